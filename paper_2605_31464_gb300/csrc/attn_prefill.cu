// Causal grouped-query attention over the prompt (prefill) on the tcgen05
// tensor cores.
//
// One CTA = two 128-row query tiles (A: rows q0 .. q0+127, B: the next 128)
// of one head of one prompt, walking 128-key tiles (two 64-token pages of the
// paged KV cache) up to the diagonal.  The two tiles share every K and V tile
// and take turns on the tensor core: while the softmax warps of one tile
// exponentiate, the MMA thread runs the other tile's products.
//   warp 0      TMA producer: both Q tiles once; K and V^T tiles into
//               two-deep rings
//   warp 1      one thread issues, per key tile j and query tile x,
//               O_x += P_x(j-1) V(j-1) and S_x(j) = Q_x K(j)^T, alternating
//               A and B; P_x is read straight from tensor memory
//   warps 2, 3  idle (they complete the first warpgroup, which hands most of
//               its registers to the softmax warpgroups)
//   warps 4..7  softmax of tile A, warps 8..11 softmax of tile B: thread r
//               owns query row r (TMEM lane r), reads its whole score row in
//               one round trip, writes
//               P = exp2(s - m) as bf16 over the first 64 columns of its own
//               S tile (which the next S of that tile overwrites only after
//               P V has read it: the tensor core runs one thread's MMAs in
//               order) and keeps the row sum l.  The reference max m is raised
//               (and O, l rescaled in place) only when a tile's max exceeds it
//               by more than 2^8, so O and l always share the same reference
//               and o = O / l is exact.
// Tensor memory: S_A, S_B (128 columns each) and O_A, O_B (HD columns each).
// The V cache is stored transposed per page ([page][kv head][hd][64 keys]) so
// that both products read K-major operands.  Every wait is bounded.
#include "kernels.h"
#include "ptx.cuh"

namespace gf {

template <int HD>
struct FaCfg {
  static constexpr int BQ = 128;                        // rows of one query tile
  static constexpr int BKV = 128;
  static constexpr int HALVES = HD / 64;                // 64-column blocks of Q and K
  static constexpr int Q_BYTES = BQ * HD * 2;           // one query tile
  static constexpr int K_BYTES = BKV * HD * 2;          // HALVES blocks of [128 keys][64]
  static constexpr int K_BLOCK = BKV * 128;
  static constexpr int V_BYTES = HD * BKV * 2;          // 2 page blocks of [HD rows][64 keys]
  static constexpr int V_BLOCK = HD * 128;
  static constexpr int SMEM = 1024 + 2 * Q_BYTES + 2 * K_BYTES + 2 * V_BYTES + 256;
  static constexpr int THREADS = 384;
  // registers per thread: 168 at launch (three warps per scheduler); the producer warpgroup keeps
  // 64 and the two softmax warpgroups take 216: 128 * 64 + 256 * 216 = 63,488 <= 384 * 168 = 64,512
  static_assert(128 * 64 + 256 * 216 <= 384 * 168, "register hand-off exceeds the launch allocation");
  static constexpr uint32_t REGS_PRODUCER = 64;
  static constexpr uint32_t REGS_SOFTMAX = 216;
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr uint32_t s_col(int x) { return (uint32_t)(x * 128); }
  static constexpr uint32_t o_col(int x) { return (uint32_t)(256 + x * HD); }
};

template <int HD>
__global__ void __launch_bounds__(384, 1) attn_prefill_tc_kernel(const __grid_constant__ CUtensorMap tmQ,
                                                                 const __grid_constant__ CUtensorMap tmK,
                                                                 const __grid_constant__ CUtensorMap tmV,
                                                                 const PrefillAttnArgs a) {
  using C = FaCfg<HD>;
  pdl_trigger();
  pdl_wait();
  constexpr uint32_t IDESC_S = idesc_bf16_f32(128, C::BKV);
  constexpr uint32_t IDESC_O = idesc_bf16_f32(128, HD);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;                   // [2][Q_BYTES]
  uint8_t* sK = sQ + 2 * C::Q_BYTES;    // [2][K_BYTES]
  uint8_t* sV = sK + 2 * C::K_BYTES;    // [2][V_BYTES]
  uint64_t* bar = reinterpret_cast<uint64_t*>(sV + 2 * C::V_BYTES);
  uint64_t* q_full = bar;
  uint64_t* k_full = bar + 1;    // [2] ring slots
  uint64_t* k_empty = bar + 3;   // [2]
  uint64_t* v_full = bar + 5;    // [2]
  uint64_t* v_empty = bar + 7;   // [2]
  uint64_t* s_full = bar + 9;    // [2] query tiles: S_x(j) completes phase j
  uint64_t* p_full = bar + 11;   // [2] query tiles: P_x(j) written (128 arrivals)
  uint64_t* o_done = bar + 13;   // [2] query tiles: P_x(j) V(j) completes phase j
  uint64_t* mma_done = bar + 15;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar + 16);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int head = blockIdx.x % a.n_q;
  const int2 item = a.items[blockIdx.x / a.n_q];
  const int b = item.x;
  const int q0 = item.y * 2 * C::BQ;
  const int seq_start = a.offsets[b];
  const int len = a.offsets[b + 1] - seq_start;
  const int past = a.past ? a.past[b] : 0;  // keys already cached before this prompt's first token
  const int kvh = head / (a.n_q / a.n_kv);
  const int32_t* pages = a.block_table + (int64_t)a.slots[b] * a.max_pages;
  const int n_keys = past + len;
  const int n_pages = (n_keys + 63) >> 6;
  // key tiles each query tile needs (0: the tile has no rows)
  int n_t[2];
#pragma unroll
  for (int x = 0; x < 2; ++x)
    n_t[x] = (q0 + x * C::BQ < len) ? (past + min(q0 + (x + 1) * C::BQ, len) + C::BKV - 1) / C::BKV : 0;
  const int n_max = max(n_t[0], n_t[1]);

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], 1);
      mbar_init(&v_full[i], 1);
      mbar_init(&v_empty[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], 128);
      mbar_init(&o_done[i], 1);
    }
    mbar_init(mma_done, 1);
    fence_mbar_init();
    fence_async_smem();
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp < 4) {
    regs_dec<C::REGS_PRODUCER>();
    if (warp == 0) {
      // -------------------------------------------------------------- TMA producer
      if (lane == 0) {
        const int q_tiles = n_t[1] > 0 ? 2 : 1;
        mbar_arrive_expect_tx(q_full, q_tiles * C::Q_BYTES);
        for (int x = 0; x < q_tiles; ++x)
#pragma unroll
          for (int h = 0; h < C::HALVES; ++h)
            tma_load_2d(sQ + x * C::Q_BYTES + h * C::Q_BYTES / C::HALVES, &tmQ, q_full, head * HD + h * 64,
                        seq_start + q0 + x * C::BQ);
        int k_issued = 0, v_issued = 0;
        bool ok = true;
        for (int j = 0; j < n_max && ok; ++j) {
          const int st = j & 1;
          const uint32_t ph = ((j >> 1) & 1) ^ 1u;
          // pages of this 128-key tile; a missing second page re-reads the first (its keys are masked)
          const int pg0 = pages[2 * j];
          const int pg1 = (2 * j + 1 < n_pages) ? pages[2 * j + 1] : pg0;
          if (!mbar_wait(&k_empty[st], ph, a.err)) { ok = false; break; }
          mbar_arrive_expect_tx(&k_full[st], C::K_BYTES);
#pragma unroll
          for (int h = 0; h < C::HALVES; ++h) {
            uint8_t* dst = sK + st * C::K_BYTES + h * C::K_BLOCK;
            tma_load_2d(dst, &tmK, &k_full[st], h * 64, (int)(a.layer_row0 + ((int64_t)pg0 * a.n_kv + kvh) * 64));
            tma_load_2d(dst + 64 * 128, &tmK, &k_full[st], h * 64,
                        (int)(a.layer_row0 + ((int64_t)pg1 * a.n_kv + kvh) * 64));
          }
          ++k_issued;
          if (!mbar_wait(&v_empty[st], ph, a.err)) { ok = false; break; }
          mbar_arrive_expect_tx(&v_full[st], C::V_BYTES);
          uint8_t* dv = sV + st * C::V_BYTES;
          tma_load_2d(dv, &tmV, &v_full[st], 0, (int)(a.layer_vrow0 + ((int64_t)pg0 * a.n_kv + kvh) * HD));
          tma_load_2d(dv + C::V_BLOCK, &tmV, &v_full[st], 0, (int)(a.layer_vrow0 + ((int64_t)pg1 * a.n_kv + kvh) * HD));
          ++v_issued;
        }
        // copies still in flight must land before the CTA exits
        mbar_wait_drain(q_full, 0);
        for (int j = max(0, k_issued - 2); j < k_issued; ++j) mbar_wait_drain(&k_full[j & 1], (j >> 1) & 1);
        for (int j = max(0, v_issued - 2); j < v_issued; ++j) mbar_wait_drain(&v_full[j & 1], (j >> 1) & 1);
      }
    } else if (warp == 1) {
      // -------------------------------------------------------------- MMA issuer
      if (lane == 0) {
        bool ok = mbar_wait(q_full, 0, a.err);
        bool any = false;
        // S_x(j) = Q_x K(j)^T into the S_x columns
        auto issue_s = [&](int x, int j) -> bool {
          const int st = j & 1;
          if (!mbar_wait(&k_full[st], (j >> 1) & 1, a.err)) return false;
          tc_fence_after();
          const uint32_t d = tmem + C::s_col(x);
          const uint32_t q_base = smem_u32(sQ + x * C::Q_BYTES), k_base = smem_u32(sK + st * C::K_BYTES);
#pragma unroll
          for (int ks = 0; ks < HD / 16; ++ks) {
            const uint32_t off = (ks & 3) * 32;
            umma_bf16(d, sdesc_k_sw128(q_base + (ks >> 2) * (C::Q_BYTES / C::HALVES) + off),
                      sdesc_k_sw128(k_base + (ks >> 2) * C::K_BLOCK + off), IDESC_S, ks > 0 ? 1u : 0u);
          }
          umma_commit(&s_full[x]);
          any = true;
          return true;
        };
        // O_x += P_x(j) V(j), P_x(j) in the first 64 columns of S_x
        auto issue_pv = [&](int x, int j) -> bool {
          const int st = j & 1;
          if (!mbar_wait(&v_full[st], (j >> 1) & 1, a.err)) return false;
          if (!mbar_wait(&p_full[x], j & 1, a.err)) return false;
          tc_fence_after();
          const uint32_t d = tmem + C::o_col(x);
          const uint32_t p_tmem = tmem + C::s_col(x);
          const uint32_t v_base = smem_u32(sV + st * C::V_BYTES);
#pragma unroll
          for (int ks = 0; ks < C::BKV / 16; ++ks) {
            umma_bf16_ts(d, p_tmem + ks * 8, sdesc_k_sw128(v_base + (ks >> 2) * C::V_BLOCK + (ks & 3) * 32), IDESC_O,
                         (j > 0 || ks > 0) ? 1u : 0u);
          }
          umma_commit(&o_done[x]);
          return true;
        };
        for (int x = 0; x < 2 && ok; ++x)
          if (n_t[x] > 0) ok = issue_s(x, 0);
        if (ok) umma_commit(&k_empty[0]);
        for (int j = 0; j < n_max && ok; ++j) {
          for (int x = 0; x < 2 && ok; ++x) {
            if (j >= n_t[x]) continue;
            ok = issue_pv(x, j);
            if (ok && j + 1 < n_t[x]) ok = issue_s(x, j + 1);
          }
          if (!ok) break;
          umma_commit(&v_empty[j & 1]);
          if (j + 1 < n_max) umma_commit(&k_empty[(j + 1) & 1]);
        }
        if (any) {
          umma_commit(mma_done);
          mbar_wait_drain(mma_done, 0);
        }
      }
    }
  } else {
    regs_inc<C::REGS_SOFTMAX>();
    // -------------------------------------------------------------- softmax warps 4..7 (A), 8..11 (B)
    const int x = (warp - 4) >> 2;
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;  // query row within the tile = TMEM lane
    const int qrow = q0 + x * C::BQ + r;  // row of this query among the prompt's packed tokens
    const int qpos = past + qrow;       // absolute position of this query row
    const int n_tiles = n_t[x];
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    const uint32_t s_addr = tmem + lane_off + C::s_col(x);
    const uint32_t o_addr = tmem + lane_off + C::o_col(x);
    float m_ref = -INFINITY, l_run = 0.f;
    bool ok = n_tiles > 0;
    // wait until P V of tile t has completed (warp-uniform)
    auto wait_o = [&](int t) -> bool {
      return __all_sync(0xffffffffu, mbar_wait(&o_done[x], t & 1, a.err));
    };
    for (int j = 0; j < n_tiles && ok; ++j) {
      if (!__all_sync(0xffffffffu, mbar_wait(&s_full[x], j & 1, a.err))) { ok = false; break; }
      tc_fence_after();
      const int key0 = j * C::BKV;
      // causal / length mask only on the diagonal and last tiles (warp-uniform)
      const bool masked = (key0 + C::BKV - 1 > past + q0 + x * C::BQ) || (key0 + C::BKV > n_keys);
      const int lim = masked ? min(qpos + 1, n_keys) - key0 : C::BKV;  // keys [0, lim) are visible
      // the whole score row in one round trip
      uint32_t v[C::BKV];
#pragma unroll
      for (int c = 0; c < C::BKV / 32; ++c) tmem_ld32(s_addr + c * 32, *reinterpret_cast<uint32_t(*)[32]>(&v[c * 32]));
      tmem_ld_wait();
      if (masked) {
#pragma unroll
        for (int i = 0; i < C::BKV; ++i)
          if (i >= lim) v[i] = __float_as_uint(-INFINITY);
      }
      // row max by a tree of independent partial maxima
      float pm[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) pm[k] = fmaxf(__uint_as_float(v[2 * k]), __uint_as_float(v[2 * k + 1]));
#pragma unroll
      for (int i = 16; i < C::BKV; i += 2)
        pm[(i >> 1) & 7] = fmax3(pm[(i >> 1) & 7], __uint_as_float(v[i]), __uint_as_float(v[i + 1]));
      const float mx = fmax3(fmax3(pm[0], pm[1], pm[2]), fmax3(pm[3], pm[4], pm[5]), fmaxf(pm[6], pm[7])) *
                       a.scale_log2;
      // raise the reference max (rescaling O and l) only when this tile exceeds it by more than 2^8
      const bool raise = mx > m_ref + 8.f;
      if (__any_sync(0xffffffffu, raise)) {
        const float m_new = raise ? mx : m_ref;
        const float f = (m_ref == -INFINITY) ? 0.f : exp2f(m_ref - m_new);
        if (j > 0) {
          if (!wait_o(j - 1)) { ok = false; break; }
          tc_fence_after();
#pragma unroll 1
          for (int c = 0; c < HD / 32; ++c) {
            uint32_t ov[32];
            tmem_ld32(o_addr + c * 32, ov);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 32; ++i) ov[i] = __float_as_uint(__uint_as_float(ov[i]) * f);
            tmem_st32(o_addr + c * 32, ov);
          }
        }
        l_run *= f;
        m_ref = m_new;
      }
      const float neg_m = (m_ref == -INFINITY) ? 0.f : -m_ref;
      const uint64_t scale2 = f32x2(a.scale_log2, a.scale_log2), shift2 = f32x2(neg_m, neg_m);
      // P = exp2(s - m) as bf16 pairs (keys 2c, 2c+1 in column c) over S columns 0..63
      uint64_t ps2[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
      for (int c = 0; c < C::BKV / 64; ++c) {
        uint32_t pk[32];
#pragma unroll
        for (int i = 0; i < 64; i += 2) {
          const uint64_t t =
              fma_f32x2(f32x2(__uint_as_float(v[c * 64 + i]), __uint_as_float(v[c * 64 + i + 1])), scale2, shift2);
          const uint64_t pp = f32x2(ex2_approx(f32x2_lo(t)), ex2_approx(f32x2_hi(t)));
          ps2[(i >> 1) & 3] = add_f32x2(ps2[(i >> 1) & 3], pp);
          pk[i >> 1] = pack_bf16(f32x2_lo(pp), f32x2_hi(pp));
        }
        tmem_st32(s_addr + c * 32, pk);
      }
      float ps[8];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        ps[2 * k] = f32x2_lo(ps2[k]);
        ps[2 * k + 1] = f32x2_hi(ps2[k]);
      }
      const float rs = ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
      l_run += rs;
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&p_full[x]);
    }
    if (ok && wait_o(n_tiles - 1)) {
      tc_fence_after();
      const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
      uint4* dst = reinterpret_cast<uint4*>(a.out + (int64_t)(seq_start + (qrow < len ? qrow : 0)) * a.ldo + head * HD);
#pragma unroll 1
      for (int c = 0; c < HD / 32; ++c) {
        uint32_t ov[32];
        tmem_ld32(o_addr + c * 32, ov);
        tmem_ld_wait();
        if (qrow < len) {
#pragma unroll
          for (int q = 0; q < 4; ++q)
            dst[c * 4 + q] = make_uint4(
                pack_bf16(__uint_as_float(ov[8 * q]) * inv, __uint_as_float(ov[8 * q + 1]) * inv),
                pack_bf16(__uint_as_float(ov[8 * q + 2]) * inv, __uint_as_float(ov[8 * q + 3]) * inv),
                pack_bf16(__uint_as_float(ov[8 * q + 4]) * inv, __uint_as_float(ov[8 * q + 5]) * inv),
                pack_bf16(__uint_as_float(ov[8 * q + 6]) * inv, __uint_as_float(ov[8 * q + 7]) * inv));
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

template <int HD>
static cudaError_t launch_hd(const CUtensorMap& tmQ, const CUtensorMap& tmK, const CUtensorMap& tmV,
                             const PrefillAttnArgs& a, int n_items, cudaStream_t s) {
  // the shared-memory limit is an attribute of the function in one device's context: set it once per context
  static DeviceOnce configured;
  const cudaError_t e = configured.run([] {
    return cudaFuncSetAttribute(attn_prefill_tc_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                FaCfg<HD>::SMEM);
  });
  if (e != cudaSuccess) return e;
  const int64_t grid = (int64_t)n_items * a.n_q;
  if (grid == 0) return cudaSuccess;
  return launch_pdl(attn_prefill_tc_kernel<HD>, dim3((unsigned)grid), dim3(FaCfg<HD>::THREADS), FaCfg<HD>::SMEM, s,
                    tmQ, tmK, tmV, a);
}

cudaError_t launch_attn_prefill(int hd, const CUtensorMap& tmQ, const CUtensorMap& tmK, const CUtensorMap& tmV,
                                const PrefillAttnArgs& a, int n_items, cudaStream_t s) {
  if (hd == 128) return launch_hd<128>(tmQ, tmK, tmV, a, n_items, s);
  if (hd == 64) return launch_hd<64>(tmQ, tmK, tmV, a, n_items, s);
  return cudaErrorInvalidValue;
}

}  // namespace gf
