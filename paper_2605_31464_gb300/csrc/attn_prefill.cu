// Causal grouped-query attention over the prompt (prefill) on the tcgen05
// tensor cores.
//
// One CTA = two 128-row query tiles (A: rows q0 .. q0+127, B: the next 128)
// of one head of one prompt, walking 128-key tiles (two 64-token pages of the
// paged KV cache) up to the diagonal.  The two tiles share every K and V tile
// and take turns on the tensor core: while the softmax warps of one tile
// exponentiate, the MMA thread runs the other tile's products.
//   warp 0      TMA producer: both Q tiles once; K(0) alone, then V(t) with
//               K(t+1) on one barrier, into two-deep rings
//   warp 1      one thread issues, per key tile j and query tile x,
//               O_x += P_x(j) V(j) and S_x(j+1) = Q_x K(j+1)^T, alternating
//               A and B; P_x is read straight from tensor memory.  The tensor
//               core queues only about one MMA beyond the one it runs, so
//               every instruction this thread spends between MMAs is idle
//               tensor time: the operand descriptors are built once and moved
//               by one add per MMA, each iteration waits once for both rings
//               and frees both with one commit, and only a tile's last P V
//               commits to o_done.
//   warps 2, 3  idle (they complete the first warpgroup, which hands most of
//               its registers to the softmax warpgroups)
//   warps 4..7  softmax of tile A, warps 8..11 softmax of tile B: thread r
//               owns query row r (TMEM lane r), reads its whole score row in
//               one tensor-memory load, writes P = exp2(s - m) as bf16 over the
//               first 64 columns of its own S tile in one store (the next S of
//               that tile overwrites them only after P V has read them: the
//               tensor core runs one thread's MMAs in order) and keeps the row
//               sum l.  o = O / l is the same for any reference m shared by O
//               and l: the first key tile sets m to its row max, and later
//               tiles are exponentiated against it without a row max unless
//               their row sum shows values that could overflow, in which case
//               m is raised, O and l rescaled, and the tile done again.
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
  // 80 and the two softmax warpgroups take 208: 128 * 80 + 256 * 208 = 63,488 <= 384 * 168 = 64,512
  static_assert(128 * 80 + 256 * 208 <= 384 * 168, "register hand-off exceeds the launch allocation");
  static constexpr uint32_t REGS_PRODUCER = 80;
  static constexpr uint32_t REGS_SOFTMAX = 208;
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
  uint64_t* vk_full = bar + 1;   // [2] V(t) and K(t+1) have landed (phase t >> 1 of slot t & 1)
  uint64_t* it_done = bar + 3;   // [2] the products of key-tile iteration j are done (phase j >> 1 of slot j & 1):
                                 //     V(j) and K(j+1) have been read
  uint64_t* k0_full = bar + 5;   // K(0) has landed
  uint64_t* k0_free = bar + 7;   // the first score products are done: K(0) has been read
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
      mbar_init(&vk_full[i], 1);
      mbar_init(&it_done[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], 128);
      mbar_init(&o_done[i], 1);
    }
    mbar_init(k0_free, 1);
    mbar_init(k0_full, 1);
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
        // pages of 128-key tile t; a missing second page re-reads the first (its keys are masked)
        auto load_k = [&](int t, uint64_t* full) {
          const int st = t & 1;
          const int pg0 = pages[2 * t];
          const int pg1 = (2 * t + 1 < n_pages) ? pages[2 * t + 1] : pg0;
#pragma unroll
          for (int h = 0; h < C::HALVES; ++h) {
            uint8_t* dst = sK + st * C::K_BYTES + h * C::K_BLOCK;
            tma_load_2d(dst, &tmK, full, h * 64, (int)(a.layer_row0 + ((int64_t)pg0 * a.n_kv + kvh) * 64));
            tma_load_2d(dst + 64 * 128, &tmK, full, h * 64, (int)(a.layer_row0 + ((int64_t)pg1 * a.n_kv + kvh) * 64));
          }
        };
        // V(t) with K(t+1) (when there is one) on one barrier: the products of iteration t read both
        auto load_pair = [&](int t, bool with_k) {
          const int st = t & 1;
          const int pg0 = pages[2 * t];
          const int pg1 = (2 * t + 1 < n_pages) ? pages[2 * t + 1] : pg0;
          mbar_arrive_expect_tx(&vk_full[st], C::V_BYTES + (t + 1 < n_max ? C::K_BYTES : 0));
          uint8_t* dv = sV + st * C::V_BYTES;
          tma_load_2d(dv, &tmV, &vk_full[st], 0, (int)(a.layer_vrow0 + ((int64_t)pg0 * a.n_kv + kvh) * HD));
          tma_load_2d(dv + C::V_BLOCK, &tmV, &vk_full[st], 0, (int)(a.layer_vrow0 + ((int64_t)pg1 * a.n_kv + kvh) * HD));
          if (with_k && t + 1 < n_max) load_k(t + 1, &vk_full[st]);
        };
        // K(0) alone; then (V(0), K(1)) and V(1) into empty slots, K(2) (counted on V(1)'s barrier) once the
        // first score products have read K(0); after iteration j, (V(j + 2), K(j + 3)) into the slots it freed
        mbar_arrive_expect_tx(k0_full, C::K_BYTES);
        load_k(0, k0_full);
        load_pair(0, true);
        int pairs = 1;
        bool ok = true;
        if (n_max > 1) {
          load_pair(1, false);
          ++pairs;
          if (n_max > 2) {
            ok = mbar_wait(k0_free, 0, a.err);
            if (ok) load_k(2, &vk_full[1]);
          }
        }
        for (int j = 0; j + 2 < n_max && ok; ++j) {
          if (!mbar_wait(&it_done[j & 1], (j >> 1) & 1, a.err)) { ok = false; break; }
          load_pair(j + 2, true);
          ++pairs;
        }
        // copies still in flight must land before the CTA exits
        mbar_wait_drain(q_full, 0);
        mbar_wait_drain(k0_full, 0);
        for (int t = max(0, pairs - 2); t < pairs; ++t) mbar_wait_drain(&vk_full[t & 1], (t >> 1) & 1);
      }
    } else if (warp == 1) {
      // -------------------------------------------------------------- MMA issuer
      if (lane == 0) {
        bool ok = mbar_wait(q_full, 0, a.err) && mbar_wait(k0_full, 0, a.err);
        tc_fence_after();
        bool any = false;
        // operand descriptors of the query tiles and ring slots, built once; an MMA's K step only
        // moves the start address
        const uint64_t dq0 = sdesc_k_sw128(smem_u32(sQ)), dq1 = sdesc_k_sw128(smem_u32(sQ + C::Q_BYTES));
        const uint64_t dk0 = sdesc_k_sw128(smem_u32(sK)), dk1 = sdesc_k_sw128(smem_u32(sK + C::K_BYTES));
        const uint64_t dv0 = sdesc_k_sw128(smem_u32(sV)), dv1 = sdesc_k_sw128(smem_u32(sV + C::V_BYTES));
        // S_x(j) = Q_x K(j)^T into the S_x columns (K(j) has landed)
        auto issue_s = [&](int x, int j) {
          const uint32_t d = tmem + C::s_col(x);
          const uint64_t qd = x ? dq1 : dq0, kd = (j & 1) ? dk1 : dk0;
#pragma unroll
          for (int ks = 0; ks < HD / 16; ++ks) {
            const uint32_t off = (ks & 3) * 32;
            umma_bf16(d, sdesc_add(qd, (ks >> 2) * (C::Q_BYTES / C::HALVES) + off),
                      sdesc_add(kd, (ks >> 2) * C::K_BLOCK + off), IDESC_S, ks > 0 ? 1u : 0u);
          }
          umma_commit(&s_full[x]);
          any = true;
        };
        // O_x += P_x(j) V(j), P_x(j) in the first 64 columns of S_x (V(j) has landed)
        auto issue_pv = [&](int x, int j) -> bool {
          if (!mbar_wait(&p_full[x], j & 1, a.err)) return false;
          tc_fence_after();
          const uint32_t d = tmem + C::o_col(x);
          const uint32_t p_tmem = tmem + C::s_col(x);
          const uint64_t vd = (j & 1) ? dv1 : dv0;
#pragma unroll
          for (int ks = 0; ks < C::BKV / 16; ++ks) {
            umma_bf16_ts(d, p_tmem + ks * 8, sdesc_add(vd, (ks >> 2) * C::V_BLOCK + (ks & 3) * 32), IDESC_O,
                         (j > 0 || ks > 0) ? 1u : 0u);
          }
          // the tile's last product: its output can be read
          if (j == n_t[x] - 1) umma_commit(&o_done[x]);
          return true;
        };
        if (ok) {
          issue_s(0, 0);
          if (n_t[1] > 0) issue_s(1, 0);
          umma_commit(k0_free);
        }
        // one wait per iteration for V(j) and K(j+1), one commit per iteration freeing both slots
        for (int j = 0; j < n_max && ok; ++j) {
          ok = mbar_wait(&vk_full[j & 1], (j >> 1) & 1, a.err);
          tc_fence_after();
          if (ok && j < n_t[0]) {
            ok = issue_pv(0, j);
            if (ok && j + 1 < n_t[0]) issue_s(0, j + 1);
          }
          if (ok && j < n_t[1]) {
            ok = issue_pv(1, j);
            if (ok && j + 1 < n_t[1]) issue_s(1, j + 1);
          }
          if (ok) umma_commit(&it_done[j & 1]);
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
    // wait until the tile's last P V has completed (one phase; warp-uniform)
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
      tmem_ld128(s_addr, v);
      tmem_ld_wait();
      if (masked) {
#pragma unroll
        for (int i = 0; i < C::BKV; ++i)
          if (i >= lim) v[i] = __float_as_uint(-INFINITY);
      }
      // P = exp2(s - m) as bf16 pairs (keys 2c, 2c+1 in column c) over S columns 0..63, and row sums
      const uint64_t scale2 = f32x2(a.scale_log2, a.scale_log2);
      uint64_t ps2[4];
      uint32_t pk[C::BKV / 2];
      auto exps = [&](float neg_m) {
        const uint64_t shift2 = f32x2(neg_m, neg_m);
#pragma unroll
        for (int k = 0; k < 4; ++k) ps2[k] = 0ull;
#pragma unroll
        for (int i = 0; i < C::BKV; i += 2) {
          const uint64_t t = fma_f32x2(f32x2(__uint_as_float(v[i]), __uint_as_float(v[i + 1])), scale2, shift2);
          const uint64_t pp = f32x2(ex2_approx(f32x2_lo(t)), ex2_approx(f32x2_hi(t)));
          ps2[(i >> 1) & 3] = add_f32x2(ps2[(i >> 1) & 3], pp);
          pk[i >> 1] = pack_bf16(f32x2_lo(pp), f32x2_hi(pp));
        }
      };
      auto row_sum = [&]() {
        float ps[8];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          ps[2 * k] = f32x2_lo(ps2[k]);
          ps[2 * k + 1] = f32x2_hi(ps2[k]);
        }
        return ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
      };
      // row max by a tree of independent partial maxima
      auto row_max = [&]() {
        float pm[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) pm[k] = fmaxf(__uint_as_float(v[2 * k]), __uint_as_float(v[2 * k + 1]));
#pragma unroll
        for (int i = 16; i < C::BKV; i += 2)
          pm[(i >> 1) & 7] = fmax3(pm[(i >> 1) & 7], __uint_as_float(v[i]), __uint_as_float(v[i + 1]));
        return fmax3(fmax3(pm[0], pm[1], pm[2]), fmax3(pm[3], pm[4], pm[5]), fmaxf(pm[6], pm[7])) * a.scale_log2;
      };
      // o = O / l is the same for any common reference m.  The first tile sets m to its row max; later
      // tiles are exponentiated against it unless that could overflow: a row sum above 2^100 (or not
      // finite) takes the tile's max as the new reference, rescales O and l, and exponentiates again.
      // An accepted tile adds at most 2^100 to l, so over at most 2^14 key tiles l < 2^114 and
      // |O| < 2^114 max|v|: finite in fp32, and every P finite in bf16, whose relative precision does
      // not depend on the scale.
      float rs;
      if (j == 0) {
        m_ref = row_max();
        exps(-m_ref);
        rs = row_sum();
      } else {
        exps(-m_ref);
        rs = row_sum();
        const bool redo = !(rs <= 0x1p100f);
        if (__any_sync(0xffffffffu, redo)) {
          // the scores again (S_x still holds them)
          tmem_ld128(s_addr, v);
          tmem_ld_wait();
          if (masked) {
#pragma unroll
            for (int i = 0; i < C::BKV; ++i)
              if (i >= lim) v[i] = __float_as_uint(-INFINITY);
          }
          const float m_new = redo ? fmaxf(row_max(), m_ref) : m_ref;
          const float f = exp2f(m_ref - m_new);
          // P_x(j-1) V(j-1) was issued before S_x(j), whose completion this thread has seen
#pragma unroll 1
          for (int c = 0; c < HD / 32; ++c) {
            uint32_t ov[32];
            tmem_ld32(o_addr + c * 32, ov);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 32; ++i) ov[i] = __float_as_uint(__uint_as_float(ov[i]) * f);
            tmem_st32(o_addr + c * 32, ov);
          }
          l_run *= f;
          m_ref = m_new;
          exps(-m_ref);
          rs = row_sum();
        }
      }
      tmem_st64(s_addr, pk);
      l_run += rs;
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&p_full[x]);
    }
    if (ok && wait_o(0)) {
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
