// Causal grouped-query attention over the prompt (prefill).
//
// One CTA = 128 query rows of one head of one prompt; 8 warps own 16 rows
// each.  Q (two 64-column halves) and every 64-key K/V tile arrive by TMA
// with 128-byte swizzling; K/V tiles are read straight from the paged KV
// cache (a tile is one 64-token page).  Scores and P.V use bf16 warp MMAs with
// fp32 accumulation and an online (running max / running sum) softmax in the
// log2 domain; the output is normalised once at the end.
#include "kernels.h"
#include "ptx.cuh"

namespace gf {

template <int HD>
struct PrefillCfg {
  static constexpr int BQ = 128;
  static constexpr int BKV = 64;
  static constexpr int HALVES = HD / 64;
  static constexpr int Q_BYTES = BQ * HD * 2;
  static constexpr int Q_HALF = BQ * 128;   // bytes of one 64-column half of Q
  static constexpr int KV_HALF = BKV * 128; // bytes of one 64-column half of a K or V tile
  static constexpr int KV_BYTES = BKV * HD * 2;
  static constexpr int SMEM = 1024 + Q_BYTES + 4 * KV_BYTES + 64;
};

template <int HD>
__global__ void __launch_bounds__(256) attn_prefill_kernel(const __grid_constant__ CUtensorMap tmQ,
                                                           const __grid_constant__ CUtensorMap tmK,
                                                           const __grid_constant__ CUtensorMap tmV,
                                                           const PrefillAttnArgs a) {
  using C = PrefillCfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;                          // [HALVES][128 rows][128 B]
  uint8_t* sK = sQ + C::Q_BYTES;               // [2 bufs][HALVES][64][128 B]
  uint8_t* sV = sK + 2 * C::KV_BYTES;
  uint64_t* bar_q = reinterpret_cast<uint64_t*>(sV + 2 * C::KV_BYTES);
  uint64_t* bar_kv = bar_q + 1;                // [2]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int head = blockIdx.x % a.n_q;
  const int2 item = a.items[blockIdx.x / a.n_q];
  const int b = item.x;
  const int q0 = item.y * C::BQ;
  const int seq_start = a.offsets[b];
  const int len = a.offsets[b + 1] - seq_start;
  const int kvh = head / (a.n_q / a.n_kv);
  const int slot = a.slots[b];
  const int32_t* pages = a.block_table + (int64_t)slot * a.max_pages;
  const int n_tiles = (min(q0 + C::BQ, len) + C::BKV - 1) / C::BKV;

  auto issue_kv = [&](int j) {
    const int buf = j & 1;
    const int64_t row = a.layer_row0 + ((int64_t)pages[j] * a.n_kv + kvh) * 64;
    mbar_arrive_expect_tx(&bar_kv[buf], 2 * C::KV_BYTES);
#pragma unroll
    for (int h = 0; h < C::HALVES; ++h) {
      tma_load_2d(sK + buf * C::KV_BYTES + h * C::KV_HALF, &tmK, &bar_kv[buf], h * 64, (int)row);
      tma_load_2d(sV + buf * C::KV_BYTES + h * C::KV_HALF, &tmV, &bar_kv[buf], h * 64, (int)row);
    }
  };

  if (threadIdx.x == 0) {
    mbar_init(bar_q, 1);
    mbar_init(&bar_kv[0], 1);
    mbar_init(&bar_kv[1], 1);
    fence_mbar_init();
    fence_async_smem();
    mbar_arrive_expect_tx(bar_q, C::Q_BYTES);
#pragma unroll
    for (int h = 0; h < C::HALVES; ++h)
      tma_load_2d(sQ + h * C::Q_HALF, &tmQ, bar_q, head * HD + h * 64, seq_start + q0);
    issue_kv(0);
    if (n_tiles > 1) issue_kv(1);
  }
  __syncthreads();

  bool ok = mbar_wait(bar_q, 0, a.err);

  // Q fragments: rows 16*warp .. +15, all HD columns.
  uint32_t qa[HD / 16][4];
  {
    const int r = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      const int chunk = kk * 2 + (lane >> 4);
      const uint32_t addr = smem_u32(sQ + (chunk >> 3) * C::Q_HALF) + sw128(r, chunk & 7);
      ldsm_x4(addr, qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3]);
    }
  }

  float o[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_run[2] = {-INFINITY, -INFINITY};
  float l_run[2] = {0.f, 0.f};
  const int g = lane >> 2, t4 = lane & 3;
  const int qpos0 = q0 + warp * 16 + g;  // position of fragment row g; row g+8 is qpos0 + 8

  int j_fail = 0;
  for (int j = 0; j < n_tiles && ok; ++j) {
    const int buf = j & 1;
    if (!mbar_wait(&bar_kv[buf], (j >> 1) & 1, a.err)) {
      ok = false;
      j_fail = j;
      break;
    }
    const uint8_t* k_t = sK + buf * C::KV_BYTES;
    const uint8_t* v_t = sV + buf * C::KV_BYTES;
    // ---- S = Q K^T (16 x 64 per warp)
    float s[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        const int key = np * 16 + (lane & 7) + (lane >> 4) * 8;
        const int chunk = kk * 2 + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(k_t + (chunk >> 3) * C::KV_HALF) + sw128(key, chunk & 7), b0, b1, b2, b3);
        mma_bf16_16816(s[2 * np], qa[kk], b0, b1);
        mma_bf16_16816(s[2 * np + 1], qa[kk], b2, b3);
      }
    }
    // ---- mask, online softmax
    const int key0 = j * C::BKV;
    const bool need_mask = (key0 + C::BKV - 1 > q0 + warp * 16) || (key0 + C::BKV > len);
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int n = 0; n < 8; ++n) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float v = s[n][e] * a.scale_log2;
        if (need_mask) {
          const int key = key0 + n * 8 + 2 * t4 + (e & 1);
          const int qp = qpos0 + (e >> 1) * 8;
          if (key > qp || key >= len) v = -INFINITY;
        }
        s[n][e] = v;
        mx[e >> 1] = fmaxf(mx[e >> 1], v);
      }
    }
    float corr[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
      const float m_new = fmaxf(m_run[r], mx[r]);
      const float m_use = (m_new == -INFINITY) ? 0.f : m_new;
      corr[r] = exp2f(m_run[r] - m_use);
      m_run[r] = m_new;
      mx[r] = m_use;
    }
    float rs[2] = {0.f, 0.f};
#pragma unroll
    for (int n = 0; n < 8; ++n) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float pv = exp2f(s[n][e] - mx[e >> 1]);
        s[n][e] = pv;
        rs[e >> 1] += pv;
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) l_run[r] = l_run[r] * corr[r] + rs[r];
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) {
      o[i][0] *= corr[0];
      o[i][1] *= corr[0];
      o[i][2] *= corr[1];
      o[i][3] *= corr[1];
    }
    // ---- O += P V
#pragma unroll
    for (int kk2 = 0; kk2 < 4; ++kk2) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * kk2][0], s[2 * kk2][1]);
      pa[1] = pack_bf16(s[2 * kk2][2], s[2 * kk2][3]);
      pa[2] = pack_bf16(s[2 * kk2 + 1][0], s[2 * kk2 + 1][1]);
      pa[3] = pack_bf16(s[2 * kk2 + 1][2], s[2 * kk2 + 1][3]);
#pragma unroll
      for (int dp = 0; dp < HD / 16; ++dp) {
        const int key = kk2 * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int chunk = dp * 2 + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(smem_u32(v_t + (chunk >> 3) * C::KV_HALF) + sw128(key, chunk & 7), b0, b1, b2, b3);
        mma_bf16_16816(o[2 * dp], pa, b0, b1);
        mma_bf16_16816(o[2 * dp + 1], pa, b2, b3);
      }
    }
    __syncthreads();  // every warp is done with this buffer
    if (threadIdx.x == 0 && j + 2 < n_tiles) issue_kv(j + 2);
  }

  if (!ok) {
    // Tiles j_fail and j_fail+1 may still be in flight: let them land before the CTA exits.
    if (threadIdx.x == 0) {
      mbar_wait_drain(bar_q, 0);
      for (int j = j_fail; j < min(n_tiles, j_fail + 2); ++j) mbar_wait_drain(&bar_kv[j & 1], (j >> 1) & 1);
    }
    return;
  }

  // ---- normalise and store
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 1);
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 2);
  }
  const float inv0 = l_run[0] > 0.f ? 1.f / l_run[0] : 0.f;
  const float inv1 = l_run[1] > 0.f ? 1.f / l_run[1] : 0.f;
  const int row0 = qpos0, row1 = qpos0 + 8;
  bf16* out0 = a.out + (int64_t)(seq_start + row0) * a.ldo + head * HD;
  bf16* out1 = a.out + (int64_t)(seq_start + row1) * a.ldo + head * HD;
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) {
    const int col = i * 8 + 2 * t4;
    if (row0 < len) *reinterpret_cast<uint32_t*>(out0 + col) = pack_bf16(o[i][0] * inv0, o[i][1] * inv0);
    if (row1 < len) *reinterpret_cast<uint32_t*>(out1 + col) = pack_bf16(o[i][2] * inv1, o[i][3] * inv1);
  }
}

template <int HD>
static cudaError_t launch_hd(const CUtensorMap& tmQ, const CUtensorMap& tmK, const CUtensorMap& tmV,
                             const PrefillAttnArgs& a, int n_items, cudaStream_t s) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(attn_prefill_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         PrefillCfg<HD>::SMEM);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  const int64_t grid = (int64_t)n_items * a.n_q;
  if (grid == 0) return cudaSuccess;
  attn_prefill_kernel<HD><<<(unsigned)grid, 256, PrefillCfg<HD>::SMEM, s>>>(tmQ, tmK, tmV, a);
  return cudaGetLastError();
}

cudaError_t launch_attn_prefill(int hd, const CUtensorMap& tmQ, const CUtensorMap& tmK, const CUtensorMap& tmV,
                                const PrefillAttnArgs& a, int n_items, cudaStream_t s) {
  if (hd == 128) return launch_hd<128>(tmQ, tmK, tmV, a, n_items, s);
  if (hd == 64) return launch_hd<64>(tmQ, tmK, tmV, a, n_items, s);
  return cudaErrorInvalidValue;
}

}  // namespace gf
