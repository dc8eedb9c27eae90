// Decode attention over the paged KV cache: one new query token per sequence.
//
// Grid (split, kv_head, sequence).  A CTA takes `chunk` keys of one sequence
// and one KV head and serves every query head of that group at once (the G
// heads of a GQA group are the 16 rows of a warp MMA, zero-padded), so each
// K/V page is read from HBM once per step.  A K page (64 tokens x head_dim)
// and a V page (stored transposed, head_dim x 64 tokens) arrive by TMA,
// double-buffered; warp w takes keys 16w..16w+15 of each page.
// Each CTA writes an unnormalised partial (running max, running sum, sum of
// p.v) for its chunk; attn_combine merges the chunks of a sequence.
// In the model's decode step the kernel also does the RoPE pass (see
// DecodeAttnArgs::qkv): the queries are rotated by every CTA for its group,
// and the new key (rotated) and value are written into the cache by the CTA
// whose chunk holds the new token, before its TMA reads that page; the merge
// kernel then zeroes the rows of the split-K sums that were read.
#include <mutex>

#include "gf.h"
#include "kernels.h"
#include "ptx.cuh"

namespace gf {

// Most pages one decode-attention CTA may read (its page numbers are kept in shared memory).
constexpr int kDecodeMaxChunkPages = 64;

#ifndef GF_DECODE_STAGES
#define GF_DECODE_STAGES 2
#endif

template <int HD>
struct DecodeCfg {
  static constexpr int STAGES = GF_DECODE_STAGES;   // pages (K + V^T) in flight per CTA
  static constexpr int HALVES = HD / 64;
  static constexpr int PAGE_HALF = 64 * 128;        // one 64-column half of a K page
  static constexpr int PAGE_BYTES = 64 * HD * 2;    // one page of K (or V^T) for one head
  static constexpr int Q_BYTES = 16 * HD * 2;
  // smem: Q [HALVES][16][128 B] | K[STAGES] | V[STAGES] | barriers | the chunk's page numbers [pg_cap];
  // the K/V area is reused to combine warps
  static constexpr int SMEM = 1024 + Q_BYTES + 2 * STAGES * PAGE_BYTES + 8 * STAGES;
  static constexpr int smem(int pg_cap) { return SMEM + 4 * pg_cap; }
};

template <int HD>
__global__ void __launch_bounds__(128) attn_decode_kernel(const __grid_constant__ CUtensorMap tmK,
                                                          const __grid_constant__ CUtensorMap tmV,
                                                          const DecodeAttnArgs a) {
  using C = DecodeCfg<HD>;
  pdl_trigger();
  pdl_wait();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK = sQ + C::Q_BYTES;
  uint8_t* sV = sK + C::STAGES * C::PAGE_BYTES;
  uint64_t* bar = reinterpret_cast<uint64_t*>(sV + C::STAGES * C::PAGE_BYTES);  // [STAGES]
  int* spage = reinterpret_cast<int*>(bar + C::STAGES);                           // [pg_cap]

  const int split = blockIdx.x;
  const int kvh = blockIdx.y;
  const int b = blockIdx.z;
  const int slot = a.handles ? a.handles[b] : b;
  const int pos = a.seq_len[slot];  // the new token's position (fused step)
  const int ctx = min(pos + a.ctx_bias, a.max_ctx);
  const int k0 = split * a.chunk;
  if (k0 >= ctx) return;
  const int k1 = min(k0 + a.chunk, ctx);
  const int p0 = k0 >> 6;
  const int n_pages = ((k1 - 1) >> 6) - p0 + 1;
  const int G = a.n_q / a.n_kv;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int32_t* pages = a.block_table + (int64_t)slot * a.max_pages;

  auto issue = [&](int i, int page) {
    const int buf = i % C::STAGES;
    const int64_t pg = (int64_t)page * a.n_kv + kvh;
    mbar_arrive_expect_tx(&bar[buf], 2 * C::PAGE_BYTES);
#pragma unroll
    for (int h = 0; h < C::HALVES; ++h)
      tma_load_2d(sK + buf * C::PAGE_BYTES + h * C::PAGE_HALF, &tmK, &bar[buf], h * 64, (int)(a.layer_row0 + pg * 64));
    tma_load_2d(sV + buf * C::PAGE_BYTES, &tmV, &bar[buf], 0, (int)(a.layer_vrow0 + pg * HD));
  };

  const bool fused = a.qkv != nullptr;
  const bool writes_kv = fused && k1 == ctx;  // this chunk holds the new token
  // The page holding the new token is read only after this CTA has written the token into it: when
  // that page is among the first STAGES, its copy waits for the block-wide barrier below; later
  // pages are issued after the per-page barrier of the main loop anyway.
  const int first_copies = min(C::STAGES, n_pages);
  const bool defer_last = writes_kv && n_pages <= C::STAGES;
  if (threadIdx.x == 0) {
    for (int i = 0; i < C::STAGES; ++i) mbar_init(&bar[i], 1);
    fence_mbar_init();
    fence_async_smem();
    for (int i = 0; i < first_copies - (defer_last ? 1 : 0); ++i) issue(i, pages[p0 + i]);
  }
  // the chunk's page numbers, so that a later copy does not wait for a load of its page number
  for (int i = threadIdx.x; i < n_pages; i += blockDim.x) spage[i] = pages[p0 + i];
  if (fused) {
    // rotated queries of this group as bf16, swizzled like TMA; rows G..15 are zero.  Each thread
    // handles up to four (row, pair) items, all loads first.
    const float* row = a.qkv + (int64_t)b * a.ldqkv;
    const float2* cs = a.rope_cs + (int64_t)pos * (HD / 2);
    constexpr int kItems = 16 * (HD / 2) / 128;  // (row, pair) items per thread over all 16 rows
    float x0[kItems], x1[kItems];
    float2 t[kItems];
#pragma unroll
    for (int u = 0; u < kItems; ++u) {
      const int c = threadIdx.x + u * 128, r = c / (HD / 2), i = c % (HD / 2);
      x0[u] = x1[u] = 0.f;
      t[u] = make_float2(0.f, 0.f);
      if (r < G) {
        x0[u] = row[(kvh * G + r) * HD + i];
        x1[u] = row[(kvh * G + r) * HD + i + HD / 2];
        t[u] = cs[i];
      }
    }
#pragma unroll
    for (int u = 0; u < kItems; ++u) {
      const int c = threadIdx.x + u * 128, r = c / (HD / 2), i = c % (HD / 2);
      const float y0 = x0[u] * t[u].x - x1[u] * t[u].y;
      const float y1 = x1[u] * t[u].x + x0[u] * t[u].y;
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int col = i + hh * (HD / 2);
        *reinterpret_cast<bf16*>(sQ + (col >> 6) * (16 * 128) + sw128(r, (col & 63) >> 3) + (col & 7) * 2) =
            __float2bfloat16(hh ? y1 : y0);
      }
    }
    if (writes_kv) {
      const int page = pages[pos >> 6], in_page = pos & 63;
      const float* kr = row + (a.n_q + kvh) * HD;
      const float* vr = row + (a.n_q + a.n_kv + kvh) * HD;
      bf16* kd = a.k_cache + (a.layer_row0 + ((int64_t)page * a.n_kv + kvh) * 64 + in_page) * HD;
      bf16* vd = a.v_cache + a.layer_vrow0 * 64 + ((int64_t)page * a.n_kv + kvh) * HD * 64 + in_page;
      const float2* cs2 = a.rope_cs + (int64_t)pos * (HD / 2);
      for (int i = threadIdx.x; i < HD / 2; i += blockDim.x) {
        const float x0 = kr[i], x1 = kr[i + HD / 2];
        const float2 t = cs2[i];
        kd[i] = __float2bfloat16(x0 * t.x - x1 * t.y);
        kd[i + HD / 2] = __float2bfloat16(x1 * t.x + x0 * t.y);
      }
      for (int d = threadIdx.x; d < HD; d += blockDim.x) vd[(int64_t)d * 64] = __float2bfloat16(vr[d]);
      fence_async_global();  // the page's TMA read (after a block-wide barrier) must see these writes
    }
  } else {
    // Q rows of this group (zero rows beyond G), 16-byte chunks, swizzled like TMA.
    for (int c = threadIdx.x; c < 16 * (HD / 8); c += blockDim.x) {
      const int r = c / (HD / 8), ch = c % (HD / 8);
      uint4 v = make_uint4(0, 0, 0, 0);
      if (r < G) v = *reinterpret_cast<const uint4*>(a.q + (int64_t)b * a.ldq + (kvh * G + r) * HD + ch * 8);
      *reinterpret_cast<uint4*>(sQ + (ch >> 3) * (16 * 128) + sw128(r, ch & 7)) = v;
    }
  }
  __syncthreads();
  if (defer_last && threadIdx.x == 0) issue(n_pages - 1, spage[n_pages - 1]);

  uint32_t qa[HD / 16][4];
  {
    const int r = (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      const int chunk = kk * 2 + (lane >> 4);
      ldsm_x4(smem_u32(sQ + (chunk >> 3) * (16 * 128)) + sw128(r, chunk & 7), qa[kk][0], qa[kk][1], qa[kk][2],
              qa[kk][3]);
    }
  }

  float o[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_run[2] = {-INFINITY, -INFINITY};
  float l_run[2] = {0.f, 0.f};
  const int t4 = lane & 3;
  bool ok = true;
  int i_fail = 0;

  for (int i = 0; i < n_pages; ++i) {
    const int buf = i % C::STAGES;
    if (!mbar_wait(&bar[buf], (i / C::STAGES) & 1, a.err)) {
      ok = false;
      i_fail = i;
      break;
    }
    const uint8_t* k_t = sK + buf * C::PAGE_BYTES;
    const uint8_t* v_t = sV + buf * C::PAGE_BYTES;
    float s[2][4];
#pragma unroll
    for (int n = 0; n < 2; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      const int key = warp * 16 + (lane & 7) + (lane >> 4) * 8;
      const int chunk = kk * 2 + ((lane >> 3) & 1);
      uint32_t b0, b1, b2, b3;
      ldsm_x4(smem_u32(k_t + (chunk >> 3) * C::PAGE_HALF) + sw128(key, chunk & 7), b0, b1, b2, b3);
      mma_bf16_16816(s[0], qa[kk], b0, b1);
      mma_bf16_16816(s[1], qa[kk], b2, b3);
    }
    const int key_base = (p0 + i) * 64 + warp * 16;
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int n = 0; n < 2; ++n) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = key_base + n * 8 + 2 * t4 + (e & 1);
        float v = s[n][e] * a.scale_log2;
        if (key < k0 || key >= k1) v = -INFINITY;
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
    for (int n = 0; n < 2; ++n) {
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
    for (int d = 0; d < HD / 8; ++d) {
      o[d][0] *= corr[0];
      o[d][1] *= corr[0];
      o[d][2] *= corr[1];
      o[d][3] *= corr[1];
    }
    uint32_t pa[4];
    pa[0] = pack_bf16(s[0][0], s[0][1]);
    pa[1] = pack_bf16(s[0][2], s[0][3]);
    pa[2] = pack_bf16(s[1][0], s[1][1]);
    pa[3] = pack_bf16(s[1][2], s[1][3]);
    // V^T page: row = head dim, 64 keys per 128-byte row; this warp's keys are chunks 2w, 2w+1
#pragma unroll
    for (int dp = 0; dp < HD / 16; ++dp) {
      const int dim = dp * 16 + (lane & 7) + (lane >> 4) * 8;
      const int chunk = warp * 2 + ((lane >> 3) & 1);
      uint32_t b0, b1, b2, b3;
      ldsm_x4(smem_u32(v_t) + sw128(dim, chunk), b0, b1, b2, b3);
      mma_bf16_16816(o[2 * dp], pa, b0, b1);
      mma_bf16_16816(o[2 * dp + 1], pa, b2, b3);
    }
    __syncthreads();
    if (threadIdx.x == 0 && i + C::STAGES < n_pages) issue(i + C::STAGES, spage[i + C::STAGES]);
  }

  if (!ok) {
    if (threadIdx.x == 0)
      for (int i = i_fail; i < min(n_pages, i_fail + C::STAGES); ++i)
        mbar_wait_drain(&bar[i % C::STAGES], (i / C::STAGES) & 1);
    return;
  }

  // ---- combine the four warps (K/V buffers are free now)
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 1);
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 2);
  }
  float* red_o = reinterpret_cast<float*>(sK);          // [4 warps][16 rows][HD]
  float* red_ml = red_o + 4 * 16 * HD;                  // [4 warps][16 rows][2]
  const int g = lane >> 2;
#pragma unroll
  for (int d = 0; d < HD / 8; ++d) {
    const int col = d * 8 + 2 * t4;
    red_o[(warp * 16 + g) * HD + col] = o[d][0];
    red_o[(warp * 16 + g) * HD + col + 1] = o[d][1];
    red_o[(warp * 16 + g + 8) * HD + col] = o[d][2];
    red_o[(warp * 16 + g + 8) * HD + col + 1] = o[d][3];
  }
  if (t4 == 0) {
    red_ml[(warp * 16 + g) * 2] = m_run[0];
    red_ml[(warp * 16 + g) * 2 + 1] = l_run[0];
    red_ml[(warp * 16 + g + 8) * 2] = m_run[1];
    red_ml[(warp * 16 + g + 8) * 2 + 1] = l_run[1];
  }
  __syncthreads();
  const int64_t part = ((int64_t)b * a.n_kv + kvh) * a.max_splits + split;
  for (int idx = threadIdx.x; idx < G * HD; idx += blockDim.x) {
    const int r = idx / HD, d = idx % HD;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, red_ml[(w * 16 + r) * 2]);
    float L = 0.f, O = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float mw = red_ml[(w * 16 + r) * 2];
      const float f = (mw == -INFINITY) ? 0.f : exp2f(mw - M);
      L += red_ml[(w * 16 + r) * 2 + 1] * f;
      O += red_o[(w * 16 + r) * HD + d] * f;
    }
    a.part_o[(part * 16 + r) * HD + d] = O;
    if (d == 0) {
      a.part_ml[(part * 16 + r) * 2] = M;
      a.part_ml[(part * 16 + r) * 2 + 1] = L;
    }
  }
}

// Merge the per-chunk partials of each (sequence, query head) and normalise.
template <int HD>
__global__ void attn_combine_kernel(const DecodeAttnArgs a) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x / a.n_q;
  const int h = blockIdx.x % a.n_q;
  const int G = a.n_q / a.n_kv;
  const int kvh = h / G, r = h % G;
  const int ctx = min(a.seq_len[a.handles ? a.handles[b] : b] + a.ctx_bias, a.max_ctx);
  const int n_splits = ctx > 0 ? min((ctx + a.chunk - 1) / a.chunk, a.max_splits) : 0;
  const int64_t base = ((int64_t)b * a.n_kv + kvh) * a.max_splits;
  float M = -INFINITY;
  for (int s = 0; s < n_splits; ++s) M = fmaxf(M, a.part_ml[((base + s) * 16 + r) * 2]);
  for (int d = threadIdx.x; d < HD; d += blockDim.x) {
    float L = 0.f, O = 0.f;
    for (int s = 0; s < n_splits; ++s) {
      const float ms = a.part_ml[((base + s) * 16 + r) * 2];
      const float f = (ms == -INFINITY) ? 0.f : exp2f(ms - M);
      L += a.part_ml[((base + s) * 16 + r) * 2 + 1] * f;
      O += a.part_o[((base + s) * 16 + r) * HD + d] * f;
    }
    a.out[(int64_t)b * a.ldo + h * HD + d] = __float2bfloat16(L > 0.f ? O / L : 0.f);
  }
  if (a.qkv) {
    // fused step: every attention CTA has read its queries and the new key and value; zero the
    // split-K sums of this query head (and of the group's key and value heads) for the next step
    float* row = a.qkv + (int64_t)b * a.ldqkv;
    for (int d = threadIdx.x; d < HD; d += blockDim.x) {
      row[h * HD + d] = 0.f;
      if (r == 0) {
        row[(a.n_q + kvh) * HD + d] = 0.f;
        row[(a.n_q + a.n_kv + kvh) * HD + d] = 0.f;
      }
    }
  }
}

template <int HD>
static cudaError_t launch_hd(const CUtensorMap& tmK, const CUtensorMap& tmV, const DecodeAttnArgs& a, int B,
                             cudaStream_t s) {
  // the shared-memory limit is an attribute of the function in one device's context: set it once per context
  static DeviceOnce configured;
  cudaError_t e = configured.run([] {
    return cudaFuncSetAttribute(attn_decode_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                DecodeCfg<HD>::smem(kDecodeMaxChunkPages));
  });
  if (e != cudaSuccess) return e;
  if (B == 0) return cudaSuccess;
  const int pg_cap = a.chunk / 64;  // pages one CTA reads
  if (a.chunk < 64 || a.chunk % 64 || pg_cap > kDecodeMaxChunkPages) return cudaErrorInvalidValue;
  dim3 grid(a.max_splits, a.n_kv, B);
  e = launch_pdl(attn_decode_kernel<HD>, grid, dim3(128), DecodeCfg<HD>::smem(pg_cap), s, tmK, tmV, a);
  if (e != cudaSuccess) return e;
  return launch_pdl(attn_combine_kernel<HD>, dim3(B * a.n_q), dim3(HD), 0, s, a);
}

cudaError_t launch_attn_decode(int hd, const CUtensorMap& tmK, const CUtensorMap& tmV, const DecodeAttnArgs& a,
                               int B, cudaStream_t s) {
  if (a.n_q / a.n_kv > 16) return cudaErrorInvalidValue;
  if (hd == 128) return launch_hd<128>(tmK, tmV, a, B, s);
  if (hd == 64) return launch_hd<64>(tmK, tmV, a, B, s);
  return cudaErrorInvalidValue;
}

}  // namespace gf

// ---------------------------------------------------------------------------
// gf_decode_attention_static: the same kernels with their scratch (the
// per-chunk partial results and the timeout word) in fixed device arrays of
// this module instead of caller or runtime allocations.
namespace {
constexpr size_t kStaticScratchBytes = size_t(16) << 20;  // 16 MiB, held by every GPU that loads the library
constexpr int kMaxDevices = 64;
// Device addresses of the arrays, looked up once per device and CUDA context (ctx = its unique id).
struct StaticAddrs {
  uint64_t ctx = 0;
  void* scratch = nullptr;
  int* err = nullptr;
};
std::mutex g_static_mu;
StaticAddrs g_static[kMaxDevices];
}  // namespace

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];
// Timeout word of the allocation-free entry point: set by a bounded wait that gave up, cleared only by
// gf_decode_attention_static_status (zero when the module is loaded).
static __device__ __align__(256) int g_static_err;

// Set-up, with the device current: the device addresses of the two arrays.  In host code their names
// stand for host-side shadows, not device memory, so the kernels get the addresses
// cudaGetSymbolAddress reports.  The lookup runs on the first call in each context of a device (it
// may load this module there, which is why the first call must not fall inside a stream capture) and
// again in a context made later, after cudaDeviceReset; it allocates nothing itself.
static int static_addrs(void** scratch, int** err) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    gf::set_error_short("no CUDA device");
    return GF_ECUDA;
  }
  if (dev < 0 || dev >= kMaxDevices) {
    gf::set_error_short("too many GPUs");
    return GF_ENOTIMPL;
  }
  const uint64_t ctx = gf::current_context_id();
  std::lock_guard<std::mutex> lock(g_static_mu);
  StaticAddrs& a = g_static[dev];
  if (ctx == 0 || a.ctx != ctx || !a.scratch) {
    void* sp = nullptr;
    void* ep = nullptr;
    if (cudaGetSymbolAddress(&sp, g_static_scratch) != cudaSuccess ||
        cudaGetSymbolAddress(&ep, g_static_err) != cudaSuccess || !sp || !ep) {
      cudaGetLastError();
      gf::set_error_short("symbol lookup");
      return GF_ECUDA;
    }
    a.ctx = ctx;
    a.scratch = sp;
    a.err = reinterpret_cast<int*>(ep);
  }
  *scratch = a.scratch;
  *err = a.err;
  return GF_OK;
}

extern "C" int gf_decode_attention_static(const void* q, const void* k_cache, const void* v_cache, int64_t num_pages,
                                          const int32_t* block_table, int32_t max_pages, const int32_t* ctx_len,
                                          int32_t max_ctx, int32_t B, int32_t n_q, int32_t n_kv, int32_t head_dim,
                                          void* out, void* stream) {
  if (!q || !k_cache || !v_cache || !block_table || !ctx_len || !out || B < 1 || n_q < 1 || n_kv < 1 ||
      n_q % n_kv || n_q / n_kv > 16 || max_ctx < 1 || max_pages < 1 || max_ctx > max_pages * 64 || num_pages < 1 ||
      num_pages * n_kv * 64 >= ((int64_t)1 << 31)) {
    gf::set_error_short("bad argument");
    return GF_EINVAL;
  }
  if (head_dim != 64 && head_dim != 128) {
    gf::set_error_short("head_dim 64/128");
    return GF_ENOTIMPL;
  }
  const size_t need = gf_decode_attention_workspace(B, n_kv, head_dim, max_ctx);
  if (need > kStaticScratchBytes) {
    gf::set_error_short("exceeds scratch");
    return GF_ECAPACITY;
  }
  void* scratch = nullptr;
  int* err = nullptr;
  const int rc = static_addrs(&scratch, &err);
  if (rc != GF_OK) return rc;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // Nothing in the scratch needs clearing: every partial the merge reads is written first by this
  // call.  The timeout word is not cleared here, so that a timeout stays visible to
  // gf_decode_attention_static_status however many calls follow it.
  CUtensorMap tk, tv;
  const uint64_t rows = (uint64_t)num_pages * n_kv * 64;
  if (gf::encode_kv_map(&tk, k_cache, head_dim, rows) ||
      gf::encode_vt_map(&tv, v_cache, head_dim, (uint64_t)num_pages * n_kv * head_dim)) {
    gf::set_error_short("tensor map");
    return GF_ECUDA;
  }
  gf::DecodeAttnArgs da{};
  da.q = reinterpret_cast<const gf::bf16*>(q);
  da.ldq = (int64_t)n_q * head_dim;
  da.handles = nullptr;
  da.seq_len = ctx_len;
  da.ctx_bias = 0;
  da.max_ctx = max_ctx;
  da.block_table = block_table;
  da.max_pages = max_pages;
  da.n_q = n_q;
  da.n_kv = n_kv;
  da.layer_row0 = 0;
  da.layer_vrow0 = 0;
  da.chunk = 256;
  da.max_splits = (max_ctx + 255) / 256;
  da.part_o = reinterpret_cast<float*>(scratch);
  da.part_ml = da.part_o + (size_t)B * n_kv * da.max_splits * 16 * head_dim;
  da.out = reinterpret_cast<gf::bf16*>(out);
  da.ldo = (int64_t)n_q * head_dim;
  da.scale_log2 = 1.4426950408889634f / sqrtf((float)head_dim);
  da.err = err;
  if (gf::launch_attn_decode(head_dim, tk, tv, da, B, s) != cudaSuccess) {
    cudaGetLastError();
    gf::set_error_short("launch failed");
    return GF_ECUDA;
  }
  return GF_OK;
}

extern "C" int gf_decode_attention_static_status(void* stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    gf::set_error_short("sync failed");
    return GF_ECUDA;
  }
  void* scratch = nullptr;
  int* err = nullptr;
  const int rc = static_addrs(&scratch, &err);
  if (rc != GF_OK) return rc;
  int h = 0;
  if (cudaMemcpyAsync(&h, err, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaMemsetAsync(err, 0, sizeof(int), s) != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    gf::set_error_short("status read");
    return GF_ECUDA;
  }
  if (h == gf::kErrTimeout) {
    gf::set_error_short("wait timed out");
    return GF_ETIMEOUT;
  }
  return GF_OK;
}

extern "C" int gf_selftest_timeout_static(uint32_t limit_ms, void* stream) {
  if (limit_ms < 1 || limit_ms > 2000) {
    gf::set_error_short("bad limit");
    return GF_EINVAL;
  }
  void* scratch = nullptr;
  int* err = nullptr;
  const int rc = static_addrs(&scratch, &err);
  if (rc != GF_OK) return rc;
  if (gf::launch_timeout_probe((uint64_t)limit_ms * 1000000ull, err, reinterpret_cast<cudaStream_t>(stream)) !=
      cudaSuccess) {
    cudaGetLastError();
    gf::set_error_short("launch failed");
    return GF_ECUDA;
  }
  return gf_decode_attention_static_status(stream);
}
