// Memory-bound kernels of the forward pass: embedding gather, RMSNorm,
// rotary embedding with the paged KV-cache write, greedy arg max, the verdict
// (restricted softmax, confidence, defer), and bookkeeping.
#include "kernels.h"
#include "ptx.cuh"

namespace gf {

// ------------------------------------------------------------------ embedding
// out[t, :] = float(table[ids[t], :]); an id outside [0, vocab) records
// GF_EINVAL in the error word and yields a zero row.  One block per token;
// every thread issues all of its 16-byte loads before using them.
constexpr int kRowThreads = 256;
constexpr int kRowVec = 8;  // 16-byte vectors per thread: rows up to 256 * 8 * 4 = 8192 fp32 / 16384 bf16

__global__ void __launch_bounds__(kRowThreads) embed_kernel(const int32_t* ids, int T, const bf16* table, int vocab,
                                                            int d, float* out, int* err) {
  pdl_trigger();
  pdl_wait();
  const int t = blockIdx.x;
  const int id = ids[t];
  float* dst = out + (int64_t)t * d;
  const int nv = d / 8;  // uint4 (8 bf16) per row
  if (id < 0 || id >= vocab) {
    if (threadIdx.x == 0) atomicCAS(err, 0, 1);
    for (int i = threadIdx.x * 4; i < d; i += kRowThreads * 4)
      *reinterpret_cast<float4*>(dst + i) = make_float4(0.f, 0.f, 0.f, 0.f);
    return;
  }
  const uint4* src = reinterpret_cast<const uint4*>(table + (int64_t)id * d);
  uint4 v[kRowVec];
#pragma unroll
  for (int k = 0; k < kRowVec; ++k) {
    const int i = threadIdx.x + k * kRowThreads;
    if (i < nv) v[k] = src[i];
  }
#pragma unroll
  for (int k = 0; k < kRowVec; ++k) {
    const int i = threadIdx.x + k * kRowThreads;
    if (i < nv) {
      const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v[k]);
      const float2 f0 = __bfloat1622float2(h[0]), f1 = __bfloat1622float2(h[1]);
      const float2 f2 = __bfloat1622float2(h[2]), f3 = __bfloat1622float2(h[3]);
      *reinterpret_cast<float4*>(dst + i * 8) = make_float4(f0.x, f0.y, f1.x, f1.y);
      *reinterpret_cast<float4*>(dst + i * 8 + 4) = make_float4(f2.x, f2.y, f3.x, f3.y);
    }
  }
}

cudaError_t launch_embed(const int32_t* ids, int T, const bf16* table, int vocab, int d, float* out, int* err,
                         cudaStream_t s) {
  if (T <= 0) return cudaSuccess;
  if (d % 8 || d > kRowThreads * kRowVec * 8) return cudaErrorInvalidValue;  // d <= 16384
  return launch_pdl(embed_kernel, dim3(T), dim3(kRowThreads), 0, s, ids, T, table, vocab, d, out, err);
}

// ------------------------------------------------------------------ RMSNorm
// y[r, :] = bf16(x[src, :] * rsqrt(mean(x[src, :]^2) + eps) * gain), src = row_idx ? row_idx[r] : r.
// One block per row: every thread loads its float4s at once, the block reduces the sum of squares.
__global__ void __launch_bounds__(kRowThreads) rmsnorm_kernel(const float* x, int64_t ldx, const int32_t* row_idx,
                                                              int rows, int d, const float* gain, float eps, bf16* y,
                                                              int64_t ldy) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[kRowThreads / 32];
  const int r = blockIdx.x;
  const int src = row_idx ? row_idx[r] : r;
  const float4* xr = reinterpret_cast<const float4*>(x + (int64_t)src * ldx);
  const int nv = d / 4;
  float4 v[kRowVec];
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < kRowVec; ++k) {
    const int i = threadIdx.x + k * kRowThreads;
    v[k] = i < nv ? xr[i] : make_float4(0.f, 0.f, 0.f, 0.f);
  }
#pragma unroll
  for (int k = 0; k < kRowVec; ++k) ss += v[k].x * v[k].x + v[k].y * v[k].y + v[k].z * v[k].z + v[k].w * v[k].w;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int w = 0; w < kRowThreads / 32; ++w) tot += red[w];
  const float inv = rsqrtf(tot / (float)d + eps);
  uint2* yr = reinterpret_cast<uint2*>(y + (int64_t)r * ldy);
  const float4* g4 = reinterpret_cast<const float4*>(gain);
#pragma unroll
  for (int k = 0; k < kRowVec; ++k) {
    const int i = threadIdx.x + k * kRowThreads;
    if (i < nv) {
      const float4 g = g4[i];
      uint2 o;
      o.x = pack_bf16(v[k].x * inv * g.x, v[k].y * inv * g.y);
      o.y = pack_bf16(v[k].z * inv * g.z, v[k].w * inv * g.w);
      yr[i] = o;
    }
  }
}

// Many rows (prefill): one warp per row, each lane's loads issued eight at a time.
__global__ void __launch_bounds__(256) rmsnorm_warp_kernel(const float* x, int64_t ldx, const int32_t* row_idx,
                                                           int rows, int d, const float* gain, float eps, bf16* y,
                                                           int64_t ldy) {
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  const int src = row_idx ? row_idx[r] : r;
  const float4* xr = reinterpret_cast<const float4*>(x + (int64_t)src * ldx);
  const int nv = d / 4;
  float ss = 0.f;
  for (int base = lane; base < nv; base += 8 * 32) {
    float4 v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = base + k * 32 < nv ? xr[base + k * 32] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int k = 0; k < 8; ++k) ss += v[k].x * v[k].x + v[k].y * v[k].y + v[k].z * v[k].z + v[k].w * v[k].w;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  const float inv = rsqrtf(ss / (float)d + eps);
  uint2* yr = reinterpret_cast<uint2*>(y + (int64_t)r * ldy);
  const float4* g4 = reinterpret_cast<const float4*>(gain);
  for (int base = lane; base < nv; base += 8 * 32) {
    float4 v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = base + k * 32 < nv ? xr[base + k * 32] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int i = base + k * 32;
      if (i < nv) {
        const float4 g = g4[i];
        uint2 o;
        o.x = pack_bf16(v[k].x * inv * g.x, v[k].y * inv * g.y);
        o.y = pack_bf16(v[k].z * inv * g.z, v[k].w * inv * g.w);
        yr[i] = o;
      }
    }
  }
}

// Folded RMSNorm (prefill): y[r, :] = bf16(x[r, :] * gain) and ss[r] = sum(x[r, :]^2); the GEMM that
// reads y applies rsqrt(ss / d + eps) to its output rows.  One warp per row.
__global__ void __launch_bounds__(256) norm_stats_kernel(const float* x, int rows, int d, const float* gain, bf16* y,
                                                         float* ss_out) {
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  const float4* xr = reinterpret_cast<const float4*>(x + (int64_t)r * d);
  const float4* g4 = reinterpret_cast<const float4*>(gain);
  uint2* yr = reinterpret_cast<uint2*>(y + (int64_t)r * d);
  const int nv = d / 4;
  float ss = 0.f;
  for (int base = lane; base < nv; base += 8 * 32) {
    float4 v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = base + k * 32 < nv ? xr[base + k * 32] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int i = base + k * 32;
      ss += v[k].x * v[k].x + v[k].y * v[k].y + v[k].z * v[k].z + v[k].w * v[k].w;
      if (i < nv) {
        const float4 g = g4[i];
        uint2 o;
        o.x = pack_bf16(v[k].x * g.x, v[k].y * g.y);
        o.y = pack_bf16(v[k].z * g.z, v[k].w * g.w);
        yr[i] = o;
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if (lane == 0) ss_out[r] = ss;
}
cudaError_t launch_norm_stats(const float* x, int rows, int d, const float* gain, bf16* y, float* ss, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (d % 4) return cudaErrorInvalidValue;
  return launch_pdl(norm_stats_kernel, dim3((rows + 7) / 8), dim3(256), 0, s, x, rows, d, gain, y, ss);
}

cudaError_t launch_rmsnorm(const float* x, int64_t ldx, const int32_t* row_idx, int rows, int d, const float* gain,
                           float eps, bf16* y, int64_t ldy, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (d % 4) return cudaErrorInvalidValue;
  if (rows >= 2048 || d > kRowThreads * kRowVec * 4)
    return launch_pdl(rmsnorm_warp_kernel, dim3((rows + 7) / 8), dim3(256), 0, s, x, ldx, row_idx, rows, d, gain, eps,
                      y, ldy);
  return launch_pdl(rmsnorm_kernel, dim3(rows), dim3(kRowThreads), 0, s, x, ldx, row_idx, rows, d, gain, eps, y,
                    ldy);
}

__global__ void last_rows_kernel(const int32_t* offsets, int B, int32_t* row_idx, int repeats) {
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < B * repeats) row_idx[i] = offsets[i / repeats + 1] - 1;
}
cudaError_t launch_last_rows(const int32_t* offsets, int B, int32_t* row_idx, cudaStream_t s, int repeats) {
  if (B <= 0 || repeats <= 0) return cudaSuccess;
  return launch_pdl(last_rows_kernel, dim3((B * repeats + 255) / 256), dim3(256), 0, s, offsets, B, row_idx,
                    repeats);
}

// ------------------------------------------------------------------ RoPE + KV write
// Prefill of models whose head_dim is not 128 (with 128 the QKV GEMM's epilogue does this, and
// decode attention does it for the decode step).
// One block per token.  q and k heads are rotated pairwise (i, i + hd/2) by
// angle pos * theta^(-2i/hd) (cos/sin from the table), rounded to bf16 and
// written to the rotated-query buffer or the key cache ([page][kv head][64
// tokens][hd]); v heads are copied to the value cache, which holds each page
// transposed ([page][kv head][hd][64 tokens]).
__global__ void rope_kv_kernel(const RopeKvArgs a) {
  pdl_trigger();
  pdl_wait();
  const int t = blockIdx.x;
  int lo = 0, hi = a.B - 1;  // item with offsets[item] <= t < offsets[item+1]
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (a.offsets[mid] <= t) lo = mid; else hi = mid - 1;
  }
  const int slot = a.slots[lo];
  const int pos = t - a.offsets[lo] + (a.past ? a.past[lo] : 0);
  const int half = a.hd / 2;
  const int heads = a.n_q + 2 * a.n_kv;
  const int page = a.block_table[(int64_t)slot * a.max_pages + (pos >> 6)];
  const int in_page = pos & 63;
  float* src = a.qkv + (int64_t)t * a.ldqkv;
  const float2* cs = a.rope_cs + (int64_t)pos * half;
  const int n = heads * half;
  // all of this thread's element pairs are loaded before any is used
  constexpr int kU = 4;
  for (int base = threadIdx.x; base < n; base += kU * blockDim.x) {
    float x0[kU], x1[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int idx = base + u * blockDim.x;
      if (idx < n) {
        const int c0 = (idx / half) * a.hd + idx % half;
        x0[u] = src[c0];
        x1[u] = src[c0 + half];
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int idx = base + u * blockDim.x;
      if (idx >= n) continue;
      const int h = idx / half, i = idx % half;
      if (h < a.n_q + a.n_kv) {
        const float2 r = cs[i];
        const bf16 y0 = __float2bfloat16(x0[u] * r.x - x1[u] * r.y);
        const bf16 y1 = __float2bfloat16(x1[u] * r.x + x0[u] * r.y);
        if (h < a.n_q) {
          bf16* dst = a.q_out + (int64_t)t * a.ldq + h * a.hd;
          dst[i] = y0;
          dst[i + half] = y1;
        } else {
          const int g = h - a.n_q;
          bf16* dst = a.k_cache + (a.layer_row0 + ((int64_t)page * a.n_kv + g) * 64 + in_page) * a.hd;
          dst[i] = y0;
          dst[i + half] = y1;
        }
      } else {
        // values are stored transposed per page: [page][kv head][hd][64 keys]
        const int g = h - a.n_q - a.n_kv;
        bf16* dst = a.v_cache + a.layer_row0 * a.hd + (((int64_t)page * a.n_kv + g) * a.hd + i) * 64 + in_page;
        dst[0] = __float2bfloat16(x0[u]);
        dst[(int64_t)half * 64] = __float2bfloat16(x1[u]);
      }
    }
  }
}

__global__ void token_map_kernel(const int32_t* offsets, const int32_t* slots, const int32_t* past, int B, int T,
                                 int2* map) {
  pdl_trigger();
  pdl_wait();
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  int lo = 0, hi = B - 1;  // item with offsets[item] <= t < offsets[item+1]
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (offsets[mid] <= t) lo = mid; else hi = mid - 1;
  }
  map[t] = make_int2(slots[lo], t - offsets[lo] + (past ? past[lo] : 0));
}
cudaError_t launch_token_map(const int32_t* offsets, const int32_t* slots, const int32_t* past, int B, int T,
                             int2* map, cudaStream_t s) {
  if (T <= 0) return cudaSuccess;
  return launch_pdl(token_map_kernel, dim3((T + 255) / 256), dim3(256), 0, s, offsets, slots, past, B, T, map);
}

cudaError_t launch_rope_kv(const RopeKvArgs& a, cudaStream_t s) {
  if (a.T <= 0) return cudaSuccess;
  return launch_pdl(rope_kv_kernel, dim3(a.T), dim3(256), 0, s, a);
}

// (cos, sin) of pos * theta^(-2i/hd), evaluated in double precision.
__global__ void rope_table_kernel(double theta, int hd, int max_seq, float2* cs) {
  const int half = hd / 2;
  const int64_t n = (int64_t)max_seq * half;
  for (int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; k < n; k += (int64_t)gridDim.x * blockDim.x) {
    const int pos = (int)(k / half), i = (int)(k % half);
    const double inv_freq = pow(theta, -2.0 * i / (double)hd);
    double sn, cn;
    sincos((double)pos * inv_freq, &sn, &cn);
    cs[k] = make_float2((float)cn, (float)sn);
  }
}
cudaError_t launch_rope_table(float theta, int hd, int max_seq, float2* cs, cudaStream_t s) {
  rope_table_kernel<<<1024, 256, 0, s>>>((double)theta, hd, max_seq, cs);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ greedy arg max
// out[b] = arg max_v logits[b, v], lowest v on ties; optionally also
// out2[b*stride + col] with col = col_base (+ *step when step is given), if col < col_limit.
__global__ void argmax_kernel(const float* logits, int64_t ld, int V, int32_t* out, int32_t* out2,
                              int64_t out2_stride, const int32_t* step, int col_base, int col_limit) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const float* row = logits + (int64_t)b * ld;
  float best = -INFINITY;
  int best_i = 0x7fffffff;
  for (int i = threadIdx.x; i < V; i += blockDim.x) {
    const float v = row[i];
    if (v > best || (v == best && i < best_i)) {
      best = v;
      best_i = i;
    }
  }
  __shared__ float sv[32];
  __shared__ int si[32];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, best, o);
    const int oi = __shfl_xor_sync(0xffffffffu, best_i, o);
    if (ov > best || (ov == best && oi < best_i)) {
      best = ov;
      best_i = oi;
    }
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    sv[warp] = best;
    si[warp] = best_i;
  }
  __syncthreads();
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
    best = lane < nw ? sv[lane] : -INFINITY;
    best_i = lane < nw ? si[lane] : 0x7fffffff;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, best, o);
      const int oi = __shfl_xor_sync(0xffffffffu, best_i, o);
      if (ov > best || (ov == best && oi < best_i)) {
        best = ov;
        best_i = oi;
      }
    }
    if (lane == 0) {
      if (best_i == 0x7fffffff) best_i = 0;  // all NaN: fall back to id 0
      out[b] = best_i;
      if (out2) {
        const int col = col_base + (step ? *step : 0);
        if (col < col_limit) out2[(int64_t)b * out2_stride + col] = best_i;
      }
    }
  }
}
cudaError_t launch_argmax(const float* logits, int64_t ld, int B, int V, int32_t* out, int32_t* out2,
                          int64_t out2_stride, cudaStream_t s, const int32_t* step, int col_base, int col_limit) {
  if (B <= 0) return cudaSuccess;
  return launch_pdl(argmax_kernel, dim3(B), dim3(1024), 0, s, logits, ld, V, out, out2, out2_stride, step, col_base,
                    col_limit);
}

// ------------------------------------------------------------------ temperature sampling
// One block per row: the largest argmax_key of the Gumbel-perturbed scores (sampling.cuh).
__global__ void sample_kernel(const float* logits, int64_t ld, int V, SampleParams sp_val, const SampleParams* sp_dev,
                              const int32_t* step, int step_bias, int32_t* out, int32_t* out2, int64_t out2_stride,
                              int col_base, int col_limit) {
  pdl_trigger();
  pdl_wait();
  const SampleParams sp = sp_dev ? *sp_dev : sp_val;
  const int s = step ? *step : 0;
  const int t = s + step_bias;
  const int b = blockIdx.x;
  const float* row = logits + (int64_t)b * ld;
  unsigned long long best = 0ull;
  for (int v = threadIdx.x; v < V; v += blockDim.x) {
    const unsigned long long k = argmax_key(sample_score(row[v], sp, t, b, v), v);
    best = k > best ? k : best;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
    best = other > best ? other : best;
  }
  __shared__ unsigned long long sk[32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) sk[warp] = best;
  __syncthreads();
  if (warp == 0) {
    best = lane < (int)(blockDim.x >> 5) ? sk[lane] : 0ull;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
      best = other > best ? other : best;
    }
    if (lane == 0) {
      const int id = best ? (int)(0xFFFFFFFFu - (uint32_t)(best & 0xFFFFFFFFull)) : 0;
      out[b] = id;
      if (out2) {
        const int col = col_base + s;
        if (col < col_limit) out2[(int64_t)b * out2_stride + col] = id;
      }
    }
  }
}
cudaError_t launch_sample(const float* logits, int64_t ld, int B, int V, SampleParams sp, const SampleParams* sp_dev,
                          const int32_t* step, int step_bias, int32_t* out, int32_t* out2, int64_t out2_stride,
                          int col_base, int col_limit, cudaStream_t s) {
  if (B <= 0) return cudaSuccess;
  return launch_pdl(sample_kernel, dim3(B), dim3(1024), 0, s, logits, ld, V, sp, sp_dev, step, step_bias, out, out2,
                    out2_stride, col_base, col_limit);
}

// One thread per (item, k) of p and per item of conf: mean and population standard deviation
// over the item's R consecutive rows.
__global__ void repeat_stats_kernel(const float* p, const float* conf, int B, int R, int K, float* p_mean,
                                    float* p_std, float* conf_mean, float* conf_std) {
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B * (K + 1)) return;
  const bool is_p = i < B * K;
  const int b = is_p ? i / K : i - B * K;
  const int k = is_p ? i % K : 0;
  const float* x = is_p ? p + (int64_t)b * R * K + k : conf + (int64_t)b * R;
  const int stride = is_p ? K : 1;
  float sum = 0.f;
  for (int j = 0; j < R; ++j) sum += x[(int64_t)j * stride];
  const float mean = sum / (float)R;
  float ss = 0.f;
  for (int j = 0; j < R; ++j) {
    const float d = x[(int64_t)j * stride] - mean;
    ss += d * d;
  }
  const float sd = sqrtf(ss / (float)R);
  if (is_p) {
    if (p_mean) p_mean[i] = mean;
    if (p_std) p_std[i] = sd;
  } else {
    if (conf_mean) conf_mean[b] = mean;
    if (conf_std) conf_std[b] = sd;
  }
}
cudaError_t launch_repeat_stats(const float* p, const float* conf, int B, int R, int K, float* p_mean, float* p_std,
                                float* conf_mean, float* conf_std, cudaStream_t s) {
  if (B <= 0 || R <= 0) return cudaSuccess;
  const int n = B * (K + 1);
  return launch_pdl(repeat_stats_kernel, dim3((n + 255) / 256), dim3(256), 0, s, p, conf, B, R, K, p_mean, p_std,
                    conf_mean, conf_std);
}

// ------------------------------------------------------------------ forked sequences
// Block (job, layer): the job's source page of this layer is copied, K rows then the transposed V rows.
__global__ void fork_pages_kernel(bf16* k_cache, bf16* v_cache, const int4* jobs, int64_t page_elems,
                                  int64_t layer_elems, int32_t* seq_len) {
  pdl_trigger();
  pdl_wait();
  const int4 j = jobs[blockIdx.x];
  if (blockIdx.y == 0 && threadIdx.x == 0) seq_len[j.y] = seq_len[j.x];
  if (j.z < 0) return;
  const int64_t src = (int64_t)blockIdx.y * layer_elems + (int64_t)j.z * page_elems;
  const int64_t dst = (int64_t)blockIdx.y * layer_elems + (int64_t)j.w * page_elems;
  const int64_t n16 = page_elems * (int64_t)sizeof(bf16) / 16;
  const uint4* ks = reinterpret_cast<const uint4*>(k_cache + src);
  const uint4* vs = reinterpret_cast<const uint4*>(v_cache + src);
  uint4* kd = reinterpret_cast<uint4*>(k_cache + dst);
  uint4* vd = reinterpret_cast<uint4*>(v_cache + dst);
  for (int64_t i = threadIdx.x; i < n16; i += blockDim.x) {
    kd[i] = ks[i];
    vd[i] = vs[i];
  }
}
cudaError_t launch_fork_pages(bf16* k_cache, bf16* v_cache, const int4* jobs, int n_jobs, int layers,
                              int64_t page_elems, int64_t layer_elems, int32_t* seq_len, cudaStream_t s) {
  if (n_jobs <= 0) return cudaSuccess;
  return launch_pdl(fork_pages_kernel, dim3(n_jobs, layers), dim3(256), 0, s, k_cache, v_cache, jobs, page_elems,
                    layer_elems, seq_len);
}

// ------------------------------------------------------------------ verdict (Sec. 2.1)
// p = softmax(logits[b, ids]); conf = max p; arg = first arg max; defer = conf < tau.
struct VerdictIds {
  int32_t v[8];
};
__global__ void verdict_kernel(const float* logits, int64_t ld, int B, VerdictIds ids, int K, float tau, float* p,
                               float* conf, int32_t* arg, uint8_t* defer) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const float* row = logits + (int64_t)b * ld;
  float z[8];
  float mx = -INFINITY;
  for (int k = 0; k < K; ++k) {
    z[k] = row[ids.v[k]];
    mx = fmaxf(mx, z[k]);
  }
  float sum = 0.f;
  for (int k = 0; k < K; ++k) {
    z[k] = expf(z[k] - mx);
    sum += z[k];
  }
  float best = -1.f;
  int best_k = 0;
  for (int k = 0; k < K; ++k) {
    const float pk = z[k] / sum;
    p[(int64_t)b * K + k] = pk;
    if (pk > best) {
      best = pk;
      best_k = k;
    }
  }
  conf[b] = best;
  arg[b] = best_k;
  defer[b] = best < tau ? 1 : 0;
}
cudaError_t launch_verdict(const float* logits, int64_t ld, int B, const int32_t* ids, int K, float tau, float* p,
                           float* conf, int32_t* arg, uint8_t* defer, cudaStream_t s) {
  if (B <= 0) return cudaSuccess;
  VerdictIds v;
  for (int k = 0; k < 8; ++k) v.v[k] = k < K ? ids[k] : 0;
  return launch_pdl(verdict_kernel, dim3((B + 127) / 128), dim3(128), 0, s, logits, ld, B, v, K, tau, p, conf, arg,
                    defer);
}

// ------------------------------------------------------------------ bookkeeping
__global__ void set_seq_len_kernel(const int32_t* offsets, const int32_t* slots, int B, int32_t* seq_len,
                                   const int32_t* past) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < B) seq_len[slots[b]] = offsets[b + 1] - offsets[b] + (past ? past[b] : 0);
}
cudaError_t launch_set_seq_len(const int32_t* offsets, const int32_t* slots, int B, int32_t* seq_len,
                               cudaStream_t s, const int32_t* past) {
  if (B <= 0) return cudaSuccess;
  return launch_pdl(set_seq_len_kernel, dim3((B + 255) / 256), dim3(256), 0, s, offsets, slots, B, seq_len, past);
}

// seq_len[handles[b]] += 1 for every b; *step += 1 when step is given (decode-step counter).
__global__ void advance_kernel(const int32_t* handles, int B, int32_t* seq_len, int32_t* step) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < B) seq_len[handles[b]] += 1;
  if (step && b == 0) *step += 1;
}
cudaError_t launch_advance(const int32_t* handles, int B, int32_t* seq_len, cudaStream_t s, int32_t* step) {
  if (B <= 0) return cudaSuccess;
  return launch_pdl(advance_kernel, dim3((B + 255) / 256), dim3(256), 0, s, handles, B, seq_len, step);
}

__global__ void finish_step_kernel(unsigned long long* keys, int B, int32_t* next, int32_t* tok, int64_t tok_stride,
                                   int32_t* step, int col_base, int col_limit, const int32_t* handles,
                                   int32_t* seq_len) {
  pdl_trigger();
  pdl_wait();
  const int s = step ? *step : 0;
  __syncthreads();
  for (int b = threadIdx.x; b < B; b += blockDim.x) {
    const unsigned long long k = keys[b];
    keys[b] = 0ull;
    const int id = k ? (int)(0xFFFFFFFFu - (uint32_t)(k & 0xFFFFFFFFull)) : 0;
    next[b] = id;
    if (tok) {
      const int col = col_base + s;
      if (col < col_limit) tok[(int64_t)b * tok_stride + col] = id;
    }
    if (seq_len) seq_len[handles[b]] += 1;
  }
  __syncthreads();
  if (seq_len && step && threadIdx.x == 0) *step = s + 1;
}
cudaError_t launch_finish_step(unsigned long long* keys, int B, int32_t* next, int32_t* tok, int64_t tok_stride,
                               int32_t* step, int col_base, int col_limit, const int32_t* handles,
                               int32_t* seq_len, cudaStream_t s) {
  if (B <= 0) return cudaSuccess;
  return launch_pdl(finish_step_kernel, dim3(1), dim3(1024), 0, s, keys, B, next, tok, tok_stride, step, col_base,
                    col_limit, handles, seq_len);
}

// prompt_b = inc_ids[inc_off[b]:inc_off[b+1]] ++ cand_ids[cand_off[b]:cand_off[b+1]], packed at prompt_off[b].
__global__ void build_prompts_kernel(const int32_t* inc_ids, const int32_t* inc_off, const int32_t* cand_ids,
                                     const int32_t* cand_off, const int32_t* prompt_off, int B, int T,
                                     int32_t* out, int shared_inc) {
  pdl_trigger();
  pdl_wait();
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < T; t += gridDim.x * blockDim.x) {
    int lo = 0, hi = B - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (prompt_off[mid] <= t) lo = mid; else hi = mid - 1;
    }
    const int j = t - prompt_off[lo];
    const int n_inc = shared_inc >= 0 ? shared_inc : inc_off[lo + 1] - inc_off[lo];
    const int inc0 = shared_inc >= 0 ? 0 : inc_off[lo];
    out[t] = j < n_inc ? inc_ids[inc0 + j] : cand_ids[cand_off[lo] + (j - n_inc)];
  }
}
cudaError_t launch_build_prompts(const int32_t* inc_ids, const int32_t* inc_off, const int32_t* cand_ids,
                                 const int32_t* cand_off, const int32_t* prompt_off, int B, int T, int32_t* out,
                                 cudaStream_t s, int shared_inc) {
  if (T <= 0) return cudaSuccess;
  int blocks = (T + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  return launch_pdl(build_prompts_kernel, dim3(blocks), dim3(256), 0, s, inc_ids, inc_off, cand_ids, cand_off,
                    prompt_off, B, T, out, shared_inc);
}

// ------------------------------------------------------------------ weight packing
// dst rows [32c, 32c+16) = gate rows [16c, 16c+16), dst rows [32c+16, 32c+32) = up rows;
// rows past F are zero.  Fp = F rounded up to 64.
__global__ void pack_gate_up_kernel(const bf16* gate, const bf16* up, int F, int Fp, int d, bf16* dst) {
  const int64_t chunks_per_row = d / 8;
  const int64_t n = (int64_t)2 * Fp * chunks_per_row;
  for (int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; k < n; k += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = k / chunks_per_row, c = k % chunks_per_row;
    const int64_t blk = r / 32, in = r % 32;
    const bool is_up = in >= 16;
    const int64_t f = blk * 16 + (in & 15);
    uint4 v = make_uint4(0, 0, 0, 0);
    if (f < F) v = *reinterpret_cast<const uint4*>((is_up ? up : gate) + f * d + c * 8);
    *reinterpret_cast<uint4*>(dst + r * d + c * 8) = v;
  }
}
cudaError_t launch_pack_gate_up(const bf16* gate, const bf16* up, int F, int Fp, int d, bf16* dst, cudaStream_t s) {
  pack_gate_up_kernel<<<2048, 256, 0, s>>>(gate, up, F, Fp, d, dst);
  return cudaGetLastError();
}

// dst = src [N][K] (row pitch ld elements) in blocks of 256 rows x 64 columns: element (n, k) at
// ((n / 256) * (Kp / 64) + k / 64) * 16384 + (n % 256) * 64 + k % 64 for n < ceil(N / 256) * 256
// and k < Kp; rows >= N and columns >= K are zero.  One 16-byte chunk of dst per step, written in
// order; vec: src and ld allow 16-byte loads.
__global__ void block_rows_kernel(const bf16* src, int64_t N, int K, int64_t ld, int Kp, bool vec, bf16* dst) {
  const int64_t kbs = Kp / 64;
  const int64_t chunks = (N + 255) / 256 * 256 * (Kp / 8);
  for (int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; c < chunks; c += (int64_t)gridDim.x * blockDim.x) {
    const int64_t blk = c >> 11;  // 256 rows x 8 chunks per block
    const int in = (int)(c & 2047);
    const int64_t n = (blk / kbs) * 256 + (in >> 3);
    const int k = (int)(blk % kbs) * 64 + (in & 7) * 8;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (n < N) {
      const bf16* row = src + n * ld;
      if (vec && k + 8 <= K) {
        v = *reinterpret_cast<const uint4*>(row + k);
      } else {
        alignas(16) unsigned short t[8];
        for (int j = 0; j < 8; ++j) t[j] = k + j < K ? __bfloat16_as_ushort(row[k + j]) : (unsigned short)0;
        v = *reinterpret_cast<const uint4*>(t);
      }
    }
    reinterpret_cast<uint4*>(dst)[c] = v;
  }
}
cudaError_t launch_block_rows(const bf16* src, int64_t N, int K, int64_t ld, int Kp, bf16* dst, cudaStream_t s) {
  if (N < 1 || K < 1 || K > Kp || Kp % 64 || ld < K) return cudaErrorInvalidValue;
  const bool vec = (reinterpret_cast<uintptr_t>(src) & 15) == 0 && ld % 8 == 0;
  block_rows_kernel<<<2048, 256, 0, s>>>(src, N, K, ld, Kp, vec, dst);
  return cudaGetLastError();
}

__global__ void bf16_to_f32_kernel(const bf16* src, int64_t n, float* dst) {
  for (int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; k < n; k += (int64_t)gridDim.x * blockDim.x)
    dst[k] = __bfloat162float(src[k]);
}
cudaError_t launch_bf16_to_f32(const bf16* src, int64_t n, float* dst, cudaStream_t s) {
  bf16_to_f32_kernel<<<256, 256, 0, s>>>(src, n, dst);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ selection (Sec. 3.1, 3.6)
// One block of 1024 threads, B <= 1024 candidates with 8 bin probabilities each:
//   s_hat[i] = sum_b p[i,b] m[b]; order = indices by decreasing s_hat (lower index first on ties,
//   bitonic sort in shared memory); disc[i] = mass of the bins whose lower edge is >= x;
//   disc_pred[i] = disc[i] >= tau.
struct BinReps {
  float m[8];
};
__global__ void __launch_bounds__(1024) select_kernel(int B, const float* p, BinReps reps, float x, float tau,
                                                       float* s_hat, int32_t* order, float* disc,
                                                       uint8_t* disc_pred) {
  pdl_trigger();
  pdl_wait();
  __shared__ float key[1024];
  __shared__ int idx[1024];
  const float lower[8] = {0.f, 0.25f, 0.5f, 0.71f, 1.0f, 1.41f, 2.0f, 4.0f};
  const int i = threadIdx.x;
  float sv = -INFINITY;
  if (i < B) {
    float acc = 0.f, d = 0.f;
#pragma unroll
    for (int b = 0; b < 8; ++b) {
      const float pb = p[(int64_t)i * 8 + b];
      acc += pb * reps.m[b];
      if (lower[b] >= x) d += pb;
    }
    sv = acc;
    s_hat[i] = acc;
    disc[i] = d;
    disc_pred[i] = d >= tau ? 1 : 0;
  }
  key[i] = sv;
  idx[i] = i < B ? i : 0x7fffffff;
  __syncthreads();
  // bitonic sort, "first" = larger key, then smaller index
  for (int size = 2; size <= 1024; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const int j = i ^ stride;
      if (j > i) {
        const bool up = (i & size) == 0;
        const float ka = key[i], kb = key[j];
        const int ia = idx[i], ib = idx[j];
        const bool a_first = ka > kb || (ka == kb && ia < ib);
        if (a_first != up) {
          key[i] = kb;
          key[j] = ka;
          idx[i] = ib;
          idx[j] = ia;
        }
      }
      __syncthreads();
    }
  }
  if (i < B) order[i] = idx[i];
}
cudaError_t launch_select(int B, const float* p, const float* m_bins, float x, float tau, float* s_hat,
                          int32_t* order, float* disc, uint8_t* disc_pred, cudaStream_t s) {
  if (B <= 0) return cudaSuccess;
  BinReps r;
  for (int b = 0; b < 8; ++b) r.m[b] = m_bins[b];
  return launch_pdl(select_kernel, dim3(1), dim3(1024), 0, s, B, p, r, x, tau, s_hat, order, disc, disc_pred);
}

// ------------------------------------------------------------------ failure detection
// Waits on a barrier that nothing completes: the bounded wait gives up after
// limit_ns, records GF_ETIMEOUT in *err and the kernel returns normally.
__global__ void timeout_probe_kernel(uint64_t limit_ns, int* err) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait_for(&bar, 0, limit_ns, err);
}
cudaError_t launch_timeout_probe(uint64_t limit_ns, int* err, cudaStream_t s) {
  timeout_probe_kernel<<<1, 32, 0, s>>>(limit_ns, err);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ inspection
__global__ void read_kv_kernel(const bf16* k_cache, const bf16* v_cache, const int32_t* block_table, int max_pages,
                               int slot, int start, int n, int n_kv, int hd, int64_t layer_row0, bf16* k_dst,
                               bf16* v_dst) {
  const int64_t total = (int64_t)n * n_kv * hd;
  for (int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; k < total; k += (int64_t)gridDim.x * blockDim.x) {
    const int i = (int)(k % hd);
    const int g = (int)((k / hd) % n_kv);
    const int t = (int)(k / ((int64_t)hd * n_kv));
    const int pos = start + t;
    const int page = block_table[(int64_t)slot * max_pages + (pos >> 6)];
    k_dst[k] = k_cache[(layer_row0 + ((int64_t)page * n_kv + g) * 64 + (pos & 63)) * hd + i];
    v_dst[k] = v_cache[layer_row0 * hd + (((int64_t)page * n_kv + g) * hd + i) * 64 + (pos & 63)];
  }
}
cudaError_t launch_read_kv(const bf16* k_cache, const bf16* v_cache, const int32_t* block_table, int max_pages,
                           int slot, int start, int n, int n_kv, int hd, int64_t layer_row0, bf16* k_dst,
                           bf16* v_dst, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  read_kv_kernel<<<1024, 256, 0, s>>>(k_cache, v_cache, block_table, max_pages, slot, start, n, n_kv, hd, layer_row0,
                                      k_dst, v_dst);
  return cudaGetLastError();
}

}  // namespace gf
