// Kernel argument structs and launch wrappers shared by the runtime.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "sampling.cuh"

namespace gf {

using bf16 = __nv_bfloat16;
struct RopeEpilogue;  // gemm_tc.cuh

// RMSNorm folded into prefill GEMMs (see GemmArgs in gemm_tc.cuh): a residual-update GEMM writes
// out = bf16(x_new * gain) and adds sum(x_new^2) per row into ss_out; a consumer GEMM reading such an
// out scales its accumulator row by rsqrt(ss_in[row] * inv_d + eps).
struct NormFold {
  bf16* out;
  const float* gain;
  float* ss_out;
  int64_t ld_out;
  const float* ss_in;
  float inv_d, eps;
};

// Launch with programmatic stream serialization: the kernel may begin while the
// previous kernel of the stream finishes; it must call pdl_wait() (ptx.cuh)
// before using that kernel's results.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args&&... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// A set-up step that holds for one CUDA context, such as raising a kernel's shared-memory limit
// (an attribute of the function as loaded in the current device's context): run() calls `f` the
// first time it is reached in each context, and does nothing later in the same context.  Contexts
// are told apart per device (up to 64 devices; beyond that `f` runs every time) by
// current_context_id(), so a context made again after cudaDeviceReset runs `f` again.  Several host
// threads may call run() at once; `f` must then be safe to repeat.
// current_context_id (runtime.cu): the unique id (cuCtxGetId) of the calling thread's current CUDA
// context, 0 if it cannot be read; a context made after cudaDeviceReset gets a new id.
uint64_t current_context_id();
struct DeviceOnce {
  std::atomic<uint64_t> ctx[64] = {};
  template <typename F>
  cudaError_t run(F&& f) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t id = current_context_id();
    if (dev >= 0 && dev < 64 && id != 0 && ctx[dev].load(std::memory_order_acquire) == id) return cudaSuccess;
    e = f();
    if (e == cudaSuccess && dev >= 0 && dev < 64 && id != 0) ctx[dev].store(id, std::memory_order_release);
    return e;
  }
};

// ------------------------------------------------------------------ GEMM
// C[M,N] (op)= A[M,K] . B[N,K]^T ; mode is a GemmMode.  tmA/tmB are 2D
// tensor maps (bf16, 128-byte swizzle) with boxes {64, 128} and {64, bn}.
int gemm_num_stages(int bn);
int gemm_smem_bytes(int bn);
// group_m: M-blocks per raster group (0 = sized so a group's A tiles fill about 28 MiB of L2).
// swap: A holds the weights (M = output features, multiple of 32), B the activations
// (N = rows <= bn, bn 32/64/128), and out is written transposed (out[n][m]); modes
// kStoreF32, kAtomicF32 and kSwiGLU only.
// argmax_keys (swap + kStoreF32 only): atomicMax per output row of the packed (value, column)
// key of its largest element (see gemm_tc.cuh); the array must start at zero.
// sample (device pointer, with argmax_keys): the keys rank the Gumbel-perturbed scores of token
// t = *sample_step + sample_step_bias instead of the logits (temperature sampling, sampling.cuh).
// w_blocked: the weight operand (A when swap, else B) is in the blocked layout of
// launch_block_rows and its map has 64-element rows: {64, ceil(rows/256)*256 * K/64}, pitch 128 B.
cudaError_t launch_gemm(const CUtensorMap& tmA, const CUtensorMap& tmB, int M, int N, int K, void* out,
                        int64_t ldo, int mode, int bn, int splits, int grid, int* err, cudaStream_t s,
                        int group_m = 0, bool swap = false, unsigned long long* argmax_keys = nullptr,
                        const SampleParams* sample = nullptr, const int32_t* sample_step = nullptr,
                        int sample_step_bias = 0, const RopeEpilogue* rope = nullptr,
                        const NormFold* norm = nullptr, bool w_blocked = false);

// ------------------------------------------------------------------ attention
struct PrefillAttnArgs {
  const int2* items;          // (item, q_tile) work list, heaviest first
  const int32_t* offsets;     // [B+1] token offsets of the packed prompts
  const int32_t* slots;       // [B] sequence slot of each prompt
  const int32_t* past;        // [B] positions already cached before this prompt's tokens, or nullptr
  const int32_t* block_table; // [slots][max_pages]
  int max_pages;
  int n_q, n_kv;
  int64_t layer_row0;         // first K-cache row (64-token page rows of hd) of this layer
  int64_t layer_vrow0;        // first V-cache row (rows of 64 keys, V stored transposed per page)
  bf16* out;                  // [T, n_q*hd]
  int64_t ldo;
  float scale_log2;           // log2(e) / sqrt(hd)
  int* err;
};
cudaError_t launch_attn_prefill(int hd, const CUtensorMap& tmQ, const CUtensorMap& tmK, const CUtensorMap& tmV,
                                const PrefillAttnArgs& a, int n_items, cudaStream_t s);

struct DecodeAttnArgs {
  const bf16* q;              // [B, n_q*hd], rotated queries of this step
  int64_t ldq;
  const int32_t* handles;     // [B] slots, or nullptr: slot = b
  const int32_t* seq_len;     // [slots]; visible keys = min(seq_len[slot] + ctx_bias, max_ctx)
  int ctx_bias;
  int max_ctx;
  const int32_t* block_table;
  int max_pages;
  int n_q, n_kv;
  int64_t layer_row0;
  int64_t layer_vrow0;
  int chunk;                  // keys per split, multiple of 64 (at most 64 pages)
  int max_splits;
  float* part_o;              // [B][n_kv][max_splits][16][hd] unnormalised partial outputs
  float* part_ml;             // [B][n_kv][max_splits][16][2] (running max in log2 units, sum)
  bf16* out;                  // [B, n_q*hd]
  int64_t ldo;
  float scale_log2;
  int* err;
  // Fused decode step (qkv != nullptr; q is then unused): the queries and the new token's key and
  // value are read from the fp32 split-K sums of the QKV projection and rotated at position
  // seq_len[slot], the key and value written into the cache, and the merge kernel sets the rows of
  // qkv that were read back to zero for the next step's split-K sums.
  float* qkv;                 // [B, ldqkv]: n_q query heads | n_kv key heads | n_kv value heads
  int64_t ldqkv;
  const float2* rope_cs;      // [position][hd/2]
  bf16* k_cache;              // rows of hd: [layer][page][n_kv][64 tokens]
  bf16* v_cache;              // [layer][page][n_kv][hd][64 tokens]
};
cudaError_t launch_attn_decode(int hd, const CUtensorMap& tmK, const CUtensorMap& tmV, const DecodeAttnArgs& a,
                               int B, cudaStream_t s);

// ------------------------------------------------------------------ elementwise / small kernels
struct RopeKvArgs {
  float* qkv;                 // [T, (n_q+2n_kv)*hd] fp32 projections
  int64_t ldqkv;
  bf16* q_out;                // [T, n_q*hd]
  int64_t ldq;
  bf16* k_cache;
  bf16* v_cache;
  const float2* rope_cs;      // [max_seq][hd/2] (cos, sin)
  // the packed prompts: offsets/slots (and past: cached positions before each prompt, or nullptr)
  const int32_t* offsets;
  const int32_t* slots;
  const int32_t* past;
  int B;
  const int32_t* block_table;
  int max_pages;
  int T, n_q, n_kv, hd;
  int64_t layer_row0;
};
cudaError_t launch_rope_kv(const RopeKvArgs& a, cudaStream_t s);
// map[t] = (slot of the prompt holding packed token t, its position) for t < T.
cudaError_t launch_token_map(const int32_t* offsets, const int32_t* slots, const int32_t* past, int B, int T,
                             int2* map, cudaStream_t s);

cudaError_t launch_embed(const int32_t* ids, int T, const bf16* table, int vocab, int d, float* out, int* err,
                         cudaStream_t s);
cudaError_t launch_rmsnorm(const float* x, int64_t ldx, const int32_t* row_idx, int rows, int d, const float* gain,
                           float eps, bf16* y, int64_t ldy, cudaStream_t s);
// The folded form (many rows): y = bf16(x * gain) un-normalised and ss[r] = sum(x[r, :]^2).
cudaError_t launch_norm_stats(const float* x, int rows, int d, const float* gain, bf16* y, float* ss, cudaStream_t s);
// row_idx[b * repeats + j] = offsets[b + 1] - 1 for j < repeats (the last prompt row, once per repeat).
cudaError_t launch_last_rows(const int32_t* offsets, int B, int32_t* row_idx, cudaStream_t s, int repeats = 1);
cudaError_t launch_argmax(const float* logits, int64_t ld, int B, int V, int32_t* out, int32_t* out2,
                          int64_t out2_stride, cudaStream_t s, const int32_t* step = nullptr, int col_base = 0,
                          int col_limit = 1 << 30);
// Temperature sampling of B rows of logits (Gumbel-max, sampling.cuh): out[b] = the draw of token
// t = (*step if step) + step_bias for row b, with the parameters *sp_dev (or sp when sp_dev is null);
// optionally also out2[b*stride + col], col = col_base (+ *step), when col < col_limit.
cudaError_t launch_sample(const float* logits, int64_t ld, int B, int V, SampleParams sp, const SampleParams* sp_dev,
                          const int32_t* step, int step_bias, int32_t* out, int32_t* out2, int64_t out2_stride,
                          int col_base, int col_limit, cudaStream_t s);
// Mean and population standard deviation over the R repeats of each of B items:
// p [B*R][K] -> p_mean/p_std [B][K]; conf [B*R] -> conf_mean/conf_std [B] (any output may be null).
cudaError_t launch_repeat_stats(const float* p, const float* conf, int B, int R, int K, float* p_mean, float* p_std,
                                float* conf_mean, float* conf_std, cudaStream_t s);
// Forked sequences: for each job (src slot, dst slot, src page, dst page) copy the page's K and V
// rows of every layer when src page >= 0, and set seq_len[dst slot] = seq_len[src slot].
cudaError_t launch_fork_pages(bf16* k_cache, bf16* v_cache, const int4* jobs, int n_jobs, int layers,
                              int64_t page_elems, int64_t layer_elems, int32_t* seq_len, cudaStream_t s);
cudaError_t launch_verdict(const float* logits, int64_t ld, int B, const int32_t* ids, int K, float tau, float* p,
                           float* conf, int32_t* arg, uint8_t* defer, cudaStream_t s);
cudaError_t launch_set_seq_len(const int32_t* offsets, const int32_t* slots, int B, int32_t* seq_len,
                               cudaStream_t s, const int32_t* past = nullptr);
cudaError_t launch_advance(const int32_t* handles, int B, int32_t* seq_len, cudaStream_t s,
                           int32_t* step = nullptr);
// Greedy tokens from the argmax keys of the LM-head GEMM: next[b] (and tok[b*stride + col],
// col = col_base (+ *step), when col < col_limit); resets the keys; with seq_len, advances
// seq_len[handles[b]] and then *step.  B <= 1024.
cudaError_t launch_finish_step(unsigned long long* keys, int B, int32_t* next, int32_t* tok, int64_t tok_stride,
                               int32_t* step, int col_base, int col_limit, const int32_t* handles,
                               int32_t* seq_len, cudaStream_t s);
// shared_inc >= 0: every prompt starts with inc_ids[0 .. shared_inc) (inc_off unused).
cudaError_t launch_build_prompts(const int32_t* inc_ids, const int32_t* inc_off, const int32_t* cand_ids,
                                 const int32_t* cand_off, const int32_t* prompt_off, int B, int T, int32_t* out,
                                 cudaStream_t s, int shared_inc = -1);
cudaError_t launch_pack_gate_up(const bf16* gate, const bf16* up, int F, int Fp, int d, bf16* dst, cudaStream_t s);
// Weight layout of the GEMMs (w_blocked): dst = src [N][K] (row pitch ld elements) in blocks of
// 256 rows x 64 columns, [ceil(N/256)][Kp/64][256][64], zero beyond row N and column K
// (Kp a multiple of 64, K <= Kp).  dst holds ceil(N/256) * 256 * Kp elements.
cudaError_t launch_block_rows(const bf16* src, int64_t N, int K, int64_t ld, int Kp, bf16* dst, cudaStream_t s);
cudaError_t launch_bf16_to_f32(const bf16* src, int64_t n, float* dst, cudaStream_t s);
cudaError_t launch_rope_table(float theta, int hd, int max_seq, float2* cs, cudaStream_t s);
cudaError_t launch_read_kv(const bf16* k_cache, const bf16* v_cache, const int32_t* block_table, int max_pages,
                           int slot, int start, int n, int n_kv, int hd, int64_t layer_row0, bf16* k_dst,
                           bf16* v_dst, cudaStream_t s);

cudaError_t launch_timeout_probe(uint64_t limit_ns, int* err, cudaStream_t s);
cudaError_t launch_select(int B, const float* p, const float* m_bins, float x, float tau, float* s_hat,
                          int32_t* order, float* disc, uint8_t* disc_pred, cudaStream_t s);

// Defined in runtime.cu for entry points of other translation units.
// K cache: rows of hd, boxes {64, 64}; V cache (transposed pages): rows of 64 keys, boxes {64, hd}.
int encode_kv_map(CUtensorMap* m, const void* base, int hd, uint64_t rows);
int encode_vt_map(CUtensorMap* m, const void* base, int hd, uint64_t rows);
void set_error_short(const char* msg);

}  // namespace gf
