/*
 * gf.h - C ABI of the GB300 surrogate forecaster.
 *
 * The surrogate of Sec. 2.1 reads x_i = (r, k_i, h) (reference kernel,
 * candidate kernel, hardware) as one token sequence, generates a brief chain
 * of reasoning by greedy decoding, and emits a distribution p_i over verdict
 * tokens.  Its confidence is q_i = max_b p_{i,b}, its predicted verdict is
 * y_hat_i = argmax_b p_{i,b}, and a forecast is used only when q_i clears a
 * threshold tau; the remaining candidates are deferred to real GPU
 * measurement (Sec. 2.1, "Selective Use").
 *
 * The language model is a pre-norm decoder-only transformer with RMSNorm,
 * rotary position embedding (rotate-half, pairs (i, i+hd/2), positions from
 * 0), grouped-query attention, SwiGLU feed-forward blocks, a final RMSNorm and
 * an untied LM head; no biases.  Weights are bf16; the residual stream is
 * fp32; matmuls accumulate in fp32.
 *
 * Conventions for every call:
 *   - Return value: GF_OK (0) or one of the GF_E* codes below; on error the
 *     outputs are unspecified and gf_last_error() (thread-local) says why.
 *   - "device" pointers are CUDA global memory of the device the model was
 *     created on; "host" pointers are ordinary host memory.  The caller owns
 *     every buffer it passes; no call frees or keeps caller memory beyond
 *     the call except where stated (gf_create borrows nothing: it copies).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Device work is enqueued on it asynchronously unless the call
 *     says it synchronises.
 *   - Token ids must lie in [0, vocab); lengths must be >= 1.
 *   - Not thread-safe per model: one host thread drives a model at a time.
 */
#ifndef GF_H_
#define GF_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
  GF_OK = 0,
  GF_EINVAL = 1,     /* bad argument: shape, id >= vocab, K outside 1..8, tau outside [0,1], bad handle */
  GF_ECAPACITY = 2,  /* KV page pool, sequence slots or prefill token budget exhausted */
  GF_ENOMEM = 3,     /* a device or host allocation failed */
  GF_ECUDA = 4,      /* a CUDA runtime or driver call failed (message in gf_last_error) */
  GF_ENOTIMPL = 5,   /* configuration the kernels do not support (e.g. head_dim not 64/128) */
  GF_ETIMEOUT = 6    /* a device-side bounded wait gave up; the kernel returned early */
};

/* Model shape and resource limits. */
typedef struct gf_config {
  int32_t layers;
  int32_t d_model;     /* multiple of 64 */
  int32_t n_q;         /* query heads */
  int32_t n_kv;        /* key/value heads; n_q % n_kv == 0, n_q / n_kv <= 16 */
  int32_t head_dim;    /* 64 or 128 */
  int32_t ffn;         /* SwiGLU width (padded to a multiple of 64 inside, with zero weights) */
  int32_t vocab;       /* multiple of 32, >= 32 */
  float rope_theta;
  float rms_eps;
  int32_t max_batch;   /* sequence slots (concurrent sequences), <= 1024 */
  int32_t max_seq;     /* tokens per sequence, prompt + generated */
  int64_t max_prefill_tokens; /* largest total prompt tokens of one gf_prefill call */
  int64_t kv_pages;    /* 64-token pages in the KV pool; 0 = max_batch * ceil(max_seq / 64) */
} gf_config;

/* Canonical weights, bf16 row-major, rows = output features (as in y = x W^T).
 * All pointers are device pointers; the per-layer members are HOST arrays of
 * `layers` device pointers.  Shapes:
 *   embed [vocab, d]; lm_head [vocab, d]; final_norm [d];
 *   attn_norm[l], ffn_norm[l] [d];
 *   wq[l] [n_q*hd, d]; wk[l], wv[l] [n_kv*hd, d]; wo[l] [d, n_q*hd];
 *   w_gate[l], w_up[l] [ffn, d]; w_down[l] [d, ffn].
 * gf_create copies them into its own packed layout; the caller may free
 * them once gf_create returns and its stream has drained. */
typedef struct gf_weights {
  const void* embed;
  const void* lm_head;
  const void* final_norm;
  const void* const* attn_norm;
  const void* const* wq;
  const void* const* wk;
  const void* const* wv;
  const void* const* wo;
  const void* const* ffn_norm;
  const void* const* w_gate;
  const void* const* w_up;
  const void* const* w_down;
} gf_weights;

typedef struct gf_model gf_model;

/* Create a model on the current CUDA device: allocates the packed weight
 * arena, the paged KV pool (page size 64 tokens) and activation buffers for
 * `max_prefill_tokens`, then packs `w` on `stream` and synchronises it. */
int gf_create(const gf_config* cfg, const gf_weights* w, void* stream, gf_model** out);

/* Free everything the model owns.  Synchronises the device first. */
void gf_destroy(gf_model* m);

/* Prefill B prompts (Sec. 2.1: the prompt holds reference and candidate
 * kernel sources and the hardware table as tokens).
 *   ids          device int32[offsets[B]], prompts packed back to back
 *   offsets      host int32[B+1], offsets[0] = 0, strictly increasing
 *   seq_handles  host int32[B] (out): one slot per prompt, for decode/release
 *   last_logits  device float[B*vocab] or NULL: logits of each prompt's last
 *                position (those that pick the first generated token)
 *   next_ids     device int32[B] or NULL: greedy arg max of last_logits
 *                (lowest id on ties)
 * Fails with GF_ECAPACITY (nothing allocated) if slots, pages or
 * max_prefill_tokens are exceeded. */
int gf_prefill(gf_model* m, int32_t B, const int32_t* ids, const int32_t* offsets, int32_t* seq_handles,
               float* last_logits, int32_t* next_ids, void* stream);

/* One greedy decode step: feed ids[b] to sequence seq_handles[b] at its next
 * position, using and extending its paged KV cache.
 *   seq_handles  host int32[B], distinct live handles
 *   ids          device int32[B]
 *   logits       device float[B*vocab] or NULL
 *   next_ids     device int32[B] or NULL: arg max of the new logits
 * ids and next_ids may alias (in-place greedy loop).  GF_ECAPACITY if a
 * sequence would exceed max_seq or the pool has no free page. */
int gf_decode_step(gf_model* m, int32_t B, const int32_t* seq_handles, const int32_t* ids, float* logits,
                   int32_t* next_ids, void* stream);

/* Return the slots and KV pages of the given sequences to the pool.  Work
 * already enqueued that reads them must be ordered before any later call
 * that reuses them (all calls of one model on one stream are). */
int gf_release(gf_model* m, int32_t B, const int32_t* seq_handles);

/* The whole forecast of Sec. 2.1 for a batch of candidates:
 *   prompt_i = incumbent ids ‖ candidate ids  (x_i = (r, k_i, h));
 *   prefill, then n_decode greedy steps (the reasoning trace), then on the
 *   logits of the last step (the last prompt position if n_decode == 0):
 *     p[i,:] = softmax(logits[i, verdict_ids[0..K-1]])   (restricted softmax)
 *     conf[i] = max_b p[i,b]                              (q_i)
 *     verdict_arg[i] = argmax_b p[i,b], lowest b on ties  (y_hat_i)
 *     defer[i] = conf[i] < tau                            (measure on the GPU)
 *   Slots are released before returning.
 *   inc_ids, cand_ids          device int32, packed
 *   inc_offsets, cand_offsets  host int32[B+1]; each item's total length >= 1
 *   verdict_ids                host int32[K], 1 <= K <= 8, ids < vocab
 *   p [B*K], conf [B] float; verdict_arg [B] int32; defer [B] uint8: device
 *   tokens  device int32[B*n_decode] or NULL: the generated tokens, row-major
 *   final_logits device float[B*vocab] or NULL: the logits the verdict reads */
int gf_forecast_batch(gf_model* m, int32_t B, const int32_t* inc_ids, const int32_t* inc_offsets,
                      const int32_t* cand_ids, const int32_t* cand_offsets, int32_t n_decode,
                      const int32_t* verdict_ids, int32_t K, float tau, float* p, float* conf,
                      int32_t* verdict_arg, uint8_t* defer, int32_t* tokens, float* final_logits, void* stream);

/* gf_forecast_batch for a batch whose candidates all share one incumbent, as
 * the candidates of one search step share the reference kernel r of
 * x_i = (r, k_i, h) (Sec. 2.1): prompt_i = prefix ‖ candidate_i.  The
 * prefix's full 64-token pages are prefilled once and every candidate's block
 * table points at them (the pages are reference-counted); the remaining
 * prefix_len % 64 tokens are prefilled with each candidate.  Results are those
 * of gf_forecast_batch with inc_ids = the prefix for every item.
 *   prefix_ids   device int32[prefix_len], prefix_len >= 0
 *   cand_ids     device int32, packed; cand_offsets host int32[B+1]
 *   every prompt needs at least one token after the shared pages;
 *   other arguments as in gf_forecast_batch. */
int gf_forecast_batch_shared(gf_model* m, int32_t B, const int32_t* prefix_ids, int32_t prefix_len,
                             const int32_t* cand_ids, const int32_t* cand_offsets, int32_t n_decode,
                             const int32_t* verdict_ids, int32_t K, float tau, float* p, float* conf,
                             int32_t* verdict_arg, uint8_t* defer, int32_t* tokens, float* final_logits,
                             void* stream);

/* gf_forecast_batch with every array in host memory: copies the ids to the
 * device, runs the forecast, copies p/conf/verdict_arg/defer (and tokens if
 * non-NULL) back, and synchronises `stream` before returning. */
int gf_forecast_batch_host(gf_model* m, int32_t B, const int32_t* inc_ids, const int32_t* inc_offsets,
                           const int32_t* cand_ids, const int32_t* cand_offsets, int32_t n_decode,
                           const int32_t* verdict_ids, int32_t K, float tau, float* p, float* conf,
                           int32_t* verdict_arg, uint8_t* defer, int32_t* tokens, void* stream);

/* gf_forecast_batch with temperature sampling instead of greedy decoding, each
 * item sampled `repeats` times (Sec. 3.1 setup: three repeats per row at
 * temperature 1.0, reported as mean and population standard deviation).
 *   Row r = i * repeats + j is repeat j of item i.  Each item's prompt is
 *   prefilled once; its repeats share the prompt's full KV pages.
 *   Token t of row r (t = 0 from the prompt's logits, t = s + 1 from decode
 *   step s) is argmax_v (logits_v / temperature + G), G = -ln(-ln U) with U
 *   from Philox4x64-10 under key (seed, 0) at counter (v, t, r / 4, 0), word
 *   r mod 4, U = (floor(w / 2^41) + 1/2) 2^-23: an exact draw from
 *   softmax(logits / temperature), reproducible from (seed, t, r, v) alone.
 *   The verdict reads each row's final logits as in gf_forecast_batch.
 *   repeats >= 1, B * repeats <= max_batch; temperature > 0 and finite.
 *   p [B*repeats*K], conf, verdict_arg, defer [B*repeats]: per row, device.
 *   p_mean, p_std [B*K], conf_mean, conf_std [B]: device float or NULL, the
 *     mean and population standard deviation (divided by repeats) over the
 *     repeats of each item.
 *   tokens device int32[B*repeats*n_decode] or NULL; final_logits device
 *     float[B*repeats*vocab] or NULL; other arguments as in gf_forecast_batch. */
int gf_forecast_batch_sampled(gf_model* m, int32_t B, const int32_t* inc_ids, const int32_t* inc_offsets,
                              const int32_t* cand_ids, const int32_t* cand_offsets, int32_t n_decode,
                              int32_t repeats, float temperature, uint64_t seed, const int32_t* verdict_ids,
                              int32_t K, float tau, float* p, float* conf, int32_t* verdict_arg, uint8_t* defer,
                              float* p_mean, float* p_std, float* conf_mean, float* conf_std, int32_t* tokens,
                              float* final_logits, void* stream);

/* Stand-alone temperature draw (the rule of gf_forecast_batch_sampled) on caller logits:
 *   logits device float[B*ld], row b is sampled row r = b, token index t = token_index >= 0;
 *   out_ids device int32[B].  V <= ld; temperature > 0 and finite. */
int gf_sample_tokens(int32_t B, const float* logits, int64_t ld, int32_t V, uint64_t seed, int32_t token_index,
                     float temperature, int32_t* out_ids, void* stream);

/* Stand-alone verdict step (Sec. 2.1) on caller logits:
 *   logits device float[B*ld] (row stride ld >= max verdict id + 1);
 *   verdict_ids host int32[K]; outputs as in gf_forecast_batch. */
int gf_verdict(int32_t B, const float* logits, int64_t ld, const int32_t* verdict_ids, int32_t K, float tau,
               float* p, float* conf, int32_t* verdict_arg, uint8_t* defer, void* stream);

/* What a search does with an 8-bin forecast (K = 8 verdict ids, one per speedup
 * bin of Table tab:speedup-bins: S <= 0.25, (0.25,0.5], (0.5,0.71], (0.71,1],
 * (1,1.41], (1.41,2], (2,4], > 4):
 *   s_hat[i] = sum_b p[i,b] m_bins[b], the expected speedup that ranks
 *              candidates (Sec. 3.1); m_bins host float[8] are the bin
 *              representatives (m_2..m_7 = 0.35 0.59 0.84 1.19 1.68 2.83 in the
 *              paper; m_1, m_8 are empirical means it does not print);
 *   order[0..B) = candidate indices by decreasing s_hat, lower index first on
 *              ties (measure the first ceil(c% * B) under a budget c);
 *   disc[i]  = Pr[g >= x_cut], the discovery-moment score (Sec. 3.6): the mass
 *              of the bins whose lower edge is >= x_cut;
 *   disc_pred[i] = disc[i] >= tau_disc.
 * p, s_hat, disc device float; order device int32; disc_pred device uint8.
 * 1 <= B <= 1024.  Enqueued on `stream`. */
int gf_select(int32_t B, const float* p, const float* m_bins, float x_cut, float tau_disc, float* s_hat,
              int32_t* order, float* disc, uint8_t* disc_pred, void* stream);

/* ---- evaluation of 8-bin forecasts (host arithmetic only; no device work, no GPU needed) ----
 * gf_speedup_bin: the bin 1..8 of a measured speedup S (Table tab:speedup-bins, upper edges
 * inclusive: S <= 0.25, (0.25,0.5], (0.5,0.71], (0.71,1], (1,1.41], (1.41,2], (2,4], > 4).
 * gf_score_forecasts: the scores of n forecasts p [n*8] (host, row i = bins 1..8 of candidate i)
 * against the measured speedups S [n] (host, > 0), with bin representatives m_bins [8]:
 *   scores[0] = speedup recovered (Sec. 3.1): 100/|C| sum_{c in C} max_{i in Top_c} S_i / max_i S_i,
 *               C = {1, 5, 10, 25, 50} %, Top_c = the first ceil(c n / 100) (at least one) candidates
 *               by decreasing sum_b p_ib m_b, lower index first on ties;
 *   scores[1] = expected calibration error (Sec. 3.1): ten equal-width buckets of q_i = max_b p_ib,
 *               (0, 0.1] ... (0.9, 1] (0 in the first), accuracy = predicted bin (arg max, lowest bin
 *               on ties) equal to the measured bin;
 *   scores[2] = forecast error (Sec. 3.1): mean |m_{predicted bin} - S_i|;
 *   scores[3] = mean Brier score (Sec. 2.2): 1/2 sum_b (p_ib - 1[b = y_i])^2, y_i the measured bin;
 *   scores[4] = mean CRPS (Sec. 2.2): 1/7 sum_{k=1..7} (F_ik - 1[y_i <= k])^2, F the cumulative p.
 * scores: host double[5].  GF_EINVAL for n < 1, a null pointer, a negative or non-finite p or a
 * non-positive speedup. */
int gf_speedup_bin(double S);
int gf_score_forecasts(int32_t n, const double* p, const double* S, const double* m_bins, double* scores);

/* ---- building blocks --------------------------------------------------------
 * The dense contraction every projection of the forward pass uses, exposed on
 * its own: out[M,N] (op)= A[M,K] . W[N,K]^T on the tcgen05 tensor cores.
 *   A, W   device bf16, row-major (K contiguous); K % 64 == 0, N % 32 == 0
 *   mode   GF_GEMM_STORE_F32:  out (float, row stride ldo) = acc
 *          GF_GEMM_ADD_F32:    out += acc (non-atomic, as on the residual stream)
 *          GF_GEMM_ATOMIC_F32: out += acc with atomics (split-K partial sums)
 *          GF_GEMM_STORE_BF16: out (bf16) = acc
 *          GF_GEMM_SWIGLU:     W rows hold blocks of 16 gate rows followed by the
 *                              16 matching up rows; out (bf16, N/2 columns) = silu(gate) * up
 *   bn     tile width 64, 128 or 256, or 0 to choose; splits: split-K factor
 *          (only with GF_GEMM_ATOMIC_F32), 0 to choose; group_m: 128-row blocks
 *          per raster group (concurrent tiles share A and W tiles in L2), 0 to choose.
 * Enqueued on `stream`; a device-side timeout is reported by gf_gemm_status. */
enum { GF_GEMM_STORE_F32 = 0, GF_GEMM_ADD_F32 = 1, GF_GEMM_ATOMIC_F32 = 2, GF_GEMM_STORE_BF16 = 3,
       GF_GEMM_SWIGLU = 4 };
int gf_gemm_bf16(const void* A, const void* W, int32_t M, int32_t N, int32_t K, void* out, int64_t ldo,
                 int32_t mode, int32_t bn, int32_t splits, int32_t group_m, void* stream);
/* Synchronise `stream`; GF_ETIMEOUT if a gf_gemm_bf16, gf_decode_attention or
 * gf_selftest_timeout launch on the current device gave up waiting since the
 * last call (the word it reads is then cleared).  The building blocks keep one
 * such word per device (and CUDA context), made by their first call there. */
int gf_gemm_status(void* stream);

/* ---- planning queries (host arithmetic only: no device work, no GPU needed) --
 * gf_plan_gemm: the tiling the model's GEMMs, and gf_gemm_bf16 with
 * bn = splits = 0, use for an M x N x K product in `mode` (GF_GEMM_*) on a GPU
 * with `sms` SMs.
 *   *swap    1: the weights are the 128-row MMA operand and the M activation
 *            rows the narrow one (decode; M <= 128).  0: M rows in 128-row tiles.
 *   *bn      tile width: activation rows per tile when swapped (32, 64 or 128),
 *            else output columns per tile (64, 128 or 256).
 *   *splits  split-K factor (> 1 only in GF_GEMM_ATOMIC_F32 mode).
 * Returns GF_OK, or GF_EINVAL for sms, M, N or K < 1, a bad mode or a null
 * output pointer.  (Inside the model a GEMM whose epilogue applies a folded
 * RMSNorm is never swapped.) */
int gf_plan_gemm(int32_t sms, int32_t M, int32_t N, int32_t K, int32_t mode, int32_t* bn, int32_t* splits,
                 int32_t* swap);
/* gf_plan_decode_chunk: keys per decode-attention CTA (1024, 512 or 256) for
 * B sequences of up to max_ctx cached tokens and n_kv KV heads: the longest
 * chunk that still gives every SM two CTAs.  Returns the chunk, or GF_EINVAL
 * for a size < 1. */
int32_t gf_plan_decode_chunk(int32_t B, int32_t n_kv, int32_t max_ctx, int32_t sms);

/* Decode attention over a paged KV cache, the step a decode token spends on
 * its context (one query token per sequence, grouped-query heads):
 *   out[b, h, :] = sum_j softmax_j(q[b,h,:] . k_j / sqrt(hd)) v_j  over the
 *   ctx_len[b] cached positions j of sequence b, kv head h / (n_q / n_kv).
 *   q            device bf16 [B, n_q*hd], already rotated
 *   k_cache      device bf16 [num_pages][n_kv][64][hd] (64-token pages)
 *   v_cache      device bf16 [num_pages][n_kv][hd][64]: each page stored
 *                transposed (head dim major, 64 tokens contiguous)
 *   block_table  device int32 [B][max_pages]: page of block j of sequence b
 *   ctx_len      device int32 [B], 1 <= ctx_len[b] <= max_ctx (a larger
 *                value is clamped to max_ctx; 0 gives a zero output row)
 *   max_ctx      host bound on ctx_len, <= 64*max_pages (sizes the grid)
 *   out          device bf16 [B, n_q*hd]
 *   workspace    device scratch for the per-chunk partial results, at least
 *                gf_decode_attention_workspace(B, n_kv, head_dim, max_ctx) bytes,
 *                owned by the caller and free for reuse once the call's work
 *                on `stream` has completed.
 * head_dim 64 or 128, n_q / n_kv <= 16.  Enqueued on `stream`. */
size_t gf_decode_attention_workspace(int32_t B, int32_t n_kv, int32_t head_dim, int32_t max_ctx);
int gf_decode_attention(const void* q, const void* k_cache, const void* v_cache, int64_t num_pages,
                        const int32_t* block_table, int32_t max_pages, const int32_t* ctx_len, int32_t max_ctx,
                        int32_t B, int32_t n_q, int32_t n_kv, int32_t head_dim, void* out, void* workspace,
                        size_t workspace_bytes, void* stream);

/* gf_decode_attention without any allocation.  The paper has no counterpart:
 * this entry point exists for callers that cannot allocate device memory
 * where they call it - for example a serving loop whose device memory is
 * already fully reserved by another allocator (a raw cudaMalloc there can
 * fail), or code that must not call cudaMalloc/cudaFree after start-up
 * because those calls can synchronise the whole device and stall other
 * streams.  Arguments and results are those of gf_decode_attention; there is
 * no workspace argument.  Instead the per-chunk partial results live in a
 * fixed 16 MiB device array of the library (every GPU that loads the library
 * holds it until the process exits):
 *   - gf_decode_attention_workspace(B, n_kv, head_dim, max_ctx) must not
 *     exceed 16 MiB (16777216 bytes), else GF_ECAPACITY ("exceeds scratch")
 *     and nothing is enqueued;
 *   - the first call on a device, with that device current, looks up the
 *     array's device address (cudaGetSymbolAddress) for the current CUDA
 *     context; make that first call before any stream capture.  A context
 *     made later on the device (after cudaDeviceReset) gets the address
 *     looked up again by its first call;
 *   - every call on a device shares the one array and it keeps the last
 *     call's contents, so calls whose work overlaps on the GPU (other streams,
 *     or other host threads) race and corrupt each other's results: order
 *     them;
 *   - a bounded wait that gives up (after 2 s) records a timeout in a word
 *     of the same fixed storage and the call's output is then unspecified.
 *     The word stays set, and later calls may give up early, until
 *     gf_decode_attention_static_status reads and clears it: call that after
 *     the work whose results you use.
 * It calls no cudaMalloc, cudaFree or other allocating routine. */
int gf_decode_attention_static(const void* q, const void* k_cache, const void* v_cache, int64_t num_pages,
                               const int32_t* block_table, int32_t max_pages, const int32_t* ctx_len,
                               int32_t max_ctx, int32_t B, int32_t n_q, int32_t n_kv, int32_t head_dim, void* out,
                               void* stream);
/* Failure report of gf_decode_attention_static on the current device:
 * synchronises `stream`, then returns GF_ETIMEOUT (and clears the word) if a
 * wait of any earlier call gave up, else GF_OK.  Allocates nothing. */
int gf_decode_attention_static_status(void* stream);

/* Failure detection self-test: launch a kernel whose bounded wait on a barrier
 * that nothing completes runs out after `limit_ms` (1..2000).  The kernel
 * records the timeout and returns; this call synchronises `stream` and
 * returns GF_ETIMEOUT when the device reported it (GF_OK would mean the wait
 * did not run out).  The CUDA context stays usable. */
int gf_selftest_timeout(uint32_t limit_ms, void* stream);
/* The same self-test recording into the timeout word of
 * gf_decode_attention_static: returns what gf_decode_attention_static_status
 * then reports (GF_ETIMEOUT, with the word cleared again). */
int gf_selftest_timeout_static(uint32_t limit_ms, void* stream);

/* ---- measurement ------------------------------------------------------------
 * Kernel classes whose launches can be bracketed by CUDA events (on the
 * launching stream) for live timing inside a run. */
enum { GF_PROF_PREFILL_GEMM = 0, GF_PROF_DECODE_GEMM = 1, GF_PROF_PREFILL_ATTN = 2, GF_PROF_DECODE_ATTN = 3,
       GF_PROF_DECODE_STEPS = 4, /* the replayed decode steps of gf_forecast_batch, as one interval */
       GF_PROF_KINDS = 5 };
/* Time every launch of the classes whose bit is set in `mask` (0 = off). */
int gf_profile_enable(gf_model* m, uint32_t mask);
/* Synchronise the device and return, for class `kind` since the last read:
 * launches, summed kernel milliseconds, algorithmic FLOPs (2*M*N*K for a
 * GEMM, 4*hd per visible query-key pair for attention) and algorithmic HBM
 * bytes (operands read once, outputs written once; for GF_PROF_DECODE_STEPS
 * every weight once per step plus the cached keys and values each step reads
 * and writes); then reset the class. */
int gf_profile_read(gf_model* m, int32_t kind, int64_t* launches, double* ms, double* flops, double* bytes);

/* ---- inspection hooks (parity tests at full size) -------------------------
 * gf_debug_capture arms a copy, during the NEXT gf_prefill or gf_decode_step,
 * of the fp32 residual stream entering layer `layer` (layer == layers: the
 * final hidden state before the final RMSNorm) for batch item `item`:
 * prefill copies that prompt's rows [len, d], decode its single row [1, d],
 * into device float dst (capacity `cap_rows` rows).  Up to 8 captures may be
 * armed at once; each fires once.  GF_EINVAL on bad layer/item/cap. */
int gf_debug_capture(gf_model* m, int32_t layer, int32_t item, float* dst, int64_t cap_rows);

/* Copy the cached keys and values of sequence `handle` at positions
 * [start, start+n) of layer `layer` into dense device bf16 arrays
 * k_dst, v_dst [n, n_kv, head_dim].  Enqueued on `stream`. */
int gf_debug_read_kv(gf_model* m, int32_t layer, int32_t handle, int32_t start, int32_t n, void* k_dst,
                     void* v_dst, void* stream);

/* Synchronise `stream` and report a device-side timeout recorded by any
 * kernel of this model since the last call (GF_ETIMEOUT), then clear it. */
int gf_device_status(gf_model* m, void* stream);

/* Pages of the KV pool not referenced by any live sequence. */
int64_t gf_free_pages(const gf_model* m);

/* Number of kernels this model has launched since creation (for accounting). */
int64_t gf_launch_count(const gf_model* m);

/* Thread-local description of the last error; never NULL. */
const char* gf_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* GF_H_ */
