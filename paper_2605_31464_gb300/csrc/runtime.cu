// Host runtime behind the C ABI (include/gf.h): model creation and weight
// packing, the paged KV pool and its block tables, and the orchestration of
// prefill, greedy decode and the verdict/defer step on one CUDA stream.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <string>
#include <tuple>
#include <vector>

#include "gf.h"
#include "gemm_tc.cuh"
#include "kernels.h"
#include "page_pool.h"

using gf::bf16;

namespace {

thread_local std::string g_err = "no error";

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_err = buf;
  return code;
}

#define CU(x)                                                                                          \
  do {                                                                                                 \
    cudaError_t e_ = (x);                                                                              \
    if (e_ != cudaSuccess)                                                                             \
      return fail(GF_ECUDA, "%s failed: %s (%s:%d)", #x, cudaGetErrorString(e_), __FILE__, __LINE__); \
  } while (0)

#define TRY(x)             \
  do {                     \
    int rc_ = (x);         \
    if (rc_ != GF_OK) return rc_; \
  } while (0)

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 2D bf16 tensor map: `outer` rows of `inner` elements, row pitch in bytes,
// box {box_inner, box_outer}, 128-byte swizzle, zero fill out of bounds.
int make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t pitch_bytes,
             uint32_t box_inner, uint32_t box_outer) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return fail(GF_ECUDA, "cuTensorMapEncodeTiled is unavailable");
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {pitch_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return fail(GF_ECUDA, "cuTensorMapEncodeTiled failed (%d): inner %llu outer %llu pitch %llu box %u x %u",
                (int)r, (unsigned long long)inner, (unsigned long long)outer, (unsigned long long)pitch_bytes,
                box_inner, box_outer);
  return GF_OK;
}

// Pinned staging buffers for host->device uploads; a slot is reused only
// after the copy that last read it has executed.
struct Staging {
  struct Slot {
    void* host = nullptr;
    size_t cap = 0;
    cudaEvent_t ev = nullptr;
  };
  std::vector<Slot> slots;
  size_t next = 0;
  void release() {
    for (auto& s : slots) {
      if (s.ev) {
        cudaEventSynchronize(s.ev);
        cudaEventDestroy(s.ev);
      }
      if (s.host) cudaFreeHost(s.host);
    }
    slots.clear();
  }
};

int upload(Staging& st, void* dst, const void* src, size_t bytes, cudaStream_t s) {
  if (bytes == 0) return GF_OK;
  if (st.slots.empty()) st.slots.resize(8);
  Staging::Slot& sl = st.slots[st.next];
  st.next = (st.next + 1) % st.slots.size();
  if (!sl.ev) CU(cudaEventCreateWithFlags(&sl.ev, cudaEventDisableTiming));
  CU(cudaEventSynchronize(sl.ev));
  if (sl.cap < bytes) {
    if (sl.host) CU(cudaFreeHost(sl.host));
    sl.host = nullptr;
    sl.cap = 0;
    size_t cap = std::max<size_t>(bytes, 1 << 16);
    if (cudaHostAlloc(&sl.host, cap, cudaHostAllocDefault) != cudaSuccess) return fail(GF_ENOMEM, "pinned staging");
    sl.cap = cap;
  }
  memcpy(sl.host, src, bytes);
  CU(cudaMemcpyAsync(dst, sl.host, bytes, cudaMemcpyHostToDevice, s));
  CU(cudaEventRecord(sl.ev, s));
  return GF_OK;
}

struct Capture {
  int layer, item;
  float* dst;
  int64_t cap;
};

}  // namespace

struct gf_model {
  gf_config cfg{};
  int dev = 0, sms = 0;
  int L = 0, d = 0, nq = 0, nkv = 0, hd = 0, ffn = 0, ffn_pad = 0, vocab = 0, qkv_dim = 0, q_dim = 0;
  int64_t num_pages = 0;
  int max_pages = 0;  // pages per sequence
  int64_t T_max = 0;
  int B_max = 0;

  std::vector<void*> allocs;
  struct Layer {
    bf16 *qkv = nullptr, *o = nullptr, *gu = nullptr, *down = nullptr;
    float *attn_norm = nullptr, *ffn_norm = nullptr;
  };
  std::vector<Layer> layers;
  bf16 *embed = nullptr, *head = nullptr;
  float* final_norm = nullptr;
  bf16 *k_cache = nullptr, *v_cache = nullptr;
  CUtensorMap tm_k{}, tm_v{};
  int32_t *bt = nullptr, *seq_len = nullptr;
  float2* rope_cs = nullptr;

  // prefill activations (T_max rows)
  float* resid = nullptr;
  bf16* xn = nullptr;
  float* qkv = nullptr;
  int2* row_map = nullptr;  // prefill token -> (slot, position)
  float *ss_attn = nullptr, *ss_ffn = nullptr;  // prefill row sums of squares for the folded RMSNorm
  bf16* q = nullptr;
  bf16* attn = nullptr;
  bf16* act = nullptr;
  int32_t* prompt_ids = nullptr;
  int32_t* in_ids = nullptr;
  // small activations (B_max rows)
  float* dres = nullptr;
  bf16* dxn = nullptr;
  float* dqkv = nullptr;
  bf16* dattn = nullptr;
  bf16* dact = nullptr;
  float *part_o = nullptr, *part_ml = nullptr;
  int dec_chunk = 256, dec_max_splits = 1;
  float* logits = nullptr;  // [B_max, vocab]
  int32_t* last_idx = nullptr;
  int32_t* next = nullptr;
  int32_t* handles = nullptr;  // decode handles
  int32_t* call = nullptr;     // prefill descriptor: offsets | slots | items
  size_t call_ints = 0;
  int32_t* fcall = nullptr;    // forecast descriptor: inc_off | cand_off | prompt_off
  float* out_small = nullptr;  // host-variant outputs on the device
  int* err = nullptr;

  // host state: block tables and the reference-counted page pool; per slot its length and
  // whether it is live; the free slots
  gf::KvPagePool pool;
  std::vector<int32_t> h_len;
  std::vector<char> live;
  std::vector<int32_t> free_slots;
  std::vector<Capture> caps;
  std::map<std::tuple<const void*, uint64_t, uint64_t, uint32_t>, CUtensorMap> maps;
  Staging staging;
  int64_t launches = 0;
  // live kernel timing (gf_profile_*)
  uint32_t prof_mask = 0;
  struct ProfRec {
    cudaEvent_t a, b;
    int kind;
    double flops, bytes;
  };
  std::vector<ProfRec> prof;
  std::vector<cudaEvent_t> ev_pool;
  void* host_out = nullptr;
  size_t host_out_cap = 0;
  // greedy tokens of gf_forecast_batch: [B_max][tok_stride], column = decode step input index
  int32_t* tok_hist = nullptr;
  int tok_stride = 0;
  int32_t* ctl = nullptr;  // [0]: device decode-step counter
  unsigned long long* keys = nullptr;  // [B_max] fused greedy arg max keys (kept at zero between uses)
  gf::SampleParams* samp = nullptr;    // sampling parameters of the running sampled forecast
  // one CUDA graph per batch size for the decode step of gf_forecast_batch
  cudaStream_t cap_stream = nullptr;
  std::map<int, cudaGraphExec_t> graphs;
  int64_t graph_launches_per_step = 0;
  double weight_bytes = 0;  // bytes of all linear weights and the LM head (read once per decode step)
};

namespace {

template <typename T>
int dalloc(gf_model* m, T** p, size_t count) {
  void* v = nullptr;
  size_t bytes = std::max<size_t>(count * sizeof(T), 256);
  if (cudaMalloc(&v, bytes) != cudaSuccess) {
    cudaGetLastError();
    return fail(GF_ENOMEM, "cudaMalloc of %zu bytes failed", bytes);
  }
  m->allocs.push_back(v);
  *p = reinterpret_cast<T*>(v);
  return GF_OK;
}

int get_map(gf_model* m, const void* base, uint64_t inner, uint64_t outer, uint32_t box_outer, CUtensorMap* out) {
  auto key = std::make_tuple(base, inner, outer, box_outer);
  auto it = m->maps.find(key);
  if (it != m->maps.end()) {
    *out = it->second;
    return GF_OK;
  }
  TRY(make_map(out, base, inner, outer, inner * 2, 64, box_outer));
  if (m->maps.size() > 4096) m->maps.clear();
  m->maps[key] = *out;
  return GF_OK;
}

cudaEvent_t pool_event(gf_model* m) {
  if (!m->ev_pool.empty()) {
    cudaEvent_t e = m->ev_pool.back();
    m->ev_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Brackets one launch with events when its kernel class is being timed.
struct ProfScope {
  gf_model* m;
  cudaStream_t s;
  int kind;
  double flops, bytes;
  cudaEvent_t a = nullptr;
  ProfScope(gf_model* m_, cudaStream_t s_, int kind_, double flops_, double bytes_)
      : m(m_), s(s_), kind(kind_), flops(flops_), bytes(bytes_) {
    if (m->prof_mask & (1u << kind)) {
      a = pool_event(m);
      cudaEventRecord(a, s);
    }
  }
  ~ProfScope() {
    if (a) {
      cudaEvent_t b = pool_event(m);
      cudaEventRecord(b, s);
      m->prof.push_back({a, b, kind, flops, bytes});
    }
  }
};

// Tile width, split-K factor and operand order for a GEMM of M rows.  Few rows
// (decode) swap the operands: the weights fill the 128-row MMA dimension and the
// rows become a narrow N, so the pipeline streams mostly weight bytes.
void plan_gemm(int sms, int M, int N, int K, int mode, int* bn, int* splits, bool* swap) {
  const int num_m = (M + 127) / 128;
  *splits = 1;
  *swap = false;
  // SwiGLU above 64 rows: non-swapped 256-wide weight tiles move fewer activation bytes per weight byte
  // than 128-wide swapped ones (measured about 10 % faster at 96-128 rows)
  const bool swap_ok = mode == gf::kStoreF32 || mode == gf::kAtomicF32 || (mode == gf::kSwiGLU && M <= 64);
  if (M <= 128 && N % 32 == 0 && swap_ok) {
    *swap = true;
    *bn = M <= 32 ? 32 : (M <= 64 ? 64 : 128);
    if (mode == gf::kAtomicF32) {
      // about one wave of (tile, split) units: more splits add atomic traffic without adding bandwidth
      const int tiles = (N + 127) / 128;
      const int kb = K / 64;
      int s = (sms + tiles / 2) / tiles;
      s = std::min(s, std::max(1, kb / 4));
      *splits = std::max(1, s);
    }
    return;
  }
  if (mode == gf::kSwiGLU || mode == gf::kRopeQKV) {
    *bn = (num_m >= 4 || (mode == gf::kSwiGLU && M > 64)) ? 256 : 128;
    return;
  }
  if (num_m >= 4) {
    *bn = 256;
    return;
  }
  if (mode != gf::kAtomicF32) {
    *bn = 128;
    return;
  }
  *bn = 64;
  const int tiles = num_m * ((N + 63) / 64);
  const int kb = K / 64;
  int s = (2 * sms + tiles - 1) / tiles;
  s = std::min(s, std::max(1, kb / 4));
  *splits = std::max(1, s);
}

// Rows of a stored weight matrix: the GEMMs read every weight matrix in blocks of 256 rows x 64
// columns (launch_block_rows), so N is rounded up to whole blocks of zero rows.
int64_t weight_rows(int64_t n) { return (n + 255) / 256 * 256; }

// n_alg / k_alg: the unpadded output width and contraction length (algorithmic work).
// W is a weight matrix of the model, stored blocked (see weight_rows).

// keys: ask the LM-head GEMM to fuse the greedy arg max (*fused tells whether it could).
int gemm(gf_model* m, const bf16* A, int M, int K, const bf16* W, int N, void* out, int64_t ldo, int mode,
         cudaStream_t s, bool decode, int64_t n_alg = 0, int64_t k_alg = 0, unsigned long long* keys = nullptr,
         bool* fused = nullptr, const gf::SampleParams* sample = nullptr, const int32_t* sample_step = nullptr,
         int sample_bias = 0, const gf::RopeEpilogue* rope = nullptr, const gf::NormFold* norm = nullptr) {
  if (M <= 0) return GF_OK;
  int bn, splits;
  bool swap;
  plan_gemm(m->sms, M, N, K, mode, &bn, &splits, &swap);
  if (norm && swap) {
    // the folded RMSNorm is applied by the non-swapped epilogues only
    swap = false;
    bn = 128;
    splits = 1;
  }
  CUtensorMap ta, tb;
  const uint64_t w_rows64 = (uint64_t)weight_rows(N) * (uint64_t)(K / 64);  // 64-element rows of W
  if (swap) {
    TRY(get_map(m, W, 64, w_rows64, 128, &ta));
    TRY(get_map(m, A, (uint64_t)K, (uint64_t)M, (uint32_t)bn, &tb));
  } else {
    TRY(get_map(m, A, (uint64_t)K, (uint64_t)M, 128, &ta));
    TRY(get_map(m, W, 64, w_rows64, (uint32_t)bn, &tb));
  }
  const double na = n_alg ? n_alg : N, ka = k_alg ? k_alg : K;
  const double out_bytes =
      (mode == gf::kSwiGLU ? na / 2 * 2 : na * (mode == gf::kStoreBF16 || mode == gf::kRopeQKV ? 2 : 4)) * M;
  ProfScope ps(m, s, decode ? GF_PROF_DECODE_GEMM : GF_PROF_PREFILL_GEMM, 2.0 * M * na * ka,
               na * ka * 2 + (double)M * ka * 2 + out_bytes * (mode == gf::kAddF32 || mode == gf::kAtomicF32 ? 2 : 1));
  const bool use_keys = keys && swap && mode == gf::kStoreF32;
  if (fused) *fused = use_keys;
  if (swap)
    CU(gf::launch_gemm(ta, tb, N, M, K, out, ldo, mode, bn, splits, m->sms, m->err, s, 0, true,
                       use_keys ? keys : nullptr, sample, sample_step, sample_bias, nullptr, nullptr, true));
  else
    CU(gf::launch_gemm(ta, tb, M, N, K, out, ldo, mode, bn, splits, m->sms, m->err, s, 0, false, nullptr, nullptr,
                       nullptr, 0, rope, norm, true));
  m->launches += 1;
  return GF_OK;
}

int64_t layer_row0(const gf_model* m, int l) { return (int64_t)l * m->num_pages * m->nkv * 64; }

// Keys per decode-attention CTA: the largest of 1024/512/256 that still gives two CTAs per SM
// (longer chunks keep each CTA's page pipeline full and leave fewer partial results to merge).
int decode_chunk(int B, int n_kv, int max_ctx, int sms) {
  for (int chunk = 1024; chunk > 256; chunk /= 2)
    if ((int64_t)B * n_kv * ((max_ctx + chunk - 1) / chunk) >= 2 * sms) return chunk;
  return 256;
}
int64_t layer_vrow0(const gf_model* m, int l) { return (int64_t)l * m->num_pages * m->nkv * m->hd; }



int fire_captures(gf_model* m, int layer, const float* base, const int32_t* offsets_host, int B, bool decode,
                  cudaStream_t s) {
  for (size_t i = 0; i < m->caps.size();) {
    Capture& c = m->caps[i];
    if (c.layer == layer && c.item < B) {
      int64_t row0 = decode ? c.item : offsets_host[c.item];
      int64_t rows = decode ? 1 : (offsets_host[c.item + 1] - offsets_host[c.item]);
      rows = std::min(rows, c.cap);
      CU(cudaMemcpyAsync(c.dst, base + row0 * m->d, rows * m->d * sizeof(float), cudaMemcpyDeviceToDevice, s));
      m->caps.erase(m->caps.begin() + i);
    } else {
      ++i;
    }
  }
  return GF_OK;
}

int alloc_pages(gf_model* m, int slot, int first, int count, gf::KvPagePool::Undo* undo) {
  if (!m->pool.alloc(slot, first, count, undo)) return fail(GF_ECAPACITY, "KV page pool exhausted");
  return GF_OK;
}

void release_slot(gf_model* m, int slot) {
  m->pool.clear(slot);
  m->h_len[slot] = 0;
  m->live[slot] = 0;
  m->free_slots.push_back(slot);
}

int upload_block_table(gf_model* m, cudaStream_t s) {
  const std::vector<int32_t>& t = m->pool.table();
  return upload(m->staging, m->bt, t.data(), t.size() * sizeof(int32_t), s);
}

// Prefill of B packed prompts already on the device.  `reserve` extra
// tokens of KV pages are allocated per sequence (decode steps to come).
// past > 0: every prompt continues a cached prefix of `past` positions (a multiple of 64) whose
// pages belong to slot `share_slot`; the prompt's tokens sit at positions past, past+1, ...
// want_head = false skips the final norm, LM head and greedy token (prefix-only prefill).
int prefill_impl(gf_model* m, int B, const int32_t* ids, const int32_t* offsets, int reserve, int32_t* handles_out,
                 float* logits_dst, int32_t* next_dst, cudaStream_t s, int32_t* tokens_col = nullptr,
                 int64_t tokens_stride = 0, int past = 0, int share_slot = -1, bool want_head = true) {
  if (B < 1 || B > m->B_max) return fail(GF_EINVAL, "batch %d outside 1..%d", B, m->B_max);
  if (!ids || !offsets) return fail(GF_EINVAL, "null ids or offsets");
  if (offsets[0] != 0) return fail(GF_EINVAL, "offsets[0] must be 0");
  for (int b = 0; b < B; ++b) {
    const int len = offsets[b + 1] - offsets[b];
    if (len < 1) return fail(GF_EINVAL, "prompt %d has length %d", b, len);
    if (past + len + reserve > m->cfg.max_seq)
      return fail(GF_ECAPACITY, "prompt %d: %d tokens (+%d) exceed max_seq %d", b, past + len, reserve,
                  m->cfg.max_seq);
  }
  const int64_t T = offsets[B];
  if (T > m->T_max) return fail(GF_ECAPACITY, "%lld prompt tokens exceed max_prefill_tokens %lld", (long long)T,
                                (long long)m->T_max);
  if ((int)m->free_slots.size() < B) return fail(GF_ECAPACITY, "no free sequence slots");
  // slots and pages
  std::vector<int32_t> slots(B);
  gf::KvPagePool::Undo undo;
  for (int b = 0; b < B; ++b) {
    slots[b] = m->free_slots.back();
    m->free_slots.pop_back();
  }
  const int shared = past / 64;
  for (int b = 0; b < B; ++b) {
    const int len = offsets[b + 1] - offsets[b];
    if (shared > 0) m->pool.share(slots[b], share_slot, shared, &undo);
    const int rc = alloc_pages(m, slots[b], shared, (past + len + reserve + 63) / 64 - shared, &undo);
    if (rc != GF_OK) {
      m->pool.rollback(undo);
      for (int bb = B - 1; bb >= 0; --bb) m->free_slots.push_back(slots[bb]);
      return rc;
    }
  }
  for (int b = 0; b < B; ++b) {
    m->live[slots[b]] = 1;
    m->h_len[slots[b]] = past + offsets[b + 1] - offsets[b];
    handles_out[b] = slots[b];
  }
  // descriptor: offsets | slots | past | work items (heaviest first)
  std::vector<int32_t> desc;
  desc.insert(desc.end(), offsets, offsets + B + 1);
  desc.insert(desc.end(), slots.begin(), slots.end());
  desc.insert(desc.end(), (size_t)B, past);
  const size_t items_at = desc.size() + (desc.size() & 1);  // int2 alignment
  desc.resize(items_at);
  // attention work items: (prompt, pair of 128-row query tiles)
  std::vector<std::pair<int, int>> items;
  for (int b = 0; b < B; ++b) {
    const int len = offsets[b + 1] - offsets[b];
    for (int qt = 0; qt < (len + 255) / 256; ++qt) items.push_back({b, qt});
  }
  std::stable_sort(items.begin(), items.end(), [&](const std::pair<int, int>& x, const std::pair<int, int>& y) {
    auto cost = [&](const std::pair<int, int>& it) {
      const int len = offsets[it.first + 1] - offsets[it.first];
      return past + std::min(it.second * 256 + 256, len);
    };
    return cost(x) > cost(y);
  });
  for (auto& it : items) {
    desc.push_back(it.first);
    desc.push_back(it.second);
  }
  if (desc.size() > m->call_ints) return fail(GF_ECAPACITY, "prefill descriptor too large");
  TRY(upload(m->staging, m->call, desc.data(), desc.size() * sizeof(int32_t), s));
  TRY(upload_block_table(m, s));
  const int32_t* d_off = m->call;
  const int32_t* d_slots = m->call + B + 1;
  const int32_t* d_past = past > 0 ? m->call + 2 * B + 1 : nullptr;
  const int2* d_items = reinterpret_cast<const int2*>(m->call + items_at);

  CU(gf::launch_embed(ids, (int)T, m->embed, m->vocab, m->d, m->resid, m->err, s));
  m->launches++;
  // head_dim 128: RoPE and the KV-cache write are fused into the QKV GEMM's epilogue
  const bool fused_rope = m->hd == 128;
  gf::RopeEpilogue re{};
  if (fused_rope) {
    CU(gf::launch_token_map(d_off, d_slots, d_past, B, (int)T, m->row_map, s));
    m->launches++;
    re.row_map = m->row_map;
    re.rope_cs = m->rope_cs;
    re.q_out = m->q;
    re.ldq = m->q_dim;
    re.k_cache = m->k_cache;
    re.v_cache = m->v_cache;
    re.block_table = m->bt;
    re.max_pages = m->max_pages;
    re.n_q = m->nq;
    re.n_kv = m->nkv;
  }
  CUtensorMap tq;
  TRY(get_map(m, m->q, (uint64_t)m->q_dim, (uint64_t)T, 128, &tq));
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)m->hd);
  // With the fused RoPE path the two RMSNorms of a layer are folded into the GEMMs around them: the
  // residual-update GEMMs write xn = bf16(x * gain) with per-row sums of squares, and the QKV and
  // gate/up GEMMs scale their output rows by rsqrt(mean square + eps).
  gf::NormFold to_qkv{}, to_gu{}, from_o{}, from_down{};
  if (fused_rope) {
    const float inv_d = 1.0f / (float)m->d;
    to_qkv = gf::NormFold{nullptr, nullptr, nullptr, 0, m->ss_attn, inv_d, m->cfg.rms_eps};
    to_gu = gf::NormFold{nullptr, nullptr, nullptr, 0, m->ss_ffn, inv_d, m->cfg.rms_eps};
    from_o = gf::NormFold{m->xn, nullptr, m->ss_ffn, m->d, nullptr, 0.f, 0.f};
    from_down = gf::NormFold{m->xn, nullptr, m->ss_attn, m->d, nullptr, 0.f, 0.f};
    CU(gf::launch_norm_stats(m->resid, (int)T, m->d, m->layers[0].attn_norm, m->xn, m->ss_attn, s));
    m->launches++;
  }
  for (int l = 0; l < m->L; ++l) {
    const gf_model::Layer& W = m->layers[l];
    TRY(fire_captures(m, l, m->resid, offsets, B, false, s));
    if (!fused_rope) {
      CU(gf::launch_rmsnorm(m->resid, m->d, nullptr, (int)T, m->d, W.attn_norm, m->cfg.rms_eps, m->xn, m->d, s));
      m->launches++;
    }
    if (fused_rope) {
      re.layer_row0 = layer_row0(m, l);
      TRY(gemm(m, m->xn, (int)T, m->d, W.qkv, m->qkv_dim, nullptr, 0, gf::kRopeQKV, s, false, 0, 0, nullptr, nullptr,
               nullptr, nullptr, 0, &re, &to_qkv));
    } else {
      TRY(gemm(m, m->xn, (int)T, m->d, W.qkv, m->qkv_dim, m->qkv, m->qkv_dim, gf::kStoreF32, s, false));
      gf::RopeKvArgs ra{};
      ra.qkv = m->qkv;
      ra.ldqkv = m->qkv_dim;
      ra.q_out = m->q;
      ra.ldq = m->q_dim;
      ra.k_cache = m->k_cache;
      ra.v_cache = m->v_cache;
      ra.rope_cs = m->rope_cs;
      ra.offsets = d_off;
      ra.slots = d_slots;
      ra.past = d_past;
      ra.B = B;
      ra.block_table = m->bt;
      ra.max_pages = m->max_pages;
      ra.T = (int)T;
      ra.n_q = m->nq;
      ra.n_kv = m->nkv;
      ra.hd = m->hd;
      ra.layer_row0 = layer_row0(m, l);
      CU(gf::launch_rope_kv(ra, s));
      m->launches++;
    }
    gf::PrefillAttnArgs pa{};
    pa.items = d_items;
    pa.offsets = d_off;
    pa.slots = d_slots;
    pa.past = d_past;
    pa.block_table = m->bt;
    pa.max_pages = m->max_pages;
    pa.n_q = m->nq;
    pa.n_kv = m->nkv;
    pa.layer_row0 = layer_row0(m, l);
    pa.layer_vrow0 = layer_vrow0(m, l);
    pa.out = m->attn;
    pa.ldo = m->q_dim;
    pa.scale_log2 = scale_log2;
    pa.err = m->err;
    {
      double pairs = 0;
      for (int b = 0; b < B; ++b) {
        const double n = offsets[b + 1] - offsets[b];
        pairs += n * (n + 1) / 2 + n * past;
      }
      ProfScope ps(m, s, GF_PROF_PREFILL_ATTN, pairs * m->nq * 4.0 * m->hd,
                   (double)T * (m->q_dim * 2 + 2 * m->nkv * m->hd * 2 + m->q_dim * 2));
      CU(gf::launch_attn_prefill(m->hd, tq, m->tm_k, m->tm_v, pa, (int)items.size(), s));
    }
    m->launches++;
    if (fused_rope) {
      CU(cudaMemsetAsync(m->ss_ffn, 0, (size_t)T * sizeof(float), s));
      from_o.gain = W.ffn_norm;
      TRY(gemm(m, m->attn, (int)T, m->q_dim, W.o, m->d, m->resid, m->d, gf::kAddF32, s, false, 0, 0, nullptr, nullptr,
               nullptr, nullptr, 0, nullptr, &from_o));
      TRY(gemm(m, m->xn, (int)T, m->d, W.gu, 2 * m->ffn_pad, m->act, m->ffn_pad, gf::kSwiGLU, s, false, 2 * m->ffn, 0,
               nullptr, nullptr, nullptr, nullptr, 0, nullptr, &to_gu));
      // the last layer's output goes to the final norm (on the last rows only), not to another QKV
      const bool next = l + 1 < m->L;
      if (next) {
        CU(cudaMemsetAsync(m->ss_attn, 0, (size_t)T * sizeof(float), s));
        from_down.gain = m->layers[l + 1].attn_norm;
      }
      TRY(gemm(m, m->act, (int)T, m->ffn_pad, W.down, m->d, m->resid, m->d, gf::kAddF32, s, false, 0, m->ffn, nullptr,
               nullptr, nullptr, nullptr, 0, nullptr, next ? &from_down : nullptr));
    } else {
      TRY(gemm(m, m->attn, (int)T, m->q_dim, W.o, m->d, m->resid, m->d, gf::kAddF32, s, false));
      CU(gf::launch_rmsnorm(m->resid, m->d, nullptr, (int)T, m->d, W.ffn_norm, m->cfg.rms_eps, m->xn, m->d, s));
      m->launches++;
      TRY(gemm(m, m->xn, (int)T, m->d, W.gu, 2 * m->ffn_pad, m->act, m->ffn_pad, gf::kSwiGLU, s, false,
               2 * m->ffn));
      TRY(gemm(m, m->act, (int)T, m->ffn_pad, W.down, m->d, m->resid, m->d, gf::kAddF32, s, false, 0, m->ffn));
    }
  }
  TRY(fire_captures(m, m->L, m->resid, offsets, B, false, s));
  if (!want_head) {
    CU(gf::launch_set_seq_len(d_off, d_slots, B, m->seq_len, s, d_past));
    m->launches++;
    return GF_OK;
  }
  CU(gf::launch_last_rows(d_off, B, m->last_idx, s));
  CU(gf::launch_rmsnorm(m->resid, m->d, m->last_idx, B, m->d, m->final_norm, m->cfg.rms_eps, m->dxn, m->d, s));
  m->launches += 2;
  float* lg = logits_dst ? logits_dst : m->logits;
  bool fused = false;
  TRY(gemm(m, m->dxn, B, m->d, m->head, m->vocab, lg, m->vocab, gf::kStoreF32, s, false, 0, 0,
           next_dst ? m->keys : nullptr, &fused));
  if (next_dst) {
    if (fused)
      CU(gf::launch_finish_step(m->keys, B, next_dst, tokens_col, tokens_stride, nullptr, 0, 1 << 30, nullptr,
                                nullptr, s));
    else
      CU(gf::launch_argmax(lg, m->vocab, B, m->vocab, next_dst, tokens_col, tokens_stride, s));
    m->launches++;
  }
  CU(gf::launch_set_seq_len(d_off, d_slots, B, m->seq_len, s, d_past));
  m->launches++;
  return GF_OK;
}

// One decode step for B live sequences whose handles are already on the
// device in m->handles (host copy in `h`).
// With `step` (a device counter), the generated token is also written to
// tokens_col[b * tokens_stride + *step + 1] and the counter advanced, so that
// the step can be captured once in a CUDA graph and replayed.
int decode_impl(gf_model* m, int B, const int32_t* h, const int32_t* ids, float* logits_dst, int32_t* next_dst,
                int32_t* tokens_col, int64_t tokens_stride, cudaStream_t s, int32_t* step = nullptr,
                bool capturing = false, bool sampled = false) {
  CU(gf::launch_embed(ids, B, m->embed, m->vocab, m->d, m->dres, m->err, s));
  m->launches++;
  CU(cudaMemsetAsync(m->dqkv, 0, (size_t)B * m->qkv_dim * sizeof(float), s));
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)m->hd);
  for (int l = 0; l < m->L; ++l) {
    const gf_model::Layer& W = m->layers[l];
    if (!capturing) TRY(fire_captures(m, l, m->dres, nullptr, B, true, s));
    CU(gf::launch_rmsnorm(m->dres, m->d, nullptr, B, m->d, W.attn_norm, m->cfg.rms_eps, m->dxn, m->d, s));
    m->launches++;
    // split-K sums of q | k | v; the attention kernel rotates them, writes the new key and value
    // into the cache and zeroes these rows again
    TRY(gemm(m, m->dxn, B, m->d, W.qkv, m->qkv_dim, m->dqkv, m->qkv_dim, gf::kAtomicF32, s, true));
    gf::DecodeAttnArgs da{};
    da.handles = m->handles;
    da.seq_len = m->seq_len;
    da.ctx_bias = 1;
    da.max_ctx = m->dec_max_splits * m->dec_chunk;
    da.block_table = m->bt;
    da.max_pages = m->max_pages;
    da.n_q = m->nq;
    da.n_kv = m->nkv;
    da.layer_row0 = layer_row0(m, l);
    da.layer_vrow0 = layer_vrow0(m, l);
    da.chunk = decode_chunk(B, m->nkv, m->cfg.max_seq, m->sms);
    da.max_splits = (m->dec_max_splits * m->dec_chunk + da.chunk - 1) / da.chunk;
    da.part_o = m->part_o;
    da.part_ml = m->part_ml;
    da.out = m->dattn;
    da.ldo = m->q_dim;
    da.scale_log2 = scale_log2;
    da.err = m->err;
    da.qkv = m->dqkv;
    da.ldqkv = m->qkv_dim;
    da.rope_cs = m->rope_cs;
    da.k_cache = m->k_cache;
    da.v_cache = m->v_cache;
    {
      double ctx = 0;
      for (int b = 0; b < B; ++b) ctx += m->h_len[h[b]] + 1;
      ProfScope ps(m, s, GF_PROF_DECODE_ATTN, ctx * m->nq * 4.0 * m->hd,
                   ctx * 2.0 * m->nkv * m->hd * 2 + (double)B * m->q_dim * 4);
      CU(gf::launch_attn_decode(m->hd, m->tm_k, m->tm_v, da, B, s));
    }
    m->launches += 2;
    TRY(gemm(m, m->dattn, B, m->q_dim, W.o, m->d, m->dres, m->d, gf::kAtomicF32, s, true));
    CU(gf::launch_rmsnorm(m->dres, m->d, nullptr, B, m->d, W.ffn_norm, m->cfg.rms_eps, m->dxn, m->d, s));
    m->launches++;
    TRY(gemm(m, m->dxn, B, m->d, W.gu, 2 * m->ffn_pad, m->dact, m->ffn_pad, gf::kSwiGLU, s, true, 2 * m->ffn));
    TRY(gemm(m, m->dact, B, m->ffn_pad, W.down, m->d, m->dres, m->d, gf::kAtomicF32, s, true, 0, m->ffn));
  }
  if (!capturing) TRY(fire_captures(m, m->L, m->dres, nullptr, B, true, s));
  CU(gf::launch_rmsnorm(m->dres, m->d, nullptr, B, m->d, m->final_norm, m->cfg.rms_eps, m->dxn, m->d, s));
  m->launches++;
  float* lg = logits_dst ? logits_dst : m->logits;
  bool fused = false;
  // sampled: token t = *step + 1 of each row is drawn (temperature sampling, sampling.cuh)
  TRY(gemm(m, m->dxn, B, m->d, m->head, m->vocab, lg, m->vocab, gf::kStoreF32, s, true, 0, 0,
           next_dst ? m->keys : nullptr, &fused, sampled ? m->samp : nullptr, step, 1));
  if (next_dst && fused) {
    // greedy tokens from the LM head's fused arg max; advances the sequences and the step counter
    CU(gf::launch_finish_step(m->keys, B, next_dst, tokens_col, tokens_stride, step, step ? 1 : 0,
                              step ? (int)tokens_stride : (1 << 30), m->handles, m->seq_len, s));
    m->launches++;
  } else {
    if (next_dst) {
      if (sampled)
        CU(gf::launch_sample(lg, m->vocab, B, m->vocab, gf::SampleParams{}, m->samp, step, 1, next_dst, tokens_col,
                             tokens_stride, 1, step ? (int)tokens_stride : (1 << 30), s));
      else if (step)
        CU(gf::launch_argmax(lg, m->vocab, B, m->vocab, next_dst, tokens_col, tokens_stride, s, step, 1,
                             (int)tokens_stride));
      else
        CU(gf::launch_argmax(lg, m->vocab, B, m->vocab, next_dst, tokens_col, tokens_stride, s));
      m->launches++;
    }
    CU(gf::launch_advance(m->handles, B, m->seq_len, s, step));
    m->launches++;
  }
  if (!capturing)
    for (int b = 0; b < B; ++b) m->h_len[h[b]] += 1;
  return GF_OK;
}

// The decode step of gf_forecast_batch for a batch of B sequences whose
// handles are in m->handles, captured once as a CUDA graph: ids and tokens
// come from m->next, logits go to m->logits, generated tokens to m->tok_hist.
int decode_graph(gf_model* m, int B, const int32_t* h, cudaGraphExec_t* out, bool sampled = false) {
  const int key = B | (sampled ? 1 << 20 : 0);
  auto it = m->graphs.find(key);
  if (it != m->graphs.end()) {
    *out = it->second;
    return GF_OK;
  }
  if (!m->cap_stream) CU(cudaStreamCreateWithFlags(&m->cap_stream, cudaStreamNonBlocking));
  const uint32_t mask = m->prof_mask;
  m->prof_mask = 0;
  const int64_t launches = m->launches;
  CU(cudaStreamBeginCapture(m->cap_stream, cudaStreamCaptureModeThreadLocal));
  int rc = decode_impl(m, B, h, m->next, m->logits, m->next, m->tok_hist, m->tok_stride, m->cap_stream, m->ctl,
                       true, sampled);
  cudaGraph_t g = nullptr;
  const cudaError_t e = cudaStreamEndCapture(m->cap_stream, &g);
  m->prof_mask = mask;
  m->graph_launches_per_step = m->launches - launches;
  m->launches = launches;
  if (rc != GF_OK) {
    if (g) cudaGraphDestroy(g);
    return rc;
  }
  if (e != cudaSuccess) return fail(GF_ECUDA, "decode-step capture failed: %s", cudaGetErrorString(e));
  cudaGraphExec_t exec = nullptr;
  const cudaError_t e2 = cudaGraphInstantiate(&exec, g, 0);
  cudaGraphDestroy(g);
  if (e2 != cudaSuccess) return fail(GF_ECUDA, "graph instantiation failed: %s", cudaGetErrorString(e2));
  if (m->graphs.size() >= 16) {
    for (auto& kv : m->graphs) cudaGraphExecDestroy(kv.second);
    m->graphs.clear();
  }
  m->graphs[key] = exec;
  *out = exec;
  return GF_OK;
}

// Validate handles and allocate the pages the next token needs.
int prepare_decode(gf_model* m, int B, const int32_t* h, cudaStream_t s) {
  if (B < 1 || B > m->B_max) return fail(GF_EINVAL, "batch %d outside 1..%d", B, m->B_max);
  std::vector<char> seen(m->B_max, 0);
  for (int b = 0; b < B; ++b) {
    if (h[b] < 0 || h[b] >= m->B_max || !m->live[h[b]]) return fail(GF_EINVAL, "handle %d is not live", h[b]);
    if (seen[h[b]]) return fail(GF_EINVAL, "handle %d repeated", h[b]);
    seen[h[b]] = 1;
    if (m->h_len[h[b]] + 1 > m->cfg.max_seq) return fail(GF_ECAPACITY, "sequence %d reached max_seq", h[b]);
  }
  gf::KvPagePool::Undo undo;
  for (int b = 0; b < B; ++b) {
    const int pos = m->h_len[h[b]];
    const int rc = alloc_pages(m, h[b], pos / 64, 1, &undo);
    if (rc != GF_OK) {
      m->pool.rollback(undo);
      return rc;
    }
  }
  if (!undo.empty()) TRY(upload_block_table(m, s));
  return GF_OK;
}

}  // namespace

// Validates a forecast call and assembles its prompts (incumbent ++ candidate) into m->prompt_ids.
// poff receives the prompt offsets; the device copy sits at m->fcall + 2 (B + 1).
int assemble_prompts(gf_model* m, int B, const int32_t* inc_ids, const int32_t* inc_offsets, const int32_t* cand_ids,
                     const int32_t* cand_offsets, int n_decode, const int32_t* verdict_ids, int K, float tau,
                     std::vector<int32_t>& poff, cudaStream_t s) {
  if (K < 1 || K > 8) return fail(GF_EINVAL, "K = %d outside 1..8", K);
  if (!(tau >= 0.f && tau <= 1.f)) return fail(GF_EINVAL, "tau outside [0, 1]");
  if (n_decode < 0) return fail(GF_EINVAL, "n_decode < 0");
  for (int k = 0; k < K; ++k)
    if (verdict_ids[k] < 0 || verdict_ids[k] >= m->vocab) return fail(GF_EINVAL, "verdict id %d >= vocab", verdict_ids[k]);
  if (inc_offsets[0] != 0 || cand_offsets[0] != 0) return fail(GF_EINVAL, "offsets must start at 0");
  poff.assign(B + 1, 0);
  for (int b = 0; b < B; ++b) {
    const int ni = inc_offsets[b + 1] - inc_offsets[b], nc = cand_offsets[b + 1] - cand_offsets[b];
    if (ni < 0 || nc < 0 || ni + nc < 1) return fail(GF_EINVAL, "item %d: bad lengths %d + %d", b, ni, nc);
    if ((ni > 0 && !inc_ids) || (nc > 0 && !cand_ids)) return fail(GF_EINVAL, "null ids");
    poff[b + 1] = poff[b] + ni + nc;
  }
  if (poff[B] > m->T_max) return fail(GF_ECAPACITY, "prompt tokens exceed max_prefill_tokens");
  std::vector<int32_t> desc;
  desc.insert(desc.end(), inc_offsets, inc_offsets + B + 1);
  desc.insert(desc.end(), cand_offsets, cand_offsets + B + 1);
  desc.insert(desc.end(), poff.begin(), poff.end());
  TRY(upload(m->staging, m->fcall, desc.data(), desc.size() * sizeof(int32_t), s));
  CU(gf::launch_build_prompts(inc_ids, m->fcall, cand_ids, m->fcall + B + 1, m->fcall + 2 * (B + 1), B, poff[B],
                              m->prompt_ids, s));
  m->launches++;
  return GF_OK;
}

// Repeats of prefilled sequences: row b * R + j is h[b] for j = 0 and otherwise a new slot whose
// block table shares h[b]'s full 64-token pages (copy-free) and owns a fresh copy of its partial
// last page plus the pages of n_decode more tokens.  jobs receives (src slot, dst slot, src page,
// dst page) per fork for launch_fork_pages (pages -1: nothing to copy).  On failure every slot of
// rows and h is released.
int fork_sequences(gf_model* m, int B, int R, const int32_t* h, int n_decode, std::vector<int32_t>& rows,
                   std::vector<int32_t>& jobs) {
  gf::KvPagePool::Undo unused;
  for (int b = 0; b < B; ++b) rows[(size_t)b * R] = h[b];
  int rc = GF_OK;
  for (int b = 0; b < B && rc == GF_OK; ++b) {
    const int len = m->h_len[h[b]], full = len / 64;
    for (int j = 1; j < R && rc == GF_OK; ++j) {
      if (m->free_slots.empty()) {
        rc = fail(GF_ECAPACITY, "no free sequence slots");
        break;
      }
      const int slot = m->free_slots.back();
      m->free_slots.pop_back();
      m->live[slot] = 1;
      m->h_len[slot] = len;
      rows[(size_t)b * R + j] = slot;
      m->pool.share(slot, h[b], full, &unused);
      rc = alloc_pages(m, slot, full, (len + n_decode + 63) / 64 - full, &unused);
      const bool partial = len % 64 != 0;
      jobs.insert(jobs.end(), {h[b], slot, partial ? m->pool.entry(h[b], full) : -1,
                               partial ? m->pool.entry(slot, full) : -1});
    }
  }
  if (rc != GF_OK) {
    for (int r = 0; r < B * R; ++r)
      if (rows[r] >= 0) release_slot(m, rows[r]);
    for (int b = 0; b < B; ++b) rows[(size_t)b * R] = -1;
  }
  return rc;
}

// Token 0 of the B x R sampled rows: the final norm of each prompt's last position (once per
// repeat), the LM head into lg and the draw (into m->next and column 0 of m->tok_hist).  The
// prompt offsets are the ones assemble_prompts left on the device.
int sampled_head(gf_model* m, int B, int R, float* lg, cudaStream_t s) {
  const int BR = B * R;
  CU(gf::launch_last_rows(m->fcall + 2 * (B + 1), B, m->last_idx, s, R));
  CU(gf::launch_rmsnorm(m->resid, m->d, m->last_idx, BR, m->d, m->final_norm, m->cfg.rms_eps, m->dxn, m->d, s));
  m->launches += 2;
  bool fused = false;
  TRY(gemm(m, m->dxn, BR, m->d, m->head, m->vocab, lg, m->vocab, gf::kStoreF32, s, false, 0, 0, m->keys, &fused,
           m->samp, nullptr, 0));
  if (fused)
    CU(gf::launch_finish_step(m->keys, BR, m->next, m->tok_hist, m->tok_stride, nullptr, 0, 1 << 30, nullptr,
                              nullptr, s));
  else
    CU(gf::launch_sample(lg, m->vocab, BR, m->vocab, gf::SampleParams{}, m->samp, nullptr, 0, m->next, m->tok_hist,
                         m->tok_stride, 0, 1 << 30, s));
  m->launches++;
  return GF_OK;
}

// The part of a forecast after the prefill: n_decode greedy steps (the first eager, the rest one
// replayed CUDA graph), the verdict on the final logits, and the release of the sequences.
int decode_verdict_release(gf_model* m, int B, std::vector<int32_t>& h, int n_decode, const int32_t* verdict_ids,
                           int K, float tau, float* p, float* conf, int32_t* verdict_arg, uint8_t* defer,
                           int32_t* tokens, float* final_logits, float* lg, cudaStream_t s,
                           bool sampled = false) {
  int rc = upload(m->staging, m->handles, h.data(), (size_t)B * sizeof(int32_t), s);
  if (rc == GF_OK && n_decode > 0) {
    lg = m->logits;
    if (cudaMemsetAsync(m->ctl, 0, sizeof(int32_t), s) != cudaSuccess) rc = fail(GF_ECUDA, "memset failed");
    // the first step runs eagerly (it also configures the kernels); the rest replay one captured graph
    if (rc == GF_OK)
      rc = decode_impl(m, B, h.data(), m->next, m->logits, m->next, m->tok_hist, m->tok_stride, s, m->ctl, false,
                       sampled);
    if (rc == GF_OK && n_decode > 1) {
      cudaGraphExec_t exec = nullptr;
      rc = decode_graph(m, B, h.data(), &exec, sampled);
      // algorithmic bytes of the replayed steps: every weight once per step, the cached K/V each
      // sequence reads, and the new K/V rows written
      double bytes = 0;
      if (m->prof_mask & (1u << GF_PROF_DECODE_STEPS)) {
        const double kv_tok = (double)m->L * m->nkv * m->hd * 2 * 2;
        for (int step = 1; step < n_decode; ++step) {
          double ctx = 0;
          for (int b = 0; b < B; ++b) ctx += m->h_len[h[b]] + step;  // context of this step's query
          bytes += m->weight_bytes + ctx * kv_tok + (double)B * kv_tok;
        }
      }
      {
        ProfScope ps(m, s, GF_PROF_DECODE_STEPS, 0.0, bytes);
        for (int step = 1; step < n_decode && rc == GF_OK; ++step) {
          const cudaError_t e = cudaGraphLaunch(exec, s);
          if (e != cudaSuccess) rc = fail(GF_ECUDA, "graph launch failed: %s", cudaGetErrorString(e));
          m->launches += m->graph_launches_per_step;
        }
      }
      if (rc == GF_OK)
        for (int b = 0; b < B; ++b) m->h_len[h[b]] += n_decode - 1;
    }
    if (rc == GF_OK && final_logits &&
        cudaMemcpyAsync(final_logits, m->logits, (size_t)B * m->vocab * sizeof(float), cudaMemcpyDeviceToDevice,
                        s) != cudaSuccess)
      rc = fail(GF_ECUDA, "logits copy failed");
  }
  if (rc == GF_OK && tokens && n_decode > 0 &&
      cudaMemcpy2DAsync(tokens, (size_t)n_decode * sizeof(int32_t), m->tok_hist, (size_t)m->tok_stride * sizeof(int32_t),
                        (size_t)n_decode * sizeof(int32_t), B, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    rc = fail(GF_ECUDA, "tokens copy failed");
  if (rc == GF_OK) {
    const cudaError_t e = gf::launch_verdict(lg, m->vocab, B, verdict_ids, K, tau, p, conf, verdict_arg, defer, s);
    if (e != cudaSuccess) rc = fail(GF_ECUDA, "verdict launch: %s", cudaGetErrorString(e));
    m->launches++;
  }
  for (int b = 0; b < B; ++b) release_slot(m, h[b]);
  return rc;
}

// Helpers for entry points defined in other translation units.
namespace gf {
// Tensor map over a KV pool viewed as `rows` rows of hd bf16 (boxes of 64 x 64); 0 on success.
int encode_kv_map(CUtensorMap* m, const void* base, int hd, uint64_t rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return 1;
  cuuint64_t dims[2] = {(cuuint64_t)hd, rows};
  cuuint64_t strides[1] = {(cuuint64_t)hd * 2};
  cuuint32_t box[2] = {64, 64};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS
             ? 0
             : 1;
}
int encode_vt_map(CUtensorMap* m, const void* base, int hd, uint64_t rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return 1;
  cuuint64_t dims[2] = {64, rows};
  cuuint64_t strides[1] = {128};
  cuuint32_t box[2] = {64, (cuuint32_t)hd};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS
             ? 0
             : 1;
}
// Record a message of at most 15 characters (kept in the string's inline buffer, so nothing is allocated).
void set_error_short(const char* msg) { g_err = msg; }

uint64_t current_context_id() {
  typedef CUresult (*GetCurrentFn)(CUcontext*);
  typedef CUresult (*GetIdFn)(CUcontext, unsigned long long*);
  static GetCurrentFn get_current = nullptr;
  static GetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<GetCurrentFn>(p);
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<GetIdFn>(p);
  });
  if (!get_current || !get_id) return 0;
  CUcontext c = nullptr;
  unsigned long long id = 0;
  if (get_current(&c) != CUDA_SUCCESS || !c || get_id(c, &id) != CUDA_SUCCESS) return 0;
  return id;
}
}  // namespace gf

// =====================================================================================================
// C ABI
// =====================================================================================================
extern "C" {

const char* gf_last_error(void) { return g_err.c_str(); }

int64_t gf_launch_count(const gf_model* m) { return m ? m->launches : 0; }

int64_t gf_free_pages(const gf_model* m) { return m ? m->pool.free_pages() : 0; }

void gf_destroy(gf_model* m) {
  if (!m) return;
  cudaDeviceSynchronize();
  for (auto& kv : m->graphs) cudaGraphExecDestroy(kv.second);
  if (m->cap_stream) cudaStreamDestroy(m->cap_stream);
  m->staging.release();
  for (void* p : m->allocs) cudaFree(p);
  if (m->host_out) cudaFreeHost(m->host_out);
  delete m;
}

int gf_create(const gf_config* cfg, const gf_weights* w, void* stream, gf_model** out) {
  if (!cfg || !w || !out) return fail(GF_EINVAL, "null argument");
  *out = nullptr;
  const gf_config& c = *cfg;
  if (c.layers < 1 || c.d_model < 64 || c.d_model % 64 || c.n_q < 1 || c.n_kv < 1 || c.n_q % c.n_kv ||
      c.ffn < 1 || c.vocab < 32 || c.max_batch < 1 || c.max_batch > 1024 || c.max_seq < 1 ||
      c.max_prefill_tokens < 1 || !(c.rms_eps >= 0.f) || !(c.rope_theta > 0.f))
    return fail(GF_EINVAL, "invalid configuration");
  if (c.head_dim != 64 && c.head_dim != 128) return fail(GF_ENOTIMPL, "head_dim must be 64 or 128");
  if (c.n_q / c.n_kv > 16) return fail(GF_ENOTIMPL, "more than 16 query heads per KV head");
  if (c.vocab % 32) return fail(GF_ENOTIMPL, "vocab must be a multiple of 32");
  if (!w->embed || !w->lm_head || !w->final_norm || !w->attn_norm || !w->wq || !w->wk || !w->wv || !w->wo ||
      !w->ffn_norm || !w->w_gate || !w->w_up || !w->w_down)
    return fail(GF_EINVAL, "null weight pointer");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  gf_model* m = new gf_model();
  m->cfg = c;
  int rc = GF_OK;
  auto bail = [&](int code) {
    gf_destroy(m);
    return code;
  };
  if (cudaGetDevice(&m->dev) != cudaSuccess) return bail(fail(GF_ECUDA, "no CUDA device"));
  cudaDeviceGetAttribute(&m->sms, cudaDevAttrMultiProcessorCount, m->dev);
  int major = 0, minor = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, m->dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, m->dev);
  if (major != 10) return bail(fail(GF_ENOTIMPL, "needs a Blackwell (sm_10x) GPU, found sm_%d%d", major, minor));
  m->L = c.layers;
  m->d = c.d_model;
  m->nq = c.n_q;
  m->nkv = c.n_kv;
  m->hd = c.head_dim;
  m->ffn = c.ffn;
  m->ffn_pad = (c.ffn + 63) / 64 * 64;
  m->vocab = c.vocab;
  m->q_dim = c.n_q * c.head_dim;
  m->qkv_dim = (c.n_q + 2 * c.n_kv) * c.head_dim;
  m->B_max = c.max_batch;
  m->T_max = c.max_prefill_tokens;
  m->max_pages = (c.max_seq + 63) / 64;
  m->num_pages = c.kv_pages > 0 ? c.kv_pages : (int64_t)c.max_batch * m->max_pages;
  if ((int64_t)m->L * m->num_pages * m->nkv * 64 >= ((int64_t)1 << 31))
    return bail(fail(GF_ENOTIMPL, "KV pool too large for 32-bit TMA row coordinates"));
  m->dec_max_splits = (c.max_seq + m->dec_chunk - 1) / m->dec_chunk;

  // ---- weights
  const int d = m->d, hd = m->hd;
  m->layers.resize(m->L);
  for (int l = 0; l < m->L && rc == GF_OK; ++l) {
    gf_model::Layer& W = m->layers[l];
    rc = dalloc(m, &W.qkv, (size_t)weight_rows(m->qkv_dim) * d);
    if (!rc) rc = dalloc(m, &W.o, (size_t)weight_rows(d) * m->q_dim);
    if (!rc) rc = dalloc(m, &W.gu, (size_t)weight_rows(2 * m->ffn_pad) * d);
    if (!rc) rc = dalloc(m, &W.down, (size_t)weight_rows(d) * m->ffn_pad);
    if (!rc) rc = dalloc(m, &W.attn_norm, d);
    if (!rc) rc = dalloc(m, &W.ffn_norm, d);
  }
  if (!rc) rc = dalloc(m, &m->embed, (size_t)m->vocab * d);
  if (!rc) rc = dalloc(m, &m->head, (size_t)weight_rows(m->vocab) * d);
  if (!rc) rc = dalloc(m, &m->final_norm, d);
  // ---- KV pool, tables
  const size_t cache_elems = (size_t)m->L * m->num_pages * m->nkv * 64 * hd;
  if (!rc) rc = dalloc(m, &m->k_cache, cache_elems);
  if (!rc) rc = dalloc(m, &m->v_cache, cache_elems);
  if (!rc) rc = dalloc(m, &m->bt, (size_t)m->B_max * m->max_pages);
  if (!rc) rc = dalloc(m, &m->seq_len, m->B_max);
  if (!rc) rc = dalloc(m, &m->rope_cs, (size_t)c.max_seq * (hd / 2));
  // ---- activations
  const size_t T = (size_t)m->T_max;
  if (!rc) rc = dalloc(m, &m->resid, T * d);
  if (!rc) rc = dalloc(m, &m->xn, T * d);
  if (!rc) rc = dalloc(m, &m->qkv, T * m->qkv_dim);
  if (!rc) rc = dalloc(m, &m->row_map, T);
  if (!rc) rc = dalloc(m, &m->ss_attn, T);
  if (!rc) rc = dalloc(m, &m->ss_ffn, T);
  if (!rc) rc = dalloc(m, &m->q, T * m->q_dim);
  if (!rc) rc = dalloc(m, &m->attn, T * m->q_dim);
  if (!rc) rc = dalloc(m, &m->act, T * m->ffn_pad);
  if (!rc) rc = dalloc(m, &m->prompt_ids, T);
  if (!rc) rc = dalloc(m, &m->in_ids, T);
  const size_t Bm = (size_t)m->B_max;
  if (!rc) rc = dalloc(m, &m->dres, Bm * d);
  if (!rc) rc = dalloc(m, &m->dxn, Bm * d);
  if (!rc) rc = dalloc(m, &m->dqkv, Bm * m->qkv_dim);
  if (!rc) rc = dalloc(m, &m->dattn, Bm * m->q_dim);
  if (!rc) rc = dalloc(m, &m->dact, Bm * m->ffn_pad);
  if (!rc) rc = dalloc(m, &m->part_o, Bm * m->nkv * m->dec_max_splits * 16 * hd);
  if (!rc) rc = dalloc(m, &m->part_ml, Bm * m->nkv * m->dec_max_splits * 16 * 2);
  if (!rc) rc = dalloc(m, &m->logits, Bm * m->vocab);
  if (!rc) rc = dalloc(m, &m->last_idx, Bm);
  if (!rc) rc = dalloc(m, &m->next, Bm);
  if (!rc) rc = dalloc(m, &m->handles, Bm);
  m->call_ints = 3 * Bm + 8 + 2 * (size_t)(T / 128 + Bm + 8);
  if (!rc) rc = dalloc(m, &m->call, m->call_ints);
  if (!rc) rc = dalloc(m, &m->fcall, 3 * Bm + 8);
  if (!rc) rc = dalloc(m, &m->out_small, Bm * 12);
  if (!rc) rc = dalloc(m, &m->err, 1);
  m->tok_stride = c.max_seq;
  if (!rc) rc = dalloc(m, &m->tok_hist, Bm * m->tok_stride);
  if (!rc) rc = dalloc(m, &m->ctl, 4);
  if (!rc) rc = dalloc(m, &m->keys, Bm);
  if (!rc) rc = dalloc(m, &m->samp, 1);
  if (rc) return bail(rc);

  // ---- pack weights: q, k, v rows stacked and gate/up interleaved (row-major, in a scratch
  // buffer), then every GEMM weight stored in 256 x 64 blocks
  auto cp = [&](void* dst, const void* src, size_t bytes) {
    return cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, s);
  };
  struct Scratch {
    bf16* p = nullptr;
    ~Scratch() {
      if (p) cudaFree(p);
    }
  } tmp;
  if (cudaMalloc(&tmp.p, std::max((size_t)m->qkv_dim, (size_t)2 * m->ffn_pad) * d * sizeof(bf16)) != cudaSuccess) {
    cudaGetLastError();
    return bail(fail(GF_ENOMEM, "weight packing scratch"));
  }
  cudaError_t e = cudaSuccess;
  const size_t qb = (size_t)m->q_dim * d * 2, kb = (size_t)m->nkv * hd * d * 2;
  for (int l = 0; l < m->L && e == cudaSuccess; ++l) {
    gf_model::Layer& W = m->layers[l];
    if (!w->wq[l] || !w->wk[l] || !w->wv[l] || !w->wo[l] || !w->w_gate[l] || !w->w_up[l] || !w->w_down[l] ||
        !w->attn_norm[l] || !w->ffn_norm[l]) {
      cudaStreamSynchronize(s);
      return bail(fail(GF_EINVAL, "null weight pointer in layer %d", l));
    }
    e = cp(tmp.p, w->wq[l], qb);
    if (e == cudaSuccess) e = cp(reinterpret_cast<char*>(tmp.p) + qb, w->wk[l], kb);
    if (e == cudaSuccess) e = cp(reinterpret_cast<char*>(tmp.p) + qb + kb, w->wv[l], kb);
    if (e == cudaSuccess) e = gf::launch_block_rows(tmp.p, m->qkv_dim, d, d, d, W.qkv, s);
    if (e == cudaSuccess)
      e = gf::launch_block_rows(reinterpret_cast<const bf16*>(w->wo[l]), d, m->q_dim, m->q_dim, m->q_dim, W.o, s);
    if (e == cudaSuccess)
      e = gf::launch_pack_gate_up(reinterpret_cast<const bf16*>(w->w_gate[l]),
                                  reinterpret_cast<const bf16*>(w->w_up[l]), m->ffn, m->ffn_pad, d, tmp.p, s);
    if (e == cudaSuccess) e = gf::launch_block_rows(tmp.p, 2 * m->ffn_pad, d, d, d, W.gu, s);
    if (e == cudaSuccess)
      e = gf::launch_block_rows(reinterpret_cast<const bf16*>(w->w_down[l]), d, m->ffn, m->ffn, m->ffn_pad, W.down,
                                s);
    if (e == cudaSuccess) e = gf::launch_bf16_to_f32(reinterpret_cast<const bf16*>(w->attn_norm[l]), d, W.attn_norm, s);
    if (e == cudaSuccess) e = gf::launch_bf16_to_f32(reinterpret_cast<const bf16*>(w->ffn_norm[l]), d, W.ffn_norm, s);
  }
  m->weight_bytes = (double)m->L * ((double)m->qkv_dim * d + (double)d * m->q_dim + 2.0 * m->ffn * d +
                                    (double)d * m->ffn) * 2 + (double)m->vocab * d * 2;
  if (e == cudaSuccess) e = cp(m->embed, w->embed, (size_t)m->vocab * d * 2);
  if (e == cudaSuccess) e = gf::launch_block_rows(reinterpret_cast<const bf16*>(w->lm_head), m->vocab, d, d, d, m->head, s);
  if (e == cudaSuccess) e = gf::launch_bf16_to_f32(reinterpret_cast<const bf16*>(w->final_norm), d, m->final_norm, s);
  if (e == cudaSuccess) e = gf::launch_rope_table(c.rope_theta, hd, c.max_seq, m->rope_cs, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(m->dqkv, 0, Bm * m->qkv_dim * sizeof(float), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(m->err, 0, sizeof(int), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(m->seq_len, 0, Bm * sizeof(int32_t), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(m->keys, 0, Bm * sizeof(unsigned long long), s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    cudaStreamSynchronize(s);  // nothing may still read the scratch buffer when it is freed
    return bail(fail(GF_ECUDA, "weight packing failed: %s", cudaGetErrorString(e)));
  }

  // ---- host state
  m->pool.init(m->B_max, m->max_pages, m->num_pages);
  m->h_len.assign(m->B_max, 0);
  m->live.assign(m->B_max, 0);
  for (int sl = m->B_max - 1; sl >= 0; --sl) m->free_slots.push_back(sl);
  const uint64_t rows = (uint64_t)m->L * m->num_pages * m->nkv * 64;
  if ((rc = make_map(&m->tm_k, m->k_cache, hd, rows, hd * 2, 64, 64))) return bail(rc);
  if ((rc = make_map(&m->tm_v, m->v_cache, 64, rows / 64 * hd, 128, 64, hd))) return bail(rc);
  if ((rc = upload_block_table(m, s))) return bail(rc);
  if (cudaStreamSynchronize(s) != cudaSuccess) return bail(fail(GF_ECUDA, "create: sync failed"));
  *out = m;
  return GF_OK;
}

int gf_prefill(gf_model* m, int32_t B, const int32_t* ids, const int32_t* offsets, int32_t* seq_handles,
               float* last_logits, int32_t* next_ids, void* stream) {
  if (!m || !seq_handles) return fail(GF_EINVAL, "null argument");
  return prefill_impl(m, B, ids, offsets, 0, seq_handles, last_logits, next_ids,
                      reinterpret_cast<cudaStream_t>(stream));
}

int gf_decode_step(gf_model* m, int32_t B, const int32_t* seq_handles, const int32_t* ids, float* logits,
                   int32_t* next_ids, void* stream) {
  if (!m || !seq_handles || !ids) return fail(GF_EINVAL, "null argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  TRY(prepare_decode(m, B, seq_handles, s));
  TRY(upload(m->staging, m->handles, seq_handles, (size_t)B * sizeof(int32_t), s));
  return decode_impl(m, B, seq_handles, ids, logits, next_ids, nullptr, 0, s);
}

int gf_release(gf_model* m, int32_t B, const int32_t* seq_handles) {
  if (!m || (B > 0 && !seq_handles)) return fail(GF_EINVAL, "null argument");
  for (int b = 0; b < B; ++b) {
    const int h = seq_handles[b];
    if (h < 0 || h >= m->B_max || !m->live[h]) return fail(GF_EINVAL, "handle %d is not live", h);
  }
  for (int b = 0; b < B; ++b) release_slot(m, seq_handles[b]);
  return GF_OK;
}

int gf_sample_tokens(int32_t B, const float* logits, int64_t ld, int32_t V, uint64_t seed, int32_t token_index,
                     float temperature, int32_t* out_ids, void* stream) {
  if (B < 0 || V < 1 || ld < V || token_index < 0) return fail(GF_EINVAL, "bad shape");
  if (!(temperature > 0.f) || !std::isfinite(temperature)) return fail(GF_EINVAL, "temperature must be > 0");
  if (B == 0) return GF_OK;
  if (!logits || !out_ids) return fail(GF_EINVAL, "null argument");
  const gf::SampleParams sp{(unsigned long long)seed, 1.0f / temperature, 0};
  CU(gf::launch_sample(logits, ld, B, V, sp, nullptr, nullptr, token_index, out_ids, nullptr, 0, 0, 0,
                       reinterpret_cast<cudaStream_t>(stream)));
  return GF_OK;
}

int gf_verdict(int32_t B, const float* logits, int64_t ld, const int32_t* verdict_ids, int32_t K, float tau,
               float* p, float* conf, int32_t* verdict_arg, uint8_t* defer, void* stream) {
  if (B < 0 || !logits || !verdict_ids || !p || !conf || !verdict_arg || !defer)
    return fail(GF_EINVAL, "null argument");
  if (K < 1 || K > 8) return fail(GF_EINVAL, "K = %d outside 1..8", K);
  if (!(tau >= 0.f && tau <= 1.f)) return fail(GF_EINVAL, "tau outside [0, 1]");
  for (int k = 0; k < K; ++k)
    if (verdict_ids[k] < 0 || verdict_ids[k] >= ld) return fail(GF_EINVAL, "verdict id %d outside the row", verdict_ids[k]);
  CU(gf::launch_verdict(logits, ld, B, verdict_ids, K, tau, p, conf, verdict_arg, defer,
                        reinterpret_cast<cudaStream_t>(stream)));
  return GF_OK;
}

int gf_forecast_batch(gf_model* m, int32_t B, const int32_t* inc_ids, const int32_t* inc_offsets,
                      const int32_t* cand_ids, const int32_t* cand_offsets, int32_t n_decode,
                      const int32_t* verdict_ids, int32_t K, float tau, float* p, float* conf,
                      int32_t* verdict_arg, uint8_t* defer, int32_t* tokens, float* final_logits, void* stream) {
  if (!m || !inc_offsets || !cand_offsets || !verdict_ids || !p || !conf || !verdict_arg || !defer)
    return fail(GF_EINVAL, "null argument");
  if (B < 1 || B > m->B_max) return fail(GF_EINVAL, "batch %d outside 1..%d", B, m->B_max);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  std::vector<int32_t> poff;
  TRY(assemble_prompts(m, B, inc_ids, inc_offsets, cand_ids, cand_offsets, n_decode, verdict_ids, K, tau, poff, s));
  std::vector<int32_t> h(B);
  float* lg = (n_decode == 0 && final_logits) ? final_logits : m->logits;
  // tok_hist[b, s] is the input of decode step s: the arg max of the logits before it
  TRY(prefill_impl(m, B, m->prompt_ids, poff.data(), n_decode, h.data(), lg, m->next, s, m->tok_hist,
                   m->tok_stride));
  return decode_verdict_release(m, B, h, n_decode, verdict_ids, K, tau, p, conf, verdict_arg, defer, tokens,
                                final_logits, lg, s);
}

int gf_forecast_batch_sampled(gf_model* m, int32_t B, const int32_t* inc_ids, const int32_t* inc_offsets,
                              const int32_t* cand_ids, const int32_t* cand_offsets, int32_t n_decode,
                              int32_t repeats, float temperature, uint64_t seed, const int32_t* verdict_ids,
                              int32_t K, float tau, float* p, float* conf, int32_t* verdict_arg, uint8_t* defer,
                              float* p_mean, float* p_std, float* conf_mean, float* conf_std, int32_t* tokens,
                              float* final_logits, void* stream) {
  if (!m || !inc_offsets || !cand_offsets || !verdict_ids || !p || !conf || !verdict_arg || !defer)
    return fail(GF_EINVAL, "null argument");
  if (repeats < 1) return fail(GF_EINVAL, "repeats = %d < 1", repeats);
  if (!(temperature > 0.f) || !std::isfinite(temperature)) return fail(GF_EINVAL, "temperature must be > 0");
  if (B < 1 || (int64_t)B * repeats > m->B_max)
    return fail(GF_EINVAL, "batch %d x %d repeats outside 1..%d rows", B, repeats, m->B_max);
  const int R = repeats, BR = B * R;
  if ((int)m->free_slots.size() < BR) return fail(GF_ECAPACITY, "no free sequence slots");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  std::vector<int32_t> poff;
  TRY(assemble_prompts(m, B, inc_ids, inc_offsets, cand_ids, cand_offsets, n_decode, verdict_ids, K, tau, poff, s));
  // each prompt is prefilled once; its repeats are forks that share its full KV pages
  std::vector<int32_t> h(B);
  TRY(prefill_impl(m, B, m->prompt_ids, poff.data(), n_decode, h.data(), nullptr, nullptr, s, nullptr, 0, 0, -1,
                   false));
  std::vector<int32_t> rows(BR, -1);
  std::vector<int32_t> jobs;
  int rc = fork_sequences(m, B, R, h.data(), n_decode, rows, jobs);
  if (rc == GF_OK) rc = upload_block_table(m, s);
  if (rc == GF_OK && !jobs.empty()) rc = upload(m->staging, m->call, jobs.data(), jobs.size() * sizeof(int32_t), s);
  if (rc == GF_OK) {
    const int64_t page_elems = (int64_t)m->nkv * 64 * m->hd;
    if (gf::launch_fork_pages(m->k_cache, m->v_cache, reinterpret_cast<const int4*>(m->call), (int)jobs.size() / 4,
                              m->L, page_elems, m->num_pages * page_elems, m->seq_len, s) != cudaSuccess)
      rc = fail(GF_ECUDA, "fork launch failed");
    m->launches++;
  }
  const gf::SampleParams sp{(unsigned long long)seed, 1.0f / temperature, 0};
  if (rc == GF_OK) rc = upload(m->staging, m->samp, &sp, sizeof(sp), s);
  // token 0 of every row from its prompt's last position: final norm, LM head and the draw
  float* lg = (n_decode == 0 && final_logits) ? final_logits : m->logits;
  if (rc == GF_OK) rc = sampled_head(m, B, R, lg, s);
  if (rc != GF_OK) {
    for (int r = 0; r < BR; ++r)
      if (rows[r] >= 0) release_slot(m, rows[r]);
    return rc;
  }
  TRY(decode_verdict_release(m, BR, rows, n_decode, verdict_ids, K, tau, p, conf, verdict_arg, defer, tokens,
                             final_logits, lg, s, true));
  if (p_mean || p_std || conf_mean || conf_std) {
    CU(gf::launch_repeat_stats(p, conf, B, R, K, p_mean, p_std, conf_mean, conf_std, s));
    m->launches++;
  }
  return GF_OK;
}

int gf_forecast_batch_shared(gf_model* m, int32_t B, const int32_t* prefix_ids, int32_t prefix_len,
                             const int32_t* cand_ids, const int32_t* cand_offsets, int32_t n_decode,
                             const int32_t* verdict_ids, int32_t K, float tau, float* p, float* conf,
                             int32_t* verdict_arg, uint8_t* defer, int32_t* tokens, float* final_logits,
                             void* stream) {
  if (!m || !cand_offsets || !verdict_ids || !p || !conf || !verdict_arg || !defer)
    return fail(GF_EINVAL, "null argument");
  if (B < 1 || B > m->B_max) return fail(GF_EINVAL, "batch %d outside 1..%d", B, m->B_max);
  if (K < 1 || K > 8) return fail(GF_EINVAL, "K = %d outside 1..8", K);
  if (!(tau >= 0.f && tau <= 1.f)) return fail(GF_EINVAL, "tau outside [0, 1]");
  if (n_decode < 0 || prefix_len < 0) return fail(GF_EINVAL, "negative length");
  if (prefix_len > 0 && !prefix_ids) return fail(GF_EINVAL, "null prefix ids");
  for (int k = 0; k < K; ++k)
    if (verdict_ids[k] < 0 || verdict_ids[k] >= m->vocab) return fail(GF_EINVAL, "verdict id %d >= vocab", verdict_ids[k]);
  if (cand_offsets[0] != 0) return fail(GF_EINVAL, "offsets must start at 0");
  // full 64-token pages of the prefix are computed once and shared; its tail is part of every prompt
  const int past = prefix_len / 64 * 64, tail = prefix_len - past;
  std::vector<int32_t> poff(B + 1, 0);
  for (int b = 0; b < B; ++b) {
    const int nc = cand_offsets[b + 1] - cand_offsets[b];
    if (nc < 0 || tail + nc < 1) return fail(GF_EINVAL, "item %d: no tokens after the shared pages", b);
    if (nc > 0 && !cand_ids) return fail(GF_EINVAL, "null ids");
    poff[b + 1] = poff[b] + tail + nc;
  }
  if (poff[B] > m->T_max || past > m->T_max) return fail(GF_ECAPACITY, "prompt tokens exceed max_prefill_tokens");
  if (past > 0 && m->free_slots.size() < (size_t)B + 1) return fail(GF_ECAPACITY, "no free sequence slots");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int32_t hp = -1;
  if (past > 0) {
    const int32_t poff1[2] = {0, past};
    TRY(prefill_impl(m, 1, prefix_ids, poff1, 0, &hp, nullptr, nullptr, s, nullptr, 0, 0, -1, false));
  }
  std::vector<int32_t> desc;
  desc.insert(desc.end(), cand_offsets, cand_offsets + B + 1);
  desc.insert(desc.end(), poff.begin(), poff.end());
  int rc = upload(m->staging, m->fcall, desc.data(), desc.size() * sizeof(int32_t), s);
  if (rc == GF_OK &&
      gf::launch_build_prompts(prefix_ids + past, nullptr, cand_ids, m->fcall, m->fcall + B + 1, B, poff[B],
                               m->prompt_ids, s, tail) != cudaSuccess)
    rc = fail(GF_ECUDA, "prompt assembly launch failed");
  m->launches++;
  std::vector<int32_t> h(B);
  float* lg = (n_decode == 0 && final_logits) ? final_logits : m->logits;
  if (rc == GF_OK)
    rc = prefill_impl(m, B, m->prompt_ids, poff.data(), n_decode, h.data(), lg, m->next, s, m->tok_hist,
                      m->tok_stride, past, hp, true);
  if (hp >= 0) release_slot(m, hp);  // the shared pages stay referenced by the candidates
  TRY(rc);
  return decode_verdict_release(m, B, h, n_decode, verdict_ids, K, tau, p, conf, verdict_arg, defer, tokens,
                                final_logits, lg, s);
}

int gf_forecast_batch_host(gf_model* m, int32_t B, const int32_t* inc_ids, const int32_t* inc_offsets,
                           const int32_t* cand_ids, const int32_t* cand_offsets, int32_t n_decode,
                           const int32_t* verdict_ids, int32_t K, float tau, float* p, float* conf,
                           int32_t* verdict_arg, uint8_t* defer, int32_t* tokens, void* stream) {
  if (!m || !inc_offsets || !cand_offsets || !p || !conf || !verdict_arg || !defer)
    return fail(GF_EINVAL, "null argument");
  if (B < 1 || B > m->B_max) return fail(GF_EINVAL, "batch %d outside 1..%d", B, m->B_max);
  if (K < 1 || K > 8) return fail(GF_EINVAL, "K = %d outside 1..8", K);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int64_t ni = inc_offsets[B], nc = cand_offsets[B];
  if (ni < 0 || nc < 0 || ni + nc > m->T_max) return fail(GF_ECAPACITY, "ids exceed max_prefill_tokens");
  TRY(upload(m->staging, m->in_ids, inc_ids, (size_t)ni * sizeof(int32_t), s));
  TRY(upload(m->staging, m->in_ids + ni, cand_ids, (size_t)nc * sizeof(int32_t), s));
  // outputs on the device: p [B*K] | conf [B] | arg [B] | defer [B]  (within out_small, B_max*12 floats)
  float* dp = m->out_small;
  float* dconf = dp + (size_t)B * 8;
  int32_t* darg = reinterpret_cast<int32_t*>(dconf + B);
  uint8_t* ddef = reinterpret_cast<uint8_t*>(darg + B);
  // the generated tokens are staged on the device right after the prompt ids
  int32_t* dtok = nullptr;
  if (tokens && n_decode > 0) {
    if (ni + nc + (int64_t)B * n_decode > m->T_max) return fail(GF_ECAPACITY, "tokens output exceeds staging");
    dtok = m->in_ids + ni + nc;
  }
  TRY(gf_forecast_batch(m, B, m->in_ids, inc_offsets, m->in_ids + ni, cand_offsets, n_decode, verdict_ids, K, tau,
                        dp, dconf, darg, ddef, dtok, nullptr, stream));
  const size_t bytes = (size_t)B * 12 * sizeof(float) + (dtok ? (size_t)B * n_decode * sizeof(int32_t) : 0);
  if (m->host_out_cap < bytes) {
    if (m->host_out) cudaFreeHost(m->host_out);
    m->host_out = nullptr;
    m->host_out_cap = 0;
    if (cudaHostAlloc(&m->host_out, bytes, cudaHostAllocDefault) != cudaSuccess) return fail(GF_ENOMEM, "pinned out");
    m->host_out_cap = bytes;
  }
  char* ho = reinterpret_cast<char*>(m->host_out);
  CU(cudaMemcpyAsync(ho, m->out_small, (size_t)B * 12 * sizeof(float), cudaMemcpyDeviceToHost, s));
  if (dtok)
    CU(cudaMemcpyAsync(ho + (size_t)B * 12 * sizeof(float), dtok, (size_t)B * n_decode * sizeof(int32_t),
                       cudaMemcpyDeviceToHost, s));
  CU(cudaStreamSynchronize(s));
  const float* hp = reinterpret_cast<const float*>(ho);
  memcpy(p, hp, (size_t)B * K * sizeof(float));
  memcpy(conf, hp + (size_t)B * 8, (size_t)B * sizeof(float));
  memcpy(verdict_arg, hp + (size_t)B * 9, (size_t)B * sizeof(int32_t));
  memcpy(defer, hp + (size_t)B * 10, (size_t)B);
  if (dtok) memcpy(tokens, ho + (size_t)B * 12 * sizeof(float), (size_t)B * n_decode * sizeof(int32_t));
  return GF_OK;
}

// Timeout word of the building blocks (gf_gemm_bf16, gf_decode_attention, gf_selftest_timeout): one
// per device and CUDA context, allocated the first time a building block runs there.
namespace {
struct ErrWord {
  uint64_t ctx = 0;
  int* ptr = nullptr;
};
std::mutex g_err_mu;
ErrWord g_err_words[64];

// *out = the current device's word (nullptr when `create` is false and none exists yet); GF_OK or
// the reason it cannot be had.
int block_err_word(bool create, int** out) {
  *out = nullptr;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return fail(GF_ECUDA, "no CUDA device");
  }
  if (dev < 0 || dev >= 64) return fail(GF_ENOTIMPL, "device ordinal %d: the building blocks serve devices 0..63", dev);
  const uint64_t ctx = gf::current_context_id();
  std::lock_guard<std::mutex> lock(g_err_mu);
  ErrWord& w = g_err_words[dev];
  if (w.ptr && w.ctx == ctx) {
    *out = w.ptr;
    return GF_OK;
  }
  if (!create) return GF_OK;
  // a word of an earlier context of this device went away with that context (cudaDeviceReset)
  w.ptr = nullptr;
  int* p = nullptr;
  if (cudaMalloc(&p, sizeof(int)) != cudaSuccess || cudaMemset(p, 0, sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    if (p) cudaFree(p);
    return fail(GF_ENOMEM, "error word allocation failed");
  }
  w.ptr = p;
  w.ctx = ctx;
  *out = p;
  return GF_OK;
}
}  // namespace

int gf_gemm_bf16(const void* A, const void* W, int32_t M, int32_t N, int32_t K, void* out, int64_t ldo,
                 int32_t mode, int32_t bn, int32_t splits, int32_t group_m, void* stream) {
  if (!A || !W || !out || M < 0 || N < 1 || K < 64) return fail(GF_EINVAL, "bad GEMM arguments");
  if (K % 64 || N % 32) return fail(GF_EINVAL, "GEMM needs K %% 64 == 0 and N %% 32 == 0");
  if (mode < GF_GEMM_STORE_F32 || mode > GF_GEMM_SWIGLU) return fail(GF_EINVAL, "bad GEMM mode");
  if (mode == GF_GEMM_SWIGLU && N % 32) return fail(GF_EINVAL, "SwiGLU GEMM needs N %% 32 == 0");
  if (bn != 0 && bn != 64 && bn != 128 && bn != 256) return fail(GF_EINVAL, "bn must be 0, 64, 128 or 256");
  if (splits > 1 && mode != GF_GEMM_ATOMIC_F32) return fail(GF_EINVAL, "split-K needs the atomic mode");
  if (ldo < (mode == GF_GEMM_SWIGLU ? N / 2 : N)) return fail(GF_EINVAL, "ldo too small");
  if (M == 0) return GF_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int* err = nullptr;
  TRY(block_err_word(true, &err));
  int dev = 0, sms = 0;
  CU(cudaGetDevice(&dev));
  CU(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  int pbn, psplits;
  bool swap = false;
  plan_gemm(sms, M, N, K, mode, &pbn, &psplits, &swap);
  const bool bn_given = bn != 0;
  if (bn_given) swap = false;  // an explicit tile width asks for the non-swapped tiling
  if (!bn_given) bn = pbn;
  if (splits <= 0) splits = bn_given ? 1 : psplits;
  CUtensorMap ta, tb;
  if (swap) {
    TRY(make_map(&ta, W, (uint64_t)K, (uint64_t)N, (uint64_t)K * 2, 64, 128));
    TRY(make_map(&tb, A, (uint64_t)K, (uint64_t)M, (uint64_t)K * 2, 64, (uint32_t)bn));
    CU(gf::launch_gemm(ta, tb, N, M, K, out, ldo, mode, bn, splits, sms, err, s, group_m, true));
  } else {
    TRY(make_map(&ta, A, (uint64_t)K, (uint64_t)M, (uint64_t)K * 2, 64, 128));
    TRY(make_map(&tb, W, (uint64_t)K, (uint64_t)N, (uint64_t)K * 2, 64, (uint32_t)bn));
    CU(gf::launch_gemm(ta, tb, M, N, K, out, ldo, mode, bn, splits, sms, err, s, group_m));
  }
  return GF_OK;
}

static_assert(GF_GEMM_STORE_F32 == gf::kStoreF32 && GF_GEMM_ADD_F32 == gf::kAddF32 &&
                  GF_GEMM_ATOMIC_F32 == gf::kAtomicF32 && GF_GEMM_STORE_BF16 == gf::kStoreBF16 &&
                  GF_GEMM_SWIGLU == gf::kSwiGLU,
              "public GEMM modes are the kernel's modes");

int gf_plan_gemm(int32_t sms, int32_t M, int32_t N, int32_t K, int32_t mode, int32_t* bn, int32_t* splits,
                 int32_t* swap) {
  if (!bn || !splits || !swap) return fail(GF_EINVAL, "null output pointer");
  if (sms < 1 || M < 1 || N < 1 || K < 1) return fail(GF_EINVAL, "sizes must be positive");
  if (mode < GF_GEMM_STORE_F32 || mode > GF_GEMM_SWIGLU) return fail(GF_EINVAL, "bad GEMM mode");
  int b = 0, sp = 1;
  bool sw = false;
  plan_gemm(sms, M, N, K, mode, &b, &sp, &sw);
  *bn = b;
  *splits = sp;
  *swap = sw ? 1 : 0;
  return GF_OK;
}

int32_t gf_plan_decode_chunk(int32_t B, int32_t n_kv, int32_t max_ctx, int32_t sms) {
  if (B < 1 || n_kv < 1 || max_ctx < 1 || sms < 1) return fail(GF_EINVAL, "sizes must be positive");
  return decode_chunk(B, n_kv, max_ctx, sms);
}

int gf_gemm_status(void* stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  CU(cudaStreamSynchronize(s));
  int* err = nullptr;  // shared by gf_gemm_bf16, gf_decode_attention and gf_selftest_timeout
  TRY(block_err_word(false, &err));
  if (!err) return GF_OK;  // no building block has run in this context
  int h = 0;
  CU(cudaMemcpyAsync(&h, err, sizeof(int), cudaMemcpyDeviceToHost, s));
  CU(cudaMemsetAsync(err, 0, sizeof(int), s));
  CU(cudaStreamSynchronize(s));
  if (h == gf::kErrTimeout) return fail(GF_ETIMEOUT, "a device-side wait timed out");
  return GF_OK;
}

size_t gf_decode_attention_workspace(int32_t B, int32_t n_kv, int32_t head_dim, int32_t max_ctx) {
  if (B < 1 || n_kv < 1 || head_dim < 1 || max_ctx < 1) return 0;
  const size_t splits = (size_t)(max_ctx + 255) / 256;
  return (size_t)B * n_kv * splits * 16 * ((size_t)head_dim + 2) * sizeof(float);
}

int gf_decode_attention(const void* q, const void* k_cache, const void* v_cache, int64_t num_pages,
                        const int32_t* block_table, int32_t max_pages, const int32_t* ctx_len, int32_t max_ctx,
                        int32_t B, int32_t n_q, int32_t n_kv, int32_t head_dim, void* out, void* workspace,
                        size_t workspace_bytes, void* stream) {
  if (!q || !k_cache || !v_cache || !block_table || !ctx_len || !out || !workspace)
    return fail(GF_EINVAL, "null argument");
  if (B < 1 || n_q < 1 || n_kv < 1 || n_q % n_kv || n_q / n_kv > 16) return fail(GF_EINVAL, "bad head counts");
  if (head_dim != 64 && head_dim != 128) return fail(GF_ENOTIMPL, "head_dim must be 64 or 128");
  if (max_ctx < 1 || max_pages < 1 || max_ctx > max_pages * 64) return fail(GF_EINVAL, "max_ctx outside 1..64*max_pages");
  if (num_pages < 1 || num_pages * n_kv * 64 >= ((int64_t)1 << 31)) return fail(GF_EINVAL, "bad page count");
  if (workspace_bytes < gf_decode_attention_workspace(B, n_kv, head_dim, max_ctx))
    return fail(GF_EINVAL, "workspace smaller than gf_decode_attention_workspace()");
  int* err = nullptr;
  TRY(block_err_word(true, &err));
  CUtensorMap tk, tv;
  const uint64_t rows = (uint64_t)num_pages * n_kv * 64;
  TRY(make_map(&tk, k_cache, head_dim, rows, head_dim * 2, 64, 64));
  TRY(make_map(&tv, v_cache, 64, (uint64_t)num_pages * n_kv * head_dim, 128, 64, head_dim));
  gf::DecodeAttnArgs da{};
  da.q = reinterpret_cast<const bf16*>(q);
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
  int sms = 0, dev = 0;
  CU(cudaGetDevice(&dev));
  CU(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  da.chunk = decode_chunk(B, n_kv, max_ctx, sms);
  da.max_splits = (max_ctx + da.chunk - 1) / da.chunk;
  da.part_o = reinterpret_cast<float*>(workspace);
  da.part_ml = da.part_o + (size_t)B * n_kv * da.max_splits * 16 * head_dim;
  da.out = reinterpret_cast<bf16*>(out);
  da.ldo = (int64_t)n_q * head_dim;
  da.scale_log2 = 1.4426950408889634f / sqrtf((float)head_dim);
  da.err = err;
  CU(gf::launch_attn_decode(head_dim, tk, tv, da, B, reinterpret_cast<cudaStream_t>(stream)));
  return GF_OK;
}

int gf_select(int32_t B, const float* p, const float* m_bins, float x_cut, float tau_disc, float* s_hat,
              int32_t* order, float* disc, uint8_t* disc_pred, void* stream) {
  if (!p || !m_bins || !s_hat || !order || !disc || !disc_pred) return fail(GF_EINVAL, "null argument");
  if (B < 1 || B > 1024) return fail(GF_EINVAL, "batch %d outside 1..1024", B);
  if (!(tau_disc >= 0.f && tau_disc <= 1.f)) return fail(GF_EINVAL, "tau outside [0, 1]");
  CU(gf::launch_select(B, p, m_bins, x_cut, tau_disc, s_hat, order, disc, disc_pred,
                       reinterpret_cast<cudaStream_t>(stream)));
  return GF_OK;
}

int gf_selftest_timeout(uint32_t limit_ms, void* stream) {
  if (limit_ms < 1 || limit_ms > 2000) return fail(GF_EINVAL, "limit_ms outside 1..2000");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int* err = nullptr;
  TRY(block_err_word(true, &err));
  CU(gf::launch_timeout_probe((uint64_t)limit_ms * 1000000ull, err, s));
  return gf_gemm_status(stream);
}

int gf_profile_enable(gf_model* m, uint32_t mask) {
  if (!m) return fail(GF_EINVAL, "null model");
  m->prof_mask = mask;
  return GF_OK;
}

int gf_profile_read(gf_model* m, int32_t kind, int64_t* launches, double* ms, double* flops, double* bytes) {
  if (!m || kind < 0 || kind >= GF_PROF_KINDS) return fail(GF_EINVAL, "bad profile request");
  CU(cudaDeviceSynchronize());
  int64_t n = 0;
  double t = 0, f = 0, by = 0;
  std::vector<gf_model::ProfRec> keep;
  for (auto& r : m->prof) {
    if (r.kind != kind) {
      keep.push_back(r);
      continue;
    }
    float e = 0.f;
    CU(cudaEventElapsedTime(&e, r.a, r.b));
    ++n;
    t += e;
    f += r.flops;
    by += r.bytes;
    m->ev_pool.push_back(r.a);
    m->ev_pool.push_back(r.b);
  }
  m->prof.swap(keep);
  if (launches) *launches = n;
  if (ms) *ms = t;
  if (flops) *flops = f;
  if (bytes) *bytes = by;
  return GF_OK;
}

int gf_debug_capture(gf_model* m, int32_t layer, int32_t item, float* dst, int64_t cap_rows) {
  if (!m || !dst || layer < 0 || layer > m->L || item < 0 || item >= m->B_max || cap_rows < 1)
    return fail(GF_EINVAL, "bad capture request");
  if (m->caps.size() >= 8) return fail(GF_ECAPACITY, "too many captures armed");
  m->caps.push_back({layer, item, dst, cap_rows});
  return GF_OK;
}

int gf_debug_read_kv(gf_model* m, int32_t layer, int32_t handle, int32_t start, int32_t n, void* k_dst,
                     void* v_dst, void* stream) {
  if (!m || !k_dst || !v_dst || layer < 0 || layer >= m->L || handle < 0 || handle >= m->B_max ||
      !m->live[handle] || start < 0 || n < 0 || start + n > m->h_len[handle])
    return fail(GF_EINVAL, "bad KV read request");
  CU(gf::launch_read_kv(m->k_cache, m->v_cache, m->bt, m->max_pages, handle, start, n, m->nkv, m->hd,
                        layer_row0(m, layer), reinterpret_cast<bf16*>(k_dst), reinterpret_cast<bf16*>(v_dst),
                        reinterpret_cast<cudaStream_t>(stream)));
  return GF_OK;
}

int gf_device_status(gf_model* m, void* stream) {
  if (!m) return fail(GF_EINVAL, "null model");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  CU(cudaStreamSynchronize(s));
  int h = 0;
  CU(cudaMemcpy(&h, m->err, sizeof(int), cudaMemcpyDeviceToHost));
  CU(cudaMemset(m->err, 0, sizeof(int)));
  if (h != 0) {
    // a kernel that gave up may have left split-K sums behind
    CU(cudaMemset(m->dqkv, 0, (size_t)m->B_max * m->qkv_dim * sizeof(float)));
  }
  if (h == gf::kErrTimeout) return fail(GF_ETIMEOUT, "a device-side wait timed out");
  if (h == 1) return fail(GF_EINVAL, "a token id outside [0, vocab) reached the device");
  if (h != 0) return fail(GF_ECUDA, "device error word %d", h);
  return GF_OK;
}

}  // extern "C"
