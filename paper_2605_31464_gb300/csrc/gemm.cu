// Host launchers for the tcgen05 GEMM (one template instantiation per tile
// width and epilogue).
#include "gemm_tc.cuh"
#include "kernels.h"

namespace gf {

int gemm_num_stages(int bn) {
  return bn == 256 ? GemmCfg<256>::STAGES : (bn == 128 ? GemmCfg<128>::STAGES : GemmCfg<64>::STAGES);
}
int gemm_smem_bytes(int bn) {
  return bn == 256 ? GemmCfg<256>::SMEM_BYTES : (bn == 128 ? GemmCfg<128>::SMEM_BYTES : GemmCfg<64>::SMEM_BYTES);
}

template <int BN, int MODE, bool SWAP>
static cudaError_t launch_one(const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmArgs& p, int grid,
                              cudaStream_t s) {
  // the shared-memory limit is an attribute of the function in one device's context: set it once per context
  static DeviceOnce configured;
  auto kern = gemm_tc_kernel<BN, MODE, SWAP>;
  const cudaError_t e = configured.run([&] {
    return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, GemmCfg<BN, SWAP>::SMEM_BYTES);
  });
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(grid), dim3(GemmCfg<BN, SWAP>::THREADS), GemmCfg<BN, SWAP>::SMEM_BYTES, s, tmA, tmB,
                    p);
}

template <int BN>
static cudaError_t dispatch_mode(const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmArgs& p, int mode,
                                 int grid, cudaStream_t s) {
  switch (mode) {
    case kStoreF32: return launch_one<BN, kStoreF32, false>(tmA, tmB, p, grid, s);
    case kAddF32: return launch_one<BN, kAddF32, false>(tmA, tmB, p, grid, s);
    case kAtomicF32: return launch_one<BN, kAtomicF32, false>(tmA, tmB, p, grid, s);
    case kStoreBF16: return launch_one<BN, kStoreBF16, false>(tmA, tmB, p, grid, s);
    case kSwiGLU: return launch_one<BN, kSwiGLU, false>(tmA, tmB, p, grid, s);
    case kRopeQKV:
      if constexpr (BN >= 128) return launch_one<BN, kRopeQKV, false>(tmA, tmB, p, grid, s);
      return cudaErrorInvalidValue;
    default: return cudaErrorInvalidValue;
  }
}

template <int BN>
static cudaError_t dispatch_swap(const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmArgs& p, int mode,
                                 int grid, cudaStream_t s) {
  switch (mode) {
    case kStoreF32: return launch_one<BN, kStoreF32, true>(tmA, tmB, p, grid, s);
    case kAtomicF32: return launch_one<BN, kAtomicF32, true>(tmA, tmB, p, grid, s);
    case kSwiGLU: return launch_one<BN, kSwiGLU, true>(tmA, tmB, p, grid, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_gemm(const CUtensorMap& tmA, const CUtensorMap& tmB, int M, int N, int K, void* out,
                        int64_t ldo, int mode, int bn, int splits, int grid, int* err, cudaStream_t s, int group_m,
                        bool swap, unsigned long long* argmax_keys, const SampleParams* sample,
                        const int32_t* sample_step, int sample_step_bias, const RopeEpilogue* rope,
                        const NormFold* norm, bool w_blocked) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  if (K % 64 != 0) return cudaErrorInvalidValue;
  if (!swap && N % 32 != 0) return cudaErrorInvalidValue;
  if (swap && (M % 32 != 0 || N > bn)) return cudaErrorInvalidValue;
  if (mode == kRopeQKV && (swap || !rope || bn < 128 || N % 128 != 0 || splits > 1)) return cudaErrorInvalidValue;
  GemmArgs p;
  p.M = M;
  p.N = N;
  p.K = K;
  p.num_m = (M + 127) / 128;
  p.num_n = (N + bn - 1) / bn;
  p.kb_total = K / 64;
  if (splits < 1) splits = 1;
  if (splits > p.kb_total) splits = p.kb_total;
  p.kb_per_split = (p.kb_total + splits - 1) / splits;
  p.splits = (p.kb_total + p.kb_per_split - 1) / p.kb_per_split;  // no empty split
  if (group_m <= 0) {
    // Concurrent CTAs walk a group of M-blocks across all N-blocks: the group's A tiles stay in L2
    // while every weight tile is streamed once per group.  Larger groups mean fewer weight re-reads
    // but crowd L2; about 28 MiB of A per group measured best (K = 3584: 32 M-blocks, 6 % faster
    // than 54 for the 7B gate/up GEMM; flat for K = 18944).
    const double a_tile = 128.0 * K * 2;
    group_m = (int)(28.0 * 1024 * 1024 / a_tile);
    group_m = group_m < 4 ? 4 : (group_m > 128 ? 128 : group_m);
  }
  p.group_m = group_m;
  p.out = out;
  p.ldo = ldo;
  p.err = err;
  p.argmax_keys = (swap && mode == kStoreF32) ? argmax_keys : nullptr;
  p.sample = p.argmax_keys ? sample : nullptr;
  p.sample_step = sample_step;
  p.sample_step_bias = sample_step_bias;
  if (rope) p.rope = *rope;
  p.norm_out = nullptr;
  p.norm_gain = nullptr;
  p.norm_ss = nullptr;
  p.ld_norm = 0;
  p.row_ss = nullptr;
  p.inv_d = 0.f;
  p.eps = 0.f;
  p.w_blocked = w_blocked ? 1 : 0;
  if (norm && !swap) {
    p.norm_out = norm->out;
    p.norm_gain = norm->gain;
    p.norm_ss = norm->ss_out;
    p.ld_norm = norm->ld_out;
    p.row_ss = norm->ss_in;
    p.inv_d = norm->inv_d;
    p.eps = norm->eps;
  }
  const int tiles = p.num_m * p.num_n * p.splits;
  if (grid > tiles) grid = tiles;
  if (grid < 1) grid = 1;
  if (swap) {
    switch (bn) {
      case 32: return dispatch_swap<32>(tmA, tmB, p, mode, grid, s);
      case 64: return dispatch_swap<64>(tmA, tmB, p, mode, grid, s);
      case 128: return dispatch_swap<128>(tmA, tmB, p, mode, grid, s);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (bn) {
    case 64: return dispatch_mode<64>(tmA, tmB, p, mode, grid, s);
    case 128: return dispatch_mode<128>(tmA, tmB, p, mode, grid, s);
    case 256: return dispatch_mode<256>(tmA, tmB, p, mode, grid, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace gf
