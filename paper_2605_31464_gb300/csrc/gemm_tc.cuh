// bf16 GEMM on the 5th-generation tensor cores:  C[M,N] (op)= A[M,K] . B[N,K]^T
//
// A (activations) and B (weights, rows = output features) are K-major bf16 in
// global memory, streamed by TMA into 128-byte-swizzled shared-memory stages.
// The weights are either row-major [N][K] or, with w_blocked, stored in blocks
// of 256 rows x 64 columns, [ceil(N/256)][K/64][256][64] (zero rows pad N), so
// that every weight box a stage loads (up to 256 rows of one 64-column slice)
// is one contiguous run of memory instead of rows K*2 bytes apart.
// One thread issues tcgen05.mma (M=128, N=BN, K=16 per instruction) into a
// double-buffered fp32 accumulator in tensor memory; four epilogue warps read
// it back with tcgen05.ld and apply the fused epilogue:
//   kStoreF32   C = acc                         (fp32)
//   kAddF32     C += acc                        (fp32 residual stream)
//   kAtomicF32  C += acc with atomics           (split-K partial sums)
//   kStoreBF16  C = bf16(acc)
//   kSwiGLU     B rows are interleaved in blocks of 16 (16 gate rows, then
//               the 16 matching up rows); the output is bf16(silu(gate) * up)
//               with N/2 columns.
//   kRopeQKV    prefill QKV projection: the columns are n_q query, n_kv key
//               and n_kv value heads of 128; query and key heads are rotated
//               (RoPE at each row's position) and, with the values, rounded
//               to bf16 and written straight to the rotated-query buffer and
//               the paged K / transposed-V cache (no fp32 QKV round trip).
// The kernel is persistent: gridDim.x CTAs walk the tile list (grouped along
// M so that concurrently running CTAs share A and B tiles in L2).
//
// SWAP (decode, few activation rows): the weights are the 128-row A operand
// and the activations the narrow B operand (N = BN >= batch rows), so each
// pipeline stage carries mostly weight bytes; the epilogue writes the
// transposed tile, out[b][n].  With the 16-row gate/up interleave a gate row
// and its up row sit 16 TMEM lanes apart in the same warp.
#pragma once

#include "ptx.cuh"
#include "sampling.cuh"

namespace gf {

enum GemmMode { kStoreF32 = 0, kAddF32 = 1, kAtomicF32 = 2, kStoreBF16 = 3, kSwiGLU = 4, kRopeQKV = 5 };

// Destination of the kRopeQKV epilogue (head_dim 128).  Row t of the GEMM is token t of the
// packed prompts, at sequence slot row_map[t].x and position row_map[t].y.
struct RopeEpilogue {
  const int2* row_map;
  const float2* rope_cs;        // [position][64] (cos, sin) of position * theta^(-2i/128)
  __nv_bfloat16* q_out;         // [T][n_q * 128]
  int64_t ldq;
  __nv_bfloat16* k_cache;       // rows of 128: [layer][page][n_kv][64 tokens]
  __nv_bfloat16* v_cache;       // transposed pages: [layer][page][n_kv][128][64 tokens]
  const int32_t* block_table;   // [slot][max_pages]
  int max_pages, n_q, n_kv;
  int64_t layer_row0;           // first K-cache row of this layer
};

struct GemmArgs {
  int M, N, K;
  int num_m, num_n, splits;
  int kb_total, kb_per_split;
  int group_m;
  void* out;
  int64_t ldo;  // elements
  int* err;
  // SWAP + kStoreF32 only: per output row b, atomicMax of argmax_key(value, column) over the tile
  // (the greedy arg max of a logits row; the lowest column wins ties)
  unsigned long long* argmax_keys;
  // with argmax_keys: when `sample` is set, the key is taken over the perturbed score
  // l * (1/T) + G (Gumbel-max draw, sampling.cuh) of token t = *sample_step + sample_step_bias
  // (t = sample_step_bias when sample_step is null); output column b is sampled row b
  const SampleParams* sample;
  const int32_t* sample_step;
  int sample_step_bias;
  RopeEpilogue rope;  // kRopeQKV only
  // RMSNorm folded into the prefill GEMMs around it (non-swapped tiles only):
  //  kAddF32 with norm_out: after the residual update also write norm_out = bf16(x_new * norm_gain[col])
  //    and add the row's sum of x_new^2 over the tile's columns into norm_ss[row] (atomically);
  //  kSwiGLU / kRopeQKV with row_ss: the accumulator row is scaled by rsqrt(row_ss[row] * inv_d + eps)
  //    before the epilogue's arithmetic, so that A = bf16(x * gain) yields RMSNorm(x) * gain . W.
  __nv_bfloat16* norm_out;
  const float* norm_gain;
  float* norm_ss;
  int64_t ld_norm;
  const float* row_ss;
  float inv_d, eps;
  int w_blocked;  // weights in 256 x 64 blocks (see the top of this file)
};

template <int BN, bool SWAP = false>
struct GemmCfg {
  static constexpr int BM = 128;
  static constexpr int BK = 64;
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  // non-swapped tiles keep 18 KB for the epilogue's staging tiles (4 warps x [32 rows][36 floats])
  static constexpr int EPI_BYTES = SWAP ? 0 : 4 * 32 * 36 * 4;
  static constexpr int STAGES_FIT = ((SWAP ? 220 : 200) * 1024) / STAGE_BYTES;
  static constexpr int STAGES = STAGES_FIT > 12 ? 12 : STAGES_FIT;
  static constexpr uint32_t TMEM_COLS = 2 * BN < 32 ? 32 : 2 * BN;  // two accumulator buffers
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 /*align*/ + 256 /*barriers*/ + EPI_BYTES;
  static constexpr int THREADS = 192;
};

// TMA coordinates of the weight box for k-block kb at weight row row0 (a multiple of the box
// height, which divides 256).  Blocked weights are addressed as a 2D map of 64-element rows:
// block (row0 / 256, kb) starts at row (row0 / 256 * kb_total + kb) * 256.
__device__ __forceinline__ void weight_coords(const GemmArgs& p, int kb, int row0, int& x, int& y) {
  if (p.w_blocked) {
    x = 0;
    y = ((row0 >> 8) * p.kb_total + kb) * 256 + (row0 & 255);
  } else {
    x = kb * 64;
    y = row0;
  }
}

__device__ __forceinline__ void gemm_tile_coords(const GemmArgs& p, int tile, int& m_blk, int& n_blk, int& split) {
  split = tile % p.splits;
  const int t = tile / p.splits;
  const int group_size = p.group_m * p.num_n;
  const int g = t / group_size;
  const int first_m = g * p.group_m;
  const int gm = min(p.num_m - first_m, p.group_m);
  const int in = t % group_size;
  m_blk = first_m + in % gm;
  n_blk = in / gm;
}

template <int MODE>
__device__ __forceinline__ void gemm_epilogue_chunk(const GemmArgs& p, int row, int col, const uint32_t (&r)[32]) {
  if (MODE == kStoreF32) {
    float4* dst = reinterpret_cast<float4*>(reinterpret_cast<float*>(p.out) + (int64_t)row * p.ldo + col);
#pragma unroll
    for (int i = 0; i < 8; ++i)
      dst[i] = make_float4(__uint_as_float(r[4 * i]), __uint_as_float(r[4 * i + 1]), __uint_as_float(r[4 * i + 2]),
                           __uint_as_float(r[4 * i + 3]));
  } else if (MODE == kAddF32) {
    float4* dst = reinterpret_cast<float4*>(reinterpret_cast<float*>(p.out) + (int64_t)row * p.ldo + col);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float4 o = dst[i];
      o.x += __uint_as_float(r[4 * i]);
      o.y += __uint_as_float(r[4 * i + 1]);
      o.z += __uint_as_float(r[4 * i + 2]);
      o.w += __uint_as_float(r[4 * i + 3]);
      dst[i] = o;
    }
  } else if (MODE == kAtomicF32) {
    float4* dst = reinterpret_cast<float4*>(reinterpret_cast<float*>(p.out) + (int64_t)row * p.ldo + col);
#pragma unroll
    for (int i = 0; i < 8; ++i)
      atomicAdd(dst + i, make_float4(__uint_as_float(r[4 * i]), __uint_as_float(r[4 * i + 1]),
                                     __uint_as_float(r[4 * i + 2]), __uint_as_float(r[4 * i + 3])));
  } else if (MODE == kStoreBF16) {
    uint4* dst = reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(p.out) + (int64_t)row * p.ldo + col);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      uint4 v;
      v.x = pack_bf16(__uint_as_float(r[8 * i + 0]), __uint_as_float(r[8 * i + 1]));
      v.y = pack_bf16(__uint_as_float(r[8 * i + 2]), __uint_as_float(r[8 * i + 3]));
      v.z = pack_bf16(__uint_as_float(r[8 * i + 4]), __uint_as_float(r[8 * i + 5]));
      v.w = pack_bf16(__uint_as_float(r[8 * i + 6]), __uint_as_float(r[8 * i + 7]));
      dst[i] = v;
    }
  }
}

template <int BN, int MODE, bool SWAP = false>
__global__ void __launch_bounds__(192, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const GemmArgs p) {
  using C = GemmCfg<BN, SWAP>;
  constexpr uint32_t IDESC = idesc_bf16_f32(C::BM, BN);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + C::STAGES * C::B_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* acc_full = empty + C::STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* mma_done = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  float* epi_smem = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(full) + 256);  // [4][32][36] (non-swapped)

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], 128);
    }
    mbar_init(mma_done, 1);
    fence_mbar_init();
    fence_async_smem();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int num_tiles = p.num_m * p.num_n * p.splits;

  pdl_trigger();
  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    if (lane == 0) {
      // The weights (A when SWAP, else B) are never written by an earlier kernel: the weight
      // halves of the first stages are requested before waiting for the previous kernel.
      int pre = 0;
      for (int tile = blockIdx.x; tile < num_tiles && pre < C::STAGES; tile += gridDim.x) {
        int m_blk, n_blk, split;
        gemm_tile_coords(p, tile, m_blk, n_blk, split);
        const int kb0 = split * p.kb_per_split;
        const int kb1 = min(kb0 + p.kb_per_split, p.kb_total);
        for (int kb = kb0; kb < kb1 && pre < C::STAGES; ++kb, ++pre) {
          mbar_arrive_expect_tx(&full[pre], C::STAGE_BYTES);
          int wx, wy;
          weight_coords(p, kb, SWAP ? m_blk * C::BM : n_blk * BN, wx, wy);
          if (SWAP)
            tma_load_2d(sA + pre * C::A_BYTES, &tmA, &full[pre], wx, wy);
          else
            tma_load_2d(sB + pre * C::B_BYTES, &tmB, &full[pre], wx, wy);
        }
      }
      pdl_wait();
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        int m_blk, n_blk, split;
        gemm_tile_coords(p, tile, m_blk, n_blk, split);
        const int kb0 = split * p.kb_per_split;
        const int kb1 = min(kb0 + p.kb_per_split, p.kb_total);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (issued < pre) {
            // barrier armed and weight half requested above: add the activation half
            if (SWAP)
              tma_load_2d(sB + stage * C::B_BYTES, &tmB, &full[stage], kb * C::BK, n_blk * BN);
            else
              tma_load_2d(sA + stage * C::A_BYTES, &tmA, &full[stage], kb * C::BK, m_blk * C::BM);
          } else {
            if (!mbar_wait(&empty[stage], phase ^ 1u, p.err)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&full[stage], C::STAGE_BYTES);
            int wx, wy;
            weight_coords(p, kb, SWAP ? m_blk * C::BM : n_blk * BN, wx, wy);
            if (SWAP) {
              tma_load_2d(sA + stage * C::A_BYTES, &tmA, &full[stage], wx, wy);
              tma_load_2d(sB + stage * C::B_BYTES, &tmB, &full[stage], kb * C::BK, n_blk * BN);
            } else {
              tma_load_2d(sA + stage * C::A_BYTES, &tmA, &full[stage], kb * C::BK, m_blk * C::BM);
              tma_load_2d(sB + stage * C::B_BYTES, &tmB, &full[stage], wx, wy);
            }
          }
          ++issued;
          if (++stage == C::STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      // Every copy this thread started must have landed before the CTA exits.
      const int outstanding = min(max(issued, pre), C::STAGES);
      for (int i = 0; i < outstanding; ++i) {
        if (--stage < 0) {
          stage = C::STAGES - 1;
          phase ^= 1u;
        }
        mbar_wait_drain(&full[stage], phase);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      bool any = false;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        int m_blk, n_blk, split;
        gemm_tile_coords(p, tile, m_blk, n_blk, split);
        const int kb0 = split * p.kb_per_split;
        const int kb1 = min(kb0 + p.kb_per_split, p.kb_total);
        if (!mbar_wait(&acc_empty[acc], acc_phase ^ 1u, p.err)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&full[stage], phase, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + stage * C::A_BYTES);
          const uint32_t b0 = smem_u32(sB + stage * C::B_BYTES);
#pragma unroll
          for (int k = 0; k < C::BK / 16; ++k) {
            umma_bf16(d_tmem, sdesc_k_sw128(a0 + k * 32), sdesc_k_sw128(b0 + k * 32), IDESC,
                      (kb > kb0 || k > 0) ? 1u : 0u);
          }
          umma_commit(&empty[stage]);
          any = true;
          if (++stage == C::STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(&acc_full[acc]);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
      // All MMAs must be complete before tensor memory is released.
      if (any) {
        umma_commit(mma_done);
        mbar_wait_drain(mma_done, 0);
      }
    }
  } else {
    // ------------------------------------------------ epilogue (warps 2..5)
    pdl_wait();  // the epilogue writes (and may read) buffers of earlier kernels
    const int quarter = warp & 3;  // tensor-memory lanes this warp may read
    const int row_in_tile = quarter * 32 + lane;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
      int m_blk, n_blk, split;
      gemm_tile_coords(p, tile, m_blk, n_blk, split);
      if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[acc], acc_phase, p.err))) break;  // warp-uniform
      tc_fence_after();
      const int row = m_blk * C::BM + row_in_tile;
      const bool row_ok = row < p.M;
      const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * BN);
      if (SWAP) {
        // TMEM lane = weight row (output feature), column = activation row (batch)
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          uint32_t r[32];
          tmem_ld32(taddr + c, r);
          tmem_ld_wait();
          if (MODE == kSwiGLU) {
            // lanes 0..15 of each warp hold gate rows, lanes 16..31 the matching up rows
            const int f = m_blk * 64 + quarter * 16 + (lane & 15);
            const bool f_ok = (lane < 16) && (f < p.M / 2);
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float u = __shfl_down_sync(0xffffffffu, __uint_as_float(r[i]), 16);
              const int bb = c + i;
              if (f_ok && bb < p.N) {
                const float g = __uint_as_float(r[i]);
                reinterpret_cast<__nv_bfloat16*>(p.out)[(int64_t)bb * p.ldo + f] =
                    __float2bfloat16(g / (1.0f + __expf(-g)) * u);
              }
            }
          } else {
            float* out = reinterpret_cast<float*>(p.out);
            if (row_ok) {
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                const int bb = c + i;
                if (bb < p.N) {
                  if (MODE == kAtomicF32)
                    atomicAdd(out + (int64_t)bb * p.ldo + row, __uint_as_float(r[i]));
                  else
                    out[(int64_t)bb * p.ldo + row] = __uint_as_float(r[i]);
                }
              }
            }
            if (MODE == kStoreF32 && p.argmax_keys) {
              // transpose-reduce the warp's 32 rows x 32 columns: after five halvings lane l holds
              // the best key of column c + l over this warp's rows
              unsigned long long k[32];
              if (p.sample) {
                const SampleParams sp = *p.sample;
                const int t = (p.sample_step ? *p.sample_step : 0) + p.sample_step_bias;
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                  // one Philox block serves the four rows c + 4q .. c + 4q + 3 (r / 4 shared)
                  uint64_t w[4];
                  philox4x64_10((uint64_t)row, (uint64_t)t, (uint64_t)((c >> 2) + q), 0ull, sp.seed, 0ull, w);
#pragma unroll
                  for (int j = 0; j < 4; ++j) {
                    const float z = fmaf(__uint_as_float(r[4 * q + j]), sp.inv_temp, gumbel_from_word(w[j]));
                    k[4 * q + j] = row_ok ? argmax_key(z, row) : 0ull;
                  }
                }
              } else {
#pragma unroll
                for (int i = 0; i < 32; ++i) k[i] = row_ok ? argmax_key(__uint_as_float(r[i]), row) : 0ull;
              }
#pragma unroll
              for (int o = 16; o >= 1; o >>= 1) {
                const bool upper = (lane & o) != 0;
#pragma unroll
                for (int j = 0; j < o; ++j) {
                  const unsigned long long send = upper ? k[j] : k[j + o];
                  const unsigned long long keep = upper ? k[j + o] : k[j];
                  const unsigned long long got = __shfl_xor_sync(0xffffffffu, send, o);
                  k[j] = keep > got ? keep : got;
                }
              }
              const int bb = c + lane;
              if (bb < p.N && k[0] != 0ull) atomicMax(p.argmax_keys + bb, k[0]);
            }
          }
        }
      } else if (MODE == kRopeQKV) {
        // each 128-column block of the tile is one head; RoPE pairs columns i and i + 64
        const RopeEpilogue& e = p.rope;
        int2 rm = make_int2(0, 0);
        if (row_ok) rm = e.row_map[row];
        const int page = row_ok ? e.block_table[(int64_t)rm.x * e.max_pages + (rm.y >> 6)] : 0;
        const int in_page = rm.y & 63;
        const float4* cs4 = reinterpret_cast<const float4*>(e.rope_cs + (int64_t)rm.y * 64);
        const float rs = (p.row_ss && row_ok) ? rsqrtf(p.row_ss[row] * p.inv_d + p.eps) : 1.f;
#pragma unroll 1
        for (int hh = 0; hh < BN / 128; ++hh) {
          const int head = n_blk * (BN / 128) + hh;
          if (head * 128 >= p.N) break;  // uniform across the CTA
#pragma unroll 1
          for (int c = 0; c < 64; c += 32) {
            uint32_t lo[32], hi[32];
            tmem_ld32(taddr + hh * 128 + c, lo);
            tmem_ld32(taddr + hh * 128 + c + 64, hi);
            tmem_ld_wait();
            if (!row_ok) continue;
            if (rs != 1.f) {
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                lo[i] = __float_as_uint(__uint_as_float(lo[i]) * rs);
                hi[i] = __float_as_uint(__uint_as_float(hi[i]) * rs);
              }
            }
            if (head < e.n_q + e.n_kv) {
              uint32_t y0[16], y1[16];
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const float4 r = cs4[(c >> 1) + j];  // (cos, sin) of pairs c + 2j and c + 2j + 1
                const float a0 = __uint_as_float(lo[2 * j]), b0 = __uint_as_float(hi[2 * j]);
                const float a1 = __uint_as_float(lo[2 * j + 1]), b1 = __uint_as_float(hi[2 * j + 1]);
                y0[j] = pack_bf16(a0 * r.x - b0 * r.y, a1 * r.z - b1 * r.w);
                y1[j] = pack_bf16(b0 * r.x + a0 * r.y, b1 * r.z + a1 * r.w);
              }
              __nv_bfloat16* dst =
                  head < e.n_q ? e.q_out + (int64_t)row * e.ldq + head * 128
                               : e.k_cache + (e.layer_row0 + ((int64_t)page * e.n_kv + (head - e.n_q)) * 64 + in_page) * 128;
              uint4* d0 = reinterpret_cast<uint4*>(dst + c);
              uint4* d1 = reinterpret_cast<uint4*>(dst + c + 64);
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                d0[q] = make_uint4(y0[4 * q], y0[4 * q + 1], y0[4 * q + 2], y0[4 * q + 3]);
                d1[q] = make_uint4(y1[4 * q], y1[4 * q + 1], y1[4 * q + 2], y1[4 * q + 3]);
              }
            } else {
              // values: [hd][64 tokens] per page, so lanes (consecutive tokens) write adjacent elements
              const int g = head - e.n_q - e.n_kv;
              __nv_bfloat16* dst = e.v_cache + e.layer_row0 * 128 + ((int64_t)page * e.n_kv + g) * 128 * 64 + in_page;
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                dst[(int64_t)(c + i) * 64] = __float2bfloat16(__uint_as_float(lo[i]));
                dst[(int64_t)(c + 64 + i) * 64] = __float2bfloat16(__uint_as_float(hi[i]));
              }
            }
          }
        }
      } else if (MODE == kSwiGLU) {
        // each 32-column chunk holds 16 gate columns then the 16 matching up columns
        const float rs = (p.row_ss && row_ok) ? rsqrtf(p.row_ss[row] * p.inv_d + p.eps) : 1.f;
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          uint32_t r[32];
          tmem_ld32(taddr + c, r);
          tmem_ld_wait();
          const int col = n_blk * BN + c;
          if (row_ok && col < p.N) {
            uint32_t o[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float g0 = __uint_as_float(r[2 * j]) * rs, g1 = __uint_as_float(r[2 * j + 1]) * rs;
              const float u0 = __uint_as_float(r[16 + 2 * j]) * rs, u1 = __uint_as_float(r[16 + 2 * j + 1]) * rs;
              o[j] = pack_bf16(g0 / (1.0f + __expf(-g0)) * u0, g1 / (1.0f + __expf(-g1)) * u1);
            }
            uint4* dst = reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(p.out) + (int64_t)row * p.ldo +
                                                  col / 2);
            dst[0] = make_uint4(o[0], o[1], o[2], o[3]);
            dst[1] = make_uint4(o[4], o[5], o[6], o[7]);
          }
        }
      } else if (MODE == kAddF32) {
        // TMEM hands each thread one row (lane = row), so a warp's global accesses would each touch 32
        // rows.  Each warp stages its 32 rows x 32 columns through shared memory instead and lane l then
        // handles columns 4 (l % 8) .. + 3 of rows 4 k + l / 8 (k = 0..7): an access covers four whole
        // 128-byte row pieces.  Row sums of squares are reduced over the eight lanes of a row.
        float* stile = epi_smem + quarter * (32 * 36);
        const int sub = lane & 7, rq = lane >> 3;
        const int row0 = m_blk * C::BM + quarter * 32;
        const int ncols = min(BN, p.N - n_blk * BN);
        float* res_base = reinterpret_cast<float*>(p.out);
        float ss[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) ss[k] = 0.f;
#pragma unroll 1
        for (int c = 0; c < ncols; c += 32) {
          uint32_t r[32];
          tmem_ld32(taddr + c, r);
          tmem_ld_wait();
          float4* srow = reinterpret_cast<float4*>(stile + lane * 36);
#pragma unroll
          for (int i = 0; i < 8; ++i)
            srow[i] = make_float4(__uint_as_float(r[4 * i]), __uint_as_float(r[4 * i + 1]), __uint_as_float(r[4 * i + 2]),
                                  __uint_as_float(r[4 * i + 3]));
          __syncwarp();
          const int col = n_blk * BN + c + 4 * sub;
          float4 x[8];
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int row = row0 + 4 * k + rq;
            x[k] = row < p.M ? *reinterpret_cast<const float4*>(res_base + (int64_t)row * p.ldo + col)
                             : make_float4(0.f, 0.f, 0.f, 0.f);
          }
          float4 g = make_float4(0.f, 0.f, 0.f, 0.f);
          if (p.norm_out) g = *reinterpret_cast<const float4*>(p.norm_gain + col);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int row = row0 + 4 * k + rq;
            const float4 a = reinterpret_cast<const float4*>(stile + (4 * k + rq) * 36)[sub];
            x[k].x += a.x;
            x[k].y += a.y;
            x[k].z += a.z;
            x[k].w += a.w;
            if (row < p.M) {
              *reinterpret_cast<float4*>(res_base + (int64_t)row * p.ldo + col) = x[k];
              if (p.norm_out) {
                ss[k] += x[k].x * x[k].x + x[k].y * x[k].y + x[k].z * x[k].z + x[k].w * x[k].w;
                *reinterpret_cast<uint2*>(p.norm_out + (int64_t)row * p.ld_norm + col) =
                    make_uint2(pack_bf16(x[k].x * g.x, x[k].y * g.y), pack_bf16(x[k].z * g.z, x[k].w * g.w));
              }
            }
          }
          __syncwarp();  // the next chunk overwrites the staging tile
        }
        if (p.norm_out) {
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            float v = ss[k];
            v += __shfl_xor_sync(0xffffffffu, v, 1);
            v += __shfl_xor_sync(0xffffffffu, v, 2);
            v += __shfl_xor_sync(0xffffffffu, v, 4);
            const int row = row0 + 4 * k + rq;
            if (sub == 0 && row < p.M) atomicAdd(p.norm_ss + row, v);
          }
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          uint32_t r[32];
          tmem_ld32(taddr + c, r);
          tmem_ld_wait();
          const int col = n_blk * BN + c;
          if (row_ok && col < p.N) gemm_epilogue_chunk<MODE>(p, row, col, r);
        }
      }
      tc_fence_before();
      mbar_arrive(&acc_empty[acc]);
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

}  // namespace gf
