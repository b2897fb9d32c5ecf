// Tensor-core GEMM for the encoder's linear layers (Eq. 4 projections, output
// projection, MLP) on the packed rows of the updated tokens.
//
// Y[r][f] = sum_k X[r][k] W[f][k].  The weight tile is the MMA's A operand (M = 128
// output features) and the token rows are its B operand (N = 16..BN_MAX rows, rounded
// up to 16), so a handful of updated tokens still fills the 128-row MMA: the kernel is
// then a weight-streaming loop.  The row count M lives in device memory (written by the
// selection kernel), so no host synchronisation is needed: every CTA reads M, derives
// the same tiling (feature tiles x row tiles x K splits sized to the grid) and walks its
// share of the work items.  K splits write fp32 partials; the last CTA to arrive on a
// tile sums the partials in split order (deterministic) and runs the epilogue.
//
// Pipeline per CTA (128 threads): warp 0 lane 0 issues TMA loads (weights with an
// evict-first L2 policy, rows evict-last), warp 1 lane 0 issues tcgen05.mma into a TMEM
// accumulator, all four warps run the epilogue from TMEM (tcgen05.ld, lane = feature).
#include "internal.h"
#include "ptx.cuh"

namespace ivit {
namespace {

constexpr int BM = 128;          // output features per tile (MMA M)
constexpr int BK = 64;           // K per stage: 128-byte rows, 128-byte swizzle
constexpr int XBOX = 32;         // rows per TMA box of the activation operand
constexpr int STAGES = 4;
constexpr int W_TILE_BYTES = BM * BK * 2;
constexpr int XBOX_BYTES = XBOX * BK * 2;

template <int BN_MAX>
struct GemmSmem {
  static constexpr int X_TILE_BYTES = BN_MAX * BK * 2;
  static constexpr int STAGE_BYTES = W_TILE_BYTES + X_TILE_BYTES;
  static constexpr int BAR_OFFSET = STAGES * STAGE_BYTES;
  static constexpr int TOTAL = BAR_OFFSET + 256 + 1024;  // barriers, flags, 1 KB alignment slack
};

__device__ __forceinline__ float gelu_f(float x, int mode) {
  if (mode == 1) return 0.5f * x * (1.f + erff(x * 0.70710678118654752f));
  const float c = 0.79788456080286536f;  // sqrt(2/pi)
  return 0.5f * x * (1.f + tanhf(c * (x + 0.044715f * x * x * x)));
}

__device__ __forceinline__ void epilogue_store(const GemmEpilogue& e, int r, int f, float y) {
  const float val = y + e.bias[f];
  switch (e.kind) {
    case kEpiF32Bias:
      e.out_f32[static_cast<size_t>(r) * e.ld_out + f] = val;
      break;
    case kEpiResid:
      e.out_f32[static_cast<size_t>(r) * e.ld_out + f] += val;
      break;
    case kEpiGelu:
      e.out_bf16[static_cast<size_t>(r) * e.ld_out + f] = __float2bfloat16_rn(gelu_f(val, e.gelu_mode));
      break;
    default: {  // kEpiQKV
      const int D = e.dim;
      if (f < D) {
        e.out_bf16[static_cast<size_t>(r) * e.ld_out + f] = __float2bfloat16_rn(val);
      } else {
        const size_t tok = static_cast<size_t>(e.rowtok[r]);
        if (f < 2 * D)
          e.cache_k[tok * D + (f - D)] = __float2bfloat16_rn(val);
        else
          e.cache_v[tok * D + (f - 2 * D)] = __float2bfloat16_rn(val);
      }
    }
  }
}

template <int BN_MAX>
__global__ void __launch_bounds__(128, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_x,
                   const GemmArgs a) {
  using L = GemmSmem<BN_MAX>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR_OFFSET);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 1);
  volatile int* sh_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);  // [0] last, [1] abort

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t smem_base = smem_u32(smem);
  const uint32_t bar_base = smem_u32(bars);
  // full[s] = bar_base + 8s, empty[s] = bar_base + 8(STAGES + s), accumulator = 8(2 STAGES)
  const uint32_t acc_bar = bar_base + 8 * (2 * STAGES);

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(bar_base + 8 * s, 1);
      mbar_init(bar_base + 8 * (STAGES + s), 1);
    }
    mbar_init(acc_bar, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tm_w);
    tma_prefetch_desc(&tm_x);
    sh_flag[0] = 0;
    sh_flag[1] = 0;
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(tmem_slot), BN_MAX);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  pdl_wait();  // outputs of the previous kernel on the stream are visible from here

  const int M = a.d_rows ? *a.d_rows : a.m_static;
  const int n_ft = (a.n_out + BM - 1) / BM;
  const int n_tt = (M + BN_MAX - 1) / BN_MAX;
  const int n_kb = (a.k + BK - 1) / BK;
  const int base = n_ft * n_tt;
  int splits = 1;
  if (base > 0 && 2 * base <= static_cast<int>(gridDim.x)) {
    splits = min(static_cast<int>(gridDim.x) / base, min(n_kb, a.max_splits));
    if (splits * base > a.ws_items) splits = max(1, a.ws_items / base);
  }
  const int n_items = base * splits;
  const uint64_t pol_w = l2_policy_evict_first();
  const uint64_t pol_x = l2_policy_evict_last();

  uint32_t p_stage = 0, p_phase = 0;  // producer ring position
  uint32_t c_stage = 0, c_phase = 0;  // MMA ring position
  uint32_t acc_phase = 0;

  for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
    const int t = item % base, sp = item / base;
    const int ft = t % n_ft, tt = t / n_ft;
    const int kb0 = static_cast<int>(static_cast<long long>(sp) * n_kb / splits);
    const int kb1 = static_cast<int>(static_cast<long long>(sp + 1) * n_kb / splits);
    const int row0 = tt * BN_MAX;
    const int rows = min(BN_MAX, M - row0);
    const int n_mma = (rows + 15) & ~15;
    const int nbox = (n_mma + XBOX - 1) / XBOX;

    if (warp == 0) {
      if (lane == 0) {
        for (int kb = kb0; kb < kb1; ++kb) {
          const uint32_t empty = bar_base + 8 * (STAGES + p_stage);
          const uint32_t full = bar_base + 8 * p_stage;
          if (!mbar_wait(empty, p_phase ^ 1)) {
            atomicExch(a.err, kErrWaitSlotEmpty);
            sh_flag[1] = 1;
            break;
          }
          const uint32_t st = smem_base + p_stage * L::STAGE_BYTES;
          mbar_arrive_expect_tx(full, W_TILE_BYTES + nbox * XBOX_BYTES);
          tma_load_2d(st, &tm_w, kb * BK, ft * BM, full, pol_w);
          for (int b = 0; b < nbox; ++b)
            tma_load_2d(st + W_TILE_BYTES + b * XBOX_BYTES, &tm_x, kb * BK, row0 + b * XBOX, full,
                        pol_x);
          if (++p_stage == STAGES) {
            p_stage = 0;
            p_phase ^= 1;
          }
        }
      }
      __syncwarp();
    } else if (warp == 1) {
      if (lane == 0) {
        const uint32_t idesc = idesc_bf16_f32(BM, n_mma);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(bar_base + 8 * c_stage, c_phase)) {
            atomicExch(a.err, kErrWaitTmaFull);
            sh_flag[1] = 1;
            break;
          }
          tc_fence_after();
          const uint32_t st = smem_base + c_stage * L::STAGE_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t ad = sdesc_kmajor_sw128(st + k * 32);
            const uint64_t bd = sdesc_kmajor_sw128(st + W_TILE_BYTES + k * 32);
            umma_bf16(tmem, ad, bd, idesc, (kb > kb0 || k > 0) ? 1u : 0u);
          }
          umma_commit(bar_base + 8 * (STAGES + c_stage));  // frees the stage when read
          if (++c_stage == STAGES) {
            c_stage = 0;
            c_phase ^= 1;
          }
        }
        umma_commit(acc_bar);  // accumulator complete
      }
      __syncwarp();
    }

    if (!mbar_wait(acc_bar, acc_phase)) {
      atomicExch(a.err, kErrWaitAccum);
      sh_flag[1] = 1;
    }
    acc_phase ^= 1;
    tc_fence_after();
    __syncthreads();
    if (sh_flag[1]) break;

    const int fl = warp * 32 + lane;  // TMEM lane == tile-local output feature
    const int f = ft * BM + fl;
    const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    if (splits == 1) {
      for (int c0 = 0; c0 < rows; c0 += 16) {
        float v[16];
        tmem_ld16(trow + c0, v);
        if (f < a.n_out) {
#pragma unroll
          for (int j = 0; j < 16; ++j)
            if (c0 + j < rows) epilogue_store(a.epi, row0 + c0 + j, f, v[j]);
        }
      }
    } else {
      float* part = a.ws + static_cast<size_t>(item) * (BN_MAX * BM);
      for (int c0 = 0; c0 < rows; c0 += 16) {
        float v[16];
        tmem_ld16(trow + c0, v);
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (c0 + j < rows) __stcg(part + (c0 + j) * BM + fl, v[j]);
      }
      __threadfence();
      __syncthreads();
      if (tid == 0) {
        const int prev = atomicAdd(&a.tile_ctr[t], 1);
        sh_flag[0] = (prev == splits - 1) ? 1 : 0;
      }
      __syncthreads();
      if (sh_flag[0]) {
        __threadfence();
        for (int c = 0; c < rows; ++c) {
          float acc = 0.f;
          for (int s2 = 0; s2 < splits; ++s2)
            acc += __ldcg(a.ws + static_cast<size_t>(s2 * base + t) * (BN_MAX * BM) + c * BM + fl);
          if (f < a.n_out) epilogue_store(a.epi, row0 + c, f, acc);
        }
        if (tid == 0) a.tile_ctr[t] = 0;  // ready for the next launch
      }
    }
    tc_fence_before();
    __syncthreads();
  }

  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, BN_MAX);
  }
}

template <int BN>
cudaError_t launch_variant(const CUtensorMap& tm_w, const CUtensorMap& tm_x, const GemmArgs& a,
                           int grid, bool pdl, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = GemmSmem<BN>::TOTAL;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<BN>, tm_w, tm_x, a);
}

}  // namespace

size_t gemm_smem_bytes(int bn_max) {
  return bn_max == 64 ? GemmSmem<64>::TOTAL : GemmSmem<256>::TOTAL;
}

cudaError_t gemm_setup(int bn_max) {
  if (bn_max == 64)
    return cudaFuncSetAttribute(gemm_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                GemmSmem<64>::TOTAL);
  return cudaFuncSetAttribute(gemm_tc_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              GemmSmem<256>::TOTAL);
}

int gemm_ctas_per_sm(int bn_max) {
  int n = 0;
  cudaError_t e;
  if (bn_max == 64)
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gemm_tc_kernel<64>, 128, GemmSmem<64>::TOTAL);
  else
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gemm_tc_kernel<256>, 128,
                                                      GemmSmem<256>::TOTAL);
  return e == cudaSuccess && n > 0 ? n : 1;
}

cudaError_t launch_gemm(int bn_max, const CUtensorMap& tm_w, const CUtensorMap& tm_x,
                        const GemmArgs& a, int grid, bool pdl, cudaStream_t s) {
  if (bn_max == 64) return launch_variant<64>(tm_w, tm_x, a, grid, pdl, s);
  return launch_variant<256>(tm_w, tm_x, a, grid, pdl, s);
}

}  // namespace ivit
