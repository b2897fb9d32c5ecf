// Tensor-core GEMM for the encoder's linear layers (Eq. 4 projections, output
// projection, MLP) on the packed rows of the updated tokens.
//
// Y[r][f] = sum_k X[r][k] W[f][k].  The weight tile is the MMA's A operand (M = 128
// output features) and the token rows are its B operand (N = 16..BN_MAX rows, rounded
// up to 16), so a handful of updated tokens still fills the 128-row MMA: the kernel is
// then a weight-streaming loop.  The row count M lives in device memory (written by the
// selection kernel), so no host synchronisation is needed: every CTA reads M and derives
// the same tiling.
//
// The grid is a set of thread-block clusters.  The CTAs of a cluster split K of one
// output tile between them (so many SMs stream one weight tile at once); each CTA
// writes its fp32 partial tile from TMEM to its slot of a global scratch (it stays in
// L2), and after a cluster barrier every CTA sums a slice of the tile's rows over all
// slots, in rank order (deterministic), and runs the epilogue.  The scratch outlives
// the CTAs, so a cluster with no further tile leaves without a second barrier.  A
// deferred launch (residual epilogue, small row counts) stops after writing its partial
// tile, into a slot of its own per tile: the layer norm that follows sums the slots, so
// neither the cluster barrier nor the reduction sits on this kernel's critical path.
// Clusters walk the output tiles (feature tile x row tile) with a stride.
//
// Pipeline per CTA (128 threads): warp 0 lane 0 issues TMA loads (weights with an
// evict-first L2 policy, rows evict-last), warp 1 lane 0 issues tcgen05.mma into a TMEM
// accumulator, all four warps drain TMEM (tcgen05.ld, lane = output feature).
#include "internal.h"
#include "ptx.cuh"

namespace ivit {
namespace {

constexpr int BM = 128;          // output features per tile (MMA M)
constexpr int BK = 64;           // K per stage: 128-byte rows, 128-byte swizzle
constexpr int XBOX = 32;         // rows per TMA box of the activation operand
constexpr int STAGES = 4;
constexpr int MAX_CLUSTER = 16;  // CTAs per cluster (non-portable size, opted in)
constexpr int W_TILE_BYTES = BM * BK * 2;
constexpr int XBOX_BYTES = XBOX * BK * 2;

template <int BN_MAX>
struct GemmSmem {
  static constexpr int X_TILE_BYTES = BN_MAX * BK * 2;
  static constexpr int STAGE_BYTES = W_TILE_BYTES + X_TILE_BYTES;
  static constexpr int BAR_OFFSET = STAGES * STAGE_BYTES;
  static constexpr int TOTAL = BAR_OFFSET + 256 + 1024;  // barriers, flags, 1 KB alignment slack
  // the split-K reduction stages at most (BN_MAX + MAX_CLUSTER) rows of partials, and the
  // rows' token indices, in the stage memory
  static_assert((BN_MAX + MAX_CLUSTER) * 128 * 4 + (BN_MAX / 2 + 4) * 4 <= BAR_OFFSET, "reduction staging");
};

// Hardware tanh (one MUFU instruction, relative error about 2^-11: below the bf16
// rounding the GELU output gets).
__device__ __forceinline__ float tanh_hw(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float gelu_f(float x, int mode) {
  if (mode == 1) return 0.5f * x * (1.f + erff(x * 0.70710678118654752f));
  const float c = 0.79788456080286536f;  // sqrt(2/pi)
  return 0.5f * x * (1.f + tanh_hw(c * (x + 0.044715f * x * x * x)));
}

// Output feature f of TMEM-drained row r; `bias` is bias[f], loaded while the MMAs run.
// `tok` is rowtok[r] for the epilogues that scatter by token (QKV keys/values,
// kEpiScatterF32), loaded by the caller together with its other loads; `old` is the
// residual stream's current value (kEpiResid), likewise.
__device__ __forceinline__ void epilogue_store(const GemmEpilogue& e, int r, int f, float y, float bias, int tok,
                                               float old) {
  const float val = y + bias;
  switch (e.kind) {
    case kEpiF32Bias:
      e.out_f32[static_cast<size_t>(r) * e.ld_out + f] = val;
      break;
    case kEpiResid:
      e.out_f32[static_cast<size_t>(r) * e.ld_out + f] = old + val;
      break;
    case kEpiGelu:
      e.out_bf16[static_cast<size_t>(r) * e.ld_out + f] = __float2bfloat16_rn(gelu_f(val, e.gelu_mode));
      break;
    case kEpiScatterF32:
      e.out_f32[static_cast<size_t>(tok) * e.ld_out + f] = val;
      break;
    default: {  // kEpiQKV
      const int D = e.dim;
      if (f < D) {
        e.out_bf16[static_cast<size_t>(r) * e.ld_out + f] = __float2bfloat16_rn(val);
      } else if (f < 2 * D) {
        e.cache_k[static_cast<size_t>(tok) * D + (f - D)] = __float2bfloat16_rn(val);
      } else {
        e.cache_v[static_cast<size_t>(tok) * D + (f - 2 * D)] = __float2bfloat16_rn(val);
      }
    }
  }
}

__device__ __forceinline__ bool epi_needs_tok(int kind) { return kind == kEpiQKV || kind == kEpiScatterF32; }

// One column (output feature f) of up to 16 consecutive rows r0 + j (j < n) drained from
// TMEM.  Every global load the epilogue needs (row -> token map, residual values) is
// issued for all 16 rows before the first store, so the rows cost one memory round trip,
// not one each.
__device__ __forceinline__ void epilogue_column16(const GemmEpilogue& e, int r0, int n, int f, float bias,
                                                  const float (&v)[16]) {
  int tok[16];
  float old[16];
  // (the QKV epilogue's queries stay in packed rows: only its keys and values need tokens)
  const bool need_tok = e.kind == kEpiScatterF32 || (e.kind == kEpiQKV && f >= e.dim);
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    tok[j] = 0;
    old[j] = 0.f;
    if (j < n) {
      if (need_tok) tok[j] = __ldcg(e.rowtok + r0 + j);
      if (e.kind == kEpiResid) old[j] = __ldcg(e.out_f32 + static_cast<size_t>(r0 + j) * e.ld_out + f);
    }
  }
#pragma unroll
  for (int j = 0; j < 16; ++j)
    if (j < n) epilogue_store(e, r0 + j, f, v[j], bias, tok[j], old[j]);
}

// Four consecutive output features f4..f4+3 (f4 % 4 == 0, all below n_out: every n_out
// the engine uses is a multiple of 4) of row r, with 8- or 16-byte stores; the bias `b`,
// `tok` and the residual's current value `o` as in epilogue_store.
__device__ __forceinline__ void epilogue_store4(const GemmEpilogue& e, int r, int f4, float4 y, float4 b, int tok,
                                               float4 o) {
  float4 val = make_float4(y.x + b.x, y.y + b.y, y.z + b.z, y.w + b.w);
  auto pack4 = [](float4 u) {
    const __nv_bfloat162 lo = __floats2bfloat162_rn(u.x, u.y), hi = __floats2bfloat162_rn(u.z, u.w);
    uint2 p;
    p.x = *reinterpret_cast<const uint32_t*>(&lo);
    p.y = *reinterpret_cast<const uint32_t*>(&hi);
    return p;
  };
  switch (e.kind) {
    case kEpiF32Bias:
      *reinterpret_cast<float4*>(e.out_f32 + static_cast<size_t>(r) * e.ld_out + f4) = val;
      break;
    case kEpiResid:
      *reinterpret_cast<float4*>(e.out_f32 + static_cast<size_t>(r) * e.ld_out + f4) =
          make_float4(o.x + val.x, o.y + val.y, o.z + val.z, o.w + val.w);
      break;
    case kEpiGelu:
      val = make_float4(gelu_f(val.x, e.gelu_mode), gelu_f(val.y, e.gelu_mode), gelu_f(val.z, e.gelu_mode),
                        gelu_f(val.w, e.gelu_mode));
      *reinterpret_cast<uint2*>(e.out_bf16 + static_cast<size_t>(r) * e.ld_out + f4) = pack4(val);
      break;
    case kEpiScatterF32:
      *reinterpret_cast<float4*>(e.out_f32 + static_cast<size_t>(tok) * e.ld_out + f4) = val;
      break;
    default: {  // kEpiQKV (D % 4 == 0: the four features lie in one of Q, K, V)
      const int D = e.dim;
      bf16* dst = f4 < D ? e.out_bf16 + static_cast<size_t>(r) * e.ld_out + f4
                         : (f4 < 2 * D ? e.cache_k + static_cast<size_t>(tok) * D + (f4 - D)
                                       : e.cache_v + static_cast<size_t>(tok) * D + (f4 - 2 * D));
      *reinterpret_cast<uint2*>(dst) = pack4(val);
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
  volatile int* sh_abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
  // split-K reduction: row -> token indices of this CTA's rows (at most BN_MAX / 2 + 1)
  int* red_tok = reinterpret_cast<int*>(smem + L::BAR_OFFSET - (BN_MAX / 2 + 4) * 4);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t smem_base = smem_u32(smem);
  const uint32_t bar_base = smem_u32(bars);
  // full[s] = bar_base + 8s, empty[s] = bar_base + 8(STAGES + s), accumulator = 8(2 STAGES),
  // (TMEM slot, abort flag), split-K reduction copies = 8(2 STAGES + 2)
  const uint32_t acc_bar = bar_base + 8 * (2 * STAGES);
  const uint32_t red_bar = bar_base + 8 * (2 * STAGES + 2);

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(bar_base + 8 * s, 1);
      mbar_init(bar_base + 8 * (STAGES + s), 1);
    }
    mbar_init(acc_bar, 1);
    mbar_init(red_bar, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tm_w);
    tma_prefetch_desc(&tm_x);
    *sh_abort = 0;
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(tmem_slot), BN_MAX);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // a deferred launch may split K over consecutive CTAs without clusters (a.vsplit)
  const int csize = a.vsplit > 0 ? a.vsplit : static_cast<int>(cluster_nctarank());
  const int crank = a.vsplit > 0 ? static_cast<int>(blockIdx.x) % a.vsplit : static_cast<int>(cluster_ctarank());
  const int cl_id = blockIdx.x / csize, n_cl = gridDim.x / csize;
  // The row count comes from the selection kernel, at least two launches back: every
  // kernel of the library triggers its dependents only after its own wait, so that
  // kernel has completed by the time this grid can start.
  const int M = a.d_rows ? *a.d_rows : a.m_static;
  const int n_ft = (a.n_out + BM - 1) / BM;
  const int n_tt = (M + BN_MAX - 1) / BN_MAX;
  const int n_kb = (a.k + BK - 1) / BK;
  const int tiles = n_ft * n_tt;
  const int kb0 = crank * n_kb / csize, kb1 = (crank + 1) * n_kb / csize;
  const bool has_k = kb1 > kb0;
  const uint64_t pol_w = l2_policy_evict_first();
  const uint64_t pol_x = l2_policy_evict_last();

  // Weights do not depend on earlier kernels: start streaming the first tile's weight
  // stages now, while the previous kernel may still be running.
  int n_pre = 0;
  if (warp == 0 && lane == 0 && cl_id < tiles && has_k) {
    const int ft = cl_id % n_ft, tt = cl_id / n_ft;
    const int n_mma = (min(BN_MAX, M - tt * BN_MAX) + 15) & ~15;
    const int nbox = (n_mma + XBOX - 1) / XBOX;
    n_pre = min(STAGES, kb1 - kb0);
    for (int i = 0; i < n_pre; ++i) {
      const uint32_t full = bar_base + 8 * i;
      mbar_arrive_expect_tx(full, W_TILE_BYTES + nbox * XBOX_BYTES);
      tma_load_2d(smem_base + i * L::STAGE_BYTES, &tm_w, (kb0 + i) * BK, ft * BM, full, pol_w);
    }
  }
  pdl_wait();  // outputs of the previous kernel on the stream are visible from here
  pdl_launch_dependents();
  stamp_begin(a.stamp);

  uint32_t p_stage = 0, p_phase = 0;  // producer ring position
  uint32_t c_stage = 0, c_phase = 0;  // MMA ring position
  uint32_t acc_phase = 0, red_phase = 0;

  for (int tile = cl_id; tile < tiles; tile += n_cl) {
    const int ft = tile % n_ft, tt = tile / n_ft;
    const int row0 = tt * BN_MAX;
    const int rows = min(BN_MAX, M - row0);
    const int n_mma = (rows + 15) & ~15;
    const int nbox = (n_mma + XBOX - 1) / XBOX;
    bool ok = *sh_abort == 0;
    // The epilogue's bias values, loaded now so that their latency hides under the main
    // loop: the direct drain takes feature ft*BM + tid, the split-K reduction features
    // ft*BM + 4*lane .. +3 (a thread's items all share its lane).
    const float bias1 = ft * BM + tid < a.n_out ? __ldg(a.epi.bias + ft * BM + tid) : 0.f;
    const float4 bias4 = ft * BM + 4 * lane < a.n_out ? __ldg(reinterpret_cast<const float4*>(a.epi.bias + ft * BM) + lane)
                                                      : make_float4(0.f, 0.f, 0.f, 0.f);

    if (ok && has_k) {
      if (warp == 0) {
        if (lane == 0) {
          const bool first = tile == cl_id;
          for (int kb = kb0; kb < kb1; ++kb) {
            const uint32_t empty = bar_base + 8 * (STAGES + p_stage);
            const uint32_t full = bar_base + 8 * p_stage;
            const uint32_t st = smem_base + p_stage * L::STAGE_BYTES;
            if (!(first && kb - kb0 < n_pre)) {  // prefetched stages already hold the weights
              if (!mbar_wait(empty, p_phase ^ 1)) {
                atomicExch(a.err, kErrWaitSlotEmpty);
                *sh_abort = 1;
                break;
              }
              mbar_arrive_expect_tx(full, W_TILE_BYTES + nbox * XBOX_BYTES);
              tma_load_2d(st, &tm_w, kb * BK, ft * BM, full, pol_w);
            }
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
              *sh_abort = 1;
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
        *sh_abort = 1;
      }
      acc_phase ^= 1;
    }
    tc_fence_after();
    __syncthreads();
    ok = *sh_abort == 0;

    const int fl = warp * 32 + lane;  // TMEM lane == tile-local output feature
    const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    if (csize == 1) {
      const int f = ft * BM + fl;
      if (ok && has_k) {
        for (int c0 = 0; c0 < rows; c0 += 16) {
          float v[16];
          tmem_ld16(trow + c0, v);
          if (f < a.n_out) epilogue_column16(a.epi, row0 + c0, min(16, rows - c0), f, bias1, v);
        }
      }
    } else {
      // Partials go to this CTA's slot of the global scratch (L2); the cluster barrier's
      // release/acquire makes them visible to the other CTAs, each of which sums a slice
      // of the tile's rows over all slots in rank order.  Global memory outlives the CTA,
      // so only a following tile of this cluster (which reuses the slots) needs a second
      // barrier.
      const int slot = a.defer ? tile * csize + crank : cl_id * csize + crank;
      float* mine = a.partials + static_cast<size_t>(slot) * BN_MAX * BM;
      if (ok && has_k) {
        // 32 accumulator columns per TMEM load (columns past n_mma are allocated, unused)
        for (int c0 = 0; c0 < rows; c0 += 32) {
          uint32_t v[32];
          tmem_ld32_async(trow + c0, v);
          tmem_ld_wait_regs(v);
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (c0 + j < rows) mine[(c0 + j) * BM + fl] = __uint_as_float(v[j]);
        }
      } else {
        for (int c = 0; c < rows; ++c) mine[c * BM + fl] = 0.f;
      }
      if (a.defer) {  // the next kernel sums the slots: no barrier, no epilogue here
        tc_fence_before();
        __syncthreads();  // TMEM is read before the next tile's MMAs
        continue;
      }
      cluster_sync();  // every partial of this tile is in the scratch
      const int c_lo = crank * rows / csize, c_hi = (crank + 1) * rows / csize, nr = c_hi - c_lo;
      if (ok && nr > 0) {
        // This CTA's rows of every slot come into the (idle) stage memory with one bulk
        // copy per slot, so the reduction costs one round trip to L2 however many rows
        // it covers; then slots are summed in rank order (deterministic).
        float* red = reinterpret_cast<float*>(smem);  // [csize][nr][BM]
        const bool need_tok = epi_needs_tok(a.epi.kind);
        if (tid == 0) {
          fence_proxy_async_global();  // the peers' generic stores, acquired above, before the copies
          mbar_arrive_expect_tx(red_bar, static_cast<uint32_t>(csize * nr * BM * 4));
          for (int s = 0; s < csize; ++s)
            bulk_load(smem_base + static_cast<uint32_t>(s * nr * BM * 4),
                      a.partials + (static_cast<size_t>(cl_id * csize + s) * BN_MAX + c_lo) * BM,
                      static_cast<uint32_t>(nr * BM * 4), red_bar);
        }
        if (need_tok && tid < nr) red_tok[tid] = __ldcg(a.epi.rowtok + row0 + c_lo + tid);
        __syncthreads();
        if (!mbar_wait(red_bar, red_phase)) {
          atomicExch(a.err, kErrWaitTmaFull);
          *sh_abort = 1;
        }
        red_phase ^= 1;
        if (*sh_abort == 0) {
          const float4* r4 = reinterpret_cast<const float4*>(red);
          for (int e = tid; e < nr * (BM / 4); e += 128) {
            const int c = e / (BM / 4), q = e % (BM / 4), f4 = ft * BM + 4 * q;
            if (f4 >= a.n_out) continue;
            float4 acc = r4[c * (BM / 4) + q];
            for (int s = 1; s < csize; ++s) {
              const float4 p = r4[(s * nr + c) * (BM / 4) + q];
              acc.x += p.x;
              acc.y += p.y;
              acc.z += p.z;
              acc.w += p.w;
            }
            float4 old = make_float4(0.f, 0.f, 0.f, 0.f);
            if (a.epi.kind == kEpiResid)
              old = __ldcg(reinterpret_cast<const float4*>(a.epi.out_f32 +
                                                           static_cast<size_t>(row0 + c_lo + c) * a.epi.ld_out + f4));
            epilogue_store4(a.epi, row0 + c_lo + c, f4, acc, bias4, need_tok ? red_tok[c] : 0, old);
          }
        }
      }
      if (tile + n_cl < tiles) cluster_sync();  // the next tile rewrites the slots
    }
    tc_fence_before();
    __syncthreads();
  }

  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, BN_MAX);
  }
  stamp_end(a.stamp);
}

// Many-tile form for single-CTA clusters (large row counts): a persistent loop over the
// tiles with warp specialisation, so the epilogue of one tile overlaps the main loop of
// the next.  Warps 0-7 drain the accumulator (warp w reads TMEM lane quarter w % 4 =
// 32 output features, rows of half w / 4 of the tile), warp 8 lane 0 issues the TMA
// loads, warp 9 lane 0 issues the MMAs; two TMEM accumulators (acc_full: MMAs done ->
// epilogue, acc_empty: all eight epilogue warps done -> MMAs).
constexpr int WS_EPI_WARPS = 8;
constexpr int WS_THREADS = (WS_EPI_WARPS + 2) * 32;

template <int BN_MAX>
__global__ void __launch_bounds__(WS_THREADS, 1)
    gemm_ws_kernel(const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_x,
                   const GemmArgs a) {
  using L = GemmSmem<BN_MAX>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR_OFFSET);
  // full[STAGES], empty[STAGES], acc_full[2], acc_empty[2], TMEM slot, abort flag
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 4);
  volatile int* sh_abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t smem_base = smem_u32(smem), bar_base = smem_u32(bars);
  const uint32_t accf = bar_base + 8 * (2 * STAGES), acce = accf + 16;

  if (tid == 0) {
    for (int st = 0; st < STAGES; ++st) {
      mbar_init(bar_base + 8 * st, 1);
      mbar_init(bar_base + 8 * (STAGES + st), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf + 8 * b, 1);
      mbar_init(acce + 8 * b, WS_EPI_WARPS);  // one arrival per epilogue warp
    }
    fence_mbar_init();
    tma_prefetch_desc(&tm_w);
    tma_prefetch_desc(&tm_x);
    *sh_abort = 0;
  }
  if (warp == WS_EPI_WARPS + 1) {
    tmem_alloc(smem_u32(tmem_slot), 2 * BN_MAX);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  const int M = a.d_rows ? *a.d_rows : a.m_static;
  const int n_ft = (a.n_out + BM - 1) / BM;
  const int n_tt = (M + BN_MAX - 1) / BN_MAX;
  const int n_kb = (a.k + BK - 1) / BK;
  const int tiles = n_ft * n_tt;

  // first tile's weight stages before the programmatic-launch wait (constants)
  // (the row count is from the selection kernel, at least two launches back)
  int n_pre = 0;
  if (warp == WS_EPI_WARPS && lane == 0 && static_cast<int>(blockIdx.x) < tiles) {
    const int ft = blockIdx.x % n_ft, tt = blockIdx.x / n_ft;
    const int rows = min(BN_MAX, M - tt * BN_MAX);
    const int nbox = (((rows + 15) & ~15) + XBOX - 1) / XBOX;
    n_pre = min(STAGES, n_kb);
    for (int i = 0; i < n_pre; ++i) {
      mbar_arrive_expect_tx(bar_base + 8 * i, W_TILE_BYTES + nbox * XBOX_BYTES);  // rows follow after the wait
      tma_load_2d(smem_base + i * L::STAGE_BYTES, &tm_w, i * BK, ft * BM, bar_base + 8 * i, l2_policy_evict_first());
    }
  }
  pdl_wait();
  pdl_launch_dependents();
  stamp_begin(a.stamp);

  if (warp == WS_EPI_WARPS) {
    if (lane == 0) {
      const uint64_t pol_w = l2_policy_evict_first(), pol_x = l2_policy_evict_last();
      uint32_t stage = 0, phase = 0;
      bool first = true;
      for (int tile = blockIdx.x; tile < tiles && *sh_abort == 0; tile += gridDim.x) {
        const int ft = tile % n_ft, tt = tile / n_ft;
        const int row0 = tt * BN_MAX, rows = min(BN_MAX, M - row0);
        const int nbox = (((rows + 15) & ~15) + XBOX - 1) / XBOX;
        for (int kb = 0; kb < n_kb; ++kb) {
          const uint32_t full = bar_base + 8 * stage, empty = bar_base + 8 * (STAGES + stage);
          const uint32_t st = smem_base + stage * L::STAGE_BYTES;
          const bool pre = first && kb < n_pre;  // weights already requested, bytes expected
          if (!pre) {
            if (!mbar_wait(empty, phase ^ 1)) {
              atomicExch(a.err, kErrWaitSlotEmpty);
              *sh_abort = 1;
              break;
            }
            mbar_arrive_expect_tx(full, W_TILE_BYTES + nbox * XBOX_BYTES);
            tma_load_2d(st, &tm_w, kb * BK, ft * BM, full, pol_w);
          }
          for (int b = 0; b < nbox; ++b)
            tma_load_2d(st + W_TILE_BYTES + b * XBOX_BYTES, &tm_x, kb * BK, row0 + b * XBOX, full, pol_x);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        first = false;
      }
    }
  } else if (warp == WS_EPI_WARPS + 1) {
    if (lane == 0) {
      uint32_t stage = 0, phase = 0;
      int iter = 0;
      for (int tile = blockIdx.x; tile < tiles && *sh_abort == 0; tile += gridDim.x, ++iter) {
        const int tt = tile / n_ft;
        const int rows = min(BN_MAX, M - tt * BN_MAX);
        const uint32_t idesc = idesc_bf16_f32(BM, (rows + 15) & ~15);
        const int b = iter & 1;
        if (!mbar_wait(acce + 8 * b, ((iter >> 1) & 1) ^ 1)) {  // accumulator b drained
          atomicExch(a.err, kErrWaitAccum);
          *sh_abort = 1;
          break;
        }
        tc_fence_after();
        const uint32_t acc = tmem + static_cast<uint32_t>(b * BN_MAX);
        for (int kb = 0; kb < n_kb; ++kb) {
          if (!mbar_wait(bar_base + 8 * stage, phase)) {
            atomicExch(a.err, kErrWaitTmaFull);
            *sh_abort = 1;
            break;
          }
          tc_fence_after();
          const uint32_t st = smem_base + stage * L::STAGE_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            umma_bf16(acc, sdesc_kmajor_sw128(st + k * 32), sdesc_kmajor_sw128(st + W_TILE_BYTES + k * 32), idesc,
                      (kb > 0 || k > 0) ? 1u : 0u);
          umma_commit(bar_base + 8 * (STAGES + stage));
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        umma_commit(accf + 8 * b);  // accumulator b complete
      }
    }
  } else {
    // epilogue warps: TMEM lane 32 (w % 4) + lane = tile-local output feature; warp w
    // takes the rows of half w / 4 of the tile (halves of a multiple of 16 rows)
    const int quarter = warp & 3, half = warp >> 2;
    const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    int iter = 0;
    for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++iter) {
      const int ft = tile % n_ft, tt = tile / n_ft;
      const int row0 = tt * BN_MAX, rows = min(BN_MAX, M - row0);
      const int b = iter & 1;
      const int f = ft * BM + quarter * 32 + lane;
      const float bias_f = f < a.n_out ? __ldg(a.epi.bias + f) : 0.f;  // loads while the MMAs run
      if (!mbar_wait(accf + 8 * b, (iter >> 1) & 1)) {
        atomicExch(a.err, kErrWaitAccum);
        *sh_abort = 1;
        break;
      }
      tc_fence_after();
      const uint32_t acc = trow + static_cast<uint32_t>(b * BN_MAX);
      const int hrows = ((rows + 31) / 32) * 16;
      const int r_lo = half * hrows, r_hi = min(rows, r_lo + hrows);
      for (int c0 = r_lo; c0 < r_hi; c0 += 16) {
        float v[16];
        tmem_ld16(acc + c0, v);
        if (f < a.n_out) epilogue_column16(a.epi, row0 + c0, min(16, r_hi - c0), f, bias_f, v);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acce + 8 * b);  // accumulator b may be overwritten
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == WS_EPI_WARPS + 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * BN_MAX);
  }
  stamp_end(a.stamp);
}

template <int BN>
cudaError_t launch_variant(const CUtensorMap& tm_w, const CUtensorMap& tm_x, const GemmArgs& a,
                           int n_clusters, int csize, cudaStream_t s) {
  if (BN == 256 && csize == 1)
    return launch_ex(gemm_ws_kernel<BN>, dim3(n_clusters), dim3(WS_THREADS), GemmSmem<BN>::TOTAL, s, 1, tm_w, tm_x,
                     a);
  // cluster dims are always given (also for a single CTA) so %cluster_nctarank is exact;
  // a launch with a virtual split (deferred partials, no cluster barrier) runs clusters of one
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_clusters * csize);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = GemmSmem<BN>::TOTAL;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = a.vsplit > 0 ? 1 : csize;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = g_use_pdl ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<BN>, tm_w, tm_x, a);
}

template <int BN>
int max_clusters_variant(int csize) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(csize);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = GemmSmem<BN>::TOTAL;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = csize;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, gemm_tc_kernel<BN>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

template <int BN>
cudaError_t setup_variant() {
  cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       GemmSmem<BN>::TOTAL);
  if (e != cudaSuccess) return e;
  if (BN == 256) {
    e = cudaFuncSetAttribute(gemm_ws_kernel<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, GemmSmem<BN>::TOTAL);
    if (e != cudaSuccess) return e;
  }
  return cudaFuncSetAttribute(gemm_tc_kernel<BN>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
}

}  // namespace

size_t gemm_smem_bytes(int bn_max) {
  return bn_max == 64 ? GemmSmem<64>::TOTAL : GemmSmem<256>::TOTAL;
}

cudaError_t gemm_setup(int bn_max) { return bn_max == 64 ? setup_variant<64>() : setup_variant<256>(); }

int gemm_max_clusters(int bn_max, int csize) {
  return bn_max == 64 ? max_clusters_variant<64>(csize) : max_clusters_variant<256>(csize);
}

cudaError_t launch_gemm(int bn_max, const CUtensorMap& tm_w, const CUtensorMap& tm_x,
                        const GemmArgs& args, int n_clusters, int csize, cudaStream_t s) {
  GemmArgs a = args;
  a.stamp = g_stamp;
  if (bn_max == 64) return launch_variant<64>(tm_w, tm_x, a, n_clusters, csize, s);
  return launch_variant<256>(tm_w, tm_x, a, n_clusters, csize, s);
}

}  // namespace ivit
