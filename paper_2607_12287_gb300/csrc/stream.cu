// Weight-streaming encoder kernel for a few dozen updated rows: every transformer
// block of an incremental call (Sec. III-B: the Q/K/V projections of Eq. 4 for the
// updated tokens, the cache scatter of Eq. 5, attention of the updated queries over all
// N tokens, the output projection and the MLP) in one cooperative launch.
//
// With ~26 updated rows the call must stream 823.5 MB of weights once; a chain of one
// kernel per operation spends most of its time in launch handoffs while HBM idles.
// Here one CTA per SM walks seven stages per layer, separated by grid barriers:
//
//   QKV | attention | out-proj | +residual, LN2 | MLP-up, GELU | MLP-down | +residual, LN1
//
// (the first stage of the call is LN1 of layer 0; the last writes the final layer norm
// into the final-token cache).
//
// GEMMs: the weight tile is the MMA's A operand (M = 128 output features) and the
// updated rows its B operand (N = 16..64 rows per pass), so a handful of rows still
// fills the MMA.  Each GEMM splits K over the CTAs (tile x split tasks, about one per
// CTA); the split partials (fp32, L2) are summed in split order (deterministic) by the
// last CTA of a tile to finish (QKV: + bias -> queries and the Eq. 5 K/V cache rows;
// MLP-up: + bias, GELU -> hidden state) or by the following row stage (out-proj,
// MLP-down: + bias + residual, then the layer norm).  Warp 0 of every CTA streams the
// weight stages (16 KB) of its tasks by TMA into a ring in shared memory, in the order
// the MMAs consume them, across stage and layer boundaries, limited only by free ring
// slots: the weight stream never waits for activations.  The activation operand of each
// task (layer-norm output, attention output or hidden state rows) comes by TMA after
// the barrier.
//
// Attention: items (view, head, query group) over all CTAs; the cached keys and values
// of the head ([N][dh] bf16, one TMA box each) are fetched as soon as the CTA's QKV work
// is done, before the barrier; after it the rows of this call's updated tokens are read
// again.  Scores, softmax (fp32, base 2) and P V run on the CUDA cores with the keys
// split over all eight compute warps.
//
// Roles (320 threads): warp 0 lane 0 weight producer; warp 1 lane 0 MMA issuer and TMA
// of the activation operands and K/V tiles; warps 2..9 epilogues, reductions, layer
// norms and attention.  Every wait is bounded; a CTA whose wait expires records an error
// and raises the abort flag that stops every CTA at its next grid barrier; copies in
// flight are drained before a CTA leaves.
#include <algorithm>

#include "internal.h"
#include "ptx.cuh"

namespace ivit {
namespace {

constexpr int SK_THREADS = 320;
constexpr int SK_SYNC_THREADS = 288;     // warps 1..9 (named barrier kBarAll)
constexpr int SK_COMPUTE_THREADS = 256;  // warps 2..9 (named barrier kBarCompute)
constexpr int SK_CWARPS = 8;
constexpr int SK_BM = 128;               // output features per tile (MMA M)
constexpr int SK_BK = 64;                // K per stage: 128-byte rows, 128-byte swizzle
constexpr int SK_PROWS = 64;             // rows per pass (MMA N <= 64)
constexpr int SK_XBOX = 32;              // rows per TMA box of the activation operand
constexpr int SK_STAGE = SK_BM * SK_BK * 2;    // 16 KB weight stage
constexpr int SK_BBLK = SK_PROWS * SK_BK * 2;  // 8 KB activation k-block (64 rows)
constexpr int SK_XBOX_BYTES = SK_XBOX * SK_BK * 2;
constexpr int SK_MISC = 2048;
constexpr int SK_QCH = 4;                // attention queries per chunk
constexpr int SK_ROW_F4 = 2;             // float4 per thread of a row stage (D <= 2048)
constexpr int kBarAll = 1, kBarCompute = 2;

enum SkGemm : int { kSkQKV = 0, kSkOut = 1, kSkUp = 2, kSkDown = 3 };

__device__ __forceinline__ void named_bar(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

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

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ float4 f4add(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}

// Shape of GEMM g: output features, K, tiles of 128 features, K splits, k-blocks.
struct SkShape {
  int n_out, k, tiles, splits, nkb, tasks;
};

__device__ __forceinline__ SkShape sk_shape(const StreamArgs& a, int g) {
  SkShape s;
  s.n_out = g == kSkQKV ? 3 * a.D : (g == kSkUp ? a.F : a.D);
  s.k = g == kSkDown ? a.F : a.D;
  s.tiles = (s.n_out + SK_BM - 1) / SK_BM;
  s.splits = a.splits[g];
  s.nkb = (s.k + SK_BK - 1) / SK_BK;
  s.tasks = s.tiles * s.splits;
  return s;
}

__device__ __forceinline__ void sk_task_geom(const SkShape& s, int t, int& tile, int& split, int& kb0, int& kb1) {
  tile = t / s.splits;
  split = t % s.splits;
  kb0 = split * s.nkb / s.splits;
  kb1 = (split + 1) * s.nkb / s.splits;
}

struct SkCtx {
  const StreamArgs* a;
  uint32_t ring, reg, bars;  // shared-memory addresses: weight ring, operand / attention region
  uint8_t* reg_ptr;
  uint32_t tmem;
  int M, passes, passes_max;
  volatile int* sh;  // [0] grid barrier ok, [1] abort, [2] last of a tile, [4] K/V tile landed
  float* red;        // [2][8] block-reduction scratch
  uint32_t c_pos;    // ring stages consumed (MMA issuer; every thread tracks it alike)
  uint32_t acc_phase, b_phase, kv_phase;
  unsigned epoch;
};

__device__ __forceinline__ uint32_t full_bar(const SkCtx& c, int s) { return c.bars + 8 * s; }
__device__ __forceinline__ uint32_t empty_bar(const SkCtx& c, int s) {
  return c.bars + 8 * (c.a->ring_stages + s);
}
__device__ __forceinline__ uint32_t acc_bar(const SkCtx& c) { return c.bars + 8 * (2 * c.a->ring_stages); }
__device__ __forceinline__ uint32_t b_bar(const SkCtx& c) { return c.bars + 8 * (2 * c.a->ring_stages + 1); }
__device__ __forceinline__ uint32_t kv_bar(const SkCtx& c) { return c.bars + 8 * (2 * c.a->ring_stages + 2); }

// Timeline accumulators (IVIT_TRACE): slot k (< 8) of kind g (< 8: 0..3 GEMMs, 4
// attention, 5 row stages) of this CTA.
__device__ __forceinline__ void sk_trace_add(const SkCtx& c, int g, int k, uint64_t ns) {
  const StreamArgs& a = *c.a;
  if (a.trace)
    a.trace[static_cast<size_t>(a.n_barriers) * (gridDim.x + 1) + (blockIdx.x * 8 + g) * 8 + k] += ns;
}

__device__ __forceinline__ bool sk_aborted(const SkCtx& c) {
  return c.sh[1] != 0 || ld_acquire_u32(c.a->sync + 2) != 0;
}

__device__ __forceinline__ void sk_raise(const SkCtx& c, int code) {
  atomicExch(c.a->err, code);
  atomicExch(c.a->sync + 2, 1u);
  c.sh[1] = 1;
}

// Grid barrier over warps 1..9 of every CTA: one acquire-release arrival per CTA on a
// monotonic counter (zeroed before the launch), then a bounded acquire spin that also
// gives up when another CTA raised the abort flag.  Returns the same value to every
// thread of the CTA: false when it expired or the call was aborted.
__device__ bool sk_grid_sync(SkCtx& c) {
  const StreamArgs& a = *c.a;
  named_bar(kBarAll, SK_SYNC_THREADS);
  if (threadIdx.x == 64) {  // warp 2 lane 0
    if (a.trace) a.trace[static_cast<size_t>(c.epoch) * gridDim.x + blockIdx.x] = globaltimer_ns();
    ++c.epoch;
    const unsigned target = c.epoch * gridDim.x;
    atom_add_acq_rel_u32(a.sync, 1u);
    bool ok = c.sh[1] == 0;
    const uint64_t t0 = globaltimer_ns();
    while (ok && ld_acquire_u32(a.sync) < target) {
      if (ld_acquire_u32(a.sync + 2) != 0) {
        ok = false;
      } else if (globaltimer_ns() - t0 > kWaitLimitNs) {
        atomicExch(a.err, kErrGridBarrier);
        atomicExch(a.sync + 2, 1u);
        ok = false;
      }
    }
    if (!ok) c.sh[1] = 1;
    c.sh[0] = ok ? 1 : 0;
    if (a.trace && blockIdx.x == 0)
      a.trace[static_cast<size_t>(a.n_barriers) * gridDim.x + c.epoch - 1] = globaltimer_ns();
  }
  named_bar(kBarAll, SK_SYNC_THREADS);
  return c.sh[0] != 0;
}

// ---------------------------------------------------------------- weight producer
// Warp 0 lane 0: every weight stage of this CTA's GEMM tasks, in the order the MMA
// issuer consumes them (layer, GEMM, task, k-block), into the ring.  A task's stages
// stay in the ring until its last pass of rows (the ring holds at least one task).
__device__ uint32_t sk_producer(SkCtx& c) {
  const StreamArgs& a = *c.a;
  const int G = static_cast<int>(gridDim.x);
  const int RS = a.ring_stages;
  const uint64_t pol = l2_policy_evict_first();
  uint32_t pos = 0;
  for (int l = 0; l < a.L; ++l) {
    for (int g = 0; g < 4; ++g) {
      const SkShape s = sk_shape(a, g);
      const CUtensorMap* map = a.wmaps + 4 * l + g;
      for (int t = blockIdx.x; t < s.tasks; t += G) {
        int tile, split, kb0, kb1;
        sk_task_geom(s, t, tile, split, kb0, kb1);
        for (int kb = kb0; kb < kb1; ++kb) {
          const int slot = static_cast<int>(pos % RS);
          const uint32_t parity = ((pos / RS) & 1u) ^ 1u;
          // wait for the slot to be free, giving up early on abort
          bool ok = mbar_try_wait(empty_bar(c, slot), parity);
          const uint64_t t0 = ok ? 0 : globaltimer_ns();
          while (!ok) {
            for (int i = 0; i < 8 && !ok; ++i) ok = mbar_try_wait(empty_bar(c, slot), parity);
            if (ok) break;
            __nanosleep(256);  // the ring is full: leave the issue slots to the compute warps
            if (sk_aborted(c)) return pos;
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
              sk_raise(c, kErrWaitSlotEmpty);
              return pos;
            }
          }
          mbar_arrive_expect_tx(full_bar(c, slot), SK_STAGE);
          tma_load_2d(c.ring + slot * SK_STAGE, map, kb * SK_BK, tile * SK_BM, full_bar(c, slot), pol);
          ++pos;
        }
      }
    }
  }
  return pos;
}

// ------------------------------------------------------------------ GEMM tasks
// MMA issuer (warp 1 lane 0): one pass of a task: the activation rows by TMA, then for
// each k-block the weight stage (A) times the rows (B) into the TMEM accumulator.  The
// weight stages are released after the last pass only.
__device__ void sk_mma_pass(SkCtx& c, int g, int kb0, int nkb, int p, int n_mma, bool release, uint32_t pos0) {
  const StreamArgs& a = *c.a;
  const int RS = a.ring_stages;
  const int nbox = (n_mma + SK_XBOX - 1) / SK_XBOX;
  const CUtensorMap* bm = a.bmaps + (g == kSkQKV || g == kSkUp ? 0 : (g == kSkOut ? 1 : 2));
  const uint64_t t0 = a.trace ? globaltimer_ns() : 0;
  fence_proxy_async_global();  // generic writes of other CTAs (acquired at the barrier) before TMA reads
  mbar_arrive_expect_tx(b_bar(c), nkb * nbox * SK_XBOX_BYTES);
  for (int j = 0; j < nkb; ++j)
    for (int b = 0; b < nbox; ++b)
      tma_load_2d(c.reg + j * SK_BBLK + b * SK_XBOX_BYTES, bm, (kb0 + j) * SK_BK, p * SK_PROWS + b * SK_XBOX, b_bar(c),
                  l2_policy_evict_last());
  bool ok = mbar_wait(b_bar(c), c.b_phase);
  if (!ok) sk_raise(c, kErrWaitTmaFull);
  const uint64_t t1 = a.trace ? globaltimer_ns() : 0;
  if (t0) sk_trace_add(c, g, 1, t1 - t0);
  tc_fence_after();
  const uint32_t idesc = idesc_bf16_f32(SK_BM, n_mma);
  for (int j = 0; ok && j < nkb; ++j) {
    const uint32_t pos = pos0 + j;
    const int slot = static_cast<int>(pos % RS);
    const bool ready = mbar_try_wait(full_bar(c, slot), (pos / RS) & 1u);
    const uint64_t tw = (a.trace && !ready) ? globaltimer_ns() : 0;
    if (!ready && !mbar_wait(full_bar(c, slot), (pos / RS) & 1u)) {
      sk_raise(c, kErrWaitTmaFull);
      ok = false;
      break;
    }
    if (tw) sk_trace_add(c, g, 0, globaltimer_ns() - tw);
    tc_fence_after();
    const uint32_t ab = c.ring + slot * SK_STAGE, bb = c.reg + j * SK_BBLK;
#pragma unroll
    for (int k = 0; k < SK_BK / 16; ++k)
      umma_bf16(c.tmem, sdesc_kmajor_sw128(ab + k * 32), sdesc_kmajor_sw128(bb + k * 32), idesc,
                (j > 0 || k > 0) ? 1u : 0u);
    if (release) umma_commit(empty_bar(c, slot));
  }
  umma_commit(acc_bar(c));  // (also when a wait failed: completes the accumulator phase)
  if (t1) sk_trace_add(c, g, 2, globaltimer_ns() - t1);
}

// Epilogue of one pass on warps 2..9: TMEM lane = tile-local output feature (warp w
// reads lanes 32 (w % 4) ..), column = row of the pass; the two warps of a lane quarter
// take alternate 16-row column chunks.  Writes the split's fp32 partial
// part[(split * M_max + row) * n_out + feature].
__device__ void sk_epilogue(const SkCtx& c, const SkShape& s, int tile, int split, int p, int n_mma) {
  const StreamArgs& a = *c.a;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = warp & 3, half = (warp - 2) >> 2;
  const int f = tile * SK_BM + q * 32 + lane;
  const uint32_t trow = c.tmem + (static_cast<uint32_t>(q * 32) << 16);
  float* base = a.part + static_cast<size_t>(split) * a.M_max * s.n_out + f;
  for (int ch = half; ch < n_mma / 16; ch += 2) {
    float v[16];
    tmem_ld16(trow + ch * 16, v);
    if (f < s.n_out) {
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int row = p * SK_PROWS + ch * 16 + j;
        if (row < c.M) __stcg(base + static_cast<size_t>(row) * s.n_out, v[j]);
      }
    }
  }
}

// Sum of the split partials of (row, features f..f+15) in split order, + bias; only the
// first n4 float4 (features below n_out, a multiple of 8) are read.
__device__ __forceinline__ void sk_sum16(const StreamArgs& a, const SkShape& s, int row, int f, const float* bias,
                                         int n4, float4 (&acc)[4]) {
  const float4* b4 = reinterpret_cast<const float4*>(bias + f);
#pragma unroll
  for (int u = 0; u < 4; ++u) acc[u] = u < n4 ? b4[u] : make_float4(0.f, 0.f, 0.f, 0.f);
  const size_t stride = static_cast<size_t>(a.M_max) * s.n_out;
  const float* p = a.part + static_cast<size_t>(row) * s.n_out + f;
  for (int sp = 0; sp < s.splits; ++sp) {
    float4 t[4];
#pragma unroll
    for (int u = 0; u < 4; ++u)
      t[u] = u < n4 ? __ldcg(reinterpret_cast<const float4*>(p + sp * stride) + u) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int u = 0; u < 4; ++u) acc[u] = f4add(acc[u], t[u]);
  }
}

__device__ __forceinline__ uint4 pack8(const float* v) {
  uint4 u;
  uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    __nv_bfloat162 t = __floats2bfloat162_rn(v[2 * e], v[2 * e + 1]);
    w[e] = *reinterpret_cast<uint32_t*>(&t);
  }
  return u;
}

// Last CTA of a (tile, pass) of the QKV or MLP-up GEMM: the tile's rows summed over the
// splits + bias, then queries and the K/V cache rows of the updated tokens (Eq. 5), or
// GELU into the hidden state.  Warps 2..9: thread -> (row, 16 features).
__device__ void sk_fixup(const SkCtx& c, int l, int g, const SkShape& s, int tile, int p) {
  const StreamArgs& a = *c.a;
  const int t = threadIdx.x - 64;
  const int rows = min(SK_PROWS, c.M - p * SK_PROWS);
  const int f = tile * SK_BM + (t & 7) * 16;
  if (f >= s.n_out) return;
  const LayerParams& lp = a.layers[l];
  const int D = a.D;
  for (int jr = t >> 3; jr < rows; jr += SK_COMPUTE_THREADS / 8) {
    const int row = p * SK_PROWS + jr;
    float4 acc[4];
    sk_sum16(a, s, row, f, g == kSkQKV ? lp.bqkv : lp.b1, min(4, (s.n_out - f) / 4), acc);
    float* v = reinterpret_cast<float*>(acc);
    if (g == kSkQKV) {
      bf16* dst;
      if (f < D) {
        dst = a.q + static_cast<size_t>(row) * D + f;
      } else {
        const size_t tok = static_cast<size_t>(a.rowtok[row]);
        const size_t lo = static_cast<size_t>(l) * a.M_max * D;
        dst = f < 2 * D ? a.cacheK + lo + tok * D + (f - D) : a.cacheV + lo + tok * D + (f - 2 * D);
      }
      reinterpret_cast<uint4*>(dst)[0] = pack8(v);
      reinterpret_cast<uint4*>(dst)[1] = pack8(v + 8);
    } else {
#pragma unroll
      for (int e = 0; e < 16; ++e) v[e] = gelu_f(v[e], a.gelu);
      bf16* dst = a.h + static_cast<size_t>(row) * a.F + f;
      if (f + 16 <= a.F) {
        reinterpret_cast<uint4*>(dst)[0] = pack8(v);
        reinterpret_cast<uint4*>(dst)[1] = pack8(v + 8);
      } else {
        for (int e = 0; f + e < a.F; ++e) dst[e] = __float2bfloat16_rn(v[e]);
      }
    }
  }
}

// All tasks of GEMM g of layer l on this CTA (warps 1..9).  Control flow is the same
// for every thread (the named barriers inside are not bounded); after an expired wait
// the roles skip their work and the next grid barrier stops the kernel.
__device__ void sk_gemm_stage(SkCtx& c, int l, int g) {
  const StreamArgs& a = *c.a;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const SkShape s = sk_shape(a, g);
  const int G = static_cast<int>(gridDim.x);
  const bool fix = g == kSkQKV || g == kSkUp;
  for (int t = blockIdx.x; t < s.tasks; t += G) {
    int tile, split, kb0, kb1;
    sk_task_geom(s, t, tile, split, kb0, kb1);
    const int nkb = kb1 - kb0;
    const uint32_t pos0 = c.c_pos;
    for (int p = 0; p < c.passes; ++p) {
      const int rows = min(SK_PROWS, c.M - p * SK_PROWS);
      const int n_mma = (rows + 15) & ~15;
      if (warp == 1) {
        if (lane == 0) {
          if (c.sh[1] == 0)
            sk_mma_pass(c, g, kb0, nkb, p, n_mma, p + 1 == c.passes, pos0);
          else
            umma_commit(acc_bar(c));
        }
        __syncwarp();
      } else if (warp >= 2) {
        const uint64_t te = (a.trace && lane == 0 && warp == 2) ? globaltimer_ns() : 0;
        const bool ok = mbar_wait(acc_bar(c), c.acc_phase);
        tc_fence_after();
        const uint64_t tf = te ? globaltimer_ns() : 0;
        if (!ok) {
          if (lane == 0) sk_raise(c, kErrWaitAccum);
        } else if (c.sh[1] == 0) {
          sk_epilogue(c, s, tile, split, p, n_mma);
        }
        tc_fence_before();
        __syncwarp();
        if (te) {
          sk_trace_add(c, g, 3, tf - te);
          sk_trace_add(c, g, 4, globaltimer_ns() - tf);
          sk_trace_add(c, g, 7, 1);
        }
      }
      c.b_phase ^= 1u;
      c.acc_phase ^= 1u;
      named_bar(kBarAll, SK_SYNC_THREADS);  // accumulator drained, operand region free
      if (fix) {
        // the last of the splits of (tile, pass) sums them
        if (threadIdx.x == 64) {
          const size_t ctr = g == kSkQKV ? (static_cast<size_t>(l) * s.tiles + tile) * c.passes_max + p
                                         : static_cast<size_t>(a.L) * a.qkv_tiles * c.passes_max +
                                               (static_cast<size_t>(l) * s.tiles + tile) * c.passes_max + p;
          c.sh[2] = atom_add_acq_rel_u32(a.sync + 4 + ctr, 1u) == static_cast<unsigned>(s.splits - 1) ? 1 : 0;
        }
        named_bar(kBarAll, SK_SYNC_THREADS);
        const uint64_t tx = (a.trace && threadIdx.x == 64) ? globaltimer_ns() : 0;
        if (c.sh[2] && warp >= 2) sk_fixup(c, l, g, s, tile, p);
        if (tx) sk_trace_add(c, g, 5, globaltimer_ns() - tx);
      }
    }
    c.c_pos = pos0 + nkb;
  }
}

// ------------------------------------------------------------------- row stages
// Block-wide sum over warps 2..9 (every compute thread gets the total).
__device__ __forceinline__ float sk_block_sum(const SkCtx& c, float v, int slot) {
  v = warp_sum(v);
  const int cw = (threadIdx.x >> 5) - 2, lane = threadIdx.x & 31;
  if (lane == 0) c.red[slot * 8 + cw] = v;
  named_bar(kBarCompute, SK_COMPUTE_THREADS);
  float t = 0.f;
#pragma unroll
  for (int w = 0; w < SK_CWARPS; ++w) t += c.red[slot * 8 + w];
  return t;
}

// One CTA per row (warps 2..9): with `splits` > 0 first x[r] += sum of the split
// partials of the out-proj / MLP-down GEMM (split order) + bias, then the layer norm
// of x[r] into dst (row r, or row rowtok[r] with `scatter`).
__device__ void sk_row_stage(const SkCtx& c, int splits, const float* __restrict__ bias,
                             const float* __restrict__ gamma, const float* __restrict__ beta, bf16* dst,
                             bool scatter) {
  const StreamArgs& a = *c.a;
  const int t = threadIdx.x - 64;
  const int D = a.D, n4 = D / 4;
  const uint64_t t0 = (a.trace && t == 0) ? globaltimer_ns() : 0;
  int done = 0;
  for (int r = blockIdx.x; r < c.M; r += gridDim.x, ++done) {
    float4* xr = reinterpret_cast<float4*>(a.x + static_cast<size_t>(r) * D);
    float4 v[SK_ROW_F4];
    float sum = 0.f;
#pragma unroll
    for (int i = 0; i < SK_ROW_F4; ++i) {
      const int ch = t + SK_COMPUTE_THREADS * i;
      v[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (ch < n4) {
        float4 xv = __ldcg(xr + ch);
        if (splits > 0) {
          float4 acc = reinterpret_cast<const float4*>(bias)[ch];
          const float* p = a.part + static_cast<size_t>(r) * D + 4 * ch;
          const size_t stride = static_cast<size_t>(a.M_max) * D;
          for (int s0 = 0; s0 < splits; s0 += 8) {  // batches of 8 loads in flight
            float4 pv[8];
#pragma unroll
            for (int u = 0; u < 8; ++u)
              pv[u] = s0 + u < splits ? __ldcg(reinterpret_cast<const float4*>(p + (s0 + u) * stride))
                                      : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int u = 0; u < 8; ++u) acc = f4add(acc, pv[u]);
          }
          xv = f4add(xv, acc);
          __stcg(xr + ch, xv);
        }
        v[i] = xv;
        sum += (xv.x + xv.y) + (xv.z + xv.w);
      }
    }
    const float mean = sk_block_sum(c, sum, 0) / D;
    float sq = 0.f;
#pragma unroll
    for (int i = 0; i < SK_ROW_F4; ++i) {
      if (t + SK_COMPUTE_THREADS * i < n4) {
        const float e0 = v[i].x - mean, e1 = v[i].y - mean, e2 = v[i].z - mean, e3 = v[i].w - mean;
        sq += (e0 * e0 + e1 * e1) + (e2 * e2 + e3 * e3);
      }
    }
    const float rstd = rsqrtf(sk_block_sum(c, sq, 1) / D + a.eps);
    const size_t orow = scatter ? static_cast<size_t>(a.rowtok[r]) : static_cast<size_t>(r);
    __nv_bfloat162* yr = reinterpret_cast<__nv_bfloat162*>(dst + orow * D);
#pragma unroll
    for (int i = 0; i < SK_ROW_F4; ++i) {
      const int ch = t + SK_COMPUTE_THREADS * i;
      if (ch < n4) {
        const float4 gg = reinterpret_cast<const float4*>(gamma)[ch];
        const float4 bb = reinterpret_cast<const float4*>(beta)[ch];
        yr[2 * ch] = __floats2bfloat162_rn(gg.x * (v[i].x - mean) * rstd + bb.x, gg.y * (v[i].y - mean) * rstd + bb.y);
        yr[2 * ch + 1] =
            __floats2bfloat162_rn(gg.z * (v[i].z - mean) * rstd + bb.z, gg.w * (v[i].w - mean) * rstd + bb.w);
      }
    }
    named_bar(kBarCompute, SK_COMPUTE_THREADS);  // red reused by the next row
  }
  if (t0 && done) {
    sk_trace_add(c, 5, 0, globaltimer_ns() - t0);
    sk_trace_add(c, 5, 7, done);
  }
}

// ------------------------------------------------------------------- attention
struct AttItem {
  int v, h, q0, q1;
};

__device__ __forceinline__ AttItem sk_att_item(const StreamArgs& a, int item) {
  AttItem it;
  const int per_view = a.H * a.att_groups;
  it.v = item / per_view;
  const int rem = item % per_view;
  it.h = rem / a.att_groups;
  const int grp = rem % a.att_groups;
  const int r_lo = a.cu_rows[it.v], r_hi = a.cu_rows[it.v + 1];
  const int nq = r_hi - r_lo;
  it.q0 = r_lo + grp * nq / a.att_groups;
  it.q1 = r_lo + (grp + 1) * nq / a.att_groups;
  return it;
}

__device__ __forceinline__ int sk_att_items(const StreamArgs& a) { return a.SV * a.H * a.att_groups; }

// Attention region layout (inside the operand region).
struct AttSmem {
  bf16 *k, *v;
  float *q;   // [QCH][dh], pre-scaled by log2(e) / sqrt(dh)
  float *p;   // [QCH][N] scores, then probabilities
  float *ml;  // [8 warps][QCH][2] per-warp max and sum
  float *o;   // [8 warps][QCH][dh] per-warp P V partials
};

__device__ __forceinline__ size_t sk_kv_bytes(int n_tok, int dh) {
  return (static_cast<size_t>(n_tok) * dh * 2 + 127) & ~static_cast<size_t>(127);
}

__device__ __forceinline__ AttSmem sk_att_smem(const SkCtx& c) {
  const StreamArgs& a = *c.a;
  AttSmem s;
  const size_t kv = sk_kv_bytes(a.N, a.dh);
  s.k = reinterpret_cast<bf16*>(c.reg_ptr);
  s.v = reinterpret_cast<bf16*>(c.reg_ptr + kv);
  s.q = reinterpret_cast<float*>(c.reg_ptr + 2 * kv);
  s.p = s.q + SK_QCH * a.dh;
  s.ml = s.p + SK_QCH * a.N;
  s.o = s.ml + SK_CWARPS * SK_QCH * 2;
  return s;
}

// Warp 1 lane 0: TMA of the cached keys and values of (view, head) of layer l.
__device__ void sk_prefetch_kv(SkCtx& c, int l, const AttItem& it) {
  const StreamArgs& a = *c.a;
  const AttSmem s = sk_att_smem(c);
  const uint32_t tile = static_cast<uint32_t>(a.N) * a.dh * 2;
  fence_proxy_async_smem();
  mbar_arrive_expect_tx(kv_bar(c), 2 * tile);
  tma_load_2d(smem_u32(s.k), a.kvmaps + 2 * l, it.h * a.dh, it.v * a.N, kv_bar(c), l2_policy_evict_last());
  tma_load_2d(smem_u32(s.v), a.kvmaps + 2 * l + 1, it.h * a.dh, it.v * a.N, kv_bar(c), l2_policy_evict_last());
}

// One attention item on warps 2..9 (the K/V tile is in flight or resident).  Warp w owns
// keys [w N / 8, (w + 1) N / 8); per chunk of up to four queries: scores (lane = key),
// block-wide max and sum of the exponentials, then P V with lanes owning output dims,
// summed over the warps in warp order.
__device__ void sk_att_item_run(SkCtx& c, int l, const AttItem& it) {
  const StreamArgs& a = *c.a;
  const int cw = (threadIdx.x >> 5) - 2, lane = threadIdx.x & 31;
  const int tid = threadIdx.x - 64;
  const int N = a.N, D = a.D, dh = a.dh;
  const AttSmem s = sk_att_smem(c);
  const uint64_t t0 = (a.trace && tid == 0) ? globaltimer_ns() : 0;
  const bool landed = mbar_wait(kv_bar(c), c.kv_phase);
  if (tid == 0) {
    if (!landed) sk_raise(c, kErrWaitTmaFull);
    c.sh[4] = landed ? 1 : 0;
  }
  named_bar(kBarCompute, SK_COMPUTE_THREADS);
  const bool run = c.sh[4] != 0;  // (the same for every thread: written before the barrier)
  named_bar(kBarCompute, SK_COMPUTE_THREADS);
  if (!run) return;
  // this call's updated keys and values of the view, final after the QKV stage
  const size_t lo = static_cast<size_t>(l) * a.M_max * D;
  const int r_lo = a.cu_rows[it.v], r_hi = a.cu_rows[it.v + 1];
  const int dh8 = dh / 8;
  for (int e = tid; e < (r_hi - r_lo) * dh8; e += SK_COMPUTE_THREADS) {
    const int tok = a.rowtok[r_lo + e / dh8], d = (e % dh8) * 8;
    const size_t gaddr = lo + static_cast<size_t>(tok) * D + it.h * dh + d;
    const int key = tok - it.v * N;
    *reinterpret_cast<uint4*>(s.k + key * dh + d) = __ldcg(reinterpret_cast<const uint4*>(a.cacheK + gaddr));
    *reinterpret_cast<uint4*>(s.v + key * dh + d) = __ldcg(reinterpret_cast<const uint4*>(a.cacheV + gaddr));
  }
  const float qscale = rsqrtf(static_cast<float>(dh)) * 1.4426950408889634f;  // log2(e) / sqrt(dh)
  const int k0 = cw * N / SK_CWARPS, k1 = (cw + 1) * N / SK_CWARPS;
  uint64_t t1 = 0;
  for (int qa = it.q0; qa < it.q1; qa += SK_QCH) {
    const int nq = min(SK_QCH, it.q1 - qa);
    for (int e = tid; e < nq * dh8; e += SK_COMPUTE_THREADS) {
      const int i = e / dh8, d = (e % dh8) * 8;
      const uint4 u = __ldcg(reinterpret_cast<const uint4*>(a.q + static_cast<size_t>(qa + i) * D + it.h * dh + d));
      const __nv_bfloat162* b2 = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float2 f = __bfloat1622float2(b2[j]);
        s.q[i * dh + d + 2 * j] = f.x * qscale;
        s.q[i * dh + d + 2 * j + 1] = f.y * qscale;
      }
    }
    named_bar(kBarCompute, SK_COMPUTE_THREADS);
    if (t0 && !t1) t1 = globaltimer_ns();
    // scores of this warp's keys for every query of the chunk
    float mx[SK_QCH];
#pragma unroll
    for (int i = 0; i < SK_QCH; ++i) mx[i] = -INFINITY;
    for (int key = k0 + lane; key < k1; key += 32) {
      float acc[SK_QCH];
#pragma unroll
      for (int i = 0; i < SK_QCH; ++i) acc[i] = 0.f;
      const bf16* kr = s.k + key * dh;
      for (int d = 0; d < dh; d += 8) {
        const uint4 raw = *reinterpret_cast<const uint4*>(kr + d);
        const __nv_bfloat162* k2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
        const float2 f0 = __bfloat1622float2(k2[0]), f1 = __bfloat1622float2(k2[1]);
        const float2 f2 = __bfloat1622float2(k2[2]), f3 = __bfloat1622float2(k2[3]);
#pragma unroll
        for (int i = 0; i < SK_QCH; ++i) {
          if (i < nq) {
            const float4 qa4 = *reinterpret_cast<const float4*>(s.q + i * dh + d);
            const float4 qb4 = *reinterpret_cast<const float4*>(s.q + i * dh + d + 4);
            acc[i] += qa4.x * f0.x + qa4.y * f0.y + qa4.z * f1.x + qa4.w * f1.y + qb4.x * f2.x + qb4.y * f2.y +
                      qb4.z * f3.x + qb4.w * f3.y;
          }
        }
      }
#pragma unroll
      for (int i = 0; i < SK_QCH; ++i) {
        if (i < nq) {
          s.p[i * N + key] = acc[i];
          mx[i] = fmaxf(mx[i], acc[i]);
        }
      }
    }
#pragma unroll
    for (int i = 0; i < SK_QCH; ++i) {
      mx[i] = warp_max(mx[i]);
      if (lane == 0 && i < nq) s.ml[(cw * SK_QCH + i) * 2] = mx[i];
    }
    named_bar(kBarCompute, SK_COMPUTE_THREADS);
    const uint64_t ts = (t0 && qa == it.q0) ? globaltimer_ns() : 0;
    if (ts) sk_trace_add(c, 4, 2, ts - t1);
    // block max per query; probabilities of this warp's keys and their sum
    float m[SK_QCH], sum[SK_QCH];
#pragma unroll
    for (int i = 0; i < SK_QCH; ++i) {
      m[i] = -INFINITY;
      sum[i] = 0.f;
      if (i < nq)
        for (int w = 0; w < SK_CWARPS; ++w) m[i] = fmaxf(m[i], s.ml[(w * SK_QCH + i) * 2]);
    }
    for (int key = k0 + lane; key < k1; key += 32) {
#pragma unroll
      for (int i = 0; i < SK_QCH; ++i) {
        if (i < nq) {
          const float pe = exp2f(s.p[i * N + key] - m[i]);
          s.p[i * N + key] = pe;
          sum[i] += pe;
        }
      }
    }
#pragma unroll
    for (int i = 0; i < SK_QCH; ++i) {
      sum[i] = warp_sum(sum[i]);
      if (lane == 0 && i < nq) s.ml[(cw * SK_QCH + i) * 2 + 1] = sum[i];
    }
    __syncwarp();
    // P V over this warp's keys, lanes own output dims
    float o[SK_QCH][4];
#pragma unroll
    for (int i = 0; i < SK_QCH; ++i)
#pragma unroll
      for (int cc = 0; cc < 4; ++cc) o[i][cc] = 0.f;
    for (int key = k0; key < k1; ++key) {
      const bf16* vr = s.v + key * dh;
      float vv[4];
#pragma unroll
      for (int cc = 0; cc < 4; ++cc) {
        const int d = lane + 32 * cc;
        vv[cc] = d < dh ? __bfloat162float(vr[d]) : 0.f;
      }
#pragma unroll
      for (int i = 0; i < SK_QCH; ++i) {
        if (i < nq) {
          const float pk = s.p[i * N + key];
#pragma unroll
          for (int cc = 0; cc < 4; ++cc) o[i][cc] += pk * vv[cc];
        }
      }
    }
#pragma unroll
    for (int i = 0; i < SK_QCH; ++i) {
      if (i < nq) {
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
          const int d = lane + 32 * cc;
          if (d < dh) s.o[(cw * SK_QCH + i) * dh + d] = o[i][cc];
        }
      }
    }
    named_bar(kBarCompute, SK_COMPUTE_THREADS);
    if (ts) sk_trace_add(c, 4, 3, globaltimer_ns() - ts);
    // O = sum_w o_w / sum_w l_w (every warp's partial is relative to the block max)
    for (int e = tid; e < nq * dh; e += SK_COMPUTE_THREADS) {
      const int i = e / dh, d = e % dh;
      float num = 0.f, den = 0.f;
      for (int w = 0; w < SK_CWARPS; ++w) {
        num += s.o[(w * SK_QCH + i) * dh + d];
        den += s.ml[(w * SK_QCH + i) * 2 + 1];
      }
      a.o[static_cast<size_t>(qa + i) * D + it.h * dh + d] = __float2bfloat16_rn(num / den);
    }
    named_bar(kBarCompute, SK_COMPUTE_THREADS);
  }
  fence_proxy_async_smem();  // generic writes to the region before later TMA writes to it
  if (t0) {
    const uint64_t t2 = globaltimer_ns();
    sk_trace_add(c, 4, 0, (t1 ? t1 : t2) - t0);
    sk_trace_add(c, 4, 1, t1 ? t2 - t1 : 0);
    sk_trace_add(c, 4, 7, 1);
  }
}

__global__ void __launch_bounds__(SK_THREADS, 1) stream_layers_kernel(const __grid_constant__ StreamArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int RS = a.ring_stages;
  uint8_t* reg = smem + static_cast<size_t>(RS) * SK_STAGE;
  uint8_t* misc = reg + a.region_bytes;
  SkCtx c;
  c.a = &a;
  c.ring = smem_u32(smem);
  c.reg = smem_u32(reg);
  c.reg_ptr = reg;
  c.bars = smem_u32(misc);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc + 1024);
  c.sh = reinterpret_cast<volatile int*>(misc + 1040);
  c.red = reinterpret_cast<float*>(misc + 1088);
  c.c_pos = 0;
  c.acc_phase = c.b_phase = c.kv_phase = 0;
  c.epoch = 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < RS; ++s) {
      mbar_init(full_bar(c, s), 1);
      mbar_init(empty_bar(c, s), 1);
    }
    mbar_init(acc_bar(c), 1);
    mbar_init(b_bar(c), 1);
    mbar_init(kv_bar(c), 1);
    fence_mbar_init();
    c.sh[0] = 1;
    c.sh[1] = 0;
    c.sh[2] = 0;
    c.sh[4] = 0;
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), SK_PROWS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  c.tmem = *tmem_slot;
  c.M = a.cu_rows[a.SV];
  c.passes = (c.M + SK_PROWS - 1) / SK_PROWS;
  c.passes_max = (a.M_max + SK_PROWS - 1) / SK_PROWS;

  if (c.M > 0) {
    if (warp == 0) {
      if (lane == 0) {
        const uint32_t issued = sk_producer(c);
        // every issued stage must land before the CTA leaves (on abort some were never
        // consumed): wait for the last ring-full of them
        const uint32_t first = issued > static_cast<uint32_t>(RS) ? issued - RS : 0u;
        for (uint32_t pos = first; pos < issued; ++pos)
          mbar_wait(full_bar(c, static_cast<int>(pos % RS)), (pos / RS) & 1u);
      }
      __syncwarp();
    } else {
      const int items = sk_att_items(a);
      const int G = static_cast<int>(gridDim.x);
      // LN1 of layer 0 (the rows were gathered by the previous kernel)
      if (warp >= 2) sk_row_stage(c, 0, nullptr, a.layers[0].ln1g, a.layers[0].ln1b, a.xn, false);
      bool ok = sk_grid_sync(c);
      for (int l = 0; ok && l < a.L; ++l) {
        const LayerParams& lp = a.layers[l];
        sk_gemm_stage(c, l, kSkQKV);
        // the operand region is free: fetch the cached K/V of this CTA's first attention
        // item (the condition depends on device data every thread reads alike)
        bool kv_pending = false;
        if (static_cast<int>(blockIdx.x) < items) {
          const AttItem it = sk_att_item(a, blockIdx.x);
          kv_pending = it.q1 > it.q0;
          if (kv_pending && warp == 1 && lane == 0) sk_prefetch_kv(c, l, it);
        }
        ok = sk_grid_sync(c);
        for (int item = blockIdx.x; item < items; item += G) {
          const AttItem it = sk_att_item(a, item);
          if (it.q1 <= it.q0) continue;
          if (!(item == static_cast<int>(blockIdx.x) && kv_pending)) {
            if (!ok) continue;
            named_bar(kBarAll, SK_SYNC_THREADS);  // the region is free (previous item done)
            if (warp == 1 && lane == 0) sk_prefetch_kv(c, l, it);
          }
          kv_pending = false;
          // a copy is in flight for this item: run it, or on abort only let it land
          if (warp >= 2) {
            if (ok)
              sk_att_item_run(c, l, it);
            else
              mbar_wait(kv_bar(c), c.kv_phase);
          }
          c.kv_phase ^= 1u;
        }
        if (!ok || !sk_grid_sync(c)) break;
        sk_gemm_stage(c, l, kSkOut);
        if (!sk_grid_sync(c)) break;
        if (warp >= 2) sk_row_stage(c, a.splits[kSkOut], lp.bo, lp.ln2g, lp.ln2b, a.xn, false);
        if (!sk_grid_sync(c)) break;
        sk_gemm_stage(c, l, kSkUp);
        if (!sk_grid_sync(c)) break;
        sk_gemm_stage(c, l, kSkDown);
        if (!sk_grid_sync(c)) break;
        if (warp >= 2) {
          if (l + 1 < a.L)
            sk_row_stage(c, a.splits[kSkDown], lp.b2, a.layers[l + 1].ln1g, a.layers[l + 1].ln1b, a.xn, false);
          else
            sk_row_stage(c, a.splits[kSkDown], lp.b2, a.lnfg, a.lnfb, a.tok_out, true);  // final LN
        }
        if (l + 1 < a.L) ok = sk_grid_sync(c);
      }
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(c.tmem, SK_PROWS);
  }
}

}  // namespace

int stream_task_kblocks(int k, int splits) { return ((k + SK_BK - 1) / SK_BK + splits - 1) / splits; }

size_t stream_region_bytes(int max_task_kblocks, int n_tok, int head_dim) {
  const size_t gemm = static_cast<size_t>(max_task_kblocks) * SK_BBLK;
  const size_t kv = (static_cast<size_t>(n_tok) * head_dim * 2 + 127) & ~static_cast<size_t>(127);
  const size_t att = 2 * kv + 4 * (static_cast<size_t>(SK_QCH) * head_dim + static_cast<size_t>(SK_QCH) * n_tok +
                                   static_cast<size_t>(SK_CWARPS) * SK_QCH * 2 +
                                   static_cast<size_t>(SK_CWARPS) * SK_QCH * head_dim);
  return (std::max(gemm, att) + 1023) & ~static_cast<size_t>(1023);
}

size_t stream_smem_bytes(int ring_stages, size_t region) {
  return 1024 + static_cast<size_t>(ring_stages) * SK_STAGE + region + SK_MISC;
}

int stream_ring_stages_for(size_t smem_limit, size_t region) {
  const long long room = static_cast<long long>(smem_limit) - 1024 - static_cast<long long>(region) - SK_MISC;
  return static_cast<int>(std::min<long long>(room / SK_STAGE, 16));
}

int stream_max_dim() { return 4 * SK_COMPUTE_THREADS * SK_ROW_F4; }

int stream_rows_per_pass() { return SK_PROWS; }

cudaError_t stream_setup(size_t smem) {
  return cudaFuncSetAttribute(stream_layers_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
}

int stream_max_ctas(size_t smem) {
  int per_sm = 0, dev = 0, sms = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, stream_layers_kernel, SK_THREADS, smem) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return per_sm * sms;
}

cudaError_t launch_stream(const StreamArgs& a, int grid, size_t smem, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(SK_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, stream_layers_kernel, a);
}

}  // namespace ivit
