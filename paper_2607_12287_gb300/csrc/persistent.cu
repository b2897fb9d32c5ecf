// Persistent encoder for small updated-row counts: every transformer block of an
// incremental step (Sec. III-B: Eq. 4 projections, Eq. 5 cache scatter, attention of
// the updated queries over all tokens, MLP) in one cooperative launch.
//
// With a few dozen updated rows the step is a weight-streaming problem whose time is
// set by the dependent chain of small operations, not by bandwidth; launching one kernel
// per operation pays a launch, a prologue and a teardown for each of them.  Here one CTA
// per SM walks the phases of every layer, separated by a grid barrier:
//
//   QKV partials | QKV reduce (+bias -> Q, K/V cache rows) | attention |
//   out-proj partials | reduce (+bias +residual) + LN2 | MLP-up partials |
//   reduce (+bias, GELU) | MLP-down partials | reduce (+bias +residual) + next LN1
//
// GEMM phases split K over the CTAs (fp32 partial tiles in L2, summed in split order in
// the following phase: deterministic).  Weights do not depend on activations, so before
// every barrier each CTA issues the TMA loads of the weight stages of its next GEMM
// item; the weight stream overlaps the barriers and the non-GEMM phases.  Stage
// barriers take two arrivals: one with the weight bytes (early), one with the
// activation bytes (after the barrier that makes the activations visible).
//
// Roles inside a CTA (256 threads): warp 0 lane 0 issues TMA, warp 1 lane 0 issues
// tcgen05.mma into a TMEM accumulator, warps 4..7 drain it (tcgen05.ld); every warp works
// in the element-wise, row-wise and attention phases.  All waits are bounded; a CTA
// whose barrier or stage wait expires records an error, drains its copies and exits.
#include "internal.h"
#include "ptx.cuh"

namespace ivit {
namespace {

constexpr int PT_THREADS = 256;
constexpr int PT_WARPS = PT_THREADS / 32;
constexpr int PT_BM = 128;                       // output features per tile (MMA M)
constexpr int PT_BN = 64;                        // updated rows per row tile (MMA N <= 64)
constexpr int PT_BK = 64;                        // K per stage
constexpr int PT_STAGES = 5;
constexpr int PT_W_BYTES = PT_BM * PT_BK * 2;    // 16 KB
constexpr int PT_XBOX = 32;
constexpr int PT_XBOX_BYTES = PT_XBOX * PT_BK * 2;
constexpr int PT_STAGE_BYTES = PT_W_BYTES + PT_BN * PT_BK * 2;
constexpr int PT_RING_BYTES = PT_STAGES * PT_STAGE_BYTES;
constexpr int PT_MISC_BYTES = 1024;
constexpr int PT_QPI = PT_WARPS;                 // queries per attention item (one per warp)
constexpr int PT_MAX_SPLITS = 16;

enum GemmId : int { kQKV = 0, kOut = 1, kUp = 2, kDown = 3 };

struct Shape {
  int n_out, k, n_ft, n_tt, n_kb, tiles, splits, items;
};

__device__ __forceinline__ Shape gemm_shape(const PersistentArgs& a, int g, int M) {
  Shape s;
  s.n_out = g == kQKV ? 3 * a.D : (g == kUp ? a.F : a.D);
  s.k = g == kDown ? a.F : a.D;
  s.n_ft = (s.n_out + PT_BM - 1) / PT_BM;
  s.n_tt = (M + PT_BN - 1) / PT_BN;
  s.n_kb = (s.k + PT_BK - 1) / PT_BK;
  s.tiles = s.n_ft * s.n_tt;
  s.splits = max(1, min(min(PT_MAX_SPLITS, s.n_kb), static_cast<int>(gridDim.x) / max(1, s.tiles)));
  s.items = s.tiles * s.splits;
  return s;
}

__device__ __forceinline__ float gelu_f(float x, int mode) {
  if (mode == 1) return 0.5f * x * (1.f + erff(x * 0.70710678118654752f));
  const float c = 0.79788456080286536f;  // sqrt(2/pi)
  return 0.5f * x * (1.f + tanhf(c * (x + 0.044715f * x * x * x)));
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

// Sum over the CTA (all threads must call); red = PT_WARPS floats of shared memory.
__device__ __forceinline__ float block_sum(float v, float* red) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[w] = v;
  __syncthreads();
  float t = lane < PT_WARPS ? red[lane] : 0.f;
  return warp_sum(t);
}

struct Ctx {
  const PersistentArgs* a;
  uint8_t* smem;
  uint32_t smem_base, bar_base;
  uint32_t tmem;
  int M;
  volatile int* sh;  // [0] barrier ok, [1] abort
  float* red;        // block-reduction scratch
  // producer state (warp 0 lane 0)
  uint32_t p_stage, p_phase;
  int pre_n, pre_stage0;  // stages prefetched for the next GEMM item
  uint32_t pre_parity0;   // ring parity of the first prefetched stage
  // MMA state (warp 1 lane 0)
  uint32_t c_stage, c_phase;
  // epilogue state (warps 4..7)
  uint32_t acc_phase;
  // attention tile (warp 0 lane 0 issues, every thread waits)
  uint32_t kv_phase;
  int kv_item;      // attention item whose K/V tile is in flight or resident (-1: none)
  unsigned epoch;   // grid barriers passed (thread 0)
};

__device__ __forceinline__ uint32_t full_bar(const Ctx& c, int s) { return c.bar_base + 8 * s; }
__device__ __forceinline__ uint32_t empty_bar(const Ctx& c, int s) {
  return c.bar_base + 8 * (PT_STAGES + s);
}
__device__ __forceinline__ uint32_t acc_bar(const Ctx& c) { return c.bar_base + 8 * (2 * PT_STAGES); }
__device__ __forceinline__ uint32_t kv_bar(const Ctx& c) { return c.bar_base + 8 * (2 * PT_STAGES + 1); }

__device__ __forceinline__ const CUtensorMap* wmap(const PersistentArgs& a, int l, int g) {
  return a.wmaps + 4 * l + g;
}
__device__ __forceinline__ const CUtensorMap* xmap(const PersistentArgs& a, int g) {
  return a.xmaps + (g == kQKV || g == kUp ? 0 : (g == kOut ? 1 : 2));
}

// Grid barrier on a monotonic arrival counter (zeroed before the launch): the k-th
// barrier of the kernel completes when the counter reaches k * gridDim.x.  One
// acquire-release atomic per CTA, then an acquire spin; bounded, and it gives up early
// when another CTA raised the abort flag.  False when it expired or was aborted.
__device__ bool grid_sync(Ctx& c) {
  const PersistentArgs& a = *c.a;
  __syncthreads();
  if (threadIdx.x == 0) {
    ++c.epoch;
    const unsigned target = c.epoch * gridDim.x;
    unsigned* count = a.gbar;
    unsigned* abort_flag = a.gbar + 2;
    atom_add_acq_rel_u32(count, 1u);
    bool ok = true;
    const uint64_t t0 = globaltimer_ns();
    while (ld_acquire_u32(count) < target) {
      if (ld_acquire_u32(abort_flag) != 0 || globaltimer_ns() - t0 > kWaitLimitNs) {
        atomicExch(a.err, kErrGridBarrier);
        atomicExch(abort_flag, 1u);
        ok = false;
        break;
      }
    }
    c.sh[0] = ok ? 1 : 0;
    if (a.trace && blockIdx.x == 0) a.trace[1 + a.trace[0]++] = globaltimer_ns();
  }
  __syncthreads();
  return c.sh[0] != 0;
}

// Producer: weight stages of this CTA's first item of GEMM (l, g), issued ahead of the
// barrier that publishes the activations.  One arrival per stage (weight bytes).
__device__ void prefetch_weights(Ctx& c, int l, int g) {
  c.pre_n = 0;
  if (l >= c.a->L) return;
  const Shape s = gemm_shape(*c.a, g, c.M);
  const int item = blockIdx.x;
  if (item >= s.items) return;
  const int t = item % s.tiles, sp = item / s.tiles, ft = t % s.n_ft;
  const int kb0 = sp * s.n_kb / s.splits, kb1 = (sp + 1) * s.n_kb / s.splits;
  const int n = min(PT_STAGES, kb1 - kb0);
  c.pre_stage0 = c.p_stage;
  c.pre_parity0 = c.p_phase;
  for (int i = 0; i < n; ++i) {
    if (!mbar_wait(empty_bar(c, c.p_stage), c.p_phase ^ 1)) {
      atomicExch(c.a->err, kErrWaitSlotEmpty);
      c.sh[1] = 1;
      break;
    }
    const uint32_t st = c.smem_base + c.p_stage * PT_STAGE_BYTES;
    mbar_arrive_expect_tx(full_bar(c, c.p_stage), PT_W_BYTES);
    tma_load_2d(st, wmap(*c.a, l, g), (kb0 + i) * PT_BK, ft * PT_BM, full_bar(c, c.p_stage),
                l2_policy_evict_first());
    ++c.pre_n;
    if (++c.p_stage == PT_STAGES) {
      c.p_stage = 0;
      c.p_phase ^= 1;
    }
  }
}

// On abort: complete every prefetched stage without activation bytes and wait for the
// weight copies already in flight, so none lands after the CTA has left.
__device__ void drain_prefetch(Ctx& c) {
  for (int i = 0; i < c.pre_n; ++i) {
    const int st = (c.pre_stage0 + i) % PT_STAGES;
    const uint32_t parity = c.pre_parity0 ^ static_cast<uint32_t>(((c.pre_stage0 + i) / PT_STAGES) & 1);
    mbar_arrive(full_bar(c, st));
    mbar_wait(full_bar(c, st), parity);
  }
  c.pre_n = 0;
}

// One GEMM phase: every item of this CTA (feature tile x row tile x K split) writes its
// fp32 partial tile [rows][128] to part[item].
__device__ void gemm_phase(Ctx& c, int l, int g) {
  const PersistentArgs& a = *c.a;
  const Shape s = gemm_shape(a, g, c.M);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const CUtensorMap* wm = wmap(a, l, g);
  const CUtensorMap* xm = xmap(a, g);
  for (int item = blockIdx.x; item < s.items; item += gridDim.x) {
    const int t = item % s.tiles, sp = item / s.tiles;
    const int ft = t % s.n_ft, tt = t / s.n_ft;
    const int kb0 = sp * s.n_kb / s.splits, kb1 = (sp + 1) * s.n_kb / s.splits;
    const int row0 = tt * PT_BN;
    const int rows = min(PT_BN, c.M - row0);
    const int n_mma = (rows + 15) & ~15;
    const int nbox = (n_mma + PT_XBOX - 1) / PT_XBOX;
    const bool first = item == static_cast<int>(blockIdx.x);
    const bool item_ok = c.sh[1] == 0;  // uniform: read after the previous __syncthreads
    if (!item_ok) break;
    if (warp == 0 && lane == 0) {
      fence_proxy_async_global();
      const uint64_t pol_w = l2_policy_evict_first(), pol_x = l2_policy_evict_last();
      int pre_st = c.pre_stage0;
      for (int kb = kb0; kb < kb1; ++kb) {
        uint32_t st_idx;
        if (first && kb - kb0 < c.pre_n) {
          st_idx = pre_st;
          pre_st = pre_st + 1 == PT_STAGES ? 0 : pre_st + 1;
        } else {
          if (!mbar_wait(empty_bar(c, c.p_stage), c.p_phase ^ 1)) {
            atomicExch(a.err, kErrWaitSlotEmpty);
            c.sh[1] = 1;
            break;
          }
          st_idx = c.p_stage;
          mbar_arrive_expect_tx(full_bar(c, st_idx), PT_W_BYTES);
          tma_load_2d(c.smem_base + st_idx * PT_STAGE_BYTES, wm, kb * PT_BK, ft * PT_BM,
                      full_bar(c, st_idx), pol_w);
          if (++c.p_stage == PT_STAGES) {
            c.p_stage = 0;
            c.p_phase ^= 1;
          }
        }
        const uint32_t st = c.smem_base + st_idx * PT_STAGE_BYTES;
        mbar_arrive_expect_tx(full_bar(c, st_idx), nbox * PT_XBOX_BYTES);
        for (int b = 0; b < nbox; ++b)
          tma_load_2d(st + PT_W_BYTES + b * PT_XBOX_BYTES, xm, kb * PT_BK, row0 + b * PT_XBOX,
                      full_bar(c, st_idx), pol_x);
      }
      if (first) c.pre_n = 0;
    } else if (warp == 1 && lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(PT_BM, n_mma);
      for (int kb = kb0; kb < kb1; ++kb) {
        if (!mbar_wait(full_bar(c, c.c_stage), c.c_phase)) {
          atomicExch(a.err, kErrWaitTmaFull);
          c.sh[1] = 1;
          break;
        }
        tc_fence_after();
        const uint32_t st = c.smem_base + c.c_stage * PT_STAGE_BYTES;
#pragma unroll
        for (int k = 0; k < PT_BK / 16; ++k)
          umma_bf16(c.tmem, sdesc_kmajor_sw128(st + k * 32), sdesc_kmajor_sw128(st + PT_W_BYTES + k * 32),
                    idesc, (kb > kb0 || k > 0) ? 1u : 0u);
        umma_commit(empty_bar(c, c.c_stage));
        if (++c.c_stage == PT_STAGES) {
          c.c_stage = 0;
          c.c_phase ^= 1;
        }
      }
      umma_commit(acc_bar(c));
    } else if (warp >= 4) {
      if (!mbar_wait(acc_bar(c), c.acc_phase)) {
        atomicExch(a.err, kErrWaitAccum);
        c.sh[1] = 1;
      }
      tc_fence_after();
      if (c.sh[1] == 0) {
        const int fl = (warp - 4) * 32 + lane;
        float* part = a.part + static_cast<size_t>(item) * (PT_BN * PT_BM);
        const uint32_t trow = c.tmem + (static_cast<uint32_t>((warp - 4) * 32) << 16);
        for (int c0 = 0; c0 < rows; c0 += 16) {
          float v[16];
          tmem_ld16(trow + c0, v);
#pragma unroll
          for (int j = 0; j < 16; ++j)
            if (c0 + j < rows) __stcg(part + (c0 + j) * PT_BM + fl, v[j]);
        }
      }
      tc_fence_before();
    }
    c.acc_phase ^= 1;
    __syncwarp();
    __syncthreads();  // TMEM drained before the next item's MMAs
  }
}

// Sum of the K-split partials of output (r, f..f+3) of GEMM shape s, in split order.
// Loads are issued in batches of 4 splits before their adds (one L2 round trip per
// batch, not per split).

__device__ __forceinline__ float4 sum_partials(const PersistentArgs& a, const Shape& s, int r, int f) {
  const int ft = f / PT_BM, tt = r / PT_BN;
  const int t = ft + tt * s.n_ft;
  const float* base = a.part + static_cast<size_t>(t) * (PT_BN * PT_BM) +
                      static_cast<size_t>(r - tt * PT_BN) * PT_BM + (f - ft * PT_BM);
  const size_t stride = static_cast<size_t>(s.tiles) * (PT_BN * PT_BM);
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int s0 = 0; s0 < s.splits; s0 += 4) {  // batches of 4 loads in flight
    float4 p[4];
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (s0 + u < s.splits) p[u] = __ldcg(reinterpret_cast<const float4*>(base + (s0 + u) * stride));
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (s0 + u < s.splits) {
        acc.x += p[u].x;
        acc.y += p[u].y;
        acc.z += p[u].z;
        acc.w += p[u].w;
      }
    }
  }
  return acc;
}

// QKV reduce: + bias; queries to q (packed rows), keys and values to this layer's cache
// at the updated tokens' rows (Eq. 5).
__device__ void qkv_reduce_phase(Ctx& c, int l) {
  const PersistentArgs& a = *c.a;
  const Shape s = gemm_shape(a, kQKV, c.M);
  const int D = a.D, n4 = 3 * D / 4;
  const LayerParams& lp = a.layers[l];
  bf16* ck = a.cacheK + static_cast<size_t>(l) * a.M_max * D;
  bf16* cv = a.cacheV + static_cast<size_t>(l) * a.M_max * D;
  const long long total = static_cast<long long>(c.M) * n4;
  for (long long e = blockIdx.x * static_cast<long long>(PT_THREADS) + threadIdx.x; e < total;
       e += static_cast<long long>(gridDim.x) * PT_THREADS) {
    const int r = static_cast<int>(e / n4), f = static_cast<int>(e % n4) * 4;
    const float4 y = sum_partials(a, s, r, f);
    const float4 b = *reinterpret_cast<const float4*>(lp.bqkv + f);
    __nv_bfloat162 v2[2] = {__floats2bfloat162_rn(y.x + b.x, y.y + b.y),
                            __floats2bfloat162_rn(y.z + b.z, y.w + b.w)};
    bf16* dst;
    if (f < D) {
      dst = a.q + static_cast<size_t>(r) * D + f;
    } else {
      const size_t tok = static_cast<size_t>(a.rowtok[r]);
      dst = f < 2 * D ? ck + tok * D + (f - D) : cv + tok * D + (f - 2 * D);
    }
    *reinterpret_cast<uint2*>(dst) = *reinterpret_cast<const uint2*>(v2);
  }
}

// Attention items: (view, head, chunk of PT_QPI updated queries), enumerated view by
// view; item i is handled by CTA i, i + grid, ...
__device__ __forceinline__ int attention_items(const PersistentArgs& a) {
  int n = 0;
  for (int v = 0; v < a.SV; ++v) n += (a.cu_rows[v + 1] - a.cu_rows[v] + PT_QPI - 1) / PT_QPI;
  return n * a.H;
}

// (view, head, first query row) of an attention item.
__device__ __forceinline__ void attention_item(const PersistentArgs& a, int item, int& v, int& h, int& q0) {
  h = item % a.H;
  int j = item / a.H;
  for (v = 0; v < a.SV; ++v) {
    const int nqb = (a.cu_rows[v + 1] - a.cu_rows[v] + PT_QPI - 1) / PT_QPI;
    if (j < nqb) break;
    j -= nqb;
  }
  q0 = a.cu_rows[v] + j * PT_QPI;
}

__device__ __forceinline__ uint8_t* attention_smem(const Ctx& c) {
  return c.smem + PT_RING_BYTES + PT_MISC_BYTES;
}

// Warp 0 lane 0: TMA of the cached keys and values of (view, head) of layer l, [N][dh]
// each, into the attention region.  Reused tokens' rows are final before the layer
// runs; the rows of this call's updated tokens are read again after the QKV reduce.
__device__ void prefetch_kv(Ctx& c, int l, int item) {
  const PersistentArgs& a = *c.a;
  c.kv_item = -1;
  if (l >= a.L || item >= attention_items(a)) return;
  int v, h, q0;
  attention_item(a, item, v, h, q0);
  uint8_t* base = attention_smem(c);
  const uint32_t tile = static_cast<uint32_t>(a.N) * a.dh * 2;
  mbar_arrive_expect_tx(kv_bar(c), 2 * tile);
  tma_load_2d(smem_u32(base), a.kvmaps + 2 * l, h * a.dh, v * a.N, kv_bar(c), l2_policy_evict_first());
  tma_load_2d(smem_u32(base + tile), a.kvmaps + 2 * l + 1, h * a.dh, v * a.N, kv_bar(c),
              l2_policy_evict_first());
  c.kv_item = item;
}

// Attention of a chunk of updated queries over all N tokens of their view, one warp per
// query: softmax(q K^T / sqrt(dh)) V with the key/value tile resident in shared memory
// (bf16, [N][dh]); lanes own keys for the scores and output dims for P V; fp32 softmax.
__device__ void attention_phase(Ctx& c, int l) {
  const PersistentArgs& a = *c.a;
  const int N = a.N, D = a.D, dh = a.dh;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint8_t* base = attention_smem(c);
  bf16* sk = reinterpret_cast<bf16*>(base);                              // [N][dh]
  bf16* sv = sk + static_cast<size_t>(N) * dh;                           // [N][dh]
  float* sq = reinterpret_cast<float*>(sv + static_cast<size_t>(N) * dh);  // [QPI][dh]
  float* sp = sq + PT_QPI * dh;                                          // [QPI][N]
  const bf16* ck = a.cacheK + static_cast<size_t>(l) * a.M_max * D;
  const bf16* cv = a.cacheV + static_cast<size_t>(l) * a.M_max * D;
  const int dh8 = dh / 8;
  const float scale = rsqrtf(static_cast<float>(dh));
  const int n_items = attention_items(a);
  for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
    int v, h, q0;
    attention_item(a, item, v, h, q0);
    const int r0 = a.cu_rows[v], r1 = a.cu_rows[v + 1];
    const int nq = min(PT_QPI, r1 - q0);
    __syncthreads();
    if (threadIdx.x == 0 && c.kv_item != item) prefetch_kv(c, l, item);  // not prefetched
    if (!mbar_wait(kv_bar(c), c.kv_phase)) {
      atomicExch(a.err, kErrWaitTmaFull);
      c.sh[1] = 1;
    }
    c.kv_phase ^= 1;
    __syncthreads();
    if (c.sh[1] != 0) return;
    // this call's updated keys/values of the view (reduced by the previous phase)
    const size_t vbase = static_cast<size_t>(v) * N;
    for (int e = threadIdx.x; e < (r1 - r0) * dh8; e += PT_THREADS) {
      const int tok = a.rowtok[r0 + e / dh8], d = (e % dh8) * 8;
      const size_t g = static_cast<size_t>(tok) * D + h * dh + d;
      const int key = tok - static_cast<int>(vbase);
      *reinterpret_cast<uint4*>(sk + key * dh + d) = __ldcg(reinterpret_cast<const uint4*>(ck + g));
      *reinterpret_cast<uint4*>(sv + key * dh + d) = __ldcg(reinterpret_cast<const uint4*>(cv + g));
    }
    for (int e = threadIdx.x; e < nq * dh8; e += PT_THREADS) {
      const int qi = e / dh8, d = (e % dh8) * 8;
      const uint4 u = __ldcg(reinterpret_cast<const uint4*>(a.q + static_cast<size_t>(q0 + qi) * D + h * dh + d));
      const __nv_bfloat162* b2 = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(b2[i]);
        sq[qi * dh + d + 2 * i] = f.x * scale;
        sq[qi * dh + d + 2 * i + 1] = f.y * scale;
      }
    }
    __syncthreads();
    if (warp < nq) {
      const float* qr = sq + warp * dh;
      float* pr = sp + warp * N;
      float sc[8];
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) sc[kk] = 0.f;
      for (int d = 0; d < dh; d += 8) {
        const float4 lo = *reinterpret_cast<const float4*>(qr + d);
        const float4 hi = *reinterpret_cast<const float4*>(qr + d + 4);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const int key = lane + 32 * kk;
          if (key < N) {
            const uint4 raw = *reinterpret_cast<const uint4*>(sk + key * dh + d);
            const __nv_bfloat162* k2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
            const float2 f0 = __bfloat1622float2(k2[0]), f1 = __bfloat1622float2(k2[1]);
            const float2 f2 = __bfloat1622float2(k2[2]), f3 = __bfloat1622float2(k2[3]);
            sc[kk] += lo.x * f0.x + lo.y * f0.y + lo.z * f1.x + lo.w * f1.y + hi.x * f2.x + hi.y * f2.y +
                      hi.z * f3.x + hi.w * f3.y;
          }
        }
      }
      float mx = -INFINITY;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk)
        if (lane + 32 * kk < N) mx = fmaxf(mx, sc[kk]);
      mx = warp_max(mx);
      float sum = 0.f;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const int key = lane + 32 * kk;
        if (key < N) {
          const float p = __expf(sc[kk] - mx);
          pr[key] = p;
          sum += p;
        }
      }
      const float inv = 1.f / warp_sum(sum);
      __syncwarp();
      float o[4] = {0.f, 0.f, 0.f, 0.f};
      for (int key = 0; key < N; ++key) {
        const float p = pr[key];
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
          const int d = lane + 32 * cc;
          if (d < dh) o[cc] += p * __bfloat162float(sv[key * dh + d]);
        }
      }
      bf16* orow = a.o + static_cast<size_t>(q0 + warp) * D + h * dh;
#pragma unroll
      for (int cc = 0; cc < 4; ++cc) {
        const int d = lane + 32 * cc;
        if (d < dh) orow[d] = __float2bfloat16_rn(o[cc] * inv);
      }
    }
  }
  // the region is free: start the next layer's tile of this CTA's first item
  __syncthreads();
  if (threadIdx.x == 0) prefetch_kv(c, l + 1, blockIdx.x);
}

// Row-wise: x[r] += (sum of partials + bias) when s is given, then layer norm of x[r]
// into dst (row r, or row rowtok[r] when scatter).  One CTA per row.
__device__ void row_phase(Ctx& c, const Shape* s, const float* bias, const float* gamma,
                          const float* beta, bf16* dst, bool scatter) {
  const PersistentArgs& a = *c.a;
  const int D = a.D, n4 = D / 4;
  constexpr int PER = 2;  // float4 chunks per thread (D <= 2048)
  for (int r = blockIdx.x; r < c.M; r += gridDim.x) {
    float4* xr = reinterpret_cast<float4*>(a.x + static_cast<size_t>(r) * D);
    float4 v[PER];
    float sum = 0.f;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int ch = threadIdx.x + PT_THREADS * i;
      v[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (ch < n4) {
        float4 xv = __ldcg(xr + ch);
        if (s) {
          const float4 y = sum_partials(a, *s, r, 4 * ch);
          const float4 b = reinterpret_cast<const float4*>(bias)[ch];
          xv.x += y.x + b.x;
          xv.y += y.y + b.y;
          xv.z += y.z + b.z;
          xv.w += y.w + b.w;
          __stcg(xr + ch, xv);
        }
        v[i] = xv;
        sum += (xv.x + xv.y) + (xv.z + xv.w);
      }
    }
    const float mean = block_sum(sum, c.red) / D;
    float sq = 0.f;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      if (threadIdx.x + PT_THREADS * i < n4) {
        const float p = v[i].x - mean, q = v[i].y - mean, u = v[i].z - mean, w = v[i].w - mean;
        sq += (p * p + q * q) + (u * u + w * w);
      }
    }
    const float rstd = rsqrtf(block_sum(sq, c.red) / D + a.eps);
    const size_t orow = scatter ? static_cast<size_t>(a.rowtok[r]) : static_cast<size_t>(r);
    __nv_bfloat162* yr = reinterpret_cast<__nv_bfloat162*>(dst + orow * D);
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int ch = threadIdx.x + PT_THREADS * i;
      if (ch < n4) {
        const float4 g = reinterpret_cast<const float4*>(gamma)[ch];
        const float4 b = reinterpret_cast<const float4*>(beta)[ch];
        yr[2 * ch] = __floats2bfloat162_rn(g.x * (v[i].x - mean) * rstd + b.x, g.y * (v[i].y - mean) * rstd + b.y);
        yr[2 * ch + 1] =
            __floats2bfloat162_rn(g.z * (v[i].z - mean) * rstd + b.z, g.w * (v[i].w - mean) * rstd + b.w);
      }
    }
  }
}

// MLP-up reduce: h = GELU(sum of partials + bias) in bf16.
__device__ void up_reduce_phase(Ctx& c, int l) {
  const PersistentArgs& a = *c.a;
  const Shape s = gemm_shape(a, kUp, c.M);
  const int F = a.F, n4 = F / 4;
  const float* b1 = a.layers[l].b1;
  const long long total = static_cast<long long>(c.M) * n4;
  for (long long e = blockIdx.x * static_cast<long long>(PT_THREADS) + threadIdx.x; e < total;
       e += static_cast<long long>(gridDim.x) * PT_THREADS) {
    const int r = static_cast<int>(e / n4), f = static_cast<int>(e % n4) * 4;
    const float4 y = sum_partials(a, s, r, f);
    const float4 b = *reinterpret_cast<const float4*>(b1 + f);
    __nv_bfloat162* dst = reinterpret_cast<__nv_bfloat162*>(a.h + static_cast<size_t>(r) * F + f);
    dst[0] = __floats2bfloat162_rn(gelu_f(y.x + b.x, a.gelu), gelu_f(y.y + b.y, a.gelu));
    dst[1] = __floats2bfloat162_rn(gelu_f(y.z + b.z, a.gelu), gelu_f(y.w + b.w, a.gelu));
  }
}

// True when this CTA may go on after a grid barrier; a CTA whose own stage or
// accumulator wait expired tells the others through the global abort flag.
__device__ __forceinline__ bool phase_ok(Ctx& c) {
  if (!grid_sync(c)) return false;
  if (c.sh[1] != 0) {
    if (threadIdx.x == 0) atomicExch(c.a->gbar + 2, 1u);
    return false;
  }
  return true;
}

__global__ void __launch_bounds__(PT_THREADS, 1)
    persistent_layers_kernel(const __grid_constant__ PersistentArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* misc = smem + PT_RING_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(misc);                 // 2*STAGES + 1
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * PT_STAGES + 1);
  Ctx c;
  c.a = &a;
  c.smem = smem;
  c.smem_base = smem_u32(smem);
  c.bar_base = smem_u32(bars);
  c.sh = reinterpret_cast<volatile int*>(tmem_slot + 2);
  c.red = reinterpret_cast<float*>(misc + 512);
  c.p_stage = c.p_phase = c.c_stage = c.c_phase = c.acc_phase = 0;
  c.pre_n = 0;
  c.pre_stage0 = 0;
  c.pre_parity0 = 0;
  c.kv_phase = 0;
  c.kv_item = -1;
  c.epoch = 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool producer = warp == 0 && lane == 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < PT_STAGES; ++s) {
      mbar_init(full_bar(c, s), 2);  // weight arrival + activation arrival
      mbar_init(empty_bar(c, s), 1);
    }
    mbar_init(acc_bar(c), 1);
    mbar_init(kv_bar(c), 1);
    fence_mbar_init();
    c.sh[0] = 1;
    c.sh[1] = 0;
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(tmem_slot), PT_BN);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  c.tmem = *tmem_slot;
  c.M = a.cu_rows[a.SV];
  if (a.trace && blockIdx.x == 0 && threadIdx.x == 0) {
    a.trace[0] = 0;
    a.trace[1 + a.trace[0]++] = globaltimer_ns();
  }

  bool ok = c.M > 0;
  if (ok) {
    if (producer) prefetch_weights(c, 0, kQKV);
    if (threadIdx.x == 0) prefetch_kv(c, 0, blockIdx.x);
    row_phase(c, nullptr, nullptr, a.layers[0].ln1g, a.layers[0].ln1b, a.xn, false);
    ok = phase_ok(c);
  }
  for (int l = 0; ok && l < a.L; ++l) {
    const LayerParams& lp = a.layers[l];
    gemm_phase(c, l, kQKV);
    if (producer) prefetch_weights(c, l, kOut);
    if (!(ok = phase_ok(c))) break;
    qkv_reduce_phase(c, l);
    if (!(ok = phase_ok(c))) break;
    attention_phase(c, l);
    if (!(ok = phase_ok(c))) break;
    gemm_phase(c, l, kOut);
    if (producer) prefetch_weights(c, l, kUp);
    if (!(ok = phase_ok(c))) break;
    {
      const Shape s = gemm_shape(a, kOut, c.M);
      row_phase(c, &s, lp.bo, lp.ln2g, lp.ln2b, a.xn, false);
    }
    if (!(ok = phase_ok(c))) break;
    gemm_phase(c, l, kUp);
    if (producer) prefetch_weights(c, l, kDown);
    if (!(ok = phase_ok(c))) break;
    up_reduce_phase(c, l);
    if (!(ok = phase_ok(c))) break;
    gemm_phase(c, l, kDown);
    if (producer) prefetch_weights(c, l + 1, kQKV);
    if (!(ok = phase_ok(c))) break;
    {
      const Shape s = gemm_shape(a, kDown, c.M);
      if (l + 1 < a.L)
        row_phase(c, &s, lp.b2, a.layers[l + 1].ln1g, a.layers[l + 1].ln1b, a.xn, false);
      else
        row_phase(c, &s, lp.b2, a.lnfg, a.lnfb, a.tok_out, true);  // final LN -> token cache
    }
    if (l + 1 < a.L && !(ok = phase_ok(c))) break;
  }
  if (!ok && producer) drain_prefetch(c);
  if (!ok && threadIdx.x == 0 && c.kv_item >= 0) mbar_wait(kv_bar(c), c.kv_phase);
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(c.tmem, PT_BN);
  }
}

}  // namespace

size_t persistent_smem_bytes(int n_tok, int head_dim) {
  // attention region: key and value tiles [N][dh] bf16, queries [QPI][dh] fp32,
  // probabilities [QPI][N] fp32
  const size_t attn = 2 * static_cast<size_t>(n_tok) * head_dim * sizeof(bf16) +
                      static_cast<size_t>(PT_QPI) * head_dim * sizeof(float) +
                      static_cast<size_t>(PT_QPI) * n_tok * sizeof(float);
  return 1024 + PT_RING_BYTES + PT_MISC_BYTES + attn;
}

size_t persistent_part_floats(int max_items) {
  return static_cast<size_t>(max_items) * PT_BN * PT_BM;
}

cudaError_t persistent_setup(size_t smem) {
  return cudaFuncSetAttribute(persistent_layers_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(smem));
}

int persistent_max_ctas(size_t smem) {
  int per_sm = 0, dev = 0, sms = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, persistent_layers_kernel, PT_THREADS, smem) !=
      cudaSuccess)
    return 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return per_sm * sms;
}

cudaError_t launch_persistent(const PersistentArgs& a, int grid, size_t smem, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(PT_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, persistent_layers_kernel, a);
}

}  // namespace ivit
