// Memory-bound kernels of the incremental encode: patchify, change score (Eq. 3),
// selection + stream compaction, gather of the updated rows, layer norm (with the
// final-token cache scatter), and attention of the updated queries over all tokens.
#include <cstdlib>
#include <cstring>

#include "internal.h"
#include "ptx.cuh"

namespace ivit {

bool g_use_pdl = true;
thread_local unsigned long long* g_stamp = nullptr;

namespace {

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

__device__ __forceinline__ bool is_cold(const ColdMask& m, int v) {
  return (m.bits[v >> 5] >> (v & 31)) & 1u;
}

// --------------------------------------------------------------------- patchify
// patches[v*N + i][(ky*P + kx)*3 + c] = frame[v][py*P + ky][px*P + kx][c] - 128 (exact in
// bf16).  When a patch row (P*3 bytes) has even length and the frames start at an even
// address, one thread per pair of adjacent columns: 2 bytes in, one bf16 pair out, so
// consecutive threads read and write contiguous runs; otherwise one thread per (token,
// ky) row with byte loads.  Columns P*P*3 .. kpad-1 stay zero (set once at allocation).
__global__ void patchify_kernel(const uint8_t* __restrict__ frames, bf16* __restrict__ patches,
                                int sv, int img_h, int img_w, int P, int kpad, unsigned long long* stamp) {
  pdl_wait();
  pdl_launch_dependents();
  stamp_begin(stamp);
  const int gw = img_w / P, gh = img_h / P, N = gw * gh;
  const int row = P * 3;
  const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
  const bool even = (reinterpret_cast<uintptr_t>(frames) & 1u) == 0;
  if ((row & 1) == 0 && even && static_cast<long long>(sv) * N * P * (row / 2) < (1LL << 30)) {
    // 32-bit index arithmetic (the divisions dominate this kernel's instruction count)
    const int pr = row / 2;  // column pairs per patch row
    const int total = sv * N * P * pr;
    for (int g = blockIdx.x * blockDim.x + threadIdx.x; g < total; g += static_cast<int>(stride)) {
      const int j = g % pr;
      const int t2 = g / pr;
      const int ky = t2 % P;
      const int tok = t2 / P;
      const int v = tok / N, i = tok % N;
      const int py = i / gw, px = i % gw;
      const unsigned short b2 = *reinterpret_cast<const unsigned short*>(
          frames + ((static_cast<size_t>(v) * img_h + py * P + ky) * img_w + px * P) * 3 + 2 * j);
      *reinterpret_cast<__nv_bfloat162*>(patches + static_cast<size_t>(tok) * kpad + ky * row + 2 * j) =
          __floats2bfloat162_rn(static_cast<float>(b2 & 0xFF) - 128.f, static_cast<float>(b2 >> 8) - 128.f);
    }
    stamp_end(stamp);
    return;
  }
  const long long total = static_cast<long long>(sv) * N * P;
  for (long long g = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; g < total; g += stride) {
    const int ky = static_cast<int>(g % P);
    const long long tok = g / P;
    const int v = static_cast<int>(tok / N), i = static_cast<int>(tok % N);
    const int py = i / gw, px = i % gw;
    const uint8_t* src =
        frames + ((static_cast<size_t>(v) * img_h + py * P + ky) * img_w + px * P) * 3;
    bf16* dst = patches + static_cast<size_t>(tok) * kpad + ky * row;
    for (int j = 0; j < row; ++j) dst[j] = __float2bfloat16_rn(static_cast<float>(src[j]) - 128.f);
  }
  stamp_end(stamp);
}

// ------------------------------------------------------------------------ score
// sim[t] = <e_t[t], e_ref[t]> / max(|e_t[t]| |e_ref[t]|, 1e-12) in fp32 (Eq. 3), one warp
// per token, 128-bit loads.  With copy_ref the reference row is replaced by e_t
// (reference = previous frame).
__global__ void score_kernel(const float* __restrict__ e_t, float* __restrict__ e_ref,
                             float* __restrict__ sims, int rows, int dim, int copy_ref,
                             unsigned long long* stamp) {
  pdl_wait();
  pdl_launch_dependents();
  stamp_begin(stamp);
  const int warps = blockDim.x >> 5;
  const int lane = threadIdx.x & 31;
  for (int r = blockIdx.x * warps + (threadIdx.x >> 5); r < rows; r += gridDim.x * warps) {
    const float4* a = reinterpret_cast<const float4*>(e_t + static_cast<size_t>(r) * dim);
    float4* b = reinterpret_cast<float4*>(e_ref + static_cast<size_t>(r) * dim);
    float dot = 0.f, na = 0.f, nb = 0.f;
    for (int c = lane; c < dim / 4; c += 32) {
      const float4 x = a[c], y = b[c];
      dot += x.x * y.x + x.y * y.y + x.z * y.z + x.w * y.w;
      na += x.x * x.x + x.y * x.y + x.z * x.z + x.w * x.w;
      nb += y.x * y.x + y.y * y.y + y.z * y.z + y.w * y.w;
      if (copy_ref) b[c] = x;
    }
    dot = warp_sum(dot);
    na = warp_sum(na);
    nb = warp_sum(nb);
    if (lane == 0) sims[r] = dot / fmaxf(sqrtf(na) * sqrtf(nb), 1e-12f);
  }
  stamp_end(stamp);
}

// ----------------------------------------------------------------------- select
// One CTA per view (blockDim >= N).  flag(i) = cold || sim < tau (threshold mode) or
// rank(i) < k with rank in (sim ascending, index ascending) order (top-k mode).  Flags
// are compacted in index order with warp ballots and a block prefix sum into idx[v][.]
// and counts[v].  The last CTA to finish turns the counts into cu_rows (exclusive
// prefix, cu_rows[sv] = total rows) and writes rowtok[r] = v*N + idx[v][r - cu_rows[v]].
__global__ void select_kernel(const float* __restrict__ sims, int N, int sv, int mode, float tau,
                              int topk, const ColdMask cold, int* __restrict__ idx,
                              int* __restrict__ counts, int* __restrict__ cu_rows,
                              int* __restrict__ rowtok, int* __restrict__ done_ctr,
                              int* __restrict__ user_counts, unsigned long long* stamp) {
  pdl_wait();
  pdl_launch_dependents();
  stamp_begin(stamp);
  extern __shared__ float s_sims[];  // [N]
  __shared__ int s_warp[32];
  __shared__ int s_last;
  const int v = blockIdx.x, i = threadIdx.x;
  const int lane = i & 31, warp = i >> 5, nwarps = blockDim.x >> 5;
  const bool c = is_cold(cold, v);
  const float s = (i < N) ? sims[static_cast<size_t>(v) * N + i] : 0.f;
  bool flag = false;
  if (mode == 1 && !c) {
    if (i < N) s_sims[i] = s;
    __syncthreads();
    if (i < N) {
      int rank = 0;
      for (int j = 0; j < N; ++j) {
        const float sj = s_sims[j];
        rank += (sj < s || (sj == s && j < i)) ? 1 : 0;
      }
      flag = rank < topk;
    }
  } else if (i < N) {
    flag = c || (s < tau);
  }
  const unsigned ballot = __ballot_sync(0xffffffffu, flag);
  if (lane == 0) s_warp[warp] = __popc(ballot);
  __syncthreads();
  if (warp == 0) {
    int x = lane < nwarps ? s_warp[lane] : 0;
    int incl = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane < nwarps) s_warp[lane] = incl - x;  // exclusive warp offsets
    if (lane == 31) s_last = incl;               // view total
  }
  __syncthreads();
  const int total = s_last;
  if (flag) {
    const int pos = s_warp[warp] + __popc(ballot & ((1u << lane) - 1u));
    idx[static_cast<size_t>(v) * N + pos] = i;
  }
  if (i == 0) {
    counts[v] = total;
    if (user_counts) user_counts[v] = total;
  }
  __threadfence();
  __syncthreads();
  if (i == 0) s_last = (atomicAdd(done_ctr, 1) == sv - 1) ? 1 : 0;
  __syncthreads();
  if (!s_last) {
    stamp_end(stamp);
    return;
  }
  __threadfence();
  if (i == 0) {
    int acc = 0;
    for (int u = 0; u < sv; ++u) {
      cu_rows[u] = acc;
      acc += __ldcg(counts + u);
    }
    cu_rows[sv] = acc;
    *done_ctr = 0;
  }
  __syncthreads();
  const int rows = __ldcg(cu_rows + sv);
  for (int r = i; r < rows; r += blockDim.x) {
    int lo = 0, hi = sv - 1;  // last view u with cu_rows[u] <= r
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (__ldcg(cu_rows + mid) <= r) lo = mid; else hi = mid - 1;
    }
    const int k = r - __ldcg(cu_rows + lo);
    rowtok[r] = lo * N + __ldcg(idx + static_cast<size_t>(lo) * N + k);
  }
  stamp_end(stamp);
}

// ----------------------------------------------------------------------- gather
// x[r] = e_t[tok] + pos[tok % N] for the packed updated rows (fp32 residual stream).
// The reference row of an updated token (e_ref[tok] <- ref_src[tok], the score vector:
// patch embedding or first-layer key) is refreshed here when the reference is the last
// refresh, or when the view was cold.  ref_src may be null (no refresh).
__global__ void gather_kernel(const int* __restrict__ total_rows, const int* __restrict__ rowtok,
                              const float* __restrict__ e_t, const float* __restrict__ pos,
                              float* __restrict__ x, const float* __restrict__ ref_src,
                              float* __restrict__ e_ref, int N, int dim, int ref_last_refresh,
                              const ColdMask cold, const RowBands bands, unsigned long long* stamp) {
  pdl_wait();
  pdl_launch_dependents();
  stamp_begin(stamp);
  const int rows = *total_rows;
  if (bands.handle && blockIdx.x == 0 && threadIdx.x == 0) {
    unsigned b = 0;
    while (b + 1 < static_cast<unsigned>(bands.n) && rows > bands.ub[b]) ++b;
    cudaGraphSetConditional(static_cast<cudaGraphConditionalHandle>(bands.handle), b);
  }
  const int warps = blockDim.x >> 5;
  const int lane = threadIdx.x & 31;
  for (int r = blockIdx.x * warps + (threadIdx.x >> 5); r < rows; r += gridDim.x * warps) {
    const int tok = rowtok[r];
    const int ti = tok % N;
    const bool refresh = ref_src && (ref_last_refresh || is_cold(cold, tok / N));
    const float4* a = reinterpret_cast<const float4*>(e_t + static_cast<size_t>(tok) * dim);
    const float4* p = reinterpret_cast<const float4*>(pos + static_cast<size_t>(ti) * dim);
    if (x) {  // (a call that only refreshes references passes no x)
      float4* y = reinterpret_cast<float4*>(x + static_cast<size_t>(r) * dim);
      for (int c = lane; c < dim / 4; c += 32) {
        const float4 u = a[c], w = p[c];
        y[c] = make_float4(u.x + w.x, u.y + w.y, u.z + w.z, u.w + w.w);
      }
    }
    if (refresh) {
      const float4* src = reinterpret_cast<const float4*>(ref_src + static_cast<size_t>(tok) * dim);
      float4* er = reinterpret_cast<float4*>(e_ref + static_cast<size_t>(tok) * dim);
      for (int c = lane; c < dim / 4; c += 32) er[c] = src[c];
    }
  }
  stamp_end(stamp);
}

// The same gather with the rows staged through shared memory by TMA bulk copies: per
// group of GATHER_RPC rows one thread issues a cp.async.bulk of each row of e_t and of
// the position embedding (contiguous, 16-byte aligned), every thread waits on the
// group's mbarrier, then sums from shared memory into x with 128-bit stores.
constexpr int GATHER_RPC = 4;

__global__ void gather_bulk_kernel(const int* __restrict__ total_rows, const int* __restrict__ rowtok,
                                   const float* __restrict__ e_t, const float* __restrict__ pos,
                                   float* __restrict__ x, const float* __restrict__ ref_src,
                                   float* __restrict__ e_ref, int N, int dim, int ref_last_refresh,
                                   const ColdMask cold, const RowBands bands, unsigned long long* stamp) {
  extern __shared__ __align__(128) float gsm[];  // [RPC][dim] e_t rows, then [RPC][dim] pos rows
  __shared__ __align__(8) uint64_t bar;
  __shared__ int s_tok[GATHER_RPC];
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    fence_mbar_init();
  }
  __syncthreads();
  pdl_wait();
  pdl_launch_dependents();
  stamp_begin(stamp);
  const int rows = *total_rows;
  if (bands.handle && blockIdx.x == 0 && threadIdx.x == 0) {
    unsigned b = 0;
    while (b + 1 < static_cast<unsigned>(bands.n) && rows > bands.ub[b]) ++b;
    cudaGraphSetConditional(static_cast<cudaGraphConditionalHandle>(bands.handle), b);
  }
  const int n4 = dim / 4;
  const uint32_t row_bytes = static_cast<uint32_t>(dim) * 4;
  float4* se = reinterpret_cast<float4*>(gsm);
  float4* sp = reinterpret_cast<float4*>(gsm + GATHER_RPC * dim);
  uint32_t phase = 0;
  for (int r0 = blockIdx.x * GATHER_RPC; r0 < rows; r0 += gridDim.x * GATHER_RPC, phase ^= 1u) {
    const int nr = min(GATHER_RPC, rows - r0);
    if (threadIdx.x == 0) {
      mbar_arrive_expect_tx(smem_u32(&bar), 2u * nr * row_bytes);
      for (int i = 0; i < nr; ++i) {
        const int tok = rowtok[r0 + i];
        s_tok[i] = tok;
        bulk_load(smem_u32(se + i * n4), e_t + static_cast<size_t>(tok) * dim, row_bytes, smem_u32(&bar));
        bulk_load(smem_u32(sp + i * n4), pos + static_cast<size_t>(tok % N) * dim, row_bytes, smem_u32(&bar));
      }
    }
    // one vote both publishes s_tok and keeps the loop uniform when a wait gives up
    if (__syncthreads_or(!mbar_wait(smem_u32(&bar), phase))) {
      if (threadIdx.x == 0) mbar_wait(smem_u32(&bar), phase);  // the copies in flight (bounded)
      break;
    }
    for (int e = threadIdx.x; e < nr * n4; e += blockDim.x) {
      const int i = e / n4, c = e - i * n4;
      const int tok = s_tok[i];
      const float4 u = se[i * n4 + c], w = sp[i * n4 + c];
      if (x) reinterpret_cast<float4*>(x + static_cast<size_t>(r0 + i) * dim)[c] =
          make_float4(u.x + w.x, u.y + w.y, u.z + w.z, u.w + w.w);
      if (ref_src && (ref_last_refresh || is_cold(cold, tok / N)))
        reinterpret_cast<float4*>(e_ref + static_cast<size_t>(tok) * dim)[c] =
            ref_src == e_t ? u : reinterpret_cast<const float4*>(ref_src + static_cast<size_t>(tok) * dim)[c];
    }
    __syncthreads();  // the tiles are read before the next group's copies overwrite them
  }
  stamp_end(stamp);
}

// -------------------------------------------------------------------- layernorm
// One warp per row.  The row (up to 2048 floats) is read once into registers with
// 128-bit loads; mean, centred second moment and the normalised output are computed
// from registers in fp32.  The affine parameters sit in shared memory (loaded before
// the wait on the previous kernel), which leaves registers for more rows in flight.
constexpr int LN_MAX_F4_PER_LANE = 16;

// Optionally the input row is gathered (row src_rowtok[r] of x) and, with kAdd, a
// second fp32 array is added to it first and the sum written back to x (the residual
// addition fused into the LN).
template <bool kAdd, bool kGather>
__global__ void layernorm_kernel(const int* __restrict__ nrows, float* __restrict__ x,
                                 const float* __restrict__ add, const int* __restrict__ src_rowtok,
                                 const float* __restrict__ gamma, const float* __restrict__ beta,
                                 bf16* __restrict__ y, const int* __restrict__ dst_rowtok, int dim,
                                 float eps, unsigned long long* stamp) {
  const int warps = blockDim.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n4 = dim / 4;
  // Before waiting on the previous kernel: the affine parameters (constant) and the row
  // count (written by the selection kernel, at least two launches back).
  __shared__ float4 sg[LN_MAX_F4_PER_LANE * 32], sb[LN_MAX_F4_PER_LANE * 32];
  const float4* g4 = reinterpret_cast<const float4*>(gamma);
  const float4* b4 = reinterpret_cast<const float4*>(beta);
  for (int c = threadIdx.x; c < n4; c += blockDim.x) {
    sg[c] = g4[c];
    sb[c] = b4[c];
  }
  __syncthreads();
  const int rows = *nrows;
  pdl_wait();
  pdl_launch_dependents();
  stamp_begin(stamp);
  for (int r = blockIdx.x * warps + (threadIdx.x >> 5); r < rows; r += gridDim.x * warps) {
    const size_t irow = kGather ? static_cast<size_t>(src_rowtok[r]) : static_cast<size_t>(r);
    const float4* xr = reinterpret_cast<const float4*>(static_cast<const float*>(x) + irow * dim);
    float4 v[LN_MAX_F4_PER_LANE];
    float sum = 0.f;
#pragma unroll
    for (int i = 0; i < LN_MAX_F4_PER_LANE; ++i) {
      const int c = lane + 32 * i;
      v[i] = c < n4 ? xr[c] : make_float4(0.f, 0.f, 0.f, 0.f);
      if (kAdd && c < n4) {
        const float4 w = reinterpret_cast<const float4*>(add + irow * dim)[c];
        v[i] = make_float4(v[i].x + w.x, v[i].y + w.y, v[i].z + w.z, v[i].w + w.w);
        reinterpret_cast<float4*>(x + irow * dim)[c] = v[i];
      }
      sum += (v[i].x + v[i].y) + (v[i].z + v[i].w);
    }
    const float mean = warp_sum(sum) / dim;
    float sq = 0.f;
#pragma unroll
    for (int i = 0; i < LN_MAX_F4_PER_LANE; ++i) {
      if (lane + 32 * i < n4) {
        const float a = v[i].x - mean, b = v[i].y - mean, c = v[i].z - mean, d = v[i].w - mean;
        sq += (a * a + b * b) + (c * c + d * d);
      }
    }
    const float rstd = rsqrtf(warp_sum(sq) / dim + eps);
    const size_t orow = dst_rowtok ? static_cast<size_t>(dst_rowtok[r]) : static_cast<size_t>(r);
    __nv_bfloat162* yr = reinterpret_cast<__nv_bfloat162*>(y + orow * dim);
#pragma unroll
    for (int i = 0; i < LN_MAX_F4_PER_LANE; ++i) {
      const int c = lane + 32 * i;
      if (c < n4) {
        const float4 u = v[i], g = sg[c], bb = sb[c];
        yr[2 * c] = __floats2bfloat162_rn(g.x * (u.x - mean) * rstd + bb.x, g.y * (u.y - mean) * rstd + bb.y);
        yr[2 * c + 1] = __floats2bfloat162_rn(g.z * (u.z - mean) * rstd + bb.z, g.w * (u.w - mean) * rstd + bb.w);
      }
    }
  }
  stamp_end(stamp);
}

// Layer norm after a deferred split-K GEMM with the residual epilogue: per row, x +=
// bias + sum_s partial_s (the splits in order, the same fp32 sum the GEMM's own
// reduction forms), x written back, then y = LN(x).  One CTA per row and one float4 of
// the row per thread, so every split's partial of every element is in flight at once
// (a row's partials are spread over the csize slots of its feature tiles).
__global__ void layernorm_sum_kernel(const int* __restrict__ nrows, float* __restrict__ x, const PendingSum ps,
                                     const float* __restrict__ gamma, const float* __restrict__ beta,
                                     bf16* __restrict__ y, const int* __restrict__ dst_rowtok, int dim, float eps,
                                     unsigned long long* stamp) {
  constexpr int MAXS = 16;
  __shared__ float red[2][32];
  const int c = threadIdx.x;  // float4 of the row
  const int n4 = dim / 4, lane = c & 31, warp = c >> 5, nw = blockDim.x >> 5;
  const bool act = c < n4;
  float4 g = make_float4(0.f, 0.f, 0.f, 0.f), b = g, bias = g;
  if (act) {  // constants: before the wait on the previous kernel
    g = reinterpret_cast<const float4*>(gamma)[c];
    b = reinterpret_cast<const float4*>(beta)[c];
    bias = reinterpret_cast<const float4*>(ps.bias)[c];
  }
  const int rows = *nrows;  // written by the selection kernel, at least two launches back
  pdl_wait();
  pdl_launch_dependents();
  stamp_begin(stamp);
  const int f = 4 * c, ft = f >> 7, fl = f & 127;
  const size_t sstride = static_cast<size_t>(ps.bn) * 128;
  for (int r = blockIdx.x; r < rows; r += gridDim.x) {
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (act) {
      const int tt = r / ps.bn, rr = r - tt * ps.bn;
      const float* p = ps.partials + (static_cast<size_t>(ft + ps.n_ft * tt) * ps.csize * ps.bn + rr) * 128 + fl;
      float4 q[MAXS];
#pragma unroll
      for (int sp = 0; sp < MAXS; ++sp)
        if (sp < ps.csize) q[sp] = __ldcg(reinterpret_cast<const float4*>(p + sp * sstride));
      float4* xr = reinterpret_cast<float4*>(x + static_cast<size_t>(r) * dim) + c;
      const float4 x0 = *xr;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int sp = 0; sp < MAXS; ++sp)
        if (sp < ps.csize) {
          acc.x += q[sp].x;
          acc.y += q[sp].y;
          acc.z += q[sp].z;
          acc.w += q[sp].w;
        }
      v = make_float4(x0.x + (acc.x + bias.x), x0.y + (acc.y + bias.y), x0.z + (acc.z + bias.z),
                      x0.w + (acc.w + bias.w));
      *xr = v;
    }
    float sum = warp_sum((v.x + v.y) + (v.z + v.w));
    if (lane == 0) red[0][warp] = sum;
    __syncthreads();
    sum = 0.f;
    for (int w = 0; w < nw; ++w) sum += red[0][w];
    const float mean = sum / dim;
    float sq = 0.f;
    if (act) {
      const float a0 = v.x - mean, a1 = v.y - mean, a2 = v.z - mean, a3 = v.w - mean;
      sq = (a0 * a0 + a1 * a1) + (a2 * a2 + a3 * a3);
    }
    sq = warp_sum(sq);
    if (lane == 0) red[1][warp] = sq;
    __syncthreads();
    sq = 0.f;
    for (int w = 0; w < nw; ++w) sq += red[1][w];
    const float rstd = rsqrtf(sq / dim + eps);
    if (act) {
      const size_t orow = dst_rowtok ? static_cast<size_t>(dst_rowtok[r]) : static_cast<size_t>(r);
      __nv_bfloat162* yr = reinterpret_cast<__nv_bfloat162*>(y + orow * dim);
      yr[2 * c] = __floats2bfloat162_rn(g.x * (v.x - mean) * rstd + b.x, g.y * (v.y - mean) * rstd + b.y);
      yr[2 * c + 1] = __floats2bfloat162_rn(g.z * (v.z - mean) * rstd + b.z, g.w * (v.w - mean) * rstd + b.w);
    }
  }
  stamp_end(stamp);
}

// -------------------------------------------------------------------- attention
// Attention of the updated queries of one view over all N keys of that view (cached
// K/V with this call's updated rows already written), per head:
//   O = softmax(Q K^T / sqrt(dh)) V.
// Grid: (query block x key split, head, view); the key splits of one query block form
// a thread-block cluster.  Each CTA brings its key range (kps <= 128 keys) of K and V
// into shared memory with one TMA load each, [keys][dh] bf16, issued before waiting on
// the QKV kernel (the cached keys of reused tokens do not change); after the wait it
// re-reads only the keys of this call's updated tokens.  Warp w owns queries
// 4w..4w+3: scores with lanes owning keys (16-byte row loads), softmax in fp32 over the
// CTA's keys, P V with lanes owning output dims; the cluster then merges its partial
// (m, l, o) through distributed shared memory:
//   M = max_s m_s,  O = sum_s exp(m_s - M) o_s / sum_s exp(m_s - M) l_s.
constexpr int ATT_WARPS = 8;
constexpr int ATT_QPW = 4;
constexpr int ATT_QB = ATT_WARPS * ATT_QPW;
constexpr int ATT_KR = 128;   // max keys per CTA (key split)

__global__ void __launch_bounds__(ATT_WARPS * 32)
    attention_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                     const bf16* __restrict__ q, const bf16* __restrict__ cache_k,
                     const bf16* __restrict__ cache_v, const int* __restrict__ cu_rows,
                     const int* __restrict__ rowtok, bf16* __restrict__ o, int N, int dim, int dh, int kps) {
  extern __shared__ __align__(128) uint8_t att_smem[];
  bf16* sk = reinterpret_cast<bf16*>(att_smem);            // [kps][dh]
  bf16* sv = sk + ATT_KR * dh;                              // [kps][dh]
  float* sq = reinterpret_cast<float*>(sv + ATT_KR * dh);   // [QB][dh] (later: partial o)
  float* sp = sq + ATT_QB * dh;                             // [WARPS][QPW][KR]
  float* sml = sp + ATT_WARPS * ATT_QPW * ATT_KR;           // [QB][2]
  uint64_t* bar = reinterpret_cast<uint64_t*>(sml + 2 * ATT_QB);
  const int ns = static_cast<int>(cluster_nctarank());
  const int rank = static_cast<int>(cluster_ctarank());
  const int v = blockIdx.z, h = blockIdx.y;
  const int qb_first = blockIdx.x / ns, qb_stride = gridDim.x / ns;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int dh8 = dh / 8;
  // Row ranges come from the selection kernel (complete before this grid can start).
  const int r_begin = cu_rows[v], r_end = cu_rows[v + 1];
  if (r_begin + qb_first * ATT_QB >= r_end) return;  // the whole cluster leaves together
  const int k_begin = rank * kps, nkr = min(N, k_begin + kps) - k_begin;
  const size_t vbase = static_cast<size_t>(v) * N;
  const uint32_t bar_addr = smem_u32(bar);
  bool ok = true;
  if (tid == 0) {
    mbar_init(bar_addr, 1);
    fence_mbar_init();
    const uint32_t bytes = static_cast<uint32_t>(kps) * dh * 2;
    mbar_arrive_expect_tx(bar_addr, 2 * bytes);
    tma_load_2d(smem_u32(sk), &tm_k, h * dh, static_cast<int>(vbase) + k_begin, bar_addr, l2_policy_evict_first());
    tma_load_2d(smem_u32(sv), &tm_v, h * dh, static_cast<int>(vbase) + k_begin, bar_addr, l2_policy_evict_first());
  }
  __syncthreads();  // barrier initialised before anyone waits on it
  pdl_wait();  // the QKV kernel's queries and new K/V rows are visible from here
  pdl_launch_dependents();
  if (!mbar_wait(bar_addr, 0)) ok = false;  // (all threads) cached tile landed
  __syncthreads();
  // re-read the keys this call updated (tokens of view v listed in rowtok)
  const int n_upd = r_end - r_begin;
  for (int e = tid; e < n_upd * dh8; e += blockDim.x) {
    const int r = e / dh8, c = e % dh8;
    const int j = rowtok[r_begin + r] - static_cast<int>(vbase) - k_begin;
    if (j >= 0 && j < nkr) {
      const size_t g = (vbase + k_begin + j) * dim + h * dh + c * 8;
      *reinterpret_cast<uint4*>(sk + j * dh + c * 8) = __ldcg(reinterpret_cast<const uint4*>(cache_k + g));
      *reinterpret_cast<uint4*>(sv + j * dh + c * 8) = __ldcg(reinterpret_cast<const uint4*>(cache_v + g));
    }
  }
  const float scale = rsqrtf(static_cast<float>(dh));
  // query blocks of this view handled by this cluster (the key tile stays resident)
  for (int qb = qb_first; r_begin + qb * ATT_QB < r_end; qb += qb_stride) {
  const int q0 = r_begin + qb * ATT_QB;
  const int nq = min(ATT_QB, r_end - q0);
  __syncthreads();  // previous block's queries and partials are consumed
  for (int e = tid; e < nq * dh8; e += blockDim.x) {
    const int qi = e / dh8, c = e % dh8;
    const uint4 u = __ldcg(reinterpret_cast<const uint4*>(q + static_cast<size_t>(q0 + qi) * dim + h * dh + c * 8));
    const __nv_bfloat162* b2 = reinterpret_cast<const __nv_bfloat162*>(&u);
    float4* dst = reinterpret_cast<float4*>(sq + qi * dh + c * 8);
    const float2 f0 = __bfloat1622float2(b2[0]), f1 = __bfloat1622float2(b2[1]);
    const float2 f2 = __bfloat1622float2(b2[2]), f3 = __bfloat1622float2(b2[3]);
    dst[0] = make_float4(f0.x * scale, f0.y * scale, f1.x * scale, f1.y * scale);
    dst[1] = make_float4(f2.x * scale, f2.y * scale, f3.x * scale, f3.y * scale);
  }
  __syncthreads();

  const int qa = warp * ATT_QPW;
  float m_run[ATT_QPW], l_run[ATT_QPW], acc[ATT_QPW][4];
#pragma unroll
  for (int a = 0; a < ATT_QPW; ++a) {
    m_run[a] = -INFINITY;
    l_run[a] = 0.f;
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[a][c] = 0.f;
  }
  if (qa < nq && ok) {
    float* spw = sp + warp * ATT_QPW * ATT_KR;
    // scores: lane owns keys lane + 32 kk of the CTA's range
    float sc[ATT_QPW][4];
#pragma unroll
    for (int a = 0; a < ATT_QPW; ++a)
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) sc[a][kk] = 0.f;
    for (int d = 0; d < dh; d += 8) {
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const int j = lane + 32 * kk;
        if (j < nkr) {
          const uint4 raw = *reinterpret_cast<const uint4*>(sk + j * dh + d);
          const __nv_bfloat162* k2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
          const float2 f0 = __bfloat1622float2(k2[0]), f1 = __bfloat1622float2(k2[1]);
          const float2 f2 = __bfloat1622float2(k2[2]), f3 = __bfloat1622float2(k2[3]);
#pragma unroll
          for (int a = 0; a < ATT_QPW; ++a) {
            const float4 lo = *reinterpret_cast<const float4*>(sq + (qa + a) * dh + d);
            const float4 hi = *reinterpret_cast<const float4*>(sq + (qa + a) * dh + d + 4);
            sc[a][kk] += lo.x * f0.x + lo.y * f0.y + lo.z * f1.x + lo.w * f1.y + hi.x * f2.x + hi.y * f2.y +
                         hi.z * f3.x + hi.w * f3.y;
          }
        }
      }
    }
#pragma unroll
    for (int a = 0; a < ATT_QPW; ++a) {
      float mx = -INFINITY;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        if (lane + 32 * kk < nkr) mx = fmaxf(mx, sc[a][kk]);
      mx = warp_max(mx);
      float sum = 0.f;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const int j = lane + 32 * kk;
        if (j < nkr) {
          const float p = __expf(sc[a][kk] - mx);
          spw[a * ATT_KR + j] = p;
          sum += p;
        }
      }
      m_run[a] = mx;
      l_run[a] = warp_sum(sum);
    }
    __syncwarp();
    // P V: lanes own dims lane + 32 c; 8 keys per step with every load issued first
    for (int j0 = 0; j0 < nkr; j0 += 8) {
      float pk[ATT_QPW][8], vk[8][4];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int j = j0 + u;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int d = lane + 32 * c;
          vk[u][c] = (j < nkr && d < dh) ? __bfloat162float(sv[j * dh + d]) : 0.f;
        }
#pragma unroll
        for (int a = 0; a < ATT_QPW; ++a) pk[a][u] = j < nkr ? spw[a * ATT_KR + j] : 0.f;
      }
#pragma unroll
      for (int u = 0; u < 8; ++u)
#pragma unroll
        for (int a = 0; a < ATT_QPW; ++a)
#pragma unroll
          for (int c = 0; c < 4; ++c) acc[a][c] += pk[a][u] * vk[u][c];
    }
  }

  if (ns == 1) {
#pragma unroll
    for (int a = 0; a < ATT_QPW; ++a) {
      const int qi = qa + a;
      if (qi < nq) {
        const float inv = 1.f / l_run[a];
        bf16* orow = o + static_cast<size_t>(q0 + qi) * dim + h * dh;
#pragma unroll
        for (int c = 0; c < 4; ++c)
          if (lane + 32 * c < dh) orow[lane + 32 * c] = __float2bfloat16_rn(acc[a][c] * inv);
      }
    }
    continue;
  }

  // partial (m, l, o) of every query of the block, then a cluster-wide merge
  __syncthreads();  // every warp is done with sq
  float* so = sq;
#pragma unroll
  for (int a = 0; a < ATT_QPW; ++a) {
    const int qi = qa + a;
#pragma unroll
    for (int c = 0; c < 4; ++c)
      if (lane + 32 * c < dh) so[qi * dh + lane + 32 * c] = acc[a][c];
    if (lane == 0) {
      sml[2 * qi] = m_run[a];
      sml[2 * qi + 1] = l_run[a];
    }
  }
  cluster_sync();
  const uint32_t so_addr = smem_u32(so), ml_addr = smem_u32(sml);
  for (int qi = rank + ns * warp; qi < nq; qi += ns * ATT_WARPS) {
    float M = -INFINITY;
    for (int s2 = 0; s2 < ns; ++s2) M = fmaxf(M, ld_dsmem_f32(mapa_shared(ml_addr + 8 * qi, s2)));
    float lsum = 0.f, out[4] = {0.f, 0.f, 0.f, 0.f};
    for (int s2 = 0; s2 < ns; ++s2) {
      const float w = __expf(ld_dsmem_f32(mapa_shared(ml_addr + 8 * qi, s2)) - M);
      lsum += w * ld_dsmem_f32(mapa_shared(ml_addr + 8 * qi + 4, s2));
#pragma unroll
      for (int c = 0; c < 4; ++c)
        if (lane + 32 * c < dh)
          out[c] += w * ld_dsmem_f32(mapa_shared(so_addr + 4 * (qi * dh + lane + 32 * c), s2));
    }
    const float inv = 1.f / lsum;
    bf16* orow = o + static_cast<size_t>(q0 + qi) * dim + h * dh;
#pragma unroll
    for (int c = 0; c < 4; ++c)
      if (lane + 32 * c < dh) orow[lane + 32 * c] = __float2bfloat16_rn(out[c] * inv);
  }
  cluster_sync();  // partials stay valid until every CTA of the cluster has read them
  }  // query blocks
}

}  // namespace

cudaError_t launch_patchify(const uint8_t* frames, bf16* patches, int sv, int img_h, int img_w,
                            int patch, int kpad, cudaStream_t s) {
  long long total = static_cast<long long>(sv) * (img_h / patch) * (img_w / patch) * patch;
  if ((patch * 3) % 2 == 0) total *= patch * 3 / 2;
  const long long blocks = (total + 255) / 256;
  const int grid = static_cast<int>(blocks < 8192 ? blocks : 8192);
  return launch_ex(patchify_kernel, dim3(grid), dim3(256), 0, s, 1, frames, patches, sv, img_h, img_w, patch, kpad,
                   g_stamp);
}

cudaError_t launch_score(const float* e_t, float* e_ref, float* sims, int rows, int dim,
                         int copy_ref, cudaStream_t s) {
  const int grid = min((rows + 7) / 8, 4096);
  return launch_ex(score_kernel, dim3(grid), dim3(256), 0, s, 1, e_t, e_ref, sims, rows, dim, copy_ref, g_stamp);
}

cudaError_t launch_select(const float* sims, int n_tok, int sv, int mode, float tau, int topk,
                          const ColdMask& cold, int* idx, int* counts, int* cu_rows, int* rowtok,
                          int* done_ctr, int* user_counts, cudaStream_t s) {
  const int threads = (n_tok + 31) / 32 * 32;
  return launch_ex(select_kernel, dim3(sv), dim3(threads), n_tok * sizeof(float), s, 1, sims, n_tok, sv,
                   mode, tau, topk, cold, idx, counts, cu_rows, rowtok, done_ctr, user_counts, g_stamp);
}

cudaError_t launch_gather(const int* cu_rows_total, const int* rowtok, const float* e_t,
                          const float* pos, float* x, const float* ref_src, float* e_ref, int n_tok,
                          int dim, int ref_last_refresh, const ColdMask& cold, int max_rows, int grid,
                          cudaStream_t s, const RowBands& bands) {
  const char* genv = std::getenv("IVIT_GATHER");  // read per launch: graphs capture it once
  const bool bulk = genv && std::strcmp(genv, "tma") == 0;
  if (bulk && dim % 4 == 0 && dim <= 2048) {
    const size_t smem = 2 * GATHER_RPC * static_cast<size_t>(dim) * sizeof(float);
    static bool attr = false;
    if (!attr) {
      const cudaError_t e = cudaFuncSetAttribute(gather_bulk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 static_cast<int>(2 * GATHER_RPC * 2048 * sizeof(float)));
      if (e != cudaSuccess) return e;
      attr = true;
    }
    grid = max(1, min(grid, (max_rows + GATHER_RPC - 1) / GATHER_RPC));
    return launch_ex(gather_bulk_kernel, dim3(grid), dim3(256), smem, s, 1, cu_rows_total, rowtok, e_t, pos, x,
                     ref_src, e_ref, n_tok, dim, ref_last_refresh, cold, bands, g_stamp);
  }
  grid = max(1, min(grid, (max_rows + 7) / 8));
  return launch_ex(gather_kernel, dim3(grid), dim3(256), 0, s, 1, cu_rows_total, rowtok, e_t, pos, x,
                   ref_src, e_ref, n_tok, dim, ref_last_refresh, cold, bands, g_stamp);
}

cudaError_t launch_layernorm(const int* rows, const float* x, const float* gamma, const float* beta,
                             bf16* y, const int* dst_rowtok, int dim, float eps, int max_rows,
                             int grid, cudaStream_t s) {
  return launch_layernorm_ex(rows, const_cast<float*>(x), nullptr, nullptr, gamma, beta, y, dst_rowtok, dim, eps,
                             max_rows, grid, s);
}

cudaError_t launch_layernorm_sum(const int* rows, float* x, const PendingSum& ps, const float* gamma,
                                 const float* beta, bf16* y, const int* dst_rowtok, int dim, float eps,
                                 int max_rows, int grid, cudaStream_t s) {
  if (dim % 4 != 0 || dim > 4096 || ps.csize < 2 || ps.csize > 16 || ps.bn < 1 || !ps.partials || !ps.bias)
    return cudaErrorInvalidValue;
  const int threads = (dim / 4 + 31) / 32 * 32;
  grid = max(1, min(grid, max_rows));
  return launch_ex(layernorm_sum_kernel, dim3(grid), dim3(threads), 0, s, 1, rows, x, ps, gamma, beta, y,
                   dst_rowtok, dim, eps, g_stamp);
}

cudaError_t launch_layernorm_ex(const int* rows, float* x, const float* add, const int* src_rowtok,
                                const float* gamma, const float* beta, bf16* y, const int* dst_rowtok, int dim,
                                float eps, int max_rows, int grid, cudaStream_t s) {
  grid = max(1, min(grid, (max_rows + 7) / 8));
  auto kern = add ? (src_rowtok ? layernorm_kernel<true, true> : layernorm_kernel<true, false>)
                  : (src_rowtok ? layernorm_kernel<false, true> : layernorm_kernel<false, false>);
  return launch_ex(kern, dim3(grid), dim3(256), 0, s, 1, rows, x, add, src_rowtok, gamma, beta, y, dst_rowtok, dim,
                   eps, g_stamp);
}

size_t attention_smem(int dh) {
  return 2 * static_cast<size_t>(ATT_KR) * dh * sizeof(bf16) +
         (ATT_QB * dh + ATT_WARPS * ATT_QPW * ATT_KR + 2 * ATT_QB) * sizeof(float) + 16;
}

int attention_keys_per_split(int n_tok) {
  int ns = (n_tok + 63) / 64;  // key splits of about 64 keys, at most 8 (portable cluster)
  ns = ns < 1 ? 1 : (ns > 8 ? 8 : ns);
  return (n_tok + ns - 1) / ns;
}

cudaError_t attention_setup() {
  return cudaFuncSetAttribute(attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(attention_smem(128)));
}

cudaError_t launch_attention(const CUtensorMap& tm_k, const CUtensorMap& tm_v, const bf16* q,
                             const bf16* cache_k, const bf16* cache_v, const int* cu_rows,
                             const int* rowtok, bf16* o, int sv, int n_tok, int dim, int heads,
                             int query_blocks, cudaStream_t s) {
  const int dh = dim / heads;
  const int kps = attention_keys_per_split(n_tok);
  const int ns = (n_tok + kps - 1) / kps;
  const int max_qb = (n_tok + ATT_QB - 1) / ATT_QB;
  const int qbs = query_blocks < 1 ? 1 : (query_blocks > max_qb ? max_qb : query_blocks);
  const dim3 grid(qbs * ns, heads, sv);
  return launch_ex(attention_kernel, grid, dim3(ATT_WARPS * 32), attention_smem(dh), s,
                   static_cast<unsigned>(ns), tm_k, tm_v, q, cache_k, cache_v, cu_rows, rowtok, o, n_tok, dim,
                   dh, kps);
}

}  // namespace ivit
