// Memory-bound kernels of the incremental encode: patchify, change score (Eq. 3),
// selection + stream compaction, gather of the updated rows, layer norm (with the
// final-token cache scatter), and attention of the updated queries over all tokens.
#include "internal.h"
#include "ptx.cuh"

namespace ivit {
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
// bf16).  One thread per (token, ky): P*3 contiguous bytes in, P*3 bf16 out.  Columns
// P*P*3 .. kpad-1 stay zero (set once at allocation).
__global__ void patchify_kernel(const uint8_t* __restrict__ frames, bf16* __restrict__ patches,
                                int sv, int img_h, int img_w, int P, int kpad) {
  pdl_wait();
  const int gw = img_w / P, gh = img_h / P, N = gw * gh;
  const long long total = static_cast<long long>(sv) * N * P;
  for (long long g = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; g < total;
       g += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int ky = static_cast<int>(g % P);
    const long long tok = g / P;
    const int v = static_cast<int>(tok / N), i = static_cast<int>(tok % N);
    const int py = i / gw, px = i % gw;
    const uint8_t* src =
        frames + ((static_cast<size_t>(v) * img_h + py * P + ky) * img_w + px * P) * 3;
    bf16* dst = patches + static_cast<size_t>(tok) * kpad + ky * P * 3;
    for (int j = 0; j < P * 3; ++j) dst[j] = __float2bfloat16_rn(static_cast<float>(src[j]) - 128.f);
  }
}

// ------------------------------------------------------------------------ score
// sim[t] = <e_t[t], e_ref[t]> / max(|e_t[t]| |e_ref[t]|, 1e-12) in fp32 (Eq. 3), one warp
// per token, 128-bit loads.  With copy_ref the reference row is replaced by e_t
// (reference = previous frame).
__global__ void score_kernel(const float* __restrict__ e_t, float* __restrict__ e_ref,
                             float* __restrict__ sims, int rows, int dim, int copy_ref) {
  pdl_wait();
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
                              int* __restrict__ user_counts) {
  pdl_wait();
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
  if (!s_last) return;
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
}

// ----------------------------------------------------------------------- gather
// x[r] = e_t[tok] + pos[tok % N] for the packed updated rows (fp32 residual stream).
// The reference row of an updated token is refreshed here when the reference is the
// last refresh, or when the view was cold.
__global__ void gather_kernel(const int* __restrict__ total_rows, const int* __restrict__ rowtok,
                              const float* __restrict__ e_t, const float* __restrict__ pos,
                              float* __restrict__ x, float* __restrict__ e_ref, int N, int dim,
                              int ref_last_refresh, const ColdMask cold) {
  pdl_wait();
  const int rows = *total_rows;
  const int warps = blockDim.x >> 5;
  const int lane = threadIdx.x & 31;
  for (int r = blockIdx.x * warps + (threadIdx.x >> 5); r < rows; r += gridDim.x * warps) {
    const int tok = rowtok[r];
    const int ti = tok % N;
    const bool refresh = ref_last_refresh || is_cold(cold, tok / N);
    const float4* a = reinterpret_cast<const float4*>(e_t + static_cast<size_t>(tok) * dim);
    const float4* p = reinterpret_cast<const float4*>(pos + static_cast<size_t>(ti) * dim);
    float4* y = reinterpret_cast<float4*>(x + static_cast<size_t>(r) * dim);
    float4* er = reinterpret_cast<float4*>(e_ref + static_cast<size_t>(tok) * dim);
    for (int c = lane; c < dim / 4; c += 32) {
      const float4 u = a[c], w = p[c];
      y[c] = make_float4(u.x + w.x, u.y + w.y, u.z + w.z, u.w + w.w);
      if (refresh) er[c] = u;
    }
  }
}

// -------------------------------------------------------------------- layernorm
// One warp per row; mean, then centred second moment, then the normalised output, in
// fp32 (the row stays in L1 between passes).
__global__ void layernorm_kernel(const int* __restrict__ nrows, const float* __restrict__ x,
                                 const float* __restrict__ gamma, const float* __restrict__ beta,
                                 bf16* __restrict__ y, const int* __restrict__ dst_rowtok, int dim,
                                 float eps) {
  pdl_wait();
  const int rows = *nrows;
  const int warps = blockDim.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n4 = dim / 4;
  for (int r = blockIdx.x * warps + (threadIdx.x >> 5); r < rows; r += gridDim.x * warps) {
    const float4* xr = reinterpret_cast<const float4*>(x + static_cast<size_t>(r) * dim);
    float sum = 0.f;
    for (int c = lane; c < n4; c += 32) {
      const float4 u = xr[c];
      sum += (u.x + u.y) + (u.z + u.w);
    }
    const float mean = warp_sum(sum) / dim;
    float sq = 0.f;
    for (int c = lane; c < n4; c += 32) {
      const float4 u = xr[c];
      const float a = u.x - mean, b = u.y - mean, cc = u.z - mean, d = u.w - mean;
      sq += (a * a + b * b) + (cc * cc + d * d);
    }
    const float rstd = rsqrtf(warp_sum(sq) / dim + eps);
    const size_t orow = dst_rowtok ? static_cast<size_t>(dst_rowtok[r]) : static_cast<size_t>(r);
    __nv_bfloat162* yr = reinterpret_cast<__nv_bfloat162*>(y + orow * dim);
    const float4* g4 = reinterpret_cast<const float4*>(gamma);
    const float4* b4 = reinterpret_cast<const float4*>(beta);
    for (int c = lane; c < n4; c += 32) {
      const float4 u = xr[c], g = g4[c], b = b4[c];
      yr[2 * c] = __floats2bfloat162_rn(g.x * (u.x - mean) * rstd + b.x, g.y * (u.y - mean) * rstd + b.y);
      yr[2 * c + 1] = __floats2bfloat162_rn(g.z * (u.z - mean) * rstd + b.z, g.w * (u.w - mean) * rstd + b.w);
    }
  }
}

// -------------------------------------------------------------------- attention
// CTA = (query block of one view, head).  Keys and values of the view are streamed in
// tiles of KT rows through shared memory (fp32, padded rows); each warp owns QPW
// queries and keeps an online softmax (running max and sum) and its output row in
// registers: lane d owns output dims d, d+32, d+64, d+96.
constexpr int ATT_WARPS = 4;
constexpr int ATT_QPW = 8;
constexpr int ATT_QB = ATT_WARPS * ATT_QPW;
constexpr int ATT_KT = 64;

__global__ void __launch_bounds__(ATT_WARPS * 32)
    attention_kernel(const bf16* __restrict__ q, const bf16* __restrict__ cache_k,
                     const bf16* __restrict__ cache_v, const int* __restrict__ cu_rows,
                     bf16* __restrict__ o, int N, int dim, int dh) {
  pdl_wait();
  extern __shared__ float sm[];
  const int ld = dh + 1;
  float* sk = sm;                       // [KT][dh+1]
  float* sv = sk + ATT_KT * ld;         // [KT][dh+1]
  float* sq = sv + ATT_KT * ld;         // [QB][dh]
  const int v = blockIdx.z, h = blockIdx.y;
  const int r_begin = cu_rows[v], r_end = cu_rows[v + 1];
  const int q0 = r_begin + blockIdx.x * ATT_QB;
  if (q0 >= r_end) return;
  const int nq = min(ATT_QB, r_end - q0);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float scale = rsqrtf(static_cast<float>(dh));

  for (int e = tid; e < nq * dh; e += blockDim.x) {
    const int qi = e / dh, d = e % dh;
    sq[qi * dh + d] = __bfloat162float(q[static_cast<size_t>(q0 + qi) * dim + h * dh + d]) * scale;
  }

  float m_run[ATT_QPW], l_run[ATT_QPW], acc[ATT_QPW][4];
#pragma unroll
  for (int a = 0; a < ATT_QPW; ++a) {
    m_run[a] = -INFINITY;
    l_run[a] = 0.f;
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[a][c] = 0.f;
  }

  const size_t vbase = static_cast<size_t>(v) * N;
  for (int k0 = 0; k0 < N; k0 += ATT_KT) {
    const int nk = min(ATT_KT, N - k0);
    __syncthreads();
    for (int e = tid; e < nk * dh; e += blockDim.x) {
      const int j = e / dh, d = e % dh;
      const size_t g = (vbase + k0 + j) * dim + h * dh + d;
      sk[j * ld + d] = __bfloat162float(cache_k[g]);
      sv[j * ld + d] = __bfloat162float(cache_v[g]);
    }
    __syncthreads();
#pragma unroll
    for (int a = 0; a < ATT_QPW; ++a) {
      const int qi = warp * ATT_QPW + a;
      if (qi >= nq) break;
      const float* qr = sq + qi * dh;
      float s0 = -INFINITY, s1 = -INFINITY;
      if (lane < nk) {
        float t = 0.f;
        for (int d = 0; d < dh; ++d) t += qr[d] * sk[lane * ld + d];
        s0 = t;
      }
      if (lane + 32 < nk) {
        float t = 0.f;
        for (int d = 0; d < dh; ++d) t += qr[d] * sk[(lane + 32) * ld + d];
        s1 = t;
      }
      const float mt = warp_max(fmaxf(s0, s1));
      const float m_new = fmaxf(m_run[a], mt);
      const float corr = __expf(m_run[a] - m_new);
      const float p0 = (lane < nk) ? __expf(s0 - m_new) : 0.f;
      const float p1 = (lane + 32 < nk) ? __expf(s1 - m_new) : 0.f;
      l_run[a] = l_run[a] * corr + warp_sum(p0 + p1);
      m_run[a] = m_new;
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[a][c] *= corr;
      for (int j = 0; j < nk; ++j) {
        const float pj = __shfl_sync(0xffffffffu, j < 32 ? p0 : p1, j & 31);
        const float* vr = sv + j * ld;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int d = lane + 32 * c;
          if (d < dh) acc[a][c] += pj * vr[d];
        }
      }
    }
  }
#pragma unroll
  for (int a = 0; a < ATT_QPW; ++a) {
    const int qi = warp * ATT_QPW + a;
    if (qi >= nq) break;
    const float inv = 1.f / l_run[a];
    bf16* orow = o + static_cast<size_t>(q0 + qi) * dim + h * dh;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int d = lane + 32 * c;
      if (d < dh) orow[d] = __float2bfloat16_rn(acc[a][c] * inv);
    }
  }
}

}  // namespace

cudaError_t launch_patchify(const uint8_t* frames, bf16* patches, int sv, int img_h, int img_w,
                            int patch, int kpad, cudaStream_t s) {
  const long long total = static_cast<long long>(sv) * (img_h / patch) * (img_w / patch) * patch;
  const long long blocks = (total + 255) / 256;
  const int grid = static_cast<int>(blocks < 4096 ? blocks : 4096);
  patchify_kernel<<<grid, 256, 0, s>>>(frames, patches, sv, img_h, img_w, patch, kpad);
  return cudaGetLastError();
}

cudaError_t launch_score(const float* e_t, float* e_ref, float* sims, int rows, int dim,
                         int copy_ref, cudaStream_t s) {
  const int grid = min((rows + 7) / 8, 4096);
  score_kernel<<<grid, 256, 0, s>>>(e_t, e_ref, sims, rows, dim, copy_ref);
  return cudaGetLastError();
}

cudaError_t launch_select(const float* sims, int n_tok, int sv, int mode, float tau, int topk,
                          const ColdMask& cold, int* idx, int* counts, int* cu_rows, int* rowtok,
                          int* done_ctr, int* user_counts, cudaStream_t s) {
  const int threads = (n_tok + 31) / 32 * 32;
  select_kernel<<<sv, threads, n_tok * sizeof(float), s>>>(sims, n_tok, sv, mode, tau, topk, cold, idx,
                                                            counts, cu_rows, rowtok, done_ctr,
                                                            user_counts);
  return cudaGetLastError();
}

cudaError_t launch_gather(const int* cu_rows_total, const int* rowtok, const float* e_t,
                          const float* pos, float* x, float* e_ref, int n_tok, int dim,
                          int ref_last_refresh, const ColdMask& cold, int max_rows, int grid,
                          cudaStream_t s) {
  grid = max(1, min(grid, (max_rows + 7) / 8));
  gather_kernel<<<grid, 256, 0, s>>>(cu_rows_total, rowtok, e_t, pos, x, e_ref, n_tok, dim,
                                     ref_last_refresh, cold);
  return cudaGetLastError();
}

cudaError_t launch_layernorm(const int* rows, const float* x, const float* gamma, const float* beta,
                             bf16* y, const int* dst_rowtok, int dim, float eps, int max_rows,
                             int grid, cudaStream_t s) {
  grid = max(1, min(grid, (max_rows + 7) / 8));
  layernorm_kernel<<<grid, 256, 0, s>>>(rows, x, gamma, beta, y, dst_rowtok, dim, eps);
  return cudaGetLastError();
}

cudaError_t launch_attention(const bf16* q, const bf16* cache_k, const bf16* cache_v,
                             const int* cu_rows, bf16* o, int sv, int n_tok, int dim, int heads,
                             cudaStream_t s) {
  const int dh = dim / heads;
  const size_t smem = (2 * ATT_KT * (dh + 1) + ATT_QB * dh) * sizeof(float);
  static bool attr_set = false;
  if (!attr_set) {
    cudaFuncSetAttribute(attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 96 * 1024);
    attr_set = true;
  }
  dim3 grid((n_tok + ATT_QB - 1) / ATT_QB, heads, sv);
  attention_kernel<<<grid, ATT_WARPS * 32, smem, s>>>(q, cache_k, cache_v, cu_rows, o, n_tok, dim, dh);
  return cudaGetLastError();
}

}  // namespace ivit
