// Token selection without any device allocation (ivit_select_noalloc).
//
// Some callers cannot call cudaMalloc at the point where they need the changed-token
// lists: code that enqueues work while a CUDA stream is being captured into a graph
// (allocation calls are not permitted there), plugins whose host framework forbids
// allocation inside its enqueue callback, and real-time loops that allocate only at
// start-up.  This entry point computes the same scores and lists as the selection step
// of ivit_encode_incremental, from two embedding sets the caller already holds, and
// keeps its only scratch -- one fp32 score per token -- in a file-scope device array of
// fixed size instead of allocating it.
#include <mutex>

#include "../../include/ivit.h"
#include "internal.h"
#include "ptx.cuh"

namespace ivit {
void set_create_error(const char* msg);  // engine.cu: message for ivit_last_error(NULL)
}

namespace {

// Scores of every token of the call.  Every device that loads the library holds this
// array until the process exits.  Calls share it: each call writes every entry it later
// reads, so nothing carries over between calls, but calls that overlap on the GPU race.
static __device__ __align__(256) float g_select_scores[IVIT_NOALLOC_MAX_TOKENS];

constexpr int kMaxDevices = 64;

// Device address of g_select_scores per device, looked up on the first call made on that
// device (with that device current) and cached.
float* scores_address(int* code) {
  static std::mutex mu;
  static float* addr[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    *code = IVIT_ERR_CUDA;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_select_scores);
    if (e != cudaSuccess) {
      *code = IVIT_ERR_CUDA;
      return nullptr;
    }
    addr[dev] = static_cast<float*>(p);
  }
  *code = IVIT_OK;
  return addr[dev];
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Eq. 3 cosine of every token against its reference, one warp per token, into scores.
__global__ void noalloc_score_kernel(const float* __restrict__ e_cur, const float* __restrict__ e_ref,
                                     float* __restrict__ scores, int rows, int dim) {
  const int warps = blockDim.x >> 5;
  const int lane = threadIdx.x & 31;
  for (int r = blockIdx.x * warps + (threadIdx.x >> 5); r < rows; r += gridDim.x * warps) {
    const float4* a = reinterpret_cast<const float4*>(e_cur + static_cast<size_t>(r) * dim);
    const float4* b = reinterpret_cast<const float4*>(e_ref + static_cast<size_t>(r) * dim);
    float dot = 0.f, na = 0.f, nb = 0.f;
    for (int c = lane; c < dim / 4; c += 32) {
      const float4 x = a[c], y = b[c];
      dot += x.x * y.x + x.y * y.y + x.z * y.z + x.w * y.w;
      na += x.x * x.x + x.y * x.y + x.z * x.z + x.w * x.w;
      nb += y.x * y.x + y.y * y.y + y.z * y.z + y.w * y.w;
    }
    dot = warp_sum(dot);
    na = warp_sum(na);
    nb = warp_sum(nb);
    if (lane == 0) scores[r] = dot / fmaxf(sqrtf(na) * sqrtf(nb), 1e-12f);
  }
}

// One CTA per view: threshold or top-k flags compacted in index order (warp ballots and
// a block prefix sum) into idx[v][0..count), the rest of the row set to -1.
__global__ void noalloc_select_kernel(const float* __restrict__ scores, int N, int mode, float tau,
                                      int topk, int* __restrict__ idx, int* __restrict__ counts) {
  extern __shared__ float s_scores[];
  __shared__ int s_warp[32];
  __shared__ int s_total;
  const int v = blockIdx.x, i = threadIdx.x;
  const int lane = i & 31, warp = i >> 5, nwarps = blockDim.x >> 5;
  const float s = (i < N) ? scores[static_cast<size_t>(v) * N + i] : 0.f;
  bool flag = false;
  if (mode == IVIT_SEL_TOPK) {
    if (i < N) s_scores[i] = s;
    __syncthreads();
    if (i < N) {
      int rank = 0;
      for (int j = 0; j < N; ++j) {
        const float sj = s_scores[j];
        rank += (sj < s || (sj == s && j < i)) ? 1 : 0;
      }
      flag = rank < topk;
    }
  } else if (i < N) {
    flag = s < tau;
  }
  const unsigned ballot = __ballot_sync(0xffffffffu, flag);
  if (lane == 0) s_warp[warp] = __popc(ballot);
  __syncthreads();
  if (warp == 0) {
    const int x = lane < nwarps ? s_warp[lane] : 0;
    int incl = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane < nwarps) s_warp[lane] = incl - x;
    if (lane == 31) s_total = incl;
  }
  __syncthreads();
  const int total = s_total;
  int* row = idx + static_cast<size_t>(v) * N;
  if (flag) row[s_warp[warp] + __popc(ballot & ((1u << lane) - 1u))] = i;
  for (int k = total + i; k < N; k += blockDim.x) row[k] = -1;
  if (i == 0) counts[v] = total;
}

}  // namespace

extern "C" int ivit_select_noalloc(const float* e_cur_dev, const float* e_ref_dev, int32_t n_views,
                                   int32_t n_tok, int32_t dim, int32_t select_mode, float threshold,
                                   int32_t topk, int32_t* idx_out_dev, int32_t* counts_out_dev,
                                   void* stream) {
  if (!e_cur_dev || !e_ref_dev || !idx_out_dev || !counts_out_dev) {
    ivit::set_create_error("ivit_select_noalloc: null pointer");
    return IVIT_ERR_ARG;
  }
  // the score kernel reads both embedding sets with 128-bit loads, the selection kernel
  // stores 32-bit indices: a misaligned pointer is an argument error, never a device fault
  if ((reinterpret_cast<uintptr_t>(e_cur_dev) & 15u) || (reinterpret_cast<uintptr_t>(e_ref_dev) & 15u) ||
      (reinterpret_cast<uintptr_t>(idx_out_dev) & 3u) || (reinterpret_cast<uintptr_t>(counts_out_dev) & 3u)) {
    ivit::set_create_error("ivit_select_noalloc: e_cur/e_ref must be 16-byte aligned, idx/counts 4-byte aligned");
    return IVIT_ERR_ARG;
  }
  if (select_mode != IVIT_SEL_THRESHOLD && select_mode != IVIT_SEL_TOPK) {
    ivit::set_create_error("ivit_select_noalloc: bad select_mode");
    return IVIT_ERR_ARG;
  }
  if (n_views <= 0 || n_tok <= 0 || n_tok > 1024 || dim <= 0 || dim % 4) {
    ivit::set_create_error("ivit_select_noalloc: need n_views >= 1, 1 <= n_tok <= 1024, dim % 4 == 0");
    return IVIT_ERR_SHAPE;
  }
  if (static_cast<long long>(n_views) * n_tok > IVIT_NOALLOC_MAX_TOKENS) {
    ivit::set_create_error(
        "ivit_select_noalloc: n_views * n_tok exceeds IVIT_NOALLOC_MAX_TOKENS (65536)");
    return IVIT_ERR_SHAPE;
  }
  int code = IVIT_OK;
  float* scores = scores_address(&code);
  if (!scores) {
    ivit::set_create_error("ivit_select_noalloc: cudaGetSymbolAddress failed");
    return code;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int rows = n_views * n_tok;
  const int grid = (rows + 7) / 8 < 4096 ? (rows + 7) / 8 : 4096;
  noalloc_score_kernel<<<grid, 256, 0, s>>>(e_cur_dev, e_ref_dev, scores, rows, dim);
  const int threads = (n_tok + 31) / 32 * 32;
  const int k = topk < 0 ? 0 : topk;
  noalloc_select_kernel<<<n_views, threads, n_tok * sizeof(float), s>>>(scores, n_tok, select_mode,
                                                                        threshold, k, idx_out_dev,
                                                                        counts_out_dev);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    ivit::set_create_error(cudaGetErrorString(e));
    return IVIT_ERR_CUDA;
  }
  return IVIT_OK;
}
