// The 2-step action combine of Sec. III-C (Eq. 9): the final action state from the two
// anchor velocities of the flow-matching solver,
//   x_T[s][i] = x_0[s][i] + alpha[s] v_0[s][i] + beta[s] v_7[s][i] + b[s][i].
// The velocity network and the adaptor that predicts (alpha, beta, b) are not part of
// this library; the caller passes their outputs.  Elementwise and HBM-bound: 128-bit
// loads and stores when the action width allows, a grid-stride loop sized to the SMs.
#include "internal.h"
#include "ptx.cuh"
#include "ivit.h"

namespace ivit {
namespace {

__global__ void action_combine_kernel(const float* __restrict__ x0, const float* __restrict__ v0,
                                      const float* __restrict__ v7, const float* __restrict__ alpha,
                                      const float* __restrict__ beta, const float* __restrict__ b,
                                      int dim, long long n, int vec4, float* __restrict__ xT) {
  pdl_wait();
  pdl_launch_dependents();
  const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
  if (vec4) {
    const long long n4 = n >> 2;
    const float4* x4 = reinterpret_cast<const float4*>(x0);
    const float4* a4 = reinterpret_cast<const float4*>(v0);
    const float4* c4 = reinterpret_cast<const float4*>(v7);
    const float4* b4 = reinterpret_cast<const float4*>(b);
    float4* y4 = reinterpret_cast<float4*>(xT);
    for (long long k = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; k < n4; k += stride) {
      const int s = static_cast<int>((k << 2) / dim);
      const float al = alpha[s], be = beta[s];
      const float4 x = x4[k], p = a4[k], q = c4[k];
      const float4 o = b ? b4[k] : make_float4(0.f, 0.f, 0.f, 0.f);
      y4[k] = make_float4(fmaf(be, q.x, fmaf(al, p.x, x.x)) + o.x, fmaf(be, q.y, fmaf(al, p.y, x.y)) + o.y,
                          fmaf(be, q.z, fmaf(al, p.z, x.z)) + o.z, fmaf(be, q.w, fmaf(al, p.w, x.w)) + o.w);
    }
  } else {
    for (long long k = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; k < n; k += stride) {
      const int s = static_cast<int>(k / dim);
      xT[k] = fmaf(beta[s], v7[k], fmaf(alpha[s], v0[k], x0[k])) + (b ? b[k] : 0.f);
    }
  }
}

}  // namespace
}  // namespace ivit

extern "C" int ivit_action_combine(const float* x0_dev, const float* v0_dev, const float* v7_dev,
                                   const float* alpha_dev, const float* beta_dev, const float* b_dev,
                                   int32_t batch, int32_t dim, float* xT_dev, void* stream) {
  if (batch < 0 || dim < 0) return IVIT_ERR_ARG;
  const long long n = static_cast<long long>(batch) * dim;
  if (n == 0) return IVIT_OK;
  if (!x0_dev || !v0_dev || !v7_dev || !alpha_dev || !beta_dev || !xT_dev) return IVIT_ERR_ARG;
  // 128-bit accesses need rows of a multiple of 4 floats and 16-byte aligned arrays;
  // any other layout takes the scalar loop (alignment 4 bytes, checked here).
  auto aligned = [](const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; };
  for (const void* p : {static_cast<const void*>(x0_dev), static_cast<const void*>(v0_dev),
                        static_cast<const void*>(v7_dev), static_cast<const void*>(alpha_dev),
                        static_cast<const void*>(beta_dev), static_cast<const void*>(b_dev),
                        static_cast<const void*>(xT_dev)})
    if (p && !aligned(p, 4)) return IVIT_ERR_ARG;
  const bool vec4 = (dim & 3) == 0 && aligned(x0_dev, 16) && aligned(v0_dev, 16) && aligned(v7_dev, 16) &&
                    aligned(xT_dev, 16) && (!b_dev || aligned(b_dev, 16));
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev))
    return IVIT_ERR_CUDA;
  const long long items = vec4 ? n / 4 : n;
  const long long blocks = (items + 255) / 256;
  const int grid = static_cast<int>(blocks < 4LL * sms ? blocks : 4LL * sms);
  const cudaError_t e = ivit::launch_ex(ivit::action_combine_kernel, dim3(grid), dim3(256), 0,
                                        static_cast<cudaStream_t>(stream), 1, x0_dev, v0_dev, v7_dev, alpha_dev,
                                        beta_dev, b_dev, static_cast<int>(dim), n, vec4 ? 1 : 0, xT_dev);
  return e == cudaSuccess ? IVIT_OK : IVIT_ERR_CUDA;
}
