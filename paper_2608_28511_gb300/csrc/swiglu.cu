// SwiGLU backward as a streaming kernel: from dA [rows, F] (the GEMM-2 input
// gradient) and the saved pre-activation h [rows, 2F] (packed gate/up blocks
// of 64) it writes dH [rows, 2F] in the same packed order:
//   s = sigmoid(g),  dg = dA u s (1 + g (1 - s)),  du = dA g s.
// HBM-bound: reads dA and h once, writes dH once, 16-byte vectors.
// Also the squared-ReLU backward of the shared expert (same access pattern).
#include "common.cuh"
#include "launch.h"

namespace moe {

template <typename T>
__global__ void __launch_bounds__(256) swiglu_bwd_kernel(const uint4* __restrict__ dA, const T* __restrict__ h,
                                                         int64_t rows, int F, T* __restrict__ dH) {
  constexpr int NV = Vec<T>::N;
  const int64_t vpr = F / NV;  // 16-byte vectors of dA per row
  const int64_t total = rows * vpr;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / vpr;
    const int f = (int)(i % vpr) * NV;
    const int64_t cg = r * 2 * F + (f / 64) * 128 + (f % 64);
    float a[NV], g[NV], u[NV], dg[NV], du[NV];
    unpack16<T>(ld_stream(dA + i), a);
    unpack16<T>(ld_stream(reinterpret_cast<const uint4*>(h + cg)), g);
    unpack16<T>(ld_stream(reinterpret_cast<const uint4*>(h + cg + 64)), u);
#pragma unroll
    for (int j = 0; j < NV; ++j) {
      const float s = 1.0f / (1.0f + __expf(-g[j]));
      dg[j] = a[j] * u[j] * s * (1.0f + g[j] * (1.0f - s));
      du[j] = a[j] * g[j] * s;
    }
    st_stream(reinterpret_cast<uint4*>(dH + cg), pack16<T>(dg));
    st_stream(reinterpret_cast<uint4*>(dH + cg + 64), pack16<T>(du));
  }
}

cudaError_t launch_swiglu_bwd(const Ctx& c, DType dt, const void* dA, const void* h, int64_t rows, int F,
                              void* dH) {
  if (rows == 0) return cudaSuccess;
  const int64_t vecs = rows * F * (int64_t)dsize(dt) / 16;
  const int64_t want = (vecs + 255) / 256;
  const int blocks = (int)(want < (int64_t)c.num_sms * 16 ? want : (int64_t)c.num_sms * 16);
  KernelScope ks("swiglu_bwd", c.stream);
  if (dt == DType::BF16)
    swiglu_bwd_kernel<bf16><<<blocks, 256, 0, c.stream>>>((const uint4*)dA, (const bf16*)h, rows, F, (bf16*)dH);
  else
    swiglu_bwd_kernel<float><<<blocks, 256, 0, c.stream>>>((const uint4*)dA, (const float*)h, rows, F,
                                                           (float*)dH);
  return cudaGetLastError();
}

// Squared-ReLU backward of the shared expert: dh = 2 max(h, 0) dA, elementwise
// over 16-byte vectors (dh may alias dA).
template <typename T>
__global__ void __launch_bounds__(256) relusq_bwd_kernel(const uint4* dA, const uint4* __restrict__ h, int64_t nvec,
                                                         uint4* dh) {
  constexpr int NV = Vec<T>::N;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nvec; i += (int64_t)gridDim.x * blockDim.x) {
    float a[NV], hv[NV];
    unpack16<T>(ld_stream(dA + i), a);
    unpack16<T>(ld_stream(h + i), hv);
#pragma unroll
    for (int j = 0; j < NV; ++j) a[j] *= 2.0f * fmaxf(hv[j], 0.f);
    st_stream(dh + i, pack16<T>(a));
  }
}

cudaError_t launch_relusq_bwd(const Ctx& c, DType dt, const void* dA, const void* h, int64_t n, void* dh) {
  if (n == 0) return cudaSuccess;
  const int64_t vecs = n * (int64_t)dsize(dt) / 16;
  const int64_t want = (vecs + 255) / 256;
  const int blocks = (int)(want < (int64_t)c.num_sms * 16 ? want : (int64_t)c.num_sms * 16);
  KernelScope ks("relusq_bwd", c.stream);
  if (dt == DType::BF16)
    relusq_bwd_kernel<bf16><<<blocks, 256, 0, c.stream>>>((const uint4*)dA, (const uint4*)h, vecs, (uint4*)dh);
  else
    relusq_bwd_kernel<float><<<blocks, 256, 0, c.stream>>>((const uint4*)dA, (const uint4*)h, vecs, (uint4*)dh);
  return cudaGetLastError();
}

}  // namespace moe
