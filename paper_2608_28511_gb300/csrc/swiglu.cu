// SwiGLU backward as a streaming kernel: from dA [rows, F] (the GEMM-2 input
// gradient) and the saved pre-activation h [rows, 2F] (packed gate/up blocks
// of 64) it writes dH [rows, 2F] in the same packed order:
//   s = sigmoid(g),  dg = dA u s (1 + g (1 - s)),  du = dA g s.
// HBM-bound: reads dA and h once, writes dH once, 16-byte vectors.  sigmoid
// takes the fast exponential and a correctly rounded reciprocal.
// Also the squared-ReLU backward of the shared expert (same access pattern).
#include "common.cuh"
#include "launch.h"

namespace moe {

// Each thread takes two 16-byte vectors of dA per pass (i and i + stride),
// with all six loads issued before any arithmetic; IDX is the index type
// (32-bit when rows * F / NV fits).
template <typename T, typename IDX>
__device__ __forceinline__ void swiglu_bwd_vec(const float (&a)[Vec<T>::N], const float (&g)[Vec<T>::N],
                                               const float (&u)[Vec<T>::N], T* __restrict__ dH, IDX cg) {
  constexpr int NV = Vec<T>::N;
  float dg[NV], du[NV];
#pragma unroll
  for (int j = 0; j < NV; ++j) {
    const float s = __frcp_rn(1.0f + __expf(-g[j]));
    dg[j] = a[j] * u[j] * s * (1.0f + g[j] * (1.0f - s));
    du[j] = a[j] * g[j] * s;
  }
  st_stream(reinterpret_cast<uint4*>(dH + cg), pack16<T>(dg));
  st_stream(reinterpret_cast<uint4*>(dH + cg + 64), pack16<T>(du));
}

template <typename T, typename IDX>
__global__ void __launch_bounds__(256) swiglu_bwd_kernel(const uint4* __restrict__ dA, const T* __restrict__ h,
                                                         int64_t rows, int F, T* __restrict__ dH) {
  constexpr int NV = Vec<T>::N;
  const IDX vpr = (IDX)(F / NV);  // 16-byte vectors of dA per row
  const IDX total = (IDX)rows * vpr;
  const IDX stride = (IDX)gridDim.x * blockDim.x;
  auto col = [&](IDX i) -> IDX {  // element offset of vector i's gate block in h / dH
    const IDX r = i / vpr;
    const IDX f = (i - r * vpr) * NV;
    return r * 2 * F + (f / 64) * 128 + (f % 64);
  };
  for (IDX i = (IDX)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += 2 * stride) {
    const IDX i2 = i + stride;
    const bool two = i2 < total;
    const IDX c1 = col(i), c2 = two ? col(i2) : c1;
    float a1[NV], g1[NV], u1[NV], a2[NV], g2[NV], u2[NV];
    const uint4 va1 = ld_stream(dA + i), vg1 = ld_stream(reinterpret_cast<const uint4*>(h + c1)),
                vu1 = ld_stream(reinterpret_cast<const uint4*>(h + c1 + 64));
    uint4 va2 = va1, vg2 = vg1, vu2 = vu1;
    if (two) {
      va2 = ld_stream(dA + i2);
      vg2 = ld_stream(reinterpret_cast<const uint4*>(h + c2));
      vu2 = ld_stream(reinterpret_cast<const uint4*>(h + c2 + 64));
    }
    unpack16<T>(va1, a1);
    unpack16<T>(vg1, g1);
    unpack16<T>(vu1, u1);
    swiglu_bwd_vec<T, IDX>(a1, g1, u1, dH, c1);
    if (two) {
      unpack16<T>(va2, a2);
      unpack16<T>(vg2, g2);
      unpack16<T>(vu2, u2);
      swiglu_bwd_vec<T, IDX>(a2, g2, u2, dH, c2);
    }
  }
}

cudaError_t launch_swiglu_bwd(const Ctx& c, DType dt, const void* dA, const void* h, int64_t rows, int F,
                              void* dH) {
  if (rows == 0) return cudaSuccess;
  const int64_t vecs = rows * F * (int64_t)dsize(dt) / 16;
  const int64_t want = (vecs + 255) / 256;
  const int blocks = (int)(want < (int64_t)c.num_sms * 16 ? want : (int64_t)c.num_sms * 16);
  KernelScope ks("swiglu_bwd", c.stream);
  // 32-bit indexing when every element offset of h fits
  const bool i32 = rows * 2 * (int64_t)F < ((int64_t)1 << 31);
  if (dt == DType::BF16) {
    if (i32)
      swiglu_bwd_kernel<bf16, int32_t><<<blocks, 256, 0, c.stream>>>((const uint4*)dA, (const bf16*)h, rows, F,
                                                                     (bf16*)dH);
    else
      swiglu_bwd_kernel<bf16, int64_t><<<blocks, 256, 0, c.stream>>>((const uint4*)dA, (const bf16*)h, rows, F,
                                                                     (bf16*)dH);
  } else {
    if (i32)
      swiglu_bwd_kernel<float, int32_t><<<blocks, 256, 0, c.stream>>>((const uint4*)dA, (const float*)h, rows, F,
                                                                      (float*)dH);
    else
      swiglu_bwd_kernel<float, int64_t><<<blocks, 256, 0, c.stream>>>((const uint4*)dA, (const float*)h, rows, F,
                                                                      (float*)dH);
  }
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
