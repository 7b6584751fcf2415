// Router kernels: warp-per-token top-K with renormalised probabilities, and
// the router backward dz = p (dp - sum_k p_k dp_k) on the chosen set.
#include <math_constants.h>

#include "common.cuh"
#include "launch.h"

namespace moe {

// One warp per token.  Lane l holds logits l, l + 32, ... (VPL per lane).  K
// rounds of a warp arg-max pick the largest remaining logit, ties to the lower
// expert index (reading R2); NaN is treated as -inf.  The probabilities are
// exp(z_k - z_max) normalised over the K chosen logits, which equals the full
// softmax renormalised over the chosen set (reading R1).
template <int VPL>
__global__ void __launch_bounds__(256) topk_kernel(const float* __restrict__ logits, int64_t T, int E, int K,
                                                   int32_t* __restrict__ idx, float* __restrict__ prob) {
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= T) return;
  const float* row = logits + t * E;
  float v[VPL];
  unsigned alive = 0;
#pragma unroll
  for (int j = 0; j < VPL; ++j) {
    const int e = lane + 32 * j;
    float z = -CUDART_INF_F;
    if (e < E) {
      z = __ldg(row + e);
      if (z != z) z = -CUDART_INF_F;
      alive |= 1u << j;
    }
    v[j] = z;
  }
  float sel_v[kMaxK];
  int sel_i[kMaxK];
#pragma unroll
  for (int k = 0; k < kMaxK; ++k) {
    if (k < K) {
      float bv = -CUDART_INF_F;
      int bi = 0x7fffffff;
#pragma unroll
      for (int j = 0; j < VPL; ++j) {
        const int e = lane + 32 * j;
        if ((alive >> j) & 1u) {
          if (v[j] > bv || (v[j] == bv && e < bi)) { bv = v[j]; bi = e; }
        }
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
        if (ov > bv || (ov == bv && oi < bi)) { bv = ov; bi = oi; }
      }
      if (lane == (bi & 31)) alive &= ~(1u << (bi >> 5));
      sel_v[k] = bv;
      sel_i[k] = bi;
    }
  }
  const float zmax = sel_v[0];
  float w[kMaxK];
  float sum = 0.f;
#pragma unroll
  for (int k = 0; k < kMaxK; ++k) {
    if (k < K) {
      w[k] = expf(sel_v[k] - zmax);
      sum += w[k];
    }
  }
  const float inv = 1.0f / sum;
#pragma unroll
  for (int k = 0; k < kMaxK; ++k) {
    if (k < K && lane == k) {
      idx[t * K + k] = sel_i[k];
      prob[t * K + k] = w[k] * inv;
    }
  }
}

cudaError_t launch_topk(const Ctx& c, const float* logits, int64_t T, int E, int K, int32_t* idx, float* prob) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  dim3 grid((unsigned)((T + warps - 1) / warps)), block(32 * warps);
  KernelScope ks("topk", c.stream);
  const int vpl = (E + 31) / 32;
  if (vpl <= 1) topk_kernel<1><<<grid, block, 0, c.stream>>>(logits, T, E, K, idx, prob);
  else if (vpl <= 2) topk_kernel<2><<<grid, block, 0, c.stream>>>(logits, T, E, K, idx, prob);
  else if (vpl <= 4) topk_kernel<4><<<grid, block, 0, c.stream>>>(logits, T, E, K, idx, prob);
  else topk_kernel<8><<<grid, block, 0, c.stream>>>(logits, T, E, K, idx, prob);
  return cudaGetLastError();
}

// One warp per token: dz[t, e] = p_k (dp_k - c) if e = idx[t, k], else 0,
// with c = sum_k p_k dp_k.  Every entry of the row is written once.
__global__ void __launch_bounds__(256) route_dz_kernel(const int32_t* __restrict__ idx,
                                                       const float* __restrict__ prob,
                                                       const float* __restrict__ dprob, int64_t T, int E, int K,
                                                       float* __restrict__ dz, bf16* __restrict__ dz_bf16) {
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= T) return;
  int my_e = -1;
  float my_p = 0.f, my_dp = 0.f;
  if (lane < K) {
    my_e = idx[t * K + lane];
    my_p = prob[t * K + lane];
    my_dp = dprob[t * K + lane];
  }
  float cdot = my_p * my_dp;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) cdot += __shfl_xor_sync(0xffffffffu, cdot, off);
  const float my_dz = my_p * (my_dp - cdot);
  for (int e0 = 0; e0 < E; e0 += 32) {
    const int e = e0 + lane;
    float val = 0.f;
    for (int k = 0; k < K; ++k) {
      const int ek = __shfl_sync(0xffffffffu, my_e, k);
      const float dk = __shfl_sync(0xffffffffu, my_dz, k);
      if (ek == e) val = dk;
    }
    if (e < E) {
      dz[t * E + e] = val;
      if (dz_bf16) dz_bf16[t * E + e] = __float2bfloat16_rn(val);
    }
  }
}

cudaError_t launch_route_dz(const Ctx& c, const int32_t* idx, const float* prob, const float* dprob, int64_t T,
                            int E, int K, float* dz, void* dz_bf16) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  dim3 grid((unsigned)((T + warps - 1) / warps)), block(32 * warps);
  KernelScope ks("route_dz", c.stream);
  route_dz_kernel<<<grid, block, 0, c.stream>>>(idx, prob, dprob, T, E, K, dz, (bf16*)dz_bf16);
  return cudaGetLastError();
}

// Deterministic reduction of split-K partial products: each output is the
// in-order sum of its S partials.
__global__ void __launch_bounds__(256) sum_splits_kernel(const float4* __restrict__ part, int S, int64_t n4,
                                                         float4* __restrict__ out) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += (int64_t)gridDim.x * blockDim.x) {
    float4 a = __ldcs(part + i);
    for (int s = 1; s < S; ++s) {
      const float4 b = __ldcs(part + (int64_t)s * n4 + i);
      a.x += b.x;
      a.y += b.y;
      a.z += b.z;
      a.w += b.w;
    }
    out[i] = a;
  }
}

cudaError_t launch_sum_splits(const Ctx& c, const float* part, int S, int64_t n, float* out) {
  const int64_t n4 = n / 4;
  const int64_t want = (n4 + 255) / 256;
  const int blocks = (int)(want < (int64_t)c.num_sms * 8 ? want : (int64_t)c.num_sms * 8);
  KernelScope ks("sum_splits", c.stream);
  sum_splits_kernel<<<blocks, 256, 0, c.stream>>>((const float4*)part, S, n4, (float4*)out);
  return cudaGetLastError();
}

}  // namespace moe
