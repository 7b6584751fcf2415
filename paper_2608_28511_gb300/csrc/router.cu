// Router kernels: top-K with renormalised probabilities, and
// the router backward dz = p (dp - sum_k p_k dp_k) on the chosen set.
#include <math_constants.h>

#include "common.cuh"
#include "launch.h"
#include "select.cuh"

namespace moe {

struct Identity {
  __device__ __forceinline__ float operator()(float z) const { return z; }
};

// Four threads per token (select.cuh): the K largest logits, ties to the lower
// expert index (reading R2), NaN as -inf, ordered by descending logit.  The
// probabilities are exp(z_k - z_max) normalised over the K chosen logits,
// which equals the full softmax renormalised over the chosen set (reading R1).
template <int KM>
__global__ void __launch_bounds__(256) topk_kernel(const float* __restrict__ logits, int64_t T, int E, int K,
                                                   int tpb, int32_t* __restrict__ idx, float* __restrict__ prob) {
  extern __shared__ __align__(16) float zs[];  // [tpb][E]
  const int tid = threadIdx.x;
  const int64_t t0 = (int64_t)blockIdx.x * tpb;
  const int n = (int)min((int64_t)tpb, T - t0);
  sel::stage_rows(logits + t0 * E, zs, n * E, Identity());
  __syncthreads();
  const int q = tid >> 2, r = tid & 3;
  const bool active = q < n;
  uint64_t win[KM];
  float unused;
  sel::quad_topk<KM>(zs + (int64_t)q * E, nullptr, E, K, r, q, active, win, &unused);
  if (!active) return;
  const float zmax = sel::unpack_key(win[0]);
  float w[KM];
  float sum = 0.f;
#pragma unroll
  for (int k = 0; k < KM; ++k) {
    w[k] = 0.f;
    if (k < K) {
      w[k] = expf(sel::unpack_key(win[k]) - zmax);
      sum += w[k];
    }
  }
  const float inv = 1.0f / sum;
  const int64_t o = (t0 + q) * K;
#pragma unroll
  for (int k = 0; k < KM; ++k) {
    if (k < K && (k & 3) == r) {
      idx[o + k] = sel::unpack_e(win[k]);
      prob[o + k] = w[k] * inv;
    }
  }
}

cudaError_t launch_topk(const Ctx& c, const float* logits, int64_t T, int E, int K, int32_t* idx, float* prob) {
  if (T == 0) return cudaSuccess;
  const int tpb = sel::tokens_per_block(E);
  const dim3 grid((unsigned)((T + tpb - 1) / tpb));
  const size_t smem = (size_t)tpb * E * 4;
  KernelScope ks("topk", c.stream);
  switch (sel::k_bound(K)) {
    case 2: topk_kernel<2><<<grid, 4 * tpb, smem, c.stream>>>(logits, T, E, K, tpb, idx, prob); break;
    case 4: topk_kernel<4><<<grid, 4 * tpb, smem, c.stream>>>(logits, T, E, K, tpb, idx, prob); break;
    case 8: topk_kernel<8><<<grid, 4 * tpb, smem, c.stream>>>(logits, T, E, K, tpb, idx, prob); break;
    default: topk_kernel<16><<<grid, 4 * tpb, smem, c.stream>>>(logits, T, E, K, tpb, idx, prob); break;
  }
  return cudaGetLastError();
}

// One warp per token: dz[t, e] = p_k (dp_k - c) if e = idx[t, k], else 0,
// with c = sum_k p_k dp_k.  Every entry of the row is written once.
__global__ void __launch_bounds__(256) route_dz_kernel(const int32_t* __restrict__ idx,
                                                       const float* __restrict__ prob,
                                                       const float* __restrict__ dprob, int64_t T, int E, int K,
                                                       float* __restrict__ dz, bf16* __restrict__ dz_bf16,
                                                       int64_t ld16) {
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
      if (dz_bf16) dz_bf16[t * ld16 + e] = __float2bfloat16_rn(val);
    }
  }
}

cudaError_t launch_route_dz(const Ctx& c, const int32_t* idx, const float* prob, const float* dprob, int64_t T,
                            int E, int K, float* dz, void* dz_bf16, int64_t ld16) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  dim3 grid((unsigned)((T + warps - 1) / warps)), block(32 * warps);
  KernelScope ks("route_dz", c.stream);
  route_dz_kernel<<<grid, block, 0, c.stream>>>(idx, prob, dprob, T, E, K, dz, (bf16*)dz_bf16,
                                                 ld16 > 0 ? ld16 : E);
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
