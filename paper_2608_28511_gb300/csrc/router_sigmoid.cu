// The paper's router variant (Sec. 5.2): sigmoid scores, an expert bias that
// shapes the choice of experts only, gate values renormalised over the chosen
// experts, and a sequence-level load-balancing loss.
//   s = sigmoid(z); choose the K largest s + b (ties to the lower expert);
//   p_k = s_k / sum_{j in S} s_j;
//   per sequence g of S tokens: f_gi = E / (K S) #{t in g : i chosen},
//   P_gi = mean over t in g of s_ti / sum_j s_tj, L = coef / GBS sum_g,i f_gi P_gi.
// All reductions run in a fixed order, so results are bit-reproducible.
#include <math_constants.h>

#include "common.cuh"
#include "launch.h"

namespace moe {

namespace {

constexpr int kTokChunk = 256;  // tokens per partial sum of the balance statistics

__device__ __forceinline__ float sigmoidf_(float z) { return 1.0f / (1.0f + __expf(-z)); }

// One warp per token: scores, the biased choice, gate values and the token's
// score sum (for the balance statistics).
template <int VPL>
__global__ void __launch_bounds__(256) topk_sigmoid_kernel(const float* __restrict__ logits,
                                                           const float* __restrict__ bias, int64_t T, int E, int K,
                                                           int32_t* __restrict__ idx, float* __restrict__ prob,
                                                           float* __restrict__ rowsum) {
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= T) return;
  const float* row = logits + t * E;
  float s[VPL], key[VPL];
  unsigned alive = 0;
  float ssum = 0.f;
#pragma unroll
  for (int j = 0; j < VPL; ++j) {
    const int e = lane + 32 * j;
    s[j] = 0.f;
    key[j] = -CUDART_INF_F;
    if (e < E) {
      s[j] = sigmoidf_(__ldg(row + e));
      key[j] = s[j] + (bias ? __ldg(bias + e) : 0.f);
      if (key[j] != key[j]) key[j] = -CUDART_INF_F;
      alive |= 1u << j;
      ssum += s[j];
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) ssum += __shfl_xor_sync(0xffffffffu, ssum, off);
  int sel_i[kMaxK];
  float sel_s[kMaxK];
  float gsum = 0.f;
#pragma unroll
  for (int k = 0; k < kMaxK; ++k) {
    if (k < K) {
      float bv = -CUDART_INF_F, bs = 0.f;
      int bi = 0x7fffffff;
#pragma unroll
      for (int j = 0; j < VPL; ++j) {
        const int e = lane + 32 * j;
        if ((alive >> j) & 1u) {
          if (key[j] > bv || (key[j] == bv && e < bi)) { bv = key[j]; bi = e; bs = s[j]; }
        }
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
        const float os = __shfl_xor_sync(0xffffffffu, bs, off);
        if (ov > bv || (ov == bv && oi < bi)) { bv = ov; bi = oi; bs = os; }
      }
      if (lane == (bi & 31)) alive &= ~(1u << (bi >> 5));
      sel_i[k] = bi;
      sel_s[k] = bs;
      gsum += bs;
    }
  }
  const float inv = 1.0f / gsum;
#pragma unroll
  for (int k = 0; k < kMaxK; ++k) {
    if (k < K && lane == k) {
      idx[t * K + k] = sel_i[k];
      prob[t * K + k] = sel_s[k] * inv;
    }
  }
  if (lane == 0) rowsum[t] = ssum;
}

// Partial balance statistics: block (g, chunk) sums, for every expert, the
// normalised scores and the choice counts of up to kTokChunk tokens of
// sequence g, in token order.
__global__ void __launch_bounds__(256) aux_partial_kernel(const float* __restrict__ logits,
                                                          const float* __restrict__ rowsum,
                                                          const int32_t* __restrict__ idx, int64_t S, int E, int K,
                                                          int nchunk, float* __restrict__ psum,
                                                          int32_t* __restrict__ pcnt) {
  const int g = blockIdx.y, ch = blockIdx.x;
  const int64_t t0 = (int64_t)g * S + (int64_t)ch * kTokChunk;
  const int64_t t1 = min((int64_t)g * S + S, t0 + kTokChunk);
  __shared__ int32_t sidx[kTokChunk * kMaxK];
  __shared__ float srs[kTokChunk];
  for (int64_t i = threadIdx.x; i < (t1 - t0) * K; i += blockDim.x) sidx[i] = idx[t0 * K + i];
  for (int64_t i = threadIdx.x; i < t1 - t0; i += blockDim.x) srs[i] = rowsum[t0 + i];
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    float acc = 0.f;
    int cnt = 0;
    for (int64_t t = t0; t < t1; ++t) {
      acc += sigmoidf_(logits[t * E + e]) / srs[t - t0];
      for (int k = 0; k < K; ++k) cnt += sidx[(t - t0) * K + k] == e;
    }
    const int64_t o = ((int64_t)g * nchunk + ch) * E + e;
    psum[o] = acc;
    pcnt[o] = cnt;
  }
}

// f [GBS, E] and the loss: one block, chunks and then (g, e) summed in order.
__global__ void __launch_bounds__(256) aux_finalize_kernel(const float* __restrict__ psum,
                                                           const int32_t* __restrict__ pcnt, int GBS, int64_t S,
                                                           int E, int K, int nchunk, float coef,
                                                           float* __restrict__ f_out, float* __restrict__ loss) {
  __shared__ float red[256];
  float part = 0.f;
  for (int i = threadIdx.x; i < GBS * E; i += blockDim.x) {
    const int g = i / E, e = i % E;
    float P = 0.f;
    int64_t cnt = 0;
    for (int ch = 0; ch < nchunk; ++ch) {
      const int64_t o = ((int64_t)g * nchunk + ch) * E + e;
      P += psum[o];
      cnt += pcnt[o];
    }
    const float f = (float)((double)E / ((double)K * (double)S) * (double)cnt);
    f_out[i] = f;
    part += f * (P / (float)S);
  }
  red[threadIdx.x] = part;
  __syncthreads();
  for (int off = 128; off > 0; off >>= 1) {
    if (threadIdx.x < off) red[threadIdx.x] += red[threadIdx.x + off];
    __syncthreads();
  }
  if (threadIdx.x == 0) loss[0] = coef / (float)GBS * red[0];
}

// One warp per token: gradient of the gate values of the chosen experts plus
// aux_grad times the balance loss with respect to the logits (all E entries),
// and its bf16 copy.
__global__ void __launch_bounds__(256) route_dz_sigmoid_kernel(
    const float* __restrict__ logits, const int32_t* __restrict__ idx, const float* __restrict__ prob,
    const float* __restrict__ dprob, const float* __restrict__ f, int64_t T, int64_t S, int E, int K, float cscale,
    float* __restrict__ dz, bf16* __restrict__ dz16, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= T) return;
  const int64_t g = t / S;
  const float* row = logits + t * E;
  const float* fg = f + g * E;
  // score sum and sum_i c_i shat_i numerator over the whole row
  float ssum = 0.f, csum = 0.f;
  for (int e = lane; e < E; e += 32) {
    const float sv = sigmoidf_(row[e]);
    ssum += sv;
    csum += cscale * fg[e] * sv;
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    ssum += __shfl_xor_sync(0xffffffffu, ssum, off);
    csum += __shfl_xor_sync(0xffffffffu, csum, off);
  }
  const float cbar = csum / ssum;  // sum_i c_i shat_i
  // gate path: chosen experts' scores, gate values and incoming gradients
  int my_e = -1;
  float my_p = 0.f, my_dp = 0.f, my_s = 0.f;
  if (lane < K) {
    my_e = idx[t * K + lane];
    if (my_e >= 0 && my_e < E) {
      my_p = prob[t * K + lane];
      my_dp = dprob[t * K + lane];
      my_s = sigmoidf_(row[my_e]);
    } else {
      set_error(err, kErrIndex);  // an out-of-range expert index contributes nothing
      my_e = -1;
    }
  }
  float dot = my_p * my_dp, gs = my_s;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    dot += __shfl_xor_sync(0xffffffffu, dot, off);
    gs += __shfl_xor_sync(0xffffffffu, gs, off);
  }
  const float my_gate = (my_dp - dot) / gs;
  for (int e0 = 0; e0 < E; e0 += 32) {
    const int e = e0 + lane;
    float gate = 0.f;
    for (int k = 0; k < K; ++k) {
      const int ek = __shfl_sync(0xffffffffu, my_e, k);
      const float gk = __shfl_sync(0xffffffffu, my_gate, k);
      if (ek == e) gate = gk;
    }
    if (e < E) {
      const float sv = sigmoidf_(row[e]);
      const float ds = gate + (cscale * fg[e] - cbar) / ssum;
      const float v = sv * (1.0f - sv) * ds;
      dz[t * E + e] = v;
      if (dz16) dz16[t * E + e] = __float2bfloat16_rn(v);
    }
  }
}

}  // namespace

size_t route_sigmoid_fwd_ws_bytes(int64_t T, int64_t S, int64_t GBS, int E) {
  const int64_t nchunk = (S + kTokChunk - 1) / kTokChunk;
  return (size_t)T * 4 + (size_t)GBS * nchunk * E * 8 + 512;
}

cudaError_t launch_route_sigmoid_select(const Ctx& c, const float* logits, const float* bias, int64_t T, int64_t S,
                                        int64_t GBS, int E, int K, float coef, int32_t* idx, float* prob,
                                        float* f_out, float* loss, void* ws) {
  if (T == 0) return cudaSuccess;
  float* rowsum = static_cast<float*>(ws);
  const int64_t nchunk = (S + kTokChunk - 1) / kTokChunk;
  float* psum = rowsum + ((T + 63) / 64) * 64;
  int32_t* pcnt = reinterpret_cast<int32_t*>(psum + GBS * nchunk * E);
  {
    const int warps = 8;
    dim3 grid((unsigned)((T + warps - 1) / warps)), block(32 * warps);
    KernelScope ks("topk_sigmoid", c.stream);
    const int vpl = (E + 31) / 32;
    if (vpl <= 1) topk_sigmoid_kernel<1><<<grid, block, 0, c.stream>>>(logits, bias, T, E, K, idx, prob, rowsum);
    else if (vpl <= 2) topk_sigmoid_kernel<2><<<grid, block, 0, c.stream>>>(logits, bias, T, E, K, idx, prob, rowsum);
    else if (vpl <= 4) topk_sigmoid_kernel<4><<<grid, block, 0, c.stream>>>(logits, bias, T, E, K, idx, prob, rowsum);
    else topk_sigmoid_kernel<8><<<grid, block, 0, c.stream>>>(logits, bias, T, E, K, idx, prob, rowsum);
  }
  cudaError_t st = cudaGetLastError();
  if (st != cudaSuccess) return st;
  {
    KernelScope ks("aux_partial", c.stream);
    aux_partial_kernel<<<dim3((unsigned)nchunk, (unsigned)GBS), 256, 0, c.stream>>>(logits, rowsum, idx, S, E, K,
                                                                                  (int)nchunk, psum, pcnt);
  }
  st = cudaGetLastError();
  if (st != cudaSuccess) return st;
  {
    KernelScope ks("aux_finalize", c.stream);
    aux_finalize_kernel<<<1, 256, 0, c.stream>>>(psum, pcnt, (int)GBS, S, E, K, (int)nchunk, coef, f_out, loss);
  }
  return cudaGetLastError();
}

cudaError_t launch_route_dz_sigmoid(const Ctx& c, const float* logits, const int32_t* idx, const float* prob,
                                    const float* dprob, const float* f, int64_t T, int64_t S, int64_t GBS, int E,
                                    int K, float coef, float aux_grad, float* dz, void* dz16) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  dim3 grid((unsigned)((T + warps - 1) / warps)), block(32 * warps);
  const float cscale = aux_grad * coef / ((float)GBS * (float)S);
  KernelScope ks("route_dz_sigmoid", c.stream);
  route_dz_sigmoid_kernel<<<grid, block, 0, c.stream>>>(logits, idx, prob, dprob, f, T, S, E, K, cscale, dz,
                                                        static_cast<bf16*>(dz16), c.err);
  return cudaGetLastError();
}

}  // namespace moe
