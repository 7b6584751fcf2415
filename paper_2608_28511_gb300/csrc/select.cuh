// Top-K selection over the E experts of each token, shared by the softmax
// router (keys = logits) and the sigmoid router (keys = sigmoid scores + expert
// bias).  Four threads per token: a block stages the rows of its tokens in
// shared memory, each thread of a token's quad keeps a sorted list of the K
// best (key, expert) pairs of every fourth column, and the quad merges its
// four lists by K rounds of a two-level shuffle maximum.  Ties go to the lower
// expert index: a pair is packed into one 64-bit integer,
//   (order-preserving bits of the key) << 32 | ~expert,
// so the larger integer is the better pair.  NaN keys count as -inf.
#pragma once

#include <math_constants.h>

#include "common.cuh"

namespace moe {
namespace sel {

// Tokens per block: the staged rows (tokens x E fp32) take at most 32 KB.
inline int tokens_per_block(int E) { return E <= 128 ? 64 : 32; }
inline int k_bound(int K) { return K <= 2 ? 2 : K <= 4 ? 4 : K <= 8 ? 8 : 16; }

__device__ __forceinline__ uint64_t pack(float key, int e) {
  if (key != key) key = -CUDART_INF_F;
  if (key == 0.f) key = 0.f;  // -0 ties with +0
  const uint32_t b = __float_as_uint(key);
  const uint32_t o = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
  return ((uint64_t)o << 32) | (uint32_t)~(uint32_t)e;
}
__device__ __forceinline__ int unpack_e(uint64_t p) { return (int)~(uint32_t)p; }
__device__ __forceinline__ float unpack_key(uint64_t p) {
  const uint32_t o = (uint32_t)(p >> 32);
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}

__device__ __forceinline__ uint64_t shfl_xor64(uint64_t v, int m) {
  const uint32_t lo = __shfl_xor_sync(0xffffffffu, (uint32_t)v, m);
  const uint32_t hi = __shfl_xor_sync(0xffffffffu, (uint32_t)(v >> 32), m);
  return ((uint64_t)hi << 32) | lo;
}

// Copies n*E consecutive floats from global memory into shared memory, with
// eight loads in flight per thread, applying f on the way.
template <typename F>
__device__ __forceinline__ void stage_rows(const float* __restrict__ src, float* __restrict__ dst, int total, F f) {
  const int step = blockDim.x, tid = threadIdx.x;
  if (((reinterpret_cast<uintptr_t>(src) & 15) == 0) && (total & 3) == 0) {
    const float4* s4 = reinterpret_cast<const float4*>(src);
    float4* d4 = reinterpret_cast<float4*>(dst);
    const int n4 = total >> 2;
    int i = tid;
    for (; i + 7 * step < n4; i += 8 * step) {
      float4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = __ldg(s4 + i + u * step);
#pragma unroll
      for (int u = 0; u < 8; ++u) d4[i + u * step] = make_float4(f(v[u].x), f(v[u].y), f(v[u].z), f(v[u].w));
    }
    for (; i < n4; i += step) {
      const float4 v = __ldg(s4 + i);
      d4[i] = make_float4(f(v.x), f(v.y), f(v.z), f(v.w));
    }
  } else {
    int i = tid;
    for (; i + 7 * step < total; i += 8 * step) {
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = __ldg(src + i + u * step);
#pragma unroll
      for (int u = 0; u < 8; ++u) dst[i + u * step] = f(v[u]);
    }
    for (; i < total; i += step) dst[i] = f(__ldg(src + i));
  }
}

// The quad's K best pairs of one staged row, best first, in every thread of
// the quad (win[0 .. K-1]; entries K .. KM-1 are 0).  row: the token's staged
// values; bias: added to the value to form the key (NULL: key = value);
// r: the thread's place in the quad; q: the token's place in the block (for a
// conflict-free column rotation); active: the token exists.  Also returns the
// quad's sum of the row's values in *rowsum (fixed order).
template <int KM>
__device__ __forceinline__ void quad_topk(const float* __restrict__ row, const float* __restrict__ bias, int E, int K,
                                          int r, int q, bool active, uint64_t (&win)[KM], float* rowsum) {
  // Sorted list in slots KM-K .. KM-1 (best first) during the scan; the slots
  // below hold walls that nothing passes, so the K-th best is slot KM-1.
  const int k0 = KM - K;
  uint64_t L[KM];
#pragma unroll
  for (int k = 0; k < KM; ++k) L[k] = k < k0 ? ~0ull : 0ull;
  float sum = 0.f;
  const int J = (E + 3) >> 2;
  int jj = q % J;
  int c = 4 * jj + r;
  float v = (active && c < E) ? row[c] : 0.f;
  for (int j = 0; j < J; ++j) {
    const int jn = jj + 1 == J ? 0 : jj + 1;
    const int cn = 4 * jn + r;
    const float vn = (active && cn < E) ? row[cn] : 0.f;  // next column, loaded ahead
    if (active && c < E) {
      sum += v;
      const uint64_t p = pack(bias ? __fadd_rn(v, bias[c]) : v, c);
      if (p > L[KM - 1]) {
        uint64_t cv = p;
#pragma unroll
        for (int k = 0; k < KM; ++k) {
          const uint64_t hi = cv > L[k] ? cv : L[k];
          cv = cv > L[k] ? L[k] : cv;
          L[k] = hi;
        }
      }
    }
    jj = jn;
    c = cn;
    v = vn;
  }
  // left-align: shift by k0 in binary steps of static size
#pragma unroll
  for (int b = 1; b < KM; b <<= 1) {
    if (k0 & b) {
#pragma unroll
      for (int k = 0; k < KM; ++k) L[k] = k + b < KM ? L[k + b] : 0ull;
    }
  }
  // merge the quad's four lists: K rounds of a quad maximum; the owner pops
#pragma unroll
  for (int k = 0; k < KM; ++k) {
    win[k] = 0ull;
    if (k < K) {
      uint64_t best = L[0];
      uint64_t o = shfl_xor64(best, 1);
      best = o > best ? o : best;
      o = shfl_xor64(best, 2);
      best = o > best ? o : best;
      win[k] = best;
      const bool pop = L[0] == best && best != 0ull;
#pragma unroll
      for (int m = 0; m < KM; ++m) L[m] = pop ? (m + 1 < KM ? L[m + 1] : 0ull) : L[m];
    }
  }
  sum += __shfl_xor_sync(0xffffffffu, sum, 1);
  sum += __shfl_xor_sync(0xffffffffu, sum, 2);
  *rowsum = sum;
}

}  // namespace sel
}  // namespace moe
