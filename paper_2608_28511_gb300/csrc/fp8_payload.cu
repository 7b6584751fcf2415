// Low-precision dispatch payload (Sec. 1, the precision lever b_x of Eq. 1):
// every dispatched row travels as FP8 E4M3 codes (one byte per hidden
// element) plus one power-of-two scale, the smallest s = 2^e (e >= -126) with
// max |x| <= 448 s; the code of x_i is the nearest E4M3 value to x_i / s
// (ties to even, saturating).  A power-of-two scale makes x_i / s exact in
// fp32 and code * s exact in bf16, so the receiver's dequantized row is exact.
#include <cuda_fp8.h>

#include "common.cuh"
#include "launch.h"

namespace moe {

namespace {

// Exponent of the row scale for a row maximum amax (finite, >= 0): the
// smallest e with amax <= 448 2^e, where 448 (the largest finite E4M3 value)
// is 0.875 2^9.
__device__ __forceinline__ int row_scale_exp(float amax) {
  if (!(amax > 0.f)) return 0;
  int k;
  const float m = frexpf(amax, &k);  // amax = m 2^k, m in [0.5, 1)
  const int e = k - 9 + (m > 0.875f ? 1 : 0);
  return e < -126 ? -126 : e;
}

// 8 bf16 values (one 16-byte vector) times inv_s -> 8 E4M3 codes.
__device__ __forceinline__ uint2 quantize8(const uint4& v, float inv_s) {
  float f[8];
  unpack16<bf16>(v, f);
  uint32_t w[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    uint32_t acc = 0;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const __nv_fp8x2_storage_t c = __nv_cvt_float2_to_fp8x2(
          make_float2(f[4 * h + 2 * j] * inv_s, f[4 * h + 2 * j + 1] * inv_s), __NV_SATFINITE, __NV_E4M3);
      acc |= (uint32_t)c << (16 * j);
    }
    w[h] = acc;
  }
  return make_uint2(w[0], w[1]);
}

// One warp per token: the row's maximum magnitude, its scale, then its codes
// written to each of its K rows (row_of_slot) with the scale.
template <int KM>
__global__ void __launch_bounds__(256) dispatch_fp8_kernel(const uint4* __restrict__ x,
                                                           const int32_t* __restrict__ row_of_slot, int64_t T,
                                                           int K, int vpr, uint2* __restrict__ xq,
                                                           float* __restrict__ scale_perm, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= T) return;
  const uint4* row = x + t * vpr;
  float amax = 0.f;
  for (int i = lane; i < vpr; i += 32) {
    float f[8];
    unpack16<bf16>(__ldg(row + i), f);
#pragma unroll
    for (int j = 0; j < 8; ++j) amax = fmaxf(amax, fabsf(f[j]));
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
  const int e = row_scale_exp(amax);
  const float inv_s = ldexpf(1.0f, -e);
  int64_t dst[KM];
#pragma unroll
  for (int k = 0; k < KM; ++k) {
    dst[k] = k < K ? (int64_t)__ldg(row_of_slot + t * K + k) : -1;
    if (dst[k] >= T * K) {  // a row outside [0, TK): recorded and skipped
      set_error(err, kErrIndex);
      dst[k] = -1;
    }
  }
  if (lane < K) {
#pragma unroll
    for (int k = 0; k < KM; ++k)
      if (k == lane && dst[k] >= 0) scale_perm[dst[k]] = ldexpf(1.0f, e);
  }
  for (int i = lane; i < vpr; i += 32) {
    const uint2 q = quantize8(__ldg(row + i), inv_s);
#pragma unroll
    for (int k = 0; k < KM; ++k)
      if (dst[k] >= 0) xq[dst[k] * vpr + i] = q;
  }
}

// x_perm[r] = codes[r] * scale[r] in bf16 (exact), 8 codes (one 16-byte
// store) per thread step, so a warp writes 512 contiguous bytes.
__global__ void __launch_bounds__(256) dequant_rows_kernel(const uint2* __restrict__ xq,
                                                           const float* __restrict__ scale, int64_t rows, int vpr,
                                                           uint4* __restrict__ out) {
  const int64_t total = rows * vpr;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const float s = __ldg(scale + i / vpr);
    const uint2 q = __ldg(xq + i);
    const uint32_t w[2] = {q.x, q.y};
    float f[8];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const __half2_raw hr = __nv_cvt_fp8x2_to_halfraw2((__nv_fp8x2_storage_t)(w[h] >> (16 * j)), __NV_E4M3);
        const float2 v = __half22float2(*reinterpret_cast<const __half2*>(&hr));
        f[4 * h + 2 * j] = v.x * s;
        f[4 * h + 2 * j + 1] = v.y * s;
      }
    }
    st_stream(out + i, pack16<bf16>(f));
  }
}

int k_bound(int K) { return K <= 2 ? 2 : K <= 4 ? 4 : K <= 8 ? 8 : 16; }

}  // namespace

cudaError_t launch_dispatch_fp8(const Ctx& c, const void* x, const int32_t* row_of_slot, int64_t T, int K, int D,
                                void* xq, float* scale_perm) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  const dim3 grid((unsigned)((T + warps - 1) / warps));
  const int vpr = D / 8;
  KernelScope ks("dispatch_fp8", c.stream);
  switch (k_bound(K)) {
    case 2: dispatch_fp8_kernel<2><<<grid, 32 * warps, 0, c.stream>>>((const uint4*)x, row_of_slot, T, K, vpr,
                       (uint2*)xq, scale_perm, c.err); break;
    case 4: dispatch_fp8_kernel<4><<<grid, 32 * warps, 0, c.stream>>>((const uint4*)x, row_of_slot, T, K, vpr,
                       (uint2*)xq, scale_perm, c.err); break;
    case 8: dispatch_fp8_kernel<8><<<grid, 32 * warps, 0, c.stream>>>((const uint4*)x, row_of_slot, T, K, vpr,
                       (uint2*)xq, scale_perm, c.err); break;
    default: dispatch_fp8_kernel<16><<<grid, 32 * warps, 0, c.stream>>>((const uint4*)x, row_of_slot, T, K,
                        vpr, (uint2*)xq, scale_perm, c.err); break;
  }
  return cudaGetLastError();
}

cudaError_t launch_dequant_rows(const Ctx& c, const void* xq, const float* scale, int64_t rows, int D, void* out) {
  if (rows == 0) return cudaSuccess;
  const int vpr = D / 8;
  const int64_t want = (rows * vpr + 255) / 256;
  const int blocks = (int)(want < (int64_t)c.num_sms * 16 ? want : (int64_t)c.num_sms * 16);
  KernelScope ks("dequant_rows", c.stream);
  dequant_rows_kernel<<<blocks, 256, 0, c.stream>>>((const uint2*)xq, scale, rows, vpr, (uint4*)out);
  return cudaGetLastError();
}

}  // namespace moe
