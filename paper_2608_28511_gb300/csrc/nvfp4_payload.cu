// NVFP4 dispatch payload (Sec. 1, the precision lever b_x of Eq. 1; Sec. 6
// names FP8 and NVFP4): every dispatched row travels as E2M1 codes (two per
// byte, element 2j in the low nibble of byte j), one E4M3 scale per block of
// 16 elements and one power-of-two scale g per row:
//   g   = the smallest 2^e (e >= -126) with max |x| <= 6 * 448 * g;
//   s_b = E4M3 nearest to max_{i in b} |x_i| / (6 g)   (fp32 ratio);
//   q_i = E2M1 nearest to x_i / (s_b g)                (fp32 ratio);
// both roundings to nearest, ties to even, saturating.  The receiver's
// q * s_b * g is exact in bf16.
#include <cuda_fp4.h>
#include <cuda_fp8.h>

#include "common.cuh"
#include "launch.h"

namespace moe {

namespace {

constexpr int kBlk = 16;  // elements per block scale

// Exponent of the row scale for a row maximum amax (finite, >= 0): the
// smallest e with amax <= 6 * 448 * 2^e, where 6 * 448 = 2688 is
// 0.65625 * 2^12.
__device__ __forceinline__ int nvfp4_row_exp(float amax) {
  if (!(amax > 0.f)) return 0;
  int k;
  const float m = frexpf(amax, &k);  // amax = m 2^k, m in [0.5, 1)
  const int e = k - 12 + (m > 0.65625f ? 1 : 0);
  return e < -126 ? -126 : e;
}

__device__ __forceinline__ float e4m3_to_float(uint8_t c) {
  const __half_raw h = __nv_cvt_fp8_to_halfraw((__nv_fp8_storage_t)c, __NV_E4M3);
  return __half2float(*reinterpret_cast<const __half*>(&h));
}

// One 16-element block (two 16-byte vectors of bf16) -> its E4M3 scale code
// and 8 bytes of E2M1 codes.
__device__ __forceinline__ void quantize_block(const uint4& v0, const uint4& v1, float six_g, float g,
                                               uint8_t* scode, uint2* codes) {
  float f[kBlk];
  unpack16<bf16>(v0, f);
  unpack16<bf16>(v1, f + 8);
  float amax = 0.f;
#pragma unroll
  for (int i = 0; i < kBlk; ++i) amax = fmaxf(amax, fabsf(f[i]));
  const __nv_fp8_storage_t sc = __nv_cvt_float_to_fp8(amax / six_g, __NV_SATFINITE, __NV_E4M3);
  *scode = (uint8_t)sc;
  const float sb = e4m3_to_float((uint8_t)sc);
  uint32_t w[2] = {0u, 0u};
  if (sb > 0.f) {
    const float den = sb * g;  // exact: an E4M3 value times a power of two
#pragma unroll
    for (int h = 0; h < 2; ++h) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int i = 8 * h + 2 * j;
        const __nv_fp4x2_storage_t b =
            __nv_cvt_float2_to_fp4x2(make_float2(f[i] / den, f[i + 1] / den), __NV_E2M1, cudaRoundNearest);
        w[h] |= (uint32_t)b << (8 * j);
      }
    }
  }
  *codes = make_uint2(w[0], w[1]);
}

// One warp per token: the row maximum and scale, then every block's scale and
// codes, written to each of the token's K rows (row_of_slot).
template <int KM>
__global__ void __launch_bounds__(256) dispatch_nvfp4_kernel(const uint4* __restrict__ x,
                                                             const int32_t* __restrict__ row_of_slot, int64_t T,
                                                             int K, int vpr, uint2* __restrict__ xq,
                                                             uint8_t* __restrict__ bscale, float* __restrict__ rscale,
                                                             uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= T) return;
  const uint4* row = x + t * vpr;
  const int nblk = vpr / 2;  // 16-element blocks per row
  float amax = 0.f;
  for (int i = lane; i < vpr; i += 32) {
    float f[8];
    unpack16<bf16>(__ldg(row + i), f);
#pragma unroll
    for (int j = 0; j < 8; ++j) amax = fmaxf(amax, fabsf(f[j]));
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
  const int e = nvfp4_row_exp(amax);
  const float g = ldexpf(1.0f, e);
  const float six_g = 6.0f * g;  // exact
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
      if (k == lane && dst[k] >= 0) rscale[dst[k]] = g;
  }
  for (int b = lane; b < nblk; b += 32) {
    uint8_t sc;
    uint2 q;
    quantize_block(__ldg(row + 2 * b), __ldg(row + 2 * b + 1), six_g, g, &sc, &q);
#pragma unroll
    for (int k = 0; k < KM; ++k) {
      if (dst[k] >= 0) {
        xq[dst[k] * nblk + b] = q;
        bscale[dst[k] * nblk + b] = sc;
      }
    }
  }
}

// x_perm[r] = code * s_b * g in bf16 (exact), 8 elements (4 code bytes, one
// 16-byte store) per thread step, so a warp writes 512 contiguous bytes.
__global__ void __launch_bounds__(256) dequant_nvfp4_kernel(const uint32_t* __restrict__ xq,
                                                            const uint8_t* __restrict__ bscale,
                                                            const float* __restrict__ rscale, int64_t rows,
                                                            int nblk, uint4* __restrict__ out) {
  const int64_t total = rows * nblk * 2;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t b = i >> 1;
    const float s = e4m3_to_float(__ldg(bscale + b)) * __ldg(rscale + b / nblk);
    const uint32_t w = __ldg(xq + i);
    float f[8];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const __half2_raw hr = __nv_cvt_fp4x2_to_halfraw2((__nv_fp4x2_storage_t)(w >> (8 * j)), __NV_E2M1);
      const float2 v = __half22float2(*reinterpret_cast<const __half2*>(&hr));
      f[2 * j] = v.x * s;
      f[2 * j + 1] = v.y * s;
    }
    st_stream(out + i, pack16<bf16>(f));
  }
}

int k_bound(int K) { return K <= 2 ? 2 : K <= 4 ? 4 : K <= 8 ? 8 : 16; }

}  // namespace

cudaError_t launch_dispatch_nvfp4(const Ctx& c, const void* x, const int32_t* row_of_slot, int64_t T, int K, int D,
                                  void* xq, uint8_t* bscale, float* rscale) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  const dim3 grid((unsigned)((T + warps - 1) / warps));
  const int vpr = D / 8;
  KernelScope ks("dispatch_nvfp4", c.stream);
  switch (k_bound(K)) {
    case 2: dispatch_nvfp4_kernel<2><<<grid, 32 * warps, 0, c.stream>>>((const uint4*)x, row_of_slot, T, K, vpr,
                       (uint2*)xq, bscale, rscale, c.err); break;
    case 4: dispatch_nvfp4_kernel<4><<<grid, 32 * warps, 0, c.stream>>>((const uint4*)x, row_of_slot, T, K, vpr,
                       (uint2*)xq, bscale, rscale, c.err); break;
    case 8: dispatch_nvfp4_kernel<8><<<grid, 32 * warps, 0, c.stream>>>((const uint4*)x, row_of_slot, T, K, vpr,
                       (uint2*)xq, bscale, rscale, c.err); break;
    default: dispatch_nvfp4_kernel<16><<<grid, 32 * warps, 0, c.stream>>>((const uint4*)x, row_of_slot, T, K,
                        vpr, (uint2*)xq, bscale, rscale, c.err); break;
  }
  return cudaGetLastError();
}

cudaError_t launch_dequant_nvfp4(const Ctx& c, const void* xq, const uint8_t* bscale, const float* rscale,
                                 int64_t rows, int D, void* out) {
  if (rows == 0) return cudaSuccess;
  const int nblk = D / kBlk;
  const int64_t want = (rows * nblk * 2 + 255) / 256;
  const int blocks = (int)(want < (int64_t)c.num_sms * 16 ? want : (int64_t)c.num_sms * 16);
  KernelScope ks("dequant_nvfp4", c.stream);
  dequant_nvfp4_kernel<<<blocks, 256, 0, c.stream>>>((const uint32_t*)xq, bscale, rscale, rows, nblk, (uint4*)out);
  return cudaGetLastError();
}

}  // namespace moe
