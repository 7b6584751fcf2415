// CUDA-core grouped GEMM (fp32 FMA, no TF32): the all-fp32 path and the
// reference engine for every GemmDesc shape the tensor-core engine handles.
//
// C(m, n) = sum_k A(m, k) B(n, k) with arbitrary element strides, grouped
// along M (per-expert row ranges), along K (per-expert reduction ranges) or
// dense, plus the router / SwiGLU epilogues, and the row gathers of GemmDesc.  Tile 64 x 128 x 16, 256
// threads; thread (ty, tx) owns rows 4 ty .. 4 ty + 3 and columns
// 4 tx .. 4 tx + 3 and 64 + 4 tx .. 64 + 4 tx + 3 of the tile, so a packed
// gate column and its up column (64 apart) land in the same thread.
#include "common.cuh"
#include "launch.h"

namespace moe {

namespace {

constexpr int BM = 64, BN = 128, BK = 16;

template <typename T>
__device__ __forceinline__ float ldf(const void* p, int64_t i) {
  return to_f32<T>(static_cast<const T*>(p)[i]);
}

__device__ __forceinline__ float silu_f(float v) { return v / (1.0f + __expf(-v)); }

template <typename TA, typename TB, typename TC>
__global__ void __launch_bounds__(256) simt_gemm_kernel(GemmDesc d) {
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tid = threadIdx.x;
  const int tx = tid & 15, ty = tid >> 4;
  const int64_t n0 = (int64_t)blockIdx.x * BN;

  int g = 0;
  int64_t row0 = 0, row_end = d.M, kbeg = 0, kend = d.K;
  if (d.group == Group::M) {
    const int64_t mt = blockIdx.y;
    int64_t acc = 0;
    g = -1;
    for (int e = 0; e < d.num_groups; ++e) {
      const int64_t lo = d.offsets[e], hi = d.offsets[e + 1];
      const int64_t nt = (hi - lo + BM - 1) / BM;
      if (mt < acc + nt) {
        g = e;
        row0 = lo + (mt - acc) * BM;
        row_end = hi;
        break;
      }
      acc += nt;
    }
    if (g < 0) return;
  } else if (d.group == Group::K) {
    g = blockIdx.z;
    row0 = (int64_t)blockIdx.y * BM;
    kbeg = d.offsets[g];
    kend = d.offsets[g + 1];
  } else {
    row0 = (int64_t)blockIdx.y * BM;
  }
  if (row0 >= row_end || n0 >= d.N) return;

  const void* Bp = static_cast<const char*>(d.B) + (int64_t)g * d.sb_g * sizeof(TB);
  const bool a_kfast = d.sa_k == 1;
  const bool b_kfast = d.sb_k == 1;

  float acc[4][8];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

  for (int64_t k0 = kbeg; k0 < kend; k0 += BK) {
    for (int i = tid; i < BM * BK; i += 256) {
      int m, k;
      if (a_kfast) { k = i % BK; m = i / BK; } else { m = i % BM; k = i / BM; }
      const int64_t gm = row0 + m, gk = k0 + k;
      float v = 0.f;
      if (gm < row_end && gk < kend) {
        const int64_t sm = (d.gather && d.group == Group::M) ? (int64_t)d.gather[gm] : gm;
        v = ldf<TA>(d.A, sm * d.sa_m + gk * d.sa_k);
      }
      As[k][m] = v;
    }
    for (int i = tid; i < BN * BK; i += 256) {
      int n, k;
      if (b_kfast) { k = i % BK; n = i / BK; } else { n = i % BN; k = i / BN; }
      const int64_t gn = n0 + n, gk = k0 + k;
      float v = 0.f;
      if (gn < d.N && gk < kend) {
        const int64_t sk = (d.gather && d.group == Group::K) ? (int64_t)d.gather[gk] : gk;
        v = ldf<TB>(Bp, gn * d.sb_n + sk * d.sb_k);
      }
      Bs[k][n] = v;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < BK; ++k) {
      float a[4], b[8];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[k][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        b[j] = Bs[k][tx * 4 + j];
        b[4 + j] = Bs[k][64 + tx * 4 + j];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }

  TC* C = static_cast<TC*>(d.C) + (d.group == Group::K ? (int64_t)g * d.sc_g : 0);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t gm = row0 + ty * 4 + i;
    if (gm >= row_end) continue;
    TC* crow = C + gm * d.ldc;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int64_t col = (j < 4) ? (tx * 4 + j) : (64 + tx * 4 + (j - 4));
      const int64_t gn = n0 + col;
      if (gn >= d.N) continue;
      float v = acc[i][j];
      switch (d.epi) {
        case Epi::Store:
          crow[gn] = from_f32<TC>(v);
          break;
        case Epi::StoreBias:
          crow[gn] = from_f32<TC>(v + (d.bias ? d.bias[gn] : 0.f));
          break;
        case Epi::Accum:
          crow[gn] = from_f32<TC>(to_f32<TC>(crow[gn]) + v);
          break;
        case Epi::SwigluFwd: {
          crow[gn] = from_f32<TC>(v);
          if (j < 4) {
            // gate at tile column c < 64, up at c + 64 (same thread, index j + 4)
            const float gt = v, up = acc[i][j + 4];
            const int64_t f = n0 / 2 + col;
            static_cast<TC*>(d.aux)[gm * (d.N / 2) + f] = from_f32<TC>(silu_f(gt) * up);
          }
          break;
        }
        case Epi::ReluSqFwd: {
          crow[gn] = from_f32<TC>(v);
          const float r = fmaxf(v, 0.f);
          static_cast<TC*>(d.aux)[gm * d.ldc + gn] = from_f32<TC>(r * r);
          break;
        }
      }
    }
  }
}

template <typename TA, typename TB, typename TC>
cudaError_t run(const Ctx& c, const GemmDesc& d) {
  dim3 block(256);
  dim3 grid((unsigned)((d.N + BN - 1) / BN), 1, 1);
  if (d.group == Group::M) {
    grid.y = (unsigned)((d.max_rows + BM - 1) / BM + d.num_groups);
  } else if (d.group == Group::K) {
    grid.y = (unsigned)((d.M + BM - 1) / BM);
    grid.z = (unsigned)d.num_groups;
  } else {
    grid.y = (unsigned)((d.M + BM - 1) / BM);
  }
  if (grid.x == 0 || grid.y == 0 || grid.z == 0) return cudaSuccess;
  simt_gemm_kernel<TA, TB, TC><<<grid, block, 0, c.stream>>>(d);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm_simt(const Ctx& c, const GemmDesc& d, const char* name) {
  KernelScope ks(name, c.stream);
  const int key = (int)d.a_type * 4 + (int)d.b_type * 2 + (int)d.c_type;
  switch (key) {
    case 0: return run<bf16, bf16, bf16>(c, d);
    case 1: return run<bf16, bf16, float>(c, d);
    case 2 + 0: return run<bf16, float, bf16>(c, d);
    case 4 + 0: return run<float, bf16, bf16>(c, d);
    case 4 + 1: return run<float, bf16, float>(c, d);
    case 4 + 2 + 1: return run<float, float, float>(c, d);
    default: return cudaErrorNotSupported;
  }
}

}  // namespace moe
