// Permute family: deterministic counting sort of the routed slots into the
// expert-grouped order (histogram + prefix sum + in-order ranking), and the
// in-HBM dispatch / combine and their backward passes.  On one GPU these
// replace the paper's six expert-parallel transfers per layer (Sec. 4.1
// footnote).  All row copies use 16-byte vectors, one warp per token.
#include "common.cuh"
#include "launch.h"

namespace moe {

constexpr int kChunk = 2048;       // slots per counting-sort chunk
constexpr int kRankWarps = 8;      // sub-chunks of kChunk / kRankWarps slots
constexpr int kSub = kChunk / kRankWarps;

static inline int64_t num_chunks(int64_t TK) { return (TK + kChunk - 1) / kChunk; }

size_t perm_workspace_bytes(int64_t TK, int E) {
  return (size_t)E * (size_t)num_chunks(TK) * sizeof(int32_t);
}

// Per-chunk expert histogram (shared-memory counters; counts are order-free,
// so the result is deterministic).  Layout: counts[e * nchunks + chunk].
__global__ void __launch_bounds__(256) perm_hist_kernel(const int32_t* __restrict__ idx, int64_t TK, int E,
                                                        int nchunks, int32_t* __restrict__ counts, uint32_t* err) {
  __shared__ int h[kMaxE];
  for (int i = threadIdx.x; i < E; i += blockDim.x) h[i] = 0;
  __syncthreads();
  const int64_t s0 = (int64_t)blockIdx.x * kChunk;
  const int64_t s1 = min(TK, s0 + kChunk);
  // every load of the thread's kChunk / 256 slots in flight before the counts
  constexpr int kPer = kChunk / 256;
  int ev[kPer];
#pragma unroll
  for (int i = 0; i < kPer; ++i) {
    const int64_t s = s0 + i * 256 + threadIdx.x;
    ev[i] = s < s1 ? __ldg(idx + s) : 0;
  }
#pragma unroll
  for (int i = 0; i < kPer; ++i) {
    if (s0 + i * 256 + threadIdx.x >= s1) continue;
    if (ev[i] >= 0 && ev[i] < E) atomicAdd(&h[ev[i]], 1);
    else set_error(err, kErrIndex);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < E; i += blockDim.x) counts[(int64_t)i * nchunks + blockIdx.x] = h[i];
}

// Ranks every slot of one chunk in slot order (= token order within an
// expert, since a token picks an expert at most once), so the permutation is
// stable in t and bit-reproducible.  Each block first derives its chunk's
// first row per expert from the whole (expert, chunk) count table: the
// exclusive scan of the experts' totals plus the expert's counts in the
// earlier chunks (block 0 also writes the offsets).  Warp w owns slots
// [w * kSub, (w+1) * kSub) of the chunk and walks them 32 at a time; lanes
// that share an expert get consecutive rows by __match_any_sync rank.  Also
// writes prob_perm.
__global__ void __launch_bounds__(kRankWarps * 32) perm_rank_kernel(
    const int32_t* __restrict__ idx, const float* __restrict__ prob, int64_t TK, int K, int E, int nchunks,
    const int32_t* __restrict__ counts, int32_t* __restrict__ offsets, int32_t* __restrict__ row_of_slot,
    int32_t* __restrict__ token_of_row, float* __restrict__ prob_perm) {
  __shared__ int cnt[kRankWarps * kMaxE];
  __shared__ int tot[kMaxE + 1];  // expert totals, then their exclusive scan
  __shared__ int pre[kMaxE];      // the expert's slots in the chunks before this one
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < kRankWarps * E; i += blockDim.x) cnt[i] = 0;
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    const int32_t* row = counts + (int64_t)e * nchunks;
    int before = 0, all = 0;
#pragma unroll 8
    for (int c = 0; c < nchunks; ++c) {
      const int v = row[c];
      before += c < (int)blockIdx.x ? v : 0;
      all += v;
    }
    pre[e] = before;
    tot[e] = all;
  }
  __syncthreads();
  if (threadIdx.x == 0) {  // E <= 256: a serial scan is a few hundred adds
    int run = 0;
    for (int e = 0; e < E; ++e) {
      const int v = tot[e];
      tot[e] = run;
      run += v;
    }
    tot[E] = run;
  }
  __syncthreads();
  if (blockIdx.x == 0)
    for (int e = threadIdx.x; e <= E; e += blockDim.x) offsets[e] = tot[e];
  const int64_t c0 = (int64_t)blockIdx.x * kChunk;
  const int64_t w0 = c0 + (int64_t)warp * kSub;
  const int64_t w1 = min(TK, w0 + kSub);
  // the warp's kSub expert indices and probabilities, all loads in flight at
  // once (expert -1 past the end)
  int ev[kSub / 32];
  float pv[kSub / 32];
#pragma unroll
  for (int i = 0; i < kSub / 32; ++i) {
    const int64_t s = w0 + i * 32 + lane;
    ev[i] = s < w1 ? __ldg(idx + s) : -1;
    pv[i] = s < w1 ? __ldg(prob + s) : 0.f;
  }
#pragma unroll
  for (int i = 0; i < kSub / 32; ++i)
    if (ev[i] >= 0 && ev[i] < E) atomicAdd(&cnt[warp * E + ev[i]], 1);
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    int run = tot[e] + pre[e];
    for (int w = 0; w < kRankWarps; ++w) {
      const int c = cnt[w * E + e];
      cnt[w * E + e] = run;
      run += c;
    }
  }
  __syncthreads();
  const unsigned lt = (1u << lane) - 1u;
#pragma unroll
  for (int i = 0; i < kSub / 32; ++i) {
    const int64_t s = w0 + i * 32 + lane;
    const int e = ev[i];
    const bool valid = (s < w1) && e >= 0 && e < E;
    const unsigned peers = __match_any_sync(0xffffffffu, valid ? e : -1);
    const int rank = __popc(peers & lt);
    const int here = valid ? cnt[warp * E + e] : 0;
    __syncwarp();
    if (valid) {
      const int row = here + rank;
      row_of_slot[s] = row;
      token_of_row[row] = (int32_t)(s / K);
      prob_perm[row] = pv[i];
      if (rank == __popc(peers) - 1) cnt[warp * E + e] = here + __popc(peers);
    } else if (s < w1) {
      row_of_slot[s] = 0;  // keeps downstream gathers in bounds; the status word is set
    }
    __syncwarp();
  }
}

cudaError_t launch_permutation(const Ctx& c, const int32_t* idx, const float* prob, int64_t T, int K, int E,
                               int32_t* offsets, int32_t* row_of_slot, int32_t* token_of_row, float* prob_perm,
                               void* ws) {
  const int64_t TK = T * K;
  const int nch = (int)num_chunks(TK);
  int32_t* counts = (int32_t*)ws;
  if (TK == 0) {
    KernelScope ks("perm_zero", c.stream);
    return cudaMemsetAsync(offsets, 0, sizeof(int32_t) * (E + 1), c.stream);
  }
  {
    KernelScope ks("perm_hist", c.stream);
    perm_hist_kernel<<<nch, 256, 0, c.stream>>>(idx, TK, E, nch, counts, c.err);
  }
  cudaError_t st = cudaGetLastError();
  if (st != cudaSuccess) return st;
  {
    KernelScope ks("perm_rank", c.stream);
    perm_rank_kernel<<<nch, kRankWarps * 32, 0, c.stream>>>(idx, prob, TK, K, E, nch, counts, offsets,
                                                            row_of_slot, token_of_row, prob_perm);
  }
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Row movers: one warp per token, lanes stride over the row's 16-byte vectors.
// KM is a compile-time bound on K (2, 4, 8 or 16) so the per-token row and
// load arrays stay in registers without the register cost of the largest K.
// ---------------------------------------------------------------------------

template <int KM>
__device__ __forceinline__ void load_rows(const int32_t* __restrict__ row_of_slot, int64_t t, int K,
                                          int32_t (&rows)[KM]) {
#pragma unroll
  for (int k = 0; k < KM; ++k) rows[k] = (k < K) ? __ldg(row_of_slot + t * K + k) : 0;
}

static inline int k_bound(int K) { return K <= 2 ? 2 : (K <= 4 ? 4 : (K <= 8 ? 8 : 16)); }

#define MOE_DISPATCH_KM(K, CALL) \
  switch (k_bound(K)) {          \
    case 2: { constexpr int KM = 2; CALL; break; }  \
    case 4: { constexpr int KM = 4; CALL; break; }  \
    case 8: { constexpr int KM = 8; CALL; break; }  \
    default: { constexpr int KM = 16; CALL; break; } \
  }

// Dispatch: each token's row is read once and written to its K rows.
template <int KM>
__global__ void __launch_bounds__(256) dispatch_rows_kernel(const uint4* __restrict__ x,
                                                            const int32_t* __restrict__ row_of_slot, int64_t T,
                                                            int K, int vpr, uint4* __restrict__ x_perm) {
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= T) return;
  int32_t rows[KM];
  load_rows<KM>(row_of_slot, t, K, rows);
  const uint4* src = x + t * vpr;
  for (int v = lane; v < vpr; v += 32) {
    const uint4 val = ld_stream(src + v);
#pragma unroll
    for (int k = 0; k < KM; ++k)
      if (k < K) st_stream(x_perm + (int64_t)rows[k] * vpr + v, val);
  }
}

cudaError_t launch_dispatch_rows(const Ctx& c, const void* x, const int32_t* row_of_slot, int64_t T, int K,
                                 int64_t row_bytes, void* x_perm) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  const unsigned grid = (unsigned)((T + warps - 1) / warps);
  const int vpr = (int)(row_bytes / 16);
  KernelScope ks("dispatch_rows", c.stream);
  MOE_DISPATCH_KM(K, (dispatch_rows_kernel<KM><<<grid, 32 * warps, 0, c.stream>>>(
                         (const uint4*)x, row_of_slot, T, K, vpr, (uint4*)x_perm)));
  return cudaGetLastError();
}

// Combine: y[t] = sum_k p_k Y_perm[row_k], fp32 accumulation, one rounding.
template <typename T, int KM>
__global__ void __launch_bounds__(256) combine_kernel(const uint4* __restrict__ y_perm,
                                                      const float* __restrict__ prob_perm,
                                                      const int32_t* __restrict__ row_of_slot, int64_t Tn, int K,
                                                      int vpr, uint4* __restrict__ y) {
  constexpr int NV = Vec<T>::N;
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= Tn) return;
  int32_t rows[KM];
  load_rows<KM>(row_of_slot, t, K, rows);
  float p[KM];
#pragma unroll
  for (int k = 0; k < KM; ++k) p[k] = (k < K) ? __ldg(prob_perm + rows[k]) : 0.f;
  for (int v = lane; v < vpr; v += 32) {
    uint4 raw[KM];
#pragma unroll
    for (int k = 0; k < KM; ++k)
      if (k < K) raw[k] = ld_stream(y_perm + (int64_t)rows[k] * vpr + v);
    float acc[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) acc[i] = 0.f;
#pragma unroll
    for (int k = 0; k < KM; ++k) {
      if (k < K) {
        float f[NV];
        unpack16<T>(raw[k], f);
#pragma unroll
        for (int i = 0; i < NV; ++i) acc[i] = fmaf(p[k], f[i], acc[i]);
      }
    }
    st_stream(y + t * vpr + v, pack16<T>(acc));
  }
}

cudaError_t launch_combine(const Ctx& c, DType dt, const void* y_perm, const float* prob_perm,
                           const int32_t* row_of_slot, int64_t T, int K, int D, void* y) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  const int vpr = (int)((int64_t)D * dsize(dt) / 16);
  const unsigned grid = (unsigned)((T + warps - 1) / warps);
  KernelScope ks("combine", c.stream);
  if (dt == DType::BF16) {
    MOE_DISPATCH_KM(K, (combine_kernel<bf16, KM><<<grid, 32 * warps, 0, c.stream>>>(
                           (const uint4*)y_perm, prob_perm, row_of_slot, T, K, vpr, (uint4*)y)));
  } else {
    MOE_DISPATCH_KM(K, (combine_kernel<float, KM><<<grid, 32 * warps, 0, c.stream>>>(
                           (const uint4*)y_perm, prob_perm, row_of_slot, T, K, vpr, (uint4*)y)));
  }
  return cudaGetLastError();
}

// Combine backward: dY_perm[row_k] = p_k dy[t]; dprob_perm[row_k] = <dy[t], Y_perm[row_k]>.
template <typename T, int KM>
__global__ void __launch_bounds__(256) combine_bwd_kernel(const uint4* __restrict__ dy,
                                                          const uint4* __restrict__ y_perm,
                                                          const float* __restrict__ prob_perm,
                                                          const int32_t* __restrict__ row_of_slot, int64_t Tn,
                                                          int K, int vpr, uint4* __restrict__ dy_perm,
                                                          float* __restrict__ dprob_perm) {
  constexpr int NV = Vec<T>::N;
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= Tn) return;
  int32_t rows[KM];
  load_rows<KM>(row_of_slot, t, K, rows);
  float p[KM], dot[KM];
#pragma unroll
  for (int k = 0; k < KM; ++k) {
    p[k] = (k < K) ? __ldg(prob_perm + rows[k]) : 0.f;
    dot[k] = 0.f;
  }
  for (int v = lane; v < vpr; v += 32) {
    const uint4 gv = ld_stream(dy + t * vpr + v);
    uint4 raw[KM];
#pragma unroll
    for (int k = 0; k < KM; ++k)
      if (k < K) raw[k] = ld_stream(y_perm + (int64_t)rows[k] * vpr + v);
    float g[NV];
    unpack16<T>(gv, g);
#pragma unroll
    for (int k = 0; k < KM; ++k) {
      if (k < K) {
        float f[NV], o[NV];
        unpack16<T>(raw[k], f);
#pragma unroll
        for (int i = 0; i < NV; ++i) {
          dot[k] = fmaf(g[i], f[i], dot[k]);
          o[i] = p[k] * g[i];
        }
        st_stream(dy_perm + (int64_t)rows[k] * vpr + v, pack16<T>(o));
      }
    }
  }
#pragma unroll
  for (int k = 0; k < KM; ++k) {
    if (k < K) {
      float s = dot[k];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
      if (lane == 0) dprob_perm[rows[k]] = s;
    }
  }
}

cudaError_t launch_combine_bwd(const Ctx& c, DType dt, const void* dy, const void* y_perm, const float* prob_perm,
                               const int32_t* row_of_slot, int64_t T, int K, int D, void* dy_perm,
                               float* dprob_perm) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  const int vpr = (int)((int64_t)D * dsize(dt) / 16);
  const unsigned grid = (unsigned)((T + warps - 1) / warps);
  KernelScope ks("combine_bwd", c.stream);
  if (dt == DType::BF16) {
    MOE_DISPATCH_KM(K, (combine_bwd_kernel<bf16, KM><<<grid, 32 * warps, 0, c.stream>>>(
                           (const uint4*)dy, (const uint4*)y_perm, prob_perm, row_of_slot, T, K, vpr,
                           (uint4*)dy_perm, dprob_perm)));
  } else {
    MOE_DISPATCH_KM(K, (combine_bwd_kernel<float, KM><<<grid, 32 * warps, 0, c.stream>>>(
                           (const uint4*)dy, (const uint4*)y_perm, prob_perm, row_of_slot, T, K, vpr,
                           (uint4*)dy_perm, dprob_perm)));
  }
  return cudaGetLastError();
}

// Dispatch backward: dx[t] = sum_k dX_perm[row_k] (fp32 accumulation; dx
// rows ldv 16-byte vectors apart); dprob[t, k] = dprob_perm[row_k].
template <typename T, int KM>
__global__ void __launch_bounds__(256) dispatch_bwd_kernel(const uint4* __restrict__ dx_perm,
                                                           const float* __restrict__ dprob_perm,
                                                           const int32_t* __restrict__ row_of_slot, int64_t Tn,
                                                           int K, int vpr, int64_t ldv, uint4* __restrict__ dx,
                                                           float* __restrict__ dprob) {
  constexpr int NV = Vec<T>::N;
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= Tn) return;
  int32_t rows[KM];
  load_rows<KM>(row_of_slot, t, K, rows);
  for (int v = lane; v < vpr; v += 32) {
    uint4 raw[KM];
#pragma unroll
    for (int k = 0; k < KM; ++k)
      if (k < K) raw[k] = ld_stream(dx_perm + (int64_t)rows[k] * vpr + v);
    float acc[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) acc[i] = 0.f;
#pragma unroll
    for (int k = 0; k < KM; ++k) {
      if (k < K) {
        float f[NV];
        unpack16<T>(raw[k], f);
#pragma unroll
        for (int i = 0; i < NV; ++i) acc[i] += f[i];
      }
    }
    st_stream(dx + t * ldv + v, pack16<T>(acc));
  }
  // the probability gradients last, off the path of the row loads
  if (lane < K) dprob[t * K + lane] = __ldg(dprob_perm + row_of_slot[t * K + lane]);
}

cudaError_t launch_dispatch_bwd(const Ctx& c, DType dt, const void* dx_perm, const float* dprob_perm,
                                const int32_t* row_of_slot, int64_t T, int K, int D, void* dx, float* dprob,
                                int64_t ldx) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  const int vpr = (int)((int64_t)D * dsize(dt) / 16);
  const int64_t ldv = (ldx > 0 ? ldx : D) * (int64_t)dsize(dt) / 16;
  const unsigned grid = (unsigned)((T + warps - 1) / warps);
  KernelScope ks("dispatch_bwd", c.stream);
  if (dt == DType::BF16) {
    MOE_DISPATCH_KM(K, (dispatch_bwd_kernel<bf16, KM><<<grid, 32 * warps, 0, c.stream>>>(
                           (const uint4*)dx_perm, dprob_perm, row_of_slot, T, K, vpr, ldv, (uint4*)dx, dprob)));
  } else {
    MOE_DISPATCH_KM(K, (dispatch_bwd_kernel<float, KM><<<grid, 32 * warps, 0, c.stream>>>(
                           (const uint4*)dx_perm, dprob_perm, row_of_slot, T, K, vpr, ldv, (uint4*)dx, dprob)));
  }
  return cudaGetLastError();
}

// Dispatch backward fused with the softmax router's backward, for a router
// that reads the dispatch input itself (no latent projection).  dz is nonzero
// only on a token's K selected experts, so dz . W_r for token t is a sum of
// K rows of W_r [E, D], the same shape as the sum over its K dX_perm rows.
// Per token t (one warp):
//   dprob[t, k] = dprob_perm[row_k];
//   dz[t, e_k]  = p_k (dprob[t, k] - sum_j p_j dprob[t, j]), 0 elsewhere
//                 (the same reduction tree as route_dz_kernel, so the same bits);
//   dx[t]       = sum_k dX_perm[row_k] + sum_k dz[t, e_k] W_r[e_k]
//                 (fp32 accumulation, rounded once).
// dz16 (bf16 copy of dz, for the router weight gradient) may be NULL.
template <typename T, int KM>
__global__ void __launch_bounds__(256, KM <= 8 ? 3 : 1) dispatch_route_bwd_kernel(
    const uint4* __restrict__ dx_perm, const float* __restrict__ dprob_perm, const int32_t* __restrict__ row_of_slot,
    const int32_t* __restrict__ idx, const float* __restrict__ prob, const uint4* __restrict__ w_router, int64_t Tn,
    int K, int E, int vpr, uint4* __restrict__ dx, float* __restrict__ dprob, float* __restrict__ dz,
    bf16* __restrict__ dz16, uint32_t* err) {
  constexpr int NV = Vec<T>::N;
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= Tn) return;
  int32_t rows[KM];
  load_rows<KM>(row_of_slot, t, K, rows);
  int my_e = -1;
  float my_p = 0.f, my_dp = 0.f;
  if (lane < K) {
    my_e = __ldg(idx + t * K + lane);
    my_p = __ldg(prob + t * K + lane);
    my_dp = __ldg(dprob_perm + __ldg(row_of_slot + t * K + lane));
  }
  float cdot = my_p * my_dp;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) cdot += __shfl_xor_sync(0xffffffffu, cdot, off);
  const float my_dz = my_p * (my_dp - cdot);
  int ek[KM];
  float dzk[KM];
#pragma unroll
  for (int k = 0; k < KM; ++k) {
    ek[k] = __shfl_sync(0xffffffffu, my_e, k);
    dzk[k] = __shfl_sync(0xffffffffu, my_dz, k);
    if (k < K && (ek[k] < 0 || ek[k] >= E)) {  // an expert index outside [0, E): recorded, its row skipped
      if (lane == 0) set_error(err, kErrIndex);
      ek[k] = -1;
    }
  }
  for (int v = lane; v < vpr; v += 32) {
    // the K dX_perm rows (HBM) first, then the K rows of W_r (L2-resident):
    // one set of K vectors in registers at a time keeps three blocks per SM
    uint4 raw[KM];
#pragma unroll
    for (int k = 0; k < KM; ++k)
      if (k < K) raw[k] = ld_stream(dx_perm + (int64_t)rows[k] * vpr + v);
    float acc[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) acc[i] = 0.f;
#pragma unroll
    for (int k = 0; k < KM; ++k) {
      if (k < K) {
        float f[NV];
        unpack16<T>(raw[k], f);
#pragma unroll
        for (int i = 0; i < NV; ++i) acc[i] += f[i];
      }
    }
#pragma unroll
    for (int k = 0; k < KM; ++k)
      if (k < K && ek[k] >= 0) raw[k] = ld_keep(w_router + (int64_t)ek[k] * vpr + v);
#pragma unroll
    for (int k = 0; k < KM; ++k) {
      if (k < K && ek[k] >= 0) {
        float f[NV];
        unpack16<T>(raw[k], f);
#pragma unroll
        for (int i = 0; i < NV; ++i) acc[i] = fmaf(dzk[k], f[i], acc[i]);
      }
    }
    st_stream(dx + t * vpr + v, pack16<T>(acc));
  }
  if (lane < K) dprob[t * K + lane] = my_dp;
  for (int e0 = 0; e0 < E; e0 += 32) {
    const int e = e0 + lane;
    float val = 0.f;
#pragma unroll
    for (int k = 0; k < KM; ++k)
      if (k < K && ek[k] == e) val = dzk[k];
    if (e < E) {
      dz[t * E + e] = val;
      if (dz16) dz16[t * E + e] = __float2bfloat16_rn(val);
    }
  }
}

cudaError_t launch_dispatch_route_bwd(const Ctx& c, DType dt, const void* dx_perm, const float* dprob_perm,
                                      const int32_t* row_of_slot, const int32_t* idx, const float* prob,
                                      const void* w_router, int64_t T, int K, int E, int D, void* dx, float* dprob,
                                      float* dz, void* dz16) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  const int vpr = (int)((int64_t)D * dsize(dt) / 16);
  const unsigned grid = (unsigned)((T + warps - 1) / warps);
  KernelScope ks("dispatch_route_bwd", c.stream);
  if (dt == DType::BF16) {
    MOE_DISPATCH_KM(K, (dispatch_route_bwd_kernel<bf16, KM><<<grid, 32 * warps, 0, c.stream>>>(
                           (const uint4*)dx_perm, dprob_perm, row_of_slot, idx, prob, (const uint4*)w_router, T, K,
                           E, vpr, (uint4*)dx, dprob, dz, (bf16*)dz16, c.err)));
  } else {
    MOE_DISPATCH_KM(K, (dispatch_route_bwd_kernel<float, KM><<<grid, 32 * warps, 0, c.stream>>>(
                           (const uint4*)dx_perm, dprob_perm, row_of_slot, idx, prob, (const uint4*)w_router, T, K,
                           E, vpr, (uint4*)dx, dprob, dz, (bf16*)dz16, c.err)));
  }
  return cudaGetLastError();
}

// w1[e, 128 i + c] = w_gate[e, 64 i + c] for c < 64, w_up[e, 64 i + c - 64] otherwise.
__global__ void __launch_bounds__(256) pack_w1_kernel(const uint4* __restrict__ wg, const uint4* __restrict__ wu,
                                                      int64_t rows_total, int F, int vpr, uint4* __restrict__ w1) {
  const int64_t r = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (r >= rows_total) return;
  const int lane = threadIdx.x & 31;
  const int64_t e = r / (2 * F);
  const int j = (int)(r % (2 * F));
  const int blk = j / 128, c = j % 128;
  const int f = blk * 64 + (c & 63);
  const uint4* src = (c < 64 ? wg : wu) + (e * F + f) * vpr;
  for (int v = lane; v < vpr; v += 32) w1[r * vpr + v] = src[v];
}

cudaError_t launch_pack_w1(const Ctx& c, DType dt, const void* w_gate, const void* w_up, int E, int F, int D,
                           void* w1) {
  const int64_t rows = (int64_t)E * 2 * F;
  const int vpr = (int)((int64_t)D * dsize(dt) / 16);
  KernelScope ks("pack_w1", c.stream);
  pack_w1_kernel<<<(unsigned)((rows + 7) / 8), 256, 0, c.stream>>>((const uint4*)w_gate, (const uint4*)w_up, rows,
                                                                   F, vpr, (uint4*)w1);
  return cudaGetLastError();
}

}  // namespace moe
