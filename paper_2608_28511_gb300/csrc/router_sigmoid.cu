// The paper's router variant (Sec. 5.2): sigmoid scores, an expert bias that
// shapes the choice of experts only, gate values renormalised over the chosen
// experts, and a sequence-level load-balancing loss.
//   s = sigmoid(z); choose the K largest s + b (ties to the lower expert);
//   p_k = s_k / sum_{j in S} s_j;
//   per sequence g of S tokens: f_gi = E / (K S) #{t in g : i chosen},
//   P_gi = mean over t in g of s_ti / sum_j s_tj, L = coef / GBS sum_g,i f_gi P_gi.
// All reductions run in a fixed order (integer atomics only), so results are
// bit-reproducible.
#include <math_constants.h>

#include "common.cuh"
#include "launch.h"
#include "select.cuh"

namespace moe {

namespace {

int64_t select_chunks(int64_t S, int E) {
  return (S + sel::tokens_per_block(E) - 1) / sel::tokens_per_block(E);
}

__device__ __forceinline__ float sigmoidf_(float z) { return __frcp_rn(1.0f + __expf(-z)); }

struct SigmoidOp {
  __device__ __forceinline__ float operator()(float z) const { return sigmoidf_(z); }
};

// Block (chunk ch of sequence g): stages the scores s = sigmoid(z) of its
// tokens, chooses each token's K experts by s + b (four threads per token),
// writes idx and the gate values s_k / sum over the chosen of s, then adds up,
// per expert, the normalised scores (in token order) and the choice counts of
// its tokens: one partial per (sequence, chunk).  With `keys` the block also
// writes every selection key s + b it compared, formed by the same fp32
// addition of the same staged operands as in the selection.
template <int KM>
__global__ void __launch_bounds__(256) select_sigmoid_kernel(
    const float* __restrict__ logits, const float* __restrict__ bias, int64_t S, int E, int K, int tpb, int nch,
    int32_t* __restrict__ idx, float* __restrict__ prob, float* __restrict__ psum, int32_t* __restrict__ pcnt,
    uint32_t* __restrict__ ticket, float* __restrict__ keys) {
  extern __shared__ __align__(16) float sm[];
  float* zs = sm;                                   // [tpb][E] scores
  float* bs = zs + tpb * E;                         // [E]
  float* inv = bs + E;                              // [tpb]
  int* cnt = reinterpret_cast<int*>(inv + tpb);     // [E]
  const int tid = threadIdx.x, ch = blockIdx.x, g = blockIdx.y;
  const int64_t t0 = (int64_t)g * S + (int64_t)ch * tpb;
  const int n = (int)min((int64_t)tpb, S - (int64_t)ch * tpb);
  sel::stage_rows(logits + t0 * E, zs, n * E, SigmoidOp());
  for (int e = tid; e < E; e += blockDim.x) {
    bs[e] = bias ? __ldg(bias + e) : 0.f;
    cnt[e] = 0;
  }
  if (ch == 0 && g == 0 && tid == 0) *ticket = 0u;  // for the finalize kernel that follows
  __syncthreads();
  if (keys) {
    float* kout = keys + t0 * E;
    for (int i = tid; i < n * E; i += blockDim.x) kout[i] = __fadd_rn(zs[i], bs[i % E]);
  }
  const int q = tid >> 2, r = tid & 3;
  const bool active = q < n;
  const float* row = zs + (int64_t)q * E;
  uint64_t win[KM];
  float ssum;
  sel::quad_topk<KM>(row, bs, E, K, r, q, active, win, &ssum);
  if (active) {
    float gsum = 0.f;
#pragma unroll
    for (int k = 0; k < KM; ++k)
      if (k < K) gsum += row[sel::unpack_e(win[k])];
    const float ginv = __frcp_rn(gsum);
    const int64_t o = (t0 + q) * K;
#pragma unroll
    for (int k = 0; k < KM; ++k) {
      if (k < K && (k & 3) == r) {
        const int e = sel::unpack_e(win[k]);
        idx[o + k] = e;
        prob[o + k] = row[e] * ginv;
        atomicAdd(cnt + e, 1);
      }
    }
    if (r == 0) inv[q] = __frcp_rn(ssum);
  }
  __syncthreads();
  const int64_t o = ((int64_t)g * nch + ch) * E;
  for (int e = tid; e < E; e += blockDim.x) {
    float acc = 0.f;
#pragma unroll 8
    for (int t = 0; t < n; ++t) acc += zs[t * E + e] * inv[t];
    psum[o + e] = acc;
    pcnt[o + e] = cnt[e];
  }
}

// f [GBS, E] and the loss.  Block (expert tile of 32, sequence g): warp w adds
// chunks w, w + 8, ...; warp 0 combines the 8 warps in order, writes f and the
// tile's sum of f P; the last block to finish adds the tiles in order.
__global__ void __launch_bounds__(256) balance_finalize_kernel(const float* __restrict__ psum,
                                                               const int32_t* __restrict__ pcnt, int64_t S, int E,
                                                               int K, int nch, float coef, int GBS,
                                                               float* __restrict__ f_out, float* __restrict__ tile_sum,
                                                               uint32_t* __restrict__ ticket,
                                                               float* __restrict__ loss) {
  __shared__ float rp[8][32];
  __shared__ int rc[8][32];
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  const int e = blockIdx.x * 32 + l, g = blockIdx.y;
  float P = 0.f;
  int c = 0;
  if (e < E) {
    for (int ch = w; ch < nch; ch += 8) {
      const int64_t o = ((int64_t)g * nch + ch) * E + e;
      P += psum[o];
      c += pcnt[o];
    }
  }
  rp[w][l] = P;
  rc[w][l] = c;
  __syncthreads();
  if (w != 0) return;
  P = 0.f;
  c = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    P += rp[i][l];
    c += rc[i][l];
  }
  float prod = 0.f;
  if (e < E) {
    const float f = (float)((double)E / ((double)K * (double)S) * (double)c);
    f_out[(int64_t)g * E + e] = f;
    prod = f * (P / (float)S);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) prod += __shfl_xor_sync(0xffffffffu, prod, off);
  const int nblk = gridDim.x * gridDim.y;
  unsigned last = 0;
  if (l == 0) {
    tile_sum[blockIdx.y * gridDim.x + blockIdx.x] = prod;
    __threadfence();
    last = atomicAdd(ticket, 1u) == (unsigned)(nblk - 1);
  }
  last = __shfl_sync(0xffffffffu, last, 0);
  if (!last) return;
  __threadfence();
  float tot = 0.f;
  for (int i = l; i < nblk; i += 32) tot += __ldcg(tile_sum + i);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, off);
  if (l == 0) {
    loss[0] = coef / (float)GBS * tot;
    *ticket = 0u;
  }
}

// One warp per token; lane l holds experts l, l + 32, ...  Gradient of the
// gate values of the chosen experts plus aux_grad times the balance loss with
// respect to all E logits, and its bf16 copy.
template <int VPL>
__global__ void __launch_bounds__(256) route_dz_sigmoid_kernel(
    const float* __restrict__ logits, const int32_t* __restrict__ idx, const float* __restrict__ prob,
    const float* __restrict__ dprob, const float* __restrict__ f, int64_t T, int64_t S, int E, int K, float cscale,
    float* __restrict__ dz, bf16* __restrict__ dz16, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= T) return;
  const float* row = logits + t * E;
  const float* fg = f + (t / S) * E;
  float s[VPL], c[VPL];
  float ssum = 0.f, csum = 0.f;
#pragma unroll
  for (int j = 0; j < VPL; ++j) {
    const int e = lane + 32 * j;
    s[j] = 0.f;
    c[j] = 0.f;
    if (e < E) {
      s[j] = sigmoidf_(__ldg(row + e));
      c[j] = cscale * __ldg(fg + e);
      ssum += s[j];
      csum += c[j] * s[j];
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    ssum += __shfl_xor_sync(0xffffffffu, ssum, off);
    csum += __shfl_xor_sync(0xffffffffu, csum, off);
  }
  const float rs = __frcp_rn(ssum);
  const float cbar = csum * rs;  // sum_i c_i s_i / sum_i s_i
  int my_e = -1;
  float my_p = 0.f, my_dp = 0.f, my_s = 0.f;
  if (lane < K) {
    my_e = idx[t * K + lane];
    if (my_e >= 0 && my_e < E) {
      my_p = prob[t * K + lane];
      my_dp = dprob[t * K + lane];
      my_s = sigmoidf_(__ldg(row + my_e));
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
  const float my_gate = (my_dp - dot) * __frcp_rn(gs);
  float gate[VPL];
#pragma unroll
  for (int j = 0; j < VPL; ++j) gate[j] = 0.f;
#pragma unroll
  for (int k = 0; k < kMaxK; ++k) {
    if (k < K) {
      const int ek = __shfl_sync(0xffffffffu, my_e, k);
      const float gk = __shfl_sync(0xffffffffu, my_gate, k);
#pragma unroll
      for (int j = 0; j < VPL; ++j)
        if (ek == lane + 32 * j) gate[j] = gk;
    }
  }
#pragma unroll
  for (int j = 0; j < VPL; ++j) {
    const int e = lane + 32 * j;
    if (e < E) {
      const float v = s[j] * (1.0f - s[j]) * (gate[j] + (c[j] - cbar) * rs);
      dz[t * E + e] = v;
      if (dz16) dz16[t * E + e] = __float2bfloat16_rn(v);
    }
  }
}

size_t align256(size_t v) { return (v + 255) & ~size_t(255); }

}  // namespace

size_t route_sigmoid_fwd_ws_bytes(int64_t T, int64_t S, int64_t GBS, int E) {
  (void)T;
  const int64_t parts = GBS * select_chunks(S, E) * E;
  const int64_t tiles = GBS * ((E + 31) / 32);
  return align256(parts * 4) * 2 + align256(tiles * 4) + 256;
}

cudaError_t launch_route_sigmoid_select(const Ctx& c, const float* logits, const float* bias, int64_t T, int64_t S,
                                        int64_t GBS, int E, int K, float coef, int32_t* idx, float* prob,
                                        float* f_out, float* loss, void* ws, float* keys) {
  if (T == 0) return cudaSuccess;
  const int tpb = sel::tokens_per_block(E);
  const int64_t nch = select_chunks(S, E);
  const int64_t parts = GBS * nch * E;
  const int64_t tiles = GBS * ((E + 31) / 32);
  char* base = static_cast<char*>(ws);
  float* psum = reinterpret_cast<float*>(base);
  int32_t* pcnt = reinterpret_cast<int32_t*>(base + align256(parts * 4));
  float* tile_sum = reinterpret_cast<float*>(base + 2 * align256(parts * 4));
  uint32_t* ticket = reinterpret_cast<uint32_t*>(base + 2 * align256(parts * 4) + align256(tiles * 4));
  {
    const size_t smem = (size_t)(tpb * E + E + tpb + E) * 4;
    dim3 grid((unsigned)nch, (unsigned)GBS);
    KernelScope ks("select_sigmoid", c.stream);
#define MOE_SELECT_SIGMOID(KM)                                                                             \
  select_sigmoid_kernel<KM><<<grid, 4 * tpb, smem, c.stream>>>(logits, bias, S, E, K, tpb, (int)nch, idx, \
                                                               prob, psum, pcnt, ticket, keys)
    switch (sel::k_bound(K)) {
      case 2: MOE_SELECT_SIGMOID(2); break;
      case 4: MOE_SELECT_SIGMOID(4); break;
      case 8: MOE_SELECT_SIGMOID(8); break;
      default: MOE_SELECT_SIGMOID(16); break;
    }
#undef MOE_SELECT_SIGMOID
  }
  cudaError_t st = cudaGetLastError();
  if (st != cudaSuccess) return st;
  {
    KernelScope ks("balance_finalize", c.stream);
    dim3 grid((unsigned)((E + 31) / 32), (unsigned)GBS);
    balance_finalize_kernel<<<grid, 256, 0, c.stream>>>(psum, pcnt, S, E, K, (int)nch, coef, (int)GBS, f_out,
                                                        tile_sum, ticket, loss);
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
  bf16* d16 = static_cast<bf16*>(dz16);
  KernelScope ks("route_dz_sigmoid", c.stream);
#define MOE_DZ_SIGMOID(VPL)                                                                                     \
  route_dz_sigmoid_kernel<VPL><<<grid, block, 0, c.stream>>>(logits, idx, prob, dprob, f, T, S, E, K, cscale, dz, \
                                                             d16, c.err)
  const int vpl = (E + 31) / 32;
  if (vpl <= 1) MOE_DZ_SIGMOID(1);
  else if (vpl <= 2) MOE_DZ_SIGMOID(2);
  else if (vpl <= 4) MOE_DZ_SIGMOID(4);
  else MOE_DZ_SIGMOID(8);
#undef MOE_DZ_SIGMOID
  return cudaGetLastError();
}

}  // namespace moe
