// Internal launcher interface between the C ABI (abi.cu) and the kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>
#include <stddef.h>

#include "moe.h"

namespace moe {

struct Ctx {
  cudaStream_t stream;
  uint32_t* err;   // device status word of the current device
  int num_sms;
  int device;
};

// Per-kernel CUDA-event timing and launch counting (implemented in abi.cu).
void prof_begin(const char* name, cudaStream_t s);
void prof_end(const char* name, cudaStream_t s);
void count_launch();

struct KernelScope {
  const char* name;
  cudaStream_t s;
  KernelScope(const char* n, cudaStream_t st) : name(n), s(st) { prof_begin(name, s); }
  ~KernelScope() { prof_end(name, s); count_launch(); }
};

enum class DType : int { BF16 = 0, F32 = 1 };

inline size_t dsize(DType t) { return t == DType::BF16 ? 2 : 4; }

// Shape validation and per-device context shared by the entry points
// (implemented in abi.cu).
struct ShapeInfo {
  int64_t T, TK;
  int K, D, E, F, H, Din;
  DType dt;
  size_t bx;
};
int abi_check_shape(const moe_shape_t* s, ShapeInfo* d);
int abi_device_ctx(void* stream, Ctx* c);
int abi_cuda_status(cudaError_t e);

// ---------------------------------------------------------------------------
// router.cu
// ---------------------------------------------------------------------------
constexpr int kMaxK = 16;
constexpr int kMaxE = 256;

cudaError_t launch_topk(const Ctx& c, const float* logits, int64_t T, int E, int K, int32_t* idx, float* prob);
// out[i] = sum over s of part[s * n + i], s = 0 .. S-1 in order (fp32).
cudaError_t launch_sum_splits(const Ctx& c, const float* part, int S, int64_t n, float* out);
// dz[T, E] fp32 (fully written) and optionally a bf16 copy whose rows are
// ld16 elements apart (0: E).
cudaError_t launch_route_dz(const Ctx& c, const int32_t* idx, const float* prob, const float* dprob, int64_t T,
                            int E, int K, float* dz, void* dz_bf16, int64_t ld16 = 0);

// ---------------------------------------------------------------------------
// router_sigmoid.cu
// ---------------------------------------------------------------------------
size_t route_sigmoid_fwd_ws_bytes(int64_t T, int64_t S, int64_t GBS, int E);
// idx/prob [T, K] from the sigmoid scores of logits [T, E] (bias [E] for the
// choice only, may be NULL), f [GBS, E] and loss [1] of the sequence-level
// balance loss.
cudaError_t launch_route_sigmoid_select(const Ctx& c, const float* logits, const float* bias, int64_t T, int64_t S,
                                        int64_t GBS, int E, int K, float coef, int32_t* idx, float* prob,
                                        float* f_out, float* loss, void* ws, float* keys = nullptr);
// dz [T, E] fp32 (fully written) and optionally a bf16 copy.
cudaError_t launch_route_dz_sigmoid(const Ctx& c, const float* logits, const int32_t* idx, const float* prob,
                                    const float* dprob, const float* f, int64_t T, int64_t S, int64_t GBS, int E,
                                    int K, float coef, float aux_grad, float* dz, void* dz16);

// ---------------------------------------------------------------------------
// permute.cu
// ---------------------------------------------------------------------------
size_t perm_workspace_bytes(int64_t TK, int E);
cudaError_t launch_permutation(const Ctx& c, const int32_t* idx, const float* prob, int64_t T, int K, int E,
                               int32_t* offsets, int32_t* row_of_slot, int32_t* token_of_row, float* prob_perm,
                               void* ws);
cudaError_t launch_dispatch_rows(const Ctx& c, const void* x, const int32_t* row_of_slot, int64_t T, int K,
                                 int64_t row_bytes, void* x_perm);
cudaError_t launch_combine(const Ctx& c, DType dt, const void* y_perm, const float* prob_perm,
                           const int32_t* row_of_slot, int64_t T, int K, int D, void* y);
cudaError_t launch_combine_bwd(const Ctx& c, DType dt, const void* dy, const void* y_perm, const float* prob_perm,
                               const int32_t* row_of_slot, int64_t T, int K, int D, void* dy_perm,
                               float* dprob_perm);
// dx rows ldx elements apart (0: D).
cudaError_t launch_dispatch_bwd(const Ctx& c, DType dt, const void* dx_perm, const float* dprob_perm,
                                const int32_t* row_of_slot, int64_t T, int K, int D, void* dx, float* dprob,
                                int64_t ldx = 0);
// permute.cu: the dispatch backward fused with the softmax router's dz and
// dx += dz . w_router (w_router [E, D]); dz16 (bf16 copy of dz) may be NULL.
cudaError_t launch_dispatch_route_bwd(const Ctx& c, DType dt, const void* dx_perm, const float* dprob_perm,
                                      const int32_t* row_of_slot, const int32_t* idx, const float* prob,
                                      const void* w_router, int64_t T, int K, int E, int D, void* dx, float* dprob,
                                      float* dz, void* dz16);
cudaError_t launch_pack_w1(const Ctx& c, DType dt, const void* w_gate, const void* w_up, int E, int F, int D,
                           void* w1);

// fp8_payload.cu: E4M3 codes [TK, D] and power-of-two row scales [TK] of the
// bf16 rows x [T, D] written to each token's K rows; and their bf16 values.
cudaError_t launch_dispatch_fp8(const Ctx& c, const void* x, const int32_t* row_of_slot, int64_t T, int K, int D,
                                void* xq, float* scale_perm);
cudaError_t launch_dequant_rows(const Ctx& c, const void* xq, const float* scale, int64_t rows, int D, void* out);

// nvfp4_payload.cu: E2M1 codes [TK, D/2] (two per byte), E4M3 block scales
// [TK, D/16] and power-of-two row scales [TK] of the bf16 rows x [T, D]
// written to each token's K rows; and their bf16 values.
cudaError_t launch_dispatch_nvfp4(const Ctx& c, const void* x, const int32_t* row_of_slot, int64_t T, int K, int D,
                                  void* xq, uint8_t* bscale, float* rscale);
cudaError_t launch_dequant_nvfp4(const Ctx& c, const void* xq, const uint8_t* bscale, const float* rscale,
                                 int64_t rows, int D, void* out);

// swiglu.cu: dH [rows, 2F] (packed) from dA [rows, F] and the saved h [rows, 2F].
cudaError_t launch_swiglu_bwd(const Ctx& c, DType dt, const void* dA, const void* h, int64_t rows, int F,
                              void* dH);
// swiglu.cu: dh = 2 max(h, 0) dA over n elements (dh may alias dA).
cudaError_t launch_relusq_bwd(const Ctx& c, DType dt, const void* dA, const void* h, int64_t n, void* dh);

// ---------------------------------------------------------------------------
// Grouped GEMM  C(m, n) = sum_k A(m, k) B(n, k), fp32 accumulation.
// ---------------------------------------------------------------------------
enum class Group : int {
  Dense = 0,  // one problem: M x N x K
  M = 1,      // group g owns rows [offsets[g], offsets[g+1]) of A and C; B advanced by g * sb_g
  K = 2,      // group g reduces over k in [offsets[g], offsets[g+1]); C advanced by g * sc_g
};

enum class Epi : int {
  Store = 0,      // C = acc
  StoreBias = 1,  // C = acc + bias[n]
  Accum = 2,      // C = C + acc
  SwigluFwd = 3,  // acc is h (packed gate/up, N = 2F): C = h, aux[m, f] = silu(g) u  (aux ld = N/2)
  ReluSqFwd = 4,  // acc is h: C = h, aux[m, n] = max(h, 0)^2  (aux ld = ldc)
  SwigluBwd = 5,  // acc is dA (N = F); aux is the saved h (packed gate/up blocks of 64, ld = ldc = 2N):
                  // C = dH in h's layout, dg = dA u s (1 + g (1 - s)), du = dA g s, s = sigmoid(g)
};

struct GemmDesc {
  Group group = Group::Dense;
  Epi epi = Epi::Store;
  int64_t M = 0, N = 0, K = 0;  // the grouped dimension is taken from offsets
  int num_groups = 1;
  const int32_t* offsets = nullptr;  // [num_groups + 1], device
  int64_t max_rows = 0;              // Group::M: total rows (upper bound for the grid)
  const void* A = nullptr;
  DType a_type = DType::BF16;
  int64_t sa_m = 0, sa_k = 0;        // element strides of A(m, k)
  const void* B = nullptr;
  DType b_type = DType::BF16;
  int64_t sb_n = 0, sb_k = 0, sb_g = 0;
  void* C = nullptr;
  DType c_type = DType::BF16;
  int64_t ldc = 0, sc_g = 0;
  const float* bias = nullptr;       // StoreBias
  void* aux = nullptr;               // SwigluFwd / ReluSqFwd activation output (c_type);
                                     // SwigluBwd: the saved h, only read
  void* scratch = nullptr;           // Group::K on the tensor-core engine: per-group tensor maps
                                     // (gemm_tc_group_scratch_bytes, 128-byte aligned)
  bool maps_ready = false;           // Group::K: the maps in scratch were already built
                                     // (gemm_tc_group_maps_pair)
  int64_t split_rows = 0;            // Group::K with offsets == nullptr: num_groups equal splits of
                                     // [0, split_rows) (split-K of a dense product)
  const int32_t* gather = nullptr;   // row indirection into a source matrix of gather_rows rows:
  int64_t gather_rows = 0;           //   Group::M: A's row m is source row gather[m];
                                     //   Group::K: B's k row k is source row gather[k]
};

cudaError_t launch_gemm_simt(const Ctx& c, const GemmDesc& d, const char* name);

// tcgen05 / TMA engine (bf16 operands only).  Returns cudaErrorNotSupported
// for a descriptor it does not handle.
bool gemm_tc_supports(const GemmDesc& d);
size_t gemm_tc_group_scratch_bytes(int num_groups);
cudaError_t launch_gemm_tc(const Ctx& c, const GemmDesc& d, const char* name);
// Builds the per-group tail maps of two Group::K GEMMs over the same groups
// (the two expert weight gradients) in one launch, into d0.scratch and
// d1.scratch.  Returns false, launching nothing, unless both are tensor-core
// GEMMs grouped by expert offsets; *err receives the launch status.
bool gemm_tc_group_maps_pair(const Ctx& c, const GemmDesc& d0, const GemmDesc& d1, cudaError_t* err);

}  // namespace moe
