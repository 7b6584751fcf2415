/*
 * moe.h -- C ABI of the GB300 (sm_103a) dropless routed MoE layer library.
 *
 * One routed Mixture-of-Experts layer, forward and backward, on one GPU.
 * The layer is the object of the paper's Eq. 1 (Sec. 1): dropless routing
 * with no capacity padding, each token dispatched to its K routed experts as a
 * hidden vector of width D (b_x bytes per element) plus one routed probability
 * (b_p = 4 bytes, fp32).  Sec. 4.1 (footnote on the all-to-all dispatcher)
 * names the six transfers of one layer: hidden dispatch, probability dispatch
 * and hidden combine forward, plus their three inverses backward.  With every
 * expert on one GPU those transfers become the in-HBM permutes below
 * (moe_dispatch, moe_combine, moe_combine_bwd, moe_dispatch_bwd).  Sec. 5.2
 * names the building blocks (grouped-GEMM experts, fused permute); the
 * LatentMoE projections (Sec. 1 levers list, Table 2) are moe_latent_proj*.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - T = S * GBS tokens, TK = T * K routed slots; slot s = t * K + k is token
 *    t's k-th routed expert.  "Rows" are the slots in expert-grouped order:
 *    expert e owns rows [expert_offsets[e], expert_offsets[e+1]), and within
 *    an expert rows are ordered by token (a counting sort, stable in t).
 *  - Every data pointer is a DEVICE pointer owned by the caller, row-major and
 *    contiguous, 16-byte aligned.  The library never allocates or frees
 *    caller-visible memory; scratch comes from the caller-provided workspace
 *    `ws` of `ws_bytes` bytes (size from moe_workspace_size).
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Every call only enqueues work on that stream and returns; there
 *    is no host synchronisation (moe_check_device_status excepted).
 *  - Activation and weight storage dtype is shape->x_dtype (MOE_BF16: b_x = 2,
 *    MOE_F32: b_x = 4).  Probabilities, logits and their gradients are fp32;
 *    weight gradients are written fp32; routing indices and the permutation
 *    are int32.  All accumulations are fp32.  MOE_F32 uses plain fp32 FMA
 *    throughout (no TF32).
 *  - Return value: MOE_OK (0) or a negative moe_status.  On error nothing has
 *    been enqueued.  Errors found on the device (an out-of-range expert index,
 *    a bounded wait that expired) set a device status word that
 *    moe_check_device_status reads.
 *
 * Weight layouts
 *  - w_router [E, Din]: logits z = x . w_router^T (Din = H for LatentMoE,
 *    else D).
 *  - w1 [E, 2F, D]: gate and up projections packed by moe_pack_w1, in blocks
 *    of 64 rows: rows [128 i, 128 i + 64) are gate rows 64 i .. 64 i + 63 and
 *    rows [128 i + 64, 128 i + 128) are the up rows of the same 64 features.
 *    The saved pre-activation h [TK, 2F] and its gradient use the same order.
 *  - w2 [E, D, F]: Y = a . w2_e^T.
 *  - Gradients dw1 / dw2 / dw_router have the layouts of w1 / w2 / w_router.
 */
#ifndef MOE_GB300_H
#define MOE_GB300_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MOE_OK = 0,
    MOE_ERR_SHAPE = -1,       /* non-positive or inconsistent sizes, K > E, E > 256, D or F not a multiple of 64, overflow */
    MOE_ERR_DTYPE = -2,       /* unknown x_dtype */
    MOE_ERR_ALIGN = -3,       /* a pointer not 16-byte aligned */
    MOE_ERR_NULL = -4,        /* a required pointer is NULL */
    MOE_ERR_WORKSPACE = -5,   /* ws_bytes smaller than moe_workspace_size() */
    MOE_ERR_CUDA = -6,        /* a CUDA runtime call or launch failed (see moe_last_cuda_error) */
    MOE_ERR_DEVICE = -7,      /* the device status word is set (moe_check_device_status) */
    MOE_ERR_UNSUPPORTED = -8, /* valid request this build does not implement */
    MOE_ERR_TOO_LARGE = -9    /* shape exceeds the fixed scratch of moe_dispatch_noalloc */
} moe_status;

typedef enum { MOE_BF16 = 0, MOE_F32 = 1 } moe_dtype;

/* Eq. 1 symbols: S sequence length, GBS global batch, K routed top-K, D
 * dispatch hidden width; plus E experts, F expert SwiGLU width, the b_x dtype
 * and H, the model width of a LatentMoE layer (0 = no latent projection). */
typedef struct {
    int64_t S;
    int64_t GBS;
    int32_t K;
    int32_t D;
    int32_t E;
    int32_t F;
    int32_t x_dtype;  /* moe_dtype */
    int32_t H;
} moe_shape_t;

/* Bytes of scratch the calls below need for this shape (the maximum over all
 * calls; one workspace may be reused by every call on one stream).  Returns
 * MOE_OK and writes *bytes, or a shape error. */
int moe_workspace_size(const moe_shape_t* shape, size_t* bytes);

/* Router (reading R1, R2, R7): logits[T, E] = x[T, Din] . w_router^T (+ bias),
 * then moe_topk.  bias [E] fp32 is optional (NULL = none) and is added in fp32
 * after the product.  Din = H when shape->H > 0, else D. */
int moe_route(const moe_shape_t* shape, const void* x, const void* w_router, const float* bias,
              float* logits, int32_t* topk_idx, float* topk_prob, void* ws, size_t ws_bytes, void* stream);

/* Top-K of given fp32 logits [T, E] (four threads per token): the K largest
 * logits (ties to the lower expert index), ordered by descending logit, and
 * renormalised probabilities p_k = exp(z_k - z_max) / sum over the K chosen
 * (equal to softmax over all E restricted to the chosen set). */
int moe_topk(const moe_shape_t* shape, const float* logits, int32_t* topk_idx, float* topk_prob, void* stream);

/* Dispatch (forward hidden and probability transfers, Sec. 4.1 footnote):
 * builds expert_offsets [E+1], row_of_slot [TK] and token_of_row [TK] by a
 * deterministic counting sort of topk_idx [T, K] (histogram + prefix sum),
 * then x_perm[row] = x[token_of_row[row]] ([TK, D]) and
 * prob_perm[row] = topk_prob[slot].  x is the dispatch input [T, D] (for
 * LatentMoE the down-projected x_lat).  x_perm may be NULL to build only the
 * permutation and prob_perm.  Expert indices outside [0, E) set the device
 * status word and are skipped. */
int moe_dispatch(const moe_shape_t* shape, const void* x, const int32_t* topk_idx, const float* topk_prob,
                 int32_t* expert_offsets, int32_t* row_of_slot, int32_t* token_of_row,
                 void* x_perm, float* prob_perm, void* ws, size_t ws_bytes, void* stream);

/* Dispatch with a low-precision payload (Sec. 1: lower-precision
 * communication, b_x of Eq. 1; readings FP1-FP2): the permutation and
 * prob_perm as moe_dispatch, and each token's row of x [T, D] (bf16 only;
 * MOE_ERR_UNSUPPORTED otherwise) sent to its K rows as FP8 E4M3 codes,
 * x_perm_q [TK, D] (one byte each), with one fp32 scale per row,
 * x_scale_perm [TK]: the smallest power of two s = 2^e, e >= -126, with
 * max_i |x_i| <= 448 s (1 for an all-zero row); code_i = the E4M3 value nearest
 * x_i / s, ties to even, saturating at +-448.  The payload per routed slot is
 * D + 4 + 4 bytes (codes, scale, probability) instead of 2 D + 4. */
int moe_dispatch_fp8(const moe_shape_t* shape, const void* x, const int32_t* topk_idx, const float* topk_prob,
                     int32_t* expert_offsets, int32_t* row_of_slot, int32_t* token_of_row, void* x_perm_q,
                     float* x_scale_perm, float* prob_perm, void* ws, size_t ws_bytes, void* stream);

/* The receiving side of moe_dispatch_fp8: x_perm[r, i] = value(code) * scale[r]
 * in bf16 ([TK, D]; exact, the scale being a power of two). */
int moe_dequant_rows(const moe_shape_t* shape, const void* x_perm_q, const float* x_scale_perm, void* x_perm,
                     void* stream);

/* Dispatch with an NVFP4 payload (Sec. 1: lower-precision communication, b_x
 * of Eq. 1; Sec. 6 names FP8 and NVFP4; readings NV1-NV3): the permutation and
 * prob_perm as moe_dispatch, and each token's row x of x [T, D] (bf16 only;
 * MOE_ERR_UNSUPPORTED otherwise) sent to its K rows in three arrays:
 *   x_rscale_perm [TK] fp32: g = the smallest power of two 2^e, e >= -126,
 *     with max_i |x_i| <= 6 * 448 * g (1 for an all-zero row);
 *   x_bscale_perm [TK, D/16] E4M3 codes: per block b of 16 consecutive
 *     elements, s_b = the E4M3 value nearest to the fp32 quotient
 *     max_{i in b} |x_i| / (6 g), ties to even, saturating;
 *   x_perm_q [TK, D/2] bytes: E2M1 codes (magnitudes 0, 0.5, 1, 1.5, 2, 3, 4,
 *     6 and a sign bit), code_i = the E2M1 value nearest to the fp32 quotient
 *     x_i / (s_b g), ties to even, saturating at +-6, zero where s_b = 0;
 *     element 2j in the low nibble of byte j.
 * The payload per routed slot is D/2 + D/16 + 4 + 4 bytes instead of 2 D + 4. */
int moe_dispatch_nvfp4(const moe_shape_t* shape, const void* x, const int32_t* topk_idx, const float* topk_prob,
                       int32_t* expert_offsets, int32_t* row_of_slot, int32_t* token_of_row, void* x_perm_q,
                       uint8_t* x_bscale_perm, float* x_rscale_perm, float* prob_perm, void* ws, size_t ws_bytes,
                       void* stream);

/* The receiving side of moe_dispatch_nvfp4: x_perm[r, i] = value(code) * s_b * g
 * in bf16 ([TK, D]; exact: at most 6 significant bits times a power of two). */
int moe_dequant_nvfp4(const moe_shape_t* shape, const void* x_perm_q, const uint8_t* x_bscale_perm,
                      const float* x_rscale_perm, void* x_perm, void* stream);

/* Dispatch that allocates nothing and takes no workspace.  The paper has no
 * counterpart: this entry point exists for callers that cannot allocate
 * device memory when they call the layer -- a host framework that has already
 * reserved all device memory for its own pool or forbids allocation inside its
 * step loop, or a runtime that cannot afford cudaMalloc's implicit device-wide
 * synchronisation -- and so cannot provide the workspace moe_dispatch needs.
 *
 * Results are identical to moe_dispatch (same arguments minus ws/ws_bytes).
 * The counting sort's per-chunk histogram table, E * ceil(T*K / 2048)
 * int32 values, lives in one fixed device array of
 * MOE_DISPATCH_NOALLOC_SCRATCH_INTS int32 (1 MiB) compiled into the library;
 * every GPU that loads the library holds its copy until the process exits.
 * The call makes no cudaMalloc / cudaFree or other allocating call.
 *  - A shape whose table does not fit (E * ceil(T*K / 2048) > 262144) returns
 *    MOE_ERR_TOO_LARGE before anything is enqueued.
 *  - The first call on a device looks up that device's copy of the array
 *    (cudaGetSymbolAddress, with the device current).  With CUDA's lazy module
 *    loading that first lookup is also when the library's module is loaded on
 *    the device and the array is placed, which may allocate device memory and
 *    synchronise; only the calls after it allocate nothing.  Make one warm-up
 *    call per device at initialisation, before any stream capture.
 *  - On a device with an ordinal of 64 or more the call returns MOE_ERR_CUDA
 *    (cudaErrorInvalidDevice) without enqueuing anything.
 *  - All calls share the one array.  Each call writes every table entry it
 *    reads before reading it, so nothing from an earlier call leaks into a
 *    result; but calls whose kernels overlap on the GPU (different streams or
 *    host threads without ordering between them) race on the array, and the
 *    caller must order them. */
#define MOE_DISPATCH_NOALLOC_SCRATCH_INTS 262144
int moe_dispatch_noalloc(const moe_shape_t* shape, const void* x, const int32_t* topk_idx,
                         const float* topk_prob, int32_t* expert_offsets, int32_t* row_of_slot,
                         int32_t* token_of_row, void* x_perm, float* prob_perm, void* stream);

/* Grouped SwiGLU expert FFN (Sec. 5.2 grouped GEMM; reading R6): for every
 * expert e and its rows, h = x_perm . w1_e^T ([rows, 2F], packed order),
 * a = silu(g) * u ([rows, F]), y_perm = a . w2_e^T ([rows, D]).  h_save and
 * act_save are written for the backward pass.  Reads expert_offsets on the
 * device (no host synchronisation). */
int moe_expert_ffn(const moe_shape_t* shape, const void* x_perm, const int32_t* expert_offsets,
                   const void* w1, const void* w2, void* h_save, void* act_save, void* y_perm,
                   void* ws, size_t ws_bytes, void* stream);

/* moe_expert_ffn with GEMM-1 reading its rows straight from the dispatch
 * input: row r of expert e is x[token_of_row[r]] (x [T, D]; for LatentMoE the
 * down-projected x_lat), copied row by row by the GEMM's producer (16-byte
 * cp.async copies), so the dispatched copy x_perm is never written
 * (moe_dispatch may then be called with x_perm = NULL).  Same results as
 * moe_expert_ffn on x_perm = x[token_of_row]; slower on GB300 than the tiled
 * copies of x_perm. */
int moe_expert_ffn_gather(const moe_shape_t* shape, const void* x, const int32_t* token_of_row,
                          const int32_t* expert_offsets, const void* w1, const void* w2, void* h_save,
                          void* act_save, void* y_perm, void* ws, size_t ws_bytes, void* stream);

/* Combine (forward hidden combine, Sec. 4.1 footnote; reading R5):
 * y[t] = sum_k prob_perm[r] * y_perm[r], r = row_of_slot[t K + k], fp32
 * accumulation, one rounding to the storage dtype.  y is [T, D]. */
int moe_combine(const moe_shape_t* shape, const void* y_perm, const float* prob_perm, const int32_t* row_of_slot,
                void* y, void* stream);

/* Combine backward (inverse of the combine): dy_perm[r] = prob_perm[r] * dy[t]
 * and dprob_perm[r] = <dy[t], y_perm[r]> (fp32) for every slot (t, k). */
int moe_combine_bwd(const moe_shape_t* shape, const void* dy, const void* y_perm, const float* prob_perm,
                    const int32_t* row_of_slot, void* dy_perm, float* dprob_perm, void* stream);

/* Expert FFN backward: dA = dy_perm . w2_e, SwiGLU backward from the saved h
 * (dg = dA u sigmoid(g) (1 + g (1 - sigmoid(g))), du = dA silu(g)),
 * dx_perm = dH . w1_e, dw2_e = dy_perm_e^T . a_e, dw1_e = dH_e^T . x_perm_e.
 * dw1 [E, 2F, D] and dw2 [E, D, F] are fp32 and fully written (zero for an
 * expert with no rows).  dH [TK, 2F] lives in the workspace.  With bf16 operands
 * the SwiGLU backward runs in dA's GEMM on its fp32 accumulator (dA is never
 * stored); with fp32 operands dA is stored in the workspace and a separate pass
 * reads it back. */
int moe_expert_ffn_bwd(const moe_shape_t* shape, const void* dy_perm, const void* x_perm, const void* h_save,
                       const void* act_save, const int32_t* expert_offsets, const void* w1, const void* w2,
                       void* dx_perm, float* dw1, float* dw2, void* ws, size_t ws_bytes, void* stream);

/* moe_expert_ffn_bwd whose GEMM-1 weight gradient gathers the rows of x
 * [T, D] by token_of_row instead of reading x_perm (same results). */
int moe_expert_ffn_bwd_gather(const moe_shape_t* shape, const void* dy_perm, const void* x,
                              const int32_t* token_of_row, const void* h_save, const void* act_save,
                              const int32_t* expert_offsets, const void* w1, const void* w2, void* dx_perm,
                              float* dw1, float* dw2, void* ws, size_t ws_bytes, void* stream);

/* Dispatch backward (inverse of the hidden and probability dispatches):
 * dx[t] = sum_k dx_perm[r] (fp32 accumulation; dx [T, D] is overwritten) and
 * dtopk_prob[t, k] = dprob_perm[r], r = row_of_slot[t K + k]. */
int moe_dispatch_bwd(const moe_shape_t* shape, const void* dx_perm, const float* dprob_perm,
                     const int32_t* row_of_slot, void* dx, float* dtopk_prob, void* stream);

/* Router backward: dlogits[t, j] = p_j (dp_j - sum_k p_k dp_k) for the K
 * chosen experts, 0 elsewhere ([T, E] fp32, fully written);
 * dx[T, Din] += dlogits . w_router (accumulated into the existing contents,
 * one rounding); dw_router [E, Din] = dlogits^T . x (fp32, overwritten).
 * The logit bias gets no gradient. */
int moe_route_bwd(const moe_shape_t* shape, const void* x, const void* w_router, const int32_t* topk_idx,
                  const float* topk_prob, const float* dtopk_prob, void* dx, float* dw_router, float* dlogits,
                  void* ws, size_t ws_bytes, void* stream);

/* moe_dispatch_bwd followed by moe_route_bwd in one pass over the tokens, for
 * a layer without latent projection (H = 0; MOE_ERR_UNSUPPORTED otherwise),
 * where the router reads the dispatch input x [T, D].  dlogits is nonzero only
 * on each token's K chosen experts, so dlogits . w_router for token t is a sum
 * of K rows of w_router [E, D]; it is added while the K rows of dx_perm are
 * summed:
 *   dx[t] = sum_k dx_perm[r_k] + sum_k dlogits[t, e_k] w_router[e_k]
 * with fp32 accumulation and ONE rounding (the two separate calls round dx
 * twice), dtopk_prob and dlogits as the two calls (dlogits bit-identical),
 * dw_router = dlogits^T . x as moe_route_bwd.  dx [T, D] is overwritten.
 * Workspace as moe_route_bwd. */
int moe_dispatch_route_bwd(const moe_shape_t* shape, const void* dx_perm, const float* dprob_perm,
                           const int32_t* row_of_slot, const void* x, const void* w_router, const int32_t* topk_idx,
                           const float* topk_prob, void* dx, float* dtopk_prob, float* dlogits, float* dw_router,
                           void* ws, size_t ws_bytes, void* stream);

/* The backward tail of a LatentMoE layer with the softmax router (H > 0,
 * bf16, (D + E) a multiple of 8; MOE_ERR_UNSUPPORTED otherwise), in place of
 * moe_dispatch_bwd into dx_lat, moe_latent_proj_bwd of the down-projection
 * and moe_route_bwd.  The router reads x [T, H], so its dx term is not a sum
 * of rows of the dispatch gradient.  Instead both gradients into x come out
 * of ONE product over the concatenated reduction dimension:
 *   dx_cat = [dx_lat | dz] [T, D + E] (bf16, written: the dispatch backward's
 *   sums in columns 0 .. D-1, the bf16 copy of dlogits in D .. D+E-1) times
 *   w_down_router [D + E, H] = w_down [D, H] stacked on w_router [E, H]
 *   (one contiguous array: the caller keeps the two weights there),
 *   dx = dx_lat . w_down + dlogits . w_router  (fp32 accumulation, one rounding;
 *   the separate calls round twice).
 * dtopk_prob, dlogits, dw_down = dx_lat^T . x and dw_router = dlogits^T . x
 * (fp32) are as the separate calls compute them.  dx [T, H] is overwritten.
 * Workspace: moe_workspace_size(). */
int moe_latent_route_bwd(const moe_shape_t* shape, const void* dx_perm, const float* dprob_perm,
                         const int32_t* row_of_slot, const void* x, const void* w_down_router,
                         const int32_t* topk_idx, const float* topk_prob, void* dx_cat, void* dx,
                         float* dtopk_prob, float* dlogits, float* dw_down, float* dw_router, void* ws,
                         size_t ws_bytes, void* stream);

/* Sigmoid router with expert bias and the sequence-level balance loss
 * (Sec. 5.2 experimental details; the paper gives no formulas, readings S1-S3):
 *   logits[T, E] = x[T, Din] . w_router^T (fp32, no logit bias);
 *   s = sigmoid(logits); the K experts with the largest s + expert_bias
 *   (ties to the lower expert index, slots by descending s + b) -> topk_idx;
 *   topk_prob[t, k] = s_k / sum over the K chosen of s (the bias shapes the
 *   choice only);
 *   sequence g = tokens g*S .. g*S+S-1 (shape->S tokens, shape->GBS sequences):
 *   aux_f[g, i] = E / (K S) * #{t in g : i chosen}  ([GBS, E] fp32, written),
 *   P[g, i] = mean over t in g of s_ti / sum_j s_tj,
 *   aux_loss[0] = aux_coef / GBS * sum_{g,i} aux_f[g, i] P[g, i]  (fp32).
 * expert_bias [E] fp32 may be NULL (zero).  Every reduction runs in a fixed
 * order: results are bit-reproducible.  A NaN aux_coef is MOE_ERR_SHAPE. */
int moe_route_sigmoid(const moe_shape_t* shape, const void* x, const void* w_router, const float* expert_bias,
                      float aux_coef, float* logits, int32_t* topk_idx, float* topk_prob, float* aux_f,
                      float* aux_loss, void* ws, size_t ws_bytes, void* stream);

/* The selection and balance-statistics stage of moe_route_sigmoid on given
 * fp32 logits [T, E] (Sec. 5.2; readings S1-S3): topk_idx, topk_prob, aux_f
 * and aux_loss exactly as moe_route_sigmoid computes them from its own
 * logits.  select_keys [T, E] fp32 (optional, NULL = not written) receives
 * every key the selection compared, s + expert_bias with s = sigmoid(logits),
 * formed by the same fp32 arithmetic: the K largest of a row, ties to the
 * lower expert, are topk_idx.  Workspace as moe_route_sigmoid. */
int moe_topk_sigmoid(const moe_shape_t* shape, const float* logits, const float* expert_bias, float aux_coef,
                     float* select_keys, int32_t* topk_idx, float* topk_prob, float* aux_f, float* aux_loss,
                     void* ws, size_t ws_bytes, void* stream);

/* Sigmoid router backward: gradient of (the downstream loss through
 * topk_prob, given as dtopk_prob [T, K]) + aux_grad * aux_loss with respect to
 * the logits, with aux_f from moe_route_sigmoid (a count: no gradient) and
 * c_gi = aux_grad * aux_coef / (GBS S) * aux_f[g, i]:
 *   dL/ds_j = [j chosen] (dp_j - sum_k p_k dp_k) / sum_{chosen} s
 *             + (c_gj - sum_i c_gi s_i / sum s) / sum_i s_i,
 *   dlogits[t, j] = s_j (1 - s_j) dL/ds_j  ([T, E] fp32, fully written);
 * then dx[T, Din] += dlogits . w_router (one rounding) and
 * dw_router [E, Din] = dlogits^T . x (fp32, overwritten), as moe_route_bwd.
 * The expert bias gets no gradient.  logits are moe_route_sigmoid's. */
int moe_route_sigmoid_bwd(const moe_shape_t* shape, const void* x, const void* w_router, const float* logits,
                          const int32_t* topk_idx, const float* topk_prob, const float* dtopk_prob,
                          const float* aux_f, float aux_coef, float aux_grad, void* dx, float* dw_router,
                          float* dlogits, void* ws, size_t ws_bytes, void* stream);

/* Shared expert (Sec. 5.2 experimental details: an ungated shared expert MLP
 * in parallel with the routed experts, its output added to the combined routed
 * output; readings SH1-SH2): with F_s hidden units (a multiple of 64),
 *   h_save[T, F_s] = x[T, Din] . w_s1^T   (w_s1 [F_s, Din]),
 *   act_save[T, F_s] = max(h, 0)^2        (squared ReLU, no gate, no biases),
 *   y[T, Din] += act . w_s2^T             (w_s2 [Din, F_s]; added to the existing
 *                                          contents, i.e. the routed output).
 * Call it after the routed output is in y (after the LatentMoE up-projection). */
int moe_shared_expert(const moe_shape_t* shape, int32_t F_s, const void* x, const void* w_s1, const void* w_s2,
                      void* h_save, void* act_save, void* y, void* stream);

/* Shared expert backward from dy [T, Din] and the saved h and act:
 *   dh[T, F_s] = 2 max(h, 0) (dy . w_s2)   (caller's buffer, overwritten),
 *   dx[T, Din] += dh . w_s1                 (added to the existing contents),
 *   dw_s1 [F_s, Din] = dh^T . x, dw_s2 [Din, F_s] = dy^T . act (fp32, overwritten). */
int moe_shared_expert_bwd(const moe_shape_t* shape, int32_t F_s, const void* dy, const void* x, const void* h_save,
                          const void* act_save, const void* w_s1, const void* w_s2, void* dh, void* dx,
                          float* dw_s1, float* dw_s2, void* stream);

/* LatentMoE projection (dense, T rows): out[T, n_out] = in[T, n_in] . w^T with
 * w [n_out, n_in].  Down-projection: n_in = H, n_out = D; up-projection:
 * n_in = D, n_out = H. */
int moe_latent_proj(const moe_shape_t* shape, int32_t n_in, int32_t n_out, const void* in, const void* w,
                    void* out, void* ws, size_t ws_bytes, void* stream);

/* LatentMoE projection backward: din = dout . w (overwritten, or added to the
 * existing contents when accumulate != 0), dw [n_out, n_in] = dout^T . in
 * (fp32, overwritten).  din may be NULL to skip it. */
int moe_latent_proj_bwd(const moe_shape_t* shape, int32_t n_in, int32_t n_out, const void* dout, const void* in,
                        const void* w, void* din, int32_t accumulate, float* dw, void* ws, size_t ws_bytes,
                        void* stream);

/* Packs w_gate [E, F, D] and w_up [E, F, D] into w1 [E, 2F, D] (layout above). */
int moe_pack_w1(const moe_shape_t* shape, const void* w_gate, const void* w_up, void* w1, void* stream);

/* Eq. 1 per-layer logical payload with L_E = 1 and constant 1:
 * S * GBS * K * (4 D b_x + 2 b_p), b_p = 4.  Host only; 0 on a bad shape. */
uint64_t moe_eq1_bytes(const moe_shape_t* shape);

/* ---- CE-MoE layout tools (host only) ------------------------------------
 * Layer composition (Sec. 4.1): from a baseline of a_star Mamba, b_star MoE
 * and c_star attention blocks (L = a_star + b_star + c_star) and a target
 * token-mixing-to-MoE ratio alpha, the CE-MoE composition keeps c = c_star,
 * sets b = d = floor(L / (alpha + 2)) MoE and dense-FFN blocks and gives the
 * rest to Mamba: a = L - b - c - d.  MOE_ERR_SHAPE if a would be negative. */
int moe_ce_composition(int32_t a_star, int32_t b_star, int32_t c_star, double alpha, int32_t* a, int32_t* b,
                       int32_t* c, int32_t* d);

/* Layer pattern of Algorithm 1 (Sec. 4.2) for a composition (a Mamba, b MoE,
 * c attention, d dense FFN; b >= c).  Writes the pattern over M, E, * and -
 * into `pattern` (NUL-terminated), the virtual-block order over A / N / R into
 * `blocks` and the pattern with A blocks in [ ] and N / R blocks in ( ) into
 * `decorated` (either may be NULL).  Readings where the algorithm is loose:
 * Distribute gives the N blocks near-equal groups of A blocks between them,
 * larger groups first; Phase 3 makes one residue block per remaining MoE,
 * attention or dense block (at least one) and shares the remaining Mamba
 * evenly, larger shares first.  Returns the pattern length, or MOE_ERR_SHAPE
 * (bad counts, or a buffer too small) / MOE_ERR_NULL. */
int moe_ce_layer_pattern(int32_t a, int32_t b, int32_t c, int32_t d, char* pattern, size_t pattern_cap,
                         char* blocks, size_t blocks_cap, char* decorated, size_t decorated_cap);

/* Synchronises `stream`, then returns MOE_OK, MOE_ERR_DEVICE if the device
 * status word of the current device is set (and clears it), or MOE_ERR_CUDA.
 * Off the timed path. */
int moe_check_device_status(void* stream);

/* Raw device status word of the current device (bit flags, 0 = clean):
 * 1 = expert index out of range, 2 = a bounded pipeline wait expired. */
int moe_device_status_word(void* stream, uint32_t* word);

/* Last cudaError_t seen by a call that returned MOE_ERR_CUDA (0 if none). */
int moe_last_cuda_error(void);

/* Human-readable text for a moe_status. */
const char* moe_strerror(int status);

/* Library version (major * 10000 + minor * 100 + patch). */
int moe_version(void);

/* Per-kernel timing.  While enabled, every kernel launch is bracketed by
 * CUDA events on its launch stream; moe_prof_get reads the accumulated
 * device time per kernel name (synchronising on the recorded events). */
int moe_prof_enable(int on);
int moe_prof_reset(void);
int moe_prof_count(void);
int moe_prof_get(int i, const char** name, int* launches, double* total_ms);

/* Kernel launches made by this library since load (all streams). */
uint64_t moe_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* MOE_GB300_H */
