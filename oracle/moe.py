"""Float64 reference for one dropless routed MoE layer, forward and backward.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``): a plain, slow, obviously
correct restatement of what the layer computes, used to check the CUDA library.

What the paper fixes, and where:
  * the layer whose expert-parallel traffic Eq. 1 (Sec. 1) counts: dropless
    routing with no capacity padding, every token sent to its K routed
    experts as a hidden vector of width D (b_x bytes per element) plus one
    routed probability (b_p bytes);
  * the six transfers of one layer per microbatch (Sec. 4.1, footnote on the
    all-to-all dispatcher): hidden-state dispatch, probability dispatch and
    hidden-state combine in the forward pass, and their inverses in the
    backward pass;
  * grouped-GEMM experts and a fused permute (Sec. 5.2, experimental details);
  * the LatentMoE variant that dispatches through a lower-dimensional latent
    width (Sec. 1 levers list; Table 2, d_latent column).
The paper does not spell out the router or the expert activation.  The
readings taken here (each also listed with its reason in the design notes):
  R1  softmax over all E logits, top-K, then renormalise over the K chosen;
  R2  selection by logit value, ties to the lower expert index, slots ordered
      by descending logit then lower index;
  R4  expert-grouped row order: counting sort by expert, stable in token;
  R5  the routed probability scales the expert output in the combine;
  R6  SwiGLU expert: a = silu(x W_gate^T) * (x W_up^T), Y = a W2^T, no biases;
  R7  an optional per-expert logit bias is added after the router product
      and receives no gradient;
  R11 LatentMoE: the router reads the model-width input; the down-projection
      feeds dispatch and the up-projection follows the combine.

All arithmetic is float64 on float64 copies of the stored (bf16/fp32) inputs.
No blocking, fusion or reordering beyond the definitions below.
"""
from __future__ import annotations

import math
from typing import Optional

import numpy as np

__all__ = [
    "router_logits", "softmax_rows", "top_k_route", "expert_permutation", "dispatch",
    "silu", "sigmoid", "expert_ffn_one", "expert_ffn", "combine", "combine_bwd",
    "expert_ffn_bwd_one", "expert_ffn_bwd", "dispatch_bwd", "route_bwd",
    "layer_forward", "layer_backward", "near_tie_tokens", "latent_project",
    "latent_project_bwd",
]


# ---------------------------------------------------------------------------
# Forward
# ---------------------------------------------------------------------------

def router_logits(x: np.ndarray, w_router: np.ndarray, bias: Optional[np.ndarray] = None) -> np.ndarray:
    """z_t = x_t . W_r^T (+ b): one logit per (token, expert).  Readings R1, R7."""
    z = np.matmul(x, w_router.T)
    if bias is not None:
        z = z + bias[None, :]
    return z


def softmax_rows(z: np.ndarray) -> np.ndarray:
    """Row-wise softmax over the E experts (max-subtracted).  Reading R1."""
    m = z.max(axis=1, keepdims=True)
    e = np.exp(z - m)
    return e / e.sum(axis=1, keepdims=True)


def top_k_route(z: np.ndarray, K: int):
    """Per token: s = softmax(z_t); S_t = the K experts of largest logit
    (ties to the lower expert index), ordered by descending logit; renormalised
    p_tk = s_tk / sum_{j in S_t} s_j.  Readings R1, R2, R3 (no epsilon).

    Returns idx [T, K] int64 and prob [T, K] float64.
    """
    T, E = z.shape
    s = softmax_rows(z)
    idx = np.empty((T, K), dtype=np.int64)
    prob = np.empty((T, K), dtype=np.float64)
    for t in range(T):
        ranked = sorted(range(E), key=lambda e: (-z[t, e], e))
        chosen = ranked[:K]
        denom = sum(s[t, e] for e in chosen)
        for k, e in enumerate(chosen):
            idx[t, k] = e
            prob[t, k] = s[t, e] / denom
    return idx, prob


def expert_permutation(idx: np.ndarray, E: int):
    """Expert-grouped order of the T*K routed slots (reading R4).

    Slot s = t*K + k holds token t's k-th choice.  Rows are the slots sorted by
    (expert, token); a token picks an expert at most once, so the order is
    unique.  Returns offsets [E+1] (offsets[e] = first row of expert e,
    offsets[E] = T*K), row_of_slot [T*K] and token_of_row [T*K].
    """
    T, K = idx.shape
    TK = T * K
    flat = [int(v) for v in idx.reshape(-1)]
    order = sorted(range(TK), key=lambda s: (flat[s], s // K))
    row_of_slot = np.empty(TK, dtype=np.int64)
    token_of_row = np.empty(TK, dtype=np.int64)
    for row, s in enumerate(order):
        row_of_slot[s] = row
        token_of_row[row] = s // K
    counts = [0] * E
    for e in flat:
        counts[e] += 1
    offsets = np.zeros(E + 1, dtype=np.int64)
    for e in range(E):
        offsets[e + 1] = offsets[e] + counts[e]
    return offsets, row_of_slot, token_of_row


def dispatch(x: np.ndarray, prob: np.ndarray, row_of_slot: np.ndarray, token_of_row: np.ndarray):
    """Pack each token's K copies into the expert-grouped buffer: the hidden
    vector (first forward transfer) and the routed probability (second forward
    transfer), Sec. 4.1 footnote.  x_perm[row] = x[token_of_row[row]]."""
    TK = token_of_row.shape[0]
    x_perm = x[token_of_row]
    prob_perm = np.empty(TK, dtype=np.float64)
    flat_p = prob.reshape(-1)
    for s in range(TK):
        prob_perm[row_of_slot[s]] = flat_p[s]
    return x_perm, prob_perm


def sigmoid(v: np.ndarray) -> np.ndarray:
    return 1.0 / (1.0 + np.exp(-v))


def silu(v: np.ndarray) -> np.ndarray:
    """silu(v) = v * sigmoid(v).  Reading R6."""
    return v * sigmoid(v)


def expert_ffn_one(X_e, wg_e, wu_e, w2_e):
    """One expert's SwiGLU FFN on its rows: g = X W_g^T, u = X W_u^T,
    a = silu(g) * u, Y = a W2^T.  Reading R6; grouped-GEMM experts, Sec. 5.2."""
    g = np.matmul(X_e, wg_e.T)
    u = np.matmul(X_e, wu_e.T)
    a = silu(g) * u
    Y = np.matmul(a, w2_e.T)
    return g, u, a, Y


def expert_ffn(x_perm, offsets, w_gate, w_up, w2):
    """Every expert on its contiguous row range [offsets[e], offsets[e+1])."""
    TK = x_perm.shape[0]
    E, F, D = w_gate.shape
    g = np.zeros((TK, F))
    u = np.zeros((TK, F))
    a = np.zeros((TK, F))
    y_perm = np.zeros((TK, w2.shape[1]))
    for e in range(E):
        lo, hi = int(offsets[e]), int(offsets[e + 1])
        if hi == lo:
            continue
        g[lo:hi], u[lo:hi], a[lo:hi], y_perm[lo:hi] = expert_ffn_one(x_perm[lo:hi], w_gate[e], w_up[e], w2[e])
    return g, u, a, y_perm


def combine(y_perm, prob_perm, row_of_slot, T: int, K: int):
    """Probability-weighted combine (third forward transfer, Sec. 4.1
    footnote; reading R5): y_t = sum_k p_tk * Y_perm[row(t, k)]."""
    y = np.zeros((T, y_perm.shape[1]))
    for t in range(T):
        for k in range(K):
            r = row_of_slot[t * K + k]
            y[t] += prob_perm[r] * y_perm[r]
    return y


# ---------------------------------------------------------------------------
# Backward (exact adjoint of the forward above, routing held fixed)
# ---------------------------------------------------------------------------

def combine_bwd(dy, y_perm, prob_perm, token_of_row):
    """Inverse of the combine: dY_perm[row] = p_row * dy[t(row)] and
    dprob_perm[row] = <dy[t(row)], Y_perm[row]>."""
    TK = token_of_row.shape[0]
    dy_perm = np.empty_like(y_perm)
    dprob_perm = np.empty(TK)
    for r in range(TK):
        t = token_of_row[r]
        dy_perm[r] = prob_perm[r] * dy[t]
        dprob_perm[r] = float(np.dot(dy[t], y_perm[r]))
    return dy_perm, dprob_perm


def expert_ffn_bwd_one(dY_e, X_e, g_e, u_e, wg_e, wu_e, w2_e):
    """Adjoint of ``expert_ffn_one``.

    dA = dY W2;  dg = dA * u * sigmoid(g) * (1 + g (1 - sigmoid(g)));
    du = dA * silu(g);  dW2 = dY^T a;  dWg = dg^T X;  dWu = du^T X;
    dX = dg W_g + du W_u.
    """
    sg = sigmoid(g_e)
    a_e = g_e * sg * u_e
    dA = np.matmul(dY_e, w2_e)
    dg = dA * u_e * sg * (1.0 + g_e * (1.0 - sg))
    du = dA * (g_e * sg)
    dw2 = np.matmul(dY_e.T, a_e)
    dwg = np.matmul(dg.T, X_e)
    dwu = np.matmul(du.T, X_e)
    dX = np.matmul(dg, wg_e) + np.matmul(du, wu_e)
    return dX, dwg, dwu, dw2


def expert_ffn_bwd(dy_perm, x_perm, g, u, offsets, w_gate, w_up, w2):
    E = w_gate.shape[0]
    dx_perm = np.zeros_like(x_perm)
    dwg = np.zeros_like(w_gate)
    dwu = np.zeros_like(w_up)
    dw2 = np.zeros_like(w2)
    for e in range(E):
        lo, hi = int(offsets[e]), int(offsets[e + 1])
        if hi == lo:
            continue
        dx_perm[lo:hi], dwg[e], dwu[e], dw2[e] = expert_ffn_bwd_one(
            dy_perm[lo:hi], x_perm[lo:hi], g[lo:hi], u[lo:hi], w_gate[e], w_up[e], w2[e])
    return dx_perm, dwg, dwu, dw2


def dispatch_bwd(dx_perm, dprob_perm, row_of_slot, T: int, K: int):
    """Inverse of the dispatch: dx_t = sum_k dX_perm[row(t, k)] and
    dprob[t, k] = dprob_perm[row(t, k)]."""
    dx = np.zeros((T, dx_perm.shape[1]))
    dprob = np.empty((T, K))
    for t in range(T):
        for k in range(K):
            r = row_of_slot[t * K + k]
            dx[t] += dx_perm[r]
            dprob[t, k] = dprob_perm[r]
    return dx, dprob


def route_bwd(x, w_router, idx, prob, dprob):
    """Adjoint of the renormalised top-K softmax and of the router product.

    With p_k = exp(z_k) / sum_{j in S} exp(z_j):  dz_j = p_j (dp_j - sum_k p_k dp_k)
    for j in S, 0 for j outside S (the selection is piecewise constant).
    Then dx_router = dz W_r and dW_r = dz^T x.  The logit bias (R7) gets no
    gradient.
    """
    T, K = idx.shape
    E = w_router.shape[0]
    dz = np.zeros((T, E))
    for t in range(T):
        c = sum(prob[t, k] * dprob[t, k] for k in range(K))
        for k in range(K):
            dz[t, idx[t, k]] = prob[t, k] * (dprob[t, k] - c)
    dx_router = np.matmul(dz, w_router)
    dw_router = np.matmul(dz.T, x)
    return dz, dx_router, dw_router


# ---------------------------------------------------------------------------
# LatentMoE projections (Sec. 1 levers list, Table 2)
# ---------------------------------------------------------------------------

def latent_project(x, w):
    """out = x . w^T  (w is [out_width, in_width])."""
    return np.matmul(x, w.T)


def latent_project_bwd(dout, x, w):
    """Adjoint of ``latent_project``: dx = dout . w, dw = dout^T . x."""
    return np.matmul(dout, w), np.matmul(dout.T, x)


# ---------------------------------------------------------------------------
# Whole layer
# ---------------------------------------------------------------------------

def layer_forward(x, w_router, w_gate, w_up, w2, K: int, bias=None, w_down=None, w_upp=None,
                  idx_override=None):
    """One layer forward.  Returns a dict with every intermediate.

    ``idx_override`` replaces the oracle's own top-K choice (used where an
    fp64 near-tie could legitimately resolve either way; the probabilities are
    then the renormalised softmax over the given set, in the given order).
    """
    E = w_router.shape[0]
    T = x.shape[0]
    out = {}
    z = router_logits(x, w_router, bias)
    if idx_override is None:
        idx, prob = top_k_route(z, K)
    else:
        idx = np.asarray(idx_override, dtype=np.int64)
        prob = np.empty((T, K))
        for t in range(T):
            m = max(z[t, e] for e in idx[t])
            ws = [math.exp(z[t, e] - m) for e in idx[t]]
            tot = sum(ws)
            for k in range(K):
                prob[t, k] = ws[k] / tot
    out.update(z=z, idx=idx, prob=prob)
    x_in = x
    if w_down is not None:
        x_in = latent_project(x, w_down)
        out["x_lat"] = x_in
    offsets, row_of_slot, token_of_row = expert_permutation(idx, E)
    x_perm, prob_perm = dispatch(x_in, prob, row_of_slot, token_of_row)
    g, u, a, y_perm = expert_ffn(x_perm, offsets, w_gate, w_up, w2)
    y = combine(y_perm, prob_perm, row_of_slot, T, K)
    out.update(offsets=offsets, row_of_slot=row_of_slot, token_of_row=token_of_row,
               x_perm=x_perm, prob_perm=prob_perm, g=g, u=u, a=a, y_perm=y_perm, y=y)
    if w_upp is not None:
        out["y_lat"] = y
        out["y"] = latent_project(y, w_upp)
    return out


def layer_backward(fwd: dict, dy, x, w_router, w_gate, w_up, w2, w_down=None, w_upp=None):
    """One layer backward given the forward dict and the upstream gradient dy."""
    T, K = fwd["idx"].shape
    out = {}
    if w_upp is not None:
        dy_lat, dw_upp = latent_project_bwd(dy, fwd["y_lat"], w_upp)
        out["dw_upp"] = dw_upp
        out["dy_lat"] = dy_lat
        dy = dy_lat
    dy_perm, dprob_perm = combine_bwd(dy, fwd["y_perm"], fwd["prob_perm"], fwd["token_of_row"])
    x_perm = fwd["x_perm"]
    dx_perm, dwg, dwu, dw2 = expert_ffn_bwd(dy_perm, x_perm, fwd["g"], fwd["u"], fwd["offsets"],
                                            w_gate, w_up, w2)
    dx_experts, dprob = dispatch_bwd(dx_perm, dprob_perm, fwd["row_of_slot"], T, K)
    dz, dx_router, dw_router = route_bwd(x, w_router, fwd["idx"], fwd["prob"], dprob)
    out.update(dy_perm=dy_perm, dprob_perm=dprob_perm, dx_perm=dx_perm, dw_gate=dwg, dw_up=dwu,
               dw2=dw2, dprob=dprob, dz=dz, dw_router=dw_router)
    if w_down is not None:
        dx_lat = dx_experts
        dx_from_lat, dw_down = latent_project_bwd(dx_lat, x, w_down)
        out.update(dx_lat=dx_lat, dw_down=dw_down, dx_experts=dx_from_lat)
        out["dx"] = dx_from_lat + dx_router
    else:
        out["dx_experts"] = dx_experts
        out["dx"] = dx_experts + dx_router
    out["dx_router"] = dx_router
    return out


def near_tie_tokens(z: np.ndarray, K: int, rel: float = 1e-4) -> np.ndarray:
    """Tokens whose routing an fp32-versus-fp64 logit difference could flip:
    some gap among the K+1 largest logits is below rel * max|z_t| (reading R2)."""
    T, E = z.shape
    flagged = []
    for t in range(T):
        v = sorted(z[t], reverse=True)[: min(K + 1, E)]
        scale = rel * max(abs(float(q)) for q in z[t])
        if any(v[i] - v[i + 1] < scale for i in range(len(v) - 1)):
            flagged.append(t)
    return np.asarray(flagged, dtype=np.int64)
