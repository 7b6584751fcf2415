"""Float64 reference for the sigmoid router with expert bias and the
sequence-level auxiliary load-balancing loss (Sec. 5.2, experimental details:
sigmoid router scores with expert bias, sequence-level auxiliary load
balancing with coefficient 1e-4).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

The paper names these parts without formulas.  Readings (each listed with its
reason in the design notes):
  S1  scores s = sigmoid(z) per expert; the expert bias b is added to the
      scores for choosing the K experts only (it shapes routing, not the
      gate values, and gets no gradient); ties to the lower expert index,
      slots ordered by descending s + b;
  S2  gate values p_k = s_k / sum_{j in S} s_j over the K chosen experts;
  S3  sequence-level balance loss: for each sequence g of S tokens,
      f_gi = E / (K S) * #{t in g : i chosen for t},
      P_gi = (1 / S) * sum_{t in g} s_ti / sum_j s_tj,
      L_aux = coef / GBS * sum_g sum_i f_gi P_gi;
      f is a count (no gradient); the gradient flows through P.
"""
from __future__ import annotations

import numpy as np

from .moe import sigmoid

__all__ = ["sigmoid_route", "seq_aux_loss", "sigmoid_route_bwd", "select_on_keys"]


def select_on_keys(keys: np.ndarray, K: int) -> np.ndarray:
    """Reading S1's choice on given selection keys [T, E]: per token the K
    largest keys, ties to the lower expert index, best first.  Given the fp32
    keys s + b that the GPU formed, this is the stage-isolated choice its
    indices must equal bit for bit (the keys' own rounding is then the same
    on both sides)."""
    T, E = keys.shape
    idx = np.empty((T, K), dtype=np.int64)
    for t in range(T):
        row = [float(v) for v in keys[t]]
        idx[t] = sorted(range(E), key=lambda e: (-row[e], e))[:K]
    return idx


def sigmoid_route(z: np.ndarray, K: int, expert_bias=None, idx_override=None, keys=None):
    """Readings S1, S2.  Returns idx [T, K] int64 and prob [T, K] float64.

    ``idx_override`` replaces the choice (where a near-tie of s + b could
    resolve either way); the gate values are then S2 over the given set.
    ``keys`` [T, E] chooses on those selection keys (``select_on_keys``)
    instead of the float64 s + b.
    """
    T, E = z.shape
    s = sigmoid(z)
    b = np.zeros(E) if expert_bias is None else np.asarray(expert_bias, dtype=np.float64)
    idx = np.empty((T, K), dtype=np.int64)
    prob = np.empty((T, K))
    chosen_on_keys = select_on_keys(keys, K) if keys is not None and idx_override is None else None
    for t in range(T):
        if idx_override is not None:
            chosen = [int(e) for e in idx_override[t]]
        elif chosen_on_keys is not None:
            chosen = [int(e) for e in chosen_on_keys[t]]
        else:
            key = [s[t, e] + b[e] for e in range(E)]
            chosen = sorted(range(E), key=lambda e: (-key[e], e))[:K]
        denom = sum(s[t, e] for e in chosen)
        for k, e in enumerate(chosen):
            idx[t, k] = e
            prob[t, k] = s[t, e] / denom
    return idx, prob


def seq_aux_loss(z: np.ndarray, idx: np.ndarray, S: int, GBS: int, coef: float):
    """Reading S3.  Returns (L_aux, f [GBS, E], P [GBS, E])."""
    T, E = z.shape
    K = idx.shape[1]
    s = sigmoid(z)
    f = np.zeros((GBS, E))
    P = np.zeros((GBS, E))
    for g in range(GBS):
        for t in range(g * S, (g + 1) * S):
            for k in range(K):
                f[g, idx[t, k]] += 1.0
            P[g] += s[t] / s[t].sum()
    f *= E / (K * S)
    P /= S
    loss = coef / GBS * float((f * P).sum())
    return loss, f, P


def sigmoid_route_bwd(x, w_router, z, idx, prob, dprob, f, S: int, GBS: int, coef: float, aux_grad: float = 1.0):
    """Gradient of (downstream loss through the gate values) + aux_grad * L_aux
    with respect to the logits z, then dx_router = dz W_r and dW_r = dz^T x.

    Gate path (j in S): p_k = s_k / sum_S s gives
        dL/ds_j = (dp_j - sum_k p_k dp_k) / sum_S s.
    Balance path (every j): with c_gi = aux_grad * coef / (GBS S) * f_gi and
    shat = s / sum_j s,  dL/ds_j = (c_gj - sum_i c_gi shat_i) / sum_i s_i.
    Then dz_j = s_j (1 - s_j) dL/ds_j.
    """
    T, E = z.shape
    K = idx.shape[1]
    s = sigmoid(z)
    dz = np.zeros((T, E))
    for t in range(T):
        g = t // S
        ds = np.zeros(E)
        sel = [int(e) for e in idx[t]]
        denom = sum(s[t, e] for e in sel)
        dot = sum(prob[t, k] * dprob[t, k] for k in range(K))
        for k, e in enumerate(sel):
            ds[e] += (dprob[t, k] - dot) / denom
        c = aux_grad * coef / (GBS * S) * f[g]
        tot = s[t].sum()
        shat = s[t] / tot
        ds += (c - float((c * shat).sum())) / tot
        dz[t] = s[t] * (1.0 - s[t]) * ds
    return dz, np.matmul(dz, w_router), np.matmul(dz.T, x)
