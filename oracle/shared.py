"""Float64 reference for the shared expert of the MoE layer (Sec. 5.2,
experimental details: each MoE layer has, in parallel with the routed experts,
an ungated shared expert MLP whose output is added to the combined routed
output).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

The paper names the part without formulas.  Readings (each listed with its
reason in the design notes):
  SH1  ungated two-layer MLP with squared-ReLU activation and no biases:
       h = x W_s1^T  [T, F_s],  a = relu(h)^2,  y_shared = a W_s2^T  [T, Din],
       with W_s1 [F_s, Din] and W_s2 [Din, F_s];
  SH2  it reads the layer input x (the model width H for LatentMoE) and its
       output is added to the layer output y (after the LatentMoE
       up-projection), so dx receives its input gradient too.
"""
from __future__ import annotations

import numpy as np

__all__ = ["relu_sq", "shared_expert", "shared_expert_bwd"]


def relu_sq(v: np.ndarray) -> np.ndarray:
    r = np.maximum(v, 0.0)
    return r * r


def shared_expert(x: np.ndarray, w_s1: np.ndarray, w_s2: np.ndarray):
    """Reading SH1.  Returns (h, a, y_shared)."""
    h = np.matmul(x, w_s1.T)
    a = relu_sq(h)
    return h, a, np.matmul(a, w_s2.T)


def shared_expert_bwd(dy: np.ndarray, x: np.ndarray, h: np.ndarray, a: np.ndarray, w_s1: np.ndarray,
                      w_s2: np.ndarray):
    """Backward of ``shared_expert`` for the upstream gradient dy [T, Din].

    dA = dy W_s2;  d relu(h)^2 / dh = 2 relu(h), so dh = 2 relu(h) dA;
    dW_s2 = dy^T a;  dW_s1 = dh^T x;  dx = dh W_s1.
    Returns (dh, dx, dw_s1, dw_s2).
    """
    dA = np.matmul(dy, w_s2)
    dh = 2.0 * np.maximum(h, 0.0) * dA
    return dh, np.matmul(dh, w_s1), np.matmul(dh.T, x), np.matmul(dy.T, a)
