"""Eq. 1 (Sec. 1): expert-parallel volume of one training step.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

V_step is proportional to L_E * S * GBS * K * (4 D b_x + 2 b_p).  Reading R12:
the proportionality constant is taken as 1 byte per logical element, so the
value is the logical payload of the six per-layer transfers of Sec. 4.1's
footnote (hidden dispatch, probability dispatch, hidden combine and their
three inverses), summed over L_E routed layers.
"""
from __future__ import annotations

__all__ = ["eq1_bytes", "six_transfer_bytes"]


def eq1_bytes(S: int, GBS: int, K: int, D: int, b_x: int, b_p: int = 4, L_E: int = 1) -> int:
    """L_E * S * GBS * K * (4 * D * b_x + 2 * b_p), Eq. 1."""
    return L_E * S * GBS * K * (4 * D * b_x + 2 * b_p)


def six_transfer_bytes(T: int, K: int, D: int, b_x: int, b_p: int = 4) -> dict:
    """Byte size of each of the six logical transfers of one layer (Sec. 4.1
    footnote), as buffers of the expert-grouped layout: T*K rows each."""
    TK = T * K
    return {
        "x_perm": TK * D * b_x,        # forward hidden-state dispatch
        "prob_perm": TK * b_p,         # forward routed-probability dispatch
        "y_perm": TK * D * b_x,        # forward hidden-state combine
        "dy_perm": TK * D * b_x,       # backward inverse of the combine
        "dx_perm": TK * D * b_x,       # backward inverse of the hidden dispatch
        "dprob_perm": TK * b_p,        # backward inverse of the probability dispatch
    }
