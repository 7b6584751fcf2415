"""Helpers shared by the GPU parity tests."""
from __future__ import annotations

import numpy as np
import torch

import oracle as O
import synth

# Tolerances of the layer (float outputs and gradients: relative Frobenius
# error against the float64 oracle; routed probabilities: absolute error).
REL_FROB = 1e-2
PROB_ABS = 1e-5
LOGIT_REL = 1e-5


def rel_frob(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    den = np.linalg.norm(b)
    if den == 0.0:
        return float(np.linalg.norm(a))
    return float(np.linalg.norm(a - b) / den)


def f64(t) -> np.ndarray:
    return t.detach().float().cpu().double().numpy() if t.dtype == torch.bfloat16 else \
        t.detach().cpu().double().numpy()


def i64(t) -> np.ndarray:
    return t.detach().cpu().numpy().astype(np.int64)


def make_layer(w: synth.Workload, T: int | None = None, seed: int | None = None, inputs: dict | None = None,
               gather: bool = False):
    """Build a MoeLayer for workload ``w`` (token count T), load seeded inputs, run forward+backward."""
    from paper_2608_28511_gb300.layer import MoeLayer
    T = w.T if T is None else T
    if inputs is None:
        inputs = synth.make_inputs(w, seed=seed, T=T)
    layer = MoeLayer(T, 1, w.K, w.D, w.E, w.F, w.dtype, w.H, gather=gather)
    layer.load(inputs)
    layer.forward()
    layer.backward()
    torch.cuda.synchronize()
    return layer, inputs


def oracle_inputs(inputs: dict) -> dict:
    return {k: synth.to_f64(v) for k, v in inputs.items()}


def rel_frob_blocks(a, b, rows: int = 128) -> float:
    """Largest relative Frobenius error over blocks of ``rows`` consecutive
    entries of the leading axis (128 tokens or rows, or one expert with
    rows = 1 on an [E, ...] weight gradient).  A block whose reference is
    exactly zero counts as exact only if the result is zero there too."""
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    assert a.shape == b.shape, (a.shape, b.shape)
    worst = 0.0
    for i in range(0, b.shape[0], rows):
        den = np.linalg.norm(b[i:i + rows])
        num = np.linalg.norm(a[i:i + rows] - b[i:i + rows])
        err = (0.0 if num == 0.0 else float("inf")) if den == 0.0 else float(num / den)
        worst = max(worst, err)
    return worst


def assert_close(a, b, rows: int = 128, tol: float = REL_FROB, what: str = "") -> None:
    """The layer's float tolerance on the whole tensor and on every block of
    ``rows`` leading-axis entries, so that an error confined to one tile, one
    expert or a few tokens cannot hide under the whole tensor's norm."""
    whole = rel_frob(a, b)
    local = rel_frob_blocks(a, b, rows)
    assert whole <= tol and local <= tol, f"{what}: relative Frobenius {whole:.3g} whole, {local:.3g} worst block"
