"""Seeded synthetic inputs for the dropless routed MoE layer.

This module is shared by the float64 oracle (``oracle/``), the tests and the
benchmark.  It holds workload shapes and random draws only: none of the
layer's arithmetic (routing, permutation, expert FFN, combine) lives here.

Shapes follow the symbols of the paper's Eq. 1 (Sec. 1): S sequence length,
GBS global batch size, K routed top-K, D dispatch hidden width, plus the
number of experts E and the expert SwiGLU width F.  The LatentMoE workload
adds the model hidden width H, projected down to D before dispatch (Sec. 1
levers list, Table 2 d_latent column).

Draw order and scales (one ``torch.Generator`` per workload, seeded):
  x, W_r, W_gate, W_up, W2, [W_down, W_up_proj], dy
each drawn as float32 N(0, 1) times its standard deviation (1 for x and dy,
1/sqrt(fan_in) for every weight), then cast to the workload's storage dtype
(bfloat16, or float32 for the tiny all-fp32 workload).

Public layouts (row-major):
  x       [T, D]        (LatentMoE: x is [T, H])
  w_router[E, D]        logits z = x . w_router^T   (LatentMoE: [E, H])
  w_gate  [E, F, D]     gate projection of each expert
  w_up    [E, F, D]     up projection of each expert
  w2      [E, D, F]     down projection of each expert, Y = a . w2_e^T
  w_down  [D, H]        LatentMoE down-projection, x_lat = x . w_down^T
  w_upp   [H, D]        LatentMoE up-projection,   out = y_lat . w_upp^T
  bias    [E] float32   per-expert logit bias (skewed workload only)
  expert_bias [E] float32  selection-only bias of the sigmoid router
                        (``make_expert_bias``, drawn separately)
  w_s1 [F_s, D], w_s2 [D, F_s]  shared expert (``make_shared_expert``, drawn
                        separately; LatentMoE: H in place of D)
  dy      [T, D]        upstream gradient (LatentMoE: [T, H])
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    S: int
    GBS: int
    D: int
    E: int
    K: int
    F: int
    dtype: str = "bf16"          # storage dtype of activations/weights: "bf16" or "f32"
    H: int = 0                   # model hidden width for LatentMoE (0 = no projection)
    skew_bias: bool = False      # add b_e = 3*ln(1/(e+1)) to the router logits
    seed: int = 0

    @property
    def T(self) -> int:
        return self.S * self.GBS

    @property
    def TK(self) -> int:
        return self.T * self.K

    @property
    def b_x(self) -> int:
        return 2 if self.dtype == "bf16" else 4

    @property
    def in_width(self) -> int:
        """Width of the layer input x (H for LatentMoE, else D)."""
        return self.H if self.H else self.D

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workloads of the layer benchmark (tiny all-fp32, baseline-style,
# CE-MoE-style wider experts, LatentMoE dispatch, skewed routing).
TINY = Workload("tiny_fp32_T256_D128_E8_K2_F256", S=128, GBS=2, D=128, E=8, K=2, F=256, dtype="f32")
BASE = Workload("base_T8192_D2048_E64_K6_F1024", S=4096, GBS=2, D=2048, E=64, K=6, F=1024)
CEMOE = Workload("cemoe_T16384_D2048_E128_K8_F1536", S=4096, GBS=4, D=2048, E=128, K=8, F=1536)
LATENT = Workload("latent_T16384_H4096_D1024_E256_K8_F768", S=4096, GBS=4, D=1024, E=256, K=8, F=768, H=4096)
SKEW = Workload("skew_T32768_D2048_E128_K8_F1024", S=8192, GBS=4, D=2048, E=128, K=8, F=1024, skew_bias=True)

# The base workload's shape with half the tokens and half the experts (the same
# ~768 rows per expert): a case for detailed profiler captures, which replay
# each kernel many times and save and restore device memory around them.
BASE_HALF = Workload("base_half_T4096_D2048_E32_K6_F1024", S=2048, GBS=2, D=2048, E=32, K=6, F=1024)
# The skewed workload with half the tokens and half the experts (the same
# logit-bias formula, so a similar head of near-capped experts and a tail of
# empty ones): about 4 GB on the device, for detailed profiler captures.
SKEW_HALF = Workload("skew_half_T16384_D2048_E64_K8_F1024", S=4096, GBS=4, D=2048, E=64, K=8, F=1024,
                     skew_bias=True)

# LatentMoE with half the tokens and half the experts (the same ~512 rows per
# expert): about 2.5 GB on the device, for detailed profiler captures.
LATENT_HALF = Workload("latent_half_T8192_H4096_D1024_E128_K8_F768", S=4096, GBS=2, D=1024, E=128, K=8, F=768,
                       H=4096)

WORKLOADS = {w.name: w for w in (TINY, BASE, CEMOE, LATENT, SKEW, BASE_HALF, SKEW_HALF, LATENT_HALF)}
ALIASES = {"C1": TINY, "C2": BASE, "C3": CEMOE, "C4": LATENT, "C5": SKEW, "C2h": BASE_HALF, "C5h": SKEW_HALF,
           "C4h": LATENT_HALF}


def get(name: str) -> Workload:
    if name in ALIASES:
        return ALIASES[name]
    return WORKLOADS[name]


def skew_bias_values(E: int) -> torch.Tensor:
    """Per-expert logit bias of the skewed workload: b_e = 3 * ln(1/(e+1)), e 0-based, in float32."""
    return torch.tensor([3.0 * math.log(1.0 / (e + 1)) for e in range(E)], dtype=torch.float32)


def make_expert_bias(E: int, seed: int, std: float = 0.05) -> torch.Tensor:
    """Expert bias [E] float32 for the sigmoid router, N(0, std) from its own
    generator (seed + 7919), so it leaves the ``make_inputs`` stream alone."""
    g = torch.Generator().manual_seed(int(seed) + 7919)
    return torch.randn(E, generator=g, dtype=torch.float32) * std


def make_shared_expert(w: Workload, F_s: int, seed: int) -> dict:
    """Shared-expert weights w_s1 [F_s, Din] and w_s2 [Din, F_s] in the storage
    dtype, N(0, 1/fan_in) from their own generator (seed + 104729)."""
    g = torch.Generator().manual_seed(int(seed) + 104729)
    X = w.in_width
    st = _storage(w.dtype)
    w1 = (torch.randn(F_s, X, generator=g, dtype=torch.float32) / math.sqrt(X)).to(st)
    w2 = (torch.randn(X, F_s, generator=g, dtype=torch.float32) / math.sqrt(F_s)).to(st)
    return {"w_s1": w1, "w_s2": w2}


def _storage(dtype: str) -> torch.dtype:
    return torch.bfloat16 if dtype == "bf16" else torch.float32


def make_inputs(w: Workload, seed: Optional[int] = None, T: Optional[int] = None) -> dict:
    """Draw every input of one layer step on the CPU, seeded.

    Returns a dict of CPU tensors in the storage dtype (see the module doc for
    layouts).  ``T`` overrides the token count (the token draws then use the
    same generator stream, so a smaller T is NOT a prefix of a larger one).
    """
    seed = w.seed if seed is None else seed
    T = w.T if T is None else T
    g = torch.Generator().manual_seed(seed)
    st = _storage(w.dtype)
    X = w.in_width

    def draw(shape, std):
        return (torch.randn(*shape, generator=g, dtype=torch.float32) * std).to(st)

    out = {}
    out["x"] = draw((T, X), 1.0)
    out["w_router"] = draw((w.E, X), 1.0 / math.sqrt(X))
    out["w_gate"] = draw((w.E, w.F, w.D), 1.0 / math.sqrt(w.D))
    out["w_up"] = draw((w.E, w.F, w.D), 1.0 / math.sqrt(w.D))
    out["w2"] = draw((w.E, w.D, w.F), 1.0 / math.sqrt(w.F))
    if w.H:
        out["w_down"] = draw((w.D, w.H), 1.0 / math.sqrt(w.H))
        out["w_upp"] = draw((w.H, w.D), 1.0 / math.sqrt(w.D))
    out["dy"] = draw((T, X), 1.0)
    out["bias"] = skew_bias_values(w.E) if w.skew_bias else None
    return out


def to_f64(t: Optional[torch.Tensor]):
    """Exact widening of a bf16/fp32 CPU tensor to a float64 numpy array."""
    if t is None:
        return None
    return t.detach().to("cpu").to(torch.float64).numpy()
