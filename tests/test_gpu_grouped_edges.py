"""The expert FFN's grouped GEMMs on expert row counts at every edge of the
engine's 256-row tiles: an empty expert, 1, 31, 32, 33, 100, 224, 225, 255,
256, 257, 480 and 513 rows.  Each output is compared per expert with the
float64 oracle's expert FFN (``expert_ffn_one`` / ``expert_ffn_bwd_one``) on
the same bf16 inputs, widened exactly:
  * GEMM-1 + SwiGLU (h and a);
  * GEMM-2 (y, from the GPU's own a);
  * the backward GEMMs (dA through the SwiGLU backward, dX, both weight
    gradients, from the GPU's own h).
One case has full-width column tiles (2F, D and F multiples of 256), the
other ragged ones (2F = 640, F = 320)."""
import itertools

import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_28511_gb300 import abi
from tests.gpu_util import REL_FROB, f64, rel_frob

pytestmark = pytest.mark.gpu

# rows per expert: empty, within one tile, exactly one tile, one tile plus 1, 224 or 257 rows
COUNTS = [0, 1, 31, 32, 33, 100, 224, 225, 255, 256, 257, 480, 513]
CASES = {"full": (512, 256), "ragged": (256, 320)}  # (D, F)


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _run(D, F, seed):
    E, TK = len(COUNTS), sum(COUNTS)
    dev = "cuda"
    g = torch.Generator().manual_seed(seed)
    bf = torch.bfloat16
    rnd = lambda *s, sc=1.0: (torch.randn(*s, generator=g) * sc).to(bf)  # noqa: E731
    shp = abi.MoeShape.of(TK, 1, 1, D, E, F, "bf16")
    off = torch.tensor([0] + list(itertools.accumulate(COUNTS)), dtype=torch.int32, device=dev)
    host = dict(x=rnd(TK, D), wg=rnd(E, F, D, sc=D ** -0.5), wu=rnd(E, F, D, sc=D ** -0.5),
                w2=rnd(E, D, F, sc=F ** -0.5), dy=rnd(TK, D))
    x, wg, wu, w2, dy = (host[k].to(dev) for k in ("x", "wg", "wu", "w2", "dy"))
    w1 = torch.empty(E, 2 * F, D, dtype=bf, device=dev)
    abi.moe_pack_w1(shp, wg, wu, w1)
    e = lambda *s, d=bf: torch.empty(*s, dtype=d, device=dev)  # noqa: E731
    h, act, y = e(TK, 2 * F), e(TK, F), e(TK, D)
    dx, dw1, dw2 = e(TK, D), e(E, 2 * F, D, d=torch.float32), e(E, D, F, d=torch.float32)
    ws = torch.empty(abi.moe_workspace_size(shp), dtype=torch.uint8, device=dev)
    abi.moe_expert_ffn(shp, x, off, w1, w2, h, act, y, ws)
    abi.moe_expert_ffn_bwd(shp, dy, x, h, act, off, w1, w2, dx, dw1, dw2, ws)
    torch.cuda.synchronize()
    assert abi.moe_check_device_status() == 0
    o = {k: v.to(torch.float64).numpy() for k, v in host.items()}
    return dict(off=off.tolist(), o=o, h=f64(h), act=f64(act), y=f64(y), dx=f64(dx), dw1=f64(dw1), dw2=f64(dw2),
                E=E, F=F)


def _halves(t, F):
    """[rows, 2F] packed [gate 64 | up 64] blocks -> gate, up [rows, F]."""
    v = t.reshape(t.shape[0], F // 64, 2, 64)
    return v[:, :, 0].reshape(t.shape[0], F), v[:, :, 1].reshape(t.shape[0], F)


@pytest.mark.parametrize("case", list(CASES))
def test_grouped_gemm_row_edges(case):
    D, F = CASES[case]
    r = _run(D, F, seed=11 if case == "full" else 12)
    off, E, o = r["off"], r["E"], r["o"]
    v = r["dw1"].reshape(E, F // 64, 2, 64, D)  # packed [gate 64 | up 64] rows
    gw1, uw1 = v[:, :, 0].reshape(E, F, D), v[:, :, 1].reshape(E, F, D)
    for ex in range(E):
        lo, hi = off[ex], off[ex + 1]
        if hi == lo:
            # an expert without rows: exactly zero weight gradients
            assert not r["dw1"][ex].any() and not r["dw2"][ex].any()
            continue
        X = o["x"][lo:hi]
        g_ref, u_ref, a_ref, y_ref = O.expert_ffn_one(X, o["wg"][ex], o["wu"][ex], o["w2"][ex])
        g_gpu, u_gpu = _halves(r["h"][lo:hi], F)
        assert rel_frob(g_gpu, g_ref) < 5e-3, (case, ex, "gate")
        assert rel_frob(u_gpu, u_ref) < 5e-3, (case, ex, "up")
        assert rel_frob(r["act"][lo:hi], a_ref) < 5e-3, (case, ex, "a")
        # GEMM-2 alone, from the GPU's own a
        assert rel_frob(r["y"][lo:hi], np.matmul(r["act"][lo:hi], o["w2"][ex].T)) < 5e-3, (case, ex, "y")
        assert rel_frob(r["y"][lo:hi], y_ref) < REL_FROB, (case, ex, "y end to end")
        # backward from the GPU's own h (the oracle's adjoint of the expert)
        dX, dwg, dwu, dw2 = O.expert_ffn_bwd_one(o["dy"][lo:hi], X, g_gpu, u_gpu, o["wg"][ex], o["wu"][ex],
                                                 o["w2"][ex])
        assert rel_frob(r["dx"][lo:hi], dX) < REL_FROB, (case, ex, "dx")
        assert rel_frob(r["dw2"][ex], dw2) < REL_FROB, (case, ex, "dw2")
        assert rel_frob(gw1[ex], dwg) < REL_FROB, (case, ex, "dw_gate")
        assert rel_frob(uw1[ex], dwu) < REL_FROB, (case, ex, "dw_up")
