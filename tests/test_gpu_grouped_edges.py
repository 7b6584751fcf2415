"""The expert FFN's grouped GEMMs on expert row counts at every edge of the
engine's 256-row tiles: an empty expert, 1, 31, 32, 33, 100, 224, 225, 255,
256, 257, 480 and 513 rows.  Each output is compared per expert with plain
PyTorch fp32 on the same bf16 inputs:
  * GEMM-1 + SwiGLU (h and a);
  * GEMM-2 (y, from the GPU's own a);
  * the backward GEMMs (dA through the SwiGLU backward, dX, both weight
    gradients, from the GPU's own h and a).
One case has full-width column tiles (2F, D and F multiples of 256), the
other ragged ones (2F = 640, F = 320)."""
import itertools

import pytest
import torch

from paper_2608_28511_gb300 import abi

pytestmark = pytest.mark.gpu

# rows per expert: empty, within one tile, exactly one tile, one tile plus 1, 224 or 257 rows
COUNTS = [0, 1, 31, 32, 33, 100, 224, 225, 255, 256, 257, 480, 513]
CASES = {"full": (512, 256), "ragged": (256, 320)}  # (D, F)


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _rel(a, b):
    a, b = a.double(), b.double()
    return float((a - b).norm() / b.norm().clamp_min(1e-30))


def _run(D, F, seed):
    E, TK = len(COUNTS), sum(COUNTS)
    dev = "cuda"
    g = torch.Generator(device=dev).manual_seed(seed)
    bf = torch.bfloat16
    rnd = lambda *s, sc=1.0: (torch.randn(*s, device=dev, generator=g) * sc).to(bf)  # noqa: E731
    shp = abi.MoeShape.of(TK, 1, 1, D, E, F, "bf16")
    off = torch.tensor([0] + list(itertools.accumulate(COUNTS)), dtype=torch.int32, device=dev)
    x = rnd(TK, D)
    wg, wu = rnd(E, F, D, sc=D ** -0.5), rnd(E, F, D, sc=D ** -0.5)
    w2 = rnd(E, D, F, sc=F ** -0.5)
    dy = rnd(TK, D)
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
    return dict(off=off.tolist(), x=x, wg=wg, wu=wu, w2=w2, dy=dy, h=h, act=act, y=y, dx=dx, dw1=dw1, dw2=dw2,
                E=E, F=F)


def _halves(t, F):
    """[rows, 2F] packed [gate 64 | up 64] blocks -> gate, up [rows, F]."""
    v = t.reshape(t.shape[0], F // 64, 2, 64)
    return v[:, :, 0].reshape(t.shape[0], F), v[:, :, 1].reshape(t.shape[0], F)


@pytest.mark.parametrize("case", list(CASES))
def test_grouped_gemm_row_edges(case):
    D, F = CASES[case]
    r = _run(D, F, seed=11 if case == "full" else 12)
    off, E = r["off"], r["E"]
    v = r["dw1"].reshape(E, F // 64, 2, 64, D)  # packed [gate 64 | up 64] rows
    gw1, uw1 = v[:, :, 0].reshape(E, F, D), v[:, :, 1].reshape(E, F, D)
    for ex in range(E):
        lo, hi = off[ex], off[ex + 1]
        if hi == lo:
            # an expert without rows: zero weight gradients
            assert torch.count_nonzero(r["dw1"][ex]) == 0 and torch.count_nonzero(r["dw2"][ex]) == 0
            continue
        X = r["x"][lo:hi].float()
        Wg, Wu, W2 = r["wg"][ex].float(), r["wu"][ex].float(), r["w2"][ex].float()
        g_ref, u_ref = X @ Wg.T, X @ Wu.T
        g_gpu, u_gpu = _halves(r["h"][lo:hi], F)
        assert _rel(g_gpu, g_ref) < 5e-3, (case, ex, "gate")
        assert _rel(u_gpu, u_ref) < 5e-3, (case, ex, "up")
        a_ref = torch.nn.functional.silu(g_gpu.float()) * u_gpu.float()
        assert _rel(r["act"][lo:hi], a_ref) < 5e-3, (case, ex, "a")
        A = r["act"][lo:hi].float()
        assert _rel(r["y"][lo:hi], A @ W2.T) < 5e-3, (case, ex, "y")
        # backward from the GPU's own h and a
        dY = r["dy"][lo:hi].float()
        dA = dY @ W2
        gs, us = g_gpu.float(), u_gpu.float()
        sg = torch.sigmoid(gs)
        dg = dA * us * sg * (1 + gs * (1 - sg))
        du = dA * gs * sg
        assert _rel(r["dx"][lo:hi], dg @ Wg + du @ Wu) < 1e-2, (case, ex, "dx")
        assert _rel(r["dw2"][ex], dY.T @ A) < 1e-2, (case, ex, "dw2")
        assert _rel(gw1[ex], dg.T @ X) < 1e-2, (case, ex, "dw_gate")
        assert _rel(uw1[ex], du.T @ X) < 1e-2, (case, ex, "dw_up")
