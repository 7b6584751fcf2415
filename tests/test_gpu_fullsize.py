"""Parity at the full benchmark sizes, in the launch configuration bench.py
times (one MoeLayer step).

Index work is checked on every token (stage-isolated: the oracle routes the
GPU's own fp32 logits and sorts the GPU's own indices).  Float outputs are
checked on samples the float64 oracle can compute one by one: sampled
tokens' y and dx (their forward and backward only touch their own K experts),
whole weight gradients of sampled experts (their forward and backward only
touch their own rows), and the router / projection weight gradients from the
GPU's upstream stage outputs.
"""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.gpu_util import LOGIT_REL, PROB_ABS, REL_FROB, assert_close, f64, i64, make_layer, rel_frob

pytestmark = pytest.mark.gpu

FULL = ["C2", "C3", "C4", "C5"]


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _w64(t):
    return t.detach().to(torch.float64).numpy()


@pytest.mark.parametrize("cfg", FULL)
def test_full_size_parity(cfg):
    w = synth.get(cfg)
    L, inp = make_layer(w)
    T, K, E = w.T, w.K, w.E
    rng = np.random.default_rng(123)
    x64 = lambda rows: _w64(inp["x"][rows])  # noqa: E731
    wr = _w64(inp["w_router"])
    bias = synth.to_f64(inp["bias"])

    # ---- routing: logits on sampled rows, top-K on every token (stage-isolated)
    rows = np.unique(np.concatenate([[0, T - 1], rng.choice(T, 256, replace=False)]))
    z_gpu = f64(L.logits)
    z_ref = O.router_logits(x64(rows), wr, bias)
    assert rel_frob(z_gpu[rows], z_ref) <= LOGIT_REL
    idx_gpu = i64(L.topk_idx)
    idx_ref, prob_ref = O.top_k_route(z_gpu, K)
    assert (idx_gpu == idx_ref).all()
    assert np.abs(f64(L.topk_prob) - prob_ref).max() <= PROB_ABS
    # routing from the fp64 logits agrees except at near-ties
    idx_own, _ = O.top_k_route(z_ref, K)
    ties = set(rows[O.near_tie_tokens(z_ref, K)].tolist())
    differ = set(rows[np.nonzero((idx_own != idx_gpu[rows]).any(axis=1))[0]].tolist())
    assert differ <= ties

    # ---- permutation: bit-exact on every slot; dispatch is an exact copy
    off, ros, tor = O.expert_permutation(idx_gpu, E)
    assert (i64(L.expert_offsets) == off).all()
    assert (i64(L.row_of_slot) == ros).all()
    assert (i64(L.token_of_row) == tor).all()
    x_disp = L.x_lat if w.H else L.x
    assert torch.equal(L.x_perm, x_disp[L.token_of_row.long()])

    # ---- sampled tokens: the first and the last 128 tokens and 64 random ones
    # in between; y and dx checked token by token, dprob per block.  The
    # oracle takes them expert by expert (rows are independent), so each
    # expert's weights are widened once.
    prob_gpu = f64(L.topk_prob)
    toks = np.concatenate([np.arange(0, 128), np.arange(T - 128, T),
                           np.sort(rng.choice(np.arange(128, T - 128), 64, replace=False))])
    n = len(toks)
    w_down = _w64(inp["w_down"]) if w.H else None
    w_upp = _w64(inp["w_upp"]) if w.H else None
    dy_all = inp["dy"]
    xt = x64(toks)
    xd = O.latent_project(xt, w_down) if w.H else xt
    dyt = _w64(dy_all[toks])
    dyd = O.latent_project_bwd(dyt, np.zeros((n, w.D)), w_upp)[0] if w.H else dyt
    idx_s, prob_s = idx_gpu[toks], prob_gpu[toks]
    Yk = np.zeros((n, K, w.D))
    dXk = np.zeros((n, K, w.D))
    dp = np.zeros((n, K))
    for e in np.unique(idx_s):
        i, k = np.nonzero(idx_s == e)
        wg, wu, w2 = _w64(inp["w_gate"][e]), _w64(inp["w_up"][e]), _w64(inp["w2"][e])
        g, u, a, Y = O.expert_ffn_one(xd[i], wg, wu, w2)
        dX, _, _, _ = O.expert_ffn_bwd_one(prob_s[i, k][:, None] * dyd[i], xd[i], g, u, wg, wu, w2)
        Yk[i, k], dXk[i, k], dp[i, k] = Y, dX, (dyd[i] * Y).sum(axis=1)
    y_ref = (prob_s[:, :, None] * Yk).sum(axis=1)
    if w.H:
        y_ref = O.latent_project(y_ref, w_upp)
    _, dx_r, _ = O.route_bwd(xt, wr, idx_s, prob_s, dp)
    dx_e = dXk.sum(axis=1)
    if w.H:
        dx_e = O.latent_project_bwd(dx_e, np.zeros((n, w.H)), w_down)[0]
    assert_close(f64(L.y)[toks], y_ref, rows=1, what="y per token")
    assert_close(f64(L.dx)[toks], dx_e + dx_r, rows=1, what="dx per token")
    assert_close(f64(L.dprob)[toks], dp, rows=128, what="dprob per block")

    # ---- sampled experts: whole weight gradients (largest, median, smallest non-empty; empty ones are zero)
    cnt = np.diff(off)
    nz = np.nonzero(cnt)[0]
    order = nz[np.argsort(cnt[nz], kind="stable")]
    for e in sorted({int(order[-1]), int(order[len(order) // 2]), int(order[0])}):
        lo, hi = int(off[e]), int(off[e + 1])
        tk = tor[lo:hi]
        pe = f64(L.prob_perm[lo:hi])[:, None]
        X_e = x64(tk)
        dY_e = _w64(dy_all[tk])
        if w.H:
            X_e = O.latent_project(X_e, w_down)
            dY_e = O.latent_project_bwd(dY_e, np.zeros((len(tk), w.D)), w_upp)[0]
        wg, wu, w2 = _w64(inp["w_gate"][e]), _w64(inp["w_up"][e]), _w64(inp["w2"][e])
        g, u, a, Y = O.expert_ffn_one(X_e, wg, wu, w2)
        _, dwg, dwu, dw2 = O.expert_ffn_bwd_one(pe * dY_e, X_e, g, u, wg, wu, w2)
        v = L.dw1[e].view(w.F // 64, 2, 64, w.D)
        gg, gu = v[:, 0].reshape(w.F, w.D), v[:, 1].reshape(w.F, w.D)
        assert_close(f64(gg), dwg, what=f"dW_gate of expert {e}")
        assert_close(f64(gu), dwu, what=f"dW_up of expert {e}")
        assert_close(f64(L.dw2[e]), dw2, what=f"dW2 of expert {e}")
    for e in np.nonzero(cnt == 0)[0][:4]:
        assert float(L.dw1[e].abs().max()) == 0.0 and float(L.dw2[e].abs().max()) == 0.0

    # ---- router gradients over all tokens from the GPU's dprob (stage-isolated)
    dz, _, dw_r = O.route_bwd(_w64(inp["x"]), wr, idx_gpu, prob_gpu, f64(L.dprob))
    assert_close(f64(L.dlogits), dz, what="dlogits")
    assert_close(f64(L.dw_router), dw_r, rows=1, what="dW_router per expert")

    # ---- LatentMoE projection weight gradients from the GPU's stage inputs
    if w.H:
        _, dwu_ref = O.latent_project_bwd(_w64(dy_all), f64(L.y_lat), w_upp)
        assert_close(f64(L.dw_upp), dwu_ref, what="dW_up_proj")
        _, dwd_ref = O.latent_project_bwd(f64(L.dx_lat), _w64(inp["x"]), w_down)
        assert_close(f64(L.dw_down), dwd_ref, what="dW_down")

    # ---- Eq. 1 payload of this workload's six transfers (I7)
    six = (L.x_perm.numel() + L.y_perm.numel() + L.dy_perm.numel() + L.dx_perm.numel()) * L.x_perm.element_size() \
        + (L.prob_perm.numel() + L.dprob_perm.numel()) * 4
    assert six == O.eq1_bytes(w.S, w.GBS, K, w.D, w.b_x, 4)


def test_full_size_graph_and_host_pipeline_match_eager_bitwise():
    """At the base workload, the two launch forms bench.py times reproduce the
    eager step bit for bit: the step replayed as one CUDA graph, and
    MoeLayer.run_host (host batches, copies overlapped with compute, one graph
    per buffer set)."""
    w = synth.get("C2")
    L, inp = make_layer(w)
    names = ("topk_idx", "row_of_slot", "x_perm", "h", "y", "dx_perm", "dw1", "dw2", "dx", "dw_router")
    eager = {n: getattr(L, n).clone() for n in names}
    g = L.capture()
    for n in names:
        getattr(L, n).zero_()
    g.replay()
    torch.cuda.synchronize()
    for n in names:
        assert torch.equal(getattr(L, n), eager[n]), n
    x_h = inp["x"].pin_memory()
    dy_h = inp["dy"].pin_memory()
    y_h = torch.empty_like(x_h).pin_memory()
    dx_h = torch.empty_like(x_h).pin_memory()
    L.prepare_host_pipeline(graphs=True)
    L.run_host([(x_h, dy_h, y_h, dx_h)] * 3)
    torch.cuda.synchronize()
    assert torch.equal(y_h, eager["y"].cpu())
    assert torch.equal(dx_h, eager["dx"].cpu())
