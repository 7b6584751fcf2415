"""Full-size parity of the next-step rows at the base workload (T=8192, D=2048,
E=64, K=6, F=1024), in the launch configuration bench.py times for them:
the sigmoid router (``--router sigmoid``), the shared expert
(``--shared-width 2688``) and the FP8 and NVFP4 payloads (``--payload``).
Index work and payload codes on every token, statistics and router gradients
over all tokens, the shared expert and the layer output on sampled tokens, the
shared expert's whole weight gradients; tolerances as in the other parity
tests."""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.gpu_util import REL_FROB, f64, i64, rel_frob

pytestmark = pytest.mark.gpu

W = synth.get("C2")


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _w64(t):
    return t.detach().to(torch.float64).numpy()


def test_sigmoid_router_full_size():
    from paper_2608_28511_gb300.layer import MoeLayer
    inp = synth.make_inputs(W)
    inp["expert_bias"] = synth.make_expert_bias(W.E, W.seed)
    L = MoeLayer(W.S, W.GBS, W.K, W.D, W.E, W.F, W.dtype, W.H, router="sigmoid")
    L.load(inp)
    L.forward()
    L.backward()
    torch.cuda.synchronize()
    z = f64(L.logits)
    bias = inp["expert_bias"].double().numpy()
    idx = i64(L.topk_idx)
    # the selection kernel's own fp32 keys s + b: the choice is bitwise on every token
    from paper_2608_28511_gb300 import abi
    keys_t = torch.empty_like(L.logits)
    idx_t = torch.empty_like(L.topk_idx)
    abi.moe_topk_sigmoid(L.shape, L.logits, L.expert_bias, L.aux_coef, keys_t, idx_t, torch.empty_like(L.topk_prob),
                         torch.empty_like(L.aux_f), torch.empty_like(L.aux_loss), L.ws)
    torch.cuda.synchronize()
    keys = f64(keys_t)
    assert np.array_equal(i64(idx_t), idx)
    assert np.array_equal(idx, O.select_on_keys(keys, W.K))
    assert np.abs(keys - (O.sigmoid(z) + bias[None, :])).max() <= 2e-6
    _, prob_at = O.sigmoid_route(z, W.K, bias, idx_override=idx)
    assert np.abs(f64(L.topk_prob) - prob_at).max() <= 1e-5
    loss_ref, f_ref, _ = O.seq_aux_loss(z, idx, W.S, W.GBS, L.aux_coef)
    assert np.array_equal(f64(L.aux_f), f_ref.astype(np.float32).astype(np.float64))
    assert abs(float(L.aux_loss[0].item()) - loss_ref) <= 1e-4 * abs(loss_ref)
    dz_ref, _, dw_ref = O.sigmoid_route_bwd(_w64(inp["x"]), _w64(inp["w_router"]), z, idx, f64(L.topk_prob),
                                            f64(L.dprob), f64(L.aux_f), W.S, W.GBS, L.aux_coef, 1.0)
    assert rel_frob(f64(L.dlogits), dz_ref) <= 1e-4
    assert rel_frob(f64(L.dw_router), dw_ref) <= REL_FROB


def test_shared_expert_full_size():
    from paper_2608_28511_gb300.layer import MoeLayer
    Fs = 2688
    inp = synth.make_inputs(W)
    inp.update(synth.make_shared_expert(W, Fs, W.seed))
    L = MoeLayer(W.S, W.GBS, W.K, W.D, W.E, W.F, W.dtype, W.H, shared_F=Fs)
    L.load(inp)
    L.forward()
    L.backward()
    torch.cuda.synchronize()
    x, w1, w2, dy = (_w64(inp[k]) for k in ("x", "w_s1", "w_s2", "dy"))
    # sampled tokens: the shared expert's pre-activation, activation and its part of y
    rng = np.random.default_rng(7)
    toks = np.unique(np.concatenate([[0, W.T - 1], rng.choice(W.T, 48, replace=False)]))
    h_ref, a_ref, y_ref = O.shared_expert(x[toks], w1, w2)
    assert rel_frob(f64(L.h_s)[toks], h_ref) <= REL_FROB
    assert rel_frob(f64(L.act_s)[toks], a_ref) <= REL_FROB
    # whole weight gradients from the GPU's saved h and act (stage-isolated)
    dh_ref, _, dw1_ref, dw2_ref = O.shared_expert_bwd(dy, x, f64(L.h_s), f64(L.act_s), w1, w2)
    assert rel_frob(f64(L.dw_s1), dw1_ref) <= REL_FROB
    assert rel_frob(f64(L.dw_s2), dw2_ref) <= REL_FROB
    assert rel_frob(f64(L.dh_s)[toks], dh_ref[toks]) <= REL_FROB


def test_fp8_payload_full_size():
    """The FP8 dispatch payload at the base workload (``--payload fp8``): every
    token's codes and row scale at all K of its rows, bit for bit against the
    oracle's quantization of the GPU's own dispatch input; the dequantized
    rows exactly; sampled tokens' layer output within the layer tolerance,
    from the dequantized rows (readings FP1-FP3)."""
    from paper_2608_28511_gb300.layer import MoeLayer
    inp = synth.make_inputs(W)
    L = MoeLayer(W.S, W.GBS, W.K, W.D, W.E, W.F, W.dtype, W.H, payload="fp8")
    L.load(inp)
    L.forward()
    L.backward()
    torch.cuda.synchronize()
    x = _w64(inp["x"])
    codes, scales = O.fp8_quantize_rows(x)
    tor = i64(L.token_of_row)
    assert np.array_equal(L.x_perm_q.cpu().numpy(), codes[tor])
    assert np.array_equal(f64(L.x_scale_perm), scales[tor])
    assert np.array_equal(f64(L.x_perm), O.fp8_dequantize_rows(codes, scales)[tor])
    # sampled tokens' y from the dequantized rows (stage-isolated routing: the GPU's indices)
    rng = np.random.default_rng(11)
    toks = np.unique(np.concatenate([[0, W.T - 1], rng.choice(W.T, 48, replace=False)]))
    x_deq = O.fp8_dequantize_rows(codes[toks], scales[toks])
    idx = i64(L.topk_idx)[toks]
    prob = f64(L.topk_prob)[toks]
    wg, wu, w2 = (_w64(inp[k]) for k in ("w_gate", "w_up", "w2"))
    y_ref = np.zeros((len(toks), W.D))
    for i in range(len(toks)):
        for k in range(W.K):
            e = idx[i, k]
            g, u = x_deq[i] @ wg[e].T, x_deq[i] @ wu[e].T
            y_ref[i] += prob[i, k] * ((O.silu(g) * u) @ w2[e].T)
    assert rel_frob(f64(L.y)[toks], y_ref) <= REL_FROB


def test_nvfp4_payload_full_size():
    """The NVFP4 dispatch payload at the base workload (``--payload nvfp4``):
    every token's E2M1 codes, E4M3 block scales and row scale at all K of its
    rows, bit for bit against the oracle's quantization of the GPU's own
    dispatch input; the dequantized rows exactly; sampled tokens' layer output
    within the layer tolerance, from the dequantized rows (readings NV1-NV3)."""
    from paper_2608_28511_gb300.layer import MoeLayer
    inp = synth.make_inputs(W)
    L = MoeLayer(W.S, W.GBS, W.K, W.D, W.E, W.F, W.dtype, W.H, payload="nvfp4")
    L.load(inp)
    L.forward()
    L.backward()
    torch.cuda.synchronize()
    x = _w64(inp["x"])
    codes, bsc, rsc = O.nvfp4_quantize_rows(x)
    tor = i64(L.token_of_row)
    assert np.array_equal(L.x_perm_q4.cpu().numpy(), codes[tor])
    assert np.array_equal(L.x_bscale_perm.cpu().numpy(), bsc[tor])
    assert np.array_equal(f64(L.x_rscale_perm), rsc[tor])
    assert np.array_equal(f64(L.x_perm), O.nvfp4_dequantize_rows(codes, bsc, rsc)[tor])
    rng = np.random.default_rng(12)
    toks = np.unique(np.concatenate([[0, W.T - 1], rng.choice(W.T, 48, replace=False)]))
    x_deq = O.nvfp4_dequantize_rows(codes[toks], bsc[toks], rsc[toks])
    idx = i64(L.topk_idx)[toks]
    prob = f64(L.topk_prob)[toks]
    wg, wu, w2 = (_w64(inp[k]) for k in ("w_gate", "w_up", "w2"))
    y_ref = np.zeros((len(toks), W.D))
    for i in range(len(toks)):
        for k in range(W.K):
            e = idx[i, k]
            g, u = x_deq[i] @ wg[e].T, x_deq[i] @ wu[e].T
            y_ref[i] += prob[i, k] * ((O.silu(g) * u) @ w2[e].T)
    assert rel_frob(f64(L.y)[toks], y_ref) <= REL_FROB
