"""GPU parity of the sigmoid router (sigmoid scores, selection-only expert
bias, sequence-level balance loss; Sec. 5.2) against the float64 oracle.

Stage-isolated checks feed the oracle the GPU's own fp32 selection keys
s + b (exported by moe_topk_sigmoid from the selection kernel itself), so the
choice of experts is compared bit for bit on every token, exact ties included
(ties go to the lower expert).  From the raw inputs the oracle's float64 keys
may order two keys that lie within fp32 rounding of each other the other way;
the end-to-end test allows exactly those tokens and checks the rest bitwise.
Float results: gate values 1e-5 absolute, balance loss 1e-5 relative, logit
gradients 1e-4 relative Frobenius (fp32 arithmetic throughout), and the
router's weight and input gradients 1e-2 relative Frobenius (bf16 GEMMs).
"""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.gpu_util import LOGIT_REL, PROB_ABS, REL_FROB, f64, i64, oracle_inputs, rel_frob

pytestmark = pytest.mark.gpu

W = synth.Workload
CASES = {
    # several sequences, ragged last GEMM tile
    "sig_bf16": W("sig_bf16", S=300, GBS=3, D=256, E=16, K=4, F=256),
    # S spans several 256-token statistic chunks with a ragged tail
    "sig_chunks": W("sig_chunks", S=777, GBS=2, D=128, E=24, K=6, F=128),
    # E > 128: eight scores per lane, K = 8
    "sig_wideE": W("sig_wideE", S=256, GBS=2, D=256, E=200, K=8, F=128),
    # every token its own sequence
    "sig_S1": W("sig_S1", S=1, GBS=96, D=128, E=8, K=2, F=128),
    "sig_fp32": W("sig_fp32", S=200, GBS=2, D=192, E=12, K=3, F=192, dtype="f32"),
    "sig_latent": W("sig_latent", S=256, GBS=2, D=256, E=32, K=4, F=192, H=512),
}
COEF = 1e-4
KEY_TIE = 1e-6

_cache = {}


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    yield
    _cache.clear()


def run(name, aux_coef=COEF, aux_grad=1.0):
    key = (name, aux_coef, aux_grad)
    if key not in _cache:
        from paper_2608_28511_gb300.layer import MoeLayer
        w = CASES[name]
        inputs = synth.make_inputs(w)
        inputs["expert_bias"] = synth.make_expert_bias(w.E, w.seed)
        L = MoeLayer(w.S, w.GBS, w.K, w.D, w.E, w.F, w.dtype, w.H, router="sigmoid", aux_coef=aux_coef,
                     aux_grad=aux_grad)
        L.load(inputs)
        L.forward()
        L.backward()
        torch.cuda.synchronize()
        _cache[key] = (w, L, inputs, oracle_inputs(inputs))
    return _cache[key]


def key_tie_tokens(z, bias, K):
    """Tokens where two of the K+1 largest float64 keys s + b lie within KEY_TIE."""
    keys = O.sigmoid(z) + bias[None, :]
    top = -np.sort(-keys, axis=1)[:, : min(K + 1, keys.shape[1])]
    return set(np.nonzero((top[:, :-1] - top[:, 1:] < KEY_TIE).any(axis=1))[0].tolist())


def gpu_keys(L, logits=None, bias="layer"):
    """Re-run the selection stage on the layer's logits with the key export:
    (keys [T, E] f64, idx [T, K]) exactly as the selection kernel formed and chose them."""
    from paper_2608_28511_gb300 import abi
    logits = L.logits if logits is None else logits
    b = L.expert_bias if isinstance(bias, str) else bias
    keys = torch.empty_like(logits)
    idx = torch.empty(logits.shape[0], L.K, dtype=torch.int32, device=logits.device)
    prob = torch.empty(logits.shape[0], L.K, dtype=torch.float32, device=logits.device)
    f = torch.empty_like(L.aux_f)
    loss = torch.empty_like(L.aux_loss)
    abi.moe_topk_sigmoid(L.shape, logits, b, L.aux_coef, keys, idx, prob, f, loss, L.ws)
    torch.cuda.synchronize()
    return f64(keys), i64(idx), f64(prob), f64(f), float(loss[0].item())


def check_choice_bitwise(L, z, bias, K):
    """The layer's indices equal the oracle's choice on the kernel's own keys,
    on every token; the keys are sigmoid(z) + b within fp32 rounding."""
    keys, idx_k, _, _, _ = gpu_keys(L)
    idx = i64(L.topk_idx)
    assert np.array_equal(idx_k, idx)                     # the export does not change the choice
    assert np.array_equal(idx, O.select_on_keys(keys, K))
    assert np.abs(keys - (O.sigmoid(z) + bias[None, :])).max() <= 2e-6
    return keys


def check_choice_from_raw(idx_gpu, idx_ref, z, bias, K):
    """From float64 keys of the raw inputs: equal except where two of the K+1
    largest keys lie within fp32 rounding (KEY_TIE); there the GPU's choice
    must still be a valid top-K of the float64 keys up to that gap."""
    ties = key_tie_tokens(z, bias, K)
    keys = O.sigmoid(z) + bias[None, :]
    for t in np.nonzero((idx_gpu != idx_ref).any(axis=1))[0]:
        assert t in ties, f"token {t}: {idx_gpu[t]} != {idx_ref[t]} without a near-tie"
        assert len(set(idx_gpu[t].tolist())) == K
        ref_keys = keys[t, idx_ref[t]]
        assert np.abs(keys[t, idx_gpu[t]] - ref_keys).max() < KEY_TIE
    return ties


names = list(CASES)


@pytest.mark.parametrize("name", names)
def test_sigmoid_route_stage(name):
    w, L, inp, o = run(name)
    z_ref = O.router_logits(o["x"], o["w_router"])
    z = f64(L.logits)
    assert rel_frob(z, z_ref) <= LOGIT_REL
    bias = o["expert_bias"]
    keys = check_choice_bitwise(L, z, bias, w.K)
    idx = i64(L.topk_idx)
    idx_ref, prob_at = O.sigmoid_route(z, w.K, bias, keys=keys)
    assert np.array_equal(idx, idx_ref)
    prob = f64(L.topk_prob)
    assert np.abs(prob - prob_at).max() <= PROB_ABS
    assert np.abs(prob.sum(axis=1) - 1.0).max() <= 1e-6


@pytest.mark.parametrize("name", names)
def test_balance_loss_stage(name):
    w, L, inp, o = run(name)
    z = f64(L.logits)
    idx = i64(L.topk_idx)
    loss_ref, f_ref, P_ref = O.seq_aux_loss(z, idx, w.S, w.GBS, COEF)
    f = f64(L.aux_f)
    assert np.array_equal(f, f_ref.astype(np.float32).astype(np.float64))
    loss = float(L.aux_loss[0].item())
    assert abs(loss - loss_ref) <= 1e-5 * abs(loss_ref)
    # invariant: every sequence makes S*K choices, so sum_i f_gi = E
    assert np.allclose(f.sum(axis=1), w.E, rtol=1e-6)


@pytest.mark.parametrize("name", names)
def test_sigmoid_route_bwd_stage(name):
    w, L, inp, o = run(name)
    z = f64(L.logits)
    idx = i64(L.topk_idx)
    dz_ref, _, dw_ref = O.sigmoid_route_bwd(o["x"], o["w_router"], z, idx, f64(L.topk_prob), f64(L.dprob),
                                            f64(L.aux_f), w.S, w.GBS, COEF, 1.0)
    assert rel_frob(f64(L.dlogits), dz_ref) <= 1e-4
    assert rel_frob(f64(L.dw_router), dw_ref) <= REL_FROB


@pytest.mark.parametrize("name", ["sig_bf16", "sig_chunks", "sig_fp32"])
def test_balance_gradient_alone(name):
    """dtopk_prob = 0 and a large coefficient isolate the balance-loss gradient;
    dx starts at zero, so dx = dlogits . w_router exactly as the oracle."""
    from paper_2608_28511_gb300 import abi
    w, L, inp, o = run(name)
    dprob0 = torch.zeros_like(L.dprob)
    dx = torch.zeros_like(L.dx)
    dw = torch.empty_like(L.dw_router)
    dz = torch.empty_like(L.dlogits)
    coef, grad = 0.5, 2.0
    abi.moe_route_sigmoid_bwd(L.shape, L.x, L.w_router, L.logits, L.topk_idx, L.topk_prob, dprob0, L.aux_f, coef,
                              grad, dx, dw, dz, L.ws)
    torch.cuda.synchronize()
    z = f64(L.logits)
    idx = i64(L.topk_idx)
    dz_ref, dx_ref, dw_ref = O.sigmoid_route_bwd(o["x"], o["w_router"], z, idx, f64(L.topk_prob),
                                                 np.zeros(idx.shape), f64(L.aux_f), w.S, w.GBS, coef, grad)
    assert np.abs(dz_ref).max() > 0
    assert rel_frob(f64(dz), dz_ref) <= 1e-4
    assert rel_frob(f64(dx), dx_ref) <= REL_FROB
    assert rel_frob(f64(dw), dw_ref) <= REL_FROB


@pytest.mark.parametrize("name", ["sig_bf16", "sig_fp32", "sig_latent"])
def test_sigmoid_layer_end_to_end(name):
    """The whole layer with the sigmoid router against the oracle run from the raw inputs."""
    w, L, inp, o = run(name)
    x, wr = o["x"], o["w_router"]
    z = O.router_logits(x, wr)
    idx_ref, _ = O.sigmoid_route(z, w.K, o["expert_bias"])
    idx = i64(L.topk_idx)
    check_choice_bitwise(L, f64(L.logits), o["expert_bias"], w.K)
    check_choice_from_raw(idx, idx_ref, z, o["expert_bias"], w.K)
    idx_use, prob = O.sigmoid_route(z, w.K, o["expert_bias"], idx_override=idx)
    x_in = O.latent_project(x, o["w_down"]) if w.H else x
    off, ros, tor = O.expert_permutation(idx_use, w.E)
    x_perm, prob_perm = O.dispatch(x_in, prob, ros, tor)
    g, u, a, y_perm = O.expert_ffn(x_perm, off, o["w_gate"], o["w_up"], o["w2"])
    y = O.combine(y_perm, prob_perm, ros, w.T, w.K)
    dy = o["dy"]
    if w.H:
        y_lat = y
        y = O.latent_project(y_lat, o["w_upp"])
        dy, _ = O.latent_project_bwd(dy, y_lat, o["w_upp"])
    assert rel_frob(f64(L.y), y) <= REL_FROB
    loss_ref, f_ref, _ = O.seq_aux_loss(z, idx_use, w.S, w.GBS, COEF)
    assert abs(float(L.aux_loss[0].item()) - loss_ref) <= 1e-4 * abs(loss_ref)
    dy_perm, dprob_perm = O.combine_bwd(dy, y_perm, prob_perm, tor)
    dx_perm, dwg, dwu, dw2 = O.expert_ffn_bwd(dy_perm, x_perm, g, u, off, o["w_gate"], o["w_up"], o["w2"])
    dx_e, dprob = O.dispatch_bwd(dx_perm, dprob_perm, ros, w.T, w.K)
    if w.H:
        dx_e, _ = O.latent_project_bwd(dx_e, x, o["w_down"])
    dz, dx_r, dw_r = O.sigmoid_route_bwd(x, wr, z, idx_use, prob, dprob, f_ref, w.S, w.GBS, COEF, 1.0)
    assert rel_frob(f64(L.dprob), dprob) <= REL_FROB
    assert rel_frob(f64(L.dlogits), dz) <= REL_FROB
    assert rel_frob(f64(L.dw_router), dw_r) <= REL_FROB
    assert rel_frob(f64(L.dx), dx_e + dx_r) <= REL_FROB


def test_sigmoid_router_deterministic():
    """Two runs on the same inputs give bit-identical routing, statistics and gradients."""
    from paper_2608_28511_gb300 import abi
    w, L, inp, o = run("sig_chunks")
    outs = []
    for _ in range(2):
        abi.moe_route_sigmoid(L.shape, L.x, L.w_router, L.expert_bias, COEF, L.logits, L.topk_idx, L.topk_prob,
                              L.aux_f, L.aux_loss, L.ws)
        abi.moe_route_sigmoid_bwd(L.shape, L.x, L.w_router, L.logits, L.topk_idx, L.topk_prob, L.dprob, L.aux_f,
                                  COEF, 1.0, L.dx, L.dw_router, L.dlogits, L.ws)
        torch.cuda.synchronize()
        outs.append([t.clone() for t in (L.topk_idx, L.topk_prob, L.aux_f, L.aux_loss[:1], L.dlogits, L.dw_router)])
    for a, b in zip(*outs):
        assert torch.equal(a, b)


def test_zero_bias_equals_no_bias():
    """A NULL expert bias and an all-zero one choose identically."""
    from paper_2608_28511_gb300 import abi
    w, L, inp, o = run("sig_bf16")
    res = []
    for b in (None, torch.zeros_like(L.expert_bias)):
        idx = torch.empty_like(L.topk_idx)
        prob = torch.empty_like(L.topk_prob)
        f = torch.empty_like(L.aux_f)
        loss = torch.empty_like(L.aux_loss)
        z = torch.empty_like(L.logits)
        abi.moe_route_sigmoid(L.shape, L.x, L.w_router, b, COEF, z, idx, prob, f, loss, L.ws)
        torch.cuda.synchronize()
        res.append((idx, prob, f, loss[:1]))
    for a, b in zip(*res):
        assert torch.equal(a, b)


def test_sigmoid_status_errors():
    from paper_2608_28511_gb300 import abi
    w, L, inp, o = run("sig_bf16")
    with pytest.raises(abi.MoeError) as e:
        abi.moe_route_sigmoid(L.shape, L.x, L.w_router, L.expert_bias, COEF, L.logits, L.topk_idx, L.topk_prob,
                              L.aux_f, L.aux_loss, L.ws[:16])
    assert e.value.status == -5
    with pytest.raises(abi.MoeError) as e:
        abi.moe_route_sigmoid(L.shape, L.x, L.w_router, L.expert_bias, float("nan"), L.logits, L.topk_idx,
                              L.topk_prob, L.aux_f, L.aux_loss, L.ws)
    assert e.value.status == -1
    with pytest.raises(abi.MoeError) as e:
        abi.moe_route_sigmoid(L.shape, L.x, L.w_router, L.expert_bias, COEF, L.logits, L.topk_idx, L.topk_prob,
                              None, L.aux_loss, L.ws)
    assert e.value.status == -4


TIE_CASES = [(128, 2, 16, 4), (96, 1, 8, 2), (64, 2, 200, 8), (100, 3, 24, 16)]


@pytest.mark.parametrize("S,GBS,E,K", TIE_CASES)
def test_exact_key_ties_go_to_the_lower_expert(S, GBS, E, K):
    """Integer logits in [-2, 2] and a bias of a few equal values: most tokens
    have exactly equal keys at the K-th place.  The kernel's choice equals the
    oracle's on its exported keys and on the float64 keys (equal (z, b) pairs
    give equal keys in both precisions; distinct pairs stay far apart), and
    its gate values and balance statistics match the oracle's."""
    from paper_2608_28511_gb300 import abi
    from paper_2608_28511_gb300.layer import MoeLayer
    T = S * GBS
    g = torch.Generator().manual_seed(S + E + K)
    z = torch.randint(-2, 3, (T, E), generator=g).to(torch.float32)
    bias = (torch.randint(0, 2, (E,), generator=g).to(torch.float32) * 0.25)
    L = MoeLayer(S, GBS, K, 64, E, 64, "bf16", router="sigmoid")
    zd, bd = z.cuda(), bias.cuda()
    keys, idx, prob, f, loss = gpu_keys(L, logits=zd, bias=bd)
    zf, bf = z.double().numpy(), bias.double().numpy()
    k64 = O.sigmoid(zf) + bf[None, :]
    tied = sum(int(np.sort(k64[t])[::-1][K - 1] == np.sort(k64[t])[::-1][K]) for t in range(T)) if K < E else 0
    assert K == E or tied > T // 4                              # the case really is tie-heavy
    assert np.array_equal(idx, O.select_on_keys(keys, K))
    idx_ref, prob_ref = O.sigmoid_route(zf, K, bf)
    assert np.array_equal(idx, idx_ref)
    assert np.abs(prob - prob_ref).max() <= PROB_ABS
    loss_ref, f_ref, _ = O.seq_aux_loss(zf, idx_ref, S, GBS, L.aux_coef)
    assert np.array_equal(f, f_ref.astype(np.float32).astype(np.float64))
    assert abs(loss - loss_ref) <= 1e-5 * abs(loss_ref)
    # the selection stage alone equals the full router on the same logits
    idx2 = torch.empty(T, K, dtype=torch.int32, device="cuda")
    prob2 = torch.empty(T, K, dtype=torch.float32, device="cuda")
    abi.moe_topk_sigmoid(L.shape, zd, bd, L.aux_coef, None, idx2, prob2, L.aux_f, L.aux_loss, L.ws)
    torch.cuda.synchronize()
    assert np.array_equal(i64(idx2), idx)
    assert np.array_equal(f64(prob2), prob)
