"""Pins for the float64 oracle against facts that do not come from the oracle.

Each test checks the oracle against brute force, a library routine, a closed
form, an invariant of the method, or finite differences, so that a dropped
term, a wrong sign or index, or a transposed operand fails at least one of
them (``test_oracle_mutations.py`` plants such mistakes to show it).
"""
import itertools
import os

import numpy as np
import pytest
import scipy.special
import torch

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rng(seed=0):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------------------
# Routing: top-K selection and renormalised probabilities
# ---------------------------------------------------------------------------

def _brute_force_topk_set(z_row, K):
    """The unique K-subset S such that every chosen expert beats every other
    one (larger logit, or equal logit and lower index)."""
    E = len(z_row)
    winners = []
    for S in itertools.combinations(range(E), K):
        rest = [j for j in range(E) if j not in S]
        if all(z_row[i] > z_row[j] or (z_row[i] == z_row[j] and i < j) for i in S for j in rest):
            winners.append(set(S))
    assert len(winners) == 1
    return winners[0]


@pytest.mark.parametrize("E,K", [(4, 2), (6, 3), (8, 2), (5, 5), (7, 1)])
def test_topk_matches_brute_force_random(E, K):
    z = _rng(E * 10 + K).normal(size=(40, E))
    idx, prob = O.top_k_route(z, K)
    for t in range(z.shape[0]):
        assert set(idx[t].tolist()) == _brute_force_topk_set(z[t], K)
        # slots ordered by descending logit, equal logits by lower index
        for k in range(K - 1):
            a, b = idx[t, k], idx[t, k + 1]
            assert z[t, a] > z[t, b] or (z[t, a] == z[t, b] and a < b)
        # renormalised probabilities = softmax restricted to the chosen set (I3)
        ref = scipy.special.softmax(z[t, idx[t]])
        np.testing.assert_allclose(prob[t], ref, rtol=1e-13, atol=0)
        assert abs(prob[t].sum() - 1.0) < 1e-12


def test_topk_ties_go_to_lower_index():
    # integer logits with many exact ties
    z = _rng(3).integers(-2, 3, size=(200, 6)).astype(np.float64)
    idx, prob = O.top_k_route(z, 3)
    for t in range(z.shape[0]):
        assert set(idx[t].tolist()) == _brute_force_topk_set(z[t], 3)
    # all-equal logits: experts 0..K-1 in order, uniform probabilities
    idx, prob = O.top_k_route(np.zeros((3, 8)), 4)
    assert (idx == np.arange(4)).all()
    np.testing.assert_allclose(prob, 0.25, rtol=0, atol=1e-15)


def test_topk_probabilities_closed_form():
    # logits ln 1, ln 2, ln 3, ln 4 with K = 2 choose experts 3, 2 with p = 4/7, 3/7
    z = np.log(np.array([[1.0, 2.0, 3.0, 4.0]]))
    idx, prob = O.top_k_route(z, 2)
    assert idx.tolist() == [[3, 2]]
    np.testing.assert_allclose(prob[0], [4 / 7, 3 / 7], rtol=1e-14)
    # softmax over all experts vs the library routine
    zz = _rng(1).normal(size=(10, 9))
    np.testing.assert_allclose(O.softmax_rows(zz), scipy.special.softmax(zz, axis=1), rtol=1e-13)


def test_router_logits_bias_and_library_matmul():
    r = _rng(5)
    x, w, b = r.normal(size=(7, 5)), r.normal(size=(3, 5)), r.normal(size=3)
    ref = torch.nn.functional.linear(torch.from_numpy(x), torch.from_numpy(w), torch.from_numpy(b)).numpy()
    np.testing.assert_allclose(O.router_logits(x, w, b), ref, rtol=1e-13, atol=1e-13)


# ---------------------------------------------------------------------------
# Permutation (I1, I2, I4) against a library stable sort
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("T,E,K", [(1, 4, 2), (3, 3, 3), (50, 8, 2), (127, 16, 4), (64, 5, 1)])
def test_permutation_vs_stable_argsort(T, E, K):
    z = _rng(T + E + K).normal(size=(T, E))
    idx, _ = O.top_k_route(z, K)
    offsets, row_of_slot, token_of_row = O.expert_permutation(idx, E)
    order = np.argsort(idx.reshape(-1), kind="stable")          # library stable sort
    assert (token_of_row == order // K).all()
    assert (row_of_slot[order] == np.arange(T * K)).all()
    # I1: row_of_slot is a bijection and every token appears exactly K times
    assert sorted(row_of_slot.tolist()) == list(range(T * K))
    assert (np.bincount(token_of_row, minlength=T) == K).all()
    # I2: offsets start at 0, are monotone, end at T*K and match the histogram
    assert offsets[0] == 0 and offsets[-1] == T * K and (np.diff(offsets) >= 0).all()
    assert (np.diff(offsets) == np.bincount(idx.reshape(-1), minlength=E)).all()
    # I4: tokens strictly increase inside each expert's range
    for e in range(E):
        seg = token_of_row[offsets[e]:offsets[e + 1]]
        assert (np.diff(seg) > 0).all()
        assert (idx.reshape(-1)[order[offsets[e]:offsets[e + 1]]] == e).all()


def test_permutation_all_tokens_one_expert_and_empty_experts():
    T, E, K = 9, 6, 1
    idx = np.full((T, K), 4)
    offsets, row_of_slot, token_of_row = O.expert_permutation(idx, E)
    assert offsets.tolist() == [0, 0, 0, 0, 0, 9, 9]
    assert token_of_row.tolist() == list(range(9))


# ---------------------------------------------------------------------------
# Expert FFN, dispatch and combine: special cases with independent answers
# ---------------------------------------------------------------------------

def _dense_swiglu_torch(x, wg, wu, w2):
    """Textbook dense SwiGLU FFN built from torch library ops (float64)."""
    tx, tg, tu, t2 = (torch.from_numpy(a) for a in (x, wg, wu, w2))
    return (torch.nn.functional.silu(tx @ tg.T) * (tx @ tu.T)) @ t2.T


def _small_layer(T=12, D=8, E=4, K=2, F=6, seed=0):
    r = _rng(seed)
    return dict(x=r.normal(size=(T, D)), w_router=r.normal(size=(E, D)) / np.sqrt(D),
                w_gate=r.normal(size=(E, F, D)) / np.sqrt(D), w_up=r.normal(size=(E, F, D)) / np.sqrt(D),
                w2=r.normal(size=(E, D, F)) / np.sqrt(F), dy=r.normal(size=(T, D)))


def test_single_expert_is_dense_swiglu():
    # I9: K = E = 1 reduces to a dense SwiGLU FFN
    p = _small_layer(E=1, K=1)
    fwd = O.layer_forward(p["x"], p["w_router"], p["w_gate"], p["w_up"], p["w2"], K=1)
    ref = _dense_swiglu_torch(p["x"], p["w_gate"][0], p["w_up"][0], p["w2"][0]).numpy()
    np.testing.assert_allclose(fwd["y"], ref, rtol=1e-12, atol=1e-12)
    assert np.allclose(fwd["prob"], 1.0)


def test_single_expert_backward_matches_autograd():
    # the dense special case's gradients from torch autograd
    p = _small_layer(E=1, K=1, seed=4)
    fwd = O.layer_forward(p["x"], p["w_router"], p["w_gate"], p["w_up"], p["w2"], K=1)
    bwd = O.layer_backward(fwd, p["dy"], p["x"], p["w_router"], p["w_gate"], p["w_up"], p["w2"])
    tx, tg, tu, t2 = (torch.from_numpy(p[k][0] if k != "x" else p[k]).clone().requires_grad_(True)
                      for k in ("x", "w_gate", "w_up", "w2"))
    y = (torch.nn.functional.silu(tx @ tg.T) * (tx @ tu.T)) @ t2.T
    (y * torch.from_numpy(p["dy"])).sum().backward()
    np.testing.assert_allclose(bwd["dx_experts"], tx.grad.numpy(), rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(bwd["dw_gate"][0], tg.grad.numpy(), rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(bwd["dw_up"][0], tu.grad.numpy(), rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(bwd["dw2"][0], t2.grad.numpy(), rtol=1e-11, atol=1e-12)
    # one expert, probability 1: no router gradient (I5 with |S| = E = 1)
    assert np.abs(bwd["dz"]).max() == 0.0


def test_identical_experts_give_dense_ffn_for_any_routing():
    # I8: renormalised probabilities sum to 1, so identical experts give FFN(x)
    p = _small_layer(E=5, K=3, seed=2)
    for k in ("w_gate", "w_up", "w2"):
        p[k][:] = p[k][0]
    fwd = O.layer_forward(p["x"], p["w_router"], p["w_gate"], p["w_up"], p["w2"], K=3)
    ref = _dense_swiglu_torch(p["x"], p["w_gate"][0], p["w_up"][0], p["w2"][0]).numpy()
    np.testing.assert_allclose(fwd["y"], ref, rtol=1e-12, atol=1e-12)


def test_combine_of_dispatch_with_identity_experts_returns_x():
    # I6
    p = _small_layer(T=20, E=6, K=3, seed=3)
    z = O.router_logits(p["x"], p["w_router"])
    idx, prob = O.top_k_route(z, 3)
    off, ros, tor = O.expert_permutation(idx, 6)
    x_perm, prob_perm = O.dispatch(p["x"], prob, ros, tor)
    y = O.combine(x_perm, prob_perm, ros, 20, 3)
    np.testing.assert_allclose(y, p["x"], rtol=1e-13, atol=1e-13)


def test_expert_ffn_per_expert_matches_library_matmul():
    p = _small_layer(T=30, E=4, K=2, seed=7)
    fwd = O.layer_forward(p["x"], p["w_router"], p["w_gate"], p["w_up"], p["w2"], K=2)
    for e in range(4):
        lo, hi = fwd["offsets"][e], fwd["offsets"][e + 1]
        ref = _dense_swiglu_torch(p["x"][fwd["token_of_row"][lo:hi]], p["w_gate"][e], p["w_up"][e], p["w2"][e])
        np.testing.assert_allclose(fwd["y_perm"][lo:hi], ref.numpy(), rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------------------
# Backward: finite differences of the forward, adjoint identities, I5
# ---------------------------------------------------------------------------

def _loss(p, K, bias=None, latent=None):
    kw = {}
    if latent is not None:
        kw = dict(w_down=latent[0], w_upp=latent[1])
    fwd = O.layer_forward(p["x"], p["w_router"], p["w_gate"], p["w_up"], p["w2"], K=K, bias=bias, **kw)
    return float((fwd["y"] * p["dy"]).sum()), fwd


@pytest.mark.parametrize("use_bias", [False, True])
def test_backward_matches_central_differences(use_bias):
    K = 2
    p = _small_layer(T=6, D=5, E=4, K=K, F=3, seed=11)
    bias = _rng(12).normal(size=4) if use_bias else None
    _, fwd = _loss(p, K, bias)
    bwd = O.layer_backward(fwd, p["dy"], p["x"], p["w_router"], p["w_gate"], p["w_up"], p["w2"])
    grads = dict(x=bwd["dx"], w_router=bwd["dw_router"], w_gate=bwd["dw_gate"], w_up=bwd["dw_up"], w2=bwd["dw2"])
    h = 1e-6
    for name, g in grads.items():
        it = np.nditer(p[name], flags=["multi_index"])
        for _ in it:
            i = it.multi_index
            old = p[name][i]
            p[name][i] = old + h
            lp, fp = _loss(p, K, bias)
            p[name][i] = old - h
            lm, fm = _loss(p, K, bias)
            p[name][i] = old
            if not ((fp["idx"] == fwd["idx"]).all() and (fm["idx"] == fwd["idx"]).all()):
                continue            # the perturbation crossed a routing boundary
            fd = (lp - lm) / (2 * h)
            assert abs(fd - g[i]) <= 1e-6 * max(1.0, abs(fd)), (name, i, fd, g[i])


def test_latent_backward_matches_central_differences():
    K, H = 2, 7
    p = _small_layer(T=5, D=4, E=3, K=K, F=3, seed=21)
    r = _rng(22)
    x_h = r.normal(size=(5, H))
    p["x"] = x_h
    p["w_router"] = r.normal(size=(3, H)) / np.sqrt(H)
    p["w_down"] = r.normal(size=(4, H)) / np.sqrt(H)
    p["w_upp"] = r.normal(size=(H, 4)) / 2.0
    p["dy"] = r.normal(size=(5, H))
    lat = (p["w_down"], p["w_upp"])
    _, fwd = _loss(p, K, None, lat)
    bwd = O.layer_backward(fwd, p["dy"], p["x"], p["w_router"], p["w_gate"], p["w_up"], p["w2"],
                           w_down=p["w_down"], w_upp=p["w_upp"])
    grads = dict(x=bwd["dx"], w_router=bwd["dw_router"], w_down=bwd["dw_down"], w_upp=bwd["dw_upp"],
                 w2=bwd["dw2"], w_gate=bwd["dw_gate"])
    h = 1e-6
    for name, g in grads.items():
        it = np.nditer(p[name], flags=["multi_index"])
        for _ in it:
            i = it.multi_index
            old = p[name][i]
            p[name][i] = old + h
            lp, fp = _loss(p, K, None, lat)
            p[name][i] = old - h
            lm, fm = _loss(p, K, None, lat)
            p[name][i] = old
            if not ((fp["idx"] == fwd["idx"]).all() and (fm["idx"] == fwd["idx"]).all()):
                continue
            fd = (lp - lm) / (2 * h)
            assert abs(fd - g[i]) <= 1e-6 * max(1.0, abs(fd)), (name, i, fd, g[i])


def test_router_gradient_invariants():
    # I5: dz rows sum to zero and vanish outside the chosen set
    p = _small_layer(T=25, E=7, K=3, seed=13)
    fwd = O.layer_forward(p["x"], p["w_router"], p["w_gate"], p["w_up"], p["w2"], K=3)
    bwd = O.layer_backward(fwd, p["dy"], p["x"], p["w_router"], p["w_gate"], p["w_up"], p["w2"])
    dz = bwd["dz"]
    np.testing.assert_allclose(dz.sum(axis=1), 0.0, atol=1e-12)
    for t in range(25):
        outside = [e for e in range(7) if e not in fwd["idx"][t]]
        assert (dz[t, outside] == 0).all()


def test_adjoint_identities_of_the_permute_family():
    T, E, K, D = 15, 5, 2, 6
    r = _rng(17)
    z = r.normal(size=(T, E))
    idx, prob = O.top_k_route(z, K)
    off, ros, tor = O.expert_permutation(idx, E)
    x = r.normal(size=(T, D))
    v = r.normal(size=(T * K, D))
    # dispatch (x -> x_perm) and the hidden part of dispatch_bwd are adjoint
    x_perm, _ = O.dispatch(x, prob, ros, tor)
    dx, _ = O.dispatch_bwd(v, np.zeros(T * K), ros, T, K)
    assert abs((x_perm * v).sum() - (x * dx).sum()) < 1e-10
    # combine is linear in Y_perm; its adjoint is the hidden part of combine_bwd
    _, prob_perm = O.dispatch(x, prob, ros, tor)
    dy = r.normal(size=(T, D))
    y = O.combine(v, prob_perm, ros, T, K)
    dy_perm, dprob_perm = O.combine_bwd(dy, v, prob_perm, tor)
    assert abs((y * dy).sum() - (v * dy_perm).sum()) < 1e-10
    # combine is also linear in prob_perm; its adjoint is dprob_perm
    assert abs((y * dy).sum() - (prob_perm * dprob_perm).sum()) < 1e-10
    # the probability dispatch and the probability part of dispatch_bwd are adjoint
    w = r.normal(size=T * K)
    _, dprob = O.dispatch_bwd(np.zeros((T * K, D)), w, ros, T, K)
    assert abs((prob_perm * w).sum() - (prob * dprob).sum()) < 1e-12


# ---------------------------------------------------------------------------
# Eq. 1 and the paper's worked numbers
# ---------------------------------------------------------------------------

def _golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                k, v = line.split()
                vals[k] = float(v)
    return vals


def test_eq1_reproduces_the_papers_worked_ratios():
    g = _golden("eq1_paper_examples.txt")
    S, GBS, K, D = 8192, 768, 6, 2688
    base = O.eq1_bytes(S, GBS, K, D, 2, 4, L_E=int(g["routed_layers_baseline"]))
    sw = O.eq1_bytes(S, GBS, K, D, 2, 4, L_E=int(g["routed_layers_switch"]))
    ce = O.eq1_bytes(S, GBS, K, D, 2, 4, L_E=int(g["routed_layers_cemoe"]))
    # all-to-all call counts scale with L_E at fixed K (Sec. 4.1)
    assert round(100 * (1 - sw / base), 1) == g["calls_reduction_switch_pct"]
    assert round(100 * (1 - ce / base), 1) == g["calls_reduction_cemoe_pct"]
    # volume with 1.5 K for the reduced variants (K_base = 8, so 1.5 K = 12
    # stays an integer)
    kf = g["volume_k_factor"]
    sw15 = O.eq1_bytes(S, GBS, 4 * 3, D, 2, 4, L_E=int(g["routed_layers_switch"]))
    ce15 = O.eq1_bytes(S, GBS, 4 * 3, D, 2, 4, L_E=int(g["routed_layers_cemoe"]))
    base8 = O.eq1_bytes(S, GBS, 8, D, 2, 4, L_E=int(g["routed_layers_baseline"]))
    assert 12 / 8 == kf
    assert round(100 * (1 - sw15 / base8), 1) == g["volume_reduction_switch_pct"]
    assert round(100 * (1 - ce15 / base8), 1) == g["volume_reduction_cemoe_pct"]
    # L_E K proxy (Sec. 4.3)
    lek0 = g["lek_baseline_LE"] * g["lek_baseline_K"]
    lek1 = g["lek_cemoe_LE"] * g["lek_cemoe_K"]
    assert lek0 == 138 and round(100 * (1 - lek1 / lek0), 1) == g["lek_reduction_pct"]
    # q = 6 transfers per layer: 23 layers -> 138 all-to-all calls
    assert g["q_per_layer"] * g["routed_layers_baseline"] == 138


@pytest.mark.parametrize("T,K,D,b_x", [(256, 2, 128, 4), (8192, 6, 2048, 2), (16384, 8, 1024, 2)])
def test_six_transfers_sum_to_eq1(T, K, D, b_x):
    # I7: the payload of the six logical transfers equals Eq. 1's per-layer term
    parts = O.six_transfer_bytes(T, K, D, b_x)
    assert len(parts) == 6
    assert sum(parts.values()) == O.eq1_bytes(T, 1, K, D, b_x, 4, L_E=1)
    # forward dispatch payload: hidden + probability per routed copy
    assert parts["x_perm"] + parts["prob_perm"] == T * K * (D * b_x + 4)


def test_eq1_bytes_published_values_for_the_workloads():
    # the per-layer Eq. 1 term of each workload, by hand: T K (4 D b_x + 2 b_p)
    assert O.eq1_bytes(128, 2, 2, 128, 4) == 256 * 2 * (4 * 128 * 4 + 8) == 1052672
    assert O.eq1_bytes(4096, 2, 6, 2048, 2) == 805699584
    assert O.eq1_bytes(4096, 4, 8, 2048, 2) == 2148532224
    assert O.eq1_bytes(4096, 4, 8, 1024, 2) == 1074790400
    assert O.eq1_bytes(8192, 4, 8, 2048, 2) == 4297064448


def test_near_tie_flags():
    z = np.array([[3.0, 1.0, 1.0 + 1e-9, 0.0], [4.0, 3.0, 2.0, 1.0]])
    flagged = O.near_tie_tokens(z, K=2)
    assert flagged.tolist() == [0]
