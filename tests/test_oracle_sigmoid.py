"""Pins for the sigmoid-router oracle (scores, expert-bias selection, gate
values, sequence-level balance loss and their gradient) against brute force,
closed forms, an independent vectorised restatement and finite differences."""
import itertools

import numpy as np
import pytest
import scipy.special

import oracle as O


def _rng(s):
    return np.random.default_rng(s)


def _winners(key, K):
    E = len(key)
    out = []
    for S in itertools.combinations(range(E), K):
        rest = [j for j in range(E) if j not in S]
        if all(key[i] > key[j] or (key[i] == key[j] and i < j) for i in S for j in rest):
            out.append(set(S))
    assert len(out) == 1
    return out[0]


@pytest.mark.parametrize("E,K", [(6, 2), (8, 3), (5, 5), (7, 1)])
def test_selection_uses_score_plus_bias_and_gates_use_scores(E, K):
    r = _rng(E + K)
    z = r.normal(size=(30, E)) * 2
    b = r.normal(size=E) * 0.3
    idx, prob = O.sigmoid_route(z, K, b)
    s = scipy.special.expit(z)                      # library sigmoid
    for t in range(30):
        assert set(idx[t].tolist()) == _winners(s[t] + b, K)
        key = s[t, idx[t]] + b[idx[t]]
        assert all(key[k] > key[k + 1] or (key[k] == key[k + 1] and idx[t, k] < idx[t, k + 1]) for k in range(K - 1))
        assert abs(prob[t].sum() - 1) < 1e-12
        np.testing.assert_allclose(prob[t] / prob[t][0], s[t, idx[t]] / s[t, idx[t][0]], rtol=1e-12)


def test_zero_bias_selects_like_the_logits():
    z = _rng(3).normal(size=(50, 9))
    idx_sig, _ = O.sigmoid_route(z, 3, None)
    idx_soft, _ = O.top_k_route(z, 3)               # sigmoid is monotone: same choice as by logit
    assert (idx_sig == idx_soft).all()


def test_large_bias_forces_the_choice():
    z = _rng(4).normal(size=(20, 6))
    b = np.array([0, 0, 0, 0, 5.0, 5.0])
    idx, _ = O.sigmoid_route(z, 2, b)
    assert (np.sort(idx, axis=1) == [4, 5]).all()


def test_balanced_routing_with_flat_scores_gives_the_coefficient():
    # every expert chosen by exactly K S / E tokens and equal scores: f = 1, P = 1/E, L = coef
    E, K, S, GBS, coef = 4, 2, 8, 3, 1e-4
    z = np.zeros((S * GBS, E))
    idx = np.array([[(2 * t) % E, (2 * t + 1) % E] for t in range(S * GBS)])
    loss, f, P = O.seq_aux_loss(z, idx, S, GBS, coef)
    np.testing.assert_allclose(f, 1.0, rtol=0, atol=1e-15)
    np.testing.assert_allclose(P, 1.0 / E, rtol=0, atol=1e-15)
    assert loss == pytest.approx(coef, rel=1e-14)


def test_balance_loss_matches_a_vectorised_restatement():
    E, K, S, GBS, coef = 7, 3, 11, 4, 1e-4
    r = _rng(9)
    z = r.normal(size=(S * GBS, E))
    idx, _ = O.sigmoid_route(z, K, r.normal(size=E) * 0.2)
    loss, f, P = O.seq_aux_loss(z, idx, S, GBS, coef)
    s = scipy.special.expit(z)
    shat = s / s.sum(axis=1, keepdims=True)
    for g in range(GBS):
        cnt = np.bincount(idx[g * S:(g + 1) * S].ravel(), minlength=E)
        np.testing.assert_allclose(f[g], cnt * E / (K * S), rtol=1e-14)
        np.testing.assert_allclose(P[g], shat[g * S:(g + 1) * S].mean(axis=0), rtol=1e-13)
    assert loss == pytest.approx(coef * np.mean([(f[g] * P[g]).sum() for g in range(GBS)]), rel=1e-13)


def _objective(z, idx, dprob, S, GBS, coef, aux_grad, f):
    """Downstream loss through the gate values of the fixed choice, plus aux_grad * L_aux."""
    s = scipy.special.expit(z)
    sel = np.take_along_axis(s, idx, axis=1)
    p = sel / sel.sum(axis=1, keepdims=True)
    shat = s / s.sum(axis=1, keepdims=True)
    P = shat.reshape(GBS, S, -1).mean(axis=1)
    return float((p * dprob).sum()) + aux_grad * coef / GBS * float((f * P).sum())


def test_router_gradient_matches_central_differences():
    E, K, S, GBS, D = 6, 2, 5, 2, 4
    r = _rng(21)
    x = r.normal(size=(S * GBS, D))
    w = r.normal(size=(E, D))
    z = x @ w.T
    idx, prob = O.sigmoid_route(z, K, r.normal(size=E) * 0.1)
    dprob = r.normal(size=(S * GBS, K))
    coef, aux_grad = 0.3, 0.7              # large so the balance path is visible in the check
    _, f, _ = O.seq_aux_loss(z, idx, S, GBS, coef)
    dz, dxr, dwr = O.sigmoid_route_bwd(x, w, z, idx, prob, dprob, f, S, GBS, coef, aux_grad)
    h = 1e-6
    for i in range(z.shape[0]):
        for j in range(E):
            zp, zm = z.copy(), z.copy()
            zp[i, j] += h
            zm[i, j] -= h
            fd = (_objective(zp, idx, dprob, S, GBS, coef, aux_grad, f)
                  - _objective(zm, idx, dprob, S, GBS, coef, aux_grad, f)) / (2 * h)
            assert abs(fd - dz[i, j]) <= 1e-7 * max(1.0, abs(fd)), (i, j, fd, dz[i, j])
    np.testing.assert_allclose(dxr, dz @ w, rtol=1e-13)
    np.testing.assert_allclose(dwr, dz.T @ x, rtol=1e-13)


@pytest.mark.parametrize("E,K", [(6, 2), (8, 3), (5, 5), (9, 4)])
def test_selection_on_given_keys_against_brute_force_with_exact_ties(E, K):
    """select_on_keys: the unique K-set that beats every other expert (larger
    key, or an equal key and a lower index), ordered best first; integer keys
    with many exact ties exercise the tie rule."""
    keys = _rng(40 + E).integers(-2, 3, size=(60, E)).astype(np.float32)
    idx = O.select_on_keys(keys, K)
    for t in range(60):
        assert set(idx[t].tolist()) == _winners(keys[t].astype(np.float64), K)
        k = keys[t, idx[t]]
        assert all(k[j] > k[j + 1] or (k[j] == k[j + 1] and idx[t, j] < idx[t, j + 1]) for j in range(K - 1))


def test_selection_on_keys_matches_the_float64_route_when_keys_are_its_own():
    r = _rng(41)
    z = r.normal(size=(40, 10)) * 2
    b = r.normal(size=10) * 0.2
    keys = scipy.special.expit(z) + b[None, :]
    idx_keys, prob_keys = O.sigmoid_route(z, 3, b, keys=keys)
    idx, prob = O.sigmoid_route(z, 3, b)
    assert (idx_keys == idx).all()
    np.testing.assert_array_equal(prob_keys, prob)


def test_gates_on_key_choice_use_scores_not_keys():
    # equal keys from different (score, bias) pairs: the choice is by key, the gates by score
    z = np.array([[0.0, np.log(3.0), 0.0]])         # s = 0.5, 0.75, 0.5
    b = np.array([0.25, 0.0, -0.5])                 # keys 0.75, 0.75, 0.0
    keys = scipy.special.expit(z) + b[None, :]
    idx, prob = O.sigmoid_route(z, 2, b, keys=keys)
    assert idx.tolist() == [[0, 1]]                 # tie at 0.75 -> lower expert first
    np.testing.assert_allclose(prob[0], [0.5 / 1.25, 0.75 / 1.25], rtol=1e-15)
