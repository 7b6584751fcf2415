"""Pins for the shared-expert oracle (ungated squared-ReLU MLP, reading SH1)
against brute force, invariants of the activation, torch autograd and finite
differences."""
import numpy as np
import pytest
import torch

import oracle as O


def _rng(s):
    return np.random.default_rng(s)


def _params(T=7, Din=6, Fs=5, seed=0):
    r = _rng(seed)
    return r.normal(size=(T, Din)), r.normal(size=(Fs, Din)) / 2, r.normal(size=(Din, Fs)) / 2, r.normal(size=(T, Din))


def test_forward_is_a_sum_of_squared_positive_projections():
    # brute force: y[t, d] = sum over f with w1_f . x_t > 0 of (w1_f . x_t)^2 w2[d, f]
    x, w1, w2, _ = _params(seed=1)
    h, a, y = O.shared_expert(x, w1, w2)
    for t in range(x.shape[0]):
        for d in range(w2.shape[0]):
            acc = 0.0
            for f in range(w1.shape[0]):
                proj = sum(w1[f, i] * x[t, i] for i in range(x.shape[1]))
                if proj > 0:
                    acc += proj * proj * w2[d, f]
            assert y[t, d] == pytest.approx(acc, rel=1e-12, abs=1e-12)


def test_degree_two_homogeneity_and_sign_gate():
    x, w1, w2, _ = _params(seed=2)
    _, _, y = O.shared_expert(x, w1, w2)
    for c in (0.5, 3.0):
        np.testing.assert_allclose(O.shared_expert(c * x, w1, w2)[2], c * c * y, rtol=1e-12, atol=1e-12)
    # every pre-activation negative: no output, no gradient
    w1n = -np.abs(w1)
    xp = np.abs(x)
    h, a, y0 = O.shared_expert(xp, w1n, w2)
    assert np.all(y0 == 0)
    dh, dx, dw1, dw2 = O.shared_expert_bwd(np.ones_like(y0), xp, h, a, w1n, w2)
    assert np.all(dx == 0) and np.all(dw1 == 0) and np.all(dw2 == 0)


def test_backward_matches_torch_autograd():
    x, w1, w2, dy = _params(T=9, Din=8, Fs=6, seed=3)
    h, a, y = O.shared_expert(x, w1, w2)
    dh, dx, dw1, dw2 = O.shared_expert_bwd(dy, x, h, a, w1, w2)
    tx, t1, t2 = (torch.tensor(v, requires_grad=True) for v in (x, w1, w2))
    ty = torch.relu(tx @ t1.T).pow(2) @ t2.T
    ty.backward(torch.tensor(dy))
    np.testing.assert_allclose(y, ty.detach().numpy(), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dx, tx.grad.numpy(), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dw1, t1.grad.numpy(), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dw2, t2.grad.numpy(), rtol=1e-12, atol=1e-12)


def test_backward_matches_central_differences():
    x, w1, w2, dy = _params(T=4, Din=5, Fs=3, seed=4)
    h, a, _ = O.shared_expert(x, w1, w2)
    _, dx, dw1, dw2 = O.shared_expert_bwd(dy, x, h, a, w1, w2)

    def loss(x_, w1_, w2_):
        return float((O.shared_expert(x_, w1_, w2_)[2] * dy).sum())

    eps = 1e-6
    for arr, grad, which in ((x, dx, 0), (w1, dw1, 1), (w2, dw2, 2)):
        for i in np.ndindex(arr.shape):
            args_p = [x.copy(), w1.copy(), w2.copy()]
            args_m = [x.copy(), w1.copy(), w2.copy()]
            args_p[which][i] += eps
            args_m[which][i] -= eps
            fd = (loss(*args_p) - loss(*args_m)) / (2 * eps)
            assert abs(fd - grad[i]) <= 1e-6 * max(1.0, abs(fd)), (which, i, fd, grad[i])
