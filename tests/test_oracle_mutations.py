"""Plant plausible mistakes in the oracle (on the CPU) and check that the pins
in ``test_oracle_pins.py`` catch each one."""
import numpy as np
import pytest

import oracle
import oracle.moe as M
import tests.test_oracle_pins as P


def _patch(monkeypatch, name, fn):
    """Replace an oracle function both in its module and in the package namespace."""
    monkeypatch.setattr(M, name, fn)
    monkeypatch.setattr(oracle, name, fn)


def _expect_failure(fn, *args):
    with pytest.raises(AssertionError):
        fn(*args)


def test_dropped_term_in_swiglu_backward_is_caught(monkeypatch):
    def bad(dY_e, X_e, g_e, u_e, wg_e, wu_e, w2_e):
        sg = M.sigmoid(g_e)
        a_e = g_e * sg * u_e
        dA = np.matmul(dY_e, w2_e)
        dg = dA * u_e * sg * (g_e * (1.0 - sg))          # "1 +" dropped
        du = dA * (g_e * sg)
        return (np.matmul(dg, wg_e) + np.matmul(du, wu_e), np.matmul(dg.T, X_e),
                np.matmul(du.T, X_e), np.matmul(dY_e.T, a_e))
    _patch(monkeypatch, "expert_ffn_bwd_one", bad)
    _expect_failure(P.test_backward_matches_central_differences, False)
    _expect_failure(P.test_single_expert_backward_matches_autograd)


def test_wrong_sign_in_router_backward_is_caught(monkeypatch):
    orig = M.route_bwd

    def bad(x, w_router, idx, prob, dprob):
        dz, dxr, dwr = orig(x, w_router, idx, prob, dprob)
        return -dz, -dxr, -dwr
    _patch(monkeypatch, "route_bwd", bad)
    _expect_failure(P.test_backward_matches_central_differences, False)


def test_tie_to_higher_index_is_caught(monkeypatch):
    orig_sorted = sorted

    def bad_topk(z, K):
        T, E = z.shape
        s = M.softmax_rows(z)
        idx = np.empty((T, K), dtype=np.int64)
        prob = np.empty((T, K))
        for t in range(T):
            chosen = orig_sorted(range(E), key=lambda e: (-z[t, e], -e))[:K]
            d = sum(s[t, e] for e in chosen)
            idx[t] = chosen
            prob[t] = [s[t, e] / d for e in chosen]
        return idx, prob
    _patch(monkeypatch, "top_k_route", bad_topk)
    _expect_failure(P.test_topk_ties_go_to_lower_index)


def test_missing_renormalisation_is_caught(monkeypatch):
    def bad_topk(z, K):
        T, E = z.shape
        s = M.softmax_rows(z)
        idx = np.empty((T, K), dtype=np.int64)
        prob = np.empty((T, K))
        for t in range(T):
            chosen = sorted(range(E), key=lambda e: (-z[t, e], e))[:K]
            idx[t] = chosen
            prob[t] = [s[t, e] for e in chosen]
        return idx, prob
    _patch(monkeypatch, "top_k_route", bad_topk)
    _expect_failure(P.test_topk_matches_brute_force_random, 6, 3)
    _expect_failure(P.test_identical_experts_give_dense_ffn_for_any_routing)


def test_transposed_down_projection_is_caught(monkeypatch):
    def bad(X_e, wg_e, wu_e, w2_e):
        g = np.matmul(X_e, wg_e.T)
        u = np.matmul(X_e, wu_e.T)
        a = M.silu(g) * u
        return g, u, a, np.matmul(a, w2_e)  # w2 used untransposed
    _patch(monkeypatch, "expert_ffn_one", bad)
    # square D = F makes the mistaken product well formed
    def square_case():
        p = P._small_layer(T=30, D=6, E=4, K=2, F=6, seed=7)
        fwd = M.layer_forward(p["x"], p["w_router"], p["w_gate"], p["w_up"], p["w2"], K=2)
        for e in range(4):
            lo, hi = fwd["offsets"][e], fwd["offsets"][e + 1]
            ref = P._dense_swiglu_torch(p["x"][fwd["token_of_row"][lo:hi]], p["w_gate"][e], p["w_up"][e], p["w2"][e])
            np.testing.assert_allclose(fwd["y_perm"][lo:hi], ref.numpy(), rtol=1e-12, atol=1e-12)
    _expect_failure(square_case)


def test_unstable_permutation_is_caught(monkeypatch):
    def bad(idx, E):
        T, K = idx.shape
        flat = idx.reshape(-1).tolist()
        order = sorted(range(T * K), key=lambda s: (flat[s], -(s // K)))
        ros = np.empty(T * K, dtype=np.int64)
        tor = np.empty(T * K, dtype=np.int64)
        for r, s in enumerate(order):
            ros[s] = r
            tor[r] = s // K
        off = np.concatenate([[0], np.cumsum(np.bincount(flat, minlength=E))])
        return off, ros, tor
    _patch(monkeypatch, "expert_permutation", bad)
    _expect_failure(P.test_permutation_vs_stable_argsort, 50, 8, 2)


def test_wrong_combine_weight_is_caught(monkeypatch):
    def bad(y_perm, prob_perm, row_of_slot, T, K):
        y = np.zeros((T, y_perm.shape[1]))
        for t in range(T):
            for k in range(K):
                r = row_of_slot[t * K + k]
                y[t] += prob_perm[row_of_slot[t * K]] * y_perm[r]   # always slot 0's weight
        return y
    _patch(monkeypatch, "combine", bad)
    _expect_failure(P.test_combine_of_dispatch_with_identity_experts_returns_x)


def test_sigmoid_router_mistakes_are_caught(monkeypatch):
    import oracle.router_sigmoid as RS
    import tests.test_oracle_sigmoid as PS
    orig_bwd = RS.sigmoid_route_bwd

    def no_sigmoid_slope(x, w_router, z, idx, prob, dprob, f, S, GBS, coef, aux_grad=1.0):
        dz, _, _ = orig_bwd(x, w_router, z, idx, prob, dprob, f, S, GBS, coef, aux_grad)
        s = M.sigmoid(z)
        dz = dz / (s * (1 - s))                       # dropped the sigmoid derivative
        return dz, dz @ w_router, dz.T @ x
    monkeypatch.setattr(RS, "sigmoid_route_bwd", no_sigmoid_slope)
    monkeypatch.setattr(oracle, "sigmoid_route_bwd", no_sigmoid_slope)
    _expect_failure(PS.test_router_gradient_matches_central_differences)

    orig_aux = RS.seq_aux_loss

    def wrong_fraction(z, idx, S, GBS, coef):
        loss, f, P = orig_aux(z, idx, S, GBS, coef)
        return loss * idx.shape[1], f * idx.shape[1], P     # missing the 1/K of the load fraction
    monkeypatch.setattr(RS, "seq_aux_loss", wrong_fraction)
    monkeypatch.setattr(oracle, "seq_aux_loss", wrong_fraction)
    _expect_failure(PS.test_balanced_routing_with_flat_scores_gives_the_coefficient)


def test_shared_expert_mistakes_are_caught(monkeypatch):
    import oracle.shared as SE
    import tests.test_oracle_shared as PSH

    def relu_slope_one(dy, x, h, a, w_s1, w_s2):
        dA = np.matmul(dy, w_s2)
        dh = np.maximum(h, 0.0) * dA                   # the factor 2 of d relu^2 dropped
        return dh, np.matmul(dh, w_s1), np.matmul(dh.T, x), np.matmul(dy.T, a)
    monkeypatch.setattr(SE, "shared_expert_bwd", relu_slope_one)
    monkeypatch.setattr(oracle, "shared_expert_bwd", relu_slope_one)
    _expect_failure(PSH.test_backward_matches_central_differences)
    monkeypatch.undo()

    def plain_relu(x, w_s1, w_s2):
        h = np.matmul(x, w_s1.T)
        a = np.maximum(h, 0.0)                         # square dropped
        return h, a, np.matmul(a, w_s2.T)
    monkeypatch.setattr(SE, "shared_expert", plain_relu)
    monkeypatch.setattr(oracle, "shared_expert", plain_relu)
    _expect_failure(PSH.test_degree_two_homogeneity_and_sign_gate)
    monkeypatch.undo()

    def transposed_down(x, w_s1, w_s2):
        h = np.matmul(x, w_s1.T)
        a = O_relu_sq(h)
        return h, a, np.matmul(a, w_s2[:, ::-1].T)      # hidden units matched to the wrong columns
    O_relu_sq = SE.relu_sq
    monkeypatch.setattr(SE, "shared_expert", transposed_down)
    monkeypatch.setattr(oracle, "shared_expert", transposed_down)
    _expect_failure(PSH.test_forward_is_a_sum_of_squared_positive_projections)


def test_fp8_payload_mistakes_are_caught(monkeypatch):
    import oracle.fp8 as F
    import tests.test_oracle_fp8 as PF

    def ties_away(v):
        neg = v < 0
        a = abs(v)
        if a >= F.E4M3_MAX:
            return F._CODES[-1] | (0x80 if neg else 0)
        best = min(zip(F._CODES, F._VALS), key=lambda cv: (abs(cv[1] - a), -cv[1]))   # ties to the larger
        return best[0] | (0x80 if neg else 0)
    monkeypatch.setattr(F, "e4m3_quantize", ties_away)
    monkeypatch.setattr(oracle, "e4m3_quantize", ties_away)
    _expect_failure(PF.test_ties_go_to_the_even_code_and_saturate)
    monkeypatch.undo()

    def scale_one_too_big(row):
        amax = float(np.max(np.abs(row)))
        if amax == 0.0:
            return 1.0
        e = -126
        while amax > F.E4M3_MAX * 2.0 ** e:
            e += 1
        return 2.0 ** (e + 1)                              # not the smallest fitting power of two
    monkeypatch.setattr(F, "fp8_row_scale", scale_one_too_big)
    monkeypatch.setattr(oracle, "fp8_row_scale", scale_one_too_big)
    _expect_failure(PF.test_row_scale_is_the_smallest_fitting_power_of_two)


def test_nvfp4_payload_mistakes_are_caught(monkeypatch):
    import oracle.nvfp4 as N
    import tests.test_oracle_nvfp4 as PN

    # rounding ties away from zero instead of to the even code
    def ties_away(v):
        neg = v < 0
        a = abs(v)
        if a >= N.E2M1_MAX:
            return N._CODES[-1] | (0x8 if neg else 0)
        best = min(zip(N._CODES, N._VALS), key=lambda cv: (abs(cv[1] - a), -cv[1]))
        return best[0] | (0x8 if neg else 0)
    monkeypatch.setattr(N, "e2m1_quantize", ties_away)
    monkeypatch.setattr(oracle, "e2m1_quantize", ties_away)
    _expect_failure(PN.test_ties_to_even_saturation_and_sign)
    monkeypatch.undo()

    # the two codes of a byte swapped (element 2j in the high nibble)
    real = N.nvfp4_quantize_rows

    def swapped_nibbles(x):
        codes, bsc, rsc = real(x)
        return ((codes >> 4) | ((codes & 0xF) << 4)).astype(np.uint8), bsc, rsc
    monkeypatch.setattr(N, "nvfp4_quantize_rows", swapped_nibbles)
    monkeypatch.setattr(oracle, "nvfp4_quantize_rows", swapped_nibbles)
    _expect_failure(PN.test_hand_computed_block)
    monkeypatch.undo()

    # block scale from the row maximum instead of the block's own maximum
    def row_amax_scales(x):
        codes, bsc, rsc = real(x)
        bsc[:] = bsc.max(axis=1, keepdims=True)
        return codes, bsc, rsc
    monkeypatch.setattr(N, "nvfp4_quantize_rows", row_amax_scales)
    monkeypatch.setattr(oracle, "nvfp4_quantize_rows", row_amax_scales)
    _expect_failure(PN.test_round_trip_and_bf16_exactness)


def test_sigmoid_key_selection_mistakes_are_caught(monkeypatch):
    import oracle.router_sigmoid as RS
    import tests.test_oracle_sigmoid as PS

    def ties_to_higher(keys, K):
        T, E = keys.shape
        return np.array([sorted(range(E), key=lambda e: (-float(keys[t, e]), -e))[:K] for t in range(T)],
                        dtype=np.int64)

    monkeypatch.setattr(RS, "select_on_keys", ties_to_higher)
    monkeypatch.setattr(oracle, "select_on_keys", ties_to_higher)
    _expect_failure(PS.test_selection_on_given_keys_against_brute_force_with_exact_ties, 8, 3)
    _expect_failure(PS.test_gates_on_key_choice_use_scores_not_keys)

    def ascending(keys, K):
        T, E = keys.shape
        return np.array([sorted(range(E), key=lambda e: (-float(keys[t, e]), e))[:K][::-1] for t in range(T)],
                        dtype=np.int64)

    monkeypatch.setattr(RS, "select_on_keys", ascending)
    monkeypatch.setattr(oracle, "select_on_keys", ascending)
    _expect_failure(PS.test_selection_on_given_keys_against_brute_force_with_exact_ties, 8, 3)
