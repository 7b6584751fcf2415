"""The gathering expert FFN (GEMM-1 and its weight gradient read the
dispatched rows straight from x by token_of_row, no x_perm copy) against the
default path that writes x_perm: every output agrees bit for bit, so the
gathering path inherits the x_perm path's stage-by-stage parity with the
oracle (``test_gpu_parity.py``).  Also checked directly against the oracle,
and on the edge shapes (one token, ragged tails, K = 16, fp32)."""
import pytest
import torch

import oracle as O
import synth
from tests.gpu_util import REL_FROB, f64, i64, make_layer, oracle_inputs, rel_frob
from tests.test_gpu_parity import CASES, EDGE

pytestmark = pytest.mark.gpu

OUTPUTS = ("topk_idx", "topk_prob", "expert_offsets", "row_of_slot", "token_of_row", "h", "act", "y_perm", "y",
           "dy_perm", "dprob_perm", "dx_perm", "dw1", "dw2", "dx", "dlogits", "dw_router")


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _bits(t):
    return t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.uint8)


CASE_LIST = list(CASES.values()) + [e for e in EDGE if e.name in ("t1", "t127", "k16", "t3_fp32")]


@pytest.mark.parametrize("w", CASE_LIST, ids=[c.name for c in CASE_LIST])
def test_gather_matches_x_perm_path_bitwise(w):
    inp = synth.make_inputs(w)
    Lg, _ = make_layer(w, inputs=inp, gather=True)
    Lp, _ = make_layer(w, inputs=inp, gather=False)
    assert Lg.x_perm is None
    for name in OUTPUTS + (("y_lat", "dx_lat", "dw_down", "dw_upp") if w.H else ()):
        a, b = getattr(Lg, name), getattr(Lp, name)
        # +0 and -0 may differ where a sum is exactly zero: compare values, then bits elsewhere
        assert torch.equal(a, b), name
        nz = b != 0
        assert torch.equal(_bits(a[nz]), _bits(b[nz])), name


def test_gather_end_to_end_against_oracle():
    w = CASES["mid_latent"]
    L, inp = make_layer(w, gather=True)
    o = oracle_inputs(inp)
    fwd = O.layer_forward(o["x"], o["w_router"], o["w_gate"], o["w_up"], o["w2"], w.K, idx_override=i64(L.topk_idx),
                          w_down=o["w_down"], w_upp=o["w_upp"])
    bwd = O.layer_backward(fwd, o["dy"], o["x"], o["w_router"], o["w_gate"], o["w_up"], o["w2"],
                           w_down=o["w_down"], w_upp=o["w_upp"])
    assert rel_frob(f64(L.y), fwd["y"]) <= REL_FROB
    assert rel_frob(f64(L.dx), bwd["dx"]) <= REL_FROB
    gg, gu = L.unpack_w1_like(L.dw1)
    assert rel_frob(f64(gg), bwd["dw_gate"]) <= REL_FROB
    assert rel_frob(f64(gu), bwd["dw_up"]) <= REL_FROB
    assert rel_frob(f64(L.dw2), bwd["dw2"]) <= REL_FROB
