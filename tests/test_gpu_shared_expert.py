"""GPU parity of the shared expert (ungated squared-ReLU MLP added to the layer
output, Sec. 5.2, readings SH1-SH2) against the float64 oracle.

Stage-isolated checks call the two entry points on the GPU's own inputs with
the accumulation targets zeroed; the end-to-end check runs the whole layer
with a shared expert against the oracle composed from the raw inputs.
Tolerance: relative Frobenius 1e-2 (bf16 storage, fp32 accumulation).
"""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.gpu_util import REL_FROB, f64, i64, oracle_inputs, rel_frob

pytestmark = pytest.mark.gpu

W = synth.Workload
CASES = {
    # F_s = 320: one full and one ragged 256-column tile
    "sh_bf16": (W("sh_bf16", S=300, GBS=2, D=256, E=16, K=4, F=256), 320),
    "sh_latent": (W("sh_latent", S=256, GBS=2, D=256, E=32, K=4, F=192, H=512), 384),
    "sh_fp32": (W("sh_fp32", S=200, GBS=1, D=192, E=12, K=3, F=192, dtype="f32"), 128),
    "sh_wide": (W("sh_wide", S=384, GBS=1, D=1024, E=8, K=2, F=768), 1536),
    "sh_t1": (W("sh_t1", S=1, GBS=1, D=128, E=8, K=2, F=128), 64),
}

_cache = {}


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    yield
    _cache.clear()


def run(name):
    if name not in _cache:
        from paper_2608_28511_gb300.layer import MoeLayer
        w, Fs = CASES[name]
        inputs = synth.make_inputs(w)
        inputs.update(synth.make_shared_expert(w, Fs, w.seed))
        L = MoeLayer(w.S, w.GBS, w.K, w.D, w.E, w.F, w.dtype, w.H, shared_F=Fs)
        L.load(inputs)
        L.forward()
        L.backward()
        torch.cuda.synchronize()
        _cache[name] = (w, Fs, L, inputs, oracle_inputs(inputs))
    return _cache[name]


names = list(CASES)


@pytest.mark.parametrize("name", names)
def test_shared_forward_stage(name):
    from paper_2608_28511_gb300 import abi
    w, Fs, L, inp, o = run(name)
    h_ref, a_ref, y_ref = O.shared_expert(o["x"], o["w_s1"], o["w_s2"])
    assert rel_frob(f64(L.h_s), h_ref) <= REL_FROB
    assert rel_frob(f64(L.act_s), a_ref) <= REL_FROB
    assert (f64(L.act_s)[h_ref < -1e-2] == 0).all()           # the ReLU gate
    y = torch.zeros_like(L.y)
    h = torch.empty_like(L.h_s)
    a = torch.empty_like(L.act_s)
    abi.moe_shared_expert(L.shape, Fs, L.x, L.w_s1, L.w_s2, h, a, y)
    torch.cuda.synchronize()
    assert torch.equal(h, L.h_s) and torch.equal(a, L.act_s)   # deterministic
    assert rel_frob(f64(y), y_ref) <= REL_FROB


@pytest.mark.parametrize("name", names)
def test_shared_backward_stage(name):
    from paper_2608_28511_gb300 import abi
    w, Fs, L, inp, o = run(name)
    h, a = f64(L.h_s), f64(L.act_s)
    dh_ref, dx_ref, dw1_ref, dw2_ref = O.shared_expert_bwd(o["dy"], o["x"], h, a, o["w_s1"], o["w_s2"])
    dh = torch.empty_like(L.dh_s)
    dx = torch.zeros_like(L.dx)
    dw1 = torch.empty_like(L.dw_s1)
    dw2 = torch.empty_like(L.dw_s2)
    abi.moe_shared_expert_bwd(L.shape, Fs, L.dy, L.x, L.h_s, L.act_s, L.w_s1, L.w_s2, dh, dx, dw1, dw2)
    torch.cuda.synchronize()
    assert rel_frob(f64(dh), dh_ref) <= REL_FROB
    assert rel_frob(f64(dx), dx_ref) <= REL_FROB
    assert rel_frob(f64(dw1), dw1_ref) <= REL_FROB
    assert rel_frob(f64(dw2), dw2_ref) <= REL_FROB
    assert torch.equal(dw1, L.dw_s1) and torch.equal(dw2, L.dw_s2)


@pytest.mark.parametrize("name", ["sh_bf16", "sh_latent", "sh_fp32"])
def test_layer_with_shared_expert_end_to_end(name):
    w, Fs, L, inp, o = run(name)
    kw = dict(w_down=o.get("w_down"), w_upp=o.get("w_upp"))
    fwd = O.layer_forward(o["x"], o["w_router"], o["w_gate"], o["w_up"], o["w2"], w.K, bias=o["bias"],
                          idx_override=i64(L.topk_idx), **kw)
    h, a, y_sh = O.shared_expert(o["x"], o["w_s1"], o["w_s2"])
    assert rel_frob(f64(L.y), fwd["y"] + y_sh) <= REL_FROB
    bwd = O.layer_backward(fwd, o["dy"], o["x"], o["w_router"], o["w_gate"], o["w_up"], o["w2"], **kw)
    _, dx_sh, dw1, dw2 = O.shared_expert_bwd(o["dy"], o["x"], h, a, o["w_s1"], o["w_s2"])
    assert rel_frob(f64(L.dx), bwd["dx"] + dx_sh) <= REL_FROB
    assert rel_frob(f64(L.dw_s1), dw1) <= REL_FROB
    assert rel_frob(f64(L.dw_s2), dw2) <= REL_FROB
    # the routed part is unchanged by the shared expert
    assert rel_frob(f64(L.dw_router), bwd["dw_router"]) <= REL_FROB


def test_shared_expert_shape_errors():
    from paper_2608_28511_gb300 import abi
    w, Fs, L, inp, o = run("sh_bf16")
    for bad in (0, 96, -64):
        with pytest.raises(abi.MoeError) as e:
            abi.moe_shared_expert(L.shape, bad, L.x, L.w_s1, L.w_s2, L.h_s, L.act_s, L.y)
        assert e.value.status == -1
    with pytest.raises(abi.MoeError) as e:
        abi.moe_shared_expert(L.shape, Fs, L.x, None, L.w_s2, L.h_s, L.act_s, L.y)
    assert e.value.status == -4
