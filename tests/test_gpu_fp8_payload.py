"""GPU parity of the FP8 dispatch payload (readings FP1-FP3) against the
float64 oracle: codes and scales bit for bit (stage-isolated: the oracle
quantizes the GPU's own dispatch input), the dequantized rows exactly, the
Eq. 1 payload bytes, and the whole layer with the quantized payload within the
layer tolerances."""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.gpu_util import REL_FROB, f64, i64, oracle_inputs, rel_frob

pytestmark = pytest.mark.gpu

W = synth.Workload
CASES = {
    "fp8_bf16": W("fp8_bf16", S=500, GBS=2, D=256, E=16, K=4, F=320),
    "fp8_skew": W("fp8_skew", S=350, GBS=2, D=256, E=16, K=4, F=256, skew_bias=True),
    "fp8_latent": W("fp8_latent", S=300, GBS=2, D=256, E=32, K=4, F=192, H=512),
    "fp8_wide": W("fp8_wide", S=384, GBS=1, D=1024, E=8, K=2, F=768),
    "fp8_k16": W("fp8_k16", S=50, GBS=1, D=64, E=32, K=16, F=64),
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
        w = CASES[name]
        inputs = synth.make_inputs(w)
        L = MoeLayer(w.S, w.GBS, w.K, w.D, w.E, w.F, w.dtype, w.H, payload="fp8")
        L.load(inputs)
        L.forward()
        L.backward()
        torch.cuda.synchronize()
        _cache[name] = (w, L, inputs, oracle_inputs(inputs))
    return _cache[name]


def _codes_of(name):
    w, L, inp, o = run(name)
    x_disp = f64(L.x_lat if w.H else L.x)
    return O.fp8_quantize_rows(x_disp)


@pytest.mark.parametrize("name", list(CASES))
def test_codes_and_scales_bit_exact(name):
    w, L, inp, o = run(name)
    codes, scales = _codes_of(name)
    tor = i64(L.token_of_row)
    assert np.array_equal(L.x_perm_q.cpu().numpy(), codes[tor])
    assert np.array_equal(f64(L.x_scale_perm), scales[tor])
    # the receiver's bf16 rows are the exact dequantized values
    assert np.array_equal(f64(L.x_perm), O.fp8_dequantize_rows(codes, scales)[tor])
    # Eq. 1 payload of the hidden + probability dispatch with b_x = 1 (and one fp32 scale per row)
    nbytes = L.x_perm_q.numel() + 4 * L.x_scale_perm.numel() + 4 * L.prob_perm.numel()
    assert nbytes == w.T * w.K * (w.D * 1 + 4 + 4)


def test_extreme_row_magnitudes():
    """Rows spanning 2^-100 .. 2^100, an all-zero row and saturating values."""
    from paper_2608_28511_gb300 import abi
    w = W("fp8_extreme", S=64, GBS=1, D=128, E=8, K=2, F=128)
    shp = abi.MoeShape.from_workload(w)
    g = torch.Generator().manual_seed(5)
    x = torch.randn(64, 128, generator=g)
    x = x * torch.pow(2.0, torch.linspace(-100, 100, 64)).unsqueeze(1)
    x[3] = 0.0
    x[7, 5] = -3.0e38
    x = x.to(torch.bfloat16)
    idx = torch.stack([torch.arange(64) % 8, (torch.arange(64) + 3) % 8], 1).to(torch.int32)
    prob = torch.full((64, 2), 0.5)
    dev = "cuda"
    xd, idxd, probd = x.to(dev), idx.to(dev), prob.to(dev)
    off = torch.empty(9, dtype=torch.int32, device=dev)
    ros = torch.empty(128, dtype=torch.int32, device=dev)
    tor = torch.empty(128, dtype=torch.int32, device=dev)
    q = torch.empty(128, 128, dtype=torch.uint8, device=dev)
    sc = torch.empty(128, device=dev)
    pp = torch.empty(128, device=dev)
    xp = torch.empty(128, 128, dtype=torch.bfloat16, device=dev)
    ws = torch.empty(abi.moe_workspace_size(shp), dtype=torch.uint8, device=dev)
    abi.moe_dispatch_fp8(shp, xd, idxd, probd, off, ros, tor, q, sc, pp, ws)
    abi.moe_dequant_rows(shp, q, sc, xp)
    torch.cuda.synchronize()
    codes, scales = O.fp8_quantize_rows(x.double().numpy())
    t = tor.cpu().numpy().astype(np.int64)
    assert np.array_equal(q.cpu().numpy(), codes[t])
    assert np.array_equal(sc.cpu().double().numpy(), scales[t])
    assert np.array_equal(xp.cpu().double().numpy(), O.fp8_dequantize_rows(codes, scales)[t])


@pytest.mark.parametrize("name", ["fp8_bf16", "fp8_skew", "fp8_wide"])
def test_layer_with_fp8_payload_end_to_end(name):
    w, L, inp, o = run(name)
    x, wr = o["x"], o["w_router"]
    idx = i64(L.topk_idx)
    fwd = O.layer_forward(x, wr, o["w_gate"], o["w_up"], o["w2"], w.K, bias=o["bias"], idx_override=idx)
    x_deq = O.fp8_dequantize_rows(*O.fp8_quantize_rows(x))
    off, ros, tor = fwd["offsets"], fwd["row_of_slot"], fwd["token_of_row"]
    x_perm, prob_perm = O.dispatch(x_deq, fwd["prob"], ros, tor)
    g, u, a, y_perm = O.expert_ffn(x_perm, off, o["w_gate"], o["w_up"], o["w2"])
    y = O.combine(y_perm, prob_perm, ros, w.T, w.K)
    assert rel_frob(f64(L.y), y) <= REL_FROB
    dy_perm, dprob_perm = O.combine_bwd(o["dy"], y_perm, prob_perm, tor)
    dx_perm, dwg, dwu, dw2 = O.expert_ffn_bwd(dy_perm, x_perm, g, u, off, o["w_gate"], o["w_up"], o["w2"])
    dx_e, dprob = O.dispatch_bwd(dx_perm, dprob_perm, ros, w.T, w.K)
    dz, dx_r, dw_r = O.route_bwd(x, wr, idx, fwd["prob"], dprob)
    assert rel_frob(f64(L.dx), dx_e + dx_r) <= REL_FROB              # straight-through (FP3)
    gg, gu = L.unpack_w1_like(L.dw1)
    assert rel_frob(f64(gg), dwg) <= REL_FROB
    assert rel_frob(f64(gu), dwu) <= REL_FROB
    assert rel_frob(f64(L.dw2), dw2) <= REL_FROB
    assert rel_frob(f64(L.dw_router), dw_r) <= REL_FROB


def test_fp8_payload_rejects_fp32():
    from paper_2608_28511_gb300 import abi
    w = W("fp8_f32", S=8, GBS=1, D=64, E=4, K=2, F=64, dtype="f32")
    shp = abi.MoeShape.from_workload(w)
    dev = "cuda"
    z = lambda *s, d=torch.float32: torch.zeros(*s, dtype=d, device=dev)  # noqa: E731
    with pytest.raises(abi.MoeError) as e:
        abi.moe_dispatch_fp8(shp, z(8, 64), z(8, 2, d=torch.int32), z(8, 2), z(5, d=torch.int32),
                             z(16, d=torch.int32), z(16, d=torch.int32), z(16, 64, d=torch.uint8), z(16), z(16),
                             z(1 << 16, d=torch.uint8))
    assert e.value.status == -8
