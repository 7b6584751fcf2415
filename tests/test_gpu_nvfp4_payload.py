"""GPU parity of the NVFP4 dispatch payload (readings NV1-NV3) against the
float64 oracle: codes, block scales and row scales bit for bit
(stage-isolated: the oracle quantizes the GPU's own dispatch input), the
dequantized rows exactly, the Eq. 1 payload bytes with b_x = 1/2 plus the
scales, and the whole layer with the quantized payload within the layer
tolerances."""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.gpu_util import REL_FROB, f64, i64, oracle_inputs, rel_frob

pytestmark = pytest.mark.gpu

W = synth.Workload
CASES = {
    "nv4_bf16": W("nv4_bf16", S=500, GBS=2, D=256, E=16, K=4, F=320),
    "nv4_skew": W("nv4_skew", S=350, GBS=2, D=256, E=16, K=4, F=256, skew_bias=True),
    "nv4_latent": W("nv4_latent", S=300, GBS=2, D=256, E=32, K=4, F=192, H=512),
    "nv4_wide": W("nv4_wide", S=384, GBS=1, D=1024, E=8, K=2, F=768),
    "nv4_k16": W("nv4_k16", S=50, GBS=1, D=64, E=32, K=16, F=64),
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
        L = MoeLayer(w.S, w.GBS, w.K, w.D, w.E, w.F, w.dtype, w.H, payload="nvfp4")
        L.load(inputs)
        L.forward()
        L.backward()
        torch.cuda.synchronize()
        _cache[name] = (w, L, inputs, oracle_inputs(inputs))
    return _cache[name]


@pytest.mark.parametrize("name", list(CASES))
def test_codes_and_scales_bit_exact(name):
    w, L, inp, o = run(name)
    codes, bsc, rsc = O.nvfp4_quantize_rows(f64(L.x_lat if w.H else L.x))
    tor = i64(L.token_of_row)
    assert np.array_equal(L.x_perm_q4.cpu().numpy(), codes[tor])
    assert np.array_equal(L.x_bscale_perm.cpu().numpy(), bsc[tor])
    assert np.array_equal(f64(L.x_rscale_perm), rsc[tor])
    # the receiver's bf16 rows are the exact dequantized values
    assert np.array_equal(f64(L.x_perm), O.nvfp4_dequantize_rows(codes, bsc, rsc)[tor])
    # Eq. 1 payload of the hidden + probability dispatch with b_x = 1/2, plus
    # one E4M3 scale per 16 elements and one fp32 scale per row
    nbytes = (L.x_perm_q4.numel() + L.x_bscale_perm.numel() + 4 * L.x_rscale_perm.numel()
              + 4 * L.prob_perm.numel())
    assert nbytes == w.T * w.K * (w.D // 2 + w.D // 16 + 4 + 4)


def _dispatch_nvfp4(x, K, E):
    """Runs moe_dispatch_nvfp4 + moe_dequant_nvfp4 on bf16 rows x [T, D]
    (CPU tensor) with a fixed round-robin routing."""
    from paper_2608_28511_gb300 import abi
    T, D = x.shape
    w = W("nv4_direct", S=T, GBS=1, D=D, E=E, K=K, F=64)
    shp = abi.MoeShape.from_workload(w)
    idx = torch.stack([(torch.arange(T) + 3 * k) % E for k in range(K)], 1).to(torch.int32)
    prob = torch.full((T, K), 1.0 / K)
    dev = "cuda"
    TK = T * K
    off = torch.empty(E + 1, dtype=torch.int32, device=dev)
    ros = torch.empty(TK, dtype=torch.int32, device=dev)
    tor = torch.empty(TK, dtype=torch.int32, device=dev)
    q = torch.empty(TK, D // 2, dtype=torch.uint8, device=dev)
    bs = torch.empty(TK, D // 16, dtype=torch.uint8, device=dev)
    rs = torch.empty(TK, device=dev)
    pp = torch.empty(TK, device=dev)
    xp = torch.empty(TK, D, dtype=torch.bfloat16, device=dev)
    ws = torch.empty(abi.moe_workspace_size(shp), dtype=torch.uint8, device=dev)
    abi.moe_dispatch_nvfp4(shp, x.to(dev), idx.to(dev), prob.to(dev), off, ros, tor, q, bs, rs, pp, ws)
    abi.moe_dequant_nvfp4(shp, q, bs, rs, xp)
    torch.cuda.synchronize()
    return (tor.cpu().numpy().astype(np.int64), q.cpu().numpy(), bs.cpu().numpy(), rs.cpu().double().numpy(),
            xp.cpu().double().numpy())


def _check_direct(x, K=2, E=8):
    t, q, bs, rs, xp = _dispatch_nvfp4(x, K, E)
    codes, bsc, rsc = O.nvfp4_quantize_rows(x.double().numpy())
    assert np.array_equal(q, codes[t])
    assert np.array_equal(bs, bsc[t])
    assert np.array_equal(rs, rsc[t])
    assert np.array_equal(xp, O.nvfp4_dequantize_rows(codes, bsc, rsc)[t])


def test_extreme_row_magnitudes():
    """Rows spanning 2^-120 .. 2^100 (the smallest ones at the clamped row
    exponent -126), an all-zero row, an all-zero block, a saturating element
    and blocks far below their row's maximum (E4M3 subnormal and zero block
    scales)."""
    g = torch.Generator().manual_seed(5)
    x = torch.randn(64, 128, generator=g)
    x = x * torch.pow(2.0, torch.linspace(-120, 100, 64)).unsqueeze(1)
    x[3] = 0.0
    x[9, 16:32] = 0.0
    x[7, 5] = -3.0e38
    x[11, :16] *= 2.0 ** -15      # block scale in the E4M3 subnormal range
    x[12, 16:32] *= 2.0 ** -30    # block scale rounds to zero: zero codes
    _check_direct(x.to(torch.bfloat16))


def test_ties_and_nibble_order():
    """Values on E2M1 rounding midpoints (ties to the even code) and a row
    whose even and odd elements differ in sign, so a swapped nibble order or a
    wrong tie rule changes the codes."""
    D = 64
    mids = torch.tensor([0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0, 6.0])
    row = torch.cat([mids, -mids]).repeat(D // 16)
    x = torch.stack([row, -row, row.flip(0), torch.linspace(-6, 6, D)])
    # row maximum 6 * 2^-7: g = 2^-15, every block's s_b = 2^8, so x / (s_b g)
    # is exactly the midpoints above
    x = (x * 2.0 ** -7).to(torch.bfloat16)
    _check_direct(x, K=1, E=4)
    t, q, bs, rs, xp = _dispatch_nvfp4(x, 1, 4)
    r = int(np.nonzero(t == 0)[0][0])
    # element 0 (0.25 -> tie between 0 and 0.5: the even code 0) and element 1
    # (0.75 -> tie between 0.5 and 1: the even code 2, value 1.0)
    assert q[r, 0] == (0x2 << 4) | 0x0


@pytest.mark.parametrize("name", ["nv4_bf16", "nv4_skew", "nv4_wide"])
def test_layer_with_nvfp4_payload_end_to_end(name):
    w, L, inp, o = run(name)
    x, wr = o["x"], o["w_router"]
    idx = i64(L.topk_idx)
    fwd = O.layer_forward(x, wr, o["w_gate"], o["w_up"], o["w2"], w.K, bias=o["bias"], idx_override=idx)
    x_deq = O.nvfp4_dequantize_rows(*O.nvfp4_quantize_rows(x))
    off, ros, tor = fwd["offsets"], fwd["row_of_slot"], fwd["token_of_row"]
    x_perm, prob_perm = O.dispatch(x_deq, fwd["prob"], ros, tor)
    g, u, a, y_perm = O.expert_ffn(x_perm, off, o["w_gate"], o["w_up"], o["w2"])
    y = O.combine(y_perm, prob_perm, ros, w.T, w.K)
    assert rel_frob(f64(L.y), y) <= REL_FROB
    dy_perm, dprob_perm = O.combine_bwd(o["dy"], y_perm, prob_perm, tor)
    dx_perm, dwg, dwu, dw2 = O.expert_ffn_bwd(dy_perm, x_perm, g, u, off, o["w_gate"], o["w_up"], o["w2"])
    dx_e, dprob = O.dispatch_bwd(dx_perm, dprob_perm, ros, w.T, w.K)
    dz, dx_r, dw_r = O.route_bwd(x, wr, idx, fwd["prob"], dprob)
    assert rel_frob(f64(L.dx), dx_e + dx_r) <= REL_FROB              # straight-through (NV3)
    gg, gu = L.unpack_w1_like(L.dw1)
    assert rel_frob(f64(gg), dwg) <= REL_FROB
    assert rel_frob(f64(gu), dwu) <= REL_FROB
    assert rel_frob(f64(L.dw2), dw2) <= REL_FROB
    assert rel_frob(f64(L.dw_router), dw_r) <= REL_FROB


def test_nvfp4_payload_rejects_fp32():
    from paper_2608_28511_gb300 import abi
    w = W("nv4_f32", S=8, GBS=1, D=64, E=4, K=2, F=64, dtype="f32")
    shp = abi.MoeShape.from_workload(w)
    dev = "cuda"
    z = lambda *s, d=torch.float32: torch.zeros(*s, dtype=d, device=dev)  # noqa: E731
    with pytest.raises(abi.MoeError) as e:
        abi.moe_dispatch_nvfp4(shp, z(8, 64), z(8, 2, d=torch.int32), z(8, 2), z(5, d=torch.int32),
                               z(16, d=torch.int32), z(16, d=torch.int32), z(16, 32, d=torch.uint8),
                               z(16, 4, d=torch.uint8), z(16), z(16), z(1 << 16, d=torch.uint8))
    assert e.value.status == -8
