"""The dispatch backward fused with the softmax router's backward
(moe_dispatch_route_bwd, what MoeLayer runs without latent projection)
against the two separate calls and against float64 sums of the GPU's own
stage inputs: dtopk_prob, dlogits and dw_router bit-identical to the separate
calls, dx within one bf16 rounding of the exact sum of the K dX_perm rows plus
dlogits . W_r (the separate calls round dx twice)."""
import numpy as np
import pytest
import torch

import synth
from tests.gpu_util import f64, i64, make_layer

pytestmark = pytest.mark.gpu

W = synth.Workload
CASES = {
    "tiny_f32": W("frb_tiny", S=256, GBS=1, D=128, E=8, K=2, F=256, dtype="f32"),
    "ragged": W("frb_ragged", S=333, GBS=1, D=192, E=24, K=6, F=128),
    "k8_e128": W("frb_k8", S=500, GBS=1, D=256, E=128, K=8, F=128),
    "k16": W("frb_k16", S=77, GBS=1, D=64, E=32, K=16, F=64),
    "skew": W("frb_skew", S=600, GBS=1, D=128, E=16, K=4, F=64, skew_bias=True),
}


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("name", list(CASES))
def test_fused_matches_separate_calls(name):
    from paper_2608_28511_gb300 import abi
    w = CASES[name]
    L, _ = make_layer(w)
    s = L.shape
    dx_sep = torch.empty_like(L.dx)
    dprob_sep = torch.empty_like(L.dprob)
    dlog_sep = torch.empty_like(L.dlogits)
    dwr_sep = torch.empty_like(L.dw_router)
    abi.moe_dispatch_bwd(s, L.dx_perm, L.dprob_perm, L.row_of_slot, dx_sep, dprob_sep)
    abi.moe_route_bwd(s, L.x, L.w_router, L.topk_idx, L.topk_prob, dprob_sep, dx_sep, dwr_sep, dlog_sep, L.ws)
    # the fused call again, into fresh buffers (the layer's own buffers hold its backward)
    dx_f = torch.full_like(L.dx, 7.0)
    dprob_f = torch.full_like(L.dprob, 7.0)
    dlog_f = torch.full_like(L.dlogits, 7.0)
    dwr_f = torch.full_like(L.dw_router, 7.0)
    abi.moe_dispatch_route_bwd(s, L.dx_perm, L.dprob_perm, L.row_of_slot, L.x, L.w_router, L.topk_idx,
                               L.topk_prob, dx_f, dprob_f, dlog_f, dwr_f, L.ws)
    torch.cuda.synchronize()
    assert abi.moe_check_device_status() == 0
    assert torch.equal(dprob_f, dprob_sep)
    assert torch.equal(dlog_f, dlog_sep)
    assert torch.equal(dwr_f, dwr_sep)
    assert torch.equal(dx_f, L.dx)                                   # the layer ran the fused call
    # dx against the exact sum of the same stage inputs
    ros = i64(L.row_of_slot).reshape(w.T, w.K)
    idx = i64(L.topk_idx)
    dxp = f64(L.dx_perm)
    wr = f64(L.w_router)                                             # [E, D]
    dz = f64(dlog_f)                                                 # [T, E], nonzero on the chosen experts
    ref = dxp[ros].sum(axis=1) + dz @ wr
    nz = np.zeros_like(dz, dtype=bool)
    nz[np.arange(w.T)[:, None], idx] = True
    assert np.all(dz[~nz] == 0.0)
    u = 2.0 ** -8 if w.dtype == "bf16" else 2.0 ** -23
    slack = 1e-5 * np.abs(ref).max()                                 # fp32 accumulation of 2K terms
    err_f = np.abs(f64(dx_f) - ref)
    assert np.all(err_f <= u * np.abs(ref) + slack)
    # the separate calls round twice: never closer in total than the fused result by more than rounding noise
    err_s = np.abs(f64(dx_sep) - ref)
    assert err_f.sum() <= err_s.sum() * 1.05 + slack


def test_fused_rejects_latent_shape():
    from paper_2608_28511_gb300 import abi
    w = W("frb_latent", S=64, GBS=1, D=64, E=8, K=2, F=64, H=128)
    shp = abi.MoeShape.from_workload(w)
    dev = "cuda"
    z = lambda *s, d=torch.float32: torch.zeros(*s, dtype=d, device=dev)  # noqa: E731
    with pytest.raises(abi.MoeError) as e:
        abi.moe_dispatch_route_bwd(shp, z(128, 64, d=torch.bfloat16), z(128), z(128, d=torch.int32),
                                   z(64, 128, d=torch.bfloat16), z(8, 128, d=torch.bfloat16), z(64, 2, d=torch.int32),
                                   z(64, 2), z(64, 128, d=torch.bfloat16), z(64, 2), z(64, 8), z(8, 128),
                                   z(1 << 20, d=torch.uint8))
    assert e.value.status == -8
