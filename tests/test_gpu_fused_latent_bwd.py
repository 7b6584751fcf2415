"""The LatentMoE backward tail in one product (moe_latent_route_bwd, what
MoeLayer runs for H > 0 with the softmax router) against the separate calls
(moe_dispatch_bwd, moe_latent_proj_bwd, moe_route_bwd) and against float64
sums of the GPU's own stage inputs: dtopk_prob, dlogits, dw_down and dw_router
bit-identical, the bf16 dlogits columns of [dx_lat | dz] equal to the rounded
dlogits, and dx within one bf16 rounding (plus the fp32 accumulation error of
a K = D + E reduction) of dx_lat . w_down + dz . w_router."""
import numpy as np
import pytest
import torch

import synth
from tests.gpu_util import f64, make_layer

pytestmark = pytest.mark.gpu

W = synth.Workload
CASES = {
    "latent": W("flb_latent", S=300, GBS=2, D=256, E=32, K=4, F=192, H=512),
    "ragged_E24": W("flb_e24", S=257, GBS=1, D=256, E=24, K=3, F=64, H=384),
    "ragged_E40": W("flb_e40", S=333, GBS=1, D=128, E=40, K=5, F=64, H=256),
    "k1": W("flb_k1", S=200, GBS=1, D=128, E=8, K=1, F=64, H=192),
}


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("name", list(CASES))
def test_fused_latent_tail_matches_separate_calls(name):
    from paper_2608_28511_gb300 import abi
    w = CASES[name]
    L, _ = make_layer(w)
    assert L.latent_fused
    s = L.shape
    # the separate calls on the same stage inputs
    dx_lat = torch.empty(w.T, w.D, dtype=torch.bfloat16, device="cuda")
    dprob = torch.empty_like(L.dprob)
    dx = torch.empty_like(L.dx)
    dwd = torch.empty_like(L.dw_down)
    dlog = torch.empty_like(L.dlogits)
    dwr = torch.empty_like(L.dw_router)
    abi.moe_dispatch_bwd(s, L.dx_perm, L.dprob_perm, L.row_of_slot, dx_lat, dprob)
    abi.moe_latent_proj_bwd(s, w.H, w.D, dx_lat, L.x, L.w_down, dx, False, dwd, L.ws)
    abi.moe_route_bwd(s, L.x, L.w_router, L.topk_idx, L.topk_prob, dprob, dx, dwr, dlog, L.ws)
    torch.cuda.synchronize()
    assert abi.moe_check_device_status() == 0
    assert torch.equal(L.dx_lat, dx_lat)
    assert torch.equal(L.dprob, dprob)
    assert torch.equal(L.dlogits, dlog)
    assert torch.equal(L.dw_down, dwd)
    assert torch.equal(L.dw_router, dwr)
    dz16 = L.dx_cat[:, w.D:]
    assert torch.equal(dz16, L.dlogits.to(torch.bfloat16))
    # dx from the same stage inputs, exactly
    a = np.concatenate([f64(L.dx_lat), f64(dz16)], axis=1)            # [T, D + E]
    b = np.concatenate([f64(L.w_down), f64(L.w_router)], axis=0)      # [D + E, H]
    ref = a @ b
    absref = np.abs(a) @ np.abs(b)
    err = np.abs(f64(L.dx) - ref)
    assert np.all(err <= 2.0 ** -8 * np.abs(ref) + 1e-4 * absref)
    # one rounding instead of two: not less accurate in total than the separate calls
    assert err.sum() <= np.abs(f64(dx) - ref).sum() * 1.05 + 1e-6


def test_fused_latent_tail_rejects_plain_layer():
    from paper_2608_28511_gb300 import abi
    w = W("flb_plain", S=64, GBS=1, D=64, E=8, K=2, F=64)
    shp = abi.MoeShape.from_workload(w)
    z = lambda *s, d=torch.float32: torch.zeros(*s, dtype=d, device="cuda")  # noqa: E731
    with pytest.raises(abi.MoeError) as e:
        abi.moe_latent_route_bwd(shp, z(128, 64, d=torch.bfloat16), z(128), z(128, d=torch.int32),
                                 z(64, 64, d=torch.bfloat16), z(72, 64, d=torch.bfloat16), z(64, 2, d=torch.int32),
                                 z(64, 2), z(64, 72, d=torch.bfloat16), z(64, 64, d=torch.bfloat16), z(64, 2),
                                 z(64, 8), z(64, 64), z(8, 64), z(1 << 20, d=torch.uint8))
    assert e.value.status == -8
