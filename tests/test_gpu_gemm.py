"""The dense GEMM shapes of the library (LatentMoE projections and their
backward) against the float64 oracle (``latent_project`` and its adjoint) on
the same bf16 inputs, over sizes with ragged M, N and K tiles.  These
exercise the tensor-core engine's K-major x K-major, K-major x MN-major and
MN-major x MN-major operand paths and its store, accumulate and fp32
epilogues."""
import pytest
import torch

import oracle as O
from paper_2608_28511_gb300 import abi
from tests.gpu_util import f64, rel_frob

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _rnd(g, *shape, scale=1.0):
    """bf16 draws on the host (seeded), copied to the device."""
    return (torch.randn(*shape, generator=g) * scale).to(torch.bfloat16).cuda()


SIZES = [(1, 64, 64), (100, 192, 320), (300, 512, 256), (1000, 320, 1024), (2048, 1024, 64), (129, 64, 576)]


@pytest.mark.parametrize("T,n_in,n_out", SIZES)
def test_dense_forward(T, n_in, n_out):
    g = torch.Generator().manual_seed(T + n_in)
    shp = abi.MoeShape.of(T, 1, 1, 64, 1, 64, "bf16", n_in)
    x = _rnd(g, T, n_in)
    w = _rnd(g, n_out, n_in, scale=n_in ** -0.5)
    out = torch.empty(T, n_out, device="cuda", dtype=torch.bfloat16)
    ws = torch.empty(abi.moe_workspace_size(shp), dtype=torch.uint8, device="cuda")
    abi.moe_latent_proj(shp, n_in, n_out, x, w, out, ws)
    torch.cuda.synchronize()
    ref = O.latent_project(f64(x), f64(w))
    assert rel_frob(f64(out), ref) < 5e-3
    assert abi.moe_check_device_status() == 0


@pytest.mark.parametrize("T,n_in,n_out", SIZES)
@pytest.mark.parametrize("accumulate", [False, True])
def test_dense_backward(T, n_in, n_out, accumulate):
    g = torch.Generator().manual_seed(7 * T + n_out)
    shp = abi.MoeShape.of(T, 1, 1, 64, 1, 64, "bf16", n_in)
    x = _rnd(g, T, n_in)
    w = _rnd(g, n_out, n_in, scale=n_in ** -0.5)
    dout = _rnd(g, T, n_out)
    din0 = _rnd(g, T, n_in)
    din = din0.clone()
    dw = torch.empty(n_out, n_in, device="cuda", dtype=torch.float32)
    ws = torch.empty(abi.moe_workspace_size(shp), dtype=torch.uint8, device="cuda")
    abi.moe_latent_proj_bwd(shp, n_in, n_out, dout, x, w, din, accumulate, dw, ws)
    torch.cuda.synchronize()
    ref_din, ref_dw = O.latent_project_bwd(f64(dout), f64(x), f64(w))
    if accumulate:
        ref_din = ref_din + f64(din0)
    assert rel_frob(f64(din), ref_din) < 5e-3
    assert rel_frob(f64(dw), ref_dw) < 1e-4
    assert abi.moe_check_device_status() == 0
