"""The dense GEMM shapes of the library (LatentMoE projections and their
backward) against plain PyTorch fp32 on the GPU, over sizes with ragged M, N
and K tiles.  These exercise the tensor-core engine's K-major x K-major,
K-major x MN-major and MN-major x MN-major operand paths and its store,
accumulate and fp32 epilogues."""
import pytest
import torch

from paper_2608_28511_gb300 import abi

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _rel(a, b):
    a, b = a.float(), b.float()
    return float((a - b).norm() / b.norm().clamp_min(1e-30))


SIZES = [(1, 64, 64), (100, 192, 320), (300, 512, 256), (1000, 320, 1024), (2048, 1024, 64), (129, 64, 576)]


@pytest.mark.parametrize("T,n_in,n_out", SIZES)
def test_dense_forward(T, n_in, n_out):
    g = torch.Generator(device="cuda").manual_seed(T + n_in)
    shp = abi.MoeShape.of(T, 1, 1, 64, 1, 64, "bf16", n_in)
    x = torch.randn(T, n_in, device="cuda", generator=g).to(torch.bfloat16)
    w = (torch.randn(n_out, n_in, device="cuda", generator=g) / n_in ** 0.5).to(torch.bfloat16)
    out = torch.empty(T, n_out, device="cuda", dtype=torch.bfloat16)
    ws = torch.empty(abi.moe_workspace_size(shp), dtype=torch.uint8, device="cuda")
    abi.moe_latent_proj(shp, n_in, n_out, x, w, out, ws)
    ref = x.float() @ w.float().T
    torch.cuda.synchronize()
    assert _rel(out, ref) < 5e-3
    assert abi.moe_check_device_status() == 0


@pytest.mark.parametrize("T,n_in,n_out", SIZES)
@pytest.mark.parametrize("accumulate", [False, True])
def test_dense_backward(T, n_in, n_out, accumulate):
    g = torch.Generator(device="cuda").manual_seed(7 * T + n_out)
    shp = abi.MoeShape.of(T, 1, 1, 64, 1, 64, "bf16", n_in)
    x = torch.randn(T, n_in, device="cuda", generator=g).to(torch.bfloat16)
    w = (torch.randn(n_out, n_in, device="cuda", generator=g) / n_in ** 0.5).to(torch.bfloat16)
    dout = torch.randn(T, n_out, device="cuda", generator=g).to(torch.bfloat16)
    din0 = torch.randn(T, n_in, device="cuda", generator=g).to(torch.bfloat16)
    din = din0.clone()
    dw = torch.empty(n_out, n_in, device="cuda", dtype=torch.float32)
    ws = torch.empty(abi.moe_workspace_size(shp), dtype=torch.uint8, device="cuda")
    abi.moe_latent_proj_bwd(shp, n_in, n_out, dout, x, w, din, accumulate, dw, ws)
    ref_din = dout.float() @ w.float()
    if accumulate:
        ref_din = ref_din + din0.float()
    ref_dw = dout.float().T @ x.float()
    torch.cuda.synchronize()
    assert _rel(din, ref_din) < 5e-3
    assert _rel(dw, ref_dw) < 1e-4
    assert abi.moe_check_device_status() == 0
