"""MoeLayer.run_host: steps on batches in pinned host memory.  The copies in
and out overlap the neighbouring steps' compute, on two copy streams and two
alternating device buffer sets.  Each batch's y and dx must equal those of a
plain device step on the same inputs, bit for bit, with and without the
captured graphs.  The batches differ from one another, so a copy that races
its step shows up."""
import pytest
import torch

import synth
from tests.gpu_util import make_layer

pytestmark = pytest.mark.gpu

CASES = [
    synth.Workload("hp_bf16", S=384, GBS=2, D=256, E=16, K=4, F=256),
    synth.Workload("hp_latent", S=256, GBS=2, D=256, E=32, K=4, F=192, H=512),
]


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("graphs", [True, False], ids=["graphs", "eager"])
@pytest.mark.parametrize("w", CASES, ids=[c.name for c in CASES])
def test_run_host_matches_device_steps(w, graphs):
    inp = synth.make_inputs(w)
    L, _ = make_layer(w, inputs=inp)
    ref, _ = make_layer(w, inputs=inp)
    g = torch.Generator().manual_seed(3)
    n = 5
    batches = []
    for _ in range(n):
        x = torch.randn(tuple(L.x.shape), generator=g).to(L.x.dtype).pin_memory()
        dy = torch.randn(tuple(L.dy.shape), generator=g).to(L.dy.dtype).pin_memory()
        batches.append((x, dy, torch.empty_like(x).pin_memory(), torch.empty_like(dy).pin_memory()))
    L.prepare_host_pipeline(graphs=graphs)
    L.run_host(batches)
    torch.cuda.synchronize()
    for x, dy, y_h, dx_h in batches:
        ref.x.copy_(x)
        ref.dy.copy_(dy)
        ref.step()
        torch.cuda.synchronize()
        assert torch.equal(y_h, ref.y.cpu())
        assert torch.equal(dx_h, ref.dx.cpu())
    # the layer is left bound to its first buffer set and still steps on the device
    L.x.copy_(batches[0][0])
    L.dy.copy_(batches[0][1])
    L.step()
    torch.cuda.synchronize()
    assert torch.equal(L.y.cpu(), batches[0][2])
