"""moe_dispatch_noalloc, the dispatch for callers that cannot allocate device
memory at the call (a framework that owns all device memory, or a loop that
must not pay cudaMalloc's device synchronisation), against moe_dispatch.

Collected last on purpose (file name), so a run that stops at the first
failure has run every other test first.  Both calls in a row are checked
against the workspace version: the second problem runs on the scratch array
the first one left behind.  Around every call after the first on the device,
the device's free memory and torch's reserved memory must not change.
"""
import pytest
import torch

from paper_2608_28511_gb300 import abi

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _routing(T, E, K, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    z = torch.randn(T, E, device="cuda", generator=g)
    idx = z.topk(K, dim=1).indices.to(torch.int32).contiguous()
    prob = torch.softmax(z.gather(1, idx.long()), dim=1).contiguous()
    return idx, prob


def _buffers(T, E, K, D):
    dev = "cuda"
    TK = T * K
    return dict(off=torch.empty(E + 1, dtype=torch.int32, device=dev),
                ros=torch.empty(TK, dtype=torch.int32, device=dev),
                tor=torch.empty(TK, dtype=torch.int32, device=dev),
                xp=torch.empty(TK, D, dtype=torch.bfloat16, device=dev),
                pp=torch.empty(TK, dtype=torch.float32, device=dev))


def _device_memory():
    """Free bytes on the device (driver view) and bytes reserved by torch's caching allocator."""
    torch.cuda.synchronize()
    return torch.cuda.mem_get_info()[0], torch.cuda.memory_reserved()


@pytest.fixture(scope="module")
def _warm():
    # The first call on a device loads the library's module there and places
    # the fixed array; the calls after it are the ones that allocate nothing.
    T, E, K, D = 64, 8, 2, 64
    shp = abi.MoeShape.of(T, 1, K, D, E, 64, "bf16")
    x = torch.zeros(T, D, dtype=torch.bfloat16, device="cuda")
    idx, prob = _routing(T, E, K, 0)
    b = _buffers(T, E, K, D)
    abi.moe_dispatch_noalloc(shp, x, idx, prob, b["off"], b["ros"], b["tor"], b["xp"], b["pp"])
    torch.cuda.synchronize()


# The second pair's last call sits exactly at the array's limit:
# E * ceil(T*K / 2048) = 256 * 1024 = 262144 int32 counts.
@pytest.mark.parametrize("calls", [[(4096, 64, 6, 256, 1), (300, 16, 4, 128, 2)],
                                   [(64, 8, 2, 64, 3), (8192, 128, 8, 128, 4)],
                                   [(8192, 128, 8, 128, 5), (262144, 256, 8, 64, 6)]])
def test_noalloc_dispatch_matches_workspace_dispatch_on_two_calls_in_a_row(calls, _warm):
    for T, E, K, D, seed in calls:
        shp = abi.MoeShape.of(T, 1, K, D, E, 64, "bf16")
        x = torch.randn(T, D, device="cuda").to(torch.bfloat16)
        idx, prob = _routing(T, E, K, seed)
        ref = _buffers(T, E, K, D)
        ws = torch.empty(abi.moe_workspace_size(shp), dtype=torch.uint8, device="cuda")
        abi.moe_dispatch(shp, x, idx, prob, ref["off"], ref["ros"], ref["tor"], ref["xp"], ref["pp"], ws)
        out = _buffers(T, E, K, D)
        before = _device_memory()
        abi.moe_dispatch_noalloc(shp, x, idx, prob, out["off"], out["ros"], out["tor"], out["xp"], out["pp"])
        after = _device_memory()
        assert after == before, f"device memory changed across the call: {before} -> {after}"
        for k in ("off", "ros", "tor", "xp", "pp"):
            assert torch.equal(out[k], ref[k]), k       # index work and copies: bit-exact
        assert abi.moe_check_device_status() == 0
        del ws, ref, out


def test_noalloc_dispatch_rejects_shapes_beyond_its_fixed_scratch():
    # E * ceil(T*K / 2048) = 256 * 1025 > 262144: refused before anything is enqueued
    shp = abi.MoeShape.of(2048 * 1025 // 8, 1, 8, 64, 256, 64, "bf16")
    with pytest.raises(abi.MoeError) as ei:
        abi.moe_dispatch_noalloc(shp, 16, 16, 16, 16, 16, 16, None, 16)
    assert ei.value.status == -9
