"""Host-side checks of the C ABI: the library builds and loads, exports every
symbol include/moe.h declares, and validates arguments before touching a GPU.
No test here launches a kernel."""
import ctypes
import os
import re
import shutil

import pytest

import oracle as O
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"),
                                reason="nvcc is needed to build the library")


@pytest.fixture(scope="module")
def L():
    from paper_2608_28511_gb300 import _build, abi
    _build.build()
    return abi


def _declared_symbols():
    text = open(os.path.join(ROOT, "include", "moe.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(moe_[a-z0-9_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(L):
    syms = _declared_symbols()
    assert len(syms) >= 20
    lib = ctypes.CDLL(L.LIB_PATH)
    for s in syms:
        assert hasattr(lib, s), s
    assert sorted(L.EXPORTS) == syms


def _prototypes():
    """{name: number of parameters} of every function include/moe.h declares."""
    text = open(os.path.join(ROOT, "include", "moe.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    out = {}
    for m in re.finditer(r"\b(moe_[a-z0-9_]+)\s*\(([^)]*)\)\s*;", text):
        params = m.group(2).strip()
        out[m.group(1)] = 0 if params in ("", "void") else params.count(",") + 1
    return out


def test_binding_signatures_match_the_header(L):
    """Each ctypes signature of the binding has as many arguments as the C
    prototype (a missing or extra argument would shift every later one)."""
    protos = _prototypes()
    assert sorted(protos) == sorted(L.EXPORTS)
    for name, (args, _res) in L._SIGS.items():
        assert len(args) == protos[name], (name, len(args), protos[name])


def test_version_and_strerror(L):
    assert L.moe_version() >= 100
    for st in (0, -1, -2, -3, -4, -5, -6, -7, -8):
        assert L.moe_strerror(st)
    assert L.moe_strerror(-99) == "unknown status"


@pytest.mark.parametrize("name", ["C1", "C2", "C3", "C4", "C5"])
def test_eq1_bytes_matches_oracle(L, name):
    w = synth.get(name)
    shp = L.MoeShape.from_workload(w)
    assert L.moe_eq1_bytes(shp) == O.eq1_bytes(w.S, w.GBS, w.K, w.D, w.b_x, 4)


def test_workspace_size_is_positive_and_monotone(L):
    small = L.moe_workspace_size(L.MoeShape.of(128, 2, 2, 128, 8, 256, "f32"))
    big = L.moe_workspace_size(L.MoeShape.of(4096, 2, 6, 2048, 64, 1024, "bf16"))
    assert 0 < small < big
    # the backward's dH scratch [T*K, 2F] dominates for the full-size layer
    assert big >= 8192 * 6 * 2 * 1024 * 2


@pytest.mark.parametrize("bad,status", [
    (dict(K=0), -1), (dict(K=9, E=8), -1), (dict(E=300), -1), (dict(K=17, E=32), -1), (dict(D=100), -1),
    (dict(F=96), -1), (dict(H=100), -1), (dict(S=0), -1), (dict(x_dtype=7), -2),
    (dict(S=1 << 20, GBS=1 << 10, K=8), -1),
])
def test_shape_validation(L, bad, status):
    args = dict(S=128, GBS=2, K=2, D=128, E=8, F=256, x_dtype=1, H=0)
    args.update(bad)
    shp = L.MoeShape(args["S"], args["GBS"], args["K"], args["D"], args["E"], args["F"], args["x_dtype"], args["H"])
    n = ctypes.c_size_t(0)
    assert L.lib().moe_workspace_size(ctypes.byref(shp), ctypes.byref(n)) == status
    assert L.lib().moe_eq1_bytes(ctypes.byref(shp)) == 0


def test_null_and_misaligned_pointers_are_rejected_before_any_launch(L):
    lib = L.lib()
    shp = L.MoeShape.of(128, 2, 2, 128, 8, 256, "f32")
    sp = ctypes.byref(shp)
    assert lib.moe_topk(sp, None, None, None, None) == -4
    assert lib.moe_topk(sp, 0x1001, 0x2000, 0x3000, None) == -3
    assert lib.moe_combine(sp, 0x1000, 0x2000, 0x3000, 0x4008, None) == -3
    assert lib.moe_dispatch(sp, 0x1000, 0x2000, 0x3000, 0x4000, 0x5000, 0x6000, 0x7000, 0x8000, 0x9000, 16,
                            None) == -5
    assert lib.moe_expert_ffn(sp, 0x1000, None, 0x3000, 0x4000, 0x5000, 0x6000, 0x7000, 0, 0, None) == -4
    assert lib.moe_latent_proj(sp, 100, 128, 0x1000, 0x2000, 0x3000, 0, 0, None) == -1
    assert lib.moe_route_bwd(sp, 0x1000, 0x2000, 0x3000, 0x4000, 0x5000, 0x6000, 0x7000, 0x8000, 0x9000, 0,
                             None) == -5


def test_python_binding_raises_on_error(L):
    shp = L.MoeShape.of(128, 2, 9, 128, 8, 256, "f32")
    with pytest.raises(L.MoeError) as ei:
        L.moe_workspace_size(shp)
    assert ei.value.status == -1


def test_layer_buffer_layout_for_the_fused_backward_tails(L):
    """Host-side layout of MoeLayer (CPU tensors, no launch): with H > 0 and
    the softmax router, w_down and w_router are consecutive row ranges of one
    [D + E, H] array and dx_lat is the first D columns of [dx_lat | dz]; the
    other configurations keep separate arrays."""
    import torch
    from paper_2608_28511_gb300.layer import MoeLayer
    D, E, H = 128, 8, 256
    La = MoeLayer(64, 1, 2, D, E, 64, "bf16", H=H, device="cpu")
    assert La.latent_fused
    assert La.w_down.is_contiguous() and La.w_router.is_contiguous()
    assert La.w_down.data_ptr() == La.w_down_router.data_ptr()
    assert La.w_router.data_ptr() == La.w_down_router.data_ptr() + D * H * 2
    assert La.dx_cat.shape == (64, D + E) and La.dx_lat.data_ptr() == La.dx_cat.data_ptr()
    assert La.dx_lat.stride() == (D + E, 1)
    for kw in ({"router": "sigmoid"}, {"dtype": "f32"}):
        args = dict(dtype="bf16", H=H, device="cpu")
        args.update(kw)
        Lb = MoeLayer(64, 1, 2, D, E, 64, **args)
        assert not Lb.latent_fused and Lb.w_down_router is None and Lb.dx_lat.is_contiguous()
    Lc = MoeLayer(64, 1, 2, D, E, 64, "bf16", device="cpu")
    assert not Lc.latent_fused and Lc.w_down is None
