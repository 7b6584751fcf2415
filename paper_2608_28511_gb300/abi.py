"""ctypes binding for ``libmoe.so`` (declared in ``include/moe.h``).

Argument marshalling only: every function here passes device pointers and
sizes straight to the C entry point of the same name and raises ``MoeError``
on a non-zero status.  Tensors may be given as torch tensors (their
``data_ptr()`` is passed) or as raw integer addresses.  Nothing here computes
any part of the layer; if the library is missing the import of a function
fails loudly instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libmoe.so")

MOE_BF16 = 0
MOE_F32 = 1

STATUS = {
    0: "MOE_OK", -1: "MOE_ERR_SHAPE", -2: "MOE_ERR_DTYPE", -3: "MOE_ERR_ALIGN", -4: "MOE_ERR_NULL",
    -5: "MOE_ERR_WORKSPACE", -6: "MOE_ERR_CUDA", -7: "MOE_ERR_DEVICE", -8: "MOE_ERR_UNSUPPORTED",
    -9: "MOE_ERR_TOO_LARGE",
}

# Every symbol include/moe.h declares.
EXPORTS = (
    "moe_workspace_size", "moe_route", "moe_topk", "moe_dispatch", "moe_expert_ffn", "moe_combine",
    "moe_combine_bwd", "moe_expert_ffn_bwd", "moe_dispatch_bwd", "moe_route_bwd", "moe_latent_proj",
    "moe_latent_proj_bwd", "moe_pack_w1", "moe_eq1_bytes", "moe_check_device_status",
    "moe_device_status_word", "moe_last_cuda_error", "moe_strerror", "moe_version", "moe_prof_enable",
    "moe_prof_reset", "moe_prof_count", "moe_prof_get", "moe_launch_count", "moe_dispatch_noalloc",
    "moe_ce_composition", "moe_ce_layer_pattern", "moe_route_sigmoid", "moe_route_sigmoid_bwd",
    "moe_shared_expert", "moe_shared_expert_bwd", "moe_expert_ffn_gather", "moe_expert_ffn_bwd_gather",
    "moe_dispatch_fp8", "moe_dequant_rows", "moe_dispatch_nvfp4", "moe_dequant_nvfp4", "moe_dispatch_route_bwd",
    "moe_latent_route_bwd", "moe_topk_sigmoid",
)


class MoeError(RuntimeError):
    def __init__(self, fn: str, status: int, msg: str):
        super().__init__(f"{fn} failed: {STATUS.get(status, status)} ({msg})")
        self.status = status


class MoeShape(ctypes.Structure):
    """moe_shape_t: Eq. 1 symbols S, GBS, K, D plus E, F, the b_x dtype and H."""
    _fields_ = [("S", ctypes.c_int64), ("GBS", ctypes.c_int64), ("K", ctypes.c_int32), ("D", ctypes.c_int32),
                ("E", ctypes.c_int32), ("F", ctypes.c_int32), ("x_dtype", ctypes.c_int32), ("H", ctypes.c_int32)]

    @classmethod
    def of(cls, S, GBS, K, D, E, F, dtype="bf16", H=0) -> "MoeShape":
        dt = MOE_BF16 if dtype in ("bf16", MOE_BF16) else MOE_F32
        return cls(int(S), int(GBS), int(K), int(D), int(E), int(F), dt, int(H))

    @classmethod
    def from_workload(cls, w, T: Optional[int] = None) -> "MoeShape":
        """From an object with S, GBS, K, D, E, F, dtype, H (T overrides S*GBS as S=T, GBS=1)."""
        if T is not None:
            return cls.of(T, 1, w.K, w.D, w.E, w.F, w.dtype, w.H)
        return cls.of(w.S, w.GBS, w.K, w.D, w.E, w.F, w.dtype, w.H)

    @property
    def T(self) -> int:
        return self.S * self.GBS


_lib = None

_VP = ctypes.c_void_p
_SZ = ctypes.c_size_t
_I32 = ctypes.c_int32
_F32 = ctypes.c_float
_SHP = ctypes.POINTER(MoeShape)

_SIGS = {
    "moe_workspace_size": ([_SHP, ctypes.POINTER(_SZ)], ctypes.c_int),
    "moe_route": ([_SHP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP], ctypes.c_int),
    "moe_topk": ([_SHP, _VP, _VP, _VP, _VP], ctypes.c_int),
    "moe_dispatch": ([_SHP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP], ctypes.c_int),
    "moe_expert_ffn": ([_SHP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP], ctypes.c_int),
    "moe_combine": ([_SHP, _VP, _VP, _VP, _VP, _VP], ctypes.c_int),
    "moe_combine_bwd": ([_SHP, _VP, _VP, _VP, _VP, _VP, _VP, _VP], ctypes.c_int),
    "moe_expert_ffn_bwd": ([_SHP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP], ctypes.c_int),
    "moe_dispatch_bwd": ([_SHP, _VP, _VP, _VP, _VP, _VP, _VP], ctypes.c_int),
    "moe_route_bwd": ([_SHP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP], ctypes.c_int),
    "moe_dispatch_route_bwd": ([_SHP] + [_VP] * 12 + [_SZ, _VP], ctypes.c_int),
    "moe_latent_route_bwd": ([_SHP] + [_VP] * 14 + [_SZ, _VP], ctypes.c_int),
    "moe_route_sigmoid": ([_SHP, _VP, _VP, _VP, _F32, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP], ctypes.c_int),
    "moe_topk_sigmoid": ([_SHP, _VP, _VP, _F32, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP], ctypes.c_int),
    "moe_route_sigmoid_bwd": ([_SHP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _F32, _F32, _VP, _VP, _VP, _VP, _SZ, _VP],
                              ctypes.c_int),
    "moe_expert_ffn_gather": ([_SHP] + [_VP] * 9 + [_SZ, _VP], ctypes.c_int),
    "moe_dispatch_fp8": ([_SHP] + [_VP] * 10 + [_SZ, _VP], ctypes.c_int),
    "moe_dequant_rows": ([_SHP, _VP, _VP, _VP, _VP], ctypes.c_int),
    "moe_dispatch_nvfp4": ([_SHP] + [_VP] * 11 + [_SZ, _VP], ctypes.c_int),
    "moe_dequant_nvfp4": ([_SHP, _VP, _VP, _VP, _VP, _VP], ctypes.c_int),
    "moe_expert_ffn_bwd_gather": ([_SHP] + [_VP] * 12 + [_SZ, _VP], ctypes.c_int),
    "moe_shared_expert": ([_SHP, _I32, _VP, _VP, _VP, _VP, _VP, _VP, _VP], ctypes.c_int),
    "moe_shared_expert_bwd": ([_SHP, _I32] + [_VP] * 11, ctypes.c_int),
    "moe_latent_proj": ([_SHP, _I32, _I32, _VP, _VP, _VP, _VP, _SZ, _VP], ctypes.c_int),
    "moe_latent_proj_bwd": ([_SHP, _I32, _I32, _VP, _VP, _VP, _VP, _I32, _VP, _VP, _SZ, _VP], ctypes.c_int),
    "moe_pack_w1": ([_SHP, _VP, _VP, _VP, _VP], ctypes.c_int),
    "moe_eq1_bytes": ([_SHP], ctypes.c_uint64),
    "moe_check_device_status": ([_VP], ctypes.c_int),
    "moe_device_status_word": ([_VP, ctypes.POINTER(ctypes.c_uint32)], ctypes.c_int),
    "moe_last_cuda_error": ([], ctypes.c_int),
    "moe_strerror": ([ctypes.c_int], ctypes.c_char_p),
    "moe_version": ([], ctypes.c_int),
    "moe_prof_enable": ([ctypes.c_int], ctypes.c_int),
    "moe_prof_reset": ([], ctypes.c_int),
    "moe_prof_count": ([], ctypes.c_int),
    "moe_prof_get": ([ctypes.c_int, ctypes.POINTER(ctypes.c_char_p), ctypes.POINTER(ctypes.c_int),
                      ctypes.POINTER(ctypes.c_double)], ctypes.c_int),
    "moe_launch_count": ([], ctypes.c_uint64),
    "moe_dispatch_noalloc": ([_SHP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP], ctypes.c_int),
    "moe_ce_composition": ([_I32, _I32, _I32, ctypes.c_double] + [ctypes.POINTER(_I32)] * 4, ctypes.c_int),
    "moe_ce_layer_pattern": ([_I32, _I32, _I32, _I32, ctypes.c_char_p, _SZ, ctypes.c_char_p, _SZ, ctypes.c_char_p,
                              _SZ], ctypes.c_int),
}


def lib() -> ctypes.CDLL:
    """Load libmoe.so (built by ``__graft_entry__.build()``); raises if absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build() "
                               "(there is no fallback implementation)")
        L = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in _SIGS.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = res
        _lib = L
    return _lib


def _p(t) -> Optional[int]:
    """Device address of a tensor (or pass an int / None through)."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not t.is_contiguous():
        raise ValueError("tensors passed to the MoE library must be contiguous")
    return t.data_ptr()


def _nbytes(t) -> int:
    if t is None:
        return 0
    return t.numel() * t.element_size()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(fn: str, st: int) -> None:
    if st != 0:
        msg = lib().moe_strerror(st).decode()
        if st == -6:
            msg += f"; cudaError {lib().moe_last_cuda_error()}"
        raise MoeError(fn, st, msg)


def _shape(shape: MoeShape):
    return ctypes.byref(shape)


# ---------------------------------------------------------------------------
# Entry points (same names and argument order as include/moe.h)
# ---------------------------------------------------------------------------

def moe_workspace_size(shape: MoeShape) -> int:
    n = _SZ(0)
    _check("moe_workspace_size", lib().moe_workspace_size(_shape(shape), ctypes.byref(n)))
    return n.value


def moe_route(shape, x, w_router, bias, logits, topk_idx, topk_prob, ws, stream=None):
    _check("moe_route", lib().moe_route(_shape(shape), _p(x), _p(w_router), _p(bias), _p(logits), _p(topk_idx),
                                        _p(topk_prob), _p(ws), _nbytes(ws), _stream(stream)))


def moe_topk(shape, logits, topk_idx, topk_prob, stream=None):
    _check("moe_topk", lib().moe_topk(_shape(shape), _p(logits), _p(topk_idx), _p(topk_prob), _stream(stream)))


def moe_dispatch(shape, x, topk_idx, topk_prob, expert_offsets, row_of_slot, token_of_row, x_perm, prob_perm, ws,
                 stream=None):
    _check("moe_dispatch", lib().moe_dispatch(_shape(shape), _p(x), _p(topk_idx), _p(topk_prob), _p(expert_offsets),
                                              _p(row_of_slot), _p(token_of_row), _p(x_perm), _p(prob_perm), _p(ws),
                                              _nbytes(ws), _stream(stream)))


def moe_dispatch_fp8(shape, x, topk_idx, topk_prob, expert_offsets, row_of_slot, token_of_row, x_perm_q,
                     x_scale_perm, prob_perm, ws, stream=None):
    _check("moe_dispatch_fp8", lib().moe_dispatch_fp8(
        _shape(shape), _p(x), _p(topk_idx), _p(topk_prob), _p(expert_offsets), _p(row_of_slot), _p(token_of_row),
        _p(x_perm_q), _p(x_scale_perm), _p(prob_perm), _p(ws), _nbytes(ws), _stream(stream)))


def moe_dequant_rows(shape, x_perm_q, x_scale_perm, x_perm, stream=None):
    _check("moe_dequant_rows", lib().moe_dequant_rows(_shape(shape), _p(x_perm_q), _p(x_scale_perm), _p(x_perm),
                                                      _stream(stream)))


def moe_dispatch_nvfp4(shape, x, topk_idx, topk_prob, expert_offsets, row_of_slot, token_of_row, x_perm_q,
                       x_bscale_perm, x_rscale_perm, prob_perm, ws, stream=None):
    _check("moe_dispatch_nvfp4", lib().moe_dispatch_nvfp4(
        _shape(shape), _p(x), _p(topk_idx), _p(topk_prob), _p(expert_offsets), _p(row_of_slot), _p(token_of_row),
        _p(x_perm_q), _p(x_bscale_perm), _p(x_rscale_perm), _p(prob_perm), _p(ws), _nbytes(ws), _stream(stream)))


def moe_dequant_nvfp4(shape, x_perm_q, x_bscale_perm, x_rscale_perm, x_perm, stream=None):
    _check("moe_dequant_nvfp4", lib().moe_dequant_nvfp4(_shape(shape), _p(x_perm_q), _p(x_bscale_perm),
                                                        _p(x_rscale_perm), _p(x_perm), _stream(stream)))


def moe_dispatch_noalloc(shape, x, topk_idx, topk_prob, expert_offsets, row_of_slot, token_of_row, x_perm,
                         prob_perm, stream=None):
    """moe_dispatch without a workspace, for callers that cannot allocate device
    memory at the call (the scratch is a fixed 1 MiB array inside the library)."""
    _check("moe_dispatch_noalloc", lib().moe_dispatch_noalloc(
        _shape(shape), _p(x), _p(topk_idx), _p(topk_prob), _p(expert_offsets), _p(row_of_slot), _p(token_of_row),
        _p(x_perm), _p(prob_perm), _stream(stream)))


def moe_expert_ffn(shape, x_perm, expert_offsets, w1, w2, h_save, act_save, y_perm, ws, stream=None):
    _check("moe_expert_ffn", lib().moe_expert_ffn(_shape(shape), _p(x_perm), _p(expert_offsets), _p(w1), _p(w2),
                                                  _p(h_save), _p(act_save), _p(y_perm), _p(ws), _nbytes(ws),
                                                  _stream(stream)))


def moe_expert_ffn_gather(shape, x, token_of_row, expert_offsets, w1, w2, h_save, act_save, y_perm, ws,
                          stream=None):
    _check("moe_expert_ffn_gather", lib().moe_expert_ffn_gather(
        _shape(shape), _p(x), _p(token_of_row), _p(expert_offsets), _p(w1), _p(w2), _p(h_save), _p(act_save),
        _p(y_perm), _p(ws), _nbytes(ws), _stream(stream)))


def moe_expert_ffn_bwd_gather(shape, dy_perm, x, token_of_row, h_save, act_save, expert_offsets, w1, w2, dx_perm,
                              dw1, dw2, ws, stream=None):
    _check("moe_expert_ffn_bwd_gather", lib().moe_expert_ffn_bwd_gather(
        _shape(shape), _p(dy_perm), _p(x), _p(token_of_row), _p(h_save), _p(act_save), _p(expert_offsets), _p(w1),
        _p(w2), _p(dx_perm), _p(dw1), _p(dw2), _p(ws), _nbytes(ws), _stream(stream)))


def moe_combine(shape, y_perm, prob_perm, row_of_slot, y, stream=None):
    _check("moe_combine", lib().moe_combine(_shape(shape), _p(y_perm), _p(prob_perm), _p(row_of_slot), _p(y),
                                            _stream(stream)))


def moe_combine_bwd(shape, dy, y_perm, prob_perm, row_of_slot, dy_perm, dprob_perm, stream=None):
    _check("moe_combine_bwd", lib().moe_combine_bwd(_shape(shape), _p(dy), _p(y_perm), _p(prob_perm),
                                                    _p(row_of_slot), _p(dy_perm), _p(dprob_perm), _stream(stream)))


def moe_expert_ffn_bwd(shape, dy_perm, x_perm, h_save, act_save, expert_offsets, w1, w2, dx_perm, dw1, dw2, ws,
                       stream=None):
    _check("moe_expert_ffn_bwd", lib().moe_expert_ffn_bwd(
        _shape(shape), _p(dy_perm), _p(x_perm), _p(h_save), _p(act_save), _p(expert_offsets), _p(w1), _p(w2),
        _p(dx_perm), _p(dw1), _p(dw2), _p(ws), _nbytes(ws), _stream(stream)))


def moe_dispatch_bwd(shape, dx_perm, dprob_perm, row_of_slot, dx, dtopk_prob, stream=None):
    _check("moe_dispatch_bwd", lib().moe_dispatch_bwd(_shape(shape), _p(dx_perm), _p(dprob_perm), _p(row_of_slot),
                                                      _p(dx), _p(dtopk_prob), _stream(stream)))


def moe_dispatch_route_bwd(shape, dx_perm, dprob_perm, row_of_slot, x, w_router, topk_idx, topk_prob, dx,
                           dtopk_prob, dlogits, dw_router, ws, stream=None):
    _check("moe_dispatch_route_bwd", lib().moe_dispatch_route_bwd(
        _shape(shape), _p(dx_perm), _p(dprob_perm), _p(row_of_slot), _p(x), _p(w_router), _p(topk_idx),
        _p(topk_prob), _p(dx), _p(dtopk_prob), _p(dlogits), _p(dw_router), _p(ws), _nbytes(ws), _stream(stream)))


def moe_latent_route_bwd(shape, dx_perm, dprob_perm, row_of_slot, x, w_down_router, topk_idx, topk_prob, dx_cat,
                         dx, dtopk_prob, dlogits, dw_down, dw_router, ws, stream=None):
    _check("moe_latent_route_bwd", lib().moe_latent_route_bwd(
        _shape(shape), _p(dx_perm), _p(dprob_perm), _p(row_of_slot), _p(x), _p(w_down_router), _p(topk_idx),
        _p(topk_prob), _p(dx_cat), _p(dx), _p(dtopk_prob), _p(dlogits), _p(dw_down), _p(dw_router), _p(ws),
        _nbytes(ws), _stream(stream)))


def moe_route_bwd(shape, x, w_router, topk_idx, topk_prob, dtopk_prob, dx, dw_router, dlogits, ws, stream=None):
    _check("moe_route_bwd", lib().moe_route_bwd(_shape(shape), _p(x), _p(w_router), _p(topk_idx), _p(topk_prob),
                                                _p(dtopk_prob), _p(dx), _p(dw_router), _p(dlogits), _p(ws),
                                                _nbytes(ws), _stream(stream)))


def moe_route_sigmoid(shape, x, w_router, expert_bias, aux_coef, logits, topk_idx, topk_prob, aux_f, aux_loss, ws,
                      stream=None):
    _check("moe_route_sigmoid", lib().moe_route_sigmoid(
        _shape(shape), _p(x), _p(w_router), _p(expert_bias), float(aux_coef), _p(logits), _p(topk_idx),
        _p(topk_prob), _p(aux_f), _p(aux_loss), _p(ws), _nbytes(ws), _stream(stream)))


def moe_topk_sigmoid(shape, logits, expert_bias, aux_coef, select_keys, topk_idx, topk_prob, aux_f, aux_loss, ws,
                     stream=None):
    _check("moe_topk_sigmoid", lib().moe_topk_sigmoid(
        _shape(shape), _p(logits), _p(expert_bias), float(aux_coef), _p(select_keys), _p(topk_idx), _p(topk_prob),
        _p(aux_f), _p(aux_loss), _p(ws), _nbytes(ws), _stream(stream)))


def moe_route_sigmoid_bwd(shape, x, w_router, logits, topk_idx, topk_prob, dtopk_prob, aux_f, aux_coef, aux_grad,
                          dx, dw_router, dlogits, ws, stream=None):
    _check("moe_route_sigmoid_bwd", lib().moe_route_sigmoid_bwd(
        _shape(shape), _p(x), _p(w_router), _p(logits), _p(topk_idx), _p(topk_prob), _p(dtopk_prob), _p(aux_f),
        float(aux_coef), float(aux_grad), _p(dx), _p(dw_router), _p(dlogits), _p(ws), _nbytes(ws),
        _stream(stream)))


def moe_shared_expert(shape, F_s, x, w_s1, w_s2, h_save, act_save, y, stream=None):
    _check("moe_shared_expert", lib().moe_shared_expert(_shape(shape), int(F_s), _p(x), _p(w_s1), _p(w_s2),
                                                        _p(h_save), _p(act_save), _p(y), _stream(stream)))


def moe_shared_expert_bwd(shape, F_s, dy, x, h_save, act_save, w_s1, w_s2, dh, dx, dw_s1, dw_s2, stream=None):
    _check("moe_shared_expert_bwd", lib().moe_shared_expert_bwd(
        _shape(shape), int(F_s), _p(dy), _p(x), _p(h_save), _p(act_save), _p(w_s1), _p(w_s2), _p(dh), _p(dx),
        _p(dw_s1), _p(dw_s2), _stream(stream)))


def moe_latent_proj(shape, n_in, n_out, x, w, out, ws, stream=None):
    _check("moe_latent_proj", lib().moe_latent_proj(_shape(shape), int(n_in), int(n_out), _p(x), _p(w), _p(out),
                                                    _p(ws), _nbytes(ws), _stream(stream)))


def moe_latent_proj_bwd(shape, n_in, n_out, dout, x, w, din, accumulate, dw, ws, stream=None):
    _check("moe_latent_proj_bwd", lib().moe_latent_proj_bwd(
        _shape(shape), int(n_in), int(n_out), _p(dout), _p(x), _p(w), _p(din), int(bool(accumulate)), _p(dw),
        _p(ws), _nbytes(ws), _stream(stream)))


def moe_pack_w1(shape, w_gate, w_up, w1, stream=None):
    _check("moe_pack_w1", lib().moe_pack_w1(_shape(shape), _p(w_gate), _p(w_up), _p(w1), _stream(stream)))


def moe_eq1_bytes(shape: MoeShape) -> int:
    return int(lib().moe_eq1_bytes(_shape(shape)))


def moe_check_device_status(stream=None) -> int:
    return int(lib().moe_check_device_status(_stream(stream)))


def moe_device_status_word(stream=None) -> int:
    w = ctypes.c_uint32(0)
    _check("moe_device_status_word", lib().moe_device_status_word(_stream(stream), ctypes.byref(w)))
    return int(w.value)


def moe_strerror(status: int) -> str:
    return lib().moe_strerror(int(status)).decode()


def moe_version() -> int:
    return int(lib().moe_version())


def moe_launch_count() -> int:
    return int(lib().moe_launch_count())


def moe_prof_enable(on: bool) -> None:
    lib().moe_prof_enable(int(bool(on)))


def moe_prof_reset() -> None:
    lib().moe_prof_reset()


def moe_prof_read() -> dict:
    """{kernel name: (launches, total device ms)} accumulated while enabled."""
    L = lib()
    out = {}
    for i in range(L.moe_prof_count()):
        name = ctypes.c_char_p()
        n = ctypes.c_int(0)
        ms = ctypes.c_double(0.0)
        _check("moe_prof_get", L.moe_prof_get(i, ctypes.byref(name), ctypes.byref(n), ctypes.byref(ms)))
        out[name.value.decode()] = (n.value, ms.value)
    return out


# ---------------------------------------------------------------------------
# CE-MoE layout tools (host only)
# ---------------------------------------------------------------------------

def moe_ce_composition(a_star: int, b_star: int, c_star: int, alpha: float) -> tuple:
    """(a, b, c, d): Mamba, MoE, attention and dense-FFN block counts (Sec. 4.1)."""
    out = [ctypes.c_int32(0) for _ in range(4)]
    _check("moe_ce_composition", lib().moe_ce_composition(int(a_star), int(b_star), int(c_star), float(alpha),
                                                          *[ctypes.byref(o) for o in out]))
    return tuple(o.value for o in out)


def moe_ce_layer_pattern(a: int, b: int, c: int, d: int) -> tuple:
    """(pattern, virtual-block order, decorated pattern) of Algorithm 1 (Sec. 4.2)."""
    cap = 4 * (a + b + c + d) + 64
    bufs = [ctypes.create_string_buffer(cap) for _ in range(3)]
    n = lib().moe_ce_layer_pattern(int(a), int(b), int(c), int(d), bufs[0], cap, bufs[1], cap, bufs[2], cap)
    if n < 0:
        _check("moe_ce_layer_pattern", n)
    return tuple(b_.value.decode() for b_ in bufs)
