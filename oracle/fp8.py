"""Float64 reference for the low-precision dispatch payload (Sec. 1, levers:
lower-precision communication, b_x in Eq. 1; Sec. 6 mentions FP8 / NVFP4).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

The paper names the lever, not a format.  Readings (each listed with its
reason in the design notes):
  FP1  payload format: FP8 E4M3 (1 sign bit, 4 exponent bits with bias 7,
       3 mantissa bits, no infinities, S.1111.111 is NaN, largest finite 448),
       one code per hidden element, so b_x = 1 byte;
  FP2  one scale per dispatched row: the smallest power of two s = 2^e,
       e >= -126, with max_i |x_i| <= 448 s (s = 1 for an all-zero row); the
       code of x_i is the E4M3 value nearest to x_i / s, ties to the even code,
       saturating at +-448, sign kept (also for zero); the receiver uses
       code * s, which a power-of-two s makes exact in bf16;
  FP3  the backward pass treats the quantization as the identity for the
       gradient (straight-through): the expert weight gradients see the
       dequantized rows, the input gradient flows to x unchanged.
"""
from __future__ import annotations

import math

import numpy as np

__all__ = ["e4m3_value", "e4m3_table", "e4m3_quantize", "e4m3_quantize_array", "fp8_row_scale",
           "fp8_quantize_rows", "fp8_dequantize_rows"]

E4M3_MAX = 448.0


def e4m3_value(code: int) -> float:
    """Value of an 8-bit E4M3 code by the format's definition (FP1)."""
    s = -1.0 if code & 0x80 else 1.0
    e = (code >> 3) & 0xF
    m = code & 0x7
    if e == 0xF and m == 0x7:
        return math.nan
    if e == 0:
        return s * (m / 8.0) * 2.0 ** -6
    return s * (1.0 + m / 8.0) * 2.0 ** (e - 7)


def e4m3_table():
    """(codes, values) of the non-negative finite codes, ordered by value."""
    codes = [c for c in range(0x80) if not math.isnan(e4m3_value(c))]
    return codes, [e4m3_value(c) for c in codes]


_CODES, _VALS = e4m3_table()


def e4m3_quantize(v: float) -> int:
    """Nearest E4M3 code to v (ties to the even code, saturating, sign kept)."""
    neg = math.copysign(1.0, v) < 0
    a = abs(v)
    if a >= E4M3_MAX:
        code = _CODES[-1]
    else:
        best, best_d = None, None
        for c, val in zip(_CODES, _VALS):
            d = abs(val - a)
            if best is None or d < best_d or (d == best_d and (c & 1) == 0):
                best, best_d = c, d
        code = best
    return code | (0x80 if neg else 0)


_VARR = np.array(_VALS)
_CARR = np.array(_CODES, dtype=np.int64)


def e4m3_quantize_array(v: np.ndarray) -> np.ndarray:
    """e4m3_quantize over an array: the two table values around |v| (sorted
    search), the nearer one, ties to the even code; same rules as the scalar."""
    v = np.asarray(v, dtype=np.float64)
    a = np.minimum(np.abs(v), E4M3_MAX)
    hi = np.clip(np.searchsorted(_VARR, a, side="left"), 0, len(_VARR) - 1)
    lo = np.clip(hi - 1, 0, len(_VARR) - 1)
    d_lo = np.abs(a - _VARR[lo])
    d_hi = np.abs(_VARR[hi] - a)
    pick_hi = (d_hi < d_lo) | ((d_hi == d_lo) & ((_CARR[hi] & 1) == 0))
    code = np.where(pick_hi, _CARR[hi], _CARR[lo])
    neg = np.signbit(v)
    return (code | np.where(neg, 0x80, 0)).astype(np.uint8)


def fp8_row_scale(row: np.ndarray) -> float:
    """FP2: the smallest power of two s = 2^e, e >= -126, with max |x| <= 448 s."""
    amax = float(np.max(np.abs(row))) if row.size else 0.0
    if amax == 0.0:
        return 1.0
    e = -126
    while amax > E4M3_MAX * 2.0 ** e:
        e += 1
    return 2.0 ** e


def fp8_quantize_rows(x: np.ndarray):
    """Rows of x [R, D] -> (codes uint8 [R, D], scales float64 [R])."""
    R, D = x.shape
    codes = np.empty((R, D), dtype=np.uint8)
    scales = np.empty(R)
    for r in range(R):
        s = fp8_row_scale(x[r])
        scales[r] = s
        codes[r] = e4m3_quantize_array(x[r] / s)
    return codes, scales


def fp8_dequantize_rows(codes: np.ndarray, scales: np.ndarray) -> np.ndarray:
    lut = np.array([e4m3_value(c) for c in range(256)])
    return lut[codes] * scales[:, None]
