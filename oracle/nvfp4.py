"""Float64 reference for the NVFP4 dispatch payload (Sec. 1: lower-precision
communication, b_x of Eq. 1; Sec. 6 names FP8 and NVFP4).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

The paper names the format, not a scaling recipe.  Readings (each listed
with its reason in the design notes):
  NV1  element format: E2M1 (1 sign bit, 2 exponent bits with bias 1,
       1 mantissa bit; magnitudes 0, 0.5, 1, 1.5, 2, 3, 4, 6), two codes per
       byte, element 2j in the low nibble of byte j;
  NV2  two-level scaling of each dispatched row x (D elements):
       * a row scale g = 2^e, the smallest with e >= -126 and
         max_i |x_i| <= 6 * 448 * g (g = 1 for an all-zero row);
       * per block b of 16 consecutive elements, a scale s_b = the E4M3 value
         nearest to r_b = max_{i in b} |x_i| / (6 g) (ties to the even code,
         saturating at 448), with r_b computed in fp32;
       * code_i = the E2M1 value nearest to x_i / (s_b g) computed in fp32
         (ties to the even code, saturating at +-6, sign kept); a block with
         s_b = 0 gets zero codes.
       The receiver uses code * s_b * g, which is exact in bf16 (at most 6
       significant bits times a power of two).  Both sides take every
       rounding decision from the same fp32 value;
  NV3  the backward pass treats the quantization as the identity for the
       gradient (straight-through), as for the FP8 payload.
Payload per dispatched row: D / 2 code bytes + D / 16 scale bytes + 4 bytes.
"""
from __future__ import annotations

import math

import numpy as np

from .fp8 import e4m3_quantize_array, e4m3_value

__all__ = ["e2m1_value", "e2m1_table", "e2m1_quantize", "e2m1_quantize_array", "nvfp4_row_scale",
           "nvfp4_quantize_rows", "nvfp4_dequantize_rows", "NVFP4_BLOCK"]

NVFP4_BLOCK = 16
E2M1_MAX = 6.0
E4M3_MAX = 448.0


def e2m1_value(code: int) -> float:
    """Value of a 4-bit E2M1 code by the format's definition (NV1)."""
    s = -1.0 if code & 0x8 else 1.0
    e = (code >> 1) & 0x3
    m = code & 0x1
    if e == 0:
        return s * m * 0.5  # subnormal: m * 2^(1 - bias) / 2
    return s * (1.0 + m / 2.0) * 2.0 ** (e - 1)


def e2m1_table():
    """(codes, values) of the non-negative codes, ordered by value."""
    codes = list(range(8))
    return codes, [e2m1_value(c) for c in codes]


_CODES, _VALS = e2m1_table()


def e2m1_quantize(v: float) -> int:
    """Nearest E2M1 code to v (ties to the even code, saturating, sign kept)."""
    neg = math.copysign(1.0, v) < 0
    a = abs(v)
    if a >= E2M1_MAX:
        code = _CODES[-1]
    else:
        best, best_d = None, None
        for c, val in zip(_CODES, _VALS):
            d = abs(val - a)
            if best is None or d < best_d or (d == best_d and (c & 1) == 0):
                best, best_d = c, d
        code = best
    return code | (0x8 if neg else 0)


_VARR = np.array(_VALS)
_CARR = np.array(_CODES, dtype=np.int64)


def e2m1_quantize_array(v: np.ndarray) -> np.ndarray:
    """e2m1_quantize over an array (the two table values around |v|, the
    nearer one, ties to the even code); same rules as the scalar form."""
    v = np.asarray(v, dtype=np.float64)
    a = np.minimum(np.abs(v), E2M1_MAX)
    hi = np.clip(np.searchsorted(_VARR, a, side="left"), 0, len(_VARR) - 1)
    lo = np.clip(hi - 1, 0, len(_VARR) - 1)
    d_lo = np.abs(a - _VARR[lo])
    d_hi = np.abs(_VARR[hi] - a)
    pick_hi = (d_hi < d_lo) | ((d_hi == d_lo) & ((_CARR[hi] & 1) == 0))
    code = np.where(pick_hi, _CARR[hi], _CARR[lo])
    return (code | np.where(np.signbit(v), 0x8, 0)).astype(np.uint8)


def nvfp4_row_scale(row: np.ndarray) -> float:
    """NV2: the smallest power of two g = 2^e, e >= -126, with max |x| <= 6 * 448 * g."""
    amax = float(np.max(np.abs(row))) if row.size else 0.0
    if amax == 0.0:
        return 1.0
    e = -126
    while amax > E2M1_MAX * E4M3_MAX * 2.0 ** e:
        e += 1
    return 2.0 ** e


def nvfp4_quantize_rows(x: np.ndarray):
    """Rows of x [R, D] (D a multiple of 16) -> (codes uint8 [R, D/2], two per
    byte, element 2j in the low nibble; block scales as E4M3 codes uint8
    [R, D/16]; row scales float64 [R])."""
    R, D = x.shape
    nb = D // NVFP4_BLOCK
    codes = np.zeros((R, D // 2), dtype=np.uint8)
    bsc = np.zeros((R, nb), dtype=np.uint8)
    rsc = np.empty(R)
    for r in range(R):
        g = nvfp4_row_scale(x[r])
        rsc[r] = g
        blocks = x[r].reshape(nb, NVFP4_BLOCK)
        amax_b = np.max(np.abs(blocks), axis=1).astype(np.float32)
        ratio = amax_b / np.float32(E2M1_MAX * g)              # fp32 division (NV2)
        bcode = e4m3_quantize_array(ratio.astype(np.float64))
        bsc[r] = bcode
        sb = np.array([e4m3_value(int(c)) for c in bcode])
        q = np.zeros((nb, NVFP4_BLOCK), dtype=np.uint8)
        live = sb > 0
        if live.any():
            den = (sb[live] * g).astype(np.float32)[:, None]   # exact: E4M3 value times 2^e
            vals = blocks[live].astype(np.float32) / den        # fp32 division (NV2)
            q[live] = e2m1_quantize_array(vals.astype(np.float64))
        flat = q.reshape(D)
        codes[r] = (flat[0::2] & 0xF) | ((flat[1::2] & 0xF) << 4)
    return codes, bsc, rsc


def nvfp4_dequantize_rows(codes: np.ndarray, bsc: np.ndarray, rsc: np.ndarray) -> np.ndarray:
    """code * s_b * g for every element, float64 [R, D]."""
    lut4 = np.array([e2m1_value(c) for c in range(16)])
    lut8 = np.array([e4m3_value(c) for c in range(256)])
    R, half = codes.shape
    D = 2 * half
    q = np.empty((R, D), dtype=np.uint8)
    q[:, 0::2] = codes & 0xF
    q[:, 1::2] = codes >> 4
    sb = np.repeat(lut8[bsc], NVFP4_BLOCK, axis=1)
    return lut4[q] * sb * rsc[:, None]
