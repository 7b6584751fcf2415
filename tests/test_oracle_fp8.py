"""Pins for the FP8 payload oracle (readings FP1-FP2): the E4M3 code table
against the format's published properties, the vectorised quantizer against
the scalar brute-force search over all codes, rounding ties, saturation, the
power-of-two row scale and the exactness of the dequantized values in bf16."""
import math

import numpy as np
import pytest
import torch

import oracle as O


def test_code_table_properties():
    codes, vals = O.e4m3_table()
    assert len(codes) == 127                      # 0x00..0x7E; 0x7F is NaN
    assert vals[0] == 0.0 and vals[-1] == 448.0   # largest finite E4M3
    assert vals[1] == 2.0 ** -9                   # smallest subnormal
    assert O.e4m3_value(0x08) == 2.0 ** -6        # smallest normal
    assert math.isnan(O.e4m3_value(0x7F)) and math.isnan(O.e4m3_value(0xFF))
    assert all(b > a for a, b in zip(vals, vals[1:]))
    # spacing: 8 values per binade above 2^-6
    assert O.e4m3_value(0x38) == 1.0 and O.e4m3_value(0x39) == 1.125
    assert O.e4m3_value(0x80) == 0.0 and math.copysign(1, O.e4m3_value(0x80)) < 0


def test_vectorised_quantizer_matches_brute_force():
    rng = np.random.default_rng(0)
    codes, vals = O.e4m3_table()
    mids = [(a + b) / 2 for a, b in zip(vals, vals[1:])]
    v = np.concatenate([rng.normal(size=3000) * 50, rng.normal(size=500) * 1e-3, np.array(vals), np.array(mids),
                        -np.array(mids), [500.0, -1e9, 448.0, 464.0, 0.0, -0.0, 2.0 ** -10, -(2.0 ** -10)]])
    got = O.e4m3_quantize_array(v)
    want = np.array([O.e4m3_quantize(float(x)) for x in v], dtype=np.uint8)
    assert (got == want).all()


def test_ties_go_to_the_even_code_and_saturate():
    assert O.e4m3_quantize(1.0625) == 0x38        # between 1.0 (0x38) and 1.125 (0x39): even
    assert O.e4m3_quantize(1.1875) == 0x3A        # between 1.125 (0x39) and 1.25 (0x3A): even
    assert O.e4m3_quantize(2.0 ** -10) == 0x00    # half the smallest subnormal -> +0
    assert O.e4m3_quantize(-(2.0 ** -10)) == 0x80
    assert O.e4m3_quantize(460.0) == 0x7E and O.e4m3_quantize(-1e6) == 0xFE
    assert O.e4m3_quantize(1.0) == 0x38 and O.e4m3_quantize(-448.0) == 0xFE


def test_row_scale_is_the_smallest_fitting_power_of_two():
    for amax in (448.0, 448.0001, 1.0, 3.5, 896.0, 1e-30, 7e3):
        row = np.array([0.5 * amax, -amax, 0.0])
        s = O.fp8_row_scale(row)
        e = math.log2(s)
        assert e == int(e)
        assert amax <= 448.0 * s
        assert s == 2.0 ** -126 or amax > 448.0 * s / 2
    assert O.fp8_row_scale(np.zeros(4)) == 1.0


def test_dequantized_rows_are_exact_in_bf16_and_close():
    rng = np.random.default_rng(3)
    x = torch.randn(40, 64).to(torch.bfloat16).double().numpy() * rng.uniform(1e-3, 1e3, size=(40, 1))
    x = torch.tensor(x).to(torch.bfloat16).double().numpy()
    codes, scales = O.fp8_quantize_rows(x)
    xd = O.fp8_dequantize_rows(codes, scales)
    assert np.array_equal(torch.tensor(xd).to(torch.bfloat16).double().numpy(), xd)
    # relative error of a normal E4M3 value is at most 2^-4; rows keep their max within [224 s, 448 s]
    big = np.abs(x) >= 2.0 ** -6 * scales[:, None]
    assert (np.abs(xd - x)[big] <= 2.0 ** -4 * np.abs(x)[big]).all()
    assert (np.abs(x).max(axis=1) > 224.0 * scales).all()
