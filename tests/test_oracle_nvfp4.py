"""Pins for the NVFP4 payload oracle (readings NV1-NV2).  They check:
  * the E2M1 code table against the format's published values;
  * the vectorised quantizer against the scalar brute-force search;
  * rounding ties, saturation and sign;
  * the power-of-two row scale and the E4M3 block scales;
  * a hand-computed block;
  * the round trip and the exactness of the dequantized values in bf16."""
import numpy as np
import torch

import oracle as O


def test_e2m1_table_is_the_published_one():
    codes, vals = O.e2m1_table()
    assert vals == [0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0]
    assert [O.e2m1_value(c | 0x8) for c in codes] == [-v for v in vals]


def test_vectorised_quantizer_matches_brute_force():
    rng = np.random.default_rng(0)
    _, vals = O.e2m1_table()
    mids = [(a + b) / 2 for a, b in zip(vals, vals[1:])]
    v = np.concatenate([rng.normal(size=3000) * 3, np.array(vals), np.array(mids), -np.array(mids),
                        [7.0, -100.0, 6.0, 0.0, -0.0, 0.24, 0.26]])
    got = O.e2m1_quantize_array(v)
    want = np.array([O.e2m1_quantize(float(x)) for x in v], dtype=np.uint8)
    assert (got == want).all()


def test_ties_to_even_saturation_and_sign():
    assert O.e2m1_quantize(0.25) == 0x0   # between 0 (0x0) and 0.5 (0x1): even
    assert O.e2m1_quantize(0.75) == 0x2   # between 0.5 (0x1) and 1.0 (0x2): even
    assert O.e2m1_quantize(1.25) == 0x2   # between 1.0 (0x2) and 1.5 (0x3): even
    assert O.e2m1_quantize(2.5) == 0x4    # between 2 (0x4) and 3 (0x5): even
    assert O.e2m1_quantize(5.0) == 0x6    # between 4 (0x6) and 6 (0x7): even
    assert O.e2m1_quantize(1e9) == 0x7 and O.e2m1_quantize(-1e9) == 0xF
    assert O.e2m1_quantize(-0.0) == 0x8   # sign kept on zero
    assert O.e2m1_quantize(2.9) == 0x5 and O.e2m1_quantize(-3.4) == 0xD


def test_row_scale_is_the_smallest_power_of_two():
    assert O.nvfp4_row_scale(np.array([6.0 * 448.0])) == 1.0
    assert O.nvfp4_row_scale(np.array([6.0 * 448.0 + 1.0])) == 2.0
    assert O.nvfp4_row_scale(np.array([1.0])) == 2.0 ** -11    # 2688 * 2^-11 = 1.3125 >= 1 > 0.65625
    assert O.nvfp4_row_scale(np.zeros(16)) == 1.0
    assert O.nvfp4_row_scale(np.array([1e-45])) == 2.0 ** -126


def test_hand_computed_block():
    # one 16-element row: amax 3.0 -> g = 2^-9 (6 * 448 * 2^-9 = 5.25 >= 3 > 2.625)
    x = np.array([[3.0, -1.5, 0.75, 0.0, 2.0, 1.0, -3.0, 0.5, 0.1, 0.2, 1.25, -2.5, 6.0 / 448 * 2, 0.0, 1.75, -0.25]])
    x[0, 12] = 0.0
    codes, bsc, rsc = O.nvfp4_quantize_rows(x)
    assert rsc[0] == 2.0 ** -9
    # r_b = 3 / (6 * 2^-9) = 256 -> E4M3 256 exactly (0x78); s_b * g = 0.5
    assert O.e4m3_value(int(bsc[0, 0])) == 256.0
    deq = O.nvfp4_dequantize_rows(codes, bsc, rsc)[0]
    # x / 0.5 -> 6, -3, 1.5, 0, 4, 2, -6, 1, 0.2, 0.4, 2.5, -5, 0, 0, 3.5, -0.5
    # E2M1  -> 6, -3, 1.5, 0, 4, 2, -6, 1, 0,   0.5, 2,   -4, 0, 0, 4,   -0.5
    want = 0.5 * np.array([6, -3, 1.5, 0, 4, 2, -6, 1, 0, 0.5, 2, -4, 0, 0, 4, -0.5])
    assert np.array_equal(deq, want)
    # element 0 in the low nibble of byte 0: 6 = code 0x7; element 1: -3 = 0xD
    assert codes[0, 0] == (0x7 | (0xD << 4))


def test_round_trip_and_bf16_exactness():
    rng = np.random.default_rng(4)
    x = rng.normal(size=(40, 64)) * np.exp(rng.normal(size=(40, 1)) * 4)
    x[3] = 0.0
    x = torch.tensor(x).to(torch.bfloat16).double().numpy()
    codes, bsc, rsc = O.nvfp4_quantize_rows(x)
    deq = O.nvfp4_dequantize_rows(codes, bsc, rsc)
    # exact in bf16
    assert np.array_equal(torch.tensor(deq).to(torch.bfloat16).double().numpy(), deq)
    # quantizing the dequantized rows reproduces the codes and scales
    c2, b2, r2 = O.nvfp4_quantize_rows(deq)
    assert np.array_equal(c2, codes) and np.array_equal(b2, bsc) and np.array_equal(r2, rsc)
    # error bound per element: half a step of the E2M1 grid, relative to the block scale
    err = np.abs(deq - x)
    sb = np.repeat(np.array([[O.e4m3_value(int(c)) for c in row] for row in bsc]), 16, axis=1) * rsc[:, None]
    assert (err <= sb * 1.0 + 1e-300).all()  # the widest E2M1 gap (4 -> 6) halves to 1 step of s_b g
    # payload bytes per row: D / 2 codes + D / 16 scales + 4
    assert codes.shape[1] + bsc.shape[1] + 4 == 64 // 2 + 64 // 16 + 4
