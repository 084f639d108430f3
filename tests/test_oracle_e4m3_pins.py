"""Pins of the low-precision (e4m3) LM-head oracle against the OCP FP8 E4M3
format's own definition: code table values, round-to-nearest-even ties,
saturation, exhaustive round trips, nearest-value brute force, and a quantised
model that must reproduce the unquantised one when every value is exact."""
import numpy as np
import pytest

import oracle as O
from oracle import e4m3 as Q

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


# values fixed by the format: 1 sign, 4 exponent bits (bias 7), 3 mantissa bits
TABLE = {
    0x00: 0.0, 0x01: 2.0 ** -9, 0x07: 7 * 2.0 ** -9, 0x08: 2.0 ** -6, 0x38: 1.0, 0x3C: 1.5,
    0x40: 2.0, 0x48: 4.0, 0x7E: 448.0, 0x7D: 416.0, 0x77: 240.0, 0xB8: -1.0, 0xFE: -448.0,
    0x81: -(2.0 ** -9),
}


def test_decode_table():
    for code, val in TABLE.items():
        assert Q.e4m3_decode([code])[0] == val, hex(code)
    assert np.isnan(Q.e4m3_decode([0x7F])[0]) and np.isnan(Q.e4m3_decode([0xFF])[0])
    assert np.signbit(Q.e4m3_decode([0x80])[0])


def test_encode_table_and_ties():
    cases = [
        (1.0, 0x38), (448.0, 0x7E), (-448.0, 0xFE), (2.0 ** -9, 0x01), (2.0 ** -6, 0x08),
        (1.0625, 0x38),            # halfway 1.0 / 1.125: even mantissa 0
        (1.1875, 0x3A),            # halfway 1.125 / 1.25: even mantissa 2
        (2.0 ** -10, 0x00),        # halfway 0 / 2^-9: even (zero)
        (3 * 2.0 ** -10, 0x02),    # halfway 2^-9 / 2^-8: even mantissa 2
        (15.5 * 2.0 ** -3, 0x40),  # 1.9375: halfway 1.875 / 2.0 rounds up into the next binade
        (500.0, 0x7E), (-1.0e6, 0xFE), (464.0, 0x7E),  # saturation
        (-1.0e-10, 0x80), (-0.0, 0x80), (0.0, 0x00),
    ]
    for y, code in cases:
        assert Q.e4m3_encode(np.float32(y)) == code, (y, hex(int(Q.e4m3_encode(np.float32(y)))))


def test_exhaustive_round_trip():
    codes = np.array([c for c in range(256) if c not in (0x7F, 0xFF)], dtype=np.uint8)
    np.testing.assert_array_equal(Q.e4m3_encode(Q.e4m3_decode(codes).astype(np.float32)), codes)
    # the finite magnitudes increase with the code
    mags = Q.e4m3_decode(np.arange(0, 0x7F, dtype=np.uint8))
    assert np.all(np.diff(mags) > 0)


def test_encode_is_a_nearest_value_brute_force():
    rng = np.random.default_rng(3)
    y = np.concatenate([rng.uniform(-460, 460, 4000), rng.normal(0, 0.02, 4000),
                        rng.uniform(-2.0 ** -6, 2.0 ** -6, 2000)]).astype(np.float32)
    finite = np.array([c for c in range(256) if c not in (0x7F, 0xFF)], dtype=np.uint8)
    vals = Q.e4m3_decode(finite)
    got = Q.e4m3_decode(Q.e4m3_encode(y))
    yc = np.clip(y.astype(np.float64), -448.0, 448.0)
    best = np.min(np.abs(vals[None, :] - yc[:, None]), axis=1)
    np.testing.assert_array_equal(np.abs(got - yc), best)


def test_quantize_rows_exact_when_representable():
    x = np.array([[448.0, -224.0, 1.0, 0.0, -2.0 ** -9],
                  [0.0, 0.0, 0.0, 0.0, 0.0],
                  [-7.0, 3.5, 0.4375, 0.0, 14.0]], dtype=np.float32)
    codes, scale = Q.quantize_rows(x)
    assert scale[0] == np.float32(1.0) and scale[1] == 0.0
    assert scale[2] == np.float32(14.0) / np.float32(448.0)
    np.testing.assert_array_equal(Q.dequantize_rows(codes, scale)[:2], x[:2].astype(np.float64))
    # row 2: scaled by 32, every value lands on the grid
    np.testing.assert_allclose(Q.dequantize_rows(codes, scale)[2], x[2], rtol=0, atol=1e-12)


def test_quantized_head_equals_exact_head_on_grid_values():
    # weights and hidden states whose rows have amax 448 and grid values: the
    # quantised model is the unquantised one, so Eq. 1-2 must agree exactly
    rng = np.random.default_rng(5)
    grid = Q.e4m3_decode(np.arange(0, 0x7F, dtype=np.uint8))
    V, D = 96, 48
    W = rng.choice(grid, size=(V, D)) * rng.choice([-1.0, 1.0], size=(V, D))
    W[:, 0] = 448.0
    H = rng.choice(grid[:60], size=(5, D)) * rng.choice([-1.0, 1.0], size=(5, D))
    H[:, 1] = -448.0
    W, H = W.astype(np.float32), H.astype(np.float32)
    lay = O.build_layout([3, 2], [2, 1], [2, 1, 2], [4, 7, 95, 0, 11], V)
    wc, ws = Q.quantize_rows(W)
    assert np.all(ws == 1.0)
    # scale the logits down so that exp does not overflow in either path
    ref = O.token_logprobs(lay, H.astype(np.float64) / 4096.0, W.astype(np.float64))
    got = O.token_logprobs(lay, Q.dequantize_rows(*Q.quantize_rows(H)) / 4096.0,
                           Q.dequantize_rows(wc, ws))
    np.testing.assert_array_equal(got, ref)
    np.testing.assert_allclose(
        Q.token_logprobs_e4m3(lay, H / np.float32(4096.0), wc, ws),
        ref, rtol=0, atol=1e-12)
