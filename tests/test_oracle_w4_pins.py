"""Pins of the 4-bit (w4) LM-head oracle against the OCP FP4 E2M1 format's own
definition and the block-exponent rule: the code table, round-to-nearest-even
ties, saturation, an exhaustive round trip, a nearest-value brute force, block
exponents worked out by hand, exact reproduction of grid values, and a
quantised model that must reproduce the unquantised one when every weight is
representable."""
import numpy as np

import oracle as O
from oracle import e4m3 as Q8
from oracle import w4 as Q4


def test_decode_table():
    # 1 sign bit, 2 exponent bits (bias 1), 1 mantissa bit
    want = [0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0]
    for c, v in enumerate(want):
        assert Q4.e2m1_decode([c])[0] == v
        assert Q4.e2m1_decode([c | 8])[0] == -v
    assert np.signbit(Q4.e2m1_decode([8])[0])


def test_encode_ties_and_saturation():
    cases = [
        (0.25, 0),    # halfway 0 / 0.5: the even code is 0
        (0.75, 2),    # halfway 0.5 / 1: code 2 (1.0)
        (1.25, 2),    # halfway 1 / 1.5: code 2
        (1.75, 4),    # halfway 1.5 / 2: code 4 (2.0)
        (2.5, 4),     # halfway 2 / 3: code 4
        (3.5, 6),     # halfway 3 / 4: code 6 (4.0)
        (5.0, 6),     # halfway 4 / 6: code 6
        (5.01, 7), (0.2, 0), (0.26, 1), (7.0, 7), (1.0e9, 7),
        (-0.25, 8), (-0.0, 8), (0.0, 0), (-3.0, 13), (-6.5, 15),
    ]
    for y, code in cases:
        assert Q4.e2m1_encode(np.float32(y)) == code, (y, int(Q4.e2m1_encode(np.float32(y))))


def test_exhaustive_round_trip():
    codes = np.arange(16, dtype=np.uint8)
    np.testing.assert_array_equal(Q4.e2m1_encode(Q4.e2m1_decode(codes).astype(np.float32)), codes)


def test_encode_is_a_nearest_value_brute_force():
    rng = np.random.default_rng(11)
    y = np.concatenate([rng.uniform(-7, 7, 20000),
                        np.repeat([0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0], 3) *
                        np.tile([1, -1, 1], 7)]).astype(np.float32)
    got = Q4.e2m1_decode(Q4.e2m1_encode(y))
    yc = np.clip(y.astype(np.float64), -6.0, 6.0)
    grid = np.array([-6, -4, -3, -2, -1.5, -1, -0.5, 0, 0.5, 1, 1.5, 2, 3, 4, 6], dtype=np.float64)
    best = np.min(np.abs(grid[None, :] - yc[:, None]), axis=1)
    np.testing.assert_array_equal(np.abs(got - yc), best)
    # on a tie the chosen magnitude has an even code
    tie = np.sum(np.isclose(np.abs(grid[None, :] - yc[:, None]), best[:, None], rtol=0,
                            atol=0), axis=1) > 1
    assert tie.sum() >= 21
    assert np.all(Q4.e2m1_encode(y[tie]) % 2 == 0)


def test_block_exponents_by_hand():
    # row amax 12 (s = 2, inv = 0.5): block 0 holds it (t = 6, e = 0); block 1's
    # amax 3 gives t = 1.5 = 6 * 2^-2 (e = -2); block 2's amax 0.1 gives
    # t = 0.05 < 6 * 2^-5 (e clamps to -5); block 3 is zeros (e = -5); the
    # last block is 16 elements long with amax 6 (t = 3, e = -1)
    D = 4 * 32 + 16
    x = np.zeros((1, D), dtype=np.float32)
    x[0, 5] = -12.0
    x[0, 40] = 3.0
    x[0, 41] = -0.75
    x[0, 70] = 0.1
    x[0, 130] = 6.0
    x[0, 131] = 1.0
    codes, exps, scale = Q4.quantize_rows_w4(x)
    assert scale[0] == np.float32(2.0)
    np.testing.assert_array_equal(exps[0], [0, -2, -5, -5, -1])
    assert codes[0, 5] == (8 | 7)         # -12 / 2 = -6
    assert codes[0, 40] == 7              # 3 * 0.5 * 4 = 6
    assert codes[0, 41] == (8 | 3)        # -0.75 * 2 = -1.5
    assert codes[0, 70] == 3              # 0.1 * 0.5 * 32 = 1.6 -> 1.5
    assert codes[0, 130] == 7 and codes[0, 131] == 2   # 6 * 0.5 * 2 = 6; 1 * 0.5 * 2 = 1
    deq = Q4.dequantize_rows_w4(codes, exps, scale)[0]
    assert deq[5] == -12.0 and deq[40] == 3.0 and deq[41] == -0.75 and deq[130] == 6.0
    assert deq[70] == 2.0 * 2.0 ** -5 * 1.5
    z = Q4.quantize_rows_w4(np.zeros((2, 64), dtype=np.float32))
    assert np.all(z[0] == 0) and np.all(z[1] == -5) and np.all(z[2] == 0)


def test_grid_rows_reproduce_exactly():
    # rows built as s * 2^e_b * value(code) with the row's largest block at e = 0
    rng = np.random.default_rng(12)
    V, D = 40, 96
    vals = Q4.e2m1_decode(rng.integers(0, 16, size=(V, D)))
    e = rng.integers(-5, 1, size=(V, D // 32))
    e[:, 0] = 0
    vals[:, 0] = 6.0   # every block's scale is set by a 6
    vals[:, 32] = -6.0
    vals[:, 64] = 6.0
    s = np.float32(2.0) ** rng.integers(-8, 8, size=V).astype(np.float32)
    x = (s[:, None] * np.exp2(np.repeat(e, 32, axis=1)) * vals).astype(np.float32)
    codes, exps, scale = Q4.quantize_rows_w4(x)
    np.testing.assert_array_equal(Q4.dequantize_rows_w4(codes, exps, scale), x.astype(np.float64))
    np.testing.assert_array_equal(exps, e)


def test_quantized_head_equals_exact_head_on_grid_values():
    # weights whose quantisation is exact and hidden states on the e4m3 grid
    # with amax 448: the 4-bit model is the unquantised model
    rng = np.random.default_rng(13)
    V, D = 80, 64
    vals = Q4.e2m1_decode(rng.integers(0, 16, size=(V, D)))
    vals[:, 0] = 6.0
    vals[:, 32] = 6.0
    e = rng.integers(-5, 1, size=(V, 2))
    e[:, 0] = 0        # the row's largest block: s = 1
    W = (vals * np.exp2(np.repeat(e, 32, axis=1))).astype(np.float32)
    grid = Q8.e4m3_decode(np.arange(0, 0x7F, dtype=np.uint8))
    H = (rng.choice(grid[:60], size=(5, D)) * rng.choice([-1.0, 1.0], size=(5, D))).astype(
        np.float32)
    H[:, 1] = -448.0
    wc, we, ws = Q4.quantize_rows_w4(W)
    assert np.all(ws == 1.0)
    lay = O.build_layout([3, 2], [2, 1], [2, 1, 2], [4, 7, 79, 0, 11], V)
    ref = O.token_logprobs(lay, H.astype(np.float64) / 4096.0, W.astype(np.float64))
    got = Q4.token_logprobs_w4(lay, H / np.float32(4096.0), wc, we, ws)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)
