"""Pins of the MXFP8 oracle (oracle/mx.py) to the format's own definition:
the shared exponent X = floor(log2(amax)) - 8 worked out by hand, saturation
of the block maximum above 448 2^X, zero and short blocks, an exact round trip
of values on the grid, and a quantised LM head that equals the unquantised one
when every weight and hidden state is representable."""
import numpy as np

import oracle as O
from oracle import mx as MX
from oracle.e4m3 import e4m3_decode


def test_block_exponent_by_hand():
    amax = np.array([1.0, 448.0, 256.0, 511.99, 0.75, 2.0 ** -20, 0.0, 2.0 ** -130,
                     3.0e38, 1.5 * 2.0 ** 100], dtype=np.float64)
    # floor(log2): 0, 8, 8, 8, -1, -20, -, -130, 127, 100
    want = [-8, 0, 0, 0, -9, -28, -127, -127, 119, 92]
    np.testing.assert_array_equal(MX.block_exponents(amax), want)


def test_block_maximum_scales_into_256_512_and_saturates_above_448():
    x = np.zeros((3, 32), dtype=np.float32)
    x[0, 0] = 480.0          # X = 0: 480 saturates to 448
    x[0, 1] = -1.0
    x[1, 0] = 1.75 * 2.0 ** 5   # X = 5 - 8 = -3: scaled 1.75 * 2^8 = 448, exact
    x[1, 1] = 2.0 ** -3      # scaled 1
    x[2, 0] = 2.0 ** 7 * 1.9375  # X = -1: scaled 1.9375 * 2^8 = 496 -> 448
    codes, exps = MX.quantize_rows_mxfp8(x)
    np.testing.assert_array_equal(exps[:, 0], [0, -3, -1])
    deq = MX.dequantize_rows_mxfp8(codes, exps)
    assert deq[0, 0] == 448.0 and deq[0, 1] == -1.0
    assert deq[1, 0] == 1.75 * 2.0 ** 5 and deq[1, 1] == 2.0 ** -3
    assert deq[2, 0] == 448.0 * 0.5
    assert codes[0, 0] == 0x7E and codes[2, 0] == 0x7E


def test_zero_and_short_blocks():
    x = np.zeros((2, 40), dtype=np.float32)
    x[1, 35] = 3.0           # the second (8-element) block: X = 1 - 8 = -7
    codes, exps = MX.quantize_rows_mxfp8(x)
    assert exps.shape == (2, 2)
    np.testing.assert_array_equal(exps[0], [-127, -127])
    np.testing.assert_array_equal(exps[1], [-127, -7])
    assert not codes[0].any()
    assert MX.dequantize_rows_mxfp8(codes, exps)[1, 35] == 3.0


def _grid_rows(rng, rows, D):
    """Rows whose every block is a power of two times E4M3 grid values with
    the block maximum's scaled magnitude in [256, 448]: representable exactly."""
    nb = -(-D // 32)
    grid = e4m3_decode(np.arange(256, dtype=np.uint8))
    grid = grid[np.isfinite(grid) & (np.abs(grid) <= 448)]
    top = grid[(np.abs(grid) >= 256)]
    X = rng.integers(-20, 10, size=(rows, nb))
    vals = rng.choice(grid, size=(rows, nb, 32))
    vals[:, :, 0] = rng.choice(top, size=(rows, nb))   # the block maximum
    x = (vals * np.exp2(X)[:, :, None]).reshape(rows, nb * 32)[:, :D]
    return x.astype(np.float32), X


def test_round_trip_on_the_grid():
    rng = np.random.default_rng(5)
    x, X = _grid_rows(rng, 17, 96)
    codes, exps = MX.quantize_rows_mxfp8(x)
    np.testing.assert_array_equal(exps, X)
    np.testing.assert_array_equal(MX.dequantize_rows_mxfp8(codes, exps), x.astype(np.float64))


def test_quantised_head_equals_unquantised_on_representable_values():
    rng = np.random.default_rng(6)
    V, D = 300, 96
    W, _ = _grid_rows(rng, V, D)
    W *= np.float32(2.0 ** -12)      # keep the logits moderate (still on the grid)
    H, _ = _grid_rows(rng, 7, D)
    H *= np.float32(2.0 ** -12)
    cand_len = [1, 3, 2]
    ids = rng.integers(0, V, size=sum(cand_len))
    lay = O.build_layout([5], [3], cand_len, ids, V)
    H = H[:lay["N"]]              # 4 rows: the shared row and 3 fed tokens
    wc, we = MX.quantize_rows_mxfp8(W)
    got = MX.token_logprobs_mxfp8(lay, H, wc, we)
    ref = O.token_logprobs(lay, H.astype(np.float64), W.astype(np.float64))
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)


def test_exponent_rule_is_what_decides_saturation():
    # a mistaken rule X = floor(log2 amax) - 7 would keep 480 unsaturated
    # (scaled 240); the format's rule saturates it, so the two disagree here
    x = np.zeros((1, 32), dtype=np.float32)
    x[0, 0] = 480.0
    x[0, 1] = 2.0 ** -9 * 3    # an element near the bottom of the range
    codes, exps = MX.quantize_rows_mxfp8(x)
    deq = MX.dequantize_rows_mxfp8(codes, exps)
    assert deq[0, 0] == 448.0
    # 3 * 2^-9 at X = 0 is the E4M3 subnormal 3 * 2^-9 (code 0x03)
    assert codes[0, 1] == 0x03 and deq[0, 1] == 3 * 2.0 ** -9
