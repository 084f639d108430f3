"""fp64 CPU oracle of the 4-bit LM head (e2m1 codes, a power-of-two exponent
per 32-element block, one float32 scale per row).

TEST INFRASTRUCTURE, like the rest of ``oracle``: only the tests, the smoke
check and the benchmark's CPU-baseline leg use it; it shares no code with the
CUDA path and imports nothing from it.

The paper runs its largest models with 4-bit weights (Q4_K_M, Appendix A):
4-bit codes in blocks of 32 that carry their own scale under a scale per
group of blocks. The 4-bit LM head here has the same two levels, in a form a
tensor core can take exactly:

* E2M1 (OCP FP4): 1 sign bit, 2 exponent bits (bias 1), 1 mantissa bit. Codes
  0..7 are the magnitudes 0, 0.5, 1, 1.5, 2, 3, 4, 6; bit 3 is the sign.
* Encoding a float32 value: round to the nearest magnitude, ties to the even
  code (the one whose mantissa bit is 0); magnitudes past 6 saturate to 6; the
  sign is kept (a negative value that rounds to zero gives code 8).
* Quantising a row x (float32 values of bf16 inputs): amax = max |x|;
  s = amax / 6 and inv = 6 / amax, each one float32 operation rounded to
  nearest. Block b holds 32 consecutive elements (the last block of a row may
  be shorter); t_b = (max |x_i| over the block) * inv in float32, and its
  exponent e_b is the smallest integer in [-5, 0] with t_b <= 6 * 2^e_b (0 when
  none is). The block's codes are the E2M1 encodings of x_i * (inv * 2^-e_b),
  one float32 multiplication rounded to nearest. A row of zeros has s = 0,
  zero codes and e_b = -5.
* The dequantised weight is s * 2^e_b * value(code). Every 2^e_b * value(code)
  is an E4M3 value (e_b >= -5 keeps it a normal number), so its product with an
  E4M3 hidden code is exact whether 2^e_b is applied as a block scale factor by
  the tensor core or folded into widened codes.
* The logit is z[n, v] = s_h[n] s_w[v] sum_k decode_e4m3(h[n, k]) w~[v, k] with
  the hidden states quantised per token as in the E4M3 head; everything after
  the logits is the oracle of Eq. 1-5 on the dequantised matrices.
"""
from __future__ import annotations

import numpy as np

from .e4m3 import dequantize_rows as e4m3_dequantize_rows
from .e4m3 import quantize_rows as e4m3_quantize_rows
from .jet_oracle import token_logprobs

__all__ = ["E2M1_VALUES", "BLOCK", "E_MIN", "e2m1_decode", "e2m1_encode", "quantize_rows_w4",
           "dequantize_rows_w4", "token_logprobs_w4"]

E2M1_VALUES = np.array([0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0])
BLOCK = 32
E_MIN = -5


def e2m1_decode(codes) -> np.ndarray:
    """Values (float64) of 4-bit codes 0..15."""
    c = np.asarray(codes, dtype=np.int64)
    mag = E2M1_VALUES[c & 7]
    return np.where(c & 8, -mag, mag)


# the midpoints between consecutive magnitudes
_MID = (E2M1_VALUES[1:] + E2M1_VALUES[:-1]) / 2


def e2m1_encode(y) -> np.ndarray:
    """Codes of float32 values: nearest magnitude, ties to the even code,
    saturating at 6, sign kept."""
    y = np.asarray(y, dtype=np.float32)
    neg = np.signbit(y)
    a = np.minimum(np.abs(y.astype(np.float64)), 6.0)
    # the number of midpoints below a is the nearer magnitude's code; a value
    # exactly on a midpoint between codes i and i + 1 takes the even one
    idx = np.searchsorted(_MID, a, side="left")
    tie = np.isin(a, _MID) & (idx % 2 == 1)
    idx = idx + tie
    return (idx | np.where(neg, 8, 0)).astype(np.uint8)


def quantize_rows_w4(x, chunk: int = 1024):
    """(codes [rows, D] uint8 0..15, exps [rows, ceil(D/32)] int8, scale [rows]
    float32) of a float32 matrix; rows are independent, so they are taken
    `chunk` at a time."""
    x = np.asarray(x)
    rows, D = x.shape
    nb = (D + BLOCK - 1) // BLOCK
    codes = np.zeros((rows, D), dtype=np.uint8)
    exps = np.empty((rows, nb), dtype=np.int8)
    scale = np.empty(rows, dtype=np.float32)
    for r0 in range(0, rows, chunk):
        xb = np.asarray(x[r0:r0 + chunk], dtype=np.float32)
        n = xb.shape[0]
        amax = np.max(np.abs(xb), axis=1).astype(np.float32)
        nz = amax > 0
        safe = np.where(nz, amax, np.float32(1))
        scale[r0:r0 + n] = np.where(nz, safe / np.float32(6.0), np.float32(0)).astype(np.float32)
        inv = np.where(nz, np.float32(6.0) / safe, np.float32(0)).astype(np.float32)
        xp = np.zeros((n, nb * BLOCK), dtype=np.float32)
        xp[:, :D] = xb
        xp = xp.reshape(n, nb, BLOCK)
        t = (np.max(np.abs(xp), axis=2) * inv[:, None]).astype(np.float32)
        # the smallest e in [E_MIN, 0] with t <= 6 * 2^e (0 when there is none)
        e = np.zeros((n, nb), dtype=np.int64)
        for ee in range(0, E_MIN - 1, -1):
            e = np.where(t <= np.float32(6.0 * 2.0 ** ee), ee, e)
        exps[r0:r0 + n] = e
        inv_b = (inv[:, None] * np.exp2(-e).astype(np.float32)).astype(np.float32)
        y = (xp * inv_b[:, :, None]).astype(np.float32)
        codes[r0:r0 + n] = e2m1_encode(y).reshape(n, nb * BLOCK)[:, :D]
    return codes, exps, scale


def dequantize_rows_w4(codes, exps, scale) -> np.ndarray:
    """float64 values s[r] * 2^e[r, b] * value(code)."""
    codes = np.asarray(codes)
    D = codes.shape[1]
    e = np.repeat(np.asarray(exps, dtype=np.float64), BLOCK, axis=1)[:, :D]
    return np.asarray(scale, dtype=np.float64)[:, None] * np.exp2(e) * e2m1_decode(codes)


class DequantizedW4Rows:
    """Read-only view of the dequantised weights that dequantises the rows a
    slice asks for."""

    def __init__(self, codes, exps, scale):
        self.codes, self.exps, self.scale = codes, exps, scale
        self.shape = codes.shape

    def __getitem__(self, rows):
        return dequantize_rows_w4(self.codes[rows], self.exps[rows], self.scale[rows])


def token_logprobs_w4(lay, H, w_codes, w_exps, w_scale, targets=None):
    """l_{c,t} (Eq. 1, Eq. 2) of the 4-bit LM head: the hidden states are
    quantised per token to E4M3 here, the weights come quantised."""
    h_codes, h_scale = e4m3_quantize_rows(H)
    return token_logprobs(lay, e4m3_dequantize_rows(h_codes, h_scale),
                          DequantizedW4Rows(w_codes, w_exps, w_scale), targets)
