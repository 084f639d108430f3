"""fp64 CPU oracle of the low-precision LM head (e4m3, one scale per row).

TEST INFRASTRUCTURE, like the rest of ``oracle``: only the tests, the smoke
check and the benchmark's CPU-baseline leg use it; it shares no code with the
CUDA path and imports nothing from it.

The paper runs its models with 8-bit (Q8_0) and 4-bit (Q4_K_M) weights
(Appendix A). The low-precision LM head here stores each row of a matrix as
OCP FP8 E4M3 codes plus one float32 scale: the weights per vocabulary row, the
hidden states per token. What this module fixes, from the format's definition:

* E4M3: 1 sign bit, 4 exponent bits (bias 7), 3 mantissa bits. Exponent field
  0 encodes subnormals m/8 * 2^-6; fields 1..15 encode (1 + m/8) * 2^(e-7),
  except S.1111.111, which is NaN. There are no infinities; the largest finite
  magnitude is 1.75 * 2^8 = 448 (code 0x7E), the smallest 2^-9 (code 0x01).
* Encoding a float32 value: round to the nearest representable magnitude, ties
  to the even mantissa; magnitudes past 448 saturate to 448; the sign is kept
  (a negative value that rounds to zero gives 0x80).
* Quantising a row x (float32 values of bf16 inputs): amax = max |x| in
  float32, s = amax / 448 and y = x * (448 / amax), each one float32 operation
  rounded to nearest; the codes are the e4m3 encodings of y. A row of zeros
  has s = 0 and zero codes.
* The quantised model's logit is z[n, v] = s_h[n] s_w[v] sum_k decode(h[n, k])
  decode(w[v, k]); everything after the logits is the oracle of Eq. 1-5 run on
  the dequantised matrices.
"""
from __future__ import annotations

import numpy as np

from .jet_oracle import token_logprobs

__all__ = ["e4m3_decode", "e4m3_encode", "quantize_rows", "dequantize_rows",
           "token_logprobs_e4m3"]

E4M3_MAX = 448.0


def e4m3_decode(codes) -> np.ndarray:
    """Values (float64) of e4m3 codes; NaN for the two NaN codes."""
    c = np.asarray(codes, dtype=np.uint8).astype(np.int64)
    sign = np.where(c & 0x80, -1.0, 1.0)
    e = (c >> 3) & 0xF
    m = c & 0x7
    mag = np.where(e == 0, m / 8.0 * 2.0 ** -6, (1.0 + m / 8.0) * np.exp2(e - 7.0))
    mag = np.where((e == 15) & (m == 7), np.nan, mag)
    return sign * mag


def _round_half_even(x: np.ndarray) -> np.ndarray:
    f = np.floor(x)
    d = x - f
    up = (d > 0.5) | ((d == 0.5) & (np.mod(f, 2.0) == 1.0))
    return f + up


def e4m3_encode(y) -> np.ndarray:
    """e4m3 codes of float32 values: nearest, ties to even, saturating at 448."""
    y = np.asarray(y, dtype=np.float32)
    neg = np.signbit(y)
    a = np.minimum(np.abs(y.astype(np.float64)), E4M3_MAX)
    # exponent of the binade a falls in; below 2^-6 the spacing stays 2^-9
    safe = np.where(a > 0, a, 1.0)
    e = np.maximum(np.floor(np.log2(safe)), -6.0)
    # guard against log2 rounding at exact powers of two
    e = np.where(np.exp2(e) > safe, e - 1, e)
    e = np.where(np.exp2(e + 1) <= safe, e + 1, e)
    e = np.maximum(e, -6.0)
    step = np.exp2(e - 3.0)
    mag = _round_half_even(a / step) * step
    mag = np.where(a > 0, np.minimum(mag, E4M3_MAX), 0.0)
    # the code of the rounded magnitude
    codes = np.zeros(y.shape, dtype=np.int64)
    sub = (mag > 0) & (mag < 2.0 ** -6)
    codes = np.where(sub, np.rint(mag / 2.0 ** -9), codes)
    nrm = mag >= 2.0 ** -6
    en = np.floor(np.log2(np.where(nrm, mag, 1.0)))
    mn = np.where(nrm, mag / np.exp2(en - 3.0) - 8.0, 0.0)
    codes = np.where(nrm, (en + 7.0) * 8.0 + mn, codes)
    codes = codes.astype(np.int64) | np.where(neg, 0x80, 0)
    return codes.astype(np.uint8)


def quantize_rows(x, block: int = 2048):
    """(codes [rows, D] uint8, scale [rows] float32) of a float32 matrix; rows
    are independent, so they are taken `block` at a time to bound memory."""
    x = np.asarray(x)
    codes = np.empty(x.shape, dtype=np.uint8)
    scale = np.empty(x.shape[0], dtype=np.float32)
    for r0 in range(0, x.shape[0], block):
        xb = np.asarray(x[r0:r0 + block], dtype=np.float32)
        amax = np.max(np.abs(xb), axis=1).astype(np.float32)
        nz = amax > 0
        inv = np.where(nz, np.float32(E4M3_MAX) / np.where(nz, amax, np.float32(1)),
                       np.float32(0)).astype(np.float32)
        y = (xb * inv[:, None]).astype(np.float32)
        codes[r0:r0 + block] = e4m3_encode(y)
        scale[r0:r0 + block] = (amax / np.float32(E4M3_MAX)).astype(np.float32)
    return codes, scale


def dequantize_rows(codes, scale) -> np.ndarray:
    """float64 values s[r] * decode(codes[r, k])."""
    return np.asarray(scale, dtype=np.float64)[:, None] * e4m3_decode(codes)


class DequantizedRows:
    """Read-only view of s[r] * decode(codes[r, :]) that dequantises the rows a
    slice asks for (the full weight matrix would take 8 bytes per element)."""

    def __init__(self, codes, scale):
        self.codes, self.scale = codes, scale
        self.shape = codes.shape

    def __getitem__(self, rows):
        return dequantize_rows(self.codes[rows], self.scale[rows])


def token_logprobs_e4m3(lay, H, w_codes, w_scale, targets=None):
    """l_{c,t} (Eq. 1, Eq. 2) of the quantised LM head: the hidden states are
    quantised per token here, the weights come quantised per vocabulary row."""
    h_codes, h_scale = quantize_rows(H)
    return token_logprobs(lay, dequantize_rows(h_codes, h_scale),
                          DequantizedRows(w_codes, w_scale), targets)
