"""fp64 CPU oracle of the MXFP8 LM head (e4m3 codes in 32-element blocks that
share a power-of-two scale, on both the weights and the hidden states).

TEST INFRASTRUCTURE, like the rest of ``oracle``: only the tests, the smoke
check and the benchmark's CPU-baseline leg use it; it shares no code with the
CUDA path and imports nothing from it.

The paper's 8-bit weights (Q8_0, Appendix A) are 8-bit codes in blocks of 32
elements with one scale per block. The microscaling (MX) form of that idea
keeps the 32-element block and restricts its scale to a power of two, which
the tensor core applies itself; here it is used for both operands of the LM
head. What this module fixes (the paper gives no kernel-level scheme, so this
is a reading, stated once):

* A block is 32 consecutive elements of a row (the last block of a row may be
  shorter). Its shared exponent is X = floor(log2(amax)) - 8, where amax is
  the largest |x| of the block and 8 is the exponent of the largest E4M3
  binade (448 = 1.75 * 2^8); X is clamped to [-127, 127], and a block of zeros
  gets X = -127. The scale factor is stored as the byte X + 127 (UE8M0).
* An element's code is the E4M3 encoding (``oracle.e4m3.e4m3_encode``: nearest,
  ties to even, saturating at 448) of x * 2^-X, which is exact in float32 (a
  power-of-two multiplication). The scaled block maximum lies in [256, 512),
  so the largest elements of some blocks saturate to 448, as the format has it.
* The dequantised value is 2^X * decode(code); the logit is
  z[n, v] = sum_k dq(h)[n, k] dq(w)[v, k] with no further per-row scale, and
  everything after the logits is the oracle of Eq. 1-5 on those matrices.
"""
from __future__ import annotations

import numpy as np

from .e4m3 import e4m3_decode, e4m3_encode
from .jet_oracle import token_logprobs

__all__ = ["BLOCK", "X_MIN", "X_MAX", "block_exponents", "quantize_rows_mxfp8",
           "dequantize_rows_mxfp8", "token_logprobs_mxfp8"]

BLOCK = 32
X_MIN, X_MAX = -127, 127
E4M3_EMAX = 8


def block_exponents(amax) -> np.ndarray:
    """X = floor(log2(amax)) - 8, clamped to [-127, 127]; -127 for amax = 0.
    floor(log2) is read off the binary exponent, so it is exact."""
    a = np.asarray(amax, dtype=np.float64)
    _, ex = np.frexp(np.where(a > 0, a, 1.0))   # a = f 2^ex with f in [0.5, 1)
    x = (ex.astype(np.int64) - 1) - E4M3_EMAX
    x = np.where(a > 0, x, X_MIN)
    return np.clip(x, X_MIN, X_MAX)


def quantize_rows_mxfp8(x, chunk: int = 1024):
    """(codes [rows, D] uint8, exps [rows, ceil(D/32)] int16) of a float32
    matrix; rows are independent, so they are taken `chunk` at a time."""
    x = np.asarray(x)
    rows, D = x.shape
    nb = (D + BLOCK - 1) // BLOCK
    codes = np.zeros((rows, D), dtype=np.uint8)
    exps = np.empty((rows, nb), dtype=np.int16)
    for r0 in range(0, rows, chunk):
        xb = np.asarray(x[r0:r0 + chunk], dtype=np.float32)
        n = xb.shape[0]
        xp = np.zeros((n, nb * BLOCK), dtype=np.float32)
        xp[:, :D] = xb
        xp = xp.reshape(n, nb, BLOCK)
        amax = np.max(np.abs(xp), axis=2)
        X = block_exponents(amax)
        exps[r0:r0 + n] = X
        # x * 2^-X: a float32 multiplication by a power of two (exact; 2^-X is
        # formed in float64 and is exactly representable in float32 for |X| <= 126,
        # and the product is rounded once to float32 for X = -127)
        y = (xp.astype(np.float64) * np.exp2(-X.astype(np.float64))[:, :, None]).astype(np.float32)
        codes[r0:r0 + n] = e4m3_encode(y).reshape(n, nb * BLOCK)[:, :D]
    return codes, exps


def dequantize_rows_mxfp8(codes, exps) -> np.ndarray:
    """float64 values 2^X[r, b] * decode(codes[r, k])."""
    codes = np.asarray(codes)
    D = codes.shape[1]
    e = np.repeat(np.asarray(exps, dtype=np.float64), BLOCK, axis=1)[:, :D]
    return np.exp2(e) * e4m3_decode(codes)


class DequantizedMxRows:
    """Read-only view of the dequantised rows a slice asks for."""

    def __init__(self, codes, exps):
        self.codes, self.exps = codes, exps
        self.shape = codes.shape

    def __getitem__(self, rows):
        return dequantize_rows_mxfp8(self.codes[rows], self.exps[rows])


def token_logprobs_mxfp8(lay, H, w_codes, w_exps, targets=None):
    """l_{c,t} (Eq. 1, Eq. 2) of the MXFP8 LM head: the hidden states are
    quantised here (per token, per 32-element block), the weights come
    quantised."""
    h_codes, h_exps = quantize_rows_mxfp8(H)
    return token_logprobs(lay, dequantize_rows_mxfp8(h_codes, h_exps),
                          DequantizedMxRows(w_codes, w_exps), targets)
