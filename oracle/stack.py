"""fp64 CPU oracle of a hybrid decoder stack over the scoring step's rows.

TEST INFRASTRUCTURE, like the rest of ``oracle``: only the tests and the smoke
check use it; it shares no code with the CUDA path and imports nothing from it.

The paper scores candidates with hybrid models whose linear-attention layers
keep a recurrent state that is restored for every candidate, and whose
attention layers reuse the prefix cache (Sec. 4.1). A stack of such layers
applied to the step's query rows - the shared row and every candidate's fed
tokens - turns the single-layer step into a decoder forward, with a fork of
the recurrent state at every linear-attention layer. The paper gives no layer
recipe; the reading here is the common pre-norm decoder layer:

    h  = RMSNorm(x) * g1
    o  = full layer:   q, k, v = h W_mix^T; cascade attention over the layer's
                       prefix keys/values plus the candidate's own fed tokens
         linear layer: q, k, v, a, b = h W_mix^T; k normalised per head;
                       alpha = sigmoid(a), beta = sigmoid(b); every candidate's
                       fed tokens run the recurrence from the layer's prefix
                       state; the shared row reads the prefix state itself
                       (o = S_prefix^T q / sqrt(dk))
    x' = x + o W_o^T
    h2 = RMSNorm(x') * g2
    x''= x' + (SiLU(h2 W_gate^T) * (h2 W_up^T)) W_down^T

RMSNorm(x) = x / sqrt(mean(x^2) + eps), eps = 1e-6. The key/value rows of
each request's shared row are the last position of the layer's prefix cache
(the shared row is the last prefix position), so only the fed rows' keys and
values come from the projection.

Storage points. The device keeps activations in bf16 between operations; the
oracle computes every operation in float64 and rounds its result to bf16 at
the same points (round to nearest even): h, h2, the mixer projection's output,
the normalised keys, the attention / recurrence outputs, x', u = SiLU(g) * up
and x''. The gates alpha, beta and the recurrent states stay unrounded.
"""
from __future__ import annotations

import math

import numpy as np

from .jet_oracle import cascade_attention, fork_state

__all__ = ["bf16", "rmsnorm", "silu", "sigmoid", "layer_forward", "stack_forward", "EPS"]

EPS = 1e-6


def bf16(x) -> np.ndarray:
    """float64 values rounded to bf16 (nearest, ties to even), as float64.
    Values are first rounded to float32, as a float32 result would be."""
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    b = f.view(np.uint32).astype(np.uint64)
    b = (b + ((b >> 16) & 1) + 0x7FFF) >> 16
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def rmsnorm(x, g, eps: float = EPS) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * g, row by row."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * np.asarray(g, np.float64)


def sigmoid(z) -> np.ndarray:
    z = np.asarray(z, dtype=np.float64)
    return 1.0 / (1.0 + np.exp(-z))


def silu(z) -> np.ndarray:
    z = np.asarray(z, dtype=np.float64)
    return z * sigmoid(z)


def _fed_rows(lay):
    """Row indices of the fed tokens, in fed-token order (every row but each
    request's shared row)."""
    rows = []
    for r in range(lay["R"]):
        rows.extend(range(int(lay["row_offset"][r]) + 1, int(lay["row_offset"][r + 1])))
    return np.asarray(rows, dtype=np.int64)


def _gate_up(w_gu, Dff):
    """(W_gate, W_up) from the interleaved [2 Dff, D] matrix: gate feature f
    is row 128 (f // 64) + f % 64, its up feature the row 64 below it."""
    f = np.arange(Dff)
    g_rows = 128 * (f // 64) + f % 64
    return w_gu[g_rows], w_gu[g_rows + 64]


def layer_forward(lay, x, kind: str, P: dict, dims: dict, rule: str = "delta"):
    """One decoder layer on the rows x [N, D] (bf16 values). P holds the
    layer's float64 tensors (g1, g2, w_mix, w_o, w_gu, w_d and k_pre/v_pre or
    s_prefix); dims holds Hq, Hkv, d, Hl, dk, dv, Dff. Returns x''."""
    N, D = x.shape
    R = lay["R"]
    fed = _fed_rows(lay)
    h = bf16(rmsnorm(x, P["g1"]))
    z = bf16(h @ P["w_mix"].T)
    if kind == "full":
        Hq, Hkv, d = dims["Hq"], dims["Hkv"], dims["d"]
        q = z[:, :Hq * d].reshape(N, Hq, d)
        k = z[:, Hq * d:(Hq + Hkv) * d].reshape(N, Hkv, d)
        v = z[:, (Hq + Hkv) * d:(Hq + 2 * Hkv) * d].reshape(N, Hkv, d)
        o = bf16(cascade_attention(lay, q, P["k_pre"], P["v_pre"], k[fed], v[fed], Hq, Hkv))
        o = o.reshape(N, Hq * d)
    else:
        Hl, dk, dv = dims["Hl"], dims["dk"], dims["dv"]
        lq = z[:, :Hl * dk].reshape(N, Hl, dk)
        lk_raw = z[:, Hl * dk:2 * Hl * dk].reshape(N, Hl, dk)
        lv = z[:, 2 * Hl * dk:Hl * (2 * dk + dv)].reshape(N, Hl, dv)
        a = z[:, Hl * (2 * dk + dv):Hl * (2 * dk + dv) + Hl]
        b = z[:, Hl * (2 * dk + dv) + Hl:Hl * (2 * dk + dv) + 2 * Hl]
        lk = bf16(lk_raw / np.linalg.norm(lk_raw, axis=-1, keepdims=True))
        alpha, beta = sigmoid(a), sigmoid(b)
        o = np.zeros((N, Hl, dv))
        lo, _ = fork_state(lay, P["s_prefix"], lq[fed], lk[fed], lv[fed], alpha[fed], beta[fed],
                           rule=rule)
        o[fed] = lo
        for r in range(R):
            n = int(lay["row_offset"][r])
            for hh in range(Hl):
                o[n, hh] = P["s_prefix"][r, hh].T @ lq[n, hh] / math.sqrt(dk)
        o = bf16(o).reshape(N, Hl * dv)
    x1 = bf16(x + o @ P["w_o"].T)
    h2 = bf16(rmsnorm(x1, P["g2"]))
    wg, wu = _gate_up(P["w_gu"], dims["Dff"])
    u = bf16(silu(h2 @ wg.T) * (h2 @ wu.T))
    return bf16(x1 + u @ P["w_d"].T)


def stack_forward(lay, x0, kinds, params, dims, rule: str = "delta"):
    """The stack's output rows (bf16 values, float64) for input rows x0."""
    x = np.asarray(x0, dtype=np.float64)
    for kind, P in zip(kinds, params):
        x = layer_forward(lay, x, kind, P, dims, rule)
    return x
