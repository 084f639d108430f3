"""Seeded synthetic inputs for the JET candidate-scoring step.

This module is shared by the fp64 oracle (``oracle/``), the tests and the
benchmark. It draws random structure (prefix lengths, candidate counts and
lengths, target token ids) and random tensors (queries, keys, values, hidden
states, LM-head weights, recurrent states) with the shapes and distributions of
the paper's workloads. It holds none of the scoring method's arithmetic: no
layout, no attention, no logsumexp, no decision rule. The only count it makes
is the number of query rows, ``N = R + sum_c (m_c - 1)``, needed to size the
per-row tensors.

The paper (Sec. 5.1, Appendix A) evaluates MMLU and BoolQ requests on Qwen
models; neither the data nor the weights are available, so these draws stand in
for them. Every draw is reproducible from ``(seed, tensor tag, chunk index)``
alone: large tensors are drawn in fixed-size chunks with independent PCG64
streams, so the values do not depend on the number of threads used.

bf16 tensors are returned as ``uint16`` bit patterns (round to nearest even
from a float32 draw); :func:`bf16_to_f32` widens them exactly.
"""
from __future__ import annotations

import dataclasses
import os
from concurrent.futures import ThreadPoolExecutor
from typing import Dict, Optional

import numpy as np

__all__ = [
    "Workload", "WORKLOADS", "Problem", "make_problem", "bf16_round",
    "bf16_to_f32", "f32_to_bf16_bits", "StackSpec", "STACKS", "stack_shapes", "stack_tensor",
    "stack_x0",
]

_CHUNK = 1 << 22  # elements per independently seeded chunk


# --------------------------------------------------------------------------
# bf16 helpers (storage format only)
# --------------------------------------------------------------------------
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even); return uint16 bits."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).copy()
    b += ((b >> 16) & 1) + 0x7FFF
    return (b >> 16).astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def bf16_round(x: np.ndarray) -> np.ndarray:
    """float32 array holding the bf16-rounded values of ``x``."""
    return bf16_to_f32(f32_to_bf16_bits(x))


# --------------------------------------------------------------------------
# workloads
# --------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class Workload:
    """Shape and distribution recipe of one synthetic workload.

    Attributes follow the paper's notation where it has one: ``R`` requests
    (questions x), ``C`` candidates per request, candidate lengths ``m_c``,
    vocabulary size ``V``. ``Hq``/``Hkv``/``d`` are the attention heads and
    head dimension, ``D`` the LM-head hidden size. ``Hl``/``dk``/``dv`` size
    the linear-attention recurrent state (0 when the workload has none).
    """
    name: str
    index: int
    R: int
    prefix: tuple          # ("fixed", P) | ("uniform", lo, hi) | ("lognormal", median, sigma, lo, hi)
    C: int
    cand_len: tuple        # ("list", (m...)) | ("geom", p, max) | ("uniform", lo, hi)
    Hq: int
    Hkv: int
    d: int
    D: int
    V: int
    dtype: str             # "f32" or "bf16"
    w_std: float           # std of the LM-head weights
    mode: str              # decision rule: "argmax", "binary", "ordinal"
    Hl: int = 0
    dk: int = 0
    dv: int = 0

    @property
    def seed(self) -> int:
        # the paper's sample seed (Appendix A) plus the workload index
        return 20260921 + self.index


WORKLOADS: Dict[str, Workload] = {w.name: w for w in [
    Workload("tiny", 0, R=1, prefix=("fixed", 128), C=4, cand_len=("list", (1, 2, 3, 4)),
             Hq=8, Hkv=2, d=64, D=512, V=8192, dtype="f32", w_std=1.0 / np.sqrt(512.0),
             mode="argmax"),
    Workload("dense27b_mc", 1, R=16, prefix=("uniform", 200, 1200), C=4,
             cand_len=("geom", 0.3, 12), Hq=24, Hkv=4, d=256, D=5120, V=151936,
             dtype="bf16", w_std=0.02, mode="argmax"),
    Workload("binary", 2, R=64, prefix=("lognormal", 400.0, 0.6, 64, 2048), C=2,
             cand_len=("uniform", 1, 2), Hq=24, Hkv=4, d=256, D=5120, V=151936,
             dtype="bf16", w_std=0.02, mode="binary"),
    Workload("ordinal_hybrid", 3, R=32, prefix=("fixed", 512), C=10,
             cand_len=("uniform", 1, 3), Hq=16, Hkv=2, d=256, D=4096, V=151936,
             dtype="bf16", w_std=0.02, mode="ordinal", Hl=16, dk=128, dv=128),
    Workload("moe_a3b_long", 4, R=256, prefix=("uniform", 2048, 8192), C=4,
             cand_len=("geom", 0.3, 12), Hq=16, Hkv=2, d=256, D=2048, V=151936,
             dtype="bf16", w_std=0.02, mode="argmax"),
]}
WORKLOAD_BY_INDEX = {w.index: w for w in WORKLOADS.values()}


def _rng(seed: int, *tags: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, *tags])))


def _threads() -> int:
    return max(1, min(16, os.cpu_count() or 1))


def _normal_chunks(seed: int, tag: int, n: int, std: float, bf16: bool) -> np.ndarray:
    """n draws from N(0, std^2), chunk-seeded, as bf16 bits or float32."""
    out = np.empty(n, dtype=np.uint16 if bf16 else np.float32)

    def fill(i: int) -> None:
        lo, hi = i * _CHUNK, min(n, (i + 1) * _CHUNK)
        x = _rng(seed, tag, i).standard_normal(hi - lo, dtype=np.float32)
        if std != 1.0:
            x *= np.float32(std)
        out[lo:hi] = f32_to_bf16_bits(x) if bf16 else x

    nchunks = (n + _CHUNK - 1) // _CHUNK
    if nchunks <= 1:
        for i in range(nchunks):
            fill(i)
    else:
        with ThreadPoolExecutor(_threads()) as ex:
            list(ex.map(fill, range(nchunks)))
    return out


# tensor tags (part of the seed of each tensor)
_TAGS = {"structure": 1, "q": 2, "k_pre": 3, "v_pre": 4, "k_cand": 5, "v_cand": 6,
         "hidden": 7, "w_lm": 8, "s_prefix": 9, "lq": 10, "lk": 11, "lv": 12,
         "alpha": 13, "beta": 14, "q_pre": 15, "lq_pre": 16, "lk_pre": 17, "lv_pre": 18,
         "alpha_pre": 19, "beta_pre": 20}


@dataclasses.dataclass
class Problem:
    """One batch of R requests: structure plus lazily drawn tensors.

    ``prefix_len[r]`` is P_r, ``n_cand[r]`` is C_r, ``cand_len`` lists m_c for
    every candidate in request order, ``target_ids`` lists y_{c,1..m_c} for
    every candidate in the same order. ``N`` is the number of query rows and
    ``F = N - R`` the number of fed candidate tokens.
    """
    work: Workload
    seed: int
    prefix_len: np.ndarray
    n_cand: np.ndarray
    cand_len: np.ndarray
    target_ids: np.ndarray
    _cache: dict = dataclasses.field(default_factory=dict, repr=False)

    @property
    def R(self) -> int:
        return int(self.prefix_len.shape[0])

    @property
    def N(self) -> int:
        return self.R + int(np.sum(self.cand_len - 1))

    @property
    def F(self) -> int:
        return self.N - self.R

    @property
    def total_prefix(self) -> int:
        return int(np.sum(self.prefix_len))

    @property
    def bf16(self) -> bool:
        return self.work.dtype == "bf16"

    # ---- tensors -----------------------------------------------------------
    def _normal(self, name: str, shape, std: float = 1.0) -> np.ndarray:
        key = (name, tuple(shape))
        if key not in self._cache:
            n = int(np.prod(shape))
            self._cache[key] = _normal_chunks(self.seed, _TAGS[name], n, std,
                                              self.bf16).reshape(shape)
        return self._cache[key]

    def tensor(self, name: str) -> np.ndarray:
        """Device-format tensor: uint16 bf16 bits for bf16 workloads, else float32.

        Linear-attention gates ``alpha``/``beta`` and the recurrent state
        ``s_prefix`` are always float32.
        """
        w = self.work
        if name == "q":
            return self._normal("q", (self.N, w.Hq, w.d))
        if name in ("k_pre", "v_pre"):
            return self._normal(name, (self.total_prefix, w.Hkv, w.d))
        if name == "q_pre":  # queries of every prefix position (the prefill)
            return self._normal("q_pre", (self.total_prefix, w.Hq, w.d))
        if name in ("k_cand", "v_cand"):
            return self._normal(name, (self.F, w.Hkv, w.d))
        if name == "hidden":
            return self._normal("hidden", (self.N, w.D))
        if name == "w_lm":
            return self._normal("w_lm", (w.V, w.D), std=w.w_std)
        if w.Hl == 0:
            raise KeyError(f"workload {w.name} has no linear-attention layer")
        if name in self._cache:
            return self._cache[name]
        if name == "s_prefix":
            n = self.R * w.Hl * w.dk * w.dv
            x = _normal_chunks(self.seed, _TAGS["s_prefix"], n, 1.0 / np.sqrt(w.dk), False)
            val = x.reshape(self.R, w.Hl, w.dk, w.dv)
        elif name in ("lq", "lv", "lq_pre", "lv_pre"):
            # fed candidate tokens (F) or, with the _pre suffix, prefix tokens
            dim = w.dk if name.startswith("lq") else w.dv
            rows = self.total_prefix if name.endswith("_pre") else self.F
            val = self._normal(name, (rows, w.Hl, dim))
        elif name in ("lk", "lk_pre"):
            rows = self.total_prefix if name.endswith("_pre") else self.F
            x = _normal_chunks(self.seed, _TAGS[name], rows * w.Hl * w.dk, 1.0, False)
            x = x.reshape(rows, w.Hl, w.dk).astype(np.float64)
            x /= np.linalg.norm(x, axis=-1, keepdims=True)  # unit-norm keys
            x = x.astype(np.float32)
            val = f32_to_bf16_bits(x).reshape(x.shape) if self.bf16 else x
        elif name in ("alpha", "beta", "alpha_pre", "beta_pre"):
            lo, hi = (0.90, 1.00) if name.startswith("alpha") else (0.0, 1.0)
            rows = self.total_prefix if name.endswith("_pre") else self.F
            g = _rng(self.seed, _TAGS[name])
            val = g.uniform(lo, hi, size=(rows, w.Hl)).astype(np.float32)
        else:
            raise KeyError(name)
        self._cache[name] = val
        return val

    def f32(self, name: str) -> np.ndarray:
        """Exact float32 values of a tensor (widened from bf16 where needed)."""
        t = self.tensor(name)
        return bf16_to_f32(t) if t.dtype == np.uint16 else t

    def drop(self, name: Optional[str] = None) -> None:
        """Forget cached tensors (all of them when ``name`` is None)."""
        if name is None:
            self._cache.clear()
        else:
            for k in [k for k in self._cache if (k[0] if isinstance(k, tuple) else k) == name]:
                del self._cache[k]


def _draw_prefix(spec: tuple, R: int, g: np.random.Generator) -> np.ndarray:
    kind = spec[0]
    if kind == "fixed":
        return np.full(R, spec[1], dtype=np.int32)
    if kind == "uniform":  # inclusive integer bounds
        return g.integers(spec[1], spec[2] + 1, size=R).astype(np.int32)
    if kind == "lognormal":
        median, sigma, lo, hi = spec[1:]
        x = np.exp(g.normal(np.log(median), sigma, size=R))
        return np.clip(np.rint(x), lo, hi).astype(np.int32)
    raise ValueError(kind)


def _draw_lengths(spec: tuple, n: int, g: np.random.Generator) -> np.ndarray:
    kind = spec[0]
    if kind == "list":
        vals = np.asarray(spec[1], dtype=np.int32)
        return np.resize(vals, n).astype(np.int32)
    if kind == "geom":  # geometric(p) on 1..max, truncated and renormalised
        p, mmax = spec[1], spec[2]
        k = np.arange(1, mmax + 1)
        w = (1.0 - p) ** (k - 1) * p
        return g.choice(k, size=n, p=w / w.sum()).astype(np.int32)
    if kind == "uniform":
        return g.integers(spec[1], spec[2] + 1, size=n).astype(np.int32)
    raise ValueError(kind)


# --------------------------------------------------------------------------
# hybrid decoder stacks (several layers over the step's query rows)
# --------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class StackSpec:
    """A stack of decoder layers: ``kinds`` lists "linear" (linear attention,
    forked per candidate) or "full" (attention over the cached prefix) per
    layer; ``Dff`` is the MLP width (a multiple of 64)."""
    kinds: tuple
    Dff: int


STACKS: Dict[str, StackSpec] = {
    # three linear-attention layers per full-attention layer, as in the
    # paper's hybrid Qwen models; MLP width 3 x D
    "hybrid4": StackSpec(("linear", "linear", "linear", "full"), 3 * 4096),
}

_STACK_NAMES = ("g1", "g2", "w_mix", "w_o", "w_gu", "w_d", "k_pre", "v_pre", "s_prefix")


def stack_shapes(work: Workload, spec: StackSpec, kind: str, total_prefix: int, R: int):
    """Shapes of one layer's tensors. w_mix is [(Hq + 2 Hkv) d, D] for a
    full layer (q, k, v heads in that order) and [Hl (2 dk + dv) + 2 Hl, D] for
    a linear layer (q, k, v, then the alpha and beta logits); w_gu holds the
    MLP gate and up rows interleaved in blocks of 64 (rows 128 t .. + 63 gate
    features 64 t .., rows 128 t + 64 .. up features 64 t ..)."""
    w = work
    out = dict(g1=(w.D,), g2=(w.D,), w_gu=(2 * spec.Dff, w.D), w_d=(w.D, spec.Dff))
    if kind == "full":
        out.update(w_mix=((w.Hq + 2 * w.Hkv) * w.d, w.D), w_o=(w.D, w.Hq * w.d),
                   k_pre=(total_prefix, w.Hkv, w.d), v_pre=(total_prefix, w.Hkv, w.d))
    else:
        out.update(w_mix=(w.Hl * (2 * w.dk + w.dv) + 2 * w.Hl, w.D), w_o=(w.D, w.Hl * w.dv),
                   s_prefix=(R, w.Hl, w.dk, w.dv))
    return out


def stack_tensor(problem: "Problem", spec: StackSpec, layer: int, name: str) -> np.ndarray:
    """One tensor of layer ``layer`` in device format (bf16 bits; the recurrent
    state float32). Norm gains are 1 + N(0, 0.1^2); weights N(0, 1/fan_in);
    prefix keys/values N(0, 1); the prefix state N(0, 1/dk)."""
    w = problem.work
    kind = spec.kinds[layer]
    shape = stack_shapes(w, spec, kind, problem.total_prefix, problem.R)[name]
    key = ("stack", spec, layer, name)
    if key in problem._cache:
        return problem._cache[key]
    tag = 100 + 16 * layer + _STACK_NAMES.index(name)
    n = int(np.prod(shape))
    if name in ("g1", "g2"):
        x = 1.0 + _normal_chunks(problem.seed, tag, n, 0.1, False)
        val = f32_to_bf16_bits(x.astype(np.float32))
    elif name == "s_prefix":
        val = _normal_chunks(problem.seed, tag, n, 1.0 / np.sqrt(w.dk), False)
    elif name in ("k_pre", "v_pre"):
        val = _normal_chunks(problem.seed, tag, n, 1.0, True)
    else:
        val = _normal_chunks(problem.seed, tag, n, 1.0 / np.sqrt(shape[1]), True)
    val = val.reshape(shape)
    problem._cache[key] = val
    return val


def stack_x0(problem: "Problem") -> np.ndarray:
    """The embeddings of the step's N query rows, [N, D] bf16 bits, N(0, 1)."""
    key = ("stack_x0", problem.N, problem.work.D)
    if key not in problem._cache:
        problem._cache[key] = _normal_chunks(problem.seed, 99, problem.N * problem.work.D, 1.0,
                                             True).reshape(problem.N, problem.work.D)
    return problem._cache[key]


def make_problem(work, R: Optional[int] = None, seed: Optional[int] = None) -> Problem:
    """Draw the structure of a batch.

    ``work`` is a :class:`Workload`, its name or its index. ``R`` overrides the
    request count: the first ``R`` requests of the full draw are kept, so
    smaller batches are prefixes of larger ones (the batch-size sweep uses
    this).
    """
    if isinstance(work, str):
        work = WORKLOADS[work]
    elif isinstance(work, int):
        work = WORKLOAD_BY_INDEX[work]
    seed = work.seed if seed is None else seed
    g = _rng(seed, _TAGS["structure"])
    Rfull = work.R if R is None else max(R, work.R)
    prefix_len = _draw_prefix(work.prefix, Rfull, g)
    n_cand = np.full(Rfull, work.C, dtype=np.int32)
    cand_len = _draw_lengths(work.cand_len, Rfull * work.C, g)
    target_ids = g.integers(0, work.V, size=int(cand_len.sum())).astype(np.int32)
    Rk = Rfull if R is None else R
    keep_c = int(n_cand[:Rk].sum())
    keep_t = int(cand_len[:keep_c].sum())
    return Problem(work, seed, prefix_len[:Rk].copy(), n_cand[:Rk].copy(),
                   cand_len[:keep_c].copy(), target_ids[:keep_t].copy())


def custom_problem(work: Workload, prefix_len, n_cand, cand_len, target_ids,
                   seed: int = 1) -> Problem:
    """A problem with explicit structure (edge cases in tests)."""
    return Problem(work, seed, np.asarray(prefix_len, dtype=np.int32),
                   np.asarray(n_cand, dtype=np.int32), np.asarray(cand_len, dtype=np.int32),
                   np.asarray(target_ids, dtype=np.int32))


def torch_tensor(problem: Problem, name: str, device=None, pin: bool = False):
    """A tensor of the problem as a torch tensor (bf16 bit patterns become
    torch.bfloat16 without any rounding); optionally pinned or on a device."""
    import torch
    a = problem.tensor(name)
    if a.dtype == np.uint16:
        t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(a))
    if pin:
        t = t.pin_memory()
    if device is not None:
        t = t.to(device)
    return t


def array_to_torch(a: np.ndarray, device=None):
    """A device-format array (bf16 bits or float32) as a torch tensor."""
    import torch
    if a.dtype == np.uint16:
        t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(a))
    return t if device is None else t.to(device)
