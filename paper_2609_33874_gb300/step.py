"""One teacher-forced candidate-scoring step: attend -> (fork) -> score -> decide.

:class:`ScoringStep` owns the device buffers of one batch shape (the layout,
outputs and workspace) and strings the C entry points together on one CUDA
stream. Inputs are torch tensors already on the device (:meth:`run`) or pinned
host tensors that are copied in first (:meth:`run_from_host`, the end-to-end
path: host -> device copies, the kernels, device -> host copies of the
results; :meth:`run_pipelined` does the same over a sequence of batches and
overlaps each batch's input copies with the previous batch's kernels).
"""
from __future__ import annotations

from typing import Dict, Optional

import torch

from . import jet

_TORCH_DTYPE = {jet.DTYPE_F32: torch.float32, jet.DTYPE_BF16: torch.bfloat16}

# per-batch inputs of the step; the LM-head weights are model state and stay resident
ATTN_INPUTS = ("q", "k_pre", "v_pre", "k_cand", "v_cand")
FORK_INPUTS = ("s_prefix", "lq", "lk", "lv", "alpha", "beta")
RESULTS = ("tok_logprob", "cand_score", "q_cand", "choice", "value")
# below this many input bytes per batch (about 5 us over the host link)
# run_pipelined copies on the compute stream instead of overlapping
_OVERLAP_MIN_BYTES = 1 << 20
_ALIGN = 256  # bytes: every packed tensor starts on this boundary


def _pack_plan(items):
    """(offsets, total bytes) of tensors laid end to end at _ALIGN boundaries;
    items is a list of (name, dtype, shape)."""
    offs, at = {}, 0
    for name, dtype, shape in items:
        at = (at + _ALIGN - 1) // _ALIGN * _ALIGN
        n = 1
        for d in shape:
            n *= int(d)
        offs[name] = (at, dtype, tuple(shape))
        at += n * torch.empty((), dtype=dtype).element_size()
    return offs, (at + _ALIGN - 1) // _ALIGN * _ALIGN


def _views(buf: torch.Tensor, offs):
    """Typed views of a uint8 buffer at the planned offsets."""
    out = {}
    for name, (o, dtype, shape) in offs.items():
        n = 1
        for d in shape:
            n *= int(d)
        nb = n * torch.empty((), dtype=dtype).element_size()
        out[name] = buf[o:o + nb].view(dtype).view(shape)
    return out


class HostBatch:
    """One batch's layout words and inputs in a single pinned host buffer, each
    at a 256-byte aligned offset, so that the batch moves to the device in one
    copy (a loader writes its batches straight into such buffers)."""

    def __init__(self, step: "ScoringStep", host: Dict[str, torch.Tensor],
                 layout_words: torch.Tensor):
        items = [("__words__", layout_words.dtype, layout_words.shape)]
        items += [(k, host[k].dtype, host[k].shape) for k in step.input_names()]
        self.offsets, nbytes = _pack_plan(items)
        self.buf = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
        v = _views(self.buf, self.offsets)
        v["__words__"].copy_(layout_words)
        for k in step.input_names():
            v[k].copy_(host[k])

    @property
    def nbytes(self) -> int:
        return self.buf.numel()


class HostResults:
    """Pinned host buffer laid out like a step's results (one copy back):
    ``views`` holds tok_logprob, cand_score, q_cand, choice and value."""

    def __init__(self, step: "ScoringStep"):
        self.buf = torch.empty(step._results.numel(), dtype=torch.uint8, pin_memory=True)
        self.views = _views(self.buf, step._result_offsets)

    def __getitem__(self, k):
        return self.views[k]


def quantize_lm_head(w_lm: torch.Tensor, stream=None):
    """e4m3 codes [V, D] and per-row float32 scales [V] of the bf16 LM-head
    weights (jet_quantize_rows_e4m3), for a step built with lm="e4m3"."""
    V, D = w_lm.shape
    w_q = torch.empty(V, D, dtype=torch.uint8, device=w_lm.device)
    w_scale = torch.empty(V, dtype=torch.float32, device=w_lm.device)
    jet.jet_quantize_rows_e4m3(w_lm, w_q, w_scale, stream=stream)
    return w_q, w_scale


def quantize_lm_head_w4(w_lm: torch.Tensor, stream=None):
    """4-bit codes and block scale factors (uint8, jet_w4_bytes(V, D) bytes) and per-row float32
    scales [V] of the bf16 LM-head weights (jet_quantize_w4), for a step built
    with lm="w4"."""
    V, D = w_lm.shape
    w4 = torch.empty(jet.jet_w4_bytes(V, D), dtype=torch.uint8, device=w_lm.device)
    w_scale = torch.empty(V, dtype=torch.float32, device=w_lm.device)
    jet.jet_quantize_w4(w_lm, w4, w_scale, stream=stream)
    return w4, w_scale


def quantize_lm_head_mxfp8(w_lm: torch.Tensor, stream=None):
    """MXFP8 codes and block scale factors (uint8, jet_mxfp8_bytes(V, D) bytes)
    of the bf16 LM-head weights (jet_quantize_mxfp8), for a step built with
    lm="mxfp8"."""
    V, D = w_lm.shape
    w_mx = torch.empty(jet.jet_mxfp8_bytes(V, D), dtype=torch.uint8, device=w_lm.device)
    jet.jet_quantize_mxfp8(w_lm, w_mx, stream=stream)
    return w_mx


class ScoringStep:
    """Device state of one batch shape.

    ``layout`` is a :class:`jet.HostLayout`; ``dims`` a :class:`jet.jet_dims`;
    ``mode`` one of ``jet.DECIDE_*``. ``hybrid`` adds the linear-attention
    fork; ``keep_fork_state`` also writes every candidate's final recurrent
    state. ``chain`` feeds the attention output to the LM head (requires
    Hq * d == D). ``lm`` selects the LM head: "bf16" (w_lm is the bf16 weight
    matrix), "e4m3" (w_lm is the pair returned by :func:`quantize_lm_head`) or
    "w4" (the pair returned by :func:`quantize_lm_head_w4`) or "mxfp8" (the
    buffer returned by :func:`quantize_lm_head_mxfp8`).
    ``rule`` selects the fork's recurrence: "delta" (gated delta rule) or "gla"
    (plain gated linear attention).
    """

    def __init__(self, layout: "jet.HostLayout", dims: "jet.jet_dims", mode: int,
                 device="cuda", hybrid: bool = False, keep_fork_state: bool = False,
                 chain: bool = False, lm: str = "bf16", rule: str = "delta"):
        if lm not in ("bf16", "e4m3", "w4", "mxfp8"):
            raise ValueError("lm must be 'bf16', 'e4m3', 'w4' or 'mxfp8'")
        self.lm = lm
        self.rule = jet.RULES[rule]
        self.dev = torch.device(device)
        self.host_layout = layout
        self.layout = layout.to_device(self.dev)
        self.dims, self.mode, self.hybrid, self.chain = dims, int(mode), hybrid, chain
        n = layout.sizes
        self.R, self.C, self.N, self.T = n.R, n.C, n.N, n.T
        self.F = n.N - n.R
        if chain and dims.Hq * dims.d != dims.D:
            raise ValueError("chain needs Hq * d == D")
        dt = _TORCH_DTYPE[dims.dtype]
        z = lambda *s, dtype=torch.float32: torch.empty(*s, dtype=dtype, device=self.dev)  # noqa: E731
        self.o = z(n.N, dims.Hq, dims.d, dtype=dt)
        # the results share one device buffer, so that they return in one copy
        self._result_offsets, rb = _pack_plan([
            ("tok_logprob", torch.float32, (n.T,)), ("cand_score", torch.float32, (n.C,)),
            ("q_cand", torch.float32, (n.C,)), ("choice", torch.int32, (n.R,)),
            ("value", torch.float32, (n.R,))])
        self._results = z(rb, dtype=torch.uint8)
        self._bind_results(self._results)
        ws = {"bf16": jet.jet_workspace_bytes, "e4m3": jet.jet_workspace_bytes_e4m3,
              "w4": jet.jet_workspace_bytes_e4m3,
              "mxfp8": jet.jet_workspace_bytes_mxfp8}[lm](n, dims)
        self.ws = z((ws + 15) // 16 * 4)  # float32 words, 16-byte multiple
        if hybrid:
            self.lo = z(self.F, dims.Hl, dims.dv, dtype=dt)
            self.s_fork = z(n.C, dims.Hl, dims.dk, dims.dv) if keep_fork_state else None
        self._dev_inputs: Optional[Dict[str, torch.Tensor]] = None
        self.overlap_min_bytes = _OVERLAP_MIN_BYTES

    def _bind_results(self, buf: torch.Tensor) -> None:
        """Point tok_logprob, cand_score, q_cand, choice and value at ``buf``
        (views made once per buffer: this runs once per pipelined batch)."""
        if getattr(self, "_bound", None) is buf:
            return
        cache = self.__dict__.setdefault("_result_views", {})
        views = cache.get(buf.data_ptr())
        if views is None:
            views = cache[buf.data_ptr()] = (buf, _views(buf, self._result_offsets))
        for k, t in views[1].items():
            setattr(self, k, t)
        self._bound = buf

    # ------------------------------------------------------------------
    def run(self, x: Dict[str, torch.Tensor], w_lm: torch.Tensor, stream=None,
            layout: Optional["jet.DeviceLayout"] = None) -> None:
        """Enqueue the whole step on ``stream`` (default: the current stream).

        ``x`` holds q, k_pre, v_pre, k_cand, v_cand, hidden (unless chained)
        and, for a hybrid step, s_prefix, lq, lk, lv, alpha, beta. ``layout``
        (default: the step's own) must have this step's sizes.
        """
        d = self.dims
        lay = self.layout if layout is None else layout
        jet.jet_prefix_attend(lay, d, x["q"], x["k_pre"], x["v_pre"], x["k_cand"], x["v_cand"],
                              self.o, self.ws, stream=stream)
        if self.hybrid:
            jet.jet_fork_state(lay, d, x["s_prefix"], x["lq"], x["lk"], x["lv"], x["alpha"],
                               x["beta"], self.lo, self.s_fork, stream=stream, rule=self.rule)
        hidden = self.o.view(self.N, d.Hq * d.d) if self.chain else x["hidden"]
        self.score(hidden, w_lm, stream=stream, layout=lay)
        jet.jet_decide(lay, self.mode, self.cand_score, self.q_cand, self.choice, self.value,
                       stream=stream)

    def score(self, hidden: torch.Tensor, w_lm, stream=None, layout=None) -> None:
        """The LM-head call of the step (bf16, e4m3, w4 or mxfp8, as the step was built)."""
        lay = self.layout if layout is None else layout
        if self.lm == "mxfp8":
            jet.jet_score_candidates_mxfp8(lay, self.dims, hidden, w_lm, self.tok_logprob,
                                           self.cand_score, self.ws, stream=stream)
        elif self.lm == "w4":
            w4, w_scale = w_lm
            jet.jet_score_candidates_w4(lay, self.dims, hidden, w4, w_scale, self.tok_logprob,
                                        self.cand_score, self.ws, stream=stream)
        elif self.lm == "e4m3":
            w_q, w_scale = w_lm
            jet.jet_score_candidates_e4m3(lay, self.dims, hidden, w_q, w_scale, self.tok_logprob,
                                          self.cand_score, self.ws, stream=stream)
        else:
            jet.jet_score_candidates(lay, self.dims, hidden, w_lm, self.tok_logprob,
                                     self.cand_score, self.ws, stream=stream)

    def input_names(self):
        names = list(ATTN_INPUTS) + ([] if self.chain else ["hidden"])
        return names + (list(FORK_INPUTS) if self.hybrid else [])

    def run_from_host(self, host: Dict[str, torch.Tensor], layout_words: torch.Tensor,
                      w_lm: torch.Tensor, out: Dict[str, torch.Tensor], stream=None) -> None:
        """End-to-end step: copy the batch's pinned host inputs (and its layout
        words) to the device, run the step, copy the results into the pinned
        host tensors of ``out`` (tok_logprob, cand_score, q_cand, choice,
        value). Everything is enqueued on ``stream``; the caller synchronises."""
        s = torch.cuda.current_stream(self.dev) if stream is None else stream
        with torch.cuda.stream(s):
            if self._dev_inputs is None:
                self._dev_inputs = {k: torch.empty_like(host[k], device=self.dev)
                                    for k in self.input_names()}
            self.layout.words.copy_(layout_words, non_blocking=True)
            for k in self.input_names():
                self._dev_inputs[k].copy_(host[k], non_blocking=True)
            self.run(self._dev_inputs, w_lm, stream=s)
            for k in RESULTS:
                out[k].copy_(getattr(self, k), non_blocking=True)

    def run_pipelined(self, batches, w_lm: torch.Tensor, outs, stream=None) -> None:
        """End to end over a sequence of batches of this step's shape: the
        host -> device copies of batch i+1 run on a copy stream while the
        kernels of batch i run on ``stream``; device inputs and layouts are
        double-buffered. ``batches`` yields :class:`HostBatch` objects (one
        copy each) or (pinned host inputs, pinned layout words) pairs;
        ``outs[i]`` receives batch i's results: a :class:`HostResults` (one
        copy, from a device buffer per pipeline slot, on a third stream, so the
        compute stream runs batch after batch without waiting for it; the
        step's own result tensors are then left untouched) or a dict of pinned
        tensors (copied from the step's result tensors on ``stream``).
        Everything is enqueued; ``stream`` ends after the last copy back, and
        the caller synchronises."""
        s = torch.cuda.current_stream(self.dev) if stream is None else stream
        if getattr(self, "_pipe", None) is None:
            self._copy_stream = torch.cuda.Stream(self.dev)
            self._out_stream = torch.cuda.Stream(self.dev)
            self._pipe = []
            for _ in range(2):
                words = torch.empty_like(self.layout.words)
                self._pipe.append(dict(
                    layout=jet.DeviceLayout(self.layout.sizes, words), inputs=None,
                    copied=torch.cuda.Event(), consumed=torch.cuda.Event(),
                    results=torch.empty_like(self._results), scored=torch.cuda.Event(),
                    read=torch.cuda.Event()))
        cs, os_ = self._copy_stream, self._out_stream
        start = torch.cuda.Event()
        start.record(s)
        cs.wait_event(start)  # after everything already enqueued on ``stream``
        os_.wait_event(start)
        own = self._results
        for i, batch in enumerate(batches):
            buf = self._pipe[i % 2]
            packed = isinstance(batch, HostBatch)
            nbytes = batch.nbytes if packed else self.host_bytes(*batch)[0]
            # a batch whose copies take a few microseconds gains nothing from
            # the overlap and would pay the two cross-stream waits: copy in order
            overlap = nbytes >= self.overlap_min_bytes
            with torch.cuda.stream(cs if overlap else s):
                if overlap and i >= 2:
                    cs.wait_event(buf["consumed"])  # batch i-2's kernels are done with it
                if packed:
                    if buf.get("packed") is None or buf["packed"].numel() != nbytes:
                        buf["packed"] = torch.empty(nbytes, dtype=torch.uint8, device=self.dev)
                        v = _views(buf["packed"], batch.offsets)
                        buf["packed_layout"] = jet.DeviceLayout(self.layout.sizes,
                                                                v.pop("__words__"))
                        buf["packed_inputs"] = v
                    buf["packed"].copy_(batch.buf, non_blocking=True)
                    inputs, layout = buf["packed_inputs"], buf["packed_layout"]
                else:
                    host, layout_words = batch
                    if buf["inputs"] is None:
                        buf["inputs"] = {k: torch.empty_like(host[k], device=self.dev)
                                         for k in self.input_names()}
                    buf["layout"].words.copy_(layout_words, non_blocking=True)
                    for k in self.input_names():
                        buf["inputs"][k].copy_(host[k], non_blocking=True)
                    inputs, layout = buf["inputs"], buf["layout"]
                if overlap:
                    buf["copied"].record(cs)
            if overlap:
                s.wait_event(buf["copied"])
            # a batch small enough to copy in order returns its results in order too
            packed_out = isinstance(outs[i], HostResults) and overlap
            if packed_out:
                # the results of batch i go to this slot's own device buffer and
                # back on a third stream, off the compute stream: batch i+1's
                # kernels follow batch i's directly
                if i >= 2:
                    s.wait_event(buf["read"])  # batch i-2's results have left
                self._bind_results(buf["results"])
            else:
                self._bind_results(own)
            self.run(inputs, w_lm, stream=s, layout=layout)
            buf["consumed"].record(s)
            if packed_out:
                buf["scored"].record(s)
                os_.wait_event(buf["scored"])
                with torch.cuda.stream(os_):
                    outs[i].buf.copy_(buf["results"], non_blocking=True)
                buf["read"].record(os_)
            else:
                with torch.cuda.stream(s):
                    if isinstance(outs[i], HostResults):
                        outs[i].buf.copy_(own, non_blocking=True)
                    else:
                        for k in RESULTS:
                            outs[i][k].copy_(getattr(self, k), non_blocking=True)
        self._bind_results(own)
        s.wait_stream(os_)  # the caller's synchronisation covers the last copies

    def host_bytes(self, host: Dict[str, torch.Tensor], layout_words: torch.Tensor):
        """(host->device, device->host) bytes one :meth:`run_from_host` moves."""
        h2d = layout_words.numel() * layout_words.element_size()
        h2d += sum(host[k].numel() * host[k].element_size() for k in self.input_names())
        d2h = sum(getattr(self, k).numel() * getattr(self, k).element_size() for k in RESULTS)
        return h2d, d2h


class DecoderStack:
    """A hybrid decoder stack's device tensors and workspace for one batch
    shape. ``layers`` is a list of dicts: kind ("linear" or "full") and the
    tensors g1, g2, w_mix, w_o, w_gu, w_d and k_pre/v_pre (full) or s_prefix
    (linear), already on the device."""

    def __init__(self, layout: "jet.HostLayout", dims: "jet.jet_dims", layers, Dff: int,
                 rule: str = "delta", device="cuda"):
        self.dev = torch.device(device)
        self.layout = layout.to_device(self.dev)
        self.dims = dims
        self.layers = [dict(L, kind=jet.LAYER_FULL if L["kind"] == "full" else jet.LAYER_LINEAR)
                       for L in layers]
        self.stack, self._keep = jet.make_stack(self.layers, Dff, jet.RULES[rule])
        n = layout.sizes
        self.N = n.N
        wsb = jet.jet_stack_workspace_bytes(n, dims, Dff)
        if wsb == 0:
            raise ValueError("invalid stack sizes")
        self.ws = torch.empty((wsb + 15) // 16 * 4, dtype=torch.float32, device=self.dev)
        self.x = torch.empty(n.N, dims.D, dtype=torch.bfloat16, device=self.dev)

    def forward(self, x0: torch.Tensor, stream=None, layout=None) -> torch.Tensor:
        """Enqueue the stack on ``stream``; returns the output rows [N, D]."""
        lay = self.layout if layout is None else layout
        jet.jet_stack_forward(lay, self.dims, self.stack, x0, self.x, self.ws, stream=stream)
        return self.x

