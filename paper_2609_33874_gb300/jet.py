"""ctypes binding of libjet (the C ABI declared in ``include/jet.h``).

The functions keep the C names (``jet_layout_build``, ``jet_prefix_attend``,
``jet_fork_state``, ``jet_score_candidates``, ``jet_decide`` ...) and only
marshal arguments: every step of the scoring path runs in the library's CUDA
kernels. Tensor arguments are torch tensors on a CUDA device (or raw device
addresses as ints); torch supplies device memory and streams only. A nonzero
status raises :class:`JetError`. If the library has not been built the import
of this module fails loudly; there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libjet.so")

JET_OK = 0
STATUS_NAMES = {0: "JET_OK", 1: "JET_ERR_ARG", 2: "JET_ERR_SHAPE", 3: "JET_ERR_RANGE",
                4: "JET_ERR_ALIGN", 5: "JET_ERR_WORKSPACE", 6: "JET_ERR_CAPACITY",
                7: "JET_ERR_UNSUPPORTED", 8: "JET_ERR_CUDA", 9: "JET_ERR_TIMEOUT",
                10: "JET_ERR_DEVICE"}
DTYPE_F32, DTYPE_BF16 = 0, 1
DECIDE_ARGMAX, DECIDE_BINARY, DECIDE_ORDINAL = 0, 1, 2
MODES = {"argmax": DECIDE_ARGMAX, "binary": DECIDE_BINARY, "ordinal": DECIDE_ORDINAL}
RECUR_DELTA, RECUR_GLA = 0, 1
RULES = {"delta": RECUR_DELTA, "gla": RECUR_GLA}


class JetError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)} "
                         f"({_lib.jet_status_string(status).decode()})")


# ---------------------------------------------------------------------------
# C structs
# ---------------------------------------------------------------------------
class jet_sizes(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("R", "C", "N", "T", "V", "total_prefix", "max_prefix", "min_cand",
                 "max_cand", "max_rows", "max_len", "reserved")]


_ARRAYS = ("prefix_offset", "cand_offset", "row_offset", "cand_row_offset", "tgt_offset",
           "target_ids", "tgt_row", "row_req", "row_cand", "row_pos", "row_tgt_offset",
           "row_tgt_index", "req_order")


class jet_layout(ctypes.Structure):
    _fields_ = [("n", jet_sizes)] + [(a, ctypes.c_void_p) for a in _ARRAYS]


class jet_dims(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("dtype", "Hq", "Hkv", "d", "D", "Hl", "dk", "dv",
                                              "max_sms")]


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libjet.so is not built ({LIB_PATH}); run "
                          "`python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(LIB_PATH)
    P, I, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    i32p = ctypes.POINTER(ctypes.c_int32)
    sig = {
        "jet_abi_version": (I, []),
        "jet_status_string": (ctypes.c_char_p, [I]),
        "jet_layout_plan": (I, [I, i32p, i32p, i32p, I, ctypes.POINTER(jet_sizes)]),
        "jet_layout_words": (SZ, [ctypes.POINTER(jet_sizes)]),
        "jet_layout_build": (I, [I, i32p, i32p, i32p, i32p, I, i32p, SZ,
                                 ctypes.POINTER(jet_layout)]),
        "jet_layout_bind": (I, [ctypes.POINTER(jet_sizes), P, ctypes.POINTER(jet_layout)]),
        "jet_workspace_bytes": (SZ, [ctypes.POINTER(jet_sizes), ctypes.POINTER(jet_dims)]),
        "jet_prefix_attend": (I, [ctypes.POINTER(jet_layout), ctypes.POINTER(jet_dims),
                                  P, P, P, P, P, P, P, SZ, P]),
        "jet_prefill_workspace_bytes": (SZ, [ctypes.POINTER(jet_sizes),
                                             ctypes.POINTER(jet_dims)]),
        "jet_prefill_attend": (I, [ctypes.POINTER(jet_layout), ctypes.POINTER(jet_dims),
                                   P, P, P, P, P, SZ, P]),
        "jet_prefill_state": (I, [ctypes.POINTER(jet_layout), ctypes.POINTER(jet_dims), I,
                                  P, P, P, P, P, P, P, P, P]),
        "jet_fork_state": (I, [ctypes.POINTER(jet_layout), ctypes.POINTER(jet_dims),
                               P, P, P, P, P, P, P, P, P]),
        "jet_fork_state_rule": (I, [ctypes.POINTER(jet_layout), ctypes.POINTER(jet_dims), I,
                                    P, P, P, P, P, P, P, P, P]),
        "jet_score_candidates": (I, [ctypes.POINTER(jet_layout), ctypes.POINTER(jet_dims),
                                     P, P, P, P, P, SZ, P]),
        "jet_score_candidates_noalloc": (I, [ctypes.POINTER(jet_layout), ctypes.POINTER(jet_dims),
                                             P, P, P, P, P]),
        "jet_quantize_rows_e4m3": (I, [P, I, I, P, P, P]),
        "jet_workspace_bytes_e4m3": (SZ, [ctypes.POINTER(jet_sizes), ctypes.POINTER(jet_dims)]),
        "jet_score_candidates_e4m3": (I, [ctypes.POINTER(jet_layout), ctypes.POINTER(jet_dims),
                                          P, P, P, P, P, P, SZ, P]),
        "jet_w4_bytes": (SZ, [ctypes.c_int64, ctypes.c_int64]),
        "jet_quantize_w4": (I, [P, ctypes.c_int64, ctypes.c_int64, P, P, P]),
        "jet_score_candidates_w4": (I, [ctypes.POINTER(jet_layout), ctypes.POINTER(jet_dims),
                                        P, P, P, P, P, P, SZ, P]),
        "jet_mxfp8_bytes": (SZ, [ctypes.c_int64, ctypes.c_int64]),
        "jet_quantize_mxfp8": (I, [P, ctypes.c_int64, ctypes.c_int64, P, P]),
        "jet_workspace_bytes_mxfp8": (SZ, [ctypes.POINTER(jet_sizes), ctypes.POINTER(jet_dims)]),
        "jet_score_candidates_mxfp8": (I, [ctypes.POINTER(jet_layout), ctypes.POINTER(jet_dims),
                                           P, P, P, P, P, SZ, P]),
        "jet_stack_workspace_bytes": (SZ, [ctypes.POINTER(jet_sizes), ctypes.POINTER(jet_dims),
                                           I]),
        "jet_stack_forward": (I, [ctypes.POINTER(jet_layout), ctypes.POINTER(jet_dims),
                                  P, P, P, P, SZ, P]),
        "jet_decide": (I, [ctypes.POINTER(jet_layout), I, P, P, P, P, P]),
        "jet_evaluate": (I, [ctypes.POINTER(jet_layout), P, P, P, P, P, P]),
        "jet_device_status": (I, [P, ctypes.POINTER(ctypes.c_int32)]),
        "jet_set_wait_budget_ns": (ctypes.c_uint64, [ctypes.c_uint64]),
        "jet_launch_count": (ctypes.c_uint64, []),
        "jet_set_test_stall": (I, [I]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = _load()
DECLARED = ("jet_abi_version", "jet_status_string", "jet_layout_plan", "jet_layout_words",
            "jet_layout_build", "jet_layout_bind", "jet_workspace_bytes", "jet_prefix_attend",
            "jet_prefill_workspace_bytes", "jet_prefill_attend", "jet_prefill_state",
            "jet_fork_state", "jet_fork_state_rule", "jet_score_candidates", "jet_score_candidates_noalloc",
            "jet_quantize_rows_e4m3", "jet_workspace_bytes_e4m3", "jet_score_candidates_e4m3",
            "jet_w4_bytes", "jet_quantize_w4", "jet_score_candidates_w4",
            "jet_mxfp8_bytes", "jet_quantize_mxfp8", "jet_workspace_bytes_mxfp8",
            "jet_score_candidates_mxfp8",
            "jet_stack_workspace_bytes", "jet_stack_forward", "jet_decide", "jet_evaluate", "jet_device_status",
            "jet_set_wait_budget_ns", "jet_launch_count", "jet_set_test_stall")


def library() -> ctypes.CDLL:
    return _lib


def _check(status: int, where: str) -> None:
    if status != JET_OK:
        raise JetError(status, where)


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _ptr32(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


def _addr(x) -> Optional[int]:
    """Device address of a tensor (or an int address); None for None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if not x.is_contiguous():
        raise ValueError("tensor arguments must be contiguous")
    return x.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ---------------------------------------------------------------------------
# layout
# ---------------------------------------------------------------------------
class HostLayout:
    """A layout built on the host: sizes, the packed int32 words and the bound struct."""

    def __init__(self, sizes: jet_sizes, words: np.ndarray, struct: jet_layout):
        self.sizes, self.words, self.struct = sizes, words, struct

    def array(self, name: str) -> np.ndarray:
        """A copy of one layout array (int32)."""
        n = self.sizes
        lens = {"prefix_offset": n.R + 1, "cand_offset": n.R + 1, "row_offset": n.R + 1,
                "cand_row_offset": n.C + 1, "tgt_offset": n.C + 1, "target_ids": n.T,
                "tgt_row": n.T, "row_req": n.N, "row_cand": n.N, "row_pos": n.N,
                "row_tgt_offset": n.N + 1, "row_tgt_index": n.T, "req_order": n.R}
        off = (getattr(self.struct, name) - self.words.ctypes.data) // 4
        return self.words[off:off + lens[name]].copy()

    def to_device(self, device=None) -> "DeviceLayout":
        import torch
        dev = torch.device("cuda") if device is None else torch.device(device)
        words = torch.from_numpy(self.words).to(dev)
        return DeviceLayout(self.sizes, words)


class DeviceLayout:
    """The same words copied to a device and bound (``jet_layout_bind``)."""

    def __init__(self, sizes: jet_sizes, words):
        self.sizes = sizes
        self.words = words  # keeps the device buffer alive
        self.struct = jet_layout()
        _check(_lib.jet_layout_bind(ctypes.byref(sizes), ctypes.c_void_p(words.data_ptr()),
                                    ctypes.byref(self.struct)), "jet_layout_bind")


def jet_layout_plan(prefix_len, n_cand, cand_len, V: int) -> jet_sizes:
    p, c, m = _i32(prefix_len), _i32(n_cand), _i32(cand_len)
    out = jet_sizes()
    _check(_lib.jet_layout_plan(len(p), _ptr32(p), _ptr32(c), _ptr32(m), int(V),
                                ctypes.byref(out)), "jet_layout_plan")
    return out


def jet_layout_words(sizes: jet_sizes) -> int:
    return int(_lib.jet_layout_words(ctypes.byref(sizes)))


def jet_layout_build(prefix_len, n_cand, cand_len, target_ids, V: int) -> HostLayout:
    p, c, m, y = _i32(prefix_len), _i32(n_cand), _i32(cand_len), _i32(target_ids)
    sizes = jet_layout_plan(p, c, m, V)
    words = np.zeros(max(1, jet_layout_words(sizes)), dtype=np.int32)
    struct = jet_layout()
    _check(_lib.jet_layout_build(len(p), _ptr32(p), _ptr32(c), _ptr32(m), _ptr32(y), int(V),
                                 _ptr32(words), words.size, ctypes.byref(struct)),
           "jet_layout_build")
    return HostLayout(sizes, words, struct)


LAYER_LINEAR, LAYER_FULL = 0, 1


class jet_stack_layer(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("reserved", ctypes.c_int32)] + [
        (n, ctypes.c_void_p) for n in ("g1", "g2", "w_mix", "w_o", "w_gu", "w_d", "k_pre",
                                       "v_pre", "s_prefix")]


class jet_stack(ctypes.Structure):
    _fields_ = [("L", ctypes.c_int32), ("Dff", ctypes.c_int32), ("rule", ctypes.c_int32),
                ("reserved", ctypes.c_int32), ("layers", ctypes.POINTER(jet_stack_layer))]


def make_stack(layers, Dff: int, rule: int = 0):
    """A jet_stack over a list of dicts (kind, g1, g2, w_mix, w_o, w_gu, w_d,
    and k_pre/v_pre or s_prefix as tensors); returns (struct, keep-alive)."""
    arr = (jet_stack_layer * max(1, len(layers)))()
    for i, Ly in enumerate(layers):
        arr[i].kind = int(Ly["kind"])
        for n in ("g1", "g2", "w_mix", "w_o", "w_gu", "w_d", "k_pre", "v_pre", "s_prefix"):
            setattr(arr[i], n, _addr(Ly.get(n)))
    st = jet_stack(len(layers), int(Dff), int(rule), 0,
                   ctypes.cast(arr, ctypes.POINTER(jet_stack_layer)))
    return st, arr


def make_dims(dtype: int, Hq=0, Hkv=0, d=0, D=0, Hl=0, dk=0, dv=0, max_sms=0) -> jet_dims:
    return jet_dims(int(dtype), int(Hq), int(Hkv), int(d), int(D), int(Hl), int(dk), int(dv),
                    int(max_sms))


def jet_workspace_bytes(sizes: jet_sizes, dims: jet_dims) -> int:
    return int(_lib.jet_workspace_bytes(ctypes.byref(sizes), ctypes.byref(dims)))


# ---------------------------------------------------------------------------
# compute entry points
# ---------------------------------------------------------------------------
def _lay(layout) -> jet_layout:
    return layout.struct if isinstance(layout, (DeviceLayout, HostLayout)) else layout


def jet_prefix_attend(layout, dims: jet_dims, q, k_pre, v_pre, k_cand, v_cand, o, ws,
                      ws_bytes: Optional[int] = None, stream=None) -> None:
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    _check(_lib.jet_prefix_attend(ctypes.byref(_lay(layout)), ctypes.byref(dims), _addr(q),
                                  _addr(k_pre), _addr(v_pre), _addr(k_cand), _addr(v_cand),
                                  _addr(o), _addr(ws), int(ws_bytes), _stream(stream)),
           "jet_prefix_attend")


def jet_prefill_workspace_bytes(sizes: jet_sizes, dims: jet_dims) -> int:
    return int(_lib.jet_prefill_workspace_bytes(ctypes.byref(sizes), ctypes.byref(dims)))


def jet_prefill_attend(layout, dims: jet_dims, q, k, v, o, ws, ws_bytes: Optional[int] = None,
                       stream=None) -> None:
    """Causal self-attention over every request's prefix (see include/jet.h)."""
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    _check(_lib.jet_prefill_attend(ctypes.byref(_lay(layout)), ctypes.byref(dims), _addr(q),
                                   _addr(k), _addr(v), _addr(o), _addr(ws), int(ws_bytes),
                                   _stream(stream)), "jet_prefill_attend")


def jet_prefill_state(layout, dims: jet_dims, q, k, v, alpha, beta, o, s_out, s_init=None,
                      rule: int = 0, stream=None) -> None:
    """The prefix scan of the recurrent state (see include/jet.h)."""
    _check(_lib.jet_prefill_state(ctypes.byref(_lay(layout)), ctypes.byref(dims), int(rule),
                                  _addr(s_init), _addr(q), _addr(k), _addr(v), _addr(alpha),
                                  _addr(beta), _addr(o), _addr(s_out), _stream(stream)),
           "jet_prefill_state")


def jet_fork_state(layout, dims: jet_dims, s_prefix, q, k, v, alpha, beta, o, s_fork=None,
                   stream=None, rule: int = None) -> None:
    """The fork with the gated delta rule, or with the recurrence `rule`
    (RECUR_DELTA or RECUR_GLA) through jet_fork_state_rule."""
    if rule is None:
        _check(_lib.jet_fork_state(ctypes.byref(_lay(layout)), ctypes.byref(dims),
                                   _addr(s_prefix), _addr(q), _addr(k), _addr(v), _addr(alpha),
                                   _addr(beta), _addr(o), _addr(s_fork), _stream(stream)),
               "jet_fork_state")
        return
    _check(_lib.jet_fork_state_rule(ctypes.byref(_lay(layout)), ctypes.byref(dims), int(rule),
                                    _addr(s_prefix), _addr(q), _addr(k), _addr(v), _addr(alpha),
                                    _addr(beta), _addr(o), _addr(s_fork), _stream(stream)),
           "jet_fork_state_rule")


def jet_score_candidates(layout, dims: jet_dims, hidden, w_lm, tok_logprob, cand_score, ws,
                         ws_bytes: Optional[int] = None, stream=None) -> None:
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    _check(_lib.jet_score_candidates(ctypes.byref(_lay(layout)), ctypes.byref(dims),
                                     _addr(hidden), _addr(w_lm), _addr(tok_logprob),
                                     _addr(cand_score), _addr(ws), int(ws_bytes),
                                     _stream(stream)), "jet_score_candidates")


def jet_score_candidates_noalloc(layout, dims: jet_dims, hidden, w_lm, tok_logprob, cand_score,
                                 stream=None) -> None:
    """jet_score_candidates with the library's own fixed scratch array, for
    callers that cannot allocate device memory (see include/jet.h)."""
    _check(_lib.jet_score_candidates_noalloc(ctypes.byref(_lay(layout)), ctypes.byref(dims),
                                             _addr(hidden), _addr(w_lm), _addr(tok_logprob),
                                             _addr(cand_score), _stream(stream)),
           "jet_score_candidates_noalloc")


def jet_quantize_rows_e4m3(x, q, scale, stream=None) -> None:
    """Per-row e4m3 codes q [rows, D] uint8 and scales [rows] float32 of the
    bf16 matrix x [rows, D] (see include/jet.h)."""
    rows, D = (int(x.shape[0]), int(x.shape[1])) if x.dim() == 2 else (0, 0)
    _check(_lib.jet_quantize_rows_e4m3(_addr(x), rows, D, _addr(q), _addr(scale),
                                       _stream(stream)), "jet_quantize_rows_e4m3")


def jet_workspace_bytes_e4m3(sizes: jet_sizes, dims: jet_dims) -> int:
    return int(_lib.jet_workspace_bytes_e4m3(ctypes.byref(sizes), ctypes.byref(dims)))


def jet_score_candidates_e4m3(layout, dims: jet_dims, hidden, w_q, w_scale, tok_logprob,
                              cand_score, ws, ws_bytes: Optional[int] = None, stream=None) -> None:
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    _check(_lib.jet_score_candidates_e4m3(ctypes.byref(_lay(layout)), ctypes.byref(dims),
                                          _addr(hidden), _addr(w_q), _addr(w_scale),
                                          _addr(tok_logprob), _addr(cand_score), _addr(ws),
                                          int(ws_bytes), _stream(stream)),
           "jet_score_candidates_e4m3")


def jet_w4_bytes(V: int, D: int) -> int:
    """Bytes of the 4-bit codes and scale factors of a [V, D] matrix (0 if invalid)."""
    return int(_lib.jet_w4_bytes(int(V), int(D)))


def jet_quantize_w4(w, w4, scale, stream=None) -> None:
    """4-bit codes and block scale factors w4 (jet_w4_bytes(V, D) bytes) and
    row scales [V] float32 of the bf16 matrix w [V, D] (see include/jet.h)."""
    V, D = (int(w.shape[0]), int(w.shape[1])) if w.dim() == 2 else (0, 0)
    _check(_lib.jet_quantize_w4(_addr(w), V, D, _addr(w4), _addr(scale), _stream(stream)),
           "jet_quantize_w4")


def jet_score_candidates_w4(layout, dims: jet_dims, hidden, w4, w_scale, tok_logprob,
                            cand_score, ws, ws_bytes: Optional[int] = None, stream=None) -> None:
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    _check(_lib.jet_score_candidates_w4(ctypes.byref(_lay(layout)), ctypes.byref(dims),
                                        _addr(hidden), _addr(w4), _addr(w_scale),
                                        _addr(tok_logprob), _addr(cand_score), _addr(ws),
                                        int(ws_bytes), _stream(stream)),
           "jet_score_candidates_w4")


def jet_mxfp8_bytes(V: int, D: int) -> int:
    """Bytes of the MXFP8 codes and scale factors of a [V, D] matrix (0 if invalid)."""
    return int(_lib.jet_mxfp8_bytes(int(V), int(D)))


def jet_quantize_mxfp8(w, out, stream=None) -> None:
    """MXFP8 codes and block scale factors (jet_mxfp8_bytes(V, D) bytes) of the
    bf16 matrix w [V, D] (see include/jet.h)."""
    V, D = (int(w.shape[0]), int(w.shape[1])) if w.dim() == 2 else (0, 0)
    _check(_lib.jet_quantize_mxfp8(_addr(w), V, D, _addr(out), _stream(stream)),
           "jet_quantize_mxfp8")


def jet_workspace_bytes_mxfp8(sizes: jet_sizes, dims: jet_dims) -> int:
    return int(_lib.jet_workspace_bytes_mxfp8(ctypes.byref(sizes), ctypes.byref(dims)))


def jet_score_candidates_mxfp8(layout, dims: jet_dims, hidden, w_mx, tok_logprob, cand_score,
                               ws, ws_bytes: Optional[int] = None, stream=None) -> None:
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    _check(_lib.jet_score_candidates_mxfp8(ctypes.byref(_lay(layout)), ctypes.byref(dims),
                                           _addr(hidden), _addr(w_mx), _addr(tok_logprob),
                                           _addr(cand_score), _addr(ws), int(ws_bytes),
                                           _stream(stream)),
           "jet_score_candidates_mxfp8")


def jet_stack_workspace_bytes(sizes: jet_sizes, dims: jet_dims, Dff: int) -> int:
    return int(_lib.jet_stack_workspace_bytes(ctypes.byref(sizes), ctypes.byref(dims), int(Dff)))


def jet_stack_forward(layout, dims: jet_dims, stack, x0, x, ws, ws_bytes: Optional[int] = None,
                      stream=None) -> None:
    """x = the decoder stack applied to x0 (see include/jet.h); ``stack`` is
    the struct returned by :func:`make_stack`."""
    ws_bytes = ws.numel() * ws.element_size() if ws_bytes is None else ws_bytes
    _check(_lib.jet_stack_forward(ctypes.byref(_lay(layout)), ctypes.byref(dims),
                                  ctypes.byref(stack), _addr(x0), _addr(x), _addr(ws),
                                  int(ws_bytes), _stream(stream)), "jet_stack_forward")


def jet_decide(layout, mode: int, cand_score, q, choice, value, stream=None) -> None:
    _check(_lib.jet_decide(ctypes.byref(_lay(layout)), int(mode), _addr(cand_score), _addr(q),
                           _addr(choice), _addr(value), _stream(stream)), "jet_decide")


def jet_evaluate(layout, cand_score, choice, gold, nll, correct, stream=None) -> None:
    """Gold NLL over equivalent labels and agreement of the choice (see include/jet.h)."""
    _check(_lib.jet_evaluate(ctypes.byref(_lay(layout)), _addr(cand_score), _addr(choice),
                             _addr(gold), _addr(nll), _addr(correct), _stream(stream)),
           "jet_evaluate")


def jet_device_status(stream=None) -> int:
    out = ctypes.c_int32(0)
    _check(_lib.jet_device_status(_stream(stream), ctypes.byref(out)), "jet_device_status")
    return int(out.value)


def jet_set_wait_budget_ns(ns: int) -> int:
    """Budget of one bounded wait in the tensor-core kernels (0: the default
    2 s); returns the previous budget."""
    return int(_lib.jet_set_wait_budget_ns(int(ns)))


def jet_launch_count() -> int:
    """Kernels the library has launched in this process so far."""
    return int(_lib.jet_launch_count())


def jet_set_test_stall(on: bool) -> bool:
    """Test hook: the tensor-core kernels launched while it is on withhold their
    first load, so that a bounded wait runs out; returns the previous setting."""
    return bool(_lib.jet_set_test_stall(1 if on else 0))
