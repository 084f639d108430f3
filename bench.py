#!/usr/bin/env python3
"""Benchmark of the JET candidate-scoring step on GB300.

A step is one pass of the whole hot path - cascade attention, the recurrent
state fork (hybrid workloads), the fused LM head with full-vocabulary
log-sum-exp and target gather, and the decision rules - over one batch of
synthetic requests whose inputs are already resident in HBM. The metric is
candidate sets (requests) scored per second.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--R R]
    python bench.py --impl reference ...   # the fp64 CPU oracle on the host cores

The default workload is the long-context batch (256 requests, prefixes of
2,048-8,192 tokens, 16/2 heads, d 256, D 2,048, V 151,936, bf16): the largest
single-GPU configuration and the one whose LM head is tensor-bound. On one GPU
the same run then times the other four workloads (`per_workload`, each with
its roofline, per-call breakdown and CPU-oracle sample) and the batch-size
sweep R = 1, 2, 4, ..., 128 of the long-context batch (`sweep`); the headline
`value` is the 256-request batch alone.

Under torchrun (N > 1) every rank scores its own batch on its own GPU
(independent replicas, no collective on the data path); rank 0 prints one
JSON line with the whole-job throughput.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

_CORES = os.cpu_count() or 1
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, str(_CORES))

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "candidate sets scored/sec"
UNIT = "sets/s"
DEFAULT_WORKLOAD = "moe_a3b_long"
# the other workloads, timed in the same default run (one GPU)
EXTRA_WORKLOADS = ("tiny", "dense27b_mc", "binary", "ordinal_hybrid")
L2_BYTES = 129 * 1024 * 1024


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(hbm=float(p["hbm_gbs"]), bf16=float(p["bf16_tflops"]),
                    bf16_sustained=float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                    sm_max_mhz=float(p.get("sm_max_mhz", 2070.0)), source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sustained=1700.0, sm_max_mhz=2070.0,
                source="fallback")


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class NvmlClocks:
    """SM clock and clock-event reasons of one GPU, polled every `period_s`
    through read-only NVML queries (clock, maximum clock, event reasons,
    power) from a background thread, so that even a timed region of a few
    tens of milliseconds holds many samples. Changes no setting."""
    REASONS = ((0x4, "sw_power_cap"), (0x8, "hw_slowdown"), (0x20, "sw_thermal_slowdown"),
               (0x40, "hw_thermal_slowdown"), (0x80, "hw_power_brake_slowdown"))

    def __init__(self, uuid: str | None, period_s: float = 0.001):
        import ctypes
        self.period = period_s
        self.samples = []
        self.t_on = self.t_off = None
        self.stop_evt = threading.Event()
        self.thread = None
        self.lib = self.h = None
        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                return
            h = ctypes.c_void_p()
            ok = False
            for cand in ([f"GPU-{uuid}", str(uuid)] if uuid else []):
                if lib.nvmlDeviceGetHandleByUUID(cand.encode(), ctypes.byref(h)) == 0:
                    ok = True
                    break
            if not ok:
                return
            self.reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                getattr(lib, "nvmlDeviceGetCurrentClocksThrottleReasons")
            mx = ctypes.c_uint()
            if lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) != 0:
                return
            self.smax = float(mx.value)
            self.lib, self.h = lib, h
        except (OSError, AttributeError):
            self.lib = None

    @property
    def available(self) -> bool:
        return self.lib is not None

    def start(self):
        if self.available:
            self.thread = threading.Thread(target=self._poll, daemon=True)
            self.thread.start()

    def _poll(self):
        import ctypes
        mhz, rsn, mw = ctypes.c_uint(), ctypes.c_ulonglong(), ctypes.c_uint()
        while not self.stop_evt.is_set():
            t = time.time()
            if self.lib.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(mhz)) == 0 and \
                    self.reasons_fn(self.h, ctypes.byref(rsn)) == 0:
                self.lib.nvmlDeviceGetPowerUsage(self.h, ctypes.byref(mw))
                self.samples.append((t, float(mhz.value), int(rsn.value), mw.value / 1e3))
            time.sleep(self.period)

    def mark(self, on: bool):
        if on:
            self.t_on = time.time()
        else:
            self.t_off = time.time()

    def stop(self):
        if not self.available:
            return None
        self.stop_evt.set()
        if self.thread:
            self.thread.join(timeout=2)
        inside = [x for x in self.samples if self.t_on and self.t_off and
                  self.t_on <= x[0] <= self.t_off]
        window = "timed"
        if not inside:
            inside, window = self.samples, "warmup+timed"
        if not inside:
            return None
        reasons = sorted({name for x in inside for bit, name in self.REASONS if x[2] & bit})
        return dict(sm_mhz=statistics.median(x[1] for x in inside), sm_max_mhz=self.smax,
                    reasons=reasons, samples=len(inside), window=window,
                    power_w_max=round(max(x[3] for x in inside), 1), source="nvml, 1 ms")


class ClockSampler:
    QUERY = ("timestamp,index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.lines = []
        self.proc = None
        self.t_on = self.t_off = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def mark(self, on: bool):
        if on:
            self.t_on = time.time()
        else:
            self.t_off = time.time()

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.15)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        rows = []
        for t, line in self.lines:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 11:
                continue
            if self.uuid and self.uuid not in f[2]:
                continue
            try:
                rows.append(dict(t=t, sm=float(f[3]), smax=float(f[4]), active=f[6],
                                 hw=f[7], hwt=f[8], swt=f[9], swp=f[10]))
            except ValueError:
                continue
        inside = [r for r in rows if self.t_on and self.t_off and self.t_on <= r["t"] <= self.t_off + 0.1]
        window = "timed"
        if not inside:
            inside, window = rows, "warmup+timed"
        if not inside:
            return None
        reasons = set()
        for r in inside:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("swp", "sw_power_cap")):
                if r[key].lower().startswith("active"):
                    reasons.add(name)
        return dict(sm_mhz=statistics.median(r["sm"] for r in inside),
                    sm_max_mhz=max(r["smax"] for r in inside), reasons=sorted(reasons),
                    samples=len(inside), window=window)


# ---------------------------------------------------------------------------
# CPU oracle (baseline and reference arm)
# ---------------------------------------------------------------------------
def oracle_step(problem):
    """The oracle's whole step on one problem: attention, fork, LM head, Eq. 3-5."""
    import oracle as O
    w = problem.work
    lay = O.build_layout(problem.prefix_len, problem.n_cand, problem.cand_len,
                         problem.target_ids, w.V)
    O.cascade_attention(lay, problem.f32("q"), problem.f32("k_pre"), problem.f32("v_pre"),
                        problem.f32("k_cand"), problem.f32("v_cand"), w.Hq, w.Hkv)
    if w.Hl:
        O.fork_state(lay, problem.f32("s_prefix"), problem.f32("lq"), problem.f32("lk"),
                     problem.f32("lv"), problem.f32("alpha"), problem.f32("beta"))
    mode = {"argmax": O.ARGMAX, "binary": O.BINARY, "ordinal": O.ORDINAL}[w.mode]
    return O.score_step(lay, problem.f32("hidden"), problem.f32("w_lm"), mode)


def step_config(args, problem, world: int) -> dict:
    """The `config` of the step's JSON line (both arms): the workload and its sizes."""
    w = problem.work
    es = 2 if w.dtype == "bf16" else 4
    return dict(workload=args.workload, R=problem.R, N=problem.N, T=len(problem.target_ids),
                C=len(problem.cand_len), total_prefix=problem.total_prefix, Hq=w.Hq, Hkv=w.Hkv,
                d=w.d, D=w.D, V=w.V, Hl=w.Hl,
                parallelism=f"replicas{world}" if world > 1 else "single",
                lm_head={"bf16": "bf16",
                         "e4m3": "e4m3, one float32 scale per weight row and per token",
                         "w4": "weights e2m1 with a power-of-two exponent per 32-element "
                               "block and a float32 scale per row; hidden e4m3 per token",
                         "mxfp8": "weights and hidden states e4m3 with a shared power-of-two "
                                  "scale per 32-element block (MXFP8)"}[args.lm],
                recurrence=(args.rule if w.Hl else None),
                l2=f"inputs larger than L2: LM-head weights {w.V * w.D * es / 1e9:.2f} GB "
                   f"streamed every step")


def oracle_sample(name: str, R: int, k: int):
    import jet_synth
    p = jet_synth.make_problem(name, R=min(k, R))
    names = ["q", "k_pre", "v_pre", "k_cand", "v_cand", "hidden", "w_lm"]
    if p.work.Hl:
        names += ["s_prefix", "lq", "lk", "lv", "alpha", "beta"]
    for n in names:  # draw the inputs before timing
        p.f32(n)
    return p


def cpu_baseline(name: str, R: int, k: int):
    p = oracle_sample(name, R, k)
    t0 = time.perf_counter()
    oracle_step(p)
    dt = time.perf_counter() - t0
    return dict(value=p.R / dt, unit=UNIT, cores=_CORES, kind="oracle",
                sample=f"first {p.R} of {R} requests of workload {name}, one pass of the "
                       f"fp64 oracle step ({dt:.1f} s), BLAS threads {_CORES}")


# ---------------------------------------------------------------------------
# helpers
# ---------------------------------------------------------------------------
def _source_hash(files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def _traffic(kernel_file: str, workload: str):
    """DRAM traffic per launch of the dominant kernel from a committed ncu
    summary, if it was taken on the current source of that kernel."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    try:
        with open(path) as f:
            rec = json.load(f).get(workload)
    except (OSError, ValueError):
        return None
    if not rec or rec.get("source_hash") != _source_hash([kernel_file]):
        return None
    return rec.get("bytes_per_launch")


def _call(ms: float, nbytes: int, peaks) -> dict:
    """An HBM-bound call: its time, algorithmic bytes and fraction of the copy peak."""
    gbs = nbytes / (ms / 1e3) / 1e9
    return dict(ms=round(ms, 4), bound="hbm", algorithmic_bytes=int(nbytes),
                achieved_gbs=round(gbs, 1), frac=round(gbs / peaks["hbm"], 4))


def aggregate(total_ms: float, e2e_ms: float, R: int, steps: int, world: int, device=None):
    """Whole-job numbers of N independent replicas: the slowest rank's timed
    regions (max over ranks) and the sets all ranks scored per second.
    Returns (total_ms, e2e_ms, ms_per_step, sets_per_s, e2e_sets_per_s)."""
    if world > 1:
        import torch
        import torch.distributed as dist
        t = torch.tensor([total_ms, e2e_ms], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms, e2e_ms = float(t[0]), float(t[1])
    ms_per_step = total_ms / steps
    return (total_ms, e2e_ms, ms_per_step, R * world / (ms_per_step / 1e3),
            R * world / (e2e_ms / 1e3))


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
def _device_inputs(problem, names, dev, src=None):
    """The step's inputs on the device: drawn for `problem`, or (src given) the
    leading rows of a larger batch's device tensors - a batch of the first R
    requests of a draw is the leading part of every packed input."""
    import jet_synth
    if src is None:
        return {k: jet_synth.torch_tensor(problem, k, device=dev) for k in names}
    P, N, F = problem.total_prefix, problem.N, problem.N - problem.R
    rows = dict(q=N, hidden=N, k_pre=P, v_pre=P, k_cand=F, v_cand=F, lq=F, lk=F, lv=F, alpha=F,
                beta=F, s_prefix=problem.R)
    return {k: src[k][:rows[k]] for k in names}


def _measure(args, problem, dev, stream, peaks, world=1, src=None, w_lm=None, clocks=None,
             e2e=False, evaluate=False):
    """Times `args.steps` scoring steps of `problem` (inputs resident in HBM)
    after `args.warmup` untimed ones, then the per-call breakdown, and returns
    the numbers of one JSON record (the headline line or a `per_workload` /
    `sweep` entry). With e2e the step is also timed end to end from pinned
    host memory."""
    import torch
    import jet_synth
    from paper_2609_33874_gb300 import jet
    from paper_2609_33874_gb300.step import ScoringStep
    w = problem.work
    R = problem.R
    dtype = jet.DTYPE_BF16 if w.dtype == "bf16" else jet.DTYPE_F32
    dims = jet.make_dims(dtype, Hq=w.Hq, Hkv=w.Hkv, d=w.d, D=w.D, Hl=w.Hl, dk=w.dk, dv=w.dv)
    hl = jet.jet_layout_build(problem.prefix_len, problem.n_cand, problem.cand_len,
                              problem.target_ids, w.V)
    low = args.lm != "bf16"   # e4m3 or 4-bit weights, e4m3 hidden states
    step = ScoringStep(hl, dims, jet.MODES[w.mode], device=dev, hybrid=w.Hl > 0,
                       keep_fork_state=w.Hl > 0, lm=args.lm, rule=args.rule)
    names = step.input_names()
    x = _device_inputs(problem, names, dev, src)
    if w_lm is None:
        w_lm = jet_synth.torch_tensor(problem, "w_lm", device=dev)
        if low:
            # model state: the weights are quantised once, outside the timed region
            from paper_2609_33874_gb300.step import (quantize_lm_head, quantize_lm_head_mxfp8,
                                                     quantize_lm_head_w4)
            w_lm = {"w4": quantize_lm_head_w4, "e4m3": quantize_lm_head,
                    "mxfp8": quantize_lm_head_mxfp8}[args.lm](w_lm)
            torch.cuda.synchronize(dev)

    # the per-call breakdown (taken outside the timed steps): attend | fork | score | decide
    call_ev = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(args.steps)]

    def one_step(i=None):
        d, lay = step.dims, step.layout
        ev = call_ev[i] if i is not None else None
        if ev:
            ev[0].record(stream)
        jet.jet_prefix_attend(lay, d, x["q"], x["k_pre"], x["v_pre"], x["k_cand"], x["v_cand"],
                              step.o, step.ws, stream=stream)
        if ev:
            ev[1].record(stream)
        if step.hybrid:
            jet.jet_fork_state(lay, d, x["s_prefix"], x["lq"], x["lk"], x["lv"], x["alpha"],
                               x["beta"], step.lo, step.s_fork, stream=stream, rule=step.rule)
        if ev:
            ev[2].record(stream)
        step.score(x["hidden"], w_lm, stream=stream)
        if ev:
            ev[3].record(stream)
        jet.jet_decide(lay, step.mode, step.cand_score, step.q_cand, step.choice, step.value,
                       stream=stream)
        if ev:
            ev[4].record(stream)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            one_step()
    torch.cuda.synchronize(dev)
    assert jet.jet_device_status(stream) == 0, "a kernel reported an error status"
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    if clocks:
        clocks.mark(True)
    n0 = jet.jet_launch_count()
    t_start.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(args.steps):
            one_step()   # no events between the calls: each call's kernels may
                         # start while the previous call's last kernel ends
    t_end.record(stream)
    launches = jet.jet_launch_count() - n0
    torch.cuda.synchronize(dev)
    if clocks:
        clocks.mark(False)
    if world > 1:
        torch.distributed.barrier()
    total_ms = t_start.elapsed_time(t_end)
    clk = clocks.stop() if clocks else None
    # the per-call breakdown: the same steps again with events between the calls
    with torch.cuda.stream(stream):
        for i in range(args.steps):
            one_step(i)
    torch.cuda.synchronize(dev)
    call_ms = {name: statistics.mean(ev[k].elapsed_time(ev[k + 1]) for ev in call_ev)
               for k, name in enumerate(("attend", "fork", "score", "decide"))}

    if evaluate:
        # evaluation helper (after the step, outside it): gold NLL + agreement,
        # with every request's first candidate taken as the gold label
        gold = torch.zeros(step.C, dtype=torch.uint8, device=dev)
        gold[torch.as_tensor(hl.array("cand_offset")[:-1], dtype=torch.long, device=dev)] = 1
        nll = torch.empty(step.R, dtype=torch.float32, device=dev)
        correct = torch.empty(step.R, dtype=torch.int32, device=dev)
        ev_a, ev_b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        n_eval = 20
        with torch.cuda.stream(stream):
            jet.jet_evaluate(step.layout, step.cand_score, step.choice, gold, nll, correct,
                             stream=stream)
            ev_a.record(stream)
            for _ in range(n_eval):
                jet.jet_evaluate(step.layout, step.cand_score, step.choice, gold, nll, correct,
                                 stream=stream)
            ev_b.record(stream)
        torch.cuda.synchronize(dev)
        call_ms["evaluate"] = ev_a.elapsed_time(ev_b) / n_eval

    e2e_ms, h2d, d2h = None, 0, 0
    if e2e:
        # end to end: pinned host inputs, copies inside the timed region. A
        # batch as a loader leaves it: its layout words and inputs in one
        # pinned buffer (HostBatch), the results back into one pinned buffer
        # (HostResults); step i+1's input copy overlaps step i's kernels
        from paper_2609_33874_gb300.step import HostBatch, HostResults
        host = {k: x[k].cpu().pin_memory() for k in names}
        words = torch.from_numpy(hl.words).pin_memory()
        batch = HostBatch(step, host, words)
        out = HostResults(step)
        e_steps = max(3, min(args.steps, 50))
        step.run_pipelined([batch] * max(3, args.warmup), w_lm,
                           [out] * max(3, args.warmup), stream=stream)
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        if world > 1:
            torch.distributed.barrier()
        e0.record(stream)
        step.run_pipelined([batch] * e_steps, w_lm, [out] * e_steps, stream=stream)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        e2e_ms = e0.elapsed_time(e1) / e_steps
        h2d, d2h = batch.nbytes, out.buf.numel()
        del host, batch, out
    assert jet.jet_device_status(stream) == 0

    total_ms, e2e_agg, ms_per_step, value, e2e_value = aggregate(
        total_ms, e2e_ms if e2e_ms is not None else total_ms / args.steps, R, args.steps, world,
        device=dev)

    # --- roofline of the dominant kernel (the LM head) ----------------------
    N, T = problem.N, len(problem.target_ids)
    es = 2 if w.dtype == "bf16" else 4
    vtiles = (w.V + 127) // 128
    lm_bytes = w.V * w.D * es + N * w.D * es + vtiles * N * 8 + T * 4
    if low:
        # w_lm codes (+ block exponents for w4) + row scales, bf16 hidden in, its
        # codes out and back, scales
        nb = (w.D + 31) // 32
        w_bytes = {"e4m3": w.V * w.D + w.V * 4, "w4": w.V * w.D // 2 + w.V * nb + w.V * 4,
                   "mxfp8": w.V * w.D + w.V * nb}[args.lm]
        # hidden: bf16 in, its codes out and back, its scales (per token, or
        # per 32-element block for mxfp8)
        h_scales = N * nb if args.lm == "mxfp8" else N * 4
        lm_bytes = w_bytes + N * w.D * 2 + 2 * N * w.D + h_scales + vtiles * N * 8 + T * 4
    lm_flops = 2.0 * N * w.D * w.V
    score_avg_s = call_ms["score"] / 1e3
    # e4m3 tensor peak (both low-precision heads multiply e4m3 operands): the
    # measured bf16 peak x the nominal 2x of 8-bit operands
    tc_peak = peaks["bf16"] * (2 if low else 1)
    ridge = tc_peak * 1e12 / (peaks["hbm"] * 1e9)
    kernel_file = ("paper_2609_33874_gb300/csrc/lmhead_tc.cu" if w.dtype == "bf16"
                   else "paper_2609_33874_gb300/csrc/lmhead_simt.cu")
    wl_key = problem_key(args, problem)
    traffic = _traffic(kernel_file, wl_key + (":" + args.lm if low else ""))
    if w.dtype != "bf16":
        # float32 FMA: SMs x 128 lanes x 2 flop x the maximum SM clock
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        alu_peak = sms * 128 * 2 * peaks["sm_max_mhz"] * 1e6 / 1e12
        ach = lm_flops / score_avg_s / 1e12
        roof = dict(bound="alu", achieved=round(ach, 3), peak=round(alu_peak, 1), unit="TFLOP/s",
                    frac=round(ach / alu_peak, 4), traffic=traffic)
    elif lm_flops / lm_bytes < ridge:
        ach = lm_bytes / score_avg_s / 1e9
        roof = dict(bound="hbm", achieved=round(ach, 1), peak=peaks["hbm"], unit="GB/s",
                    frac=round(ach / peaks["hbm"], 4), traffic=traffic)
    else:
        ach = lm_flops / score_avg_s / 1e12
        roof = dict(bound="tensor", achieved=round(ach, 1), peak=round(tc_peak, 1), unit="TFLOP/s",
                    frac=round(ach / tc_peak, 4), traffic=traffic)
        roof["frac_of_sustained"] = round(ach / (peaks["bf16_sustained"] * (2 if low else 1)), 4)
    roof.update(kernel="jet_score_candidates" + (f"_{args.lm} (quantise hidden + {args.lm} LM head "
                                                 "+ lse merge)" if low else
                                                 " (LM head + lse merge)"),
                algorithmic_bytes=lm_bytes, algorithmic_flops=lm_flops,
                avg_launch_ms=round(score_avg_s * 1e3, 4), peak_source=peaks["source"])

    # every call of the step against its own roofline (algorithmic bytes only)
    F = N - R
    attn_bytes = (2 * problem.total_prefix * w.Hkv * w.d * es + 2 * F * w.Hkv * w.d * es
                  + 2 * N * w.Hq * w.d * es)
    calls = dict(attend=_call(call_ms["attend"], attn_bytes, peaks),
                 score=dict(ms=round(call_ms["score"], 4), bound=roof["bound"],
                            frac=roof["frac"]),
                 decide=dict(ms=round(call_ms["decide"], 4)))
    if "evaluate" in call_ms:
        calls["evaluate"] = dict(ms=round(call_ms["evaluate"], 4),
                                 note="outside the step: gold NLL over equivalent labels and "
                                      "agreement, back to back")
    if w.Hl:
        fork_bytes = (R * w.Hl * w.dk * w.dv * 4 + len(problem.cand_len) * w.Hl * w.dk * w.dv * 4
                      + F * w.Hl * (2 * w.dk + 2 * w.dv) * es + F * w.Hl * 8)
        calls["fork"] = _call(call_ms["fork"], fork_bytes, peaks)
    rec = dict(value=round(value, 2), unit=UNIT, ms_per_step=round(ms_per_step, 4),
               clocks=clk, gpu_launches=int(launches), roofline=roof, calls=calls,
               config=step_config(args, problem, world))
    if e2e:
        rec["e2e"] = dict(value=round(e2e_value, 2), unit=UNIT, h2d_bytes_per_step=h2d,
                          d2h_bytes_per_step=d2h, ms_per_step=round(e2e_agg, 4))
    del x, step
    return rec, w_lm


def problem_key(args, problem) -> str:
    """Name of a timed batch: the workload, and R where it is a smaller batch."""
    full = problem.work.R
    return args.workload if problem.R == full else f"{args.workload}:R={problem.R}"


def run_gpu(args):
    import torch
    world, rank, local = _dist()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)

    from paper_2609_33874_gb300 import build as _build
    if rank == 0:
        _build.build()
    if world > 1:
        torch.distributed.barrier()
    import jet_synth

    w = jet_synth.WORKLOADS[args.workload]
    R = args.R or w.R
    problem = jet_synth.make_problem(w, R=R)
    stream = torch.cuda.Stream(dev)
    peaks = _peaks()
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    clocks = NvmlClocks(uuid)
    if not clocks.available:
        clocks = ClockSampler(uuid)
    clocks.start()

    # --- the headline batch: device-resident steps, per-call breakdown, e2e
    from paper_2609_33874_gb300.step import ScoringStep  # noqa: F401  (loads the library)
    head, w_lm = _measure(args, problem, dev, stream, peaks, world=world, clocks=clocks,
                          e2e=not args.no_e2e, evaluate=True)
    low = args.lm != "bf16"
    result = dict(
        metric=METRIC, value=head["value"], unit=UNIT, n_gpus=world, steps=args.steps,
        warmup=args.warmup, ms_per_step=head["ms_per_step"], higher_is_better=True,
        scaling="weak", vs_baseline=None,
        dtype=(f"bf16 (LM head {args.lm})" if low else "bf16") if w.dtype == "bf16" else "f32",
        data="synthetic",
        config=head["config"],
        clocks=head["clocks"],
        e2e=head.get("e2e"),
        gpu_launches=head["gpu_launches"],
        roofline=head["roofline"],
        calls=head["calls"],
    )
    extras = world == 1 and not args.headline_only
    if rank == 0 and world == 1 and not args.no_cpu_baseline and not low:
        result["cpu_baseline"] = cpu_baseline(args.workload, R, args.cpu_sample)

    if extras and args.workload == DEFAULT_WORKLOAD and R == w.R:
        # the batch-size sweep: the first R requests of the same draw, sliced
        # from the headline batch's device inputs
        src = _device_inputs(problem, _input_names(problem), dev)
        sweep = []
        r = 1
        while r < R:
            sub = jet_synth.make_problem(w, R=r)
            rec, _ = _measure(args, sub, dev, stream, peaks, src=src, w_lm=w_lm)
            sweep.append(dict(R=r, N=sub.N, value=rec["value"], ms_per_step=rec["ms_per_step"],
                              gpu_launches=rec["gpu_launches"], roofline=_brief(rec["roofline"]),
                              calls=rec["calls"]))
            r *= 2
        sweep.append(dict(R=R, N=problem.N, value=head["value"], ms_per_step=head["ms_per_step"],
                          gpu_launches=head["gpu_launches"], roofline=_brief(head["roofline"]),
                          calls=head["calls"]))
        result["sweep"] = sweep
        del src
    del w_lm
    torch.cuda.empty_cache()

    if extras and args.workload == DEFAULT_WORKLOAD and not low:
        # the other workloads: the same step, timed the same way, each with its
        # own roofline, per-call breakdown and CPU-oracle sample
        per = {}
        saved = args.workload
        for name in EXTRA_WORKLOADS:
            args.workload = name
            wp = jet_synth.make_problem(name)
            rec, wl = _measure(args, wp, dev, stream, peaks)
            del wl
            torch.cuda.empty_cache()
            if not args.no_cpu_baseline:
                rec["cpu_baseline"] = cpu_baseline(name, wp.R, args.cpu_sample)
            rec["dtype"] = "bf16" if wp.work.dtype == "bf16" else "f32"
            per[name] = rec
            wp.drop()
        args.workload = saved
        result["per_workload"] = per
    if world > 1:
        torch.distributed.destroy_process_group()
    if rank == 0:
        print(json.dumps(result), flush=True)


def _input_names(problem):
    """The step's input names for this problem's workload."""
    names = ["q", "k_pre", "v_pre", "k_cand", "v_cand", "hidden"]
    if problem.work.Hl:
        names += ["s_prefix", "lq", "lk", "lv", "alpha", "beta"]
    return names


def _brief(roof):
    return {k: roof[k] for k in ("bound", "achieved", "peak", "unit", "frac") if k in roof}


# ---------------------------------------------------------------------------
# the prefill (a "next" row, one GPU): causal attention over the prefixes
# ---------------------------------------------------------------------------
def _time_stream(fn, stream, warmup, steps):
    """Average milliseconds of fn() over `steps` calls on `stream` (CUDA events
    on that stream, after `warmup` untimed calls) and the library's kernel
    launches inside the timed calls."""
    import torch
    from paper_2609_33874_gb300 import jet
    with torch.cuda.stream(stream):
        for _ in range(warmup):
            fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    n0 = jet.jet_launch_count()
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(steps):
            fn()
    e1.record(stream)
    launches = jet.jet_launch_count() - n0
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / steps, launches


def _roof(flops, nbytes, ms, peaks):
    """The binding roofline of a kernel with the given algorithmic work."""
    tf = flops / (ms / 1e3) / 1e12
    gbs = nbytes / (ms / 1e3) / 1e9
    ridge = peaks["bf16"] * 1e12 / (peaks["hbm"] * 1e9)
    if flops / nbytes >= ridge:
        return dict(bound="tensor", achieved=round(tf, 1), peak=peaks["bf16"], unit="TFLOP/s",
                    frac=round(tf / peaks["bf16"], 4))
    return dict(bound="hbm", achieved=round(gbs, 1), peak=peaks["hbm"], unit="GB/s",
                frac=round(gbs / peaks["hbm"], 4))


def run_prefill(args):
    """Times the prefill of the workload's prefixes (inputs resident in HBM):
    jet_prefill_attend (causal self-attention) and, for hybrid workloads,
    jet_prefill_state (the recurrent-state scan of a linear-attention layer).
    Prints one JSON line: prefix tokens per second through both, with each
    part's roofline."""
    import torch
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    from paper_2609_33874_gb300 import build as _build
    _build.build()
    import jet_synth
    from paper_2609_33874_gb300 import jet
    w = jet_synth.WORKLOADS[args.workload]
    R = args.R or w.R
    p = jet_synth.make_problem(w, R=R)
    if w.dtype != "bf16":
        print(json.dumps(dict(metric="prefix tokens prefilled/sec", unavailable="bf16 only")))
        return
    hl = jet.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    lay = hl.to_device(dev)
    stream = torch.cuda.Stream(dev)
    peaks = _peaks()
    P = p.prefix_len.astype(np.float64)
    parts = {}

    dims = jet.make_dims(jet.DTYPE_BF16, Hq=w.Hq, Hkv=w.Hkv, d=w.d, D=w.D)
    q, k, v = (jet_synth.torch_tensor(p, n, device=dev) for n in ("q_pre", "k_pre", "v_pre"))
    o = torch.empty(p.total_prefix, w.Hq, w.d, dtype=torch.bfloat16, device=dev)
    wsb = jet.jet_prefill_workspace_bytes(hl.sizes, dims)
    ws = torch.empty((wsb + 15) // 16 * 4, dtype=torch.float32, device=dev)
    ms, n_att = _time_stream(
        lambda: jet.jet_prefill_attend(lay, dims, q, k, v, o, ws, stream=stream),
        stream, args.warmup, args.steps)
    assert jet.jet_device_status(stream) == 0
    del q, k, v, o, ws
    # S = QK^T and O = PV over the causal triangle (keys 0..p of position p)
    flops = float(np.sum(4.0 * w.Hq * w.d * P * (P + 1) / 2))
    nbytes = p.total_prefix * (2 * w.Hq + 2 * w.Hkv) * w.d * 2  # Q, O, K, V once
    roof = _roof(flops, nbytes, ms, peaks)
    roof.update(kernel="jet_prefill_attend (work list + attend_prefix_tc_kernel, causal)",
                algorithmic_flops=flops, algorithmic_bytes=nbytes, traffic=None,
                peak_source=peaks["source"])
    parts["attend"] = dict(ms=round(ms, 4), roofline=roof, launches=n_att)

    if w.Hl > 0:
        ldims = jet.make_dims(jet.DTYPE_BF16, Hl=w.Hl, dk=w.dk, dv=w.dv, D=w.D)
        t = {n: jet_synth.torch_tensor(p, n, device=dev)
             for n in ("lq_pre", "lk_pre", "lv_pre", "alpha_pre", "beta_pre", "s_prefix")}
        lo = torch.empty(p.total_prefix, w.Hl, w.dv, dtype=torch.bfloat16, device=dev)
        s_out = torch.empty(R, w.Hl, w.dk, w.dv, dtype=torch.float32, device=dev)
        rule = jet.RULES[args.rule]
        ms_s, n_scan = _time_stream(
            lambda: jet.jet_prefill_state(lay, ldims, t["lq_pre"], t["lk_pre"], t["lv_pre"],
                                          t["alpha_pre"], t["beta_pre"], lo, s_out,
                                          s_init=t["s_prefix"], rule=rule, stream=stream),
            stream, args.warmup, args.steps)
        assert jet.jet_device_status(stream) == 0
        # q, k, v and the output once, the gates, and the start and final states
        sbytes = (p.total_prefix * w.Hl * ((2 * w.dk + 2 * w.dv) * 2 + 8)
                  + 2 * R * w.Hl * w.dk * w.dv * 4)
        # per token and head: u = k^T S, the rank-one update, o = S^T q
        sflops = float(p.total_prefix * w.Hl * w.dk * w.dv * (6 if args.rule == "delta" else 4))
        # the recurrence's own work against the fp32 FMA peak (152 SMs x 128
        # lanes x 2 flop per clock at the maximum SM clock), the bound of the
        # sequential form; bf16 128 x 128 states run the chunked form, which
        # moves most of that work onto the tensor cores and is bound by its
        # per-chunk chain of MMAs and barriers
        alu_peak = 152 * 128 * 2 * peaks["sm_max_mhz"] * 1e6 / 1e12
        tf_s = sflops / (ms_s / 1e3) / 1e12
        sroof = dict(bound="alu", achieved=round(tf_s, 2), peak=round(alu_peak, 1),
                     unit="TFLOP/s", frac=round(tf_s / alu_peak, 4),
                     hbm_frac=round(sbytes / (ms_s / 1e3) / 1e9 / peaks["hbm"], 4))
        chunked = w.dtype == "bf16" and w.dk == 128 and w.dv == 128
        sroof.update(kernel=(f"jet_prefill_state ({'scan_tc_kernel, chunked' if chunked else 'scan_kernel'}"
                             f", {args.rule} rule)"),
                     peak_basis="recurrence work (6 or 4 dk dv flop per token and head) against "
                                "fp32 FMA: 152 SMs x 128 lanes x 2 flop x max SM clock",
                     algorithmic_flops=sflops, algorithmic_bytes=sbytes, traffic=None,
                     peak_source=peaks["source"])
        parts["state"] = dict(ms=round(ms_s, 4), roofline=sroof, launches=n_scan)
        del t, lo, s_out
    p.drop()
    total_ms = sum(x["ms"] for x in parts.values())
    dom = max(parts.values(), key=lambda x: x["ms"])
    print(json.dumps(dict(
        metric="prefix tokens prefilled/sec", value=round(p.total_prefix / (total_ms / 1e3), 1),
        unit="tokens/s", n_gpus=1, steps=args.steps, warmup=args.warmup,
        ms_per_step=round(total_ms, 4), higher_is_better=True, dtype="bf16", data="synthetic",
        config=dict(workload=args.workload, R=R, total_prefix=p.total_prefix,
                    max_prefix=int(P.max()), Hq=w.Hq, Hkv=w.Hkv, d=w.d, Hl=w.Hl,
                    rule=args.rule if w.Hl > 0 else None),
        roofline=dom["roofline"], parts=parts,
        gpu_launches=sum(x["launches"] for x in parts.values()))), flush=True)


def run_stack(args):
    """Times a hybrid decoder stack over the workload's rows followed by the
    LM head and the decision (inputs resident in HBM) and prints one JSON
    line: candidate sets per second through the whole forward, with the
    stack's projections against their roofline."""
    import torch
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    from paper_2609_33874_gb300 import build as _build
    _build.build()
    import jet_synth
    from paper_2609_33874_gb300 import jet
    from paper_2609_33874_gb300.step import DecoderStack, ScoringStep
    w = jet_synth.WORKLOADS[args.workload]
    spec = jet_synth.STACKS[args.stack]
    R = args.R or w.R
    p = jet_synth.make_problem(w, R=R)
    hl = jet.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    dims = jet.make_dims(jet.DTYPE_BF16, Hq=w.Hq, Hkv=w.Hkv, d=w.d, D=w.D, Hl=w.Hl, dk=w.dk,
                         dv=w.dv)
    layers = []
    for l, kind in enumerate(spec.kinds):
        names = ["g1", "g2", "w_mix", "w_o", "w_gu", "w_d"] + (
            ["k_pre", "v_pre"] if kind == "full" else ["s_prefix"])
        L = {n: jet_synth.array_to_torch(jet_synth.stack_tensor(p, spec, l, n), dev)
             for n in names}
        L["kind"] = kind
        layers.append(L)
    stack = DecoderStack(hl, dims, layers, spec.Dff, rule=args.rule, device=dev)
    step = ScoringStep(hl, dims, jet.MODES[w.mode], device=dev)
    x0 = jet_synth.array_to_torch(jet_synth.stack_x0(p), dev)
    w_lm = jet_synth.torch_tensor(p, "w_lm", device=dev)
    p.drop()
    stream = torch.cuda.Stream(dev)

    def one():
        x = stack.forward(x0, stream=stream)
        step.score(x, w_lm, stream=stream)
        jet.jet_decide(step.layout, step.mode, step.cand_score, step.q_cand, step.choice,
                       step.value, stream=stream)

    ms, n_fwd = _time_stream(one, stream, args.warmup, args.steps)
    ms_stack, _ = _time_stream(lambda: stack.forward(x0, stream=stream), stream, 2, args.steps)
    assert jet.jet_device_status(stream) == 0
    N = p.N
    # the stack's projections: weight bytes once per call, 2 N K O flops each
    wts = 0
    for l, kind in enumerate(spec.kinds):
        sh = jet_synth.stack_shapes(w, spec, kind, p.total_prefix, R)
        wts += sum(int(np.prod(sh[n])) for n in ("w_mix", "w_o", "w_gu", "w_d"))
    flops = 2.0 * N * wts
    nbytes = wts * 2 + len(spec.kinds) * N * w.D * 2 * 8  # weights + the rows' passes
    peaks = _peaks()
    roof = _roof(flops, nbytes, ms_stack, peaks)
    roof.update(kernel="jet_stack_forward (proj_tc_kernel projections, rmsnorm, attention, fork)",
                algorithmic_flops=flops, algorithmic_bytes=nbytes, traffic=None,
                peak_source=peaks["source"])
    print(json.dumps(dict(
        metric="candidate sets scored/sec (decoder stack + LM head)",
        value=round(R / (ms / 1e3), 1), unit="sets/s", n_gpus=1, steps=args.steps,
        warmup=args.warmup, ms_per_step=round(ms, 4), higher_is_better=True, dtype="bf16",
        data="synthetic",
        config=dict(workload=args.workload, stack=args.stack, kinds=list(spec.kinds),
                    Dff=spec.Dff, R=R, N=N, D=w.D, rule=args.rule),
        roofline=roof, parts=dict(stack_ms=round(ms_stack, 4),
                                  score_and_decide_ms=round(ms - ms_stack, 4)),
        gpu_launches=n_fwd)), flush=True)


# ---------------------------------------------------------------------------
# reference arm: the fp64 oracle on the host cores
# ---------------------------------------------------------------------------
def run_reference(args):
    world, rank, _ = _dist()
    if rank != 0:
        return
    import jet_synth
    w = jet_synth.WORKLOADS[args.workload]
    R = args.R or w.R
    k = args.ref_sample or args.cpu_sample
    p = oracle_sample(args.workload, R, k)
    for _ in range(args.warmup):
        oracle_step(p)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_step(p)
    dt = (time.perf_counter() - t0) / args.steps
    value = p.R / dt
    desc = (f"first {p.R} of {R} requests of workload {args.workload} per step, fp64 oracle "
            f"step, BLAS threads {_CORES}")
    print(json.dumps(dict(
        impl="reference", metric=METRIC, value=round(value, 4), unit=UNIT, n_gpus=world,
        steps=args.steps, warmup=args.warmup, ms_per_step=round(dt * 1e3, 2),
        higher_is_better=True, scaling="weak", vs_baseline=None, dtype="f64", data="synthetic",
        config=step_config(args, jet_synth.make_problem(w, R=R), world),
        cpu_baseline=dict(value=round(value, 4), unit=UNIT, cores=_CORES, kind="oracle",
                          sample=desc),
        e2e=dict(value=round(value, 4), unit=UNIT, h2d_bytes_per_step=0, d2h_bytes_per_step=0),
    )), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--R", type=int, default=0, help="requests per batch (default: the workload's)")
    ap.add_argument("--cpu-sample", type=int, default=16,
                    help="requests in the CPU-oracle baseline sample")
    ap.add_argument("--ref-sample", type=int, default=0,
                    help="requests per step of the reference arm (default: --cpu-sample, so "
                         "that both CPU figures time the same sample)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true",
                    help="skip the end-to-end timing (profiling runs: device inputs only)")
    ap.add_argument("--headline-only", action="store_true",
                    help="time the headline batch only (no per-workload lines, no sweep)")
    ap.add_argument("--rule", default="delta", choices=["delta", "gla"],
                    help="recurrence of the linear-attention fork (hybrid workloads)")
    ap.add_argument("--lm", default="bf16", choices=["bf16", "e4m3", "w4", "mxfp8"],
                    help="LM head precision: bf16 (the workload's), e4m3 codes with one "
                         "scale per weight row and per token (the paper's 8-bit weights), or "
                         "w4: 4-bit weights in 32-element blocks (the paper's 4-bit weights), "
                         "or mxfp8: e4m3 weights and hidden states in 32-element blocks with "
                         "power-of-two block scales")
    ap.add_argument("--stack", default=None,
                    help="time a hybrid decoder stack (e.g. hybrid4) over the workload's rows, "
                         "then the LM head and the decision (one GPU)")
    ap.add_argument("--prefill", action="store_true",
                    help="time the prefill (causal attention over the workload's prefixes) "
                         "instead of the scoring step (one GPU)")
    ap.add_argument("--sweep", action="store_true",
                    help="one line per batch size R = 1, 2, 4, ... up to the workload's R "
                         "(one GPU; no CPU baseline)")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)  # at least three untimed warm-up steps
    if args.impl == "reference":
        run_reference(args)
    elif args.stack:
        run_stack(args)
    elif args.prefill:
        run_prefill(args)
    elif args.sweep:
        import jet_synth
        if _dist()[0] > 1:
            ap.error("--sweep runs on one GPU")
        args.no_cpu_baseline = True
        full = jet_synth.WORKLOADS[args.workload].R
        args.headline_only = True
        r = 1
        while r <= full:
            args.R = r
            run_gpu(args)
            r *= 2
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
