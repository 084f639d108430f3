"""Failure detection without a GPU fault. Every wait between the roles of the
tensor-core kernels (attention, LM head, decoder-stack projections) is
bounded: a wait that runs past its budget makes the kernel stop issuing work,
let its copies and tensor-core operations in flight finish, free its tensor
memory and return, with JET_ERR_TIMEOUT in the device status word. A wait
that ends in time never reaches the budget check, so these tests make one
that cannot end: the test hook jet_set_test_stall has each kernel withhold its
first load (a barrier nothing will complete), with a 1 ms budget. Each call
must return and report the timeout, and the next call without the hook must
compute the right answer on the same context."""
import dataclasses

import numpy as np
import pytest

import jet_synth
from gpu_common import TOL_ATTN_BF16, build_step, check_attention, check_scores, oracle_layout

pytestmark = pytest.mark.gpu

JET_OK, JET_ERR_TIMEOUT = 0, 9
BUDGET_NS = 1_000_000  # 1 ms: the stalled wait gives up quickly


@pytest.fixture(scope="module")
def cuda(jet):
    import torch
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required for -m gpu tests")
    yield jet
    jet.jet_set_test_stall(False)
    jet.jet_set_wait_budget_ns(0)


def _problem(seed=5):
    # bf16 dense27b_mc layer shapes with a smaller vocabulary
    w = dataclasses.replace(jet_synth.WORKLOADS["dense27b_mc"], V=20000)
    rng = np.random.default_rng(seed)
    prefix = [1800, 900, 1500, 600]
    n_cand = [4, 4, 2, 3]
    cand_len = rng.integers(1, 8, size=sum(n_cand))
    ids = rng.integers(0, w.V, size=int(cand_len.sum()))
    return jet_synth.custom_problem(w, prefix, n_cand, cand_len, ids, seed=seed)


def _stalled(cuda, fn):
    """Run fn with the hook on and a short budget; return the device status."""
    old_budget = cuda.jet_set_wait_budget_ns(BUDGET_NS)
    cuda.jet_set_test_stall(True)
    try:
        fn()
        return cuda.jet_device_status()
    finally:
        cuda.jet_set_test_stall(False)
        cuda.jet_set_wait_budget_ns(old_budget)


def test_hooks_are_process_settings(cuda):
    old = cuda.jet_set_wait_budget_ns(123)
    assert cuda.jet_set_wait_budget_ns(0) == 123
    assert cuda.jet_set_wait_budget_ns(old) == 2_000_000_000  # 0 restores the default
    assert cuda.jet_set_test_stall(True) is False
    assert cuda.jet_set_test_stall(False) is True
    assert cuda.jet_device_status() == JET_OK


def test_step_wait_runs_out_then_recovers(cuda):
    # the whole step (attention, LM head, decision) with the hook: the calls
    # return and the status reads JET_ERR_TIMEOUT, twice in a row; then the
    # same step without it gives the oracle's answer on the same context
    import torch
    p = _problem()
    lay = oracle_layout(p)
    step, x, w_lm = build_step(cuda, p)
    for _ in range(2):
        assert _stalled(cuda, lambda: step.run(x, w_lm)) == JET_ERR_TIMEOUT
    assert cuda.jet_device_status() == JET_OK
    step.run(x, w_lm)
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == JET_OK
    got = dict(o=step.o.float().cpu().numpy(), ell=step.tok_logprob.cpu().numpy(),
               s=step.cand_score.cpu().numpy(), q=step.q_cand.cpu().numpy(),
               choice=step.choice.cpu().numpy(), value=step.value.cpu().numpy())
    check_attention(lay, p, got["o"], list(range(p.N)), TOL_ATTN_BF16)
    check_scores(lay, p, got, list(range(p.R)))


@pytest.mark.parametrize("call", ["attend", "score", "score_e4m3", "score_w4"])
def test_each_kernel_reports_timeout(cuda, call):
    # each tensor-core kernel on its own: the attention kernel (scheduler,
    # producer, MMA and softmax roles) and the LM head in its three formats
    # (producer, MMA, epilogue and, for 4-bit weights, converter roles); a
    # second call without the hook gives the same results as a first one
    import torch
    from paper_2609_33874_gb300.step import ScoringStep, quantize_lm_head, quantize_lm_head_w4
    p = _problem(seed=6)
    w = p.work
    lm = {"score_e4m3": "e4m3", "score_w4": "w4"}.get(call, "bf16")
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    dims = cuda.make_dims(cuda.DTYPE_BF16, Hq=w.Hq, Hkv=w.Hkv, d=w.d, D=w.D)
    step = ScoringStep(hl, dims, cuda.MODES[w.mode], device="cuda", lm=lm)
    x = {k: jet_synth.torch_tensor(p, k, device="cuda") for k in step.input_names()}
    w_lm = jet_synth.torch_tensor(p, "w_lm", device="cuda")
    if lm == "e4m3":
        w_lm = quantize_lm_head(w_lm)
    elif lm == "w4":
        w_lm = quantize_lm_head_w4(w_lm)

    def attend():
        cuda.jet_prefix_attend(step.layout, step.dims, x["q"], x["k_pre"], x["v_pre"],
                               x["k_cand"], x["v_cand"], step.o, step.ws)

    def score():
        step.score(x["hidden"], w_lm)

    fn = attend if call == "attend" else score
    out = (lambda: step.o.clone()) if call == "attend" else (lambda: step.tok_logprob.clone())
    fn()
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == JET_OK
    ref = out()
    assert _stalled(cuda, fn) == JET_ERR_TIMEOUT
    fn()
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == JET_OK
    assert torch.equal(out(), ref)


def test_stack_projection_wait_runs_out(cuda):
    # a decoder stack (tensor-core projections, attention, fork) with the hook
    # reports the timeout; without it, its rows equal a run that never saw one
    import torch
    from paper_2609_33874_gb300.step import DecoderStack
    small = dataclasses.replace(jet_synth.WORKLOADS["tiny"], dtype="bf16", D=1024, Hq=4, Hkv=2,
                                d=64, Hl=2, dk=128, dv=64, V=3000, w_std=0.05)
    spec = jet_synth.StackSpec(("linear", "full"), 2048)
    cl = [1, 3, 4, 2, 5]
    p = jet_synth.custom_problem(small, [70, 33], [3, 2], cl, np.arange(sum(cl)) * 7 % small.V,
                                 seed=44)
    w = p.work
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    dims = cuda.make_dims(cuda.DTYPE_BF16, Hq=w.Hq, Hkv=w.Hkv, d=w.d, D=w.D, Hl=w.Hl, dk=w.dk,
                          dv=w.dv)
    layers = []
    for l, kind in enumerate(spec.kinds):
        names = ["g1", "g2", "w_mix", "w_o", "w_gu", "w_d"] + (
            ["k_pre", "v_pre"] if kind == "full" else ["s_prefix"])
        L = {n: jet_synth.array_to_torch(jet_synth.stack_tensor(p, spec, l, n), "cuda")
             for n in names}
        L["kind"] = kind
        layers.append(L)
    st = DecoderStack(hl, dims, layers, spec.Dff)
    x0 = jet_synth.array_to_torch(jet_synth.stack_x0(p), "cuda")
    ref = st.forward(x0).clone()
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == JET_OK
    assert _stalled(cuda, lambda: st.forward(x0)) == JET_ERR_TIMEOUT
    got = st.forward(x0)
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == JET_OK
    assert torch.equal(got, ref)


@pytest.mark.parametrize("rule", ["delta", "gla"])
def test_prefix_scan_wait_runs_out(cuda, rule):
    # the chunked prefix-state scan on the tensor cores (bf16, 128 x 128
    # states; several chunks per request, so copies of later chunks are in
    # flight when the first wait gives up): the hooked call reports the
    # timeout, the next one equals a run that never saw one
    import torch
    w = dataclasses.replace(jet_synth.WORKLOADS["ordinal_hybrid"], Hl=2, dtype="bf16")
    pl = [200, 64, 130]
    R = len(pl)
    p = jet_synth.custom_problem(w, pl, [1] * R, [1] * R, [0] * R, seed=61)
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    dims = cuda.make_dims(cuda.DTYPE_BF16, Hl=w.Hl, dk=w.dk, dv=w.dv, D=w.D)
    t = {n: jet_synth.torch_tensor(p, n, device="cuda")
         for n in ("lq_pre", "lk_pre", "lv_pre", "alpha_pre", "beta_pre", "s_prefix")}
    o = torch.empty(p.total_prefix, w.Hl, w.dv, dtype=torch.bfloat16, device="cuda")
    s_out = torch.empty(R, w.Hl, w.dk, w.dv, dtype=torch.float32, device="cuda")
    lay = hl.to_device("cuda")

    def fn():
        cuda.jet_prefill_state(lay, dims, t["lq_pre"], t["lk_pre"], t["lv_pre"], t["alpha_pre"],
                               t["beta_pre"], o, s_out, s_init=t["s_prefix"],
                               rule=cuda.RULES[rule])

    fn()
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == JET_OK
    ref_o, ref_s = o.clone(), s_out.clone()
    assert _stalled(cuda, fn) == JET_ERR_TIMEOUT
    fn()
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == JET_OK
    assert torch.equal(o, ref_o) and torch.equal(s_out, ref_s)
