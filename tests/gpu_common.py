"""Shared helpers of the GPU parity tests: run a problem through the C ABI and
compute the oracle's answer for the same seeded inputs."""
import numpy as np

import jet_synth
import oracle as O

# acceptance bars (per-candidate / per-token |delta log-prob| 2e-3; argmax
# identical above a 1e-2 top-two gap; derived bars for q(true) and the
# ordinal expectation; bf16 attention output 1e-2 absolute)
TOL_LOGPROB = 2e-3
ARGMAX_GAP = 1e-2
TOL_BINARY = 1e-3
TOL_ORDINAL = 9e-3
TOL_ATTN_BF16 = 1e-2
TOL_ATTN_F32 = 1e-4
TOL_FORK_REL = 1e-4


def dims_for(jet, w):
    dtype = jet.DTYPE_BF16 if w.dtype == "bf16" else jet.DTYPE_F32
    return jet.make_dims(dtype, Hq=w.Hq, Hkv=w.Hkv, d=w.d, D=w.D, Hl=w.Hl, dk=w.dk, dv=w.dv)


def build_step(jet, problem, device="cuda", chain=False, keep_fork=True, rule="delta"):
    from paper_2609_33874_gb300.step import ScoringStep
    w = problem.work
    hl = jet.jet_layout_build(problem.prefix_len, problem.n_cand, problem.cand_len,
                              problem.target_ids, w.V)
    step = ScoringStep(hl, dims_for(jet, w), jet.MODES[w.mode], device=device,
                       hybrid=w.Hl > 0, keep_fork_state=keep_fork, chain=chain, rule=rule)
    names = step.input_names()
    x = {k: jet_synth.torch_tensor(problem, k, device=device) for k in names}
    w_lm = jet_synth.torch_tensor(problem, "w_lm", device=device)
    return step, x, w_lm


def run_problem(jet, problem, device="cuda", chain=False, keep_fork=True, rule="delta"):
    import torch
    step, x, w_lm = build_step(jet, problem, device, chain, keep_fork, rule)
    step.run(x, w_lm)
    torch.cuda.synchronize()
    assert jet.jet_device_status() == 0
    out = dict(o=step.o.float().cpu().numpy(), ell=step.tok_logprob.cpu().numpy(),
               s=step.cand_score.cpu().numpy(), q=step.q_cand.cpu().numpy(),
               choice=step.choice.cpu().numpy(), value=step.value.cpu().numpy())
    if step.hybrid:
        out["lo"] = step.lo.float().cpu().numpy()
        out["s_fork"] = None if step.s_fork is None else step.s_fork.cpu().numpy()
    return out, step


def oracle_layout(problem):
    return O.build_layout(problem.prefix_len, problem.n_cand, problem.cand_len,
                          problem.target_ids, problem.work.V)


def check_scores(lay, problem, got, requests, hidden=None, w_lm=None):
    """Oracle l, s and decisions for the given requests; compare with `got`."""
    w = problem.work
    H = problem.f32("hidden") if hidden is None else hidden
    W = problem.f32("w_lm") if w_lm is None else w_lm
    tg = []
    cands = []
    for r in requests:
        for c in range(int(lay["cand_offset"][r]), int(lay["cand_offset"][r + 1])):
            cands.append(c)
            tg.extend(range(int(lay["tgt_offset"][c]), int(lay["tgt_offset"][c + 1])))
    tg = np.asarray(tg)
    ell = O.token_logprobs(lay, H, W, tg)
    err = np.abs(got["ell"][tg] - ell)
    assert err.max() <= TOL_LOGPROB, f"token log-prob error {err.max()}"
    full = np.zeros(lay["T"])
    full[tg] = ell
    s = O.candidate_scores(lay, full)
    cands = np.asarray(cands)
    serr = np.abs(got["s"][cands] - s[cands])
    assert serr.max() <= TOL_LOGPROB, f"candidate score error {serr.max()}"
    mode = {"argmax": O.ARGMAX, "binary": O.BINARY, "ordinal": O.ORDINAL}[w.mode]
    q, choice, value = O.decide(lay, s, mode)
    for r in requests:
        c0, c1 = int(lay["cand_offset"][r]), int(lay["cand_offset"][r + 1])
        sr = np.sort(s[c0:c1])[::-1]
        if len(sr) == 1 or sr[0] - sr[1] > ARGMAX_GAP:
            assert got["choice"][r] == choice[r], f"request {r}"
        if w.mode == "binary":
            assert abs(got["value"][r] - value[r]) <= TOL_BINARY
        if w.mode == "ordinal":
            assert abs(got["value"][r] - value[r]) <= TOL_ORDINAL
        np.testing.assert_allclose(got["q"][c0:c1], q[c0:c1], atol=2 * TOL_LOGPROB)
    return ell, s


def check_invariants(lay, got):
    """Properties that hold at any size: l <= 0, q sums to one, the choice is
    the (first) maximiser of s."""
    assert np.all(np.isfinite(got["ell"])) and np.all(got["ell"] <= 1e-6)
    for r in range(lay["R"]):
        c0, c1 = int(lay["cand_offset"][r]), int(lay["cand_offset"][r + 1])
        assert abs(got["q"][c0:c1].sum() - 1) < 1e-5
        assert got["choice"][r] == int(np.argmax(got["s"][c0:c1]))


def check_attention(lay, problem, got_o, rows, tol):
    w = problem.work
    ref = O.cascade_attention(lay, problem.f32("q"), problem.f32("k_pre"), problem.f32("v_pre"),
                              problem.f32("k_cand"), problem.f32("v_cand"), w.Hq, w.Hkv, rows=rows)
    err = np.abs(got_o[rows] - ref)
    assert err.max() <= tol, f"attention error {err.max()} (tol {tol})"
    return ref


def check_fork(lay, problem, got, requests, rule="delta"):
    sub = [r for r in requests]
    s_prefix = problem.f32("s_prefix")
    ref_o, ref_s = O.fork_state(lay, s_prefix, problem.f32("lq"), problem.f32("lk"),
                                problem.f32("lv"), problem.f32("alpha"), problem.f32("beta"),
                                rule=rule)
    for r in sub:
        c0, c1 = int(lay["cand_offset"][r]), int(lay["cand_offset"][r + 1])
        if got.get("s_fork") is not None:
            ref = ref_s[c0:c1]
            err = np.abs(got["s_fork"][c0:c1] - ref) / (np.abs(ref).max() + 1e-30)
            assert err.max() <= TOL_FORK_REL, f"fork state error {err.max()}"
        f0 = int(lay["row_offset"][r]) - r
        f1 = int(lay["row_offset"][r + 1]) - r - 1
        if f1 > f0:
            err = np.abs(got["lo"][f0:f1] - ref_o[f0:f1])
            tol = TOL_ATTN_BF16 if problem.bf16 else TOL_ATTN_F32
            assert err.max() <= tol, f"fork output error {err.max()}"
