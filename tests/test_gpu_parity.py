"""GPU parity: the CUDA path through the C ABI against the fp64 oracle on the
same seeded inputs. Small cases compare every output; the full-size workloads
(in the launch configuration the benchmark times) compare sampled requests
and rows, plus properties that hold at any size."""
import numpy as np
import pytest

import jet_synth
import oracle as O
from gpu_common import (TOL_ATTN_BF16, TOL_ATTN_F32, build_step, check_attention, check_fork,
                        check_invariants, check_scores, oracle_layout, run_problem)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cuda(jet):
    import torch
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required for -m gpu tests")
    return jet


def _custom(base, prefix_len, n_cand, cand_len, seed=3, **over):
    import dataclasses
    w = dataclasses.replace(jet_synth.WORKLOADS[base], **over)
    rng = np.random.default_rng(seed)
    ids = rng.integers(0, w.V, size=int(np.sum(cand_len)))
    return jet_synth.custom_problem(w, prefix_len, n_cand, cand_len, ids, seed=seed)


# ---------------------------------------------------------------------------
# tiny workload (float32): every output
# ---------------------------------------------------------------------------
def test_tiny_full_step(cuda):
    p = jet_synth.make_problem("tiny")
    got, _ = run_problem(cuda, p)
    lay = oracle_layout(p)
    check_attention(lay, p, got["o"], list(range(p.N)), TOL_ATTN_F32)
    check_scores(lay, p, got, [0])
    check_invariants(lay, got)


def test_tiny_chained(cuda):
    # the attention output feeds the LM head (Hq * d == D)
    p = jet_synth.make_problem("tiny")
    got, _ = run_problem(cuda, p, chain=True)
    lay = oracle_layout(p)
    o = O.cascade_attention(lay, p.f32("q"), p.f32("k_pre"), p.f32("v_pre"), p.f32("k_cand"),
                            p.f32("v_cand"), 8, 2)
    check_scores(lay, p, got, [0], hidden=o.reshape(p.N, -1))


# ---------------------------------------------------------------------------
# attention: ragged prefixes, head dims, dtypes, edge cases
# ---------------------------------------------------------------------------
ATTN_CASES = [
    # (base, prefix_len, n_cand, cand_len, overrides)
    ("tiny", [1], [1], [1], {}),                                   # P = 1, one token
    ("tiny", [33, 95, 64], [2, 1, 3], [1, 5, 2, 3, 1, 4], {}),     # ragged tails of 32-key tiles
    ("tiny", [700], [4], [12, 1, 7, 3], dict(dtype="bf16")),
    ("tiny", [257, 31], [3, 2], [2, 2, 2, 1, 9], dict(Hq=6, Hkv=3, d=128, dtype="bf16")),
    ("tiny", [513, 129, 1000], [4, 4, 1], [1, 3, 1, 2, 5, 1, 1, 2, 1], dict(Hq=24, Hkv=4, d=256,
                                                                          dtype="bf16")),
    ("tiny", [5, 6], [1, 1], [1, 1], dict(Hq=4, Hkv=4, d=64)),     # no fed tokens at all
]


@pytest.mark.parametrize("case", range(len(ATTN_CASES)))
def test_attention_cases(cuda, case):
    base, pl, nc, cl, over = ATTN_CASES[case]
    p = _custom(base, pl, nc, cl, seed=10 + case, **over)
    got, _ = run_problem(cuda, p)
    lay = oracle_layout(p)
    tol = TOL_ATTN_BF16 if p.bf16 else TOL_ATTN_F32
    check_attention(lay, p, got["o"], list(range(p.N)), tol)


def test_attention_longest_first_list_with_splits(cuda):
    # Enough long prefixes that the planned chunk reaches 16 key tiles (1,088
    # keys here: half of one SM's share of all tiles), so the persistent kernel
    # takes its items from the longest-first work list, while every request
    # still splits into several near-equal chunks (up to 15 for the longest).
    pl = [8000] * 39 + [16000]
    p = _custom("tiny", pl, [2] * 40, [1, 2] * 40, seed=50, Hq=8, Hkv=1, d=128, dtype="bf16")
    got, _ = run_problem(cuda, p)
    lay = oracle_layout(p)
    rows = []
    for r in (0, 17, 38, 39):
        rows.extend(range(int(lay["row_offset"][r]), int(lay["row_offset"][r + 1])))
    check_attention(lay, p, got["o"], rows, TOL_ATTN_BF16)


# ---------------------------------------------------------------------------
# LM head: ragged vocabulary and rows, targets at the vocabulary edges
# ---------------------------------------------------------------------------
LM_CASES = [
    (dict(V=1000, D=72), [4, 9], [3, 2], [1, 4, 2, 6, 3]),          # V % 128 != 0, D % 32 != 0
    (dict(V=129, D=64, dtype="bf16"), [2], [5], [1, 1, 2, 1, 40]),  # 41 rows, one vocab tail
    (dict(V=20000, D=256, dtype="bf16", w_std=0.05), [3] * 7, [4] * 7, [3] * 28),
    (dict(V=8192, D=512, dtype="bf16"), [1] * 3, [1, 2, 3], [1, 12, 1, 1, 2, 3]),
    # more than 256 rows: two token tiles; hidden size not a multiple of 64
    (dict(V=5000, D=200, dtype="bf16"), [2] * 3, [10] * 3, [10] * 30),
    # three token tiles, vocabulary tail of one row
    (dict(V=1025, D=128, dtype="bf16"), [2] * 6, [10] * 6, [11] * 60),
    (dict(V=4096, D=64, dtype="bf16"), [2], [1], [1]),                  # a single row
    # an odd number of vocabulary tiles, the last one ragged
    (dict(V=1100, D=96, dtype="bf16"), [5] * 4, [6] * 4, [4] * 24),
    # exactly 256 rows: the largest single token tile (512 TMEM columns)
    (dict(V=3000, D=128, dtype="bf16"), [3] * 4, [21] * 4, [4] * 84),
]


@pytest.mark.parametrize("case", range(len(LM_CASES)))
def test_lm_head_cases(cuda, case):
    over, pl, nc, cl = LM_CASES[case]
    p = _custom("tiny", pl, nc, cl, seed=20 + case, **over)
    # targets at 0 and V - 1
    p.target_ids[0] = 0
    p.target_ids[-1] = p.work.V - 1
    got, _ = run_problem(cuda, p)
    lay = oracle_layout(p)
    check_scores(lay, p, got, list(range(p.R)))
    check_invariants(lay, got)


def test_all_vocabulary_targets_sum_to_one(cuda):
    # one request with every vocabulary entry as a single-token candidate:
    # the GPU's probabilities over V sum to one (Eq. 1)
    V = 3000
    w = dict(V=V, D=128, dtype="bf16")
    p = _custom("tiny", [7], [V], [1] * V, seed=30, **w)
    p.target_ids[:] = np.arange(V)
    got, _ = run_problem(cuda, p)
    assert abs(np.exp(got["ell"].astype(np.float64)).sum() - 1.0) < 1e-4
    check_scores(oracle_layout(p), p, got, [0])


# ---------------------------------------------------------------------------
# recurrent-state fork
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("keep", [True, False])
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_fork_small(cuda, keep, dtype):
    p = _custom("ordinal_hybrid", [3, 4, 2], [10, 3, 1], [1, 2, 3, 1, 1, 3, 2, 2, 1, 3, 4, 1, 6, 1],
                seed=40, V=4096, D=256, Hl=3, dv=64, dtype=dtype)
    got, _ = run_problem(cuda, p, keep_fork=keep)
    lay = oracle_layout(p)
    check_fork(lay, p, got, list(range(p.R)))
    check_scores(lay, p, got, list(range(p.R)))


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("rule", ["delta", "gla"])
def test_fork_long_candidates(cuda, dtype, rule):
    # candidates of up to 40 tokens: a candidate runs through several 16-token
    # windows of fed tokens (its state carried across them); both recurrences
    p = _custom("ordinal_hybrid", [5, 9], [4, 3], [20, 40, 1, 33, 7, 12, 2], seed=41, V=4096,
                D=256, Hl=2, dv=96, dtype=dtype)
    got, _ = run_problem(cuda, p, rule=rule)
    lay = oracle_layout(p)
    check_fork(lay, p, got, list(range(p.R)), rule=rule)


@pytest.mark.parametrize("rule", ["delta", "gla"])
def test_fork_window_splits(cuda, rule):
    # short candidates that straddle the 16-token windows of fed tokens at
    # several offsets, beside one-token candidates and a request with none fed
    cl = [2] + [3] * 9 + [1, 4, 2, 5, 3, 1, 6, 2] + [1, 1]
    p = _custom("ordinal_hybrid", [6, 3], [18, 2], cl, seed=42, V=4096, D=256, Hl=2, dv=64,
                dtype="bf16")
    got, _ = run_problem(cuda, p, keep_fork=True, rule=rule)
    lay = oracle_layout(p)
    check_fork(lay, p, got, list(range(p.R)), rule=rule)


def test_fork_gla_full_size(cuda):
    # the hybrid workload's shape with the gated linear-attention recurrence
    p = jet_synth.make_problem("ordinal_hybrid")
    got, _ = run_problem(cuda, p, keep_fork=True, rule="gla")
    check_fork(oracle_layout(p), p, got, [0, 17, 31], rule="gla")


# ---------------------------------------------------------------------------
# full-size workloads: sampled outputs against the oracle
# ---------------------------------------------------------------------------
FULL = {
    "dense27b_mc": dict(requests=[0, 7, 15], rows=12),
    "binary": dict(requests=[0, 31, 63], rows=12),
    "ordinal_hybrid": dict(requests=[0, 17, 31], rows=12),
    "moe_a3b_long": dict(requests=[0, 100, 255], rows=8),
}


@pytest.mark.parametrize("name", list(FULL))
def test_full_size_workload(cuda, name):
    p = jet_synth.make_problem(name)
    got, _ = run_problem(cuda, p, keep_fork=True)
    lay = oracle_layout(p)
    check_invariants(lay, got)
    req = FULL[name]["requests"]
    check_scores(lay, p, got, req)
    rng = np.random.default_rng(5)
    rows = []
    for r in req:
        n0, n1 = int(lay["row_offset"][r]), int(lay["row_offset"][r + 1])
        rows.extend(rng.choice(np.arange(n0, n1), size=min(FULL[name]["rows"] // len(req) + 1,
                                                            n1 - n0), replace=False).tolist())
    check_attention(lay, p, got["o"], sorted(set(rows)), TOL_ATTN_BF16)
    if p.work.Hl:
        check_fork(lay, p, got, req)


# ---------------------------------------------------------------------------
# failure detection: an invalid device layout is reported, never faults
# ---------------------------------------------------------------------------
def test_corrupt_device_layout_is_flagged(cuda):
    import torch
    p = jet_synth.make_problem("tiny")
    step, x, w_lm = build_step(cuda, p)
    hl = step.host_layout
    # point one row's target index past T: the LM-head kernel must skip it
    words = torch.from_numpy(hl.words.copy())
    off = (hl.struct.row_tgt_index - hl.words.ctypes.data) // 4
    words[off] = hl.sizes.T + 1000
    step.layout.words.copy_(words.to(step.layout.words.device))
    step.run(x, w_lm)
    assert cuda.jet_device_status() == 10  # JET_ERR_DEVICE
    assert cuda.jet_device_status() == 0   # cleared by the read
    step.layout.words.copy_(torch.from_numpy(hl.words).to(step.layout.words.device))
    step.run(x, w_lm)
    assert cuda.jet_device_status() == 0


def test_lm_head_sm_budget_gives_identical_results(cuda):
    # fewer persistent CTAs change which CTA computes a tile, not the tile's arithmetic
    import torch
    p = jet_synth.make_problem("binary")
    step, x, w_lm = build_step(cuda, p)
    step.run(x, w_lm)
    torch.cuda.synchronize()
    ref = step.tok_logprob.clone()
    d = step.dims
    capped = cuda.make_dims(d.dtype, Hq=d.Hq, Hkv=d.Hkv, d=d.d, D=d.D, max_sms=37)
    cuda.jet_score_candidates(step.layout, capped, x["hidden"], w_lm, step.tok_logprob,
                              step.cand_score, step.ws)
    torch.cuda.synchronize()
    assert torch.equal(step.tok_logprob, ref)
    bad = cuda.make_dims(d.dtype, Hq=d.Hq, Hkv=d.Hkv, d=d.d, D=d.D, max_sms=-1)
    with pytest.raises(cuda.JetError):
        cuda.jet_score_candidates(step.layout, bad, x["hidden"], w_lm, step.tok_logprob,
                                  step.cand_score, step.ws)


def test_end_to_end_from_host(cuda):
    import torch
    p = jet_synth.make_problem("tiny")
    step, _, w_lm = build_step(cuda, p)
    host = {k: jet_synth.torch_tensor(p, k, pin=True) for k in step.input_names()}
    words = torch.from_numpy(step.host_layout.words).pin_memory()
    out = {k: torch.empty_like(getattr(step, k), device="cpu").pin_memory()
           for k in ("tok_logprob", "cand_score", "q_cand", "choice", "value")}
    step.run_from_host(host, words, w_lm, out)
    torch.cuda.synchronize()
    got = dict(ell=out["tok_logprob"].numpy(), s=out["cand_score"].numpy(),
               q=out["q_cand"].numpy(), choice=out["choice"].numpy(), value=out["value"].numpy())
    lay = oracle_layout(p)
    check_scores(lay, p, got, [0])
    h2d, d2h = step.host_bytes(host, words)
    assert h2d > 0 and d2h > 0


@pytest.mark.parametrize("packed", [False, True])
@pytest.mark.parametrize("overlap", [True, False])
def test_end_to_end_pipelined(cuda, overlap, packed):
    """Four batches of one shape with their own hidden states and targets,
    copied in on the copy stream while the previous batch computes (or in
    order on the compute stream): each batch's results must be its own (the
    double buffers are reused from the third batch on). ``packed``: every
    batch in one pinned buffer (HostBatch), the results back into one
    (HostResults)."""
    import torch
    from paper_2609_33874_gb300.step import HostBatch, HostResults
    p0 = jet_synth.make_problem("tiny")
    rng = np.random.default_rng(7)
    probs = [jet_synth.custom_problem(p0.work, p0.prefix_len, p0.n_cand, p0.cand_len,
                                      rng.integers(0, p0.work.V, size=len(p0.target_ids)),
                                      seed=1000 + i) for i in range(4)]
    step, _, w_lm = build_step(cuda, p0)
    step.overlap_min_bytes = 0 if overlap else 1 << 40
    batches, outs = [], []
    for p in probs:
        hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, p.work.V)
        host = {k: jet_synth.torch_tensor(p, k, pin=True) for k in step.input_names()}
        words = torch.from_numpy(hl.words).pin_memory()
        if packed:
            batches.append(HostBatch(step, host, words))
            outs.append(HostResults(step))
        else:
            batches.append((host, words))
            outs.append({k: torch.empty_like(getattr(step, k), device="cpu").pin_memory()
                         for k in ("tok_logprob", "cand_score", "q_cand", "choice", "value")})
    step.run_pipelined(batches, w_lm, outs)
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == 0
    W = p0.f32("w_lm")
    for p, out in zip(probs, outs):
        got = dict(ell=out["tok_logprob"].numpy(), s=out["cand_score"].numpy(),
                   q=out["q_cand"].numpy(), choice=out["choice"].numpy(),
                   value=out["value"].numpy())
        check_scores(oracle_layout(p), p, got, range(len(p.prefix_len)), w_lm=W)


# ---------------------------------------------------------------------------
# candidate isolation on the GPU (Sec. 4.1): a candidate's log-probabilities
# do not depend on which other candidates share its batch or in what order
# ---------------------------------------------------------------------------
def _row_map(n_cand, cand_len):
    """Per request its shared row, per candidate its fed rows, per candidate
    its targets (row and target order of the teacher-forced layout)."""
    shared, fed, tgts = [], [], []
    row = tgt = c = 0
    for nc in n_cand:
        shared.append(row)
        row += 1
        for _ in range(nc):
            m = int(cand_len[c])
            fed.append(list(range(row, row + m - 1)))
            tgts.append(list(range(tgt, tgt + m)))
            row += m - 1
            tgt += m
            c += 1
    return shared, fed, tgts


def test_candidates_are_isolated(cuda):
    import torch
    n_cand, cand_len = [4, 3], [3, 1, 4, 2, 2, 5, 1]
    p = _custom("tiny", [40, 33], n_cand, cand_len, seed=51, V=3000, D=128, dtype="bf16")
    step, x, w_lm = build_step(cuda, p)
    step.run(x, w_lm)
    torch.cuda.synchronize()
    ell0, s0 = step.tok_logprob.cpu().numpy(), step.cand_score.cpu().numpy()
    o0 = step.o.float().cpu().numpy()
    # request 0's candidates reordered, request 1's second candidate removed
    keep = [3, 0, 2, 1, 4, 6]
    n_new = [4, 2]
    shared, fed, tgts = _row_map(n_cand, cand_len)
    ids = np.asarray(p.target_ids)
    q = _custom("tiny", [40, 33], n_new, [cand_len[c] for c in keep], seed=51, V=3000, D=128,
                dtype="bf16")
    q.target_ids[:] = np.concatenate([ids[tgts[c]] for c in keep])
    rows = [shared[0]] + sum((fed[c] for c in keep[:4]), []) + [shared[1]] + \
        sum((fed[c] for c in keep[4:]), [])
    R = len(n_cand)
    req_of = np.repeat(np.arange(R), [1 + sum(cand_len[c] - 1 for c in range(sum(n_cand[:r]),
                                                  sum(n_cand[:r + 1]))) for r in range(R)])
    fed_rows = [r for r in rows if r not in shared]
    fed_idx = torch.tensor([r - int(req_of[r]) - 1 for r in fed_rows], dtype=torch.long)
    step2, _, _ = build_step(cuda, q)
    sel = torch.tensor(rows, dtype=torch.long)
    x2 = dict(x)
    x2["q"] = x["q"][sel.to(x["q"].device)].contiguous()
    x2["hidden"] = x["hidden"][sel.to(x["hidden"].device)].contiguous()
    for k in ("k_cand", "v_cand"):
        x2[k] = x[k][fed_idx.to(x[k].device)].contiguous()
    step2.run(x2, w_lm)
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == 0
    ell1, s1 = step2.tok_logprob.cpu().numpy(), step2.cand_score.cpu().numpy()
    np.testing.assert_allclose(s1, s0[keep], rtol=0, atol=1e-5)
    np.testing.assert_allclose(ell1, np.concatenate([ell0[tgts[c]] for c in keep]), rtol=0,
                               atol=1e-5)
    # the attention rows too: each row sees the prefix and its own candidate only
    np.testing.assert_allclose(step2.o.float().cpu().numpy(), o0[rows], rtol=0, atol=1e-2)


# ---------------------------------------------------------------------------
# evaluation helpers: gold NLL over equivalent labels, agreement
# ---------------------------------------------------------------------------
def test_evaluate_against_oracle(cuda):
    import torch
    rng = np.random.default_rng(80)
    R = 300
    n_cand = rng.integers(1, 40, size=R)
    C = int(n_cand.sum())
    hl = cuda.jet_layout_build([4] * R, n_cand, [1] * C, rng.integers(0, 64, size=C), 64)
    lay = O.build_layout([4] * R, n_cand, [1] * C, hl.array("target_ids"), 64)
    # scores with request-wide offsets up to 1e3, repeated values (ties) and
    # requests without any gold label
    s = (rng.normal(0, 5, C) + np.repeat(rng.uniform(-1e3, 1e3, R), n_cand)).astype(np.float32)
    s[rng.random(C) < 0.1] = np.float32(7.0)
    gold = (rng.random(C) < 0.3).astype(np.uint8)
    gold[: n_cand[0]] = 0
    dl = hl.to_device("cuda")
    d_s = torch.from_numpy(s).cuda()
    q = torch.empty(C, device="cuda")
    choice = torch.empty(R, dtype=torch.int32, device="cuda")
    value = torch.empty(R, device="cuda")
    cuda.jet_decide(dl, cuda.DECIDE_ARGMAX, d_s, q, choice, value)
    nll = torch.empty(R, device="cuda")
    correct = torch.empty(R, dtype=torch.int32, device="cuda")
    cuda.jet_evaluate(dl, d_s, choice, torch.from_numpy(gold).cuda(), nll, correct)
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == 0
    _, ref_choice, _ = O.decide(lay, s.astype(np.float64), O.ARGMAX)
    np.testing.assert_array_equal(choice.cpu().numpy(), ref_choice)
    ref_nll, ref_correct = O.evaluate(lay, s.astype(np.float64), ref_choice, gold.astype(bool))
    got = nll.cpu().numpy().astype(np.float64)
    inf = np.isinf(ref_nll)
    assert inf.any() and np.array_equal(np.isinf(got), inf)
    np.testing.assert_allclose(got[~inf], ref_nll[~inf], rtol=1e-5, atol=2e-5)
    assert ref_nll[~inf].max() > 200.0   # gold probabilities below float32's range stay finite
    np.testing.assert_array_equal(correct.cpu().numpy(), ref_correct)
