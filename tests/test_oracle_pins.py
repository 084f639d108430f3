"""Pins of the fp64 oracle against facts the paper and the mathematics fix.

Nothing here re-types the oracle's formulas: each test checks a worked example
printed in the paper, a closed form, an invariant, or an independent
formulation (full-sequence causal attention, exhaustive enumeration on a
16-token toy model).
"""
import math
import os

import numpy as np
import pytest

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    out = {}
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            key, *vals = line.split()
            if key == "visible":
                rows.append(vals)
            else:
                out[key] = [int(v) for v in vals]
    return out, rows


# ---------------------------------------------------------------------------
# Eq. 4 worked example and the decision rules (Sec. 3.2, Sec. 3.3)
# ---------------------------------------------------------------------------
def test_eq4_worked_example():
    vals = np.loadtxt(os.path.join(GOLDEN, "eq4_example.txt"))
    L, q_expected = vals[:, 0], vals[:, 1]
    lay = O.build_layout([5], [2], [1, 1], [0, 1], 4)
    q, choice, value = O.decide(lay, np.log(L), O.ARGMAX)
    np.testing.assert_allclose(q, q_expected, rtol=0, atol=1e-12)
    assert choice[0] == 0


def test_decide_shift_invariance_and_argmax_of_q():
    rng = np.random.default_rng(0)
    lay = O.build_layout([3, 4], [5, 3], [1] * 8, list(range(8)), 16)
    s = rng.normal(size=8) * 3
    q1, c1, v1 = O.decide(lay, s, O.ORDINAL)
    q2, c2, v2 = O.decide(lay, s + 1234.5, O.ORDINAL)
    np.testing.assert_allclose(q1, q2, atol=1e-12)
    np.testing.assert_array_equal(c1, c2)
    # Eq. 5: argmax q = argmax s, and q sums to one per request
    for r, (a, b) in enumerate([(0, 5), (5, 8)]):
        assert c1[r] == int(np.argmax(q1[a:b]))
        assert abs(q1[a:b].sum() - 1) < 1e-12


def test_decide_ties_lowest_index_and_binary_half():
    lay = O.build_layout([3], [4], [1] * 4, [0, 1, 2, 3], 8)
    s = np.array([-2.0, -1.0, -1.0, -3.0])
    _, choice, _ = O.decide(lay, s, O.ARGMAX)
    assert choice[0] == 1  # tie between 1 and 2 resolved to the lower index
    lay2 = O.build_layout([3], [2], [1, 1], [0, 1], 8)
    q, choice, value = O.decide(lay2, np.array([-0.7, -0.7]), O.BINARY)
    assert value[0] == 0.5 and choice[0] == 0
    with pytest.raises(ValueError):
        O.decide(lay, s, O.BINARY)


def test_decide_ordinal_one_hot_and_uniform():
    K = 10
    lay = O.build_layout([3], [K], [1] * K, list(range(K)), 16)
    for i in range(K):
        s = np.full(K, -1e4)
        s[i] = 0.0
        _, _, value = O.decide(lay, s, O.ORDINAL)
        assert abs(value[0] - i) < 1e-12
    _, _, value = O.decide(lay, np.zeros(K), O.ORDINAL)
    assert abs(value[0] - (K - 1) / 2) < 1e-12   # expectation of the uniform zero-based index


# ---------------------------------------------------------------------------
# layout (Sec. 3.1, Eq. 1; Sec. 4.1)
# ---------------------------------------------------------------------------
def test_layout_golden_small():
    g, visible = _read_golden("layout_small.txt")
    lay = O.build_layout(g["prefix_len"], g["n_cand"], g["cand_len"], g["target_ids"], g["V"][0])
    for key in ("R", "C", "N", "T"):
        assert lay[key] == g[key][0], key
    for key in ("prefix_offset", "cand_offset", "row_offset", "cand_row_offset", "tgt_offset",
                "tgt_row", "row_req", "row_cand", "row_pos", "row_tgt_offset", "row_tgt_index",
                "target_ids"):
        np.testing.assert_array_equal(lay[key], g[key], err_msg=key)
    for vals in visible:
        n, p0, p1 = int(vals[0]), int(vals[1]), int(vals[2])
        fed = [] if vals[3] == "-" else [int(v) for v in vals[3:]]
        (q0, q1), got = O.visible_keys(lay, n)
        assert (q0, q1) == (p0, p1) and got == fed, n


def test_layout_counts_random():
    rng = np.random.default_rng(1)
    for _ in range(20):
        R = int(rng.integers(1, 6))
        n_cand = rng.integers(1, 5, size=R)
        cand_len = rng.integers(1, 6, size=int(n_cand.sum()))
        ids = rng.integers(0, 50, size=int(cand_len.sum()))
        lay = O.build_layout(rng.integers(1, 9, size=R), n_cand, cand_len, ids, 50)
        assert lay["N"] == R + int((cand_len - 1).sum())
        assert lay["T"] == int(cand_len.sum())
        for c in range(lay["C"]):
            js = range(lay["tgt_offset"][c], lay["tgt_offset"][c + 1])
            rows = [int(lay["tgt_row"][j]) for j in js]
            r = int(lay["row_req"][rows[0]])
            assert rows[0] == lay["row_offset"][r]           # first token from the prefix row
            first = int(lay["cand_row_offset"][c])
            assert rows[1:] == list(range(first, first + len(rows) - 1))
        # targets grouped by row are a permutation of all targets
        assert sorted(lay["row_tgt_index"].tolist()) == list(range(lay["T"]))


def test_layout_rejects_bad_input():
    with pytest.raises(ValueError):
        O.build_layout([3], [1], [0], [], 8)          # m_c = 0
    with pytest.raises(ValueError):
        O.build_layout([3], [1], [1], [8], 8)         # id == V
    with pytest.raises(ValueError):
        O.build_layout([3], [2], [1], [1], 8)         # one length for two candidates


# ---------------------------------------------------------------------------
# Eq. 1 / Eq. 2: full-vocabulary normalisation and closed forms
# ---------------------------------------------------------------------------
def _all_tokens_layout(V):
    # one request whose V single-token candidates are every vocabulary entry:
    # the shared row then carries a target for every v in V
    return O.build_layout([4], [V], [1] * V, list(range(V)), V)


@pytest.mark.parametrize("w_scale", [0.3, 30.0])
def test_probabilities_sum_to_one_over_vocab(w_scale):
    V, D = 257, 24
    rng = np.random.default_rng(2)
    lay = _all_tokens_layout(V)
    H = rng.normal(size=(lay["N"], D))
    W = rng.normal(size=(V, D)) * w_scale
    ell = O.token_logprobs(lay, H, W)
    assert np.all(np.isfinite(ell))
    assert abs(np.exp(ell).sum() - 1.0) < 1e-12


def test_zero_weights_give_uniform_distribution():
    V, D = 8192, 16
    lay = O.build_layout([4, 2], [3, 1], [1, 2, 3, 4], [5, 0, 8191, 7, 7, 7, 1, 2, 3, 4], V)
    H = np.random.default_rng(3).normal(size=(lay["N"], D))
    res = O.score_step(lay, H, np.zeros((V, D)), O.ARGMAX)
    np.testing.assert_allclose(res["ell"], -math.log(V), rtol=0, atol=1e-12)
    np.testing.assert_allclose(res["s"], -np.array([1, 2, 3, 4]) * math.log(V), atol=1e-11)
    # q_c proportional to V^{-m_c} within request 0 (lengths 1, 2, 3)
    w = np.array([V ** -1.0, V ** -2.0, V ** -3.0])
    np.testing.assert_allclose(res["q"][:3], w / w.sum(), rtol=1e-12)
    assert res["choice"][0] == 0 and res["choice"][1] == 0


@pytest.mark.parametrize("a", [3.0, 1000.0])
def test_two_valued_logits_closed_form(a):
    # z_y = a for one token y, z_v = 0 for every other v:
    # p_y = e^a / (e^a + V - 1); computed as a - log(e^a + V - 1) stably
    V, D, y = 1000, 8, 17
    W = np.zeros((V, D))
    W[y, 0] = 1.0
    lay = O.build_layout([2], [2], [1, 1], [y, 3], V)
    H = np.zeros((lay["N"], D))
    H[:, 0] = a
    ell = O.token_logprobs(lay, H, W)
    log_den = a + math.log1p((V - 1) * math.exp(-a))
    assert abs(ell[0] - (a - log_den)) < 1e-12
    assert abs(ell[1] - (0.0 - log_den)) < 1e-12


def test_logit_shift_invariance():
    # adding the same constant to every logit of a row leaves l unchanged (Eq. 2)
    V, D = 300, 10
    rng = np.random.default_rng(4)
    lay = O.build_layout([3, 3], [2, 2], [2, 1, 3, 1], rng.integers(0, V, 7), V)
    H = rng.normal(size=(lay["N"], D))
    W = rng.normal(size=(V, D))
    base = O.token_logprobs(lay, H, W)
    H2 = np.concatenate([H, np.ones((lay["N"], 1))], axis=1)
    W2 = np.concatenate([W, np.full((V, 1), 5000.0)], axis=1)
    np.testing.assert_allclose(O.token_logprobs(lay, H2, W2), base, atol=1e-9)


# ---------------------------------------------------------------------------
# cascade attention against an independent full-sequence formulation
# ---------------------------------------------------------------------------
def _causal_attention_full(q_seq, k_seq, v_seq, Hq, Hkv):
    """Plain causal self-attention over one full token sequence."""
    L, _, d = q_seq.shape
    g = Hq // Hkv
    out = np.zeros_like(q_seq)
    for i in range(L):
        for h in range(Hq):
            s = k_seq[: i + 1, h // g] @ q_seq[i, h] / math.sqrt(d)
            p = np.exp(s - s.max())
            out[i, h] = (p / p.sum()) @ v_seq[: i + 1, h // g]
    return out


def test_cascade_equals_full_sequence_causal_attention():
    rng = np.random.default_rng(5)
    Hq, Hkv, d = 6, 2, 8
    prefix_len, n_cand = [5, 3], [3, 2]
    cand_len = [1, 3, 2, 4, 1]
    lay = O.build_layout(prefix_len, n_cand, cand_len, rng.integers(0, 9, sum(cand_len)), 9)
    N, R = lay["N"], lay["R"]
    # one query/key/value per sequence position: prefix positions and fed tokens
    k_pre = rng.normal(size=(sum(prefix_len), Hkv, d))
    v_pre = rng.normal(size=(sum(prefix_len), Hkv, d))
    k_cand = rng.normal(size=(N - R, Hkv, d))
    v_cand = rng.normal(size=(N - R, Hkv, d))
    q = rng.normal(size=(N, Hq, d))
    got = O.cascade_attention(lay, q, k_pre, v_pre, k_cand, v_cand, Hq, Hkv)
    # independent route: materialise prefix || candidate for each candidate and
    # run causal attention; the shared row is the last prefix position
    row = 0
    fed = 0
    c = 0
    for r in range(R):
        p0 = sum(prefix_len[:r])
        P = prefix_len[r]
        shared = row
        row += 1
        for _ in range(n_cand[r]):
            m = cand_len[c]
            nf = m - 1
            qs = np.concatenate([np.zeros((P - 1, Hq, d)), q[[shared]], q[row:row + nf]])
            ks = np.concatenate([k_pre[p0:p0 + P], k_cand[fed:fed + nf]])
            vs = np.concatenate([v_pre[p0:p0 + P], v_cand[fed:fed + nf]])
            ref = _causal_attention_full(qs, ks, vs, Hq, Hkv)
            np.testing.assert_allclose(got[shared], ref[P - 1], atol=1e-12)
            np.testing.assert_allclose(got[row:row + nf], ref[P:], atol=1e-12)
            row += nf
            fed += nf
            c += 1


def test_cascade_zero_query_averages_visible_values():
    # q = 0 gives equal weights: the output is the mean of exactly the visible values
    rng = np.random.default_rng(6)
    Hq, Hkv, d = 4, 4, 3
    lay = O.build_layout([4], [2], [3, 2], [1, 2, 3, 4, 5], 8)
    N = lay["N"]
    v_pre = rng.normal(size=(4, Hkv, d))
    v_cand = rng.normal(size=(N - 1, Hkv, d))
    out = O.cascade_attention(lay, np.zeros((N, Hq, d)), rng.normal(size=(4, Hkv, d)), v_pre,
                              rng.normal(size=(N - 1, Hkv, d)), v_cand, Hq, Hkv)
    np.testing.assert_allclose(out[0], v_pre.mean(0), atol=1e-12)
    np.testing.assert_allclose(out[2], np.concatenate([v_pre, v_cand[:2]]).mean(0), atol=1e-12)
    np.testing.assert_allclose(out[3], np.concatenate([v_pre, v_cand[2:3]]).mean(0), atol=1e-12)


def test_gqa_head_grouping():
    # each key/value head carries a constant value vector: query head h must
    # return the constant of key/value head floor(h / g)
    Hq, Hkv, d = 8, 2, 4
    lay = O.build_layout([3], [1], [2], [0, 1], 4)
    consts = np.array([[1.0] * d, [-2.0] * d])
    v_pre = np.broadcast_to(consts, (3, Hkv, d)).copy()
    v_cand = np.broadcast_to(consts, (1, Hkv, d)).copy()
    rng = np.random.default_rng(7)
    out = O.cascade_attention(lay, rng.normal(size=(2, Hq, d)), rng.normal(size=(3, Hkv, d)), v_pre,
                              rng.normal(size=(1, Hkv, d)), v_cand, Hq, Hkv)
    for h in range(Hq):
        np.testing.assert_allclose(out[:, h], consts[h // 4][None, :].repeat(2, 0), atol=1e-12)


# ---------------------------------------------------------------------------
# 16-token toy model: exhaustive enumeration (Eq. 1-3 and the alignment)
# ---------------------------------------------------------------------------
def _toy(seed, Vt=16, dm=6, Hq=2, Hkv=1, d=3):
    rng = np.random.default_rng(seed)
    return dict(Vt=Vt, Hq=Hq, Hkv=Hkv, d=d, E=rng.normal(size=(Vt, dm)),
                Wq=rng.normal(size=(dm, Hq * d)), Wk=rng.normal(size=(dm, Hkv * d)),
                Wv=rng.normal(size=(dm, Hkv * d)), Wlm=rng.normal(size=(Vt, Hq * d)) * 1.5)


def _toy_oracle_scores(toy, x, cands):
    """Candidate scores through the oracle's layout, cascade attention, LM head, Eq. 3."""
    Vt, Hq, Hkv, d = toy["Vt"], toy["Hq"], toy["Hkv"], toy["d"]
    lay = O.build_layout([len(x)], [len(cands)], [len(y) for y in cands],
                         [t for y in cands for t in y], Vt)
    N = lay["N"]
    emb = toy["E"]
    k_pre = (emb[x] @ toy["Wk"]).reshape(len(x), Hkv, d)
    v_pre = (emb[x] @ toy["Wv"]).reshape(len(x), Hkv, d)
    # the token at each row: the last prefix token, or the fed token y_{c,t}
    tok = []
    for n in range(N):
        c = int(lay["row_cand"][n])
        tok.append(x[-1] if c < 0 else cands[c][int(lay["row_pos"][n]) - 1])
    tok = np.asarray(tok)
    q = (emb[tok] @ toy["Wq"]).reshape(N, Hq, d)
    fed = tok[lay["row_cand"] >= 0]
    k_cand = (emb[fed] @ toy["Wk"]).reshape(-1, Hkv, d)
    v_cand = (emb[fed] @ toy["Wv"]).reshape(-1, Hkv, d)
    o = O.cascade_attention(lay, q, k_pre, v_pre, k_cand, v_cand, Hq, Hkv)
    ell = O.token_logprobs(lay, o.reshape(N, Hq * d), toy["Wlm"])
    return lay, O.candidate_scores(lay, ell)


def _toy_full_sequence_score(toy, x, y):
    """log p(y | x) by running the toy model on the whole sequence x || y."""
    Hq, Hkv, d = toy["Hq"], toy["Hkv"], toy["d"]
    seq = np.asarray(list(x) + list(y))
    L = len(seq)
    e = toy["E"][seq]
    h = _causal_attention_full((e @ toy["Wq"]).reshape(L, Hq, d), (e @ toy["Wk"]).reshape(L, Hkv, d),
                               (e @ toy["Wv"]).reshape(L, Hkv, d), Hq, Hkv).reshape(L, Hq * d)
    total = 0.0
    for t in range(len(y)):
        z = toy["Wlm"] @ h[len(x) - 1 + t]
        total += z[y[t]] - (z.max() + math.log(np.exp(z - z.max()).sum()))
    return total


@pytest.mark.parametrize("m", [1, 2, 3])
def test_toy_enumeration_sums_to_one(m):
    toy = _toy(8)
    x = [3, 14, 1, 5, 9]
    cands = [list(np.unravel_index(i, (16,) * m)) for i in range(16 ** m)]
    cands = [[int(t) for t in y] for y in cands]
    lay, s = _toy_oracle_scores(toy, x, cands)
    # sum over all length-m continuations of prod_t p(y_t | x, y_<t) = 1
    assert abs(np.exp(s).sum() - 1.0) < 1e-12
    # the argmax decision is the maximum-likelihood continuation
    _, choice, _ = O.decide(lay, s, O.ARGMAX)
    assert choice[0] == int(np.argmax(s))


def test_toy_scores_equal_independent_recomputation():
    toy = _toy(9)
    x = [7, 2, 2, 11]
    rng = np.random.default_rng(10)
    cands = [[int(t) for t in rng.integers(0, 16, size=m)] for m in (1, 2, 3, 4, 5, 3)]
    cands.append(list(cands[2]))  # a duplicate candidate (Sec. 3.3)
    lay, s = _toy_oracle_scores(toy, x, cands)
    for c, y in enumerate(cands):
        assert abs(s[c] - _toy_full_sequence_score(toy, x, y)) < 1e-12
    assert s[2] == s[len(cands) - 1]
    # duplicates tie; the fixed ordering picks the lower index
    s2 = s.copy()
    s2[:] = -50.0
    s2[2] = s2[len(cands) - 1] = s[2]
    _, choice, _ = O.decide(lay, s2, O.ARGMAX)
    assert choice[0] == 2


# ---------------------------------------------------------------------------
# recurrent-state fork (Sec. 4.1, Sec. 5.6)
# ---------------------------------------------------------------------------
def _unit(v):
    return v / np.linalg.norm(v)


def _fork_case(R_pref, n_cand, cand_len, Hl=2, dk=8, dv=6, seed=11):
    rng = np.random.default_rng(seed)
    lay = O.build_layout([3] * len(n_cand), n_cand, cand_len, [0] * sum(cand_len), 4)
    F = lay["N"] - lay["R"]
    data = dict(
        s_prefix=rng.normal(size=(lay["R"], Hl, dk, dv)) / math.sqrt(dk),
        lq=rng.normal(size=(F, Hl, dk)), lk=np.apply_along_axis(_unit, -1, rng.normal(size=(F, Hl, dk))),
        lv=rng.normal(size=(F, Hl, dv)), alpha=rng.uniform(0.9, 1.0, size=(F, Hl)),
        beta=rng.uniform(0, 1, size=(F, Hl)))
    return lay, data


def test_fork_delta_rule_write_then_read():
    # alpha = beta = 1 and a unit key: after writing (k, v) the state reads v back at k
    lay, dat = _fork_case(1, [2], [2, 2])
    dat["alpha"][:] = 1.0
    dat["beta"][:] = 1.0
    dk = dat["lk"].shape[-1]
    dat["lq"] = dat["lk"] * math.sqrt(dk)   # o = S^T q / sqrt(dk) = S^T k
    o, s_fork = O.fork_state(lay, dat["s_prefix"], dat["lq"], dat["lk"], dat["lv"], dat["alpha"], dat["beta"])
    np.testing.assert_allclose(o, dat["lv"], atol=1e-12)
    for c in range(2):
        f = c  # one fed token per candidate, in candidate order
        for h in range(2):
            np.testing.assert_allclose(s_fork[c, h].T @ dat["lk"][f, h], dat["lv"][f, h], atol=1e-12)


def test_fork_orthogonal_writes_do_not_interfere():
    lay, dat = _fork_case(1, [1], [3], dk=8)
    dat["alpha"][:] = 1.0
    dat["beta"][:] = 1.0
    basis = np.linalg.qr(np.random.default_rng(12).normal(size=(8, 8)))[0]
    for h in range(2):
        dat["lk"][0, h] = basis[:, 0]
        dat["lk"][1, h] = basis[:, 1]
    _, s_fork = O.fork_state(lay, dat["s_prefix"], dat["lq"], dat["lk"], dat["lv"], dat["alpha"], dat["beta"])
    for h in range(2):
        np.testing.assert_allclose(s_fork[0, h].T @ basis[:, 0], dat["lv"][0, h], atol=1e-12)
        np.testing.assert_allclose(s_fork[0, h].T @ basis[:, 1], dat["lv"][1, h], atol=1e-12)


def test_fork_pure_decay_and_single_token_copy():
    lay, dat = _fork_case(1, [3], [1, 2, 3])
    dat["beta"][:] = 0.0
    o, s_fork = O.fork_state(lay, dat["s_prefix"], dat["lq"], dat["lk"], dat["lv"], dat["alpha"], dat["beta"])
    S = dat["s_prefix"][0]
    np.testing.assert_array_equal(s_fork[0], S)      # m = 1: an untouched copy
    a = dat["alpha"]
    # candidate 1: one fed token (index 0); candidate 2: fed tokens 1, 2
    np.testing.assert_allclose(s_fork[1], a[0][:, None, None] * S, rtol=1e-13)
    np.testing.assert_allclose(s_fork[2], (a[1] * a[2])[:, None, None] * S, rtol=1e-13)


def test_fork_equals_fresh_recurrence_and_is_isolated():
    rng = np.random.default_rng(13)
    Hl, dk, dv, P = 2, 8, 5, 6
    lens = [3, 1, 4, 2]
    lay, dat = _fork_case(1, [len(lens)], lens, Hl, dk, dv, seed=14)
    # prefix tokens, run from a zero state, give the stored prefix state S_r
    pk = np.apply_along_axis(_unit, -1, rng.normal(size=(P, Hl, dk)))
    pv, pq = rng.normal(size=(P, Hl, dv)), rng.normal(size=(P, Hl, dk))
    pa, pb = rng.uniform(0.9, 1, size=(P, Hl)), rng.uniform(0, 1, size=(P, Hl))
    S_r = np.zeros((1, Hl, dk, dv))
    for t in range(P):
        for h in range(Hl):
            S_r[0, h], _ = O.gated_delta_step(S_r[0, h], pq[t, h], pk[t, h], pv[t, h], pa[t, h], pb[t, h])
    o, s_fork = O.fork_state(lay, S_r, dat["lq"], dat["lk"], dat["lv"], dat["alpha"], dat["beta"])
    fed = 0
    for c, m in enumerate(lens):
        for h in range(Hl):
            S = np.zeros((dk, dv))
            for t in range(P):
                S, _ = O.gated_delta_step(S, pq[t, h], pk[t, h], pv[t, h], pa[t, h], pb[t, h])
            for t in range(m - 1):
                f = fed + t
                S, o_ref = O.gated_delta_step(S, dat["lq"][f, h], dat["lk"][f, h], dat["lv"][f, h],
                                              dat["alpha"][f, h], dat["beta"][f, h])
                assert np.max(np.abs(o[f, h] - o_ref)) < 1e-10
            assert np.max(np.abs(s_fork[c, h] - S)) < 1e-10
        fed += m - 1
    # isolation: reversing the candidate order leaves every candidate's result
    # bit-identical (no state leaks from one candidate into the next)
    order = list(reversed(range(len(lens))))
    lens_r = [lens[c] for c in order]
    lay_r = O.build_layout([3], [len(lens)], lens_r, [0] * sum(lens), 4)
    starts = np.concatenate([[0], np.cumsum(np.asarray(lens) - 1)])
    perm = np.concatenate([np.arange(starts[c], starts[c] + lens[c] - 1) for c in order]).astype(int)
    o_r, s_r = O.fork_state(lay_r, S_r, dat["lq"][perm], dat["lk"][perm], dat["lv"][perm],
                            dat["alpha"][perm], dat["beta"][perm])
    for i, c in enumerate(order):
        assert np.array_equal(s_r[i], s_fork[c])
    np.testing.assert_array_equal(o_r, o[perm])


# ---------------------------------------------------------------------------
# evaluation helpers: gold NLL over equivalent labels, agreement
# ---------------------------------------------------------------------------
def _eval_layout(n_cand):
    cand_len = [1] * int(sum(n_cand))
    return O.build_layout([4] * len(n_cand), n_cand, cand_len, list(range(len(cand_len))), 64)


def test_evaluate_closed_forms():
    lay = _eval_layout([2, 2, 3, 2, 4])
    s = np.array([0.0, 0.0,            # equal scores, one gold: nll = log 2
                  -1.0, -3.0,          # both gold: nll = 0
                  1.0, 2.0, 3.0,       # gold = the two lowest: -log((e+e^2)/(e+e^2+e^3))
                  5.0, 5.0,            # no gold: infinite
                  -2.0, 0.5, 0.5, -9.0])  # gold = two tied maxima, choice = first of them
    gold = np.array([0, 1, 1, 1, 1, 1, 0, 0, 0, 0, 1, 1, 0], bool)
    q, choice, _ = O.decide(lay, s, O.ARGMAX)
    nll, correct = O.evaluate(lay, s, choice, gold)
    assert abs(nll[0] - math.log(2)) < 1e-15 and abs(nll[1]) < 1e-15
    e = np.exp([1.0, 2.0, 3.0])
    assert abs(nll[2] + math.log((e[0] + e[1]) / e.sum())) < 1e-14
    assert nll[3] == math.inf
    assert abs(nll[4] + math.log(q[10] + q[11])) < 1e-14
    # choice: ties to the lowest index; accepted when that label is gold
    np.testing.assert_array_equal(choice, [0, 0, 2, 0, 1])
    np.testing.assert_array_equal(correct, [0, 1, 0, 0, 1])


def test_evaluate_singleton_gold_is_minus_log_q_and_shift_invariant():
    rng = np.random.default_rng(9)
    lay = _eval_layout([5, 3, 7])
    s = rng.normal(0, 4, lay["C"])
    gold = np.zeros(lay["C"], bool)
    gold[[2, 6, 12]] = True
    q, choice, _ = O.decide(lay, s, O.ARGMAX)
    nll, _ = O.evaluate(lay, s, choice, gold)
    np.testing.assert_allclose(nll, -np.log(q[[2, 6, 12]]), rtol=1e-13)
    nll2, _ = O.evaluate(lay, s + 123.0, choice, gold)
    np.testing.assert_allclose(nll2, nll, rtol=1e-12)
    # gold = every candidate: probability one
    nll3, correct3 = O.evaluate(lay, s, choice, np.ones(lay["C"], bool))
    np.testing.assert_allclose(nll3, 0.0, atol=1e-14)
    assert correct3.all()


# ---------------------------------------------------------------------------
# recurrence variant: plain gated linear attention
# ---------------------------------------------------------------------------
def test_gla_closed_form_from_zero_state():
    # S_T = sum_t (prod_{s>t} alpha_s) beta_t k_t v_t^T from S_0 = 0
    rng = np.random.default_rng(31)
    dk, dv, Tn = 8, 5, 6
    k = rng.normal(size=(Tn, dk)); v = rng.normal(size=(Tn, dv)); q = rng.normal(size=(Tn, dk))
    a = rng.uniform(0.9, 1.0, Tn); b = rng.uniform(0, 1, Tn)
    S = np.zeros((dk, dv))
    for t in range(Tn):
        S, o = O.gated_linear_step(S, q[t], k[t], v[t], a[t], b[t])
    ref = sum(np.prod(a[t + 1:]) * b[t] * np.outer(k[t], v[t]) for t in range(Tn))
    np.testing.assert_allclose(S, ref, rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(o, ref.T @ q[-1] / math.sqrt(dk), rtol=1e-12)


def test_gla_and_delta_agree_only_without_overlap():
    # the two rules coincide when the key is orthogonal to what the state holds
    dk, dv = 6, 3
    S0 = np.zeros((dk, dv)); S0[:3] = np.arange(9.0).reshape(3, 3)
    k = np.zeros(dk); k[4] = 1.0
    v = np.array([1.0, -2.0, 0.5]); q = np.ones(dk)
    d1, _ = O.gated_delta_step(S0, q, k, v, 0.95, 0.7)
    g1, _ = O.gated_linear_step(S0, q, k, v, 0.95, 0.7)
    np.testing.assert_allclose(d1, g1, rtol=0, atol=1e-15)
    k2 = np.zeros(dk); k2[1] = 1.0            # overlaps row 1 of the state
    d2, _ = O.gated_delta_step(S0, q, k2, v, 0.95, 0.7)
    g2, _ = O.gated_linear_step(S0, q, k2, v, 0.95, 0.7)
    # delta erases beta of the old row before writing; gla only adds
    np.testing.assert_allclose(g2[1] - d2[1], 0.95 * 0.7 * S0[1], rtol=1e-14)


def test_fork_rule_selects_the_recurrence():
    lay = O.build_layout([3, 2], [2, 1], [3, 1, 2], [1, 2, 3, 4, 5, 6], 8)
    rng = np.random.default_rng(33)
    R, F, Hl, dk, dv = 2, lay["N"] - 2, 2, 4, 3
    sp = rng.normal(size=(R, Hl, dk, dv))
    lq, lk, lv = (rng.normal(size=(F, Hl, n)) for n in (dk, dk, dv))
    al, be = rng.uniform(0.9, 1, (F, Hl)), rng.uniform(0, 1, (F, Hl))
    od, sd = O.fork_state(lay, sp, lq, lk, lv, al, be)
    og, sg = O.fork_state(lay, sp, lq, lk, lv, al, be, rule="gla")
    assert not np.allclose(sd, sg)
    # candidate 0 of request 0 feeds fed tokens 0, 1 (m = 3): replay it by hand
    S = sp[0, 1].copy()
    for f in (0, 1):
        S = al[f, 1] * S + be[f, 1] * np.outer(lk[f, 1], lv[f, 1])
    np.testing.assert_allclose(sg[0, 1], S, rtol=1e-13)


# ---------------------------------------------------------------------------
# prefill: causal attention over each request's prefix
# ---------------------------------------------------------------------------
def test_prefill_first_position_and_zero_query():
    rng = np.random.default_rng(41)
    P = [5, 3]
    q = rng.normal(size=(8, 4, 6)); k = rng.normal(size=(8, 2, 6)); v = rng.normal(size=(8, 2, 6))
    q[6] = 0.0
    out = O.prefill_attention(P, q, k, v, 4, 2)
    # position 0 of each request sees only its own key: the output is its value
    np.testing.assert_allclose(out[0], v[0][[0, 0, 1, 1]], rtol=1e-14)
    np.testing.assert_allclose(out[5], v[5][[0, 0, 1, 1]], rtol=1e-14)
    # a zero query averages exactly the visible values (request 1, position 1 = row 6)
    np.testing.assert_allclose(out[6, 2], v[5:7, 1].mean(axis=0), rtol=1e-14)


def test_prefill_last_position_equals_the_shared_row():
    # the shared row of the scoring step is the last prefix position: the
    # prefill's output there equals cascade attention of that row
    rng = np.random.default_rng(42)
    P = [6, 4]
    lay = O.build_layout(P, [1, 1], [1, 1], [3, 5], 8)
    d, Hq, Hkv = 8, 6, 3
    qp = rng.normal(size=(10, Hq, d)); kp = rng.normal(size=(10, Hkv, d))
    vp = rng.normal(size=(10, Hkv, d))
    q_rows = qp[[5, 9]]                      # the shared rows' queries
    casc = O.cascade_attention(lay, q_rows, kp, vp, np.zeros((0, Hkv, d)), np.zeros((0, Hkv, d)),
                               Hq, Hkv)
    pre = O.prefill_attention(P, qp, kp, vp, Hq, Hkv, rows=[5, 9])
    np.testing.assert_allclose(pre, casc, rtol=1e-13)


def test_prefill_is_causal():
    # changing a later key or value never changes an earlier position
    rng = np.random.default_rng(43)
    P = [7]
    q = rng.normal(size=(7, 2, 4)); k = rng.normal(size=(7, 1, 4)); v = rng.normal(size=(7, 1, 4))
    a = O.prefill_attention(P, q, k, v, 2, 1)
    k2, v2 = k.copy(), v.copy()
    k2[4:] += 3.0
    v2[4:] -= 1.0
    b = O.prefill_attention(P, q, k2, v2, 2, 1)
    np.testing.assert_array_equal(a[:4], b[:4])
    assert not np.allclose(a[4:], b[4:])


# ---------------------------------------------------------------------------
# prefill of the recurrent state
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("rule", ["delta", "gla"])
def test_prefill_state_then_fork_equals_one_scan(rule):
    # scanning prefix ++ candidate tokens in one pass equals forking the
    # candidate from the scanned prefix state (the state the fork reuses)
    rng = np.random.default_rng(51)
    Hl, dk, dv = 2, 4, 3
    P = [4, 3]
    cand = [[2, 3], [1]]                          # candidate lengths m_c
    lay = O.build_layout(P, [2, 1], [2, 3, 1], list(range(6)), 8)
    F = lay["N"] - lay["R"]
    pk = rng.normal(size=(7, Hl, dk)); pq = rng.normal(size=(7, Hl, dk)); pv = rng.normal(size=(7, Hl, dv))
    pa, pb = rng.uniform(0.9, 1, (7, Hl)), rng.uniform(0, 1, (7, Hl))
    fk = rng.normal(size=(F, Hl, dk)); fq = rng.normal(size=(F, Hl, dk)); fv = rng.normal(size=(F, Hl, dv))
    fa, fb = rng.uniform(0.9, 1, (F, Hl)), rng.uniform(0, 1, (F, Hl))
    s0 = rng.normal(size=(2, Hl, dk, dv))
    o_pre, s_pre = O.prefill_state(P, s0, pq, pk, pv, pa, pb, rule)
    _, s_fork = O.fork_state(lay, s_pre, fq, fk, fv, fa, fb, rule=rule)
    # candidate 1 of request 0 (m = 3) feeds fed tokens 1, 2: scan prefix 0 + those
    cat = lambda x, y: np.concatenate([x[0:4], y[1:3]])  # noqa: E731
    _, s_one = O.prefill_state([6], s0[:1], cat(pq, fq), cat(pk, fk), cat(pv, fv),
                               cat(pa, fa), cat(pb, fb), rule)
    np.testing.assert_allclose(s_fork[1], s_one[0], rtol=1e-12, atol=1e-13)
    # the outputs of the prefix positions are the one-pass scan's first outputs
    o_one, _ = O.prefill_state([4], s0[:1], pq[:4], pk[:4], pv[:4], pa[:4], pb[:4], rule)
    np.testing.assert_allclose(o_pre[:4], o_one, rtol=1e-13)


def test_prefill_state_zero_init_and_empty_writes():
    rng = np.random.default_rng(52)
    Hl, dk, dv = 1, 3, 2
    k = rng.normal(size=(2, Hl, dk)); q = rng.normal(size=(2, Hl, dk)); v = rng.normal(size=(2, Hl, dv))
    a = np.full((2, Hl), 0.5); b = np.zeros((2, Hl))       # beta = 0: nothing is written
    s0 = rng.normal(size=(1, Hl, dk, dv))
    _, s = O.prefill_state([2], s0, q, k, v, a, b)
    np.testing.assert_allclose(s, 0.25 * s0, rtol=1e-15)      # two decays of 1/2
    _, z = O.prefill_state([2], None, q, k, v, a, b)
    assert np.all(z == 0)
