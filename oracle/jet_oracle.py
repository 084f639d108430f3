"""fp64 CPU oracle of the JET candidate-scoring step.

TEST INFRASTRUCTURE. Only the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg use this module; the product path never imports
it. It shares no code with the CUDA path (``paper_2609_33874_gb300``) and
imports nothing from it. Both sides only share the seeded input generator
``jet_synth``.

Everything here is written for a reader checking it against the paper, not for
speed: plain loops over requests, candidates, rows and heads; numpy's matmul
is the only library primitive used for a contraction. All arithmetic is
float64. Inputs are the exact values of the device inputs (bf16 or float32
widened to float64).

What each function computes, and where the paper defines it:

* :func:`build_layout` - teacher-forcing alignment of candidate tokens to
  query rows (Sec. 3.1, Eq. 1: the logit z_{c,t,.} is conditioned on
  (x, y_{c,<t}); Sec. 4.1: the prefix output gives every candidate's first
  token).
* :func:`cascade_attention` - candidate rows attend to the shared prefix plus
  their own earlier candidate tokens (Sec. 4.1, Fig. 1 "KV-cache text
  models"). Readings where the paper is silent: scale 1/sqrt(d), grouped-query
  head h uses key/value head floor(h / (Hq/Hkv)), no positional encoding.
* :func:`prefill_attention` - causal self-attention over each request's
  prefix, the prefill whose K/V the scoring step reuses (Sec. 4.1).
* :func:`prefill_state` - the prefix recurrent state: the prefix tokens fed
  through the recurrence in order, the state every candidate forks from.
* :func:`fork_state` - every candidate continues an unmodified copy of the
  prefix recurrent state (Sec. 4.1: for hybrid models the paper puts the prefix
  state back, unchanged, before each candidate; Sec. 5.6). The recurrence itself is not
  given by the paper; the reading used is the gated delta rule
  S <- alpha (S - beta k (k^T S)) + beta k v^T, read out as o = S^T q / sqrt(dk).
  ``rule="gla"`` selects the plain gated linear-attention variant
  S <- alpha S + beta k v^T (no erase term), a second reading of the
  unnamed recurrence.
* :func:`token_logprobs` - Eq. 1 and Eq. 2: log-softmax over the full
  vocabulary, evaluated at the target token.
* :func:`candidate_scores` - Eq. 3: s(c|x) = sum_t l_{c,t}, no length
  normalisation, no end-of-turn token.
* :func:`decide` - Eq. 4 (normalisation over candidates, max-shifted) and
  Eq. 5 with the decision rules of Sec. 3.3 (argmax with ties to the lowest
  index, binary q(true) with C = {false, true}, ordinal expected zero-based
  index).
* :func:`evaluate` - gold negative log-likelihood with the probabilities of
  labels that carry the gold answer text summed (Sec. 3.3), and agreement of
  the choice with the gold answer (Sec. 5.1).
"""
from __future__ import annotations

import math
from typing import Dict

import numpy as np

__all__ = ["build_layout", "cascade_attention", "prefill_attention", "prefill_state", "fork_state",
           "token_logprobs", "candidate_scores", "decide", "evaluate", "score_step"]

ARGMAX, BINARY, ORDINAL = 0, 1, 2


# ----------------------------------------------------------------------------
# (a1) layout: which row predicts which target, which rows see which keys
# ----------------------------------------------------------------------------
def build_layout(prefix_len, n_cand, cand_len, target_ids, V) -> Dict[str, np.ndarray]:
    """Teacher-forced row/target layout of a batch (Sec. 3.1, Eq. 1; Sec. 4.1).

    For request r with prefix x (P_r tokens) and candidates y_c = (y_{c,1} ..
    y_{c,m_c}):

    * its first row is the last prefix position; its logits condition on x
      alone, so they give p(y_{c,1} | x) for every candidate c (Sec. 4.1:
      the prefix output supplies the first-token probabilities);
    * then, candidate by candidate, one row per fed token y_{c,t} for
      t = 1 .. m_c - 1; the row fed with y_{c,t} conditions on (x, y_{c,<=t})
      and so predicts y_{c,t+1};
    * the last token y_{c,m_c} is only ever a target.

    Returns int32 arrays:
      prefix_offset[R+1]  start of request r's prefix in the packed prefix K/V
      cand_offset[R+1]    first candidate of request r
      row_offset[R+1]     first row of request r (its shared row)
      cand_row_offset[C+1] first fed row of candidate c (C+1-th entry = N)
      tgt_offset[C+1]     first target of candidate c
      tgt_row[T]          row whose logits predict target j
      target_ids[T]       the target token ids, in candidate order
      row_req[N], row_cand[N] (-1 for a shared row), row_pos[N] (t of the fed
                          token, 0 for a shared row)
      row_tgt_offset[N+1], row_tgt_index[T]  targets grouped by row, in
                          increasing target index within each row
    """
    prefix_len = [int(x) for x in prefix_len]
    n_cand = [int(x) for x in n_cand]
    cand_len = [int(x) for x in cand_len]
    target_ids = [int(x) for x in target_ids]
    R = len(prefix_len)
    C = sum(n_cand)
    if len(cand_len) != C:
        raise ValueError("cand_len must list one length per candidate")
    if any(m < 1 for m in cand_len):
        raise ValueError("every candidate needs at least one token")
    if len(target_ids) != sum(cand_len):
        raise ValueError("target_ids must list m_c ids per candidate")
    if any(not (0 <= y < V) for y in target_ids):
        raise ValueError("token id outside the vocabulary")

    prefix_offset, cand_offset, row_offset = [0], [0], []
    cand_row_offset, tgt_offset, tgt_row, tgt_ids = [], [], [], []
    row_req, row_cand, row_pos = [], [], []
    c_global = 0
    y_pos = 0
    for r in range(R):
        prefix_offset.append(prefix_offset[-1] + prefix_len[r])
        cand_offset.append(cand_offset[-1] + n_cand[r])
        shared_row = len(row_req)
        row_offset.append(shared_row)
        row_req.append(r)
        row_cand.append(-1)
        row_pos.append(0)
        for _ in range(n_cand[r]):
            c = c_global
            m = cand_len[c]
            y = target_ids[y_pos:y_pos + m]
            y_pos += m
            first_fed_row = len(row_req)
            cand_row_offset.append(first_fed_row)
            for t in range(1, m):           # rows fed with y_{c,1} .. y_{c,m-1}
                row_req.append(r)
                row_cand.append(c)
                row_pos.append(t)
            tgt_offset.append(len(tgt_row))
            for t in range(1, m + 1):       # targets y_{c,1} .. y_{c,m}
                if t == 1:
                    row = shared_row        # conditioned on x only
                else:
                    row = first_fed_row + (t - 2)  # the row fed with y_{c,t-1}
                tgt_row.append(row)
                tgt_ids.append(y[t - 1])
            c_global += 1
    N = len(row_req)
    T = len(tgt_row)
    row_offset.append(N)
    cand_row_offset.append(N)
    tgt_offset.append(T)

    by_row = [[] for _ in range(N)]
    for j, n in enumerate(tgt_row):
        by_row[n].append(j)
    row_tgt_offset, row_tgt_index = [0], []
    for n in range(N):
        row_tgt_index.extend(by_row[n])
        row_tgt_offset.append(len(row_tgt_index))

    i32 = lambda a: np.asarray(a, dtype=np.int32)  # noqa: E731
    return dict(R=R, C=C, N=N, T=T, V=int(V),
                prefix_len=i32(prefix_len), n_cand=i32(n_cand), cand_len=i32(cand_len),
                prefix_offset=i32(prefix_offset), cand_offset=i32(cand_offset),
                row_offset=i32(row_offset), cand_row_offset=i32(cand_row_offset),
                tgt_offset=i32(tgt_offset), tgt_row=i32(tgt_row), target_ids=i32(tgt_ids),
                row_req=i32(row_req), row_cand=i32(row_cand), row_pos=i32(row_pos),
                row_tgt_offset=i32(row_tgt_offset), row_tgt_index=i32(row_tgt_index))


def _fed_index(lay, n: int) -> int:
    """Index of row n's fed token in the packed candidate K/V (shared rows omitted)."""
    return n - int(lay["row_req"][n]) - 1


# ----------------------------------------------------------------------------
# (a2) shared-prefix cascade attention
# ----------------------------------------------------------------------------
def visible_keys(lay, n: int):
    """(prefix key range, list of fed-token indices) visible to row n.

    A shared row sees the whole prefix (it is the last prefix position). The
    row fed with y_{c,t} sees the prefix and candidate c's fed tokens
    y_{c,1..t}, never another candidate's (Sec. 4.1).
    """
    r = int(lay["row_req"][n])
    p0, p1 = int(lay["prefix_offset"][r]), int(lay["prefix_offset"][r + 1])
    c = int(lay["row_cand"][n])
    if c < 0:
        return (p0, p1), []
    first = int(lay["cand_row_offset"][c])
    return (p0, p1), [_fed_index(lay, m) for m in range(first, n + 1)]


def cascade_attention(lay, q, k_pre, v_pre, k_cand, v_cand, Hq: int, Hkv: int, rows=None):
    """O[n, h] = softmax_j(q[n,h] . k_j / sqrt(d)) weighted sum of v_j over row n's
    visible keys; key/value head floor(h / (Hq/Hkv)). All float64.

    ``rows`` selects the rows to compute (default: all); the result has one
    entry per selected row."""
    N, _, d = q.shape
    rows = list(range(N)) if rows is None else [int(n) for n in rows]
    g = Hq // Hkv
    out = np.zeros((len(rows), Hq, d), dtype=np.float64)
    scale = 1.0 / math.sqrt(d)
    for i, n in enumerate(rows):
        (p0, p1), fed = visible_keys(lay, n)
        qn = np.asarray(q[n], np.float64)
        for h in range(Hq):
            kh = h // g
            K = np.concatenate([np.asarray(k_pre[p0:p1, kh], np.float64),
                                np.asarray(k_cand[fed, kh], np.float64).reshape(len(fed), d)])
            Vv = np.concatenate([np.asarray(v_pre[p0:p1, kh], np.float64),
                                 np.asarray(v_cand[fed, kh], np.float64).reshape(len(fed), d)])
            scores = (K @ qn[h]) * scale
            w = np.exp(scores - scores.max())
            out[i, h] = (w / w.sum()) @ Vv
    return out


def prefill_attention(prefix_len, q, k, v, Hq: int, Hkv: int, rows=None):
    """Causal self-attention over every request's prefix, the prefill that
    produces the shared prefix (Sec. 4.1): position p of request r attends to
    the request's keys 0..p. q is [sum P, Hq, d]; k, v are [sum P, Hkv, d].
    ``rows`` selects prefix rows (default: all). All float64."""
    prefix_len = np.asarray(prefix_len, np.int64)
    offset = np.concatenate([[0], np.cumsum(prefix_len)])
    total, _, d = q.shape
    rows = list(range(total)) if rows is None else [int(n) for n in rows]
    g = Hq // Hkv
    scale = 1.0 / math.sqrt(d)
    out = np.zeros((len(rows), Hq, d), dtype=np.float64)
    for i, n in enumerate(rows):
        r = int(np.searchsorted(offset, n, side="right") - 1)
        p0 = int(offset[r])
        qn = np.asarray(q[n], np.float64)
        for h in range(Hq):
            K = np.asarray(k[p0:n + 1, h // g], np.float64)
            Vv = np.asarray(v[p0:n + 1, h // g], np.float64)
            scores = (K @ qn[h]) * scale
            w = np.exp(scores - scores.max())
            out[i, h] = (w / w.sum()) @ Vv
    return out


# ----------------------------------------------------------------------------
# (a3) recurrent-state fork
# ----------------------------------------------------------------------------
def gated_delta_step(S, q, k, v, alpha, beta):
    """One recurrence step on a (dk, dv) state; returns (new state, output)."""
    S = alpha * (S - beta * np.outer(k, k @ S)) + beta * np.outer(k, v)
    return S, (S.T @ q) / math.sqrt(S.shape[0])


def gated_linear_step(S, q, k, v, alpha, beta):
    """The plain gated linear-attention variant of the step: decay and write,
    S <- alpha S + beta k v^T, without the delta rule's erase term."""
    S = alpha * S + beta * np.outer(k, v)
    return S, (S.T @ q) / math.sqrt(S.shape[0])


RULES = {"delta": gated_delta_step, "gla": gated_linear_step}


def fork_state(lay, s_prefix, lq, lk, lv, alpha, beta, rule: str = "delta"):
    """Per candidate: restore the unchanged prefix state S_r, then feed the
    candidate's tokens y_{c,1..m_c-1} (Sec. 4.1).

    Returns (o[F, Hl, dv], s_fork[C, Hl, dk, dv]) where F = N - R fed tokens in
    row order and s_fork is each candidate's state after its last fed token
    (a copy of S_r when m_c = 1). ``rule`` names the recurrence: "delta" (the
    gated delta rule) or "gla" (plain gated linear attention).
    """
    step = RULES[rule]
    s_prefix = np.asarray(s_prefix, np.float64)
    R, Hl, dk, dv = s_prefix.shape
    C, N = lay["C"], lay["N"]
    o = np.zeros((N - R, Hl, dv), np.float64)
    s_fork = np.zeros((C, Hl, dk, dv), np.float64)
    for r in range(R):
        for c in range(int(lay["cand_offset"][r]), int(lay["cand_offset"][r + 1])):
            m = int(lay["cand_len"][c])
            first = int(lay["cand_row_offset"][c])
            for h in range(Hl):
                S = s_prefix[r, h].copy()          # restore the prefix state
                for t in range(1, m):
                    f = _fed_index(lay, first + t - 1)
                    S, o[f, h] = step(
                        S, np.asarray(lq[f, h], np.float64), np.asarray(lk[f, h], np.float64),
                        np.asarray(lv[f, h], np.float64), float(alpha[f, h]), float(beta[f, h]))
                s_fork[c, h] = S
    return o, s_fork


def prefill_state(prefix_len, s_init, lq, lk, lv, alpha, beta, rule: str = "delta"):
    """The prefix recurrent state (the prefill of a linear-attention layer):
    request r's P_r prefix tokens fed in order through the recurrence from
    s_init[r] (zeros when s_init is None). Token arrays are [sum P, Hl, .].
    Returns (o [sum P, Hl, dv], s_out [R, Hl, dk, dv]); s_out is the state
    jet_fork_state forks from (Sec. 4.1)."""
    step = RULES[rule]
    prefix_len = np.asarray(prefix_len, np.int64)
    R = len(prefix_len)
    total, Hl, dk = np.asarray(lk).shape
    dv = np.asarray(lv).shape[2]
    o = np.zeros((total, Hl, dv), np.float64)
    s_out = np.zeros((R, Hl, dk, dv), np.float64)
    p0 = 0
    for r in range(R):
        for h in range(Hl):
            S = np.zeros((dk, dv)) if s_init is None else np.asarray(s_init[r, h], np.float64).copy()
            for p in range(p0, p0 + int(prefix_len[r])):
                S, o[p, h] = step(S, np.asarray(lq[p, h], np.float64),
                                  np.asarray(lk[p, h], np.float64),
                                  np.asarray(lv[p, h], np.float64),
                                  float(alpha[p, h]), float(beta[p, h]))
            s_out[r, h] = S
        p0 += int(prefix_len[r])
    return o, s_out


# ----------------------------------------------------------------------------
# (a4) LM head, full-vocabulary log-softmax, target gather
# ----------------------------------------------------------------------------
def row_logsumexp(H, W, rows=None, vocab_chunk: int = 8192):
    """lse[n] = a_n + log sum_v exp(z_{n,v} - a_n), z_{n,v} = h_n . W_v, a_n = max_v z
    (Eq. 2), over the full vocabulary. Returns (lse, z) for the selected rows;
    z holds every logit of those rows. W may be any float array; it is widened
    to float64 one vocabulary slice at a time to bound memory."""
    H = np.asarray(H)
    rows = np.arange(H.shape[0]) if rows is None else np.asarray(rows)
    h = np.asarray(H[rows], np.float64)
    V = W.shape[0]
    z = np.empty((len(rows), V), np.float64)
    for v0 in range(0, V, vocab_chunk):
        z[:, v0:v0 + vocab_chunk] = h @ np.asarray(W[v0:v0 + vocab_chunk], np.float64).T
    a = z.max(axis=1)
    lse = a + np.log(np.exp(z - a[:, None]).sum(axis=1))
    return lse, z


def token_logprobs(lay, H, W, targets=None):
    """l_{c,t} = z_{c,t,y} - a - log sum_v exp(z_{c,t,v} - a) (Eq. 1, Eq. 2) for
    every target (or the selected target indices)."""
    targets = np.arange(lay["T"]) if targets is None else np.asarray(targets)
    rows = np.unique(lay["tgt_row"][targets])
    lse, z = row_logsumexp(H, W, rows)
    pos = {int(n): i for i, n in enumerate(rows)}
    ell = np.empty(len(targets), np.float64)
    for i, j in enumerate(targets):
        k = pos[int(lay["tgt_row"][j])]
        ell[i] = z[k, int(lay["target_ids"][j])] - lse[k]
    return ell


def candidate_scores(lay, ell):
    """s(c|x) = sum_{t=1..m_c} l_{c,t} (Eq. 3), summed in t order."""
    C = lay["C"]
    s = np.zeros(C, np.float64)
    for c in range(C):
        acc = 0.0
        for j in range(int(lay["tgt_offset"][c]), int(lay["tgt_offset"][c + 1])):
            acc += float(ell[j])
        s[c] = acc
    return s


# ----------------------------------------------------------------------------
# (a5) decision rules
# ----------------------------------------------------------------------------
def decide(lay, s, mode: int):
    """Per request: q(c) = exp(s_c - M) / sum_d exp(s_d - M), M = max_d s_d (Eq. 4);
    choice = argmax_c s_c, ties to the lowest candidate index (Eq. 5, Sec. 3.3);
    value = q(true) = q[1] for binary (C = {false, true}); sum_i i q(i) with
    zero-based i for ordinal (Sec. 3.3); value = q[choice] for argmax."""
    R = lay["R"]
    q = np.zeros(lay["C"], np.float64)
    choice = np.zeros(R, np.int32)
    value = np.zeros(R, np.float64)
    for r in range(R):
        c0, c1 = int(lay["cand_offset"][r]), int(lay["cand_offset"][r + 1])
        sr = np.asarray(s[c0:c1], np.float64)
        M = sr.max()
        e = np.exp(sr - M)
        qr = e / e.sum()
        q[c0:c1] = qr
        best = 0
        for i in range(1, c1 - c0):
            if sr[i] > sr[best]:
                best = i
        choice[r] = best
        if mode == BINARY:
            if c1 - c0 != 2:
                raise ValueError("binary decisions need exactly two candidates")
            value[r] = qr[1]
        elif mode == ORDINAL:
            value[r] = sum(i * qr[i] for i in range(c1 - c0))
        else:
            value[r] = qr[best]
    return q, choice, value


# ----------------------------------------------------------------------------
# evaluation: gold negative log-likelihood and agreement (Sec. 3.3, Sec. 5.1)
# ----------------------------------------------------------------------------
def evaluate(lay, s, choice, gold):
    """Per request, with q from Eq. 4 and gold[c] true for every candidate
    whose label carries the gold answer text: nll = -log sum_{gold c} q(c)
    (equivalent labels' probabilities are summed, Sec. 3.3; infinite when no
    candidate is gold), correct = gold[choice] (any label with the gold text
    is accepted; for binary requests the choice is the argmax of {false,
    true}, i.e. q(true) > 1/2, Sec. 5.1)."""
    def logsumexp(x):
        m = x.max()
        return m + math.log(np.exp(x - m).sum())

    R = lay["R"]
    nll = np.zeros(R, np.float64)
    correct = np.zeros(R, np.int32)
    for r in range(R):
        c0, c1 = int(lay["cand_offset"][r]), int(lay["cand_offset"][r + 1])
        sr = np.asarray(s[c0:c1], np.float64)
        g = np.asarray(gold[c0:c1], bool)
        # -log sum_{gold} q(c) with q = e^(s_c) / sum_d e^(s_d) (Eq. 4), written
        # as the difference of two log-sum-exps so that it stays exact where
        # q itself would underflow
        nll[r] = logsumexp(sr) - logsumexp(sr[g]) if g.any() else math.inf
        correct[r] = int(g[int(choice[r])])
    return nll, correct


def score_step(lay, H, W, mode: int):
    """Eq. 1 through Eq. 5 for a batch whose LM-head inputs H are given."""
    ell = token_logprobs(lay, H, W)
    s = candidate_scores(lay, ell)
    q, choice, value = decide(lay, s, mode)
    return dict(ell=ell, s=s, q=q, choice=choice, value=value)
