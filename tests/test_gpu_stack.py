"""GPU parity of the hybrid decoder stack (jet_stack_forward) through the C ABI
against the oracle's stack with the same storage points, on the same seeded
inputs: a small ragged batch with both layer kinds and both recurrence rules,
the stack's rows fed through the LM head (token log-probabilities and
candidate scores against the oracle's, split into the LM head's own error and
the stack's rounding carried through it), and the full-size four-layer hybrid
stack on the ordinal_hybrid batch with the full-vocabulary LM head after it."""
import dataclasses

import numpy as np
import pytest

import jet_synth
import oracle as O
from oracle import stack as S
from gpu_common import TOL_LOGPROB, oracle_layout

pytestmark = pytest.mark.gpu

# The device and the oracle round to bf16 at the same points. Between them,
# the device accumulates in float32 and its attention multiplies bf16-rounded
# probabilities (P in bf16 for the PV product), which moves an attention
# output by up to ~2^-9 of its size before the output's own rounding. Through
# W_o that shift reaches every element of x, so about half of the stored
# elements land one bf16 ulp (2^-8 relative) away from the oracle's, and a
# shifted value feeds the next layer scaled by weights of size 1/sqrt(fan_in)
# and averaged with the rest. Each layer adds such a perturbation of its own,
# so the bars grow with the depth L: each element within 8 ulps of its row's
# rms per layer (L 2^-5), the mean within half an ulp per layer (L 2^-9).
TOL_STACK_ROW_PER_LAYER = 2.0 ** -5
TOL_STACK_MEAN_PER_LAYER = 2.0 ** -9


@pytest.fixture(scope="module")
def cuda(jet):
    import torch
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required for -m gpu tests")
    return jet


def _layers(p, spec, device="cuda"):
    out = []
    for l, kind in enumerate(spec.kinds):
        names = ["g1", "g2", "w_mix", "w_o", "w_gu", "w_d"] + (
            ["k_pre", "v_pre"] if kind == "full" else ["s_prefix"])
        L = {n: jet_synth.array_to_torch(jet_synth.stack_tensor(p, spec, l, n), device)
             for n in names}
        L["kind"] = kind
        out.append(L)
    return out


def _oracle_params(p, spec, l):
    kind = spec.kinds[l]
    names = ["g1", "g2", "w_mix", "w_o", "w_gu", "w_d"] + (
        ["k_pre", "v_pre"] if kind == "full" else ["s_prefix"])
    P = {}
    for n in names:
        a = jet_synth.stack_tensor(p, spec, l, n)
        P[n] = (jet_synth.bf16_to_f32(a) if a.dtype == np.uint16 else a).astype(np.float64)
    return P


def _oracle_stack(p, spec, rule):
    w = p.work
    lay = oracle_layout(p)
    dims = dict(Hq=w.Hq, Hkv=w.Hkv, d=w.d, Hl=w.Hl, dk=w.dk, dv=w.dv, Dff=spec.Dff)
    x = jet_synth.bf16_to_f32(jet_synth.stack_x0(p)).astype(np.float64)
    for l, kind in enumerate(spec.kinds):
        x = S.layer_forward(lay, x, kind, _oracle_params(p, spec, l), dims, rule)
    return x


def _gpu_stack(cuda, p, spec, rule):
    import torch
    from paper_2609_33874_gb300.step import DecoderStack
    w = p.work
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    dims = cuda.make_dims(cuda.DTYPE_BF16, Hq=w.Hq, Hkv=w.Hkv, d=w.d, D=w.D, Hl=w.Hl, dk=w.dk,
                          dv=w.dv)
    st = DecoderStack(hl, dims, _layers(p, spec), spec.Dff, rule=rule)
    x0 = jet_synth.array_to_torch(jet_synth.stack_x0(p), "cuda")
    outs = []
    for _ in range(2):  # a second call on the same buffers gives the same rows
        x = st.forward(x0)
        torch.cuda.synchronize()
        assert cuda.jet_device_status() == 0
        outs.append(x.float().cpu().numpy())
    np.testing.assert_array_equal(outs[0], outs[1])
    return outs[1], st


def _check_rows(got, ref, L):
    rms = np.sqrt(np.mean(ref * ref, axis=1, keepdims=True))
    rel = np.abs(got - ref) / rms
    print(f"stack rows ({L} layers): max {rel.max():.3e} mean {rel.mean():.3e} "
          f"share exact {np.mean(got == ref):.4f}")
    assert rel.max() <= L * TOL_STACK_ROW_PER_LAYER, f"stack row error {rel.max()}"
    assert rel.mean() <= L * TOL_STACK_MEAN_PER_LAYER, f"stack mean error {rel.mean()}"


SMALL = dataclasses.replace(jet_synth.WORKLOADS["tiny"], dtype="bf16", D=256, Hq=4, Hkv=2, d=64,
                            Hl=2, dk=128, dv=64, V=3000, w_std=0.05)


@pytest.mark.parametrize("rule", ["delta", "gla"])
def test_stack_small(cuda, rule):
    spec = jet_synth.StackSpec(("linear", "full", "linear"), 256)
    cl = [1, 3, 4, 2, 5]
    p = jet_synth.custom_problem(SMALL, [70, 33], [3, 2], cl,
                                 np.arange(sum(cl)) * 7 % SMALL.V, seed=41)
    got, _ = _gpu_stack(cuda, p, spec, rule)
    _check_rows(got, _oracle_stack(p, spec, rule), len(spec.kinds))


def _score_gpu(cuda, p, x):
    """The device LM head (jet_score_candidates) on the hidden states x."""
    import torch
    w = p.work
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    dims = cuda.make_dims(cuda.DTYPE_BF16, D=w.D)
    w_lm = jet_synth.torch_tensor(p, "w_lm", device="cuda")
    ell = torch.empty(hl.sizes.T, dtype=torch.float32, device="cuda")
    s = torch.empty(hl.sizes.C, dtype=torch.float32, device="cuda")
    wsb = cuda.jet_workspace_bytes(hl.sizes, dims)
    ws = torch.empty((wsb + 15) // 16 * 4, dtype=torch.float32, device="cuda")
    cuda.jet_score_candidates(hl.to_device("cuda"), dims, x, w_lm, ell, s, ws)
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == 0
    return ell.cpu().numpy(), s.cpu().numpy()


# Scores chained after the stack. The stack's rows differ from the oracle's by
# bf16 rounding (the row bars above); a log-probability l = z_y - lse(z) moves
# with its row's hidden state h as dl = g . dh + O(|dh|^2), with the gradient
# g = W_y - sum_v p_v W_v (p the row's softmax). Three checks follow:
#  1. the device LM head on the device's own stack rows against the oracle's
#     LM head on those same rows: the scoring bar TOL_LOGPROB, token by token
#     and per candidate;
#  2. the whole chained difference (device stack + head against oracle stack +
#     head) minus the part the row difference explains, g . dh: TOL_LOGPROB,
#     i.e. the chain adds nothing to the stack's rounding beyond the scoring bar;
#  3. the whole chained difference against a bar fixed by oracle quantities
#     alone: the row bar allows a mean relative element error of L 2^-9 of the
#     row's rms, so an rms error of at most 1.5 L 2^-9 rms(h) (heavier tails
#     than a Gaussian's 1.25); with element errors of unrelated signs g . dh has
#     a standard deviation of |g| rms(dh), held here to five of them.
CHAIN_SIGMAS = 5.0
CHAIN_RMS_PER_MEAN = 1.5


def _chained_checks(lay, got, ref, W, ell_gpu, s_gpu, L, targets=None, cands=None):
    T, C = int(lay["T"]), int(lay["C"])
    targets = np.arange(T) if targets is None else np.asarray(targets)
    cands = np.arange(C) if cands is None else np.asarray(cands)
    # 1. the LM head on the device's rows
    head = O.token_logprobs(lay, got, W, targets)
    err_head = np.abs(ell_gpu[targets] - head)
    assert err_head.max() <= TOL_LOGPROB, f"LM head on the stack rows: {err_head.max()}"
    # 2./3. the chain against the oracle's stack and head
    tg_row = lay["tgt_row"][targets]
    rows = np.unique(tg_row)
    lse, z = O.row_logsumexp(ref, W, rows)
    pos = {int(n): i for i, n in enumerate(rows)}
    k = np.array([pos[int(n)] for n in tg_row])
    y = lay["target_ids"][targets].astype(np.int64)
    ell_ref = z[k, y] - lse[k]
    prob = np.exp(z - lse[:, None])
    EW = np.zeros((len(rows), W.shape[1]), np.float64)
    for v0 in range(0, W.shape[0], 8192):
        EW += prob[:, v0:v0 + 8192] @ np.asarray(W[v0:v0 + 8192], np.float64)
    grad = np.asarray(W[y], np.float64) - EW[k]
    dh = (got - ref)[tg_row]
    dl = ell_gpu[targets] - ell_ref
    resid = np.abs(dl - np.sum(grad * dh, axis=1))
    rms_h = np.sqrt(np.mean(ref[tg_row] ** 2, axis=1))
    bar = TOL_LOGPROB + CHAIN_SIGMAS * np.linalg.norm(grad, axis=1) * (
        CHAIN_RMS_PER_MEAN * L * TOL_STACK_MEAN_PER_LAYER) * rms_h
    print(f"chained log-probs ({L} layers, {len(targets)} targets): head on device rows "
          f"max {err_head.max():.3e}; chain max |dl| {np.abs(dl).max():.3e} "
          f"(mean {np.abs(dl).mean():.3e}, fixed bar {bar.min():.3e} .. {bar.max():.3e}); "
          f"after removing g.dh max {resid.max():.3e}")
    assert resid.max() <= TOL_LOGPROB, f"chain beyond the row difference: {resid.max()}"
    assert np.all(np.abs(dl) <= bar), f"chained log-prob error {np.abs(dl).max()}"
    # per candidate: sums of the targets above, in t order (Eq. 3)
    pos_t = {int(j): i for i, j in enumerate(targets)}
    ds_head, ds = [], []
    for c in cands:
        ts = range(int(lay["tgt_offset"][c]), int(lay["tgt_offset"][c + 1]))
        idx = [pos_t[j] for j in ts]
        ds_head.append(abs(s_gpu[c] - head[idx].sum()))
        ds.append(abs(s_gpu[c] - ell_ref[idx].sum()))
        assert ds[-1] <= bar[idx].sum()
    print(f"chained scores: head on device rows max {max(ds_head):.3e}; chain max {max(ds):.3e}")
    assert max(ds_head) <= TOL_LOGPROB, f"candidate score on the stack rows: {max(ds_head)}"


def test_stack_then_scores(cuda):
    # the stack's rows are the LM head's hidden states
    spec = jet_synth.StackSpec(("full", "linear"), 128)
    cl = [2, 1, 6, 3]
    p = jet_synth.custom_problem(SMALL, [40, 90], [2, 2], cl,
                                 np.arange(sum(cl)) * 13 % SMALL.V, seed=42)
    got, st = _gpu_stack(cuda, p, spec, "delta")
    ref = _oracle_stack(p, spec, "delta")
    _check_rows(got, ref, len(spec.kinds))
    ell, s = _score_gpu(cuda, p, st.x)
    _chained_checks(oracle_layout(p), got, ref, p.f32("w_lm"), ell, s, len(spec.kinds))


def test_stack_full_size_hybrid4(cuda):
    # four layers (3 linear : 1 full) on the ordinal_hybrid batch (32 requests,
    # 337 rows, D = 4,096, MLP width 12,288), then the full-vocabulary LM head
    # (V = 151,936) on sampled requests
    spec = jet_synth.STACKS["hybrid4"]
    p = jet_synth.make_problem("ordinal_hybrid")
    got, st = _gpu_stack(cuda, p, spec, "delta")
    ref = _oracle_stack(p, spec, "delta")
    _check_rows(got, ref, len(spec.kinds))
    ell, s = _score_gpu(cuda, p, st.x)
    lay = oracle_layout(p)
    reqs = [0, 13, p.R - 1]
    cands = np.concatenate([np.arange(lay["cand_offset"][r], lay["cand_offset"][r + 1])
                            for r in reqs])
    targets = np.concatenate([np.arange(lay["tgt_offset"][c], lay["tgt_offset"][c + 1])
                              for c in cands])
    _chained_checks(lay, got, ref, p.f32("w_lm"), ell, s, len(spec.kinds), targets, cands)


def test_stack_edges(cuda):
    import torch
    from paper_2609_33874_gb300.step import DecoderStack
    # every candidate a single token: no fed rows (F = 0), a one-token prefix
    spec = jet_synth.StackSpec(("linear", "full"), 128)
    p = jet_synth.custom_problem(SMALL, [1, 5], [2, 3], [1, 1, 1, 1, 1], [3, 4, 5, 6, 7], seed=43)
    got, st = _gpu_stack(cuda, p, spec, "delta")
    _check_rows(got, _oracle_stack(p, spec, "delta"), len(spec.kinds))
    # in place (x = x0) gives the same rows as out of place
    x0 = jet_synth.array_to_torch(jet_synth.stack_x0(p), "cuda")
    xin = x0.clone()
    cuda.jet_stack_forward(st.layout, st.dims, st.stack, xin, xin, st.ws)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(xin.float().cpu().numpy(), got)
    # no layers: a copy
    w = p.work
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    empty = DecoderStack(hl, st.dims, [], 128)
    y = empty.forward(x0)
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == 0
    assert torch.equal(y, x0)
