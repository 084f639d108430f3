"""GPU parity of the hybrid decoder stack (jet_stack_forward) through the C ABI
against the oracle's stack with the same storage points, on the same seeded
inputs: a small ragged batch with both layer kinds and both recurrence rules,
the stack's rows fed through the LM head (token log-probabilities and
candidate scores against the oracle's), and the full-size four-layer hybrid
stack on the ordinal_hybrid batch."""
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


def test_stack_then_scores(cuda):
    # the stack's rows are the LM head's hidden states
    import torch
    spec = jet_synth.StackSpec(("full", "linear"), 128)
    cl = [2, 1, 6, 3]
    p = jet_synth.custom_problem(SMALL, [40, 90], [2, 2], cl,
                                 np.arange(sum(cl)) * 13 % SMALL.V, seed=42)
    got, st = _gpu_stack(cuda, p, spec, "delta")
    ref = _oracle_stack(p, spec, "delta")
    _check_rows(got, ref, len(spec.kinds))
    w = p.work
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    dims = cuda.make_dims(cuda.DTYPE_BF16, D=w.D)
    w_lm = jet_synth.torch_tensor(p, "w_lm", device="cuda")
    ell = torch.empty(hl.sizes.T, dtype=torch.float32, device="cuda")
    s = torch.empty(hl.sizes.C, dtype=torch.float32, device="cuda")
    wsb = cuda.jet_workspace_bytes(hl.sizes, dims)
    ws = torch.empty((wsb + 15) // 16 * 4, dtype=torch.float32, device="cuda")
    cuda.jet_score_candidates(hl.to_device("cuda"), dims, st.x, w_lm, ell, s, ws)
    torch.cuda.synchronize()
    lay = oracle_layout(p)
    ref_ell = O.token_logprobs(lay, ref, p.f32("w_lm"))
    # the scoring step's own bar, plus what the hidden-state difference can
    # move a log-probability: |dl| <= 2 max_v |W_v . dH| <= 2 max_v |W_v| |dH|
    W = p.f32("w_lm").astype(np.float64)
    dh = np.linalg.norm(got - ref, axis=1)
    tol_rows = TOL_LOGPROB + 2 * np.linalg.norm(W, axis=1).max() * dh
    tg_row = lay["tgt_row"]
    err = np.abs(ell.cpu().numpy() - ref_ell)
    print(f"log-prob error max {err.max():.3e}, bar {tol_rows[tg_row].min():.3e} .. "
          f"{tol_rows[tg_row].max():.3e}")
    assert np.all(err <= tol_rows[tg_row]), f"token log-prob error {err.max()}"
    ref_s = O.candidate_scores(lay, ref_ell)
    tol_c = np.array([tol_rows[tg_row[int(lay["tgt_offset"][c]):int(lay["tgt_offset"][c + 1])]]
                      .sum() for c in range(lay["C"])])
    assert np.all(np.abs(s.cpu().numpy() - ref_s) <= tol_c)


def test_stack_full_size_hybrid4(cuda):
    # four layers (3 linear : 1 full) on the ordinal_hybrid batch (32 requests,
    # 337 rows, D = 4,096, MLP width 12,288)
    spec = jet_synth.STACKS["hybrid4"]
    p = jet_synth.make_problem("ordinal_hybrid")
    got, _ = _gpu_stack(cuda, p, spec, "delta")
    _check_rows(got, _oracle_stack(p, spec, "delta"), len(spec.kinds))


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
