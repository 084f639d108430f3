"""GPU parity of the prefill - causal self-attention over every request's
prefix - through the C ABI against the oracle on the same seeded inputs:
ragged prefixes around the 64-key tile and the query-block size, every head
dimension, and the full-size dense27b_mc prefixes (sampled rows); and of the
prefix scan of a linear-attention layer's recurrent state (both rules, both
dtypes, prefixes around the 32-token staging window, the full hybrid prefixes)."""
import dataclasses

import numpy as np
import pytest

import jet_synth
import oracle as O
from gpu_common import TOL_ATTN_BF16, TOL_FORK_REL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cuda(jet):
    import torch
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required for -m gpu tests")
    return jet


def _prefill(cuda, p):
    import torch
    w = p.work
    R = p.R
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    dims = cuda.make_dims(cuda.DTYPE_BF16, Hq=w.Hq, Hkv=w.Hkv, d=w.d, D=w.D)
    q = jet_synth.torch_tensor(p, "q_pre", device="cuda")
    k = jet_synth.torch_tensor(p, "k_pre", device="cuda")
    v = jet_synth.torch_tensor(p, "v_pre", device="cuda")
    o = torch.empty(p.total_prefix, w.Hq, w.d, dtype=torch.bfloat16, device="cuda")
    wsb = cuda.jet_prefill_workspace_bytes(hl.sizes, dims)
    assert wsb > 0 and R >= 1
    ws = torch.empty((wsb + 15) // 16 * 4, dtype=torch.float32, device="cuda")
    cuda.jet_prefill_attend(hl.to_device("cuda"), dims, q, k, v, o, ws)
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == 0
    return o.float().cpu().numpy()


def _sample_rows(prefix_len, rng, per=12):
    off = np.concatenate([[0], np.cumsum(prefix_len)])
    rows = []
    for r, P in enumerate(prefix_len):
        pick = set(range(min(3, P))) | set(range(max(0, P - 3), P))
        pick |= set(rng.integers(0, P, size=min(per, P)).tolist())
        rows.extend(int(off[r]) + x for x in sorted(pick))
    return rows


def _check(p, got, rows):
    w = p.work
    ref = O.prefill_attention(p.prefix_len, p.f32("q_pre"), p.f32("k_pre"), p.f32("v_pre"),
                              w.Hq, w.Hkv, rows=rows)
    err = np.abs(got[rows] - ref)
    assert err.max() <= TOL_ATTN_BF16, f"prefill error {err.max()}"


PREFILL_CASES = [
    ([1, 63, 64, 65, 300], dict(Hq=8, Hkv=2, d=64)),      # tile edges, 16-row blocks
    ([700, 129, 5], dict(Hq=6, Hkv=3, d=128)),             # 64-row blocks
    ([1000, 257, 21, 22], dict(Hq=24, Hkv=4, d=256)),      # 21-row blocks: ragged last block
    ([513, 512, 17], dict(Hq=16, Hkv=2, d=256)),
    ([130], dict(Hq=4, Hkv=4, d=64)),                      # g = 1: 128-row blocks
]


@pytest.mark.parametrize("case", range(len(PREFILL_CASES)))
def test_prefill_cases(cuda, case):
    pl, over = PREFILL_CASES[case]
    w = dataclasses.replace(jet_synth.WORKLOADS["tiny"], dtype="bf16", **over)
    R = len(pl)
    p = jet_synth.custom_problem(w, pl, [1] * R, [1] * R, [0] * R, seed=90 + case)
    got = _prefill(cuda, p)
    rows = list(range(p.total_prefix)) if p.total_prefix <= 400 else \
        _sample_rows(p.prefix_len, np.random.default_rng(case))
    _check(p, got, rows)


def test_prefill_full_size_dense27b_mc(cuda):
    p = jet_synth.make_problem("dense27b_mc")
    got = _prefill(cuda, p)
    _check(p, got, _sample_rows(p.prefix_len, np.random.default_rng(7), per=4))


# ---------------------------------------------------------------------------
# prefill of the recurrent state (the prefix scan)
# ---------------------------------------------------------------------------
def _scan(cuda, p, rule, with_init):
    import torch
    w = p.work
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    dims = cuda.make_dims(cuda.DTYPE_BF16 if p.bf16 else cuda.DTYPE_F32, Hl=w.Hl, dk=w.dk,
                          dv=w.dv, D=w.D)
    t = {n: jet_synth.torch_tensor(p, n, device="cuda")
         for n in ("lq_pre", "lk_pre", "lv_pre", "alpha_pre", "beta_pre")}
    s_init = jet_synth.torch_tensor(p, "s_prefix", device="cuda") if with_init else None
    dt = torch.bfloat16 if p.bf16 else torch.float32
    o = torch.empty(p.total_prefix, w.Hl, w.dv, dtype=dt, device="cuda")
    s_out = torch.empty(p.R, w.Hl, w.dk, w.dv, dtype=torch.float32, device="cuda")
    cuda.jet_prefill_state(hl.to_device("cuda"), dims, t["lq_pre"], t["lk_pre"], t["lv_pre"],
                           t["alpha_pre"], t["beta_pre"], o, s_out, s_init=s_init,
                           rule=cuda.RULES[rule])
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == 0
    return o.float().cpu().numpy(), s_out.cpu().numpy()


def _check_scan_out(got, ref, bf16):
    # outputs are stored in the workload's dtype: bf16 rounds each to 8
    # significant bits (relative 2^-9), float32 to 24; the state itself is
    # float32 throughout
    atol, rtol = (1e-3, 8e-3) if bf16 else (1e-5, 1e-5)
    err = np.abs(got - ref) - (atol + rtol * np.abs(ref))
    assert err.max() <= 0, f"scan output error {np.abs(got - ref).max()}"


@pytest.mark.parametrize("rule", ["delta", "gla"])
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_prefill_state(cuda, rule, dtype):
    # prefixes around the 32-token staging window; with and without a start state
    w = dataclasses.replace(jet_synth.WORKLOADS["ordinal_hybrid"], Hl=3, dv=64, dtype=dtype)
    pl = [1, 31, 32, 33, 70]
    R = len(pl)
    p = jet_synth.custom_problem(w, pl, [1] * R, [1] * R, [0] * R, seed=95)
    for with_init in (False, True):
        got_o, got_s = _scan(cuda, p, rule, with_init)
        ref_o, ref_s = O.prefill_state(p.prefix_len, p.f32("s_prefix") if with_init else None,
                                       p.f32("lq_pre"), p.f32("lk_pre"), p.f32("lv_pre"),
                                       p.f32("alpha_pre"), p.f32("beta_pre"), rule)
        rel = np.abs(got_s - ref_s).max() / np.abs(ref_s).max()
        assert rel <= TOL_FORK_REL, f"state error {rel}"
        _check_scan_out(got_o, ref_o, p.bf16)


@pytest.mark.parametrize("rule", ["delta", "gla"])
def test_prefill_state_full_hybrid(cuda, rule):
    # the hybrid workload's prefixes (32 requests x 512 tokens, 16 heads): the
    # chunked scan in the launch configuration the bench times
    p = jet_synth.make_problem("ordinal_hybrid")
    got_o, got_s = _scan(cuda, p, rule, True)
    sub = [0, 13, 31]
    off = np.concatenate([[0], np.cumsum(p.prefix_len)])
    rows = np.concatenate([np.arange(off[r], off[r + 1]) for r in sub])
    sel = lambda n: p.f32(n)[rows]  # noqa: E731
    ref_o, ref_s = O.prefill_state(p.prefix_len[sub], p.f32("s_prefix")[sub], sel("lq_pre"),
                                   sel("lk_pre"), sel("lv_pre"), sel("alpha_pre"),
                                   sel("beta_pre"), rule)
    rel = np.abs(got_s[sub] - ref_s).max() / np.abs(ref_s).max()
    assert rel <= TOL_FORK_REL, f"state error {rel}"
    _check_scan_out(got_o[rows], ref_o, True)


@pytest.mark.parametrize("dv", [32, 160])
def test_prefill_state_column_tails(cuda, dv):
    # dv % 64 == 32: the last 64-column block of each head is half full
    w = dataclasses.replace(jet_synth.WORKLOADS["ordinal_hybrid"], Hl=2, dv=dv, dtype="bf16")
    pl = [17, 48, 3]
    R = len(pl)
    p = jet_synth.custom_problem(w, pl, [1] * R, [1] * R, [0] * R, seed=96)
    got_o, got_s = _scan(cuda, p, "delta", True)
    ref_o, ref_s = O.prefill_state(p.prefix_len, p.f32("s_prefix"), p.f32("lq_pre"),
                                   p.f32("lk_pre"), p.f32("lv_pre"), p.f32("alpha_pre"),
                                   p.f32("beta_pre"), "delta")
    rel = np.abs(got_s - ref_s).max() / np.abs(ref_s).max()
    assert rel <= TOL_FORK_REL, f"state error {rel}"
    _check_scan_out(got_o, ref_o, True)


@pytest.mark.parametrize("rule", ["delta", "gla"])
@pytest.mark.parametrize("alpha_scale", [1.0, 0.1])
def test_prefill_state_chunked(cuda, rule, alpha_scale):
    # bf16 with 128 x 128 states runs the chunked scan on the tensor cores
    # (chunks of 64 tokens): prefixes around the chunk edges, with and without
    # a start state; alpha_scale 0.1 makes every decay strong (a ~ 0.09-0.1,
    # products far below float32's normal range within a chunk)
    import torch
    w = dataclasses.replace(jet_synth.WORKLOADS["ordinal_hybrid"], Hl=3, dtype="bf16")
    assert w.dk == 128 and w.dv == 128
    pl = [1, 63, 64, 65, 128, 130, 200]
    R = len(pl)
    p = jet_synth.custom_problem(w, pl, [1] * R, [1] * R, [0] * R, seed=97)
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    dims = cuda.make_dims(cuda.DTYPE_BF16, Hl=w.Hl, dk=w.dk, dv=w.dv, D=w.D)
    t = {n: jet_synth.torch_tensor(p, n, device="cuda")
         for n in ("lq_pre", "lk_pre", "lv_pre", "alpha_pre", "beta_pre")}
    alpha = (p.f32("alpha_pre") * np.float32(alpha_scale)).astype(np.float32)
    t["alpha_pre"] = torch.from_numpy(alpha).cuda()
    for with_init in (False, True):
        s_init = jet_synth.torch_tensor(p, "s_prefix", device="cuda") if with_init else None
        o = torch.empty(p.total_prefix, w.Hl, w.dv, dtype=torch.bfloat16, device="cuda")
        s_out = torch.empty(R, w.Hl, w.dk, w.dv, dtype=torch.float32, device="cuda")
        outs = []
        for _ in range(2):  # two calls in a row give the same answer
            cuda.jet_prefill_state(hl.to_device("cuda"), dims, t["lq_pre"], t["lk_pre"],
                                   t["lv_pre"], t["alpha_pre"], t["beta_pre"], o, s_out,
                                   s_init=s_init, rule=cuda.RULES[rule])
            torch.cuda.synchronize()
            assert cuda.jet_device_status() == 0
            outs.append((o.float().cpu().numpy(), s_out.cpu().numpy()))
        np.testing.assert_array_equal(outs[0][1], outs[1][1])
        got_o, got_s = outs[1]
        ref_o, ref_s = O.prefill_state(p.prefix_len, p.f32("s_prefix") if with_init else None,
                                       p.f32("lq_pre"), p.f32("lk_pre"), p.f32("lv_pre"), alpha,
                                       p.f32("beta_pre"), rule)
        rel = np.abs(got_s - ref_s).max() / np.abs(ref_s).max()
        print(f"chunked scan {rule} alpha x{alpha_scale} init={with_init}: state rel {rel:.2e}, "
              f"out max {np.abs(got_o - ref_o).max():.2e}")
        assert rel <= TOL_FORK_REL, f"state error {rel}"
        _check_scan_out(got_o, ref_o, True)


def test_prefill_state_chunked_long(cuda):
    # long prefixes through the chunked scan: 2,000 and 1,500 tokens (32 and
    # 24 chunks, the last ones ragged), so a start state is carried through
    # many chunk boundaries and both K buffers are reused many times
    w = dataclasses.replace(jet_synth.WORKLOADS["ordinal_hybrid"], Hl=2, dtype="bf16")
    pl = [2000, 1500]
    R = len(pl)
    p = jet_synth.custom_problem(w, pl, [1] * R, [1] * R, [0] * R, seed=98)
    got_o, got_s = _scan(cuda, p, "delta", True)
    ref_o, ref_s = O.prefill_state(p.prefix_len, p.f32("s_prefix"), p.f32("lq_pre"),
                                   p.f32("lk_pre"), p.f32("lv_pre"), p.f32("alpha_pre"),
                                   p.f32("beta_pre"), "delta")
    rel = np.abs(got_s - ref_s).max() / np.abs(ref_s).max()
    print(f"chunked scan over 2,000 / 1,500 tokens: state rel {rel:.2e}")
    assert rel <= TOL_FORK_REL, f"state error {rel}"
    _check_scan_out(got_o, ref_o, True)
