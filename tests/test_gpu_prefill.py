"""GPU parity of the prefill - causal self-attention over every request's
prefix - through the C ABI against the oracle on the same seeded inputs:
ragged prefixes around the 64-key tile and the query-block size, every head
dimension, and the full-size dense27b_mc prefixes (sampled rows)."""
import dataclasses

import numpy as np
import pytest

import jet_synth
import oracle as O
from gpu_common import TOL_ATTN_BF16

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
