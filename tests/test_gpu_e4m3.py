"""GPU parity of the e4m3 LM head through the C ABI: the quantiser against the
oracle's own quantisation of the same bf16 inputs (bit-exact codes and
scales), and token log-probabilities / candidate scores against the oracle's
quantised model (each side quantises the weights and hidden states itself)."""
import dataclasses

import numpy as np
import pytest

import jet_synth
import oracle as O
from oracle import e4m3 as Q
from gpu_common import TOL_LOGPROB, oracle_layout

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cuda(jet):
    import torch
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required for -m gpu tests")
    return jet


def _bf16_device(x32):
    import torch
    bits = jet_synth.f32_to_bf16_bits(x32)
    return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).cuda()


def _quantize_on_gpu(cuda, x_dev):
    import torch
    rows, D = x_dev.shape
    q = torch.empty(rows, D, dtype=torch.uint8, device="cuda")
    s = torch.empty(rows, dtype=torch.float32, device="cuda")
    cuda.jet_quantize_rows_e4m3(x_dev, q, s)
    torch.cuda.synchronize()
    return q.cpu().numpy(), s.cpu().numpy()


def test_quantize_rows_bit_exact(cuda):
    rng = np.random.default_rng(61)
    rows, D = 96, 528
    x = rng.standard_normal((rows, D)).astype(np.float32)
    x *= np.float32(10.0) ** rng.uniform(-30, 30, size=(rows, 1)).astype(np.float32)
    x[0] = 0.0                                   # a row of zeros: scale 0
    x[1] = -0.0                                  # negative zeros keep their sign bit
    x[2] = 0.0
    x[2, 17] = -3.0                              # one spike: scaled to exactly -448
    x[3] = rng.uniform(-1e-3, 1e-3, D)           # values that fall in the subnormal codes
    x[3, 5] = 1.0
    x[4] = np.linspace(-448.0, 448.0, D)         # ties and saturation at the grid's edge
    x = jet_synth.bf16_round(x)
    q, s = _quantize_on_gpu(cuda, _bf16_device(x))
    codes, scale = Q.quantize_rows(x)
    np.testing.assert_array_equal(s.view(np.uint32), scale.view(np.uint32))
    np.testing.assert_array_equal(q, codes)


def _score_e4m3(cuda, p):
    """Run jet_score_candidates_e4m3 on problem p; W quantised on the GPU."""
    import torch
    w = p.work
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    lay = hl.to_device("cuda")
    dims = cuda.make_dims(cuda.DTYPE_BF16, Hq=w.Hq, Hkv=w.Hkv, d=w.d, D=w.D)
    hidden = jet_synth.torch_tensor(p, "hidden", device="cuda")
    w_lm = jet_synth.torch_tensor(p, "w_lm", device="cuda")
    w_q = torch.empty(w.V, w.D, dtype=torch.uint8, device="cuda")
    w_s = torch.empty(w.V, dtype=torch.float32, device="cuda")
    cuda.jet_quantize_rows_e4m3(w_lm, w_q, w_s)
    del w_lm
    ell = torch.empty(hl.sizes.T, dtype=torch.float32, device="cuda")
    s = torch.empty(hl.sizes.C, dtype=torch.float32, device="cuda")
    wsb = cuda.jet_workspace_bytes_e4m3(hl.sizes, dims)
    ws = torch.empty((wsb + 15) // 16 * 4, dtype=torch.float32, device="cuda")
    cuda.jet_score_candidates_e4m3(lay, dims, hidden, w_q, w_s, ell, s, ws)
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == 0
    return ell.cpu().numpy(), s.cpu().numpy()


def _check(p, ell, s, requests):
    lay = oracle_layout(p)
    wc, wsc = Q.quantize_rows(p.f32("w_lm"))
    tg, cands = [], []
    for r in requests:
        for c in range(int(lay["cand_offset"][r]), int(lay["cand_offset"][r + 1])):
            cands.append(c)
            tg.extend(range(int(lay["tgt_offset"][c]), int(lay["tgt_offset"][c + 1])))
    tg = np.asarray(tg)
    ref = Q.token_logprobs_e4m3(lay, p.f32("hidden"), wc, wsc, tg)
    err = np.abs(ell[tg] - ref)
    assert err.max() <= TOL_LOGPROB, f"token log-prob error {err.max()}"
    full = np.zeros(lay["T"])
    full[tg] = ref
    sref = O.candidate_scores(lay, full)
    serr = np.abs(s[cands] - sref[cands])
    assert serr.max() <= TOL_LOGPROB, f"candidate score error {serr.max()}"
    assert np.all(np.isfinite(ell)) and np.all(ell <= 1e-6)


E4M3_CASES = [
    (dict(V=1000, D=96), [4, 9], [3, 2], [1, 4, 2, 6, 3]),           # V % 128 != 0
    (dict(V=129, D=64), [2], [5], [1, 1, 2, 1, 40]),                 # one vocabulary tail row
    (dict(V=20000, D=256, w_std=0.05), [3] * 7, [4] * 7, [3] * 28),
    (dict(V=1100, D=96), [5] * 4, [6] * 4, [4] * 24),                # odd tile count, ragged last tile
    (dict(V=5000, D=208), [2] * 3, [10] * 3, [10] * 30),             # two token tiles; D % 128 != 0
    (dict(V=1025, D=128), [2] * 6, [10] * 6, [11] * 60),             # three token tiles
]


@pytest.mark.parametrize("case", range(len(E4M3_CASES)))
def test_e4m3_lm_head_cases(cuda, case):
    over, pl, nc, cl = E4M3_CASES[case]
    wl = dataclasses.replace(jet_synth.WORKLOADS["tiny"], dtype="bf16", **over)
    rng = np.random.default_rng(70 + case)
    ids = rng.integers(0, wl.V, size=int(np.sum(cl)))
    ids[0], ids[-1] = 0, wl.V - 1
    p = jet_synth.custom_problem(wl, pl, nc, cl, ids, seed=70 + case)
    ell, s = _score_e4m3(cuda, p)
    _check(p, ell, s, list(range(p.R)))


def test_e4m3_full_size_dense27b_mc(cuda):
    # the benchmark's shape (V = 151,936, D = 5,120): sampled requests
    p = jet_synth.make_problem("dense27b_mc")
    ell, s = _score_e4m3(cuda, p)
    _check(p, ell, s, [0, 7, 15])


def test_e4m3_rejects_unsupported(cuda):
    import torch
    p = jet_synth.make_problem("tiny")
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, p.work.V)
    dims = cuda.make_dims(cuda.DTYPE_F32, D=512)   # float32 hidden: no e4m3 path
    x = torch.empty(16, dtype=torch.float32, device="cuda")
    with pytest.raises(cuda.JetError) as e:
        cuda.jet_score_candidates_e4m3(hl.to_device("cuda"), dims, x, x, x, x, x, x)
    assert e.value.status == 7
