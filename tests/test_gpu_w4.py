"""GPU parity of the 4-bit (w4) LM head through the C ABI: the quantiser's
codes, block exponents and scales against the oracle's own quantisation of the
same bf16 weights (bit-exact, after reading back the code and scale-factor
layout the library documents), and token log-probabilities / candidate scores against the
oracle's 4-bit model (each side quantises the weights and hidden states
itself)."""
import dataclasses

import numpy as np
import pytest

import jet_synth
import oracle as O
from oracle import w4 as Q4
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


def untile(buf, V, D):
    """(codes [Vp, Kp] 0..15, exps [Vp, Kp / 32] int8) from the documented
    layout: a row-major code region of Vp = 128 ceil(V / 128) rows of
    Kp = 128 ceil(D / 128) codes, element 2 j of a row in the low nibble of its
    byte j; then one 512-byte chunk of UE8M0 scale factors per (vocabulary
    tile vt, K slice kb), chunk index vt * ceil(D / 128) + kb, holding row
    32 j + i of the tile's factor for block c of the slice at byte
    16 i + 4 j + c (factor = 127 + e)."""
    nvt, nkb = -(-V // 128), -(-D // 128)
    Vp, Kp = nvt * 128, nkb * 128
    b = np.asarray(buf, dtype=np.uint8)
    assert b.size == Vp * Kp // 2 + nvt * nkb * 512
    by = b[:Vp * Kp // 2].reshape(Vp, Kp // 2)
    codes = np.stack([by & 15, by >> 4], axis=-1).reshape(Vp, Kp)
    sf = b[Vp * Kp // 2:].reshape(nvt, nkb, 32, 4, 4)          # [vt, kb, i, j, c]
    e = sf.astype(np.int16) - 127
    exps = e.transpose(0, 3, 2, 1, 4).reshape(Vp, nkb * 4).astype(np.int8)  # row 32 j + i
    return codes, exps


def _quantize_on_gpu(cuda, w_dev):
    import torch
    V, D = w_dev.shape
    nbytes = cuda.jet_w4_bytes(V, D)
    assert nbytes == -(-V // 128) * -(-D // 128) * 8704
    w4 = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    sc = torch.empty(V, dtype=torch.float32, device="cuda")
    cuda.jet_quantize_w4(w_dev, w4, sc)
    return w4, sc


def test_quantize_w4_bit_exact(cuda):
    import torch
    rng = np.random.default_rng(81)
    V, D = 300, 208          # a partial vocabulary tile, D % 128 != 0, a 16-element last block
    x = rng.standard_normal((V, D)).astype(np.float32)
    x *= np.float32(10.0) ** rng.uniform(-20, 20, size=(V, 1)).astype(np.float32)
    # blocks spread over the exponent range, and blocks far below it (clamped)
    x *= (2.0 ** -rng.integers(0, 9, size=(V, (D + 31) // 32))).repeat(32, axis=1)[:, :D]
    x[0] = 0.0                                    # a row of zeros
    x[1] = -0.0
    x[2] = 0.0
    x[2, 100] = -5.0                              # one spike
    x[3] = np.tile([6.0, 0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0, -0.25, -5.0], 21)[:D]  # ties
    x[4] = 0.0
    x[4, :32] = 6.0                               # block exponents 0, -1, ..., -5 and clamp
    for b in range(1, 7):
        x[4, 32 * b:32 * b + 16] = 6.0 * 2.0 ** -b
    x = jet_synth.bf16_round(x)
    w4, sc = _quantize_on_gpu(cuda, _bf16_device(x))
    torch.cuda.synchronize()
    codes, exps = untile(w4.cpu().numpy(), V, D)
    rc, re_, rs = Q4.quantize_rows_w4(x)
    np.testing.assert_array_equal(sc.cpu().numpy().view(np.uint32), rs.view(np.uint32))
    np.testing.assert_array_equal(codes[:V, :D], rc)
    nb = (D + 31) // 32
    np.testing.assert_array_equal(exps[:V, :nb], re_)
    # padding: codes past D and rows past V are zero; their blocks have e = -5
    assert np.all(codes[:, D:] == 0) and np.all(codes[V:] == 0)
    assert np.all(exps[:, nb:] == -5) and np.all(exps[V:] == -5)


def _score_w4(cuda, p):
    import torch
    w = p.work
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    lay = hl.to_device("cuda")
    dims = cuda.make_dims(cuda.DTYPE_BF16, Hq=w.Hq, Hkv=w.Hkv, d=w.d, D=w.D)
    hidden = jet_synth.torch_tensor(p, "hidden", device="cuda")
    w_lm = jet_synth.torch_tensor(p, "w_lm", device="cuda")
    w4, w_s = _quantize_on_gpu(cuda, w_lm)
    del w_lm
    ell = torch.empty(hl.sizes.T, dtype=torch.float32, device="cuda")
    s = torch.empty(hl.sizes.C, dtype=torch.float32, device="cuda")
    wsb = cuda.jet_workspace_bytes_e4m3(hl.sizes, dims)
    ws = torch.empty((wsb + 15) // 16 * 4, dtype=torch.float32, device="cuda")
    out = []
    for _ in range(2):  # two calls in a row give the same answer
        cuda.jet_score_candidates_w4(lay, dims, hidden, w4, w_s, ell, s, ws)
        torch.cuda.synchronize()
        assert cuda.jet_device_status() == 0
        out.append((ell.cpu().numpy(), s.cpu().numpy()))
    np.testing.assert_array_equal(out[0][0], out[1][0])
    return out[1]


def _check(p, ell, s, requests):
    lay = oracle_layout(p)
    wc, we, wsc = Q4.quantize_rows_w4(p.f32("w_lm"))
    tg, cands = [], []
    for r in requests:
        for c in range(int(lay["cand_offset"][r]), int(lay["cand_offset"][r + 1])):
            cands.append(c)
            tg.extend(range(int(lay["tgt_offset"][c]), int(lay["tgt_offset"][c + 1])))
    tg = np.asarray(tg)
    ref = Q4.token_logprobs_w4(lay, p.f32("hidden"), wc, we, wsc, tg)
    err = np.abs(ell[tg] - ref)
    assert err.max() <= TOL_LOGPROB, f"token log-prob error {err.max()}"
    full = np.zeros(lay["T"])
    full[tg] = ref
    sref = O.candidate_scores(lay, full)
    serr = np.abs(s[cands] - sref[cands])
    assert serr.max() <= TOL_LOGPROB, f"candidate score error {serr.max()}"
    assert np.all(np.isfinite(ell)) and np.all(ell <= 1e-6)


W4_CASES = [
    (dict(V=1000, D=96), [4, 9], [3, 2], [1, 4, 2, 6, 3]),           # V % 128 != 0, one K slice
    (dict(V=129, D=64), [2], [5], [1, 1, 2, 1, 40]),                 # one vocabulary tail row
    (dict(V=20000, D=256, w_std=0.05), [3] * 7, [4] * 7, [3] * 28),
    (dict(V=1100, D=96), [5] * 4, [6] * 4, [4] * 24),                # odd tile count, ragged last tile
    (dict(V=5000, D=208), [2] * 3, [10] * 3, [10] * 30),             # two token tiles; D % 128 != 0
    (dict(V=1025, D=400), [2] * 6, [10] * 6, [11] * 60),             # three token tiles
]


@pytest.mark.parametrize("case", range(len(W4_CASES)))
def test_w4_lm_head_cases(cuda, case):
    over, pl, nc, cl = W4_CASES[case]
    wl = dataclasses.replace(jet_synth.WORKLOADS["tiny"], dtype="bf16", **over)
    rng = np.random.default_rng(90 + case)
    ids = rng.integers(0, wl.V, size=int(np.sum(cl)))
    ids[0], ids[-1] = 0, wl.V - 1
    p = jet_synth.custom_problem(wl, pl, nc, cl, ids, seed=90 + case)
    ell, s = _score_w4(cuda, p)
    _check(p, ell, s, list(range(p.R)))


def test_w4_full_size_dense27b_mc(cuda):
    # the benchmark's shape (V = 151,936, D = 5,120): sampled requests
    p = jet_synth.make_problem("dense27b_mc")
    ell, s = _score_w4(cuda, p)
    _check(p, ell, s, [0, 7, 15])


def test_w4_rejects_unsupported(cuda):
    import torch
    p = jet_synth.make_problem("tiny")
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, p.work.V)
    dims = cuda.make_dims(cuda.DTYPE_F32, D=512)   # float32 hidden: no 4-bit path
    x = torch.empty(16, dtype=torch.float32, device="cuda")
    with pytest.raises(cuda.JetError) as e:
        cuda.jet_score_candidates_w4(hl.to_device("cuda"), dims, x, x, x, x, x, x)
    assert e.value.status == 7
