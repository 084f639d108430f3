"""GPU parity of the MXFP8 LM head through the C ABI: the quantiser's codes and
block exponents against the oracle's own quantisation of the same bf16 weights
(bit-exact, after reading back the layout include/jet.h documents), and token
log-probabilities / candidate scores against the oracle's MXFP8 model (each
side quantises the weights and the hidden states itself)."""
import dataclasses

import numpy as np
import pytest

import jet_synth
import oracle as O
from oracle import mx as MX
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


def read_back(buf, V, D):
    """(codes [V, D] uint8, exps [Vp, 4 ceil(D / 128)] int) from the documented
    layout: codes row-major (V D bytes rounded up to 256), then a 512-byte
    chunk per (128-row tile vt, 128-element slice kb), chunk vt ceil(D/128) + kb,
    byte 16 i + 4 j + c = 127 + X of block c of the slice in row 128 vt + 32 j + i."""
    nvt, nkb = -(-V // 128), -(-D // 128)
    b = np.asarray(buf, dtype=np.uint8)
    off = -(-(V * D) // 256) * 256
    assert b.size == off + nvt * nkb * 512
    codes = b[:V * D].reshape(V, D)
    sf = b[off:].reshape(nvt, nkb, 32, 4, 4).astype(np.int64) - 127   # [vt, kb, i, j, c]
    exps = sf.transpose(0, 3, 2, 1, 4).reshape(nvt * 128, nkb * 4)     # row 128 vt + 32 j + i
    return codes, exps


def _quantize_on_gpu(cuda, w_dev):
    import torch
    V, D = w_dev.shape
    nbytes = cuda.jet_mxfp8_bytes(V, D)
    out = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    cuda.jet_quantize_mxfp8(w_dev, out)
    return out


def test_quantize_mxfp8_bit_exact(cuda):
    import torch
    rng = np.random.default_rng(71)
    V, D = 300, 208          # a partial vocabulary tile, D % 128 != 0, a 16-element last block
    x = rng.standard_normal((V, D)).astype(np.float32)
    x *= np.float32(10.0) ** rng.uniform(-25, 25, size=(V, 1)).astype(np.float32)
    x *= (2.0 ** -rng.integers(0, 12, size=(V, (D + 31) // 32))).repeat(32, axis=1)[:, :D]
    x[0] = 0.0                                     # a row of zeros
    x[1] = -0.0
    x[2, :32] = 480.0                              # a block whose maximum saturates
    x[2, 32:64] = 1.75 * 2.0 ** 5                  # ... and one exactly on the top code
    x[3] = 1e-38                                   # tiny (subnormal-range) blocks
    x[4, ::7] = 3.0e38                             # the largest binade
    x = jet_synth.bf16_round(x)
    out = _quantize_on_gpu(cuda, _bf16_device(x))
    torch.cuda.synchronize()
    assert cuda.jet_device_status() == 0
    codes, exps = read_back(out.cpu().numpy(), V, D)
    rc, re_ = MX.quantize_rows_mxfp8(x)
    np.testing.assert_array_equal(codes, rc)
    nb = (D + 31) // 32
    np.testing.assert_array_equal(exps[:V, :nb], re_)
    # blocks past D are blocks of zeros; rows past V carry the factor of 1
    assert np.all(exps[:V, nb:] == -127) and np.all(exps[V:] == 0)


def _score_mx(cuda, p):
    import torch
    w = p.work
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, w.V)
    lay = hl.to_device("cuda")
    dims = cuda.make_dims(cuda.DTYPE_BF16, Hq=w.Hq, Hkv=w.Hkv, d=w.d, D=w.D)
    hidden = jet_synth.torch_tensor(p, "hidden", device="cuda")
    w_lm = jet_synth.torch_tensor(p, "w_lm", device="cuda")
    w_mx = _quantize_on_gpu(cuda, w_lm)
    del w_lm
    ell = torch.empty(hl.sizes.T, dtype=torch.float32, device="cuda")
    s = torch.empty(hl.sizes.C, dtype=torch.float32, device="cuda")
    wsb = cuda.jet_workspace_bytes_mxfp8(hl.sizes, dims)
    ws = torch.empty((wsb + 15) // 16 * 4, dtype=torch.float32, device="cuda")
    out = []
    for _ in range(2):  # two calls in a row give the same answer
        cuda.jet_score_candidates_mxfp8(lay, dims, hidden, w_mx, ell, s, ws)
        torch.cuda.synchronize()
        assert cuda.jet_device_status() == 0
        out.append((ell.cpu().numpy(), s.cpu().numpy()))
    np.testing.assert_array_equal(out[0][0], out[1][0])
    return out[1]


def _check(p, ell, s, requests):
    lay = oracle_layout(p)
    wc, we = MX.quantize_rows_mxfp8(p.f32("w_lm"))
    tg, cands = [], []
    for r in requests:
        for c in range(int(lay["cand_offset"][r]), int(lay["cand_offset"][r + 1])):
            cands.append(c)
            tg.extend(range(int(lay["tgt_offset"][c]), int(lay["tgt_offset"][c + 1])))
    tg = np.asarray(tg)
    ref = MX.token_logprobs_mxfp8(lay, p.f32("hidden"), wc, we, tg)
    err = np.abs(ell[tg] - ref)
    assert err.max() <= TOL_LOGPROB, f"token log-prob error {err.max()}"
    full = np.zeros(lay["T"])
    full[tg] = ref
    sref = O.candidate_scores(lay, full)
    serr = np.abs(s[cands] - sref[cands])
    assert serr.max() <= TOL_LOGPROB, f"candidate score error {serr.max()}"
    assert np.all(np.isfinite(ell)) and np.all(ell <= 1e-6)


MX_CASES = [
    (dict(V=1000, D=96), [4, 9], [3, 2], [1, 4, 2, 6, 3]),           # V % 128 != 0, one K slice
    (dict(V=129, D=64), [2], [5], [1, 1, 2, 1, 40]),                 # one vocabulary tail row
    (dict(V=20000, D=256, w_std=0.05), [3] * 7, [4] * 7, [3] * 28),
    (dict(V=1100, D=96), [5] * 4, [6] * 4, [4] * 24),                # odd tile count, ragged last tile
    (dict(V=5000, D=208), [2] * 3, [10] * 3, [10] * 30),             # two token tiles of 144 rows
    (dict(V=1025, D=400), [2] * 6, [10] * 6, [11] * 60),             # three token tiles of 208 rows
    (dict(V=3000, D=128), [2] * 2, [10] * 2, [11] * 20),             # one tile of 208 rows (> 128)
]


@pytest.mark.parametrize("case", range(len(MX_CASES)))
def test_mx_lm_head_cases(cuda, case):
    over, pl, nc, cl = MX_CASES[case]
    wl = dataclasses.replace(jet_synth.WORKLOADS["tiny"], dtype="bf16", **over)
    rng = np.random.default_rng(60 + case)
    ids = rng.integers(0, wl.V, size=int(np.sum(cl)))
    ids[0], ids[-1] = 0, wl.V - 1
    p = jet_synth.custom_problem(wl, pl, nc, cl, ids, seed=60 + case)
    ell, s = _score_mx(cuda, p)
    _check(p, ell, s, list(range(p.R)))


def test_mx_full_size_dense27b_mc(cuda):
    # the benchmark's shape (V = 151,936, D = 5,120): sampled requests
    p = jet_synth.make_problem("dense27b_mc")
    ell, s = _score_mx(cuda, p)
    _check(p, ell, s, [0, 7, 15])


def test_mx_rejects_unsupported(cuda):
    import torch
    p = jet_synth.make_problem("tiny")
    hl = cuda.jet_layout_build(p.prefix_len, p.n_cand, p.cand_len, p.target_ids, p.work.V)
    dims = cuda.make_dims(cuda.DTYPE_F32, D=512)   # float32 hidden: no MXFP8 path
    x = torch.empty(16, dtype=torch.float32, device="cuda")
    with pytest.raises(cuda.JetError) as e:
        cuda.jet_score_candidates_mxfp8(hl.to_device("cuda"), dims, x, x, x, x, x)
    assert e.value.status == 7
