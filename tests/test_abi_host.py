"""Host-side tests of the C ABI: exported symbols, the layout builder against
the oracle's independent layout (bit-exact), and argument validation. No call
here reaches a kernel: every compute call is made with an argument the library
must reject before launching."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle as O

FIELDS = ("prefix_offset", "cand_offset", "row_offset", "cand_row_offset", "tgt_offset",
          "target_ids", "tgt_row", "row_req", "row_cand", "row_pos", "row_tgt_offset",
          "row_tgt_index")


def test_exports_every_declared_symbol(jet, repo_root):
    header = open(os.path.join(repo_root, "include", "jet.h")).read()
    declared = set(re.findall(r"^\s*(?:jet_status|size_t|int32_t|uint64_t|const char\*)\s+(jet_\w+)\s*\(",
                              header, flags=re.M))
    assert len(declared) >= 12
    lib = ctypes.CDLL(jet.LIB_PATH)
    for name in sorted(declared):
        assert hasattr(lib, name), name
    assert set(jet.DECLARED) == declared
    assert lib.jet_abi_version() == 1


def _compare(jet, prefix_len, n_cand, cand_len, ids, V):
    ref = O.build_layout(prefix_len, n_cand, cand_len, ids, V)
    lay = jet.jet_layout_build(prefix_len, n_cand, cand_len, ids, V)
    s = lay.sizes
    assert (s.R, s.C, s.N, s.T, s.V) == (ref["R"], ref["C"], ref["N"], ref["T"], V)
    assert s.total_prefix == int(np.sum(prefix_len))
    assert s.max_prefix == int(np.max(prefix_len))
    assert s.max_len == int(np.max(cand_len))
    assert s.min_cand == int(np.min(n_cand)) and s.max_cand == int(np.max(n_cand))
    rows = np.diff(ref["row_offset"])
    assert s.max_rows == int(rows.max())
    for f in FIELDS:
        got = lay.array(f)
        assert got.dtype == np.int32
        np.testing.assert_array_equal(got, ref[f], err_msg=f)
    # scheduling order: the requests by decreasing prefix length, ties in index order
    order = lay.array("req_order")
    np.testing.assert_array_equal(order, np.argsort(-np.asarray(prefix_len), kind="stable"))


def test_layout_matches_oracle_golden(jet):
    _compare(jet, [3, 2], [2, 1], [1, 3, 2], [11, 21, 22, 23, 31, 32], 64)


@pytest.mark.parametrize("seed", range(12))
def test_layout_matches_oracle_random(jet, seed):
    rng = np.random.default_rng(100 + seed)
    R = int(rng.integers(1, 40))
    n_cand = rng.integers(1, 12, size=R)
    cand_len = rng.integers(1, 13, size=int(n_cand.sum()))
    V = int(rng.integers(2, 200000))
    ids = rng.integers(0, V, size=int(cand_len.sum()))
    ids[0] = 0
    ids[-1] = V - 1
    _compare(jet, rng.integers(1, 3000, size=R), n_cand, cand_len, ids, V)


def test_layout_edge_cases(jet):
    _compare(jet, [1], [1], [1], [0], 1)                      # one token, V = 1
    _compare(jet, [5], [3], [1, 1, 1], [7, 7, 7], 8)          # duplicates, single-token only
    _compare(jet, [5, 6], [1, 1], [12, 12], list(range(24)), 24)
    V = 151936
    _compare(jet, [9], [4], [2, 2, 2, 2], [V - 1, 0, V - 2, 151935, 151872, 1, 128, 127], V)


def test_layout_plan_workload_sizes(jet):
    import jet_synth
    for name, (N, T) in {"tiny": (7, 10)}.items():
        p = jet_synth.make_problem(name)
        s = jet.jet_layout_plan(p.prefix_len, p.n_cand, p.cand_len, p.work.V)
        assert (s.N, s.T) == (N, T)
        assert s.N == p.N


def test_layout_rejects_bad_input(jet):
    with pytest.raises(jet.JetError) as e:
        jet.jet_layout_build([3], [1], [0], [], 8)
    assert e.value.status == 2  # JET_ERR_SHAPE
    with pytest.raises(jet.JetError) as e:
        jet.jet_layout_build([3], [1], [1], [8], 8)
    assert e.value.status == 3  # JET_ERR_RANGE
    with pytest.raises(jet.JetError) as e:
        jet.jet_layout_build([3], [1], [1], [-1], 8)
    assert e.value.status == 3
    with pytest.raises(jet.JetError) as e:
        jet.jet_layout_build([0], [1], [1], [1], 8)
    assert e.value.status == 2
    with pytest.raises(jet.JetError) as e:
        jet.jet_layout_plan([3], [1], [1], 0)
    assert e.value.status == 1  # JET_ERR_ARG
    # words buffer too small
    lib = jet.library()
    p, c, m, y = (np.array(v, np.int32) for v in ([3], [2], [2, 1], [1, 2, 3]))
    out = jet.jet_layout()
    small = np.zeros(4, np.int32)
    P = ctypes.POINTER(ctypes.c_int32)
    st = lib.jet_layout_build(1, p.ctypes.data_as(P), c.ctypes.data_as(P), m.ctypes.data_as(P),
                              y.ctypes.data_as(P), 8, small.ctypes.data_as(P), small.size,
                              ctypes.byref(out))
    assert st == 5  # JET_ERR_WORKSPACE


# ---------------------------------------------------------------------------
# compute entry points: rejected before any launch
# ---------------------------------------------------------------------------
FAKE = 1 << 40          # 16-byte aligned address that is never dereferenced
MIS = FAKE + 4          # misaligned


def _setup(jet):
    lay = jet.jet_layout_build([4, 3], [2, 2], [1, 3, 2, 1], list(range(7)), 16)
    dims = jet.make_dims(jet.DTYPE_BF16, Hq=8, Hkv=2, d=64, D=64, Hl=2, dk=128, dv=64)
    return lay, dims


def _attend(jet, lay, dims, q=FAKE, ws=FAKE, ws_bytes=None):
    ws_bytes = jet.jet_workspace_bytes(lay.sizes, dims) if ws_bytes is None else ws_bytes
    return jet.library().jet_prefix_attend(ctypes.byref(lay.struct), ctypes.byref(dims), q, FAKE,
                                           FAKE, FAKE, FAKE, FAKE, ws, ws_bytes, None)


def test_attend_validation(jet):
    lay, dims = _setup(jet)
    bad = jet.make_dims(jet.DTYPE_BF16, Hq=6, Hkv=4, d=64, D=64)
    assert _attend(jet, lay, bad) == 2                     # Hq % Hkv != 0
    bad = jet.make_dims(jet.DTYPE_BF16, Hq=8, Hkv=2, d=96, D=64)
    assert _attend(jet, lay, bad) == 7                     # unsupported head dim
    bad = jet.make_dims(5, Hq=8, Hkv=2, d=64, D=64)
    assert _attend(jet, lay, bad) == 7                     # unsupported dtype
    assert _attend(jet, lay, dims, q=MIS) == 4             # misaligned
    assert _attend(jet, lay, dims, q=None) == 1            # null
    assert _attend(jet, lay, dims, ws_bytes=16) == 5       # workspace too small
    assert _attend(jet, lay, dims, ws=None) == 5
    assert _attend(jet, lay, dims, ws=MIS) == 4
    assert jet.library().jet_prefix_attend(None, ctypes.byref(dims), FAKE, FAKE, FAKE, FAKE, FAKE,
                                           FAKE, FAKE, 1 << 30, None) == 1


def test_score_and_decide_validation(jet):
    lay, dims = _setup(jet)
    lib = jet.library()
    ws = jet.jet_workspace_bytes(lay.sizes, dims)
    assert ws > 0
    bad = jet.make_dims(jet.DTYPE_BF16, D=60)
    assert lib.jet_score_candidates(ctypes.byref(lay.struct), ctypes.byref(bad), FAKE, FAKE, FAKE,
                                    FAKE, FAKE, ws, None) == 2
    assert lib.jet_score_candidates(ctypes.byref(lay.struct), ctypes.byref(dims), FAKE, MIS, FAKE,
                                    FAKE, FAKE, ws, None) == 4
    assert lib.jet_score_candidates(ctypes.byref(lay.struct), ctypes.byref(dims), FAKE, FAKE, FAKE,
                                    FAKE, FAKE, 64, None) == 5
    # binary decisions need exactly two candidates per request
    assert lib.jet_decide(ctypes.byref(lay.struct), jet.DECIDE_ARGMAX + 7, FAKE, FAKE, FAKE, FAKE,
                          None) == 1
    lay3 = jet.jet_layout_build([4], [3], [1, 1, 1], [0, 1, 2], 16)
    assert lib.jet_decide(ctypes.byref(lay3.struct), jet.DECIDE_BINARY, FAKE, FAKE, FAKE, FAKE,
                          None) == 2
    assert lib.jet_decide(ctypes.byref(lay.struct), jet.DECIDE_ORDINAL, FAKE, None, FAKE, FAKE,
                          None) == 1


def test_fork_validation(jet):
    lay, dims = _setup(jet)
    lib = jet.library()
    bad = jet.make_dims(jet.DTYPE_BF16, Hl=2, dk=64, dv=64)
    args = [FAKE] * 9
    assert lib.jet_fork_state(ctypes.byref(lay.struct), ctypes.byref(bad), *args) == 7
    bad = jet.make_dims(jet.DTYPE_BF16, Hl=2, dk=128, dv=48)
    assert lib.jet_fork_state(ctypes.byref(lay.struct), ctypes.byref(bad), *args) == 7
    mis = [FAKE] * 9
    mis[7] = MIS  # s_fork
    assert lib.jet_fork_state(ctypes.byref(lay.struct), ctypes.byref(dims), *mis) == 4
    nul = [FAKE] * 9
    nul[4] = None  # alpha
    assert lib.jet_fork_state(ctypes.byref(lay.struct), ctypes.byref(dims), *nul) == 1


def test_fork_rule_validation(jet):
    lay, dims = _setup(jet)
    lib = jet.library()
    args = [FAKE] * 9
    assert lib.jet_fork_state_rule(ctypes.byref(lay.struct), ctypes.byref(dims), 7, *args) == 1
    bad = jet.make_dims(jet.DTYPE_BF16, Hl=2, dk=64, dv=64)
    assert lib.jet_fork_state_rule(ctypes.byref(lay.struct), ctypes.byref(bad), jet.RECUR_GLA,
                                   *args) == 7


def test_prefill_state_validation(jet):
    lay, dims = _setup(jet)
    lib = jet.library()
    L, D = ctypes.byref(lay.struct), ctypes.byref(dims)
    # rule, s_init (nullable), q, k, v, alpha, beta, o, s_out, stream
    args = [FAKE] * 8 + [None]
    assert lib.jet_prefill_state(L, D, 5, *args) == 1                      # unknown rule
    bad = jet.make_dims(jet.DTYPE_BF16, Hl=2, dk=64, dv=64)
    assert lib.jet_prefill_state(L, ctypes.byref(bad), jet.RECUR_DELTA, *args) == 7
    nul = list(args)
    nul[5] = None  # beta
    assert lib.jet_prefill_state(L, D, jet.RECUR_GLA, *nul) == 1
    mis = list(args)
    mis[0] = MIS   # s_init is optional but must be aligned when given
    assert lib.jet_prefill_state(L, D, jet.RECUR_DELTA, *mis) == 4
    mis = list(args)
    mis[7] = MIS   # s_out
    assert lib.jet_prefill_state(L, D, jet.RECUR_DELTA, *mis) == 4


def test_w4_validation(jet):
    lay, dims = _setup(jet)
    lib = jet.library()
    assert jet.jet_w4_bytes(300, 208) == 3 * 2 * 8704
    assert jet.jet_w4_bytes(128, 128) == 8704
    assert jet.jet_w4_bytes(0, 128) == 0 and jet.jet_w4_bytes(10, 24) == 0
    # quantiser: rows, shape, null and alignment
    assert lib.jet_quantize_w4(FAKE, 0, 64, FAKE, FAKE, None) == 1
    assert lib.jet_quantize_w4(FAKE, 4, 24, FAKE, FAKE, None) == 2     # D % 16 != 0
    assert lib.jet_quantize_w4(None, 4, 64, FAKE, FAKE, None) == 1
    assert lib.jet_quantize_w4(FAKE, 4, 64, MIS, FAKE, None) == 4
    # scoring: float32 dims have no 4-bit path; workspace and alignment checks
    L = ctypes.byref(lay.struct)
    f32 = jet.make_dims(jet.DTYPE_F32, D=64)
    args = [FAKE] * 6
    assert lib.jet_score_candidates_w4(L, ctypes.byref(f32), *args, 1 << 30, None) == 7
    bf = jet.make_dims(jet.DTYPE_BF16, D=64)
    assert lib.jet_score_candidates_w4(L, ctypes.byref(bf), *args, 16, None) == 5
    mis = list(args)
    mis[1] = MIS   # w4
    assert lib.jet_score_candidates_w4(L, ctypes.byref(bf), *mis, 1 << 30, None) == 4


def test_stack_validation(jet):
    lay, dims = _setup(jet)   # Hq 8, Hkv 2, d 64, D 64, Hl 2, dk 128, dv 64
    lib = jet.library()
    L = ctypes.byref(lay.struct)
    ws = jet.jet_stack_workspace_bytes(lay.sizes, dims, 128)
    assert ws > 0 and jet.jet_stack_workspace_bytes(lay.sizes, dims, 100) == 0
    full = dict(kind="full", **{n: FAKE for n in ("g1", "g2", "w_mix", "w_o", "w_gu", "w_d",
                                                  "k_pre", "v_pre")})
    lin = dict(kind="linear", **{n: FAKE for n in ("g1", "g2", "w_mix", "w_o", "w_gu", "w_d",
                                                   "s_prefix")})

    def call(layers, Dff=128, rule=0, d=dims, ws_bytes=ws):
        arr = [dict(L2, kind=jet.LAYER_FULL if L2["kind"] == "full" else
                    (jet.LAYER_LINEAR if L2["kind"] == "linear" else L2["kind"]))
               for L2 in layers]
        st, keep = jet.make_stack(arr, Dff, rule)
        return lib.jet_stack_forward(L, ctypes.byref(d), ctypes.byref(st), FAKE, FAKE, FAKE,
                                     ws_bytes, None)

    assert call([full, lin], ws_bytes=16) == 5                        # workspace
    assert call([full, lin], Dff=96) == 2                             # Dff % 64 != 0
    assert call([full], rule=9) == 1                                  # unknown rule
    assert call([dict(full, kind=7)]) == 1                            # unknown kind
    assert call([dict(lin, s_prefix=None)]) == 1                      # null state
    assert call([dict(full, w_gu=MIS)]) == 4                          # misaligned weight
    odd = jet.make_dims(jet.DTYPE_BF16, Hq=8, Hkv=2, d=64, D=64, Hl=3, dk=128, dv=64)
    assert call([lin], d=odd) == 7                                    # Hl odd
    f32 = jet.make_dims(jet.DTYPE_F32, Hq=8, Hkv=2, d=64, D=64, Hl=2, dk=128, dv=64)
    assert call([full], d=f32) == 7                                   # bf16 only
    assert call([]) == 0                                              # no layers: a copy


def test_e4m3_validation(jet):
    lay, dims = _setup(jet)
    lib = jet.library()
    ws = jet.jet_workspace_bytes_e4m3(lay.sizes, dims)
    assert ws > jet.jet_workspace_bytes(lay.sizes, jet.make_dims(jet.DTYPE_BF16, D=64)) - 1
    # quantiser: shape, rows, null and alignment
    assert lib.jet_quantize_rows_e4m3(FAKE, 4, 24, FAKE, FAKE, None) == 2   # D % 16 != 0
    assert lib.jet_quantize_rows_e4m3(FAKE, -1, 64, FAKE, FAKE, None) == 1
    assert lib.jet_quantize_rows_e4m3(None, 4, 64, FAKE, FAKE, None) == 1
    assert lib.jet_quantize_rows_e4m3(FAKE, 4, 64, MIS, FAKE, None) == 4
    assert lib.jet_quantize_rows_e4m3(FAKE, 0, 64, None, None, None) == 0  # nothing to do
    # scoring: the e4m3 head takes bf16 hidden states and D % 16 == 0
    f32 = jet.make_dims(jet.DTYPE_F32, D=64)
    args = (FAKE, FAKE, FAKE, FAKE, FAKE, FAKE)
    assert lib.jet_score_candidates_e4m3(ctypes.byref(lay.struct), ctypes.byref(f32), *args,
                                         ws, None) == 7
    bad = jet.make_dims(jet.DTYPE_BF16, D=72)
    assert lib.jet_score_candidates_e4m3(ctypes.byref(lay.struct), ctypes.byref(bad), *args,
                                         ws, None) == 2
    assert lib.jet_score_candidates_e4m3(ctypes.byref(lay.struct), ctypes.byref(dims), *args,
                                         64, None) == 5
    mis = (FAKE, MIS, FAKE, FAKE, FAKE, FAKE)  # w_q
    assert lib.jet_score_candidates_e4m3(ctypes.byref(lay.struct), ctypes.byref(dims), *mis,
                                         ws, None) == 4


def test_empty_batch_is_a_no_op(jet):
    lay = jet.jet_layout_build([], [], [], [], 16)
    assert lay.sizes.R == 0 and lay.sizes.N == 0
    dims = jet.make_dims(jet.DTYPE_BF16, Hq=8, Hkv=2, d=64, D=64, Hl=2, dk=128, dv=64)
    lib = jet.library()
    assert lib.jet_prefix_attend(ctypes.byref(lay.struct), ctypes.byref(dims), *([None] * 7), 0,
                                 None) == 0
    assert lib.jet_score_candidates(ctypes.byref(lay.struct), ctypes.byref(dims), *([None] * 5), 0,
                                    None) == 0
    assert lib.jet_decide(ctypes.byref(lay.struct), 0, None, None, None, None, None) == 0
    assert lib.jet_fork_state(ctypes.byref(lay.struct), ctypes.byref(dims), *([None] * 9)) == 0


def test_status_strings(jet):
    lib = jet.library()
    for s in range(11):
        assert lib.jet_status_string(s)
    assert lib.jet_status_string(99) == b"unknown status"
