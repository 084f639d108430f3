"""Pins of the hybrid decoder-stack oracle: the bf16 rounding and the small
functions against their definitions, and the whole stack against an
independent token-by-token decoder (one candidate's tokens fed one at a time
with a growing key/value cache and a stepped recurrent state), which teacher
forcing must reproduce; plus candidate isolation and the shared row's
independence from the candidates."""
import math

import numpy as np

import oracle as O
from oracle import stack as S

DIMS = dict(Hq=4, Hkv=2, d=16, Hl=2, dk=16, dv=8, Dff=128)
D = 64


def test_bf16_rounding_table():
    cases = [(1.0 + 2.0 ** -8, 1.0),              # halfway: the even neighbour
             (1.0 + 3 * 2.0 ** -8, 1.0 + 2.0 ** -6),  # halfway above an odd mantissa: up
             (1.0 + 2.0 ** -8 + 2.0 ** -20, 1.0 + 2.0 ** -7),
             (-3.0, -3.0), (0.0, 0.0), (2.0 ** -126, 2.0 ** -126),
             (2.0 ** -133, 2.0 ** -133), (2.0 ** -140, 0.0)]  # bf16 subnormals end at 2^-133
    for x, want in cases:
        assert S.bf16(x) == want, (x, S.bf16(x), want)
    assert np.signbit(S.bf16(-0.0))


def test_rmsnorm_sigmoid_silu():
    x = np.array([[3.0, 4.0]])
    np.testing.assert_allclose(S.rmsnorm(x, [1.0, 2.0], eps=0.0),
                               [[3 / math.sqrt(12.5), 8 / math.sqrt(12.5)]], rtol=1e-15)
    # scale invariance without eps; a constant row maps to the gains
    rng = np.random.default_rng(1)
    y = rng.standard_normal((3, 10))
    np.testing.assert_allclose(S.rmsnorm(7.5 * y, 1.0, eps=0.0), S.rmsnorm(y, 1.0, eps=0.0),
                               rtol=1e-13)
    np.testing.assert_allclose(S.rmsnorm(np.full((1, 5), -2.0), np.arange(5.0), eps=0.0),
                               -np.arange(5.0)[None], rtol=1e-15)
    assert S.sigmoid(0.0) == 0.5 and S.silu(0.0) == 0.0
    z = rng.standard_normal(20)
    np.testing.assert_allclose(S.silu(z) - S.silu(-z), z, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(S.sigmoid(z) + S.sigmoid(-z), 1.0, rtol=1e-15)


def _params(rng, kinds, total_prefix, R):
    out = []
    Hq, Hkv, d, Hl, dk, dv, Dff = (DIMS[k] for k in ("Hq", "Hkv", "d", "Hl", "dk", "dv", "Dff"))
    for kind in kinds:
        P = dict(g1=S.bf16(1 + 0.1 * rng.standard_normal(D)),
                 g2=S.bf16(1 + 0.1 * rng.standard_normal(D)),
                 w_gu=S.bf16(rng.standard_normal((2 * Dff, D)) / math.sqrt(D)),
                 w_d=S.bf16(rng.standard_normal((D, Dff)) / math.sqrt(Dff)))
        if kind == "full":
            P["w_mix"] = S.bf16(rng.standard_normal(((Hq + 2 * Hkv) * d, D)) / math.sqrt(D))
            P["w_o"] = S.bf16(rng.standard_normal((D, Hq * d)) / math.sqrt(Hq * d))
            P["k_pre"] = S.bf16(rng.standard_normal((total_prefix, Hkv, d)))
            P["v_pre"] = S.bf16(rng.standard_normal((total_prefix, Hkv, d)))
        else:
            P["w_mix"] = S.bf16(rng.standard_normal((Hl * (2 * dk + dv) + 2 * Hl, D)) /
                                math.sqrt(D))
            P["w_o"] = S.bf16(rng.standard_normal((D, Hl * dv)) / math.sqrt(Hl * dv))
            P["s_prefix"] = rng.standard_normal((R, Hl, dk, dv)) / math.sqrt(dk)
        out.append(P)
    return out


KINDS = ("linear", "full", "linear")


def _decode_one(x_rows, P_list, r, p0, P_len):
    """Independent token-by-token decoder for request r's rows x_rows (the
    shared row first, then one candidate's fed tokens in order)."""
    Hq, Hkv, d, Hl, dk, dv, Dff = (DIMS[k] for k in ("Hq", "Hkv", "d", "Hl", "dk", "dv", "Dff"))
    g = Hq // Hkv
    x = np.array(x_rows, dtype=np.float64)
    for kind, P in zip(KINDS, P_list):
        out = np.empty_like(x)
        if kind == "full":
            K = [P["k_pre"][p0 + j] for j in range(P_len)]  # the cache, incl. the shared row
            V = [P["v_pre"][p0 + j] for j in range(P_len)]
        else:
            St = P["s_prefix"][r].copy()
        for t in range(x.shape[0]):
            h = S.bf16(S.rmsnorm(x[t], P["g1"]))
            z = S.bf16(P["w_mix"] @ h)
            if kind == "full":
                q = z[:Hq * d].reshape(Hq, d)
                if t > 0:  # a fed token appends its own key and value
                    K.append(z[Hq * d:(Hq + Hkv) * d].reshape(Hkv, d))
                    V.append(z[(Hq + Hkv) * d:].reshape(Hkv, d))
                o = np.zeros((Hq, d))
                for hh in range(Hq):
                    kk = np.array([k[hh // g] for k in K])
                    vv = np.array([v[hh // g] for v in V])
                    sc = kk @ q[hh] / math.sqrt(d)
                    p = np.exp(sc - sc.max())
                    o[hh] = p @ vv / p.sum()
                o = S.bf16(o).reshape(-1)
            else:
                lq = z[:Hl * dk].reshape(Hl, dk)
                kr = z[Hl * dk:2 * Hl * dk].reshape(Hl, dk)
                lk = S.bf16(kr / np.linalg.norm(kr, axis=-1, keepdims=True))
                lv = z[2 * Hl * dk:Hl * (2 * dk + dv)].reshape(Hl, dv)
                al = S.sigmoid(z[Hl * (2 * dk + dv):Hl * (2 * dk + dv) + Hl])
                be = S.sigmoid(z[Hl * (2 * dk + dv) + Hl:])
                o = np.zeros((Hl, dv))
                for hh in range(Hl):
                    if t > 0:  # the shared row only reads the prefix state
                        St[hh], _ = O.gated_delta_step(St[hh], lq[hh], lk[hh], lv[hh], al[hh],
                                                       be[hh])
                    o[hh] = St[hh].T @ lq[hh] / math.sqrt(dk)
                o = S.bf16(o).reshape(-1)
            x1 = S.bf16(x[t] + P["w_o"] @ o)
            h2 = S.bf16(S.rmsnorm(x1, P["g2"]))
            f = np.arange(Dff)
            gr = 128 * (f // 64) + f % 64
            u = S.bf16(S.silu(P["w_gu"][gr] @ h2) * (P["w_gu"][gr + 64] @ h2))
            out[t] = S.bf16(x1 + P["w_d"] @ u)
        x = out
    return x


def _problem(rng):
    prefix_len, n_cand, cand_len = [5, 3], [2, 3], [3, 1, 2, 4, 2]
    ids = list(range(sum(cand_len)))
    lay = O.build_layout(prefix_len, n_cand, cand_len, ids, 50)
    params = _params(rng, KINDS, sum(prefix_len), len(prefix_len))
    x0 = S.bf16(rng.standard_normal((lay["N"], D)))
    return lay, params, x0, prefix_len, n_cand, cand_len


def test_teacher_forcing_equals_token_by_token_decoding():
    rng = np.random.default_rng(7)
    lay, params, x0, prefix_len, n_cand, cand_len = _problem(rng)
    got = S.stack_forward(lay, x0, KINDS, params, DIMS)
    p0 = 0
    c = 0
    for r in range(len(prefix_len)):
        row0 = int(lay["row_offset"][r])
        for _ in range(n_cand[r]):
            c0 = int(lay["cand_row_offset"][c])
            m = cand_len[c]
            rows = [row0] + list(range(c0, c0 + m - 1))
            want = _decode_one(x0[rows], params, r, p0, prefix_len[r])
            np.testing.assert_allclose(got[rows], want, rtol=0, atol=1e-9)
            c += 1
        p0 += prefix_len[r]


def test_candidate_isolation_and_shared_row():
    # dropping request 0's first candidate changes no other row's output
    rng = np.random.default_rng(8)
    lay, params, x0, prefix_len, n_cand, cand_len = _problem(rng)
    full = S.stack_forward(lay, x0, KINDS, params, DIMS)
    lay2 = O.build_layout(prefix_len, [1, 3], cand_len[1:], list(range(sum(cand_len[1:]))), 50)
    c0 = int(lay["cand_row_offset"][0])
    keep = [n for n in range(lay["N"]) if not (c0 <= n < c0 + cand_len[0] - 1)]
    part = S.stack_forward(lay2, x0[keep], KINDS, params, DIMS)
    np.testing.assert_array_equal(part, full[keep])
    # the shared rows depend on nothing but their own input and the caches
    x1 = x0.copy()
    x1[[n for n in range(lay["N"]) if n not in (0, int(lay["row_offset"][1]))]] += 1.0
    other = S.stack_forward(lay, x1, KINDS, params, DIMS)
    for r in range(2):
        n = int(lay["row_offset"][r])
        np.testing.assert_array_equal(other[n], full[n])
