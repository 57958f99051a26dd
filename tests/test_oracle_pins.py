"""Pins of the fp64 oracle against facts fixed by the paper and by mathematics.

Each test checks the oracle against something other than itself: hand-derived
examples (tests/golden), closed forms, an independent formulation (complex
rotation, a library softmax, exact rational arithmetic), invariants the method
states (§4.1-§4.2, Eqs. 2-3) or brute force on tiny inputs.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
from scipy.special import softmax

from oracle import kvm_oracle as O

GOLD = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(1234)


def _gold(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def _unit(x):
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


# ---------------------------------------------------------------- input widening
@pytest.mark.parametrize("bits,value", [
    (0x3F80, 1.0), (0xC040, -3.0), (0x0000, 0.0), (0x4049, 3.140625), (0x3F81, 1.0 + 2.0 ** -7),
    (0xBF00, -0.5), (0x7F7F, (2.0 - 2.0 ** -7) * 2.0 ** 127), (0x0080, 2.0 ** -126), (0x0001, 2.0 ** -133),
    (0x7F80, math.inf), (0xFF80, -math.inf)])
def test_bf16_widening_on_fixed_bit_patterns(bits, value):
    """bf16 = sign | 8 exponent bits (bias 127) | 7 fraction bits: each bit
    pattern's value written out by hand, including a subnormal and the
    infinities."""
    got = O.bf16_to_f64(np.array([bits], dtype=np.uint16))[0]
    assert got == value
    assert got.dtype == np.float64 if hasattr(got, "dtype") else True


def test_bf16_widening_sign_of_zero_and_nan():
    z = O.bf16_to_f64(np.array([0x8000], dtype=np.uint16))[0]
    assert z == 0.0 and math.copysign(1.0, z) == -1.0
    assert math.isnan(O.bf16_to_f64(np.array([0x7FC0], dtype=np.uint16))[0])


# ---------------------------------------------------------------- golden
def test_golden_gdn_hand_example():
    g = _gold("gdn_hand_2d.json")
    q = np.array(g["q"])[:, None, :]
    k = np.array(g["k"])[:, None, :]
    v = np.array(g["v"])[:, None, :]
    a = np.array(g["alpha"])[:, None]
    b = np.array(g["beta"])[:, None]
    S0 = np.array(g["S0"])[None]
    o, S = O.gdn_recurrent(q, k, v, a, b, S0)
    np.testing.assert_allclose(o[:, 0], g["o"], atol=1e-12)
    np.testing.assert_allclose(S[0], g["S"], atol=1e-12)


def test_golden_attention_hand_example():
    g = _gold("attn_hand.json")
    cache = O.AttnCache(np.array(g["cache_k"]), np.array(g["cache_v"]), np.array(g["cache_pos"]))
    out, new = O.tail_attn_prefill(cache, np.array(g["q"]), np.array(g["k_new"]),
                                   np.array(g["v_new"]), g["cursor"], 0, 1e4)
    np.testing.assert_allclose(out, g["out"], atol=1e-12)
    assert list(new.pos) == [0, g["cursor"]]


def test_golden_rope_hand_example():
    g = _gold("rope_hand.json")
    x = np.array(g["x"], dtype=np.float64)[:, None, :]
    pos = np.full(x.shape[0], g["pos"])
    out = O.rope(x, pos, g["R"], g["theta"])
    np.testing.assert_allclose(out[:, 0], g["out"], atol=1e-12)


# ---------------------------------------------------------------- RoPE
def test_rope_matches_complex_rotation():
    """RoFormer's complex form: z_d = x_d + i x_{d+R/2} times exp(i pos w_d)."""
    D, R, theta = 16, 8, 1e4
    x = rng.standard_normal((5, 3, D))
    pos = np.array([0, 1, 17, 4096, 479547])
    out = O.rope(x, pos, R, theta)
    h = R // 2
    for n in range(5):
        for d in range(h):
            w = theta ** (-(2 * d) / R)
            z = complex(x[n, 0, d], x[n, 0, d + h]) * complex(math.cos(pos[n] * w), math.sin(pos[n] * w))
            assert abs(out[n, 0, d] - z.real) < 1e-9
            assert abs(out[n, 0, d + h] - z.imag) < 1e-9
    np.testing.assert_array_equal(out[:, :, R:], x[:, :, R:])


def test_rope_relative_position_and_norm():
    D, R, theta = 64, 64, 1e4
    q = rng.standard_normal((1, 1, D))
    k = rng.standard_normal((1, 1, D))
    for m, n, delta in [(10, 3, 1000), (5, 5, 123456), (0, 40, 400000)]:
        a = O.rope(q, [m], R, theta)[0, 0] @ O.rope(k, [n], R, theta)[0, 0]
        b = O.rope(q, [m + delta], R, theta)[0, 0] @ O.rope(k, [n + delta], R, theta)[0, 0]
        assert abs(a - b) < 1e-8 * max(1.0, abs(a))
    r = O.rope(q, [479547], R, theta)
    assert abs(np.linalg.norm(r) - np.linalg.norm(q)) < 1e-12
    np.testing.assert_array_equal(O.rope(q, [0], R, theta), q)


def test_rope_frequency_values():
    w = O.rope_frequencies(64, 1e4)
    assert w[0] == 1.0
    assert abs(w[1] - 10 ** (-0.125)) < 1e-15
    assert abs(w[31] - 1e4 ** (-62 / 64)) < 1e-18


# ---------------------------------------------------------------- attention
def test_attention_single_key_returns_value():
    cache = O.AttnCache(np.zeros((2, 0, 8)), np.zeros((2, 0, 8)), np.zeros(0))
    q = rng.standard_normal((1, 4, 8))
    k = rng.standard_normal((1, 2, 8))
    v = rng.standard_normal((1, 2, 8))
    out, _ = O.tail_attn_prefill(cache, q, k, v, 7, 8, 1e4)
    for h in range(4):
        np.testing.assert_allclose(out[0, h], v[0, h // 2], atol=1e-14)


def test_attention_constant_values_weights_sum_to_one():
    L, M, D = 9, 3, 8
    cache = O.AttnCache(rng.standard_normal((1, L, D)), np.ones((1, L, D)) * 2.5, np.arange(L))
    out, _ = O.tail_attn_prefill(cache, rng.standard_normal((M, 2, D)), rng.standard_normal((M, 1, D)),
                                 np.ones((M, 1, D)) * 2.5, L, 4, 1e4)
    np.testing.assert_allclose(out, 2.5, atol=1e-13)


def _masked_reference(cache_full, keep, q, k_new, v_new, p, R, theta):
    """Library softmax over the UNcompacted cache with removed keys at -inf."""
    M, Hq, D = q.shape
    Hkv = cache_full.K.shape[0]
    g = Hq // Hkv
    pos_new = p + np.arange(M)
    qr = O.rope(q, pos_new, R, theta)
    kr = O.rope(k_new, pos_new, R, theta)
    out = np.zeros_like(qr)
    L = cache_full.K.shape[1]
    for i in range(M):
        for h in range(Hq):
            keys = np.concatenate([cache_full.K[h // g], kr[:, h // g]])
            vals = np.concatenate([cache_full.V[h // g], v_new[:, h // g]])
            allow = np.concatenate([keep, np.arange(M) <= i])
            s = np.where(allow, keys @ qr[i, h] / math.sqrt(D), -np.inf)
            out[i, h] = softmax(s) @ vals
    return out


def test_removed_equals_masked():
    """Eq. 2: attention over the compacted cache equals attention over the
    full cache with the removed entries masked out."""
    L, M, D, Hq, Hkv, R = 40, 5, 16, 4, 2, 8
    full = O.AttnCache(rng.standard_normal((Hkv, L, D)), rng.standard_normal((Hkv, L, D)), np.arange(L))
    begins, ends = [3, 20], [7, 31]
    K, V, pos, _ = O.kv_compact(full.K, full.V, full.pos, begins, ends)
    q = rng.standard_normal((M, Hq, D))
    kn = rng.standard_normal((M, Hkv, D))
    vn = rng.standard_normal((M, Hkv, D))
    out, _ = O.tail_attn_prefill(O.AttnCache(K, V, pos), q, kn, vn, 50, R, 1e4)
    ref = _masked_reference(full, O.keep_mask(L, begins, ends), q, kn, vn, 50, R, 1e4)
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_gqa_equals_mha_with_replicated_kv():
    L, M, D, Hq, Hkv, R = 12, 4, 8, 4, 2, 8
    K = rng.standard_normal((Hkv, L, D))
    V = rng.standard_normal((Hkv, L, D))
    q = rng.standard_normal((M, Hq, D))
    kn = rng.standard_normal((M, Hkv, D))
    vn = rng.standard_normal((M, Hkv, D))
    out, _ = O.tail_attn_prefill(O.AttnCache(K, V, np.arange(L)), q, kn, vn, L, R, 1e4)
    rep = [0, 0, 1, 1]
    out2, _ = O.tail_attn_prefill(O.AttnCache(K[rep], V[rep], np.arange(L)), q, kn[:, rep], vn[:, rep],
                                  L, R, 1e4)
    np.testing.assert_allclose(out, out2, atol=1e-13)


def test_attention_brute_force_tiny():
    """Scalar brute force: complex-form rotation and an explicit softmax."""
    D, R, theta, L, M = 4, 2, 10.0, 3, 2
    Kc = rng.standard_normal((1, L, D))
    Vc = rng.standard_normal((1, L, D))
    q = rng.standard_normal((M, 1, D))
    kn = rng.standard_normal((M, 1, D))
    vn = rng.standard_normal((M, 1, D))
    p = 11
    out, _ = O.tail_attn_prefill(O.AttnCache(Kc, Vc, np.arange(L)), q, kn, vn, p, R, theta)

    def rot(x, pos):
        z = complex(x[0], x[1]) * complex(math.cos(pos), math.sin(pos))   # R = 2: w_0 = 1
        return [z.real, z.imag, x[2], x[3]]

    for i in range(M):
        qi = rot(q[i, 0], p + i)
        keys = [list(Kc[0, j]) for j in range(L)] + [rot(kn[j, 0], p + j) for j in range(i + 1)]
        vals = [list(Vc[0, j]) for j in range(L)] + [list(vn[j, 0]) for j in range(i + 1)]
        sc = [sum(a * b for a, b in zip(qi, kk)) / 2.0 for kk in keys]
        ws = [math.exp(s) for s in sc]
        tot = sum(ws)
        for d in range(D):
            ref = sum(w * vv[d] for w, vv in zip(ws, vals)) / tot
            assert abs(out[i, 0, d] - ref) < 1e-12


def test_attention_relative_shift_invariance():
    """Shifting every position by the same amount leaves the outputs alone."""
    D, R, Hq, Hkv = 16, 16, 2, 1
    toks = {"q": rng.standard_normal((10, Hq, D)), "k": rng.standard_normal((10, Hkv, D)),
            "v": rng.standard_normal((10, Hkv, D))}
    empty = O.AttnCache(np.zeros((Hkv, 0, D)), np.zeros((Hkv, 0, D)), np.zeros(0))
    a, _ = O.tail_attn_prefill(empty, toks["q"], toks["k"], toks["v"], 0, R, 1e4)
    b, cb = O.tail_attn_prefill(empty, toks["q"], toks["k"], toks["v"], 250000, R, 1e4)
    np.testing.assert_allclose(a, b, atol=1e-9)
    assert list(cb.pos) == list(range(250000, 250010))


# ---------------------------------------------------------------- delta rule
def _gdn_inputs(M, H, dk, dv, unit=True):
    k = rng.standard_normal((M, H, dk))
    if unit:
        k = _unit(k)
    return (rng.standard_normal((M, H, dk)), k, rng.standard_normal((M, H, dv)),
            1 / (1 + np.exp(-rng.normal(3, 0.5, (M, H)))), 1 / (1 + np.exp(-rng.standard_normal((M, H)))),
            rng.standard_normal((H, dv, dk)) * 0.2)


def test_gdn_identity_gates_keep_state():
    q, k, v, a, b, S0 = _gdn_inputs(7, 2, 4, 3)
    o, S = O.gdn_recurrent(q, k, v, np.ones_like(a), np.zeros_like(b), S0)
    np.testing.assert_allclose(S, S0, atol=1e-15)
    np.testing.assert_allclose(o, np.einsum("hvk,thk->thv", S0, q), atol=1e-13)


def test_gdn_unit_key_recall():
    """alpha = beta = 1 and |k| = 1: the delta rule stores v exactly, S_t k_t = v_t."""
    q, k, v, a, b, S0 = _gdn_inputs(6, 3, 8, 5)
    M = k.shape[0]
    for t in range(1, M + 1):
        _, S = O.gdn_recurrent(q[:t], k[:t], v[:t], np.ones_like(a[:t]), np.ones_like(b[:t]), S0)
        for h in range(3):
            np.testing.assert_allclose(S[h] @ k[t - 1, h], v[t - 1, h], atol=1e-12)


def test_gdn_general_key_identity():
    """S_t k_t = alpha (1 - beta |k|^2) S_{t-1} k_t + beta |k|^2 v_t for any k."""
    q, k, v, a, b, S0 = _gdn_inputs(5, 2, 6, 4, unit=False)
    Sp = S0
    for t in range(5):
        _, S = O.gdn_recurrent(q[t:t + 1], k[t:t + 1], v[t:t + 1], a[t:t + 1], b[t:t + 1], Sp)
        for h in range(2):
            kk = k[t, h] @ k[t, h]
            ref = a[t, h] * (1 - b[t, h] * kk) * (Sp[h] @ k[t, h]) + b[t, h] * kk * v[t, h]
            np.testing.assert_allclose(S[h] @ k[t, h], ref, atol=1e-11)
        Sp = S


def test_gdn_orthonormal_keys_closed_form():
    """Orthonormal keys never interfere: S_n = sum_j (prod_{u>j} alpha_u) beta_j v_j k_j^T."""
    d = 6
    Qm, _ = np.linalg.qr(rng.standard_normal((d, d)))
    k = Qm.T[:, None, :]                       # d tokens, 1 head
    v = rng.standard_normal((d, 1, 3))
    a = rng.uniform(0.5, 1.0, (d, 1))
    b = rng.uniform(0.1, 1.0, (d, 1))
    _, S = O.gdn_recurrent(rng.standard_normal((d, 1, d)), k, v, a, b, np.zeros((1, 3, d)))
    ref = np.zeros((3, d))
    for j in range(d):
        ref += np.prod(a[j + 1:, 0]) * b[j, 0] * np.outer(v[j, 0], k[j, 0])
    np.testing.assert_allclose(S[0], ref, atol=1e-13)


def test_gdn_exact_rational_brute_force():
    """Exact rational arithmetic (fractions) on a tiny 2x2 case, three tokens."""
    toks = [((Fraction(1, 2), Fraction(1, 3)), (Fraction(3, 5), Fraction(4, 5)), (Fraction(1), Fraction(-2)),
             Fraction(7, 8), Fraction(1, 4)),
            ((Fraction(-1), Fraction(2)), (Fraction(1), Fraction(0)), (Fraction(1, 3), Fraction(1, 2)),
             Fraction(3, 4), Fraction(2, 3)),
            ((Fraction(2), Fraction(1)), (Fraction(5, 13), Fraction(12, 13)), (Fraction(-3, 2), Fraction(1)),
             Fraction(9, 10), Fraction(1, 2))]
    S = [[Fraction(1, 5), Fraction(-1, 2)], [Fraction(1, 3), Fraction(1)]]
    S0 = np.array([[float(x) for x in r] for r in S])[None]
    outs = []
    for q, k, v, al, be in toks:
        # S <- al*S*(I - be k k^T) + be v k^T, written entrywise
        P = [[(1 if i == j else 0) - be * k[i] * k[j] for j in range(2)] for i in range(2)]
        S = [[al * sum(S[r][m] * P[m][c] for m in range(2)) + be * v[r] * k[c] for c in range(2)]
             for r in range(2)]
        outs.append([sum(S[r][c] * q[c] for c in range(2)) for r in range(2)])
    f = lambda i: np.array([[float(x) for x in t[i]] for t in toks])[:, None, :]
    o, Sn = O.gdn_recurrent(f(0), f(1), f(2), np.array([[float(t[3])] for t in toks]),
                            np.array([[float(t[4])] for t in toks]), S0)
    np.testing.assert_allclose(o[:, 0], [[float(x) for x in r] for r in outs], atol=1e-14)
    np.testing.assert_allclose(Sn[0], [[float(x) for x in r] for r in S], atol=1e-14)


@pytest.mark.parametrize("M,C", [(150, 64), (64, 64), (1, 64), (37, 16), (200, 32)])
def test_gdn_chunked_equals_recurrent(M, C):
    q, k, v, a, b, S0 = _gdn_inputs(M, 3, 16, 12)
    o1, S1 = O.gdn_recurrent(q, k, v, a, b, S0)
    o2, S2 = O.gdn_chunked(q, k, v, a, b, S0, C)
    np.testing.assert_allclose(o2, o1, atol=1e-11, rtol=1e-11)
    np.testing.assert_allclose(S2, S1, atol=1e-11, rtol=1e-11)


def test_gdn_resume_equals_uninterrupted():
    """Continuing from a carried state equals running the whole sequence."""
    q, k, v, a, b, S0 = _gdn_inputs(30, 2, 8, 8)
    o, S = O.gdn_recurrent(q, k, v, a, b, S0)
    o1, Sm = O.gdn_recurrent(q[:13], k[:13], v[:13], a[:13], b[:13], S0)
    o2, S2 = O.gdn_recurrent(q[13:], k[13:], v[13:], a[13:], b[13:], Sm)
    np.testing.assert_allclose(np.concatenate([o1, o2]), o, atol=1e-13)
    np.testing.assert_allclose(S2, S, atol=1e-13)


# ---------------------------------------------------------------- compaction
def test_compact_counts_positions_order():
    L = 100
    K = rng.standard_normal((2, L, 4))
    pos = np.arange(L) * 3 + 7
    begins, ends = [0, 10, 50, 99], [2, 20, 51, 100]
    K2, V2, p2, gather = O.kv_compact(K, K.copy(), pos, begins, ends)
    assert K2.shape[1] == L - (2 + 10 + 1 + 1)
    assert np.all(np.diff(p2) > 0)
    np.testing.assert_array_equal(K2, K[:, gather])
    removed = set().union(*[set(range(b, e)) for b, e in zip(begins, ends)])
    assert list(gather) == [i for i in range(L) if i not in removed]


def test_compact_identity_and_composition():
    L = 60
    K = rng.standard_normal((1, L, 2))
    pos = np.arange(L)
    K1, _, p1, g1 = O.kv_compact(K, K, pos, [], [])
    np.testing.assert_array_equal(K1, K)
    np.testing.assert_array_equal(g1, np.arange(L))
    # two compactions in sequence == one compaction with the union of spans
    Ka, _, pa, ga = O.kv_compact(K, K, pos, [5, 30], [10, 33])        # 52 left
    Kb, _, pb, gb = O.kv_compact(Ka, Ka, pa, [0, 40], [3, 52])
    Ku, _, pu, gu = O.kv_compact(K, K, pos, [0, 5, 30, 48], [3, 10, 33, 60])
    np.testing.assert_array_equal(Kb, Ku)
    np.testing.assert_array_equal(pb, pu)
    np.testing.assert_array_equal(ga[gb], gu)


@pytest.mark.parametrize("begins,ends", [([5, 3], [6, 4]), ([2, 4], [5, 7]), ([3], [3]), ([-1], [2]),
                                         ([8], [11]), ([1, 2], [2])])
def test_span_validation_rejects(begins, ends):
    with pytest.raises(O.SpanError):
        O.keep_mask(10, begins, ends)


# ---------------------------------------------------------------- whole round
def _stack():
    return dict(layer_kind=[0, 1, 0, 1], Hkv=2, D=16, H=2, dk=8, dv=6, R=8, theta=1e4)


def _tokens(n, st):
    ins = {}
    for l, kind in enumerate(st["layer_kind"]):
        if kind == 1:
            ins[l] = {"q": rng.standard_normal((n, 4, st["D"])), "k": _unit(rng.standard_normal((n, 2, st["D"]))),
                      "v": rng.standard_normal((n, 2, st["D"]))}
        else:
            q, k, v, a, b, _ = _gdn_inputs(n, st["H"], st["dk"], st["dv"])
            ins[l] = {"q": q, "k": k, "v": v, "alpha": a, "beta": b}
    return ins


def _cut(ins, a, b):
    return {l: {k: x[a:b] for k, x in d.items()} for l, d in ins.items()}


def test_zero_removal_tail_update_equals_refill():
    """With nothing removed, causality makes the true-tail update identical to
    a refill of the concatenated sequence (outputs, state, cache)."""
    st = _stack()
    N, M = 23, 9
    ins = _tokens(N + M, st)
    args = (st["Hkv"], st["D"], st["H"], st["dk"], st["dv"], st["R"], st["theta"])
    _, pre = O.refill(st["layer_kind"], _cut(ins, 0, N), *args)
    assert pre.cursor == N
    outs, post = O.maintenance_round(pre, st["layer_kind"], [], [], _cut(ins, N, N + M), st["R"], st["theta"])
    ref_outs, ref = O.refill(st["layer_kind"], ins, *args)
    for l in outs:
        np.testing.assert_allclose(outs[l], ref_outs[l][N:], atol=1e-12)
    for l in post.states:
        np.testing.assert_allclose(post.states[l], ref.states[l], atol=1e-12)
    for l in post.caches:
        np.testing.assert_allclose(post.caches[l].K, ref.caches[l].K, atol=1e-12)
        np.testing.assert_array_equal(post.caches[l].pos, ref.caches[l].pos)
    assert post.cursor == ref.cursor == N + M


def test_removal_leaves_recurrent_state_and_cursor_alone():
    """§4.1: removal does not roll back R; §4.2: holes, cursor keeps moving."""
    st = _stack()
    N, M = 30, 6
    ins = _tokens(N + M, st)
    args = (st["Hkv"], st["D"], st["H"], st["dk"], st["dv"], st["R"], st["theta"])
    _, pre = O.refill(st["layer_kind"], _cut(ins, 0, N), *args)
    tail = _cut(ins, N, N + M)
    o_a, a = O.maintenance_round(pre, st["layer_kind"], [4, 12], [9, 20], tail, st["R"], st["theta"])
    o_b, b = O.maintenance_round(pre, st["layer_kind"], [], [], tail, st["R"], st["theta"])
    for l in a.states:
        np.testing.assert_array_equal(a.states[l], b.states[l])
        np.testing.assert_array_equal(o_a[l], o_b[l])
    assert a.cursor == b.cursor == N + M
    for l in a.caches:
        c = a.caches[l]
        assert c.live == N - 13 + M
        assert list(c.pos[-M:]) == list(range(N, N + M))
        assert np.all(np.diff(c.pos) > 0)
        # survivors keep their stored (already rotated) keys byte for byte
        keep = O.keep_mask(N, [4, 12], [9, 20])
        np.testing.assert_array_equal(c.K[:, :N - 13], pre.caches[l].K[:, keep])
    # with a removal the result is not a refill of the surviving text (§4.1)
    surv = np.nonzero(O.keep_mask(N, [4, 12], [9, 20]))[0]
    txt = {l: {k: np.concatenate([x[:N][surv], x[N:N + M]]) for k, x in d.items()} for l, d in ins.items()}
    r_outs, r = O.refill(st["layer_kind"], txt, *args)
    assert not np.allclose(r.states[0], a.states[0])
    assert not np.allclose(r_outs[1][-M:], o_a[1])


# ---------------------------------------------------------------- placement variants (§5.2)
def test_rerotation_round_trip_is_identity():
    """Turning stored keys from p to q and back to p gives the keys back."""
    D, R, theta = 16, 8, 1e4
    n = 7
    x = rng.standard_normal((n, 2, D))
    p = rng.integers(0, 500_000, n)
    q = rng.integers(0, 500_000, n)
    cache = O.AttnCache(np.transpose(O.rope(x, p, R, theta), (1, 0, 2)), rng.standard_normal((2, n, D)), p)
    there = O.rerotate_keys(cache, 0, n, q, R, theta)
    back = O.rerotate_keys(there, 0, n, p, R, theta)
    np.testing.assert_allclose(back.K, cache.K, atol=1e-9)
    np.testing.assert_array_equal(back.V, cache.V)
    np.testing.assert_array_equal(back.pos, p)
    assert not np.allclose(there.K, cache.K)


def test_rerotation_equals_rotation_at_the_target_position():
    """A key stored at p, turned to q, equals the raw key rotated at q in
    RoFormer's complex form (an independent statement of the rotation)."""
    D, R, theta = 16, 8, 1e4
    n = 5
    x = rng.standard_normal((n, 2, D))
    p = np.array([3, 90, 1000, 261_955, 479_547])
    q = np.array([10_003, 2, 479_547, 20, 0])
    cache = O.AttnCache(np.transpose(O.rope(x, p, R, theta), (1, 0, 2)), np.zeros((2, n, D)), p)
    moved = O.rerotate_keys(cache, 1, 4, q[1:4], R, theta)
    h = R // 2
    for j in range(1, 4):
        for kv in range(2):
            for d in range(h):
                w = theta ** (-(2 * d) / R)
                z = complex(x[j, kv, d], x[j, kv, d + h]) * complex(math.cos(q[j] * w), math.sin(q[j] * w))
                assert abs(moved.K[kv, j, d] - z.real) < 1e-8
                assert abs(moved.K[kv, j, d + h] - z.imag) < 1e-8
    np.testing.assert_array_equal(moved.K[:, [0, 4]], cache.K[:, [0, 4]])
    assert list(moved.pos) == [3, 2, 479_547, 20, 479_547]


def test_explicit_true_tail_positions_equal_the_default():
    st = _stack()
    N, M = 20, 7
    ins = _tokens(N + M, st)
    args = (st["Hkv"], st["D"], st["H"], st["dk"], st["dv"], st["R"], st["theta"])
    _, pre = O.refill(st["layer_kind"], _cut(ins, 0, N), *args)
    tail = _cut(ins, N, N + M)
    o_a, a = O.maintenance_round(pre, st["layer_kind"], [2], [5], tail, st["R"], st["theta"])
    o_b, b = O.maintenance_round(pre, st["layer_kind"], [2], [5], tail, st["R"], st["theta"],
                                 positions=np.arange(N, N + M))
    for l in o_a:
        np.testing.assert_array_equal(o_a[l], o_b[l])
    for l in a.caches:
        np.testing.assert_array_equal(a.caches[l].K, b.caches[l].K)
        np.testing.assert_array_equal(a.caches[l].pos, b.caches[l].pos)
    assert a.cursor == b.cursor == N + M


def test_gapped_prefill_brute_force():
    """Fresh gapped prefill (§5.2): the text read from an empty state with
    gaps between records' position ids.  Each output row is recomputed with
    scalar loops: keys rotated in the complex form at their ids, causal in
    reading order, softmax by hand."""
    Hq, Hkv, D, R, theta = 4, 2, 8, 8, 1e4
    pos = np.array([0, 1, 2, 10_000, 10_001, 20_000, 20_001, 20_002])
    M = len(pos)
    q = rng.standard_normal((M, Hq, D))
    k = _unit(rng.standard_normal((M, Hkv, D)))
    v = rng.standard_normal((M, Hkv, D))
    empty = O.AttnCache(np.zeros((Hkv, 0, D)), np.zeros((Hkv, 0, D)), np.zeros(0, np.int64))
    out, cache = O.tail_attn_prefill(empty, q, k, v, 0, R, theta, positions=pos)
    h = R // 2

    def rot(x, p):
        y = list(x)
        for d in range(h):
            w = theta ** (-(2 * d) / R)
            z = complex(x[d], x[d + h]) * complex(math.cos(p * w), math.sin(p * w))
            y[d], y[d + h] = z.real, z.imag
        return y

    for i in range(M):
        for hq in range(Hq):
            kv = hq // (Hq // Hkv)
            qi = rot(q[i, hq], pos[i])
            sc = [sum(a * b for a, b in zip(qi, rot(k[j, kv], pos[j]))) / math.sqrt(D) for j in range(i + 1)]
            mx = max(sc)
            w = [math.exp(x - mx) for x in sc]
            ref = [sum(w[j] * v[j, kv, d] for j in range(i + 1)) / sum(w) for d in range(D)]
            np.testing.assert_allclose(out[i, hq], ref, atol=1e-10)
    np.testing.assert_array_equal(cache.pos, pos)


def test_slot_positions_change_attention_but_not_the_recurrence():
    """Slot-preserving placement (§5.2) changes only the rotary ids of the
    replacement: attention outputs differ from the true tail, the recurrent
    layers (which carry no positions) do not; the cursor does not move past
    the largest id used."""
    st = _stack()
    N, M = 30, 6
    ins = _tokens(N + M, st)
    args = (st["Hkv"], st["D"], st["H"], st["dk"], st["dv"], st["R"], st["theta"])
    _, pre = O.refill(st["layer_kind"], _cut(ins, 0, N), *args)
    tail = _cut(ins, N, N + M)
    o_t, t = O.maintenance_round(pre, st["layer_kind"], [10], [16], tail, st["R"], st["theta"])
    o_s, s = O.maintenance_round(pre, st["layer_kind"], [10], [16], tail, st["R"], st["theta"],
                                 positions=np.arange(10, 16))
    for l in t.states:
        np.testing.assert_array_equal(t.states[l], s.states[l])
        np.testing.assert_array_equal(o_t[l], o_s[l])
    for l in t.caches:
        assert not np.allclose(o_t[l], o_s[l])
        assert list(s.caches[l].pos[-M:]) == list(range(10, 16))
    assert t.cursor == N + M and s.cursor == N


def test_relative_shift_invariance_with_explicit_positions():
    """Shifting every id (the cache's rotation and the tail's) by the same
    amount leaves attention outputs unchanged (relative positions only)."""
    Hq, Hkv, D, R, theta = 4, 2, 16, 8, 1e4
    L, M, shift = 9, 5, 123_457
    kraw = _unit(rng.standard_normal((L, Hkv, D)))
    vals = rng.standard_normal((Hkv, L, D))
    cpos = np.array([0, 3, 4, 8, 20, 21, 22, 40, 41])
    tpos = np.array([100, 7, 300, 301, 5])
    q = rng.standard_normal((M, Hq, D))
    k = _unit(rng.standard_normal((M, Hkv, D)))
    v = rng.standard_normal((M, Hkv, D))
    outs = []
    for s in (0, shift):
        cache = O.AttnCache(np.transpose(O.rope(kraw, cpos + s, R, theta), (1, 0, 2)), vals, cpos + s)
        o, _ = O.tail_attn_prefill(cache, q, k, v, 0, R, theta, positions=tpos + s)
        outs.append(o)
    np.testing.assert_allclose(outs[0], outs[1], atol=1e-8)


# ---------------------------------------------------------------- maintenance delimiters (§4.2)
def test_delimiters_leave_no_kv_but_keep_their_effect():
    st = _stack()
    N, M = 25, 10
    ins = _tokens(N + M, st)
    args = (st["Hkv"], st["D"], st["H"], st["dk"], st["dv"], st["R"], st["theta"])
    _, pre = O.refill(st["layer_kind"], _cut(ins, 0, N), *args)
    tail = _cut(ins, N, N + M)
    delim = ([0, 7], [2, 8])                     # tail tokens 0, 1 and 7 are delimiters
    o_d, d = O.maintenance_round(pre, st["layer_kind"], [3], [6], tail, st["R"], st["theta"], delimiters=delim)
    o_k, k = O.maintenance_round(pre, st["layer_kind"], [3], [6], tail, st["R"], st["theta"])
    # the round itself is the same round: every output, every recurrent state
    for l in o_d:
        np.testing.assert_array_equal(o_d[l], o_k[l])
    for l in d.states:
        np.testing.assert_array_equal(d.states[l], k.states[l])
    # their ids stay consumed; their KV are gone and nothing else is
    assert d.cursor == k.cursor == N + M
    keep = np.ones(N - 3 + M, bool)
    keep[[N - 3 + 0, N - 3 + 1, N - 3 + 7]] = False
    for l in d.caches:
        assert d.caches[l].live == N - 3 + M - 3
        np.testing.assert_array_equal(d.caches[l].K, k.caches[l].K[:, keep])
        np.testing.assert_array_equal(d.caches[l].pos, k.caches[l].pos[keep])
        assert N + 0 not in d.caches[l].pos and N + 7 not in d.caches[l].pos
    # their indirect effect remains: without the delimiter tokens the state differs
    plain = {l: {kk: np.delete(x, [0, 1, 7], axis=0) for kk, x in dd.items()} for l, dd in tail.items()}
    _, nd = O.maintenance_round(pre, st["layer_kind"], [3], [6], plain, st["R"], st["theta"])
    assert not np.allclose(nd.states[0], d.states[0])
    # a later round attends over the cache without the delimiters' keys
    nxt = _tokens(3, st)
    o2, _ = O.maintenance_round(d, st["layer_kind"], [], [], nxt, st["R"], st["theta"])
    c = d.caches[1]
    qr = O.rope(nxt[1]["q"], np.arange(N + M, N + M + 3), st["R"], st["theta"])
    kr = O.rope(nxt[1]["k"], np.arange(N + M, N + M + 3), st["R"], st["theta"])
    keys = np.concatenate([c.K[0], kr[:1, 0]])
    vals = np.concatenate([c.V[0], nxt[1]["v"][:1, 0]])
    np.testing.assert_allclose(o2[1][0, 0], O.attend_row(qr[0, 0], keys, vals), atol=1e-12)


# ---------------------------------------------------------------- attention probes (§5.3)
def _probe_cache(L=23, Hkv=2, D=16, R=8, theta=1e4):
    pos = np.sort(rng.choice(np.arange(1000), size=L, replace=False))
    kraw = _unit(rng.standard_normal((L, Hkv, D)))
    K = np.transpose(O.rope(kraw, pos, R, theta), (1, 0, 2))
    return O.AttnCache(K, rng.standard_normal((Hkv, L, D)), pos)


def test_probe_rows_are_the_attention_weights():
    """Each probe row sums to 1 over the keys its query sees, and weighting
    the values by it reproduces the attention output of that query (the
    reference softmax reconstructs the attention)."""
    c = _probe_cache()
    n_q, Hq = 5, 4
    q = rng.standard_normal((n_q, Hq, 16))
    qr = O.rotate_probe_queries(c, q, 8, 1e4)
    d = O.probe_distributions(c, qr)
    np.testing.assert_allclose(d.sum(axis=2), 1.0, atol=1e-12)
    for i in range(n_q):
        lim = c.live - n_q + i + 1
        assert np.all(d[i, :, lim:] == 0)
        for h in range(Hq):
            kv = h // 2
            np.testing.assert_allclose(d[i, h] @ c.V[kv], O.attend_row(qr[i, h], c.K[kv, :lim], c.V[kv, :lim]),
                                       atol=1e-12)
    a = O.attention_probe(c, q, 8, 1e4)
    assert abs(a.sum() - 1.0) < 1e-12


def test_probe_holes_excluded_equals_masking():
    """Probe over the compacted cache = probe over the cache before removal
    with the removed keys' scores at -inf (scipy softmax), renumbered."""
    c = _probe_cache(L=30)
    n_q, Hq = 4, 4
    q = rng.standard_normal((n_q, Hq, 16))
    K, V, pos, gather = O.kv_compact(c.K, c.V, c.pos, [3, 12], [7, 20])
    cc = O.AttnCache(K, V, pos)
    got = O.probe_distributions(cc, O.rotate_probe_queries(cc, q, 8, 1e4))
    qr = O.rope(q, pos[-n_q:], 8, 1e4)
    keep = O.keep_mask(30, [3, 12], [7, 20])
    for i in range(n_q):
        lim_old = gather[cc.live - n_q + i] + 1
        for h in range(Hq):
            sc = c.K[h // 2, :lim_old] @ qr[i, h] / 4.0
            sc = np.where(keep[:lim_old], sc, -np.inf)
            ref = softmax(sc)
            np.testing.assert_allclose(got[i, h, :cc.live - n_q + i + 1], ref[keep[:lim_old]], atol=1e-12)


def test_probe_brute_force_tiny():
    c = _probe_cache(L=6, Hkv=1, D=4, R=4)
    q = rng.standard_normal((2, 2, 4))
    qr = O.rotate_probe_queries(c, q, 4, 1e4)
    got = O.attention_probe(c, q, 4, 1e4)
    acc = [0.0] * 6
    for i in range(2):
        for h in range(2):
            lim = 6 - 2 + i + 1
            sc = [sum(qr[i, h, d] * c.K[0, j, d] for d in range(4)) / 2.0 for j in range(lim)]
            mx = max(sc)
            w = [math.exp(x - mx) for x in sc]
            for j in range(lim):
                acc[j] += w[j] / sum(w) / 4
    np.testing.assert_allclose(got, acc, atol=1e-12)


def test_effective_group_count_closed_forms():
    for n in (1, 2, 7, 34):
        assert abs(O.effective_group_count(np.ones(n)) - n) < 1e-12
        assert abs(O.effective_group_count(np.full(n, 0.37)) - n) < 1e-12      # scale-free
    assert abs(O.effective_group_count([0, 0, 5.0, 0]) - 1.0) < 1e-12
    p = 0.2
    assert abs(O.effective_group_count([p, 1 - p]) - math.exp(-(p * math.log(p) + (1 - p) * math.log(1 - p)))) < 1e-12
    m = O.group_mass([0.1, 0.2, 0.3, 0.4], [0, -1, 0, 2], 3)
    np.testing.assert_allclose(m, [0.4, 0.0, 0.4])


def test_total_variation_is_the_largest_event_difference():
    """TVD = max over events A of |P(A) - Q(A)| (its definition as a
    supremum), checked by enumerating every subset of a small support."""
    import itertools
    for _ in range(20):
        p = rng.random(6)
        p /= p.sum()
        q = rng.random(6)
        q /= q.sum()
        best = max(abs(sum(p[list(A)]) - sum(q[list(A)])) for r in range(7) for A in itertools.combinations(range(6), r))
        assert abs(O.total_variation(p, q) - best) < 1e-12
    assert O.total_variation([1, 0], [0, 1]) == 1.0
    assert O.total_variation([0.3, 0.7], [0.3, 0.7]) == 0.0


# ---------------------------------------------------------------- short convolution (§4.1)
def test_short_conv_from_zero_state_is_numpy_convolution():
    """From a zero state the carried convolution is the causal part of the
    full convolution with the reversed taps (numpy's convolve)."""
    M, C = 11, 5
    x = rng.standard_normal((M, C))
    w = rng.standard_normal((C, 4))
    y, st = O.short_conv(x, np.zeros((3, C)), w)
    for c in range(C):
        np.testing.assert_allclose(y[:, c], np.convolve(x[:, c], w[c, ::-1])[:M], atol=1e-12)
    np.testing.assert_array_equal(st, x[-3:])


def test_short_conv_state_carry_equals_one_pass():
    """Rounds of 5, 1, 2 and 7 tokens, each continuing from the state the
    previous one left, give the convolution of the whole sequence (numpy's
    convolve), and the state is always the last three inputs."""
    C = 4
    x = rng.standard_normal((15, C))
    w = rng.standard_normal((C, 4))
    st = np.zeros((3, C))
    parts, at = [], 0
    for m in (5, 1, 2, 7):
        y, st = O.short_conv(x[at:at + m], st, w)
        parts.append(y)
        at += m
        seen = np.concatenate([np.zeros((3, C)), x[:at]])
        np.testing.assert_array_equal(st, seen[-3:])
    y = np.concatenate(parts)
    for c in range(C):
        np.testing.assert_allclose(y[:, c], np.convolve(x[:, c], w[c, ::-1])[:15], atol=1e-12)


def test_silu_and_identity_taps():
    from scipy.special import expit
    x = rng.standard_normal(50) * 4
    np.testing.assert_allclose(O.silu(x), x * expit(x), atol=1e-12)
    assert O.silu(0.0) == 0.0
    w = np.tile([0.0, 0.0, 0.0, 1.0], (3, 1))            # only the current token
    q = rng.standard_normal((6, 1, 1))
    k = rng.standard_normal((6, 1, 1))
    v = rng.standard_normal((6, 1, 1))
    q2, k2, v2, st = O.gdn_conv_inputs(q, k, v, rng.standard_normal((3, 3)), w)
    np.testing.assert_allclose(q2, O.silu(q), atol=1e-12)
    np.testing.assert_allclose(v2, O.silu(v), atol=1e-12)
    np.testing.assert_allclose(np.abs(k2), 1.0, atol=1e-12)   # d_k = 1: unit norm is +-1
    np.testing.assert_array_equal(st[:, 0], q[-3:, 0, 0])


def test_zero_removal_tail_update_equals_refill_with_conv_state():
    """The refill equivalence (causality) holds with the convolution state
    carried across the round boundary: outputs, S and conv state."""
    st = _stack()
    N, M = 17, 9
    ins = _tokens(N + M, st)
    Cch = st["H"] * (2 * st["dk"] + st["dv"])
    convw = {l: rng.standard_normal((Cch, 4)) * 0.5 for l, kd in enumerate(st["layer_kind"]) if kd == 0}
    args = (st["Hkv"], st["D"], st["H"], st["dk"], st["dv"], st["R"], st["theta"])
    _, pre = O.refill(st["layer_kind"], _cut(ins, 0, N), *args, conv_weights=convw)
    outs, post = O.maintenance_round(pre, st["layer_kind"], [], [], _cut(ins, N, N + M), st["R"], st["theta"],
                                     conv_weights=convw)
    ref_outs, ref = O.refill(st["layer_kind"], ins, *args, conv_weights=convw)
    for l in outs:
        np.testing.assert_allclose(outs[l], ref_outs[l][N:], atol=1e-12)
    for l in post.states:
        np.testing.assert_allclose(post.states[l], ref.states[l], atol=1e-12)
        np.testing.assert_array_equal(post.conv[l], ref.conv[l])
    # without carrying the conv state (restarting it from zero) the outputs differ
    cold = pre.copy()
    cold.conv = {}
    o_cold, _ = O.maintenance_round(cold, st["layer_kind"], [], [], _cut(ins, N, N + M), st["R"], st["theta"],
                                    conv_weights=convw)
    assert not np.allclose(o_cold[0][:3], outs[0][:3])
