"""Pins of the CPU oracle against facts fixed outside it.

Each test checks the oracle against something it does not share code with:
hand-derived closed forms (tests/golden), an independent pure-Python brute
force (tests/brute_force.py), mathematical invariants, special cases that
reduce to a library routine (torch's softmax / scaled-dot-product attention
in fp64 on the CPU), and the retained-length arithmetic of Eq. 8.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import timebill_oracle as orc
from tests import brute_force as bf

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _frac_expr(s):
    """'a/b + c/d' -> float (exact rational arithmetic first)."""
    tot = Fraction(0)
    for term in s.split("+"):
        tot += Fraction(term.strip())
    return float(tot)


# --------------------------------------------------------------------------
# Eq. 8: retained length
# --------------------------------------------------------------------------

@pytest.mark.parametrize("n,w,alpha,k,r", [
    (512, 16, 0.5, 256, 272),          # tiny config
    (4096, 32, 0.0, 4064, 4096),       # alpha = 0 keeps the prompt (clamped to P)
    (4096, 32, 0.25, 3072, 3104),
    (4096, 32, 0.5, 2048, 2080),
    (4096, 32, 0.75, 1024, 1056),
    (32768, 32, 0.5, 16384, 16416),
    (32768, 32, 0.95, 1639, 1671),     # ceil(1638.4)
    (131072, 64, 0.9, 13108, 13172),   # ceil(13107.2)
    (10, 1, 0.3, 7, 8),                # 0.7 * 10 in binary is 7.000000000000001
    (6, 2, 0.6666666666666666, 2, 4),  # (1 - 2/3) * 6 in binary is 2.0000000000000004
    (100, 4, 1.0, 0, 4),               # alpha = 1 keeps the window only
    (8, 8, 0.5, 0, 8),                 # W = N: no prefix to score
])
def test_retained_count_values(n, w, alpha, k, r):
    assert orc.retained_count(n, w, alpha) == (k, r)


def test_retained_count_is_ceil_of_eq8_and_monotone():
    # Eq. 8: (1 - alpha) N tokens survive; where that product is an exact
    # integer (alpha * N integral with alpha a dyadic rational) k equals it.
    for n in (64, 1000, 4096, 32768):
        for num in range(0, 17):
            alpha = num / 16.0
            k, _ = orc.retained_count(n, 1, alpha)
            exact = Fraction(16 - num, 16) * n
            assert k == min(math.ceil(exact), n - 1)
        ks = [orc.retained_count(n, 8, a / 100.0)[0] for a in range(101)]
        assert all(x >= y for x, y in zip(ks, ks[1:]))


@pytest.mark.parametrize("bad", [(-1e-12,), (1.0000001,), (float("nan"),)])
def test_retained_count_rejects_bad_alpha(bad):
    with pytest.raises(ValueError):
        orc.retained_count(100, 4, bad[0])


def test_decode_length_matches_eq8_shape():
    # Eq. 8: the cache grows by one row per decode step on top of what
    # eviction kept: lengths at steps 1..S are R+1..R+S (the step's own token
    # appended before attending), an arithmetic progression with slope 1.
    for n, w, a in [(512, 16, 0.5), (131072, 64, 0.9)]:
        k, R = orc.retained_count(n, w, a)
        lens = [R + s for s in range(1, 6)]
        assert np.all(np.diff(lens) == 1)
        assert lens[0] - 1 == math.ceil((1 - a) * n - 1e-9 * n) + w


# --------------------------------------------------------------------------
# Hand-derived closed forms (tests/golden)
# --------------------------------------------------------------------------

def _golden_vote_inputs(gd):
    c = np.array(gd["c"], dtype=np.float64)
    a = np.array(gd["a"], dtype=np.float64)
    hkv, N = c.shape
    hq, W, d = len(a), 2, 4
    K = np.zeros((hkv, N, d))
    K[:, :, 0] = np.log(c)
    q = np.zeros((hq, W, d))
    q[:, :, 0] = 2.0 * a[:, None]
    return q, K


def test_golden_window_vote():
    with open(os.path.join(GOLDEN, "window_vote_closed_form.json")) as f:
        gd = json.load(f)
    q, K = _golden_vote_inputs(gd)
    N = K.shape[1]
    assert orc.retained_count(N, 2, gd["alpha"]) == (gd["k_expected"], gd["R_expected"])
    S = orc.window_scores(q, K)
    S_exp = np.array([[_frac_expr(x) for x in row] for row in gd["S_expected"]])
    np.testing.assert_allclose(S, S_exp, rtol=1e-13, atol=0)
    k = gd["k_expected"]
    for case in gd["cases"]:
        pooled = orc.max_pool(S, case["pool_k"])
        if "pooled_expected" in case:
            P_exp = np.array([[_frac_expr(x) for x in row] for row in case["pooled_expected"]])
            np.testing.assert_allclose(pooled, P_exp, rtol=1e-13, atol=0)
        for g in range(K.shape[0]):
            idx = orc.select_indices(pooled[g], k, N)
            assert idx.tolist() == case["idx_expected"][g], (case, g)


def test_golden_decode():
    with open(os.path.join(GOLDEN, "decode_closed_form.json")) as f:
        gd = json.load(f)
    c = np.array(gd["c"], dtype=np.float64)
    v = np.array(gd["v"], dtype=np.float64)
    Kc = np.zeros((1, len(c), 4))
    Kc[0, :, 0] = np.log(c)
    Vc = v[None]
    q = np.array([[2.0, 0, 0, 0]])
    for case in gd["cases"]:
        out = orc.decode_attention(q, Kc, Vc, case["len"])
        exp = np.array([_frac_expr(x) if "/" in x else float(x) for x in case["out_expected"]])
        np.testing.assert_allclose(out[0], exp, rtol=1e-13, atol=1e-15)


# --------------------------------------------------------------------------
# Brute force on tiny random inputs
# --------------------------------------------------------------------------

def _rand_case(seed, hkv, G, W, N, d, scale=1.0):
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((hkv * G, W, d))
    K = rng.standard_normal((hkv, N, d)) * scale
    V = rng.standard_normal((hkv, N, d))
    return q, K, V


@pytest.mark.parametrize("seed,hkv,G,W,N,d,pool_k", [
    (0, 1, 1, 1, 9, 2, 1),
    (1, 2, 2, 3, 20, 4, 3),
    (2, 1, 3, 5, 33, 8, 7),
    (3, 3, 1, 2, 17, 3, 5),
    (4, 2, 3, 4, 64, 8, 7),
    (5, 1, 2, 8, 12, 5, 9),   # pool wider than half the prefix
])
def test_oracle_matches_brute_force(seed, hkv, G, W, N, d, pool_k):
    q, K, V = _rand_case(seed, hkv, G, W, N, d, scale=1.5)
    S = orc.window_scores(q, K)
    S_bf = np.array(bf.scores(q.tolist(), K.tolist(), G))
    np.testing.assert_allclose(S, S_bf, rtol=1e-12, atol=1e-15)
    pooled = orc.max_pool(S, pool_k)
    for g in range(hkv):
        pb = bf.pool(S_bf[g].tolist(), pool_k)
        np.testing.assert_allclose(pooled[g], pb, rtol=1e-12, atol=1e-15)
        for alpha in (0.0, 0.1, 0.35, 0.5, 0.77, 0.9, 1.0):
            k, R = orc.retained_count(N, W, alpha)
            assert k == bf.budget(N, W, alpha)
            idx = orc.select_indices(pooled[g], k, N)
            # compare on the brute force's own pooled values: identical up to
            # rounding, so use the oracle's to keep exact ties exact
            assert idx.tolist() == bf.select(pooled[g].tolist(), k, N)
            assert len(idx) == R
            Kc = orc.gather_rows(K[g], idx)
            assert np.array_equal(Kc, K[g][idx])
            for length in (1, R // 2 + 1, R):
                qd = q[g * G, 0]
                out = orc.decode_attention(q[g * G:g * G + 1, 0], Kc[None], orc.gather_rows(V[g], idx)[None], length)
                ref = bf.attention(qd.tolist(), Kc.tolist(), V[g][idx].tolist(), length)
                np.testing.assert_allclose(out[0], ref, rtol=1e-12, atol=1e-14)


def test_score_evict_batch_matches_per_request():
    rng = np.random.default_rng(11)
    hkv, G, W, d = 2, 2, 3, 4
    ns = [15, 7, 22]
    rows = sum(ns)
    off = np.concatenate([[0], np.cumsum(ns)[:-1]])
    q = rng.standard_normal((3, hkv * G, W, d))
    K = rng.standard_normal((hkv, rows, d))
    V = rng.standard_normal((hkv, rows, d))
    alphas = [0.2, 0.5, 0.9]
    res = orc.score_evict(q, K, V, ns, alphas, off, W, 3)
    for b, r in enumerate(res):
        Kb = K[:, off[b]:off[b] + ns[b]]
        S_bf = bf.scores(q[b].tolist(), Kb.tolist(), G)
        np.testing.assert_allclose(r["S"], S_bf, rtol=1e-12)
        for g in range(hkv):
            k = bf.budget(ns[b], W, alphas[b])
            assert r["idx"][g].tolist() == bf.select(r["pooled"][g].tolist(), k, ns[b])
            assert np.array_equal(r["Vc"][g], V[g, off[b]:off[b] + ns[b]][r["idx"][g]])


# --------------------------------------------------------------------------
# Invariants and special cases
# --------------------------------------------------------------------------

def test_invariants_on_a_medium_case():
    q, K, V = _rand_case(21, 2, 3, 6, 400, 16)
    N, W = 400, 6
    S = orc.window_scores(q, K)
    # every softmax row sums to one: prefix mass + window mass = G * W
    d = 16
    sig = 1 / math.sqrt(d)
    P = N - W
    for g in range(2):
        win_mass = 0.0
        for h in range(g * 3, g * 3 + 3):
            for w in range(W):
                lg = sig * K[g, :P + w + 1] @ q[h, w]
                e = np.exp(lg - lg.max())
                win_mass += e[P:].sum() / e.sum()
        assert abs(S[g].sum() + win_mass - 3 * W) < 1e-10
    pooled = orc.max_pool(S, 7)
    assert np.all(pooled >= S)
    assert np.array_equal(orc.max_pool(S, 1), S)
    for alpha in np.linspace(0, 1, 11):
        k, R = orc.retained_count(N, W, float(alpha))
        for g in range(2):
            idx = orc.select_indices(pooled[g], k, N)
            assert len(idx) == R
            assert np.all(np.diff(idx) > 0)
            assert set(range(P, N)) <= set(idx.tolist())
            # everything kept outranks everything dropped
            kept = idx[idx < P]
            dropped = np.setdiff1d(np.arange(P), kept)
            if len(kept) and len(dropped):
                assert pooled[g][kept].min() >= pooled[g][dropped].max()
    k0, R0 = orc.retained_count(N, W, 0.0)
    assert orc.select_indices(pooled[0], k0, N).tolist() == list(range(N))


def test_single_window_row_is_plain_softmax():
    import torch
    q, K, _ = _rand_case(5, 1, 1, 1, 50, 8)
    S = orc.window_scores(q, K)
    logits = torch.from_numpy(K[0]) @ torch.from_numpy(q[0, 0]) / math.sqrt(8)
    p = torch.softmax(logits, dim=0).numpy()
    np.testing.assert_allclose(S[0], p[:49], rtol=1e-13)


def test_constant_keys_pin_the_tie_rule():
    rng = np.random.default_rng(3)
    N, W = 40, 4
    q = rng.standard_normal((2, W, 8))
    K = np.tile(rng.standard_normal((1, 1, 8)), (1, N, 1))
    S = orc.window_scores(q, K)
    pooled = orc.max_pool(S, 7)
    assert np.all(pooled == pooled[0, 0])
    for alpha in (0.1, 0.5, 0.9):
        k, _ = orc.retained_count(N, W, alpha)
        assert orc.select_indices(pooled[0], k, N).tolist() == list(range(k)) + list(range(N - W, N))


def test_head_to_group_mapping_is_contiguous():
    # Queries only in head 1; with Hq=4, Hkv=2 head 1 belongs to group 0.
    # Group 0's scores then differ from uniform and group 1's stay uniform.
    rng = np.random.default_rng(8)
    N, W, d = 30, 2, 4
    q = np.zeros((4, W, d))
    q[1] = rng.standard_normal((W, d)) * 3
    K = rng.standard_normal((2, N, d))
    S = orc.window_scores(q, K)
    P = N - W
    uniform = np.array([sum(1.0 / (P + w + 1) for w in range(W)) * 2] * P)
    np.testing.assert_allclose(S[1], uniform, rtol=1e-13)
    assert np.abs(S[0] - uniform).max() > 1e-3


def test_planted_heavy_hitters_survive():
    from paper_2512_21859_gb300 import inputs
    wl = inputs.WORKLOADS["tiny"]
    lay = inputs.make_layer(wl, 0)
    q = inputs.as_f32(lay["q_win"], wl.dtype)
    K = inputs.as_f32(lay["K"], wl.dtype)
    V = inputs.as_f32(lay["V"], wl.dtype)
    res = orc.score_evict(q, K, V, lay["n"], lay["alpha"], lay["kv_offset"], wl.window, wl.pool_k)[0]
    P = int(lay["n"][0]) - wl.window
    for g in range(wl.hkv):
        kept = set(res["idx"][g].tolist())
        for j in lay["heavy"][0]:
            assert j in kept
            for t in range(max(0, j - 3), min(P, j + 4)):
                assert t in kept


def test_decode_full_cache_equals_sdpa():
    import torch
    q, K, V = _rand_case(9, 2, 3, 1, 70, 16)
    N, W = 70, 1
    k, R = orc.retained_count(N, W, 0.0)
    pooled = orc.max_pool(orc.window_scores(q, K), 7)
    idx = [orc.select_indices(pooled[g], k, N) for g in range(2)]
    Kc = np.stack([K[g][idx[g]] for g in range(2)])
    Vc = np.stack([V[g][idx[g]] for g in range(2)])
    assert np.array_equal(Kc, K)
    qd = np.random.default_rng(1).standard_normal((6, 16))
    out = orc.decode_attention(qd, Kc, Vc, N)
    qt = torch.from_numpy(qd)[:, None, :]                      # [Hq][1][d]
    kt = torch.from_numpy(K).repeat_interleave(3, dim=0)        # [Hq][N][d]
    vt = torch.from_numpy(V).repeat_interleave(3, dim=0)
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt)[:, 0].numpy()
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-14)


def test_decode_invariances():
    rng = np.random.default_rng(4)
    q = rng.standard_normal((2, 8))
    Kc = rng.standard_normal((1, 25, 8))
    Vc = rng.standard_normal((1, 25, 8))
    base = orc.decode_attention(q, Kc, Vc, 25)
    perm = rng.permutation(25)
    np.testing.assert_allclose(orc.decode_attention(q, Kc[:, perm], Vc[:, perm], 25), base, rtol=1e-12)
    # rows past len are ignored
    Kc2 = Kc.copy()
    Kc2[:, 20:] = 1e6
    np.testing.assert_allclose(orc.decode_attention(q, Kc2, Vc, 20), orc.decode_attention(q, Kc, Vc, 20))
    # one row: the output is that row's value
    np.testing.assert_allclose(orc.decode_attention(q, Kc, Vc, 1), np.tile(Vc[0, 0], (2, 1)))
    # a convex combination of the values
    assert np.all(base <= Vc[0].max(axis=0) + 1e-12) and np.all(base >= Vc[0].min(axis=0) - 1e-12)


# --------------------------------------------------------------------------
# The packed-batch decode the GPU parity tests compare against
# --------------------------------------------------------------------------

def _packed_decode_case(seed=21):
    """Four requests whose caches are drawn first as separate arrays and
    only then packed at non-contiguous row offsets, with filler rows (huge
    values) between and after them, so that a wrong offset or a wrong
    request index changes the result."""
    rng = np.random.default_rng(seed)
    hkv, G, d = 2, 3, 5
    lens = [7, 0, 12, 1]
    caps = [9, 3, 14, 4]
    caches = [(rng.standard_normal((hkv, c, d)), rng.standard_normal((hkv, c, d))) for c in caps]
    q = rng.standard_normal((len(lens), hkv * G, d))
    gaps = [2, 1, 5, 3]
    offs, rows = [], 0
    for c, gap in zip(caps, gaps):
        rows += gap
        offs.append(rows)
        rows += c
    Kp = np.full((hkv, rows + 2, d), 1e3)
    Vp = np.full((hkv, rows + 2, d), -1e3)
    for (Kb, Vb), o, c in zip(caches, offs, caps):
        Kp[:, o:o + c] = Kb
        Vp[:, o:o + c] = Vb
    return q, caches, Kp, Vp, lens, offs, G


def test_decode_batch_matches_unpacked_brute_force():
    q, caches, Kp, Vp, lens, offs, G = _packed_decode_case()
    out = orc.decode_batch(q, Kp, Vp, lens, offs)
    assert out.shape == q.shape
    for b, (Kb, Vb) in enumerate(caches):
        for h in range(q.shape[1]):
            g = h // G
            if lens[b] == 0:
                assert np.all(out[b, h] == 0.0)
                continue
            ref = bf.attention(q[b, h].tolist(), Kb[g].tolist(), Vb[g].tolist(), lens[b])
            np.testing.assert_allclose(out[b, h], ref, rtol=1e-12, atol=1e-14)
    # one request alone through the single-request routine on its own arrays
    Kb, Vb = caches[2]
    np.testing.assert_allclose(out[2], orc.decode_attention(q[2], Kb, Vb, lens[2]), rtol=1e-13)
    # a length-1 request returns its first value row, its heads' own group
    np.testing.assert_allclose(out[3], np.repeat(caches[3][1][:, 0], G, axis=0), rtol=1e-13)
