"""The pins must catch plausible mistakes in the oracle.

Each case plants one mistake in a copy of the oracle's source (on the CPU,
never in the CUDA path) and checks that at least one pin then fails: the
hand-derived closed forms of tests/golden or the brute force.
"""
import inspect
import math
import json
import os
import types

import numpy as np
import pytest

from oracle import timebill_oracle as orc
from tests import brute_force as bf
from tests.test_oracle_pins import GOLDEN, _frac_expr, _golden_vote_inputs, _packed_decode_case

SRC = inspect.getsource(orc)

MUTANTS = {
    "scale 1/d instead of 1/sqrt(d)": ("sigma = 1.0 / math.sqrt(d)\n    # visible", "sigma = 1.0 / d\n    # visible"),
    "window row sees one key too few": ("<= (P + np.arange(W))", "< (P + np.arange(W))"),
    "window row sees the whole window": ("<= (P + np.arange(W))[:, None]", "<= (P + W - 1 + 0 * np.arange(W))[:, None]"),
    "window keys also scored": ("S[g] += prob[:, :P].sum(axis=0)", "S[g] += prob[:, 1:P + 1].sum(axis=0)"),
    "interleaved head mapping": ("for h in range(g * G, (g + 1) * G):\n            logits", "for h in range(g, hq, hkv):\n            logits"),
    "pool misses right neighbours": ("out[..., :-t] = np.maximum(out[..., :-t], S[..., t:])", "pass"),
    "pool one wider": ("range(1, pool_k // 2 + 1)", "range(1, pool_k // 2 + 2)"),
    "ties to the higher index": ("np.lexsort((np.arange(P), -pooled))", "np.lexsort((-np.arange(P), -pooled))"),
    "budget rounds instead of ceil": ("k = math.ceil((1.0 - alpha) * n - 1e-9 * n)", "k = round((1.0 - alpha) * n)"),
    "budget counts the window inside": ("return k, k + window", "return max(k - window, 0), max(k - window, 0) + window"),
    "decode scale dropped": ("s = sigma * (kk @ q[h])", "s = kk @ q[h]"),
    "decode attends one row too many": ("kk = np.asarray(Kc[g, :length]", "kk = np.asarray(Kc[g, :length + 1]"),
    "packed decode slices one row late": ("Kc[:, off:off + L], Vc[:, off:off + L]", "Kc[:, off + 1:off + 1 + L], Vc[:, off + 1:off + 1 + L]"),
    "packed decode reads the next request's offset": ("off, L = int(cache_offset[b]), int(lens[b])", "off, L = int(cache_offset[min(b + 1, B - 1)]), int(lens[b])"),
    "packed decode writes the wrong request": ("        out[b] = decode_attention(q[b]", "        out[B - 1 - b] = decode_attention(q[b]"),
    "packed decode takes one request's length for all": ("off, L = int(cache_offset[b]), int(lens[b])", "off, L = int(cache_offset[b]), int(lens[0])"),
    "decoding steps counted from i = 0": ("for i in range(1, n_w):", "for i in range(0, n_w):"),
    "decode step over N_kv without the eviction": ("p * ((1.0 - alpha) * n_x + i - 1) + q", "p * (n_x + i - 1) + q"),
    "per-step constant dropped": ("t_decode += p * ((1.0 - alpha) * n_x + i - 1) + q", "t_decode += p * ((1.0 - alpha) * n_x + i - 1)"),
    "pessimistic length rounded down": ("int(min(math.ceil(k * n_hat), n_max))", "int(min(math.floor(k * n_hat), n_max))"),
    "lse rows see one key too few": ("visible = np.arange(N)[None, :] <= last_seen[:, None]", "visible = np.arange(N)[None, :] < last_seen[:, None]"),
    "lse without the max added back": ("out[h] = m + np.log(", "out[h] = np.log("),
    "scores from lse over the window keys too": ("logits = sigma * (q[h] @ k[h // G, :P].T)      # [W][P]\n        S[h // G] += np.exp(logits - L[h][:, None]).sum(axis=0)", "logits = sigma * (q[h] @ k[h // G, 1:P + 1].T)      # [W][P]\n        S[h // G] += np.exp(logits - L[h][:, None]).sum(axis=0)"),
    "avg pool over the in-range count": ("    return total / pool_k\n", "    return total / np.convolve(np.ones(L), np.ones(pool_k), 'same')\n"),
    "avg pool one narrower": ("    for t in range(pool_k):\n        total += Z[..., t:t + L]", "    for t in range(pool_k - 1):\n        total += Z[..., t:t + L]"),
    "literal budget keeps the window on top": ("        k -= window\n", "        k -= 0\n"),
    "predictor overhead ignored": ("return t_predict + wcet(a, b, c, p, q, n_x, al, n_w) - budget", "return wcet(a, b, c, p, q, n_x, al, n_w) - budget"),
    "fit without the constant column": ("for k in range(degree, -1, -1)], axis=1)", "for k in range(degree, 0, -1)], axis=1)"),
    "MAPE relative to the fit": ("np.abs(fit - ta) / ta", "np.abs(fit - ta) / fit"),
    "MAPE without the percent": ("mape = 100.0 * float(", "mape = float("),
}


def _mutant(name):
    old, new = MUTANTS[name]
    assert SRC.count(old) == 1, name
    mod = types.ModuleType("oracle_mutant")
    exec(compile(SRC.replace(old, new), "oracle_mutant", "exec"), mod.__dict__)
    return mod


def _pins_pass(m):
    """Run a compact version of the pins against module m; False on any miss."""
    try:
        with open(os.path.join(GOLDEN, "window_vote_closed_form.json")) as f:
            gd = json.load(f)
        q, K = _golden_vote_inputs(gd)
        if m.retained_count(6, 2, gd["alpha"]) != (2, 4):
            return False
        if m.retained_count(131072, 64, 0.9) != (13108, 13172):
            return False
        S = m.window_scores(q, K)
        S_exp = np.array([[_frac_expr(x) for x in r] for r in gd["S_expected"]])
        if not np.allclose(S, S_exp, rtol=1e-12, atol=0):
            return False
        for case in gd["cases"]:
            pooled = m.max_pool(S, case["pool_k"])
            for g in range(2):
                if m.select_indices(pooled[g], 2, 6).tolist() != case["idx_expected"][g]:
                    return False
        rng = np.random.default_rng(2)
        qq = rng.standard_normal((3, 5, 8))
        KK = rng.standard_normal((1, 33, 8)) * 1.5
        VV = rng.standard_normal((1, 33, 8))
        S2 = m.window_scores(qq, KK)
        S2_bf = np.array(bf.scores(qq.tolist(), KK.tolist(), 3))
        if not np.allclose(S2, S2_bf, rtol=1e-12):
            return False
        pb = bf.pool(S2_bf[0].tolist(), 7)
        if not np.allclose(m.max_pool(S2, 7)[0], pb, rtol=1e-12):
            return False
        # exact ties: constant keys
        Kt = np.tile(KK[:, :1], (1, 33, 1))
        pt = m.max_pool(m.window_scores(qq, Kt), 7)[0]
        if m.select_indices(pt, 10, 33).tolist() != bf.select(pt.tolist(), 10, 33):
            return False
        out = m.decode_attention(qq[:1, 0], KK, VV, 20)
        ref = bf.attention(qq[0, 0].tolist(), KK[0].tolist(), VV[0].tolist(), 20)
        if not np.allclose(out[0], ref, rtol=1e-12):
            return False
        # the packed-batch decode against the brute force on unpacked caches
        qb, caches, Kp, Vp, lens, offs, Gb = _packed_decode_case()
        ob = m.decode_batch(qb, Kp, Vp, lens, offs)
        for b, (Kb, Vb) in enumerate(caches):
            for h in (0, qb.shape[1] - 1):
                want = [0.0] * qb.shape[2] if lens[b] == 0 else bf.attention(
                    qb[b, h].tolist(), Kb[h // Gb].tolist(), Vb[h // Gb].tolist(), lens[b])
                if not np.allclose(ob[b, h], want, rtol=1e-12, atol=1e-14):
                    return False
        # the budgeted eviction ratio: the hand example of tests/test_alpha_star.py
        al = m.alpha_star(1e-9, 2e-6, 1e-4, 1e-6, 5e-5, 1000, 10, 1.0, 100, 3e-4, 8e-3, 0.95)
        want = 1.0 - (8e-3 - 3e-4 - (1e-3 + 2e-3 + 1e-4) - 9 * 5e-5 - 36e-6) / 9e-3
        if abs(al - want) > 1e-12 or m.pessimistic_length(10, 1.25, 100) != 13:
            return False
        # the window normalisers and the scores rebuilt from them: brute force
        rng = np.random.default_rng(5)
        qq, KK2 = rng.standard_normal((4, 5, 8)), rng.standard_normal((2, 23, 8))
        lse = m.window_lse(qq, KK2)
        G2 = 2
        for h in (0, 3):
            for w in (0, 4):
                lg = [float(qq[h, w] @ KK2[h // G2, j]) / math.sqrt(8) for j in range(18 + w + 1)]
                mx = max(lg)
                if abs(lse[h, w] - (mx + math.log(math.fsum(math.exp(x - mx) for x in lg)))) > 1e-12:
                    return False
        if not np.allclose(m.window_scores_from_lse(qq, KK2, lse), np.array(bf.scores(qq.tolist(), KK2.tolist(), G2)),
                           rtol=1e-12, atol=0):
            return False
        # the eviction variants: the literal Eq. 8 budget and the average pool
        if m.retained_count(100, 16, 0.5, budget_includes_window=True) != (34, 50):
            return False
        ap = m.avg_pool(np.full(12, 2.0), 7)
        if not (np.allclose(ap[3:9], 2.0) and np.allclose(ap[:3], 2.0 * np.array([4, 5, 6]) / 7)):
            return False
        # the least-squares fit: the hand line of tests/test_time_fit.py
        coef, mape = m.fit_time_model([0, 1, 2], [1, 3, 2], 1)
        if not np.allclose(coef, [0.5, 1.5], atol=1e-14) or abs(mape - 100.0 * (0.5 + 1 / 3 + 0.25) / 3) > 1e-12:
            return False
        return True
    except (ValueError, IndexError, AssertionError):
        return False


def test_unmutated_oracle_passes():
    assert _pins_pass(orc)


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name):
    assert not _pins_pass(_mutant(name)), name
