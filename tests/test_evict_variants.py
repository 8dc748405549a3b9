"""Eviction variants: Eq. 8 read literally (TB_EVICT_BUDGET_INCLUDES_WINDOW)
and SnapKV's average pooling (TB_EVICT_AVG_POOL).

Oracle pins (no GPU): hand-computed budgets, the average pool against
pure-Python neighbour sums, its special cases (kernel 1, constant scores),
and the whole variant eviction against brute force. The C ABI's host budget
(tb_retained_count_ex) against the oracle. GPU parity (@gpu): tb_score_evict
and tb_select_topk with the flags against the oracle, including a prefix long
enough for the non-cluster select path.
"""
import math

import numpy as np
import pytest

from oracle import timebill_oracle as orc
from paper_2512_21859_gb300 import inputs
from tests import brute_force as bf


# ---------------------------------------------------------------------------
# oracle pins
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("n,w,alpha,want", [
    (100, 16, 0.5, (34, 50)),     # 50 rows in all, 16 of them the window
    (100, 16, 0.9, (0, 16)),      # the budget is below the window: the window alone
    (100, 16, 0.0, (84, 100)),    # nothing evicted
    (100, 16, 0.84, (0, 16)),     # ceil(16) - 16 = 0
    (100, 16, 0.83, (1, 17)),     # ceil(17) - 16 = 1
    (10, 1, 0.3, (6, 7)),         # the 1e-9 n guard: (1 - 0.3) 10 lands a hair above 7
    (131072, 64, 0.9, (13044, 13108)),
])
def test_budget_includes_window_hand(n, w, alpha, want):
    assert orc.retained_count(n, w, alpha, budget_includes_window=True) == want
    # the same count of rows, the window inside it, never fewer than the window
    rows = math.ceil((1 - alpha) * n - 1e-9 * n)
    assert want[1] == min(max(rows, w), n)


def _avg_brute(row, pool_k):
    half = pool_k // 2
    out = []
    for j in range(len(row)):
        tot = 0.0
        for t in range(j - half, j + half + 1):
            if 0 <= t < len(row):
                tot += row[t]
        out.append(tot / pool_k)
    return out


@pytest.mark.parametrize("pool_k", [1, 3, 7, 13])
def test_avg_pool_against_neighbour_sums(pool_k):
    rng = np.random.default_rng(pool_k)
    S = rng.exponential(1.0, size=(2, 40))
    got = orc.avg_pool(S, pool_k)
    for g in range(2):
        np.testing.assert_allclose(got[g], _avg_brute(S[g].tolist(), pool_k), rtol=1e-14)


def test_avg_pool_special_cases():
    S = np.arange(1.0, 11.0)
    np.testing.assert_array_equal(orc.avg_pool(S, 1), S)                  # kernel 1: identity
    c = orc.avg_pool(np.full(12, 2.0), 7)
    np.testing.assert_allclose(c[3:9], 2.0)                                # interior: the value
    np.testing.assert_allclose(c[:3], 2.0 * np.array([4, 5, 6]) / 7)       # edges: zeros padded in
    np.testing.assert_allclose(c[-3:], 2.0 * np.array([6, 5, 4]) / 7)


@pytest.mark.parametrize("seed", range(3))
def test_variant_eviction_against_brute_force(seed):
    rng = np.random.default_rng(seed)
    hq, hkv, W, d, n = 4, 2, 5, 8, 41
    q = rng.standard_normal((1, hq, W, d))
    K = rng.standard_normal((hkv, n, d))
    V = rng.standard_normal((hkv, n, d))
    for alpha in (0.3, 0.6, 0.95):
        res = orc.score_evict(q, K, V, [n], [alpha], [0], W, 7, pool="avg",
                              budget_includes_window=True)[0]
        S = bf.scores(q[0].tolist(), K.tolist(), hq // hkv)
        kk = max(0, min(math.ceil((1 - alpha) * n - 1e-9 * n) - W, n - W))
        assert res["k"] == kk and res["R"] == kk + W
        for g in range(hkv):
            pooled = _avg_brute(S[g], 7)
            np.testing.assert_allclose(res["pooled"][g], pooled, rtol=1e-12)
            assert res["idx"][g].tolist() == bf.select(pooled, kk, n)


# ---------------------------------------------------------------------------
# the host budget of the C ABI (no GPU)
# ---------------------------------------------------------------------------

@pytest.fixture(scope="module")
def tbh():
    from paper_2512_21859_gb300 import build, binding
    build.build()
    binding.load()
    return binding


def test_abi_budget_matches_oracle(tbh):
    rng = np.random.default_rng(3)
    for _ in range(2000):
        w = int(rng.integers(1, 65))
        n = int(rng.integers(w, 200000))
        a = float(rng.choice([rng.uniform(0, 1), round(float(rng.uniform(0, 1)), 2)]))
        for flag in (0, tbh.TB_EVICT_BUDGET_INCLUDES_WINDOW):
            assert tbh.tb_retained_count_ex(n, w, a, flag) == orc.retained_count(n, w, a, bool(flag))
        # the pool bit does not touch the budget
        assert tbh.tb_retained_count_ex(n, w, a, tbh.TB_EVICT_AVG_POOL) == orc.retained_count(n, w, a)


# ---------------------------------------------------------------------------
# GPU parity
# ---------------------------------------------------------------------------

def _gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2512_21859_gb300 import binding as tb, build
    build.build()
    tb.load()
    return torch, tb


VARIANTS = [
    ("bf16", 28, 4, 128, 32, 7, [5000, 700], [0.5, 0.9], 2),
    ("bf16", 28, 4, 128, 32, 7, [5000, 700], [0.5, 0.9], 1),
    ("bf16", 28, 4, 128, 32, 7, [3000], [0.3], 3),
    ("bf16", 32, 8, 128, 64, 5, [2100, 64], [0.8, 0.5], 3),
    ("f32", 4, 2, 64, 16, 7, [512, 97], [0.5, 0.2], 3),
]


@pytest.mark.gpu
@pytest.mark.parametrize("case", range(len(VARIANTS)))
def test_gpu_variant_evict(case):
    torch, tb = _gpu()
    from tests.gpu_common import check_index_set, from_dev, request_slices, run_evict
    dtype, hq, hkv, d, W, pk, ns, alphas, flags = VARIANTS[case]
    wl = inputs.Workload(name="var", layers=1, hq=hq, hkv=hkv, head_dim=d, dtype=dtype, batch=len(ns),
                         window=W, pool_k=pk, decode_steps=1, seed=500 + case, n_fixed=ns[0], alpha=0.5,
                         heavy_frac=0.01, unit_keys=dtype == "bf16")
    lay = inputs.make_layer(wl, 0, n_override=ns)
    lay["alpha"] = np.asarray(alphas, dtype=np.float64)
    res = run_evict(wl, lay, flags=flags)
    ref = orc.score_evict(inputs.as_f32(lay["q_win"], dtype), inputs.as_f32(lay["K"], dtype),
                          inputs.as_f32(lay["V"], dtype), lay["n"], lay["alpha"], lay["kv_offset"], W, pk,
                          pool="avg" if flags & tb.TB_EVICT_AVG_POOL else "max",
                          budget_includes_window=bool(flags & tb.TB_EVICT_BUDGET_INCLUDES_WINDOW))
    desc = res["desc"]
    Kc, Vc = from_dev(res["Kc_t"], dtype), from_dev(res["Vc_t"], dtype)
    for b, n in enumerate(ns):
        s0, i0, P, R = request_slices(desc, b)
        r = ref[b]
        assert R == r["R"]
        for g in range(hkv):
            check_index_set(res["idx"][g, i0:i0 + R], r["pooled"][g], r["k"], n, W)
            np.testing.assert_allclose(res["pooled"][g, s0:s0 + P], r["pooled"][g], rtol=2e-6, atol=0)
            off, oo = int(lay["kv_offset"][b]), int(desc.out_offset[b])
            gi = res["idx"][g, i0:i0 + R]
            assert np.array_equal(Kc[g, oo:oo + R], lay["K"][g, off + gi])
            assert np.array_equal(Vc[g, oo:oo + R], lay["V"][g, off + gi])


@pytest.mark.gpu
@pytest.mark.parametrize("P_long", [False, True])
def test_gpu_avg_select_exact_on_quantised_scores(P_long):
    """Scores on a 1/64 grid: every window sum is exact in fp32, so the
    average-pooled order, ties included, must match the oracle exactly. The
    long prefix (> 8 x 16K keys) takes the non-cluster select path."""
    torch, tb = _gpu()
    from tests.gpu_common import request_slices
    rng = np.random.default_rng(17 + P_long)
    W, pk, hkv = 16, 7, 2
    ns = [140000] if P_long else [int(x) for x in rng.integers(W, 20000, size=4)] + [W + 1]
    alphas = list(rng.uniform(0, 1, size=len(ns)))
    desc = tb.EvictDesc(hq=hkv, hkv=hkv, head_dim=64, window=W, pool_k=pk, dtype=tb.TB_F32,
                        n=ns, alpha=alphas, flags=tb.TB_EVICT_AVG_POOL)
    score_rows, idx_rows = tb.tb_evict_layout(desc)
    S = (np.floor(rng.exponential(1.0, size=(hkv, max(score_rows, 1))) * 64) / 64).astype(np.float32)
    S_t = torch.from_numpy(S).cuda()
    idx = torch.full((hkv, idx_rows), -1, dtype=torch.int32, device="cuda")
    pooled = torch.zeros_like(S_t)
    ws = torch.empty(tb.tb_evict_workspace_size(desc), dtype=torch.uint8, device="cuda")
    tb.tb_select_topk(desc, S_t, idx, pooled, ws)
    gi, gp = idx.cpu().numpy(), pooled.cpu().numpy()
    for b, nb in enumerate(ns):
        s0, i0, P, R = request_slices(desc, b)
        for g in range(hkv):
            op = orc.avg_pool(S[g, s0:s0 + P].astype(np.float64), pk)
            np.testing.assert_allclose(gp[g, s0:s0 + P], op, rtol=2.5e-7, atol=0)
            assert np.array_equal(gi[g, i0:i0 + R], orc.select_indices(op, R - W, nb))
