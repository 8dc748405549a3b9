"""The eviction ratio a time budget allows (Prob. 13, closed form Eq. 14).

Oracle pins: the oracle solves Prob. 13 from its definition (the WCET of
Eq. 12 summed step by step, bisection on the constraint). It is pinned here
by a hand-computed example, the problem's own conditions (feasibility,
minimality, the [0, alpha_max] range) and its degenerate cases. The C ABI's
closed form (tb_alpha_star, tb_wcet; host code, no GPU) is then checked
against the oracle on a seeded grid of models, budgets and lengths.
"""
import math

import numpy as np
import pytest

from oracle import timebill_oracle as orc


# ---------------------------------------------------------------------------
# oracle pins
# ---------------------------------------------------------------------------

def test_oracle_hand_example():
    # prefill free, one step = 1 us per cached token: N_x = 1000, N_W = 10
    # -> nine decoding steps over 1000 (1 - a) + i - 1 tokens, i = 1..9:
    # WCET = 1e-6 (9000 (1 - a) + 36). Budget 5 ms: a = 1 - (5e-3 - 36e-6) / 9e-3.
    want = 1.0 - (5e-3 - 36e-6) / 9e-3
    got = orc.alpha_star(0, 0, 0, 1e-6, 0, 1000, 10, 1.0, 100, 0.0, 5e-3, 0.95)
    assert got == pytest.approx(want, abs=1e-14)
    assert orc.wcet(0, 0, 0, 1e-6, 0, 1000, 0.25, 10) == pytest.approx(1e-6 * (9000 * 0.75 + 36))
    # prefill and predictor overhead come off the budget; q adds per step
    got = orc.alpha_star(1e-9, 2e-6, 1e-4, 1e-6, 5e-5, 1000, 10, 1.0, 100, 3e-4, 8e-3, 0.95)
    prefill = 1e-9 * 1e6 + 2e-6 * 1000 + 1e-4
    want = 1.0 - (8e-3 - 3e-4 - prefill - 9 * 5e-5 - 36e-6) / 9e-3
    assert got == pytest.approx(want, abs=1e-12)


@pytest.mark.parametrize("seed", range(5))
def test_oracle_solves_the_problem(seed):
    rng = np.random.default_rng(seed)
    for _ in range(20):
        a, b, c = rng.uniform(0, 1e-9), rng.uniform(0, 1e-5), rng.uniform(0, 1e-3)
        p, q = rng.uniform(1e-8, 1e-6), rng.uniform(0, 1e-4)
        n_x, n_hat, k = int(rng.integers(100, 4000)), float(rng.integers(1, 300)), float(rng.uniform(1, 3))
        n_max, t_pred, amax = int(rng.integers(50, 600)), float(rng.uniform(0, 1e-3)), 0.95
        n_w = orc.pessimistic_length(n_hat, k, n_max)
        w0 = orc.wcet(a, b, c, p, q, n_x, 0.0, n_w)
        T = t_pred + w0 * float(rng.uniform(0.3, 1.2))
        al = orc.alpha_star(a, b, c, p, q, n_x, n_hat, k, n_max, t_pred, T, amax)
        assert 0.0 <= al <= amax
        fits = t_pred + orc.wcet(a, b, c, p, q, n_x, al, n_w) <= T * (1 + 1e-12)
        if al < amax:
            assert fits  # feasible
        if 0.0 < al:
            # minimal: a slightly smaller ratio breaks the budget
            assert t_pred + orc.wcet(a, b, c, p, q, n_x, max(0.0, al - 1e-9), n_w) > T * (1 - 1e-12) or al == 0.0
        if not fits:
            assert al == amax  # nothing in range fits: the most eviction allowed


def test_oracle_degenerate_cases():
    # a budget that fits everything keeps the whole cache; one that fits nothing caps at alpha_max
    assert orc.alpha_star(0, 0, 0, 1e-6, 0, 1000, 10, 1.0, 100, 0.0, 1.0, 0.95) == 0.0
    assert orc.alpha_star(0, 0, 0, 1e-6, 0, 1000, 10, 1.0, 100, 0.0, 1e-9, 0.95) == 0.95
    # one token to generate: no decoding step, alpha cannot change the estimate
    assert orc.pessimistic_length(1, 1.0, 100) == 1
    assert orc.wcet(0, 0, 1e-3, 1e-6, 1e-4, 1000, 0.7, 1) == pytest.approx(1e-3)
    # N_W is the pessimistic length: k N_hat rounded up, capped at N_max
    assert orc.pessimistic_length(10, 1.25, 100) == 13
    assert orc.pessimistic_length(10, 5.0, 30) == 30


def test_oracle_alpha_feeds_the_retained_count():
    # the ratio found here is what Eq. 8 then turns into a cache length
    al = orc.alpha_star(0, 0, 0, 1e-6, 0, 1000, 10, 1.0, 100, 0.0, 5e-3, 0.95)
    k_keep, r = orc.retained_count(1000, 16, al)
    assert k_keep == math.ceil((1 - al) * 1000 - 1e-9 * 1000) and r == k_keep + 16


# ---------------------------------------------------------------------------
# the C ABI against the oracle (host code: runs without a GPU)
# ---------------------------------------------------------------------------

@pytest.fixture(scope="module")
def tb():
    from paper_2512_21859_gb300 import build, binding
    build.build()
    binding.load()
    return binding


@pytest.mark.parametrize("seed", range(4))
def test_abi_matches_oracle(tb, seed):
    rng = np.random.default_rng(100 + seed)
    for _ in range(40):
        coef = dict(a=rng.uniform(0, 1e-9), b=rng.uniform(0, 1e-5), c=rng.uniform(0, 1e-3),
                    p=rng.uniform(1e-8, 1e-6), q=rng.uniform(0, 1e-4))
        n_x, n_hat, k = int(rng.integers(1, 8000)), float(rng.integers(0, 400)), float(rng.uniform(1, 4))
        n_max, t_pred = int(rng.integers(1, 800)), float(rng.uniform(0, 1e-3))
        amax = float(rng.choice([0.0, 0.5, 0.95]))
        n_w = orc.pessimistic_length(n_hat, k, n_max)
        w0 = orc.wcet(coef["a"], coef["b"], coef["c"], coef["p"], coef["q"], n_x, 0.0, max(n_w, 1))
        T = t_pred + w0 * float(rng.uniform(0.2, 1.3))
        m = tb.TimeModel(coef["a"], coef["b"], coef["c"], coef["p"], coef["q"])
        got, got_nw = tb.tb_alpha_star(m, n_x, n_hat, k, n_max, t_pred, T, amax)
        want = orc.alpha_star(coef["a"], coef["b"], coef["c"], coef["p"], coef["q"], n_x, n_hat, k,
                              n_max, t_pred, T, amax)
        assert got_nw == max(1, n_w)
        assert got == pytest.approx(want, abs=1e-9), (coef, n_x, n_hat, k, n_max, t_pred, T, amax)
        al = float(rng.uniform(0, 1))
        assert tb.tb_wcet(m, n_x, al, max(n_w, 1)) == pytest.approx(
            orc.wcet(coef["a"], coef["b"], coef["c"], coef["p"], coef["q"], n_x, al, max(n_w, 1)),
            rel=1e-12, abs=1e-15)


@pytest.mark.parametrize("kw", [dict(n_x=0), dict(n_max=0), dict(n_hat=-1.0), dict(k=0.5),
                                dict(alpha_max=1.0), dict(alpha_max=-0.1), dict(p=0.0),
                                dict(budget=float("nan")), dict(q=float("inf"))])
def test_abi_rejects_bad_inputs(tb, kw):
    args = dict(n_x=1000, n_hat=10.0, k=1.0, n_max=100, t_predict=0.0, budget=5e-3, alpha_max=0.95,
                a=0.0, b=0.0, c=0.0, p=1e-6, q=0.0)
    args.update(kw)
    m = tb.TimeModel(args["a"], args["b"], args["c"], args["p"], args["q"])
    with pytest.raises(tb.TbError) as e:
        tb.tb_alpha_star(m, args["n_x"], args["n_hat"], args["k"], args["n_max"], args["t_predict"],
                         args["budget"], args["alpha_max"])
    assert e.value.status == tb.TB_ERR_INVALID_ARG
    with pytest.raises(tb.TbError):
        tb.tb_wcet(m, 0, 0.5, 10)
