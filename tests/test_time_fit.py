"""Profiling-based fitting of the time model (Eq. 6a / 6b by least squares).

Oracle pins: hand-solved fits, exact recovery of a polynomial, the
least-squares solution solved again in exact rational arithmetic (normal
equations with Fractions), and the defining property of least squares (the
residual is orthogonal to every column). The C ABI (tb_fit_time_model;
host code, no GPU) is then checked against the oracle.
"""
from fractions import Fraction

import numpy as np
import pytest

from oracle import timebill_oracle as orc


def _exact_ls(x, t, degree):
    """Least squares in exact arithmetic: the normal equations V^T V c = V^T t
    solved by Gauss-Jordan elimination over the rationals."""
    xs = [Fraction(v) for v in x]
    ts = [Fraction(v) for v in t]
    cols = [[xi ** k for xi in xs] for k in range(degree, -1, -1)]
    n = degree + 1
    M = [[sum(a * b for a, b in zip(cols[i], cols[j])) for j in range(n)] +
         [sum(a * b for a, b in zip(cols[i], ts))] for i in range(n)]
    for c in range(n):
        piv = next(r for r in range(c, n) if M[r][c] != 0)
        M[c], M[piv] = M[piv], M[c]
        M[c] = [v / M[c][c] for v in M[c]]
        for r in range(n):
            if r != c and M[r][c] != 0:
                f = M[r][c]
                M[r] = [a - f * b for a, b in zip(M[r], M[c])]
    return [M[i][n] for i in range(n)]


def test_oracle_hand_line():
    # (0,1) (1,3) (2,2): mean x 1, mean t 2, Sxt = 1, Sxx = 2 -> p = 1/2, q = 3/2;
    # fitted 1.5, 2, 2.5 -> |err|/t = 1/2, 1/3, 1/4
    coef, mape = orc.fit_time_model([0, 1, 2], [1, 3, 2], 1)
    assert coef == pytest.approx([0.5, 1.5], abs=1e-14)
    assert mape == pytest.approx(100.0 * (0.5 + 1 / 3 + 0.25) / 3, abs=1e-12)


def test_oracle_hand_quadratic():
    # three points determine the parabola t = x^2 - 2x + 3 exactly
    coef, mape = orc.fit_time_model([1, 2, 3], [2, 3, 6], 2)
    assert coef == pytest.approx([1.0, -2.0, 3.0], abs=1e-12)
    assert mape == pytest.approx(0.0, abs=1e-12)


def test_oracle_recovers_the_paper_scale_model():
    # prefill over N_x in [0, 32768] and decode steps over N_kv in the same range
    x = np.arange(0, 32769, 1024, dtype=np.float64)
    a, b, c = 3e-12, 2e-7, 1e-3
    coef, mape = orc.fit_time_model(x, a * x * x + b * x + c, 2)
    assert coef == pytest.approx([a, b, c], rel=1e-6)
    assert mape < 1e-7
    coef, mape = orc.fit_time_model(x, 4e-9 * x + 2.5e-5, 1)
    assert coef == pytest.approx([4e-9, 2.5e-5], rel=1e-9)
    assert mape < 1e-9


@pytest.mark.parametrize("degree", [1, 2])
@pytest.mark.parametrize("seed", range(3))
def test_oracle_matches_exact_rational_least_squares(degree, seed):
    rng = np.random.default_rng(seed)
    x = rng.integers(0, 50, 12)
    x[:3] = [0, 7, 31]  # at least three distinct abscissae
    t = rng.integers(1, 1000, 12)
    want = [float(v) for v in _exact_ls(x.tolist(), t.tolist(), degree)]
    coef, mape = orc.fit_time_model(x, t, degree)
    assert coef == pytest.approx(want, rel=1e-9, abs=1e-12)
    fit = np.polyval(want, x.astype(np.float64))
    assert mape == pytest.approx(100.0 * np.mean(np.abs(fit - t) / t), rel=1e-9)


@pytest.mark.parametrize("degree", [1, 2])
def test_oracle_residual_is_orthogonal(degree):
    rng = np.random.default_rng(7)
    x = np.sort(rng.uniform(0, 32768, 40))
    t = 1e-6 * x + 1e-3 + rng.normal(0, 1e-4, 40) + 1e-3
    coef, _ = orc.fit_time_model(x, t, degree)
    r = np.polyval(coef, x) - t
    for k in range(degree + 1):
        col = x ** k
        assert abs(col @ r) <= 1e-9 * np.linalg.norm(col) * np.linalg.norm(t)


# ---------------------------------------------------------------------------
# the C ABI against the oracle (host code: runs without a GPU)
# ---------------------------------------------------------------------------

@pytest.fixture(scope="module")
def tb():
    from paper_2512_21859_gb300 import build, binding
    build.build()
    binding.load()
    return binding


@pytest.mark.parametrize("degree", [1, 2])
@pytest.mark.parametrize("seed", range(4))
def test_abi_matches_oracle(tb, degree, seed):
    rng = np.random.default_rng(200 + seed)
    for _ in range(10):
        m = int(rng.integers(degree + 1, 60))
        x = rng.uniform(0, float(rng.choice([1.0, 4096.0, 32768.0, 131072.0])), m)
        x[: degree + 1] = np.arange(degree + 1) * 3.0 + 1.0
        t = (rng.uniform(0, 1e-11) * x * x * (degree == 2) + rng.uniform(1e-9, 1e-6) * x
             + rng.uniform(1e-5, 1e-3)) * rng.uniform(0.9, 1.1, m)
        got, gmape = tb.tb_fit_time_model(x, t, degree)
        want, wmape = orc.fit_time_model(x, t, degree)
        # compare the fitted times (well conditioned) and the MAPE
        np.testing.assert_allclose(np.polyval(got, x), np.polyval(want, x), rtol=1e-9)
        assert gmape == pytest.approx(wmape, rel=1e-9, abs=1e-12)


def test_abi_hand_examples(tb):
    coef, mape = tb.tb_fit_time_model([0.0, 1.0, 2.0], [1.0, 3.0, 2.0], 1)
    assert coef == pytest.approx([0.5, 1.5], abs=1e-14)
    assert mape == pytest.approx(100.0 * (0.5 + 1 / 3 + 0.25) / 3, abs=1e-12)
    coef, mape = tb.tb_fit_time_model([1.0, 2.0, 3.0], [2.0, 3.0, 6.0], 2)
    assert coef == pytest.approx([1.0, -2.0, 3.0], abs=1e-12)


@pytest.mark.parametrize("x,t,degree", [
    ([1.0, 2.0], [1.0, 2.0], 2),             # fewer points than coefficients
    ([1.0, 1.0, 1.0], [1.0, 2.0, 3.0], 1),   # one distinct abscissa
    ([1.0, 2.0, 2.0], [1.0, 2.0, 3.0], 2),   # two distinct abscissae for three coefficients
    ([1.0, 2.0, 3.0], [1.0, 0.0, 3.0], 1),   # a non-positive time
    ([1.0, float("nan"), 3.0], [1.0, 2.0, 3.0], 1),
    ([1.0, 2.0, 3.0], [1.0, 2.0, float("inf")], 1),
    ([1.0, 2.0, 3.0, 4.0], [1.0, 2.0, 3.0, 4.0], 3),
    ([1.0, 2.0, 3.0], [1.0, 2.0, 3.0], 0),
])
def test_abi_rejects_bad_inputs(tb, x, t, degree):
    with pytest.raises(tb.TbError) as e:
        tb.tb_fit_time_model(x, t, degree)
    assert e.value.status == tb.TB_ERR_INVALID_ARG


def test_bench_fit_report(tb):
    # the bench's report of a fit: exact Eq. 6b data gives back p and q with
    # no error on the fitted or the held-out points
    import bench
    x = list(range(1024, 32769, 1024))
    t = [0.0005 * n + 4.0 for n in x]
    rep = bench._fit_report(tb, x, t, 1)
    assert rep["p_us_per_token"] == pytest.approx(0.0005) and rep["q_us"] == pytest.approx(4.0)
    assert rep["mape_pct"] < 1e-9 and rep["holdout_mape_pct"] < 1e-9
    assert len(rep["points"]) == len(x)
    rep = bench._fit_report(tb, x, [1e-9 * n * n + 0.001 * n + 2.0 for n in x], 2)
    assert rep["a_us_per_token2"] == pytest.approx(1e-9, rel=1e-6)
