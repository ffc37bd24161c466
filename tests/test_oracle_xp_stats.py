"""Pins of the oracle's cross-play matrix consumers (no GPU).

What fixes the values: App. B "Upper bound estimation" (a teammate's recorded bound is
raised to any cross-play score that exceeds it), Sec. 3 (returns are reported relative to
the best response's; J_AHT is the expectation over the evaluation teammates), App. A
ROTATE (cooperative regret = best-response return minus the ego's return) and App. A
BRDiv (matched teammate/best-response returns up, mismatched cross-play down).
"""
import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def test_worked_3x3_by_hand():
    # rows: policies in the ego seat, columns: teammates
    xp = np.array([[3, 1, 0], [2, 4, 1], [0, 0, 2]], np.float32)
    r = oracle.xp_stats(xp)
    # column maxima
    assert r["upper"].tolist() == [3.0, 4.0, 2.0]
    np.testing.assert_array_equal(r["regret"], [[0, 3, 2], [1, 0, 1], [3, 4, 0]])
    np.testing.assert_allclose(r["norm"], [[1, 1 / 4, 0], [2 / 3, 1, 1 / 2], [0, 0, 1]], rtol=1e-15)
    np.testing.assert_allclose(r["j_aht"], [4 / 3, 7 / 3, 2 / 3], rtol=1e-15)
    np.testing.assert_allclose(r["j_norm"], [(1 + 1 / 4) / 3, (2 / 3 + 1 + 1 / 2) / 3, 1 / 3], rtol=1e-15)
    assert r["max_regret"].tolist() == [3.0, 1.0, 4.0]
    assert r["worst"].tolist() == [1, 0, 1]  # row 1: regrets 1, 0, 1 -> the lower index
    # matched mean 9/3 = 3, mismatched mean (1 + 0 + 2 + 1 + 0 + 0) / 6 = 2/3
    assert r["brdiv"] == pytest.approx(3 - 2 / 3, rel=1e-15)


def test_upper_bound_refinement_keeps_higher_prior():
    rng = np.random.default_rng(1)
    xp = rng.uniform(0, 10, (5, 7)).astype(np.float32)
    prior = np.array([100, -np.inf, 0, 5, 20, -3, 9.5])
    r = oracle.xp_stats(xp, prior)
    np.testing.assert_array_equal(r["upper"], np.maximum(prior, xp.max(axis=0).astype(np.float64)))
    # a second pass with the refined bounds changes nothing
    r2 = oracle.xp_stats(xp, r["upper"])
    np.testing.assert_array_equal(r2["upper"], r["upper"])
    # a NaN bound is never exceeded, so it stays NaN (strict comparison)
    r3 = oracle.xp_stats(xp, np.full(7, np.nan))
    assert np.isnan(r3["upper"]).all()


@pytest.mark.parametrize("shape", [(1, 1), (4, 9), (16, 16), (64, 64), (33, 17)])
def test_invariants_random(shape):
    rng = np.random.default_rng(shape[0] * 100 + shape[1])
    xp = rng.uniform(0.1, 3.0, shape).astype(np.float32)
    r = oracle.xp_stats(xp)
    col_max = xp.max(axis=0).astype(np.float64)
    assert (r["regret"] >= 0).all()
    # the best row of each column has zero regret and normalised return exactly 1
    best = xp.argmax(axis=0)
    assert (r["regret"][best, np.arange(shape[1])] == 0).all()
    assert (r["norm"][best, np.arange(shape[1])] == 1).all()
    assert (r["norm"] <= 1).all() and (r["norm"] > 0).all()
    np.testing.assert_allclose(r["norm"] * col_max, xp, rtol=1e-15)
    np.testing.assert_allclose(r["j_aht"], xp.astype(np.float64).mean(axis=1), rtol=1e-14)
    np.testing.assert_allclose(r["j_norm"], (xp / col_max).mean(axis=1), rtol=1e-6)
    np.testing.assert_array_equal(r["max_regret"], r["regret"].max(axis=1))
    np.testing.assert_array_equal(r["worst"], r["regret"].argmax(axis=1))  # first maximum
    if shape[0] == shape[1]:
        n = shape[0]
        x = xp.astype(np.float64)
        tr = np.trace(x)
        want = tr / n - ((x.sum() - tr) / (n * (n - 1)) if n > 1 else 0.0)
        assert r["brdiv"] == pytest.approx(want, rel=1e-12, abs=1e-12)
    else:
        assert r["brdiv"] is None


def test_brdiv_special_cases():
    n = 6
    a, b = 5.0, 1.5
    m = np.full((n, n), b, np.float32)
    np.fill_diagonal(m, a)
    assert oracle.xp_stats(m)["brdiv"] == a - b
    assert oracle.xp_stats(np.full((n, n), 2.5, np.float32))["brdiv"] == 0.0
    assert oracle.xp_stats(np.array([[7.25]], np.float32))["brdiv"] == 7.25
    # relabelling teammates and their best responses together leaves it unchanged
    rng = np.random.default_rng(3)
    x = rng.uniform(0, 1, (n, n)).astype(np.float32)
    p = rng.permutation(n)
    assert oracle.xp_stats(x[p][:, p])["brdiv"] == pytest.approx(oracle.xp_stats(x)["brdiv"], rel=1e-14)
    # a mismatched row raises the cross-play term and lowers the objective
    y = x.copy()
    y[0, 1] += 1.0
    assert oracle.xp_stats(y)["brdiv"] < oracle.xp_stats(x)["brdiv"]


def test_nonpositive_bound_gives_nan_normalisation():
    xp = np.array([[0, 2], [0, 1]], np.float32)  # teammate 0: every return 0
    r = oracle.xp_stats(xp)
    assert r["upper"].tolist() == [0.0, 2.0]
    assert np.isnan(r["norm"][:, 0]).all() and not np.isnan(r["norm"][:, 1]).any()
    assert np.isnan(r["j_norm"]).all()
    np.testing.assert_array_equal(r["regret"], [[0, 0], [0, 1]])
    assert r["worst"].tolist() == [0, 1]
