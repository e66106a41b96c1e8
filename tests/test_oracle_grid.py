"""Oracle pins for a general permissible set P (Sec. 5 and App. E define the DP and
the interval quantities for any sorted P; here P spans X: first = min x,
last = max x).  Checked against brute force over all codebooks drawn from P, the
per-entry definitions, a hand-computed case and the P = X special case."""
import itertools

import numpy as np
import pytest

from paper_2608_18147_gb300 import workloads


def uniform_grid(x, n):
    g = np.linspace(float(x.min()), float(x.max()), n).astype(np.float32)
    g[0], g[-1] = x.min(), x.max()
    return np.unique(g)


def test_grid_equal_to_unique_values_is_the_plain_histogram(oracle_mod):
    x = workloads.signed_lognormal(500, 2)
    a = oracle_mod.Hist(x).arrays()
    b = oracle_mod.Hist(x, np.unique(x)).arrays()
    for k in a:
        np.testing.assert_array_equal(a[k], b[k])
    ra = oracle_mod.solve_budget(x, 6, 1.5)
    rb = oracle_mod.solve_budget(x, 6, 1.5, grid=np.unique(x))
    assert ra["lam"] == rb["lam"] and ra["mse"] == rb["mse"]
    np.testing.assert_array_equal(ra["Q"], rb["Q"])


def test_grid_hand_computed_case(oracle_mod):
    # X = {0, 0.25, 1}, P = {0, 0.5, 1}: Q = P puts 0.25 in (0, 0.5]: MSE = 0.25 * 0.25,
    # up-probability 0.5 -> H(I,B) over intervals (0,0.5] (first: down mass 1 + 0.5) and (0.5,1]
    x = np.array([0.0, 0.25, 1.0], np.float32)
    H = oracle_mod.Hist(x, np.array([0.0, 0.5, 1.0], np.float32))
    arr = H.arrays()
    np.testing.assert_array_equal(arr["w"], [1, 1, 1])
    np.testing.assert_array_equal(arr["N"], [0, 1, 2, 3])
    mse, hs, hx = H.eval_idx([0, 1, 2])
    assert mse == 0.0625
    h = lambda y: 0.0 if y == 0 else -y * np.log2(y)
    # first interval (0, 0.5] holds 0.25 (U = D = 0.5) plus x = 0 (down); second holds 1 (U = 1)
    assert hs == pytest.approx(h(0.5 / 3) + h(1.5 / 3) + h(1.0 / 3) + h(0.0), rel=1e-15)
    # Xhat: 0 w.p. (1 + 0.5)/3, 0.5 w.p. 0.5/3, 1 w.p. 1/3
    assert hx == pytest.approx(h(1.5 / 3) + h(0.5 / 3) + h(1.0 / 3), rel=1e-15)


@pytest.mark.parametrize("seed", [0, 1])
def test_grid_metrics_match_the_per_entry_definitions(oracle_mod, seed):
    x = workloads.student_t(400, seed, scale=1.0)
    g = uniform_grid(x, 33)
    H = oracle_mod.Hist(x, g)
    rng = np.random.default_rng(seed)
    for _ in range(5):
        inner = np.sort(rng.choice(np.arange(1, g.size - 1), size=5, replace=False))
        a = np.concatenate([[0], inner, [g.size - 1]])
        got = H.eval_idx(a)
        want = oracle_mod.eval_direct(x, g[a].astype(np.float64))
        np.testing.assert_allclose(got, want, rtol=1e-12)


@pytest.mark.parametrize("lam", [0.0, 0.05, 0.5])
def test_grid_dp_equals_brute_force_over_the_grid(oracle_mod, lam):
    """eq. apx_rec over P: the DP's best surrogate Lagrangian equals the minimum over every
    codebook drawn from P that contains both endpoints (at most s values)."""
    x = workloads.signed_lognormal(60, 7)
    g = uniform_grid(x, 10)
    H = oracle_mod.Hist(x, g)
    s = 5
    lp = lam * H.norm2
    r = H.apx_dp(s, lp, tables=False)
    best = np.inf
    for m in range(2, s + 1):
        for inner in itertools.combinations(range(1, g.size - 1), m - 2):
            a = [0, *inner, g.size - 1]
            mse, hs, _ = H.eval_idx(a)
            best = min(best, mse + lp * hs)
    assert r["best"] == pytest.approx(best, rel=1e-12, abs=1e-300)
    mse, hs, _ = H.eval_idx(r["Q_idx"])
    assert mse + lp * hs == pytest.approx(best, rel=1e-12, abs=1e-300)


def test_grid_rejects_sets_that_do_not_span_x(oracle_mod):
    x = np.array([1.0, 2.0, 3.0], np.float32)
    for P in ([1.5, 3.0], [1.0, 2.5], [1.0, 3.0, 2.0], [1.0, 1.0, 3.0]):
        with pytest.raises(oracle_mod.OracleError):
            oracle_mod.Hist(x, np.array(P, np.float32))
