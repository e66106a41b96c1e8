"""Oracle pins for a general permissible set P (Sec. 5 and App. E define the DP and
the interval quantities for any sorted P with p_1 <= x_1 and p_last >= x_d; the first
value ranges over L = {a : p_a <= x_1}, the last over R = {b : p_b >= x_d}).  Checked
against brute force over all codebooks drawn from P, the per-entry definitions, a
hand-computed case, the App. F.1 example and the P = X special case."""
import itertools
from fractions import Fraction

import numpy as np
import pytest

from conftest import read_golden

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


def wide_grid(x, n, below, above):
    """n evenly spaced values from min x - below to max x + above, with min x and
    max x themselves in the set (so L and R hold several values)."""
    lo, hi = float(x.min()), float(x.max())
    g = np.linspace(lo - below, hi + above, n).astype(np.float32)
    return np.unique(np.concatenate([g, np.array([lo, hi], np.float32)]))


def test_grid_first_and_last_value_sets(oracle_mod):
    x = np.array([1.0, 2.0, 2.0, 3.0], np.float32)
    H = oracle_mod.Hist(x, np.array([0.0, 0.5, 1.0, 2.0, 3.0, 4.0], np.float32))
    assert (H.nL, H.nR) == (3, 2)
    assert (oracle_mod.Hist(x).nL, oracle_mod.Hist(x).nR) == (1, 1)
    H = oracle_mod.Hist(x, np.array([-1.0, 2.5, 5.0], np.float32))   # neither end in X
    assert (H.nL, H.nR) == (1, 1)
    np.testing.assert_array_equal(H.arrays()["w"], [0, 3, 1])
    # the first value's own mass n_a is zero when p_a < x_1: x_1 itself rounds within (p_a, p_b]
    mse, hs, hx = H.eval_idx([0, 1, 2])
    assert mse == pytest.approx((2.5 - 1) * (1 + 1) + 2 * (2.5 - 2) * (2 + 1) + (5 - 3) * (3 - 2.5), rel=1e-15)


@pytest.mark.parametrize("lam", [0.0, 0.02, 0.3])
@pytest.mark.parametrize("seed", [3, 4])
def test_grid_with_several_end_candidates_equals_brute_force(oracle_mod, lam, seed):
    """eqs. apx_base (min over a in L) and apx_final (min over j in R) against every
    spanning codebook drawn from a grid that extends past X on both sides, scored by
    the per-entry definitions (no prefix sums)."""
    x = workloads.signed_lognormal(48, seed)
    span = float(x.max() - x.min())
    g = wide_grid(x, 11, 0.3 * span, 0.25 * span)
    H = oracle_mod.Hist(x, g)
    assert H.nL >= 2 and H.nR >= 2 and g.size <= 16
    s = 4
    lp = lam * H.norm2
    bf = oracle_mod.brute_grid(x, g, s, lp, np.inf)
    r = H.apx_dp(s, lp, tables=False)
    assert r["best"] == pytest.approx(bf["surrogate"], rel=1e-12, abs=1e-300)
    a = r["Q_idx"]
    assert a[0] < H.nL and a[-1] >= H.p - H.nR
    mse, hs, hx = H.eval_idx(a)
    dm, ds, dx = oracle_mod.eval_direct(x, g[a].astype(np.float64))
    np.testing.assert_allclose([mse, hs, hx], [dm, ds, dx], rtol=1e-12, atol=1e-300)
    # the optimal DP of Sec. 4 / App. E reaches the true-Lagrangian brute-force optimum
    best, qo = H.opt_dp(s, lp)
    assert best == pytest.approx(bf["true"], rel=1e-12, abs=1e-300)
    dm, _, dx = oracle_mod.eval_direct(x, g[qo].astype(np.float64))
    assert dm + lp * dx == pytest.approx(bf["true"], rel=1e-12, abs=1e-300)
    # exactly s values (the outer minimum at i = s only)
    r = H.apx_dp(s, lp, exact_s=True, tables=False)
    assert r["m"] == s


def test_brute_grid_on_the_unique_values_is_the_plain_brute_force(oracle_mod):
    x = workloads.normal(40, 5)[:12]
    g = np.unique(x)
    for lp in (0.0, 0.01 * float(np.sum(x.astype(np.float64) ** 2))):
        a = oracle_mod.brute(x, 5, lp, 1.5)
        b = oracle_mod.brute_grid(x, g, 5, lp, 1.5)
        for k in ("surrogate", "true", "mse_surr_budget", "mse_opt_budget_minus1", "mse_min"):
            assert a[k] == b[k]


def test_appF1_example_through_the_grid_dp(oracle_mod):
    """App. F.1: X = half 0s, half 2s, P = (0,1,2,3,4), s = 2.  R = {2, 3, 4}; the three
    codebooks of the table come out of eval_idx with the printed vNMSEs, no multiplier
    makes B = {0, 3} the Lagrangian optimum, and B is the hard-budget optimum at b = 0.95."""
    g = read_golden("appF1_lagrangian_gap.txt")
    d = 64
    x = np.array([0.0] * (d // 2) + [2.0] * (d // 2), np.float32)
    P = np.array([0, 1, 2, 3, 4], np.float32)
    H = oracle_mod.Hist(x, P)
    assert (H.nL, H.nR) == (1, 3)
    vn = {}
    for row in g["row"]:
        qs, _, _, v = [t.strip() for t in row.split(";")]
        a = [int(float(t)) for t in qs.split()]
        mse, hs, hx = H.eval_idx(a)
        assert mse / H.norm2 == pytest.approx(float(Fraction(v)), abs=1e-15)
        assert hs == pytest.approx(hx, rel=1e-14)
        vn[a[1]] = (mse, hx)
    for lam in np.geomspace(1e-3, 1e3, 121):
        r = H.apx_dp(2, lam * H.norm2, tables=False)
        assert list(r["Q_idx"]) in ([0, 2], [0, 4])
        J = {b: m + lam * H.norm2 * h for b, (m, h) in vn.items()}
        assert r["best"] == pytest.approx(min(J.values()), rel=1e-13)
    bf = oracle_mod.brute_grid(x, P, 2, 0.0, 0.95)
    assert bf["masks"][2] == 0b01001                     # {0, 3}
    assert bf["mse_surr_budget"] / H.norm2 == pytest.approx(0.5, abs=1e-15)
