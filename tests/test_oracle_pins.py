"""Pins of the CPU oracle to what the paper and the mathematics fix.

Every check here compares the oracle with something other than itself: values
printed in the paper (tests/golden), the per-entry definitions, brute-force
enumeration, closed forms, the entropy sandwich and one-bit lemma of Sec. 5,
the lambda = 0 reduction to ASQ, and metamorphic invariances.
"""
import math
from fractions import Fraction

import numpy as np
import pytest

from conftest import read_golden
from paper_2608_18147_gb300 import workloads


def frac(s):
    return Fraction(s)


def hbits(fr):
    return -float(fr) * math.log2(float(fr)) if fr > 0 else 0.0


# ----------------------------------------------------------- paper examples

def test_sec3_worked_example(oracle_mod):
    g = read_golden("sec3_worked_example.txt")
    x = np.array(g["x"][0].split(), np.float32)
    Q = [float(t) for t in g["Q"][0].split()]
    f = [frac(t) for t in g["freq"][0].split()]
    mse, hs, hx = oracle_mod.eval_direct(x, Q)
    # frequencies printed in the paper -> entropy; and the paper's rounded value
    assert hx == pytest.approx(sum(hbits(t) for t in f), rel=1e-14)
    assert abs(hx - float(g["H_approx"][0])) < float(g["H_tol"][0])
    # the middle entry is rounded down w.p. 9/10: variance (10-1)(1-0) of Sec. 2
    pdown = frac(g["p_down_middle"][0])
    assert mse == pytest.approx(float(pdown * (1 - 0) ** 2 + (1 - pdown) * (10 - 1) ** 2), rel=1e-14)
    # one interval: the surrogate equals the true entropy (B determines Xhat)
    assert hs == pytest.approx(hx, rel=1e-14)
    # the same numbers through the prefix-sum path (Q subset of X)
    H = oracle_mod.Hist(x)
    assert H.eval_idx([0, 2]) == pytest.approx((mse, hs, hx), rel=1e-14)


def test_appF1_lagrangian_gap_table(oracle_mod):
    g = read_golden("appF1_lagrangian_gap.txt")
    d = 64
    x = np.array([0.0] * (d // 2) + [2.0] * (d // 2), np.float32)
    norm2 = float(np.sum(x.astype(np.float64) ** 2))
    for row in g["row"]:
        qs, dist, H3, vn = [t.strip() for t in row.split(";")]
        Q = [float(t) for t in qs.split()]
        mse, hs, hx = oracle_mod.eval_direct(x, Q)
        dist = [frac(t) for t in dist.split()]
        assert hx == pytest.approx(sum(hbits(t) for t in dist), rel=1e-14)
        assert round(hx, 3) == pytest.approx(float(H3), abs=1e-12)
        assert mse / norm2 == pytest.approx(float(frac(vn)), abs=1e-15)
        assert hs == pytest.approx(hx, rel=1e-14)  # two values: one interval
    for row in g["H6"]:
        qs, h6 = [t.strip() for t in row.split(";")]
        _, _, hx = oracle_mod.eval_direct(x, [float(t) for t in qs.split()])
        assert abs(hx - float(h6)) < 5e-7
    # the two multiplier thresholds printed with the table
    hA = oracle_mod.eval_direct(x, [0, 4])[2]
    hB = oracle_mod.eval_direct(x, [0, 3])[2]
    hC = oracle_mod.eval_direct(x, [0, 2])[2]
    assert 0.5 / (hC - hB) > float(g["lambda_gt"][0])
    assert 0.5 / (hB - hA) < float(g["lambda_lt"][0])


def test_appF2_nonadjacent_example(oracle_mod):
    g = read_golden("appF2_nonadjacent.txt")
    d = 99
    x = np.array([0.0] * (d // 3) + [1.0] * (d // 3) + [2.0] * (d // 3), np.float32)
    norm2 = float(np.sum(x.astype(np.float64) ** 2))
    assert norm2 / d == pytest.approx(float(frac(g["norm2_per_d"][0])), rel=1e-14)
    H = oracle_mod.Hist(x)
    assert H.p == 3
    for row in g["row"]:
        qs, dist, Hs, mpd, vn = [t.strip() for t in row.split(";")]
        Q = [float(t) for t in qs.split()]
        mse, hs, hx = oracle_mod.eval_direct(x, Q)
        dist = [frac(t) for t in dist.split()]
        assert hx == pytest.approx(sum(hbits(t) for t in dist), rel=1e-14)
        Hexp = math.log2(3) if Hs.split()[1] == "log2(3)" else float(Hs.split()[1])
        assert hx == pytest.approx(Hexp, rel=1e-14)
        assert mse / d == pytest.approx(float(frac(mpd.split()[1])), abs=1e-15)
        assert mse / norm2 == pytest.approx(float(frac(vn.split()[1])), abs=1e-15)
        # weighted-histogram path agrees with the per-entry definitions
        idx = [int(np.searchsorted(H.arrays()["v"], q)) for q in Q]
        assert H.eval_idx(idx) == pytest.approx((mse, hs, hx), rel=1e-13, abs=1e-13)


# --------------------------------------------- prefix sums and interval costs

def test_prefix_sums_exact(oracle_mod):
    rng = np.random.default_rng(3)
    x = rng.choice(np.float32([-2.5, -1.0, -0.0, 0.0, 0.375, 1.0, 3.0, 7.25]), 200)
    H = oracle_mod.Hist(x)
    a = H.arrays()
    vals = sorted(set(float(t) for t in x))
    assert list(a["v"]) == vals  # -0.0 and 0.0 are one value
    cnt = [int(np.sum(x == np.float32(v))) for v in vals]
    assert list(a["w"]) == cnt
    N = S = S2 = Fraction(0)
    for t, v in enumerate(vals):
        assert a["N"][t] == N
        assert Fraction(a["S_hi"][t]) + Fraction(a["S_lo"][t]) == S
        assert Fraction(a["S2_hi"][t]) + Fraction(a["S2_lo"][t]) == S2
        N += cnt[t]
        S += cnt[t] * Fraction(v)
        S2 += cnt[t] * Fraction(v) ** 2
    assert H.norm2 == float(S2)


def test_pair_costs_match_definition(oracle_mod):
    """App. E prefix-difference C, U, D equal the Sec. 5 sums over X_{k,j}."""
    rng = np.random.default_rng(4)
    x = np.round(rng.standard_normal(300) * 4) / 4  # many duplicates
    x = x.astype(np.float32)
    H = oracle_mod.Hist(x)
    v = H.arrays()["v"].astype(np.float64)
    xs = x.astype(np.float64)
    for _ in range(200):
        k, j = sorted(rng.choice(H.p, 2, replace=False))
        sel = xs[(xs > v[k]) & (xs <= v[j])]
        C = np.sum((v[j] - sel) * (sel - v[k]))
        U = np.sum((sel - v[k]) / (v[j] - v[k]))
        D = np.sum((v[j] - sel) / (v[j] - v[k]))
        c, u, dd = H.pair(k, j)
        assert c == pytest.approx(C, rel=1e-12, abs=1e-12)
        assert u == pytest.approx(U, rel=1e-12, abs=1e-12)
        assert dd == pytest.approx(D, rel=1e-12, abs=1e-12)
        assert u + dd == pytest.approx(sel.size, rel=1e-14)


def test_pair_costs_exact_rational(oracle_mod):
    """Exact rational check: the binary128 path returns correctly rounded C."""
    rng = np.random.default_rng(5)
    x = (rng.standard_normal(64) * 3).astype(np.float32)
    H = oracle_mod.Hist(x)
    v = [Fraction(float(t)) for t in H.arrays()["v"]]
    for k, j in [(0, 63), (5, 6), (10, 40), (62, 63), (0, 1)]:
        Cx = sum((v[j] - v[t]) * (v[t] - v[k]) for t in range(k + 1, j + 1))
        c, u, dd = H.pair(k, j)
        assert c == float(Cx)


# ---------------------------------------------------- entropy and evaluation

def _random_codebook(rng, p, m):
    inner = np.sort(rng.choice(np.arange(1, p - 1), m - 2, replace=False)) if m > 2 else []
    return np.concatenate([[0], inner, [p - 1]]).astype(np.int64)


@pytest.mark.parametrize("seed", range(6))
def test_eval_prefix_equals_direct_and_sandwich(oracle_mod, seed):
    rng = np.random.default_rng(seed)
    x = (np.round(rng.standard_normal(500) * 6) / 6).astype(np.float32)
    H = oracle_mod.Hist(x)
    v = H.arrays()["v"].astype(np.float64)
    for m in (2, 3, 5, 9):
        a = _random_codebook(rng, H.p, m)
        e1 = H.eval_idx(a)
        e2 = oracle_mod.eval_direct(x, v[a])
        assert e1 == pytest.approx(e2, rel=1e-11, abs=1e-11)
        mse, hs, hx = e1
        # eq. apx_entropy_sandwich: H(Xhat) <= H(I,B) <= H(Xhat) + 1
        assert hx <= hs + 1e-12
        assert hs <= hx + 1.0 + 1e-12


def test_s2_closed_form(oracle_mod):
    """s = 2: Q = {x_1, x_d} and H(I,B) = H(Xhat) (one interval)."""
    x = workloads.normal(300, seed=7)
    H = oracle_mod.Hist(x)
    lp = 0.3 * H.norm2
    r = H.apx_dp(2, lp)
    assert list(r["Q_idx"]) == [0, H.p - 1]
    mse, hs, hx = H.eval_idx(r["Q_idx"])
    xs = x.astype(np.float64)
    assert mse == pytest.approx(np.sum((xs.max() - xs) * (xs - xs.min())), rel=1e-12)
    assert hs == pytest.approx(hx, rel=1e-13)
    assert r["best"] == pytest.approx(mse + lp * hs, rel=1e-13)


# ----------------------------------------------------- DPs vs brute force

def _tiny(seed, d=14, dup=True):
    rng = np.random.default_rng(seed)
    if dup:
        x = rng.choice((rng.standard_normal(9) * 2).astype(np.float32), d)
    else:
        x = (rng.standard_normal(d) * 2).astype(np.float32)
    return x


@pytest.mark.parametrize("seed", range(8))
@pytest.mark.parametrize("lam", [0.0, 0.01, 0.2, 3.0])
def test_apx_dp_equals_bruteforce_surrogate(oracle_mod, seed, lam):
    """Eq. apx_rec is an exact DP for MSE + lambda' H(I,B) over spanning Q subset of X."""
    x = _tiny(seed, d=12 + seed % 3, dup=seed % 2 == 0)
    H = oracle_mod.Hist(x)
    for s in (2, 3, 4, 6):
        lp = lam * H.norm2
        r = H.apx_dp(s, lp)
        b = oracle_mod.brute(x, s, lp, 10.0)
        assert r["best"] == pytest.approx(b["surrogate"], rel=1e-12, abs=1e-12)
        mse, hs, hx = H.eval_idx(r["Q_idx"])
        assert mse + lp * hs == pytest.approx(r["best"], rel=1e-12, abs=1e-12)
        assert r["m"] <= s


@pytest.mark.parametrize("seed", range(8))
@pytest.mark.parametrize("lam", [0.0, 0.05, 0.5, 4.0])
def test_opt_dp_equals_bruteforce_true(oracle_mod, seed, lam):
    """Sec. 4's DP minimises the true Lagrangian MSE + lambda' H(Xhat)."""
    x = _tiny(100 + seed, d=12 + seed % 3, dup=seed % 2 == 1)
    H = oracle_mod.Hist(x)
    for s in (2, 3, 5):
        lp = lam * H.norm2
        best, Q = H.opt_dp(s, lp)
        b = oracle_mod.brute(x, s, lp, 10.0)
        assert best == pytest.approx(b["true"], rel=1e-12, abs=1e-12)
        mse, hs, hx = H.eval_idx(Q)
        assert mse + lp * hx == pytest.approx(best, rel=1e-12, abs=1e-12)


@pytest.mark.parametrize("seed", range(6))
def test_lambda_zero_is_asq(oracle_mod, seed):
    """lambda = 0 is classic ASQ (Sec. 3): approx DP = eq. asqdp = brute-force min MSE."""
    x = _tiny(200 + seed, d=13)
    H = oracle_mod.Hist(x)
    for s in (2, 3, 4, 7):
        a = H.apx_dp(s, 0.0)["best"]
        q = H.asq_dp(s)
        b = oracle_mod.brute(x, s, 0.0, 100.0)["mse_min"]
        assert a == pytest.approx(q, rel=1e-12, abs=1e-12)
        assert a == pytest.approx(b, rel=1e-12, abs=1e-12)
    # larger input: apx DP at lambda=0 equals the ASQ recurrence
    x = workloads.signed_lognormal(200, seed)
    H = oracle_mod.Hist(x)
    assert H.apx_dp(6, 0.0)["best"] == pytest.approx(H.asq_dp(6), rel=1e-12)


@pytest.mark.parametrize("seed", range(10))
def test_one_bit_lemma_bruteforce(oracle_mod, seed):
    """Sec. 5 lemma: MSE(Q_APX(b)) <= OPT(b-1) and H(Xhat) of Q_APX(b) <= b."""
    x = _tiny(300 + seed, d=14)
    for s in (3, 4, 6):
        for b in (1.25, 1.5, 2.0, 2.5):
            r = oracle_mod.brute(x, s, 0.0, b)
            if math.isfinite(r["mse_surr_budget"]):
                assert r["hx_of_surr_budget"] <= b + 1e-12
            assert r["mse_surr_budget"] <= r["mse_opt_budget_minus1"] * (1 + 1e-12) + 1e-12


@pytest.mark.parametrize("seed", range(3))
def test_lagrangian_sandwich_vs_optimal_dp(oracle_mod, seed):
    """J_true(Q_apx) <= J_surr,apx(lambda) <= J_opt(lambda) + lambda' (eq. apx_entropy_sandwich)."""
    x = workloads.normal(160, seed)
    H = oracle_mod.Hist(x)
    H.cache()
    for lam in (0.01, 0.1, 1.0):
        lp = lam * H.norm2
        r = H.apx_dp(6, lp)
        jopt, Qo = H.opt_dp(6, lp)
        mse, hs, hx = H.eval_idx(r["Q_idx"])
        assert mse + lp * hx <= r["best"] * (1 + 1e-12)
        assert r["best"] <= (jopt + lp) * (1 + 1e-12)
        assert jopt <= mse + lp * hx + 1e-9 * abs(jopt)  # the optimum is optimal


# ------------------------------------------------------------- the search

def test_search_schedule_and_selection(oracle_mod):
    x = workloads.normal(1024, 0)
    H = oracle_mod.Hist(x)
    H.cache()
    r = H.search(8, 2.0)
    tr = r["trace"]
    assert r["status"] == 0
    assert tr[0, 0] == 0.0
    # first round is the 7 geometric midpoints of [1e-8, 1e3]
    np.testing.assert_array_equal(tr[1:8, 0], oracle_mod.midpoints7(1e-8, 1e3))
    t = oracle_mod.midpoints7(1e-8, 1e3)
    assert np.allclose(np.diff(np.log(np.concatenate([[1e-8], t, [1e3]]))), math.log(1e11) / 8, rtol=1e-12)
    # H(I,B) of the exact Lagrangian minimisers is non-increasing in lambda
    order = np.argsort(tr[:, 0], kind="stable")
    hs = tr[order, 2]
    assert np.all(np.diff(hs) <= 1e-12)
    # answer = least MSE among feasible evaluated points, feasible by construction
    feas = tr[tr[:, 5] == 1]
    assert r["h_surrogate"] <= 2.0
    assert r["mse"] == feas[:, 1].min()
    assert r["mse"] == pytest.approx(H.eval_idx(r["Q_idx"])[0], rel=1e-14)


def test_search_bracket_schedule(oracle_mod):
    """Each round's 7 points are the midpoints of the bracket around the first feasible point."""
    x = workloads.signed_lognormal(800, 3)
    H = oracle_mod.Hist(x)
    H.cache()
    r = H.search(8, 2.5, rounds=4)
    tr = r["trace"]
    lo, hi = 1e-8, 1e3
    for rnd in range(4):
        pts = tr[1 + 7 * rnd: 8 + 7 * rnd]
        np.testing.assert_array_equal(pts[:, 0], oracle_mod.midpoints7(lo, hi))
        feas = np.flatnonzero(pts[:, 5] == 1)
        if feas.size:
            f = feas[0]
            lo, hi = (pts[f - 1, 0] if f > 0 else lo), pts[f, 0]
        else:
            lo = pts[6, 0]
    assert tr.shape[0] == 1 + 7 * 4


def test_search_unconstrained_budget_returns_lambda0(oracle_mod):
    x = workloads.normal(512, 1)
    H = oracle_mod.Hist(x)
    r = H.search(4, 8.0)
    assert r["lam"] == 0.0 and r["n_evaluated"] == 1
    assert r["mse"] == pytest.approx(H.asq_dp(4), rel=1e-12)


def test_search_infeasible(oracle_mod):
    x = workloads.normal(256, 2)
    H = oracle_mod.Hist(x)
    r = H.search(4, 0.0)
    assert r["status"] == oracle_mod.EINFEASIBLE


# --------------------------------------------------------------- refinement

@pytest.mark.parametrize("seed", range(3))
def test_refinement_monotone_and_bounded_by_optimum(oracle_mod, seed):
    """Sec. 6: the refined Q is never worse than the start; the optimal DP bounds it."""
    x = workloads.signed_lognormal(150, seed)
    H = oracle_mod.Hist(x)
    H.cache()
    for lam in (0.02, 0.2):
        lp = lam * H.norm2
        a = H.apx_dp(7, lp)["Q_idx"]
        rf = H.refine(a, lp, max_rounds=8, tol=0.0)
        J = rf["J"]
        assert np.all(np.diff(J) <= 1e-12 * abs(J[0]))
        jopt, _ = H.opt_dp(7, lp)
        mse, hs, hx = H.eval_idx(rf["Q_idx"])
        assert mse + lp * hx >= jopt * (1 - 1e-12)
        assert mse + lp * hx == pytest.approx(J[-1], rel=1e-12)
        assert len(rf["Q_idx"]) == len(a)  # values move, never merge


def test_refinement_colour_step_is_exact_coordinate_minimum(oracle_mod):
    """After convergence no single interior value can improve J by moving (brute force)."""
    x = workloads.normal(160, 9)
    H = oracle_mod.Hist(x)
    H.cache()
    lp = 0.02 * H.norm2
    a = H.apx_dp(12, lp)["Q_idx"]
    assert len(a) >= 9  # every colour class has members
    rf = H.refine(a, lp, max_rounds=50, tol=0.0)
    q = rf["Q_idx"]
    assert rf["rounds"] < 50

    def J(c):
        mse, hs, hx = H.eval_idx(c)
        return mse + lp * hx
    j0 = J(q)
    for l in range(1, len(q) - 1):
        for c in range(q[l - 1] + 1, q[l + 1]):
            t = q.copy()
            t[l] = c
            assert J(t) >= j0 * (1 - 1e-12)


def test_refinement_budget_guard(oracle_mod):
    x = workloads.student_t(2000, 3)
    H = oracle_mod.Hist(x)
    H.cache()
    b = 2.0
    r = H.search(8, b)
    rf = H.refine(r["Q_idx"], r["lam"] * H.norm2, budget=b, guard=True, max_rounds=5)
    assert H.eval_idx(rf["Q_idx"])[2] <= b


# ------------------------------------------------------------ metamorphic

def test_scale_by_power_of_two_is_exact(oracle_mod):
    """vNMSE is scale free (Sec. 2); c = 2^k scales every binary64 step exactly."""
    x = workloads.student_t(700, 4, scale=1.0)
    for c in (2.0 ** -20, 0.25, 8.0):
        H1, H2 = oracle_mod.Hist(x), oracle_mod.Hist((x * np.float32(c)).astype(np.float32))
        for lam in (0.0, 0.05, 0.7):
            r1 = H1.apx_dp(8, lam * H1.norm2)
            r2 = H2.apx_dp(8, lam * H2.norm2)
            np.testing.assert_array_equal(r1["Q_idx"], r2["Q_idx"])
            np.testing.assert_array_equal(r1["bp"], r2["bp"])
            assert r2["best"] == r1["best"] * c * c


def test_permutation_invariance(oracle_mod):
    x = workloads.mixture(900, 5)
    y = np.random.default_rng(1).permutation(x)
    r1 = oracle_mod.Hist(x).search(8, 2.5)
    r2 = oracle_mod.Hist(y).search(8, 2.5)
    np.testing.assert_array_equal(r1["Q_idx"], r2["Q_idx"])
    assert r1["lam"] == r2["lam"] and r1["mse"] == r2["mse"]


# ------------------------------------------------------------ quantization

def test_splitmix64_reference_outputs(oracle_mod):
    """SplitMix64 (Steele, Lea, Flood 2014) seeded with 0: first three outputs."""
    g = 0x9E3779B97F4A7C15
    outs = [oracle_mod.splitmix64((t * g) % 2 ** 64) for t in (1, 2, 3)]
    assert outs == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_unbiased_by_exact_expectation():
    """Sec. 2: a (b-x)/(b-a) + b (x-a)/(b-a) = x, in exact rationals."""
    rng = np.random.default_rng(6)
    for _ in range(200):
        a, x, b = sorted(Fraction(float(t)) for t in rng.standard_normal(3).astype(np.float32))
        if a == b:
            continue
        pu = (x - a) / (b - a)
        assert a * (1 - pu) + b * pu == x
        assert (b - x) * (x - a) == pu * (b - x) ** 2 + (1 - pu) * (a - x) ** 2  # Var, Sec. 2


def test_quantizer_decision_rule_bias_bound(oracle_mod):
    """Exact probability of rounding up under the 24-bit rule is within 2^-22 of (x-a)/(b-a)."""
    rng = np.random.default_rng(7)
    k = np.arange(2 ** 24, dtype=np.float32) * np.float32(2.0 ** -24)
    for _ in range(6):
        a, x, b = np.sort(rng.standard_normal(3).astype(np.float32))
        d1, d2 = np.float32(x - a), np.float32(b - a)
        pup = np.count_nonzero(k * d2 < d1) / 2 ** 24
        assert abs(pup - (float(x) - float(a)) / (float(b) - float(a))) <= 2.0 ** -22


def test_quantize_semantics_and_monte_carlo(oracle_mod):
    Q = np.array([-1.0, -0.25, 0.5, 2.0], np.float32)
    x = np.concatenate([Q, np.full(200000, 0.1, np.float32), np.full(200000, -0.7, np.float32)])
    idx, counts, he = oracle_mod.quantize(x, Q, seed=12345)
    assert list(idx[:4]) == [0, 1, 2, 3]  # values on Q are deterministic
    assert counts.sum() == x.size and np.array_equal(np.bincount(idx, minlength=4), counts)
    f = counts / x.size
    assert he == pytest.approx(-np.sum(f[f > 0] * np.log2(f[f > 0])), rel=1e-12)
    for val, lo in ((0.1, 1), (-0.7, 0)):
        sel = idx[4:][x[4:] == np.float32(val)]
        assert set(np.unique(sel)) <= {lo, lo + 1}
        xh = Q[sel].astype(np.float64)
        se = np.std(xh) / math.sqrt(xh.size)
        assert abs(xh.mean() - float(np.float32(val))) < 5 * se
    # the counter-based draws depend on (seed, index) only
    i2, _, _ = oracle_mod.quantize(x, Q, seed=12345)
    assert np.array_equal(idx, i2)
    i3, _, _ = oracle_mod.quantize(x, Q, seed=54321)
    assert not np.array_equal(idx, i3)


def test_quantize_rejects_non_spanning(oracle_mod):
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.quantize(np.array([0.0, 3.0], np.float32), np.array([0.0, 1.0], np.float32), 1)


def _splitmix64_np(z):
    """SplitMix64 output function, vectorised (pinned by the reference outputs above)."""
    z = z.astype(np.uint64)
    z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
    z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
    return z ^ (z >> np.uint64(31))


def test_quantize_first_draw_is_first_splitmix_output(oracle_mod):
    """Entry 0 consumes the first SplitMix64 output of the seed: k = 0xE220A8 for seed 0."""
    k = 0xE220A8397B1DCDAF >> 40
    u = k / 2 ** 24  # 0.8833...
    Q = np.array([0.0, 1.0], np.float32)
    up = np.array([np.float32(u + 0.01)], np.float32)
    dn = np.array([np.float32(u - 0.01)], np.float32)
    assert oracle_mod.quantize(up, Q, 0)[0][0] == 1
    assert oracle_mod.quantize(dn, Q, 0)[0][0] == 0


def test_quantize_exact_at_dyadic_probability(oracle_mod):
    """Pr[up] is exactly (x-a)/(b-a) when it is a multiple of 2^-24: the draw u = p rounds down."""
    with np.errstate(over="ignore"):
        i = np.arange(1, 1 << 25, dtype=np.uint64)
        k = _splitmix64_np(i * np.uint64(0x9E3779B97F4A7C15)) >> np.uint64(40)
    hit = np.flatnonzero(k == (1 << 23))[0]          # an entry whose draw is exactly 1/2
    miss = np.flatnonzero(k == (1 << 23) - 1)[0]     # and one just below
    Q = np.array([0.0, 1.0], np.float32)
    x = np.full(max(hit, miss) + 1, 0.5, np.float32)
    idx, _, _ = oracle_mod.quantize(x, Q, 0)
    assert idx[hit] == 0 and idx[miss] == 1
    # and over all 2^24 draws the rule rounds up with probability exactly 1/2
    kk = np.arange(2 ** 24, dtype=np.float32) * np.float32(2.0 ** -24)
    assert np.count_nonzero(kk * np.float32(1.0) < np.float32(0.5)) == 2 ** 23


def _exact_refine_round_lambda0(xs, a):
    """One Sec. 6 round at lambda = 0 in exact rationals: colours 0, 1, 2; each
    interior value with index % 3 == colour moves to the unique value strictly
    between its neighbours minimising C[left, c] + C[c, right]; ties keep the
    current value, else the lowest candidate."""
    v = sorted(set(xs))

    def Cx(k, j):
        return sum((Fraction(v[j]) - Fraction(t)) * (Fraction(t) - Fraction(v[k]))
                   for t in xs if v[k] < t <= v[j])
    a = list(a)
    for col in range(3):
        new = list(a)
        for l in range(1, len(a) - 1):
            if l % 3 != col:
                continue
            best, bc = Cx(a[l - 1], a[l]) + Cx(a[l], a[l + 1]), a[l]
            for c in range(a[l - 1] + 1, a[l + 1]):
                val = Cx(a[l - 1], c) + Cx(c, a[l + 1])
                if val < best:
                    best, bc = val, c
            new[l] = bc
        a = new
    return a


@pytest.mark.parametrize("seed", range(12))
def test_refinement_round_exact_with_ties(oracle_mod, seed):
    rng = np.random.default_rng(seed)
    xs = [float(t) for t in rng.integers(0, 13, 40)] + [0.0, 12.0]
    x = np.array(xs, np.float32)
    H = oracle_mod.Hist(x)
    m = min(6, H.p)
    a = _random_codebook(rng, H.p, m)
    want = _exact_refine_round_lambda0(xs, a)
    got = H.refine(a, 0.0, max_rounds=1, tol=-1.0)["Q_idx"]
    assert list(got) == want


def test_refinement_tie_keeps_current(oracle_mod):
    """X = {0, 2, 8, 10}: moving the middle value between 2 and 8 ties exactly (MSE 12)."""
    x = np.array([0, 2, 8, 10], np.float32)
    H = oracle_mod.Hist(x)
    assert list(H.refine([0, 1, 3], 0.0, max_rounds=1, tol=-1.0)["Q_idx"]) == [0, 1, 3]
    assert list(H.refine([0, 2, 3], 0.0, max_rounds=1, tol=-1.0)["Q_idx"]) == [0, 2, 3]
