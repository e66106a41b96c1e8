"""Pins of the oracle's single-decision helpers (Sec. 5, eqs. apx_base and apx_rec).

``or_dp_decision`` (one output of eq. apx_rec against a caller-given previous
layer) and ``or_dp_candidate`` (one candidate of eq. apx_rec, or of eq. apx_base
with ``first``) are what the full-size GPU tests use to check sampled outputs
one by one, so they are pinned here against things other than themselves:

* brute force over every chain of codebook values that ends at j: the value of
  dp(i, j) in eq. apx_rec is the least surrogate cost of a chain
  v_0 = a_1 < ... < a_i = v_j, each link costing C + lambda' Phi (the first link
  Phi^first), summed link by link from the left.  Floating-point addition is
  monotone, so that least left-to-right sum equals the DP's value bit for bit,
  and the brute force also gives the lowest arg-min k and the second-best
  candidate of every decision;
* the interval costs C, U, D of App. E (``or_pair``, pinned against exact
  rationals in test_oracle_pins.py) with Phi = h(U/d) + h(D/d) and
  Phi^first = h(U/d) + h((D + n_a)/d) written out here from Sec. 5;
* the full tables of ``or_apx_dp`` (itself pinned against brute force over
  spanning codebooks) at every (i, j) on larger inputs, with duplicates, ragged
  sizes and s up to 16, at lambda' = 0, small and large.
"""
import itertools
import math

import numpy as np
import pytest

from paper_2608_18147_gb300 import workloads


def h(y):
    """h(y) = -y log2 y, h(0) = 0 (Sec. 4)."""
    return -y * math.log2(y) if y > 0.0 else 0.0


def link(H, k, j, lam_prime, first):
    """C[k, j] + lambda' Phi[k, j] (Phi^first[k, j] for the first interval), Sec. 5."""
    C, U, D = H.pair(k, j)
    d = float(H.d)
    if first:
        w = H.arrays()["w"]
        phi = h(U / d) + h((D + float(w[k])) / d)
    else:
        phi = h(U / d) + h(D / d)
    return C + lam_prime * phi


def chain_minima(H, s, lam_prime):
    """bf[i][j]: least left-to-right sum over chains 0 = a_1 < ... < a_i = j (i values)."""
    p = H.p
    W = {(k, j): link(H, k, j, lam_prime, False) for j in range(p) for k in range(j)}
    W1 = {j: link(H, 0, j, lam_prime, True) for j in range(1, p)}
    bf = np.full((s + 1, p), np.inf)
    for i in range(2, s + 1):
        for j in range(i - 1, p):
            best = math.inf
            for mid in itertools.combinations(range(1, j), i - 2):
                chain = (0,) + mid + (j,)
                v = W1[chain[1]]
                for r in range(1, len(chain) - 1):
                    v = v + W[(chain[r], chain[r + 1])]
                best = min(best, v)
            bf[i, j] = best
    return bf, W


def _tiny(seed, d, dup):
    rng = np.random.default_rng(seed)
    if dup:
        return rng.choice((rng.standard_normal(7) * 3).astype(np.float32), d)
    return (rng.standard_normal(d) * 3).astype(np.float32)


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("lam", [0.0, 0.03, 0.7])
def test_decision_equals_chain_bruteforce(oracle_mod, seed, lam):
    """eq. apx_rec, one output at a time: or_dp_decision's minimum, lowest arg-min and
    second-best equal the brute force over chains, and so do or_apx_dp's tables."""
    x = _tiny(400 + seed, d=9 + seed % 3, dup=seed % 2 == 0)
    H = oracle_mod.Hist(x)
    p = H.p
    s = min(6, p)
    lp = lam * H.norm2
    bf, W = chain_minima(H, s, lp)
    r = H.apx_dp(s, lp)
    for i in range(3, s + 1):
        prev = bf[i - 1]
        for j in range(i - 1, p):
            cands = [(prev[k] + W[(k, j)], k) for k in range(i - 2, j)]
            vals = sorted(v for v, _ in cands)
            best = vals[0]
            arg = min(k for v, k in cands if v == best)
            second = vals[1] if len(vals) > 1 else math.inf
            b, a, s2 = H.dp_decision(prev, i, j, lp)
            assert b == bf[i, j] == best
            assert a == arg
            assert s2 == second
            assert r["dp"][i, j] == best
            assert r["bp"][i, j] == arg
    # the base layer (eq. apx_base, L = {0}) and the traced optimum (eq. apx_final)
    for j in range(1, p):
        assert r["dp"][2, j] == bf[2, j]
        assert r["bp"][2, j] == 0
    assert r["best"] == min(bf[i, p - 1] for i in range(2, s + 1))


@pytest.mark.parametrize("seed", range(4))
def test_candidate_is_the_link_cost(oracle_mod, seed):
    """or_dp_candidate: prev_k + (C + lambda' Phi) for eq. apx_rec and
    C + lambda' Phi^first (first interval, own mass n_a) for eq. apx_base."""
    x = _tiny(500 + seed, d=40, dup=True)
    H = oracle_mod.Hist(x)
    rng = np.random.default_rng(seed)
    for lam in (0.0, 0.05, 2.0):
        lp = lam * H.norm2
        for _ in range(30):
            j = int(rng.integers(1, H.p))
            k = int(rng.integers(0, j))
            prev_k = float(rng.uniform(0.0, 10.0))
            assert H.dp_candidate(prev_k, k, j, lp) == prev_k + link(H, k, j, lp, False)
            assert H.dp_candidate(0.0, k, j, lp, first=True) == link(H, k, j, lp, True)
        # the first interval at k = 0 is the base layer of eq. apx_base
        r = H.apx_dp(3, lp)
        for j in range(1, H.p):
            assert H.dp_candidate(0.0, 0, j, lp, first=True) == r["dp"][2, j]


def _inputs():
    return [
        ("normal_ragged", workloads.normal(301, 3)),
        ("lognormal_dups", np.repeat(workloads.signed_lognormal(130, 4), 3)[:377]),
        ("studentt", workloads.student_t(257, 5)),
    ]


@pytest.mark.parametrize("name,x", _inputs())
@pytest.mark.parametrize("s", [3, 8, 16])
def test_decision_matches_full_tables(oracle_mod, name, x, s):
    """Every output of or_apx_dp's tables (value, lowest arg-min, relative margin to the
    second-best) is reproduced by or_dp_decision fed the table's previous layer."""
    H = oracle_mod.Hist(x)
    H.cache()
    for lam in (0.0, 1e-4, 0.05, 3.0):
        lp = lam * H.norm2
        r = H.apx_dp(s, lp)
        dp, bp, mg = r["dp"], r["bp"], r["margin"]
        for i in range(3, s + 1):
            for j in range(i - 1, H.p):
                b, a, s2 = H.dp_decision(dp[i - 1], i, j, lp)
                assert b == dp[i, j]
                assert a == bp[i, j]
                m = (s2 - b) / b if b > 0.0 else (math.inf if s2 > b else 0.0)
                assert m == mg[i, j] or (math.isinf(m) and math.isinf(mg[i, j]))


def test_base_layer_over_first_value_set(oracle_mod):
    """eq. apx_base with a first-value set L of several grid points: the base layer is the
    least or_dp_candidate(first) over a in L, a < j, lowest a on ties."""
    x = workloads.normal(200, 7)
    lo, hi = float(x.min()), float(x.max())
    grid = np.linspace(lo - 1.0, hi + 0.5, 64).astype(np.float32)
    grid = np.unique(np.concatenate([grid, np.float32([lo, hi])]))
    H = oracle_mod.Hist(x, grid)
    assert H.nL > 1 and H.nR > 1
    for lam in (0.0, 0.02, 1.0):
        lp = lam * H.norm2
        r = H.apx_dp(5, lp)
        for j in range(1, H.p):
            vals = [(H.dp_candidate(0.0, a, j, lp, first=True), a) for a in range(min(H.nL, j))]
            best = min(v for v, _ in vals)
            assert r["dp"][2, j] == best
            assert r["bp"][2, j] == min(a for v, a in vals if v == best)


def test_decision_ties_take_lowest_k(oracle_mod):
    """Exact ties (evenly spaced integer values, equal weights: symmetric interval costs)
    go to the lowest k (the tie rule of eq. apx_rec), in or_dp_decision and or_apx_dp."""
    x = np.repeat(np.arange(9, dtype=np.float32), 2)
    H = oracle_mod.Hist(x)
    s = 5
    lp = 0.0  # MSE only: the costs are integers, so equal sums are exact ties
    bf, W = chain_minima(H, s, lp)
    r = H.apx_dp(s, lp)
    ties = 0
    for i in range(3, s + 1):
        prev = bf[i - 1]
        for j in range(i - 1, H.p):
            cands = [(prev[k] + W[(k, j)], k) for k in range(i - 2, j)]
            best = min(v for v, _ in cands)
            winners = [k for v, k in cands if v == best]
            ties += len(winners) > 1
            b, a, _ = H.dp_decision(prev, i, j, lp)
            assert (b, a) == (best, min(winners))
            assert (r["dp"][i, j], r["bp"][i, j]) == (best, min(winners))
    assert ties > 0


@pytest.mark.parametrize("name,x", _inputs() + [("tiny", np.float32([0.5, -1.0, 2.0])),
                                                ("single", np.float32([1.0, 1.0]))])
@pytest.mark.parametrize("s", [2, 3, 8, 16])
def test_column_order_equals_layer_order(oracle_mod, name, x, s):
    """or_apx_dp_columns (each pair's link cost computed once for all layers) returns
    or_apx_dp's tables, codebook and optimum bit for bit: the recurrence of eq. apx_rec
    does not depend on the order its outputs are visited in."""
    for grid in (None, "grid"):
        g = None
        if grid:
            lo, hi = float(x.min()), float(x.max())
            g = np.unique(np.concatenate([np.linspace(lo - 0.5, hi + 0.5, 40).astype(np.float32),
                                          np.float32([lo, hi])]))
        H = oracle_mod.Hist(x, g)
        for lam in (0.0, 0.01, 1.5):
            lp = lam * H.norm2
            for exact_s in (False, True):
                if exact_s and s > H.p > 1:  # exactly s values do not exist: both report it
                    for cols in (False, True):
                        with pytest.raises(oracle_mod.OracleError) as e:
                            H.apx_dp(s, lp, exact_s=True, columns=cols)
                        assert e.value.code == oracle_mod.EINFEASIBLE
                    continue
                a = H.apx_dp(s, lp, exact_s=exact_s)
                b = H.apx_dp(s, lp, exact_s=exact_s, columns=True)
                assert a["m"] == b["m"] and a["best"] == b["best"]
                assert np.array_equal(a["Q_idx"], b["Q_idx"])
                if H.p > 1:
                    assert np.array_equal(a["dp"], b["dp"])
                    assert np.array_equal(a["bp"], b["bp"])
                    assert np.array_equal(a["margin"], b["margin"])


@pytest.mark.parametrize("name,x", _inputs())
@pytest.mark.parametrize("s", [3, 9, 16])
def test_column_prefix_equals_the_whole_dp_on_its_columns(oracle_mod, name, x, s):
    """or_apx_dp_columns_prefix (the column-by-column DP stopped before column jend) gives
    or_apx_dp's tables bit for bit on every column j < jend, since dp(i, j) reads only
    columns k < j (eq. apx_rec), and leaves the later columns unset."""
    H = oracle_mod.Hist(x)
    for lam in (0.0, 0.05):
        lp = lam * H.norm2
        full = H.apx_dp(s, lp)
        for jend in sorted({1, 2, max(1, H.p // 3), H.p}):
            pr = H.apx_dp_columns_prefix(s, lp, jend)
            for key in ("dp", "bp", "margin"):
                assert np.array_equal(pr[key][:, :jend], full[key][:, :jend]), (key, jend)
            assert np.isinf(pr["dp"][:, jend:]).all() and (pr["bp"][:, jend:] == -1).all()
    with pytest.raises(oracle_mod.OracleError):
        H.apx_dp_columns_prefix(s, 0.0, H.p + 1)
