"""Pins of the oracle's linear-space traceback (Sec. 5, last paragraph: Hirschberg's
method on eq. apx_rec) to what fixes it: brute force over every spanning codebook on tiny
inputs (the surrogate Lagrangian MSE + lambda' H(I,B)), the answer of eq. apx_final, and
or_apx_dp's codebook wherever that one is unique (no decision on its traced path within
1e-9 of the second best)."""
import numpy as np
import pytest

from paper_2608_18147_gb300 import workloads


def _tiny(seed, d, dup):
    rng = np.random.default_rng(seed)
    if dup:
        return rng.choice((rng.standard_normal(9) * 2).astype(np.float32), d)
    return (rng.standard_normal(d) * 2).astype(np.float32)


@pytest.mark.parametrize("seed", range(8))
@pytest.mark.parametrize("lam", [0.0, 0.02, 0.3, 3.0])
def test_linear_traceback_equals_bruteforce(oracle_mod, seed, lam):
    x = _tiny(600 + seed, d=12 + seed % 3, dup=seed % 2 == 0)
    H = oracle_mod.Hist(x)
    for s in (2, 3, 4, 6):
        lp = lam * H.norm2
        Q, m, best = H.apx_dp_linear(s, lp)
        b = oracle_mod.brute(x, s, lp, 10.0)
        mse, hs, _ = H.eval_idx(Q)
        assert mse + lp * hs == pytest.approx(b["surrogate"], rel=1e-12, abs=1e-12)
        assert best == pytest.approx(b["surrogate"], rel=1e-12, abs=1e-12)
        assert m <= s and Q[0] == 0 and Q[-1] == H.p - 1 and np.all(np.diff(Q) > 0)


def _inputs():
    return [("normal", workloads.normal(700, 1)), ("lognormal", workloads.signed_lognormal(513, 2)),
            ("studentt", workloads.student_t(640, 3)), ("dups", np.repeat(workloads.normal(150, 4), 4))]


@pytest.mark.parametrize("name,x", _inputs())
@pytest.mark.parametrize("s", [3, 8, 16])
def test_linear_traceback_matches_backpointer_traceback(oracle_mod, name, x, s):
    """The same optimum as or_apx_dp (eq. apx_final), the same number of values, and the same
    codebook whenever or_apx_dp's traced decisions are all unique by more than 1e-9."""
    H = oracle_mod.Hist(x)
    H.cache()
    same = 0
    for lam in (0.0, 1e-3, 0.05, 0.5, 5.0):
        lp = lam * H.norm2
        for exact_s in (False, True):
            r = H.apx_dp(s, lp, exact_s=exact_s)
            Q, m, best = H.apx_dp_linear(s, lp, exact_s=exact_s)
            assert best == r["best"] and m == r["m"]
            mse, hs, _ = H.eval_idx(Q)
            assert mse + lp * hs == pytest.approx(r["best"], rel=1e-12, abs=1e-15)
            path = r["Q_idx"]
            margin = min([r["margin"][i, path[i - 1]] for i in range(3, r["m"] + 1)] or [np.inf])
            if margin > 1e-9:
                assert np.array_equal(Q, path)
                same += 1
    assert same > 0
