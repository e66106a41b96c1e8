"""The optimal DP of Sec. 4 on the GPU (ecasq_opt_dp) against the oracle's naive
O(s p^3) recurrence, brute force and the lambda = 0 special case (pytest -m gpu)."""
import numpy as np
import pytest

from paper_2608_18147_gb300 import workloads

pytestmark = pytest.mark.gpu

VAL_RTOL = 1e-12
MET_RTOL = 1e-9


@pytest.fixture(scope="module")
def E():
    import torch
    assert torch.cuda.is_available(), "these tests need a CUDA GPU"
    import paper_2608_18147_gb300 as E
    E.lib()
    return E


def _compare(E, H, x, v, s, lams, P=None, exact_s=False):
    Q, m, met = E.ecasq_opt_dp(x, s, lams, P=P, flags=E.EXACT_S if exact_s else 0)
    for g, lam in enumerate(lams):
        lp = lam * H.norm2
        best, qo = H.opt_dp(s, lp, exact_s)
        assert met[g, 0] == pytest.approx(best, rel=VAL_RTOL, abs=1e-300), (g, lam)
        q = Q[g, :m[g]].cpu().numpy()
        mse, hs, hx = H.eval_idx(qo)
        if not np.array_equal(q, v[qo]):
            # a different optimum is allowed only at an exact-arithmetic tie
            a = np.searchsorted(v, q)
            gm, _, gx = H.eval_idx(a)
            assert gm + lp * gx == pytest.approx(best, rel=1e-9)
        else:
            np.testing.assert_allclose(met[g, 1:], [mse, hs, hx], rtol=MET_RTOL, atol=1e-300)
        # the optimum is the traced codebook's true Lagrangian
        assert met[g, 0] == pytest.approx(met[g, 1] + lp * met[g, 3], rel=1e-9, abs=1e-300)
    return Q, m, met


@pytest.mark.parametrize("d,s", [(300, 6), (1200, 5)])
def test_opt_dp_matches_oracle(E, oracle_mod, d, s):
    """p = 1200 spans two shared-memory k tiles (1024 each) per column."""
    x = workloads.normal(d, 4)
    H = oracle_mod.Hist(x)
    v = H.arrays()["v"]
    _compare(E, H, x, v, s, [0.0, 0.003, 0.05, 0.4])


def test_opt_dp_on_a_grid_with_several_end_candidates(E, oracle_mod):
    x = workloads.signed_lognormal(2000, 6)
    span = float(x.max() - x.min())
    g = np.unique(np.concatenate([np.linspace(x.min() - 0.2 * span, x.max() + 0.1 * span, 150).astype(np.float32),
                                  np.array([x.min(), x.max()], np.float32)]))
    H = oracle_mod.Hist(x, g)
    assert H.nL > 1 and H.nR > 1
    _compare(E, H, x, g, 7, [0.0, 0.01, 0.2, 2.0], P=g)
    _compare(E, H, x, g, 7, [0.05], P=g, exact_s=True)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_opt_dp_equals_brute_force(E, oracle_mod, seed):
    x = workloads.signed_lognormal(12, seed)
    H = oracle_mod.Hist(x)
    for lam in (0.0, 0.02, 0.3):
        lp = lam * H.norm2
        _, _, met = E.ecasq_opt_dp(x, 5, [lam])
        assert met[0, 0] == pytest.approx(oracle_mod.brute(x, 5, lp, 0.0)["true"], rel=1e-12, abs=1e-300)


def test_opt_dp_at_zero_multiplier_is_the_least_mse(E, oracle_mod):
    x = workloads.student_t(800, 3, scale=1.0)
    H = oracle_mod.Hist(x)
    for s in (3, 8):
        _, _, met = E.ecasq_opt_dp(x, s, [0.0])
        assert met[0, 0] == pytest.approx(H.asq_dp(s), rel=1e-12)


def test_opt_dp_never_worse_than_the_approximate_dp(E, oracle_mod):
    """Both solve the true Lagrangian's feasible set; the optimal DP minimises it exactly."""
    x = workloads.signed_lognormal(3000, 8)
    lams = [0.001, 0.01, 0.1, 1.0]
    Qo, mo, mo_met = E.ecasq_opt_dp(x, 8, lams)
    Qa, ma, ma_met = E.ecasq_dp_pass(x, 8, lams)
    n2 = float(np.sum(x.astype(np.float64) ** 2))
    for g, lam in enumerate(lams):
        true_apx = ma_met[g, 1] + lam * n2 * ma_met[g, 3]
        assert mo_met[g, 0] <= true_apx * (1 + 1e-12)
