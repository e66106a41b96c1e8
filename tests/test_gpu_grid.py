"""ecasq_solve_grid: the codebook drawn from a caller-given permissible set P
(Sec. 5, App. E for general P) against the oracle on the same P (pytest -m gpu)."""
import numpy as np
import pytest

from paper_2608_18147_gb300 import workloads

pytestmark = pytest.mark.gpu

MET_RTOL = 1e-9


@pytest.fixture(scope="module")
def E():
    import torch
    assert torch.cuda.is_available(), "these tests need a CUDA GPU"
    import paper_2608_18147_gb300 as E
    E.lib()
    return E


def _check(res, o, Q):
    assert res["status"] == o["status"]
    assert res["lambda"] == o["lam"]
    np.testing.assert_array_equal(Q.cpu().numpy(), o["Q"])
    np.testing.assert_allclose([res["mse"], res["h_surrogate"], res["h_exact"]],
                               [o["mse"], o["h_surrogate"], o["h_exact"]], rtol=MET_RTOL)


def test_grid_of_unique_values_equals_plain_solve(E):
    x = workloads.signed_lognormal(3000, 1)
    Q1, r1 = E.ecasq_solve(x, 8, budget_bits=2.0)
    Q2, r2 = E.ecasq_solve_grid(x, np.unique(x), 8, budget_bits=2.0)
    np.testing.assert_array_equal(Q1.cpu().numpy(), Q2.cpu().numpy())
    for k in ("lambda", "mse", "h_surrogate", "h_exact", "p", "passes"):
        assert r1[k] == r2[k], k


@pytest.mark.parametrize("n,refine", [(256, 0), (256, 5), (1024, 0), (97, 0)])
def test_uniform_grid_matches_oracle(E, oracle_mod, n, refine):
    x = workloads.make("lognormal_d16384_s16")
    g = E.uniform_grid(x, n)
    Q, res = E.ecasq_solve_grid(x, g, 16, budget_bits=2.0, refine_max_rounds=refine, refine_rel_tol=1e-9)
    o = oracle_mod.solve_budget(x, 16, 2.0, grid=g, refine_rounds=refine, refine_tol=1e-9)
    assert res["p"] == g.size
    _check(res, o, Q)
    assert np.all(np.isin(Q.cpu().numpy(), g))


def test_grid_larger_than_x_and_fast_kernel_sizes(E, oracle_mod):
    x = workloads.student_t(200, 3, scale=1.0)          # n > d
    g = E.uniform_grid(x, 300)
    Q, res = E.ecasq_solve_grid(x, g, 6, budget_bits=1.5)
    _check(res, oracle_mod.solve_budget(x, 6, 1.5, grid=g), Q)
    x = workloads.student_t(20000, 4, scale=1.0)        # n = 4096: the fast kernel, resident costs
    g = E.uniform_grid(x, 4096)
    Q, res = E.ecasq_solve_grid(x, g, 8, budget_bits=2.5, flags=E.RESIDENT_COSTS)
    _check(res, oracle_mod.solve_budget(x, 8, 2.5, grid=g), Q)


def test_grid_that_does_not_span_x_is_rejected(E):
    x = np.array([1.0, 2.0, 3.0, 2.5], np.float32)
    for P in ([1.5, 3.0], [1.0, 2.5], [1.0, 3.0, 2.0], [1.0, 1.0, 3.0], [1.0, np.inf, 3.0]):
        with pytest.raises(E.EcasqError) as ei:
            E.ecasq_solve_grid(x, np.array(P, np.float32), 4, budget_bits=1.0)
        assert ei.value.code == E.native.EINVAL


def wide_grid(x, n, below, above):
    lo, hi = float(x.min()), float(x.max())
    g = np.linspace(lo - below, hi + above, n).astype(np.float32)
    return np.unique(np.concatenate([g, np.array([lo, hi], np.float32)]))


@pytest.mark.parametrize("refine", [0, 3])
def test_grid_with_several_first_and_last_candidates(E, oracle_mod, refine):
    """L = {p_a <= min x} and R = {p_b >= max x} with several members each (eqs. apx_base,
    apx_final): the base layer minimises over a in L, the final selection over j in R."""
    x = workloads.signed_lognormal(5000, 11)
    span = float(x.max() - x.min())
    g = wide_grid(x, 300, 0.05 * span, 0.08 * span)
    import torch
    ws = torch.empty(int(E.lib().ecasq_workspace_size_grid(x.size, g.size, 8, 0)), dtype=torch.uint8,
                     device="cuda")
    Q, res = E.ecasq_solve_grid(x, g, 8, budget_bits=2.0, ws=ws, refine_max_rounds=refine, refine_rel_tol=1e-9)
    H = oracle_mod.Hist(x, g)
    st = E.native.ws_status(ws)
    assert (st["grid_nL"], st["grid_nR"]) == (H.nL, H.nR)
    assert H.nL > 1 and H.nR > 1
    _check(res, oracle_mod.solve_budget(x, 8, 2.0, grid=g, refine_rounds=refine, refine_tol=1e-9), Q)


def test_appF1_example_on_the_gpu(E, oracle_mod):
    """App. F.1: X = half 0s, half 2s; P = (0,1,2,3,4); s = 2.  At every multiplier the
    GPU returns the oracle's codebook ({0,2} or {0,4}, never {0,3}); the budgeted solve
    at b = 0.95 returns {0, 4}, the best Lagrangian point under the budget."""
    x = np.array([0.0] * 32 + [2.0] * 32, np.float32)
    P = np.arange(5, dtype=np.float32)
    H = oracle_mod.Hist(x, P)
    for lam in (0.01, 1.0, 4.0, 5.5, 6.5, 20.0):
        Q, res = E.ecasq_solve_grid(x, P, 2, lambda_=lam)
        o = H.apx_dp(2, lam * H.norm2, tables=False)
        np.testing.assert_array_equal(Q.cpu().numpy(), P[o["Q_idx"]])
        assert Q.cpu().numpy().tolist() in ([0.0, 2.0], [0.0, 4.0])
    Q, res = E.ecasq_solve_grid(x, P, 2, budget_bits=0.95)
    _check(res, oracle_mod.solve_budget(x, 2, 0.95, grid=P), Q)
    assert Q.cpu().numpy().tolist() == [0.0, 4.0]


@pytest.mark.parametrize("case", ["uniform", "wide", "dynamic_range", "ties"])
def test_grid_dp_equals_reference_kernel(E, case):
    """The grid DP (cached pair costs, fp32 band, binary64 re-scoring) returns what the
    binary64 reference kernel returns, bit for bit, at every evaluated multiplier."""
    rng = np.random.default_rng(5)
    if case == "uniform":
        x = workloads.student_t(30000, 8, scale=1.0)
        g = E.uniform_grid(x, 2000)
    elif case == "wide":
        x = workloads.signed_lognormal(8000, 12)
        g = wide_grid(x, 700, 1.0, 3.0)
    elif case == "dynamic_range":    # fp32 copies of tiny intervals underflow after scaling
        x = np.concatenate([rng.standard_normal(3000) * 1e-25, rng.standard_normal(40) * 1e15]).astype(np.float32)
        g = np.unique(np.concatenate([np.sort(x)[::7], [x.min(), x.max()]]).astype(np.float32))
    else:                            # many zero-mass intervals: exact ties between candidates
        x = np.repeat(np.arange(12, dtype=np.float32), 50)
        g = np.linspace(0, 11, 400).astype(np.float32)
    for b in (1.0, 2.5):
        Q1, r1 = E.ecasq_solve_grid(x, g, 8, budget_bits=b)
        Q2, r2 = E.ecasq_solve_grid(x, g, 8, budget_bits=b, flags=E.DP_REFERENCE)
        np.testing.assert_array_equal(Q1.cpu().numpy(), Q2.cpu().numpy())
        for k in ("status", "lambda", "mse", "h_surrogate", "h_exact", "passes", "lambdas_evaluated"):
            assert r1[k] == r2[k], k
