"""ecasq_solve_batched: every row's result equals ecasq_solve on that row alone
(same schedule, same codebook, multiplier and metrics), and matches the oracle
(pytest -m gpu).  Rows of length <= 1024 with <= 128 unique values run the
batched path; others fall back to the single-row solve inside the same call."""
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


def _per_row(E, X, s, **kw):
    out = []
    for r in range(X.shape[0]):
        try:
            Q, res = E.ecasq_solve(X[r], s, **kw)
            out.append((Q.cpu().numpy(), res))
        except E.EcasqError as e:
            out.append((None, {"status": e.code}))
    return out


def _compare(E, X, s, **kw):
    Qb, mb, resb = E.ecasq_solve_batched(X, s, **kw)
    Qb, mb = Qb.cpu().numpy(), mb.cpu().numpy()
    for r, (Q1, r1) in enumerate(_per_row(E, X, s, **kw)):
        assert resb[r]["status"] == r1["status"], r
        if Q1 is None:
            continue
        assert mb[r] == r1["m"] == resb[r]["m"], r
        np.testing.assert_array_equal(Qb[r, :mb[r]], Q1, err_msg=f"row {r}")
        for key in ("lambda", "mse", "h_surrogate", "h_exact", "p", "passes", "lambdas_evaluated", "candidates"):
            assert resb[r][key] == r1[key], (r, key)
    return Qb, mb, resb


def test_batched_kv_rows_equal_single_solves(E):
    X = workloads.make("kvrows_8192x128_s8")[:48]
    _compare(E, X, 8, budget_bits=3.0)


def test_batched_matches_oracle(E, oracle_mod):
    X = workloads.make("kvrows_8192x128_s8")[100:106]
    Qb, mb, resb = E.ecasq_solve_batched(X, 8, budget_bits=3.0)
    for r in range(X.shape[0]):
        o = oracle_mod.solve_budget(X[r], 8, 3.0)
        assert resb[r]["status"] == o["status"]
        assert resb[r]["lambda"] == o["lam"]
        np.testing.assert_array_equal(Qb[r, :mb[r]].cpu().numpy(), o["Q"])
        np.testing.assert_allclose([resb[r]["mse"], resb[r]["h_surrogate"], resb[r]["h_exact"]],
                                   [o["mse"], o["h_surrogate"], o["h_exact"]], rtol=MET_RTOL)


def test_batched_edge_rows(E):
    rng = np.random.default_rng(4)
    d = 37  # not a multiple of 4
    X = rng.standard_normal((6, d)).astype(np.float32)
    X[1] = 2.5                                  # one unique value
    X[2, ::2] = X[2, 1]                         # many duplicates
    X[3] = np.round(X[3] * 2) / 2               # few unique values
    X[4, :5] = -0.0; X[4, 5:10] = 0.0           # -0 and +0 are one value
    _compare(E, X, 6, budget_bits=1.5)
    _compare(E, X, 6, lambda_=0.05)             # fixed multiplier
    _compare(E, X, 6, budget_bits=1.5, flags=E.EXACT_S)


def test_batched_long_and_many_unique_rows(E):
    rng = np.random.default_rng(5)
    X = rng.standard_normal((5, 1024)).astype(np.float32)
    X[0] = np.round(X[0] * 8) / 8               # <= 128 unique values: batched path
    X[2] = np.round(X[2] * 4) / 4
    _compare(E, X, 8, budget_bits=2.0)          # rows 1, 3, 4 (> 128 unique) fall back inside the call
    Y = rng.standard_normal((2, 1500)).astype(np.float32)  # d > 1024: row-by-row path
    _compare(E, Y, 8, budget_bits=2.0)
