"""Two-way time-sharing on the GPU (Sec. 7): ecasq_solve_timeshare and
ecasq_quantize_timeshare against the oracle on the same inputs (pytest -m gpu)."""
import math

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


def _check_ts(E, Qm, Qp, res, ts, o, v):
    np.testing.assert_array_equal(Qm.cpu().numpy(), v[o["minus_idx"]])
    np.testing.assert_array_equal(Qp.cpu().numpy(), v[o["plus_idx"]])
    assert ts["m_plus"] == o["plus_idx"].size
    if o["beta"] == 0.0:
        assert ts["beta"] == 0.0
    else:
        assert ts["beta"] == pytest.approx(o["beta"], rel=MET_RTOL)
        assert ts["lambda_plus"] == o["lam_plus"]
    assert res["lambda"] == o["lam_minus"]
    np.testing.assert_allclose([ts["mse"], ts["h_surrogate"], ts["h_exact"]],
                               [o["mse"], o["h_surrogate"], o["h_exact"]], rtol=MET_RTOL)


def test_appF1_time_sharing_on_the_gpu(E, oracle_mod):
    x = np.array([0.0] * 32 + [2.0] * 32, np.float32)
    P = np.arange(5, dtype=np.float32)
    Qm, Qp, res, ts = E.ecasq_solve_timeshare(x, 2, 0.95, P=P)
    o = oracle_mod.Hist(x, P).timeshare(2, 0.95)
    _check_ts(E, Qm, Qp, res, ts, o, P)
    assert Qm.cpu().numpy().tolist() == [0.0, 4.0] and Qp.cpu().numpy().tolist() == [0.0, 2.0]
    assert round(ts["beta"], 2) == 0.74 and round(ts["vnmse"], 2) == 0.26


@pytest.mark.parametrize("budget", [1.5, 2.5])
def test_time_sharing_matches_oracle(E, oracle_mod, budget):
    x = workloads.signed_lognormal(3000, 21)
    Qm, Qp, res, ts = E.ecasq_solve_timeshare(x, 8, budget)
    H = oracle_mod.Hist(x)
    H.cache()
    o = H.timeshare(8, budget)
    _check_ts(E, Qm, Qp, res, ts, o, H.arrays()["v"])
    assert ts["beta"] > 0.0
    assert ts["h_surrogate"] == pytest.approx(budget, rel=1e-12)


def test_time_sharing_fast_kernel_and_grid(E, oracle_mod):
    x = workloads.make("lognormal_d16384_s16")
    Qm, Qp, res, ts = E.ecasq_solve_timeshare(x, 16, 2.0, flags=E.RESIDENT_COSTS)
    H = oracle_mod.Hist(x)
    H.cache()
    _check_ts(E, Qm, Qp, res, ts, H.timeshare(16, 2.0), H.arrays()["v"])
    g = E.uniform_grid(x, 256)
    Qm, Qp, res, ts = E.ecasq_solve_timeshare(x, 16, 2.0, P=g)
    _check_ts(E, Qm, Qp, res, ts, oracle_mod.Hist(x, g).timeshare(16, 2.0), g)


def test_no_time_sharing_when_lambda_zero_is_feasible(E):
    x = workloads.normal(1000, 2)
    Qm, Qp, res, ts = E.ecasq_solve_timeshare(x, 4, 30.0)
    assert ts["beta"] == 0.0 and ts["m_plus"] == 0 and Qp.numel() == 0
    assert res["lambda"] == 0.0 and math.isnan(ts["lambda_plus"])


@pytest.mark.parametrize("d,beta", [(100003, 0.3), (4099, 0.0), (4099, 1.0), (1, 0.5)])
def test_time_shared_encode_bit_exact(E, oracle_mod, d, beta):
    x = workloads.signed_lognormal(d, 9)
    Qm = np.unique(np.concatenate([np.quantile(x, np.linspace(0, 1, 7)).astype(np.float32), [x.min(), x.max()]]))
    Qp = np.unique(np.concatenate([np.quantile(x, np.linspace(0, 1, 12)).astype(np.float32), [x.min(), x.max()]]))
    if d > 1:
        x[::97] = Qm[len(Qm) // 2]                     # entries equal to a codebook value
    idx, sel, counts, rate = E.ecasq_quantize_timeshare(x, Qm, Qp, beta, 77, 31337)
    oi, osel, oc, orate = oracle_mod.quantize_timeshare(x, Qm, Qp, beta, 77, 31337)
    np.testing.assert_array_equal(idx.cpu().numpy(), oi)
    np.testing.assert_array_equal(sel.cpu().numpy(), osel)
    np.testing.assert_array_equal(counts.cpu().numpy().astype(np.uint32), oc)
    assert rate == pytest.approx(orate, rel=1e-12, abs=1e-300)
    if beta in (0.0, 1.0):
        assert np.all(osel == (1 if beta == 1.0 else 0))
