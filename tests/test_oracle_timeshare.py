"""Oracle pins for two-way time-sharing (Sec. 7, App. F.1): the App. F.1 example with
its printed fraction and vNMSE, dominance over every single quantizer under the
budget (brute force), and the time-shared encode's partition and rounding."""
import math

import numpy as np
import pytest

from conftest import read_golden
from paper_2608_18147_gb300 import workloads


def test_appF1_time_sharing(oracle_mod):
    g = read_golden("appF1_lagrangian_gap.txt")
    b = float(g["ts_budget"][0])
    x = np.array([0.0] * 32 + [2.0] * 32, np.float32)
    P = np.arange(5, dtype=np.float32)
    H = oracle_mod.Hist(x, P)
    ts = H.timeshare(2, b)
    assert list(ts["minus_idx"]) == [0, 4]          # A
    assert list(ts["plus_idx"]) == [0, 2]           # C
    assert round(ts["beta"], 2) == float(g["ts_alpha"][0])
    hA = -(0.75 * math.log2(0.75) + 0.25 * math.log2(0.25))
    assert ts["beta"] == pytest.approx((b - hA) / (1.0 - hA), rel=1e-14)
    assert round(ts["mse"] / H.norm2, 2) == float(g["ts_vnmse"][0])
    assert ts["mse"] / H.norm2 < 0.5                # better than B, the hard-budget single optimum
    assert ts["h_surrogate"] == pytest.approx(b, rel=1e-14)


@pytest.mark.parametrize("seed", [0, 1, 2])
@pytest.mark.parametrize("s", [3, 4])
def test_time_sharing_dominates_every_single_quantizer(oracle_mod, seed, s):
    """The mixture meets the budget and has no more MSE than any codebook drawn from X
    with H(I,B) <= b (Sec. 7: the MSE is linear in the mixing probability)."""
    x = workloads.signed_lognormal(12, seed)
    H = oracle_mod.Hist(x)
    h_lo = H.eval_idx([0, H.p - 1])[1]
    h_hi = H.eval_idx(list(range(H.p)))[1]
    for b in np.linspace(h_lo + 0.05, min(h_hi, 2.2) - 0.05, 7):
        ts = H.timeshare(s, float(b))
        single = oracle_mod.brute(x, s, 0.0, float(b))["mse_surr_budget"]
        assert ts["h_surrogate"] <= b * (1 + 1e-12)
        assert ts["mse"] <= single * (1 + 1e-12) + 1e-300
        assert ts["mse"] <= ts["minus"]["mse"]
        if ts["beta"] > 0:
            assert ts["plus"]["h_surrogate"] > b > ts["minus"]["h_surrogate"]
            assert ts["plus"]["mse"] < ts["minus"]["mse"]
            assert ts["h_surrogate"] == pytest.approx(b, rel=1e-12)


def test_no_time_sharing_when_unconstrained(oracle_mod):
    x = workloads.normal(500, 3)
    H = oracle_mod.Hist(x)
    ts = H.timeshare(4, 20.0)                       # lambda = 0 is feasible (Everett: no mixing)
    assert ts["beta"] == 0.0 and ts["plus_idx"].size == 0
    r = H.search(4, 20.0)
    np.testing.assert_array_equal(ts["minus_idx"], r["Q_idx"])
    assert ts["mse"] == r["mse"]


def test_time_shared_encode(oracle_mod):
    x = workloads.signed_lognormal(20000, 5)
    g = np.unique(np.concatenate([np.linspace(x.min(), x.max(), 64).astype(np.float32),
                                  np.array([x.min(), x.max()], np.float32)]))
    H = oracle_mod.Hist(x, g)
    ts = H.timeshare(8, 2.0)
    assert 0.0 < ts["beta"] < 1.0
    v = H.arrays()["v"]
    Qm, Qp = v[ts["minus_idx"]], v[ts["plus_idx"]]
    idx, sel, counts, rate = oracle_mod.quantize_timeshare(x, Qm, Qp, ts["beta"], 11, 12345)
    # the partition: a fraction beta of the entries, independently (5 sigma)
    n = x.size
    assert abs(sel.mean() - ts["beta"]) < 5 * math.sqrt(ts["beta"] * (1 - ts["beta"]) / n)
    # each part rounds exactly as the plain encode with its own codebook (same counter i)
    im, _, _ = oracle_mod.quantize(x, Qm, 11)
    ip, _, _ = oracle_mod.quantize(x, Qp, 11)
    np.testing.assert_array_equal(idx[sel == 0], im[sel == 0])
    np.testing.assert_array_equal(idx[sel == 1], ip[sel == 1])
    cm = np.bincount(idx[sel == 0], minlength=Qm.size)
    cp = np.bincount(idx[sel == 1], minlength=Qp.size)
    np.testing.assert_array_equal(counts, np.concatenate([cm, cp]))
    bits = 0.0
    for c in (cm, cp):
        c = c[c > 0].astype(np.float64)
        bits -= float(np.sum(c * np.log2(c / c.sum())))
    assert rate == pytest.approx(bits / n, rel=1e-12)
    # beta = 0: every entry takes Q-, identical to the plain encode
    idx0, sel0, counts0, _ = oracle_mod.quantize_timeshare(x, Qm, None, 0.0, 11, 12345)
    assert not sel0.any()
    np.testing.assert_array_equal(idx0, im)
