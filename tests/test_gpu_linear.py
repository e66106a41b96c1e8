"""The linear-space traceback (Sec. 5, last paragraph: Hirschberg's method on eq. apx_rec)
on the GPU against the oracle's (pytest -m gpu): the same codebook, m and optimum, and the
metrics of that codebook within 1e-9 relative; where the two codebooks differ (exact or
near ties of the split sums, binary64 rounding of the two sides' interval costs), the GPU's
codebook must reach the same optimum.  Also the backpointer traceback's codebook wherever
that one is unique, and a workspace linear in d."""
import numpy as np
import pytest

from paper_2608_18147_gb300 import workloads

pytestmark = pytest.mark.gpu

MET_RTOL = 1e-9
OPT_RTOL = 1e-12


@pytest.fixture(scope="module")
def E():
    import torch
    assert torch.cuda.is_available(), "these tests need a CUDA GPU"
    import paper_2608_18147_gb300 as E
    E.lib()
    return E


def _inputs():
    rng = np.random.default_rng(21)
    return {
        "normal1000": workloads.normal(1000, 1),
        "lognormal2049": workloads.signed_lognormal(2049, 2),
        "studentt3000": workloads.student_t(3000, 3, scale=1.0),
        "dups": rng.choice(np.float32([-3, -1.5, 0.0, 0.25, 2, 5.5, 7.0]), 901),
    }


@pytest.mark.parametrize("name", list(_inputs()))
@pytest.mark.parametrize("s", [3, 8, 16])
def test_linear_traceback_matches_oracle(E, oracle_mod, name, s):
    x = _inputs()[name]
    H = oracle_mod.Hist(x)
    v = H.arrays()["v"]
    differ = 0
    for lam in (0.0, 0.01, 0.5):
        lp = lam * H.norm2
        for exact_s in (False, True):
            if exact_s and s > H.p:
                with pytest.raises(E.EcasqError):
                    E.ecasq_dp_linear(x, s, lam, flags=E.EXACT_S)
                continue
            Qg, met = E.ecasq_dp_linear(x, s, lam, flags=E.EXACT_S if exact_s else 0)
            Qo, mo, best = H.apx_dp_linear(s, lp, exact_s=exact_s)
            a = np.searchsorted(v, Qg.cpu().numpy())
            assert np.array_equal(v[a], Qg.cpu().numpy())  # values of x
            assert a.size == mo
            assert met[0] == pytest.approx(best, rel=OPT_RTOL)
            mse, hs, hx = H.eval_idx(a)
            np.testing.assert_allclose(met[1:], [mse, hs, hx], rtol=MET_RTOL)
            if not np.array_equal(a, Qo):
                differ += 1
                assert mse + lp * hs == pytest.approx(best, rel=OPT_RTOL)
    assert differ <= 2


def test_linear_traceback_matches_backpointer_traceback(E, oracle_mod):
    x = workloads.student_t(4000, 9, scale=1.0)
    H = oracle_mod.Hist(x)
    H.cache()
    s, same = 16, 0
    for lam in (0.0, 1e-3, 0.05, 0.5):
        r = H.apx_dp(s, lam * H.norm2)
        path = r["Q_idx"]
        margin = min([r["margin"][i, path[i - 1]] for i in range(3, r["m"] + 1)] or [np.inf])
        Qg, met = E.ecasq_dp_linear(x, s, lam)
        Qp, mp, metp = E.ecasq_dp_pass(x, s, [lam])
        assert met[0] == pytest.approx(metp[0][0], rel=OPT_RTOL)
        if margin > 1e-9:
            np.testing.assert_array_equal(Qg.cpu().numpy(), Qp[0, :mp[0]].cpu().numpy())
            same += 1
    assert same > 0


def test_linear_traceback_edge_cases_and_workspace(E):
    import torch
    Q, met = E.ecasq_dp_linear(np.full(40, 2.5, np.float32), 8, 0.1)
    assert Q.numel() == 1 and float(Q[0]) == 2.5 and met[0] == 0.0
    Q, met = E.ecasq_dp_linear(np.float32([1.0, -2.0, 1.0, -2.0]), 8, 0.1)
    assert Q.cpu().numpy().tolist() == [-2.0, 1.0]
    with pytest.raises(E.EcasqError):
        E.ecasq_dp_linear(np.float32([1.0, -2.0, 3.0]), 8, 0.1, flags=E.EXACT_S)
    with pytest.raises(E.EcasqError):
        E.ecasq_dp_linear(np.float32([1.0, 2.0]), 8, -1.0)
    L = E.lib()
    for d in (1000, 1 << 20):
        nb = L.ecasq_workspace_size_linear(d)
        assert nb < 130 * d + (1 << 16)  # linear in d, no table of backpointers
        assert nb < E.ecasq_workspace_size(d, 16) / 8
    torch.cuda.synchronize()
