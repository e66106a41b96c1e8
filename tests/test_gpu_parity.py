"""GPU-vs-oracle parity through the C ABI (run on a GB300: pytest -m gpu).

Bar: integer and index outputs bit-exact (sort, histogram, backpointers,
codebooks, quantized indices) except where the oracle's best two candidates
differ by under 1e-9 relative; DP values within 1e-12 relative (binary64 on both
sides, same formulas); MSE / entropies within 1e-9 relative, tighter than the
1e-6 the method's accuracy target asks.
"""
from fractions import Fraction

import numpy as np
import pytest

from paper_2608_18147_gb300 import workloads

pytestmark = pytest.mark.gpu

TIE = 1e-9          # decisions whose oracle margin is below this may differ
DP_RTOL = 1e-12     # DP values (binary64 on both sides, same formulas)
MET_RTOL = 1e-9     # MSE and entropies


@pytest.fixture(scope="module")
def E():
    import torch
    assert torch.cuda.is_available(), "these tests need a CUDA GPU"
    import paper_2608_18147_gb300 as E
    E.lib()
    return E


def inputs_small():
    rng = np.random.default_rng(11)
    return {
        "normal1024": workloads.normal(1024, 0),
        "dups": rng.choice(np.float32([-3, -1.5, -0.0, 0.0, 0.25, 2, 5.5]), 777),
        "one": np.array([1.25], np.float32),
        "two_values": np.array([1.0, -2.0, 1.0, 1.0, -2.0], np.float32),
        "const": np.full(50, 3.5, np.float32),
        "ragged2049": workloads.signed_lognormal(2049, 3),
        "tiny_offset": (np.float32(1000.0) + workloads.normal(300, 4) * np.float32(0.01)).astype(np.float32),
    }


# ---------------------------------------------------------- histogram (A1-A3)

@pytest.mark.parametrize("name", list(inputs_small()))
def test_prepare_parity(E, oracle_mod, name):
    x = inputs_small()[name]
    g = E.ecasq_prepare(x)
    H = oracle_mod.Hist(x)
    a = H.arrays()
    assert g["p"] == H.p
    np.testing.assert_array_equal(g["v"].cpu().numpy(), a["v"])
    np.testing.assert_array_equal(g["w"].cpu().numpy(), a["w"])
    np.testing.assert_array_equal(g["N"].cpu().numpy(), a["N"])
    for key in ("S", "S2"):
        gh, gl = g[key + "_hi"].cpu().numpy(), g[key + "_lo"].cpu().numpy()
        oh, ol = a[key + "_hi"], a[key + "_lo"]
        scale = max(abs(float(oh[-1])), 1e-300)
        for t in range(0, H.p + 1, max(1, H.p // 50)):
            diff = (Fraction(float(gh[t])) + Fraction(float(gl[t]))) - (Fraction(float(oh[t])) + Fraction(float(ol[t])))
            assert abs(float(diff)) <= 2.0 ** -96 * scale


# ---------------------------------------------------------------- DP tables

def _dp_parity(E, oracle_mod, x, s, lams, flags, exact_s=False):
    import torch
    d = x.size
    ws = E.workspace(d, s)
    Qg, mg, met = E.ecasq_dp_pass(x, s, lams, flags=flags | (E.EXACT_S if exact_s else 0), ws=ws)
    H = oracle_mod.Hist(x)
    if H.p <= 20000:
        H.cache()
    v = H.arrays()["v"]
    report = []
    for g, lam in enumerate(lams):
        r = H.apx_dp(s, lam * H.norm2, exact_s=exact_s)
        dp, bp = E.ecasq_dp_tables(ws, g, s, d)
        dp, bp = dp.cpu().numpy(), bp.cpu().numpy()
        fin = np.isfinite(r["dp"])
        np.testing.assert_array_equal(np.isfinite(dp), fin)
        np.testing.assert_allclose(dp[fin], r["dp"][fin], rtol=DP_RTOL, atol=0)
        decided = r["bp"] >= 0
        np.testing.assert_array_equal(bp >= 0, decided)
        mism = (bp != r["bp"]) & decided
        assert np.all(r["margin"][mism] < TIE), "backpointer mismatch with margin >= 1e-9"
        # the traced codebook and its metrics
        if not np.any(mism):
            assert mg[g] == r["m"]
            np.testing.assert_array_equal(Qg[g, :mg[g]].cpu().numpy(), v[r["Q_idx"]])
        mse, hs, hx = H.eval_idx(r["Q_idx"])
        np.testing.assert_allclose(met[g], [r["best"], mse, hs, hx], rtol=MET_RTOL, atol=1e-300)
        report.append(int(mism.sum()))
    return report


@pytest.mark.parametrize("lams", [[0.0], [0.0, 1e-4, 0.01, 0.05, 0.2, 0.6, 2.0, 40.0]])
@pytest.mark.parametrize("flags_name", ["DP_REFERENCE", "EXACT_TABLES"])
def test_dp_parity_normal1024(E, oracle_mod, lams, flags_name):
    x = workloads.normal(1024, 0)
    _dp_parity(E, oracle_mod, x, 8, lams, getattr(E, flags_name))


@pytest.mark.parametrize("name,s,lams", [
    ("ragged2049", 6, [0.0, 0.03, 0.4]),
    ("ragged2049", 16, [0.0, 1e-3, 0.05, 0.4, 3.0]),
    ("dups", 8, [0.0, 0.1]),
    ("tiny_offset", 9, [0.0, 0.02, 0.5]),
    ("normal1024", 3, [0.0, 0.3]),
    ("normal1024", 23, [0.0, 0.01, 0.2, 1.0, 5.0, 20.0, 100.0]),
    ("ragged2049", 32, [0.0, 1e-3, 0.02, 0.3, 2.0, 9.0, 30.0, 100.0]),  # 8 layers per thread, 2 splits
    ("normal1024", 18, [0.0, 0.05, 0.4]),                                # 8 layers per thread, 2 groups
])
def test_dp_fast_parity(E, oracle_mod, name, s, lams):
    """The fast kernel (fp32 filter + certified band + exact re-scoring) against the oracle."""
    x = inputs_small()[name]
    _dp_parity(E, oracle_mod, x, s, lams, E.EXACT_TABLES)


def _eps_layer(i):
    """Certified relative error of the fast kernel's fp32 minima at layer i."""
    u = 2.0 ** -24
    eps = 1.0001 * u
    for _ in range(3, i + 1):
        eps = max(eps, 24 * u) + 1.0001 * u
    return eps


@pytest.mark.parametrize("name,s,lams", [
    ("normal1024", 8, [0.0, 1e-4, 0.01, 0.2, 2.0]),
    ("ragged2049", 16, [0.0, 1e-3, 0.05, 0.4]),
])
def test_dp_fast_closure_mode(E, oracle_mod, name, s, lams):
    """Default fast mode: only the outputs eq. apx_final and the traceback read are
    resolved exactly; the codebooks and metrics equal the oracle's, resolved entries
    match exactly and the rest lie within their certified fp32 bound."""
    x = inputs_small()[name]
    ws = E.workspace(x.size, s)
    Qg, mg, met = E.ecasq_dp_pass(x, s, lams, ws=ws)
    st = E.native.ws_status(ws)
    assert st["bound_viol"] == 0 and st["timeout"] == 0
    H = oracle_mod.Hist(x)
    H.cache()
    v = H.arrays()["v"]
    for g, lam in enumerate(lams):
        r = H.apx_dp(s, lam * H.norm2)
        dp, bp = [t.cpu().numpy() for t in E.ecasq_dp_tables(ws, g, s, x.size)]
        res = bp >= -1
        assert res[:, -1][2:].all()  # every dp(i, p-1) is resolved
        fin = np.isfinite(r["dp"]) & res
        np.testing.assert_allclose(dp[fin], r["dp"][fin], rtol=DP_RTOL)
        mism = (bp != r["bp"]) & res & (r["bp"] >= 0)
        assert np.all(r["margin"][mism] < TIE)
        unres = (bp == -2)
        for i in range(3, s + 1):
            row = unres[i] & np.isfinite(r["dp"][i])
            if row.any():
                err = np.abs(dp[i][row] - r["dp"][i][row])
                assert np.all(err <= _eps_layer(i) * 1.001 * r["dp"][i][row])
        assert mg[g] == r["m"]
        np.testing.assert_array_equal(Qg[g, :mg[g]].cpu().numpy(), v[r["Q_idx"]])
        mse, hs, hx = H.eval_idx(r["Q_idx"])
        np.testing.assert_allclose(met[g], [r["best"], mse, hs, hx], rtol=MET_RTOL)


def test_dp_fast_matches_reference_16k(E, oracle_mod):
    """d = 16384 (signed LogNormal), s = 16, 8 multipliers: fast vs reference DP tables, and
    sampled decisions against the oracle given the GPU's previous layer."""
    x = workloads.signed_lognormal(16384, 0)
    s = 16
    lams = [0.0, 1e-5, 1e-3, 0.01, 0.05, 0.2, 1.0, 10.0]
    wsf, wsr = E.workspace(x.size, s), E.workspace(x.size, s)
    Ql, ml, metl = E.ecasq_dp_pass(x, s, lams, flags=0, ws=wsf)  # default closure mode
    stl = E.native.ws_status(wsf)
    Qf, mf, metf = E.ecasq_dp_pass(x, s, lams, flags=E.EXACT_TABLES, ws=wsf)
    stf = E.native.ws_status(wsf)
    Qr, mr, metr = E.ecasq_dp_pass(x, s, lams, flags=E.DP_REFERENCE, ws=wsr)
    assert stf["bound_viol"] == 0 and stf["timeout"] == 0
    H = oracle_mod.Hist(x)
    rng = np.random.default_rng(5)
    for g in range(len(lams)):
        dpf, bpf = [t.cpu().numpy() for t in E.ecasq_dp_tables(wsf, g, s, x.size)]
        dpr, bpr = [t.cpu().numpy() for t in E.ecasq_dp_tables(wsr, g, s, x.size)]
        np.testing.assert_array_equal(np.isfinite(dpf), np.isfinite(dpr))
        fin = np.isfinite(dpr)
        np.testing.assert_allclose(dpf[fin], dpr[fin], rtol=DP_RTOL)
        mism = np.argwhere((bpf != bpr) & (bpr >= 0))
        lp = lams[g] * H.norm2
        for i, j in mism[:50]:  # any disagreement must be a near-tie for the oracle
            best, arg, second = H.dp_decision(dpr[i - 1], int(i), int(j), lp)
            vf = H.dp_candidate(dpr[i - 1][bpf[i, j]], bpf[i, j], j, lp)
            assert vf <= best * (1 + TIE)
        assert mism.shape[0] <= 1e-6 * bpr.size + 5
        for _ in range(6):  # sampled decisions straight from the oracle's formulas
            i = int(rng.integers(3, s + 1))
            j = int(rng.integers(i - 1, x.size if H.p == x.size else H.p))
            best, arg, second = H.dp_decision(dpf[i - 1], i, j, lp)
            assert dpf[i, j] == pytest.approx(best, rel=DP_RTOL)
            if second > best * (1 + TIE):
                assert bpf[i, j] == arg
        assert mf[g] == mr[g] == ml[g]
        np.testing.assert_array_equal(Qf[g].cpu().numpy(), Qr[g].cpu().numpy())
        np.testing.assert_array_equal(Ql[g].cpu().numpy(), Qr[g].cpu().numpy())
    np.testing.assert_allclose(metl, metr, rtol=MET_RTOL)
    assert stl["bound_viol"] == 0 and stl["members"] < stf["members"]


@pytest.mark.parametrize("name", ["dups", "ragged2049", "tiny_offset", "two_values"])
def test_dp_reference_parity_edge_inputs(E, oracle_mod, name):
    x = inputs_small()[name]
    _dp_parity(E, oracle_mod, x, 6, [0.0, 0.03, 0.4], E.DP_REFERENCE)
    if oracle_mod.Hist(x).p >= 6:
        _dp_parity(E, oracle_mod, x, 6, [0.1], E.DP_REFERENCE, exact_s=True)
    else:  # exactly s values cannot be drawn from fewer unique values: both sides say so
        with pytest.raises(E.EcasqError) as ei:
            E.ecasq_dp_pass(x, 6, [0.1], flags=E.DP_REFERENCE | E.EXACT_S)
        assert ei.value.code == E.native.EINFEASIBLE
        with pytest.raises(oracle_mod.OracleError):
            oracle_mod.Hist(x).apx_dp(6, 0.1, exact_s=True)


def test_dp_reference_parity_s_exceeds_p(E, oracle_mod):
    x = np.array([0.5, -1.0, 2.0, 0.5, 7.0], np.float32)  # p = 4 < s
    _dp_parity(E, oracle_mod, x, 8, [0.0, 0.2], E.DP_REFERENCE)


# --------------------------------------------------------------- the search

@pytest.mark.parametrize("flags_name", ["DP_REFERENCE", "FAST"])
def test_solve_parity_normal1024(E, oracle_mod, flags_name):
    flags = getattr(E, flags_name, 0)
    x = workloads.normal(1024, 0)
    Q, res = E.ecasq_solve(x, 8, budget_bits=2.0, flags=flags)
    o = oracle_mod.solve_budget(x, 8, 2.0)
    assert res["status"] == o["status"] == 0
    assert res["lambda"] == o["lam"]
    np.testing.assert_array_equal(Q.cpu().numpy(), o["Q"])
    np.testing.assert_allclose([res["mse"], res["h_surrogate"], res["h_exact"]],
                               [o["mse"], o["h_surrogate"], o["h_exact"]], rtol=MET_RTOL)
    assert res["h_surrogate"] <= 2.0


def test_solve_with_refinement_parity(E, oracle_mod):
    x = workloads.normal(1024, 0)
    Q, res = E.ecasq_solve(x, 8, budget_bits=2.0, refine_max_rounds=5, refine_rel_tol=1e-9)
    o = oracle_mod.solve_budget(x, 8, 2.0, refine_rounds=5, refine_tol=1e-9)
    np.testing.assert_array_equal(Q.cpu().numpy(), o["Q"])
    assert res["refine_rounds"] == o.get("refine_rounds", 0)
    np.testing.assert_allclose([res["mse"], res["h_exact"]], [o["mse"], o["h_exact"]], rtol=MET_RTOL)
    assert res["h_exact"] <= 2.0


def test_solve_unconstrained_and_infeasible(E, oracle_mod):
    x = workloads.normal(512, 1)
    Q, res = E.ecasq_solve(x, 4, budget_bits=8.0, flags=E.DP_REFERENCE)
    o = oracle_mod.solve_budget(x, 4, 8.0)
    assert res["lambda"] == 0.0 and o["lam"] == 0.0
    np.testing.assert_array_equal(Q.cpu().numpy(), o["Q"])
    Q, res = E.ecasq_solve(x[:256], 4, budget_bits=0.0, flags=E.DP_REFERENCE)
    assert res["status"] == E.native.EINFEASIBLE


def test_solve_degenerate_inputs(E, oracle_mod):
    Q, res = E.ecasq_solve(np.full(33, -2.0, np.float32), 8, budget_bits=1.0)
    assert res["m"] == 1 and Q.cpu().numpy().tolist() == [-2.0] and res["mse"] == 0.0
    Q, res = E.ecasq_solve(np.array([3.0], np.float32), 8, budget_bits=1.0)
    assert res["m"] == 1
    x = np.array([1.0, -2.0, 1.0, 1.0, -2.0], np.float32)
    Q, res = E.ecasq_solve(x, 8, budget_bits=1.0, flags=E.DP_REFERENCE)
    assert Q.cpu().numpy().tolist() == [-2.0, 1.0] and res["mse"] == 0.0


def test_nonfinite_and_workspace_errors(E):
    import torch
    x = workloads.normal(100, 0)
    x[17] = np.nan
    with pytest.raises(E.EcasqError) as ei:
        E.ecasq_solve(x, 4, budget_bits=2.0)
    assert ei.value.code == E.native.ENONFINITE
    x[17] = np.inf
    with pytest.raises(E.EcasqError):
        E.ecasq_solve(x, 4, budget_bits=2.0)
    small = torch.empty(1024, dtype=torch.uint8, device="cuda")
    with pytest.raises(E.EcasqError) as ei:
        E.ecasq_solve(workloads.normal(100, 0), 4, budget_bits=2.0, ws=small)
    assert ei.value.code == E.native.EWORKSPACE


# --------------------------------------------------------------- refinement

@pytest.mark.parametrize("seed", [0, 1])
def test_refine_parity(E, oracle_mod, seed):
    x = workloads.signed_lognormal(600, seed)
    H = oracle_mod.Hist(x)
    H.cache()
    v = H.arrays()["v"]
    lam = 0.05
    a0 = H.apx_dp(9, lam * H.norm2)["Q_idx"]
    for guard_budget in (-1.0, 2.2):
        o = H.refine(a0, lam * H.norm2, budget=guard_budget if guard_budget >= 0 else np.inf,
                     guard=guard_budget >= 0, max_rounds=6, tol=0.0)
        Q, res = E.ecasq_refine(x, v[a0], lam, budget_bits=guard_budget, max_rounds=6, rel_tol=0.0)
        np.testing.assert_array_equal(Q.cpu().numpy(), v[o["Q_idx"]])
        assert res["refine_rounds"] == o["rounds"]
        np.testing.assert_allclose(res["objective"], o["J"][-1], rtol=MET_RTOL)


def test_refine_rejects_codebook_outside_x(E):
    x = workloads.normal(100, 0)
    Q = np.array([x.min(), 0.123456, x.max()], np.float32)
    with pytest.raises(E.EcasqError) as ei:
        E.ecasq_refine(x, Q, 0.1)
    assert ei.value.code == E.native.ERANGE


def test_evaluate_parity(E, oracle_mod):
    x = inputs_small()["dups"]
    H = oracle_mod.Hist(x)
    v = H.arrays()["v"]
    for a in ([0, H.p - 1], [0, 2, 3, H.p - 1], list(range(H.p))):
        got = E.ecasq_evaluate(x, v[a])
        np.testing.assert_allclose(got, H.eval_idx(a), rtol=MET_RTOL, atol=1e-15)


# -------------------------------------------------------------- quantization

@pytest.mark.parametrize("d,offset", [(1, 0), (7, 0), (1001, 1), (4096, 0), (100003, 3)])
def test_quantize_bit_exact(E, oracle_mod, d, offset):
    import torch
    x = workloads.student_t(d + offset, d, scale=1.0)
    xg = torch.as_tensor(x).cuda()[offset:]  # misaligned start when offset > 0
    xs = x[offset:]
    Q = np.unique(np.concatenate([[xs.min(), xs.max()], np.quantile(xs, [0.2, 0.5, 0.7]).astype(np.float32)]))
    Q = np.sort(Q.astype(np.float32))
    for seed in (0, 12345, 2 ** 63 + 7):
        idx, counts, he = E.ecasq_quantize(xg, Q, seed)
        oi, oc, oh = oracle_mod.quantize(xs, Q, seed)
        np.testing.assert_array_equal(idx.cpu().numpy(), oi)
        np.testing.assert_array_equal(counts.cpu().numpy().astype(np.uint32), oc)
        assert he == pytest.approx(oh, rel=1e-12, abs=1e-15)


@pytest.mark.parametrize("m", [1, 2, 3, 5, 8, 9, 16, 17, 32, 33, 256])
@pytest.mark.parametrize("offset", [0, 1])
def test_quantize_bit_exact_codebook_sizes(E, oracle_mod, m, offset):
    """Every search depth of the short-codebook kernel (m <= 16: 0 to 4 unrolled steps),
    both sides of the per-thread-histogram limits (16 and 32 values) and the cap, on an
    input long enough for several grid-stride steps per thread."""
    import torch
    d = 3_000_001
    x = workloads.signed_lognormal(d + offset, 11)
    xg = torch.as_tensor(x).cuda()[offset:]
    xs = x[offset:]
    if m == 1:  # a constant input: every entry equals the single value
        xs = np.full_like(xs, np.float32(2.5))
        xg = torch.as_tensor(xs).cuda()
    Q = np.unique(np.quantile(xs, np.linspace(0.0, 1.0, m)).astype(np.float32))
    Q[0], Q[-1] = xs.min(), xs.max()
    assert Q.size == m
    idx, counts, he = E.ecasq_quantize(xg, Q, 99)
    oi, oc, oh = oracle_mod.quantize(xs, Q, 99)
    np.testing.assert_array_equal(idx.cpu().numpy(), oi)
    np.testing.assert_array_equal(counts.cpu().numpy().astype(np.uint32), oc)
    assert int(oc.sum()) == d
    assert he == pytest.approx(oh, rel=1e-12, abs=1e-15)


def test_quantize_rejects_out_of_range(E):
    x = np.array([0.0, 2.0], np.float32)
    with pytest.raises(E.EcasqError) as ei:
        E.ecasq_quantize(x, np.array([0.0, 1.0], np.float32), 1)
    assert ei.value.code == E.native.ERANGE
