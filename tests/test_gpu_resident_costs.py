"""ECASQ_RESIDENT_COSTS: the interval costs C and Phi (Sec. 5, App. E) built once
per call into the workspace and streamed to every DP pass.  The tiles are
computed by the same code as the fused kernel's producer, so every fp32
minimum and every exact decision equals the fused mode's; the results match
the oracle under the same bar as the other fast-DP tests (pytest -m gpu)."""
import numpy as np
import pytest

from paper_2608_18147_gb300 import workloads

pytestmark = pytest.mark.gpu

TIE = 1e-9
DP_RTOL = 1e-12
MET_RTOL = 1e-9


@pytest.fixture(scope="module")
def E():
    import torch
    assert torch.cuda.is_available(), "these tests need a CUDA GPU"
    import paper_2608_18147_gb300 as E
    E.lib()
    return E


def _free():
    import torch
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _tables(E, ws, G, s, d):
    out = []
    for g in range(G):
        dp, bp = E.ecasq_dp_tables(ws, g, s, d)
        out.append((dp.cpu().numpy(), bp.cpu().numpy()))
    return out


@pytest.mark.parametrize("flags_name", ["DEFAULT", "EXACT_TABLES"])
@pytest.mark.parametrize("name,s", [("lognormal16k", 16), ("ragged2049", 9), ("mixture12k", 32), ("ragged5000", 18)])
def test_resident_costs_bit_identical_to_fused(E, name, s, flags_name):
    """Same codebooks and metrics with and without resident costs; the same
    exact tables; the same fp32 minima where the closure left outputs unresolved.
    At s = 32 and s = 18 the resident kernel runs eight layers per thread (the fused
    kernel seven)."""
    x = {"lognormal16k": lambda: workloads.signed_lognormal(16384, 0),
         "ragged2049": lambda: workloads.student_t(2049, 3, scale=1.0),
         "mixture12k": lambda: workloads.mixture(12288, 2),
         "ragged5000": lambda: workloads.student_t(5000, 6, scale=1.0)}[name]()
    flags = getattr(E, flags_name, 0)
    lams = [0.0, 1e-5, 1e-3, 0.01, 0.05, 0.2, 1.0, 10.0]
    wsf = E.workspace(x.size, s)
    wsr = E.workspace(x.size, s, flags=E.RESIDENT_COSTS)
    assert wsr.numel() > wsf.numel()
    Qf, mf, metf = E.ecasq_dp_pass(x, s, lams, flags=flags, ws=wsf)
    stf = E.native.ws_status(wsf)
    Qr, mr, metr = E.ecasq_dp_pass(x, s, lams, flags=flags | E.RESIDENT_COSTS, ws=wsr)
    str_ = E.native.ws_status(wsr)
    for st in (stf, str_):
        assert st["timeout"] == 0 and st["bound_viol"] == 0
        if name == "lognormal16k":
            assert st["big_bands"] > 0  # both branches of the many-member exact stage run
            # the exact stage's bound (the band's fp32 argmin in binary64) spares some members
            assert st["rescored"] < st["members"]
    assert mf == mr
    np.testing.assert_array_equal(Qf.cpu().numpy(), Qr.cpu().numpy())
    np.testing.assert_array_equal(metf, metr)
    for (dpf, bpf), (dpr, bpr) in zip(_tables(E, wsf, len(lams), s, x.size), _tables(E, wsr, len(lams), s, x.size)):
        if flags & E.EXACT_TABLES:
            np.testing.assert_array_equal(dpf, dpr)
            np.testing.assert_array_equal(bpf, bpr)
            continue
        # Exactly resolved outputs agree exactly.  The band members the need stage
        # lists may differ in the last bits between the modes (the fused mode
        # re-derives C and Phi from double-double anchors, the resident mode reads
        # the wavefront's own values), so the sets of resolved outputs may differ.
        both = (bpf >= -1) & (bpr >= -1)
        np.testing.assert_array_equal(dpf[both], dpr[both])
        np.testing.assert_array_equal(bpf[both], bpr[both])
        # Outputs resolved in neither hold the wavefront's fp32 minimum: bit-identical.
        neither = (bpf == -2) & (bpr == -2)
        assert neither.any()
        np.testing.assert_array_equal(dpf[neither], dpr[neither])
    del wsf, wsr
    _free()


def test_resident_costs_dp_parity(E, oracle_mod):
    """All outputs resolved exactly: DP values within 1e-12 of the oracle's,
    backpointers equal except at oracle near-ties, codebooks and metrics equal."""
    x = workloads.student_t(2049, 3, scale=1.0)
    s, lams = 16, [0.0, 1e-3, 0.05, 0.4, 3.0]
    ws = E.workspace(x.size, s, flags=E.RESIDENT_COSTS)
    Qg, mg, met = E.ecasq_dp_pass(x, s, lams, flags=E.EXACT_TABLES | E.RESIDENT_COSTS, ws=ws)
    H = oracle_mod.Hist(x)
    H.cache()
    v = H.arrays()["v"]
    for g, lam in enumerate(lams):
        r = H.apx_dp(s, lam * H.norm2)
        dp, bp = [t.cpu().numpy() for t in E.ecasq_dp_tables(ws, g, s, x.size)]
        fin = np.isfinite(r["dp"])
        np.testing.assert_array_equal(np.isfinite(dp), fin)
        np.testing.assert_allclose(dp[fin], r["dp"][fin], rtol=DP_RTOL, atol=0)
        decided = r["bp"] >= 0
        mism = (bp != r["bp"]) & decided
        assert np.all(r["margin"][mism] < TIE)
        assert mg[g] == r["m"]
        np.testing.assert_array_equal(Qg[g, :mg[g]].cpu().numpy(), v[r["Q_idx"]])
        mse, hs, hx = H.eval_idx(r["Q_idx"])
        np.testing.assert_allclose(met[g], [r["best"], mse, hs, hx], rtol=MET_RTOL)


def test_resident_costs_solve_parity(E, oracle_mod):
    x = workloads.normal(1024, 0)
    Q, res = E.ecasq_solve(x, 8, budget_bits=2.0, refine_max_rounds=5, refine_rel_tol=1e-9,
                           flags=E.RESIDENT_COSTS)
    o = oracle_mod.solve_budget(x, 8, 2.0, refine_rounds=5, refine_tol=1e-9)
    assert res["status"] == o["status"] == 0
    assert res["lambda"] == o["lam"]
    np.testing.assert_array_equal(Q.cpu().numpy(), o["Q"])
    np.testing.assert_allclose([res["mse"], res["h_exact"]], [o["mse"], o["h_exact"]], rtol=MET_RTOL)


def test_resident_costs_workspace_checks(E):
    d, s = 4096, 8
    base = E.ecasq_workspace_size(d, s)
    assert E.ecasq_workspace_size_flags(d, s, 1, 0) == base
    nJ = (d + 63) // 64
    assert E.ecasq_workspace_size_flags(d, s, 1, E.RESIDENT_COSTS) >= base + nJ * (nJ + 1) // 2 * 35328
    x = workloads.normal(d, 2)
    small = E.workspace(d, s)  # no room for the resident tiles
    with pytest.raises(E.EcasqError) as ei:
        E.ecasq_solve(x, s, budget_bits=2.0, flags=E.RESIDENT_COSTS, ws=small)
    assert ei.value.code == E.native.EWORKSPACE
    with pytest.raises(E.EcasqError) as ei:
        E.ecasq_dp_pass(x, s, [0.1], flags=E.RESIDENT_COSTS, ws=small)
    assert ei.value.code == E.native.EWORKSPACE
    # the same workspace serves later calls on different data (tiles rebuilt per call)
    ws = E.workspace(d, s, flags=E.RESIDENT_COSTS)
    for seed in (3, 4):
        y = workloads.signed_lognormal(d, seed)
        Qa, ra = E.ecasq_solve(y, s, budget_bits=1.5, flags=E.RESIDENT_COSTS, ws=ws)
        Qb, rb = E.ecasq_solve(y, s, budget_bits=1.5)
        np.testing.assert_array_equal(Qa.cpu().numpy(), Qb.cpu().numpy())
        assert ra["lambda"] == rb["lambda"] and ra["mse"] == rb["mse"]
    del ws, small
    _free()


def test_full_size_sampled_decisions(E, oracle_mod):
    """The benchmark workload (Student-t, d = 2^17, s = 16) in the benchmark's
    launch configuration (resident costs): every output resolved exactly, sampled
    outputs recomputed one by one by the oracle from the GPU's previous layer."""
    x = workloads.make("studentt_d131072_s16")
    s = 16
    lams = [0.0, 1e-4, 1e-3, 0.01, 0.1, 0.4, 2.0, 30.0]
    ws = E.workspace(x.size, s, flags=E.RESIDENT_COSTS)
    Qg, mg, met = E.ecasq_dp_pass(x, s, lams, flags=E.EXACT_TABLES | E.RESIDENT_COSTS, ws=ws)
    st = E.native.ws_status(ws)
    assert st["timeout"] == 0 and st["bound_viol"] == 0
    H = oracle_mod.Hist(x)
    v = H.arrays()["v"]
    rng = np.random.default_rng(17)
    for g, lam in enumerate(lams):
        dp, bp = [t.cpu().numpy() for t in E.ecasq_dp_tables(ws, g, s, x.size)]
        lp = lam * H.norm2
        samples = [(s, H.p - 1), (3, H.p - 1)] + [(int(rng.integers(3, s + 1)), int(rng.integers(s, H.p)))
                                                  for _ in range(4)]
        for i, j in samples:
            best, arg, second = H.dp_decision(dp[i - 1], i, j, lp)
            assert dp[i, j] == pytest.approx(best, rel=DP_RTOL)
            if second > best * (1 + TIE):
                assert bp[i, j] == arg
        # the traced codebook: consecutive backpointers and its metrics
        m = mg[g]
        q = Qg[g, :m].cpu().numpy()
        idx = np.searchsorted(v, q)
        np.testing.assert_array_equal(v[idx], q)
        assert idx[0] == 0 and idx[-1] == H.p - 1
        for r in range(m - 1, 1, -1):
            assert bp[r + 1, idx[r]] == idx[r - 1]
        mse, hs, hx = H.eval_idx(idx)
        np.testing.assert_allclose(met[g][1:], [mse, hs, hx], rtol=MET_RTOL)
    del ws
    _free()


@pytest.mark.parametrize("flags_name", ["DEFAULT", "EXACT_TABLES"])
@pytest.mark.parametrize("name,s", [("lognormal16k", 16), ("ragged20001", 9), ("mixture12k", 32)])
def test_streamed_costs_bit_identical_to_fused(E, name, s, flags_name):
    """ECASQ_STREAMED_COSTS builds the cost tiles band by band into a bounded buffer and runs
    the wavefront over each band: the same fp32 values as the fused producer's, so the same
    tables (resolved and unresolved outputs alike), codebooks and metrics, over several bands."""
    if name == "lognormal16k":
        x = workloads.signed_lognormal(16384, 0)
    elif name == "ragged20001":
        x = workloads.student_t(20001, 4, scale=1.0)
    else:
        x = workloads.mixture(12288, 2)
    flags = getattr(E, flags_name, 0)
    lams = [0.0, 1e-5, 1e-3, 0.01, 0.05, 0.2, 1.0, 10.0]
    wsf = E.workspace(x.size, s)
    wss = E.workspace(x.size, s, flags=E.STREAMED_COSTS)
    full = E.ecasq_workspace_size_flags(x.size, s, 1, E.RESIDENT_COSTS)
    assert wsf.numel() < wss.numel() < full
    Qf, mf, metf = E.ecasq_dp_pass(x, s, lams, flags=flags, ws=wsf)
    n0 = E.ecasq_kernel_launches()
    Qs, ms, mets = E.ecasq_dp_pass(x, s, lams, flags=flags | E.STREAMED_COSTS, ws=wss)
    n1 = E.ecasq_kernel_launches()
    Qf2, _, _ = E.ecasq_dp_pass(x, s, lams, flags=flags, ws=wsf)
    n2 = E.ecasq_kernel_launches()
    assert (n1 - n0) - (n2 - n1) >= 3  # at least two bands: a build and a wavefront launch each
    for ws in (wsf, wss):
        st = E.native.ws_status(ws)
        assert st["timeout"] == 0 and st["bound_viol"] == 0
    assert mf == ms
    np.testing.assert_array_equal(Qf.cpu().numpy(), Qs.cpu().numpy())
    np.testing.assert_array_equal(metf, mets)
    for (dpf, bpf), (dps, bps) in zip(_tables(E, wsf, len(lams), s, x.size), _tables(E, wss, len(lams), s, x.size)):
        np.testing.assert_array_equal(dpf, dps)
        np.testing.assert_array_equal(bpf, bps)
    del wsf, wss
    _free()


def test_streamed_costs_budgeted_solve_matches_oracle(E, oracle_mod):
    """The budgeted solve (multiplier search, refinement) with streamed costs against the oracle."""
    x = workloads.mixture(9000, 5)
    Q, res = E.ecasq_solve(x, 12, budget_bits=3.0, refine_max_rounds=5, refine_rel_tol=1e-9,
                           flags=E.STREAMED_COSTS)
    o = oracle_mod.solve_budget(x, 12, 3.0, refine_rounds=5, refine_tol=1e-9)
    assert res["lambda"] == o["lam"]
    np.testing.assert_array_equal(Q.cpu().numpy(), o["Q"])
    np.testing.assert_allclose([res["mse"], res["h_surrogate"], res["h_exact"]],
                               [o["mse"], o["h_surrogate"], o["h_exact"]], rtol=MET_RTOL)


@pytest.mark.parametrize("name,s", [("lognormal16k", 16), ("studentt9000", 12), ("normal5000", 10)])
def test_two_part_publish_bit_identical_to_one_part(E, name, s):
    """Publishing each column block in two parts (rows 2..8 after layer 8, then the rest) lets the
    next block start its last tile and first layers early; the results are those of the one-part
    publish: the same tables, resolved and unresolved outputs alike."""
    if name == "lognormal16k":
        x = workloads.signed_lognormal(16384, 0)
    elif name == "studentt9000":
        x = workloads.student_t(9000, 6)
    else:
        x = workloads.normal(5000, 7)
    lams = [0.0, 1e-4, 0.01, 0.1, 0.4, 1.0, 3.0, 30.0]
    for costs_flag in (E.RESIDENT_COSTS, E.STREAMED_COSTS):
        ws1 = E.workspace(x.size, s, flags=costs_flag)
        ws2 = E.workspace(x.size, s, flags=costs_flag)
        Q1, m1, met1 = E.ecasq_dp_pass(x, s, lams, flags=costs_flag | E.ONE_PART_PUBLISH, ws=ws1)
        Q2, m2, met2 = E.ecasq_dp_pass(x, s, lams, flags=costs_flag, ws=ws2)
        for ws in (ws1, ws2):
            st = E.native.ws_status(ws)
            assert st["timeout"] == 0 and st["bound_viol"] == 0
        assert m1 == m2
        np.testing.assert_array_equal(Q1.cpu().numpy(), Q2.cpu().numpy())
        np.testing.assert_array_equal(met1, met2)
        for (dp1, bp1), (dp2, bp2) in zip(_tables(E, ws1, len(lams), s, x.size), _tables(E, ws2, len(lams), s, x.size)):
            np.testing.assert_array_equal(dp1, dp2)
            np.testing.assert_array_equal(bp1, bp2)
        del ws1, ws2
        _free()


@pytest.mark.parametrize("name,s,b,mode", [("studentt16k", 16, 2.5, "RESIDENT_COSTS"),
                                           ("lognormal16k", 16, 1.0, "RESIDENT_COSTS"),
                                           ("studentt20001", 12, 2.5, "RESIDENT_COSTS"),
                                           ("normal8192", 10, 2.0, "RESIDENT_COSTS"),
                                           ("studentt16k", 16, 2.5, "STREAMED_COSTS"),
                                           ("mixture12k", 32, 4.0, "RESIDENT_COSTS"),   # 8 layers per thread
                                           ("ragged5000", 18, 2.5, "STREAMED_COSTS")])
def test_seeded_search_bit_identical_to_unseeded(E, name, s, b, mode):
    """Later passes of the search start their tile skipping from the fp32 minima of the
    bracket's evaluated upper end (an upper bound of theirs: candidates are non-decreasing
    in lambda').  Same multiplier, codebook and metrics as without; with every output
    resolved exactly, the same last-pass tables; fewer tiles walked."""
    x = {"studentt16k": lambda: workloads.student_t(16384, 0),
         "lognormal16k": lambda: workloads.signed_lognormal(16384, 0),
         "studentt20001": lambda: workloads.student_t(20001, 5, scale=1.0),
         "normal8192": lambda: workloads.normal(8192, 7),
         "mixture12k": lambda: workloads.mixture(12288, 2),
         "ragged5000": lambda: workloads.student_t(5000, 6, scale=1.0)}[name]()
    cost = getattr(E, mode)  # streamed costs: bands of column blocks, tile skipping and seeds as resident
    out = {}
    for extra in (0, E.UNSEEDED_SEARCH):
        ws = E.workspace(x.size, s, flags=cost)
        Q, res = E.ecasq_solve(x, s, budget_bits=b, refine_max_rounds=0,
                               flags=cost | E.EXACT_TABLES | extra, ws=ws)
        st = E.native.ws_status(ws)
        assert st["timeout"] == 0 and st["bound_viol"] == 0
        out[extra] = (Q.cpu().numpy(), res, st, _tables(E, ws, st["last_G"], s, x.size))
        del ws
        _free()
    (Qs, rs, sts, ts), (Qu, ru, stu, tu) = out[0], out[E.UNSEEDED_SEARCH]
    assert rs["passes"] == ru["passes"] >= 3
    np.testing.assert_array_equal(Qs, Qu)
    for k in ("lambda", "m", "mse", "h_exact", "h_surrogate", "status"):
        assert rs[k] == ru[k], k
    for (dps, bps), (dpu, bpu) in zip(ts, tu):
        np.testing.assert_array_equal(dps, dpu)
        np.testing.assert_array_equal(bps, bpu)
    assert sts["tiles_run"] <= stu["tiles_run"]
    assert stu["tiles_skipped"] > 0  # tile skipping runs at every s here (even layer groups)
    if name == "studentt16k":  # five seeded passes at multipliers where most tiles are skipped
        assert sts["tiles_run"] < 0.95 * stu["tiles_run"]


@pytest.mark.parametrize("lam", [0.0, 0.05])
@pytest.mark.parametrize("name,s,mode", [("studentt16k", 16, "RESIDENT_COSTS"),
                                         ("lognormal16k", 16, "RESIDENT_COSTS"),
                                         ("mixture12k", 17, "RESIDENT_COSTS"),  # 8 layers per thread
                                         ("ragged5000", 18, "STREAMED_COSTS")])  # 8 layers per thread
def test_self_seeded_pass_bit_identical(E, name, s, mode, lam):
    """A fixed-multiplier pass seeded with its own fp32 minima: every running minimum
    starts at the output's final value, the tightest seed that the monotonicity of the
    candidates in lambda' (Sec. 5) allows, so the seeded band starts with no run and
    tiles within the band join it without a reset (a walk whose band started empty
    once dropped a tile 0 that joined it first).  Same codebook, metrics and exact
    tables as the plain pass, no certificate violation, and fewer tiles walked."""
    x = {"studentt16k": lambda: workloads.student_t(16384, 0),
         "lognormal16k": lambda: workloads.signed_lognormal(16384, 0),
         "mixture12k": lambda: workloads.mixture(12288, 2),
         "ragged5000": lambda: workloads.student_t(5000, 6, scale=1.0)}[name]()
    cost = getattr(E, mode)
    out = {}
    for extra in (0, E.TEST_SELF_SEED):
        ws = E.workspace(x.size, s, flags=cost)
        Q, res = E.ecasq_solve(x, s, lambda_=lam, refine_max_rounds=0, flags=cost | E.EXACT_TABLES | extra, ws=ws)
        st = E.native.ws_status(ws)
        assert st["timeout"] == 0 and st["bound_viol"] == 0
        out[extra] = (Q.cpu().numpy(), res, st, _tables(E, ws, 1, s, x.size))
        del ws
        _free()
    (Q0, r0, st0, t0), (Q1, r1, st1, t1) = out[0], out[E.TEST_SELF_SEED]
    assert r1["passes"] == r0["passes"] + 1
    np.testing.assert_array_equal(Q0, Q1)
    for k in ("lambda", "m", "mse", "h_exact", "h_surrogate", "status"):
        assert r0[k] == r1[k], k
    (dp0, bp0), (dp1, bp1) = t0[0], t1[0]
    np.testing.assert_array_equal(dp0, dp1)
    np.testing.assert_array_equal(bp0, bp1)
    # the counters add up over a call's passes: the seeded pass is the second one
    assert st1["tiles_run"] <= 2 * st0["tiles_run"]
    assert st0["tiles_skipped"] > 0  # 8 layers per thread at s = 17 and 18: tile skipping with one multiplier
    assert st1["tiles_run"] - st0["tiles_run"] < st0["tiles_run"]
