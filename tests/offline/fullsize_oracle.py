"""Full-size check, oracle half: the CPU oracle's approximate DP (Sec. 5, eqs. apx_base,
apx_rec, apx_final) at the multiplier the GPU's budgeted solve selected, over the whole
input, compared with what fullsize_gpu.py wrote.

    python tests/offline/fullsize_oracle.py fullsize_out/studentt_d131072_s16.json

The oracle runs or_apx_dp_columns (each pair's link cost computed once for all layers;
the same tables as or_apx_dp) on this host's OpenMP threads.  Checks, with the parity
bar of the GPU tests:
  * every exactly resolved GPU output the file holds: dp within 1e-12 relative of the
    oracle's, the same backpointer unless the oracle's best two candidates are within
    1e-9 relative (then the GPU's choice, re-scored by the oracle, is within 1e-9 of the
    minimum);
  * the codebook and m equal the oracle's, unless a decision on the oracle's traced path
    had a margin under 1e-9 (then the two objectives agree within 1e-9);
  * MSE, H(I,B) and H(Xhat) of the GPU's codebook, evaluated by the oracle, within 1e-9
    relative of the GPU's own figures, and H(I,B) within the budget.
With --columns F (0 < F < 1) the oracle runs only the first ceil(F p) columns of its DP
(or_apx_dp_columns_prefix: dp(i, j) reads only columns k < j, so those columns are the
whole DP's; the work shrinks by F^2): the outputs of those columns are compared as above,
the GPU's codebook metrics are checked by the oracle's evaluation, and the codebook and
refinement comparisons, which need every column, are skipped.
Writes <name>.report.json next to the input (or to --out) and prints it.
"""
import argparse
import json
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
for p in (ROOT, os.path.join(ROOT, "tests")):
    if p not in sys.path:
        sys.path.insert(0, p)

TIE = 1e-9
DP_RTOL = 1e-12
MET_RTOL = 1e-9


def check(meta_path, out_dir=None, frac=None):
    import oracle
    from paper_2608_18147_gb300 import workloads
    meta = json.load(open(meta_path))
    tables = np.load(meta_path[:-len(".json")] + ".npz")
    name, s = meta["workload"], meta["s"]
    x = workloads.make(name, 0)
    oracle.build()
    t0 = time.perf_counter()
    H = oracle.Hist(x)
    assert H.p == meta["p"], (H.p, meta["p"])
    lp = meta["lam"] * H.norm2
    jend = H.p if frac is None else max(1, min(H.p, int(np.ceil(frac * H.p))))
    if jend < H.p:
        r = H.apx_dp_columns_prefix(s, lp, jend)
    else:
        r = H.apx_dp(s, lp, columns=True)
    wall = time.perf_counter() - t0
    dp_o, bp_o, mg_o = r["dp"], r["bp"], r["margin"]
    cols = tables["cols"] if "cols" in tables.files else np.arange(H.p)
    dp_g, bp_g = tables["dp"], tables["bp"]
    keep = cols < jend  # the stored outputs of the columns the oracle ran
    cols, dp_g, bp_g = cols[keep], dp_g[:, keep], bp_g[:, keep]
    rep = dict(workload=name, d=int(x.size), p=int(H.p), s=s, lam=meta["lam"], oracle_wall_s=wall,
               oracle_threads=oracle.num_threads(), oracle_host=os.uname().machine,
               columns_run=int(jend), stored_columns_compared=int(keep.sum()),
               outputs_compared=0, dp_max_rel=0.0, bp_mismatch=0, bp_mismatch_near_tie=0, bp_invalid=0)
    for i in range(2, s + 1):
        o, g = dp_o[i, cols], dp_g[i]
        fin = np.isfinite(o)
        assert np.array_equal(fin, np.isfinite(g)), "finite pattern differs at layer %d" % i
        rel = np.abs(g[fin] - o[fin]) / np.maximum(np.abs(o[fin]), 1e-300)
        rep["dp_max_rel"] = max(rep["dp_max_rel"], float(rel.max()) if rel.size else 0.0)
        rep["outputs_compared"] += int(fin.sum())
        diff = np.nonzero(fin & (bp_o[i, cols] != bp_g[i]))[0]
        for t in diff:
            j = int(cols[t])
            rep["bp_mismatch"] += 1
            if mg_o[i, j] < TIE:
                rep["bp_mismatch_near_tie"] += 1
                k = int(bp_g[i][t])
                v = H.dp_candidate(dp_o[i - 1, k], k, j, lp)
                if not (0 <= k < j and v <= dp_o[i, j] * (1 + TIE)):
                    rep["bp_invalid"] += 1
            else:
                rep["bp_invalid"] += 1
    v = H.arrays()["v"]
    a_gpu = np.searchsorted(v, np.float32(meta["Q"]))
    a_pass = np.searchsorted(v, np.float32(meta["pass_Q"]))
    rep["pass_codebook_equal_solve"] = bool(np.array_equal(a_gpu, a_pass))
    mse, hs, hx = H.eval_idx(a_gpu)
    rep["metrics_oracle_of_gpu_codebook"] = [mse, hs, hx]
    rep["metrics_gpu"] = [meta["mse"], meta["h_surrogate"], meta["h_exact"]]
    rep["metrics_max_rel"] = max(abs(a - b) / abs(b) for a, b in zip(rep["metrics_gpu"], [mse, hs, hx]) if b)
    rep["feasible"] = bool(hs <= meta["budget_bits"])
    if jend < H.p:  # the codebook and the refinement need every column
        ok = (rep["dp_max_rel"] <= DP_RTOL and rep["bp_invalid"] == 0 and rep["metrics_max_rel"] <= MET_RTOL
              and rep["feasible"] and rep["pass_codebook_equal_solve"])
        return _finish(rep, ok, meta_path, out_dir, name)
    rep["codebook_equal"] = bool(np.array_equal(a_gpu, r["Q_idx"]))
    rep["m_gpu"], rep["m_oracle"] = int(meta["m"]), int(r["m"])
    # margins of the decisions on the oracle's traced path
    path = r["Q_idx"]
    rep["path_min_margin"] = float(min([mg_o[i, path[i - 1]] for i in range(3, r["m"] + 1)] or [np.inf]))
    rep["objective_oracle"] = r["best"]
    rep["objective_of_gpu_codebook"] = mse + lp * hs
    rep["objective_rel"] = abs(rep["objective_of_gpu_codebook"] - r["best"]) / abs(r["best"])
    ref_ok = True
    if "refined" in meta:
        # Sec. 6 refinement of the oracle's own DP codebook at the same multiplier, the same
        # budget guard and stop rule, against the GPU's refined solve
        g = meta["refined"]
        t1 = time.perf_counter()
        rf = H.refine(r["Q_idx"], lp, budget=meta["budget_bits"], guard=True, max_rounds=g["max_rounds"],
                      tol=g["tol"])
        a_ref = np.searchsorted(v, np.float32(g["Q"]))
        mo = H.eval_idx(rf["Q_idx"])
        rep["refine"] = dict(rounds_gpu=g["rounds"], rounds_oracle=rf["rounds"],
                             codebook_equal=bool(np.array_equal(a_ref, rf["Q_idx"])),
                             last_rel_gpu=g["last_rel"],
                             last_rel_oracle=float((rf["J"][-2] - rf["J"][-1]) / abs(rf["J"][-2])),
                             metrics_max_rel=max(abs(a - b) / abs(b) for a, b in
                                                 zip([g["mse"], g["h_surrogate"], g["h_exact"]], mo) if b),
                             stopped_by_rule=rf["rounds"] < g["max_rounds"], oracle_wall_s=time.perf_counter() - t1)
        ref_ok = (rep["refine"]["codebook_equal"] and rep["refine"]["rounds_gpu"] == rep["refine"]["rounds_oracle"]
                  and rep["refine"]["metrics_max_rel"] <= MET_RTOL)
    ok = ref_ok and (rep["dp_max_rel"] <= DP_RTOL and rep["bp_invalid"] == 0 and rep["metrics_max_rel"] <= MET_RTOL
          and rep["feasible"] and rep["pass_codebook_equal_solve"]
          and (rep["codebook_equal"] or (rep["path_min_margin"] < TIE and rep["objective_rel"] <= TIE)))
    return _finish(rep, ok, meta_path, out_dir, name)


def _finish(rep, ok, meta_path, out_dir, name):
    rep["pass"] = bool(ok)
    out = os.path.join(out_dir or os.path.dirname(meta_path), name + ".report.json")
    with open(out, "w") as f:
        json.dump(rep, f, indent=1)
    print(json.dumps(rep), flush=True)
    return ok


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("meta", nargs="+")
    ap.add_argument("--out", default=None)
    ap.add_argument("--columns", type=float, default=None,
                    help="run the oracle's DP over this fraction of the columns only (0 < F < 1)")
    args = ap.parse_args()
    ok = all([check(m, args.out, args.columns) for m in args.meta])
    sys.exit(0 if ok else 1)


if __name__ == "__main__":
    main()
