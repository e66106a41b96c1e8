"""CPU oracle for ECASQ (arxiv 2608.18147) -- test infrastructure only.

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product (the CUDA library and its
Python binding) never touches it, and the two share no code.

The arithmetic lives in ``ecasq_oracle.c`` (plain C, binary64 results,
binary128 prefix sums); this module compiles it on first use with gcc and
wraps it with ctypes.  Each wrapper names the passage of the paper it follows.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ecasq_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, EINVAL, ENONFINITE, EINFEASIBLE, ERANGE, ENOMEM = 0, -1, -2, -3, -7, -8


def build(force: bool = False) -> str:
    """Compile the oracle into oracle/_build/liboracle.so (gcc, OpenMP)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + ".%d.tmp" % os.getpid()
    cmd = ["gcc", "-O2", "-std=gnu11", "-fopenmp", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = C.CDLL(build())
        P = C.c_void_p
        i32, i64, u64, dbl = C.c_int32, C.c_int64, C.c_uint64, C.c_double
        pf = C.POINTER(C.c_float)
        pd = C.POINTER(C.c_double)
        pi32 = C.POINTER(C.c_int32)
        pi64 = C.POINTER(C.c_int64)
        sig = {
            "or_hist_new": (P, [pf, i64, pi32]),
            "or_hist_new_grid": (P, [pf, i64, pf, i64, pi32]),
            "or_hist_free": (None, [P]),
            "or_hist_info": (None, [P, pi64, pi64, pd]),
            "or_hist_ends": (None, [P, pi64, pi64]),
            "or_hist_arrays": (None, [P, pf, pi64, pi64, pd, pd, pd, pd]),
            "or_hist_cache": (i32, [P]),
            "or_pair": (None, [P, i64, i64, pd]),
            "or_phi": (dbl, [P, i64, i64, i32]),
            "or_apx_dp": (i32, [P, i32, dbl, i32, pd, pi32, pd, pi64, pi32, pd]),
            "or_apx_dp_columns": (i32, [P, i32, dbl, i32, pd, pi32, pd, pi64, pi32, pd]),
            "or_apx_dp_columns_prefix": (i32, [P, i32, dbl, i64, pd, pi32, pd]),
            "or_apx_dp_linear": (i32, [P, i32, dbl, i32, pi64, pi32, pd]),
            "or_dp_decision": (None, [P, pd, i32, i64, dbl, pd, pi64, pd]),
            "or_dp_candidate": (dbl, [P, dbl, i64, i64, dbl, i32]),
            "or_eval_idx": (i32, [P, pi64, i32, pd]),
            "or_eval_direct": (i32, [pf, i64, pd, i32, pd]),
            "or_asq_dp": (i32, [P, i32, pd]),
            "or_opt_dp": (i32, [P, i32, dbl, i32, pd, pi64, pi32]),
            "or_brute": (i32, [pf, i64, i32, dbl, dbl, pd, pi64]),
            "or_brute_grid": (i32, [pf, i64, pf, i64, i32, dbl, dbl, pd, pi64]),
            "or_midpoints7": (None, [dbl, dbl, pd]),
            "or_search": (i32, [P, i32, dbl, dbl, dbl, i32, i32, pi64, pi32, pd, pd, i32, pi32]),
            "or_refine": (i32, [P, pi64, i32, dbl, dbl, i32, i32, dbl, pi32, pd]),
            "or_timeshare": (i32, [P, i32, dbl, dbl, dbl, i32, i32, pi64, pi32, pi64, pi32, pd, pd, pd]),
            "or_quantize_timeshare": (i32, [pf, i64, pf, i32, pf, i32, dbl, u64, u64, C.POINTER(C.c_uint8),
                                            C.POINTER(C.c_uint8), C.POINTER(C.c_uint32), pd]),
            "or_splitmix64": (u64, [u64]),
            "or_quantize": (i32, [pf, i64, pf, i32, u64, C.POINTER(C.c_uint8),
                                  C.POINTER(C.c_uint32), pd]),
            "or_num_threads": (i32, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def _ptr(a, ctype):
    return a.ctypes.data_as(C.POINTER(ctype))


def _f32(x):
    return np.ascontiguousarray(np.asarray(x, dtype=np.float32).ravel())


class OracleError(RuntimeError):
    def __init__(self, code, what):
        super().__init__("%s failed with oracle status %d" % (what, code))
        self.code = code


def num_threads() -> int:
    return int(_load().or_num_threads())


class Hist:
    """Sorted weighted histogram of x with App. E prefix sums (Sec. 2, App. E)."""

    def __init__(self, x, grid=None):
        """grid: optional candidate set P (ascending fp32, first <= min x, last >= max x);
        by default P = the unique values of x.  nL, nR: sizes of the first- and
        last-value sets L = {0..nL-1}, R = {p-nR..p-1} of Sec. 5."""
        lib = _load()
        self._x = _f32(x)
        st = C.c_int32(0)
        if grid is None:
            self._h = lib.or_hist_new(_ptr(self._x, C.c_float), self._x.size, C.byref(st))
        else:
            self._grid = _f32(grid)
            self._h = lib.or_hist_new_grid(_ptr(self._x, C.c_float), self._x.size, _ptr(self._grid, C.c_float),
                                           self._grid.size, C.byref(st))
        if not self._h:
            raise OracleError(st.value, "or_hist_new" if grid is None else "or_hist_new_grid")
        d, p, n2 = C.c_int64(), C.c_int64(), C.c_double()
        lib.or_hist_info(self._h, C.byref(d), C.byref(p), C.byref(n2))
        self.d, self.p, self.norm2 = d.value, p.value, n2.value
        nL, nR = C.c_int64(), C.c_int64()
        lib.or_hist_ends(self._h, C.byref(nL), C.byref(nR))
        self.nL, self.nR = nL.value, nR.value

    def __del__(self):
        h = getattr(self, "_h", None)
        if h and _lib is not None:
            _lib.or_hist_free(h)
            self._h = None

    def arrays(self):
        p = self.p
        v = np.empty(p, np.float32)
        w = np.empty(p, np.int64)
        N = np.empty(p + 1, np.int64)
        Sh, Sl, S2h, S2l = (np.empty(p + 1, np.float64) for _ in range(4))
        _load().or_hist_arrays(self._h, _ptr(v, C.c_float), _ptr(w, C.c_int64), _ptr(N, C.c_int64),
                               _ptr(Sh, C.c_double), _ptr(Sl, C.c_double),
                               _ptr(S2h, C.c_double), _ptr(S2l, C.c_double))
        return dict(v=v, w=w, N=N, S_hi=Sh, S_lo=Sl, S2_hi=S2h, S2_lo=S2l)

    def cache(self):
        st = _load().or_hist_cache(self._h)
        if st != OK:
            raise OracleError(st, "or_hist_cache")

    def pair(self, k, j):
        """(C_P, U_P, D_P)[k, j] of App. E (0-based unique indices, k < j)."""
        out = np.empty(3, np.float64)
        _load().or_pair(self._h, int(k), int(j), _ptr(out, C.c_double))
        return float(out[0]), float(out[1]), float(out[2])

    def phi(self, k, j, first=False):
        return float(_load().or_phi(self._h, int(k), int(j), int(bool(first))))

    def apx_dp(self, s, lam_prime, exact_s=False, tables=True, columns=False):
        """Approximate DP of Sec. 5 at multiplier lambda' (eqs. apx_base/rec/final).
        columns: evaluate it column by column (or_apx_dp_columns: the same tables, each
        pair's link cost computed once for all layers; for inputs too large to memoise)."""
        p = self.p
        rows = s + 1
        dp = np.empty(rows * p, np.float64) if tables else None
        bp = np.empty(rows * p, np.int32) if tables else None
        mg = np.empty(rows * p, np.float64) if tables else None
        Q = np.empty(s + 1, np.int64)
        m = C.c_int32()
        best = C.c_double()
        nul = lambda a, t: _ptr(a, t) if a is not None else None
        fn = _load().or_apx_dp_columns if columns else _load().or_apx_dp
        st = fn(self._h, int(s), float(lam_prime), int(bool(exact_s)),
                               nul(dp, C.c_double), nul(bp, C.c_int32), nul(mg, C.c_double),
                               _ptr(Q, C.c_int64), C.byref(m), C.byref(best))
        if st != OK:
            raise OracleError(st, "or_apx_dp")
        out = dict(Q_idx=Q[:m.value].copy(), m=m.value, best=best.value)
        if tables:
            out.update(dp=dp.reshape(rows, p), bp=bp.reshape(rows, p), margin=mg.reshape(rows, p))
        return out

    def apx_dp_columns_prefix(self, s, lam_prime, jend):
        """The approximate DP's tables (dp, bp, margin; (s+1) x p) for the columns j < jend
        only, evaluated column by column as apx_dp(columns=True) does; later columns are
        left at +inf / -1 / +inf and no codebook is formed."""
        p, rows = self.p, s + 1
        dp = np.empty(rows * p, np.float64)
        bp = np.empty(rows * p, np.int32)
        mg = np.empty(rows * p, np.float64)
        st = _load().or_apx_dp_columns_prefix(self._h, int(s), float(lam_prime), int(jend), _ptr(dp, C.c_double),
                                              _ptr(bp, C.c_int32), _ptr(mg, C.c_double))
        if st != OK:
            raise OracleError(st, "or_apx_dp_columns_prefix")
        return dict(dp=dp.reshape(rows, p), bp=bp.reshape(rows, p), margin=mg.reshape(rows, p))

    def apx_dp_linear(self, s, lam_prime, exact_s=False):
        """Linear-space traceback of the approximate DP (Sec. 5, Hirschberg's method):
        (codebook indices, m, dp(m, p-1)); O(p) memory."""
        Q = np.empty(s + 1, np.int64)
        m = C.c_int32()
        best = C.c_double()
        st = _load().or_apx_dp_linear(self._h, int(s), float(lam_prime), int(bool(exact_s)), _ptr(Q, C.c_int64),
                                      C.byref(m), C.byref(best))
        if st != OK:
            raise OracleError(st, "or_apx_dp_linear")
        return Q[:m.value].copy(), m.value, best.value

    def dp_decision(self, prev, i, j, lam_prime):
        """min over k of prev[k] + C[k,j] + lambda' Phi[k,j] (eq. apx_rec), one output."""
        prev = np.ascontiguousarray(prev, dtype=np.float64)
        b, s2 = C.c_double(), C.c_double()
        a = C.c_int64()
        _load().or_dp_decision(self._h, _ptr(prev, C.c_double), int(i), int(j), float(lam_prime),
                               C.byref(b), C.byref(a), C.byref(s2))
        return b.value, a.value, s2.value

    def dp_candidate(self, prev_k, k, j, lam_prime, first=False):
        return float(_load().or_dp_candidate(self._h, float(prev_k), int(k), int(j),
                                             float(lam_prime), int(bool(first))))

    def eval_idx(self, a):
        """(MSE, H(I,B), H(Xhat)) of the codebook v[a] (Sec. 2, 3, eq. apx_additive_entropy)."""
        a = np.ascontiguousarray(a, dtype=np.int64)
        out = np.empty(3, np.float64)
        st = _load().or_eval_idx(self._h, _ptr(a, C.c_int64), a.size, _ptr(out, C.c_double))
        if st != OK:
            raise OracleError(st, "or_eval_idx")
        return float(out[0]), float(out[1]), float(out[2])

    def asq_dp(self, s):
        """Least MSE with at most s values by eq. asqdp (lambda = 0)."""
        b = C.c_double()
        st = _load().or_asq_dp(self._h, int(s), C.byref(b))
        if st != OK:
            raise OracleError(st, "or_asq_dp")
        return b.value

    def opt_dp(self, s, lam_prime, exact_s=False):
        """Optimal DP of Sec. 4 / App. E; returns (best objective, codebook indices)."""
        b = C.c_double()
        Q = np.empty(s + 1, np.int64)
        m = C.c_int32()
        st = _load().or_opt_dp(self._h, int(s), float(lam_prime), int(bool(exact_s)),
                               C.byref(b), _ptr(Q, C.c_int64), C.byref(m))
        if st != OK:
            raise OracleError(st, "or_opt_dp")
        return b.value, Q[:m.value].copy()

    def search(self, s, budget, lo=1e-8, hi=1e3, rounds=6, exact_s=False):
        """Budgeted solve: lambda search of the approximate DP (Sec. 3, Sec. 5)."""
        cap = 8 * rounds + 16
        trace = np.empty(6 * cap, np.float64)
        nt = C.c_int32()
        Q = np.empty(s + 1, np.int64)
        m = C.c_int32()
        res = np.zeros(4, np.float64)
        st = _load().or_search(self._h, int(s), float(budget), float(lo), float(hi), int(rounds),
                               int(bool(exact_s)), _ptr(Q, C.c_int64), C.byref(m),
                               _ptr(res, C.c_double), _ptr(trace, C.c_double), cap, C.byref(nt))
        if st not in (OK, EINFEASIBLE):
            raise OracleError(st, "or_search")
        n = min(nt.value, cap)
        return dict(status=st, Q_idx=Q[:m.value].copy(), m=m.value, lam=res[0], mse=res[1],
                    h_surrogate=res[2], h_exact=res[3], trace=trace[:6 * n].reshape(n, 6).copy(),
                    n_evaluated=nt.value)

    def timeshare(self, s, budget, lo=1e-8, hi=1e3, rounds=6, exact_s=False):
        """Two-way time-sharing of Sec. 7 around the budget (reading in the C file)."""
        Qm = np.empty(s + 1, np.int64)
        Qp = np.empty(s + 1, np.int64)
        mm, mp = C.c_int32(), C.c_int32()
        mmet, pmet = np.empty(3), np.empty(3)
        out = np.empty(6)
        st = _load().or_timeshare(self._h, int(s), float(budget), float(lo), float(hi), int(rounds),
                                  int(bool(exact_s)), _ptr(Qm, C.c_int64), C.byref(mm), _ptr(Qp, C.c_int64),
                                  C.byref(mp), _ptr(mmet, C.c_double), _ptr(pmet, C.c_double),
                                  _ptr(out, C.c_double))
        if st != OK:
            raise OracleError(st, "or_timeshare")
        return dict(beta=out[0], lam_minus=out[1], lam_plus=out[2], mse=out[3], h_surrogate=out[4],
                    h_exact=out[5], minus_idx=Qm[:mm.value].copy(), plus_idx=Qp[:mp.value].copy(),
                    minus=dict(mse=mmet[0], h_surrogate=mmet[1], h_exact=mmet[2]),
                    plus=dict(mse=pmet[0], h_surrogate=pmet[1], h_exact=pmet[2]))

    def refine(self, a, lam_prime, budget=np.inf, guard=False, max_rounds=5, tol=0.0):
        """Three-colour refinement of Sec. 6 (true Lagrangian, reading in the C file)."""
        a = np.array(a, dtype=np.int64)
        ru = C.c_int32()
        J = np.full(max_rounds + 1, np.nan)
        st = _load().or_refine(self._h, _ptr(a, C.c_int64), a.size, float(lam_prime), float(budget),
                               int(bool(guard)), int(max_rounds), float(tol), C.byref(ru),
                               _ptr(J, C.c_double))
        if st != OK:
            raise OracleError(st, "or_refine")
        return dict(Q_idx=a, rounds=ru.value, J=J[:ru.value + 1].copy())


def eval_direct(x, Q):
    """(MSE, H(I,B), H(Xhat)) from the per-entry definitions for any spanning Q."""
    x = _f32(x)
    Q = np.ascontiguousarray(Q, dtype=np.float64)
    out = np.empty(3, np.float64)
    st = _load().or_eval_direct(_ptr(x, C.c_float), x.size, _ptr(Q, C.c_double), Q.size,
                                _ptr(out, C.c_double))
    if st != OK:
        raise OracleError(st, "or_eval_direct")
    return float(out[0]), float(out[1]), float(out[2])


def brute(x, s, lam_prime, budget):
    """Exhaustive search over spanning codebooks drawn from x (p <= 20)."""
    x = _f32(x)
    out = np.empty(6, np.float64)
    masks = np.empty(4, np.int64)
    st = _load().or_brute(_ptr(x, C.c_float), x.size, int(s), float(lam_prime), float(budget),
                          _ptr(out, C.c_double), _ptr(masks, C.c_int64))
    if st != OK:
        raise OracleError(st, "or_brute")
    return dict(surrogate=out[0], true=out[1], mse_surr_budget=out[2], mse_opt_budget_minus1=out[3],
                hx_of_surr_budget=out[4], mse_min=out[5], masks=masks.copy())


def brute_grid(x, grid, s, lam_prime, budget):
    """Exhaustive search over spanning codebooks drawn from the permissible set `grid`
    (at most 16 values); masks are bitmasks over the grid."""
    x = _f32(x)
    g = _f32(grid)
    out = np.empty(6, np.float64)
    masks = np.empty(4, np.int64)
    st = _load().or_brute_grid(_ptr(x, C.c_float), x.size, _ptr(g, C.c_float), g.size, int(s),
                               float(lam_prime), float(budget), _ptr(out, C.c_double), _ptr(masks, C.c_int64))
    if st != OK:
        raise OracleError(st, "or_brute_grid")
    return dict(surrogate=out[0], true=out[1], mse_surr_budget=out[2], mse_opt_budget_minus1=out[3],
                hx_of_surr_budget=out[4], mse_min=out[5], masks=masks.copy())


def midpoints7(lo, hi):
    t = np.empty(7, np.float64)
    _load().or_midpoints7(float(lo), float(hi), _ptr(t, C.c_double))
    return t


def splitmix64(z):
    return int(_load().or_splitmix64(C.c_uint64(z & 0xFFFFFFFFFFFFFFFF)))


def quantize(x, Q, seed):
    """Stochastic quantization of Sec. 2 with the counter-based decision rule."""
    x = _f32(x)
    Q = _f32(Q)
    idx = np.empty(x.size, np.uint8)
    counts = np.empty(Q.size, np.uint32)
    he = C.c_double()
    st = _load().or_quantize(_ptr(x, C.c_float), x.size, _ptr(Q, C.c_float), Q.size,
                             C.c_uint64(seed & 0xFFFFFFFFFFFFFFFF), _ptr(idx, C.c_uint8),
                             _ptr(counts, C.c_uint32), C.byref(he))
    if st != OK:
        raise OracleError(st, "or_quantize")
    return idx, counts, he.value


def quantize_timeshare(x, Qm, Qp, beta, seed, seed_ts):
    """Time-shared stochastic quantization (Sec. 7): (idx, sel, counts, rate)."""
    x = _f32(x)
    Qm = _f32(Qm)
    if Qp is None or len(Qp) == 0:
        Qp, mp = np.zeros(1, np.float32), 0
    else:
        Qp = _f32(Qp)
        mp = Qp.size
    idx = np.empty(x.size, np.uint8)
    sel = np.empty(x.size, np.uint8)
    counts = np.empty(Qm.size + mp, np.uint32)
    rate = C.c_double()
    st = _load().or_quantize_timeshare(_ptr(x, C.c_float), x.size, _ptr(Qm, C.c_float), Qm.size,
                                       _ptr(Qp, C.c_float), mp, float(beta),
                                       C.c_uint64(seed & 0xFFFFFFFFFFFFFFFF), C.c_uint64(seed_ts & 0xFFFFFFFFFFFFFFFF),
                                       _ptr(idx, C.c_uint8), _ptr(sel, C.c_uint8), _ptr(counts, C.c_uint32),
                                       C.byref(rate))
    if st != OK:
        raise OracleError(st, "or_quantize_timeshare")
    return idx, sel, counts, rate.value


def solve_budget(x, s, budget, lo=1e-8, hi=1e3, rounds=6, refine_rounds=0, refine_tol=0.0,
                 guard=True, exact_s=False, grid=None):
    """Full budgeted pipeline: search, then optional refinement at the chosen lambda
    (codebook drawn from `grid` when given, else from the unique values of x)."""
    H = Hist(x, grid)
    if H.p <= 20000:
        H.cache()
    r = H.search(s, budget, lo, hi, rounds, exact_s)
    out = dict(r)
    if refine_rounds > 0 and r["status"] == OK and r["m"] >= 3:
        rf = H.refine(r["Q_idx"], r["lam"] * H.norm2, budget, guard, refine_rounds, refine_tol)
        out["Q_idx"] = rf["Q_idx"]
        out["refine_rounds"] = rf["rounds"]
        out["refine_J"] = rf["J"]
        mse, hs, hx = H.eval_idx(rf["Q_idx"])
        out.update(mse=mse, h_surrogate=hs, h_exact=hx)
    v = H.arrays()["v"]
    out["Q"] = v[out["Q_idx"]]
    out["norm2"] = H.norm2
    out["p"] = H.p
    return out
