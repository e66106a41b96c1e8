"""Thin ctypes binding of include/ecasq.h.

Every function here has the C entry point's name and only marshals
arguments: torch CUDA tensors become device pointers, the current torch
stream becomes the cudaStream_t, and host results come back as Python
values.  All arithmetic runs in libecasq.so; there is no fallback -- if the
library cannot be loaded, every call raises.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

import numpy as np

from . import build as _build

OK, EINVAL, ENONFINITE, EINFEASIBLE, EWORKSPACE, ECUDA, ETIMEOUT, ERANGE = 0, -1, -2, -3, -4, -5, -6, -7
EXACT_S, NO_REFINE_GUARD, DP_REFERENCE, TIME_KERNELS, EXACT_TABLES, RESIDENT_COSTS, STREAMED_COSTS = 1, 2, 4, 8, 16, 32, 64
ONE_PART_PUBLISH = 128  # fast DP: publish every column block once (no two-part publish)
UNSEEDED_SEARCH = 256  # fast DP search: no seeded tile skipping (same results)
TEST_STALL = 1 << 30  # test hook of the bounded waits (include/ecasq.h)
TEST_SELF_SEED = 1 << 29  # test hook: a fixed-multiplier pass seeded with its own fp32 minima (same results)

_lock = threading.Lock()
_lib = None


class Params(C.Structure):
    _fields_ = [("s", C.c_int32), ("flags", C.c_uint32), ("budget_bits", C.c_double), ("lambda_", C.c_double),
                ("lambda_lo", C.c_double), ("lambda_hi", C.c_double), ("search_rounds", C.c_int32),
                ("refine_max_rounds", C.c_int32), ("refine_rel_tol", C.c_double)]


class Result(C.Structure):
    _fields_ = [("status", C.c_int32), ("m", C.c_int32), ("passes", C.c_int32), ("lambdas_evaluated", C.c_int32),
                ("refine_rounds", C.c_int32), ("reserved", C.c_int32), ("d", C.c_int64), ("p", C.c_int64),
                ("lambda_", C.c_double), ("lambda_prime", C.c_double), ("norm2", C.c_double), ("mse", C.c_double),
                ("vnmse", C.c_double), ("h_surrogate", C.c_double), ("h_exact", C.c_double), ("r_tot", C.c_double),
                ("objective", C.c_double), ("candidates", C.c_int64), ("rescored", C.c_int64),
                ("dp_kernel_ms", C.c_double), ("dp_kernel_launches", C.c_int32), ("reserved2", C.c_int32),
                ("refine_last_rel", C.c_double)]

    def as_dict(self):
        out = {}
        for name, _ in self._fields_:
            key = "lambda" if name == "lambda_" else name
            out[key] = getattr(self, name)
        return out


class Timeshare(C.Structure):
    _fields_ = [("beta", C.c_double), ("lambda_plus", C.c_double), ("mse", C.c_double), ("vnmse", C.c_double),
                ("h_surrogate", C.c_double), ("h_exact", C.c_double), ("plus_mse", C.c_double),
                ("plus_h_surrogate", C.c_double), ("plus_h_exact", C.c_double), ("m_plus", C.c_int32),
                ("reserved", C.c_int32)]

    def as_dict(self):
        return {name: getattr(self, name) for name, _ in self._fields_}


class EcasqError(RuntimeError):
    def __init__(self, code, where):
        self.code = code
        msg = lib().ecasq_strerror(code).decode() if _lib is not None else str(code)
        super().__init__("%s: %s (status %d)" % (where, msg, code))


def lib_path() -> str:
    return _build.LIB


def lib():
    """Load libecasq.so (building it first if it is missing or stale)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.build()
        L = C.CDLL(path)
        vp, i32, i64, u32, u64, dbl, sz = C.c_void_p, C.c_int32, C.c_int64, C.c_uint32, C.c_uint64, C.c_double, C.c_size_t
        pd = C.POINTER(C.c_double)
        pi32 = C.POINTER(C.c_int32)
        pi64 = C.POINTER(C.c_int64)
        PP = C.POINTER(Params)
        PR = C.POINTER(Result)
        sig = {
            "ecasq_version": (C.c_int, []),
            "ecasq_strerror": (C.c_char_p, [C.c_int]),
            "ecasq_workspace_size": (sz, [i64, i32, i64]),
            "ecasq_workspace_size_flags": (sz, [i64, i32, i64, u32]),
            "ecasq_solve": (C.c_int, [vp, i64, PP, vp, sz, vp, PR, vp]),
            "ecasq_solve_grid": (C.c_int, [vp, i64, vp, i64, PP, vp, sz, vp, PR, vp]),
            "ecasq_workspace_size_grid": (sz, [i64, i64, i32, u32]),
            "ecasq_workspace_size_opt": (sz, [i64, i64, i32, i32]),
            "ecasq_workspace_size_prep": (sz, [i64]),
            "ecasq_opt_dp": (C.c_int, [vp, i64, vp, i64, i32, pd, i32, u32, vp, sz, vp, pi32, pd, vp]),
            "ecasq_solve_timeshare": (C.c_int, [vp, i64, vp, i64, PP, vp, sz, vp, vp, PR, C.POINTER(Timeshare), vp]),
            "ecasq_quantize_timeshare": (C.c_int, [vp, i64, vp, i32, vp, i32, dbl, u64, u64, vp, vp, vp, vp, sz, pd,
                                                   vp]),
            "ecasq_dp_pass": (C.c_int, [vp, i64, i32, pd, i32, u32, vp, sz, vp, pi32, pd, vp]),
            "ecasq_dp_tables": (C.c_int, [vp, sz, i32, vp, vp, pi64, vp]),
            "ecasq_workspace_size_linear": (sz, [i64]),
            "ecasq_dp_linear": (C.c_int, [vp, i64, i32, dbl, u32, vp, sz, vp, pi32, pd, vp]),
            "ecasq_refine": (C.c_int, [vp, i64, vp, i32, dbl, dbl, i32, dbl, u32, vp, sz, PR, vp]),
            "ecasq_evaluate": (C.c_int, [vp, i64, vp, i32, vp, sz, pd, vp]),
            "ecasq_quantize": (C.c_int, [vp, i64, vp, i32, u64, vp, vp, vp, sz, pd, vp]),
            "ecasq_quantize_noalloc": (C.c_int, [vp, i64, vp, i32, u64, vp, vp, pd, vp]),
            "ecasq_solve_batched": (C.c_int, [vp, i64, i64, PP, vp, sz, vp, vp, PR, vp]),
            "ecasq_prepare": (C.c_int, [vp, i64, vp, sz, vp, vp, vp, vp, vp, pi64, vp]),
            "ecasq_kernel_launches": (i64, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
        return L


def exported_symbols():
    """Names declared in include/ecasq.h that the loaded library exports."""
    L = lib()
    names = []
    for name in ("ecasq_version", "ecasq_strerror", "ecasq_workspace_size", "ecasq_workspace_size_flags",
                 "ecasq_solve", "ecasq_solve_grid", "ecasq_workspace_size_grid", "ecasq_solve_timeshare",
                 "ecasq_quantize_timeshare", "ecasq_workspace_size_opt", "ecasq_workspace_size_prep", "ecasq_opt_dp",
                 "ecasq_dp_pass",
                 "ecasq_dp_tables", "ecasq_workspace_size_linear", "ecasq_dp_linear", "ecasq_refine", "ecasq_evaluate", "ecasq_quantize", "ecasq_quantize_noalloc",
                 "ecasq_solve_batched",
                 "ecasq_prepare", "ecasq_kernel_launches"):
        if hasattr(L, name):
            names.append(name)
    return names


# ------------------------------------------------------------------ helpers

def _torch():
    import torch
    return torch


def _stream():
    torch = _torch()
    return C.c_void_p(torch.cuda.current_stream().cuda_stream)


def _ptr(t):
    return C.c_void_p(t.data_ptr())


def _dev_f32(x):
    torch = _torch()
    if not isinstance(x, torch.Tensor):
        x = torch.as_tensor(np.ascontiguousarray(x, dtype=np.float32))
    if x.dtype != torch.float32:
        raise TypeError("x must be float32")
    if not x.is_cuda:
        x = x.cuda()
    return x.contiguous()


def _check(rc, where, ok=(OK,)):
    if rc not in ok:
        raise EcasqError(rc, where)
    return rc


def ws_status(ws):
    """Counters the library leaves at the start of a workspace after a call
    (unique values, device-side flags, fast-DP statistics)."""
    raw = ws[:120].cpu().numpy().tobytes()
    (p, nonfinite, range_err, timeout, bound_viol, norm2, rescored, overflow, last_s, last_G, last_d, members,
     big_bands, tiles_run, tiles_skipped, grid_nL, grid_nR, tiles_fetched) = __import__("struct").unpack("<qiiiidqqiiqqqqqqqq", raw)
    return dict(p=p, nonfinite=nonfinite, range_err=range_err, timeout=timeout, bound_viol=bound_viol, norm2=norm2,
                rescored=rescored, overflow=overflow, last_s=last_s, last_G=last_G, last_d=last_d, members=members,
                big_bands=big_bands, tiles_run=tiles_run, tiles_skipped=tiles_skipped, grid_nL=grid_nL,
                grid_nR=grid_nR, tiles_fetched=tiles_fetched)


def ecasq_workspace_size(d, s, rows=1) -> int:
    return int(lib().ecasq_workspace_size(int(d), int(s), int(rows)))


def ecasq_workspace_size_flags(d, s, rows=1, flags=0) -> int:
    return int(lib().ecasq_workspace_size_flags(int(d), int(s), int(rows), int(flags)))


def workspace(d, s, rows=1, flags=0):
    """A device workspace (torch uint8 tensor; CUDA allocations are 256-byte aligned)."""
    torch = _torch()
    n = ecasq_workspace_size_flags(d, s, rows, flags)
    if n == 0:
        raise EcasqError(EINVAL, "ecasq_workspace_size")
    return torch.empty(n, dtype=torch.uint8, device="cuda")


def make_params(s, budget_bits=0.0, lambda_=-1.0, lambda_lo=0.0, lambda_hi=0.0, search_rounds=0,
                refine_max_rounds=0, refine_rel_tol=0.0, flags=0):
    return Params(int(s), int(flags), float(budget_bits), float(lambda_), float(lambda_lo), float(lambda_hi),
                  int(search_rounds), int(refine_max_rounds), float(refine_rel_tol))


# --------------------------------------------------------------- entry points

def ecasq_solve(x, s, budget_bits=0.0, lambda_=-1.0, ws=None, **kw):
    """Budgeted (or fixed-multiplier) solve; returns (Q tensor [m], result dict)."""
    torch = _torch()
    x = _dev_f32(x)
    d = x.numel()
    if ws is None:
        ws = workspace(d, s, flags=kw.get("flags", 0))
    prm = make_params(s, budget_bits, lambda_, **kw)
    Q = torch.zeros(s, dtype=torch.float32, device="cuda")
    res = Result()
    rc = lib().ecasq_solve(_ptr(x), d, C.byref(prm), _ptr(ws), ws.numel(), _ptr(Q), C.byref(res), _stream())
    _check(rc, "ecasq_solve", ok=(OK, EINFEASIBLE))
    return Q[:res.m].clone(), res.as_dict()


def ecasq_solve_grid(x, P, s, budget_bits=0.0, lambda_=-1.0, ws=None, **kw):
    """Budgeted solve with the codebook drawn from the candidate set P (strictly ascending,
    P[0] <= min x, P[-1] >= max x)."""
    torch = _torch()
    x = _dev_f32(x)
    P = _dev_f32(P)
    d, n = x.numel(), P.numel()
    if ws is None:
        nb = int(lib().ecasq_workspace_size_grid(d, n, int(s), int(kw.get("flags", 0))))
        if nb == 0:
            raise EcasqError(EINVAL, "ecasq_workspace_size_grid")
        ws = torch.empty(nb, dtype=torch.uint8, device="cuda")
    prm = make_params(s, budget_bits, lambda_, **kw)
    Q = torch.zeros(s, dtype=torch.float32, device="cuda")
    res = Result()
    rc = lib().ecasq_solve_grid(_ptr(x), d, _ptr(P), n, C.byref(prm), _ptr(ws), ws.numel(), _ptr(Q), C.byref(res),
                                _stream())
    _check(rc, "ecasq_solve_grid", ok=(OK, EINFEASIBLE))
    return Q[:res.m].clone(), res.as_dict()


def ecasq_solve_timeshare(x, s, budget_bits, P=None, ws=None, **kw):
    """Budgeted solve with two-way time-sharing (Sec. 7): (Q- tensor, Q+ tensor or empty,
    result dict of Q-, time-sharing dict).  P: optional permissible set as in ecasq_solve_grid."""
    torch = _torch()
    x = _dev_f32(x)
    d = x.numel()
    flags = int(kw.get("flags", 0))
    if P is not None:
        P = _dev_f32(P)
        n = P.numel()
        nb = int(lib().ecasq_workspace_size_grid(d, n, int(s), flags))
    else:
        n = 0
        nb = int(lib().ecasq_workspace_size_flags(d, int(s), 1, flags))
    if ws is None:
        if nb == 0:
            raise EcasqError(EINVAL, "workspace size")
        ws = torch.empty(nb, dtype=torch.uint8, device="cuda")
    prm = make_params(s, budget_bits, -1.0, **kw)
    Qm = torch.zeros(s, dtype=torch.float32, device="cuda")
    Qp = torch.zeros(s, dtype=torch.float32, device="cuda")
    res = Result()
    ts = Timeshare()
    rc = lib().ecasq_solve_timeshare(_ptr(x), d, _ptr(P) if P is not None else None, n, C.byref(prm), _ptr(ws),
                                     ws.numel(), _ptr(Qm), _ptr(Qp), C.byref(res), C.byref(ts), _stream())
    _check(rc, "ecasq_solve_timeshare", ok=(OK, EINFEASIBLE))
    return Qm[:res.m].clone(), Qp[:ts.m_plus].clone(), res.as_dict(), ts.as_dict()


def ecasq_quantize_timeshare(x, Qm, Qp, beta, seed, seed_ts, ws=None, with_sel=True):
    """Time-shared stochastic quantization (Sec. 7): (idx, sel or None, counts [mm + mp], rate)."""
    torch = _torch()
    x = _dev_f32(x)
    d = x.numel()
    Qm = _dev_f32(Qm)
    Qp = _dev_f32(Qp) if Qp is not None and len(Qp) else None
    mm, mp = Qm.numel(), (Qp.numel() if Qp is not None else 0)
    if ws is None:
        ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    idx = torch.empty(d, dtype=torch.uint8, device="cuda")
    sel = torch.empty(d, dtype=torch.uint8, device="cuda") if with_sel else None
    counts = torch.empty(mm + mp, dtype=torch.int32, device="cuda")
    rate = C.c_double()
    rc = lib().ecasq_quantize_timeshare(_ptr(x), d, _ptr(Qm), mm, _ptr(Qp) if Qp is not None else None, mp,
                                        float(beta), C.c_uint64(int(seed) & 0xFFFFFFFFFFFFFFFF),
                                        C.c_uint64(int(seed_ts) & 0xFFFFFFFFFFFFFFFF), _ptr(idx),
                                        _ptr(sel) if sel is not None else None, _ptr(counts), _ptr(ws), ws.numel(),
                                        C.byref(rate), _stream())
    _check(rc, "ecasq_quantize_timeshare")
    return idx, sel, counts, rate.value


def ecasq_opt_dp(x, s, lambdas, P=None, flags=0, ws=None):
    """Optimal DP of Sec. 4 at up to 8 fixed multipliers (vNMSE scale): (Q [G, s] tensor,
    m list, metrics [G, 4] = optimum, MSE, H(I,B), H(Xhat)).  P: optional permissible set."""
    torch = _torch()
    x = _dev_f32(x)
    d = x.numel()
    lams = np.ascontiguousarray(np.atleast_1d(lambdas), dtype=np.float64)
    G = lams.size
    n = 0
    if P is not None:
        P = _dev_f32(P)
        n = P.numel()
    if ws is None:
        nb = int(lib().ecasq_workspace_size_opt(d, n if P is not None else d, int(s), G))
        if nb == 0:
            raise EcasqError(EINVAL, "ecasq_workspace_size_opt")
        ws = torch.empty(nb, dtype=torch.uint8, device="cuda")
    Q = torch.zeros((G, s), dtype=torch.float32, device="cuda")
    m = (C.c_int32 * G)()
    met = np.zeros(4 * G, np.float64)
    rc = lib().ecasq_opt_dp(_ptr(x), d, _ptr(P) if P is not None else None, n, int(s),
                            lams.ctypes.data_as(C.POINTER(C.c_double)), G, int(flags), _ptr(ws), ws.numel(), _ptr(Q),
                            m, met.ctypes.data_as(C.POINTER(C.c_double)), _stream())
    _check(rc, "ecasq_opt_dp")
    return Q, list(m), met.reshape(G, 4)


def uniform_grid(x, n):
    """n equally spaced fp32 candidates from min x to max x, both endpoints exact."""
    x = np.asarray(x, dtype=np.float32)
    lo, hi = float(x.min()), float(x.max())
    g = np.linspace(lo, hi, n).astype(np.float32)
    g[0], g[-1] = np.float32(lo), np.float32(hi)
    return np.unique(g)


def ecasq_dp_pass(x, s, lambdas, flags=0, ws=None):
    """One DP pass at up to 8 multipliers: (Q [G, s] tensor, m list, metrics [G, 4])."""
    torch = _torch()
    x = _dev_f32(x)
    d = x.numel()
    lams = np.ascontiguousarray(lambdas, dtype=np.float64)
    G = lams.size
    if ws is None:
        ws = workspace(d, s, flags=flags)
    Q = torch.zeros((G, s), dtype=torch.float32, device="cuda")
    m = (C.c_int32 * G)()
    met = np.zeros(4 * G, np.float64)
    rc = lib().ecasq_dp_pass(_ptr(x), d, int(s), lams.ctypes.data_as(C.POINTER(C.c_double)), G, int(flags),
                             _ptr(ws), ws.numel(), _ptr(Q), m, met.ctypes.data_as(C.POINTER(C.c_double)), _stream())
    _check(rc, "ecasq_dp_pass")
    return Q, list(m), met.reshape(G, 4)


def ecasq_dp_linear(x, s, lambda_, flags=0, ws=None):
    """Linear-space traceback of the approximate DP at one multiplier (vNMSE scale):
    (Q tensor [m], metrics [4] = dp(m, p-1), MSE, H(I,B), H(Xhat))."""
    torch = _torch()
    x = _dev_f32(x)
    d = x.numel()
    if ws is None:
        nb = int(lib().ecasq_workspace_size_linear(d))
        if nb == 0:
            raise EcasqError(EINVAL, "ecasq_workspace_size_linear")
        ws = torch.empty(nb, dtype=torch.uint8, device=x.device)
    Q = torch.zeros(s, dtype=torch.float32, device=x.device)
    m = C.c_int32()
    met = np.zeros(4, np.float64)
    rc = lib().ecasq_dp_linear(_ptr(x), d, int(s), float(lambda_), int(flags), _ptr(ws), ws.numel(), _ptr(Q),
                               C.byref(m), met.ctypes.data_as(C.POINTER(C.c_double)), _stream())
    _check(rc, "ecasq_dp_linear")
    return Q[:m.value].clone(), met


def ecasq_dp_tables(ws, g, s, p_max):
    """DP tables of multiplier g of the last pass: (dp [(s+1), p] f64, bp [(s+1), p] i32) tensors."""
    torch = _torch()
    dp = torch.empty((s + 1) * p_max, dtype=torch.float64, device="cuda")
    bp = torch.empty((s + 1) * p_max, dtype=torch.int32, device="cuda")
    p = C.c_int64()
    rc = lib().ecasq_dp_tables(_ptr(ws), ws.numel(), int(g), _ptr(dp), _ptr(bp), C.byref(p), _stream())
    _check(rc, "ecasq_dp_tables")
    n = (s + 1) * p.value
    return dp[:n].view(s + 1, p.value), bp[:n].view(s + 1, p.value)


def ecasq_refine(x, Q, lambda_, budget_bits=-1.0, max_rounds=5, rel_tol=0.0, flags=0, ws=None):
    """Three-colour refinement (Sec. 6) of Q at multiplier lambda_; returns (Q, result dict)."""
    torch = _torch()
    x = _dev_f32(x)
    d = x.numel()
    Q = _dev_f32(Q).clone()
    m = Q.numel()
    if ws is None:
        ws = workspace(d, 2)
    res = Result()
    rc = lib().ecasq_refine(_ptr(x), d, _ptr(Q), m, float(lambda_), float(budget_bits), int(max_rounds),
                            float(rel_tol), int(flags), _ptr(ws), ws.numel(), C.byref(res), _stream())
    _check(rc, "ecasq_refine")
    return Q, res.as_dict()


def ecasq_evaluate(x, Q, ws=None):
    """(MSE, H(I,B), H(Xhat)) of a codebook Q subset of x."""
    x = _dev_f32(x)
    d = x.numel()
    Q = _dev_f32(Q)
    if ws is None:
        ws = workspace(d, 2)
    out = np.zeros(3, np.float64)
    rc = lib().ecasq_evaluate(_ptr(x), d, _ptr(Q), Q.numel(), _ptr(ws), ws.numel(),
                              out.ctypes.data_as(C.POINTER(C.c_double)), _stream())
    _check(rc, "ecasq_evaluate")
    return float(out[0]), float(out[1]), float(out[2])


def ecasq_quantize(x, Q, seed, ws=None, idx=None, counts=None):
    """Stochastic quantization (Sec. 2): (idx uint8 tensor, counts tensor, empirical entropy)."""
    torch = _torch()
    x = _dev_f32(x)
    d = x.numel()
    Q = _dev_f32(Q)
    m = Q.numel()
    if ws is None:
        ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    if idx is None:
        idx = torch.empty(d, dtype=torch.uint8, device=x.device)
    if counts is None:
        counts = torch.empty(m, dtype=torch.int32, device=x.device)
    _out_tensor(idx, d, (torch.uint8,), "ecasq_quantize", "idx")
    _out_tensor(counts, m, _count_dtypes(), "ecasq_quantize", "counts")
    if not (idx.device == x.device == counts.device == ws.device):
        raise EcasqError(EINVAL, "ecasq_quantize: x, idx, counts and ws must be on one device")
    he = C.c_double()
    rc = lib().ecasq_quantize(_ptr(x), d, _ptr(Q), m, C.c_uint64(int(seed) & 0xFFFFFFFFFFFFFFFF), _ptr(idx),
                              _ptr(counts), _ptr(ws), ws.numel(), C.byref(he), _stream())
    _check(rc, "ecasq_quantize")
    return idx, counts, he.value


def _out_tensor(t, n, dtypes, where, name):
    """An output buffer the kernel writes through a raw pointer: a contiguous CUDA tensor
    of one of `dtypes` with at least n elements (else EINVAL before any device work)."""
    torch = _torch()
    ok = (isinstance(t, torch.Tensor) and t.is_cuda and t.dtype in dtypes and t.is_contiguous()
          and t.numel() >= n)
    if not ok:
        raise EcasqError(EINVAL, "%s: %s must be a contiguous CUDA tensor of %s with at least %d elements"
                         % (where, name, "/".join(str(d) for d in dtypes), n))
    return t


def _count_dtypes():
    torch = _torch()
    u32 = getattr(torch, "uint32", None)
    return (torch.int32,) + ((u32,) if u32 is not None else ())


def ecasq_quantize_noalloc(x, Q, seed, idx, counts):
    """ecasq_quantize without a workspace; idx (uint8 [d]) and counts (int32 [m])
    are the caller's device tensors, on the device of x.  Returns the empirical entropy."""
    torch = _torch()
    where = "ecasq_quantize_noalloc"
    _out_tensor(idx, 0, (torch.uint8,), where, "idx")
    _out_tensor(counts, 0, _count_dtypes(), where, "counts")
    x = _dev_f32(x)
    Q = _dev_f32(Q)
    _out_tensor(idx, x.numel(), (torch.uint8,), where, "idx")
    _out_tensor(counts, Q.numel(), _count_dtypes(), where, "counts")
    if not (idx.device == x.device == Q.device == counts.device):
        raise EcasqError(EINVAL, "%s: x, Q, idx and counts must be on one device" % where)
    he = C.c_double()
    rc = lib().ecasq_quantize_noalloc(_ptr(x), x.numel(), _ptr(Q), Q.numel(),
                                      C.c_uint64(int(seed) & 0xFFFFFFFFFFFFFFFF), _ptr(idx), _ptr(counts),
                                      C.byref(he), _stream())
    _check(rc, "ecasq_quantize_noalloc")
    return he.value


class BatchResults:
    """The per-row results of ecasq_solve_batched as a read-only sequence of dicts, each
    built from the C records when it is read (building 10^4 dicts up front costs more
    than the solve of short rows)."""

    def __init__(self, records):
        self._records = records

    def __len__(self):
        return len(self._records)

    def __getitem__(self, i):
        if isinstance(i, slice):
            return [self._records[t].as_dict() for t in range(*i.indices(len(self._records)))]
        return self._records[i].as_dict()

    def __iter__(self):
        for r in self._records:
            yield r.as_dict()

    def field(self, name):
        """One field of every row, as a numpy array."""
        return np.array([getattr(r, "lambda_" if name == "lambda" else name) for r in self._records])


def ecasq_solve_batched(X, s, budget_bits=0.0, lambda_=-1.0, ws=None, **kw):
    """Independent budgeted solves of the rows of X [rows, d]: (Q [rows, s], m [rows], results);
    results is a BatchResults sequence (one dict per row, built when read)."""
    torch = _torch()
    X = _dev_f32(X)
    rows, d = X.shape
    if ws is None:
        ws = workspace(d, s, rows, flags=kw.get("flags", 0))
    prm = make_params(s, budget_bits, lambda_, **kw)
    Q = torch.zeros((rows, s), dtype=torch.float32, device="cuda")
    m = torch.zeros(rows, dtype=torch.int32, device="cuda")
    res = (Result * rows)()
    rc = lib().ecasq_solve_batched(_ptr(X), rows, d, C.byref(prm), _ptr(ws), ws.numel(), _ptr(Q), _ptr(m), res,
                                   _stream())
    _check(rc, "ecasq_solve_batched", ok=(OK, EINFEASIBLE))
    return Q, m, BatchResults(res)


def ecasq_prepare(x, ws=None):
    """Weighted histogram and App. E prefix sums: dict of tensors v, w, N, S, S2 and p."""
    torch = _torch()
    x = _dev_f32(x)
    d = x.numel()
    if ws is None:
        ws = torch.empty(int(lib().ecasq_workspace_size_prep(d)), dtype=torch.uint8, device="cuda")
    v = torch.empty(d, dtype=torch.float32, device="cuda")
    w = torch.empty(d, dtype=torch.int64, device="cuda")
    N = torch.empty(d + 1, dtype=torch.int64, device="cuda")
    S = torch.empty(2 * (d + 1), dtype=torch.float64, device="cuda")
    S2 = torch.empty(2 * (d + 1), dtype=torch.float64, device="cuda")
    p = C.c_int64()
    rc = lib().ecasq_prepare(_ptr(x), d, _ptr(ws), ws.numel(), _ptr(v), _ptr(w), _ptr(N), _ptr(S), _ptr(S2),
                             C.byref(p), _stream())
    _check(rc, "ecasq_prepare")
    p = p.value
    return dict(p=p, v=v[:p], w=w[:p], N=N[:p + 1], S_hi=S[:p + 1], S_lo=S[p + 1:2 * p + 2],
                S2_hi=S2[:p + 1], S2_lo=S2[p + 1:2 * p + 2])


def ecasq_kernel_launches() -> int:
    """Kernels the library has launched in this process so far."""
    return int(lib().ecasq_kernel_launches())
