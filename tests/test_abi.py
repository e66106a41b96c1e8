"""The C-ABI library builds, loads and exports every symbol include/ecasq.h
declares (no GPU needed: nothing here launches a kernel)."""
import os
import re

import pytest

from conftest import ROOT


def declared_symbols():
    with open(os.path.join(ROOT, "include", "ecasq.h")) as f:
        txt = f.read()
    return sorted(set(re.findall(r"\b(ecasq_[a-z_]+)\s*\(", txt)))


def test_header_declares_the_entry_points():
    names = declared_symbols()
    for n in ("ecasq_solve", "ecasq_refine", "ecasq_quantize", "ecasq_solve_batched", "ecasq_workspace_size",
              "ecasq_dp_pass", "ecasq_strerror"):
        assert n in names


def test_library_exports_every_declared_symbol():
    import ctypes
    from paper_2608_18147_gb300 import native
    L = native.lib()
    missing = [n for n in declared_symbols() if not hasattr(L, n)]
    assert not missing, missing
    # exported with C linkage (no mangling), visible to dlsym
    for n in declared_symbols():
        assert ctypes.cast(getattr(L, n), ctypes.c_void_p).value


def test_host_only_calls():
    from paper_2608_18147_gb300 import native
    L = native.lib()
    assert L.ecasq_version() >= 10000
    assert L.ecasq_strerror(0) == b"ok"
    assert b"workspace" in L.ecasq_strerror(-4)
    assert native.ecasq_workspace_size(1024, 8) > 1024 * 4
    assert native.ecasq_workspace_size(0, 8) == 0
    assert native.ecasq_workspace_size(100, 1) == 0
    assert native.ecasq_workspace_size(100, 257) == 0
    # resident interval costs: 35328 bytes per 64 x 64 tile (C, Phi, column minima) on top of the base size
    base = native.ecasq_workspace_size(4096, 8)
    assert native.ecasq_workspace_size_flags(4096, 8, 1, 0) == base
    assert native.ecasq_workspace_size_flags(4096, 8, 1, native.RESIDENT_COSTS) == base + 64 * 65 // 2 * 35328
    assert native.ecasq_workspace_size_flags(2 ** 31 - 1, 8, 1, native.RESIDENT_COSTS) == 0  # beyond size_t
    assert native.ecasq_workspace_size_flags(0, 8, 1, native.RESIDENT_COSTS) == 0
    # preparation alone: the sort, histogram and sums (linear in d), far below a solve's
    assert 80 * 2 ** 20 < native.lib().ecasq_workspace_size_prep(2 ** 20) < 100 * 2 ** 20
    assert native.lib().ecasq_workspace_size_prep(0) == 0
    assert native.lib().ecasq_workspace_size_prep(2 ** 20) < native.ecasq_workspace_size(2 ** 20, 2)
    # workspace grows with d and s
    assert native.ecasq_workspace_size(4096, 16) > native.ecasq_workspace_size(4096, 8)
    assert native.ecasq_workspace_size(8192, 8) > native.ecasq_workspace_size(4096, 8)


def test_bad_arguments_rejected_before_any_launch():
    import ctypes as C
    from paper_2608_18147_gb300 import native
    L = native.lib()
    prm = native.make_params(1, 2.0)  # s < 2
    res = native.Result()
    assert L.ecasq_solve(None, 10, C.byref(prm), None, 0, None, C.byref(res), None) == native.EINVAL
    prm = native.make_params(8, -1.0)  # budget < 0 in search mode
    assert L.ecasq_solve(C.c_void_p(256), 10, C.byref(prm), C.c_void_p(256), 1 << 30, C.c_void_p(256),
                         C.byref(res), None) == native.EINVAL
    prm = native.make_params(8, 2.0)
    # misaligned / too small workspace
    assert L.ecasq_solve(C.c_void_p(256), 10, C.byref(prm), C.c_void_p(257), 1 << 30, C.c_void_p(256),
                         C.byref(res), None) == native.EWORKSPACE
    assert L.ecasq_solve(C.c_void_p(256), 10, C.byref(prm), C.c_void_p(256), 16, C.c_void_p(256),
                         C.byref(res), None) == native.EWORKSPACE
    # time-sharing needs a budget search without refinement (Sec. 7)
    ts = native.Timeshare()
    v = C.c_void_p(256)
    for bad in (native.make_params(8, 2.0, 0.5), native.make_params(8, 2.0, refine_max_rounds=2)):
        assert L.ecasq_solve_timeshare(v, 10, None, 0, C.byref(bad), v, 1 << 30, v, v, C.byref(res), C.byref(ts),
                                       None) == native.EINVAL
    assert L.ecasq_solve_timeshare(v, 10, None, 0, C.byref(prm), v, 1 << 30, v, v, C.byref(res), None,
                                   None) == native.EINVAL
    rate = C.c_double()
    for beta, mp in ((1.5, 2), (-0.1, 2), (0.5, 0)):
        assert L.ecasq_quantize_timeshare(v, 10, v, 2, v, mp, beta, 1, 2, v, None, v, v, 256, C.byref(rate),
                                          None) == native.EINVAL


def test_product_path_does_not_touch_the_oracle():
    pkg = os.path.join(ROOT, "paper_2608_18147_gb300")
    for dirpath, _, files in os.walk(pkg):
        if "_build" in dirpath:
            continue
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                with open(os.path.join(dirpath, f)) as fh:
                    txt = fh.read()
                assert "import oracle" not in txt and "from oracle" not in txt, f
                assert "ecasq_oracle" not in txt and "liboracle" not in txt, f


def test_quantize_wrappers_refuse_host_output_buffers():
    """The bindings pass idx and counts to the kernel as raw device pointers, so they
    refuse anything that is not a CUDA tensor of the right type (EINVAL) before any call
    into the library or any device work."""
    import numpy as np
    import torch
    from paper_2608_18147_gb300 import native
    x = np.linspace(-1.0, 1.0, 64, dtype=np.float32)
    Q = np.float32([-1.0, 0.0, 1.0])
    cases = [(np.zeros(64, np.uint8), np.zeros(3, np.int32)),
             (torch.zeros(64, dtype=torch.uint8), torch.zeros(3, dtype=torch.int32)),
             (torch.zeros(64, dtype=torch.int64), torch.zeros(3, dtype=torch.int32)),
             (None, None)]
    for idx, cnt in cases:
        with pytest.raises(native.EcasqError) as ei:
            native.ecasq_quantize_noalloc(x, Q, 0, idx, cnt)
        assert ei.value.code == native.EINVAL


def test_binding_constants_match_the_header():
    """Every ECASQ_* flag and status code the header defines has the same value in the
    binding (native.py restates them for ctypes callers)."""
    from paper_2608_18147_gb300 import native
    with open(os.path.join(ROOT, "include", "ecasq.h")) as f:
        txt = f.read()
    defs = {}
    for name, val in re.findall(r"^#define\s+ECASQ_([A-Z0-9_]+)\s+([-()0-9u <]+?)\s*(?:/\*|$)", txt, re.M):
        expr = re.sub(r"(\d)u\b", r"\1", val)  # 1u << 30, (-1), 256u
        assert re.fullmatch(r"[-()0-9 <]+", expr), (name, val)
        defs[name] = eval(expr, {"__builtins__": {}})
    codes = {"OK", "EINVAL", "ENONFINITE", "EINFEASIBLE", "EWORKSPACE", "ECUDA", "ETIMEOUT", "ERANGE"}
    flags = {"EXACT_S", "NO_REFINE_GUARD", "DP_REFERENCE", "TIME_KERNELS", "EXACT_TABLES", "RESIDENT_COSTS",
             "STREAMED_COSTS", "ONE_PART_PUBLISH", "UNSEEDED_SEARCH", "TEST_STALL", "TEST_SELF_SEED"}
    for name in codes | flags:
        assert name in defs, name
        assert getattr(native, name) == defs[name], (name, getattr(native, name), defs[name])
    assert len({defs[n] for n in flags}) == len(flags)  # distinct bits
    assert all(bin(defs[n]).count("1") == 1 for n in flags)
