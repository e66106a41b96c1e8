"""Host-side pieces of the ctypes binding (no GPU): the structures it passes through the
C ABI have the header's layout, and the batched solve's result sequence behaves as a
read-only sequence of dicts."""
import os
import re
import subprocess

import numpy as np
import pytest

from conftest import ROOT

STRUCTS = {"ecasq_params_t": "Params", "ecasq_result_t": "Result", "ecasq_timeshare_t": "Timeshare"}


def _header_fields(txt, tname):
    body = re.search(r"typedef struct \w+ \{([^}]*)\} %s;" % tname, txt).group(1)
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    names = []
    for decl in body.split(";"):
        decl = decl.strip()
        if decl:
            names += [n.strip() for n in decl.split(None, 1)[1].split(",")]
    return names


def test_struct_layouts_match_the_header(tmp_path):
    """sizeof and every field offset of the three structures, from a C program compiled
    against include/ecasq.h, equal the ctypes structures' (field names map lambda <-> lambda_)."""
    from paper_2608_18147_gb300 import native
    with open(os.path.join(ROOT, "include", "ecasq.h")) as f:
        txt = f.read()
    src = ["#include <stdio.h>", "#include <stddef.h>", '#include "ecasq.h"', "int main(void) {"]
    fields = {}
    for tname in STRUCTS:
        fields[tname] = _header_fields(txt, tname)
        src.append('printf("%s sizeof %%zu\\n", sizeof(%s));' % (tname, tname))
        for f in fields[tname]:
            src.append('printf("%s %s %%zu\\n", offsetof(%s, %s));' % (tname, f, tname, f))
    src += ["return 0;", "}"]
    c = tmp_path / "layout.c"
    c.write_text("\n".join(src))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(c), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split("\n")
    got = {(a, b): int(v) for a, b, v in (line.split() for line in out if line)}
    for tname, cls in STRUCTS.items():
        S = getattr(native, cls)
        assert [("lambda" if n == "lambda_" else n) for n, _ in S._fields_] == fields[tname], tname
        assert got[(tname, "sizeof")] == __import__("ctypes").sizeof(S), tname
        for n, _ in S._fields_:
            assert got[(tname, "lambda" if n == "lambda_" else n)] == getattr(S, n).offset, (tname, n)


def test_batch_results_is_a_lazy_sequence_of_dicts():
    from paper_2608_18147_gb300 import native
    recs = (native.Result * 3)()
    for i, r in enumerate(recs):
        r.m, r.lambda_, r.mse, r.status = 4 + i, 0.5 * i, 1.0 + i, (0, -3, 0)[i]
    res = native.BatchResults(recs)
    assert len(res) == 3
    assert res[1]["m"] == 5 and res[1]["lambda"] == 0.5 and res[1]["status"] == -3
    assert res[-1]["mse"] == 3.0
    assert [d["m"] for d in res] == [4, 5, 6]
    assert [d["m"] for d in res[1:]] == [5, 6]
    assert res[0] == recs[0].as_dict()
    np.testing.assert_array_equal(res.field("lambda"), [0.0, 0.5, 1.0])
    np.testing.assert_array_equal(res.field("status"), [0, -3, 0])
    with pytest.raises(IndexError):
        res[3]
