"""The min-plus wavefront's bounded device waits (run on a GB300: pytest -m gpu).

A column block of the wavefront may be consumed only after its owner published it;
every wait on such a flag gives up after a spin limit, records a timeout in the
workspace's status record, raises the kernel's abort flag (so the other CTAs stop
waiting too) and returns.  The ECASQ_TEST_STALL hook makes that happen on purpose
without faulting anything: block 0 is never published and the spin limit drops to
2^14 spins.  The call must return ECASQ_ETIMEOUT within a short time, and the next
call on the same workspace must run normally and give the same results as a call on
a fresh workspace.
"""
import time

import numpy as np
import pytest

from paper_2608_18147_gb300 import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def E():
    import torch
    assert torch.cuda.is_available(), "these tests need a CUDA GPU"
    import paper_2608_18147_gb300 as E
    E.lib()
    return E


@pytest.mark.parametrize("resident", [True, False])
def test_stalled_block_times_out_and_workspace_recovers(E, resident):
    import torch
    x = workloads.student_t(3000, 8, scale=1.0)
    s = 16
    lams = [0.0, 0.01, 0.1, 1.0]
    flags = E.RESIDENT_COSTS if resident else 0
    ws = E.workspace(x.size, s, flags=flags)
    Q0, m0, met0 = E.ecasq_dp_pass(x, s, lams, flags=flags, ws=ws)
    for attempt in range(2):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        with pytest.raises(E.EcasqError) as ei:
            E.ecasq_dp_pass(x, s, lams, flags=flags | E.TEST_STALL, ws=ws)
        dt = time.perf_counter() - t0
        assert ei.value.code == E.native.ETIMEOUT
        assert dt < 20.0  # every CTA stopped waiting: the abort flag reached them
        st = E.native.ws_status(ws)
        assert st["timeout"] == 1
        # the same workspace, a normal call: same codebooks and metrics as before the stall
        Q1, m1, met1 = E.ecasq_dp_pass(x, s, lams, flags=flags, ws=ws)
        assert E.native.ws_status(ws)["timeout"] == 0
        assert m1 == m0
        assert torch.equal(Q1, Q0)
        np.testing.assert_array_equal(met1, met0)


def test_stalled_solve_reports_timeout(E):
    """The budgeted solve passes the status through (no partial answer)."""
    x = workloads.signed_lognormal(2500, 9)
    with pytest.raises(E.EcasqError) as ei:
        E.ecasq_solve(x, 8, budget_bits=2.0, flags=E.TEST_STALL)
    assert ei.value.code == E.native.ETIMEOUT
    Q, res = E.ecasq_solve(x, 8, budget_bits=2.0)
    assert res["status"] == 0 and res["m"] >= 2
