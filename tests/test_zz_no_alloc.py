"""ecasq_quantize_noalloc (fixed device scratch, no workspace) against
ecasq_quantize on the same inputs: identical indices, counts and empirical
entropy, on consecutive calls.  The file name sorts last so that it also runs
after every other test module (it must pass alone and after them)."""
import numpy as np
import pytest

from paper_2608_18147_gb300 import workloads

pytestmark = pytest.mark.gpu

H_RTOL = 1e-12  # empirical entropy: same counts, same host arithmetic


@pytest.fixture(scope="module")
def E():
    import torch
    assert torch.cuda.is_available(), "these tests need a CUDA GPU"
    import paper_2608_18147_gb300 as E
    E.lib()
    return E


def _case(d, seed):
    x = workloads.student_t(d, seed, scale=1.0)
    Q = np.unique(np.concatenate([[x.min(), x.max()],
                                  np.quantile(x, [0.1, 0.3, 0.5, 0.8]).astype(np.float32)]).astype(np.float32))
    return x, np.sort(Q)


@pytest.mark.parametrize("d", [1, 1000, 100003])
def test_noalloc_matches_workspace_entry_point_on_consecutive_calls(E, d):
    import torch
    x, Q = _case(d, 5)
    xg = torch.as_tensor(x).cuda()
    Qg = torch.as_tensor(Q).cuda()
    m = Qg.numel()
    for seed in (3, 2 ** 64 - 1):  # two calls in a row, each checked
        idx_ref, cnt_ref, h_ref = E.ecasq_quantize(xg, Qg, seed)
        idx = torch.empty(d, dtype=torch.uint8, device="cuda")
        cnt = torch.empty(m, dtype=torch.int32, device="cuda")
        h = E.ecasq_quantize_noalloc(xg, Qg, seed, idx, cnt)
        assert torch.equal(idx, idx_ref)
        assert torch.equal(cnt, cnt_ref)
        assert h == pytest.approx(h_ref, rel=H_RTOL, abs=1e-15)


def test_noalloc_error_flag_starts_at_zero_on_every_call(E):
    """An out-of-range call sets the scratch's error flag; the next valid call
    must not see it (every call zeroes the flag before its launch)."""
    import torch
    x, Q = _case(4096, 9)
    xg = torch.as_tensor(x).cuda()
    Qg = torch.as_tensor(Q).cuda()
    idx = torch.empty(x.size, dtype=torch.uint8, device="cuda")
    cnt = torch.empty(Qg.numel(), dtype=torch.int32, device="cuda")
    narrow = Qg[1:-1].contiguous()  # x reaches outside [narrow[0], narrow[-1]]: the kernel's own check flags it
    with pytest.raises(E.EcasqError) as ei:
        E.ecasq_quantize_noalloc(xg, narrow, 1, idx, torch.empty(narrow.numel(), dtype=torch.int32, device="cuda"))
    assert ei.value.code == E.native.ERANGE
    for seed in (1, 2):
        h = E.ecasq_quantize_noalloc(xg, Qg, seed, idx, cnt)
        idx_ref, cnt_ref, h_ref = E.ecasq_quantize(xg, Qg, seed)
        assert torch.equal(idx, idx_ref) and torch.equal(cnt, cnt_ref)
        assert h == pytest.approx(h_ref, rel=H_RTOL, abs=1e-15)


def test_noalloc_takes_no_device_memory(E):
    """After the first call on the device (set-up), further calls leave the
    device's free memory unchanged."""
    import torch
    x, Q = _case(1 << 16, 13)
    xg = torch.as_tensor(x).cuda()
    Qg = torch.as_tensor(Q).cuda()
    idx = torch.empty(x.size, dtype=torch.uint8, device="cuda")
    cnt = torch.empty(Qg.numel(), dtype=torch.int32, device="cuda")
    E.ecasq_quantize_noalloc(xg, Qg, 0, idx, cnt)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for seed in (1, 2):
        E.ecasq_quantize_noalloc(xg, Qg, seed, idx, cnt)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0


def test_noalloc_rejects_sizes_beyond_its_limits(E):
    import ctypes as C
    L = E.lib()
    p = C.c_void_p(256)
    he = C.c_double()
    assert L.ecasq_quantize_noalloc(p, 16, p, 257, 0, p, p, C.byref(he), None) == E.native.EINVAL  # m > 256
    assert L.ecasq_quantize_noalloc(p, 1 << 31, p, 4, 0, p, p, C.byref(he), None) == E.native.EINVAL  # d >= 2^31
    assert L.ecasq_quantize_noalloc(p, 0, p, 4, 0, p, p, C.byref(he), None) == E.native.EINVAL
    assert L.ecasq_quantize_noalloc(None, 16, p, 4, 0, p, p, C.byref(he), None) == E.native.EINVAL
