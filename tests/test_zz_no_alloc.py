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
    """After the first call on the device (set-up), further calls make no allocation
    through torch's allocator and take no device memory of their own: a cudaMalloc
    reserves at least a 2 MiB page, so the device's free memory may move by less than
    that (other users of the GPU) but must not drop by a page."""
    import torch
    x, Q = _case(1 << 16, 13)
    xg = torch.as_tensor(x).cuda()
    Qg = torch.as_tensor(Q).cuda()
    idx = torch.empty(x.size, dtype=torch.uint8, device="cuda")
    cnt = torch.empty(Qg.numel(), dtype=torch.int32, device="cuda")
    E.ecasq_quantize_noalloc(xg, Qg, 0, idx, cnt)
    torch.cuda.synchronize()
    n_alloc0 = torch.cuda.memory_stats().get("allocation.all.allocated", 0)
    reserved0 = torch.cuda.memory_reserved()
    free0 = torch.cuda.mem_get_info()[0]
    for seed in (1, 2):
        E.ecasq_quantize_noalloc(xg, Qg, seed, idx, cnt)
    torch.cuda.synchronize()
    assert torch.cuda.memory_stats().get("allocation.all.allocated", 0) == n_alloc0
    assert torch.cuda.memory_reserved() == reserved0
    assert free0 - torch.cuda.mem_get_info()[0] < 2 * 2 ** 20


def test_noalloc_rejects_bad_output_buffers_before_launch(E):
    """idx and counts are written through raw pointers: a buffer that is too short, of
    the wrong type, not contiguous or on the host is refused (EINVAL) and left untouched."""
    import torch
    x, Q = _case(4096, 21)
    xg = torch.as_tensor(x).cuda()
    Qg = torch.as_tensor(Q).cuda()
    m = Qg.numel()
    good_idx = torch.full((x.size,), 7, dtype=torch.uint8, device="cuda")
    good_cnt = torch.full((m,), 7, dtype=torch.int32, device="cuda")
    bad = [
        (torch.empty(x.size - 1, dtype=torch.uint8, device="cuda"), good_cnt),           # idx too short
        (good_idx, torch.empty(m - 1, dtype=torch.int32, device="cuda")),                # counts too short
        (torch.empty(x.size, dtype=torch.int32, device="cuda"), good_cnt),               # idx not uint8
        (good_idx, torch.empty(m, dtype=torch.float32, device="cuda")),                  # counts not int32
        (torch.empty(2 * x.size, dtype=torch.uint8, device="cuda")[::2], good_cnt),      # idx strided
        (torch.empty(x.size, dtype=torch.uint8), good_cnt),                              # idx on the host
        (good_idx, torch.empty(m, dtype=torch.int32)),                                   # counts on the host
    ]
    for idx, cnt in bad:
        with pytest.raises(E.EcasqError) as ei:
            E.ecasq_quantize_noalloc(xg, Qg, 1, idx, cnt)
        assert ei.value.code == E.native.EINVAL
    torch.cuda.synchronize()
    assert bool((good_idx == 7).all()) and bool((good_cnt == 7).all())


def test_noalloc_rejects_sizes_beyond_its_limits(E):
    import ctypes as C
    L = E.lib()
    p = C.c_void_p(256)
    he = C.c_double()
    assert L.ecasq_quantize_noalloc(p, 16, p, 257, 0, p, p, C.byref(he), None) == E.native.EINVAL  # m > 256
    assert L.ecasq_quantize_noalloc(p, 1 << 31, p, 4, 0, p, p, C.byref(he), None) == E.native.EINVAL  # d >= 2^31
    assert L.ecasq_quantize_noalloc(p, 0, p, 4, 0, p, p, C.byref(he), None) == E.native.EINVAL
    assert L.ecasq_quantize_noalloc(None, 16, p, 4, 0, p, p, C.byref(he), None) == E.native.EINVAL
