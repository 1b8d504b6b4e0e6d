"""pe_fleet_windows_noalloc: the fleet window counts for callers that cannot
allocate device memory (their device memory belongs to another allocator,
or their control loop must not add allocations to its timeline).  It must
give exactly the results of pe_fleet_windows with a caller workspace, and of
the CPU oracle, call after call, although every call reuses the same fixed
scratch array that keeps the previous call's contents.  Collected last on
purpose."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_11226_gb300 import pe
from paper_2608_11226_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_11226_gb300 import build
    build.build()
    assert torch.cuda.is_available()


def _inputs(n, length, seed):
    fw = W.make_fleet(n_compositions=n, length=length, seed=seed)
    dev = [torch.from_numpy(x).cuda() for x in (fw.traces, fw.job_of_gpu, fw.offsets)]
    return fw, dev


def _with_workspace(fw, dev, windows):
    N = fw.offsets.shape[0]
    counts = torch.empty((N, len(windows)), dtype=torch.int32, device="cuda")
    peaks = torch.empty_like(counts)
    ws = torch.empty(pe.fleet_workspace_bytes(fw.n_jobs, fw.traces.shape[1], fw.horizon),
                     dtype=torch.uint8, device="cuda")
    pe.fleet_windows(dev[0], dev[1], fw.n_jobs, dev[2], fw.horizon, windows, fw.budget_q, counts,
                     peaks, ws)
    torch.cuda.synchronize()
    return counts.cpu().numpy(), peaks.cpu().numpy()


def _noalloc(fw, dev, windows, stream=None):
    N = fw.offsets.shape[0]
    counts = torch.full((N, len(windows)), -7, dtype=torch.int32, device="cuda")
    peaks = torch.full_like(counts, -7)
    torch.cuda.synchronize()
    pe.fleet_windows_noalloc(dev[0], dev[1], fw.n_jobs, dev[2], fw.horizon, windows, fw.budget_q,
                             counts, peaks, stream=stream)
    torch.cuda.synchronize()
    return counts.cpu().numpy(), peaks.cpu().numpy()


def _oracle(fw, windows):
    return O.fleet_windows(fw.traces, fw.job_of_gpu, fw.n_jobs, fw.offsets, fw.horizon, windows,
                           fw.budget_q)


def test_noalloc_matches_workspace_entry_point_two_calls_in_a_row():
    # two different calls back to back: a larger one, then a smaller one that
    # leaves part of the previous call's scratch contents untouched
    for n, length, seed, windows in ((300, 40000, 0, [1, 60, 600]), (97, 2500, 5, [1, 20, 60, 600])):
        fw, dev = _inputs(n, length, seed)
        c_ref, p_ref = _with_workspace(fw, dev, windows)
        c, p = _noalloc(fw, dev, windows)
        assert np.array_equal(c, c_ref) and np.array_equal(p, p_ref)
        if n < 100:
            oc, op = _oracle(fw, windows)
            assert np.array_equal(c, oc) and np.array_equal(p, op)


def _fits(length):
    """Whether a fleet of trace length `length` (H = L) fits the static
    scratch: the entry point rejects an oversized request on the host, before
    touching any device buffer."""
    fw = W.make_fleet(n_compositions=1, length=1000, seed=0)
    tr = torch.zeros((fw.traces.shape[0], length), dtype=torch.float32, device="cuda")
    job = torch.from_numpy(fw.job_of_gpu).cuda()
    off = torch.zeros((1, fw.n_jobs), dtype=torch.int32, device="cuda")
    c = torch.zeros((1, 1), dtype=torch.int32, device="cuda")
    try:
        # N = 0: nothing is counted even when the request fits
        pe.fleet_windows_noalloc(tr, job, fw.n_jobs, off[:0], length, [1], fw.budget_q, c, c)
        return True
    except pe.PEError as e:
        assert e.status == pe.PE_EINVAL and "static scratch" in str(e)
        return False


def test_noalloc_just_under_its_limit_and_on_a_side_stream():
    """The largest fleet that fits (one prefix copy filling the array up to
    its last words, where the maxima and the flag sit), on a non-default
    stream, against the workspace entry point and the oracle."""
    lo, hi = 2000, 200000
    assert _fits(lo) and not _fits(hi)
    while hi - lo > 1:
        mid = (lo + hi) // 2
        lo, hi = (mid, hi) if _fits(mid) else (lo, mid)
    fw, dev = _inputs(6, lo, 11)
    windows = [1, 60, 600]
    side = torch.cuda.Stream()
    c, p = _noalloc(fw, dev, windows, stream=side)
    c_ref, p_ref = _with_workspace(fw, dev, windows)
    oc, op = _oracle(fw, windows)
    assert np.array_equal(c, c_ref) and np.array_equal(p, p_ref)
    assert np.array_equal(c, oc) and np.array_equal(p, op)
    # a second call in a row on the default stream, after the near-full one
    fw2, dev2 = _inputs(40, 3000, 12)
    c2, p2 = _noalloc(fw2, dev2, windows)
    oc2, op2 = _oracle(fw2, windows)
    assert np.array_equal(c2, oc2) and np.array_equal(p2, op2)


def test_noalloc_zero_compositions_is_a_noop():
    fw, dev = _inputs(1, 3000, 2)
    counts = torch.full((1, 3), -7, dtype=torch.int32, device="cuda")
    pe.fleet_windows_noalloc(dev[0], dev[1], fw.n_jobs, dev[2][:0], fw.horizon, [1, 60, 600],
                             fw.budget_q, counts, counts)
    torch.cuda.synchronize()
    assert (counts.cpu().numpy() == -7).all()


def test_noalloc_rejects_requests_beyond_its_scratch():
    fw, dev = _inputs(4, 380000, 0)   # 8 jobs x 760,000 int32 = 24 MB > 4 MiB
    counts = torch.zeros((4, 3), dtype=torch.int32, device="cuda")
    peaks = torch.zeros_like(counts)
    with pytest.raises(pe.PEError) as e:
        pe.fleet_windows_noalloc(dev[0], dev[1], fw.n_jobs, dev[2], fw.horizon, [1, 60, 600],
                                 fw.budget_q, counts, peaks)
    assert e.value.status == pe.PE_EINVAL and "static scratch" in str(e.value)
    torch.cuda.synchronize()
    assert int(counts.abs().sum()) == 0
