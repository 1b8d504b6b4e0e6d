"""pe_fleet_windows_noalloc: the fleet window counts for callers that cannot
allocate device memory (their device memory belongs to another allocator,
or their control loop cannot afford an allocation's synchronisation).  It
must give exactly the results of pe_fleet_windows with a caller workspace,
call after call, although every call reuses the same fixed scratch array
that keeps the previous call's contents.  Collected last on purpose."""
import numpy as np
import pytest
import torch

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


def _noalloc(fw, dev, windows):
    N = fw.offsets.shape[0]
    counts = torch.full((N, len(windows)), -7, dtype=torch.int32, device="cuda")
    peaks = torch.full_like(counts, -7)
    pe.fleet_windows_noalloc(dev[0], dev[1], fw.n_jobs, dev[2], fw.horizon, windows, fw.budget_q,
                             counts, peaks)
    torch.cuda.synchronize()
    return counts.cpu().numpy(), peaks.cpu().numpy()


def test_noalloc_matches_workspace_entry_point_two_calls_in_a_row():
    # two different calls back to back: a larger one, then a smaller one that
    # leaves part of the previous call's scratch contents untouched
    for n, length, seed, windows in ((300, 40000, 0, [1, 60, 600]), (97, 2500, 5, [1, 20, 60, 600])):
        fw, dev = _inputs(n, length, seed)
        c_ref, p_ref = _with_workspace(fw, dev, windows)
        c, p = _noalloc(fw, dev, windows)
        assert np.array_equal(c, c_ref) and np.array_equal(p, p_ref)


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
