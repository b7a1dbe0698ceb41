"""sieve_search_noalloc, the search entry point that allocates no device memory.

Some callers cannot call cudaMalloc: a host process without a device
allocator, a plug-in whose host application owns every allocation, code that
runs while the caller's own memory pool is being reset.  For them the library
offers an entry point whose scratch is a fixed array inside libsieve.  These
tests call it through the C ABI and check it against sieve_search, the
workspace-taking entry point, on two calls in a row (the second call runs on
the leftovers of the first), and check that a call needing more scratch than
the fixed array is refused.  This file is collected last on purpose."""
import ctypes as C

import numpy as np
import pytest
import torch

import paper_2608_03199_gb300 as sieve
import synth
from parity import TOL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def setup():
    assert torch.cuda.is_available()
    dev = torch.device("cuda:0")
    wl = synth.make_workload("tiny", device="cpu")
    index = sieve.build_layout(wl["X"].to(dev), wl["assign"].to(dev), 64, wl["centroids"].to(dev))
    return index, wl["Q"].to(dev), wl["qids"].to(dev), dev


def _noalloc(index, Q, qids, tau, k, nprobe, W, lookahead, outs, order=None, stats=True):
    v = index.view()
    p = sieve._params(tau, k, nprobe, W, lookahead, 0, 0)
    st = sieve.StatsC()
    rc = sieve.lib().sieve_search_noalloc(
        C.byref(v), C.c_void_p(Q.data_ptr()), Q.shape[0], C.c_void_p(qids.data_ptr()),
        None if order is None else C.c_void_p(order.data_ptr()),
        C.byref(p), C.c_void_p(outs[0].data_ptr()), C.c_void_p(outs[1].data_ptr()),
        C.c_void_p(outs[2].data_ptr()), C.c_void_p(outs[3].data_ptr()),
        C.byref(st) if stats else None, C.c_void_p(torch.cuda.current_stream().cuda_stream))
    torch.cuda.synchronize()
    return rc, st


def test_noalloc_matches_search_on_two_calls(setup):
    index, Q, qids, dev = setup
    nq, k = Q.shape[0], 10
    outs = (torch.empty((nq, k), dtype=torch.int64, device=dev),
            torch.empty((nq, k), dtype=torch.float32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev))
    for W, lookahead in ((4, True), (2, False)):
        ref = sieve.search(index, Q, 0.90, k, 16, W, lookahead=lookahead, query_ids=qids)
        torch.cuda.synchronize()
        for t in outs:
            t.fill_(7)
        rc, st = _noalloc(index, Q, qids, 0.90, k, 16, W, lookahead, outs)
        assert rc == 0, sieve.lib().sieve_status_str(rc)
        assert st.status == 0 and st.items == int(ref[3].sum().item())
        assert torch.equal(outs[0], ref[0])
        assert torch.equal(outs[2], ref[2]) and torch.equal(outs[3], ref[3])
        valid = (torch.arange(k, device=dev)[None, :] < ref[2][:, None])
        diff = (outs[1] - ref[1]).abs()[valid]
        assert diff.numel() == 0 or diff.max().item() <= TOL
        assert torch.isneginf(outs[1][~valid]).all()


def test_noalloc_refuses_calls_beyond_its_scratch(setup):
    index, Q, qids, dev = setup
    nq = 200_000
    big_Q = Q[:1].repeat(nq, 1).contiguous()
    big_ids = torch.zeros(nq, dtype=torch.int64, device=dev)
    need = sieve.workspace_size(index, nq, 0.90, 10, 16, 4)
    assert need > sieve.NOALLOC_SCRATCH_BYTES
    outs = (torch.empty((nq, 10), dtype=torch.int64, device=dev),
            torch.empty((nq, 10), dtype=torch.float32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev))
    rc, _ = _noalloc(index, big_Q, big_ids, 0.90, 10, 16, 4, True, outs)
    assert rc == -6
    assert sieve.lib().sieve_status_str(rc).startswith(b"call needs more scratch")


def test_noalloc_takes_no_device_memory(setup):
    """A repeated call (its kernels already loaded by the first) leaves the
    device's free memory where it was: the scratch is the fixed array."""
    index, Q, qids, dev = setup
    nq, k = Q.shape[0], 10
    outs = (torch.empty((nq, k), dtype=torch.int64, device=dev),
            torch.empty((nq, k), dtype=torch.float32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev))
    rc, _ = _noalloc(index, Q, qids, 0.90, k, 16, 4, True, outs, stats=False)
    assert rc == 0
    free_before = torch.cuda.mem_get_info(dev)[0]
    rc, _ = _noalloc(index, Q, qids, 0.90, k, 16, 4, True, outs, stats=False)
    free_after = torch.cuda.mem_get_info(dev)[0]
    assert rc == 0
    assert free_after >= free_before, (free_before, free_after)


def test_noalloc_reports_device_errors_without_stats(setup):
    """An order entry outside [0, nlist) is caught on the device; the
    host-driven rounds read the status word, so the call returns
    SIEVE_EINVAL even without a stats pointer."""
    index, Q, qids, dev = setup
    nq, k, nprobe = Q.shape[0], 10, 16
    order = sieve.rank_partitions(index, Q, nprobe)
    order[nq // 2, 0] = index.nlist          # one past the last partition
    outs = (torch.empty((nq, k), dtype=torch.int64, device=dev),
            torch.empty((nq, k), dtype=torch.float32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev))
    rc, _ = _noalloc(index, Q, qids, 0.90, k, nprobe, 4, True, outs, order=order, stats=False)
    assert rc == -1
    # and the same array serves a correct call right after
    ref = sieve.search(index, Q, 0.90, k, nprobe, 4, query_ids=qids)
    rc, _ = _noalloc(index, Q, qids, 0.90, k, nprobe, 4, True, outs, stats=False)
    assert rc == 0 and torch.equal(outs[0], ref[0]) and torch.equal(outs[3], ref[3])
