"""Bounded device waits give up cleanly (failure detection without a GPU fault).

Every wait inside the tensor-core pipelines is an mbarrier poll with an
iteration limit.  ``wait_limit`` shortens the limit of one of them, the scan
epilogue's wait for an accumulator, which has no asynchronous work of its own
outstanding; the copies and MMAs the kernel issued are still drained with the
full limit before it frees its tensor memory and returns.  With a limit of one
poll that wait gives up (the MMAs of a tile take far longer than one poll), the
call reports SIEVE_ETIMEOUT, and the same context then runs a correct search.
"""
import pytest
import torch

import paper_2608_03199_gb300 as sieve
import synth

pytestmark = pytest.mark.gpu

ETIMEOUT = -7


@pytest.fixture(scope="module")
def setup():
    assert torch.cuda.is_available()
    dev = torch.device("cuda:0")
    wl = synth.make_workload("tiny", device="cpu")
    c = wl["cfg"]
    index = sieve.build_layout(wl["X"].to(dev), wl["assign"].to(dev), c.nlist,
                               wl["centroids"].to(dev))
    assert index.tc_rows is not None   # the bulk tensor-core scan runs
    Q, qids = wl["Q"].to(dev), wl["qids"].to(dev)
    order = sieve.rank_partitions(index, Q, c.nprobe)
    return c, index, Q, qids, order


def _same(a, b):
    return all(torch.equal(x, y) for x, y in zip(a[:4], b[:4]))


@pytest.mark.parametrize("scan_path", ["tensor", "screen"])
def test_epilogue_wait_gives_up_and_the_context_survives(setup, scan_path):
    c, index, Q, qids, order = setup
    kw = dict(query_ids=qids, order=order, scan_path=scan_path)
    ref = sieve.search(index, Q, c.tau, c.k, c.nprobe, c.W, **kw)
    torch.cuda.synchronize()
    timeouts = 0
    for trial in range(4):
        loop = trial % 2          # host-driven rounds return the status without stats
        try:
            out = sieve.search(index, Q, c.tau, c.k, c.nprobe, c.W, loop=loop, stats=True,
                               wait_limit=1, **kw)
            # the wait may have been met within its single poll: then the
            # search is complete and must be exact
            assert _same(out, ref)
        except sieve.SieveError as e:
            assert e.status == ETIMEOUT, e
            timeouts += 1
        # the next search on the same context and workspace is correct
        again = sieve.search(index, Q, c.tau, c.k, c.nprobe, c.W, stats=True, **kw)
        assert again[4]["status"] == 0
        assert _same(again, ref)
    assert timeouts >= 1, "a one-poll accumulator wait never gave up"


def test_graph_mode_timeout_is_read_back(setup):
    """In graph mode without stats the call returns at once; the status word
    read afterwards (sieve_search_status) holds SIEVE_ETIMEOUT."""
    c, index, Q, qids, order = setup
    ws = sieve.Workspace()
    seen = []
    for _ in range(3):
        sieve.search(index, Q, c.tau, c.k, c.nprobe, c.W, query_ids=qids, order=order,
                     workspace=ws, wait_limit=1, scan_path="tensor")
        seen.append(sieve.search_status(ws))
    assert set(seen) <= {0, ETIMEOUT} and ETIMEOUT in seen
    ref = sieve.search(index, Q, c.tau, c.k, c.nprobe, c.W, query_ids=qids, order=order,
                       scan_path="tensor")
    out = sieve.search(index, Q, c.tau, c.k, c.nprobe, c.W, query_ids=qids, order=order,
                       workspace=ws, scan_path="tensor", check=True)
    assert sieve.search_status(ws) == 0
    assert _same(out, ref)
