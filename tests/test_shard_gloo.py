"""The multi-process host logic on CPU: world_size-2 gloo process groups.

Queries shard over processes with the index replicated (a query's result
depends only on the query and the index, Algorithm 1 / Sec. 4.3), so the
only exchange is the host-side gather of the shards' results.  The per-rank
search here is the oracle (no GPU); what is under test is the sharding, the
gather, the timing reductions and the per-rank inputs of the weak-scaling
bench.
"""
import os
import socket
import sys

import numpy as np
import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _small_cfg():
    import synth
    return synth.scaled("tiny", n=6_000, d=32, ncomp=12, nlist=40, nq=203, dup_frac=0.08,
                        dup_counts=("uniform", 2, 8), dup_sigma=(0.03, 0.08), tau=0.88,
                        nprobe=12, W=3, seed=21)


def _worker(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import oracle
        import synth
        from paper_2608_03199_gb300 import shard

        cfg = _small_cfg()
        w = synth.to_numpy(synth.make_workload(cfg, device="cpu"))
        idx = {k: w[k] for k in ("X", "ids", "assign", "centroids")}
        lo, hi = shard.query_shard(cfg.nq, world, rank)
        part = oracle.search(idx, w["Q"][lo:hi], cfg.tau, cfg.k, cfg.nprobe, cfg.W,
                             qids=w["qids"][lo:hi], threads=1)
        ids, sc, cnt, pr = shard.gather_results(part["ids"], part["scores"], part["count"],
                                                part["probes"], cfg.nq)
        full = oracle.search(idx, w["Q"], cfg.tau, cfg.k, cfg.nprobe, cfg.W, qids=w["qids"],
                             threads=1)
        assert np.array_equal(ids.numpy(), full["ids"])
        assert np.array_equal(sc.numpy(), full["scores"].astype(np.float32))
        assert np.array_equal(cnt.numpy(), full["count"])
        assert np.array_equal(pr.numpy(), full["probes"])

        # reductions used by the bench timing
        assert shard.max_over_ranks(1.5 + rank) == 1.5 + world - 1
        assert shard.sum_over_ranks(rank + 1) == world * (world + 1) / 2
        shard.barrier()

        # weak-scaling inputs: the same index on every rank, a different query batch
        wr = synth.to_numpy(synth.make_workload(cfg, device="cpu", query_stream=rank))
        import hashlib
        h_index = hashlib.sha256(wr["X"].tobytes() + wr["centroids"].tobytes()
                                 + wr["assign"].tobytes()).digest()[:8]
        h_q = hashlib.sha256(wr["qids"].tobytes()).digest()[:8]
        t = torch.tensor([int.from_bytes(h_index, "little", signed=True),
                          int.from_bytes(h_q, "little", signed=True)], dtype=torch.int64)
        got = [torch.empty_like(t) for _ in range(world)]
        dist.all_gather(got, t)
        assert all(int(g[0]) == int(got[0][0]) for g in got), "index differs across ranks"
        assert len({int(g[1]) for g in got}) == world, "ranks share a query batch"
        open(os.path.join(out_dir, f"ok{rank}"), "w").write("ok")
    finally:
        dist.destroy_process_group()


def test_query_shard_partition():
    from paper_2608_03199_gb300.shard import query_shard
    for nq in (0, 1, 5, 203, 1000):
        for world in (1, 2, 3, 8):
            spans = [query_shard(nq, world, r) for r in range(world)]
            assert spans[0][0] == 0 and spans[-1][1] == nq
            for (a, b), (c, _) in zip(spans, spans[1:]):
                assert b == c
            sizes = [b - a for a, b in spans]
            assert max(sizes) - min(sizes) <= 1 and sizes == sorted(sizes, reverse=True)
    with pytest.raises(ValueError):
        query_shard(10, 2, 2)


def test_single_process_gather_is_identity():
    from paper_2608_03199_gb300 import shard
    ids = torch.arange(12).reshape(4, 3)
    sc = torch.rand(4, 3)
    cnt = torch.tensor([3, 2, 0, 1], dtype=torch.int32)
    pr = torch.tensor([4, 5, 6, 7], dtype=torch.int32)
    out = shard.gather_results(ids, sc, cnt, pr, 4)
    for a, b in zip(out, (ids, sc, cnt, pr)):
        assert torch.equal(a, b)


def test_gloo_world2_shard_gather(tmp_path):
    import oracle
    oracle.build()
    import torch.multiprocessing as mp
    mp.spawn(_worker, args=(2, _free_port(), str(tmp_path)), nprocs=2, join=True)
    assert (tmp_path / "ok0").exists() and (tmp_path / "ok1").exists()
