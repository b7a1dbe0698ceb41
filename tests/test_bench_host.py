"""Host-side logic of bench.py that runs without a GPU: the pooled filtered
top-k recall against exhaustive search (the paper's quality measure, Sec. 6.1)
checked against the oracle's brute force, and the rule that says which scan
the automatic path takes."""
import types

import numpy as np
import torch

import bench
import oracle
import synth


def test_bruteforce_recall_against_the_oracle():
    wl = synth.make_workload("tiny", device="cpu")
    cfg = wl["cfg"]
    w = synth.to_numpy(wl)
    bf = oracle.bruteforce(w["X"], w["ids"], w["Q"], cfg.tau, cfg.k, qids=w["qids"])
    ids = torch.from_numpy(bf["ids"])
    cnt = torch.from_numpy(bf["count"]).to(torch.int32)
    one = torch.clamp(cnt, max=1)
    none = torch.zeros_like(cnt)
    r = bench.bruteforce_recall(wl["X"], wl["ids"], wl["Q"], wl["qids"], cfg.tau, cfg.k,
                                {"exact": (ids, cnt), "first": (ids, one), "empty": (ids, none)},
                                sample=1000)
    assert r["sample_queries"] == 1000
    assert r["exact_neighbours"] == int(bf["count"].sum())
    assert r["exact"] == 1.0
    assert abs(r["first"] - int(np.minimum(bf["count"], 1).sum()) / int(bf["count"].sum())) < 1e-12
    assert r["empty"] == 0.0


def test_automatic_scan_rule():
    cfg = types.SimpleNamespace(nprobe=64)
    auto = types.SimpleNamespace(scan_path="auto")
    assert not bench.uses_screen(auto, cfg, 8, True)
    assert bench.uses_screen(auto, cfg, 16, True)
    assert bench.uses_screen(auto, cfg, 64, True)
    assert not bench.uses_screen(auto, cfg, 64, False)          # no tensor layout
    assert bench.uses_screen(types.SimpleNamespace(scan_path="screen"), cfg, 8, True)
    assert not bench.uses_screen(types.SimpleNamespace(scan_path="tensor"), cfg, 64, True)
    assert not bench.uses_screen(auto, types.SimpleNamespace(nprobe=12), 64, True)


def test_cpu_baseline_times_both_modes():
    """The oracle's CPU timing (the bench's cpu_baseline leg) on the tiny
    workload: the W = 8-style window and fixed probing, each on a bounded
    sample, with the thread count reported."""
    wl = synth.make_workload("tiny", device="cpu")
    cfg = wl["cfg"]
    out = bench.cpu_baseline(bench.host_arrays(wl), cfg, 0.5)
    assert out["kind"] == "oracle" and out["cores"] >= 1 and out["value"] > 0
    assert out["fixed_probe"]["value"] > 0
    assert f"W={cfg.nprobe}" in out["fixed_probe"]["sample"]
