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
    cfg = types.SimpleNamespace(nprobe=64, tau=0.9, d=96)
    auto = types.SimpleNamespace(scan_path="auto")
    assert not bench.uses_screen(auto, cfg, 8, True)
    assert bench.uses_screen(auto, cfg, 16, True)
    assert bench.uses_screen(auto, cfg, 64, True)
    assert not bench.uses_screen(auto, cfg, 64, False)          # no tensor layout
    assert bench.uses_screen(types.SimpleNamespace(scan_path="screen"), cfg, 8, True)
    assert not bench.uses_screen(types.SimpleNamespace(scan_path="tensor"), cfg, 64, True)
    assert not bench.uses_screen(auto, types.SimpleNamespace(nprobe=12, tau=0.9, d=96), 64, True)
    assert not bench.uses_screen(auto, cfg, 64, True, tau=0.5)       # loose threshold
    wide = types.SimpleNamespace(nprobe=64, tau=0.9, d=256)         # d >= 192: at any window
    assert bench.uses_screen(auto, wide, 8, True)
    assert bench.uses_screen(auto, wide, 2, True)
    assert not bench.uses_screen(auto, wide, 8, True, tau=0.5)


def test_cpu_baseline_times_both_modes():
    """The oracle's CPU timing (the bench's cpu_baseline leg) on the tiny
    workload: the W = 8-style window and fixed probing, each on a bounded
    sample, with the thread count reported."""
    wl = synth.make_workload("tiny", device="cpu")
    cfg = wl["cfg"]
    out, parity = bench.cpu_baseline(bench.host_arrays(wl), cfg, 0.5)
    assert out["kind"] == "oracle" and out["cores"] >= 1 and out["value"] > 0
    assert out["fixed_probe"]["value"] > 0
    assert f"W={cfg.nprobe}" in out["fixed_probe"]["sample"]
    assert isinstance(out["cpu_model"], str) and out["cpu_model"]
    assert parity == {}


def test_parity_sample_counts_divergences():
    """The bench's parity record: the oracle's own results compare as all
    exact; a planted wrong id and a wrong probe count on two queries are
    counted as unexplained (their decisions sit far from any flip)."""
    wl = synth.make_workload("tiny", device="cpu")
    cfg = wl["cfg"]
    w = bench.host_arrays(wl)
    idx = {k: w[k] for k in ("X", "ids", "assign", "centroids")}
    ref = oracle.search(idx, w["Q"], cfg.tau, cfg.k, cfg.nprobe, cfg.W, qids=w["qids"])
    got = [ref["ids"].copy(), ref["scores"].astype(np.float32), ref["count"].copy(),
           ref["probes"].copy()]
    rep = bench.parity_sample(oracle, idx, w["Q"], w["qids"], cfg, cfg.W, ref, tuple(got))
    assert rep["queries"] == len(w["Q"]) and rep["exact"] == rep["queries"]
    assert rep["allowed"] == 0 and rep["unexplained"] == 0 and rep["max_score_err"] < 1e-7
    # two planted mistakes: a query's probe count off by one, another's first id
    tg, kg, cg = oracle.fragility(idx, w["Q"], cfg.tau, cfg.k, cfg.nprobe,
                                  oracle.rank(w["Q"], w["centroids"], cfg.nprobe),
                                  ref["probes"] + 1, qids=w["qids"])
    far = np.flatnonzero((tg > 1e-3) & (kg > 1e-3) & (cg > 1e-3) & (ref["count"] > 0))
    a, b = far[0], far[1]
    got[3][a] += 1
    got[0][b, 0] = 10**9
    rep = bench.parity_sample(oracle, idx, w["Q"], w["qids"], cfg, cfg.W, ref, tuple(got))
    assert rep["exact"] == rep["queries"] - 2 and rep["unexplained"] == 2
