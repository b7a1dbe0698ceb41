#!/usr/bin/env python
"""Throughput of the threshold-aware IVF search on GB300 (one JSON line).

A step is one ``sieve_search`` call over one batch of queries: centroid
ranking, then device-resident rounds of issue / bucketing / grouped scan with
the fused tau, top-k and stop-line epilogue / merge until every query has
stopped.  The default workload is the largest single-GPU configuration, the
100M x 96 corpus (65,536 partitions, 1M database-drawn queries, tau 0.90,
k 10, nprobe 256, W 8 against fixed probing, lookahead on), synthetic and
seeded (``synth``), with the index resident in HBM; ``--config`` picks
another (tiny, 1m, 10m512, 10m256, 100m) and ``--all-configs`` runs every
configuration in its own process and prints one line per configuration plus
a summary line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl sieve|reference]

With N > 1 (torchrun) each rank searches its own query batch against its own
replica of the index (queries shard with no data-path exchange: weak scaling);
the step time is the maximum over ranks.  ``--impl reference`` times the fp64
CPU oracle on the host cores instead (rank 0 only).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402
from paper_2608_03199_gb300 import shard  # noqa: E402

METRIC = ("queries/s at W=8 (tau-filtered top-10) + speedup vs fixed-probe; "
          "% HBM/tensor roofline")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("sieve", "reference"), default="sieve")
    ap.add_argument("--config", default="100m")
    ap.add_argument("--all-configs", action="store_true",
                    help="every configuration, each in its own process (a line per "
                         "configuration, then a summary line with a per_config dict)")
    ap.add_argument("--skip-cpu-baseline", action="store_true")
    ap.add_argument("--skip-e2e", action="store_true")
    ap.add_argument("--sweep", action="store_true",
                    help="operating-envelope sweeps (W, lookahead, tau, k, nprobe, batch): one "
                         "JSON line per setting instead of the benchmark line")
    ap.add_argument("--shards", type=int, default=0,
                    help="sharded layout: split the corpus into this many coarse shards, each "
                         "with its own IVF index (one JSON line instead of the benchmark line)")
    ap.add_argument("--nlist-per-shard", type=int, default=1500)
    ap.add_argument("--nprobe", type=int, default=0, help="nprobe per shard (0: the workload's)")
    ap.add_argument("--skip-calibration", action="store_true",
                    help="skip the in-call window calibration measurement")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="target CPU seconds for the oracle sample")
    ap.add_argument("--scan-path", choices=("auto", "simt", "tensor", "screen"), default="auto",
                    help="which units score the partition groups (sieve_params.scan_path: "
                         "tensor = three fp16 products per pair, screen = one product per pair "
                         "and an fp32 rescore of the candidates, auto = the screen from "
                         "tau 0.85 up, at a window of 16 or d >= 192)")
    ap.add_argument("--rq", action="store_true",
                    help="the quantized local search (RaBitQ-style 7-bit codes) on the workload")
    ap.add_argument("--ncu-case", choices=("w8", "fixed", "rqw8", "rank"), default=None,
                    help="run exactly one search (W = the config's W, or fixed probe) and exit: "
                         "a small, single-call target for an ncu capture; 'rank': one centroid "
                         "ranking of --ncu-queries queries against seeded centroids of the "
                         "config's nlist x d (under 1 GB on the device)")
    ap.add_argument("--ncu-queries", type=int, default=20_000)
    return ap.parse_args()


def workload_desc(cfg):
    return (f"{cfg.name}: {cfg.n:,} x {cfg.d} fp32 unit-norm rows, {cfg.ncomp} components"
            f"{'' if cfg.zipf is None else f' Zipf({cfg.zipf})'}, planted near-duplicates, "
            f"nlist {cfg.nlist}, {cfg.nq:,} database-drawn queries, tau {cfg.tau}, k {cfg.k}, "
            f"nprobe {cfg.nprobe}, W {cfg.W}, lookahead on")


# ---------------------------------------------------------------------------
class ClockSampler:
    """nvidia-smi samples (every 200 ms) while the GPU is busy."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,utilization.gpu,"
              "clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 10:
                continue
            try:
                rows.append({"sm": float(parts[1]), "max": float(parts[2]), "util": float(parts[4]),
                             "hw": parts[6], "hwt": parts[7], "swt": parts[8], "pcap": parts[9]})
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        busy = [r for r in rows if r["util"] >= 50] or rows
        reasons = set()
        for r in busy:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("pcap", "sw_power_cap")):
                if r[key].lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r["sm"] for r in busy),
                "sm_max_mhz": max(r["max"] for r in busy), "reasons": sorted(reasons),
                "samples": len(busy)}


# ---------------------------------------------------------------------------
def measured_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return {}


# the sources that define each profiled kernel and the layout it streams
_SCAN_SOURCES = ("common.cuh", "search.cuh", "scan_tc.cu", "tcgen05.cuh", "tc_bulk.cuh",
                 "tc_pipeline.cuh", "tc_layout.cu", "rq.cu")
_RANK_SOURCES = ("common.cuh", "search.cuh", "rank_tc.cu", "tcgen05.cuh", "tc_bulk.cuh",
                 "tc_pipeline.cuh", "tc_layout.cu")
KERNEL_SOURCES = {"k_scan_bulk": _SCAN_SOURCES, "k_scan_rq": _SCAN_SOURCES,
                  "k_scan_screen": _SCAN_SOURCES, "k_rank_bulk + k_rank_screen": _RANK_SOURCES}


def kernel_source_sha(kernel):
    """Hash of the files that define one kernel (not the host API)."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_03199_gb300", "csrc")
    for f in KERNEL_SOURCES.get(kernel, ()):
        p = os.path.join(csrc, f)
        if os.path.exists(p):
            h.update(open(p, "rb").read())
    return h.hexdigest()[:16]


def committed_traffic(kernel, workload, launches):
    """DRAM bytes per launch from the committed ncu summary, if the kernel
    sources are unchanged since it was taken: the capture's bytes over all of
    one search's launches, averaged over this step's launch count (the same
    averaging as the achieved rate; launches past the last busy round move
    no bytes)."""
    try:
        t = json.load(open(os.path.join(ROOT, "profiles", "traffic.json")))
    except Exception:
        return None
    e = t.get(kernel, {}).get(workload)
    if not e or e.get("source_sha") != kernel_source_sha(kernel) or "dram_bytes_per_search" not in e:
        return None
    return e["dram_bytes_per_search"] / max(1, launches)


def uses_screen(args, cfg, W, bulk, tau=None):
    """Whether the bulk scan screens (sieve_params.scan_path; the automatic
    path screens when tau >= 0.85, from a window of 16 up or at d >= 192)."""
    tau = cfg.tau if tau is None else tau
    return bulk and (args.scan_path == "screen" or
                     (args.scan_path == "auto" and (min(W, cfg.nprobe) >= 16 or cfg.d >= 192) and tau >= 0.85))


def rank_passes(cfg, bulk):
    """(contraction passes of the tensor-core ranking, products per score of
    the first pass): with the tensor-core layout (d <= 256), more than 2,048
    centroids and 2 nprobe to 2,048 groups of 64 (or 32), a first pass of
    group maxima on the screen (one product per score); else one pass."""
    if cfg.nlist <= 2048 or not bulk or cfg.d > 256:
        return 1, 0
    for g in (64, 32):
        ng = -(-cfg.nlist // g)
        if 2 * cfg.nprobe <= ng <= 2048:
            return 2, 1
    return 1, 0


def roofline(prof, cfg, dev, bulk=True, rank_on_tensor=True, rq=False, screen=False):
    """Roofline entry for the kernel with the largest share of the step.
    bulk: the index carries the tensor-core layout, so the tensor-core scan
    runs as k_scan_bulk (else k_scan_tc) and the ranking as k_rank_bulk;
    screen: the bulk scan screens with one product per pair (k_scan_screen);
    rank_on_tensor: the ranking runs on the tensor cores (every scan path
    but the FP32 one)."""
    km, kl = dict(prof["kernel_ms"]), dict(prof["kernel_launches"])
    # the ranking's contraction is timed on its own ("rank_mma", a part of
    # "rank"); the rest of "rank" is its selection
    if km.get("rank_mma", 0) > 0:
        km["rank_select"] = km["rank"] - km["rank_mma"]
        kl["rank_select"] = kl["rank"] - kl["rank_mma"]
        del km["rank"], kl["rank"]
    top = max(km, key=lambda k: km[k])
    props = torch.cuda.get_device_properties(dev)
    peaks = measured_peaks()
    clock_mhz = peaks.get("sm_max_mhz", 2070.0)
    fp32_tflops = props.multi_processor_count * 128 * 2 * clock_mhz * 1e6 / 1e12
    hbm = peaks.get("hbm_gbs", 6800.0)
    d = cfg.d
    launches = max(1, kl[top])
    ms_per_launch = km[top] / launches
    name = {"scan_tc": "k_scan_rq" if rq else ("k_scan_screen" if screen else "k_scan_bulk") if bulk
            else "k_scan_tc"}.get(top, f"k_{top}")
    out = {"kernel": name, "launches": kl[top], "ms_per_launch": ms_per_launch}
    # fp16 dense peak: the measured bf16 cuBLAS peak (fp16 and bf16 share the
    # nominal 2.25 PFLOP/s rate); the burst figure, as the kernel is timed alone
    f16_tflops = peaks.get("bf16_tflops", 1889.4)
    if top == "scan_tc" and rq:
        flops = 2.0 * d * prof["pairs_tc"]
        ach = flops / launches / (ms_per_launch * 1e-3) / 1e12
        out.update(bound="tensor", achieved=ach, peak=f16_tflops / 2, unit="TFLOP/s",
                   frac=ach / (f16_tflops / 2),
                   peak_source=(f"codes exact in fp16, queries split: two kind::f16 MMAs per "
                                f"estimate; fp16 dense peak {f16_tflops:.0f} TFLOP/s = measured "
                                f"bf16 cuBLAS burst (of measured), so the algorithmic peak is half"),
                   tensor_pipe_tflops=2 * ach)
    elif top == "scan_tc" and screen and bulk:
        flops = 2.0 * d * prof["pairs_tc"]
        ach = flops / launches / (ms_per_launch * 1e-3) / 1e12
        out.update(bound="tensor", achieved=ach, peak=f16_tflops, unit="TFLOP/s",
                   frac=ach / f16_tflops,
                   peak_source=(f"screen: one kind::f16 MMA per product (hi halves), the rare "
                                f"candidates rescored in FP32; fp16 dense peak {f16_tflops:.0f} "
                                f"TFLOP/s = measured bf16 cuBLAS burst (of measured)"),
                   tensor_pipe_tflops=ach,
                   l2_stream_gbs=2.0 * d * prof["rows_read_tc"] / launches
                   / (ms_per_launch * 1e-3) / 1e9)
    elif top == "scan_tc":
        flops = 2.0 * d * prof["pairs_tc"]
        ach = flops / launches / (ms_per_launch * 1e-3) / 1e12
        out.update(bound="tensor", achieved=ach, peak=f16_tflops / 3, unit="TFLOP/s",
                   frac=ach / (f16_tflops / 3),
                   peak_source=(f"fp16 split: three kind::f16 MMAs per product; fp16 dense peak "
                                f"{f16_tflops:.0f} TFLOP/s = measured bf16 cuBLAS burst (of measured), "
                                f"so the algorithmic peak is a third of it"),
                   tensor_pipe_tflops=3 * ach)
    elif top == "scan":
        flops = 2.0 * d * (prof["pairs"] - prof["pairs_tc"])
        ach = flops / launches / (ms_per_launch * 1e-3) / 1e12
        bytes_ = 4.0 * d * (prof["rows_read"] - prof["rows_read_tc"] + prof["items"])
        out.update(bound="alu", achieved=ach, peak=fp32_tflops, unit="TFLOP/s",
                   frac=ach / fp32_tflops,
                   peak_source=f"FP32 FMA: {props.multi_processor_count} SMs x 128 lanes x 2 "
                               f"x {clock_mhz:.0f} MHz (measured max clock)",
                   hbm_view={"achieved_gbs": bytes_ / launches / (ms_per_launch * 1e-3) / 1e9,
                             "peak_gbs": hbm})
    elif top == "rank_mma":
        # the score contraction of the ranking (tensor cores, three fp16
        # products per score in the pass that keeps candidates); its
        # algorithmic work is every query-centroid score once, spread over
        # all its launches: with many centroids a first pass of group maxima
        # (one product per score, on the screen, with the tensor-core layout)
        # sets each query's starting threshold
        passes, first_products = rank_passes(cfg, bulk)
        name = "k_rank_bulk" + (" + k_rank_screen" if passes == 2 and bulk else "") if bulk \
            else "k_rank_tc"
        flops = 2.0 * cfg.nq * cfg.nlist * d
        ach = flops / launches / (ms_per_launch * 1e-3) / 1e12
        # K steps of 16 issued (the zero padding of the last K-block is skipped)
        d_mma = 16 * -(-d // 16)
        out.update(kernel=name, bound="tensor", achieved=ach, peak=f16_tflops / 3,
                   unit="TFLOP/s", frac=ach / (f16_tflops / 3),
                   peak_source=(f"fp16 split: three kind::f16 MMAs per score; fp16 dense peak "
                                f"{f16_tflops:.0f} TFLOP/s = measured bf16 cuBLAS burst (of "
                                f"measured), a third of it; achieved = every score once over "
                                f"the summed time of all contraction launches"),
                   passes=passes,
                   tensor_pipe_tflops=(3 + first_products) * ach * d_mma / d,
                   rank_select_ms=km.get("rank_select"))
    elif top == "rank_select":
        out.update(kernel="ranking selection (k_select / k_compact_final)", bound="alu",
                   achieved=None, peak=None, unit=None, frac=None)
    elif top == "rank" and rank_on_tensor:
        name = "k_rank_bulk" if bulk else "k_rank_tc"
        flops = 2.0 * cfg.nq * cfg.nlist * d
        ach = flops / (km[top] * 1e-3) / 1e12
        out.update(kernel=name + " + selection", bound="tensor", achieved=ach, peak=f16_tflops / 3,
                   unit="TFLOP/s", frac=ach / (f16_tflops / 3),
                   peak_source=(f"fp16 split: three kind::f16 MMAs per score; fp16 dense peak "
                                f"{f16_tflops:.0f} TFLOP/s = measured bf16 cuBLAS burst (of "
                                f"measured), a third of it; the time is every launch of the "
                                f"ranking, selection included"),
                   tensor_pipe_tflops=3 * ach)
    elif top == "rank":
        flops = 2.0 * cfg.nq * cfg.nlist * d
        ach = flops / (km[top] * 1e-3) / 1e12
        out.update(bound="alu", achieved=ach, peak=fp32_tflops, unit="TFLOP/s",
                   frac=ach / fp32_tflops,
                   peak_source=f"FP32 FMA: {props.multi_processor_count} SMs x 128 lanes x 2 "
                               f"x {clock_mhz:.0f} MHz (measured max clock)")
    else:
        out.update(bound="hbm", achieved=None, peak=hbm, unit="GB/s", frac=None)
    out["traffic"] = committed_traffic(out["kernel"], cfg.name, kl[top])
    return out


# ---------------------------------------------------------------------------
def dist_setup(gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def barrier(world):
    if world > 1:
        shard.barrier()


def max_over_ranks(x, world, dev):
    return shard.max_over_ranks(x, device=dev) if world > 1 else x


def time_steps(fn, steps, warmup, world, dev):
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    barrier(world)
    st = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(steps):
        fn()
    e1.record(st)
    torch.cuda.synchronize()
    barrier(world)
    ms = e0.elapsed_time(e1) / steps
    return max_over_ranks(ms, world, dev)


def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo), for the record."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.processor() or platform.machine()


PARITY_TOL = 1e-5   # scores; and how close to a rounding flip a divergence may sit


def parity_sample(oracle, idx, Q, qids, cfg, W, ref, got):
    """GPU results of the first queries against the oracle's on the same
    queries: ids, counts and probes identical, or the query differs where
    the oracle's fragility tags put a decision within 1e-5 of a flip (a
    similarity that close to tau, a k-th / (k+1)-th gap or two centroid
    scores that close: allowed, counted); scores within 1e-5."""
    g_ids, g_sc, g_cnt, g_pr = got
    same = ((g_pr == ref["probes"]) & (g_cnt == ref["count"]) & (g_ids == ref["ids"]).all(axis=1))
    bad = np.flatnonzero(~same)
    allowed = np.zeros(len(same), bool)
    if len(bad):
        order = oracle.rank(Q[bad], idx["centroids"], cfg.nprobe)
        upto = np.maximum(g_pr[bad], ref["probes"][bad]).astype(np.int32)
        tg, kg, cg = oracle.fragility(idx, Q[bad], cfg.tau, cfg.k, cfg.nprobe, order, upto,
                                      qids=qids[bad])
        allowed[bad] = (tg < PARITY_TOL) | (kg < PARITY_TOL) | (cg < PARITY_TOL)
    valid = np.arange(cfg.k)[None, :] < ref["count"][:, None]
    with np.errstate(invalid="ignore"):
        err = np.where(valid & same[:, None], np.abs(g_sc.astype(np.float64) - ref["scores"]), 0.0)
    return {"queries": int(len(same)), "W": W, "exact": int(same.sum()),
            "allowed": int(allowed.sum()), "unexplained": int((~same & ~allowed).sum()),
            "max_score_err": float(err.max()) if err.size else 0.0}


def cpu_baseline(w, cfg, target_s, gpu_w=None, gpu_fixed=None):
    """The oracle (fp64, OpenMP over queries) on a bounded query sample, timed
    at the workload's W and at fixed probing.  gpu_w / gpu_fixed (host numpy
    (ids, scores, count, probes) of every query, nullable): the GPU's results
    of the same calls, compared with the oracle's on the timed samples."""
    import oracle
    idx = {k: w[k] for k in ("X", "ids", "assign", "centroids")}
    threads = oracle.default_threads()

    def sized(W, budget, least):
        """Queries that fill the budget: two probe calls separate a call's
        fixed cost (the oracle builds its partition lists from the rows) from
        the cost per query."""
        lo = min(cfg.nq, 64)
        hi = min(cfg.nq, 4 * lo)
        ts = []
        for m in (lo, hi):
            t0 = time.perf_counter()
            oracle.search(idx, w["Q"][:m], cfg.tau, cfg.k, cfg.nprobe, W, qids=w["qids"][:m],
                          threads=threads)
            ts.append(time.perf_counter() - t0)
        per_q = max((ts[1] - ts[0]) / max(1, hi - lo), ts[1] / hi * 0.05, 1e-9)
        fixed = max(0.0, ts[0] - lo * per_q)
        return int(min(cfg.nq, max(least, (budget - fixed) / per_q)))

    # at the workload's window: at least 10,000 queries (the whole batch when smaller)
    sample = sized(cfg.W, target_s, min(cfg.nq, 10_000))
    t0 = time.perf_counter()
    ref = oracle.search(idx, w["Q"][:sample], cfg.tau, cfg.k, cfg.nprobe, cfg.W,
                        qids=w["qids"][:sample], threads=threads)
    dt = time.perf_counter() - t0
    # fixed probing (W = nprobe) on a smaller sample: a third of the time budget
    fsample = sized(cfg.nprobe, target_s / 3, min(cfg.nq, 64))
    t0 = time.perf_counter()
    fref = oracle.search(idx, w["Q"][:fsample], cfg.tau, cfg.k, cfg.nprobe, cfg.nprobe,
                         qids=w["qids"][:fsample], threads=threads)
    fdt = time.perf_counter() - t0
    out = {"value": sample / dt, "unit": "queries/s", "cores": threads, "kind": "oracle",
           "cpu_model": cpu_model(),
           "sample": f"first {sample:,} of the {cfg.nq:,} queries, W={cfg.W}, "
                     f"{dt:.1f} s on {threads} host threads",
           "fixed_probe": {"value": fsample / fdt, "unit": "queries/s",
                           "sample": f"first {fsample:,} queries, W={cfg.nprobe}, {fdt:.1f} s"}}
    parity = {}
    if gpu_w is not None:
        parity[f"W{cfg.W}"] = parity_sample(oracle, idx, w["Q"][:sample], w["qids"][:sample], cfg,
                                            cfg.W, ref, tuple(a[:sample] for a in gpu_w))
    if gpu_fixed is not None:
        parity["fixed_probe"] = parity_sample(oracle, idx, w["Q"][:fsample], w["qids"][:fsample],
                                              cfg, cfg.nprobe, fref,
                                              tuple(a[:fsample] for a in gpu_fixed))
    return out, parity


def bruteforce_recall(X, ids, Q, qids, tau, k, results, sample=1000, seed=777):
    """Pooled filtered top-k recall against exhaustive search, the paper's
    quality measure (Sec. 6.1): on a seeded sample of the queries, the number
    of exact filtered top-k neighbours (score >= tau, the query's own row
    excluded) that a result set holds, over the number of exact neighbours.
    The exact sets come from fp32 inner products of each sampled query with
    every row (a plain matmul: it evaluates the outputs, it is not the
    search).  results: {name: (ids [nq][k] i64, count [nq] i32)} on the
    device."""
    nq = Q.shape[0]
    g = torch.Generator(device="cpu").manual_seed(seed)
    pick = torch.sort(torch.randperm(nq, generator=g)[:min(sample, nq)]).values.to(Q.device)
    chunk = max(1, int(2 ** 28 // max(1, X.shape[0])))       # <= 1 GiB of scores at a time
    tf32 = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    hits = {name: 0 for name in results}
    total = 0
    try:
        for lo in range(0, pick.numel(), chunk):
            p = pick[lo:lo + chunk]
            S = Q[p] @ X.T
            S[ids[None, :] == qids[p][:, None]] = float("-inf")
            S[S < tau] = float("-inf")
            val, pos = torch.topk(S, k, dim=1)
            valid = val > float("-inf")
            gt = torch.where(valid, ids[pos], torch.full_like(pos, -2))
            total += int(valid.sum().item())
            for name, (r_ids, r_cnt) in results.items():
                r = r_ids[p]
                r = torch.where(torch.arange(k, device=r.device)[None, :] < r_cnt[p][:, None].long(),
                                r, torch.full_like(r, -3))
                hits[name] += int((r[:, :, None] == gt[:, None, :]).any(-1).sum().item())
            del S
    finally:
        torch.backends.cuda.matmul.allow_tf32 = tf32
    out = {name: (h / total if total else 1.0) for name, h in hits.items()}
    out.update(sample_queries=int(pick.numel()), exact_neighbours=total,
               ground_truth="fp32 inner products with every row, score >= tau, own row excluded")
    return out


def host_arrays(wl):
    return {k: wl[k].detach().cpu().numpy() for k in ("X", "ids", "assign", "centroids", "Q", "qids")}


# ---------------------------------------------------------------------------
def run_reference(args, cfg, world, rank):
    if rank != 0:
        return 0
    import oracle
    dev = torch.device("cuda:0") if torch.cuda.is_available() else torch.device("cpu")
    wl = synth.make_workload(cfg, device=dev)
    w = host_arrays(wl)
    del wl
    idx = {k: w[k] for k in ("X", "ids", "assign", "centroids")}
    threads = oracle.default_threads()
    probe = min(cfg.nq, 64)
    t0 = time.perf_counter()
    oracle.search(idx, w["Q"][:probe], cfg.tau, cfg.k, cfg.nprobe, cfg.W, qids=w["qids"][:probe],
                  threads=threads)
    per_q = (time.perf_counter() - t0) / probe
    budget = 150.0 / max(1, args.steps + args.warmup)       # whole run within a few minutes
    sample = int(min(cfg.nq, max(16, budget / max(per_q, 1e-9))))
    times = []
    for i in range(args.warmup + args.steps):
        lo = (i * sample) % max(1, cfg.nq - sample + 1)
        t0 = time.perf_counter()
        oracle.search(idx, w["Q"][lo:lo + sample], cfg.tau, cfg.k, cfg.nprobe, cfg.W,
                      qids=w["qids"][lo:lo + sample], threads=threads)
        if i >= args.warmup:
            times.append(time.perf_counter() - t0)
    step_s = sum(times) / len(times)
    value = sample / step_s
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "queries/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": step_s * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_desc(cfg), "queries_per_step": sample},
        "cpu_baseline": {"value": value, "unit": "queries/s", "cores": threads, "kind": "oracle",
                         "sample": f"{sample:,} queries per step of the {cfg.nq:,}-query batch"},
        "e2e": {"value": value, "unit": "queries/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def run_sieve(args, cfg, world, rank, local):
    import paper_2608_03199_gb300 as sieve

    assert torch.cuda.is_available(), "bench.py needs a CUDA device"
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        torch.distributed.init_process_group("nccl", device_id=dev)
    sieve.lib()
    wl = synth.make_workload(cfg, device=dev, query_stream=rank)
    index = sieve.build_layout(wl["X"], wl["assign"], cfg.nlist, wl["centroids"])
    Q, qids = wl["Q"], wl["qids"]
    torch.cuda.synchronize()

    ws = sieve.Workspace()
    nq, k = cfg.nq, cfg.k
    outs = (torch.empty((nq, k), dtype=torch.int64, device=dev),
            torch.empty((nq, k), dtype=torch.float32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev))

    def step(W):
        return lambda: sieve.search(index, Q, cfg.tau, k, cfg.nprobe, W, lookahead=True,
                                    query_ids=qids, workspace=ws, out=outs,
                                    scan_path=args.scan_path)

    clocks = ClockSampler(local)
    clocks.start()
    ms = time_steps(step(cfg.W), args.steps, args.warmup, world, dev)
    clock_rec = clocks.stop()
    ms_fixed = time_steps(step(cfg.nprobe), max(3, args.steps // 5), 2, world, dev)

    # one profiled step (host-driven rounds, CUDA events around every launch)
    prof = sieve.search(index, Q, cfg.tau, k, cfg.nprobe, cfg.W, lookahead=True, query_ids=qids,
                        profile=True, workspace=ws, scan_path=args.scan_path)[4]
    probes = outs[3]
    sieve.search(index, Q, cfg.tau, k, cfg.nprobe, cfg.W, lookahead=True, query_ids=qids,
                 workspace=ws, out=outs, scan_path=args.scan_path)
    mean_probes = float(probes.float().mean().item())
    hit_frac = float((outs[2] > 0).float().mean().item())
    # quality context: pooled filtered top-k recall of W = 8 and of fixed
    # probing against exhaustive search on a query sample
    fixed = sieve.search(index, Q, cfg.tau, k, cfg.nprobe, cfg.nprobe, lookahead=True,
                         query_ids=qids, workspace=ws, scan_path=args.scan_path)
    recall_bf = bruteforce_recall(wl["X"], wl["ids"], Q, qids, cfg.tau, k,
                                  {f"W{cfg.W}": (outs[0], outs[2]), "fixed_probe": (fixed[0], fixed[2])})
    # host copies of both result sets, for the oracle comparison of the
    # cpu_baseline leg (the first queries are the oracle's sample)
    keep = min(nq, 200_000)
    gpu_w = tuple(t[:keep].cpu().numpy() for t in outs)
    gpu_fixed = tuple(t[:keep].cpu().numpy() for t in fixed)
    del fixed

    # in-call window calibration (Appendix A): a 2% sample fully probed, a 0.5%
    # sample-relative loss target, the rest under the selected window
    calib = None
    if not args.skip_calibration:
        g = torch.Generator(device="cpu").manual_seed(12345 + rank)
        ns = max(1, (cfg.nq * 2 + 99) // 100)
        sample = torch.sort(torch.randperm(cfg.nq, generator=g)[:ns]).values.to(dev)
        cws = sieve.Workspace()

        def cstep():
            return sieve.calibrated_search(index, Q, cfg.tau, k, cfg.nprobe, sample, 0.005,
                                           query_ids=qids, workspace=cws,
                                           scan_path=args.scan_path)
        info = cstep()[4]
        csteps = max(3, args.steps // 20)
        torch.cuda.synchronize()
        barrier(world)
        t0 = time.perf_counter()
        for _ in range(csteps):
            cstep()
        torch.cuda.synchronize()
        barrier(world)
        c_ms = max_over_ranks((time.perf_counter() - t0) / csteps * 1e3, world, dev)
        calib = {"value": nq * world / (c_ms * 1e-3), "unit": "queries/s", "ms_per_step": c_ms,
                 "W": info["W"], "sample": ns, "loss_target": 0.005,
                 "sample_neighbours": info["Z"],
                 "speedup_vs_fixed": ms_fixed / c_ms,
                 "timing": "host clock around whole calls (each reads W back once)"}

    # end to end through the C ABI with host buffers
    e2e = None
    if not args.skip_e2e:
        Qh = Q.cpu().pin_memory()
        qh = qids.cpu().pin_memory()
        houts = (torch.empty((nq, k), dtype=torch.int64, pin_memory=True),
                 torch.empty((nq, k), dtype=torch.float32, pin_memory=True),
                 torch.empty(nq, dtype=torch.int32, pin_memory=True),
                 torch.empty(nq, dtype=torch.int32, pin_memory=True))
        hws = sieve.Workspace()

        def hstep():
            sieve.search_host(index, Qh, cfg.tau, k, cfg.nprobe, cfg.W, lookahead=True,
                              query_ids_host=qh, workspace=hws, out=houts,
                              scan_path=args.scan_path)
        hsteps = max(3, args.steps // 5)
        for _ in range(2):
            hstep()
        barrier(world)
        t0 = time.perf_counter()
        for _ in range(hsteps):
            hstep()
        torch.cuda.synchronize()
        barrier(world)
        e2e_ms = max_over_ranks((time.perf_counter() - t0) / hsteps * 1e3, world, dev)
        e2e = {"value": nq * world / (e2e_ms * 1e-3), "unit": "queries/s",
               "ms_per_step": e2e_ms, "h2d_bytes_per_step": nq * cfg.d * 4 + nq * 8,
               "d2h_bytes_per_step": nq * (k * 12 + 8)}

    line = {
        "metric": METRIC,
        "value": nq * world / (ms * 1e-3),
        "unit": "queries/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "arithmetic": "fp32 inputs; scores from three fp16 tensor-core products per pair "
                      "(scaled hi/lo split), fp32 accumulation",
        "data": "synthetic",
        "config": {"workload": workload_desc(cfg), "nq_per_gpu": nq, "parallelism": f"query-shard x{world}",
                   "scan_path": args.scan_path,
                   "l2": f"inputs larger than L2 (index {cfg.n * cfg.d * 4 / 1e9:.2f} GB "
                         f"streamed per step)"},
        "fixed_probe": {"value": nq * world / (ms_fixed * 1e-3), "ms_per_step": ms_fixed,
                        "W": cfg.nprobe,
                        "scan": "screen" if uses_screen(args, cfg, cfg.nprobe, index.tc_rows is not None)
                        else "three products"},
        "speedup_vs_fixed": ms_fixed / ms,
        "calibrated": calib,
        "mean_probes": mean_probes,
        "queries_with_results": hit_frac,
        "recall_vs_bruteforce": recall_bf,
        "roofline": roofline(prof, cfg, dev, bulk=index.tc_rows is not None,
                             rank_on_tensor=args.scan_path != "simt",
                             screen=uses_screen(args, cfg, cfg.W, index.tc_rows is not None)),
        "profile": {"kernel_ms": prof["kernel_ms"], "kernel_launches": prof["kernel_launches"],
                    "rounds": prof["rounds"], "items": prof["items"], "groups": prof["groups"],
                    "mean_group": prof["items"] / max(1, prof["groups"]),
                    "pairs": prof["pairs"], "rows_read": prof["rows_read"],
                    "pairs_tc": prof["pairs_tc"], "rows_read_tc": prof["rows_read_tc"]},
        "gpu_launches": args.steps * int(sum(v for k, v in prof["kernel_launches"].items()
                                             if k != "rank_mma")),
        "clocks": clock_rec,
        "e2e": e2e,
    }
    if rank == 0 and world == 1 and not args.skip_cpu_baseline:
        line["cpu_baseline"], line["parity"] = cpu_baseline(host_arrays(wl), cfg, args.cpu_seconds,
                                                            gpu_w, gpu_fixed)
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def run_sweep(args, cfg):
    """Operating-envelope sweeps on one workload (not the benchmark line): one
    JSON line per setting with the time per call, queries/s, mean probes and
    the pooled recall of the kept neighbours against fixed probing (the same
    index, tau, k and nprobe).  Varied one at a time from the workload's own
    setting: W under the three schedules of the execution ablation (serial
    traversal, continuous batching, continuous batching with lookahead), tau
    from 0.10 to 0.95, k, nprobe, and the batch size."""
    import paper_2608_03199_gb300 as sieve
    dev = torch.device("cuda:0")
    sieve.lib()
    wl = synth.make_workload(cfg, device=dev)
    index = sieve.build_layout(wl["X"], wl["assign"], cfg.nlist, wl["centroids"])
    Q, qids = wl["Q"], wl["qids"]
    ws = sieve.Workspace()

    def timed(nq, tau, k, nprobe, W, lookahead, serial=False):
        run = lambda: sieve.search(index, Q[:nq], tau, k, nprobe, W, lookahead=lookahead,
                                   query_ids=qids[:nq], workspace=ws, serial=serial)
        for _ in range(2):
            out = run()
        torch.cuda.synchronize()
        reps = max(3, min(50, int(2e5 // max(nq, 1))))
        if serial:
            reps = 3
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            out = run()
        e1.record()
        torch.cuda.synchronize()
        return out, e0.elapsed_time(e1) / reps

    def recall(out, ref):
        a_ids, a_cnt = out[0].cpu().numpy(), out[2].cpu().numpy()
        f_ids, f_cnt = ref[0].cpu().numpy(), ref[2].cpu().numpy()
        kept = sum(len(set(a_ids[i, :a_cnt[i]]) & set(f_ids[i, :f_cnt[i]])) for i in range(len(a_cnt)))
        tot = int(f_cnt.sum())
        return kept / tot if tot else 1.0

    settings = []
    # the execution ablation of Sec. 6.3: serial traversal (every (query, rank)
    # its own partition call), continuous batching (one rank per query per
    # round, regrouped by partition), and continuous batching with lookahead
    for W in (cfg.sweep_W or (2, 4, 8, 16, cfg.nprobe)):
        for la, ser in ((False, True), (False, False), (True, False)):
            settings.append(("W", cfg.nq, cfg.tau, cfg.k, cfg.nprobe, W, la, ser))
    # threshold selectivity (Sec. 6.4): loose thresholds make most probes hit
    for tau in (0.10, 0.30, 0.50, 0.70, 0.85, 0.90, 0.95):
        settings.append(("tau", cfg.nq, tau, cfg.k, cfg.nprobe, cfg.W, True))
    for k in (5, 10, 20, 50):
        settings.append(("k", cfg.nq, cfg.tau, k, cfg.nprobe, cfg.W, True))
    for nprobe in sorted({16, 32, cfg.nprobe, min(2 * cfg.nprobe, cfg.nlist)}):
        settings.append(("nprobe", cfg.nq, cfg.tau, cfg.k, nprobe, min(cfg.W, nprobe), True))
    for nq in sorted({1, 100, 1_000, 10_000, cfg.nq}):
        if nq <= cfg.nq:
            settings.append(("batch", nq, cfg.tau, cfg.k, cfg.nprobe, cfg.W, True))
    fixed_cache = {}
    for setting in settings:
        axis, nq, tau, k, nprobe, W, la = setting[:7]
        ser = setting[7] if len(setting) > 7 else False
        key = (nq, tau, k, nprobe)
        if key not in fixed_cache:
            fixed_cache[key] = timed(nq, tau, k, nprobe, nprobe, True)
        ref, ms_fixed = fixed_cache[key]
        out, ms = timed(nq, tau, k, nprobe, W, la, ser)
        schedule = ("serial traversal" if ser else
                    "continuous batching + lookahead" if la else "continuous batching")
        print(json.dumps({"sweep": axis, "nq": nq, "tau": tau, "k": k, "nprobe": nprobe, "W": W,
                          "lookahead": la, "schedule": schedule, "ms": round(ms, 4),
                          "queries_per_s": round(nq / (ms * 1e-3)),
                          "fixed_ms": round(ms_fixed, 4), "speedup_vs_fixed": round(ms_fixed / ms, 3),
                          "mean_probes": round(float(out[3].float().mean()), 3),
                          "recall_vs_fixed": round(recall(out, ref), 5)}), flush=True)
    return 0


def run_sharded(args, cfg):
    """The sharded layout of the paper's public-100M workloads (Sec. 6.1): the
    corpus split into --shards coarse shards, each with its own IVF index of
    --nlist-per-shard partitions, searched at nprobe per shard with its own
    stopping, then the global top-k.  One JSON line (not the benchmark line):
    W = the workload's W against fixed probing on every shard."""
    import gc
    import paper_2608_03199_gb300 as sieve
    dev = torch.device("cuda:0")
    sieve.lib()
    nprobe = args.nprobe or cfg.nprobe
    w = synth.make_sharded_workload(cfg, args.shards, args.nlist_per_shard, device=dev)
    shards = []
    for sh in w["shards"]:
        idx = sieve.build_layout(sh["X"], sh["assign"], sh["centroids"].shape[0], sh["centroids"])
        shards.append(sieve.Index(idx.vectors, sh["ids"][idx.ids], idx.list_offsets, idx.centroids,
                                  idx.tc_rows, idx.tc_row_blocks, idx.tc_centroids))
        sh.clear()
    Q, qids = w["Q"], w["qids"]
    del w
    gc.collect()
    torch.cuda.empty_cache()
    ws = sieve.Workspace()

    def timed(W, reps):
        run = lambda: sieve.sharded_search(shards, Q, cfg.tau, cfg.k, nprobe, W, query_ids=qids,
                                           workspace=ws)
        out = run()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            out = run()
        e1.record()
        torch.cuda.synchronize()
        return out, e0.elapsed_time(e1) / reps

    out, ms = timed(cfg.W, max(3, args.steps // 40))
    fx, ms_fixed = timed(nprobe, 3)
    f_ids, f_cnt = fx[0].cpu().numpy(), fx[2].cpu().numpy()

    def recall(o):
        a_ids, a_cnt = o[0].cpu().numpy(), o[2].cpu().numpy()
        kept = sum(len(set(a_ids[i, :a_cnt[i]]) & set(f_ids[i, :f_cnt[i]])) for i in range(len(a_cnt)))
        return kept / max(1, int(f_cnt.sum()))

    # every shard calibrates its own window on one 2% sample (0.5% loss target)
    g = torch.Generator(device="cpu").manual_seed(4242)
    ns = max(1, (cfg.nq * 2 + 99) // 100)
    sample = torch.sort(torch.randperm(cfg.nq, generator=g)[:ns]).values.to(dev)
    crun = lambda: sieve.sharded_calibrated_search(shards, Q, cfg.tau, cfg.k, nprobe, sample, 0.005,
                                                   query_ids=qids, workspace=ws)
    cout = crun()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(3):
        cout = crun()
    torch.cuda.synchronize()
    c_ms = (time.perf_counter() - t0) / 3 * 1e3
    print(json.dumps({
        "sharded": True, "workload": workload_desc(cfg), "shards": args.shards,
        "nlist_per_shard": args.nlist_per_shard, "nprobe_per_shard": nprobe, "W": cfg.W,
        "nq": cfg.nq, "ms_per_call": ms, "queries_per_s": cfg.nq / (ms * 1e-3),
        "fixed_ms_per_call": ms_fixed, "speedup_vs_fixed": ms_fixed / ms,
        "mean_probes_over_shards": float(out[3].float().mean()),
        "recall_vs_fixed": recall(out),
        "calibrated": {"Ws": cout[5], "sample": ns, "loss_target": 0.005, "ms_per_call": c_ms,
                       "queries_per_s": cfg.nq / (c_ms * 1e-3), "speedup_vs_fixed": ms_fixed / c_ms,
                       "mean_probes_over_shards": float(cout[3].float().mean()),
                       "recall_vs_fixed": recall(cout),
                       "timing": "host clock around whole calls (one read-back per shard)"},
        "timing": "CUDA events around whole calls (every shard's search and the merge)"}))
    return 0


def run_rq(args, cfg):
    """The quantized local search (RaBitQ-style codes, the paper's IVF_RQ7)
    on one workload: index build times, the search at the workload's W and
    at fixed probing, the kept neighbours against the exact search, the
    roofline of the scan over codes and the oracle's quantized search on a
    bounded query sample.  One JSON line."""
    import paper_2608_03199_gb300 as sieve
    dev = torch.device("cuda:0")
    sieve.lib()
    wl = synth.make_workload(cfg, device=dev)
    index = sieve.build_layout(wl["X"], wl["assign"], cfg.nlist, wl["centroids"])
    Q, qids = wl["Q"], wl["qids"]
    P_host = synth.make_rotation(cfg.d, seed=1234)
    P = torch.from_numpy(P_host).to(dev)
    torch.cuda.synchronize()
    e0, e1, e2 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
    e0.record()
    codes, factors = sieve.rq_encode(index, P, 7)
    e1.record()
    rqi = sieve.build_rq_layout(index, P, 7, codes=codes, factors=factors)
    e2.record()
    torch.cuda.synchronize()
    enc_ms, lay_ms = e0.elapsed_time(e1), e1.elapsed_time(e2)
    ws = sieve.Workspace()
    nq, k = cfg.nq, cfg.k
    outs = (torch.empty((nq, k), dtype=torch.int64, device=dev),
            torch.empty((nq, k), dtype=torch.float32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev),
            torch.empty(nq, dtype=torch.int32, device=dev))

    def step(W):
        return lambda: sieve.rq_search(index, rqi, Q, cfg.tau, k, cfg.nprobe, W, query_ids=qids,
                                       workspace=ws, out=outs)
    clocks = ClockSampler(0)
    clocks.start()
    ms = time_steps(step(cfg.W), args.steps, args.warmup, 1, dev)
    clock_rec = clocks.stop()
    ms_fixed = time_steps(step(cfg.nprobe), max(3, args.steps // 5), 2, 1, dev)
    prof = sieve.rq_search(index, rqi, Q, cfg.tau, k, cfg.nprobe, cfg.W, query_ids=qids,
                           profile=True, workspace=ws)[4]
    step(cfg.W)()
    rq_ids = outs[0].cpu().numpy()
    rq_cnt = outs[2].cpu().numpy()
    mean_probes = float(outs[3].float().mean().item())
    ex = sieve.search(index, Q, cfg.tau, k, cfg.nprobe, cfg.W, lookahead=True, query_ids=qids)
    ex_ids, ex_cnt = ex[0].cpu().numpy(), ex[2].cpu().numpy()
    kept = sum(len(set(rq_ids[i, :rq_cnt[i]]) & set(ex_ids[i, :ex_cnt[i]])) for i in range(nq))
    line = {
        "metric": METRIC + " (quantized local search)",
        "value": nq / (ms * 1e-3), "unit": "queries/s", "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "u8 codes (fp16 u - mid on the tensor cores), f32 queries",
        "data": "synthetic",
        "config": {"workload": workload_desc(cfg), "bits": 7, "rotation": "seeded Haar (QR)",
                   "l2": "inputs larger than L2 (codes 0.51 GB streamed per step)"},
        "index_build_ms": {"encode": enc_ms, "layout": lay_ms},
        "fixed_probe": {"value": nq / (ms_fixed * 1e-3), "ms_per_step": ms_fixed, "W": cfg.nprobe},
        "speedup_vs_fixed": ms_fixed / ms,
        "mean_probes": mean_probes,
        "kept_vs_exact": {"common": kept, "exact": int(ex_cnt.sum()), "quantized": int(rq_cnt.sum())},
        "roofline": roofline(prof, cfg, dev, bulk=True, rq=True),
        "profile": {"kernel_ms": prof["kernel_ms"], "kernel_launches": prof["kernel_launches"],
                    "rounds": prof["rounds"], "items": prof["items"], "pairs": prof["pairs"]},
        "gpu_launches": args.steps * int(sum(v for k, v in prof["kernel_launches"].items()
                                             if k != "rank_mma")),
        "clocks": clock_rec,
    }
    if not args.skip_cpu_baseline:
        import oracle
        w = host_arrays(wl)
        idx = {kk: w[kk] for kk in ("X", "ids", "assign", "centroids")}
        threads = oracle.default_threads()
        t0 = time.perf_counter()
        hc, hf = oracle.rq_encode(idx, P_host, 7, threads=threads)
        enc_s = time.perf_counter() - t0
        probe = min(nq, 64)
        t0 = time.perf_counter()
        oracle.rq_search(idx, hc, hf, P_host, w["Q"][:probe], cfg.tau, k, cfg.nprobe, cfg.W,
                         qids=w["qids"][:probe], threads=threads)
        per_q = (time.perf_counter() - t0) / probe
        sample = int(min(nq, max(probe, args.cpu_seconds / max(per_q, 1e-9))))
        t0 = time.perf_counter()
        oracle.rq_search(idx, hc, hf, P_host, w["Q"][:sample], cfg.tau, k, cfg.nprobe, cfg.W,
                         qids=w["qids"][:sample], threads=threads)
        dt = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": sample / dt, "unit": "queries/s", "cores": threads,
                                "kind": "oracle",
                                "sample": f"first {sample:,} of the {nq:,} queries, W={cfg.W}, "
                                          f"{dt:.1f} s on {threads} host threads (encoding the "
                                          f"index took {enc_s:.1f} s more)"}
    print(json.dumps(line))
    return 0


ALL_CONFIGS = ("tiny", "1m", "10m256", "10m512", "100m")


def run_all_configs(args):
    """Every configuration in its own process (the index and its layouts of
    one configuration leave the device before the next is built): each
    prints its own benchmark line, then one summary line with per_config."""
    per = {}
    for name in ALL_CONFIGS:
        cmd = [sys.executable, os.path.abspath(__file__), "--config", name, "--steps",
               str(args.steps), "--warmup", str(args.warmup), "--cpu-seconds", str(args.cpu_seconds),
               "--scan-path", args.scan_path, "--skip-calibration"]
        if args.skip_e2e:
            cmd.append("--skip-e2e")
        if args.skip_cpu_baseline:
            cmd.append("--skip-cpu-baseline")
        r = subprocess.run(cmd, capture_output=True, text=True)
        lines = [x for x in r.stdout.splitlines() if x.startswith("{")]
        if r.returncode != 0 or not lines:
            per[name] = {"error": f"rc={r.returncode}: {r.stderr.strip().splitlines()[-1:]}"}
            continue
        print(lines[-1], flush=True)
        b = json.loads(lines[-1])
        roof = b.get("roofline") or {}
        per[name] = {"value": b["value"], "ms_per_step": b["ms_per_step"],
                     "fixed_probe_value": b["fixed_probe"]["value"],
                     "speedup_vs_fixed": b["speedup_vs_fixed"], "mean_probes": b["mean_probes"],
                     "top_kernel": roof.get("kernel"), "frac": roof.get("frac"),
                     "roofline_unit": roof.get("unit"), "parity": b.get("parity"),
                     "clocks": b.get("clocks")}
    print(json.dumps({"all_configs": True, "metric": METRIC, "unit": "queries/s",
                      "steps": args.steps, "warmup": args.warmup, "per_config": per}))
    return 0 if all("error" not in v for v in per.values()) else 1


def run_ncu_case(args, cfg):
    """One search call on the benchmark workload, nothing else on the GPU after it."""
    import paper_2608_03199_gb300 as sieve
    dev = torch.device("cuda:0")
    sieve.lib()
    if args.ncu_case == "rank":
        # the ranking alone, on its own shape: unit centroids of the config's
        # nlist x d, queries near seeded centroids
        g = torch.Generator(device=dev).manual_seed(cfg.seed)
        C = torch.randn(cfg.nlist, cfg.d, device=dev, generator=g)
        C /= C.norm(dim=1, keepdim=True)
        Q = C[torch.randint(0, cfg.nlist, (args.ncu_queries,), device=dev, generator=g)]
        Q = Q + 0.1 * torch.randn(Q.shape, device=dev, generator=g)
        Q /= Q.norm(dim=1, keepdim=True)
        index = sieve.build_layout(C.clone(), torch.arange(cfg.nlist, dtype=torch.int32, device=dev),
                                   cfg.nlist, C)
        order = sieve.rank_partitions(index, Q, cfg.nprobe)
        torch.cuda.synchronize()
        print(json.dumps({"ncu_case": "rank", "nq": args.ncu_queries, "nlist": cfg.nlist, "d": cfg.d,
                          "nprobe": cfg.nprobe, "first": int(order[0, 0])}))
        return 0
    wl = synth.make_workload(cfg, device=dev)
    index = sieve.build_layout(wl["X"], wl["assign"], cfg.nlist, wl["centroids"])
    W = cfg.nprobe if args.ncu_case == "fixed" else cfg.W
    # host-driven rounds: ncu does not profile kernels inside a CUDA graph with
    # conditional nodes; the kernels and their arguments are the same
    if args.ncu_case == "rqw8":
        P = torch.from_numpy(synth.make_rotation(cfg.d, seed=1234)).to(dev)
        rqi = sieve.build_rq_layout(index, P, 7)
        out = sieve.rq_search(index, rqi, wl["Q"], cfg.tau, cfg.k, cfg.nprobe, W,
                              query_ids=wl["qids"], stats=True, loop=1)
    else:
        out = sieve.search(index, wl["Q"], cfg.tau, cfg.k, cfg.nprobe, W, lookahead=True,
                           query_ids=wl["qids"], stats=True, loop=1, scan_path=args.scan_path)
    print(json.dumps({"ncu_case": args.ncu_case, "W": W, "rounds": out[4]["rounds"],
                      "items": out[4]["items"], "pairs": out[4]["pairs"]}))
    return 0


def main():
    args = parse()
    cfg = synth.CONFIGS[args.config]
    world, rank, local = dist_setup(args.gpus)
    if args.all_configs:
        return run_all_configs(args)
    if args.ncu_case:
        return run_ncu_case(args, cfg)
    if args.sweep:
        return run_sweep(args, cfg)
    if args.rq:
        return run_rq(args, cfg)
    if args.shards:
        return run_sharded(args, cfg)
    if args.impl == "reference":
        return run_reference(args, cfg, world, rank)
    return run_sieve(args, cfg, world, rank, local)


if __name__ == "__main__":
    sys.exit(main())
