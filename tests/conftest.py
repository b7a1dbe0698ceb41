import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs through the C ABI)")


def pytest_terminal_summary(terminalreporter):
    """The divergence count of every parity comparison of the session: queries
    identical to the oracle, queries that differ where the oracle's fragility
    tags put a decision within 1e-5 of a rounding flip (allowed), and
    queries that differ without one (unexplained, which fail their test)."""
    parity = sys.modules.get("parity")
    reports = getattr(parity, "REPORTS", None)
    if not reports:
        return
    tr = terminalreporter
    tr.section("parity against the oracle")
    tot = [0, 0, 0, 0]
    worst = 0.0
    for label, nq, exact, allowed, unexplained, err in reports:
        tr.write_line(f"{label}: {nq} queries, {exact} exact, {allowed} allowed, "
                      f"{unexplained} unexplained, max score err {err:.2e}")
        for i, v in enumerate((nq, exact, allowed, unexplained)):
            tot[i] += v
        worst = max(worst, err)
    tr.write_line(f"total: {len(reports)} comparisons, {tot[0]} queries, {tot[1]} exact, "
                  f"{tot[2]} allowed, {tot[3]} unexplained, max score err {worst:.2e}")


@pytest.fixture(scope="session")
def tiny():
    """The tiny workload (20K x 64, nlist 64, 1K queries), host numpy arrays."""
    import synth
    wl = synth.make_workload("tiny", device="cpu")
    out = synth.to_numpy(wl)
    out["cfg"] = wl["cfg"]
    return out


@pytest.fixture(scope="session")
def deep():
    """A small workload whose duplicates spread over several partitions, so
    queries hit at ranks beyond 1 and the stop line moves (2K queries would be
    slow for the brute-force pins, so 400)."""
    import synth
    cfg = synth.scaled("tiny", n=12_000, d=32, ncomp=16, nlist=96, nq=400, dup_frac=0.08,
                       dup_counts=("uniform", 2, 12), dup_sigma=(0.03, 0.09), tau=0.88,
                       nprobe=24, W=3, seed=11)
    wl = synth.make_workload(cfg, device="cpu")
    out = synth.to_numpy(wl)
    out["cfg"] = cfg
    return out


def index_of(w):
    return {"X": w["X"], "ids": w["ids"], "assign": w["assign"], "centroids": w["centroids"]}
