import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs through the C ABI)")


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
