"""The C-ABI library builds for sm_103a, loads, and exports every function that
include/*.h declares (no compute calls: this runs without a GPU)."""
import ctypes
import glob
import os
import re

import paper_2608_03199_gb300 as sieve

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^[A-Za-z_][\w \*]*?\b(sieve_\w+)\s*\(", text, flags=re.M):
            names.add(m.group(1))
    return names


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("sieve_rank_partitions", "sieve_search", "sieve_search_host",
                     "sieve_build_layout", "sieve_search_workspace_size", "sieve_status_str"):
        assert required in names


def test_library_exports_every_declared_symbol():
    path = sieve.build()
    lib = ctypes.CDLL(path)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing
    assert set(declared_functions()) <= set(sieve._SIGNATURES), "binding lacks a declared call"


def test_host_only_calls_without_gpu():
    lib = sieve.lib()
    assert lib.sieve_version().startswith(b"libsieve")
    assert lib.sieve_status_str(-1) == b"invalid argument"
    n = ctypes.c_size_t()
    assert lib.sieve_layout_workspace_size(1000, 16, ctypes.byref(n)) == 0 and n.value > 0
    assert lib.sieve_layout_workspace_size(-1, 16, ctypes.byref(n)) == -1
    v = sieve.IndexViewC(n=1000, nlist=16, d=64, vectors=16, ids=16, list_offsets=16, centroids=16)
    p = sieve._params(0.9, 10, 8, 4, True, 0, 0)
    assert lib.sieve_search_workspace_size(ctypes.byref(v), 100, ctypes.byref(p), 0,
                                           ctypes.byref(n)) == 0
    small = n.value
    assert lib.sieve_search_workspace_size(ctypes.byref(v), 100, ctypes.byref(p), 1,
                                           ctypes.byref(n)) == 0 and n.value > small
    for bad in (sieve._params(0.9, 0, 8, 4, True, 0, 0), sieve._params(0.9, 65, 8, 4, True, 0, 0),
                sieve._params(0.9, 10, 17, 4, True, 0, 0), sieve._params(0.9, 10, 8, 0, True, 0, 0),
                sieve._params(float("nan"), 10, 8, 4, True, 0, 0)):
        assert lib.sieve_search_workspace_size(ctypes.byref(v), 100, ctypes.byref(bad), 0,
                                               ctypes.byref(n)) == -1
    v.d = 62
    assert lib.sieve_search_workspace_size(ctypes.byref(v), 100, ctypes.byref(p), 0,
                                           ctypes.byref(n)) == -1
    # the status query rejects a missing or misaligned workspace before any copy
    st = ctypes.c_int32(5)
    assert lib.sieve_search_status(None, 1 << 20, ctypes.byref(st), None) == -1
    assert lib.sieve_search_status(ctypes.c_void_p(16), 1 << 20, ctypes.byref(st), None) == -1
    assert lib.sieve_search_status(ctypes.c_void_p(256), 1 << 20, None, None) == -1
    assert st.value == 5


def test_scan_path_values_without_gpu():
    """scan_path 0..3 (automatic, FP32 FMA, three fp16 products, the screen)
    are accepted; anything else is SIEVE_EINVAL before any device work."""
    lib = sieve.lib()
    n = ctypes.c_size_t()
    v = sieve.IndexViewC(n=1000, nlist=16, d=64, vectors=16, ids=16, list_offsets=16, centroids=16)
    for path in ("auto", "simt", "tensor", "screen", 0, 1, 2, 3):
        p = sieve._params(0.9, 10, 8, 4, True, 0, 0, scan_path=path)
        assert lib.sieve_search_workspace_size(ctypes.byref(v), 100, ctypes.byref(p), 0,
                                               ctypes.byref(n)) == 0
    for serial in (0, 1):
        p = sieve._params(0.9, 10, 8, 4, True, 0, 0, serial=serial)
        assert lib.sieve_search_workspace_size(ctypes.byref(v), 100, ctypes.byref(p), 0,
                                               ctypes.byref(n)) == 0
    p = sieve._params(0.9, 10, 8, 4, True, 0, 0)
    p.serial = 2
    assert lib.sieve_search_workspace_size(ctypes.byref(v), 100, ctypes.byref(p), 0,
                                           ctypes.byref(n)) == -1
    p.serial, p.wait_limit = 0, -1
    assert lib.sieve_search_workspace_size(ctypes.byref(v), 100, ctypes.byref(p), 0,
                                           ctypes.byref(n)) == -1
    for path in (-1, 4):
        p = sieve._params(0.9, 10, 8, 4, True, 0, 0, scan_path=path)
        assert lib.sieve_search_workspace_size(ctypes.byref(v), 100, ctypes.byref(p), 0,
                                               ctypes.byref(n)) == -1


def test_screen_scores_rejects_bad_arguments_without_gpu():
    """sieve_screen_scores checks its arguments on the host before any device
    work: it needs the centroids' tensor layout and d <= 256, and its output
    rows must hold every centroid at a 32-float stride (SIEVE_EINVAL)."""
    lib = sieve.lib()
    ok = dict(n=1000, nlist=100, d=64, vectors=16, ids=16, list_offsets=16, centroids=16,
              tc_centroids=16)
    q, out = ctypes.c_void_p(256), ctypes.c_void_p(512)
    v = sieve.IndexViewC(**{**ok, "tc_centroids": None})
    assert lib.sieve_screen_scores(ctypes.byref(v), q, 10, out, 128, None) == -1   # no layout
    v = sieve.IndexViewC(**{**ok, "d": 260})
    assert lib.sieve_screen_scores(ctypes.byref(v), q, 10, out, 128, None) == -1   # d > 256
    v = sieve.IndexViewC(**ok)
    assert lib.sieve_screen_scores(ctypes.byref(v), q, 10, out, 96, None) == -1    # ld < nlist
    assert lib.sieve_screen_scores(ctypes.byref(v), q, 10, out, 112, None) == -1   # ld % 32
    assert lib.sieve_screen_scores(ctypes.byref(v), q, -1, out, 128, None) == -1   # nq < 0
    assert lib.sieve_screen_scores(ctypes.byref(v), ctypes.c_void_p(260), 10, out, 128, None) == -1
    assert lib.sieve_screen_scores(ctypes.byref(v), q, 10, None, 128, None) == -1
