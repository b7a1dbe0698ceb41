"""Python binding of libsieve: threshold-aware IVF search on one GB300 (sm_103a).

This module only marshals arguments: it takes torch tensors (device memory and
streams come from PyTorch), passes raw pointers and sizes to the C ABI declared
in ``include/sieve.h``, and returns tensors.  Every step of the search runs in
libsieve's CUDA kernels; there is no CPU or PyTorch fallback.  If the library
cannot be built or loaded the calls raise.

Entry points (same names as the C ABI):

* :func:`build_layout`      -- partition-contiguous storage of an IVF index
* :func:`rank_partitions`   -- per-query top-nprobe centroid order
* :func:`search`            -- SieveIVF search on device tensors
* :func:`search_host`       -- the same with host queries and host results
* :func:`rq_encode`, :func:`build_rq_layout`, :func:`rq_search` -- the local
  search over RaBitQ-style codes (the paper's IVF_RQ7 index)
"""
from __future__ import annotations

import ctypes as C
import threading
from dataclasses import dataclass

import numpy as np
import torch

from . import _build

SIEVE_OK = 0
_STATUS = {0: "ok", -1: "invalid argument", -2: "CUDA error", -3: "workspace", -4: "round limit",
           -5: "unsupported device", -6: "exceeds the no-allocation scratch",
           -7: "device wait timed out"}


class SieveError(RuntimeError):
    def __init__(self, status: int, what: str, cuda_error: int = 0):
        msg = f"{what}: status {status} ({_STATUS.get(status, '?')})"
        if status == -2:
            msg += f", cudaError {cuda_error}"
        super().__init__(msg)
        self.status = status


class IndexViewC(C.Structure):
    _fields_ = [("n", C.c_int64), ("nlist", C.c_int64), ("d", C.c_int32), ("reserved0", C.c_int32),
                ("vectors", C.c_void_p), ("ids", C.c_void_p), ("list_offsets", C.c_void_p),
                ("centroids", C.c_void_p), ("tc_rows", C.c_void_p), ("tc_row_blocks", C.c_void_p),
                ("tc_centroids", C.c_void_p)]


class ParamsC(C.Structure):
    _fields_ = [("tau", C.c_float), ("k", C.c_int32), ("nprobe", C.c_int32), ("W", C.c_int32),
                ("lookahead", C.c_int32), ("loop", C.c_int32), ("profile", C.c_int32),
                ("scan_path", C.c_int32), ("serial", C.c_int32), ("wait_limit", C.c_int32),
                ("max_items_per_round", C.c_int64)]


class StatsC(C.Structure):
    _fields_ = [("rounds", C.c_int64), ("items", C.c_int64), ("groups", C.c_int64),
                ("tiles", C.c_int64), ("rows_read", C.c_int64), ("pairs", C.c_int64),
                ("rows_read_tc", C.c_int64), ("pairs_tc", C.c_int64),
                ("status", C.c_int32), ("reserved0", C.c_int32),
                ("kernel_ms", C.c_float * 12), ("kernel_launches", C.c_int32 * 12)]


class RqViewC(C.Structure):
    _fields_ = [("bits", C.c_int32), ("reserved0", C.c_int32), ("rq_rows", C.c_void_p),
                ("rq_row_blocks", C.c_void_p), ("rq_factors", C.c_void_p),
                ("rq_rotation", C.c_void_p)]


KERNELS = ("rank", "init", "issue", "bucket", "scatter", "scan", "merge", "round_end", "finalize",
           "scan_tc", "rq_rotate", "rank_mma")
SCAN_PATHS = {"auto": 0, "simt": 1, "tensor": 2, "screen": 3}


_lib = None
_lib_lock = threading.Lock()

# every function include/sieve.h declares, with its ctypes signature
_SIGNATURES = {
    "sieve_layout_workspace_size": (C.c_int32, [C.c_int64, C.c_int64, C.POINTER(C.c_size_t)]),
    "sieve_build_layout": (C.c_int32, [C.c_void_p, C.c_void_p, C.c_int64, C.c_int32, C.c_int64,
                                       C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_size_t,
                                       C.c_void_p]),
    "sieve_rank_workspace_size": (C.c_int32, [C.POINTER(IndexViewC), C.c_int64, C.c_int32,
                                              C.POINTER(C.c_size_t)]),
    "sieve_tc_layout_size": (C.c_int32, [C.POINTER(IndexViewC), C.POINTER(C.c_size_t),
                                         C.POINTER(C.c_size_t)]),
    "sieve_build_tc_layout": (C.c_int32, [C.POINTER(IndexViewC), C.c_void_p, C.c_void_p, C.c_void_p,
                                          C.c_void_p]),
    "sieve_rank_partitions": (C.c_int32, [C.POINTER(IndexViewC), C.c_void_p, C.c_int64, C.c_int32,
                                          C.c_void_p, C.c_void_p, C.c_void_p, C.c_size_t,
                                          C.c_void_p]),
    "sieve_screen_scores": (C.c_int32, [C.POINTER(IndexViewC), C.c_void_p, C.c_int64, C.c_void_p,
                                        C.c_int64, C.c_void_p]),
    "sieve_search_workspace_size": (C.c_int32, [C.POINTER(IndexViewC), C.c_int64,
                                                C.POINTER(ParamsC), C.c_int32,
                                                C.POINTER(C.c_size_t)]),
    "sieve_search": (C.c_int32, [C.POINTER(IndexViewC), C.c_void_p, C.c_int64, C.c_void_p,
                                 C.c_void_p, C.POINTER(ParamsC), C.c_void_p, C.c_void_p,
                                 C.c_void_p, C.c_void_p, C.POINTER(StatsC), C.c_void_p,
                                 C.c_size_t, C.c_void_p]),
    "sieve_search_status": (C.c_int32, [C.c_void_p, C.c_size_t, C.POINTER(C.c_int32), C.c_void_p]),
    "sieve_search_host": (C.c_int32, [C.POINTER(IndexViewC), C.c_void_p, C.c_int64, C.c_void_p,
                                      C.POINTER(ParamsC), C.c_void_p, C.c_void_p, C.c_void_p,
                                      C.c_void_p, C.POINTER(StatsC), C.c_void_p, C.c_size_t,
                                      C.c_void_p]),
    "sieve_search_noalloc": (C.c_int32, [C.POINTER(IndexViewC), C.c_void_p, C.c_int64,
                                         C.c_void_p, C.c_void_p, C.POINTER(ParamsC), C.c_void_p,
                                         C.c_void_p, C.c_void_p, C.c_void_p, C.POINTER(StatsC),
                                         C.c_void_p]),
    "sieve_calibrated_search_workspace_size": (C.c_int32, [C.POINTER(IndexViewC), C.c_int64,
                                                           C.c_int64, C.POINTER(ParamsC),
                                                           C.POINTER(C.c_size_t)]),
    "sieve_calibrated_search": (C.c_int32, [C.POINTER(IndexViewC), C.c_void_p, C.c_int64,
                                            C.c_void_p, C.POINTER(ParamsC), C.c_void_p, C.c_int64,
                                            C.c_double, C.c_int64, C.c_int32, C.c_void_p,
                                            C.c_void_p, C.c_void_p, C.c_void_p,
                                            C.POINTER(C.c_int32), C.c_void_p,
                                            C.POINTER(C.c_int64), C.c_void_p, C.c_size_t,
                                            C.c_void_p]),
    "sieve_sharded_search_workspace_size": (C.c_int32, [C.POINTER(IndexViewC), C.c_int32,
                                                        C.c_int64, C.POINTER(ParamsC),
                                                        C.c_void_p, C.POINTER(C.c_size_t)]),
    "sieve_sharded_search": (C.c_int32, [C.POINTER(IndexViewC), C.c_int32, C.c_void_p, C.c_int64,
                                         C.c_void_p, C.POINTER(ParamsC), C.c_void_p, C.c_void_p,
                                         C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                         C.c_void_p, C.c_size_t, C.c_void_p]),
    "sieve_merge_shard_results": (C.c_int32, [C.c_int32, C.c_int64, C.c_int32, C.c_void_p,
                                              C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                              C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                              C.c_void_p]),
    "sieve_rq_encode": (C.c_int32, [C.POINTER(IndexViewC), C.c_void_p, C.c_int32, C.c_void_p,
                                    C.c_void_p, C.c_void_p]),
    "sieve_rq_layout_size": (C.c_int32, [C.POINTER(IndexViewC), C.POINTER(C.c_size_t),
                                         C.POINTER(C.c_size_t), C.POINTER(C.c_size_t)]),
    "sieve_build_rq_layout": (C.c_int32, [C.POINTER(IndexViewC), C.c_void_p, C.c_void_p,
                                          C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                          C.c_void_p, C.c_void_p, C.c_void_p]),
    "sieve_rq_search_workspace_size": (C.c_int32, [C.POINTER(IndexViewC), C.c_int64,
                                                   C.POINTER(ParamsC), C.POINTER(C.c_size_t)]),
    "sieve_rq_search": (C.c_int32, [C.POINTER(IndexViewC), C.POINTER(RqViewC), C.c_void_p,
                                    C.c_int64, C.c_void_p, C.c_void_p, C.c_void_p,
                                    C.POINTER(ParamsC), C.c_void_p, C.c_void_p, C.c_void_p,
                                    C.c_void_p, C.POINTER(StatsC), C.c_void_p, C.c_size_t,
                                    C.c_void_p]),
    "sieve_status_str": (C.c_char_p, [C.c_int32]),
    "sieve_last_cuda_error": (C.c_int32, []),
    "sieve_version": (C.c_char_p, []),
}


def build(force: bool = False) -> str:
    """Compile libsieve for sm_103a (in-tree); returns the library path."""
    return _build.build(force=force)


def lib():
    """The loaded libsieve (built on first use)."""
    global _lib
    with _lib_lock:
        if _lib is None:
            path = _build.build()
            handle = C.CDLL(path)
            for name, (res, args) in _SIGNATURES.items():
                fn = getattr(handle, name)
                fn.restype = res
                fn.argtypes = args
            _lib = handle
        return _lib


def library_path() -> str:
    return _build.LIB


def _check(status: int, what: str):
    if status != SIEVE_OK:
        raise SieveError(status, what, lib().sieve_last_cuda_error())


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return C.c_void_p(stream.cuda_stream)


def _need_cuda(t, dtype, name, ndim=None):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims")
    return t


@dataclass
class Index:
    """A device-resident IVF index in the layout libsieve reads.

    ``tc_rows`` / ``tc_row_blocks`` / ``tc_centroids`` optionally hold the
    tensor-core layout (see :func:`add_tc_layout`)."""
    vectors: torch.Tensor        # [n][d] f32, partition-contiguous
    ids: torch.Tensor            # [n] i64
    list_offsets: torch.Tensor   # [nlist+1] i64
    centroids: torch.Tensor      # [nlist][d] f32
    tc_rows: torch.Tensor | None = None
    tc_row_blocks: torch.Tensor | None = None
    tc_centroids: torch.Tensor | None = None

    def view(self) -> IndexViewC:
        v = IndexViewC()
        v.n = self.vectors.shape[0]
        v.nlist = self.centroids.shape[0]
        v.d = self.vectors.shape[1]
        v.vectors = self.vectors.data_ptr()
        v.ids = self.ids.data_ptr()
        v.list_offsets = self.list_offsets.data_ptr()
        v.centroids = self.centroids.data_ptr()
        if self.tc_rows is not None:
            v.tc_rows = self.tc_rows.data_ptr()
            v.tc_row_blocks = self.tc_row_blocks.data_ptr()
            v.tc_centroids = self.tc_centroids.data_ptr()
        return v

    def without_tc_layout(self) -> "Index":
        return Index(self.vectors, self.ids, self.list_offsets, self.centroids)

    @property
    def nlist(self):
        return self.centroids.shape[0]

    @property
    def d(self):
        return self.vectors.shape[1]


# widest rows the bulk tensor-core pipelines take (their A operand lives in
# tensor memory: at most four 64-element K-blocks)
TC_BULK_MAX_D = 256


def add_tc_layout(index: Index, stream=None) -> Index:
    """The same index with its tensor-core layout built (sieve_build_tc_layout)."""
    base = index.without_tc_layout()
    v = base.view()
    rb, cb = C.c_size_t(), C.c_size_t()
    _check(lib().sieve_tc_layout_size(C.byref(v), C.byref(rb), C.byref(cb)), "sieve_tc_layout_size")
    dev = index.vectors.device
    rows = torch.empty(max(rb.value, 256), dtype=torch.uint8, device=dev)
    blocks = torch.empty(index.nlist + 1, dtype=torch.int64, device=dev)
    cent = torch.empty(max(cb.value, 256), dtype=torch.uint8, device=dev)
    _check(lib().sieve_build_tc_layout(C.byref(v), _ptr(rows), _ptr(blocks), _ptr(cent),
                                       _stream(stream)), "sieve_build_tc_layout")
    return Index(index.vectors, index.ids, index.list_offsets, index.centroids, rows, blocks, cent)


def build_layout(X, assign, nlist, centroids, stream=None, tc_layout=None) -> Index:
    """Index from rows X [n][d] and their partitions assign [n] (sieve_build_layout),
    with its tensor-core layout when ``tc_layout`` is True, or by default when
    d <= 256 (the width the bulk tensor-core pipelines take).

    ids of the index are the row numbers of X."""
    _need_cuda(X, torch.float32, "X", 2)
    _need_cuda(assign, torch.int32, "assign", 1)
    _need_cuda(centroids, torch.float32, "centroids", 2)
    n, d = X.shape
    L = lib()
    nbytes = C.c_size_t()
    _check(L.sieve_layout_workspace_size(n, nlist, C.byref(nbytes)), "sieve_layout_workspace_size")
    ws = torch.empty(max(nbytes.value, 1), dtype=torch.uint8, device=X.device)
    Xs = torch.empty_like(X)
    ids = torch.empty(n, dtype=torch.int64, device=X.device)
    off = torch.empty(nlist + 1, dtype=torch.int64, device=X.device)
    _check(L.sieve_build_layout(_ptr(X), _ptr(assign), n, d, nlist, _ptr(Xs), _ptr(ids), _ptr(off),
                                _ptr(ws), nbytes.value, _stream(stream)), "sieve_build_layout")
    index = Index(Xs, ids, off, centroids.contiguous())
    if tc_layout is None:
        tc_layout = d <= TC_BULK_MAX_D
    return add_tc_layout(index, stream) if tc_layout else index


def rank_partitions(index: Index, Q, nprobe, return_scores=False, stream=None):
    """int32 [nq][nprobe] centroid order per query (sieve_rank_partitions)."""
    _need_cuda(Q, torch.float32, "Q", 2)
    nq = Q.shape[0]
    order = torch.empty((nq, nprobe), dtype=torch.int32, device=Q.device)
    sc = torch.empty((nq, nprobe), dtype=torch.float32, device=Q.device) if return_scores else None
    v = index.view()
    nbytes = C.c_size_t()
    _check(lib().sieve_rank_workspace_size(C.byref(v), nq, nprobe, C.byref(nbytes)),
           "sieve_rank_workspace_size")
    ws = torch.empty(max(nbytes.value, 256), dtype=torch.uint8, device=Q.device)
    _check(lib().sieve_rank_partitions(C.byref(v), _ptr(Q), nq, nprobe, _ptr(order), _ptr(sc),
                                       _ptr(ws), ws.numel(), _stream(stream)), "sieve_rank_partitions")
    return (order, sc) if return_scores else order


def screen_scores(index: Index, Q, stream=None):
    """fp32 [nq][nlist]: the ranking's first-pass (screen) score of every
    (query, centroid) pair, one fp16 product of the hi halves summed on the
    tensor cores (sieve_screen_scores); needs the centroids' tensor layout."""
    _need_cuda(Q, torch.float32, "Q", 2)
    nq = Q.shape[0]
    nlist = index.centroids.shape[0]
    ld = (nlist + 31) // 32 * 32
    out = torch.empty((nq, ld), dtype=torch.float32, device=Q.device)
    v = index.view()
    _check(lib().sieve_screen_scores(C.byref(v), _ptr(Q), nq, _ptr(out), ld, _stream(stream)),
           "sieve_screen_scores")
    return out[:, :nlist]


def _params(tau, k, nprobe, W, lookahead, loop, max_items_per_round, profile=0, scan_path="auto",
            serial=False, wait_limit=0):
    p = ParamsC()
    p.serial = 1 if serial else 0
    p.wait_limit = int(wait_limit)
    p.profile = int(profile)
    p.scan_path = SCAN_PATHS[scan_path] if isinstance(scan_path, str) else int(scan_path)
    p.tau = float(tau)
    p.k = int(k)
    p.nprobe = int(nprobe)
    p.W = int(min(W, 2**31 - 1))
    p.lookahead = 1 if lookahead else 0
    p.loop = int(loop)
    p.max_items_per_round = int(max_items_per_round)
    return p


def workspace_size(index: Index, nq, tau, k, nprobe, W, lookahead=True, max_items_per_round=0,
                   host_io=False) -> int:
    v = index.view()
    p = _params(tau, k, nprobe, W, lookahead, 0, max_items_per_round)
    nbytes = C.c_size_t()
    _check(lib().sieve_search_workspace_size(C.byref(v), nq, C.byref(p), 1 if host_io else 0,
                                             C.byref(nbytes)), "sieve_search_workspace_size")
    return nbytes.value


class Workspace:
    """A reusable device scratch buffer (grown on demand)."""

    def __init__(self, device=None):
        self.device = device
        self.buf = None

    def get(self, nbytes, device):
        if self.buf is None or self.buf.numel() < nbytes or self.buf.device != device:
            self.buf = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=device)
        return self.buf


_default_ws = {}


def _workspace(ws, nbytes, device):
    if ws is None:
        key = (device, torch.cuda.current_stream(device).cuda_stream)
        ws = _default_ws.setdefault(key, Workspace())
    return ws.get(nbytes, device)


def _stats_dict(st):
    out = {f: getattr(st, f) for f, _ in StatsC._fields_ if not f.startswith("kernel")}
    out["kernel_ms"] = dict(zip(KERNELS, list(st.kernel_ms)))
    out["kernel_launches"] = dict(zip(KERNELS, list(st.kernel_launches)))
    return out


def search(index: Index, Q, tau, k, nprobe, W, lookahead=True, query_ids=None, order=None,
           max_items_per_round=0, loop=0, stats=False, profile=False, scan_path="auto",
           workspace=None, out=None, stream=None, check=False, serial=False, wait_limit=0):
    """SieveIVF search on device tensors (sieve_search).

    Returns (ids [nq][k] i64, scores [nq][k] f32, count [nq] i32, probes [nq] i32),
    plus a dict of counters when ``stats`` or ``profile`` (both synchronize the
    stream; ``profile`` also times every kernel launch with CUDA events).
    ``check``: read the device status word after the call
    (sieve_search_status, which synchronizes the stream) and raise on a
    device-side error; stats and host-driven rounds check it anyway.
    ``serial``: the serial traversal (every (query, rank) item its own
    partition call; the same results)."""
    stats = stats or profile
    _need_cuda(Q, torch.float32, "Q", 2)
    if query_ids is not None:
        _need_cuda(query_ids, torch.int64, "query_ids", 1)
    if order is not None:
        _need_cuda(order, torch.int32, "order", 2)
    nq = Q.shape[0]
    dev = Q.device
    p = _params(tau, k, nprobe, W, lookahead, loop, max_items_per_round, profile, scan_path, serial,
                wait_limit)
    v = index.view()
    nbytes = C.c_size_t()
    _check(lib().sieve_search_workspace_size(C.byref(v), nq, C.byref(p), 0, C.byref(nbytes)),
           "sieve_search_workspace_size")
    ws = _workspace(workspace, nbytes.value, dev)
    if out is None:
        out = (torch.empty((nq, k), dtype=torch.int64, device=dev),
               torch.empty((nq, k), dtype=torch.float32, device=dev),
               torch.empty(nq, dtype=torch.int32, device=dev),
               torch.empty(nq, dtype=torch.int32, device=dev))
    ids, scores, count, probes = out
    st = StatsC() if stats else None
    _check(lib().sieve_search(C.byref(v), _ptr(Q), nq, _ptr(query_ids), _ptr(order), C.byref(p),
                              _ptr(ids), _ptr(scores), _ptr(count), _ptr(probes),
                              C.byref(st) if st is not None else None, _ptr(ws), ws.numel(),
                              _stream(stream)), "sieve_search")
    if check and nq > 0:
        _check(search_status(ws, stream), "sieve_search (device status)")
    if stats:
        return ids, scores, count, probes, _stats_dict(st)
    return ids, scores, count, probes


def search_status(ws, stream=None) -> int:
    """The device status word of the last search that used the workspace
    tensor ``ws`` (sieve_search_status; synchronizes the stream): 0 or a
    negative SIEVE_E* code."""
    if isinstance(ws, Workspace):
        ws = ws.buf
    v = C.c_int32(0)
    _check(lib().sieve_search_status(_ptr(ws), ws.numel(), C.byref(v), _stream(stream)),
           "sieve_search_status")
    return int(v.value)


@dataclass
class RQIndex:
    """RaBitQ-style codes of an index (the paper's IVF_RQ7: RaBitQ with 7
    bits) in the layout the quantized scan reads.  ``codes`` [n][d] u8 and
    ``factors`` [n] f32 are in the index's row order; the rest is their scan
    layout (:func:`build_rq_layout`)."""
    bits: int
    codes: torch.Tensor
    factors: torch.Tensor
    rows: torch.Tensor            # fp16 (u - mid) tiles, 16 KB per block K-block
    row_blocks: torch.Tensor      # [nlist+1] i64
    block_factors: torch.Tensor   # [blocks * 128] f32
    rotation: torch.Tensor        # tensor-core layout of P^T

    def view(self) -> RqViewC:
        v = RqViewC()
        v.bits = self.bits
        v.rq_rows = self.rows.data_ptr()
        v.rq_row_blocks = self.row_blocks.data_ptr()
        v.rq_factors = self.block_factors.data_ptr()
        v.rq_rotation = self.rotation.data_ptr()
        return v


def rq_encode(index: Index, P, bits=7, stream=None):
    """Codes [n][d] u8 and factors [n] f32 of the index's rows for the
    orthogonal rotation P [d][d] (float64, device) (sieve_rq_encode)."""
    _need_cuda(P, torch.float64, "P", 2)
    n, d = index.vectors.shape
    dev = index.vectors.device
    codes = torch.empty((n, d), dtype=torch.uint8, device=dev)
    factors = torch.empty(n, dtype=torch.float32, device=dev)
    v = index.view()
    _check(lib().sieve_rq_encode(C.byref(v), _ptr(P), int(bits), _ptr(codes), _ptr(factors),
                                 _stream(stream)), "sieve_rq_encode")
    return codes, factors


def build_rq_layout(index: Index, P, bits=7, codes=None, factors=None, stream=None) -> RQIndex:
    """The quantized index: codes (encoded here unless given) and their scan
    layout (sieve_build_rq_layout)."""
    _need_cuda(P, torch.float64, "P", 2)
    if codes is None or factors is None:
        codes, factors = rq_encode(index, P, bits, stream)
    _need_cuda(codes, torch.uint8, "codes", 2)
    _need_cuda(factors, torch.float32, "factors", 1)
    v = index.view()
    rb, fb, ob = C.c_size_t(), C.c_size_t(), C.c_size_t()
    _check(lib().sieve_rq_layout_size(C.byref(v), C.byref(rb), C.byref(fb), C.byref(ob)),
           "sieve_rq_layout_size")
    dev = index.vectors.device
    rows = torch.empty(max(rb.value, 256), dtype=torch.uint8, device=dev)
    blocks = torch.empty(index.nlist + 1, dtype=torch.int64, device=dev)
    bfac = torch.empty(max(fb.value // 4, 64), dtype=torch.float32, device=dev)
    rot = torch.empty(max(ob.value, 256), dtype=torch.uint8, device=dev)
    _check(lib().sieve_build_rq_layout(C.byref(v), _ptr(codes), _ptr(factors), int(bits), _ptr(P),
                                       _ptr(rows), _ptr(blocks), _ptr(bfac), _ptr(rot),
                                       _stream(stream)), "sieve_build_rq_layout")
    return RQIndex(int(bits), codes, factors, rows, blocks, bfac, rot)


def rq_search(index: Index, rq: RQIndex, Q, tau, k, nprobe, W, lookahead=True, query_ids=None,
              order=None, cscores=None, max_items_per_round=0, loop=0, stats=False,
              profile=False, workspace=None, out=None, stream=None):
    """search() with the quantized local search over rq's codes
    (sieve_rq_search): a row qualifies iff its estimate <q, c_p> +
    f <u - mid, P^T q> >= tau.  A precomputed ``order`` needs its ``cscores``."""
    stats = stats or profile
    _need_cuda(Q, torch.float32, "Q", 2)
    if query_ids is not None:
        _need_cuda(query_ids, torch.int64, "query_ids", 1)
    if order is not None:
        _need_cuda(order, torch.int32, "order", 2)
    if cscores is not None:
        _need_cuda(cscores, torch.float32, "cscores", 2)
    nq = Q.shape[0]
    dev = Q.device
    p = _params(tau, k, nprobe, W, lookahead, loop, max_items_per_round, profile, "auto")
    v = index.view()
    rv = rq.view()
    nbytes = C.c_size_t()
    _check(lib().sieve_rq_search_workspace_size(C.byref(v), nq, C.byref(p), C.byref(nbytes)),
           "sieve_rq_search_workspace_size")
    ws = _workspace(workspace, nbytes.value, dev)
    if out is None:
        out = (torch.empty((nq, k), dtype=torch.int64, device=dev),
               torch.empty((nq, k), dtype=torch.float32, device=dev),
               torch.empty(nq, dtype=torch.int32, device=dev),
               torch.empty(nq, dtype=torch.int32, device=dev))
    ids, scores, count, probes = out
    st = StatsC() if stats else None
    _check(lib().sieve_rq_search(C.byref(v), C.byref(rv), _ptr(Q), nq, _ptr(query_ids), _ptr(order),
                                 _ptr(cscores), C.byref(p), _ptr(ids), _ptr(scores), _ptr(count),
                                 _ptr(probes), C.byref(st) if st is not None else None, _ptr(ws),
                                 ws.numel(), _stream(stream)), "sieve_rq_search")
    if stats:
        return ids, scores, count, probes, _stats_dict(st)
    return ids, scores, count, probes


def calibrated_search(index: Index, Q, tau, k, nprobe, sample, eps, min_queries=10_000,
                      fallback_W=8, lookahead=True, query_ids=None, max_items_per_round=0,
                      scan_path="auto", workspace=None, stream=None):
    """In-call window calibration (sieve_calibrated_search, Appendix A).

    sample: int64 device tensor of strictly increasing row indices of Q (the
    queries that are fully probed).  Returns (ids, scores, count, probes,
    info) with info = dict(W = the selected window, hist = numpy [nprobe + 1]
    counts of neighbours by required window, Z = their total).  The call
    synchronizes the stream once."""
    _need_cuda(Q, torch.float32, "Q", 2)
    _need_cuda(sample, torch.int64, "sample", 1)
    if query_ids is not None:
        _need_cuda(query_ids, torch.int64, "query_ids", 1)
    nq, ns = Q.shape[0], sample.shape[0]
    dev = Q.device
    p = _params(tau, k, nprobe, nprobe, lookahead, 0, max_items_per_round, 0, scan_path)
    v = index.view()
    nbytes = C.c_size_t()
    _check(lib().sieve_calibrated_search_workspace_size(C.byref(v), nq, ns, C.byref(p),
                                                        C.byref(nbytes)),
           "sieve_calibrated_search_workspace_size")
    ws = _workspace(workspace, nbytes.value, dev)
    ids = torch.empty((nq, k), dtype=torch.int64, device=dev)
    scores = torch.empty((nq, k), dtype=torch.float32, device=dev)
    count = torch.empty(nq, dtype=torch.int32, device=dev)
    probes = torch.empty(nq, dtype=torch.int32, device=dev)
    W = C.c_int32(0)
    Z = C.c_int64(0)
    hist = np.zeros(nprobe + 1, np.int64)
    _check(lib().sieve_calibrated_search(C.byref(v), _ptr(Q), nq, _ptr(query_ids), C.byref(p),
                                         _ptr(sample), ns, float(eps), int(min_queries),
                                         int(fallback_W), _ptr(ids), _ptr(scores), _ptr(count),
                                         _ptr(probes), C.byref(W),
                                         hist.ctypes.data_as(C.c_void_p), C.byref(Z), _ptr(ws),
                                         ws.numel(), _stream(stream)), "sieve_calibrated_search")
    return ids, scores, count, probes, {"W": W.value, "hist": hist, "Z": Z.value}


def sharded_search(shards, Q, tau, k, nprobe, W, lookahead=True, query_ids=None,
                   max_items_per_round=0, scan_path="auto", workspace=None, stream=None):
    """sieve_sharded_search over a list of Index shards (distinct ids across
    shards): each shard searches the batch with its own ranking and stopping
    (W: one window, or one per shard), the global top-k merges them.
    Returns (ids, scores, count, probes = partitions over all shards,
    shard_probes [nq][nshards])."""
    _need_cuda(Q, torch.float32, "Q", 2)
    if query_ids is not None:
        _need_cuda(query_ids, torch.int64, "query_ids", 1)
    nq, ns = Q.shape[0], len(shards)
    dev = Q.device
    Ws = list(W) if isinstance(W, (list, tuple)) else [W] * ns
    p = _params(tau, k, nprobe, max(Ws), lookahead, 0, max_items_per_round, 0, scan_path)
    views = (IndexViewC * ns)(*[sh.view() for sh in shards])
    wps = (C.c_int32 * ns)(*[int(min(w, 2**31 - 1)) for w in Ws])
    nbytes = C.c_size_t()
    _check(lib().sieve_sharded_search_workspace_size(views, ns, nq, C.byref(p), wps, C.byref(nbytes)),
           "sieve_sharded_search_workspace_size")
    ws = _workspace(workspace, nbytes.value, dev)
    ids = torch.empty((nq, k), dtype=torch.int64, device=dev)
    scores = torch.empty((nq, k), dtype=torch.float32, device=dev)
    count = torch.empty(nq, dtype=torch.int32, device=dev)
    probes = torch.empty(nq, dtype=torch.int32, device=dev)
    shard_probes = torch.empty((nq, ns), dtype=torch.int32, device=dev)
    _check(lib().sieve_sharded_search(views, ns, _ptr(Q), nq, _ptr(query_ids), C.byref(p), wps,
                                      _ptr(ids), _ptr(scores), _ptr(count), _ptr(probes),
                                      _ptr(shard_probes), _ptr(ws), ws.numel(), _stream(stream)),
           "sieve_sharded_search")
    return ids, scores, count, probes, shard_probes


def sharded_calibrated_search(shards, Q, tau, k, nprobe, sample, eps, min_queries=10_000,
                              fallback_W=8, lookahead=True, query_ids=None, scan_path="auto",
                              workspace=None, stream=None):
    """Every shard calibrates its own window on the same sample
    (sieve_calibrated_search per shard, Appendix A), then the global top-k
    (sieve_merge_shard_results).  Returns (ids, scores, count, probes,
    shard_probes, Ws) with Ws the window each shard selected."""
    nq, ns = Q.shape[0], len(shards)
    dev = Q.device
    ids = torch.empty((ns, nq, k), dtype=torch.int64, device=dev)
    scores = torch.empty((ns, nq, k), dtype=torch.float32, device=dev)
    count = torch.empty((ns, nq), dtype=torch.int32, device=dev)
    probes = torch.empty((ns, nq), dtype=torch.int32, device=dev)
    Ws = []
    for s, sh in enumerate(shards):
        out = calibrated_search(sh, Q, tau, k, nprobe, sample, eps, min_queries=min_queries,
                                fallback_W=fallback_W, lookahead=lookahead, query_ids=query_ids,
                                scan_path=scan_path, workspace=workspace, stream=stream)
        ids[s].copy_(out[0])
        scores[s].copy_(out[1])
        count[s].copy_(out[2])
        probes[s].copy_(out[3])
        Ws.append(out[4]["W"])
    o_ids = torch.empty((nq, k), dtype=torch.int64, device=dev)
    o_sc = torch.empty((nq, k), dtype=torch.float32, device=dev)
    o_cnt = torch.empty(nq, dtype=torch.int32, device=dev)
    o_pr = torch.empty(nq, dtype=torch.int32, device=dev)
    o_sp = torch.empty((nq, ns), dtype=torch.int32, device=dev)
    _check(lib().sieve_merge_shard_results(ns, nq, k, _ptr(ids), _ptr(scores), _ptr(count),
                                           _ptr(probes), _ptr(o_ids), _ptr(o_sc), _ptr(o_cnt),
                                           _ptr(o_pr), _ptr(o_sp), _stream(stream)),
           "sieve_merge_shard_results")
    return o_ids, o_sc, o_cnt, o_pr, o_sp, Ws


def search_host(index: Index, Q_host, tau, k, nprobe, W, lookahead=True, query_ids_host=None,
                max_items_per_round=0, loop=0, scan_path="auto", workspace=None, out=None,
                stream=None):
    """sieve_search_host: host (CPU, ideally pinned) queries in, host results out.

    The call copies the queries to the device, searches, copies the results
    back and synchronizes the stream."""
    if Q_host.is_cuda or Q_host.dtype != torch.float32 or not Q_host.is_contiguous():
        raise TypeError("Q_host must be a contiguous float32 CPU tensor")
    if query_ids_host is not None and (query_ids_host.is_cuda or query_ids_host.dtype != torch.int64):
        raise TypeError("query_ids_host must be an int64 CPU tensor")
    nq = Q_host.shape[0]
    dev = index.vectors.device
    p = _params(tau, k, nprobe, W, lookahead, loop, max_items_per_round, 0, scan_path)
    v = index.view()
    nbytes = C.c_size_t()
    _check(lib().sieve_search_workspace_size(C.byref(v), nq, C.byref(p), 1, C.byref(nbytes)),
           "sieve_search_workspace_size")
    ws = _workspace(workspace, nbytes.value, dev)
    if out is None:
        out = (torch.empty((nq, k), dtype=torch.int64, pin_memory=True),
               torch.empty((nq, k), dtype=torch.float32, pin_memory=True),
               torch.empty(nq, dtype=torch.int32, pin_memory=True),
               torch.empty(nq, dtype=torch.int32, pin_memory=True))
    ids, scores, count, probes = out
    _check(lib().sieve_search_host(C.byref(v), _ptr(Q_host), nq, _ptr(query_ids_host), C.byref(p),
                                   _ptr(ids), _ptr(scores), _ptr(count), _ptr(probes), None,
                                   _ptr(ws), ws.numel(), _stream(stream)), "sieve_search_host")
    return ids, scores, count, probes


NOALLOC_SCRATCH_BYTES = 64 << 20


def search_noalloc(index: Index, Q, tau, k, nprobe, W, lookahead=True, query_ids=None,
                   order=None, max_items_per_round=0, out=None, stream=None):
    """sieve_search_noalloc: the search with no device allocation in the call.

    For callers that cannot allocate device memory: the scratch is a fixed
    array inside libsieve (NOALLOC_SCRATCH_BYTES per GPU, held until exit);
    the caller passes the output tensors in ``out`` to keep the call itself
    allocation-free.  Returns (ids, scores, count, probes), complete once the
    stream has passed the call."""
    _need_cuda(Q, torch.float32, "Q", 2)
    nq = Q.shape[0]
    if out is None:
        dev = Q.device
        out = (torch.empty((nq, k), dtype=torch.int64, device=dev),
               torch.empty((nq, k), dtype=torch.float32, device=dev),
               torch.empty(nq, dtype=torch.int32, device=dev),
               torch.empty(nq, dtype=torch.int32, device=dev))
    ids, scores, count, probes = out
    p = _params(tau, k, nprobe, W, lookahead, 1, max_items_per_round)
    v = index.view()
    _check(lib().sieve_search_noalloc(C.byref(v), _ptr(Q), nq, _ptr(query_ids), _ptr(order),
                                      C.byref(p), _ptr(ids), _ptr(scores), _ptr(count),
                                      _ptr(probes), None, _stream(stream)), "sieve_search_noalloc")
    return ids, scores, count, probes
