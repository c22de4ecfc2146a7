"""Plain CPU oracle for AGNES hyperbatch sampling + gathering (arXiv 2601.01473).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s cpu_baseline / ``--impl reference`` legs may import this
package.  It wraps ``agnes_oracle.c`` (plain, single-threaded C) with ctypes
and shares no code with the CUDA library; it never imports the product
package.

What it computes is the per-minibatch definition of Algorithm 1 (Sec. 3.5):
for each minibatch, K hops of uniform sampling without replacement of up to
``fanout`` neighbours per frontier node (Philox4x32-10 keyed on
(seed, minibatch, hop, node, slot); Floyd's algorithm), union / dedup of the
sampled ids into ascending new nodes, relabelling of every sampled edge into
the hop's source list, and the gather of one feature row per final node.
Blocks enter only through the blocks-touched statistics (Sec. 3.2, Sec. 3.3).
"""
from __future__ import annotations

import ctypes
from dataclasses import dataclass

import numpy as np

from . import build as _build

MAX_HOPS = 8

_lib = None


class _OrcGraph(ctypes.Structure):
    _fields_ = [
        ("num_nodes", ctypes.c_int64),
        ("num_edges", ctypes.c_int64),
        ("offsets", ctypes.c_void_p),
        ("offsets_bits", ctypes.c_int32),
        ("indices", ctypes.c_void_p),
        ("features", ctypes.c_void_p),
        ("row_bytes", ctypes.c_int64),
    ]


class _OrcMinibatch(ctypes.Structure):
    _fields_ = [
        ("K", ctypes.c_int32),
        ("num_dst", ctypes.c_int64 * MAX_HOPS),
        ("num_src", ctypes.c_int64 * MAX_HOPS),
        ("num_edges", ctypes.c_int64 * MAX_HOPS),
        ("indptr", ctypes.c_void_p * MAX_HOPS),
        ("nbr", ctypes.c_void_p * MAX_HOPS),
        ("col", ctypes.c_void_p * MAX_HOPS),
        ("nodes", ctypes.c_void_p),
        ("num_nodes", ctypes.c_int64),
        ("feats", ctypes.c_void_p),
        ("dst", ctypes.c_void_p * MAX_HOPS),
    ]


FRONTIER = {"src": 0, "sampled": 1}  # ORC_FRONTIER_SRC / ORC_FRONTIER_SAMPLED


def lib() -> ctypes.CDLL:
    """Loads (building first if stale) the oracle's shared library."""
    global _lib
    if _lib is None:
        path = _build.build_oracle()
        L = ctypes.CDLL(path)
        L.orc_philox4x32_10.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
        L.orc_philox4x32_10.restype = None
        L.orc_mulhi64.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        L.orc_mulhi64.restype = ctypes.c_uint64
        L.orc_sample_positions.argtypes = [
            ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p]
        L.orc_sample_positions.restype = ctypes.c_int64
        L.orc_build_adj_blocks.argtypes = [
            ctypes.POINTER(_OrcGraph), ctypes.c_int64, ctypes.c_void_p,
            ctypes.POINTER(ctypes.c_int64)]
        L.orc_build_adj_blocks.restype = ctypes.c_int
        L.orc_sample_minibatch.argtypes = [
            ctypes.POINTER(_OrcGraph), ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p,
            ctypes.c_int32, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int,
            ctypes.POINTER(_OrcMinibatch)]
        L.orc_sample_minibatch.restype = ctypes.c_int
        L.orc_sample_minibatch_mode.argtypes = [
            ctypes.POINTER(_OrcGraph), ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p,
            ctypes.c_int32, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int, ctypes.c_int32,
            ctypes.POINTER(_OrcMinibatch)]
        L.orc_sample_minibatch_mode.restype = ctypes.c_int
        L.orc_free_minibatch.argtypes = [ctypes.POINTER(_OrcMinibatch)]
        L.orc_free_minibatch.restype = None
        L.orc_hyperbatch_stats.argtypes = [
            ctypes.POINTER(_OrcGraph), ctypes.POINTER(_OrcMinibatch), ctypes.c_int32,
            ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p]
        L.orc_hyperbatch_stats.restype = ctypes.c_int
        _lib = L
    return _lib


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data if a is not None and a.size > 0 else 0


class OracleError(RuntimeError):
    pass


# ----------------------------------------------------------------------------
# Primitives
# ----------------------------------------------------------------------------

def philox4x32_10(ctr, key):
    """Philox4x32-10 of a 4-word counter under a 2-word key (SC'11)."""
    c = np.asarray(ctr, dtype=np.uint32)
    k = np.asarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().orc_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return tuple(int(x) for x in out)


def mulhi64(a: int, b: int) -> int:
    """floor(a * b / 2**64) for unsigned 64-bit a, b."""
    return int(lib().orc_mulhi64(a, b))


def sample_positions(seed: int, g: int, hop: int, v: int, deg: int, k: int) -> list:
    """Neighbour positions node v draws at ``hop`` of minibatch g, slot order."""
    out = np.zeros(max(min(deg, k), 1), dtype=np.int64)
    n = lib().orc_sample_positions(seed, g, hop, v, deg, k, _ptr(out))
    return [int(x) for x in out[:n]]


# ----------------------------------------------------------------------------
# Graph + minibatch
# ----------------------------------------------------------------------------

@dataclass
class Graph:
    """CSR graph and feature matrix in host memory (numpy)."""

    offsets: np.ndarray  # int32 or int64, N+1
    indices: np.ndarray  # int32, E
    features: np.ndarray | None = None  # any dtype, shape [N, dim]

    def __post_init__(self):
        self.offsets = np.ascontiguousarray(self.offsets)
        if self.offsets.dtype not in (np.int32, np.int64):
            raise OracleError("offsets must be int32 or int64")
        self.indices = np.ascontiguousarray(self.indices, dtype=np.int32)
        if self.features is not None:
            self.features = np.ascontiguousarray(self.features)
        self._struct = _OrcGraph()
        s = self._struct
        s.num_nodes = self.offsets.shape[0] - 1
        s.num_edges = self.indices.shape[0]
        s.offsets = _ptr(self.offsets)
        s.offsets_bits = 32 if self.offsets.dtype == np.int32 else 64
        s.indices = _ptr(self.indices)
        if self.features is not None:
            rows = self.features.reshape(self.features.shape[0], -1)
            s.features = _ptr(self.features)
            s.row_bytes = rows.shape[1] * rows.dtype.itemsize if rows.shape[0] else 0
        else:
            s.features = 0
            s.row_bytes = 0

    @property
    def num_nodes(self) -> int:
        return int(self._struct.num_nodes)

    @property
    def row_bytes(self) -> int:
        return int(self._struct.row_bytes)


def build_adj_blocks(graph: Graph, block_bytes: int):
    """Greedy block packing of adjacency objects; returns (node_block, num_blocks)."""
    nb = ctypes.c_int64(0)
    node_block = np.zeros(max(graph.num_nodes, 1), dtype=np.int32)
    rc = lib().orc_build_adj_blocks(ctypes.byref(graph._struct), block_bytes,
                                    _ptr(node_block), ctypes.byref(nb))
    if rc != 0:
        raise OracleError(f"orc_build_adj_blocks failed ({rc})")
    return node_block[: graph.num_nodes], int(nb.value)


def _copy(ptr, n, dtype):
    if n == 0:
        return np.zeros(0, dtype=dtype)
    ctype = np.ctypeslib.as_ctypes_type(np.dtype(dtype))
    arr = np.ctypeslib.as_array(ctypes.cast(ptr, ctypes.POINTER(ctype)), shape=(n,))
    return arr.copy()


def _to_dict(mb: _OrcMinibatch, row_bytes: int, feat_dtype, feat_shape_tail):
    K = mb.K
    hops = []
    for h in range(K):
        nd, ne = int(mb.num_dst[h]), int(mb.num_edges[h])
        hops.append({
            "num_dst": nd,
            "num_src": int(mb.num_src[h]),
            "num_edges": ne,
            "indptr": _copy(mb.indptr[h], nd + 1, np.int64),
            "nbr": _copy(mb.nbr[h], ne, np.int32),
            "col": _copy(mb.col[h], ne, np.int32),
            "dst": _copy(mb.dst[h], nd, np.int32),
        })
    n = int(mb.num_nodes)
    out = {"hops": hops, "nodes": _copy(mb.nodes, n, np.int32), "num_nodes": n}
    if mb.feats:
        raw = _copy(mb.feats, n * row_bytes, np.uint8)
        out["feats"] = raw.view(feat_dtype).reshape((n,) + feat_shape_tail)
    return out


def _feat_meta(graph: Graph):
    if graph.features is None:
        return np.uint8, ()
    return graph.features.dtype, tuple(graph.features.shape[1:])


def sample_minibatch(graph: Graph, targets, fanouts, seed: int, gid: int, gather: bool = True,
                     frontier: str = "src"):
    """Samples + gathers one minibatch with global id ``gid`` (see module doc).
    ``frontier`` = "src" (dst_{h+1} = src_h) or "sampled" (dst_{h+1} = the
    distinct ids sampled at hop h: Algorithm 1's N_in <- N_out)."""
    t = np.ascontiguousarray(targets, dtype=np.int32)
    f = np.ascontiguousarray(fanouts, dtype=np.int32)
    mb = _OrcMinibatch()
    rc = lib().orc_sample_minibatch_mode(ctypes.byref(graph._struct), _ptr(t), t.shape[0],
                                         _ptr(f), f.shape[0], seed, gid, int(gather),
                                         FRONTIER[frontier], ctypes.byref(mb))
    if rc != 0:
        raise OracleError(f"orc_sample_minibatch failed ({rc})")
    try:
        dt, tail = _feat_meta(graph)
        return _to_dict(mb, graph.row_bytes, dt, tail)
    finally:
        lib().orc_free_minibatch(ctypes.byref(mb))


def hyperbatch(graph: Graph, targets, fanouts, seed: int, first_gid: int, gather: bool,
               adj_block_bytes: int, feat_block_bytes: int, threads: int = 1,
               frontier: str = "src"):
    """Runs every minibatch of a hyperbatch (targets: [H, B]) and the
    blocks-touched statistics.  Returns (list of per-minibatch dicts, stats
    list of K+1 ints).  threads > 1 runs independent minibatches on host
    threads (the C functions are reentrant and ctypes releases the GIL)."""
    t = np.ascontiguousarray(targets, dtype=np.int32)
    H = t.shape[0]
    f = np.ascontiguousarray(fanouts, dtype=np.int32)
    arr = (_OrcMinibatch * H)()
    status = [None] * H

    def run(j):
        status[j] = lib().orc_sample_minibatch_mode(
            ctypes.byref(graph._struct), _ptr(t[j]), t.shape[1], _ptr(f), f.shape[0],
            seed, first_gid + j, int(gather), FRONTIER[frontier], ctypes.byref(arr[j]))

    try:
        if threads > 1:
            import concurrent.futures as cf
            with cf.ThreadPoolExecutor(max_workers=threads) as ex:
                list(ex.map(run, range(H)))
        else:
            for j in range(H):
                run(j)
        for j in range(H):
            if status[j] != 0:
                raise OracleError(f"orc_sample_minibatch failed ({status[j]}) for minibatch {j}")
        rpb = feat_rows_per_block(graph, feat_block_bytes)
        stats = np.zeros(f.shape[0] + 1, dtype=np.int64)
        rc = lib().orc_hyperbatch_stats(ctypes.byref(graph._struct), arr, H, adj_block_bytes,
                                        rpb, _ptr(stats))
        if rc != 0:
            raise OracleError(f"orc_hyperbatch_stats failed ({rc})")
        dt, tail = _feat_meta(graph)
        mbs = [_to_dict(arr[j], graph.row_bytes, dt, tail) for j in range(H)]
        return mbs, [int(x) for x in stats]
    finally:
        for j in range(H):
            if status[j] == 0:
                lib().orc_free_minibatch(ctypes.byref(arr[j]))


def feat_rows_per_block(graph: Graph, feat_block_bytes: int) -> int:
    """Feature rows per feature block (at least one row per block)."""
    rb = graph.row_bytes if graph.row_bytes > 0 else 1
    return max(1, feat_block_bytes // rb)


__all__ = [
    "Graph", "OracleError", "philox4x32_10", "mulhi64", "sample_positions",
    "build_adj_blocks", "sample_minibatch", "hyperbatch", "feat_rows_per_block", "lib",
]

