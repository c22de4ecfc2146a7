"""Python binding of libagnes.so (include/agnes.h): argument marshalling only.

Every step of sampling and gathering runs in the library's CUDA kernels; this
module converts tensors to pointers, calls the C ABI and wraps the returned
device buffers as zero-copy torch tensors.  There is no CPU fallback: if the
shared library is missing or a call fails, an exception is raised.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libagnes.so")
MAX_HOPS = 8
MAX_FANOUT = 1024

F32, F16 = 0, 1
FEATURE_IO = {"blocks": 0, "rows": 1}  # AGNES_FEATURE_IO_* and AGNES_TOPOLOGY_IO_* values
FRONTIER = {"src": 0, "sampled": 1}    # AGNES_FRONTIER_SRC / _SAMPLED
LAUNCH = {"direct": 0, "graph": 1, "graph_pdl": 2}  # AGNES_LAUNCH_DIRECT / _GRAPH / _GRAPH_PDL
_DTYPES = {torch.float32: F32, torch.float16: F16}
_TORCH_OF = {F32: torch.float32, F16: torch.float16}

STATUS = {0: "AGNES_OK", 1: "AGNES_EINVAL", 2: "AGNES_ERANGE", 3: "AGNES_ENOMEM",
          4: "AGNES_ECUDA", 5: "AGNES_ESTATE", 6: "AGNES_ETIMEOUT", 7: "AGNES_EKERNEL"}


class AgnesError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS.get(status, status)}: {message}")
        self.status = status
        self.message = message


class _GraphDesc(ctypes.Structure):
    _fields_ = [
        ("num_nodes", ctypes.c_int64),
        ("num_edges", ctypes.c_int64),
        ("offsets", ctypes.c_void_p),
        ("offsets_bits", ctypes.c_int32),
        ("indices", ctypes.c_void_p),
        ("features", ctypes.c_void_p),
        ("feat_dtype", ctypes.c_int32),
        ("feat_dim", ctypes.c_int64),
        ("features_on_host", ctypes.c_int32),
        ("adj_block_bytes", ctypes.c_int64),
        ("feat_block_bytes", ctypes.c_int64),
        ("topology_on_host", ctypes.c_int32),
        ("graph_buffer_bytes", ctypes.c_int64),
        ("feature_cache_bytes", ctypes.c_int64),
        ("feature_cache_threshold", ctypes.c_int64),
        ("feature_io", ctypes.c_int32),
        ("topology_io", ctypes.c_int32),
    ]


class _View(ctypes.Structure):
    _fields_ = [
        ("K", ctypes.c_int32),
        ("num_dst", ctypes.c_int64 * MAX_HOPS),
        ("num_src", ctypes.c_int64 * MAX_HOPS),
        ("num_edges", ctypes.c_int64 * MAX_HOPS),
        ("indptr", ctypes.c_void_p * MAX_HOPS),
        ("col", ctypes.c_void_p * MAX_HOPS),
        ("nodes", ctypes.c_void_p),
        ("num_nodes", ctypes.c_int64),
        ("feats", ctypes.c_void_p),
        ("feat_dtype", ctypes.c_int32),
        ("feat_dim", ctypes.c_int64),
    ]


class _HyperbatchView(ctypes.Structure):
    _fields_ = [
        ("K", ctypes.c_int32), ("H", ctypes.c_int32),
        ("indptr", ctypes.c_void_p * MAX_HOPS), ("indptr_stride", ctypes.c_int64 * MAX_HOPS),
        ("col", ctypes.c_void_p * MAX_HOPS), ("col_stride", ctypes.c_int64 * MAX_HOPS),
        ("nodes", ctypes.c_void_p), ("nodes_stride", ctypes.c_int64),
        ("feats", ctypes.c_void_p), ("feats_stride_rows", ctypes.c_int64),
        ("feat_dtype", ctypes.c_int32), ("feat_dim", ctypes.c_int64),
        ("node_size", ctypes.c_void_p), ("edges", ctypes.c_void_p),
        ("src_size", ctypes.c_void_p),
    ]


class _Counters(ctypes.Structure):
    _fields_ = [
        ("K", ctypes.c_int32),
        ("frontier", ctypes.c_int64 * MAX_HOPS),
        ("edges", ctypes.c_int64 * MAX_HOPS),
        ("rows", ctypes.c_int64),
        ("distinct_rows", ctypes.c_int64),
        ("row_bytes", ctypes.c_int64),
        ("streamed_bytes", ctypes.c_int64),
        ("streamed_blocks", ctypes.c_int64),
        ("topo_loaded_blocks", ctypes.c_int64),
        ("topo_loaded_bytes", ctypes.c_int64),
        ("topo_hit_blocks", ctypes.c_int64),
        ("topo_waves", ctypes.c_int64),
        ("fcache_hit_blocks", ctypes.c_int64),
        ("fcache_loaded_blocks", ctypes.c_int64),
        ("graph_captures", ctypes.c_int64), ("graph_launches", ctypes.c_int64),
        ("graph_programmatic_edges", ctypes.c_int64),
        ("topo_cached_requests", ctypes.c_int64),
    ]


class _GraphInfo(ctypes.Structure):
    _fields_ = [
        ("num_nodes", ctypes.c_int64), ("num_edges", ctypes.c_int64),
        ("adj_blocks", ctypes.c_int64), ("adj_block_starts", ctypes.c_int64),
        ("feat_blocks", ctypes.c_int64), ("feat_rows_per_block", ctypes.c_int64),
        ("tiles", ctypes.c_int64), ("row_bytes", ctypes.c_int64),
    ]


# Exported entry points and their argument types (mirrors include/agnes.h).
_P = ctypes.c_void_p
SIGNATURES = {
    "agnes_load_graph": ([ctypes.POINTER(_GraphDesc), ctypes.c_int, _P, ctypes.POINTER(_P)],
                         ctypes.c_int),
    "agnes_prepare_hyperbatch": ([_P, _P, ctypes.c_int32, ctypes.c_int32, _P, ctypes.c_int32,
                                  ctypes.c_uint64, ctypes.c_uint64, _P], ctypes.c_int),
    "agnes_fetch_minibatch": ([_P, ctypes.c_int32, ctypes.POINTER(_View)], ctypes.c_int),
    "agnes_fetch_hyperbatch": ([_P, ctypes.POINTER(_HyperbatchView)], ctypes.c_int),
    "agnes_hyperbatch_stats": ([_P, _P], ctypes.c_int),
    "agnes_hyperbatch_counters": ([_P, ctypes.POINTER(_Counters)], ctypes.c_int),
    "agnes_get_graph_info": ([_P, ctypes.POINTER(_GraphInfo)], ctypes.c_int),
    "agnes_copy_adj_blocks": ([_P, _P, _P, ctypes.c_int64], ctypes.c_int),
    "agnes_set_profiling": ([_P, ctypes.c_int32], ctypes.c_int),
    "agnes_phase_times": ([_P, ctypes.c_int32, _P, ctypes.c_int32, ctypes.POINTER(ctypes.c_int32)],
                          ctypes.c_int),
    "agnes_hop_indptr_noalloc": ([_P, _P, ctypes.c_int64, ctypes.c_int32, _P, _P], ctypes.c_int),
    "agnes_set_frontier_mode": ([_P, ctypes.c_int32], ctypes.c_int),
    "agnes_set_launch_mode": ([_P, ctypes.c_int32], ctypes.c_int),
    "agnes_set_pipeline_depth": ([_P, ctypes.c_int32], ctypes.c_int),
    "agnes_wait_hyperbatches": ([_P, _P], ctypes.c_int),
    "agnes_fetch_previous_hyperbatch": ([_P, _P], ctypes.c_int),
    "agnes_fetch_earlier_hyperbatch": ([_P, ctypes.c_int32, _P], ctypes.c_int),
    "agnes_sage_mean_layer": ([_P, ctypes.c_int32, _P, ctypes.c_int32, ctypes.c_int64,
                               ctypes.c_int64, _P, _P, ctypes.c_int32, _P, ctypes.c_int32,
                               ctypes.c_int64, _P], ctypes.c_int),
    "agnes_free": ([_P], ctypes.c_int),
    "agnes_status_string": ([ctypes.c_int], ctypes.c_char_p),
    "agnes_last_error": ([_P], ctypes.c_char_p),
}

_lib = None


def lib() -> ctypes.CDLL:
    """The loaded libagnes.so.  Raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -m paper_2601_01473_gb300.build` (needs nvcc)")
        L = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = res
        _lib = L
    return _lib


def _check(rc: int, ctx=None):
    if rc != 0:
        msg = lib().agnes_last_error(ctx)
        raise AgnesError(rc, msg.decode() if msg else "")


def _stream_handle(stream) -> int | None:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream or None
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream or None
    return int(stream) or None


class _CudaArray:
    """Minimal __cuda_array_interface__ over library-owned device memory."""

    def __init__(self, ptr: int, shape, typestr: str):
        self.__cuda_array_interface__ = {
            "shape": tuple(int(s) for s in shape), "typestr": typestr,
            "data": (int(ptr) if ptr else 0, False), "version": 2, "strides": None,
        }


def _wrap(ptr: int, shape, dtype: torch.dtype, device) -> torch.Tensor:
    n = 1
    for s in shape:
        n *= int(s)
    if n == 0 or not ptr:
        return torch.empty(shape, dtype=dtype, device=device)
    typestr = {torch.int32: "<i4", torch.int64: "<i8", torch.float32: "<f4",
               torch.float16: "<f2"}[dtype]
    return torch.as_tensor(_CudaArray(ptr, shape, typestr), device=device)


@dataclass
class Hop:
    num_dst: int
    num_src: int
    num_edges: int
    indptr: torch.Tensor  # int64 [num_dst + 1], device
    col: torch.Tensor     # int32 [num_edges], device


@dataclass
class MinibatchView:
    hops: list
    nodes: torch.Tensor   # int32 [num_nodes], device (src_K, global ids)
    feats: torch.Tensor   # [num_nodes, feat_dim], device


class HyperbatchView:
    """Every minibatch of a hyperbatch: one zero-copy tensor per output
    buffer ([H, capacity, ...]) plus host size tables; ``view(j)`` slices
    minibatch j out of them."""

    def __init__(self, v: _HyperbatchView, device, tensors=None):
        K, H = v.K, v.H
        self.K, self.H = K, H
        import numpy as np
        sz = np.ctypeslib.as_array(ctypes.cast(v.node_size, ctypes.POINTER(ctypes.c_int32)),
                                   shape=((K + 1) * H,)).reshape(K + 1, H).copy()
        ed = np.ctypeslib.as_array(ctypes.cast(v.edges, ctypes.POINTER(ctypes.c_int32)),
                                   shape=(K * H,)).reshape(K, H).copy()
        ss = np.ctypeslib.as_array(ctypes.cast(v.src_size, ctypes.POINTER(ctypes.c_int32)),
                                   shape=(K * H,)).reshape(K, H).copy()
        self.node_size, self.edges, self.src_size = sz, ed, ss
        if tensors is None:  # wrappers of the ctx's output buffers
            tensors = ([_wrap(v.indptr[h], (H, v.indptr_stride[h]), torch.int64, device)
                        for h in range(K)],
                       [_wrap(v.col[h], (H, v.col_stride[h]), torch.int32, device)
                        for h in range(K)],
                       _wrap(v.nodes, (H, v.nodes_stride), torch.int32, device),
                       _wrap(v.feats, (H, v.feats_stride_rows, v.feat_dim),
                             _TORCH_OF[v.feat_dtype], device))
        self.indptr, self.col, self.nodes, self.feats = tensors
        self._tensors = tensors

    @staticmethod
    def _key(v: _HyperbatchView):
        """What the buffer wrappers depend on: addresses, strides, shapes."""
        K = v.K
        return (K, v.H, v.nodes, v.nodes_stride, v.feats, v.feats_stride_rows, v.feat_dim,
                v.feat_dtype, tuple(v.indptr[h] for h in range(K)),
                tuple(v.indptr_stride[h] for h in range(K)), tuple(v.col[h] for h in range(K)),
                tuple(v.col_stride[h] for h in range(K)))

    def view(self, j: int) -> "MinibatchView":
        hops = []
        for h in range(self.K):
            nd, ns, ne = int(self.node_size[h, j]), int(self.src_size[h, j]), int(self.edges[h, j])
            hops.append(Hop(nd, ns, ne, self.indptr[h][j, :nd + 1], self.col[h][j, :ne]))
        n = int(self.node_size[self.K, j])
        return MinibatchView(hops, self.nodes[j, :n], self.feats[j, :n])


class Graph:
    """A graph loaded into libagnes (one agnes_ctx)."""

    def __init__(self, offsets, indices, features, adj_block_bytes: int = 1 << 20,
                 feat_block_bytes: int | None = None, device: int = 0, stream=None,
                 features_on_host: bool = False, topology_on_host: bool = False,
                 graph_buffer_bytes: int = 0, feature_cache_bytes: int = 0,
                 feature_cache_threshold: int = 0, feature_io: str = "blocks",
                 topology_io: str = "blocks"):
        if offsets.dtype not in (torch.int32, torch.int64):
            raise TypeError("offsets must be int32 or int64")
        if indices.dtype != torch.int32:
            raise TypeError("indices must be int32")
        if features.dtype not in _DTYPES or features.dim() != 2:
            raise TypeError("features must be a 2-D float32 or float16 tensor")
        for name, t in (("offsets", offsets), ("indices", indices), ("features", features)):
            if not t.is_contiguous():
                raise ValueError(f"{name} must be contiguous")
        self._keep = (offsets, indices, features)  # borrowed by the library
        self.device = torch.device("cuda", device)
        self.feat_dtype = features.dtype
        self.feat_dim = features.shape[1]
        d = _GraphDesc()
        d.num_nodes = offsets.numel() - 1
        d.num_edges = indices.numel()
        d.offsets = offsets.data_ptr()
        d.offsets_bits = 32 if offsets.dtype == torch.int32 else 64
        d.indices = indices.data_ptr() if indices.numel() else None
        d.features = features.data_ptr()
        d.feat_dtype = _DTYPES[features.dtype]
        d.feat_dim = features.shape[1]
        d.features_on_host = int(features_on_host)
        d.adj_block_bytes = adj_block_bytes
        d.feat_block_bytes = feat_block_bytes if feat_block_bytes is not None else adj_block_bytes
        d.topology_on_host = int(topology_on_host)
        d.graph_buffer_bytes = graph_buffer_bytes
        d.feature_cache_bytes = feature_cache_bytes
        d.feature_cache_threshold = feature_cache_threshold
        if feature_io not in FEATURE_IO:
            raise ValueError(f"feature_io must be one of {sorted(FEATURE_IO)}")
        d.feature_io = FEATURE_IO[feature_io]
        if topology_io not in FEATURE_IO:
            raise ValueError(f"topology_io must be one of {sorted(FEATURE_IO)}")
        d.topology_io = FEATURE_IO[topology_io]
        ctx = ctypes.c_void_p()
        with torch.cuda.device(self.device):
            rc = lib().agnes_load_graph(ctypes.byref(d), device, _stream_handle(stream),
                                        ctypes.byref(ctx))
        _check(rc, None)
        self._ctx = ctx
        self._H = 0
        self._K = 0

    # -- lifetime --------------------------------------------------------------
    def close(self):
        if getattr(self, "_ctx", None):
            lib().agnes_free(self._ctx)
            self._ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # -- calls -------------------------------------------------------------------
    def prepare(self, targets, fanouts, seed: int, first_minibatch_id: int = 0, stream=None):
        """Enqueues one hyperbatch.  targets: [H, B] int32 (CUDA or CPU tensor)."""
        if targets.dtype != torch.int32 or targets.dim() != 2 or not targets.is_contiguous():
            raise TypeError("targets must be a contiguous [H, B] int32 tensor")
        fan = (ctypes.c_int32 * len(fanouts))(*fanouts)
        H, B = targets.shape
        self._targets = targets  # keep alive until the copy has run
        with torch.cuda.device(self.device):
            rc = lib().agnes_prepare_hyperbatch(self._ctx, targets.data_ptr(), H, B, fan,
                                                len(fanouts), seed & (2**64 - 1),
                                                first_minibatch_id, _stream_handle(stream))
        _check(rc, self._ctx)
        self._H, self._K = H, len(fanouts)

    def fetch(self, j: int) -> MinibatchView:
        v = _View()
        _check(lib().agnes_fetch_minibatch(self._ctx, j, ctypes.byref(v)), self._ctx)
        hops = []
        for h in range(v.K):
            nd, ns, ne = v.num_dst[h], v.num_src[h], v.num_edges[h]
            hops.append(Hop(nd, ns, ne, _wrap(v.indptr[h], (nd + 1,), torch.int64, self.device),
                            _wrap(v.col[h], (ne,), torch.int32, self.device)))
        nodes = _wrap(v.nodes, (v.num_nodes,), torch.int32, self.device)
        feats = _wrap(v.feats, (v.num_nodes, v.feat_dim), _TORCH_OF[v.feat_dtype], self.device)
        return MinibatchView(hops, nodes, feats)

    def fetch_all(self) -> HyperbatchView:
        """All minibatches of the last hyperbatch (one wait, one size read-back).
        The output buffers' tensor wrappers are reused while the ctx's
        workspace stays where it is (same hyperbatch shape)."""
        v = _HyperbatchView()
        _check(lib().agnes_fetch_hyperbatch(self._ctx, ctypes.byref(v)), self._ctx)
        key = HyperbatchView._key(v)
        cached = getattr(self, "_hv_cache", None)
        hv = HyperbatchView(v, self.device, cached[1] if cached and cached[0] == key else None)
        self._hv_cache = (key, hv._tensors)
        return hv

    def set_frontier(self, mode: str) -> None:
        """"src" (dst_{h+1} = src_h, the default) or "sampled" (dst_{h+1} =
        the distinct ids sampled at hop h: Algorithm 1's N_in <- N_out);
        applies from the next prepare."""
        if mode not in FRONTIER:
            raise ValueError(f"frontier must be one of {sorted(FRONTIER)}")
        _check(lib().agnes_set_frontier_mode(self._ctx, FRONTIER[mode]), self._ctx)

    def set_launch_mode(self, mode: str) -> None:
        """How the resident path is issued: "direct" (every kernel launched by
        each prepare), "graph" (captured once per hyperbatch shape, replayed as
        one CUDA graph launch) or "graph_pdl" (the default: the graph with
        programmatic kernel-to-kernel edges); the results are the same."""
        if mode not in LAUNCH:
            raise ValueError(f"launch mode must be one of {sorted(LAUNCH)}")
        _check(lib().agnes_set_launch_mode(self._ctx, LAUNCH[mode]), self._ctx)

    def fetch_previous(self) -> HyperbatchView:
        """At pipeline depth > 1: the hyperbatch prepared before the last one
        (agnes_fetch_previous_hyperbatch)."""
        v = _HyperbatchView()
        _check(lib().agnes_fetch_previous_hyperbatch(self._ctx, ctypes.byref(v)), self._ctx)
        return HyperbatchView(v, self.device)

    def fetch_earlier(self, ago: int) -> HyperbatchView:
        """At pipeline depth d: the hyperbatch prepared ``ago`` prepares
        before the last one, 0 <= ago < d (agnes_fetch_earlier_hyperbatch)."""
        v = _HyperbatchView()
        _check(lib().agnes_fetch_earlier_hyperbatch(self._ctx, int(ago), ctypes.byref(v)),
               self._ctx)
        return HyperbatchView(v, self.device)

    def set_pipeline_depth(self, depth: int) -> None:
        """Hyperbatches in flight (agnes_set_pipeline_depth): 1, or up to
        AGNES_MAX_PIPELINE_DEPTH (4) to let consecutive prepares overlap on
        the ctx's internal streams, one workspace each."""
        _check(lib().agnes_set_pipeline_depth(self._ctx, int(depth)), self._ctx)

    def wait(self, stream=None) -> None:
        """Orders ``stream`` (default: the current stream) after every
        hyperbatch still in flight (agnes_wait_hyperbatches)."""
        _check(lib().agnes_wait_hyperbatches(self._ctx, _stream_handle(stream)), self._ctx)

    def sage_mean_layer(self, hop: int, x: torch.Tensor, w: torch.Tensor, bias=None,
                        out_dtype: torch.dtype = torch.float32, stream=None) -> torch.Tensor:
        """One GraphSAGE-mean layer (agnes_sage_mean_layer) over hop ``hop`` of
        every minibatch of the last hyperbatch.  ``x`` is [H, rows, d_in]
        (minibatch j's src_hop rows first), ``w`` is [d_out, 2 d_in] fp16
        ([W_self | W_neigh]), ``bias`` [d_out] fp32 or None.  Returns
        [H, max |dst_hop|, d_out]; rows past a minibatch's |dst_hop| are
        unspecified."""
        if x.dim() != 3 or x.dtype not in _DTYPES or not x.is_contiguous():
            raise TypeError("x must be a contiguous [H, rows, d_in] float32/float16 tensor")
        if w.dtype != torch.float16 or w.dim() != 2 or not w.is_contiguous():
            raise TypeError("w must be a contiguous [d_out, 2*d_in] float16 tensor")
        if bias is not None and (bias.dtype != torch.float32 or not bias.is_contiguous()):
            raise TypeError("bias must be a contiguous float32 tensor")
        H, rows, d_in = x.shape
        d_out = w.shape[0]
        sizes = self.fetch_all().node_size
        max_dst = int(sizes[hop].max()) if 0 <= hop < sizes.shape[0] - 1 else 0
        out = torch.empty((H, max(max_dst, 1), d_out), dtype=out_dtype, device=x.device)
        _check(lib().agnes_sage_mean_layer(
            self._ctx, hop, x.data_ptr(), _DTYPES[x.dtype], rows, d_in, w.data_ptr(),
            bias.data_ptr() if bias is not None else None, d_out, out.data_ptr(),
            _DTYPES[out_dtype], out.shape[1], _stream_handle(stream)), self._ctx)
        return out

    def sizes(self, j: int) -> dict:
        """Host-side sizes of minibatch j (no device data touched)."""
        v = _View()
        _check(lib().agnes_fetch_minibatch(self._ctx, j, ctypes.byref(v)), self._ctx)
        return {"num_dst": list(v.num_dst[:v.K]), "num_src": list(v.num_src[:v.K]),
                "num_edges": list(v.num_edges[:v.K]), "num_nodes": v.num_nodes}

    def stats(self) -> list:
        out = (ctypes.c_int64 * (self._K + 1))()
        _check(lib().agnes_hyperbatch_stats(self._ctx, out), self._ctx)
        return list(out)

    def counters(self) -> dict:
        c = _Counters()
        _check(lib().agnes_hyperbatch_counters(self._ctx, ctypes.byref(c)), self._ctx)
        return {"frontier": list(c.frontier[:c.K]), "edges": list(c.edges[:c.K]),
                "rows": c.rows, "distinct_rows": c.distinct_rows, "row_bytes": c.row_bytes,
                "streamed_bytes": c.streamed_bytes, "streamed_blocks": c.streamed_blocks,
                "topo_loaded_blocks": c.topo_loaded_blocks, "topo_loaded_bytes": c.topo_loaded_bytes,
                "topo_hit_blocks": c.topo_hit_blocks, "topo_waves": c.topo_waves,
                "fcache_hit_blocks": c.fcache_hit_blocks,
                "fcache_loaded_blocks": c.fcache_loaded_blocks,
                "graph_captures": c.graph_captures, "graph_launches": c.graph_launches,
                "graph_programmatic_edges": c.graph_programmatic_edges,
                "topo_cached_requests": c.topo_cached_requests}

    def info(self) -> dict:
        g = _GraphInfo()
        _check(lib().agnes_get_graph_info(self._ctx, ctypes.byref(g)), self._ctx)
        return {k: getattr(g, k) for k, _ in _GraphInfo._fields_}

    def adj_blocks(self):
        """(start_node, start_block) int32 CPU tensors of the object index table."""
        n = self.info()["adj_block_starts"]
        sn = torch.zeros(max(n, 1), dtype=torch.int32)
        sb = torch.zeros(max(n, 1), dtype=torch.int32)
        _check(lib().agnes_copy_adj_blocks(self._ctx, sn.data_ptr(), sb.data_ptr(), n), self._ctx)
        return sn[:n], sb[:n]

    def set_profiling(self, mode):
        """CUDA-event timing of later prepares: True or "phases" (every phase),
        "gather" (the gather only, two events), False or "off"."""
        if mode is True or mode == "phases":
            m = 1
        elif mode == "gather":
            m = 2
        elif mode is False or mode == "off":
            m = 0
        else:
            raise ValueError("profiling mode must be True/'phases', 'gather' or False/'off'")
        _check(lib().agnes_set_profiling(self._ctx, m), self._ctx)

    def phase_times(self, ago: int = 0) -> list:
        """Per-phase milliseconds of the prepare issued ``ago`` calls before
        the latest (profiling must have been on for it)."""
        buf = (ctypes.c_float * (2 + 3 * MAX_HOPS))()
        n = ctypes.c_int32(0)
        _check(lib().agnes_phase_times(self._ctx, ago, buf, len(buf), ctypes.byref(n)), self._ctx)
        return list(buf[:n.value])
