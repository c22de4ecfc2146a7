"""Seeded synthetic inputs: RMAT graphs in CSR form, N(0,1) features, train
splits and hyperbatch targets.

This module feeds both the CUDA path and the oracle, so it holds none of the
method's arithmetic: no Philox, no neighbour sampling, no blocks.  Its
randomness is a 32-bit integer mixing hash evaluated with plain torch integer
ops, so a given (seed, sizes) produces the same bytes on the CPU and on a GPU;
small cases are built on the CPU, full-size ones on the GPU.

RMAT (Chakrabarti, Zhan, Faloutsos, SDM'04): each edge descends ``scale``
levels of the adjacency matrix, picking quadrant (0,0), (0,1), (1,0), (1,1)
with probabilities a, b, c, 1-a-b-c.  Endpoints >= N are redrawn with a fresh
hash stream, duplicate edges and self-loops are dropped, and the CSR rows
are the out-neighbour lists in ascending id.
"""
from __future__ import annotations

import math
from statistics import NormalDist

import torch

M32 = 0xFFFFFFFF
_GOLD = 0x9E3779B1


def _mix32(x: torch.Tensor) -> torch.Tensor:
    """Integer avalanche of 32-bit values held in int64 (no overflow)."""
    x = (((x >> 16) ^ x) * 0x45D9F3B) & M32
    x = (((x >> 16) ^ x) * 0x45D9F3B) & M32
    return (x >> 16) ^ x


def _salt(*parts: int) -> int:
    """Python-side hash of a tuple of ints into 32 bits (same mixing)."""
    h = 0x2545F491
    for p in parts:
        for word in (p & M32, (p >> 32) & M32):
            h ^= word
            h = (((h >> 16) ^ h) * 0x45D9F3B) & M32
            h = (((h >> 16) ^ h) * 0x45D9F3B) & M32
            h = (h >> 16) ^ h
    return h


def hash32(idx: torch.Tensor, *salt: int) -> torch.Tensor:
    """Uniform 32-bit values (int64 tensor) for counters 0 <= idx < 2**62.
    The counter is split into 31-bit pieces so no product overflows int64."""
    s = _salt(*salt)
    lo = idx & 0x7FFFFFFF
    hi = idx >> 31
    x = _mix32((lo * _GOLD + s) & M32)
    return _mix32(x ^ ((hi * 0x85EBCA77 + (s ^ 0x5BD1E995)) & M32))


# ----------------------------------------------------------------------------
# RMAT edges
# ----------------------------------------------------------------------------

def _rmat_pairs(idx: torch.Tensor, scale: int, thr, seed: int, attempt: int):
    """src, dst (int64) of the RMAT edges with counters idx for one draw
    attempt.  Each 32-bit hash supplies two 16-bit quadrant draws."""
    t_a, t_ab, t_abc = thr
    src = torch.zeros_like(idx)
    dst = torch.zeros_like(idx)
    for lvl in range(0, scale, 2):
        h = hash32(idx, seed, attempt, lvl, 0x524D4154)
        for half in range(2):
            if lvl + half >= scale:
                break
            u = (h >> (16 * half)) & 0xFFFF
            sbit = (u >= t_ab).to(torch.int64)
            dbit = (((u >= t_a) & (u < t_ab)) | (u >= t_abc)).to(torch.int64)
            src = (src << 1) | sbit
            dst = (dst << 1) | dbit
    return src, dst


def rmat_edges(num_nodes: int, num_edges: int, a: float, b: float, c: float, seed: int,
               device="cpu", chunk: int = 1 << 26) -> torch.Tensor:
    """Sorted unique edge keys src * N + dst (int64) of an RMAT graph without
    self-loops.  ``num_edges`` raw edges are drawn before dedup; an edge with
    an endpoint >= N is redrawn (same edge counter, next attempt)."""
    if not (0 < a and 0 <= b and 0 <= c and a + b + c < 1):
        raise ValueError("RMAT probabilities must satisfy a > 0, b, c >= 0, a+b+c < 1")
    if num_nodes >= 1 << 31:
        raise ValueError("node ids must fit in int32")
    scale = max(1, math.ceil(math.log2(max(num_nodes, 2))))
    thr = (round(a * 65536), round((a + b) * 65536), round((a + b + c) * 65536))
    keys = []
    for first in range(0, num_edges, chunk):
        idx = torch.arange(first, min(num_edges, first + chunk), dtype=torch.int64, device=device)
        src, dst = _rmat_pairs(idx, scale, thr, seed, 0)
        bad = (src >= num_nodes) | (dst >= num_nodes)
        attempt = 1
        while bool(bad.any()):
            ids = torch.nonzero(bad).flatten()
            s2, d2 = _rmat_pairs(idx[ids], scale, thr, seed, attempt)
            src[ids] = s2
            dst[ids] = d2
            bad = (src >= num_nodes) | (dst >= num_nodes)
            attempt += 1
            if attempt > 256:
                raise RuntimeError("RMAT redraw did not converge")
        keep = src != dst
        keys.append(src[keep] * num_nodes + dst[keep])
        del src, dst, bad, keep, idx
    key = torch.cat(keys) if keys else torch.zeros(0, dtype=torch.int64, device=device)
    del keys
    return torch.unique(key, sorted=True)


def csr_from_keys(keys: torch.Tensor, num_nodes: int, offsets_dtype=torch.int64):
    """CSR (offsets, indices int32) from sorted unique keys src * N + dst."""
    src = torch.div(keys, num_nodes, rounding_mode="floor")
    indices = (keys - src * num_nodes).to(torch.int32)
    counts = torch.bincount(src, minlength=num_nodes)
    del src
    offsets = torch.zeros(num_nodes + 1, dtype=torch.int64, device=keys.device)
    torch.cumsum(counts, 0, out=offsets[1:])
    if offsets_dtype == torch.int32:
        if int(offsets[-1]) >= 1 << 31:
            raise ValueError("too many edges for int32 offsets")
        offsets = offsets.to(torch.int32)
    return offsets, indices


def rmat_csr(num_nodes: int, avg_degree: float, a: float, b: float, c: float, seed: int,
             device="cpu", offsets_dtype=torch.int64):
    """RMAT graph with ``avg_degree * num_nodes`` raw edges, as CSR."""
    keys = rmat_edges(num_nodes, int(avg_degree * num_nodes), a, b, c, seed, device)
    out = csr_from_keys(keys, num_nodes, offsets_dtype)
    del keys
    return out


# ----------------------------------------------------------------------------
# Features, splits, targets
# ----------------------------------------------------------------------------

_NORMAL_TABLE: dict = {}


def _normal_table(device) -> torch.Tensor:
    """N(0,1) quantiles at the 65536 midpoints (u + 1/2) / 65536, float32."""
    key = str(device)
    if key not in _NORMAL_TABLE:
        nd = NormalDist()
        vals = [nd.inv_cdf((u + 0.5) / 65536.0) for u in range(65536)]
        _NORMAL_TABLE[key] = torch.tensor(vals, dtype=torch.float64).to(torch.float32).to(device)
    return _NORMAL_TABLE[key]


def normal_features(num_nodes: int, dim: int, dtype, seed: int, device="cpu",
                    chunk_rows: int = 1 << 20) -> torch.Tensor:
    """[N, dim] features ~ N(0,1) (inverse-CDF of 16-bit uniforms), as dtype."""
    table = _normal_table(device)
    out = torch.empty((num_nodes, dim), dtype=dtype, device=device)
    half = (dim + 1) // 2
    for r0 in range(0, num_nodes, chunk_rows):
        r1 = min(num_nodes, r0 + chunk_rows)
        rows = torch.arange(r0, r1, dtype=torch.int64, device=device)
        ctr = (rows[:, None] * half + torch.arange(half, dtype=torch.int64, device=device))
        ctr = ctr.flatten()
        h = hash32(ctr, seed, 0x46454154)
        u = torch.stack([h & 0xFFFF, h >> 16], dim=1).view(r1 - r0, 2 * half)[:, :dim]
        out[r0:r1] = table[u].to(dtype)
    return out


def permutation(n: int, seed: int, device="cpu") -> torch.Tensor:
    """A seeded permutation of [0, n) (int64), by sorting hashed keys."""
    ids = torch.arange(n, dtype=torch.int64, device=device)
    key = (hash32(ids, seed, 0x5045524D) << 31) | ids
    return torch.argsort(key)


def train_split(num_nodes: int, frac: float, seed: int, device="cpu") -> torch.Tensor:
    """A seeded random subset of round(frac * N) node ids (int32)."""
    n = max(1, round(frac * num_nodes))
    return permutation(num_nodes, seed, device)[:n].to(torch.int32)


def hyperbatch_targets(pool: torch.Tensor, H: int, B: int, seed: int, step: int) -> torch.Tensor:
    """[H, B] int32 targets: the first H*B ids of a seeded permutation of
    ``pool`` (distinct within the hyperbatch), one row per minibatch."""
    if H * B > pool.numel():
        raise ValueError(f"pool of {pool.numel()} ids cannot supply {H}x{B} distinct targets")
    perm = permutation(pool.numel(), _salt(seed, step, 0x54475453), pool.device)
    return pool[perm[: H * B]].view(H, B).to(torch.int32).contiguous()
