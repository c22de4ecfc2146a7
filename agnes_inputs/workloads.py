"""The synthetic workloads: RMAT graphs shaped like the paper's datasets
(Table 3: PA ~111M nodes / 1.62B edges; FR 68M nodes / 2.29B edges, heavily
skewed) with the sampling setup of Sec. 4.1 (block 1 MB, fanouts per hop,
minibatches of ~1000 targets, hyperbatches of many minibatches).

Every input is seeded and synthetic; these graphs stand in for the paper's
datasets, which are not used.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace

import torch

from . import synth


@dataclass(frozen=True)
class Workload:
    name: str
    num_nodes: int
    raw_degree: float          # RMAT edges drawn per node (before dedup / self-loop removal)
    a: float
    b: float
    c: float
    offsets_dtype: str         # "int32" | "int64"
    feat_dtype: str            # "float32" | "float16"
    feat_dim: int
    adj_block_bytes: int
    feat_block_bytes: int
    H: int                     # minibatches per hyperbatch
    B: int                     # targets per minibatch
    fanouts: tuple = field(default_factory=tuple)
    train_frac: float | None = None   # targets drawn from a random split of this size
    seed: int = 0

    def describe(self) -> str:
        return (f"RMAT(a={self.a},b={self.b},c={self.c}) N={self.num_nodes} "
                f"raw_deg={self.raw_degree} off={self.offsets_dtype} "
                f"feat={self.feat_dtype}x{self.feat_dim} block={self.adj_block_bytes}B "
                f"H={self.H}xB={self.B} fanouts={list(self.fanouts)}"
                + (f" train={self.train_frac}" if self.train_frac else ""))

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


KB, MB = 1024, 1024 * 1024

WORKLOADS = {
    # 100K-node RMAT, int32 CSR, fp32 x128, 64 KB blocks, 8 x 1024 targets, [10, 5]
    "rmat100k": Workload("rmat100k", 100_000, 16, 0.57, 0.19, 0.19, "int32", "float32", 128,
                         64 * KB, 64 * KB, 8, 1024, (10, 5), None, 0),
    # 10M-node RMAT, avg degree 20, int64 offsets, fp32 x128, 1 MB blocks, 64 x 1024, [15,10,5]
    "rmat10m": Workload("rmat10m", 10_000_000, 20, 0.57, 0.19, 0.19, "int64", "float32", 128,
                        MB, MB, 64, 1024, (15, 10, 5), None, 0),
    # 100M-node RMAT, ~1.6B edges, fp16 x128, 1 MB blocks, 128 x 1024 targets from a 1% train
    # split, [15,10,5]: shaped like ogbn-papers100M (PA)
    "rmat100m": Workload("rmat100m", 100_000_000, 16, 0.57, 0.19, 0.19, "int64", "float16", 128,
                         MB, MB, 128, 1024, (15, 10, 5), 0.01, 0),
    # skewed social-like RMAT, 65M nodes, ~1.8B edges, max degree > 1M, fp16 x256, [25,10]:
    # shaped like com-friendster (FR)
    "rmat65m_skew": Workload("rmat65m_skew", 65_000_000, 28, 0.6, 0.2, 0.15, "int64", "float16",
                             256, MB, MB, 64, 1024, (25, 10), None, 0),
    # small stand-ins with the same structure, for parity tests the oracle finishes in seconds
    "mini100m": Workload("mini100m", 2_000_000, 16, 0.57, 0.19, 0.19, "int64", "float16", 128,
                         MB, MB, 16, 1024, (15, 10, 5), 0.05, 1),
    # profiling stand-in for rmat100m: same cell density per (tile, minibatch) at hop 3
    # (~6 entries) with ~4 GB on the device
    "prof5m": Workload("prof5m", 5_000_000, 16, 0.57, 0.19, 0.19, "int64", "float16", 128,
                       MB, MB, 128, 64, (15, 10, 5), 0.05, 3),
    # profiling stand-in for the dedup kernels: rmat100m's hop-3 cell density (~5 entries per
    # (tile, minibatch) cell) over 1.5M cells, 16-wide features, a few GB on the device
    "prof_cells": Workload("prof_cells", 10_000_000, 16, 0.57, 0.19, 0.19, "int64", "float16", 16,
                           MB, MB, 512, 100, (15, 10, 5), 0.05, 4),
    "mini_skew": Workload("mini_skew", 1_000_000, 28, 0.6, 0.2, 0.15, "int64", "float16", 256,
                          MB, MB, 8, 1024, (25, 10), None, 2),
}


def _torch_dtype(name: str):
    return {"int32": torch.int32, "int64": torch.int64, "float32": torch.float32,
            "float16": torch.float16}[name]


def build_graph(w: Workload, device="cpu"):
    """(offsets, indices, features) of the workload's graph on ``device``."""
    offsets, indices = synth.rmat_csr(w.num_nodes, w.raw_degree, w.a, w.b, w.c, w.seed,
                                      device=device, offsets_dtype=_torch_dtype(w.offsets_dtype))
    features = synth.normal_features(w.num_nodes, w.feat_dim, _torch_dtype(w.feat_dtype),
                                     w.seed + 1, device=device)
    return offsets, indices, features


def target_pool(w: Workload, device="cpu") -> torch.Tensor:
    """Node ids targets are drawn from (a random train split, or every node)."""
    if w.train_frac:
        return synth.train_split(w.num_nodes, w.train_frac, w.seed + 2, device)
    return torch.arange(w.num_nodes, dtype=torch.int32, device=device)


def build_workload(w: Workload, device="cpu"):
    offsets, indices, features = build_graph(w, device)
    return {"offsets": offsets, "indices": indices, "features": features,
            "pool": target_pool(w, device)}


def targets_for_step(w: Workload, pool: torch.Tensor, step: int) -> torch.Tensor:
    """[H, B] int32 targets of hyperbatch ``step`` (distinct within it)."""
    return synth.hyperbatch_targets(pool, w.H, w.B, w.seed + 3, step)
