"""Seeded synthetic workloads shared by the CUDA path's tests/bench and the
oracle.  Holds input generation only (see synth.py), never the method."""
from .synth import (csr_from_keys, hash32, hyperbatch_targets, normal_features, permutation,
                    rmat_csr, rmat_edges, train_split)
from .workloads import WORKLOADS, Workload, build_graph, build_workload, target_pool, targets_for_step

__all__ = ["csr_from_keys", "hash32", "hyperbatch_targets", "normal_features", "permutation",
           "rmat_csr", "rmat_edges", "train_split", "WORKLOADS", "Workload", "build_graph",
           "build_workload", "target_pool", "targets_for_step"]
