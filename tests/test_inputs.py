"""The seeded input generators (CPU)."""
import numpy as np
import torch

from agnes_inputs import synth, WORKLOADS


def test_rmat_csr_is_sorted_unique_without_self_loops():
    off, ind = synth.rmat_csr(5000, 8, 0.57, 0.19, 0.19, seed=1)
    off, ind = off.numpy(), ind.numpy()
    assert off[0] == 0 and off[-1] == len(ind)
    assert np.all(np.diff(off) >= 0)
    for v in range(0, 5000, 37):
        row = ind[off[v]:off[v + 1]]
        assert np.all(np.diff(row) > 0)
        assert v not in row
        assert np.all((row >= 0) & (row < 5000))


def test_rmat_is_skewed_toward_low_ids():
    off, _ = synth.rmat_csr(1 << 14, 16, 0.57, 0.19, 0.19, seed=2)
    deg = np.diff(off.numpy())
    assert deg[:64].mean() > 8 * deg.mean()
    assert deg.max() > 50 * np.median(deg[deg > 0])


def test_generators_are_deterministic():
    a = synth.rmat_csr(3000, 6, 0.6, 0.2, 0.15, seed=9)
    b = synth.rmat_csr(3000, 6, 0.6, 0.2, 0.15, seed=9)
    assert torch.equal(a[0], b[0]) and torch.equal(a[1], b[1])
    c = synth.rmat_csr(3000, 6, 0.6, 0.2, 0.15, seed=10)
    assert not torch.equal(a[1][:100], c[1][:100])


def test_features_look_standard_normal():
    f = synth.normal_features(20000, 32, torch.float32, seed=3).numpy()
    assert abs(f.mean()) < 0.01 and abs(f.std() - 1) < 0.01
    h = synth.normal_features(64, 32, torch.float16, seed=3)
    assert h.dtype == torch.float16 and torch.allclose(h.float(), torch.tensor(f[:64]), atol=2e-3)


def test_targets_distinct_within_hyperbatch():
    pool = synth.train_split(100000, 0.05, seed=4)
    assert len(torch.unique(pool)) == len(pool) == 5000
    t = synth.hyperbatch_targets(pool, 4, 1024, 5, 0)
    assert t.shape == (4, 1024) and t.dtype == torch.int32
    assert len(torch.unique(t)) == 4096
    assert set(t.flatten().tolist()) <= set(pool.tolist())
    assert not torch.equal(t, synth.hyperbatch_targets(pool, 4, 1024, 5, 1))


def test_workload_table_matches_the_configs():
    w = WORKLOADS["rmat100m"]
    assert (w.num_nodes, w.H, w.B, w.fanouts, w.feat_dim) == (100_000_000, 128, 1024, (15, 10, 5), 128)
    assert WORKLOADS["rmat100k"].fanouts == (10, 5)
    assert WORKLOADS["rmat65m_skew"].fanouts == (25, 10)
