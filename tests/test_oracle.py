"""Pins for the CPU oracle (no GPU).

Each test checks the oracle against something other than itself: published
known-answer vectors, a library routine (cuRAND's host generator), exact
integer arithmetic, distributional properties of Floyd's algorithm, a
brute-force BFS that the sampler must reduce to at full fanout, a hand-worked
block-packing example, and invariants that any correct result satisfies.
"""
import ctypes
import itertools
import math
import os
import random

import numpy as np
import pytest
import torch

import oracle
from agnes_inputs import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------------------
# Philox4x32-10
# ----------------------------------------------------------------------------

def _kat_rows():
    rows = []
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            vals = [int(x, 16) for x in line.split()]
            rows.append((vals[0:4], vals[4:6], tuple(vals[6:10])))
    return rows


@pytest.mark.parametrize("ctr,key,expect", _kat_rows())
def test_philox_known_answer_vectors(ctr, key, expect):
    assert oracle.philox4x32_10(ctr, key) == expect


def _curand():
    for name in ("libcurand.so", "libcurand.so.10"):
        for d in ("/usr/local/cuda/lib64", "/usr/local/cuda/targets/sbsa-linux/lib", ""):
            try:
                return ctypes.CDLL(os.path.join(d, name) if d else name)
            except OSError:
                continue
    return None


@pytest.mark.parametrize("seed", [0, 1, 0x123456789ABCDEF0, 0xFFFFFFFFFFFFFFFF])
def test_philox_matches_curand_host_generator(seed):
    """cuRAND's host Philox4_32_10 generator emits block i as the Philox of
    counter (0, 0, lo32(i), hi32(i)) under key (lo32(seed), hi32(seed))."""
    L = _curand()
    if L is None:
        pytest.skip("libcurand not available")
    gen = ctypes.c_void_p()
    if L.curandCreateGeneratorHost(ctypes.byref(gen), 161) != 0:  # PHILOX4_32_10
        pytest.skip("curand host generator unavailable")
    try:
        assert L.curandSetPseudoRandomGeneratorSeed(gen, ctypes.c_ulonglong(seed)) == 0
        n = 4 * 64
        out = np.zeros(n, dtype=np.uint32)
        assert L.curandGenerate(gen, out.ctypes.data_as(ctypes.c_void_p), ctypes.c_size_t(n)) == 0
    finally:
        L.curandDestroyGenerator(gen)
    key = [seed & 0xFFFFFFFF, seed >> 32]
    for i in range(64):
        assert oracle.philox4x32_10([0, 0, i, 0], key) == tuple(int(x) for x in out[4 * i:4 * i + 4])


def test_mulhi64_exact():
    rng = random.Random(7)
    cases = [(0, 0), (1, 1), (2**64 - 1, 2**64 - 1), (2**64 - 1, 1), (2**63, 2), (2**32, 2**32)]
    cases += [(rng.getrandbits(64), rng.getrandbits(64)) for _ in range(2000)]
    cases += [(rng.getrandbits(64), rng.randrange(1, 1 << 20)) for _ in range(2000)]
    for a, b in cases:
        assert oracle.mulhi64(a, b) == (a * b) >> 64


def test_range_reduction_is_uniform_over_small_ranges():
    """t = floor(r * m / 2^64) over Philox outputs is uniform on [0, m)."""
    from scipy.stats import chisquare
    m = 7
    counts = [0] * m
    key = [12345, 0]
    for i in range(20000):
        x = oracle.philox4x32_10([i, 0, 0, 0], key)
        r = (x[1] << 32) | x[0]
        counts[oracle.mulhi64(r, m)] += 1
    assert chisquare(counts).pvalue > 1e-4


# ----------------------------------------------------------------------------
# Floyd sampling of positions
# ----------------------------------------------------------------------------

def test_degree_at_most_fanout_takes_all_in_order():
    for deg in range(0, 12):
        for k in (deg, deg + 1, 25):
            if k < 1:
                continue
            assert oracle.sample_positions(3, 9, 1, 42, deg, k) == list(range(deg))


def test_positions_distinct_and_in_range():
    rng = random.Random(1)
    for _ in range(3000):
        deg = rng.randrange(2, 400)
        k = rng.randrange(1, deg)
        pos = oracle.sample_positions(rng.getrandbits(64), rng.getrandbits(64),
                                      rng.randrange(1, 9), rng.randrange(0, 1 << 31), deg, k)
        assert len(pos) == k
        assert len(set(pos)) == k
        assert all(0 <= p < deg for p in pos)


@pytest.mark.parametrize("deg,k", [(5, 2), (6, 3), (8, 4), (7, 1), (4, 3)])
def test_floyd_subsets_are_uniform(deg, k):
    """Every k-subset of the deg positions is equally likely (Floyd 1987)."""
    from scipy.stats import chisquare
    subsets = {s: i for i, s in enumerate(itertools.combinations(range(deg), k))}
    counts = [0] * len(subsets)
    trials = 400 * len(subsets)
    for v in range(trials):
        pos = oracle.sample_positions(99, 5, 2, v, deg, k)
        counts[subsets[tuple(sorted(pos))]] += 1
    assert chisquare(counts).pvalue > 1e-4


def test_inclusion_probability_is_k_over_deg():
    deg, k, trials = 40, 10, 20000
    hits = np.zeros(deg)
    for g in range(trials):
        for p in oracle.sample_positions(11, g, 3, 17, deg, k):
            hits[p] += 1
    expect = trials * k / deg
    sd = math.sqrt(trials * (k / deg) * (1 - k / deg))
    assert np.all(np.abs(hits - expect) < 5 * sd)


def test_draws_depend_on_every_key_field():
    base = oracle.sample_positions(1, 2, 3, 4, 1000, 8)
    assert oracle.sample_positions(1, 2, 3, 4, 1000, 8) == base
    for args in [(9, 2, 3, 4), (1, 9, 3, 4), (1, 2, 4, 4), (1, 2, 3, 9),
                 (1 << 40, 2, 3, 4), (1, 2 << 40, 3, 4)]:
        assert oracle.sample_positions(*args, 1000, 8) != base


# ----------------------------------------------------------------------------
# Block packing
# ----------------------------------------------------------------------------

def _read_kv(path):
    out = {}
    with open(path) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, *v = line.split()
                out[k] = [int(x) for x in v]
    return out


def _graph_from_degrees(degrees, bits=64, rng=None):
    offsets = np.zeros(len(degrees) + 1, dtype=np.int64)
    offsets[1:] = np.cumsum(degrees)
    n = len(degrees)
    rng = rng or np.random.default_rng(0)
    indices = np.concatenate([np.sort(rng.choice(max(n, d + 1), size=d, replace=False))
                              for d in degrees] or [np.zeros(0)]).astype(np.int32)
    indices = np.minimum(indices, max(n - 1, 0)).astype(np.int32)
    off = offsets.astype(np.int32 if bits == 32 else np.int64)
    return oracle.Graph(off, indices)


def test_block_packing_hand_worked_example():
    kv = _read_kv(os.path.join(GOLDEN, "block_packing_example.txt"))
    g = _graph_from_degrees(kv["degrees"], bits=kv["offsets_bits"][0])
    nb, n = oracle.build_adj_blocks(g, kv["block_bytes"][0])
    assert list(nb) == kv["node_block"]
    assert n == kv["num_blocks"][0]


def _check_packing(degrees, hdr, bb, node_block, num_blocks):
    """Properties that characterise greedy in-order packing."""
    sizes = [hdr + 4 * d for d in degrees]
    used = {}
    for v, s in enumerate(sizes):
        b = node_block[v]
        if v > 0:
            assert b >= node_block[v - 1]
        if s > bb:
            span = -(-s // bb)
            if v > 0:
                assert b > node_block[v - 1]  # starts a fresh block
            if v + 1 < len(sizes):
                assert node_block[v + 1] == b + span  # next object after its blocks
            else:
                assert num_blocks == b + span
            continue
        used[b] = used.get(b, 0) + s
        assert used[b] <= bb
        if v > 0 and b != node_block[v - 1] and sizes[v - 1] <= bb:
            # greedy: v did not fit in the rest of the previous block
            prev = node_block[v - 1]
            assert b == prev + 1
            assert sum(sizes[u] for u in range(v) if node_block[u] == prev) + s > bb
    if sizes and sizes[-1] <= bb:
        assert num_blocks == node_block[-1] + 1


@pytest.mark.parametrize("bits", [32, 64])
@pytest.mark.parametrize("bb", [16, 64, 100, 4096])
def test_block_packing_properties(bits, bb):
    rng = np.random.default_rng(bb + bits)
    degrees = list(rng.integers(0, 6, size=200))
    degrees[7] = 60   # big objects in the middle,
    degrees[8] = 70   # back to back,
    degrees[-1] = 90  # and at the end
    g = _graph_from_degrees(degrees, bits=bits)
    node_block, num_blocks = oracle.build_adj_blocks(g, bb)
    _check_packing(degrees, bits // 8, bb, list(node_block), num_blocks)


# ----------------------------------------------------------------------------
# Whole minibatch
# ----------------------------------------------------------------------------

def _random_graph(n, max_deg, seed, bits=64, row=8, dtype=np.float32):
    rng = np.random.default_rng(seed)
    degrees = rng.integers(0, max_deg + 1, size=n)
    rows = [np.sort(rng.choice(n, size=min(d, n), replace=False)) for d in degrees]
    degrees = np.array([len(r) for r in rows])
    offsets = np.zeros(n + 1, dtype=np.int64)
    offsets[1:] = np.cumsum(degrees)
    indices = np.concatenate(rows).astype(np.int32) if len(rows) else np.zeros(0, np.int32)
    feats = rng.standard_normal((n, row)).astype(dtype)
    return oracle.Graph(offsets.astype(np.int32 if bits == 32 else np.int64), indices, feats)


def _bfs_expansion(g, targets, K):
    """K-hop full-neighbourhood expansion with Python sets (brute force)."""
    off, idx = g.offsets.astype(np.int64), g.indices
    nodes = list(int(t) for t in targets)
    hops = []
    for _ in range(K):
        dst = list(nodes)
        nbr = []
        for v in dst:
            nbr.extend(int(u) for u in idx[off[v]:off[v + 1]])
        new = sorted(set(nbr) - set(dst))
        src = dst + new
        where = {u: i for i, u in enumerate(src)}
        hops.append((len(dst), nbr, [where[u] for u in nbr]))
        nodes = src
    return nodes, hops


@pytest.mark.parametrize("seed", range(6))
def test_full_fanout_equals_bfs(seed):
    g = _random_graph(48, 5, seed)
    rng = np.random.default_rng(100 + seed)
    targets = rng.choice(48, size=5, replace=False)
    K = 3
    got = oracle.sample_minibatch(g, targets, [8] * K, seed=seed, gid=seed)
    nodes, hops = _bfs_expansion(g, targets, K)
    assert list(got["nodes"]) == nodes
    for h, (nd, nbr, col) in enumerate(hops):
        assert got["hops"][h]["num_dst"] == nd
        assert list(got["hops"][h]["nbr"]) == nbr
        assert list(got["hops"][h]["col"]) == col
    np.testing.assert_array_equal(got["feats"], g.features[nodes])


def _check_minibatch_invariants(g, targets, fanouts, mb):
    off, idx = g.offsets.astype(np.int64), g.indices
    nodes = mb["nodes"]
    assert list(nodes[: len(targets)]) == list(targets)
    prev_src = len(targets)
    for h, hop in enumerate(mb["hops"]):
        k = fanouts[h]
        nd = hop["num_dst"]
        assert nd == prev_src
        dst = nodes[:nd]
        ip = hop["indptr"]
        assert ip[0] == 0 and len(ip) == nd + 1
        for i, v in enumerate(dst):
            deg = off[v + 1] - off[v]
            row = idx[off[v]:off[v + 1]]
            got = hop["nbr"][ip[i]:ip[i + 1]]
            assert len(got) == min(deg, k)
            if deg <= k:
                assert list(got) == list(row)
            else:
                assert len(set(got.tolist())) == k
                assert set(got.tolist()) <= set(row.tolist())
        ns = hop["num_src"]
        src = nodes[:ns]
        new = src[nd:]
        assert np.all(np.diff(new) > 0)
        assert not (set(new.tolist()) & set(dst.tolist()))
        assert set(hop["nbr"].tolist()) <= set(src.tolist())
        assert set(new.tolist()) <= set(hop["nbr"].tolist())
        assert np.all(hop["col"] < ns)
        np.testing.assert_array_equal(src[hop["col"]], hop["nbr"])
        prev_src = ns
    assert mb["num_nodes"] == prev_src
    np.testing.assert_array_equal(mb["feats"], g.features[nodes])


@pytest.mark.parametrize("bits", [32, 64])
def test_invariants_on_rmat(bits):
    off, ind = synth.rmat_csr(4096, 12, 0.57, 0.19, 0.19, seed=3,
                              offsets_dtype=torch.int32 if bits == 32 else torch.int64)
    feats = synth.normal_features(4096, 16, torch.float16, seed=3)
    g = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    targets = synth.permutation(4096, 5)[:64].numpy().astype(np.int32)
    fanouts = [6, 4, 3]
    mb = oracle.sample_minibatch(g, targets, fanouts, seed=77, gid=12)
    _check_minibatch_invariants(g, targets, fanouts, mb)


def test_samples_of_a_node_do_not_depend_on_the_rest_of_the_frontier():
    g = _random_graph(300, 40, 4)
    deg = np.diff(g.offsets)
    v = int(np.argmax(deg))
    alone = oracle.sample_minibatch(g, [v], [5], seed=1, gid=3)
    others = [u for u in range(300) if u != v][:20]
    mixed = oracle.sample_minibatch(g, others[:10] + [v] + others[10:], [5], seed=1, gid=3)
    ip = mixed["hops"][0]["indptr"]
    assert list(mixed["hops"][0]["nbr"][ip[10]:ip[11]]) == list(alone["hops"][0]["nbr"])
    other_g = oracle.sample_minibatch(g, [v], [5], seed=1, gid=4)
    assert list(other_g["hops"][0]["nbr"]) != list(alone["hops"][0]["nbr"])


def test_invalid_inputs_are_rejected():
    g = _random_graph(20, 3, 0)
    with pytest.raises(oracle.OracleError):
        oracle.sample_minibatch(g, [1, 2, 1], [2], 0, 0)
    with pytest.raises(oracle.OracleError):
        oracle.sample_minibatch(g, [1, 20], [2], 0, 0)
    with pytest.raises(oracle.OracleError):
        oracle.sample_minibatch(g, [1], [], 0, 0)
    with pytest.raises(oracle.OracleError):
        oracle.sample_minibatch(g, [1], [0], 0, 0)


def test_hyperbatch_stats_are_distinct_blocks_of_frontiers():
    g = _random_graph(500, 12, 9, row=32)
    rng = np.random.default_rng(1)
    H, B, fan = 4, 8, [4, 3]
    targets = rng.choice(500, size=(H, B), replace=True)
    for j in range(H):
        targets[j] = rng.choice(500, size=B, replace=False)
    adj_bb, feat_bb = 256, 1024
    mbs, stats = oracle.hyperbatch(g, targets, fan, 5, 10, True, adj_bb, feat_bb)
    node_block, _ = oracle.build_adj_blocks(g, adj_bb)
    rpb = oracle.feat_rows_per_block(g, feat_bb)
    for h in range(len(fan)):
        blocks = set()
        for mb in mbs:
            blocks |= {int(node_block[v]) for v in mb["nodes"][: mb["hops"][h]["num_dst"]]}
        assert stats[h] == len(blocks)
    fb = set()
    for mb in mbs:
        fb |= {int(v) // rpb for v in mb["nodes"]}
    assert stats[-1] == len(fb)
    # one minibatch never touches more blocks than the hyperbatch
    _, one = oracle.hyperbatch(g, targets[:1], fan, 5, 10, False, adj_bb, feat_bb)
    assert all(a <= b for a, b in zip(one, stats))
    # minibatch ids, not hyperbatch positions, key the draws
    solo = oracle.sample_minibatch(g, targets[2], fan, 5, 12)
    np.testing.assert_array_equal(solo["nodes"], mbs[2]["nodes"])


def test_golden_fixture_is_reproduced():
    """Regression pin: tests/golden/oracle_tiny.json (written by
    tests/golden/make_golden.py from the oracle) is reproduced exactly."""
    import json
    with open(os.path.join(GOLDEN, "oracle_tiny.json")) as f:
        d = json.load(f)
    g = oracle.Graph(np.array(d["offsets"], np.int32), np.array(d["indices"], np.int32),
                     np.array(d["features"], np.float32))
    mbs, stats = oracle.hyperbatch(g, np.array(d["targets"], np.int32), d["fanouts"], d["seed"],
                                   d["first_gid"], True, d["adj_block_bytes"],
                                   d["feat_block_bytes"])
    assert stats == d["stats"]
    for mb, ref in zip(mbs, d["minibatches"]):
        assert mb["nodes"].tolist() == ref["nodes"]
        for hop, rh in zip(mb["hops"], ref["hops"]):
            assert hop["num_dst"] == rh["num_dst"]
            assert hop["indptr"].tolist() == rh["indptr"]
            assert hop["col"].tolist() == rh["col"]
