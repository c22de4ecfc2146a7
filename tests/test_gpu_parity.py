"""Parity of the CUDA path (through the C ABI) with the oracle: bit-exact
sampled subgraphs, relabelled edges, node lists, gathered feature bytes and
blocks-touched statistics, on small seeded inputs that span many tiles and
blocks, plus edge cases and error reporting."""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from agnes_inputs import WORKLOADS, build_workload, synth, targets_for_step
from paper_2601_01473_gb300 import AgnesError, Graph

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _bytes(t: torch.Tensor) -> np.ndarray:
    t = t.detach().cpu().contiguous()
    return t.view(torch.uint8).numpy().reshape(-1) if t.numel() else np.zeros(0, np.uint8)


def compare(g: Graph, og: oracle.Graph, targets: np.ndarray, fanouts, seed, gid0, adj_bb, feat_bb,
            check_stats=True, only=None, frontier="src"):
    """Compares every (or the listed) minibatch of g's last hyperbatch with
    the oracle."""
    H = targets.shape[0]
    js = range(H) if only is None else only
    if check_stats:
        ref, ref_stats = oracle.hyperbatch(og, targets, fanouts, seed, gid0, True, adj_bb, feat_bb,
                                           frontier=frontier)
        assert g.stats() == ref_stats
    else:
        ref = {j: oracle.sample_minibatch(og, targets[j], fanouts, seed, gid0 + j,
                                          frontier=frontier) for j in js}
    for j in js:
        v, r = g.fetch(j), ref[j]
        assert np.array_equal(v.nodes.cpu().numpy(), r["nodes"]), f"nodes of minibatch {j}"
        for h in range(len(fanouts)):
            hv, hr = v.hops[h], r["hops"][h]
            assert (hv.num_dst, hv.num_src, hv.num_edges) == (
                hr["num_dst"], hr["num_src"], hr["num_edges"]), f"sizes of hop {h}, mb {j}"
            assert np.array_equal(hv.indptr.cpu().numpy(), hr["indptr"]), f"indptr {h} mb {j}"
            assert np.array_equal(hv.col.cpu().numpy(), hr["col"]), f"col {h} mb {j}"
        assert np.array_equal(_bytes(v.feats), r["feats"].view(np.uint8).reshape(-1)
                              if r["feats"].size else np.zeros(0, np.uint8)), f"feats mb {j}"


def make(n, deg, a=0.57, b=0.19, c=0.19, seed=0, bits=64, dtype=torch.float16, dim=64):
    off, ind = synth.rmat_csr(n, deg, a, b, c, seed,
                              offsets_dtype=torch.int32 if bits == 32 else torch.int64)
    feats = synth.normal_features(n, dim, dtype, seed + 100)
    return off, ind, feats


def load(off, ind, feats, adj_bb, feat_bb):
    dev = torch.device("cuda:0")
    return Graph(off.to(dev), ind.to(dev), feats.to(dev), adj_block_bytes=adj_bb,
                 feat_block_bytes=feat_bb)


def test_golden_fixture(cuda_device):
    with open(os.path.join(GOLDEN, "oracle_tiny.json")) as f:
        d = json.load(f)
    off = torch.tensor(d["offsets"], dtype=torch.int32)
    ind = torch.tensor(d["indices"], dtype=torch.int32)
    feats = torch.tensor(d["features"], dtype=torch.float32)
    targets = torch.tensor(d["targets"], dtype=torch.int32)
    g = load(off, ind, feats, d["adj_block_bytes"], d["feat_block_bytes"])
    g.prepare(targets.to(cuda_device), d["fanouts"], d["seed"], d["first_gid"])
    assert g.stats() == d["stats"]
    for j, ref in enumerate(d["minibatches"]):
        v = g.fetch(j)
        assert v.nodes.cpu().tolist() == ref["nodes"]
        for hv, hr in zip(v.hops, ref["hops"]):
            assert hv.num_dst == hr["num_dst"]
            assert hv.indptr.cpu().tolist() == hr["indptr"]
            assert hv.col.cpu().tolist() == hr["col"]
    g.close()


@pytest.mark.parametrize("fanouts,H,B", [
    ((1024,), 3, 40),          # the largest fanout: 32 chunks of the wide sampler
    ((100, 3), 4, 60),         # several chunks, then a small hop
    ((2,) * 8, 3, 50),         # the most hops
])
def test_parity_extreme_fanouts_and_hops(cuda_device, fanouts, H, B):
    """Skewed graph whose hubs have far more than 1024 neighbours."""
    off, ind = synth.rmat_csr(20000, 60, 0.6, 0.2, 0.15, 13, offsets_dtype=torch.int64)
    assert int((off[1:] - off[:-1]).max()) > 2 * max(fanouts)
    feats = synth.normal_features(20000, 16, torch.float32, 14)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    # targets include the highest-degree nodes
    deg = off[1:] - off[:-1]
    hubs = torch.argsort(deg, descending=True)[:H * B // 4].to(torch.int32)
    rest = synth.hyperbatch_targets(torch.arange(20000, dtype=torch.int32), H, B, 2, 0)
    targets = rest.clone()
    for j in range(H):  # put hubs into every minibatch, keeping the targets distinct
        row = targets[j].tolist()
        extra = [h for h in hubs.tolist() if h not in row][:B // 4]
        targets[j, :len(extra)] = torch.tensor(extra, dtype=torch.int32)
        assert len(set(targets[j].tolist())) == B
    g = load(off, ind, feats, 16384, 16384)
    g.prepare(targets.to(cuda_device), list(fanouts), 99, 7)
    compare(g, og, targets.numpy(), list(fanouts), 99, 7, 16384, 16384)
    g.close()


def _hub_graph(N: int, hub_degrees, seed: int):
    """A sparse RMAT graph plus hub nodes with the given numbers of distinct
    random neighbours (as CSR)."""
    off, ind = synth.rmat_csr(N, 6, 0.57, 0.19, 0.19, seed)
    deg = (off[1:] - off[:-1]).long()
    src = torch.repeat_interleave(torch.arange(N, dtype=torch.int64), deg)
    keys = [src * N + ind.long()]
    hubs = []
    for i, d in enumerate(hub_degrees):
        h = int(synth.permutation(N, seed + 1)[i])
        nbrs = synth.permutation(N, seed + 10 + i)[:d + 1].long()
        nbrs = nbrs[nbrs != h][:d]
        keys.append(h * N + nbrs)
        hubs.append(h)
    keys = torch.unique(torch.cat(keys))
    off, ind = synth.csr_from_keys(keys, N)
    return off, ind, hubs


@pytest.mark.parametrize("fanouts,H,B", [
    ((4096, 6), 3, 12),   # four chunks of 1024 past the shared-memory sampler, then a small hop
    ((65536,), 2, 4),     # the largest fanout
])
def test_parity_fanouts_past_shared_memory(cuda_device, fanouts, H, B):
    """Fanouts above 1024 up to the 2^16 maximum, where each warp keeps the
    positions Floyd's algorithm has chosen in a hash set in global memory, on
    a graph whose hubs have more than 2^17 neighbours; every minibatch holds
    two hubs and is bit-exact against the oracle."""
    N = 300_000
    off, ind, hubs = _hub_graph(N, [140_000, 180_000, 220_000, 260_000], 21)
    deg = off[1:] - off[:-1]
    assert all(int(deg[h]) > 1 << 17 for h in hubs)
    feats = synth.normal_features(N, 8, torch.float32, 22)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    targets = synth.hyperbatch_targets(torch.arange(N, dtype=torch.int32), H, B, 23, 0)
    for j in range(H):  # two hubs per minibatch, targets kept distinct
        row = [t for t in targets[j].tolist() if t not in hubs][:B - 2]
        targets[j] = torch.tensor([hubs[(2 * j) % 4], hubs[(2 * j + 1) % 4]] + row,
                                  dtype=torch.int32)
    g = load(off, ind, feats, 1 << 20, 1 << 16)
    g.prepare(targets.to(cuda_device), list(fanouts), 5, 31)
    compare(g, og, targets.numpy(), list(fanouts), 5, 31, 1 << 20, 1 << 16)
    g.prepare(targets.to(cuda_device), list(fanouts), 6, 31)  # the sets are cleared per node
    compare(g, og, targets.numpy(), list(fanouts), 6, 31, 1 << 20, 1 << 16, check_stats=False)
    g.close()


@pytest.mark.parametrize("bits,dtype,fanouts", [
    (32, torch.float32, (10, 5)),
    (64, torch.float16, (15, 10, 5)),
    (64, torch.float16, (25, 10)),
    (32, torch.float16, (3,)),
    (64, torch.float32, (1, 1, 1, 1)),
    (64, torch.float16, (40, 3)),      # fanout above one warp
    (32, torch.float32, (33, 2)),
    (64, torch.float16, (4, 8, 16, 32)),
])
def test_parity_small_rmat(cuda_device, bits, dtype, fanouts):
    off, ind, feats = make(30000, 12, seed=len(fanouts) * 7 + bits, bits=bits, dtype=dtype)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    targets = synth.hyperbatch_targets(torch.arange(30000, dtype=torch.int32), 5, 100, 11, bits)
    adj_bb, feat_bb = 8192, 4096
    g = load(off, ind, feats, adj_bb, feat_bb)
    g.prepare(targets.to(cuda_device), list(fanouts), 0xDEADBEEF12345678, 1000)
    compare(g, og, targets.numpy(), list(fanouts), 0xDEADBEEF12345678, 1000, adj_bb, feat_bb)
    g.close()


@pytest.mark.parametrize("frontier", ["src", "sampled"])
def test_parity_edge_capacity_past_packed_bucket(cuda_device, frontier):
    """Hop 2's edge capacity per minibatch (41,984 frontier slots x 30) passes
    2^20, so that hop keeps the sampled bucket as (id, edge index) pairs and
    the sampler's separate rank array; hop 1 packs its entries into 4 bytes.
    Both layouts in one hyperbatch, every minibatch against the oracle."""
    n, B, fanouts = 60000, 1024, [40, 30]
    assert min(n, B * (1 + fanouts[0])) * fanouts[1] > 1 << 20 > B * fanouts[0]
    off, ind, feats = make(n, 12, seed=77, bits=64, dtype=torch.float16)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    targets = synth.hyperbatch_targets(torch.arange(n, dtype=torch.int32), 2, B, 12, 64)
    g = load(off, ind, feats, 8192, 4096)
    g.set_frontier(frontier)
    g.prepare(targets.to(cuda_device), fanouts, 0x5EED, 40)
    compare(g, og, targets.numpy(), fanouts, 0x5EED, 40, 8192, 4096, frontier=frontier)
    g.close()


def test_block_table_matches_oracle(cuda_device):
    for bits, bb in ((32, 64), (64, 256), (64, 4096), (32, 65536)):
        off, ind, feats = make(20000, 20, a=0.6, b=0.2, c=0.15, seed=bb, bits=bits)
        og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
        node_block, nb = oracle.build_adj_blocks(og, bb)
        starts = np.flatnonzero(np.r_[True, node_block[1:] != node_block[:-1]])
        g = load(off, ind, feats, bb, 4096)
        sn, sb = g.adj_blocks()
        assert np.array_equal(sn.numpy(), starts)
        assert np.array_equal(sb.numpy(), node_block[starts])
        assert g.info()["adj_blocks"] == nb
        g.close()


def test_degenerate_graphs(cuda_device):
    # a star plus isolated nodes: most targets have degree 0
    n = 5000
    deg = np.zeros(n, np.int64)
    deg[0] = n - 1
    deg[1:50] = 1
    off = torch.tensor(np.r_[0, np.cumsum(deg)], dtype=torch.int64)
    rows = [np.arange(1, n)] + [np.array([0])] * 49
    ind = torch.tensor(np.concatenate(rows), dtype=torch.int32)
    feats = synth.normal_features(n, 8, torch.float32, 1)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    g = load(off, ind, feats, 1024, 64)
    for targets in (np.arange(4000, 4064, dtype=np.int32).reshape(1, 64),   # all degree 0
                    np.array([[0, 1, 2, 3], [4999, 10, 0, 7]], np.int32),
                    np.arange(n, dtype=np.int32).reshape(1, n)):          # B = N
        for fan in ([5], [2, 2], [1024]):
            g.prepare(torch.tensor(targets).to(cuda_device), fan, 3, 9)
            compare(g, og, targets, fan, 3, 9, 1024, 64)
    g.close()


def test_hyperbatch_size_and_block_size_do_not_change_results(cuda_device):
    """Global minibatch 502 gives the same output inside hyperbatches of 16, 3
    and 1 minibatches and under different block sizes."""
    off, ind, feats = make(40000, 14, seed=21)
    targets = synth.hyperbatch_targets(torch.arange(40000, dtype=torch.int32), 16, 128, 4, 0)
    fan, seed = [8, 4, 2], 99
    ref = None
    # (first row, H, block bytes): row 2 of targets is global minibatch 502
    for first, H, bb in ((0, 16, 1 << 20), (1, 3, 65536), (2, 1, 4096), (0, 16, 2048)):
        g = load(off, ind, feats, bb, bb)
        g.prepare(targets[first:first + H].contiguous().to(cuda_device), fan, seed, 500 + first)
        v = g.fetch(2 - first)
        got = (v.nodes.cpu().numpy(), [h.col.cpu().numpy() for h in v.hops], _bytes(v.feats))
        if ref is None:
            ref = got
        else:
            assert np.array_equal(got[0], ref[0])
            assert all(np.array_equal(a, b) for a, b in zip(got[1], ref[1]))
            assert np.array_equal(got[2], ref[2])
        g.close()


def test_host_targets_equal_device_targets(cuda_device):
    off, ind, feats = make(20000, 10, seed=3)
    targets = synth.hyperbatch_targets(torch.arange(20000, dtype=torch.int32), 4, 256, 1, 0)
    g = load(off, ind, feats, 16384, 16384)
    g.prepare(targets.to(cuda_device), [10, 5], 5, 0)
    a = [g.fetch(j).nodes.cpu().clone() for j in range(4)]
    g.prepare(targets.pin_memory(), [10, 5], 5, 0)
    b = [g.fetch(j).nodes.cpu().clone() for j in range(4)]
    g.prepare(targets.clone(), [10, 5], 5, 0)  # pageable host memory
    c = [g.fetch(j).nodes.cpu().clone() for j in range(4)]
    assert all(torch.equal(x, y) and torch.equal(x, z) for x, y, z in zip(a, b, c))
    g.close()


@pytest.mark.parametrize("dtype,dim", [(torch.float16, 3), (torch.float32, 100),
                                       (torch.float32, 32), (torch.float16, 256),
                                       (torch.float32, 1000)])
def test_row_sizes(cuda_device, dtype, dim):
    off, ind, feats = make(8000, 8, seed=dim, dtype=dtype, dim=dim)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    targets = synth.hyperbatch_targets(torch.arange(8000, dtype=torch.int32), 3, 50, 2, dim)
    rb = feats.shape[1] * feats.element_size()
    g = load(off, ind, feats, 4096, max(4096, rb))
    g.prepare(targets.to(cuda_device), [6, 3], 17, 3)
    compare(g, og, targets.numpy(), [6, 3], 17, 3, 4096, max(4096, rb))
    g.close()


def test_invalid_targets_are_reported_and_ctx_stays_usable(cuda_device):
    off, ind, feats = make(3000, 6, seed=8)
    g = load(off, ind, feats, 4096, 4096)
    bad_range = torch.tensor([[1, 2, 3000]], dtype=torch.int32)
    bad_dup = torch.tensor([[5, 9, 5, 7]], dtype=torch.int32)
    for bad in (bad_range, bad_dup, torch.tensor([[-1, 4]], dtype=torch.int32)):
        g.prepare(bad.to(cuda_device), [3], 1, 0)
        with pytest.raises(AgnesError) as e:
            g.fetch(0)
        assert e.value.status == 1
    with pytest.raises(AgnesError):
        g.prepare(torch.tensor([[1]], dtype=torch.int32, device=cuda_device), [0], 1, 0)
    with pytest.raises(AgnesError):
        g.prepare(torch.tensor([[1]], dtype=torch.int32, device=cuda_device), [65537], 1, 0)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    ok = np.array([[1, 2, 3, 4]], np.int32)
    g.prepare(torch.tensor(ok).to(cuda_device), [3, 2], 1, 0)
    compare(g, og, ok, [3, 2], 1, 0, 4096, 4096)
    g.close()


@pytest.mark.parametrize("name", ["rmat100k", "mini100m", "mini_skew"])
def test_workload_parity_all_minibatches(cuda_device, name):
    w = WORKLOADS[name]
    data = build_workload(w, "cpu")
    og = oracle.Graph(data["offsets"].numpy(), data["indices"].numpy(), data["features"].numpy())
    g = load(data["offsets"], data["indices"], data["features"], w.adj_block_bytes,
             w.feat_block_bytes)
    targets = targets_for_step(w, data["pool"], 0)
    g.prepare(targets.to(cuda_device), list(w.fanouts), w.seed, 0)
    compare(g, og, targets.numpy(), list(w.fanouts), w.seed, 0, w.adj_block_bytes,
            w.feat_block_bytes)
    c = g.counters()
    assert c["rows"] == sum(g.sizes(j)["num_nodes"] for j in range(w.H))
    assert 0 < c["distinct_rows"] <= c["rows"]
    g.close()


@pytest.mark.parametrize("io", ["blocks", "rows"])
@pytest.mark.parametrize("dtype,dim,fbb,H", [
    (torch.float32, 16, 1024, 6),     # ~1900 feature blocks: many batches, the slot ring wraps
    (torch.float16, 128, 4096, 3),
    (torch.float16, 128, 1 << 20, 1),  # one block per batch
    (torch.float32, 12, 1008, 2),     # 48-byte rows, 21 rows per block: odd vector counts
])
def test_streamed_features_match_oracle(cuda_device, dtype, dim, fbb, H, io):
    """Features in pinned host memory, read over the host link block by block
    through the HBM slot ring, or row by row: same bytes as the oracle, over
    two hyperbatches in a row."""
    off, ind, feats = make(30000, 10, seed=dim + H, dtype=dtype, dim=dim)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    host_feats = feats.pin_memory()
    g = Graph(off.to(cuda_device), ind.to(cuda_device), host_feats, adj_block_bytes=8192,
              feat_block_bytes=fbb, features_on_host=True, feature_io=io)
    rb = dim * feats.element_size()
    for step in range(2):
        targets = synth.hyperbatch_targets(torch.arange(30000, dtype=torch.int32), H, 200, 7, step)
        g.prepare(targets.to(cuda_device), [8, 4], 21, 100 * step)
        compare(g, og, targets.numpy(), [8, 4], 21, 100 * step, 8192, fbb)
        c = g.counters()
        assert c["streamed_blocks"] == g.stats()[-1]
        if io == "blocks":
            assert 0 < c["streamed_bytes"] <= c["streamed_blocks"] * (fbb // rb) * rb
        else:  # each distinct row crosses the host link once
            assert c["streamed_bytes"] == c["distinct_rows"] * rb
    g.close()


@pytest.mark.parametrize("io", ["blocks", "rows"])
@pytest.mark.parametrize("cache_blocks,threshold", [
    (200, 0),          # cache holds ~1/5 of the blocks: the hottest ones
    (100000, 0),       # cache holds every block: from the third hyperbatch on, all hits
    (300, 10**9),      # no block's count exceeds the threshold: nothing cached
])
def test_feature_cache_matches_oracle(cuda_device, cache_blocks, threshold, io):
    """Streamed features with the access-count feature cache: same bytes as
    the oracle over several hyperbatches, while cached blocks are read in
    place instead of being copied again."""
    n, dim, fbb = 30000, 64, 4096
    off, ind, feats = make(n, 10, seed=5, dtype=torch.float16, dim=dim)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    g = Graph(off.to(cuda_device), ind.to(cuda_device), feats.pin_memory(), adj_block_bytes=8192,
              feat_block_bytes=fbb, features_on_host=True, feature_cache_bytes=cache_blocks * fbb,
              feature_cache_threshold=threshold, feature_io=io)
    nfb = -(-n // (fbb // (dim * 2)))
    prev_hits = prev_loads = 0
    for step in range(4):
        targets = synth.hyperbatch_targets(torch.arange(n, dtype=torch.int32), 3, 100, 11, step)
        g.prepare(targets.to(cuda_device), [6, 3], 4, 50 * step)
        compare(g, og, targets.numpy(), [6, 3], 4, 50 * step, 8192, fbb)
        c = g.counters()
        hits, loads = c["fcache_hit_blocks"] - prev_hits, c["fcache_loaded_blocks"] - prev_loads
        prev_hits, prev_loads = c["fcache_hit_blocks"], c["fcache_loaded_blocks"]
        assert c["streamed_blocks"] + hits == g.stats()[-1]
        assert loads <= c["streamed_blocks"]
        if step == 0 or threshold >= 10**9:
            assert hits == 0 and loads == 0
        if cache_blocks >= nfb and step >= 2:
            assert hits > 0
    if cache_blocks >= nfb:
        assert prev_loads <= nfb  # nothing is evicted, so no block is loaded twice
    if threshold < 10**9:
        assert prev_loads > 0 and prev_hits > 0
        assert prev_loads <= min(cache_blocks, nfb) * 3
    g.close()


def test_feature_cache_needs_host_features(cuda_device):
    off, ind, feats = make(2000, 6, seed=4, dim=16)
    with pytest.raises(AgnesError) as e:
        Graph(off.to(cuda_device), ind.to(cuda_device), feats.to(cuda_device),
              adj_block_bytes=4096, feat_block_bytes=4096, feature_cache_bytes=1 << 20)
    assert e.value.status == 1


@pytest.mark.parametrize("bb,fan,H,B", [
    (8192, [8, 4, 2], 4, 200),       # small cells (short tiles)
    (1 << 20, [15, 10, 5], 3, 300),  # 4096-id tiles: cells of hundreds of entries
    (4096, [5, 5], 6, 100),
])
def test_sampled_frontier_matches_oracle(cuda_device, bb, fan, H, B):
    """Algorithm 1's literal frontier (N_in <- N_out): bit-exact blocks, node
    lists, features and blocks-touched statistics, then the default frontier
    again on the same ctx."""
    off, ind, feats = make(30000, 12, seed=bb % 97 + len(fan))
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    g = load(off, ind, feats, bb, bb)
    targets = synth.hyperbatch_targets(torch.arange(30000, dtype=torch.int32), H, B, 5, 0)
    g.set_frontier("sampled")
    g.prepare(targets.to(cuda_device), fan, 13, 7)
    compare(g, og, targets.numpy(), fan, 13, 7, bb, bb, frontier="sampled")
    allv = g.fetch_all()
    if len(fan) > 1:  # the sampled frontier is a strict subset of src somewhere
        assert (allv.node_size[1] < allv.src_size[0]).any()
    g.set_frontier("src")
    g.prepare(targets.to(cuda_device), fan, 13, 7)
    compare(g, og, targets.numpy(), fan, 13, 7, bb, bb, frontier="src")
    allv = g.fetch_all()
    assert np.array_equal(allv.node_size[1:len(fan)], allv.src_size[:len(fan) - 1])
    with pytest.raises(ValueError):
        g.set_frontier("bogus")
    g.close()


def test_fetch_all_equals_per_minibatch_fetch(cuda_device):
    off, ind, feats = make(20000, 10, seed=31)
    targets = synth.hyperbatch_targets(torch.arange(20000, dtype=torch.int32), 5, 128, 3, 0)
    g = load(off, ind, feats, 16384, 16384)
    g.prepare(targets.to(cuda_device), [9, 4, 2], 8, 40)
    allv = g.fetch_all()
    assert (allv.K, allv.H) == (3, 5)
    for j in range(5):
        a, b = g.fetch(j), allv.view(j)
        assert torch.equal(a.nodes, b.nodes) and torch.equal(a.feats, b.feats)
        for ha, hb in zip(a.hops, b.hops):
            assert (ha.num_dst, ha.num_src, ha.num_edges) == (hb.num_dst, hb.num_src, hb.num_edges)
            assert torch.equal(ha.indptr, hb.indptr) and torch.equal(ha.col, hb.col)
    g.close()


def test_capacity_overflow_is_erange(cuda_device):
    off, ind, feats = make(3000, 6, seed=9)
    g = load(off, ind, feats, 4096, 4096)
    big = torch.zeros((65535, 1), dtype=torch.int32, device=cuda_device)
    with pytest.raises(AgnesError) as e:  # 65535 x 1 x (1+1024)^2 output rows > 2^31
        g.prepare(big, [1024, 1024], 1, 0)
    assert e.value.status == 2
    g.close()


@pytest.mark.parametrize("a,b,c,bb,buf_blocks,fan", [
    (0.57, 0.19, 0.19, 8192, 40, [8, 4]),      # buffer << topology: many waves, LRU evictions
    (0.6, 0.2, 0.15, 4096, 64, [25, 10]),     # skewed: objects larger than a block
    (0.57, 0.19, 0.19, 16384, 100000, [6, 4, 2]),  # buffer holds everything: hits from hop 2 on
])
def test_streamed_topology_matches_oracle(cuda_device, a, b, c, bb, buf_blocks, fan):
    """Neighbour lists in pinned host memory, loaded block by block into an
    HBM graph buffer with LRU + pinning: same samples as the oracle."""
    off, ind = synth.rmat_csr(30000, 14, a, b, c, seed=int(bb + buf_blocks),
                              offsets_dtype=torch.int64)
    feats = synth.normal_features(30000, 32, torch.float16, 5)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    max_obj = 8 + 4 * int((off[1:] - off[:-1]).max())
    host_ind = ind.pin_memory()
    buf = max(buf_blocks, 2 * (-(-max_obj // bb)) + 2) * bb
    g = Graph(off.to(cuda_device), host_ind, feats.to(cuda_device), adj_block_bytes=bb,
              feat_block_bytes=4096, topology_on_host=True, graph_buffer_bytes=buf)
    for step in range(2):
        targets = synth.hyperbatch_targets(torch.arange(30000, dtype=torch.int32), 4, 150, 9, step)
        g.prepare(targets.to(cuda_device), fan, 77, 10 * step)
        compare(g, og, targets.numpy(), fan, 77, 10 * step, bb, 4096)
    cnt = g.counters()
    assert cnt["topo_loaded_blocks"] > 0 and cnt["topo_waves"] >= 2 * len(fan)
    if buf_blocks >= 100000:
        assert cnt["topo_hit_blocks"] > 0
    g.close()


@pytest.mark.parametrize("a,b,c,fan", [
    (0.57, 0.19, 0.19, [8, 4]),
    (0.6, 0.2, 0.15, [25, 10]),      # skewed: hubs with neighbour lists of many blocks
    (0.57, 0.19, 0.19, [6, 4, 2]),
])
def test_topology_read_in_place_matches_oracle(cuda_device, a, b, c, fan):
    """Neighbour lists in pinned host memory, read in place over the host
    link (AGNES_TOPOLOGY_IO_ROWS): same samples as the oracle."""
    off, ind = synth.rmat_csr(30000, 14, a, b, c, seed=len(fan) * 7, offsets_dtype=torch.int64)
    feats = synth.normal_features(30000, 32, torch.float16, 6)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    g = Graph(off.to(cuda_device), ind.pin_memory(), feats.to(cuda_device), adj_block_bytes=4096,
              feat_block_bytes=4096, topology_on_host=True, topology_io="rows")
    for step in range(2):
        targets = synth.hyperbatch_targets(torch.arange(30000, dtype=torch.int32), 4, 150, 9, step)
        g.prepare(targets.to(cuda_device), fan, 77, 10 * step)
        compare(g, og, targets.numpy(), fan, 77, 10 * step, 4096, 4096)
    cnt = g.counters()
    assert cnt["topo_loaded_blocks"] == 0 and cnt["topo_waves"] == 0
    g.close()


@pytest.mark.parametrize("cache_bytes,mode", [(128 << 10, "graph_pdl"), (128 << 10, "direct"),
                                              (4096, "graph_pdl"), (64 << 20, "graph_pdl")])
def test_topology_cache_matches_oracle(cuda_device, cache_bytes, mode):
    """In-place neighbour reads with a topology cache (graph_buffer_bytes in
    rows mode): the hottest block runs are copied into HBM between
    hyperbatches and read there, the rest in place; samples match the oracle
    whatever is cached (a 1-slot cache, a partial one, one larger than the
    topology), in graph and direct launch modes."""
    off, ind = synth.rmat_csr(30000, 14, 0.6, 0.2, 0.15, seed=31, offsets_dtype=torch.int64)
    feats = synth.normal_features(30000, 32, torch.float16, 6)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    g = Graph(off.to(cuda_device), ind.pin_memory(), feats.to(cuda_device), adj_block_bytes=4096,
              feat_block_bytes=4096, topology_on_host=True, topology_io="rows",
              graph_buffer_bytes=cache_bytes)
    g.set_launch_mode(mode)
    fan = [8, 5, 3]
    slots = cache_bytes // 4096
    for step in range(11):  # picks before hyperbatches 1 and 9 (0-based)
        targets = synth.hyperbatch_targets(torch.arange(30000, dtype=torch.int32), 4, 150, 9, step)
        g.prepare(targets.to(cuda_device), fan, 5, 10 * step)
        compare(g, og, targets.numpy(), fan, 5, 10 * step, 4096, 4096)
        cnt = g.counters()
        if step == 0:
            assert cnt["topo_loaded_blocks"] == 0 and cnt["topo_cached_requests"] == 0
        if step == 1:
            assert 0 < cnt["topo_loaded_blocks"] <= slots and cnt["topo_cached_requests"] > 0
    assert cnt["topo_loaded_blocks"] <= 2 * slots
    assert cnt["topo_hit_blocks"] == 0 and cnt["topo_waves"] == 0
    g.close()


def test_graph_buffer_smaller_than_an_object_is_rejected(cuda_device):
    off, ind = synth.rmat_csr(5000, 30, 0.6, 0.2, 0.15, seed=1)
    feats = synth.normal_features(5000, 8, torch.float32, 2)
    with pytest.raises(AgnesError) as e:
        Graph(off.to(cuda_device), ind.pin_memory(), feats.to(cuda_device), adj_block_bytes=1024,
              feat_block_bytes=1024, topology_on_host=True, graph_buffer_bytes=1024)
    assert e.value.status == 1
