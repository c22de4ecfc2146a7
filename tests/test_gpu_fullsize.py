"""Full-size parity: each workload at its full size, in the launch
configuration bench.py times (one hyperbatch of H minibatches through the C
ABI), checked against the oracle on the host: sampled minibatches bit-exact
(subgraphs, node lists, gathered feature bytes) and the blocks-touched
statistics over the whole hyperbatch."""
import os

import numpy as np
import pytest
import torch

import oracle
from agnes_inputs import WORKLOADS, build_graph, target_pool, targets_for_step
from paper_2601_01473_gb300 import Graph

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


def _bytes(t):
    t = t.detach().cpu().contiguous()
    return t.view(torch.uint8).numpy().reshape(-1)


@pytest.mark.timeout(900)
@pytest.mark.parametrize("name,sample", [
    ("rmat10m", (0, 31, 63)),
    ("rmat100m", (0, 77, 127)),
    ("rmat65m_skew", (0, 40, 63)),
])
def test_fullsize_parity(cuda_device, name, sample):
    w = WORKLOADS[name]
    offsets, indices, features = build_graph(w, cuda_device)
    targets = targets_for_step(w, target_pool(w, cuda_device), 0)
    deg = offsets[1:] - offsets[:-1]
    max_deg = int(deg.max())
    print(f"\n{name}: N={offsets.numel() - 1} E={indices.numel()} max_deg={max_deg}")
    if name == "rmat65m_skew":
        assert max_deg > 1_000_000
    torch.cuda.empty_cache()
    g = Graph(offsets, indices, features, w.adj_block_bytes, w.feat_block_bytes)
    gid0 = 1000
    g.prepare(targets, list(w.fanouts), w.seed, gid0)
    got_stats = g.stats()
    views = {j: g.fetch(j) for j in sample}
    got = {j: (v.nodes.cpu().numpy(), [(h.num_dst, h.num_src, h.num_edges, h.indptr.cpu().numpy(),
                                        h.col.cpu().numpy()) for h in v.hops], _bytes(v.feats))
           for j, v in views.items()}
    del views
    og = oracle.Graph(offsets.cpu().numpy(), indices.cpu().numpy(), features.cpu().numpy())
    g.close()
    del offsets, indices, features
    torch.cuda.empty_cache()
    t = targets.cpu().numpy()
    for j in sample:
        r = oracle.sample_minibatch(og, t[j], list(w.fanouts), w.seed, gid0 + j)
        nodes, hops, feats = got[j]
        assert np.array_equal(nodes, r["nodes"]), f"nodes of minibatch {j}"
        for h, (nd, ns, ne, ip, col) in enumerate(hops):
            rh = r["hops"][h]
            assert (nd, ns, ne) == (rh["num_dst"], rh["num_src"], rh["num_edges"])
            assert np.array_equal(ip, rh["indptr"]), f"indptr hop {h} mb {j}"
            assert np.array_equal(col, rh["col"]), f"col hop {h} mb {j}"
        assert np.array_equal(feats, r["feats"].view(np.uint8).reshape(-1)), f"feats mb {j}"
    _, ref_stats = oracle.hyperbatch(og, t, list(w.fanouts), w.seed, gid0, False,
                                     w.adj_block_bytes, w.feat_block_bytes,
                                     threads=os.cpu_count() or 1)
    assert got_stats == ref_stats


@pytest.mark.timeout(1200)
def test_config5_variants_parity(cuda_device):
    """Config 5 at full size: rmat100m's graph as a sweep point (256 KB blocks,
    H = 16), with its features in pinned host memory (row I/O through a 4 GB
    feature cache, block I/O, row I/O pipelined over tile ranges), and with
    its neighbour lists read in place from pinned host memory (without and
    with a 1 GB topology cache).  Sampled minibatches bit-exact against the
    oracle."""
    w = WORKLOADS["rmat100m"]
    offsets, indices, features = build_graph(w, cuda_device)
    pool = target_pool(w, cuda_device)
    ws = w.with_(H=16, adj_block_bytes=256 * 1024, feat_block_bytes=256 * 1024)
    targets = targets_for_step(ws, pool, 3)
    fan = list(w.fanouts)
    sample = (0, 9, 15)
    host_feats = features.cpu().pin_memory()
    host_ind = indices.cpu().pin_memory()
    got = {}
    variants = {
        "sweep": dict(offsets=offsets, indices=indices, features=features),
        "rows+cache": dict(offsets=offsets, indices=indices, features=host_feats,
                           features_on_host=True, feature_io="rows",
                           feature_cache_bytes=4 << 30),
        "blocks": dict(offsets=offsets, indices=indices, features=host_feats,
                       features_on_host=True),
        "rows": dict(offsets=offsets, indices=indices, features=host_feats,
                     features_on_host=True, feature_io="rows"),
        "topology rows": dict(offsets=offsets, indices=host_ind, features=features,
                              topology_on_host=True, topology_io="rows"),
        "topology rows+cache": dict(offsets=offsets, indices=host_ind, features=features,
                                    topology_on_host=True, topology_io="rows",
                                    graph_buffer_bytes=1 << 30),
    }
    for name, kw in variants.items():
        g = Graph(adj_block_bytes=ws.adj_block_bytes, feat_block_bytes=ws.feat_block_bytes, **kw)
        for step in range(3):  # blocks admitted after the first load in the second; hits from the third
            g.prepare(targets, fan, w.seed, 500)
        got[name] = {j: (g.fetch(j).nodes.cpu().numpy(),
                         [(h.indptr.cpu().numpy(), h.col.cpu().numpy()) for h in g.fetch(j).hops],
                         _bytes(g.fetch(j).feats)) for j in sample}
        if name == "rows+cache":
            assert g.counters()["fcache_hit_blocks"] > 0
        if name == "topology rows+cache":
            assert g.counters()["topo_cached_requests"] > 0
        g.close()
    og = oracle.Graph(offsets.cpu().numpy(), host_ind.numpy(), host_feats.numpy())
    t = targets.cpu().numpy()
    for j in sample:
        r = oracle.sample_minibatch(og, t[j], fan, w.seed, 500 + j)
        for name in variants:
            nodes, hops, feats = got[name][j]
            assert np.array_equal(nodes, r["nodes"]), f"{name}: nodes of minibatch {j}"
            for h, (ip, col) in enumerate(hops):
                assert np.array_equal(ip, r["hops"][h]["indptr"]), f"{name}: indptr {h} mb {j}"
                assert np.array_equal(col, r["hops"][h]["col"]), f"{name}: col {h} mb {j}"
            assert np.array_equal(feats, r["feats"].view(np.uint8).reshape(-1)), f"{name}: feats {j}"
