"""Full-size parity: each workload at its full size, in the launch
configuration bench.py times (one hyperbatch of H minibatches through the C
ABI), checked against the oracle run over the whole hyperbatch on the host:
every minibatch bit-exact (subgraphs, node lists, gathered feature bytes) and
the blocks-touched statistics of the hyperbatch."""
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


def _check_hyperbatch(g, og, targets, fanouts, seed, gid0, adj_bb, feat_bb, features, byte_sample):
    """Every minibatch of g's last hyperbatch against the oracle run over the
    whole hyperbatch on the host cores: subgraph sizes, indptr, col and node
    lists element by element, the blocks-touched statistics exactly.  Feature
    rows: every minibatch's gathered bytes equal the feature rows of the
    oracle's node list (indexed on the device), and the minibatches of
    byte_sample are also compared with the oracle's own gather."""
    t = np.ascontiguousarray(targets.cpu().numpy())
    ref, ref_stats = oracle.hyperbatch(og, t, fanouts, seed, gid0, False, adj_bb, feat_bb,
                                       threads=os.cpu_count() or 1)
    assert g.stats() == ref_stats
    hv = g.fetch_all()
    K = len(fanouts)
    word = {2: torch.int16, 4: torch.int32}[features.element_size()]
    feats_words = features.view(word)
    for j in range(t.shape[0]):
        r = ref[j]
        n = int(hv.node_size[K, j])
        nodes = hv.nodes[j, :n].cpu().numpy()
        assert np.array_equal(nodes, r["nodes"]), f"nodes of minibatch {j}"
        for h in range(K):
            nd, ns, ne = int(hv.node_size[h, j]), int(hv.src_size[h, j]), int(hv.edges[h, j])
            rh = r["hops"][h]
            assert (nd, ns, ne) == (rh["num_dst"], rh["num_src"], rh["num_edges"]), (h, j)
            assert np.array_equal(hv.indptr[h][j, :nd + 1].cpu().numpy(), rh["indptr"]), (h, j)
            assert np.array_equal(hv.col[h][j, :ne].cpu().numpy(), rh["col"]), (h, j)
        want = feats_words.index_select(0, torch.from_numpy(r["nodes"]).to(features.device).long())
        assert torch.equal(hv.feats[j, :n].view(word), want), f"feats of minibatch {j}"
    for j in byte_sample:
        r = oracle.sample_minibatch(og, t[j], fanouts, seed, gid0 + j)
        n = int(hv.node_size[K, j])
        assert np.array_equal(_bytes(hv.feats[j, :n]), r["feats"].view(np.uint8).reshape(-1)), j


@pytest.mark.timeout(900)
@pytest.mark.parametrize("name", ["rmat10m", "rmat100m", "rmat65m_skew"])
def test_fullsize_parity(cuda_device, name):
    """Configs 2-4 at full size, in bench.py's launch configuration: every
    minibatch of one hyperbatch."""
    w = WORKLOADS[name]
    offsets, indices, features = build_graph(w, cuda_device)
    targets = targets_for_step(w, target_pool(w, cuda_device), 0)
    deg = offsets[1:] - offsets[:-1]
    max_deg = int(deg.max())
    print(f"\n{name}: N={offsets.numel() - 1} E={indices.numel()} max_deg={max_deg}")
    if name == "rmat65m_skew":
        assert max_deg > 1_000_000
    torch.cuda.empty_cache()
    og = oracle.Graph(offsets.cpu().numpy(), indices.cpu().numpy(), features.cpu().numpy())
    g = Graph(offsets, indices, features, w.adj_block_bytes, w.feat_block_bytes)
    gid0 = 1000
    g.prepare(targets, list(w.fanouts), w.seed, gid0)
    _check_hyperbatch(g, og, targets, list(w.fanouts), w.seed, gid0, w.adj_block_bytes,
                      w.feat_block_bytes, features, (0, w.H - 1))
    g.close()


@pytest.mark.timeout(1200)
@pytest.mark.parametrize("H,block", [(256, 4 << 20), (1, 256 << 10), (64, 512 << 10)])
def test_config5_extremes_parity(cuda_device, H, block):
    """Config 5's sweep at its extremes on rmat100m's graph: the largest
    hyperbatch with the largest blocks (the largest workspace, H x capK of
    about 277M output rows), one minibatch per hyperbatch with the smallest
    blocks, and a middle point; every minibatch checked."""
    w = WORKLOADS["rmat100m"]
    offsets, indices, features = build_graph(w, cuda_device)
    ws = w.with_(H=H, adj_block_bytes=block, feat_block_bytes=block)
    targets = targets_for_step(ws, target_pool(w, cuda_device), 7)
    torch.cuda.empty_cache()
    og = oracle.Graph(offsets.cpu().numpy(), indices.cpu().numpy(), features.cpu().numpy())
    g = Graph(offsets, indices, features, block, block)
    gid0 = 77_000
    for step in range(2):  # a second hyperbatch replays the captured launch sequence
        g.prepare(targets, list(w.fanouts), w.seed, gid0)
    _check_hyperbatch(g, og, targets, list(w.fanouts), w.seed, gid0, block, block, features,
                      (0, H - 1) if H > 1 else (0,))
    g.close()


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
