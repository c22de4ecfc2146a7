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
