"""The resident path replayed as one captured CUDA graph per hyperbatch shape
(the default) against the oracle and against direct launches, over a
sequence of hyperbatches that changes, between calls, only the key (seed,
minibatch ids: the graph is replayed) or the shape (H, fanouts, frontier
mode, profiling: it is captured again); and a caller's own capture of
prepare, which takes the direct path inside the caller's graph."""
import numpy as np
import pytest
import torch

import oracle
from agnes_inputs import synth
from test_gpu_parity import _bytes, compare, load, make

pytestmark = pytest.mark.gpu

ADJ, FEAT = 16384, 8192


def _snapshot(g):
    v = g.fetch_all()
    out = {"node_size": v.node_size.copy(), "src_size": v.src_size.copy(),
           "edges": v.edges.copy(), "nodes": v.nodes.clone(), "feats": _bytes(v.feats)}
    for h in range(v.K):
        out[f"indptr{h}"] = v.indptr[h].clone()
        out[f"col{h}"] = v.col[h].clone()
    out["stats"] = g.stats()
    return out


def _same(a, b):
    """Equal sizes, and equal contents within the sizes of every minibatch."""
    assert np.array_equal(a["node_size"], b["node_size"])
    assert np.array_equal(a["src_size"], b["src_size"])
    assert np.array_equal(a["edges"], b["edges"])
    assert a["stats"] == b["stats"]
    K, H = a["edges"].shape
    for j in range(H):
        n = int(a["node_size"][K, j])
        assert torch.equal(a["nodes"][j, :n], b["nodes"][j, :n])
        for h in range(K):
            nd, ne = int(a["node_size"][h, j]), int(a["edges"][h, j])
            assert torch.equal(a[f"indptr{h}"][j, :nd + 1], b[f"indptr{h}"][j, :nd + 1])
            assert torch.equal(a[f"col{h}"][j, :ne], b[f"col{h}"][j, :ne])
    fa, fb = a["feats"], b["feats"]
    assert fa.size == fb.size
    cap = int(a["nodes"].shape[1])
    row_bytes = fa.size // (H * cap)
    for j in range(H):
        n = int(a["node_size"][K, j])
        base = j * cap * row_bytes
        assert np.array_equal(fa[base:base + n * row_bytes], fb[base:base + n * row_bytes])


def test_graph_replays_match_the_oracle_and_direct_launches(cuda_device):
    off, ind, feats = make(30000, 10, seed=5, dim=32)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    pdl = load(off, ind, feats, ADJ, FEAT)  # the default launch mode
    graphed = load(off, ind, feats, ADJ, FEAT)
    graphed.set_launch_mode("graph")
    direct = load(off, ind, feats, ADJ, FEAT)
    direct.set_launch_mode("direct")
    ctxs = (pdl, graphed, direct)
    pool = torch.arange(30000, dtype=torch.int32)
    # (H, fanouts, seed, first minibatch id, frontier, profiling)
    seq = [(6, [6, 4, 3], 1, 0, "src", False),
           (6, [6, 4, 3], 2, 6, "src", False),      # new key: replay
           (6, [6, 4, 3], 1, 100, "src", False),    # new key: replay
           (3, [5, 5], 7, 0, "src", False),         # new shape: capture
           (6, [6, 4, 3], 9, 12, "sampled", False),  # new shape and frontier: capture
           (6, [6, 4, 3], 9, 18, "src", True),      # frontier and profiling: capture
           (6, [6, 4, 3], 3, 24, "src", True),      # replay, phase events re-pointed
           (6, [6, 4, 3], 4, 30, "src", "gather")]  # gather events only: capture
    for step, (H, fan, seed, gid, frontier, prof) in enumerate(seq):
        targets = synth.hyperbatch_targets(pool, H, 150, 3, step)
        for g in ctxs:
            g.set_frontier(frontier)
            g.set_profiling(prof)
            g.prepare(targets.to(cuda_device), fan, seed, gid)
        compare(pdl, og, targets.numpy(), fan, seed, gid, ADJ, FEAT, frontier=frontier)
        ref = _snapshot(pdl)
        for g in ctxs[1:]:
            _same(ref, _snapshot(g))
        if prof:
            for g in ctxs:
                t = g.phase_times(0)
                n = 1 if prof == "gather" else 2 + 3 * len(fan)
                assert len(t) == n and all(x >= 0 for x in t)
    for g in ctxs[:2]:
        c = g.counters()
        assert c["graph_captures"] == 5 and c["graph_launches"] == len(seq)
    assert pdl.counters()["graph_programmatic_edges"] > 20
    assert graphed.counters()["graph_programmatic_edges"] == 0
    d = direct.counters()
    assert d["graph_captures"] == 0 and d["graph_launches"] == 0
    for g in ctxs:
        g.close()


def test_prepare_inside_a_callers_capture(cuda_device):
    off, ind, feats = make(20000, 8, seed=6, dim=16, dtype=torch.float32)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    g = load(off, ind, feats, ADJ, FEAT)
    pool = torch.arange(20000, dtype=torch.int32)
    targets = synth.hyperbatch_targets(pool, 4, 100, 3, 0).to(cuda_device)
    fan = [5, 3]
    s = torch.cuda.Stream(cuda_device)
    g.prepare(targets, fan, 11, 40, s)  # allocates the workspace outside the capture
    torch.cuda.synchronize()
    cg = torch.cuda.CUDAGraph()
    with torch.cuda.graph(cg, stream=s):
        g.prepare(targets, fan, 11, 40, torch.cuda.current_stream())
    torch.cuda.synchronize()
    other = synth.hyperbatch_targets(pool, 4, 100, 3, 1).to(cuda_device)
    g.prepare(other, fan, 2, 0, s)
    torch.cuda.synchronize()
    compare(g, og, other.cpu().numpy(), fan, 2, 0, ADJ, FEAT)
    with torch.cuda.stream(s):  # the replay writes the ctx's buffers: ordered by the caller
        cg.replay()
    torch.cuda.synchronize()
    compare(g, og, targets.cpu().numpy(), fan, 11, 40, ADJ, FEAT)
    assert g.counters()["graph_launches"] == 2  # the prepare inside the capture took the direct path
    g.close()


def test_prepares_on_two_streams_run_in_call_order(cuda_device):
    off, ind, feats = make(20000, 8, seed=7, dim=16)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    g = load(off, ind, feats, ADJ, FEAT)
    pool = torch.arange(20000, dtype=torch.int32)
    s1, s2 = torch.cuda.Stream(cuda_device), torch.cuda.Stream(cuda_device)
    fan = [6, 4]
    t1 = synth.hyperbatch_targets(pool, 5, 120, 3, 0).to(cuda_device)
    t2 = synth.hyperbatch_targets(pool, 5, 120, 3, 1).to(cuda_device)
    torch.cuda.synchronize()
    for _ in range(3):
        g.prepare(t1, fan, 4, 0, s1)
        g.prepare(t2, fan, 5, 5, s2)  # waits for the prepare on s1
    compare(g, og, t2.cpu().numpy(), fan, 5, 5, ADJ, FEAT)
    g.close()


@pytest.mark.parametrize("depth", [2, 3, 4])
def test_pipeline_depth_matches_oracle_and_overlaps_safely(cuda_device, depth):
    """Several hyperbatches in flight (agnes_set_pipeline_depth 2 .. 4): a
    sequence of prepares on one caller stream (more than the sets, so every
    set is reused), each checked against the oracle through fetch, the
    hyperbatch before the last through agnes_fetch_previous_hyperbatch while
    the last is in flight, a device-side consumer ordered with
    agnes_wait_hyperbatches, and a return to depth 1."""
    from paper_2601_01473_gb300 import AgnesError
    off, ind, feats = make(30000, 12, seed=51, dim=32)
    og = oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())
    g = load(off, ind, feats, ADJ, FEAT)
    g.set_pipeline_depth(depth)
    pool = torch.arange(30000, dtype=torch.int32)
    fan = [6, 4, 3]
    tgts = [synth.hyperbatch_targets(pool, 6, 200, 53, s) for s in range(5)]
    st = torch.cuda.Stream(cuda_device)
    with torch.cuda.stream(st):
        dev = [t.to(cuda_device, non_blocking=True) for t in tgts]
    for s in range(5):
        g.prepare(dev[s], fan, 7, 100 * s, st)
        if s >= 1:  # the previous hyperbatch, while this one may still run
            prev = g.fetch_previous()
            r = oracle.sample_minibatch(og, tgts[s - 1][2].numpy(), fan, 7, 100 * (s - 1) + 2)
            n = int(prev.node_size[3, 2])
            assert np.array_equal(prev.nodes[2, :n].cpu().numpy(), r["nodes"])
        if s >= depth - 1:  # the oldest one still held
            old = g.fetch_earlier(depth - 1)
            a = s - (depth - 1)
            r = oracle.sample_minibatch(og, tgts[a][4].numpy(), fan, 7, 100 * a + 4)
            n = int(old.node_size[3, 4])
            assert np.array_equal(old.nodes[4, :n].cpu().numpy(), r["nodes"])
        compare(g, og, tgts[s].numpy(), fan, 7, 100 * s, ADJ, FEAT)
    with pytest.raises(AgnesError):
        g.fetch_earlier(depth)
    # a device consumer on the caller's stream, ordered by the wait call
    g.prepare(dev[0], fan, 9, 0, st)
    g.prepare(dev[1], fan, 9, 600, st)
    g.wait(st)
    with torch.cuda.stream(st):
        v = g.fetch_all()
        copy = v.nodes.clone()
    st.synchronize()
    assert torch.equal(copy, v.nodes)
    compare(g, og, tgts[1].numpy(), fan, 9, 600, ADJ, FEAT)
    g.set_pipeline_depth(1)
    g.prepare(dev[2], fan, 9, 900, st)
    compare(g, og, tgts[2].numpy(), fan, 9, 900, ADJ, FEAT)
    g.close()


def test_pipeline_depth_two_needs_a_resident_graph(cuda_device):
    off, ind, feats = make(3000, 6, seed=52)
    dev = torch.device("cuda:0")
    from paper_2601_01473_gb300 import AgnesError, Graph
    g = Graph(off.to(dev), ind.to(dev), feats.pin_memory(), adj_block_bytes=4096,
              feat_block_bytes=4096, features_on_host=True)
    with pytest.raises(AgnesError) as e:
        g.set_pipeline_depth(2)
    assert e.value.status == 1
    with pytest.raises(AgnesError):
        g.set_pipeline_depth(3)
    g.close()
    r = load(off, ind, feats, 4096, 4096)
    for bad in (0, 5):  # 1 .. AGNES_MAX_PIPELINE_DEPTH
        with pytest.raises(AgnesError) as e:
            r.set_pipeline_depth(bad)
        assert e.value.status == 1
    r.set_pipeline_depth(4)
    r.close()
