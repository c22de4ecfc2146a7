"""Pins for the oracle's literal Algorithm 1 frontier (N_in <- N_out, the
"sampled" frontier): brute-force neighbourhoods at full fanout, set
identities at any fanout, agreement with the default frontier where the
two must agree, and the per-node sample keys."""
import numpy as np
import pytest
import torch

import oracle
from agnes_inputs import synth


def _graph(n, deg, seed):
    off, ind = synth.rmat_csr(n, deg, 0.57, 0.19, 0.19, seed, offsets_dtype=torch.int64)
    feats = synth.normal_features(n, 4, torch.float32, seed + 1)
    return off.numpy(), ind.numpy(), oracle.Graph(off.numpy(), ind.numpy(), feats.numpy())


def test_full_fanout_frontier_is_the_neighbourhood_of_the_previous_frontier():
    off, ind, g = _graph(300, 5, 1)
    targets = np.array([3, 17, 42, 99, 150], np.int32)
    fan = [1024, 1024, 1024]
    mb = oracle.sample_minibatch(g, targets, fan, 5, 0, frontier="sampled")
    frontier = list(targets)
    for h in range(3):
        assert mb["hops"][h]["dst"].tolist() == frontier
        reached = set()
        for v in frontier:
            reached.update(int(u) for u in ind[off[v]:off[v + 1]])
        if h + 1 < 3:
            frontier = sorted(reached)
    # the last hop's src is its dst followed by the reached ids not in it, ascending
    last = mb["hops"][2]
    new = sorted(reached - set(last["dst"].tolist()))
    assert mb["nodes"].tolist() == last["dst"].tolist() + new


@pytest.mark.parametrize("fan", [[5, 3, 2], [10, 4], [2, 2, 2, 2]])
def test_sampled_frontier_identities(fan):
    off, ind, g = _graph(5000, 8, 2)
    targets = synth.hyperbatch_targets(torch.arange(5000, dtype=torch.int32), 1, 64, 1, 0)[0]
    mb = oracle.sample_minibatch(g, targets.numpy(), fan, 9, 7, frontier="sampled")
    for h, hop in enumerate(mb["hops"]):
        dst, nbr, col = hop["dst"], hop["nbr"], hop["col"]
        new = sorted(set(nbr.tolist()) - set(dst.tolist()))
        src = dst.tolist() + new
        assert hop["num_src"] == len(src)
        assert [src[c] for c in col.tolist()] == nbr.tolist()
        if h + 1 < len(fan):
            nxt = mb["hops"][h + 1]["dst"].tolist()
            assert nxt == sorted(set(nbr.tolist()))   # N_out: distinct sampled ids, ascending
            assert set(nxt) <= set(src)
    assert mb["nodes"].tolist()[:mb["hops"][-1]["num_dst"]] == mb["hops"][-1]["dst"].tolist()


def test_modes_agree_where_they_must():
    off, ind, g = _graph(4000, 8, 3)
    targets = synth.hyperbatch_targets(torch.arange(4000, dtype=torch.int32), 1, 50, 2, 0)[0].numpy()
    a = oracle.sample_minibatch(g, targets, [6, 4, 3], 11, 3, frontier="src")
    b = oracle.sample_minibatch(g, targets, [6, 4, 3], 11, 3, frontier="sampled")
    # hop 1 is the same in both (same frontier: the targets)
    for key in ("dst", "indptr", "nbr", "col"):
        assert np.array_equal(a["hops"][0][key], b["hops"][0][key])
    # a node in both hop-2 frontiers draws the same samples (the key does not see the frontier)
    for h in (1, 2):
        ha, hb = a["hops"][h], b["hops"][h]
        pa = {int(v): i for i, v in enumerate(ha["dst"])}
        common = 0
        for i, v in enumerate(hb["dst"].tolist()):
            if v in pa:
                j = pa[v]
                sa = ha["nbr"][ha["indptr"][j]:ha["indptr"][j + 1]]
                sb = hb["nbr"][hb["indptr"][i]:hb["indptr"][i + 1]]
                assert np.array_equal(sa, sb)
                common += 1
        assert common > 0
    # one hop: no next frontier, so the modes coincide
    a1 = oracle.sample_minibatch(g, targets, [7], 11, 3, frontier="src")
    b1 = oracle.sample_minibatch(g, targets, [7], 11, 3, frontier="sampled")
    assert np.array_equal(a1["nodes"], b1["nodes"]) and np.array_equal(a1["feats"], b1["feats"])


def test_sampled_frontier_is_never_larger_than_src():
    off, ind, g = _graph(3000, 10, 4)
    targets = synth.hyperbatch_targets(torch.arange(3000, dtype=torch.int32), 1, 40, 3, 0)[0].numpy()
    b = oracle.sample_minibatch(g, targets, [8, 8, 8], 1, 1, frontier="sampled")
    for h in range(2):
        assert b["hops"][h + 1]["num_dst"] <= b["hops"][h]["num_src"]
