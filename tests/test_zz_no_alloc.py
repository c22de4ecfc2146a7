"""agnes_hop_indptr_noalloc, the entry point for callers that must not
allocate device memory (see include/agnes.h), checked through the C ABI
against the indptr that agnes_prepare_hyperbatch produces for the same
nodes, on two calls in a row.  Kept in a file of its own that pytest collects
last."""
import ctypes

import pytest
import torch

from agnes_inputs import synth
from paper_2601_01473_gb300 import Graph, agnes

pytestmark = pytest.mark.gpu


def _noalloc(g: Graph, nodes: torch.Tensor, fanout: int, out: torch.Tensor) -> int:
    stream = torch.cuda.current_stream().cuda_stream or None
    return agnes.lib().agnes_hop_indptr_noalloc(g._ctx, nodes.data_ptr(), nodes.numel(), fanout,
                                                out.data_ptr(), stream)


@pytest.mark.parametrize("bits", [32, 64])
def test_noalloc_indptr_matches_prepare(cuda_device, bits):
    n = 50000
    off, ind = synth.rmat_csr(n, 12, 0.57, 0.19, 0.19, seed=41,
                              offsets_dtype=torch.int32 if bits == 32 else torch.int64)
    feats = synth.normal_features(n, 8, torch.float32, 42)
    g = Graph(off.to(cuda_device), ind.to(cuda_device), feats.to(cuda_device),
              adj_block_bytes=16384, feat_block_bytes=16384)
    targets = synth.hyperbatch_targets(torch.arange(n, dtype=torch.int32), 2, 3000, 43, bits)
    for call, fanout in enumerate((7, 25)):  # two calls in a row
        t = targets[call].contiguous().to(cuda_device)
        g.prepare(t.view(1, -1), [fanout], 5, call)
        ref = g.fetch(0).hops[0].indptr.clone()
        out = torch.full((t.numel() + 1,), -7, dtype=torch.int64, device=cuda_device)
        assert _noalloc(g, t, fanout, out) == 0, agnes.lib().agnes_last_error(g._ctx)
        torch.cuda.synchronize()
        assert torch.equal(out, ref)
    g.close()


def test_noalloc_rejects_oversized_and_bad_input(cuda_device):
    n = 1000
    off, ind = synth.rmat_csr(n, 5, 0.57, 0.19, 0.19, seed=44)
    feats = synth.normal_features(n, 8, torch.float32, 45)
    g = Graph(off.to(cuda_device), ind.to(cuda_device), feats.to(cuda_device),
              adj_block_bytes=4096, feat_block_bytes=4096)
    nodes = torch.arange(10, dtype=torch.int32, device=cuda_device)
    out = torch.zeros(11, dtype=torch.int64, device=cuda_device)
    L = agnes.lib()
    stream = torch.cuda.current_stream().cuda_stream or None
    too_many = (1 << 24) + 1
    assert L.agnes_hop_indptr_noalloc(g._ctx, nodes.data_ptr(), too_many, 3, out.data_ptr(),
                                      stream) == 2
    assert b"at most" in L.agnes_last_error(g._ctx)
    assert L.agnes_hop_indptr_noalloc(g._ctx, nodes.data_ptr(), 10, 0, out.data_ptr(), stream) == 1
    bad = torch.tensor([1, 2, n], dtype=torch.int32, device=cuda_device)
    assert _noalloc(g, bad, 3, out[:4]) == 1
    # the shared scratch's error word is cleared per call: a valid call succeeds next
    assert _noalloc(g, nodes, 3, out) == 0
    torch.cuda.synchronize()
    deg = (off[1:11] - off[:10]).clamp(max=3).to(torch.int64)
    assert torch.equal(out.cpu(), torch.cat([torch.zeros(1, dtype=torch.int64), deg.cumsum(0)]))
    g.close()


@pytest.mark.parametrize("n", [600_000, 1 << 24])
def test_noalloc_carries_partials_across_chunk_groups(cuda_device, n):
    """Node lists longer than one 256-chunk group of the partial-sum scan
    (524,288 nodes), up to the stated maximum of 2^24 nodes, against a torch
    prefix sum of min(deg, fanout); ids repeat, which the call allows."""
    N = 50000
    off, ind = synth.rmat_csr(N, 12, 0.57, 0.19, 0.19, seed=46, offsets_dtype=torch.int64)
    feats = synth.normal_features(N, 8, torch.float32, 47)
    g = Graph(off.to(cuda_device), ind.to(cuda_device), feats.to(cuda_device),
              adj_block_bytes=16384, feat_block_bytes=16384)
    gen = torch.Generator().manual_seed(n)
    nodes = torch.randint(0, N, (n,), generator=gen, dtype=torch.int32)
    deg = (off[1:] - off[:-1]).to(torch.int64)
    for fanout in (5, 1000):  # two calls in a row on the shared scratch
        out = torch.full((n + 1,), -3, dtype=torch.int64, device=cuda_device)
        assert _noalloc(g, nodes.to(cuda_device), fanout, out) == 0, \
            agnes.lib().agnes_last_error(g._ctx)
        torch.cuda.synchronize()
        ref = torch.cat([torch.zeros(1, dtype=torch.int64),
                         deg[nodes.long()].clamp(max=fanout).cumsum(0)])
        assert torch.equal(out.cpu(), ref)
    g.close()
