"""The GraphSAGE-mean consumer layer (agnes_sage_mean_layer, tcgen05) against
the fp64 oracle, within the elementwise bound the oracle derives for fp16
operands and fp32 accumulation, on every row of every minibatch: several
128-row tiles per minibatch with ragged tails, rows without edges, stacked
layers, both input and output dtypes."""
import numpy as np
import pytest
import torch

from agnes_inputs import synth
from oracle.sage import error_bound, sage_mean
from paper_2601_01473_gb300 import AgnesError, Graph

pytestmark = pytest.mark.gpu


def _graph(cuda_device, n, deg, dim, dtype, seed):
    off, ind = synth.rmat_csr(n, deg, 0.57, 0.19, 0.19, seed, offsets_dtype=torch.int64)
    feats = synth.normal_features(n, dim, dtype, seed + 1)
    g = Graph(off.to(cuda_device), ind.to(cuda_device), feats.to(cuda_device),
              adj_block_bytes=16384, feat_block_bytes=16384)
    return g


def _weights(d_in, d_out, seed, device):
    gen = torch.Generator().manual_seed(seed)
    w = (torch.randn(d_out, 2 * d_in, generator=gen) / (2 * d_in) ** 0.5).to(torch.float16)
    b = (torch.randn(d_out, generator=gen) * 0.1).to(torch.float32)
    return w.to(device), b.to(device)


def _check_layer(allv, hop, x, w, b, out, x_f16, out_f16):
    """Every dst row of every minibatch within the oracle's derived bound;
    returns the largest err / bound over all of them."""
    wn = w.float().cpu().numpy().astype(np.float64)
    bn = b.cpu().numpy().astype(np.float64) if b is not None else None
    xs = x.float().cpu().numpy()
    outs = out.float().cpu().numpy()
    worst = 0.0
    for j in range(allv.H):
        nd = int(allv.node_size[hop, j])
        ns = int(allv.src_size[hop, j])
        ne = int(allv.edges[hop, j])
        indptr = allv.indptr[hop][j, :nd + 1].cpu().numpy()
        col = allv.col[hop][j, :ne].cpu().numpy()
        assert indptr[-1] == ne and (ne == 0 or col.max() < ns)
        ref, a, m = sage_mean(indptr, col, xs[j, :ns].astype(np.float64), wn, bn, nd)
        bound = error_bound(a, m, wn, bn, ref, x_exact_f16=x_f16, out_f16=out_f16)
        err = np.abs(outs[j, :nd].astype(np.float64) - ref)
        assert np.all(err <= bound), (
            f"minibatch {j}: max err {err.max()} at {np.unravel_index(err.argmax(), err.shape)}")
        if nd:
            worst = max(worst, float((err / (bound + 1e-30)).max()))
    return worst


@pytest.mark.parametrize("dim,dtype,d_out,out_dtype", [
    (128, torch.float16, 128, torch.float32),
    (128, torch.float16, 256, torch.float16),
    (64, torch.float32, 32, torch.float32),
    (16, torch.float16, 96, torch.float32),
])
def test_sage_layer_matches_oracle(cuda_device, dim, dtype, d_out, out_dtype):
    g = _graph(cuda_device, 40000, 10, dim, dtype, seed=dim + d_out)
    targets = synth.hyperbatch_targets(torch.arange(40000, dtype=torch.int32), 5, 300, 3, 0)
    g.prepare(targets.to(cuda_device), [10, 5], 17, 0)
    allv = g.fetch_all()
    K = 2
    assert allv.node_size[K - 1].max() > 3 * 128  # several tiles per minibatch
    w, b = _weights(dim, d_out, 1, cuda_device)
    out = g.sage_mean_layer(K - 1, allv.feats, w, b, out_dtype=out_dtype)
    torch.cuda.synchronize()
    worst = _check_layer(allv, K - 1, allv.feats, w, b, out, dtype == torch.float16,
                         out_dtype == torch.float16)
    # the next layer consumes the first one's output (rows = src_{K-2})
    w2, b2 = _weights(d_out, 64, 2, cuda_device)
    x2 = out.contiguous()
    out2 = g.sage_mean_layer(K - 2, x2, w2, None, out_dtype=torch.float32)
    torch.cuda.synchronize()
    worst = max(worst, _check_layer(allv, K - 2, x2, w2, None, out2,
                                    out_dtype == torch.float16, False))
    print(f"sage layer worst err/bound: {worst:.3g}")
    g.close()


def test_sage_layer_rejects_bad_shapes(cuda_device):
    g = _graph(cuda_device, 5000, 6, 64, torch.float16, seed=3)
    targets = synth.hyperbatch_targets(torch.arange(5000, dtype=torch.int32), 2, 50, 3, 0)
    g.prepare(targets.to(cuda_device), [4, 2], 1, 0)
    allv = g.fetch_all()
    w, b = _weights(64, 48, 1, cuda_device)  # d_out not a multiple of 32
    with pytest.raises(AgnesError) as e:
        g.sage_mean_layer(1, allv.feats, w, b)
    assert e.value.status == 1
    w, b = _weights(64, 64, 1, cuda_device)
    with pytest.raises(AgnesError) as e:
        g.sage_mean_layer(2, allv.feats, w, b)  # hop out of range
    assert e.value.status == 1
    big = torch.zeros((2, allv.feats.shape[1], 256), dtype=torch.float16, device=cuda_device)
    w, b = _weights(256, 256, 1, cuda_device)  # operands do not fit shared memory
    with pytest.raises(AgnesError) as e:
        g.sage_mean_layer(1, big, w, b)
    assert e.value.status == 2
    g.close()
