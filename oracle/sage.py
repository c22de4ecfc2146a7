"""GraphSAGE-mean layer over one sampled hop, in fp64: the consumer of the
prepared minibatch.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s cpu_baseline / ``--impl reference`` legs may import this
module.  It shares no code with the CUDA library.

Eq. (1) (Sec. 3.1, GNN preliminaries) writes a layer as an aggregation of the
in-neighbours' embeddings followed by an update of the node's own embedding
with that aggregate.  The instance computed here, for every dst node i of a
hop's bipartite block (dst is a prefix of src), is

    agg_i = mean over the block's edges (i, u) of x[u]       (0 if i has none)
    out_i = ReLU(W_self x[i] + W_neigh agg_i + b)

with W = [W_self | W_neigh] a d_out x 2 d_in matrix (the update's fully
connected layer) and b a d_out vector.
"""
from __future__ import annotations

import numpy as np


def sage_mean(indptr, col, x, w, b, num_dst: int):
    """Returns (out, a, m): the layer's output (num_dst x d_out), the update's
    input a = [x_dst | agg] (num_dst x 2 d_in), and m, per (row, feature), a
    bound on the error of forming that mean in fp32 ((deg_i + 1) 2^-24 times
    the mean absolute neighbour value: deg_i - 1 additions and one division,
    each rounded to nearest; zero where the row has no edges), used by
    :func:`error_bound`.  Everything in fp64."""
    x = np.asarray(x, dtype=np.float64)
    w = np.asarray(w, dtype=np.float64)
    b = np.zeros(w.shape[0]) if b is None else np.asarray(b, dtype=np.float64)
    indptr = np.asarray(indptr, dtype=np.int64)
    col = np.asarray(col, dtype=np.int64)
    d_in = x.shape[1]
    if w.shape[1] != 2 * d_in:
        raise ValueError("w must be d_out x 2*d_in")
    agg = np.zeros((num_dst, d_in))
    m = np.zeros((num_dst, d_in))
    for i in range(num_dst):
        s, e = int(indptr[i]), int(indptr[i + 1])
        if e > s:
            nb = x[col[s:e]]
            agg[i] = nb.sum(axis=0) / (e - s)
            m[i] = (e - s + 1) * 2.0 ** -24 * np.abs(nb).sum(axis=0) / (e - s)
    a = np.concatenate([x[:num_dst], agg], axis=1)
    out = np.maximum(a @ w.T + b, 0.0)
    return out, a, m


def error_bound(a, m, w, b, out, x_exact_f16: bool, out_f16: bool):
    """Elementwise bound on |kernel - oracle| for a kernel that forms agg in
    fp32, rounds the update's inputs to fp16 (exact for fp16 inputs), and
    accumulates the K = 2 d_in fp16 x fp16 products in fp32 (a tensor-core
    contraction):

      input rounding   sum_k |w_nk| (2^-11 |a_ik| + 2^-25 + m_ik): rounding
                       to fp16 is within 2^-11 relative for normal values and
                       within 2^-25 absolute for subnormal ones (binary16's
                       subnormal spacing is 2^-24); m is the fp32 mean's own
                       error (:func:`sage_mean`); the self half has neither
                       rounding term when x is fp16;
      accumulation     (K + 1) 2^-22 sum_k |a_ik w_nk|: the products are exact
                       in fp32; the accumulator takes them in steps of one or
                       more products, and each step may truncate (relative
                       error below 2^-23) both its inputs' alignment and its
                       result, at most 2K + 2 times in all, each time on a
                       magnitude no larger than sum_k |a_ik w_nk|;
      bias add         2^-22 |b_n|;
      output rounding  2^-11 |out_in| + 2^-25 for an fp16 output.

    ReLU is 1-Lipschitz and does not enlarge any of these."""
    a = np.asarray(a, dtype=np.float64)
    w = np.abs(np.asarray(w, dtype=np.float64))
    d_in = a.shape[1] // 2
    K = 2 * d_in
    rel = np.abs(a) * 2.0 ** -11 + 2.0 ** -25
    if x_exact_f16:
        rel[:, :d_in] = 0.0
    m_full = np.concatenate([np.zeros_like(m), m], axis=1)
    bound = (rel + m_full) @ w.T
    bound += (np.abs(a) @ w.T) * ((K + 1) * 2.0 ** -22)
    if b is not None:
        bound += np.abs(np.asarray(b, dtype=np.float64)) * 2.0 ** -22
    if out_f16:
        bound += np.abs(out) * 2.0 ** -11 + 2.0 ** -25
    return bound
