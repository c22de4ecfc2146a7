"""Pins for the GraphSAGE-mean layer oracle (no GPU): a hand-worked example,
special cases that reduce to known functions, a pure-Python brute force of
the mean aggregation, and invariances of the layer."""
import numpy as np
import pytest

from oracle.sage import error_bound, sage_mean


def test_hand_worked_example():
    # src rows x0..x3; dst = first 3 rows; row 0 <- {x1, x2}, row 1 <- {x3}, row 2 <- {}
    x = np.array([[1, 2], [3, 4], [5, 6], [7, 8]], dtype=np.float64)
    indptr = np.array([0, 2, 3, 3])
    col = np.array([1, 2, 3])
    w_self = np.array([[1, 0], [0, -1]])
    w_neigh = np.array([[0, 1], [1, 0]])
    w = np.concatenate([w_self, w_neigh], axis=1)
    b = np.array([0.5, 0.0])
    out, a, _ = sage_mean(indptr, col, x, w, b, 3)
    # row 0: [1,-2] + W_neigh [4,5] = [5,4] -> [6.5, 2]
    # row 1: [3,-4] + W_neigh [7,8] = [8,7] -> [11.5, 3]
    # row 2: [5,-6] + 0 + b -> [5.5, -6] -> ReLU [5.5, 0]
    assert out.tolist() == [[6.5, 2.0], [11.5, 3.0], [5.5, 0.0]]
    assert a.tolist() == [[1, 2, 4, 5], [3, 4, 7, 8], [5, 6, 0, 0]]


def _random_block(rng, n_src, n_dst, max_deg, d):
    deg = rng.integers(0, max_deg + 1, n_dst)
    indptr = np.concatenate([[0], np.cumsum(deg)])
    col = rng.integers(0, n_src, int(indptr[-1]))
    x = rng.standard_normal((n_src, d))
    return indptr, col, x


def test_identity_self_weights_give_relu_of_the_dst_rows():
    rng = np.random.default_rng(1)
    indptr, col, x = _random_block(rng, 50, 20, 6, 8)
    w = np.concatenate([np.eye(8), np.zeros((8, 8))], axis=1)
    out, _, _ = sage_mean(indptr, col, x, w, None, 20)
    assert np.array_equal(out, np.maximum(x[:20], 0))


def test_identity_neighbour_weights_give_the_brute_force_mean():
    rng = np.random.default_rng(2)
    indptr, col, x = _random_block(rng, 40, 15, 5, 4)
    x = np.abs(x)  # positive, so ReLU is the identity on the mean
    w = np.concatenate([np.zeros((4, 4)), np.eye(4)], axis=1)
    out, _, _ = sage_mean(indptr, col, x, w, None, 15)
    for i in range(15):
        nbrs = list(col[indptr[i]:indptr[i + 1]])
        for f in range(4):
            if nbrs:
                total = 0.0
                for u in nbrs:
                    total += float(x[u][f])
                want = total / len(nbrs)
            else:
                want = 0.0
            assert out[i][f] == pytest.approx(want, rel=1e-12, abs=1e-15)


def test_positive_homogeneity_and_edge_order_invariance():
    rng = np.random.default_rng(3)
    indptr, col, x = _random_block(rng, 64, 30, 7, 6)
    w = rng.standard_normal((5, 12))
    b = rng.standard_normal(5)
    out, _, _ = sage_mean(indptr, col, x, w, b, 30)
    out2, _, _ = sage_mean(indptr, col, x, 2 * w, 2 * b, 30)
    assert np.allclose(out2, 2 * out, rtol=1e-13, atol=1e-13)
    col_p = col.copy()
    for i in range(30):
        s, e = indptr[i], indptr[i + 1]
        col_p[s:e] = rng.permutation(col[s:e])
    out3, _, _ = sage_mean(indptr, col_p, x, w, b, 30)
    assert np.allclose(out3, out, rtol=1e-12, atol=1e-12)


def test_rows_without_edges_use_only_the_self_half():
    rng = np.random.default_rng(4)
    x = rng.standard_normal((10, 3))
    w = rng.standard_normal((2, 6))
    b = rng.standard_normal(2)
    out, _, _ = sage_mean(np.zeros(6, np.int64), np.zeros(0, np.int64), x, w, b, 5)
    assert np.allclose(out, np.maximum(x[:5] @ w[:, :3].T + b, 0), rtol=1e-14, atol=1e-14)


def test_error_bound_covers_fp16_rounding_of_the_inputs():
    """The bound covers what it claims: rounding a (the update's input) to
    fp16 and accumulating in fp32 stays inside it."""
    rng = np.random.default_rng(5)
    indptr, col, x = _random_block(rng, 200, 100, 10, 16)
    x = x.astype(np.float16).astype(np.float64)
    w = rng.standard_normal((8, 32)).astype(np.float16).astype(np.float64)
    b = rng.standard_normal(8).astype(np.float32).astype(np.float64)
    out, a, m = sage_mean(indptr, col, x, w, b, 100)
    a16 = a.astype(np.float16).astype(np.float32)
    pre = (a16 @ w.astype(np.float32).T).astype(np.float32) + b.astype(np.float32)
    approx = np.maximum(pre, 0).astype(np.float64)
    bound = error_bound(a, m, w, b, out, x_exact_f16=True, out_f16=False)
    assert np.all(np.abs(approx - out) <= bound)


def _trunc_f32(v):
    """Rounds float64 values to float32 toward zero."""
    r = v.astype(np.float32)
    over = np.abs(r.astype(np.float64)) > np.abs(v)
    r[over] = np.nextafter(r[over], np.float32(0))
    return r


def test_error_bound_covers_truncating_accumulation_subnormals_and_f16_output():
    """A simulated kernel at the bound's worst assumptions: the mean summed in
    fp32, inputs rounded to fp16 (some aggregates cancel to fp16 subnormals),
    every product added into an fp32 accumulator that truncates, the bias
    added in fp32, the result rounded to fp16; fp32 features, so the self half
    is rounded too."""
    rng = np.random.default_rng(6)
    n_src, n_dst, d = 120, 60, 24
    indptr, col, x = _random_block(rng, n_src, n_dst, 6, d)
    # the first 20 dst rows take a pair of nearly opposite neighbours, so
    # their means cancel to about 1e-6 (fp16 subnormals)
    x[1::2] = -x[0::2] + rng.standard_normal((n_src // 2, d)) * 1e-6
    deg = np.diff(indptr)
    deg[:20] = 2
    rest = col[indptr[20]:]
    indptr = np.concatenate([[0], np.cumsum(deg)])
    col = np.concatenate([np.stack([np.arange(20) * 2, np.arange(20) * 2 + 1], 1).ravel(),
                          rest])
    w = rng.standard_normal((16, 2 * d)).astype(np.float16).astype(np.float64)
    b = rng.standard_normal(16).astype(np.float32).astype(np.float64)
    out, a, m = sage_mean(indptr, col, x, w, b, n_dst)
    x32 = x.astype(np.float32)
    agg32 = np.zeros((n_dst, d), np.float32)
    for i in range(n_dst):
        s, e = indptr[i], indptr[i + 1]
        if e > s:
            acc = np.zeros(d, np.float32)
            for u in col[s:e]:
                acc = (acc + x32[u]).astype(np.float32)
            agg32[i] = (acc / np.float32(e - s)).astype(np.float32)
    a16 = np.concatenate([x32[:n_dst], agg32], axis=1).astype(np.float16).astype(np.float64)
    assert np.any((a16 != 0) & (np.abs(a16) < 2.0 ** -14))  # subnormals occur
    acc = np.zeros((n_dst, 16), np.float32)
    for k in range(2 * d):
        acc = _trunc_f32(acc.astype(np.float64) + np.outer(a16[:, k], w[:, k]))
    pre = (acc + b.astype(np.float32)).astype(np.float32)
    approx = np.maximum(pre, 0).astype(np.float16).astype(np.float64)
    bound = error_bound(a, m, w, b, out, x_exact_f16=False, out_f16=True)
    assert np.all(np.abs(approx - out) <= bound)


def test_error_bound_rejects_a_kernel_that_rounds_its_inputs_to_bf16():
    """The bound is tight enough to catch a real precision loss: inputs
    rounded to bf16 (8 significant bits) instead of fp16 break it."""
    rng = np.random.default_rng(7)
    indptr, col, x = _random_block(rng, 200, 100, 10, 16)
    x = x.astype(np.float16).astype(np.float64)
    w = rng.standard_normal((8, 32)).astype(np.float16).astype(np.float64)
    out, a, m = sage_mean(indptr, col, x, w, None, 100)
    bits = a.astype(np.float32).view(np.uint32)
    a_bf16 = ((bits + 0x7FFF + ((bits >> 16) & 1)) & 0xFFFF0000).view(np.float32)
    approx = np.maximum(a_bf16.astype(np.float64) @ w.T, 0)
    bound = error_bound(a, m, w, None, out, x_exact_f16=True, out_f16=False)
    assert np.any(np.abs(approx - out) > bound)
