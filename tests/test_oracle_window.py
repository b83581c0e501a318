"""Pins for the observation-window score oracle (Sec. 4, SnapKV's score as a
ContourKV plug-in): a numpy computation of the same definition (one matrix
product per cell, masked softmax rows, a sliding maximum), the invariant that
each query's softmax row sums to one (so the votes of a cell sum to w), and
causality inside the window.  CPU only."""
import numpy as np
import pytest

import oracle
import workloads


def bf16(x):
    return workloads.f32_to_bf16_bits(np.asarray(x, np.float32))


def numpy_window_score(Qb, Kb, scale, pool):
    Q = workloads.bf16_bits_to_f32(Qb).astype(np.float64)
    K = workloads.bf16_bits_to_f32(Kb).astype(np.float64)
    cells, w, d = Q.shape
    T = K.shape[1]
    pos = np.arange(T)
    out_s, out_v = np.zeros((cells, T)), np.zeros((cells, T))
    for c in range(cells):
        L = scale * Q[c] @ K[c].T                           # [w][T]
        vis = pos[None, :] <= (T - w + np.arange(w))[:, None]
        L = np.where(vis, L, -np.inf)
        A = np.exp(L - L.max(axis=1, keepdims=True))
        A /= A.sum(axis=1, keepdims=True)
        vote = A.sum(axis=0)
        lim, h = T - w, pool // 2
        sc = vote.copy()
        for j in range(lim):
            sc[j] = vote[max(0, j - h):min(lim, j + h + 1)].max()
        out_s[c], out_v[c] = sc, vote
    return out_s, out_v


@pytest.mark.parametrize("cells,T,w,d,pool", [(2, 40, 8, 16, 7), (3, 17, 1, 8, 3), (1, 64, 32, 32, 7),
                                              (2, 33, 33, 8, 5), (2, 50, 4, 8, 1)])
def test_window_score_matches_numpy(cells, T, w, d, pool):
    rng = np.random.default_rng(T + w)
    Q = bf16(rng.normal(size=(cells, w, d)))
    K = bf16(rng.normal(size=(cells, T, d)) * 1.5)
    scale = 1 / np.sqrt(d)
    s, v = oracle.window_score(Q, K, scale, pool)
    ws, wv = numpy_window_score(Q, K, scale, pool)
    np.testing.assert_allclose(v, wv, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(s, ws, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(v.sum(axis=1), w, rtol=1e-12)  # every query's row sums to one


def test_window_causality_and_a_single_query():
    rng = np.random.default_rng(3)
    T, d = 20, 8
    Q = bf16(rng.normal(size=(1, 1, d)))
    K = bf16(rng.normal(size=(1, T, d)))
    s, v = oracle.window_score(Q, K, 0.5, 1)
    # one query at the last position: its own softmax row, no pooling (pool = 1)
    l = 0.5 * workloads.bf16_bits_to_f32(K[0]).astype(np.float64) @ workloads.bf16_bits_to_f32(Q[0, 0])
    p = np.exp(l - l.max())
    np.testing.assert_allclose(v[0], p / p.sum(), rtol=1e-12)
    np.testing.assert_allclose(s[0], v[0], rtol=0, atol=0)
    # w = 3: the key at the last position gets a vote from the last query only
    Q3 = bf16(rng.normal(size=(1, 3, d)))
    s3, v3 = oracle.window_score(Q3, K, 0.5, 1)
    q = workloads.bf16_bits_to_f32(Q3[0, 2]).astype(np.float64)
    l = 0.5 * workloads.bf16_bits_to_f32(K[0]).astype(np.float64) @ q
    p = np.exp(l - l.max())
    assert v3[0, T - 1] == pytest.approx(p[T - 1] / p.sum(), rel=1e-12)
