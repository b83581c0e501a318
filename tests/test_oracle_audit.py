"""Pins for the selector-audit oracle (Sec. 2.3, App. C's settings): each
rule's kept set rebuilt with numpy sorts from its definition, and its es from
the forced-weight output m_A = sum_A p v / p(A); set sizes; the rules that
ignore the logits (StreamingLLM).  CPU only."""
import numpy as np
import pytest

import oracle
from tests.test_gpu_small import rows_batch


def softmax(l):
    l = l.astype(np.float64)
    p = np.exp(l - l.max())
    return p / p.sum()


def es_of(p, V, mask):
    mu = p @ V
    S = np.flatnonzero(mask)
    return np.linalg.norm(p[S] @ V[S] / p[S].sum() - mu)


def numpy_sets(L, V, R, s):
    """L: [rows][n] logits of groups of R rows; returns sets [rows][5] masks."""
    rows, n = L.shape
    P = np.array([softmax(l) for l in L])
    out = []
    for g in range(rows // R):
        Pg = P[g * R:(g + 1) * R]
        G = Pg.sum(0)
        r = s // 2
        cand = np.arange(n - r)
        h = np.zeros(n, bool)
        h[n - r:] = True
        h[cand[np.lexsort((cand, -G[cand]))[: s - r]]] = True
        w = max(1, min(32, s // 2))
        vote = Pg[max(0, R - w):].sum(0)
        lim = n - w
        pooled = np.array([vote[max(0, j - 3):min(lim, j + 4)].max() for j in range(lim)])
        sn = np.zeros(n, bool)
        sn[lim:] = True
        c2 = np.arange(lim)
        sn[c2[np.lexsort((c2, -pooled))[: s - w]]] = True
        for i in range(R):
            l = L[g * R + i].astype(np.float64)
            sinks = min(4, s // 2)
            st = np.zeros(n, bool)
            st[:sinks] = True
            st[n - (s - sinks):] = True
            qs = []
            for Pq in (max(2, s // 4), 16):
                q = np.zeros(n, bool)
                if not (Pq == 16 and s < 16) and s // Pq >= 1:
                    np_ = -(-n // Pq)
                    pm = np.array([l[p * Pq:(p + 1) * Pq].max() for p in range(np_)])
                    pages = np.lexsort((np.arange(np_), -pm))[: s // Pq]
                    for p in pages:
                        q[p * Pq:(p + 1) * Pq] = True
                qs.append(q)
            out.append([st, h, sn, qs[0], qs[1]])
    return out, P


@pytest.mark.parametrize("R,n,d,s", [(6, 60, 32, 8), (1, 40, 32, 4), (40, 100, 64, 16), (3, 90, 32, 32),
                                     (4, 33, 32, 1), (5, 70, 32, 64)])
def test_selector_sets_and_es_match_numpy(R, n, d, s):
    rng = np.random.default_rng(R * 100 + n + s)
    rows = R * 2
    L = (rng.normal(size=(rows, n)) * rng.uniform(0.5, 3, size=(rows, 1))).astype(np.float32)
    L[:, 0] += 5
    L[:, -5:] += 1.0  # recency bump
    L[0, 10:14] = L[0, 20]  # equal logits across pages
    V = rng.normal(size=(2, n, d)).astype(np.float32)
    b = rows_batch(L, V, np.full((rows, 1), s), R=R)
    o = oracle.selector_audit(b, [s])
    want, P = numpy_sets(L, V, R, s)
    for r in range(rows):
        Vg = V[r // R].astype(np.float64)
        for sel in range(5):
            m = want[r][sel]
            got = np.array([(int(o["bits"][r, sel, 0, j >> 5]) >> (j & 31)) & 1 for j in range(n)], bool)
            np.testing.assert_array_equal(got, m, err_msg=f"row {r} rule {sel}")
            if m.any():
                assert o["es"][r, sel, 0] == pytest.approx(es_of(P[r], Vg, m), rel=1e-10)
            else:
                assert np.isnan(o["es"][r, sel, 0])
        # set sizes: s keys for the first three rules; whole pages for Quest
        for sel in range(3):
            assert want[r][sel].sum() == s
        Pq = max(2, s // 4)
        assert want[r][3].sum() <= (s // Pq) * Pq


def test_streamingllm_ignores_the_logits():
    rng = np.random.default_rng(1)
    V = rng.normal(size=(1, 50, 32)).astype(np.float32)
    a = oracle.selector_audit(rows_batch(rng.normal(size=(1, 50)).astype(np.float32), V, [[8]]), [8])
    b = oracle.selector_audit(rows_batch(rng.normal(size=(1, 50)).astype(np.float32) * 3, V, [[8]]), [8])
    np.testing.assert_array_equal(a["bits"][:, 0], b["bits"][:, 0])
    bits = a["bits"][0, 0, 0]
    kept = [j for j in range(50) if (int(bits[j >> 5]) >> (j & 31)) & 1]
    assert kept == [0, 1, 2, 3, 46, 47, 48, 49]
