"""fp64 CPU oracle for forced-weight subset evaluation -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline and
reference legs may import this package.  The product path (the CUDA library and
its binding) never does, and the oracle never imports the product: the two
share nothing but the seeded generators in ``workloads``.

The arithmetic lives in ``fw_oracle.c`` (plain C, double precision, straight
from the paper's definitions).  This module compiles it with gcc and marshals
numpy arrays into it.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fw_oracle.c")
_SO = os.path.join(_HERE, "_fw_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle shared library (gcc, OpenMP, -O2)."""
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _SO)
    return _SO


class _Rows(C.Structure):
    _fields_ = [("num_groups", C.c_int64), ("rows_per_group", C.c_int32), ("d", C.c_int32),
                ("logits", C.c_void_p), ("logit_off", C.c_void_p), ("n", C.c_void_p),
                ("v", C.c_void_p), ("v_off", C.c_void_p), ("v_dtype", C.c_int32)]


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = C.CDLL(_SO)
            vp = C.c_void_p
            L.orc_eval_instance.argtypes = [C.c_int, C.c_int, vp, vp, vp, vp, vp, vp]
            L.orc_dense_and_topk_gap.argtypes = [C.POINTER(_Rows), C.c_int, vp] + [vp] * 9 + [C.c_int, vp]
            L.orc_swap_refine.argtypes = [C.POINTER(_Rows), C.c_int, vp, C.c_int, C.c_int] + [vp] * 8
            L.orc_best_subset.argtypes = [C.POINTER(_Rows), vp, vp, vp, vp, C.c_int, vp, vp]
            L.orc_colex_rank.argtypes = [C.c_int, vp]
            L.orc_colex_rank.restype = C.c_uint64
            L.orc_contour_alloc.argtypes = [vp, C.c_int, C.c_int, C.c_int, C.c_int64, C.c_int,
                                            vp, vp, vp, vp, vp, vp]
            L.orc_contour_alloc_capped.argtypes = [vp, C.c_int, C.c_int, C.c_int, C.c_int64, C.c_int, C.c_int,
                                                   vp, vp, vp, vp, vp, vp]
            L.orc_ragged_compact_to.argtypes = [vp, vp, C.c_int, C.c_int, C.c_int, vp, vp, vp, vp, vp, vp, vp]
            L.orc_ragged_append.argtypes = [vp, vp, vp, vp, vp, vp, vp, C.c_int, C.c_int, C.c_int, vp]
            L.orc_window_score.argtypes = [vp, vp, C.c_int, C.c_int, C.c_int, C.c_int, C.c_double, C.c_int, vp, vp]
            L.orc_selector_audit.argtypes = [C.POINTER(_Rows), C.c_int, vp, C.c_int, vp, vp, C.c_int, vp, vp]
            L.orc_ragged_compact.argtypes = [vp, vp, C.c_int, C.c_int, C.c_int, C.c_int, vp, vp, vp, vp]
            L.orc_group_vote.argtypes = [C.POINTER(_Rows), C.c_int, vp, C.c_int, vp, vp, vp, vp, C.c_int,
                                         vp, vp, vp]
            L.orc_pool_best_subset.argtypes = [C.POINTER(_Rows), C.c_int, vp, vp, C.c_int, C.c_int64,
                                               vp, vp, vp, vp, vp, vp, vp]
            L.orc_candidate_set.argtypes = [C.POINTER(_Rows), C.c_int64, C.c_int, C.c_int, vp, vp]
            L.orc_swap_scores.argtypes = [C.POINTER(_Rows), C.c_int64, vp, vp, C.c_int, vp, vp]
            L.orc_num_threads.restype = C.c_int
            _lib = L
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _host(a, dtype=None):
    """numpy view of a host array or a torch tensor (copied to the host)."""
    if hasattr(a, "detach"):
        import torch

        t = a.detach()
        if t.dtype == torch.bfloat16:
            t = t.view(torch.int16)
        a = t.cpu().numpy()
        if a.dtype == np.int16:
            a = a.view(np.uint16)
    a = np.ascontiguousarray(a)
    if dtype is not None:
        a = np.ascontiguousarray(a, dtype=dtype)
    return a


class HostRows:
    """A row batch on the host in the oracle's layout (keeps arrays alive)."""

    def __init__(self, batch):
        self.R = int(batch.rows_per_group)
        self.d = int(batch.d)
        self.n = _host(batch.n_host, np.int32)
        self.logits = _host(batch.logits, np.float32)
        self.logit_off = _host(batch.logit_off, np.int64)
        self.v = _host(batch.v)
        self.v_off = _host(batch.v_off, np.int64)
        if batch.v_dtype == "bf16":
            self.v = self.v.view(np.uint16)
            self.v_dtype = 1
        elif self.v.dtype == np.float64:
            self.v_dtype = 2
        else:
            self.v = np.ascontiguousarray(self.v, np.float32)
            self.v_dtype = 0
        self.k = _host(batch.k, np.int32)
        self.nb = int(self.k.shape[1])
        self.num_rows = len(self.n) * self.R
        self.max_n = int(self.n.max())
        self.c = _Rows(len(self.n), self.R, self.d, _p(self.logits).value, _p(self.logit_off).value,
                       _p(self.n).value, _p(self.v).value, _p(self.v_off).value, self.v_dtype)


def eval_instance(p, v, in_A):
    """Definition 2.1 / Lemma 2.1 quantities for one instance given by masses p,
    points v ([n][d]) and a kept-set mask.  Returns dict."""
    p = np.ascontiguousarray(p, np.float64)
    v = np.ascontiguousarray(np.atleast_2d(v).reshape(len(p), -1), np.float64)
    m = np.ascontiguousarray(in_A, np.uint8)
    n, d = v.shape
    mu = np.zeros(d)
    mA = np.zeros(d)
    out = np.zeros(6)
    st = lib().orc_eval_instance(n, d, _p(p), _p(v), _p(m), _p(mu), _p(mA), _p(out))
    assert st == 0, st
    return dict(mu=mu, m_A=mA, kept_mass=out[0], dropped=out[1], gap=out[2], phi=out[3],
                form1=out[4], form2=out[5])


def dense_and_topk_gap(batch, words=None):
    """a1-a4 on every row and budget.  Returns dict of numpy arrays (fp64)."""
    H = batch if isinstance(batch, HostRows) else HostRows(batch)
    rows, nb, d = H.num_rows, H.nb, H.d
    words = words or (H.max_n + 31) // 32
    out = dict(o=np.zeros((rows, d)), o_kept=np.zeros((rows, nb, d)), gap=np.zeros((rows, nb)),
               dropped=np.zeros((rows, nb)), kept_mass=np.zeros((rows, nb)), phi=np.zeros((rows, nb)),
               form1=np.zeros((rows, nb)), form2=np.zeros((rows, nb)),
               kept_bits=np.zeros((rows, nb, words), np.uint32), status=np.zeros(rows, np.int32))
    st = lib().orc_dense_and_topk_gap(C.byref(H.c), nb, _p(H.k), _p(out["o"]), _p(out["o_kept"]),
                                      _p(out["gap"]), _p(out["dropped"]), _p(out["kept_mass"]),
                                      _p(out["phi"]), _p(out["form1"]), _p(out["form2"]),
                                      _p(out["kept_bits"]), words, _p(out["status"]))
    assert st == 0, st
    return out


def swap_refine(batch, E, max_swaps=64):
    H = batch if isinstance(batch, HostRows) else HostRows(batch)
    rows, nb = H.num_rows, H.nb
    out = dict(n_swaps=np.zeros((rows, nb), np.int32),
               swap_out=np.full((rows, nb, max_swaps), -1, np.int32),
               swap_in=np.full((rows, nb, max_swaps), -1, np.int32),
               refined_gap=np.zeros((rows, nb)), topk_gap=np.zeros((rows, nb)),
               capped=np.zeros((rows, nb), np.int32), margin=np.zeros((rows, nb)),
               pool_margin=np.zeros((rows, nb)))
    st = lib().orc_swap_refine(C.byref(H.c), nb, _p(H.k), int(E), int(max_swaps),
                               _p(out["n_swaps"]), _p(out["swap_out"]), _p(out["swap_in"]),
                               _p(out["refined_gap"]), _p(out["topk_gap"]), _p(out["capped"]),
                               _p(out["margin"]), _p(out["pool_margin"]))
    assert st == 0, st
    return out


def best_subset(batch):
    H = batch if isinstance(batch, HostRows) else HostRows(batch)
    rows = H.num_rows
    kk = np.ascontiguousarray(H.k[:, 0], np.int32)
    kmax = int(kk.max())
    out = dict(best_rank=np.zeros(rows, np.uint64), best_gap=np.zeros(rows),
               best_idx=np.full((rows, kmax), -1, np.int32), second_gap=np.zeros(rows),
               topk_gap=np.zeros(rows))
    st = lib().orc_best_subset(C.byref(H.c), _p(kk), _p(out["best_rank"]), _p(out["best_gap"]),
                               _p(out["best_idx"]), kmax, _p(out["second_gap"]), _p(out["topk_gap"]))
    assert st == 0, st
    return out


def pool_best_subset(batch, E, max_subsets=1 << 24):
    """f2, ES_pool (Definition 2.2): the exact best size-k subset of the
    candidate set (top-mass set + E extras of largest single-key error) for
    every row and budget slot.  E: extras per budget slot (length nb).
    Returns dict of numpy arrays (best_gap, best_idx, topk_gap, second_gap,
    n_subsets, pool_margin, status) and the call status."""
    H = batch if isinstance(batch, HostRows) else HostRows(batch)
    rows, nb = H.num_rows, H.nb
    E = np.ascontiguousarray(np.broadcast_to(np.asarray(E, np.int32), (nb,)), np.int32)
    kmax = int(H.k.max())
    out = dict(best_gap=np.zeros((rows, nb)), best_idx=np.full((rows, nb, kmax), -1, np.int32),
               topk_gap=np.zeros((rows, nb)), second_gap=np.zeros((rows, nb)),
               n_subsets=np.zeros((rows, nb), np.int64), pool_margin=np.zeros((rows, nb)),
               status=np.zeros(rows, np.int32))
    st = lib().orc_pool_best_subset(C.byref(H.c), nb, _p(H.k), _p(E), kmax, int(max_subsets),
                                    _p(out["best_gap"]), _p(out["best_idx"]), _p(out["topk_gap"]),
                                    _p(out["second_gap"]), _p(out["n_subsets"]), _p(out["pool_margin"]),
                                    _p(out["status"]))
    out["call_status"] = st
    return out


def candidate_set(batch, row, k, E):
    """Definition 2.2's candidate set of one row at budget k: (pool key indices
    ascending, pool-boundary margin)."""
    H = batch if isinstance(batch, HostRows) else HostRows(batch)
    g = int(row) // H.R
    pool = np.zeros(int(H.n[g]) + 1, np.int32)
    margin = np.zeros(1)
    P = lib().orc_candidate_set(C.byref(H.c), int(row), int(k), int(E), _p(pool), _p(margin))
    assert P >= 0, P
    return pool[:P].copy(), float(margin[0])


def swap_scores(batch, row, in_A, add):
    """One balancing round scored in full: es(A - i + j) for every kept key i
    (ascending; rows of the result) and every j in `add` (columns), and es(A).
    in_A: boolean mask over the row's keys."""
    H = batch if isinstance(batch, HostRows) else HostRows(batch)
    m = np.ascontiguousarray(in_A, np.uint8)
    add = np.ascontiguousarray(add, np.int32)
    na = int(m.sum())
    out = np.zeros((na, len(add)))
    cur = np.zeros(1)
    got = lib().orc_swap_scores(C.byref(H.c), int(row), _p(m), _p(add), len(add), _p(out), _p(cur))
    assert got == na, got
    return out, float(cur[0])


def group_vote(batch, s, eval_rows=None, words=None):
    """f1, the group vote: one kept set per group of rows (the s keys of
    largest summed mass G), every row scored against it.  s: [groups][nb]
    budgets.  eval_rows: optional boolean [rows]; rows left out are not scored
    (their gap / dropped stay 0).  Returns dict of numpy arrays."""
    H = batch if isinstance(batch, HostRows) else HostRows(batch)
    s = np.ascontiguousarray(_host(s), np.int32)
    if s.ndim == 1:
        s = s[:, None].copy()
    G, nb = s.shape
    assert G == len(H.n)
    words = words or (H.max_n + 31) // 32
    ev = None if eval_rows is None else np.ascontiguousarray(eval_rows, np.uint8)
    out = dict(mass=np.zeros((G, H.max_n)), margin=np.zeros((G, nb)),
               bits=np.zeros((G, nb, words), np.uint32), gap=np.zeros((H.num_rows, nb)),
               dropped=np.zeros((H.num_rows, nb)), status=np.zeros(H.num_rows, np.int32))
    st = lib().orc_group_vote(C.byref(H.c), nb, _p(s), H.max_n, _p(ev), _p(out["mass"]), _p(out["margin"]),
                              _p(out["bits"]), words, _p(out["gap"]), _p(out["dropped"]), _p(out["status"]))
    assert st == 0, st
    return out


def colex_rank(combo):
    c = np.ascontiguousarray(sorted(combo), np.int32)
    return int(lib().orc_colex_rank(len(c), _p(c)))


def contour_alloc(scores, floor, total_budget, uniform_s):
    s = _host(scores, np.float32)
    cells, T = s.shape
    out = dict(counts=np.zeros(cells, np.int32), offsets=np.zeros(cells + 1, np.int64),
               kept_pos=np.zeros(int(total_budget), np.int32), tau=np.zeros(1, np.float32),
               dropped_uniform=np.zeros(cells), dropped_alloc=np.zeros(cells))
    st = lib().orc_contour_alloc(_p(s), cells, T, int(floor), int(total_budget), int(uniform_s),
                                 _p(out["counts"]), _p(out["offsets"]), _p(out["kept_pos"]),
                                 _p(out["tau"]), _p(out["dropped_uniform"]), _p(out["dropped_alloc"]))
    out["status"] = st
    out["tau"] = float(out["tau"][0])
    return out


def contour_alloc_capped(scores, floor, total_budget, uniform_s, cap):
    """f3: the ContourKV allocation truncated to `cap` entries per cell."""
    s = _host(scores, np.float32)
    cells, T = s.shape
    out = dict(counts=np.zeros(cells, np.int32), offsets=np.zeros(cells + 1, np.int64),
               kept_pos=np.full(int(total_budget), -1, np.int32), tau=np.zeros(1, np.float32),
               dropped_uniform=np.zeros(cells), dropped_alloc=np.zeros(cells))
    st = lib().orc_contour_alloc_capped(_p(s), cells, T, int(floor), int(total_budget), int(uniform_s), int(cap),
                                        _p(out["counts"]), _p(out["offsets"]), _p(out["kept_pos"]),
                                        _p(out["tau"]), _p(out["dropped_uniform"]), _p(out["dropped_alloc"]))
    out["status"] = st
    out["tau"] = float(out["tau"][0])
    return out


def ragged_compact(K, V, offsets, kept_pos):
    K = _host(K)
    V = _host(V)
    cells, T, d = K.shape
    off = np.ascontiguousarray(offsets, np.int64)
    kp = np.ascontiguousarray(kept_pos, np.int32)
    tot = int(off[-1])
    Ko = np.zeros((tot, d), K.dtype)
    Vo = np.zeros((tot, d), V.dtype)
    st = lib().orc_ragged_compact(_p(K), _p(V), cells, T, d, K.dtype.itemsize, _p(off), _p(kp),
                                  _p(Ko), _p(Vo))
    assert st == 0, st
    return Ko, Vo


def ragged_compact_to(K, V, offsets, kept_pos, base, capacity, K_store, V_store):
    """f3: kept rows into a store with room per cell; K_store / V_store (numpy,
    [rows][d]) are updated in place.  Returns the per-cell status."""
    K, V = _host(K), _host(V)
    cells, T, d = K.shape
    off = np.ascontiguousarray(offsets, np.int64)
    kp = np.ascontiguousarray(kept_pos, np.int32)
    b = np.ascontiguousarray(base, np.int64)
    cap = np.ascontiguousarray(capacity, np.int32)
    status = np.zeros(cells, np.int32)
    assert K_store.flags.c_contiguous and V_store.flags.c_contiguous
    st = lib().orc_ragged_compact_to(_p(K), _p(V), cells, T, d * K.dtype.itemsize, _p(off), _p(kp), _p(b), _p(cap),
                                     _p(K_store), _p(V_store), _p(status))
    assert st == 0, st
    return status


def ragged_append(K_store, V_store, base, capacity, counts, new_K, new_V):
    """f3: decode-time append of new_K / new_V ([cells][m][d]); counts (numpy
    int32) and the stores are updated in place.  Returns the per-cell status."""
    new_K, new_V = _host(new_K), _host(new_V)
    cells, m, d = new_K.shape
    b = np.ascontiguousarray(base, np.int64)
    cap = np.ascontiguousarray(capacity, np.int32)
    assert counts.dtype == np.int32 and counts.flags.c_contiguous
    status = np.zeros(cells, np.int32)
    st = lib().orc_ragged_append(_p(K_store), _p(V_store), _p(b), _p(cap), _p(counts), _p(new_K), _p(new_V), cells, m,
                                 d * new_K.dtype.itemsize, _p(status))
    assert st == 0, st
    return status


def window_score(Qw, K, scale, pool=7):
    """f3: the observation-window score.  Qw: bf16 bits (uint16) [cells][w][d],
    K: [cells][T][d].  Returns (scores, votes), fp64 [cells][T]."""
    Qw = np.ascontiguousarray(_host(Qw)).view(np.uint16)
    K = np.ascontiguousarray(_host(K)).view(np.uint16)
    cells, w, d = Qw.shape
    T = K.shape[1]
    scores = np.zeros((cells, T))
    votes = np.zeros((cells, T))
    st = lib().orc_window_score(_p(Qw), _p(K), cells, T, d, w, float(scale), int(pool), _p(scores), _p(votes))
    assert st == 0, st
    return scores, votes


SELECTORS = ("streamingllm", "h2o", "snapkv", "quest", "quest16")


def selector_audit(batch, s):
    """f4: the deployed selectors' kept sets and their es (App. C settings).
    s: budgets (nb).  Returns es [rows][5][nb], bits [rows][5][nb][words],
    G [groups][max_n], pooled [groups][nb][max_n]."""
    H = batch if isinstance(batch, HostRows) else HostRows(batch)
    s = np.ascontiguousarray(np.atleast_1d(s), np.int32)
    nb = len(s)
    words = (H.max_n + 31) // 32
    G = len(H.n)
    out = dict(es=np.zeros((H.num_rows, 5, nb)), bits=np.zeros((H.num_rows, 5, nb, words), np.uint32),
               G=np.zeros((G, H.max_n)), pooled=np.zeros((G, nb, H.max_n)))
    st = lib().orc_selector_audit(C.byref(H.c), nb, _p(s), H.max_n, _p(out["es"]), _p(out["bits"]), words,
                                  _p(out["G"]), _p(out["pooled"]))
    assert st == 0, st
    return out


def num_threads() -> int:
    return int(lib().orc_num_threads())
