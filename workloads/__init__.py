"""Seeded synthetic inputs for forced-weight subset evaluation.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic (no softmax, no selection, no sums).  Both the CUDA library
and the CPU oracle are fed from here, never from each other.

The paper measures on attention rows captured from frozen language models and
on long-context benchmarks (Sec. 2.2, Sec. 4, App. B).  None of those models or
datasets exist here, so the generators below produce stand-ins with the same
shapes and the same qualitative structure: a large attention sink at position
0, a recency bump over the last few hundred keys, per-row temperatures, values
that are shared by the rows of one KV head or GQA group, and heavy-tailed
importance scores for the cache allocator.

Layout ("row batch"): rows come in groups of ``R`` consecutive rows that share
one value block and one length.  Group ``g`` has ``n[g]`` keys; its logits are
``R`` rows of ``n[g]`` floats stored contiguously from ``logit_off[g]``; its
values are an ``n[g] x d`` row-major block from ``v_off[g]``.  Budgets ``k`` are
``[rows][nb]`` int32.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Any, List, Sequence

import numpy as np

# --------------------------------------------------------------------------
# backends: numpy (host) and torch (device).  Same distributions, different
# streams; a test feeds ONE generated batch to both the kernels and the oracle.
# --------------------------------------------------------------------------


class _NumpyRng:
    name = "numpy"

    def __init__(self, seed: int):
        self.g = np.random.Generator(np.random.Philox(seed))

    def normal(self, shape, std=1.0):
        return (self.g.standard_normal(shape, dtype=np.float32) * np.float32(std)).astype(np.float32)

    def uniform(self, shape, lo, hi):
        return self.g.uniform(lo, hi, size=shape).astype(np.float32)

    def gumbel(self, shape):
        # -log(-log U), U in (0, 1) open
        u = self.g.random(shape, dtype=np.float64)
        u = np.clip(u, 1e-300, 1.0 - 2.0 ** -53)
        return (-np.log(-np.log(u))).astype(np.float32)

    # plumbing
    def f32(self, a):
        return np.asarray(a, dtype=np.float32)

    def arange(self, n):
        return np.arange(n, dtype=np.float32)

    def exp(self, a):
        return np.exp(a).astype(np.float32)

    def cat(self, parts):
        return np.concatenate([np.ravel(p) for p in parts]) if parts else np.zeros(0, np.float32)

    def to_bf16(self, a):
        return f32_to_bf16_bits(np.asarray(a, dtype=np.float32))

    def i32(self, a):
        return np.asarray(a, dtype=np.int32)

    def i64(self, a):
        return np.asarray(a, dtype=np.int64)


class _TorchRng:
    name = "torch"

    def __init__(self, seed: int, device: str):
        import torch

        self.torch = torch
        self.device = device
        self.g = torch.Generator(device=device)
        self.g.manual_seed(seed)

    def normal(self, shape, std=1.0):
        t = self.torch.randn(shape, generator=self.g, device=self.device, dtype=self.torch.float32)
        return t.mul_(std) if std != 1.0 else t

    def uniform(self, shape, lo, hi):
        t = self.torch.rand(shape, generator=self.g, device=self.device, dtype=self.torch.float32)
        return t.mul_(hi - lo).add_(lo)

    def gumbel(self, shape):
        u = self.torch.rand(shape, generator=self.g, device=self.device, dtype=self.torch.float64)
        u = u.clamp_(1e-300, 1.0 - 2.0 ** -53)
        return (-(-u.log()).log()).float()

    def f32(self, a):
        return self.torch.as_tensor(a, dtype=self.torch.float32, device=self.device)

    def arange(self, n):
        return self.torch.arange(n, dtype=self.torch.float32, device=self.device)

    def exp(self, a):
        return self.torch.exp(a)

    def cat(self, parts):
        return self.torch.cat([p.reshape(-1) for p in parts])

    def to_bf16(self, a):
        return a.to(self.torch.bfloat16)

    def i32(self, a):
        return self.torch.as_tensor(np.asarray(a, dtype=np.int32), device=self.device)

    def i64(self, a):
        return self.torch.as_tensor(np.asarray(a, dtype=np.int64), device=self.device)


def make_rng(seed: int, backend: str = "numpy", device: str = "cuda"):
    if backend == "numpy":
        return _NumpyRng(seed)
    if backend == "torch":
        return _TorchRng(seed, device)
    raise ValueError(backend)


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even float32 -> bfloat16, returned as uint16 bit patterns."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    nan = np.isnan(a)
    out = rounded.astype(np.uint16)
    out[nan] = 0x7FC0
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


# --------------------------------------------------------------------------
# containers
# --------------------------------------------------------------------------


@dataclasses.dataclass
class RowBatch:
    """Groups of ``rows_per_group`` rows that share a value block and a length."""

    rows_per_group: int
    d: int
    n: Any            # int32 [G]
    logits: Any       # float32, flat
    logit_off: Any    # int64 [G]
    v: Any            # float32 or bf16 (uint16 bits in numpy), flat
    v_off: Any        # int64 [G]
    v_dtype: str      # "f32" | "bf16"
    k: Any            # int32 [rows][nb]
    nb: int
    n_host: np.ndarray  # int32 [G], always on the host
    name: str = ""

    @property
    def num_groups(self) -> int:
        return int(len(self.n_host))

    @property
    def num_rows(self) -> int:
        return self.num_groups * self.rows_per_group

    @property
    def max_n(self) -> int:
        return int(self.n_host.max()) if len(self.n_host) else 0


@dataclasses.dataclass
class CacheBatch:
    """ContourKV input: per-cell importance scores and the K/V cache."""

    cells: int
    T: int
    d: int
    scores: Any  # float32 [cells][T]
    K: Any       # bf16 [cells][T][d]
    V: Any       # bf16 [cells][T][d]
    floor: int
    total_budget: int
    uniform_s: int


def _assemble(rng, groups, rows_per_group, d, v_dtype, budgets_per_group, name, lay_v=True):
    """groups: list of (n, logits[R][n], v[n][d]) in backend arrays."""
    n_host = np.array([g[0] for g in groups], dtype=np.int32)
    lo = np.zeros(len(groups), dtype=np.int64)
    vo = np.zeros(len(groups), dtype=np.int64)
    acc_l = 0
    acc_v = 0
    for i, (n, _, _) in enumerate(groups):
        lo[i] = acc_l
        vo[i] = acc_v
        acc_l += rows_per_group * n
        acc_v += n * d
    logits = rng.cat([g[1] for g in groups])
    v = rng.cat([g[2] for g in groups])
    if v_dtype == "bf16":
        v = rng.to_bf16(v)
    k = np.asarray(budgets_per_group, dtype=np.int32)
    k = np.repeat(k, rows_per_group, axis=0)
    nb = k.shape[1]
    return RowBatch(
        rows_per_group=rows_per_group, d=d, n=rng.i32(n_host), logits=logits,
        logit_off=rng.i64(lo), v=v, v_off=rng.i64(vo), v_dtype=v_dtype,
        k=rng.i32(k), nb=nb, n_host=n_host, name=name)


# --------------------------------------------------------------------------
# the five workloads
# --------------------------------------------------------------------------

# Exact best-subset toy: 256 rows, n=20, k=5, d=64, logits ~ N(0, 2^2) with a
# +6 sink at index 0, V ~ N(0, 1) per row, seed 0.
def exact_toy(seed: int = 0, rows: int = 256, n: int = 20, k: int = 5, d: int = 64,
              backend: str = "numpy", device: str = "cuda") -> RowBatch:
    rng = make_rng(seed, backend, device)
    groups = []
    for _ in range(rows):
        l = rng.normal((1, n), 2.0)
        l[0, 0] = l[0, 0] + 6.0
        v = rng.normal((n, d))
        groups.append((n, l, v))
    return _assemble(rng, groups, 1, d, "f32", [[k]] * rows, "exact_toy_n20_k5_d64")


# Exact enumeration at measurement scale: 168,192 rows in five groups with
# d = 64,128,128,128,64, n=24, k=6; logits Gumbel(0,1)*tau, tau ~ U[0.5,3] per
# row, +6 sink at index 0; V ~ N(0,1) per row.  The per-group row counts follow
# the paper's per-family instance counts (six rows per head, every layer, three
# documents, four budgets; plus the 7B arm).
ENUM_GROUPS = ((24192, 64), (36864, 128), (18432, 128), (32256, 128), (56448, 64))


def exact_enum(seed: int = 0, rows_scale: float = 1.0, n: int = 24, k: int = 6,
               backend: str = "numpy", device: str = "cuda",
               groups: Sequence = ENUM_GROUPS) -> List[RowBatch]:
    out = []
    for gi, (rows, d) in enumerate(groups):
        rows = max(1, int(round(rows * rows_scale)))
        rng = make_rng(seed * 1000 + 17 * gi + 1, backend, device)
        tau = rng.uniform((rows, 1), 0.5, 3.0)
        l = rng.gumbel((rows, n)) * tau
        l[:, 0] = l[:, 0] + 6.0
        v = rng.normal((rows, n, d))
        out.append(_batch_rows_own_v(rng, l, v, n, d, k, f"exact_enum_d{d}"))
    return out


# Adversarial inputs for the exact search (n <= 32), each a stress on a
# different part of it:
#   flat      n=24, k=6, d=64: logits Gumbel*0.3 and no sink, so many subsets
#             have es close to the best and few bounds exclude anything;
#   near_dup  n=24, k=6, d=64: values = one point + eps*N(0,1) (eps cycling
#             through 1e-2, 1e-3, 1e-4), logits as in exact_enum: es of every
#             subset within a few eps of the others;
#   planted   n=32, k=4, d=32: uniform logits and integer points in the first
#             dimension (the rest 0), with one random 4-subset planted so that
#             its mean equals the mean of all 32 points -- es = 0 exactly, and
#             every other 4-subset with that mean ties with it (App. A.2 builds
#             its hardness instances the same way);
#   planted_half  n=16, k=8, d=32: App. A.2's construction itself, uniform
#             masses and a planted split of the points into two halves of
#             equal sum (es = 0 exactly for the planted half, usually many
#             more).
# Uniform masses over 16 or 32 keys and integer points keep every quantity a
# short binary fraction, so es = 0 holds exactly in floating point too.
ADVERSARIAL_KINDS = ("flat", "near_dup", "planted", "planted_half")


def exact_adversarial(kind: str, rows: int = 512, seed: int = 0) -> RowBatch:
    rng = _NumpyRng(seed * 1000 + 300 + ADVERSARIAL_KINDS.index(kind))
    if kind == "flat":
        n, k, d = 24, 6, 64
        l = rng.gumbel((rows, n)) * np.float32(0.3)
        v = rng.normal((rows, n, d))
    elif kind == "near_dup":
        n, k, d = 24, 6, 64
        tau = rng.uniform((rows, 1), 0.5, 3.0)
        l = rng.gumbel((rows, n)) * tau
        l[:, 0] += 6.0
        eps = np.array([1e-2, 1e-3, 1e-4], np.float32)[np.arange(rows) % 3][:, None, None]
        v = (rng.normal((rows, 1, d)) + eps * rng.normal((rows, n, d))).astype(np.float32)
    elif kind in ("planted", "planted_half"):
        n, k, d = (32, 4, 32) if kind == "planted" else (16, 8, 32)
        l = np.zeros((rows, n), np.float32)
        w = np.floor(rng.uniform((rows, n), -8.0, 9.0)).astype(np.int64)
        v = np.zeros((rows, n, d), np.float32)
        for r in range(rows):
            perm = rng.g.permutation(n)
            A, out = perm[:k], perm[k:]
            # make sum(all) = (n / k) * sum(A) by moving one point outside A
            w[r, out[0]] += (n // k) * w[r, A].sum() - w[r].sum()
            v[r, :, 0] = w[r]
    else:
        raise ValueError(kind)
    return _batch_rows_own_v(rng, l.astype(np.float32), v.astype(np.float32), n, d, k, f"adversarial_{kind}")


def _batch_rows_own_v(rng, l, v, n, d, k, name):
    """Each row is its own group (R = 1): rows are contiguous, V blocks too."""
    rows = l.shape[0]
    n_host = np.full(rows, n, dtype=np.int32)
    lo = np.arange(rows, dtype=np.int64) * n
    vo = np.arange(rows, dtype=np.int64) * (n * d)
    kk = np.full((rows, 1), k, dtype=np.int32) if np.isscalar(k) else np.asarray(k, np.int32)
    return RowBatch(rows_per_group=1, d=d, n=rng.i32(n_host), logits=l.reshape(-1),
                    logit_off=rng.i64(lo), v=v.reshape(-1), v_off=rng.i64(vo), v_dtype="f32",
                    k=rng.i32(kk), nb=kk.shape[1], n_host=n_host, name=name)


def _sink_recency(rng, n):
    i = rng.arange(n)
    bump = rng.exp(-(float(n - 1) - i) / 256.0) * 2.0
    return bump


# Long-row top-k gap + swap: 8 KV heads x 512 query rows, n=32,768, d=128,
# V bf16 ~ N(0,1) shared per head, logits N(0,1.5^2) + 8*[i=0] +
# 2*exp(-(n-1-i)/256); budgets k/n in {1/16, 1/8, 1/4}.
def long_rows(seed: int = 0, heads: int = 8, rows_per_head: int = 512, n: int = 32768,
              d: int = 128, fracs=(1 / 16, 1 / 8, 1 / 4), backend: str = "numpy",
              device: str = "cuda") -> RowBatch:
    rng = make_rng(seed * 1000 + 3, backend, device)
    bump = _sink_recency(rng, n)
    groups = []
    for _ in range(heads):
        l = rng.normal((rows_per_head, n), 1.5) + bump
        l[:, 0] = l[:, 0] + 8.0
        v = rng.normal((n, d))
        groups.append((n, l, v))
    ks = [max(1, int(round(f * n))) for f in fracs]
    return _assemble(rng, groups, rows_per_head, d, "bf16", [ks] * heads,
                     f"long_rows_n{n}_d{d}")


# ContourKV allocation + ragged compaction: 32 layers x 8 KV heads = 256 cells,
# T=32,768 tokens, d=128; K, V bf16 ~ N(0,1); scores lognormal(0, sigma_h),
# sigma_h ~ U[0.5, 2.5] per cell; global budget = 1/8 of the tokens; recency
# floor of 32 positions per cell.
def contour_cache(seed: int = 0, cells: int = 256, T: int = 32768, d: int = 128,
                  floor: int = 32, budget_frac: float = 1 / 8, backend: str = "numpy",
                  device: str = "cuda", with_kv: bool = True) -> CacheBatch:
    rng = make_rng(seed * 1000 + 4, backend, device)
    sigma = rng.uniform((cells, 1), 0.5, 2.5)
    z = rng.normal((cells, T))
    scores = rng.exp(z * sigma)
    if with_kv:
        K = rng.to_bf16(rng.normal((cells, T, d)))
        V = rng.to_bf16(rng.normal((cells, T, d)))
    else:
        K = V = None
    total = int(round(cells * T * budget_frac))
    return CacheBatch(cells=cells, T=T, d=d, scores=scores, K=K, V=V, floor=floor,
                      total_budget=total, uniform_s=total // cells)


# Window queries for the observation-window score: the last w query rows of
# every cell of a contour_cache, bf16 ~ N(0, 1) like its keys (w = 32, the
# largest SnapKV window of App. C).
def window_queries(seed: int = 0, cells: int = 256, w: int = 32, d: int = 128, backend: str = "numpy",
                   device: str = "cuda"):
    rng = make_rng(seed * 1000 + 5, backend, device)
    return rng.to_bf16(rng.normal((cells, w, d)))


# Mixed-profile sweep: 168,192 rows from five head profiles (rows, d, n),
# GQA groups of 4 rows sharing a bf16 V block, logits tau*N(0,1) + sink +8 +
# recency bump, tau ~ U[0.3, 4] per row, budget per group
# {1/32, 1/16, 1/8, 1/4}[g mod 4] * n.  Profiles with equal d are returned as
# one ragged batch.
MIXED_PROFILES = (("A", 36864, 64, 1024), ("B", 24192, 128, 4096), ("C", 32256, 64, 4096),
                  ("D", 56448, 64, 8192), ("E", 18432, 128, 16384))


def mixed_profiles(seed: int = 0, rows_scale: float = 1.0, gqa: int = 4,
                   backend: str = "numpy", device: str = "cuda",
                   profiles: Sequence = MIXED_PROFILES) -> List[RowBatch]:
    fr = (1 / 32, 1 / 16, 1 / 8, 1 / 4)
    by_d = {}
    for pi, (pname, rows, d, n) in enumerate(profiles):
        rng = make_rng(seed * 1000 + 50 + pi, backend, device)
        ngroups = max(1, int(round(rows * rows_scale / gqa)))
        bump = _sink_recency(rng, n)
        gl = by_d.setdefault(d, ([], [], rng))
        for g in range(ngroups):
            tau = rng.uniform((gqa, 1), 0.3, 4.0)
            l = rng.normal((gqa, n)) * tau + bump
            l[:, 0] = l[:, 0] + 8.0
            v = rng.normal((n, d))
            gl[0].append((n, l, v))
            gl[1].append([max(1, int(round(fr[g % 4] * n)))])
    out = []
    for d, (groups, budgets, rng) in sorted(by_d.items()):
        out.append(_assemble(rng, groups, gqa, d, "bf16", budgets, f"mixed_d{d}"))
    return out


def total_subsets(n: int, k: int) -> int:
    return math.comb(n, k)
