"""GPU parity for the group vote (one kept set per KV head by the mass summed
over the head's query rows, every row scored against it).

Sets: the CUDA path sums the masses in fp32, the oracle in fp64.  Where the
oracle's relative margin between the last kept and the first dropped summed
mass is at least VOTE_MARGIN, the sets must be equal bit for bit.  Below it the
CUDA set must still hold exactly s keys, every key whose oracle mass is above
the boundary by more than VOTE_MARGIN and none below it by more than that; its
gaps are then compared with the oracle's es of that same set.  VOTE_MARGIN
covers the fp32 error of a summed mass: each p_j carries a few ulp (exp, the
division by Z, Z's own rounding) and a sum over up to 512 rows adds at most
512 ulp, about 3e-5, in the worst case.
"""
import numpy as np
import pytest

import oracle
import workloads
from tests.parity import assert_close, np_
from tests.test_gpu_small import rows_batch

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

VOTE_MARGIN = 1e-4


@pytest.fixture(scope="module")
def fw():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_25230_gb300 import fw as _fw

    return _fw


def unpack(words, n):
    w = np.ascontiguousarray(words, np.uint32)
    return np.unpackbits(w.view(np.uint8), bitorder="little")[:n].astype(bool)


def row_host(H, r):
    """fp64 masses and values of row r of a HostRows (inputs for the oracle)."""
    g, i = divmod(int(r), H.R)
    n, d = int(H.n[g]), H.d
    off = int(H.logit_off[g]) + i * n
    l = H.logits[off:off + n].astype(np.float64)
    p = np.exp(l - l.max())
    p /= p.sum()
    V = H.v[int(H.v_off[g]):int(H.v_off[g]) + n * d]
    if H.v_dtype == 1:
        V = (V.astype(np.uint32) << 16).view(np.float32)
    return p, V.reshape(n, d).astype(np.float64)


def group_budgets(b):
    k = b.k.cpu().numpy() if hasattr(b.k, "cpu") else np.asarray(b.k)
    return np.ascontiguousarray(k[::b.rows_per_group], np.int32)


def run_vote(fw, b, s):
    rows = fw.rows_from_batch(b)
    k = b.k if hasattr(b.k, "cuda") else torch.from_numpy(np.asarray(b.k)).cuda()
    top = fw.dense_and_topk_gap(rows, k.to(torch.int32).contiguous(), o_kept=False, kept_bits=False, phi=False)
    v = fw.group_vote(rows, torch.from_numpy(np.ascontiguousarray(s, np.int32)).cuda(), top)
    torch.cuda.synchronize()
    return rows, top, v


def check_vote(H, s, v, rows_idx=None):
    """Compare the CUDA vote with the oracle's; rows_idx limits the scored rows.
    Returns the number of (group, budget) sets compared bit for bit."""
    words = (H.max_n + 31) // 32
    ev = None
    if rows_idx is not None:
        ev = np.zeros(H.num_rows, bool)
        ev[rows_idx] = True
    ov = oracle.group_vote(H, s, eval_rows=ev, words=words)
    rows_idx = np.arange(H.num_rows) if rows_idx is None else np.asarray(rows_idx)
    assert np.all(np_(v["row_status"]) == 0)
    assert np.all(ov["status"] == 0)
    bits = np_(v["bits"]).view(np.uint32)
    want_gap, want_drop = ov["gap"].copy(), ov["dropped"].copy()
    strict = 0
    for g in range(len(H.n)):
        n = int(H.n[g])
        for b in range(s.shape[1]):
            mine, theirs = unpack(bits[g, b], n), unpack(ov["bits"][g, b], n)
            assert not bits[g, b][(n + 31) // 32:].any()
            if ov["margin"][g, b] >= VOTE_MARGIN:
                np.testing.assert_array_equal(mine, theirs, err_msg=f"group {g} budget {b}")
                strict += 1
                continue
            G = ov["mass"][g, :n]
            gs = np.sort(G)[::-1][s[g, b] - 1]
            assert mine.sum() == s[g, b]
            assert mine[G > gs * (1 + VOTE_MARGIN)].all() and not mine[G < gs * (1 - VOTE_MARGIN)].any()
            if not np.array_equal(mine, theirs):
                for r in rows_idx[rows_idx // H.R == g]:
                    p, V = row_host(H, r)
                    e = oracle.eval_instance(p, V, mine)
                    want_gap[r, b], want_drop[r, b] = e["gap"], e["dropped"]
    on = []
    for r in rows_idx:
        p, V = row_host(H, r)
        on.append(np.linalg.norm(oracle.eval_instance(p, V, np.ones(len(p), bool))["mu"]))
    on = np.array(on)
    assert_close(np_(v["gap"])[rows_idx], want_gap[rows_idx], on, "vote gap")
    assert_close(np_(v["dropped"])[rows_idx], want_drop[rows_idx], np.ones_like(on), "vote dropped")
    return strict


@pytest.mark.parametrize("n,d,R,v_dtype", [(20, 64, 1, "f32"), (33, 128, 3, "bf16"), (1000, 64, 7, "f32"),
                                           (4097, 128, 5, "bf16"), (300, 256, 2, "f32")])
def test_vote_shapes(fw, n, d, R, v_dtype):
    rng = np.random.default_rng(n + d + R)
    G = 6
    L = (rng.normal(size=(G * R, n)) * rng.uniform(0.3, 4, size=(G * R, 1))).astype(np.float32)
    L[:, 0] += 8
    V = rng.normal(size=(G, n, d)).astype(np.float32)
    # unsorted budgets, s = 1 and s = n among them
    s = np.stack([rng.permutation([1, max(1, n // 16), n // 4, n]) for _ in range(G)]).astype(np.int32)
    b = rows_batch(L, V, np.repeat(s, R, axis=0), v_dtype=v_dtype, R=R)
    _, _, v = run_vote(fw, b, s)
    strict = check_vote(oracle.HostRows(b), s, v)
    assert strict >= s.size // 4  # s = 1 and s = n alone are a quarter each
    full = s == n
    assert np.all(np_(v["dropped"])[np.repeat(full, R, axis=0)] == 0)  # s = n drops nothing


def test_vote_long_rows_reduced(fw):
    # the long-row workload's structure (8 KV heads of 512 query rows, 32,768
    # keys) at a size the oracle checks in seconds
    b = workloads.long_rows(seed=0, heads=2, rows_per_head=12, n=4096)
    s = group_budgets(b)
    _, _, v = run_vote(fw, b, s)
    check_vote(oracle.HostRows(b), s, v)


def test_vote_mixed_profiles_reduced(fw):
    # GQA groups of 4 query rows sharing a bf16 value block, five length profiles
    for b in workloads.mixed_profiles(seed=0, rows_scale=2e-3):
        s = group_budgets(b)
        _, _, v = run_vote(fw, b, s)
        check_vote(oracle.HostRows(b), s, v)


def test_vote_exact_ties_keep_lower_indices(fw):
    # equal logits in every row: every p_j, hence every summed mass, is the same
    # float, and only the tie rule decides the set
    n, R, G, d = 70, 3, 4, 64
    L = np.zeros((G * R, n), np.float32)
    V = np.random.default_rng(1).normal(size=(G, n, d)).astype(np.float32)
    s = np.array([[1, 5, 70], [33, 2, 64], [69, 7, 31], [10, 11, 12]], np.int32)
    b = rows_batch(L, V, np.repeat(s, R, axis=0), R=R)
    _, _, v = run_vote(fw, b, s)
    bits = np_(v["bits"]).view(np.uint32)
    for g in range(G):
        for j in range(3):
            assert np.array_equal(np.nonzero(unpack(bits[g, j], n))[0], np.arange(s[g, j]))
    check_vote(oracle.HostRows(b), s, v)


def test_vote_bad_budget_and_nonfinite_flag_their_group(fw):
    rng = np.random.default_rng(2)
    n, R, G, d = 24, 2, 4, 64
    L = rng.normal(size=(G * R, n)).astype(np.float32)
    L[5, 3] = np.inf  # a logit of group 2
    V = rng.normal(size=(G, n, d)).astype(np.float32)
    s = np.array([[3], [0], [5], [n + 1]], np.int32)
    b = rows_batch(L, V, np.full((G * R, 1), 4, np.int32), R=R)
    _, _, v = run_vote(fw, b, s)
    st = np_(v["row_status"])
    assert list(st) == [0, 0, 1, 1, 6, 6, 1, 1]
    o = oracle.group_vote(oracle.HostRows(b), s)
    assert list(o["status"]) == list(st)
    bits = np_(v["bits"]).view(np.uint32)
    assert np.array_equal(unpack(bits[0, 0], n), unpack(o["bits"][0, 0], n))
    assert not bits[1].any() and not bits[3].any()  # no set for an out-of-range budget
    assert_close(np_(v["gap"])[:2], o["gap"][:2], np.ones(2), "vote gap")


def test_vote_group_of_one_is_own_top_k_set(fw):
    # one row per group: the vote is the row's own top-mass set (Sec. 2.1),
    # so its bits and gap match the gap call's own kept set
    rng = np.random.default_rng(3)
    rows, n, d = 64, 2000, 128
    L = (rng.normal(size=(rows, n)) * 2).astype(np.float32)
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    s = np.tile(np.array([[50, 400, 1000]], np.int32), (rows, 1))
    b = rows_batch(L, V, s, v_dtype="bf16")
    rws = fw.rows_from_batch(b)
    top = fw.dense_and_topk_gap(rws, torch.from_numpy(s).cuda())
    v = fw.group_vote(rws, torch.from_numpy(s).cuda(), top)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(np_(v["bits"]), np_(top["kept_bits"]))
    np.testing.assert_allclose(np_(v["gap"]), np_(top["gap"]), rtol=1e-4, atol=1e-6)
    check_vote(oracle.HostRows(b), s, v)


def test_vote_long_rows_full_scale_sampled(fw):
    """8 KV heads x 512 query rows x 32,768 keys, budgets 2,048 / 4,096 / 8,192:
    every group's set checked, the scores of 48 rows (six per head: the first,
    the last and four drawn at random)."""
    b = workloads.long_rows(seed=0, backend="torch", device="cuda")
    s = group_budgets(b)
    _, _, v = run_vote(fw, b, s)
    H = oracle.HostRows(b)
    rng = np.random.default_rng(0)
    pick = np.sort(np.concatenate([[g * H.R, g * H.R + H.R - 1] for g in range(len(H.n))] +
                                  [g * H.R + 1 + rng.choice(H.R - 2, 4, replace=False) for g in range(len(H.n))]))
    check_vote(H, s, v, rows_idx=pick)
    gap, dr = np_(v["gap"]), np_(v["dropped"])
    assert np.all(np.isfinite(gap))
    assert np.all(np.diff(dr, axis=1) <= 1e-7)  # larger budgets drop less mass
