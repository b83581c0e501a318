"""GPU parity for the selector audit (fw_selector_audit: StreamingLLM, H2O,
SnapKV, Quest, Quest-16 with App. C's settings, each kept set scored with es)
against the fp64 oracle.  StreamingLLM and Quest sets are bit-exact (positions
and exact logit maxima decide them).  H2O and SnapKV rank fp32 sums of masses
over the group's rows; where their set differs from the oracle's, it must be a
valid top-m under the oracle's fp64 scores up to 1e-4 relative (the same
reading as the group vote), and its es is compared with the oracle's es of
that very set."""
import numpy as np
import pytest

import oracle
import workloads
from tests.parity import assert_close, np_, row_onorm
from tests.test_gpu_pool import row_host
from tests.test_gpu_small import rows_batch

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

BAND = 1e-4


@pytest.fixture(scope="module")
def fw():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_25230_gb300 import fw as _fw

    return _fw


def unpack(words, n):
    w = np.asarray(words).view(np.uint32)
    return ((w[np.arange(n) >> 5] >> (np.arange(n) & 31)) & 1).astype(bool)


def valid_top(mask, score, cand, m):
    """mask restricted to the candidates is a top-m of score within BAND."""
    sel = mask[:cand]
    if sel.sum() != m:
        return False
    if m == 0 or m == cand:
        return True
    return score[:cand][sel].min() >= score[:cand][~sel].max() * (1 - BAND)


def check_audit(fw, batch, s):
    rows = fw.rows_from_batch(batch)
    k = torch.as_tensor(np.asarray(batch.k)).cuda()
    top = fw.dense_and_topk_gap(rows, k)
    out = fw.selector_audit(rows, s, top, bits=True)
    torch.cuda.synchronize()
    H = oracle.HostRows(batch)
    o = oracle.selector_audit(H, s)
    on = row_onorm(oracle.dense_and_topk_gap(H)["o"])
    es, bits = np_(out["es"]), np_(out["bits"])
    want = o["es"].copy()
    for r in range(H.num_rows):
        g = r // H.R
        n = int(H.n[g])
        for b, sb in enumerate(s):
            for sel in range(5):
                mine, theirs = unpack(bits[r, sel, b], n), unpack(o["bits"][r, sel, b], n)
                if np.array_equal(mine, theirs):
                    continue
                assert sel in (1, 2), (r, sel, b)  # only the summed-mass rules may differ
                if sel == 1:
                    rr = sb // 2
                    assert mine[n - rr:].all() and valid_top(mine, o["G"][g], n - rr, sb - rr), (r, b)
                else:
                    w = max(1, min(32, sb // 2))
                    assert mine[n - w:].all() and valid_top(mine, o["pooled"][g, b], n - w, sb - w), (r, b)
                p, Vr = row_host(H, r)
                want[r, sel, b] = oracle.eval_instance(p, Vr, mine)["gap"]
    nan = np.isnan(want)
    np.testing.assert_array_equal(np.isnan(es), nan)
    assert_close(np.where(nan, 0, es), np.where(nan, 0, want), on, "selector es")
    return out, o


def test_audit_long_rows_reduced(fw):
    b = workloads.long_rows(seed=2, heads=2, rows_per_head=40, n=4096)
    check_audit(fw, b, [4, 8, 16, 32])


def test_audit_deployed_budgets(fw):
    b = workloads.long_rows(seed=3, heads=2, rows_per_head=12, n=2048, d=64)
    check_audit(fw, b, [64, 128, 256, 1024])


def test_audit_mixed_profiles_and_small_rows(fw):
    for b in workloads.mixed_profiles(seed=5, rows_scale=3e-4):
        check_audit(fw, b, [4, 8, 16, 32])
    for b in workloads.exact_enum(seed=0, rows_scale=8 / 24192)[:2]:
        check_audit(fw, b, [4, 6, 12, 24])


def test_audit_ties_and_budget_edges(fw):
    rng = np.random.default_rng(7)
    R, n, d = 5, 100, 32
    L = np.round(rng.normal(size=(2 * R, n)) * 2).astype(np.float32)  # many equal logits and masses
    V = rng.normal(size=(2, n, d)).astype(np.float32)
    check_audit(fw, rows_batch(L, V, np.ones((2 * R, 1), np.int32), R=R), [1, 2, 100, 17])
