"""The C ABI: libfw.so builds for sm_103a, loads, and exports every entry
point include/fw.h declares; host-side argument checks reject bad input
before any launch.  No GPU needed."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "fw.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(fw_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_25230_gb300 import _build

    path = _build.build()
    return C.CDLL(path)


def test_header_declares_the_five_calls():
    syms = declared_symbols()
    for name in ("fw_dense_and_topk_gap", "fw_swap_refine", "fw_best_subset", "fw_contour_alloc",
                 "fw_ragged_compact", "fw_group_vote", "fw_pool_best_subset", "fw_sync_status"):
        assert name in syms


def test_every_declared_symbol_is_exported(lib):
    for name in declared_symbols():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    lib.fw_status_string.restype = C.c_char_p
    assert lib.fw_status_string(0) == b"ok"
    assert b"invalid" in lib.fw_status_string(1)


def test_host_validation_rejects_bad_arguments(lib):
    from paper_2608_25230_gb300 import fw

    before = fw.launch_count()
    rows = fw.FwRows(1, 1, 48, 4, 0, None, None, None, None, None)  # d = 48 unsupported
    out = fw.FwGapOut()
    st = fw._lib.fw_dense_and_topk_gap(C.byref(rows), None, 1, C.byref(out), None, 0, None)
    assert st in (fw.FW_ERR_UNSUPPORTED, fw.FW_ERR_INVALID_ARG)
    rows = fw.FwRows(1, 1, 64, 4, 0, None, None, None, None, None)  # null pointers
    assert fw._lib.fw_dense_and_topk_gap(C.byref(rows), None, 1, C.byref(out), None, 0, None) == fw.FW_ERR_INVALID_ARG
    # ContourKV: budget below the floors, and a misaligned compaction row
    assert fw._lib.fw_contour_alloc(C.c_void_p(16), 4, 64, 32, 10, 2, *([C.c_void_p(16)] * 6), None, 0,
                                    None) == fw.FW_ERR_INVALID_ARG
    assert fw._lib.fw_ragged_compact(C.c_void_p(16), C.c_void_p(16), 1, 1, 24, C.c_void_p(16), C.c_void_p(16), 1,
                                     C.c_void_p(16), C.c_void_p(16), None) == fw.FW_ERR_INVALID_ARG
    # best subset needs n <= 32
    rows = fw.FwRows(1, 1, 64, 33, 0, *([C.c_void_p(256)] * 5))
    assert fw._lib.fw_best_subset(C.byref(rows), C.c_void_p(256), *([C.c_void_p(256)] * 3), 8, None, None,
                                  C.c_void_p(256), 1 << 20, None) == fw.FW_ERR_UNSUPPORTED
    # value rows must be 16-byte aligned; the long-row selector stages at most 96 pool keys
    rows = fw.FwRows(1, 1, 64, 64, 1, C.c_void_p(256), C.c_void_p(256), C.c_void_p(256), C.c_void_p(264),
                     C.c_void_p(256))
    assert fw._lib.fw_dense_and_topk_gap(C.byref(rows), C.c_void_p(256), 1, C.byref(out), C.c_void_p(256), 1 << 30,
                                         None) == fw.FW_ERR_INVALID_ARG
    rows = fw.FwRows(1, 1, 64, 64, 1, *([C.c_void_p(256)] * 5))
    top = fw.FwGapOut()
    top.o = top.row_max = top.row_sum = top.thr_key = top.thr_idx = 256
    prm = fw.FwSwapParams(97, 4)
    assert fw._lib.fw_swap_refine(C.byref(rows), C.c_void_p(256), 1, C.byref(top), C.byref(prm),
                                  *([C.c_void_p(256)] * 6), C.c_void_p(256), 1 << 40, None) == fw.FW_ERR_UNSUPPORTED
    # group vote: budgets per call, the gap call's outputs, the bit-mask width and the workspace
    P = C.c_void_p(256)
    assert fw._lib.fw_group_vote(C.byref(rows), P, 5, C.byref(top), P, P, P, 2, P, P, 1 << 30,
                                 None) == fw.FW_ERR_INVALID_ARG
    nosum = fw.FwGapOut()
    nosum.o = nosum.row_max = 256
    assert fw._lib.fw_group_vote(C.byref(rows), P, 1, C.byref(nosum), P, P, P, 2, P, P, 1 << 30,
                                 None) == fw.FW_ERR_INVALID_ARG
    assert fw._lib.fw_group_vote(C.byref(rows), P, 1, C.byref(top), P, P, P, 1, P, P, 1 << 30,
                                 None) == fw.FW_ERR_INVALID_ARG
    need = fw._lib.fw_group_vote_workspace(C.byref(rows), 2)
    assert need >= 64 * 4
    assert fw._lib.fw_group_vote(C.byref(rows), P, 2, C.byref(top), P, P, None, 0, None, P, need - 1,
                                 None) == fw.FW_ERR_WORKSPACE
    # ES_pool: budget slots, extras, the gap call's thresholds, k_max and the workspace
    E2 = (C.c_int32 * 2)(4, 4)
    assert fw._lib.fw_pool_best_subset(C.byref(rows), P, 5, E2, C.byref(top), P, P, 32, None, None, None, P, 1 << 30,
                                       None) == fw.FW_ERR_INVALID_ARG
    Eneg = (C.c_int32 * 2)(4, -1)
    assert fw._lib.fw_pool_best_subset(C.byref(rows), P, 2, Eneg, C.byref(top), P, P, 32, None, None, None, P, 1 << 30,
                                       None) == fw.FW_ERR_INVALID_ARG
    assert fw._lib.fw_pool_best_subset(C.byref(rows), P, 2, E2, C.byref(nosum), P, P, 32, None, None, None, P, 1 << 30,
                                       None) == fw.FW_ERR_INVALID_ARG
    assert fw._lib.fw_pool_best_subset(C.byref(rows), P, 2, E2, C.byref(top), P, P, 33, None, None, None, P, 1 << 30,
                                       None) == fw.FW_ERR_INVALID_ARG
    need = fw._lib.fw_pool_best_subset_workspace(C.byref(rows), 2)
    assert need >= 2 * 64 * 4
    assert fw._lib.fw_pool_best_subset(C.byref(rows), P, 2, E2, C.byref(top), P, P, 32, None, None, None, P, need - 1,
                                       None) == fw.FW_ERR_WORKSPACE
    # the status read-back rejects a negative row count before it touches the device
    first = C.c_int64(7)
    assert fw._lib.fw_sync_status(P, -1, C.byref(first), None) == fw.FW_ERR_INVALID_ARG and first.value == -1
    assert fw.launch_count() == before  # nothing was launched
