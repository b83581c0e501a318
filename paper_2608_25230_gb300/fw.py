"""Thin ctypes binding of libfw.so (include/fw.h).

Marshalling only: every step of the computation runs in the library's CUDA
kernels.  torch provides device memory and the current stream; the library
never allocates.  If libfw.so is missing this module raises on import -- there
is no fallback path.
"""
from __future__ import annotations

import ctypes as C
import math
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libfw.so")

FW_OK, FW_ERR_INVALID_ARG, FW_ERR_UNSUPPORTED, FW_ERR_CUDA = 0, 1, 2, 3
FW_ERR_TIMEOUT, FW_ERR_WORKSPACE, FW_ERR_NONFINITE = 4, 5, 6
FW_F32, FW_BF16 = 0, 1

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with __graft_entry__.build() "
                      "(nvcc, sm_103a); there is no CPU fallback")
_lib = C.CDLL(LIB_PATH)

vp = C.c_void_p


class FwRows(C.Structure):
    _fields_ = [("num_groups", C.c_int64), ("rows_per_group", C.c_int32), ("d", C.c_int32),
                ("max_n", C.c_int32), ("v_dtype", C.c_int32), ("logits", vp), ("logit_off", vp),
                ("n", vp), ("v", vp), ("v_off", vp)]


class FwGapOut(C.Structure):
    _fields_ = [("o", vp), ("o_kept", vp), ("gap", vp), ("dropped", vp), ("phi", vp), ("row_max", vp),
                ("row_sum", vp), ("thr_key", vp), ("thr_idx", vp), ("kept_bits", vp),
                ("kept_words", C.c_int32), ("row_status", vp)]


class FwBestSubsetStats(C.Structure):
    _fields_ = [("rows_exhaustive", C.c_int64), ("candidates", C.c_int64), ("inner_nodes", C.c_uint64),
                ("inner_leaves", C.c_uint64), ("inner_ops", C.c_uint64), ("skipped", C.c_uint64)]


class FwSwapParams(C.Structure):
    _fields_ = [("E", C.c_int32), ("max_swaps", C.c_int32)]


_lib.fw_dense_and_topk_gap.argtypes = [C.POINTER(FwRows), vp, C.c_int32, C.POINTER(FwGapOut), vp, C.c_size_t, vp]
_lib.fw_dense_and_topk_gap_workspace.argtypes = [C.POINTER(FwRows), C.c_int32]
_lib.fw_dense_and_topk_gap_workspace.restype = C.c_size_t
_lib.fw_swap_refine.argtypes = [C.POINTER(FwRows), vp, C.c_int32, C.POINTER(FwGapOut), C.POINTER(FwSwapParams),
                                vp, vp, vp, vp, vp, vp, vp, C.c_size_t, vp]
_lib.fw_swap_refine_workspace.argtypes = [C.POINTER(FwRows), C.c_int32, C.POINTER(FwSwapParams)]
_lib.fw_swap_refine_workspace.restype = C.c_size_t
_lib.fw_best_subset.argtypes = [C.POINTER(FwRows), vp, vp, vp, vp, C.c_int32, vp, vp, vp, C.c_size_t, vp]
_lib.fw_best_subset_workspace.argtypes = [C.POINTER(FwRows)]
_lib.fw_best_subset_workspace.restype = C.c_size_t
_lib.fw_fp32_fma_probe.argtypes = [C.c_int32, C.c_int32, vp, vp]
_lib.fw_fp32_fma_probe.restype = C.c_int
_lib.fw_best_subset_read_stats.argtypes = [C.POINTER(FwRows), vp, C.POINTER(FwBestSubsetStats), vp]
_lib.fw_best_subset_read_stats.restype = C.c_int
_lib.fw_contour_alloc.argtypes = [vp, C.c_int32, C.c_int32, C.c_int32, C.c_int64, C.c_int32, vp, vp, vp, vp, vp,
                                  vp, vp, C.c_size_t, vp]
_lib.fw_contour_alloc_workspace.argtypes = [C.c_int32, C.c_int32]
_lib.fw_contour_alloc_workspace.restype = C.c_size_t
_lib.fw_contour_alloc_capped.argtypes = [vp, C.c_int32, C.c_int32, C.c_int32, C.c_int64, C.c_int32, C.c_int32, vp, vp,
                                         vp, vp, vp, vp, vp, C.c_size_t, vp]
_lib.fw_contour_alloc_capped.restype = C.c_int
_lib.fw_contour_alloc_capped_workspace.argtypes = [C.c_int32, C.c_int32]
_lib.fw_contour_alloc_capped_workspace.restype = C.c_size_t
_lib.fw_ragged_compact_to.argtypes = [vp, vp, C.c_int32, C.c_int32, C.c_int32, vp, vp, vp, vp, vp, vp, vp, vp]
_lib.fw_ragged_compact_to.restype = C.c_int
_lib.fw_ragged_append.argtypes = [vp, vp, vp, vp, vp, vp, vp, C.c_int32, C.c_int32, C.c_int32, vp, vp]
_lib.fw_ragged_append.restype = C.c_int
_lib.fw_window_score.argtypes = [vp, vp, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_float, C.c_int32, vp, vp,
                                 vp, C.c_size_t, vp]
_lib.fw_window_score.restype = C.c_int
_lib.fw_window_score_workspace.argtypes = [C.c_int32, C.c_int32]
_lib.fw_window_score_workspace.restype = C.c_size_t
_lib.fw_selector_audit.argtypes = [C.POINTER(FwRows), vp, C.c_int32, C.POINTER(FwGapOut), vp, vp, C.c_int32, vp,
                                   C.c_size_t, vp]
_lib.fw_selector_audit.restype = C.c_int
_lib.fw_selector_audit_workspace.argtypes = [C.POINTER(FwRows), C.c_int32]
_lib.fw_selector_audit_workspace.restype = C.c_size_t
_lib.fw_ragged_compact.argtypes = [vp, vp, C.c_int32, C.c_int32, C.c_int32, vp, vp, C.c_int64, vp, vp, vp]
_lib.fw_group_vote.argtypes = [C.POINTER(FwRows), vp, C.c_int32, C.POINTER(FwGapOut), vp, vp, vp, C.c_int32, vp,
                               vp, C.c_size_t, vp]
_lib.fw_group_vote_workspace.argtypes = [C.POINTER(FwRows), C.c_int32]
_lib.fw_group_vote_workspace.restype = C.c_size_t
_lib.fw_pool_best_subset.argtypes = [C.POINTER(FwRows), vp, C.c_int32, vp, C.POINTER(FwGapOut), vp, vp, C.c_int32,
                                     vp, vp, vp, vp, C.c_size_t, vp]
_lib.fw_pool_best_subset_workspace.argtypes = [C.POINTER(FwRows), C.c_int32]
_lib.fw_pool_best_subset_workspace.restype = C.c_size_t
_lib.fw_sync_status.argtypes = [vp, C.c_int64, C.POINTER(C.c_int64), vp]
_lib.fw_status_string.argtypes = [C.c_int]
_lib.fw_status_string.restype = C.c_char_p
_lib.fw_launch_count.restype = C.c_uint64
for _f in ("fw_dense_and_topk_gap", "fw_swap_refine", "fw_best_subset", "fw_contour_alloc", "fw_ragged_compact",
           "fw_group_vote", "fw_pool_best_subset", "fw_sync_status"):
    getattr(_lib, _f).restype = C.c_int


class FwError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__(f"{where}: {_lib.fw_status_string(status).decode()} ({status})")


def _check(st, where):
    if st != FW_OK:
        raise FwError(st, where)


def launch_count() -> int:
    return int(_lib.fw_launch_count())


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return C.c_void_p(s.cuda_stream)


def _ws(nbytes, device):
    # 256-byte aligned scratch for the library (torch's caching allocator aligns to 512)
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


class Rows:
    """Device-side row batch (fw_rows) built from tensors."""

    def __init__(self, *, rows_per_group, d, n_host, logits, logit_off, n, v, v_off, v_dtype):
        self.rows_per_group = int(rows_per_group)
        self.d = int(d)
        self.n_host = n_host
        self.num_groups = int(len(n_host))
        self.num_rows = self.num_groups * self.rows_per_group
        self.max_n = int(max(n_host)) if self.num_groups else 1
        self.logits, self.logit_off, self.n, self.v, self.v_off = logits, logit_off, n, v, v_off
        self.v_dtype = FW_BF16 if v_dtype == "bf16" else FW_F32
        self.device = logits.device
        self.c = FwRows(self.num_groups, self.rows_per_group, self.d, self.max_n, self.v_dtype,
                        _ptr(logits), _ptr(logit_off), _ptr(n), _ptr(v), _ptr(v_off))


def _to_dev(a, dtype, device):
    if isinstance(a, torch.Tensor):
        return a.to(device=device, dtype=dtype).contiguous()
    import numpy as np

    return torch.from_numpy(np.ascontiguousarray(a)).to(device=device, dtype=dtype).contiguous()


def rows_from_batch(batch, device="cuda") -> Rows:
    """Copy a workloads.RowBatch (numpy or torch) to the device."""
    import numpy as np

    if batch.v_dtype == "bf16":
        v = batch.v
        if isinstance(v, torch.Tensor):
            v = v.to(device).contiguous().view(torch.int16)
        else:
            v = torch.from_numpy(np.ascontiguousarray(v).view(np.int16)).to(device)
    else:
        v = _to_dev(batch.v, torch.float32, device)
    return Rows(rows_per_group=batch.rows_per_group, d=batch.d, n_host=np.asarray(batch.n_host),
                logits=_to_dev(batch.logits, torch.float32, device),
                logit_off=_to_dev(batch.logit_off, torch.int64, device),
                n=_to_dev(batch.n, torch.int32, device), v=v,
                v_off=_to_dev(batch.v_off, torch.int64, device), v_dtype=batch.v_dtype)


def dense_and_topk_gap(rows: Rows, k: torch.Tensor, *, o_kept=True, kept_bits=True, phi=True, stream=None):
    """fw_dense_and_topk_gap.  k: int32 [rows][nb] on the device.  Returns a dict
    of device tensors (the fw_gap_out fields)."""
    dev = rows.device
    R, d = rows.num_rows, rows.d
    nb = int(k.shape[1])
    words = (rows.max_n + 31) // 32
    f32 = dict(dtype=torch.float32, device=dev)
    out = dict(o=torch.empty(R, d, **f32), gap=torch.empty(R, nb, **f32), dropped=torch.empty(R, nb, **f32),
               row_max=torch.empty(R, **f32), row_sum=torch.empty(R, **f32),
               thr_key=torch.empty(R, nb, dtype=torch.int32, device=dev),
               thr_idx=torch.empty(R, nb, dtype=torch.int32, device=dev),
               row_status=torch.empty(R, dtype=torch.int32, device=dev))
    if o_kept:
        out["o_kept"] = torch.empty(R, nb, d, **f32)
    if phi:
        out["phi"] = torch.empty(R, nb, **f32)
    if kept_bits:
        out["kept_bits"] = torch.empty(R, nb, words, dtype=torch.int32, device=dev)
    c_out = gap_out_struct(out, words)
    nbytes = _lib.fw_dense_and_topk_gap_workspace(C.byref(rows.c), nb)
    ws = _ws(nbytes, dev)
    st = _lib.fw_dense_and_topk_gap(C.byref(rows.c), _ptr(k), nb, C.byref(c_out), _ptr(ws), ws.numel(),
                                    _stream(stream))
    _check(st, "fw_dense_and_topk_gap")
    out["_ws"] = ws
    out["_c"] = c_out
    return out


def gap_out_struct(out, words):
    return FwGapOut(_ptr(out.get("o")), _ptr(out.get("o_kept")), _ptr(out["gap"]), _ptr(out["dropped"]),
                    _ptr(out.get("phi")), _ptr(out.get("row_max")), _ptr(out.get("row_sum")),
                    _ptr(out.get("thr_key")), _ptr(out.get("thr_idx")), _ptr(out.get("kept_bits")),
                    int(words), _ptr(out.get("row_status")))


def swap_refine(rows: Rows, k: torch.Tensor, topk: dict, *, E: int, max_swaps: int = 64, stream=None):
    dev = rows.device
    R = rows.num_rows
    nb = int(k.shape[1])
    prm = FwSwapParams(int(E), int(max_swaps))
    out = dict(n_swaps=torch.empty(R, nb, dtype=torch.int32, device=dev),
               swap_out=torch.empty(R, nb, max_swaps, dtype=torch.int32, device=dev),
               swap_in=torch.empty(R, nb, max_swaps, dtype=torch.int32, device=dev),
               refined_gap=torch.empty(R, nb, dtype=torch.float32, device=dev),
               topk_gap=torch.empty(R, nb, dtype=torch.float32, device=dev),
               capped=torch.empty(R, nb, dtype=torch.int32, device=dev))
    nbytes = _lib.fw_swap_refine_workspace(C.byref(rows.c), nb, C.byref(prm))
    ws = _ws(nbytes, dev)
    st = _lib.fw_swap_refine(C.byref(rows.c), _ptr(k), nb, C.byref(topk["_c"]), C.byref(prm),
                             _ptr(out["n_swaps"]), _ptr(out["swap_out"]), _ptr(out["swap_in"]),
                             _ptr(out["refined_gap"]), _ptr(out["topk_gap"]), _ptr(out["capped"]), _ptr(ws),
                             ws.numel(), _stream(stream))
    _check(st, "fw_swap_refine")
    out["_ws"] = ws
    return out


def group_vote(rows: Rows, s: torch.Tensor, topk: dict, *, bits=True, stream=None):
    """fw_group_vote.  s: int32 [groups][nb] budgets on the device; topk: the
    dict dense_and_topk_gap returned for the same rows.  Returns gap, dropped,
    row_status ([rows][nb] / [rows]) and bits ([groups][nb][words])."""
    dev = rows.device
    R, nb = rows.num_rows, int(s.shape[1])
    words = (rows.max_n + 31) // 32
    out = dict(gap=torch.empty(R, nb, dtype=torch.float32, device=dev),
               dropped=torch.empty(R, nb, dtype=torch.float32, device=dev),
               row_status=torch.empty(R, dtype=torch.int32, device=dev))
    if bits:
        out["bits"] = torch.empty(rows.num_groups, nb, words, dtype=torch.int32, device=dev)
    nbytes = _lib.fw_group_vote_workspace(C.byref(rows.c), nb)
    ws = _ws(nbytes, dev)
    st = _lib.fw_group_vote(C.byref(rows.c), _ptr(s), nb, C.byref(topk["_c"]), _ptr(out["gap"]),
                            _ptr(out["dropped"]), _ptr(out.get("bits")), words, _ptr(out["row_status"]), _ptr(ws),
                            ws.numel(), _stream(stream))
    _check(st, "fw_group_vote")
    out["_ws"] = ws
    return out


def best_subset(rows: Rows, k: torch.Tensor, *, k_max=None, stream=None, ws=None):
    """fw_best_subset.  k: int32 [rows] (or [rows][1]) on the device."""
    dev = rows.device
    R = rows.num_rows
    k = k.reshape(-1)
    if k_max is None:  # one device read; pass k_max to avoid it
        k_max = int(k.max().item()) if k.numel() else 1
    k_max = int(k_max)
    out = dict(best_rank=torch.empty(R, dtype=torch.int64, device=dev),
               best_gap=torch.empty(R, dtype=torch.float32, device=dev),
               best_idx=torch.empty(R, k_max, dtype=torch.int32, device=dev),
               topk_gap=torch.empty(R, dtype=torch.float32, device=dev),
               row_status=torch.empty(R, dtype=torch.int32, device=dev))
    nbytes = _lib.fw_best_subset_workspace(C.byref(rows.c))
    if ws is None or ws.numel() < nbytes:
        ws = _ws(nbytes, dev)
    st = _lib.fw_best_subset(C.byref(rows.c), _ptr(k), _ptr(out["best_rank"]), _ptr(out["best_gap"]),
                             _ptr(out["best_idx"]), k_max, _ptr(out["topk_gap"]), _ptr(out["row_status"]),
                             _ptr(ws), ws.numel(), _stream(stream))
    _check(st, "fw_best_subset")
    out["_ws"] = ws
    return out


def best_subset_stats(rows: Rows, out: dict, stream=None) -> dict:
    """fw_best_subset_read_stats for the call that returned `out` (waits for
    the stream): rows sent to the exhaustive path, re-scored candidates, and
    the walk's inner enumerations, leaves, fp32 operations and skipped nodes."""
    st = FwBestSubsetStats()
    _check(_lib.fw_best_subset_read_stats(C.byref(rows.c), _ptr(out["_ws"]), C.byref(st), _stream(stream)),
           "fw_best_subset_read_stats")
    return {name: int(getattr(st, name)) for name, _ in FwBestSubsetStats._fields_}


def pool_best_subset(rows: Rows, k: torch.Tensor, topk: dict, *, E, k_max: int = 32, stream=None):
    """fw_pool_best_subset (ES_pool, Definition 2.2).  k: int32 [rows][nb] on
    the device (the budgets of the gap call `topk`); E: extras per budget slot
    (host sequence of nb ints).  Returns best_gap, best_idx, topk_gap, n_cand,
    row_status."""
    dev, R, nb = rows.device, rows.num_rows, int(k.shape[1])
    E = [int(e) for e in E]
    if len(E) != nb:
        raise ValueError("E needs one entry per budget slot")
    Eh = (C.c_int32 * nb)(*E)
    out = dict(best_gap=torch.empty(R, nb, dtype=torch.float32, device=dev),
               best_idx=torch.empty(R, nb, int(k_max), dtype=torch.int32, device=dev),
               topk_gap=torch.empty(R, nb, dtype=torch.float32, device=dev),
               n_cand=torch.empty(R, nb, dtype=torch.int64, device=dev),
               row_status=torch.empty(R, dtype=torch.int32, device=dev))
    ws = _ws(_lib.fw_pool_best_subset_workspace(C.byref(rows.c), nb), dev)
    st = _lib.fw_pool_best_subset(C.byref(rows.c), _ptr(k), nb, Eh, C.byref(topk["_c"]), _ptr(out["best_gap"]),
                                  _ptr(out["best_idx"]), int(k_max), _ptr(out["topk_gap"]), _ptr(out["n_cand"]),
                                  _ptr(out["row_status"]), _ptr(ws), ws.numel(), _stream(stream))
    _check(st, "fw_pool_best_subset")
    out["_ws"] = ws
    return out


def sync_status(row_status: torch.Tensor, stream=None):
    """fw_sync_status: wait for the stream, then (status, first bad row) of a
    per-row status array (FW_OK, -1 when every row is fine)."""
    first = C.c_int64(-1)
    st = _lib.fw_sync_status(_ptr(row_status), int(row_status.numel()), C.byref(first), _stream(stream))
    return int(st), int(first.value)


def _contour_outputs(cells, total_budget, dev, out):
    if out is not None:  # caller-owned buffers of the same shapes, reused across calls
        return out
    return dict(counts=torch.empty(cells, dtype=torch.int32, device=dev),
                offsets=torch.empty(cells + 1, dtype=torch.int64, device=dev),
                kept_pos=torch.empty(int(total_budget), dtype=torch.int32, device=dev),
                tau=torch.empty(1, dtype=torch.float32, device=dev),
                dropped_uniform=torch.empty(cells, dtype=torch.float32, device=dev),
                dropped_alloc=torch.empty(cells, dtype=torch.float32, device=dev))


def _contour_ws(nbytes, dev, workspace):
    if workspace is None:
        return _ws(nbytes, dev)
    if workspace.numel() * workspace.element_size() < nbytes:
        raise ValueError(f"workspace holds {workspace.numel() * workspace.element_size()} bytes, {nbytes} needed")
    return workspace


def contour_alloc(scores: torch.Tensor, *, floor: int, total_budget: int, uniform_s: int, stream=None, out=None,
                  workspace=None):
    """fw_contour_alloc.  out (a dict as returned) and workspace (a uint8
    tensor of fw_contour_alloc_workspace bytes) may be passed to reuse
    buffers across calls."""
    dev = scores.device
    cells, T = scores.shape
    out = _contour_outputs(cells, total_budget, dev, out)
    ws = _contour_ws(_lib.fw_contour_alloc_workspace(cells, T), dev, workspace)
    st = _lib.fw_contour_alloc(_ptr(scores), cells, T, int(floor), int(total_budget), int(uniform_s),
                               _ptr(out["counts"]), _ptr(out["offsets"]), _ptr(out["kept_pos"]), _ptr(out["tau"]),
                               _ptr(out["dropped_uniform"]), _ptr(out["dropped_alloc"]), _ptr(ws), ws.numel(),
                               _stream(stream))
    _check(st, "fw_contour_alloc")
    out["_ws"] = ws
    return out


def contour_alloc_capped(scores: torch.Tensor, *, floor: int, total_budget: int, uniform_s: int, cap: int,
                         stream=None, out=None, workspace=None):
    """fw_contour_alloc_capped: the allocation truncated to `cap` entries per
    cell.  kept_pos holds total_budget entries; offsets[-1] of them are valid.
    out and workspace as for contour_alloc (the capped workspace size)."""
    dev = scores.device
    cells, T = scores.shape
    out = _contour_outputs(cells, total_budget, dev, out)
    ws = _contour_ws(_lib.fw_contour_alloc_capped_workspace(cells, T), dev, workspace)
    st = _lib.fw_contour_alloc_capped(_ptr(scores), cells, T, int(floor), int(total_budget), int(uniform_s), int(cap),
                                      _ptr(out["counts"]), _ptr(out["offsets"]), _ptr(out["kept_pos"]),
                                      _ptr(out["tau"]), _ptr(out["dropped_uniform"]), _ptr(out["dropped_alloc"]),
                                      _ptr(ws), ws.numel(), _stream(stream))
    _check(st, "fw_contour_alloc_capped")
    out["_ws"] = ws
    return out


def ragged_compact(K: torch.Tensor, V: torch.Tensor, offsets: torch.Tensor, kept_pos: torch.Tensor, total: int,
                   *, out=None, stream=None):
    cells, T, d = K.shape
    row_bytes = d * K.element_size()
    if out is None:
        Ko = torch.empty(int(total), d, dtype=K.dtype, device=K.device)
        Vo = torch.empty(int(total), d, dtype=V.dtype, device=V.device)
    else:
        Ko, Vo = out
    st = _lib.fw_ragged_compact(_ptr(K), _ptr(V), cells, T, row_bytes, _ptr(offsets), _ptr(kept_pos), int(total),
                                _ptr(Ko), _ptr(Vo), _stream(stream))
    _check(st, "fw_ragged_compact")
    return Ko, Vo


def ragged_compact_to(K: torch.Tensor, V: torch.Tensor, offsets: torch.Tensor, kept_pos: torch.Tensor,
                      base: torch.Tensor, capacity: torch.Tensor, K_store: torch.Tensor, V_store: torch.Tensor,
                      status: torch.Tensor = None, stream=None):
    """fw_ragged_compact_to: kept rows into a store with room per cell."""
    cells, T, d = K.shape
    st = _lib.fw_ragged_compact_to(_ptr(K), _ptr(V), cells, T, d * K.element_size(), _ptr(offsets), _ptr(kept_pos),
                                   _ptr(base), _ptr(capacity), _ptr(K_store), _ptr(V_store), _ptr(status),
                                   _stream(stream))
    _check(st, "fw_ragged_compact_to")


def ragged_append(K_store: torch.Tensor, V_store: torch.Tensor, base: torch.Tensor, capacity: torch.Tensor,
                  counts: torch.Tensor, new_K: torch.Tensor, new_V: torch.Tensor, status: torch.Tensor = None,
                  stream=None):
    """fw_ragged_append: new_K / new_V [cells][m][d] behind each cell's rows."""
    cells, m, d = new_K.shape
    st = _lib.fw_ragged_append(_ptr(K_store), _ptr(V_store), _ptr(base), _ptr(capacity), _ptr(counts), _ptr(new_K),
                               _ptr(new_V), cells, m, d * new_K.element_size(), _ptr(status), _stream(stream))
    _check(st, "fw_ragged_append")


def window_score(Qw: torch.Tensor, K: torch.Tensor, *, scale: float = None, pool: int = 7, out=None, stream=None):
    """fw_window_score.  Qw: bf16 (or int16 bits) [cells][w][d]; K: [cells][T][d].
    Returns (scores [cells][T] fp32, status [cells])."""
    cells, w, d = Qw.shape
    T = K.shape[1]
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    scores = out if out is not None else torch.empty(cells, T, dtype=torch.float32, device=K.device)
    status = torch.empty(cells, dtype=torch.int32, device=K.device)
    ws = _ws(_lib.fw_window_score_workspace(cells, T), K.device)
    st = _lib.fw_window_score(_ptr(Qw), _ptr(K), cells, T, d, w, C.c_float(scale), int(pool), _ptr(scores),
                              _ptr(status), _ptr(ws), ws.numel(), _stream(stream))
    _check(st, "fw_window_score")
    return scores, status


SELECTORS = ("streamingllm", "h2o", "snapkv", "quest", "quest16")


def selector_audit(rows: Rows, s, topk: dict, *, bits=False, stream=None):
    """fw_selector_audit: es of every deployed rule's kept set ([rows][5][nb],
    rules in SELECTORS order) at the host budgets s; optionally the sets."""
    dev, R = rows.device, rows.num_rows
    s = [int(x) for x in s]
    nb = len(s)
    words = (rows.max_n + 31) // 32
    out = dict(es=torch.empty(R, len(SELECTORS), nb, dtype=torch.float32, device=dev))
    if bits:
        out["bits"] = torch.empty(R, len(SELECTORS), nb, words, dtype=torch.int32, device=dev)
    sh = (C.c_int32 * nb)(*s)
    ws = _ws(_lib.fw_selector_audit_workspace(C.byref(rows.c), nb), dev)
    st = _lib.fw_selector_audit(C.byref(rows.c), sh, nb, C.byref(topk["_c"]), _ptr(out["es"]), _ptr(out.get("bits")),
                                words, _ptr(ws), ws.numel(), _stream(stream))
    _check(st, "fw_selector_audit")
    out["_ws"] = ws
    return out


def raw():
    """The loaded ctypes library (for callers that marshal their own arguments)."""
    return _lib


def fp32_fma_probe(blocks: int, iters: int, out: torch.Tensor, stream=None):
    """fw_fp32_fma_probe (a measurement aid): blocks x 256 threads x 16 chains x
    iters fp32 FMAs; out: float32 [blocks * 256] on the device."""
    _check(_lib.fw_fp32_fma_probe(int(blocks), int(iters), _ptr(out), _stream(stream)), "fw_fp32_fma_probe")
