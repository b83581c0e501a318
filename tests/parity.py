"""Comparison rules between the CUDA path and the fp64 oracle.

Floating-point outputs (gaps, dropped mass, outputs, Phi) must satisfy
    |gpu - oracle| <= 1e-4 * |oracle| + 1e-6 * ||o||
with ||o|| the norm of that row's dense output.  Integer and index outputs
(kept sets, swaps, ranks, counts, offsets, positions, bytes) must be equal,
except where the oracle itself records a decision closer than 1e-6 relative
(a near-tie that no fp64 evaluation order can settle).
"""
import numpy as np

REL = 1e-4
ABS_FLOOR = 1e-6
NEAR_TIE = 1e-6


def close(gpu, orc, onorm, rel=REL, floor=ABS_FLOOR):
    """Boolean array: element-wise within tolerance.  onorm broadcasts against
    the leading (row) axis."""
    gpu = np.asarray(gpu, np.float64)
    orc = np.asarray(orc, np.float64)
    onorm = np.asarray(onorm, np.float64)
    while onorm.ndim < orc.ndim:
        onorm = onorm[..., None]
    return np.abs(gpu - orc) <= rel * np.abs(orc) + floor * onorm


def assert_close(gpu, orc, onorm, what, rel=REL, floor=ABS_FLOOR):
    ok = close(gpu, orc, onorm, rel, floor)
    if not ok.all():
        bad = np.argwhere(~ok)[:5]
        g = np.asarray(gpu, np.float64)
        o = np.asarray(orc, np.float64)
        detail = ", ".join(f"{tuple(b)}: gpu={g[tuple(b)]:.9g} oracle={o[tuple(b)]:.9g}" for b in bad)
        raise AssertionError(f"{what}: {int((~ok).sum())} of {ok.size} outside tolerance; {detail}")


def np_(t):
    return t.detach().cpu().numpy()


def row_onorm(orc_o):
    return np.linalg.norm(np.asarray(orc_o, np.float64), axis=-1)
