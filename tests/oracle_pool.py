"""Worker for running the oracle over row ranges in a spawn-started process
pool (kept free of torch so that workers start quickly)."""
import numpy as np

import oracle as O


def shared_rows_chunk(args):
    """Oracle shared-row backward over rows [r0, r1) of the inputs stored in
    a (2, rows, cols) uint16 .npy file (x, g as bf16 bits).  Returns the
    binary64 gradient sums and term-magnitude sums of the range."""
    path, r0, r1, fmt, alpha, crs, dgs, sub = args
    mm = np.load(path, mmap_mode="r")
    x = np.ascontiguousarray(mm[0, r0:r1])
    g = np.ascontiguousarray(mm[1, r0:r1])
    out = O.bwd(x, g, fmt, crs=crs, dgs=dgs, alpha=alpha, sub=sub, shared=True, want_gx=False,
                want_abs=True, want_f64=True)
    return out["gcrs64"], out["gdgs64"], out["gcrs_abs"], out["gdgs_abs"]


def step_reference(lo, hi, first, switch_bits):
    """The value of a monotone step function of the binary32 bit patterns
    lo .. hi-1 (positive floats: order of bits = order of values): `first`
    below the first switch, one more from each pattern in `switch_bits` on."""
    pos = np.clip(np.asarray(switch_bits, np.int64) - lo, 0, hi - lo)
    counts = np.diff(np.concatenate([[0], pos, [hi - lo]]))
    return np.repeat(np.arange(first, first + len(counts)), counts)


def format_sweep_chunk(args):
    """Oracle format conversion over the binary32 patterns lo .. hi-1 against
    the step function (first, switch_bits), the result capped at `cap`.
    Returns the first pattern where they differ, or -1."""
    kind, lo, hi, first, switch_bits, cap = args
    x = np.arange(lo, hi, dtype=np.uint32).view(np.float32)
    if kind == "e4m3":
        got = O.e4m3_encode(x).astype(np.int64)
    else:
        got = O.e8m0_exponent(x, O.MX_CEIL if kind == "e8m0_ceil" else O.MX_FLOOR).astype(np.int64)
    ref = np.minimum(step_reference(lo, hi, first, switch_bits), cap)
    bad = np.flatnonzero(got != ref)
    return int(lo + bad[0]) if bad.size else -1
