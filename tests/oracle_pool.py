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
