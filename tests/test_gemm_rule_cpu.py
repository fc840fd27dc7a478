"""CPU: the FP4 GEMM's tolerance (gpu_helpers.gemm_bound, reading R18:
exact products, binary32 accumulation in the tensor core) accepts a binary32
evaluation in the tensor core's structure -- exact products, each K = 64
step's sum rounded once and added to a binary32 accumulator -- and rejects
plausible mistakes in a GEMM over the same exports: a missing per-tensor
alpha, a dropped last K step, a block scale taken from the neighbouring
block, the even and odd elements of a byte swapped, and the scales of B's
rows taken from the neighbouring row."""
import numpy as np
import pytest

import oracle as O
from gpu_helpers import assert_gemm_close

M, N, K = 48, 40, 512


def export(rows, seed, fmt):
    rng = np.random.default_rng(seed)
    x = (rng.standard_t(5, (rows, K)) * 0.02).astype(np.float32)
    x[:, rng.choice(K, 4, replace=False)] *= 20.0      # outlier columns
    block = 32 if fmt == O.MXFP4 else 16
    c = rng.uniform(0.9, 1.1, rows * K // block).astype(np.float32).reshape(rows, -1)
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    r = O.fwd(x, fmt, crs=c, alpha=a, want_y=False, want_codes=True)
    return r["codes"], r["scales"], a


def decode(codes, scales, fmt):
    """binary64 values of an export (the oracle's decoders, as in O.fp4_gemm)."""
    block = 32 if fmt == O.MXFP4 else 16
    nib = np.empty((codes.shape[0], codes.shape[1] * 2), np.int64)
    nib[:, 0::2] = codes & 15
    nib[:, 1::2] = codes >> 4
    val = np.array([O.e2m1_value(c) for c in range(16)], np.float64)[nib]
    if fmt == O.MXFP4:
        s = np.ldexp(1.0, scales.astype(np.int64) - 127)
    else:
        s = np.array([O.e4m3_decode(b) for b in range(256)], np.float64)[scales]
    return val * np.repeat(s, block, axis=1)


def tensor_core_f32(A, B, alpha):
    """Exact products, each K = 64 step summed exactly and rounded to
    binary32, added to a binary32 accumulator; alpha applied to the sum."""
    acc = np.zeros((A.shape[0], B.shape[0]), np.float32)
    for k0 in range(0, A.shape[1], 64):
        step = (A[:, k0:k0 + 64] @ B[:, k0:k0 + 64].T).astype(np.float32)
        acc = (acc + step).astype(np.float32)
    return (acc * np.float32(alpha)).astype(np.float64)


@pytest.fixture(params=[O.MXFP4, O.NVFP4], ids=["mxfp4", "nvfp4"])
def case(request):
    fmt = request.param
    ca, sa, aa = export(M, 1, fmt)
    cb, sb, ab = export(N, 2, fmt)
    ref = O.fp4_gemm(ca, sa, cb, sb, fmt, aa, ab)
    mag = O.fp4_gemm(ca & 0x77, sa, cb & 0x77, sb, fmt, aa, ab)
    alpha = float(np.float32(aa) * np.float32(ab)) if fmt == O.NVFP4 else 1.0
    return fmt, ca, sa, cb, sb, alpha, ref, mag


def test_tensor_core_order_is_inside(case):
    fmt, ca, sa, cb, sb, alpha, ref, mag = case
    got = tensor_core_f32(decode(ca, sa, fmt), decode(cb, sb, fmt), alpha)
    assert_gemm_close(got, ref, mag, K)


def mistakes(fmt, ca, sa, cb, sb, alpha):
    A, B = decode(ca, sa, fmt), decode(cb, sb, fmt)
    sa_shift = sa.copy()
    sa_shift[:, 1] = sa[:, 0]                                  # block 1 scaled like block 0
    swapped = ((ca & 15) << 4) | (ca >> 4)                     # even / odd elements swapped
    sb_rows = sb[np.arange(N) ^ 1]                             # B scales of the neighbouring row
    out = {
        "dropped last K step": tensor_core_f32(A[:, :K - 64], B[:, :K - 64], alpha),
        "block scale of the neighbouring block": tensor_core_f32(decode(ca, sa_shift, fmt), B, alpha),
        "nibbles swapped": tensor_core_f32(decode(swapped.astype(np.uint8), sa, fmt), B, alpha),
        "B scales of the neighbouring row": tensor_core_f32(A, decode(cb, sb_rows, fmt), alpha),
    }
    if fmt == O.NVFP4:
        out["alpha missing"] = tensor_core_f32(A, B, 1.0)
    return out


def test_mistakes_fall_outside(case):
    fmt, ca, sa, cb, sb, alpha, ref, mag = case
    for what, got in mistakes(fmt, ca, sa, cb, sb, alpha).items():
        with pytest.raises(AssertionError):
            assert_gemm_close(got, ref, mag, K, what)
