"""Helpers shared by the GPU parity tests: host <-> device marshalling and
the comparison rules (bit-exact for codes, scale bytes, values and input
gradients; a relative bound for the reduced coefficient gradients)."""
import numpy as np
import torch

import oracle as O

# Coefficient-gradient tolerance: |gpu - ref| <= REL * |ref| + floor * S_abs,
# S_abs being the same sum over |mask * g * x| terms (computed by the oracle).
# REL is the 1e-5 relative bound; the floor only matters under near-total
# cancellation and is the error bound of a double-fp32 (Sum2 / renormalised
# pair) evaluation: n * 2^-48 for the n-term chains the kernels use, taken as
# 2^-40 for per-row sums (8 to 32 terms) and 2^-30 for sums over all rows.
REL = 1e-5
FLOOR_ROW = 2.0 ** -40
FLOOR_SHARED = 2.0 ** -30


def dev(a: np.ndarray) -> torch.Tensor:
    """Host array (float32, or uint16 bf16 bits) -> CUDA tensor."""
    if a.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).cuda()
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


def host(t: torch.Tensor) -> np.ndarray:
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def bits(a: np.ndarray) -> np.ndarray:
    a = np.ascontiguousarray(a)
    if a.dtype.itemsize == 4:
        return a.view(np.uint32)
    return a.view(np.uint16) if a.dtype.itemsize == 2 else a.view(np.uint8)


def assert_bits_equal(got: np.ndarray, ref: np.ndarray, what: str):
    assert got.shape == ref.shape, (what, got.shape, ref.shape)
    g, r = bits(got), bits(ref)
    bad = np.flatnonzero(g.reshape(-1) != r.reshape(-1))
    if bad.size:
        i = bad[0]
        raise AssertionError(f"{what}: {bad.size} of {g.size} differ; first at flat index {i}: "
                             f"gpu {g.reshape(-1)[i]:#x} vs oracle {r.reshape(-1)[i]:#x}")


def assert_grad_close(got: np.ndarray, ref: np.ndarray, ref_abs: np.ndarray, floor: float,
                      what: str):
    got = got.astype(np.float64).reshape(-1)
    ref = ref.astype(np.float64).reshape(-1)
    ref_abs = ref_abs.astype(np.float64).reshape(-1)
    # a gradient whose exact value, or whose sum of |terms|, is outside the
    # fp32 range is reported as non-finite (the documented precondition); it
    # carries no value to compare
    over = ~np.isfinite(ref) | (ref_abs > 2.0 ** 127)
    assert np.all(~np.isfinite(got[~np.isfinite(ref)])), f"{what}: overflowed gradient reported finite"
    got, ref, ref_abs = got[~over], ref[~over], ref_abs[~over]
    # the oracle's fp32 rounding of ref itself is within 2^-24 relative
    bound = REL * np.abs(ref) + floor * ref_abs + 2.0 ** -126
    err = np.abs(got - ref)
    bad = np.flatnonzero(~(err <= bound))
    if bad.size:
        i = bad[np.argmax(err[bad] / bound[bad])]
        raise AssertionError(f"{what}: {bad.size} of {got.size} outside tolerance; worst at {i}: "
                             f"gpu {got[i]!r} oracle {ref[i]!r} abs-sum {ref_abs[i]!r}")


def oracle_dtype(a: np.ndarray) -> int:
    return O.BF16 if a.dtype == np.uint16 else O.F32
