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
    """Host array (float32, float16, or uint16 bf16 bits) -> CUDA tensor."""
    if a.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).cuda()
    if a.dtype == np.float16:
        return torch.from_numpy(np.ascontiguousarray(a)).cuda()
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


# Above this sum of |terms| a binary32 product or partial sum of the
# device's double-binary32 reduction can overflow (the raw sums carry the
# coefficient factors c_eff^2 <= 2 and one rounding on top of the scaled sum).
OVERFLOW_ABS = 2.0 ** 126


def assert_grad_close(got: np.ndarray, ref: np.ndarray, ref_abs: np.ndarray, floor: float,
                      what: str):
    """The coefficient-gradient rule: a gradient whose exact value is outside
    the binary32 range (the oracle's rounded value is infinite) must be
    non-finite; one whose sum of |terms| exceeds OVERFLOW_ABS may be
    non-finite (an intermediate overflowed; any infinity in a TwoSum chain
    turns the pair into NaN) or else must be within tolerance; every other
    gradient must be finite and within tolerance,
    |gpu - ref| <= REL |ref| + floor * ref_abs (+ the oracle's own rounding)."""
    got = got.astype(np.float64).reshape(-1)
    ref = ref.astype(np.float64).reshape(-1)
    ref_abs = ref_abs.astype(np.float64).reshape(-1)
    out_of_range = ~np.isfinite(ref)
    bad = np.flatnonzero(out_of_range & np.isfinite(got))
    if bad.size:
        i = bad[0]
        raise AssertionError(f"{what}: {bad.size} gradients beyond the binary32 range reported finite; "
                             f"first at {i}: gpu {got[i]!r}")
    may_overflow = ref_abs > OVERFLOW_ABS
    bad = np.flatnonzero(~np.isfinite(got) & ~out_of_range & ~may_overflow)
    if bad.size:
        i = bad[0]
        raise AssertionError(f"{what}: {bad.size} non-finite gradients where nothing can overflow; "
                             f"first at {i}: gpu {got[i]!r} oracle {ref[i]!r} abs-sum {ref_abs[i]!r}")
    keep = ~out_of_range & np.isfinite(got)
    got, ref, ref_abs = got[keep], ref[keep], ref_abs[keep]
    # the oracle's fp32 rounding of ref itself is within 2^-24 relative
    bound = REL * np.abs(ref) + floor * ref_abs + 2.0 ** -126
    err = np.abs(got - ref)
    bad = np.flatnonzero(~(err <= bound))
    if bad.size:
        i = bad[np.argmax(err[bad] / bound[bad])]
        raise AssertionError(f"{what}: {bad.size} of {got.size} outside tolerance; worst at {i}: "
                             f"gpu {got[i]!r} oracle {ref[i]!r} abs-sum {ref_abs[i]!r}")


def oracle_dtype(a: np.ndarray) -> int:
    return {np.dtype(np.uint16): O.BF16, np.dtype(np.float16): O.F16}.get(a.dtype, O.F32)


# ---------------------------------------------------------------------------
# AdamW: the device updates in binary32 from its own binary32 gradient, the
# oracle in binary64 from the exact gradient.  The bound is interval
# arithmetic over both: the gradient anywhere within its tolerance, every
# binary32 operation of the update rounded (u = 2^-24 per operation), the
# bias corrections 1 - beta^t (device: -expm1(t * log1p(-(1 - beta)))) within
# 16 u.  A value outside the interval is wrong.
# ---------------------------------------------------------------------------
U32 = 2.0 ** -24


def adamw_bounds(p, m, v, g, g_abs, floor, lr, beta1, beta2, eps, wd, step):
    """Intervals (lo, hi) for the device's new p, m, v (float64 arrays)."""
    f = lambda a: float(np.float32(a))
    lr, b1, b2, eps, wd = f(lr), f(beta1), f(beta2), f(eps), f(wd)
    o1, o2 = 1.0 - b1, 1.0 - b2
    p, m, v = (np.asarray(a, np.float64) for a in (p, m, v))
    g = np.asarray(g, np.float64)
    dg = (REL + 2 * U32) * np.abs(g) + floor * np.asarray(g_abs, np.float64) + 2.0 ** -126
    gl, gh = g - dg, g + dg
    gmax = np.maximum(np.abs(gl), np.abs(gh))
    tiny = 2.0 ** -148
    # first moment
    rm = 3 * U32 * (b1 * np.abs(m) + o1 * gmax) + tiny
    ml, mh = b1 * m + o1 * gl - rm, b1 * m + o1 * gh + rm
    # second moment
    g2h = gmax * gmax
    g2l = np.where((gl <= 0) & (gh >= 0), 0.0, np.minimum(gl * gl, gh * gh))
    rv = 4 * U32 * (b2 * v + o2 * g2h) + tiny
    vl, vh = b2 * v + o2 * g2l - rv, b2 * v + o2 * g2h + rv
    # denominator sqrt(v) / sqrt(1 - beta2^t) + eps
    R = 1.0 / np.sqrt(1.0 - b2 ** step)
    dl = np.sqrt(np.maximum(vl, 0.0)) * R
    dh = np.sqrt(np.maximum(vh, 0.0)) * R
    dl = dl * (1 - 20 * U32) + eps * (1 - U32)
    dh = dh * (1 + 20 * U32) + eps * (1 + U32)
    # m / den over the corners (den > 0), plus the division's error (the
    # device's approximate division: within 2 ulp; the square root's 2 ulp
    # are inside the denominator's slack above)
    c = np.stack([ml / dl, ml / dh, mh / dl, mh / dh])
    ul, uh = c.min(0), c.max(0)
    umax = np.maximum(np.abs(ul), np.abs(uh))
    ul, uh = ul - 3 * U32 * umax, uh + 3 * U32 * umax
    # p (1 - lr wd) - lr / (1 - beta1^t) * (m / den)
    S = lr / (1.0 - b1 ** step)
    pd = p * (1.0 - lr * wd)
    rp = 3 * U32 * np.abs(pd) + 23 * U32 * S * umax + tiny
    pl, ph = pd - S * uh - rp, pd - S * ul + rp
    return (pl, ph), (ml, mh), (vl, vh)


def assert_adamw_close(got, p0, m0, v0, ref, floor, lr, hp, step, what):
    """got: the device's new (p, m, v); p0, m0, v0: the values before the
    step; ref: the oracle's bwd_adamw entry for this array (its exact
    gradient 'grad', 'grad_abs', and new 'p')."""
    (pl, ph), (ml, mh), (vl, vh) = adamw_bounds(
        p0, m0, v0, ref["grad"], ref["grad_abs"], floor, lr, hp["beta1"], hp["beta2"], hp["eps"],
        hp["weight_decay"], step)
    for name, val, lo, hi in (("p", got[0], pl, ph), ("m", got[1], ml, mh), ("v", got[2], vl, vh)):
        val = np.asarray(val, np.float64).reshape(lo.shape)
        bad = np.flatnonzero(~((val >= lo) & (val <= hi)))
        if bad.size:
            i = bad[0]
            raise AssertionError(f"{what} {name}: {bad.size} of {val.size} outside the AdamW bound; "
                                 f"first at {i}: gpu {val.reshape(-1)[i]!r} not in "
                                 f"[{lo.reshape(-1)[i]!r}, {hi.reshape(-1)[i]!r}]")
    # the interval contains the oracle's exact step
    assert np.all((ref["p"] >= pl) & (ref["p"] <= ph)), f"{what}: oracle p outside its bound"


def gemm_bound(K, mag, ref):
    """Tolerance of the FP4 GEMM (R18): exact products, binary32 accumulation
    inside the tensor core -- (K/16 + 8) 2^-23 sum|A B| + 2^-23 |D|."""
    return (K / 16 + 8) * 2.0 ** -23 * np.asarray(mag) + 2.0 ** -23 * np.abs(ref) + 1e-30


def assert_gemm_close(got, ref, mag, K, what="D"):
    """got: the device's D (any float array); ref, mag: the oracle's D and
    its sum of |products| (binary64)."""
    got = np.asarray(got, np.float64)
    err = np.abs(got - ref)
    bad = np.argwhere(~(err <= gemm_bound(K, mag, ref)))
    assert bad.size == 0, (f"{what}: {len(bad)} of {got.size} outside the bound; first {tuple(bad[0])}: "
                           f"got {got[tuple(bad[0])]!r} ref {ref[tuple(bad[0])]!r}")
