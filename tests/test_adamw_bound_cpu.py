"""The AdamW tolerance of the GPU tests, checked on the CPU: a binary32
evaluation in the device's operation order, from any gradient within the
gradient tolerance and with its square root and division off by up to 2 ulp
(the device's approximate forms), lies inside the interval; the same
evaluation with a plausible mistake in the update does not."""
import numpy as np
import pytest

import oracle as O
from gpu_helpers import FLOOR_ROW, REL, adamw_bounds

F = np.float32


def ulps(a, k):
    """Binary32 values a moved by k units in the last place."""
    a = np.asarray(a, F)
    towards = F(np.inf) if k > 0 else F(-np.inf)
    for _ in range(abs(k)):
        a = np.nextafter(a, towards)
    return a


def device_order_f32(p, g, m, v, lr, b1, b2, eps, wd, t, mistake=None, sqrt_ulps=0, div_ulps=0):
    """The fused kernel's update in binary32 (each line one rounding); the
    kernel's square root and division are approximations within 2 ulp,
    modelled by moving the correctly rounded ones by sqrt_ulps / div_ulps."""
    p, g, m, v = (np.asarray(a, F) for a in (p, g, m, v))
    lr, b1, b2, eps, wd = F(lr), F(b1), F(b2), F(eps), F(wd)
    o1, o2 = F(1) - b1, F(1) - b2
    tt = F(t)
    bc1 = -np.expm1(tt * np.log1p(-o1))
    bc2 = -np.expm1(tt * np.log1p(-o2))
    if mistake == "no_bias_correction":
        bc1 = bc2 = F(1)
    rbc2 = F(1) / np.sqrt(bc2)
    step = lr / bc1
    decay = F(1.0 - float(lr) * float(wd))
    if mistake == "no_decay":
        decay = F(1)
    if mistake == "swapped_betas":
        b1, b2, o1, o2 = b2, b1, o2, o1
    m = b1 * m + o1 * g
    v = b2 * v + o2 * (g * g)
    den = ulps(np.sqrt(v), sqrt_ulps) * rbc2 + eps
    if mistake == "eps_inside_sqrt":
        den = np.sqrt(v * rbc2 * rbc2 + eps)
    return p * decay - step * ulps(m / den, div_ulps), m, v


def cases(rng, n):
    p = rng.uniform(0.5, 1.5, n)
    g = rng.standard_normal(n) * 10.0 ** rng.uniform(-8, 2, n)
    g_abs = np.abs(g) * rng.uniform(1, 50, n)
    m = rng.standard_normal(n) * 10.0 ** rng.uniform(-6, 0, n)
    v = 10.0 ** rng.uniform(-12, 1, n)
    return p, g, g_abs, m, v


@pytest.mark.parametrize("step", [1, 2, 7, 1000, 10 ** 6])
@pytest.mark.parametrize("lr", [1e-3, 5e-3, 2e-2, 5e-2])
def test_device_order_within_bound(step, lr):
    rng = np.random.default_rng(step * 7 + int(lr * 1e4))
    n = 20000
    p, g, g_abs, m, v = cases(rng, n)
    m = m.astype(F).astype(np.float64)
    v = v.astype(F).astype(np.float64)
    p = p.astype(F).astype(np.float64)
    if step == 1:
        m[:] = 0
        v[:] = 0
    hp = (0.9, 0.999, 1e-8, 0.01)
    (pl, ph), (ml, mh), (vl, vh) = adamw_bounds(p, m, v, g, g_abs, FLOOR_ROW, lr, *hp, step)
    # the exact step is inside
    pe, me, ve = O.adamw(p, g, m, v, lr, *hp, step)
    assert np.all((pe >= pl) & (pe <= ph)) and np.all((me >= ml) & (me <= mh))
    assert np.all((ve >= vl) & (ve <= vh))
    # the device's binary32 step from any gradient within tolerance is inside
    dg = REL * np.abs(g) + FLOOR_ROW * g_abs
    for s in (-1.0, 1.0, None):
        gd = g + (dg * s if s is not None else dg * rng.uniform(-1, 1, n))
        for su, du in ((0, 0), (2, 2), (-2, -2), (2, -2), (-2, 2)):
            pd, md, vd = device_order_f32(p, gd.astype(F), m, v, lr, *hp, step, sqrt_ulps=su, div_ulps=du)
            for val, lo, hi in ((pd, pl, ph), (md, ml, mh), (vd, vl, vh)):
                val = val.astype(np.float64)
                assert np.all((val >= lo) & (val <= hi)), (su, du)


@pytest.mark.parametrize("mistake", ["no_bias_correction", "no_decay", "swapped_betas",
                                     "eps_inside_sqrt"])
def test_mistakes_fall_outside(mistake):
    rng = np.random.default_rng(5)
    n = 4000
    p, g, g_abs, m, v = cases(rng, n)
    p = p.astype(F).astype(np.float64)
    m = (np.sign(g) * np.abs(m)).astype(F).astype(np.float64)
    v = (g * g * rng.uniform(0.5, 2, n)).astype(F).astype(np.float64)
    hp = (0.9, 0.999, 1e-8, 0.01)
    (pl, ph), _, _ = adamw_bounds(p, m, v, g, g_abs, FLOOR_ROW, 5e-2, *hp, 3)
    pd, _, _ = device_order_f32(p, g.astype(F), m, v, 5e-2, *hp, 3, mistake=mistake)
    out = ~((pd >= pl) & (pd <= ph))
    assert out.mean() > 0.5, (mistake, out.mean())
