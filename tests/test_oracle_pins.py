"""Pins for the CPU oracle (no GPU).

Each test ties the oracle to something other than itself: values worked by
hand from the paper's definitions, library conversions (torch float8 /
bfloat16), brute-force or independent numpy formulations, invariants the
paper states, and finite differences of the STE surrogate.  A plausible slip
in the oracle (dropped term, sign, index, transposed operand, off-by-one in an
exponent rule, wrong tie rule) fails at least one of them.
"""
import math
import os

import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_01847_gb300 import workloads as W


def f32(a):
    return np.asarray(a, dtype=np.float32)


# ---------------------------------------------------------------------------
# independent numpy restatements used only as pins
# ---------------------------------------------------------------------------
def e2m1_ref(u):
    """E2M1 round-to-nearest-even by spacing: 0.5 below 2, 1 in [2,4), 2 from
    4, saturated at 6; np.round rounds half to even, which on each spacing is
    the even E2M1 code.  Returns signed float64 values."""
    u = np.asarray(u, dtype=np.float64)
    a = np.abs(u)
    q = np.where(a < 2, np.round(a * 2) / 2, np.where(a < 4, np.round(a), 2 * np.round(a / 2)))
    q = np.minimum(q, 6.0)
    return np.copysign(q, u)


GRID = np.array([0, 0.5, 1, 1.5, 2, 3, 4, 6], np.float64)


def code_to_value(code):
    code = np.asarray(code).astype(np.int64)
    mag = GRID[code & 7]
    return np.where(code & 8, -mag, mag)


def e8m0_ceil_ref(m):
    """Smallest e with m <= 6 * 2^e (Eq. 3's ceiling of log2(m / 6), exact),
    clamped to [-127, 127]: start one below floor(log2 m) - 2 and step up
    while 6 * 2^e < m (binary64 products, exact)."""
    m = f32(m).astype(np.float64)
    out = np.full(m.shape, -127, np.int64)
    nz = m > 0
    _, ex = np.frexp(m[nz])                       # m in [2^(ex-1), 2^ex)
    e = ex.astype(np.int64) - 4
    for _ in range(3):
        e = np.where(6.0 * np.exp2(e.astype(np.float64)) < m[nz], e + 1, e)
    out[nz] = e
    return np.clip(out, -127, 127)


def e8m0_floor_ref(m):
    m = f32(m)
    out = np.full(m.shape, -127, np.int64)
    nz = m > 0
    mant, ex = np.frexp(m[nz].astype(np.float64))   # m = mant * 2^ex, mant in [0.5,1)
    out[nz] = (ex - 1) - 2
    return np.clip(out, -127, 127)


def torch_e4m3(r):
    return torch.from_numpy(f32(r)).to(torch.float8_e4m3fn).view(torch.uint8).numpy()


def torch_bf16_bits(f):
    return torch.from_numpy(f32(f)).to(torch.bfloat16).view(torch.int16).numpy().astype(np.uint16)


# ---------------------------------------------------------------------------
# hand-worked blocks (computed by hand from Eq. 1-3, 6-7)
# ---------------------------------------------------------------------------
def test_hand_mxfp4_block_crs():
    # m = 1.5 -> fl(1.5/6) = 0.25 = 2^-2 -> e = -2, E8M0 byte 125 (0x7D), S^dq = 0.25
    x = np.zeros((1, 32), np.float32)
    x[0, :4] = [0.7, -0.26, 0.13, 1.5]
    out = O.fwd(x, O.MXFP4, want_codes=True)
    assert out["scales"][0, 0] == 0x7D
    # c = 1: u = [2.8, -1.04, 0.52, 6.0] -> codes [5, 0xA, 1, 7], y = [0.75, -0.25, 0.125, 1.5]
    assert list(out["codes"][0, :2]) == [0xA5, 0x71]
    assert np.all(out["codes"][0, 2:] == 0)
    assert list(out["y"][0, :4]) == [0.75, -0.25, 0.125, 1.5]
    assert np.all(out["y"][0, 4:] == 0)
    # c = 1.25: S^q = 0.3125, u = [2.24, -0.832, 0.416, 4.8] -> codes [4, 0xA, 1, 6]
    crs = np.array([[1.25]], np.float32)
    out = O.fwd(x, O.MXFP4, crs=crs, want_codes=True)
    assert out["scales"][0, 0] == 0x7D            # S^dq is unchanged by c
    assert list(out["codes"][0, :2]) == [0xA4, 0x61]
    assert list(out["y"][0, :4]) == [0.5, -0.25, 0.125, 1.0]
    # STE backward with g = 1 on the first four: gx = g * fl(S^dq / S^q) = fl(0.25 / 0.3125)
    g = np.zeros_like(x)
    g[0, :4] = 1
    b = O.bwd(x, g, O.MXFP4, crs=crs)
    assert np.all(b["gx"][0, :4] == np.float32(0.8))
    assert np.all(b["gx"][0, 4:] == 0)
    # dL/dc = -(0.7 - 0.26 + 0.13 + 1.5) / 1.25^2 = -1.3248 (inputs as float32)
    expect = -(float(np.float32(0.7)) + float(np.float32(-0.26)) + float(np.float32(0.13)) + 1.5) / 1.5625
    assert b["gcrs"][0, 0] == pytest.approx(expect, rel=1e-7)
    assert expect == pytest.approx(-1.3248, abs=1e-6)


def test_hand_gx_rounding_order():
    """The STE input gradient rounds the scale ratio once (dy/dx = S^dq / S^q,
    Sec. 3.2): gx = fl(g * fl(S^dq / S^q)).  Evaluating the chain rule term by
    term instead, fl(fl(g * S^dq) / S^q), rounds differently for some g; this
    block is one of them.  Worked by hand, binary32, integers x 2^-k exact:

      S^dq = 0.25 (the block above, m = 1.5), c = 1.25, S^q = 0.3125 (exact)
      rho  = fl(0.25 / 0.3125) = fl(0.8):  0.8 * 2^24 = 13421772.8
             -> 13421773 * 2^-24                              (0x3F4CCCCD)
      g    = 1.125 = 9 / 8
      ratio order:   g * rho = 9 * 13421773 * 2^-27 = 120795957 * 2^-27
             in [0.5, 1) the spacing is 2^-24: 120795957 / 8 = 15099494.625
             -> 15099495 * 2^-24 = 0.90000004                  (0x3F666667)
      chain order:   fl(g * S^dq) = 0.28125 (exact), 0.28125 / 0.3125 = 0.9:
             0.9 * 2^24 = 15099494.4 -> 15099494 * 2^-24 = 0.9 (0x3F666666)
    The oracle (and the kernels, which it checks bit for bit) take the ratio
    order: the expected bits are the first ones."""
    x = np.zeros((1, 32), np.float32)
    x[0, :4] = [0.7, -0.26, 0.13, 1.5]
    crs = np.array([[1.25]], np.float32)
    g = np.zeros_like(x)
    g[0, :4] = 1.125
    gx = O.bwd(x, g, O.MXFP4, crs=crs)["gx"]
    assert list(gx[0, :4].view(np.uint32)) == [0x3F666667] * 4
    assert np.all(gx[0, 4:] == 0)
    # the two orders really differ here (numpy binary32 arithmetic)
    chain = np.float32(np.float32(np.float32(1.125) * np.float32(0.25)) / np.float32(0.3125))
    assert chain.view(np.uint32) == 0x3F666666
    # the same bits through a DGS coefficient (c_eff = c^k = 1.25), sub-block 8
    dgs = np.array([[1.25, 1.0, 1.0, 1.0]], np.float32)
    gx = O.bwd(x, g, O.MXFP4, dgs=dgs)["gx"]
    assert list(gx[0, :4].view(np.uint32)) == [0x3F666667] * 4


def test_hand_mxfp4_ties():
    # S^q = 0.25 (m = 1.5): 0.625 -> u = 2.5 (tie 2|3 -> 2, code 4); 1.25 -> 5
    # (tie 4|6 -> 4, code 6); 0.0625 -> 0.25 (tie 0|0.5 -> 0); -0.0625 -> -0 (0x8)
    x = np.zeros((1, 32), np.float32)
    x[0, :6] = [1.5, 0.625, 1.25, 0.0625, -0.0625, 0.1875]
    out = O.fwd(x, O.MXFP4, want_codes=True)
    codes = [(out["codes"][0, i // 2] >> (4 * (i % 2))) & 15 for i in range(6)]
    # 0.1875 -> u = 0.75 (tie 0.5|1 -> 1.0, code 2)
    assert codes == [7, 4, 6, 0, 8, 2]
    y = out["y"][0, :6]
    assert list(y) == [1.5, 0.5, 1.0, 0.0, 0.0, 0.25]
    assert not np.signbit(y[3]) and np.signbit(y[4])   # -0 kept for the negative tie


def test_hand_nvfp4_blocks():
    # amax = 0.65625 = 21/32 and 2688 = 21 * 128 -> alpha = 2^-12 exactly
    x = np.zeros((1, 32), np.float32)
    x[0, 0] = 0.65625
    x[0, 16] = 0.1
    a = O.alpha(x)
    assert a == 2.0 ** -12
    out = O.fwd(x, O.NVFP4, alpha=a, want_codes=True)
    # block 0: r = 0.65625 / (6 * 2^-12) = 448 -> E4M3 0x7E, S^dq = 448 * 2^-12
    assert out["scales"][0, 0] == 0x7E
    assert out["y"][0, 0] == np.float32(0.65625)
    # block 1: r = fl(0.1 / (6 * 2^-12)) = 68.27 -> nearest E4M3 is 72 (0x69),
    # S^dq = 72 * 2^-12 = 0.017578125, u = 0.1 / S^dq = 5.69 -> 6 (code 7)
    assert out["scales"][0, 1] == 0x69
    assert out["codes"][0, 8] & 15 == 7
    assert out["y"][0, 16] == np.float32(6 * 0.017578125)


def test_alpha_closed_form():
    for k in (-20, -3, 0, 5):
        x = np.zeros((3, 16), np.float32)
        x[1, 7] = -2688.0 * 2.0 ** k
        assert O.alpha(x) == 2.0 ** k
    assert O.alpha(np.zeros((2, 16), np.float32)) == 0.0


# ---------------------------------------------------------------------------
# format codecs against libraries / brute force
# ---------------------------------------------------------------------------
def test_e4m3_decode_matches_torch():
    b = np.arange(256, dtype=np.uint8)
    ref = torch.from_numpy(b).view(torch.float8_e4m3fn).float().numpy()
    ours = np.array([O.e4m3_decode(int(i)) for i in b], np.float32)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan) and nan.sum() == 2   # 0x7F, 0xFF
    assert np.array_equal(ours[~nan].view(np.uint32), ref[~nan].view(np.uint32))


def _near_boundaries(hi_max):
    """Every float32 whose upper 16 bits are <= hi_max and whose lower 16 bits
    are one of a few patterns around 0 and 0x8000: this hits every E4M3 (and
    bf16) rounding midpoint and its neighbours one ulp away."""
    hi = np.arange(0, hi_max + 1, dtype=np.uint32) << 16
    lo = np.array([0x0000, 0x0001, 0x0002, 0x7FFF, 0x8000, 0x8001, 0xFFFE, 0xFFFF], np.uint32)
    return (hi[:, None] | lo[None, :]).reshape(-1).view(np.float32)


def test_e4m3_encode_matches_torch_rne():
    r = _near_boundaries(0x43E7)                      # up to ~463.9 (midpoint 448|480 is 464)
    r = r[np.isfinite(r) & (r < 464.0)]
    rng = np.random.default_rng(7)
    r = np.concatenate([r, rng.uniform(0, 463.9, 200000).astype(np.float32)])
    assert np.array_equal(O.e4m3_encode(r), torch_e4m3(r))


def test_e4m3_saturates():
    big = f32([448.0, 464.0, 470.0, 1e4, 3e38, np.inf])
    assert np.all(O.e4m3_encode(big) == 0x7E)


def test_e2m1_matches_independent_rounding():
    rng = np.random.default_rng(11)
    mids = np.array([0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0, 6.0], np.float32)
    near = np.concatenate([np.nextafter(mids, np.float32(0)), mids, np.nextafter(mids, np.float32(9))])
    u = np.concatenate([rng.uniform(-8, 8, 400000).astype(np.float32),
                        near, -near, f32([0.0, -0.0, 7.9, -100.0, 1e30])])
    codes = O.e2m1_codes(u)
    ref = e2m1_ref(u)
    got = code_to_value(codes)
    assert np.array_equal(got, ref)
    # sign bit is the sign of u, also when the value rounds to zero
    assert np.array_equal((codes >> 3).astype(bool), np.signbit(u))


def test_e2m1_brute_force_grid():
    """Tiny blocks: each code is the argmin over all 15 signed E2M1 values."""
    vals = np.array(sorted(set(list(GRID) + list(-GRID))), np.float64)
    rng = np.random.default_rng(3)
    u = rng.uniform(-7, 7, 20000).astype(np.float32)
    codes = O.e2m1_codes(u)
    d = np.abs(u[:, None].astype(np.float64) - vals[None, :])
    best = vals[np.argmin(d, axis=1)]
    got = code_to_value(codes)
    not_tie = np.sort(d, axis=1)[:, 1] > np.sort(d, axis=1)[:, 0]
    assert np.array_equal(got[not_tie], best[not_tie])
    assert np.all(np.abs(got - u) <= np.min(d, axis=1) + 0.0)


def test_e8m0_ceil_and_floor_rules():
    rng = np.random.default_rng(5)
    pieces = []
    for e in range(-150, 126):                        # around 6 * 2^e for every e
        base = np.float32(6.0) * np.float32(2.0) ** np.float32(e) if e > -150 else np.float32(0)
        if not np.isfinite(base) or base == 0:
            continue
        pieces.append(np.array([base, np.nextafter(base, np.float32(0)),
                                np.nextafter(base, np.float32(np.inf))], np.float32))
        pieces.append(np.float32(2.0) ** np.float32(e) * f32([1, 1.5, 1.9999999]))
    subn = np.arange(1, 5000, dtype=np.uint32).view(np.float32)
    rand = rng.integers(1, 0x7F800000, 2_000_000, dtype=np.uint32).view(np.float32)
    m = np.concatenate(pieces + [subn, rand, f32([0.0, 3.4e38])])
    m = m[np.isfinite(m) & (m >= 0)]
    assert np.array_equal(O.e8m0_exponent(m, O.MX_CEIL), e8m0_ceil_ref(m))
    assert np.array_equal(O.e8m0_exponent(m, O.MX_FLOOR), e8m0_floor_ref(m))


CHUNK = 1 << 24


def _sweep(kind, top, first, switch_bits, cap):
    """Every binary32 pattern below `top` (from 1; from 0 for E4M3), in
    chunks over a spawn-started process pool."""
    import concurrent.futures as cf
    import multiprocessing as mp
    import oracle_pool
    lo0 = 0 if kind == "e4m3" else 1
    jobs = [(kind, lo, min(lo + CHUNK, top), first, switch_bits, cap) for lo in range(lo0, top, CHUNK)]
    with cf.ProcessPoolExecutor(max_workers=min(16, os.cpu_count() or 1),
                                mp_context=mp.get_context("spawn")) as ex:
        bad = [b for b in ex.map(oracle_pool.format_sweep_chunk, jobs) if b >= 0]
    assert not bad, (kind, hex(bad[0]))


def test_e8m0_exhaustive():
    """Every positive finite binary32 m: the ceiling rule is the smallest e
    with m <= 6 * 2^e (it steps up right after each 6 * 2^e), the floor rule
    floor(log2 m) - 2 (it steps up at each power of two), both clamped to
    [-127, 127]."""
    six = [int(np.float32(6.0 * 2.0 ** e).view(np.uint32)) + 1 for e in range(-127, 126)]
    pow2 = [int(np.float32(2.0 ** k).view(np.uint32)) for k in range(-124, 128)]
    _sweep("e8m0_ceil", 0x7F800000, -127, six, 127)
    _sweep("e8m0_floor", 0x7F800000, -127, pow2, 127)


def test_e4m3_exhaustive():
    """Every binary32 r in [0, 500]: the code is the nearest finite E4M3
    value (the table decoded from bias-7 arithmetic), ties to the even code,
    saturating at 448 -- a step function that switches at each midpoint of
    two neighbouring values, after it when the lower code is even."""
    vals = [O.e4m3_decode(b) for b in range(0x7F)]          # 0x00 .. 0x7E, increasing
    assert all(a < b for a, b in zip(vals, vals[1:]))
    switches = []
    for c in range(0x7E):
        mid = (vals[c] + vals[c + 1]) / 2.0
        assert float(np.float32(mid)) == mid                  # every midpoint is a binary32
        bits = int(np.float32(mid).view(np.uint32))
        switches.append(bits + 1 if c % 2 == 0 else bits)
    _sweep("e4m3", int(np.float32(500.0).view(np.uint32)) + 1, 0, switches, 0x7E)


def test_e8m0_ceil_never_saturates():
    """Under the ceiling rule the block maximum never exceeds 6 * 2^e, so at
    c = 1 no element saturates; and 2^e is the tightest such power."""
    rng = np.random.default_rng(9)
    m = rng.integers(0x00800000, 0x7F000000, 1_000_000, dtype=np.uint32).view(np.float32)
    # where fl(m / 6) is subnormal it can round onto 2^-127: 0x01400001 is
    # just above 6 * 2^-127 and needs e = -126
    m = np.concatenate([m, np.array([0x01400000, 0x01400001, 0x01400002], np.uint32).view(np.float32)])
    e = O.e8m0_exponent(m, O.MX_CEIL).astype(np.float64)
    ok = e < 127
    ratio = m[ok].astype(np.float64) / np.exp2(e[ok])
    assert np.all(ratio <= 6.0)
    inner = ok & (e > -127)
    assert np.all(m[inner].astype(np.float64) / np.exp2(e[inner] - 1) > 6.0)


def test_bf16_rne_matches_torch():
    r = _near_boundaries(0xFFFF)
    r = r[np.isfinite(r)]
    rng = np.random.default_rng(13)
    r = np.concatenate([r, rng.standard_normal(100000).astype(np.float32),
                        f32([3.4e38, -3.4e38, 1e-45, -1e-45])])
    assert np.array_equal(O.bf16_rne(r), torch_bf16_bits(r))


# ---------------------------------------------------------------------------
# invariants the paper states
# ---------------------------------------------------------------------------
def rtn_reference(x, fmt, alpha=0.0, block=None):
    """Standard MXFP4 / NVFP4 round-to-nearest (Eq. 1-3), written in numpy
    with torch's float8 conversion for E4M3: the c = 1 baseline."""
    x = f32(x)
    block = block or (32 if fmt == O.MXFP4 else 16)
    rows, cols = x.shape
    xb = x.reshape(rows, cols // block, block)
    m = np.abs(xb).max(axis=2)
    if fmt == O.MXFP4:
        s = np.exp2(e8m0_ceil_ref(m)).astype(np.float32)
    else:
        den = np.float32(alpha) * np.float32(6)
        with np.errstate(divide="ignore", invalid="ignore"):
            r = (m / den).astype(np.float32)
        r = np.where(m == 0, np.float32(0), np.minimum(r, np.float32(448)))
        delta = torch.from_numpy(torch_e4m3(r)).view(torch.float8_e4m3fn).float().numpy()
        s = (delta * np.float32(alpha)).astype(np.float32)
    s3 = s[:, :, None]
    with np.errstate(divide="ignore", invalid="ignore"):
        u = (xb / s3).astype(np.float32)
    q = e2m1_ref(u).astype(np.float32)
    y = (q * s3).astype(np.float32)
    y = np.where(s3 == 0, np.float32(0), y)
    return y.reshape(rows, cols)


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_crs_at_one_equals_rtn(fmt):
    """Starting from c = 1 the method is the baseline (Sec. 3.3): with all
    coefficients 1 the fake-quant equals standard RTN bit for bit."""
    w = W.WORKLOADS["w256x512_f32"]
    x = W.draw_values(w, 64, 512, 42)
    x[3, 16:32] = 0                                  # an all-zero block
    x[5, :32] *= 1e-30                               # tiny values (subnormal scales)
    block = 32 if fmt == O.MXFP4 else 16
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    ones_c = np.ones((64, 512 // block), np.float32)
    ones_d = np.ones((64, 512 // 8), np.float32)
    y = O.fwd(x, fmt, crs=ones_c, dgs=ones_d, alpha=a)["y"]
    ref = rtn_reference(x, fmt, alpha=a)
    assert np.array_equal(y.view(np.uint32), ref.view(np.uint32))
    y0 = O.fwd(x, fmt, alpha=a)["y"]
    assert np.array_equal(y0.view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_dgs_with_block_sized_subblocks_is_crs(fmt):
    """Sub-block size equal to the block size reduces DGS to CRS (Sec. 3.4,
    Table 5)."""
    w = W.WORKLOADS["llama3_8b_block"]
    x = W.to_bf16_bits(W.draw_values(w, 32, 256, 17))
    g = W.to_bf16_bits(W.draw_grad(32, 256, 18))
    block = 32 if fmt == O.MXFP4 else 16
    coef = W.draw_coefs(w, 32 * 256 // block, 19).reshape(32, -1)
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    f_c = O.fwd(x, fmt, crs=coef, alpha=a, sub=block, want_codes=True)
    f_d = O.fwd(x, fmt, dgs=coef, alpha=a, sub=block, want_codes=True)
    for k in ("y", "codes", "scales"):
        assert np.array_equal(f_c[k], f_d[k])
    b_c = O.bwd(x, g, fmt, crs=coef, alpha=a, sub=block)
    b_d = O.bwd(x, g, fmt, dgs=coef, alpha=a, sub=block)
    assert np.array_equal(b_c["gx"], b_d["gx"])
    assert np.array_equal(b_c["gcrs"], b_d["gdgs"])


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_dequant_of_export_equals_forward(fmt, dtype):
    """The deployed model (codes + scale bytes, Fig. 3(d)) reproduces the
    fake-quantized forward output exactly."""
    w = W.WORKLOADS["w256x512_f32"]
    x = W.draw_values(w, 40, 512, 23)
    x[1, :64] = 0
    crs = W.draw_coefs(w, 40 * 512 // 32, 24).reshape(40, -1)
    dgs = W.draw_coefs(w, 40 * 512 // 8, 25).reshape(40, -1)
    if dtype == "bf16":
        x = W.to_bf16_bits(x)
    block = 32 if fmt == O.MXFP4 else 16
    if fmt == O.NVFP4:
        crs = W.draw_coefs(w, 40 * 512 // 16, 24).reshape(40, -1)
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    out = O.fwd(x, fmt, crs=crs, dgs=dgs, alpha=a, want_codes=True)
    dq = O.dequant(out["codes"], out["scales"], fmt, alpha=a, block=block,
                   dtype=O.F32 if dtype == "f32" else O.BF16)
    assert np.array_equal(dq, out["y"])


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_input_gradient_at_c1_is_g(fmt):
    """At c = 1 the two scales coincide, S^dq / S^q = 1, and the STE passes
    the gradient through unchanged (live blocks)."""
    w = W.WORKLOADS["w256x512_f32"]
    x = W.draw_values(w, 16, 512, 31)
    g = W.draw_grad(16, 512, 32)
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    b = O.bwd(x, g, fmt, alpha=a)
    assert np.array_equal(b["gx"], g)


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_input_gradient_is_g_over_c(fmt):
    """dy/dx of the relaxed surrogate is S^dq / S^q = 1 / (c_i c_i^k): the
    input gradient equals g / c_eff up to the roundings of S^q, of the ratio
    and of the product, i.e. within 2^-22 relative."""
    rng = np.random.default_rng(41)
    block = 32 if fmt == O.MXFP4 else 16
    x = (rng.standard_normal((8, 4 * block)) * 0.02).astype(np.float32)
    g = rng.standard_normal(x.shape).astype(np.float32)
    crs = rng.uniform(0.8, 1.2, (8, 4)).astype(np.float32)
    dgs = rng.uniform(0.8, 1.2, (8, 4 * block // 8)).astype(np.float32)
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    b = O.bwd(x, g, fmt, crs=crs, dgs=dgs, alpha=a)
    ceff = np.repeat(crs.astype(np.float64), block, 1) * np.repeat(dgs.astype(np.float64), 8, 1)
    expect = g.astype(np.float64) / ceff
    np.testing.assert_allclose(b["gx"].astype(np.float64), expect, rtol=2.0 ** -22, atol=0)


# ---------------------------------------------------------------------------
# gradients: finite differences of the STE surrogate, autograd restatement
# ---------------------------------------------------------------------------
def surrogate_loss(x, g, crs, dgs, sdq_mask, block, sub):
    """Identity-STE surrogate: ytilde = (x / S^q) * S^dq = x / (c_i c_i^k) on
    live sub-blocks, so L = sum g * x / (c_i c_i^k); evaluated in float64."""
    rows, cols = x.shape
    c = np.repeat(crs, block, axis=1)
    d = np.repeat(dgs, sub, axis=1)
    return float(np.sum(g * x / (c * d) * sdq_mask))


@pytest.mark.parametrize("fmt,sub", [(O.MXFP4, 8), (O.MXFP4, 32), (O.NVFP4, 8), (O.NVFP4, 4)])
def test_coefficient_gradients_finite_difference(fmt, sub):
    rng = np.random.default_rng(100 + sub)
    block = 32 if fmt == O.MXFP4 else 16
    rows, cols = 3, 2 * block
    x = rng.standard_normal((rows, cols)).astype(np.float32)
    g = rng.standard_normal((rows, cols)).astype(np.float32)
    crs = rng.uniform(0.8, 1.2, (rows, cols // block)).astype(np.float32)
    dgs = rng.uniform(0.8, 1.2, (rows, cols // sub)).astype(np.float32)
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    b = O.bwd(x, g, fmt, crs=crs, dgs=dgs, alpha=a, sub=sub)
    x64, g64 = x.astype(np.float64), g.astype(np.float64)
    c64, d64 = crs.astype(np.float64), dgs.astype(np.float64)
    live = np.ones_like(x64)
    for arr, grad in ((c64, b["gcrs"]), (d64, b["gdgs"])):
        for idx in np.ndindex(arr.shape):
            h = 1e-6 * arr[idx]
            old = arr[idx]
            arr[idx] = old + h
            lp = surrogate_loss(x64, g64, c64, d64, live, block, sub)
            arr[idx] = old - h
            lm = surrogate_loss(x64, g64, c64, d64, live, block, sub)
            arr[idx] = old
            fd = (lp - lm) / (2 * h)
            assert grad[idx] == pytest.approx(fd, rel=1e-6, abs=1e-9)


def test_shared_row_gradients_sum_over_rows():
    """Shared coefficients: the gradient is the per-row gradient summed over
    rows (checked against the oracle's own per-row mode with broadcast
    coefficients, and against finite differences)."""
    rng = np.random.default_rng(77)
    rows, cols, block, sub = 5, 64, 32, 8
    x = rng.standard_normal((rows, cols)).astype(np.float32)
    g = rng.standard_normal((rows, cols)).astype(np.float32)
    crs = rng.uniform(0.9, 1.1, (1, cols // block)).astype(np.float32)
    dgs = rng.uniform(0.9, 1.1, (1, cols // sub)).astype(np.float32)
    sh = O.bwd(x, g, O.MXFP4, crs=crs, dgs=dgs, shared=True)
    pr = O.bwd(x, g, O.MXFP4, crs=np.repeat(crs, rows, 0), dgs=np.repeat(dgs, rows, 0))
    assert np.array_equal(sh["gx"], pr["gx"])
    np.testing.assert_allclose(sh["gcrs"][0], pr["gcrs"].astype(np.float64).sum(0), rtol=1e-6)
    np.testing.assert_allclose(sh["gdgs"][0], pr["gdgs"].astype(np.float64).sum(0), rtol=1e-6)
    fw = O.fwd(x, O.MXFP4, crs=crs, dgs=dgs, shared=True)
    fw2 = O.fwd(x, O.MXFP4, crs=np.repeat(crs, rows, 0), dgs=np.repeat(dgs, rows, 0))
    assert np.array_equal(fw["y"], fw2["y"])


def torch_fake_quant(x, crs, dgs, sdq, block, sub):
    """PyTorch autograd restatement of y = STE(Q(x / S^q)) * S^dq with
    S^q = S^dq * (c * c^k): the straight-through trick u + (Q(u) - u).detach()."""
    rows, cols = x.shape
    c = crs.repeat_interleave(block, dim=1)
    d = dgs.repeat_interleave(sub, dim=1)
    s = sdq.repeat_interleave(block, dim=1)
    s_q = s * (c * d)
    u = x / s_q
    q = torch.from_numpy(e2m1_ref(u.detach().numpy())).to(u.dtype)
    return (u + (q - u).detach()) * s


def torch_ste_ratio(x, crs, dgs, sdq, block, sub):
    """The same forward written as y = x * rho + (Q(x / S^q) * S^dq - x * rho).detach()
    with the scale ratio rho = S^dq / S^q: autograd's input gradient is g * rho."""
    c = crs.repeat_interleave(block, dim=1)
    d = dgs.repeat_interleave(sub, dim=1)
    s = sdq.repeat_interleave(block, dim=1)
    s_q = s * (c * d)
    rho = (s / s_q).detach()
    q = torch.from_numpy(e2m1_ref((x / s_q).detach().numpy())).to(x.dtype)
    return x * rho + (q * s - x * rho).detach()


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_autograd_restatement(fmt):
    rng = np.random.default_rng(55)
    block = 32 if fmt == O.MXFP4 else 16
    sub = 8
    rows, cols = 6, 4 * block
    x = (rng.standard_normal((rows, cols)) * 0.02).astype(np.float32)
    g = rng.standard_normal((rows, cols)).astype(np.float32)
    crs = rng.uniform(0.8, 1.2, (rows, cols // block)).astype(np.float32)
    dgs = rng.uniform(0.8, 1.2, (rows, cols // sub)).astype(np.float32)
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    ours = O.bwd(x, g, fmt, crs=crs, dgs=dgs, alpha=a)
    fw = O.fwd(x, fmt, crs=crs, dgs=dgs, alpha=a)
    # S^dq from the scale bytes, as the deployed model rebuilds it
    sb = fw["scales"].astype(np.int64)
    if fmt == O.MXFP4:
        sdq = np.exp2(sb - 127).astype(np.float32)
    else:
        dl = torch.from_numpy(fw["scales"]).view(torch.float8_e4m3fn).float().numpy()
        sdq = (dl * np.float32(a)).astype(np.float32)
    # float32 autograd: forward values and input gradient bit-identical
    xt = torch.from_numpy(x).requires_grad_(True)
    ct = torch.from_numpy(crs).requires_grad_(True)
    dt = torch.from_numpy(dgs).requires_grad_(True)
    y = torch_fake_quant(xt, ct, dt, torch.from_numpy(sdq), block, sub)
    assert np.array_equal(y.detach().numpy(), fw["y"])
    x2 = torch.from_numpy(x).requires_grad_(True)
    y2 = torch_ste_ratio(x2, ct, dt, torch.from_numpy(sdq), block, sub)
    y2.backward(torch.from_numpy(g))
    assert np.array_equal(y2.detach().numpy(), fw["y"])
    assert np.array_equal(x2.grad.numpy(), ours["gx"])
    # float64 autograd for the coefficient gradients
    x6 = torch.from_numpy(x.astype(np.float64))
    c6 = torch.from_numpy(crs.astype(np.float64)).requires_grad_(True)
    d6 = torch.from_numpy(dgs.astype(np.float64)).requires_grad_(True)
    y6 = torch_fake_quant(x6, c6, d6, torch.from_numpy(sdq.astype(np.float64)), block, sub)
    y6.backward(torch.from_numpy(g.astype(np.float64)))
    np.testing.assert_allclose(ours["gcrs"], c6.grad.numpy(), rtol=1e-5, atol=1e-12)
    np.testing.assert_allclose(ours["gdgs"], d6.grad.numpy(), rtol=1e-5, atol=1e-12)


def test_clipped_ste_masks_saturated():
    """Clipped STE: no gradient where |x / S^q| > 6 (only possible for c < 1
    under the ceiling rule)."""
    x = np.zeros((1, 32), np.float32)
    x[0, :3] = [1.5, 1.45, 0.1]          # S^dq = 0.25
    crs = np.array([[0.9]], np.float32)   # S^q = 0.225: 1.5/0.225 = 6.67, 1.45/.225 = 6.44
    g = np.ones_like(x)
    b = O.bwd(x, g, O.MXFP4, crs=crs, ste=O.STE_CLIPPED)
    assert b["gx"][0, 0] == 0 and b["gx"][0, 1] == 0 and b["gx"][0, 2] != 0
    bi = O.bwd(x, g, O.MXFP4, crs=crs, ste=O.STE_IDENTITY)
    assert bi["gx"][0, 0] != 0
    # only element 2 (x = 0.1) plus the zeros contribute: T = 0.1
    assert b["gcrs"][0, 0] == pytest.approx(-float(np.float32(0.1)) / 0.81, rel=1e-6)


def test_clipped_ste_keeps_the_saturation_boundary():
    """Clipped STE mask [|u| <= 6] (Sec. 3.2 with the clamp convention): an
    element exactly at |u| = 6 keeps its gradient.  MXFP4 block max 1.5 ->
    S^dq = 0.25 (ceiling rule), c = 1: x = 1.5 and -1.5 give u = +-6, x = 0.75
    gives u = 3; at c = 1 the ratio is 1, so gx = g on all three, and the CRS
    gradient is -(sum g x) / c^2 = -(1.5 * 1 + (-1.5) * 2 + 0.75 * 4)."""
    x = np.zeros((1, 32), np.float32)
    x[0, :3] = [1.5, -1.5, 0.75]
    g = np.zeros_like(x)
    g[0, :3] = [1.0, 2.0, 4.0]
    crs = np.ones((1, 1), np.float32)
    b = O.bwd(x, g, O.MXFP4, crs=crs, ste=O.STE_CLIPPED)
    assert list(b["gx"][0, :3]) == [1.0, 2.0, 4.0]
    assert b["gcrs"][0, 0] == pytest.approx(-1.5, rel=1e-12)


def test_nvfp4_all_zero_tensor_is_dead():
    x = np.zeros((4, 32), np.float32)
    g = np.ones_like(x)
    a = O.alpha(x)
    assert a == 0.0
    out = O.fwd(x, O.NVFP4, alpha=a, want_codes=True)
    assert np.all(out["scales"] == 0) and np.all(out["codes"] == 0)
    assert np.all(out["y"].view(np.uint32) == 0)
    b = O.bwd(x, g, O.NVFP4, crs=np.ones((4, 2), np.float32), alpha=a)
    assert np.all(b["gx"].view(np.uint32) == 0) and np.all(b["gcrs"] == 0)


def test_oracle_rejects_bad_inputs():
    x = np.ones((2, 32), np.float32)
    with pytest.raises(O.OracleError):
        O.fwd(x, O.MXFP4, crs=np.zeros((2, 1), np.float32))     # c must be > 0
    x[0, 0] = np.nan
    with pytest.raises(O.OracleError):
        O.fwd(x, O.MXFP4)
    with pytest.raises(O.OracleError):
        O.fwd(np.ones((2, 30), np.float32), O.MXFP4)            # cols % block


# ---------------------------------------------------------------------------
# learnable full-precision scale S^fp (Eq. 4): S^dq = Q_fmt(S^fp)
# ---------------------------------------------------------------------------
def absmax_sfp(x, fmt, alpha=0.0):
    """The paper's initialisation of S^fp "via absmax": fl(m / 6) for MXFP4,
    fl(m / fl(alpha * 6)) (the unrounded Delta) for NVFP4, in float32."""
    block = 32 if fmt == O.MXFP4 else 16
    xf = W.bf16_bits_to_f32(x) if x.dtype == np.uint16 else x
    rows, cols = xf.shape
    m = np.abs(xf.reshape(rows, cols // block, block)).max(axis=2).astype(np.float32)
    if fmt == O.MXFP4:
        return (m / np.float32(6)).astype(np.float32)
    den = np.float32(alpha) * np.float32(6)
    return (m / den).astype(np.float32)


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_absmax_initialised_sfp_is_the_absmax_scale(fmt):
    """S^fp initialised via absmax (Sec. 3.2) gives S^dq = Q_fmt(S^fp) equal
    to the absmax scale of Eq. 2-3: every output is identical."""
    w = W.WORKLOADS["llama3_8b_block"]
    x = W.to_bf16_bits(W.draw_values(w, 24, 256, 61))
    x[0, :32] = 0
    g = W.to_bf16_bits(W.draw_grad(24, 256, 62))
    block = 32 if fmt == O.MXFP4 else 16
    crs = W.draw_coefs(w, 24 * 256 // block, 63).reshape(24, -1)
    dgs = W.draw_coefs(w, 24 * 256 // 8, 64).reshape(24, -1)
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    sfp = absmax_sfp(x, fmt, a)
    f0 = O.fwd(x, fmt, crs=crs, dgs=dgs, alpha=a, want_codes=True)
    f1 = O.fwd(x, fmt, crs=crs, dgs=dgs, alpha=a, want_codes=True, sfp=sfp)
    for k in ("y", "codes", "scales"):
        assert np.array_equal(f0[k], f1[k]), k
    b0 = O.bwd(x, g, fmt, crs=crs, dgs=dgs, alpha=a)
    b1 = O.bwd(x, g, fmt, crs=crs, dgs=dgs, alpha=a, sfp=sfp, want_gsfp=True)
    for k in ("gx", "gcrs", "gdgs"):
        assert np.array_equal(b0[k], b1[k]), k


def test_hand_mxfp4_sfp_gradient():
    """dL/dS^dq = sum g (q - x / S^q): block [0.7, -0.26, 0.13, 1.5, 0...],
    S^dq = 0.25, c = 1.25 (S^q = 0.3125), g = 1 on the first four:
    (2 - 2.24) + (-1 + 0.832) + (0.5 - 0.416) + (4 - 4.8) = -1.124."""
    x = np.zeros((1, 32), np.float32)
    x[0, :4] = [0.7, -0.26, 0.13, 1.5]
    g = np.zeros_like(x)
    g[0, :4] = 1
    b = O.bwd(x, g, O.MXFP4, crs=np.array([[1.25]], np.float32), sfp=np.array([[0.25]], np.float32),
              want_gsfp=True)
    u = x[0, :4].astype(np.float64) / 0.3125
    expect = float(np.sum(np.array([2.0, -1.0, 0.5, 4.0]) - u))
    assert b["gsfp"][0, 0] == pytest.approx(expect, rel=1e-7)
    assert expect == pytest.approx(-1.124, abs=1e-6)


def test_hand_mxfp4_sfp_gradient_clipped_ste():
    """dL/dS^dq = sum g (q - mask x / S^q) with the clipped mask [|u| <= 6]
    applied to the STE term only (q is the forward's value): block
    [1.5, 1.45, 0.1, 0...], S^fp = 0.25 -> S^dq = 0.25, c = 0.9 (S^q = 0.225),
    u = [6.67, 6.44, 0.44] -> q = [6, 6, 0.5], g = 1 on the three:
    clipped (6 - 0) + (6 - 0) + (0.5 - 0.1 / 0.225) = 12.0556;
    identity (6 - 6.667) + (6 - 6.444) + (0.5 - 0.444) = -1.0556."""
    x = np.zeros((1, 32), np.float32)
    x[0, :3] = [1.5, 1.45, 0.1]
    g = np.zeros_like(x)
    g[0, :3] = 1
    crs = np.array([[0.9]], np.float32)
    sfp = np.array([[0.25]], np.float32)
    sq = 0.25 * float(np.float32(0.9))
    xs = x[0, :3].astype(np.float64)
    q = np.array([6.0, 6.0, 0.5])
    expect = {O.STE_CLIPPED: float(np.sum(q - np.array([0.0, 0.0, 1.0]) * xs / sq)),
              O.STE_IDENTITY: float(np.sum(q - xs / sq))}
    assert expect[O.STE_CLIPPED] == pytest.approx(12.0556, abs=1e-4)
    assert expect[O.STE_IDENTITY] == pytest.approx(-1.0556, abs=1e-4)
    for ste, e in expect.items():
        b = O.bwd(x, g, O.MXFP4, crs=crs, sfp=sfp, ste=ste, want_gsfp=True)
        assert b["gsfp"][0, 0] == pytest.approx(e, rel=1e-7)


def test_sfp_rounding_rules():
    """Q_E8M0 rounds S^fp up to a power of two; Q_E4M3 is round-to-nearest-even
    (checked against torch's float8_e4m3fn)."""
    x = np.full((4, 32), 0.01, np.float32)
    sfp = np.array([[2.0 ** -5], [2.0 ** -5 * 1.0000001], [2.0 ** -5 * 1.9], [3e-3]], np.float32)
    sc = O.fwd(x, O.MXFP4, sfp=sfp)["scales"][:, 0].astype(int) - 127
    assert list(sc) == [-5, -4, -4, int(np.ceil(np.log2(np.float64(np.float32(3e-3)))))]
    rng = np.random.default_rng(71)
    d = rng.uniform(0, 460, 512).astype(np.float32)
    xn = np.full((512, 16), 0.01, np.float32)
    out = O.fwd(xn, O.NVFP4, alpha=1.0 / 2688, sfp=d.reshape(-1, 1))
    assert np.array_equal(out["scales"][:, 0], torch_e4m3(d))


def torch_fake_quant_sfp(x, sfp, crs, dgs, fmt, alpha, block, sub):
    """Autograd restatement with the scale learned through Q_fmt by STE:
    S^dq = S^fp + (Q_fmt(S^fp) - S^fp).detach() (times alpha for NVFP4)."""
    c = crs.repeat_interleave(block, dim=1)
    d = dgs.repeat_interleave(sub, dim=1)
    sf = sfp.detach().numpy().astype(np.float32)
    if fmt == O.MXFP4:
        q = np.exp2(np.ceil(np.log2(sf.astype(np.float64))))
        s = sfp + (torch.from_numpy(q) - sfp).detach()
    else:
        # the forward's scale is fl(alpha * Delta) in binary32; the STE carries
        # d S^dq / d Delta^fp = alpha; Q_E4M3 saturates at 448 (torch's cast
        # gives NaN above it)
        dq = torch.from_numpy(torch_e4m3(np.minimum(sf, np.float32(448)))).view(
            torch.float8_e4m3fn).float()
        sdq = (dq * torch.tensor(alpha, dtype=torch.float32)).double()
        s = sdq + alpha * (sfp - sfp.detach())
    s = s.repeat_interleave(block, dim=1)
    u = x / (s * (c * d))
    qv = torch.from_numpy(e2m1_ref(u.detach().numpy()))
    return (u + (qv - u).detach()) * s


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_sfp_gradient_autograd(fmt):
    rng = np.random.default_rng(81)
    block = 32 if fmt == O.MXFP4 else 16
    rows, cols = 5, 4 * block
    x = (rng.standard_normal((rows, cols)) * 0.02).astype(np.float32)
    g = rng.standard_normal((rows, cols)).astype(np.float32)
    crs = rng.uniform(0.8, 1.2, (rows, cols // block)).astype(np.float32)
    dgs = rng.uniform(0.8, 1.2, (rows, cols // 8)).astype(np.float32)
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    sfp = (absmax_sfp(x, fmt, a) * rng.uniform(0.7, 1.3, (rows, cols // block))).astype(np.float32)
    ours = O.bwd(x, g, fmt, crs=crs, dgs=dgs, alpha=a, sfp=sfp, want_gsfp=True)
    s6 = torch.from_numpy(sfp.astype(np.float64)).requires_grad_(True)
    y = torch_fake_quant_sfp(torch.from_numpy(x.astype(np.float64)), s6,
                             torch.from_numpy(crs.astype(np.float64)),
                             torch.from_numpy(dgs.astype(np.float64)), fmt, float(a), block, 8)
    y.backward(torch.from_numpy(g.astype(np.float64)))
    np.testing.assert_allclose(ours["gsfp"], s6.grad.numpy(), rtol=1e-5, atol=1e-12)
    # the forward of the restatement is the oracle's (values, through fp64)
    fw = O.fwd(x, fmt, crs=crs, dgs=dgs, alpha=a, sfp=sfp)
    np.testing.assert_allclose(y.detach().numpy(), fw["y"].astype(np.float64), rtol=1e-6, atol=0)


# ---------------------------------------------------------------------------
# AdamW on the learnable arrays (Sec. 4.1: AdamW, constant learning rate)
# ---------------------------------------------------------------------------
HP = dict(lr_coef=5e-2, lr_scale=2e-2, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)


def fp32(v):
    return float(np.float32(v))


def test_adamw_matches_torch():
    """Five AdamW steps of the oracle equal torch.optim.AdamW in float64 (the
    library routine the paper's PyTorch setup calls)."""
    rng = np.random.default_rng(91)
    p0 = rng.uniform(0.5, 1.5, 64)
    m = np.zeros(64)
    v = np.zeros(64)
    lr, b1, b2, eps, wd = fp32(3e-2), fp32(0.9), fp32(0.999), fp32(1e-8), fp32(0.01)
    pt = torch.tensor(p0, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([pt], lr=lr, betas=(b1, b2), eps=eps, weight_decay=wd)
    p = p0.copy()
    for t in range(1, 6):
        g = rng.standard_normal(64) * 10.0 ** rng.uniform(-6, 1, 64)
        pt.grad = torch.tensor(g)
        opt.step()
        p, m, v = O.adamw(p, g, m, v, lr, b1, b2, eps, wd, t)
        np.testing.assert_allclose(p, pt.detach().numpy(), rtol=1e-14, atol=0)
        np.testing.assert_allclose(m, opt.state[pt]["exp_avg"].numpy(), rtol=1e-14, atol=0)
        np.testing.assert_allclose(v, opt.state[pt]["exp_avg_sq"].numpy(), rtol=1e-14, atol=0)


def test_adamw_first_step_closed_form():
    """From zero moments the first step is p (1 - lr wd) - lr g / (|g| + eps)."""
    g = np.array([3.0, -2e-3, 0.0, 1e-9, -7.5])
    p = np.array([1.0, 0.9, 1.1, 2.0, 0.5])
    lr, wd, eps = fp32(5e-3), fp32(0.01), fp32(1e-8)
    pn, mn, vn = O.adamw(p, g, np.zeros(5), np.zeros(5), lr, 0.9, 0.999, eps, wd, 1)
    np.testing.assert_allclose(pn, p * (1 - lr * wd) - lr * g / (np.abs(g) + eps), rtol=1e-13, atol=0)
    np.testing.assert_allclose(mn, (1 - fp32(0.9)) * g, rtol=1e-15, atol=0)
    np.testing.assert_allclose(vn, (1 - fp32(0.999)) * g * g, rtol=1e-15, atol=0)
    with pytest.raises(O.OracleError):
        O.adamw(p, g, mn, vn, lr, 0.9, 0.999, eps, wd, 0)


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_bwd_adamw_equals_autograd_and_torch_adamw(fmt):
    """The fused backward + AdamW of the oracle equals autograd of the STE
    restatement followed by torch.optim.AdamW on S^fp (lr_scale) and c_i,
    c_i^k (lr_coef), from moments of an earlier step."""
    rng = np.random.default_rng(93)
    block = 32 if fmt == O.MXFP4 else 16
    rows, cols = 4, 4 * block
    x = (rng.standard_normal((rows, cols)) * 0.02).astype(np.float32)
    g = rng.standard_normal((rows, cols)).astype(np.float32)
    crs = rng.uniform(0.8, 1.2, (rows, cols // block)).astype(np.float32)
    dgs = rng.uniform(0.8, 1.2, (rows, cols // 8)).astype(np.float32)
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    sfp = (absmax_sfp(x, fmt, a) * rng.uniform(0.7, 1.3, (rows, cols // block))).astype(np.float32)
    params = {"crs": crs, "dgs": dgs, "sfp": sfp}
    moments = {k: (rng.standard_normal(v.shape).astype(np.float32) * np.float32(0.1),
                   rng.uniform(0.01, 1.0, v.shape).astype(np.float32)) for k, v in params.items()}
    step = 7
    ours = O.bwd_adamw(x, g, fmt, params, moments, HP, step, alpha=a)
    t = {k: torch.from_numpy(v.astype(np.float64)).requires_grad_(True) for k, v in params.items()}
    y = torch_fake_quant_sfp(torch.from_numpy(x.astype(np.float64)), t["sfp"], t["crs"], t["dgs"],
                             fmt, float(a), block, 8)
    y.backward(torch.from_numpy(g.astype(np.float64)))
    opt = torch.optim.AdamW(
        [{"params": [t["sfp"]], "lr": fp32(HP["lr_scale"])},
         {"params": [t["crs"], t["dgs"]], "lr": fp32(HP["lr_coef"])}],
        betas=(fp32(HP["beta1"]), fp32(HP["beta2"])), eps=fp32(HP["eps"]),
        weight_decay=fp32(HP["weight_decay"]))
    for k, (m, v) in moments.items():
        opt.state[t[k]] = {"step": torch.tensor(float(step - 1)),
                           "exp_avg": torch.from_numpy(m.astype(np.float64)),
                           "exp_avg_sq": torch.from_numpy(v.astype(np.float64))}
    grads = {k: t[k].grad.numpy().copy() for k in t}
    opt.step()
    for k in params:
        np.testing.assert_allclose(ours[k]["grad"], grads[k], rtol=1e-5, atol=1e-12)
        lr = fp32(HP["lr_scale"] if k == "sfp" else HP["lr_coef"])
        # gradients agree to ~1e-7 relative; the step moves by about lr
        np.testing.assert_allclose(ours[k]["p"], t[k].detach().numpy(), rtol=0, atol=1e-5 * lr)
        np.testing.assert_allclose(ours[k]["m"], opt.state[t[k]]["exp_avg"].numpy(), rtol=1e-5,
                                   atol=1e-12)
        np.testing.assert_allclose(ours[k]["v"], opt.state[t[k]]["exp_avg_sq"].numpy(), rtol=1e-5,
                                   atol=0)
    # arrays that are not learned are not in the result
    part = O.bwd_adamw(x, g, fmt, {"dgs": dgs}, {"dgs": moments["dgs"]}, HP, step, alpha=a)
    assert set(part) == {"gx", "dgs"}


# ---------------------------------------------------------------------------
# deployment view: MMA scale-factor tiles and the FP4 GEMM on the export
# ---------------------------------------------------------------------------
def test_mma_scale_tiles_hand_offsets():
    R, C = 130, 5
    s = np.zeros((R, C), np.uint8)
    marks = {(0, 0): 1, (1, 0): 2, (31, 0): 3, (32, 0): 4, (64, 1): 5, (96, 3): 6, (0, 4): 7,
             (128, 0): 8, (129, 4): 9, (127, 3): 10}
    for (r, c), v in marks.items():
        s[r, c] = v
    t = O.mma_scale_tiles(s)
    assert t.size == 2 * 2 * 512                       # 2 x 2 tiles (rows and columns padded)
    where = {0: 1, 16: 2, 496: 3, 4: 4, 9: 5, 15: 6, 512: 7, 1024: 8, 1552: 9,
             31 * 16 + 3 * 4 + 3: 10}
    for off, v in where.items():
        assert t[off] == v, (off, t[off], v)
    assert np.count_nonzero(t) == len(marks)


def test_mma_scale_tiles_is_a_permutation():
    rng = np.random.default_rng(101)
    R, C = 256, 8
    s = rng.integers(1, 256, (R, C), dtype=np.uint8)
    t = O.mma_scale_tiles(s)
    assert t.size == R * C
    assert np.array_equal(np.sort(t), np.sort(s.reshape(-1)))
    # each 16-byte line of a tile holds rows r, r+32, r+64, r+96 (4 columns each)
    line = t[:16].reshape(4, 4)
    assert np.array_equal(line, s[[0, 32, 64, 96], :4])


def _dequant_independent(codes, scales, fmt):
    """Dense values of an export through torch's float8 decoders and the
    pins' own E2M1 grid (nothing of the oracle)."""
    k = codes.shape[1] * 2
    nib = np.empty((codes.shape[0], k), np.int64)
    nib[:, 0::2] = codes & 15
    nib[:, 1::2] = codes >> 4
    val = np.array([code_to_value(c) for c in range(16)])[nib]
    block = 32 if fmt == O.MXFP4 else 16
    if fmt == O.MXFP4:
        s = torch.from_numpy(scales.copy()).view(torch.float8_e8m0fnu).double().numpy()
    else:
        s = torch.from_numpy(scales.copy()).view(torch.float8_e4m3fn).double().numpy()
    return val * np.repeat(s, block, axis=1)


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_fp4_gemm_matches_independent_dequant(fmt):
    rng = np.random.default_rng(103)
    M, N, K = 40, 24, 256
    xa = (rng.standard_normal((M, K)) * 0.5).astype(np.float32)
    xb = (rng.standard_t(4, (N, K)) * 0.02).astype(np.float32)
    aa = O.alpha(xa) if fmt == O.NVFP4 else 0.0
    ab = O.alpha(xb) if fmt == O.NVFP4 else 0.0
    ea = O.fwd(xa, fmt, alpha=aa, want_y=False, want_codes=True)
    eb = O.fwd(xb, fmt, alpha=ab, want_y=False, want_codes=True)
    d = O.fp4_gemm(ea["codes"], ea["scales"], eb["codes"], eb["scales"], fmt, aa, ab)
    ref = _dequant_independent(ea["codes"], ea["scales"], fmt) @ \
        _dequant_independent(eb["codes"], eb["scales"], fmt).T
    if fmt == O.NVFP4:
        ref = ref * (float(np.float32(aa)) * float(np.float32(ab)))
    np.testing.assert_allclose(d, ref, rtol=1e-14, atol=0)


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_fp4_gemm_is_the_product_of_fake_quantized_operands(fmt):
    """W4A4 on the export equals the product of the fake-quantized tensors:
    exactly for MXFP4 (y = q 2^e has no rounding); for NVFP4 up to the
    rounding of fl(alpha * Delta) in y (2^-23 relative per product)."""
    rng = np.random.default_rng(107)
    M, N, K = 32, 48, 512
    xa = (rng.standard_normal((M, K))).astype(np.float32)
    xb = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    ca = rng.uniform(0.9, 1.1, (M, K // O.default_block(fmt))).astype(np.float32)
    aa = O.alpha(xa) if fmt == O.NVFP4 else 0.0
    ab = O.alpha(xb) if fmt == O.NVFP4 else 0.0
    fa = O.fwd(xa, fmt, crs=ca, alpha=aa, want_codes=True)
    fb = O.fwd(xb, fmt, alpha=ab, want_codes=True)
    d = O.fp4_gemm(fa["codes"], fa["scales"], fb["codes"], fb["scales"], fmt, aa, ab)
    ya, yb = fa["y"].astype(np.float64), fb["y"].astype(np.float64)
    if fmt == O.MXFP4:
        np.testing.assert_allclose(d, ya @ yb.T, rtol=1e-13, atol=0)
    else:
        bound = 2.0 ** -22 * (np.abs(ya) @ np.abs(yb).T)
        assert np.all(np.abs(d - ya @ yb.T) <= bound)


# ---------------------------------------------------------------------------
# binary16 I/O
# ---------------------------------------------------------------------------
def test_f16_decode_all_patterns_matches_numpy():
    h = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    ours = O.f16_decode(h)
    ref = h.view(np.float16).astype(np.float32)
    fin = np.isfinite(ref)
    assert np.array_equal(ours[fin].view(np.uint32), ref[fin].view(np.uint32))
    assert np.all(np.isnan(ours[np.isnan(ref)])) and np.array_equal(ours[np.isinf(ref)], ref[np.isinf(ref)])


def test_f16_rne_matches_numpy():
    """Every binary16 value, the midpoints between neighbours and one binary32
    ulp either side of each (ties to even, subnormals, the overflow
    threshold 65520), plus random patterns."""
    h = np.arange(0, 0x7C00, dtype=np.uint32).astype(np.uint16)
    v = h.view(np.float16).astype(np.float64)
    mids = ((v[:-1] + v[1:]) / 2).astype(np.float32)
    ulp = lambda a, d: np.nextafter(a, np.float32(d * np.inf)).astype(np.float32)
    cand = np.concatenate([v.astype(np.float32), mids, ulp(mids, 1), ulp(mids, -1),
                           np.array([65504, 65519.996, 65520, 65536, 1e9, 2 ** -25, 2 ** -24,
                                     3 * 2 ** -26, 2 ** -26], np.float32)])
    rng = np.random.default_rng(111)
    cand = np.concatenate([cand, rng.integers(0, 1 << 32, 2_000_000, dtype=np.uint64)
                           .astype(np.uint32).view(np.float32)])
    cand = cand[np.isfinite(cand)]
    cand = np.concatenate([cand, -cand])
    with np.errstate(over="ignore"):
        ref = cand.astype(np.float16).view(np.uint16)
    assert np.array_equal(O.f16_rne(cand), ref)


@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_f16_io_is_the_f32_path_rounded(fmt):
    """binary16 I/O: x widened exactly, every quantity computed as for
    binary32 inputs, y and gx rounded to binary16 at the end."""
    rng = np.random.default_rng(113)
    block = 32 if fmt == O.MXFP4 else 16
    x16 = (rng.standard_normal((12, 4 * block)) * 0.3).astype(np.float16)
    g16 = rng.standard_normal((12, 4 * block)).astype(np.float16)
    crs = rng.uniform(0.8, 1.2, (12, 4)).astype(np.float32)
    x32, g32 = x16.astype(np.float32), g16.astype(np.float32)
    a = O.alpha(x16) if fmt == O.NVFP4 else 0.0
    assert a == (O.alpha(x32) if fmt == O.NVFP4 else 0.0)
    f16 = O.fwd(x16, fmt, crs=crs, alpha=a, want_codes=True)
    f32 = O.fwd(x32, fmt, crs=crs, alpha=a, want_codes=True)
    assert np.array_equal(f16["codes"], f32["codes"]) and np.array_equal(f16["scales"], f32["scales"])
    assert np.array_equal(f16["y"].view(np.uint16), O.f16_rne(f32["y"]))
    b16 = O.bwd(x16, g16, fmt, crs=crs, alpha=a)
    b32 = O.bwd(x32, g32, fmt, crs=crs, alpha=a)
    assert np.array_equal(b16["gx"].view(np.uint16), O.f16_rne(b32["gx"]))
    assert np.array_equal(b16["gcrs"], b32["gcrs"])
