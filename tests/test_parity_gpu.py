"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on the
same seeded inputs.  Codes, scale bytes, dequantized values and input
gradients must be bit-exact; coefficient gradients within 1e-5 relative
(with the cancellation floor documented in gpu_helpers)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_01847_gb300 import build as B
from paper_2608_01847_gb300 import focus as F
from paper_2608_01847_gb300 import workloads as W
from gpu_helpers import (FLOOR_ROW, FLOOR_SHARED, assert_bits_equal, assert_grad_close, dev,
                         host)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    F.lib()


FMT = {"mx": O.MXFP4, "nv": O.NVFP4}


def run_case(x, g, fmt, crs=None, dgs=None, sub=8, shared=False, ste=O.STE_IDENTITY,
             rule=O.MX_CEIL, alpha=None, pad=0, check_alpha=True, offset=0):
    """Run alpha (NVFP4), fwd, pack and bwd on GPU and oracle; compare all.
    pad / offset: the device inputs are columns [offset, offset + cols) of
    a buffer [rows, offset + cols + pad] (ld > cols, rows off 32-byte
    boundaries when offset or the pitch is not a multiple of 32 bytes)."""
    rows, cols = x.shape
    block = 32 if fmt == O.MXFP4 else 16
    xd, gd = dev(x), dev(g)
    if pad or offset:
        xb = torch.zeros((rows, offset + cols + pad), dtype=xd.dtype, device="cuda")
        gb = torch.zeros_like(xb)
        xb[:, offset:offset + cols] = xd
        gb[:, offset:offset + cols] = gd
        xd, gd = xb[:, offset:offset + cols], gb[:, offset:offset + cols]
    cd = dev(crs) if crs is not None else None
    dd = dev(dgs) if dgs is not None else None
    a_dev = None
    a = 0.0
    if fmt == O.NVFP4:
        if alpha is None:
            a_dev = F.focus_nvfp4_alpha(xd)
            a = O.alpha(x)
            if check_alpha:
                assert_bits_equal(host(a_dev), np.array([a], np.float32), "alpha")
        else:
            a = float(np.float32(alpha))
            a_dev = torch.tensor([a], dtype=torch.float32, device="cuda")
    kw = dict(sub_block=sub, shared=shared, mx_rule=rule)
    y, sb = F.focus_fq_fwd(xd, fmt, cd, dd, a_dev, want_scales=True, **kw)
    codes, sb2 = F.focus_pack(xd, fmt, cd, dd, a_dev, **kw)
    gx, gc, gdg = F.focus_fq_bwd(xd, gd, fmt, cd, dd, a_dev, ste=ste, want_gcrs=True,
                                 want_gdgs=True, **kw)
    torch.cuda.synchronize()
    ref = O.fwd(x, fmt, crs=crs, dgs=dgs, alpha=a, sub=sub, shared=shared, mx_rule=rule,
                want_codes=True)
    rb = O.bwd(x, g, fmt, crs=crs, dgs=dgs, alpha=a, sub=sub, shared=shared, ste=ste,
               mx_rule=rule, want_abs=True)
    assert_bits_equal(host(y), ref["y"], "y")
    assert_bits_equal(host(sb), ref["scales"], "scale bytes (fwd)")
    assert_bits_equal(host(sb2), ref["scales"], "scale bytes (pack)")
    assert_bits_equal(host(codes), ref["codes"], "codes")
    assert_bits_equal(host(gx), rb["gx"], "gx")
    floor = FLOOR_SHARED if shared else FLOOR_ROW
    assert_grad_close(host(gc), rb["gcrs"], rb["gcrs_abs"], floor, "dL/dc")
    assert_grad_close(host(gdg), rb["gdgs"], rb["gdgs_abs"], floor, "dL/dc^k")
    return dict(y=y, codes=codes, gx=gx, gcrs=gc, gdgs=gdg)


def seeded(rows, cols, dtype="bf16", seed=0, scale=0.02, nu=5.0, coef=(0.8, 1.2)):
    w = W.Workload("t", (W.TensorSpec("t", rows, cols),), dtype, ("mxfp4",), "weight", nu, scale,
                   "entries", 0.01, 20.0, coef, seed)
    x, g = W.host_tensor(w, 0)
    return w, x, g


# ---------------------------------------------------------------------------
# 256x512 fp32 weight, MXFP4, CRS / DGS / both (the small config)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("mode", ["crs", "dgs", "both", "none"])
def test_w256x512_f32_mxfp4(mode):
    w = W.WORKLOADS["w256x512_f32"]
    x, g = W.host_tensor(w, 0)
    crs, dgs = W.host_coefs(w, 0, 32, 8)
    run_case(x, g, O.MXFP4, crs if mode in ("crs", "both") else None,
             dgs if mode in ("dgs", "both") else None)


# ---------------------------------------------------------------------------
# several tiles + ragged tails, strided rows, both dtypes and formats
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("dtype", ["bf16", "f32", "f16"])
@pytest.mark.parametrize("rows,cols,pad", [(37, 352, 0), (5, 4096, 0), (129, 96, 32), (1, 32, 0),
                                           (3000, 160, 0), (17, 1216, 16)])
def test_shapes(fmt, dtype, rows, cols, pad):
    w, x, g = seeded(rows, cols, dtype, seed=rows * 7 + cols)
    block = 32 if fmt == "mx" else 16
    crs = W.draw_coefs(w, rows * cols // block, 5).reshape(rows, -1)
    dgs = W.draw_coefs(w, rows * cols // 8, 6).reshape(rows, -1)
    run_case(x, g, FMT[fmt], crs, dgs, pad=pad)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("dtype", ["bf16", "f16", "f32"])
@pytest.mark.parametrize("pad,offset", [(8, 0), (0, 8), (8, 8), (24, 0)])
def test_rows_on_16_byte_boundaries(fmt, dtype, pad, offset):
    """Rows that start on 16-byte but not 32-byte boundaries (row pitch
    cols + 8 sixteen-bit elements, or a view starting 8 elements into a
    wider buffer; for fp32, 4-element steps): the kernels take two 128-bit
    accesses per 32-byte piece, results bit for bit the oracle's, with
    every phase (and the shared-row backward) on several tiles and a ragged
    tail."""
    w, x, g = seeded(300, 672, dtype, seed=41 + pad + offset)
    if dtype == "f32":
        pad, offset = pad // 2, offset // 2
    esz = 4 if dtype == "f32" else 2
    assert ((672 + pad + offset) * esz) % 32 == 16 or (offset * esz) % 32 == 16
    block = 32 if fmt == "mx" else 16
    crs = W.draw_coefs(w, 300 * 672 // block, 5).reshape(300, -1)
    dgs = W.draw_coefs(w, 300 * 672 // 8, 6).reshape(300, -1)
    run_case(x, g, FMT[fmt], crs, dgs, pad=pad, offset=offset)
    run_case(x, g, FMT[fmt], crs[:1], dgs[:1], shared=True, pad=pad, offset=offset)


@pytest.mark.parametrize("fmt,sub", [("mx", 2), ("mx", 4), ("mx", 8), ("mx", 16), ("mx", 32),
                                     ("nv", 2), ("nv", 4), ("nv", 8), ("nv", 16)])
@pytest.mark.parametrize("dtype", ["bf16", "f32", "f16"])
def test_sub_block_sizes(fmt, sub, dtype):
    rows, cols = 77, 640
    w, x, g = seeded(rows, cols, dtype, seed=sub)
    block = 32 if fmt == "mx" else 16
    crs = W.draw_coefs(w, rows * cols // block, 8).reshape(rows, -1)
    dgs = W.draw_coefs(w, rows * cols // sub, 9).reshape(rows, -1)
    run_case(x, g, FMT[fmt], crs, dgs, sub=sub)
    run_case(x, g, FMT[fmt], None, dgs, sub=sub)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("dtype", ["bf16", "f32", "f16"])
def test_clipped_ste_and_floor_rule(fmt, dtype):
    rows, cols = 64, 512
    w, x, g = seeded(rows, cols, dtype, seed=3, coef=(0.6, 1.0))   # c < 1: saturation happens
    block = 32 if fmt == "mx" else 16
    crs = W.draw_coefs(w, rows * cols // block, 10).reshape(rows, -1)
    dgs = W.draw_coefs(w, rows * cols // 8, 11).reshape(rows, -1)
    run_case(x, g, FMT[fmt], crs, dgs, ste=O.STE_CLIPPED)
    if fmt == "mx":
        run_case(x, g, FMT[fmt], crs, dgs, rule=O.MX_FLOOR)
        run_case(x, g, FMT[fmt], crs, dgs, rule=O.MX_FLOOR, ste=O.STE_CLIPPED)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("dtype", ["bf16", "f32", "f16"])
@pytest.mark.parametrize("rows,cols", [(300, 256), (1030, 96), (3, 4096)])
def test_shared_row_coefficients(fmt, dtype, rows, cols):
    w, x, g = seeded(rows, cols, dtype, seed=rows, scale=1.0, nu=None, coef=(0.9, 1.1))
    block = 32 if fmt == "mx" else 16
    crs = W.draw_coefs(w, cols // block, 12).reshape(1, -1)
    dgs = W.draw_coefs(w, cols // 8, 13).reshape(1, -1)
    run_case(x, g, FMT[fmt], crs, dgs, shared=True)
    run_case(x, g, FMT[fmt], crs, None, shared=True)


def test_nvfp4_frozen_alpha_saturates():
    """A frozen alpha smaller than the tensor's own (weights, Sec. 3.2) drives
    block ratios past 448: the E4M3 scale saturates."""
    w, x, g = seeded(64, 256, "bf16", seed=21)
    a = O.alpha(x) * 0.25
    run_case(x, g, O.NVFP4, alpha=a)


# ---------------------------------------------------------------------------
# crafted inputs: every rounding boundary of E2M1, E4M3 and E8M0
# ---------------------------------------------------------------------------
def test_e2m1_boundaries_through_api():
    """Blocks whose max is exactly 6 have S^dq = 1 (ceiling rule), so u = x:
    push dense sweeps and every E2M1 midpoint +-1 ulp through the kernels."""
    mids = np.array([0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0], np.float32)
    vals = [mids, np.nextafter(mids, np.float32(0)), np.nextafter(mids, np.float32(9)),
            np.linspace(0, 6, 20000, dtype=np.float32), np.float32([0.0, 1e-45, 1e-38, 6.0])]
    v = np.concatenate(vals)
    v = np.concatenate([v, -v])
    per = 31
    nblk = (v.size + per - 1) // per
    v = np.concatenate([v, np.zeros(nblk * per - v.size, np.float32)]).reshape(nblk, per)
    x = np.concatenate([np.full((nblk, 1), 6.0, np.float32), v], axis=1)   # blocks of 32
    rows = 64
    x = np.concatenate([x, np.zeros(((-nblk) % rows, 32), np.float32)]).reshape(rows, -1)
    g = np.ones_like(x)
    run_case(x, g, O.MXFP4)


def test_e4m3_boundaries_through_api():
    """alpha = fl(1/6) makes fl(alpha * 6) = 1, so each NVFP4 block's ratio is
    its own max: blocks with every E4M3 midpoint +-1 ulp as their max."""
    a = np.float32(1.0) / np.float32(6.0)
    assert np.float32(a * np.float32(6.0)) == 1.0
    codes = np.arange(0, 0x7F)
    vals = np.array([O.e4m3_decode(int(c)) for c in codes], np.float64)
    mids = ((vals[:-1] + vals[1:]) / 2).astype(np.float32)
    r = np.concatenate([mids, np.nextafter(mids, np.float32(0)), np.nextafter(mids, np.float32(999)),
                        vals.astype(np.float32), np.float32([448.0, 460.0, 470.0, 1e6])])
    r = r[r > 0]
    n = r.size
    x = np.zeros((n, 16), np.float32)
    x[:, 0] = r
    x[:, 1] = -r * np.float32(0.37)
    x[:, 5] = r * np.float32(0.81)
    rows = 16
    x = np.concatenate([x, np.zeros(((-n) % rows, 16), np.float32)]).reshape(rows, -1)
    g = np.ones_like(x)
    run_case(x, g, O.NVFP4, alpha=a)


@pytest.mark.parametrize("rule", [O.MX_CEIL, O.MX_FLOOR])
def test_e8m0_boundaries_through_api(rule):
    es = np.arange(-140, 126)
    base = (np.float32(6.0) * np.exp2(es).astype(np.float32)).astype(np.float32)
    base = base[np.isfinite(base) & (base > 0)]
    m = np.concatenate([base, np.nextafter(base, np.float32(0)), np.nextafter(base, np.float32(np.inf)),
                        np.exp2(es).astype(np.float32)])
    m = m[np.isfinite(m) & (m > 0)]
    n = m.size
    x = np.zeros((n, 32), np.float32)
    x[:, 3] = m
    x[:, 7] = -m * np.float32(0.5)
    x[:, 20] = m * np.float32(0.1)
    rows = 8
    x = np.concatenate([x, np.zeros(((-n) % rows, 32), np.float32)]).reshape(rows, -1)
    g = np.ones_like(x)
    run_case(x, g, O.MXFP4, rule=rule)


def test_degenerate_blocks():
    """All-zero blocks, tiny blocks (subnormal MXFP4 scales 2^-127), huge
    values near FLT_MAX, isolated outliers."""
    rng = np.random.default_rng(1)
    x = rng.standard_normal((48, 256)).astype(np.float32)
    x[0] = 0
    x[1, :32] = 0
    x[2] *= np.float32(1e-39)
    x[3] *= np.float32(1e-44)
    x[4, :32] = np.float32(3.0e38) * np.sign(x[4, :32])
    x[5, 7] = 1e30
    g = rng.standard_normal(x.shape).astype(np.float32)
    crs = rng.uniform(0.9, 1.1, (48, 8)).astype(np.float32)
    run_case(x, g, O.MXFP4, crs=crs)
    run_case(W.to_bf16_bits(x), W.to_bf16_bits(g), O.MXFP4, crs=crs)
    xn = x.copy()
    xn[4] = 1.0
    run_case(xn, g, O.NVFP4, crs=rng.uniform(0.9, 1.1, (48, 16)).astype(np.float32))


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_gradient_overflow_rule(dtype):
    """Sub-blocks of alternating +a, -a with g = 1 cancel exactly (T = 0).
    The kernels sum even and odd elements in two interleaved binary32 chains:
    at a = 2^125 each chain peaks at 4a = 2^127, nothing overflows, and the
    gradient is exactly 0; at a = 2^126 a chain reaches 2^128 and overflows,
    and the pair turns into NaN -- allowed only because the sum of |terms|
    (2^129) is beyond the binary32 range (the comparison rule of
    assert_grad_close)."""
    x = np.ones((2, 64), np.float32)
    x[0, :32] = np.float32(2.0 ** 125) * np.tile(np.float32([1, -1]), 16)
    x[1, :32] = np.float32(2.0 ** 126) * np.tile(np.float32([1, -1]), 16)
    g = np.ones_like(x)
    if dtype == "bf16":
        x, g = W.to_bf16_bits(x), W.to_bf16_bits(g)
    crs = np.ones((2, 2), np.float32)
    dgs = np.ones((2, 8), np.float32)
    out = run_case(x, g, O.MXFP4, crs=crs, dgs=dgs)
    gc, gd = host(out["gcrs"]), host(out["gdgs"])
    assert gc[0, 0] == 0 and np.all(gd[0, :4] == 0)
    assert np.isnan(gc[1, 0]) and np.all(np.isnan(gd[1, :4]))
    # the second block of each row (ones) is unaffected
    assert np.isfinite(gc[:, 1]).all() and np.isfinite(gd[:, 4:]).all()


def test_nvfp4_all_zero_tensor():
    x = np.zeros((8, 64), np.float32)
    g = np.ones_like(x)
    out = run_case(x, g, O.NVFP4, crs=np.ones((8, 4), np.float32))
    assert not torch.any(out["gx"])


def test_empty_tensors():
    for fmt in (O.MXFP4, O.NVFP4):
        x = torch.zeros((0, 64), dtype=torch.bfloat16, device="cuda")
        a = F.focus_nvfp4_alpha(x)
        torch.cuda.synchronize()
        assert a.item() == 0.0
        y = F.focus_fq_fwd(x, fmt, None, None, a)
        codes, sb = F.focus_pack(x, fmt, None, None, a)
        crs = torch.ones((1, 64 // (32 if fmt == O.MXFP4 else 16)), device="cuda")
        gx, gc, _ = F.focus_fq_bwd(x, x, fmt, crs, None, a, shared=True)
        torch.cuda.synchronize()
        assert y.numel() == 0 and codes.numel() == 0 and torch.all(gc == 0)


def test_deterministic():
    w, x, g = seeded(500, 1024, "bf16", seed=99, scale=1.0, nu=None)
    crs = W.draw_coefs(w, 1024 // 32, 1).reshape(1, -1)
    dgs = W.draw_coefs(w, 1024 // 8, 2).reshape(1, -1)
    xd, gd, cd, dd = dev(x), dev(g), dev(crs), dev(dgs)
    r1 = F.focus_fq_bwd(xd, gd, O.MXFP4, cd, dd, shared=True)
    r2 = F.focus_fq_bwd(xd, gd, O.MXFP4, cd, dd, shared=True)
    torch.cuda.synchronize()
    for a, b in zip(r1, r2):
        assert torch.equal(a.view(torch.int16) if a.dtype == torch.bfloat16 else a.view(torch.int32),
                           b.view(torch.int16) if b.dtype == torch.bfloat16 else b.view(torch.int32))


# ---------------------------------------------------------------------------
# learnable full-precision scale S^fp (Eq. 4)
# ---------------------------------------------------------------------------
def absmax_sfp_host(x, fmt, alpha):
    block = 32 if fmt == O.MXFP4 else 16
    xf = W.bf16_bits_to_f32(x) if x.dtype == np.uint16 else x
    rows, cols = xf.shape
    m = np.abs(xf.reshape(rows, cols // block, block)).max(axis=2).astype(np.float32)
    den = np.float32(6) if fmt == O.MXFP4 else np.float32(alpha) * np.float32(6)
    return (m / den).astype(np.float32)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("dtype", ["bf16", "f32", "f16"])
@pytest.mark.parametrize("sub", [8, 4])
@pytest.mark.parametrize("ste", [O.STE_IDENTITY, O.STE_CLIPPED])
def test_learnable_scale(fmt, dtype, sub, ste):
    rows, cols = 96, 640
    w, x, g = seeded(rows, cols, dtype, seed=7 + sub, coef=(0.8, 1.2))
    f = FMT[fmt]
    block = 32 if f == O.MXFP4 else 16
    crs = W.draw_coefs(w, rows * cols // block, 14).reshape(rows, -1)
    dgs = W.draw_coefs(w, rows * cols // sub, 15).reshape(rows, -1)
    a = O.alpha(x) if f == O.NVFP4 else 0.0
    jitter = W.draw_coefs(w, rows * cols // block, 16).reshape(rows, -1)
    sfp = (absmax_sfp_host(x, f, a) * jitter).astype(np.float32)
    sfp[3, :2] = 0.0                                   # zero scale: dead blocks
    xd, gd, cd, dd, sd = dev(x), dev(g), dev(crs), dev(dgs), dev(sfp)
    a_dev = torch.tensor([a], dtype=torch.float32, device="cuda") if f == O.NVFP4 else None
    kw = dict(sub_block=sub, sfp=sd)
    y, sb = F.focus_fq_fwd(xd, f, cd, dd, a_dev, want_scales=True, **kw)
    codes, sb2 = F.focus_pack(xd, f, cd, dd, a_dev, **kw)
    gx, gc, gdg, gs = F.focus_fq_bwd(xd, gd, f, cd, dd, a_dev, ste=ste, **kw)
    torch.cuda.synchronize()
    ref = O.fwd(x, f, crs=crs, dgs=dgs, alpha=a, sub=sub, sfp=sfp, want_codes=True)
    rb = O.bwd(x, g, f, crs=crs, dgs=dgs, alpha=a, sub=sub, ste=ste, sfp=sfp, want_abs=True,
               want_gsfp=True)
    assert_bits_equal(host(y), ref["y"], "y")
    assert_bits_equal(host(sb), ref["scales"], "scale bytes")
    assert_bits_equal(host(sb2), ref["scales"], "scale bytes (pack)")
    assert_bits_equal(host(codes), ref["codes"], "codes")
    assert_bits_equal(host(gx), rb["gx"], "gx")
    assert_grad_close(host(gc), rb["gcrs"], rb["gcrs_abs"], FLOOR_ROW, "dL/dc")
    assert_grad_close(host(gdg), rb["gdgs"], rb["gdgs_abs"], FLOOR_ROW, "dL/dc^k")
    assert_grad_close(host(gs), rb["gsfp"], rb["gsfp_abs"], FLOOR_ROW, "dL/dS^fp")


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_absmax_sfp_matches_absmax_path_on_gpu(fmt):
    """S^fp initialised via absmax reproduces the absmax path bit for bit;
    the S^fp gradient is also available without S^fp (at the absmax scale)."""
    w, x, g = seeded(64, 512, "bf16", seed=31)
    f = FMT[fmt]
    block = 32 if f == O.MXFP4 else 16
    crs = W.draw_coefs(w, 64 * 512 // block, 17).reshape(64, -1)
    a = O.alpha(x) if f == O.NVFP4 else 0.0
    sfp = absmax_sfp_host(x, f, a)
    xd, gd, cd, sd = dev(x), dev(g), dev(crs), dev(sfp)
    a_dev = torch.tensor([a], dtype=torch.float32, device="cuda") if f == O.NVFP4 else None
    y0 = F.focus_fq_fwd(xd, f, cd, None, a_dev)
    y1 = F.focus_fq_fwd(xd, f, cd, None, a_dev, sfp=sd)
    r0 = F.focus_fq_bwd(xd, gd, f, cd, None, a_dev, want_gsfp=True)
    r1 = F.focus_fq_bwd(xd, gd, f, cd, None, a_dev, sfp=sd)
    torch.cuda.synchronize()
    assert torch.equal(y0.view(torch.int16), y1.view(torch.int16))
    assert torch.equal(r0[0].view(torch.int16), r1[0].view(torch.int16))
    assert torch.equal(r0[1], r1[1]) and torch.equal(r0[3], r1[3])
    rb = O.bwd(x, g, f, crs=crs, alpha=a, want_abs=True, want_gsfp=True)
    assert_grad_close(host(r0[3]), rb["gsfp"], rb["gsfp_abs"], FLOOR_ROW, "dL/dS^fp at absmax")


# ---------------------------------------------------------------------------
# export in the block-scaled MMA scale-factor layout
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("dtype", ["bf16", "f32", "f16"])
@pytest.mark.parametrize("rows,cols", [(256, 512), (300, 96), (1, 48 * 2), (129, 1216)])
def test_pack_mma_layout(fmt, dtype, rows, cols):
    f = FMT[fmt]
    block = 32 if f == O.MXFP4 else 16
    if cols % block:
        cols = cols * 2
    w, x, g = seeded(rows, cols, dtype, seed=rows + cols)
    crs = W.draw_coefs(w, rows * cols // block, 21).reshape(rows, -1)
    dgs = W.draw_coefs(w, rows * cols // 8, 22).reshape(rows, -1)
    xd, cd, dd = dev(x), dev(crs), dev(dgs)
    a = O.alpha(x) if f == O.NVFP4 else 0.0
    a_dev = torch.tensor([a], dtype=torch.float32, device="cuda") if f == O.NVFP4 else None
    # poison the tile buffer: padding must come back as zeros
    desc = F.make_desc(xd, f, 8)
    tiles = torch.full((F.focus_mma_scale_bytes(desc),), 0xA5, dtype=torch.uint8, device="cuda")
    codes, tiles = F.focus_pack_mma(xd, f, cd, dd, a_dev, scale_tiles=tiles)
    codes_rm, scales_rm = F.focus_pack(xd, f, cd, dd, a_dev)
    torch.cuda.synchronize()
    ref = O.fwd(x, f, crs=crs, dgs=dgs, alpha=a, want_y=False, want_codes=True)
    assert_bits_equal(host(codes), ref["codes"], "codes (mma export)")
    assert_bits_equal(host(codes_rm), ref["codes"], "codes (row-major export)")
    assert_bits_equal(host(tiles), O.mma_scale_tiles(ref["scales"]), "scale tiles")


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_f16_overflow_and_subnormals(fmt):
    """binary16 I/O at the edges: values whose dequantized result or input
    gradient leaves the binary16 range (-> inf, as the oracle rounds) and
    subnormal inputs."""
    f = FMT[fmt]
    block = 32 if f == O.MXFP4 else 16
    rows, cols = 8, 4 * block
    rng = np.random.default_rng(7)
    x = (rng.standard_normal((rows, cols)) * 0.2).astype(np.float32)
    x[0] *= 2.0 ** 15                       # near the top of the binary16 range
    x[1] *= 2.0 ** -16                      # subnormal binary16 inputs
    x[2, :block] = 60000.0
    x[2, 1] = -65504.0
    g = rng.standard_normal((rows, cols)).astype(np.float32)
    g[3] = np.clip(g[3] * 16000.0, -65000.0, 65000.0)   # finite in binary16; g / c overflows
    crs = np.full((rows, cols // block), 0.7, np.float32)   # c < 1: y above x
    run_case(x.astype(np.float16), g.astype(np.float16), f, crs, None)
