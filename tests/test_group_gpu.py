"""GPU: the group entry points (one launch for several tensors) give exactly
the per-tensor entry points' results, bit for bit, and the oracle's."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_01847_gb300 import build as B
from paper_2608_01847_gb300 import focus as F
from paper_2608_01847_gb300 import workloads as W
from gpu_helpers import FLOOR_ROW, assert_bits_equal, assert_grad_close, dev, host

pytestmark = pytest.mark.gpu

FMT = {"mx": O.MXFP4, "nv": O.NVFP4}
# a layer's worth of shapes: different sizes, one tensor much larger, an empty one
SHAPES = [(96, 640), (32, 640), (160, 1024), (0, 640), (301, 640), (64, 2048)]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    F.lib()


def tensors(fmt, dtype, sub, seed, sfp=False):
    block = 32 if fmt == O.MXFP4 else 16
    out = []
    for i, (rows, cols) in enumerate(SHAPES):
        w = W.Workload("t", (W.TensorSpec("t", rows, cols),), dtype, ("mxfp4",), "weight", 5.0, 0.02,
                       "entries", 0.01, 20.0, (0.8, 1.2), seed + i)
        x, g = W.host_tensor(w, 0)
        crs = W.draw_coefs(w, rows * cols // block, 3).reshape(rows, cols // block)
        dgs = W.draw_coefs(w, rows * cols // sub, 4).reshape(rows, cols // sub)
        it = {"x": dev(x), "g": dev(g), "crs": dev(crs), "dgs": dev(dgs), "host": (x, g, crs, dgs)}
        if sfp:
            jit = W.draw_coefs(w, rows * cols // block, 5).reshape(rows, cols // block)
            it["sfp"] = dev((jit * np.float32(0.01 if fmt == O.MXFP4 else 20.0)).astype(np.float32))
        out.append(it)
    return out


def same(a, b, what):
    assert a.shape == b.shape, what
    if a.numel() == 0:
        return
    assert torch.equal(a.contiguous().view(torch.uint8), b.contiguous().view(torch.uint8)), what


@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("dtype", ["bf16", "f16", "f32"])
@pytest.mark.parametrize("sub", [8, 4])
def test_group_equals_per_tensor(fmt, dtype, sub):
    f = FMT[fmt]
    ts = tensors(f, dtype, sub, seed=10 * sub + len(dtype))
    # alpha: group vs per tensor
    alphas = F.focus_nvfp4_alpha_group([t["x"] for t in ts])
    for i, t in enumerate(ts):
        a1 = F.focus_nvfp4_alpha(t["x"])
        same(alphas[i:i + 1], a1, f"alpha {i}")
        t["alpha"] = alphas[i:i + 1] if f == O.NVFP4 else None
    kw = dict(sub_block=sub)
    ys = F.focus_fq_fwd_group([{k: t.get(k) for k in ("x", "crs", "dgs", "alpha")} for t in ts], f, **kw)
    packs = F.focus_pack_group([{k: t.get(k) for k in ("x", "crs", "dgs", "alpha")} for t in ts], f, **kw)
    bw = F.focus_fq_bwd_group([dict({k: t.get(k) for k in ("x", "g", "crs", "dgs", "alpha")},
                                    gx=None, gcrs=None, gdgs=None) for t in ts], f, **kw)
    torch.cuda.synchronize()
    for i, t in enumerate(ts):
        y1 = F.focus_fq_fwd(t["x"], f, t["crs"], t["dgs"], t["alpha"], **kw)
        c1, s1 = F.focus_pack(t["x"], f, t["crs"], t["dgs"], t["alpha"], **kw)
        gx1, gc1, gd1 = F.focus_fq_bwd(t["x"], t["g"], f, t["crs"], t["dgs"], t["alpha"], **kw)
        torch.cuda.synchronize()
        same(ys[i], y1, f"y {i}")
        same(packs[i][0], c1, f"codes {i}")
        same(packs[i][1], s1, f"scales {i}")
        same(bw[i]["gx"], gx1, f"gx {i}")
        same(bw[i]["gcrs"], gc1, f"gcrs {i}")
        same(bw[i]["gdgs"], gd1, f"gdgs {i}")


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_group_learnable_scale_equals_per_tensor(fmt):
    f = FMT[fmt]
    ts = tensors(f, "bf16", 8, seed=77, sfp=True)
    ts[1].pop("sfp")                       # a tensor without S^fp in the same group
    alphas = F.focus_nvfp4_alpha_group([t["x"] for t in ts])
    for i, t in enumerate(ts):
        t["alpha"] = alphas[i:i + 1] if f == O.NVFP4 else None
    keys = ("x", "g", "crs", "dgs", "alpha", "sfp")
    bw = F.focus_fq_bwd_group([dict({k: t.get(k) for k in keys}, gx=None, gcrs=None, gdgs=None, gsfp=None)
                               for t in ts], f)
    ys = F.focus_fq_fwd_group([{k: t.get(k) for k in ("x", "crs", "dgs", "alpha", "sfp")} for t in ts], f)
    torch.cuda.synchronize()
    for i, t in enumerate(ts):
        r = F.focus_fq_bwd(t["x"], t["g"], f, t["crs"], t["dgs"], t["alpha"], sfp=t.get("sfp"),
                           want_gsfp=True)
        y1 = F.focus_fq_fwd(t["x"], f, t["crs"], t["dgs"], t["alpha"], sfp=t.get("sfp"))
        torch.cuda.synchronize()
        same(ys[i], y1, f"y {i}")
        for name, a in zip(("gx", "gcrs", "gdgs", "gsfp"), r):
            same(bw[i][name], a, f"{name} {i}")


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_group_against_oracle(fmt):
    f = FMT[fmt]
    ts = tensors(f, "bf16", 8, seed=91)
    alphas = F.focus_nvfp4_alpha_group([t["x"] for t in ts])
    for i, t in enumerate(ts):
        t["alpha"] = alphas[i:i + 1] if f == O.NVFP4 else None
    ys = F.focus_fq_fwd_group([{k: t.get(k) for k in ("x", "crs", "dgs", "alpha")} for t in ts], f)
    bw = F.focus_fq_bwd_group([dict({k: t.get(k) for k in ("x", "g", "crs", "dgs", "alpha")},
                                    gx=None, gcrs=None, gdgs=None) for t in ts], f)
    torch.cuda.synchronize()
    for i, t in enumerate(ts):
        x, g, crs, dgs = t["host"]
        if x.size == 0:
            continue
        a = O.alpha(x) if f == O.NVFP4 else 0.0
        if f == O.NVFP4:
            assert_bits_equal(host(alphas[i:i + 1]), np.array([a], np.float32), f"alpha {i}")
        ref = O.fwd(x, f, crs=crs, dgs=dgs, alpha=a)
        rb = O.bwd(x, g, f, crs=crs, dgs=dgs, alpha=a, want_abs=True)
        assert_bits_equal(host(ys[i]), ref["y"], f"y {i}")
        assert_bits_equal(host(bw[i]["gx"]), rb["gx"], f"gx {i}")
        assert_grad_close(host(bw[i]["gcrs"]), rb["gcrs"], rb["gcrs_abs"], FLOOR_ROW, f"dL/dc {i}")
        assert_grad_close(host(bw[i]["gdgs"]), rb["gdgs"], rb["gdgs_abs"], FLOOR_ROW, f"dL/dc^k {i}")
