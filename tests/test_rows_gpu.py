"""GPU: with per-row coefficients every row is an independent problem (its
blocks, its c_i and c_i^k, its S^fp; alpha is the whole tensor's and is passed
in), so the forward, the backward (with and without S^fp), the fused AdamW
backward and the export over consecutive row ranges give exactly the results
of one call over the whole tensor: a caller may cut a tensor into row ranges
(to stream it in pieces, to bound a workspace) and call the entry points on
each.  Pinned here on ragged boundaries, one-row ranges and ranges that start
at any row."""
import pytest
import torch

import oracle as O
from paper_2608_01847_gb300 import build as B
from paper_2608_01847_gb300 import focus as F
from paper_2608_01847_gb300 import workloads as W
from gpu_helpers import dev

pytestmark = pytest.mark.gpu

FMT = {"mx": O.MXFP4, "nv": O.NVFP4}
ROWS, COLS = 1037, 1536
CUTS = [0, 1, 130, 131, 600, 1036, ROWS]   # ragged: one-row chunks, odd starts


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    F.lib()


def inputs(fmt, sub, seed):
    block = 32 if fmt == O.MXFP4 else 16
    w = W.Workload("t", (W.TensorSpec("t", ROWS, COLS),), "bf16", ("mxfp4",), "weight", 5.0, 0.02,
                   "entries", 0.01, 20.0, (0.8, 1.2), seed)
    x, g = W.host_tensor(w, 0)
    crs = W.draw_coefs(w, ROWS * COLS // block, 3).reshape(ROWS, COLS // block)
    dgs = W.draw_coefs(w, ROWS * COLS // sub, 4).reshape(ROWS, COLS // sub)
    x, g, crs, dgs = dev(x), dev(g), dev(crs), dev(dgs)
    alpha = F.focus_nvfp4_alpha(x) if fmt == O.NVFP4 else None
    m = x.float().abs().view(ROWS, COLS // block, block).amax(-1)
    den = alpha * 6.0 if alpha is not None else 6.0
    gen = torch.Generator(device="cuda")
    gen.manual_seed(seed)
    sfp = (m / den * (torch.rand(m.shape, generator=gen, device="cuda") * 0.2 + 0.9)).contiguous()
    return x, g, crs, dgs, alpha, sfp


def same(a, b, what):
    assert a.shape == b.shape, what
    assert torch.equal(a.contiguous().view(torch.uint8), b.contiguous().view(torch.uint8)), what


def spans():
    return list(zip(CUTS[:-1], CUTS[1:]))


@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("use_sfp", [False, True])
def test_row_chunks_equal_whole(fmt, use_sfp):
    f, sub = FMT[fmt], 8
    x, g, crs, dgs, alpha, sfp = inputs(f, sub, 505 if fmt == "mx" else 606)
    sfp = sfp if use_sfp else None
    kw = dict(sub_block=sub)
    y = F.focus_fq_fwd(x, f, crs, dgs, alpha, sfp=sfp, **kw)
    bwd = F.focus_fq_bwd(x, g, f, crs, dgs, alpha, sfp=sfp, **kw)
    codes, scales = F.focus_pack(x, f, crs, dgs, alpha, sfp=sfp, **kw)
    # the same calls on row ranges, writing into row slices of one buffer
    y2, codes2, scales2 = (torch.full_like(t, 7) for t in (y, codes, scales))
    bwd2 = [torch.full_like(t, 7) for t in bwd]
    rs = lambda t, a, b: None if t is None else t[a:b]
    for a, b in spans():
        F.focus_fq_fwd(x[a:b], f, crs[a:b], dgs[a:b], alpha, sfp=rs(sfp, a, b), y=y2[a:b], **kw)
        out = dict(gx=bwd2[0][a:b], gcrs=bwd2[1][a:b], gdgs=bwd2[2][a:b])
        if use_sfp:
            out["gsfp"] = bwd2[3][a:b]
        F.focus_fq_bwd(x[a:b], g[a:b], f, crs[a:b], dgs[a:b], alpha, sfp=rs(sfp, a, b), **out, **kw)
        F.focus_pack(x[a:b], f, crs[a:b], dgs[a:b], alpha, sfp=rs(sfp, a, b), codes=codes2[a:b],
                     scale_bytes=scales2[a:b], **kw)
    torch.cuda.synchronize()
    same(y2, y, "y")
    for name, got, ref in zip(("gx", "gcrs", "gdgs", "gsfp"), bwd2, bwd):
        same(got, ref, name)
    same(codes2, codes, "codes")
    same(scales2, scales, "scales")


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_row_chunks_equal_whole_adamw(fmt):
    f, sub = FMT[fmt], 8
    x, g, crs, dgs, alpha, sfp = inputs(f, sub, 707 if fmt == "mx" else 808)
    hp = dict(lr_coef=1e-3, lr_scale=5e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)
    runs = []
    for chunked in (False, True):
        p = {"crs": crs.clone(), "dgs": dgs.clone(), "sfp": sfp.clone()}
        mom = {k: (torch.zeros_like(v), torch.zeros_like(v)) for k, v in p.items()}
        step = torch.zeros(1, dtype=torch.int64, device="cuda")
        gx = torch.full_like(x, 7)
        for it in range(2):   # two steps: the second reads the first's moments
            step.add_(1)
            gi = g if it == 0 else -g
            parts = spans() if chunked else [(0, ROWS)]
            for a, b in parts:
                F.focus_fq_bwd_adamw(x[a:b], gi[a:b], f, step, hp, crs=p["crs"][a:b], dgs=p["dgs"][a:b],
                                     sfp=p["sfp"][a:b],
                                     moments={k: (m[a:b], v[a:b]) for k, (m, v) in mom.items()},
                                     alpha=alpha, sub_block=sub, gx=gx[a:b])
        torch.cuda.synchronize()
        runs.append((gx, p, mom))
    (gx1, p1, m1), (gx2, p2, m2) = runs
    same(gx2, gx1, "gx")
    for k in p1:
        same(p2[k], p1[k], k)
        same(m2[k][0], m1[k][0], k + " m")
        same(m2[k][1], m1[k][1], k + " v")
