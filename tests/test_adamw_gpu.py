"""GPU parity of the backward fused with one AdamW step (Sec. 3.2 STE,
Sec. 4.1 AdamW) against the oracle.

Input gradients must be bit-exact and coefficient / scale gradients within
the gradient tolerance, exactly as for the plain backward.  The updated
parameters and moments must lie inside the interval that the gradient
tolerance and binary32 rounding of the update allow (gpu_helpers.adamw_bounds,
itself checked on the CPU in test_adamw_bound_cpu.py).  The fused call must
also give bit-identical gradients to focus_fq_bwd, and a captured CUDA graph
that advances the device step counter must replay the eager sequence bit for
bit."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_01847_gb300 import build as B
from paper_2608_01847_gb300 import focus as F
from paper_2608_01847_gb300 import workloads as W
from gpu_helpers import (FLOOR_ROW, FLOOR_SHARED, assert_adamw_close, assert_bits_equal,
                         assert_grad_close, dev, host)

pytestmark = pytest.mark.gpu

FMT = {"mx": O.MXFP4, "nv": O.NVFP4}
# the paper's rates (Sec. 4.1) and PyTorch's AdamW defaults for the rest
HP = {O.MXFP4: dict(lr_coef=5e-2, lr_scale=2e-2, beta1=0.9, beta2=0.999, eps=1e-8,
                    weight_decay=0.01),
      O.NVFP4: dict(lr_coef=1e-3, lr_scale=5e-3, beta1=0.9, beta2=0.999, eps=1e-8,
                    weight_decay=0.01)}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    F.lib()


def seeded(rows, cols, dtype, seed):
    w = W.Workload("t", (W.TensorSpec("t", rows, cols),), dtype, ("mxfp4",), "weight", 5.0, 0.02,
                   "entries", 0.01, 20.0, (0.8, 1.2), seed)
    x, g = W.host_tensor(w, 0)
    return w, x, g


def absmax_sfp_host(x, fmt, alpha):
    block = 32 if fmt == O.MXFP4 else 16
    xf = W.bf16_bits_to_f32(x) if x.dtype == np.uint16 else x
    rows, cols = xf.shape
    m = np.abs(xf.reshape(rows, cols // block, block)).max(axis=2).astype(np.float32)
    den = np.float32(6) if fmt == O.MXFP4 else np.float32(alpha) * np.float32(6)
    return (m / den).astype(np.float32)


def make_state(w, shape, step, seed):
    """Moments as after step - 1 updates (zero before the first)."""
    if step == 1:
        return np.zeros(shape, np.float32), np.zeros(shape, np.float32)
    n = int(np.prod(shape))
    m = (W.draw_coefs(w, n, seed) - np.float32(1.0)) * np.float32(0.5)
    v = (W.draw_coefs(w, n, seed + 1) - np.float32(0.7)) * np.float32(0.02)
    return m.reshape(shape), v.reshape(shape)


def run_adamw(x, g, fmt, learn, step, sub=8, shared=False, ste=O.STE_IDENTITY, seed=0,
              grads_out=True, dtype_tag="bf16"):
    rows, cols = x.shape
    block = 32 if fmt == O.MXFP4 else 16
    crow = 1 if shared else rows
    w, _, _ = seeded(8, 64, dtype_tag, seed)
    params = {}
    if "crs" in learn:
        params["crs"] = W.draw_coefs(w, crow * (cols // block), seed + 3).reshape(crow, -1)
    if "dgs" in learn:
        params["dgs"] = W.draw_coefs(w, crow * (cols // sub), seed + 4).reshape(crow, -1)
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    if "sfp" in learn:
        jit = W.draw_coefs(w, rows * (cols // block), seed + 5).reshape(rows, -1)
        params["sfp"] = (absmax_sfp_host(x, fmt, a) * jit).astype(np.float32)
    moments = {k: make_state(w, v.shape, step, seed + 10 + 2 * i)
               for i, (k, v) in enumerate(sorted(params.items()))}
    hp = HP[fmt]
    xd, gd = dev(x), dev(g)
    pd = {k: dev(v) for k, v in params.items()}
    md = {k: (dev(m), dev(v)) for k, (m, v) in moments.items()}
    a_dev = torch.tensor([a], dtype=torch.float32, device="cuda") if fmt == O.NVFP4 else None
    t_dev = torch.tensor([step], dtype=torch.int64, device="cuda")
    go = {}
    if grads_out:
        if "crs" in params:
            go["gcrs"] = torch.empty_like(pd["crs"])
        if "dgs" in params:
            go["gdgs"] = torch.empty_like(pd["dgs"])
        if "sfp" in params:
            go["gsfp"] = torch.empty_like(pd["sfp"])
    gx = F.focus_fq_bwd_adamw(xd, gd, fmt, t_dev, hp, crs=pd.get("crs"), dgs=pd.get("dgs"),
                              sfp=pd.get("sfp"), moments=md, alpha=a_dev, sub_block=sub,
                              shared=shared, ste=ste, **go)
    torch.cuda.synchronize()
    ref = O.bwd_adamw(x, g, fmt, params, moments, hp, step, alpha=a, sub=sub, shared=shared,
                      ste=ste)
    assert_bits_equal(host(gx), ref["gx"], "gx")
    floor = FLOOR_SHARED if shared else FLOOR_ROW
    gname = {"crs": "gcrs", "dgs": "gdgs", "sfp": "gsfp"}
    for k in params:
        lr = hp["lr_scale"] if k == "sfp" else hp["lr_coef"]
        if grads_out:
            r = ref[k]
            assert_grad_close(host(go[gname[k]]), r["grad"].astype(np.float32), r["grad_abs"],
                              floor, f"dL/d{k}")
        assert_adamw_close((host(pd[k]), host(md[k][0]), host(md[k][1])), params[k],
                           moments[k][0], moments[k][1], ref[k], floor, lr, hp, step, k)
    return dict(params=params, moments=moments, a=a, dev=pd, mom=md, go=go, gx=gx)


# ---------------------------------------------------------------------------
# per-row coefficients: formats, dtypes, learned subsets, steps, sub-blocks
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("dtype", ["bf16", "f32", "f16"])
@pytest.mark.parametrize("learn", [("crs", "dgs", "sfp"), ("crs", "dgs"), ("dgs",), ("sfp",),
                                   ("crs", "sfp")])
@pytest.mark.parametrize("step", [1, 7, 1000])
def test_fused_adamw_per_row(fmt, dtype, learn, step):
    rows, cols = 203, 448 if fmt == "mx" else 464      # several CTAs, ragged tail
    _, x, g = seeded(rows, cols, dtype, seed=rows + step)
    run_adamw(x, g, FMT[fmt], learn, step, seed=step, dtype_tag=dtype)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("sub", [2, 4, 16])
def test_fused_adamw_sub_blocks(fmt, sub):
    _, x, g = seeded(64, 512, "bf16", seed=sub)
    run_adamw(x, g, FMT[fmt], ("crs", "dgs", "sfp"), 3, sub=sub, seed=sub)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_fused_adamw_clipped_ste_without_gradient_outputs(fmt):
    _, x, g = seeded(100, 256, "bf16", seed=41)
    run_adamw(x, g, FMT[fmt], ("crs", "dgs", "sfp"), 5, ste=O.STE_CLIPPED, seed=41,
              grads_out=False)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("learn", [("crs", "dgs"), ("dgs",)])
def test_fused_adamw_shared_rows(fmt, learn):
    _, x, g = seeded(777, 256, "bf16", seed=51)
    run_adamw(x, g, FMT[fmt], learn, 4, shared=True, seed=51)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_fused_adamw_shared_rows_empty_batch(fmt):
    """No rows: the gradient is a sum over nothing (zero) and the step still
    applies (weight decay and the moments' decay)."""
    f = FMT[fmt]
    block = 32 if f == O.MXFP4 else 16
    cols = 256
    w, _, _ = seeded(8, 64, "bf16", 3)
    c = W.draw_coefs(w, cols // block, 61).reshape(1, -1)
    m, v = make_state(w, c.shape, 9, 62)
    x = torch.empty((0, cols), dtype=torch.bfloat16, device="cuda")
    cd, md, vd = dev(c), dev(m), dev(v)
    t_dev = torch.tensor([9], dtype=torch.int64, device="cuda")
    a_dev = torch.zeros(1, dtype=torch.float32, device="cuda")
    F.focus_fq_bwd_adamw(x, x, f, t_dev, HP[f], crs=cd, moments={"crs": (md, vd)}, alpha=a_dev,
                         shared=True, want_gx=False)
    torch.cuda.synchronize()
    zero = np.zeros(c.shape)
    pn, mn, vn = O.adamw(c, zero, m, v, HP[f]["lr_coef"], HP[f]["beta1"], HP[f]["beta2"],
                         HP[f]["eps"], HP[f]["weight_decay"], 9)
    ref = {"grad": zero, "grad_abs": zero, "p": pn}
    assert_adamw_close((host(cd), host(md), host(vd)), c, m, v, ref, FLOOR_SHARED,
                       HP[f]["lr_coef"], HP[f], 9, "empty batch")


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_fused_gradients_equal_plain_backward(fmt):
    """The fused call computes exactly the plain backward's gradients."""
    f = FMT[fmt]
    _, x, g = seeded(150, 320 if f == O.MXFP4 else 336, "bf16", seed=71)
    r = run_adamw(x, g, f, ("crs", "dgs", "sfp"), 2, seed=71)
    p, a = r["params"], r["a"]
    a_dev = torch.tensor([a], dtype=torch.float32, device="cuda") if f == O.NVFP4 else None
    gx, gc, gdg, gs = F.focus_fq_bwd(dev(x), dev(g), f, dev(p["crs"]), dev(p["dgs"]), a_dev,
                                     sfp=dev(p["sfp"]))
    torch.cuda.synchronize()
    assert torch.equal(gx.view(torch.int16), r["gx"].view(torch.int16))
    assert torch.equal(gc, r["go"]["gcrs"]) and torch.equal(gdg, r["go"]["gdgs"])
    assert torch.equal(gs, r["go"]["gsfp"])


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_graph_replay_advances_the_step(fmt):
    """Three replays of a captured graph (step counter advanced inside it)
    equal three eager calls bit for bit."""
    f = FMT[fmt]
    block = 32 if f == O.MXFP4 else 16
    w, x, g = seeded(96, 512, "bf16", seed=81)
    rows, cols = x.shape
    c0 = W.draw_coefs(w, rows * cols // block, 82).reshape(rows, -1)
    d0 = W.draw_coefs(w, rows * cols // 8, 83).reshape(rows, -1)
    a = O.alpha(x) if f == O.NVFP4 else 0.0
    s0 = absmax_sfp_host(x, f, a)
    xd, gd = dev(x), dev(g)
    a_dev = torch.tensor([a], dtype=torch.float32, device="cuda")

    def fresh():
        st = {k: dev(v) for k, v in (("crs", c0), ("dgs", d0), ("sfp", s0))}
        mom = {k: (torch.zeros_like(v), torch.zeros_like(v)) for k, v in st.items()}
        return st, mom, torch.zeros(1, dtype=torch.int64, device="cuda")

    def one(st, mom, t):
        t.add_(1)
        F.focus_fq_bwd_adamw(xd, gd, f, t, HP[f], crs=st["crs"], dgs=st["dgs"], sfp=st["sfp"],
                             moments=mom, alpha=a_dev, want_gx=False)

    e_st, e_mom, e_t = fresh()
    for _ in range(3):
        one(e_st, e_mom, e_t)
    g_st, g_mom, g_t = fresh()
    one(g_st, g_mom, g_t)             # warm-up outside capture (first call resolves launches)
    g_st, g_mom, g_t2 = fresh()
    g_t.copy_(g_t2)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        with torch.cuda.graph(graph, stream=s):
            one(g_st, g_mom, g_t)
    torch.cuda.current_stream().wait_stream(s)
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    assert int(g_t.item()) == 3
    for k in ("crs", "dgs", "sfp"):
        assert torch.equal(g_st[k], e_st[k]), k
        assert torch.equal(g_mom[k][0], e_mom[k][0]) and torch.equal(g_mom[k][1], e_mom[k][1]), k
