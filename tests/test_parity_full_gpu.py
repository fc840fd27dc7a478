"""GPU parity at the workloads' full sizes.

Every tensor of each configuration is drawn on the GPU at its real shape and
run through the same entry points, with the same launch configuration, as the
benchmark.  Per-row results are then checked against the oracle on sampled
rows (first, last and 30 random rows of every tensor): codes, scale bytes,
values and input gradients bit for bit, coefficient gradients within the
gradient tolerance.  alpha is checked against the oracle over the whole
tensor.  With coefficients shared by all rows, the gradients are sums over
all 262,144 rows of the activation workload: the oracle computes them over
every row, split across a spawn-started process pool, and the partial sums
are added in binary64.
"""
import concurrent.futures as cf
import multiprocessing as mp
import os

import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_01847_gb300 import build as B
from paper_2608_01847_gb300 import focus as F
from paper_2608_01847_gb300 import workloads as W
import oracle_pool
from gpu_helpers import FLOOR_ROW, FLOOR_SHARED, assert_bits_equal, assert_grad_close, host

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    F.lib()
    O.build()


def _check_tensor(w, idx, fmt, sub=8, seed=0):
    """Full-size run of one tensor; sampled-row comparison with the oracle."""
    block = 32 if fmt == O.MXFP4 else 16
    x, g = W.device_tensor(w, idx, "cuda")
    crs, dgs = W.device_coefs(w, idx, block, sub, "cuda")
    rows, cols = x.shape
    a_dev = F.focus_nvfp4_alpha(x) if fmt == O.NVFP4 else None
    y, sb = F.focus_fq_fwd(x, fmt, crs, dgs, a_dev, sub_block=sub, want_scales=True)
    gx, gc, gd = F.focus_fq_bwd(x, g, fmt, crs, dgs, a_dev, sub_block=sub)
    codes, sb2 = F.focus_pack(x, fmt, crs, dgs, a_dev, sub_block=sub)
    torch.cuda.synchronize()
    xh = host(x)
    a = 0.0
    if fmt == O.NVFP4:
        a = O.alpha(xh)
        assert_bits_equal(host(a_dev), np.array([a], np.float32), f"alpha {w.tensors[idx].name}")
    rng = np.random.default_rng(seed + idx)
    rs = np.unique(np.concatenate([[0, rows - 1], rng.choice(rows, min(30, rows), replace=False)]))
    ri = torch.from_numpy(rs).cuda()
    xs = xh[rs]
    gs = host(g.index_select(0, ri))
    cs, ds = host(crs.index_select(0, ri)), host(dgs.index_select(0, ri))
    ref = O.fwd(xs, fmt, crs=cs, dgs=ds, alpha=a, sub=sub, want_codes=True)
    rb = O.bwd(xs, gs, fmt, crs=cs, dgs=ds, alpha=a, sub=sub, want_abs=True)
    name = f"{w.name}/{w.tensors[idx].name}"
    assert_bits_equal(host(y.index_select(0, ri)), ref["y"], f"{name} y")
    assert_bits_equal(host(sb.index_select(0, ri)), ref["scales"], f"{name} scale bytes")
    assert_bits_equal(host(sb2.index_select(0, ri)), ref["scales"], f"{name} scale bytes (pack)")
    assert_bits_equal(host(codes.index_select(0, ri)), ref["codes"], f"{name} codes")
    assert_bits_equal(host(gx.index_select(0, ri)), rb["gx"], f"{name} gx")
    assert_grad_close(host(gc.index_select(0, ri)), rb["gcrs"], rb["gcrs_abs"], FLOOR_ROW, f"{name} dL/dc")
    assert_grad_close(host(gd.index_select(0, ri)), rb["gdgs"], rb["gdgs_abs"], FLOOR_ROW,
                      f"{name} dL/dc^k")
    del x, g, crs, dgs, y, gx, gc, gd, codes, sb, sb2
    torch.cuda.empty_cache()


@pytest.mark.parametrize("name,fmt", [
    ("qwen3_4b_layer", O.NVFP4),
    ("llama3_8b_block", O.MXFP4), ("llama3_8b_block", O.NVFP4),
    ("llama_70b_layer", O.MXFP4), ("llama_70b_layer", O.NVFP4),
    ("act_262144x4096", O.MXFP4), ("act_262144x4096", O.NVFP4),
])
def test_full_size_per_row(name, fmt):
    w = W.WORKLOADS[name]
    for idx in range(len(w.tensors)):
        _check_tensor(w, idx, fmt)


def test_full_size_sweep_4gb():
    w = W.sweep_workload(1 << 32)
    _check_tensor(w, 0, O.NVFP4)


# ---------------------------------------------------------------------------
# shared-row coefficients over all rows of the activation workload
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("fmt", [O.MXFP4, O.NVFP4])
def test_full_size_shared_rows(fmt, tmp_path):
    w = W.WORKLOADS["act_262144x4096"]
    block = 32 if fmt == O.MXFP4 else 16
    sub = 8
    x, g = W.device_tensor(w, 0, "cuda")
    crs, dgs = W.device_coefs(w, 0, block, sub, "cuda", shared=True)
    a_dev = F.focus_nvfp4_alpha(x) if fmt == O.NVFP4 else None
    gx, gc, gd = F.focus_fq_bwd(x, g, fmt, crs, dgs, a_dev, sub_block=sub, shared=True)
    torch.cuda.synchronize()
    rows, cols = x.shape
    a = float(host(a_dev)[0]) if fmt == O.NVFP4 else 0.0
    # inputs for the pool through one memory-mapped file
    path = os.path.join(tmp_path, "xg.npy")
    arr = np.lib.format.open_memmap(path, mode="w+", dtype=np.uint16, shape=(2, rows, cols))
    arr[0] = host(x)
    arr[1] = host(g)
    arr.flush()
    del arr
    ch, dh = host(crs), host(dgs)
    if fmt == O.NVFP4:
        assert a == O.alpha(np.load(path, mmap_mode="r")[0])
    nproc = max(1, min(32, os.cpu_count() or 1))
    bounds = np.linspace(0, rows, nproc + 1).astype(int)
    jobs = [(path, int(bounds[i]), int(bounds[i + 1]), fmt, a, ch, dh, sub)
            for i in range(nproc) if bounds[i + 1] > bounds[i]]
    with cf.ProcessPoolExecutor(max_workers=nproc, mp_context=mp.get_context("spawn")) as ex:
        parts = list(ex.map(oracle_pool.shared_rows_chunk, jobs))
    ref_c = sum(p[0] for p in parts)
    ref_d = sum(p[1] for p in parts)
    abs_c = sum(p[2] for p in parts)
    abs_d = sum(p[3] for p in parts)
    # the partials are added in binary64 from unrounded values: the tolerance
    # is the shared-row one (1e-5 relative, 2^-30 cancellation floor)
    assert_grad_close(host(gc)[0], ref_c[0], abs_c[0], FLOOR_SHARED, "shared dL/dc")
    assert_grad_close(host(gd)[0], ref_d[0], abs_d[0], FLOOR_SHARED, "shared dL/dc^k")
    # input gradient: sampled rows against the per-row oracle (same formula)
    rng = np.random.default_rng(5)
    rs = np.unique(np.concatenate([[0, rows - 1], rng.choice(rows, 30, replace=False)]))
    xs = np.load(path, mmap_mode="r")[0][rs]
    gs = np.load(path, mmap_mode="r")[1][rs]
    rb = O.bwd(np.ascontiguousarray(xs), np.ascontiguousarray(gs), fmt, crs=ch, dgs=dh, alpha=a,
               sub=sub, shared=True)
    assert_bits_equal(host(gx.index_select(0, torch.from_numpy(rs).cuda())), rb["gx"], "shared gx")


# ---------------------------------------------------------------------------
# learnable S^fp and the fused AdamW step at full size (sampled rows)
# ---------------------------------------------------------------------------
def _sfp_init(x, fmt, a_dev, seed):
    """S^fp as the benchmark initialises it: the absmax scale moved by U(0.9, 1.1)."""
    block = 32 if fmt == O.MXFP4 else 16
    rows, cols = x.shape
    m = x.float().abs().view(rows, cols // block, block).amax(-1)
    den = a_dev * 6.0 if fmt == O.NVFP4 else torch.full((1,), 6.0, device=x.device)
    gen = torch.Generator(device=x.device)
    gen.manual_seed(seed)
    return (m / den * (torch.rand(m.shape, generator=gen, device=x.device) * 0.2 + 0.9)).contiguous()


@pytest.mark.parametrize("name,fmt,idx", [("qwen3_4b_layer", O.NVFP4, 4), ("llama_70b_layer", O.MXFP4, 6)])
def test_full_size_learnable_scale(name, fmt, idx):
    w = W.WORKLOADS[name]
    block = 32 if fmt == O.MXFP4 else 16
    x, g = W.device_tensor(w, idx, "cuda")
    crs, dgs = W.device_coefs(w, idx, block, 8, "cuda")
    a_dev = F.focus_nvfp4_alpha(x) if fmt == O.NVFP4 else torch.zeros(1, device="cuda")
    sfp = _sfp_init(x, fmt, a_dev, 11)
    y, sb = F.focus_fq_fwd(x, fmt, crs, dgs, a_dev, want_scales=True, sfp=sfp)
    codes, _ = F.focus_pack(x, fmt, crs, dgs, a_dev, sfp=sfp)
    gx, gc, gd, gs = F.focus_fq_bwd(x, g, fmt, crs, dgs, a_dev, sfp=sfp)
    torch.cuda.synchronize()
    rows = x.shape[0]
    a = float(host(a_dev)[0]) if fmt == O.NVFP4 else 0.0
    rng = np.random.default_rng(idx + 100)
    rs = np.unique(np.concatenate([[0, rows - 1], rng.choice(rows, 24, replace=False)]))
    ri = torch.from_numpy(rs).cuda()
    sel = lambda t: host(t.index_select(0, ri))
    xs, gsel, cs, ds, ss = sel(x), sel(g), sel(crs), sel(dgs), sel(sfp)
    ref = O.fwd(xs, fmt, crs=cs, dgs=ds, alpha=a, sfp=ss, want_codes=True)
    rb = O.bwd(xs, gsel, fmt, crs=cs, dgs=ds, alpha=a, sfp=ss, want_abs=True, want_gsfp=True)
    assert_bits_equal(sel(y), ref["y"], f"{name} y")
    assert_bits_equal(sel(sb), ref["scales"], f"{name} scale bytes")
    assert_bits_equal(sel(codes), ref["codes"], f"{name} codes")
    assert_bits_equal(sel(gx), rb["gx"], f"{name} gx")
    assert_grad_close(sel(gc), rb["gcrs"], rb["gcrs_abs"], FLOOR_ROW, f"{name} dL/dc")
    assert_grad_close(sel(gd), rb["gdgs"], rb["gdgs_abs"], FLOOR_ROW, f"{name} dL/dc^k")
    assert_grad_close(sel(gs), rb["gsfp"], rb["gsfp_abs"], FLOOR_ROW, f"{name} dL/dS^fp")


@pytest.mark.parametrize("name,fmt,idx", [("qwen3_4b_layer", O.NVFP4, 4), ("llama_70b_layer", O.MXFP4, 6)])
def test_full_size_fused_adamw(name, fmt, idx):
    from gpu_helpers import assert_adamw_close
    hp = dict(lr_coef=5e-2 if fmt == O.MXFP4 else 1e-3, lr_scale=2e-2 * 2.0 ** -7 if fmt == O.MXFP4 else 5e-3,
              beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)
    w = W.WORKLOADS[name]
    block = 32 if fmt == O.MXFP4 else 16
    x, g = W.device_tensor(w, idx, "cuda")
    crs, dgs = W.device_coefs(w, idx, block, 8, "cuda")
    a_dev = F.focus_nvfp4_alpha(x) if fmt == O.NVFP4 else torch.zeros(1, device="cuda")
    sfp = _sfp_init(x, fmt, a_dev, 12)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(idx)
    params = {"crs": crs, "dgs": dgs, "sfp": sfp}
    before = {k: v.clone() for k, v in params.items()}
    moments = {k: ((torch.rand(v.shape, generator=gen, device="cuda") - 0.5) * 0.1,
                   torch.rand(v.shape, generator=gen, device="cuda") * 0.01) for k, v in params.items()}
    mom0 = {k: (m.clone(), v.clone()) for k, (m, v) in moments.items()}
    step = torch.tensor([7], dtype=torch.int64, device="cuda")
    gx = F.focus_fq_bwd_adamw(x, g, fmt, step, hp, crs=crs, dgs=dgs, sfp=sfp, moments=moments, alpha=a_dev)
    torch.cuda.synchronize()
    rows = x.shape[0]
    a = float(host(a_dev)[0]) if fmt == O.NVFP4 else 0.0
    rng = np.random.default_rng(idx + 200)
    rs = np.unique(np.concatenate([[0, rows - 1], rng.choice(rows, 24, replace=False)]))
    ri = torch.from_numpy(rs).cuda()
    sel = lambda t: host(t.index_select(0, ri))
    p0 = {k: sel(v) for k, v in before.items()}
    m0 = {k: (sel(m), sel(v)) for k, (m, v) in mom0.items()}
    ref = O.bwd_adamw(sel(x), sel(g), fmt, p0, m0, hp, 7, alpha=a)
    assert_bits_equal(sel(gx), ref["gx"], f"{name} gx")
    for k in params:
        lr = hp["lr_scale"] if k == "sfp" else hp["lr_coef"]
        assert_adamw_close((sel(params[k]), sel(moments[k][0]), sel(moments[k][1])), p0[k], m0[k][0], m0[k][1],
                           ref[k], FLOOR_ROW, lr, hp, 7, f"{name} {k}")
