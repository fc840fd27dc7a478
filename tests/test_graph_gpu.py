"""GPU: the launch structure the benchmark uses -- each tensor's alpha,
forward, backward and pack chained on its own stream, the block kernels and
the alpha reduction as programmatic dependent launches, captured in one CUDA
graph and replayed -- gives exactly the results of the same calls made one
after another on one stream, bit for bit, on every replay.  A dependent
launch that read its predecessor's output too early (alpha before the
forward, the forward's inputs) would show here."""
import pytest
import torch

import oracle as O
from paper_2608_01847_gb300 import build as B
from paper_2608_01847_gb300 import focus as F
from paper_2608_01847_gb300 import workloads as W
from gpu_helpers import dev

pytestmark = pytest.mark.gpu

FMT = {"mx": O.MXFP4, "nv": O.NVFP4}
# tensors of different sizes, one large enough for the eight-times grid
# (at least 16 rounds of resident CTAs)
SHAPES = [(96, 640), (1024, 2048), (301, 640), (24576, 4096)]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    F.lib()


def tensors(fmt, sub, seed):
    block = 32 if fmt == O.MXFP4 else 16
    out = []
    for i, (rows, cols) in enumerate(SHAPES):
        w = W.Workload("t", (W.TensorSpec("t", rows, cols),), "bf16", ("mxfp4",), "weight", 5.0, 0.02,
                       "entries", 0.01, 20.0, (0.8, 1.2), seed + i)
        x, g = W.host_tensor(w, 0)
        crs = W.draw_coefs(w, rows * cols // block, 3).reshape(rows, cols // block)
        dgs = W.draw_coefs(w, rows * cols // sub, 4).reshape(rows, cols // sub)
        out.append({"x": dev(x), "g": dev(g), "crs": dev(crs), "dgs": dev(dgs)})
    return out


def outputs(t, fmt):
    """Fresh output buffers of one tensor's four phases."""
    x = t["x"]
    rows, cols = x.shape
    block = 32 if fmt == O.MXFP4 else 16
    ws = torch.empty(max(16, F.focus_workspace_bytes(F.make_desc(x, fmt, 8, False), F.FOCUS_WS_BWD),
                         F.focus_workspace_bytes(F.make_desc(x, fmt, 8, False), F.FOCUS_WS_ALPHA)),
                     dtype=torch.uint8, device="cuda")
    return {"alpha": torch.full((1,), -1.0, dtype=torch.float32, device="cuda"),
            "y": torch.empty_like(x), "gx": torch.empty_like(x),
            "gcrs": torch.empty_like(t["crs"]), "gdgs": torch.empty_like(t["dgs"]),
            "codes": torch.empty((rows, cols // 2), dtype=torch.uint8, device="cuda"),
            "scales": torch.empty((rows, cols // block), dtype=torch.uint8, device="cuda"), "ws": ws}


def chain(t, o, fmt, sub):
    """alpha -> forward -> backward -> pack of one tensor on the current stream."""
    alpha = None
    if fmt == O.NVFP4:
        F.focus_nvfp4_alpha(t["x"], o["alpha"], o["ws"])
        alpha = o["alpha"]
    F.focus_fq_fwd(t["x"], fmt, t["crs"], t["dgs"], alpha, sub_block=sub, y=o["y"])
    F.focus_fq_bwd(t["x"], t["g"], fmt, t["crs"], t["dgs"], alpha, sub_block=sub, gx=o["gx"],
                   gcrs=o["gcrs"], gdgs=o["gdgs"], ws=o["ws"])
    F.focus_pack(t["x"], fmt, t["crs"], t["dgs"], alpha, sub_block=sub, codes=o["codes"],
                 scale_bytes=o["scales"])


def same(a, b, what):
    assert a.shape == b.shape, what
    assert torch.equal(a.contiguous().view(torch.uint8), b.contiguous().view(torch.uint8)), what


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_chained_graph_equals_sequential(fmt):
    f, sub = FMT[fmt], 8
    ts = tensors(f, sub, seed=77 if fmt == "mx" else 91)
    # reference: the calls one after another on one stream, no graph
    ref = [outputs(t, f) for t in ts]
    for t, o in zip(ts, ref):
        chain(t, o, f, sub)
    torch.cuda.synchronize()
    # the benchmark's structure: one stream per tensor, forked from and joined
    # back to the capturing stream, all captured in one graph
    got = [outputs(t, f) for t in ts]
    graph = torch.cuda.CUDAGraph()
    side = [torch.cuda.Stream() for _ in ts]
    cap = torch.cuda.Stream()
    cap.wait_stream(torch.cuda.current_stream())
    with torch.cuda.graph(graph, stream=cap):
        main = torch.cuda.current_stream()
        for t, o, st in zip(ts, got, side):
            st.wait_stream(main)
            with torch.cuda.stream(st):
                chain(t, o, f, sub)
        for st in side:
            main.wait_stream(st)
    torch.cuda.current_stream().wait_stream(cap)
    for replay in range(3):
        for o in got:   # poison the outputs: every replay must rewrite them
            for k, v in o.items():
                if k != "ws":
                    v.fill_(7 if v.dtype == torch.uint8 else float("nan"))
        graph.replay()
        torch.cuda.synchronize()
        for i, (r, o) in enumerate(zip(ref, got)):
            for k in ("y", "gx", "gcrs", "gdgs", "codes", "scales") + (("alpha",) if f == O.NVFP4 else ()):
                same(o[k], r[k], f"replay {replay}, tensor {i}, {k}")
