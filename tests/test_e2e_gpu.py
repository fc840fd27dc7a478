"""GPU: the benchmark's end-to-end step -- inputs copied from pinned host
memory (one copy per tensor: the inputs share an allocation), each tensor's
phases, outputs copied back (one copy per tensor), three chained streams
captured in one graph -- returns to the host exactly what the same phases
called one after another on device-resident inputs produce, bit for bit.
The device inputs and outputs are poisoned before the replay, so every
value the host receives must have travelled through the pipeline."""
import pytest
import torch

import bench
from paper_2608_01847_gb300 import build as B
from paper_2608_01847_gb300 import focus as F
from paper_2608_01847_gb300 import workloads as W

pytestmark = pytest.mark.gpu

SHAPES = [(96, 640), (301, 1024), (2048, 2048), (64, 4096)]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    F.lib()


def host_view(t, host_buf, dev_buf, a):
    """The host mirror's bytes of device array `a` (a view of `dev_buf`)."""
    off = a.data_ptr() - dev_buf.data_ptr()
    n = a.numel() * a.element_size()
    return host_buf[off:off + n].view(a.dtype).view(a.shape)


@pytest.mark.parametrize("fmt,shared,sfp", [("nvfp4", False, False), ("mxfp4", False, True),
                                            ("nvfp4", True, False)])
def test_pipeline_returns_the_step_results(fmt, shared, sfp):
    w = W.Workload("e2e", tuple(W.TensorSpec(f"t{i}", r, c) for i, (r, c) in enumerate(SHAPES)), "bf16",
                   ("mxfp4", "nvfp4"), "weight", 5.0, 0.02, "entries", 0.01, 20.0, (0.9, 1.1), 314)
    case = bench.Case(workload="e2e", fmt=fmt, shared=shared, sfp=sfp)
    ts = [bench.Tensor(case, w, i, torch.device("cuda")) for i in range(len(SHAPES))]
    phases = case.phases()
    # reference: the phases called directly on the device-resident inputs
    for ph in phases:
        for t in ts:
            t.run(ph)
    torch.cuda.synchronize()
    ref = [[o.clone() for o in t.outputs()] for t in ts]
    for t in ts:
        t.host_in = t.in_buf.cpu().pin_memory()
        t.host_out = torch.full_like(t.out_buf, 0x5A, device="cpu").pin_memory()
    graph = bench.PipelineGraph(ts, phases, torch.device("cuda"))
    for t in ts:   # poison: the replay must bring every input in and every output out
        t.in_buf.fill_(0xA5)
        t.out_buf.fill_(0xC3)
    torch.cuda.synchronize()
    graph.replay()
    torch.cuda.synchronize()
    for i, t in enumerate(ts):
        for j, (a, r) in enumerate(zip(t.outputs(), ref[i])):
            got = host_view(t, t.host_out, t.out_buf, a)
            assert torch.equal(got.view(torch.uint8), r.cpu().contiguous().view(torch.uint8)), (i, j)
