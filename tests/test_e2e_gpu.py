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


@pytest.mark.parametrize("piece_elems", [1 << 27, 1 << 19])
@pytest.mark.parametrize("fmt,shared,sfp,adam", [("nvfp4", False, False, False), ("mxfp4", False, True, False),
                                                 ("nvfp4", True, False, False), ("mxfp4", False, False, True),
                                                 ("nvfp4", False, True, True)])
def test_pipeline_returns_the_step_results(fmt, shared, sfp, adam, piece_elems):
    """piece_elems 2^19: the 2048 x 2048 tensor moves and computes in 8 row
    pieces (values, codes and scale bytes leaving while the gradients still
    arrive), the others whole."""
    w = W.Workload("e2e", tuple(W.TensorSpec(f"t{i}", r, c) for i, (r, c) in enumerate(SHAPES)), "bf16",
                   ("mxfp4", "nvfp4"), "weight", 5.0, 0.02, "entries", 0.01, 20.0, (0.9, 1.1), 314)
    case = bench.Case(workload="e2e", fmt=fmt, shared=shared, sfp=sfp, adam=adam)
    step = torch.ones(1, dtype=torch.int64, device="cuda") if adam else None
    ts = [bench.Tensor(case, w, i, torch.device("cuda"), step) for i in range(len(SHAPES))]
    phases = case.phases()
    # the fused optimizer updates the learned arrays in place: keep their
    # values (and the moments) to restore them before the pipeline's step
    learned = []
    if adam:
        for t in ts:
            learned += [t.crs, t.dgs] + ([t.sfp] if t.sfp is not None else [])
            learned += [a for mv in t.moments.values() for a in mv]
    saved = [a.clone() for a in learned]
    # reference: the phases called directly on the device-resident inputs
    for ph in phases:
        for t in ts:
            t.run(ph)
    torch.cuda.synchronize()
    ref = [[o.clone() for o in t.outputs()] for t in ts]
    ref_learned = [a.clone() for a in learned]
    for a, v in zip(learned, saved):
        a.copy_(v)
    for t in ts:
        t.host_in = t.in_buf.cpu().pin_memory()
        t.host_out = torch.full_like(t.out_buf, 0x5A, device="cpu").pin_memory()
    graph = bench.PipelineGraph(ts, phases, torch.device("cuda"), piece_elems=piece_elems)
    # every input byte crosses once (copy spans may include the arena's
    # alignment padding between neighbouring arrays)
    arrays = [a for t in ts for a in t.inputs()]
    extra = graph.h2d - sum(a.numel() * a.element_size() for a in arrays)
    assert 0 <= extra < bench.ARENA_ALIGN * len(arrays), extra
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
    for a, r in zip(learned, ref_learned):   # the optimizer's step, in HBM
        assert torch.equal(a.view(torch.int32), r.view(torch.int32))


@pytest.mark.parametrize("fmt,shared,sfp", [("nvfp4", False, False), ("mxfp4", False, True),
                                            ("nvfp4", True, False)])
def test_staged_steps_return_the_step_results(fmt, shared, sfp):
    """The benchmark's end-to-end steps without the fused optimizer: two
    buffer sets on two streams, each step an input graph, a compute graph
    and an output graph, step k's inputs crossing while step k - 1 returns
    its outputs.
    Three steps (sets A, B, A) from poisoned device buffers: each set's host
    mirror receives exactly the results of the phases called directly."""
    w = W.Workload("e2e", tuple(W.TensorSpec(f"t{i}", r, c) for i, (r, c) in enumerate(SHAPES)), "bf16",
                   ("mxfp4", "nvfp4"), "weight", 5.0, 0.02, "entries", 0.01, 20.0, (0.9, 1.1), 314)
    case = bench.Case(workload="e2e", fmt=fmt, shared=shared, sfp=sfp)
    dev = torch.device("cuda")
    sets = [[bench.Tensor(case, w, i, dev, None) for i in range(len(SHAPES))] for _ in range(2)]
    phases = case.phases()
    for ph in phases:
        for t in sets[0]:
            t.run(ph)
    torch.cuda.synchronize()
    ref = [[o.clone() for o in t.outputs()] for t in sets[0]]
    for t, t2 in zip(*sets):
        t.host_in = t.in_buf.cpu().pin_memory()
        t2.host_in = t.host_in
        for u in (t, t2):
            u.host_out = torch.full_like(u.out_buf, 0x5A, device="cpu").pin_memory()
    staged = bench.StagedE2E(sets, phases, dev)
    arrays = [a for t in sets[0] for a in t.inputs()]
    extra = staged.h2d - sum(a.numel() * a.element_size() for a in arrays)
    assert 0 <= extra < bench.ARENA_ALIGN * len(arrays), extra
    for ts in sets:   # poison: every input must come in, every output go out
        for t in ts:
            t.in_buf.fill_(0xA5)
            t.out_buf.fill_(0xC3)
    torch.cuda.synchronize()
    main = torch.cuda.current_stream()
    staged.fork(main)
    for _ in range(3):
        staged.step()
    staged.join(main)
    torch.cuda.synchronize()
    for ts in sets:
        for i, t in enumerate(ts):
            for j, (a, r) in enumerate(zip(t.outputs(), ref[i])):
                got = host_view(t, t.host_out, t.out_buf, a)
                assert torch.equal(got.view(torch.uint8), r.cpu().contiguous().view(torch.uint8)), (i, j)
