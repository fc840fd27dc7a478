"""CPU: the benchmark's input / output arenas -- the arrays a step copies
between host and device placed in one allocation, so that each tensor moves
with one copy per direction: the views keep values, shapes and dtypes, sit
on aligned offsets without overlap, and the copy spans cover exactly the
arrays asked for, neighbours merged."""
import types

import pytest
import torch

import bench


def make():
    g = torch.Generator().manual_seed(3)
    o = types.SimpleNamespace(
        x=torch.randn(37, 64, generator=g).to(torch.bfloat16),
        g=torch.randn(37, 64, generator=g).to(torch.bfloat16),
        crs=torch.rand(37, 4, generator=g),
        dgs=torch.rand(37, 8, generator=g),
        codes=torch.randint(0, 255, (37, 32), generator=g, dtype=torch.uint8),
        scales=torch.randint(0, 255, (37, 3), generator=g, dtype=torch.uint8))
    return o


def test_pack_arena_keeps_values_and_aligns():
    o = make()
    names = ("x", "g", "crs", "dgs", "codes", "scales")
    before = {n: getattr(o, n).clone() for n in names}
    buf = bench.pack_arena(o, names, "cpu")
    base = buf.data_ptr()
    ends = []
    for n in names:
        v = getattr(o, n)
        assert v.dtype == before[n].dtype and v.shape == before[n].shape, n
        assert torch.equal(v, before[n]), n
        assert v.is_contiguous(), n
        off = v.data_ptr() - base
        assert off % bench.ARENA_ALIGN == 0, n
        ends.append((off, off + v.numel() * v.element_size()))
    for (s0, e0), (s1, _) in zip(ends, ends[1:]):
        assert e0 <= s1   # in order, no overlap
    assert ends[-1][1] <= buf.numel()
    # a write through a view lands in the arena
    o.crs[5, 2] = 123.0
    assert torch.equal(buf[ends[2][0]:ends[2][1]].view(torch.float32).view(37, 4), o.crs)


def test_arena_spans_merge_neighbours_only():
    o = make()
    names = ("x", "g", "crs", "dgs", "codes", "scales")
    buf = bench.pack_arena(o, names, "cpu")
    span = lambda a: (a.data_ptr() - buf.data_ptr(), a.data_ptr() - buf.data_ptr() + a.numel() * a.element_size())
    # all: one span from the first array's start to the last array's end
    assert bench.arena_spans(buf, [getattr(o, n) for n in names]) == [(0, span(o.scales)[1])]
    # order of the list does not matter
    assert bench.arena_spans(buf, [o.g, o.x]) == [(0, span(o.g)[1])]
    # a hole (crs left out) splits the copy in two
    assert bench.arena_spans(buf, [o.x, o.g, o.dgs]) == [(0, span(o.g)[1]), span(o.dgs)]
    # one array alone: exactly its bytes, no padding
    assert bench.arena_spans(buf, [o.scales]) == [span(o.scales)]


def test_arena_spans_rejects_foreign_arrays():
    o = make()
    buf = bench.pack_arena(o, ("x", "g"), "cpu")
    with pytest.raises(ValueError):
        bench.arena_spans(buf, [torch.zeros(1 << 16)])


def test_arena_mirror_round_trip():
    """A host mirror of the arena's layout moved span by span gives back every
    array: the copy the end-to-end step makes, on CPU tensors."""
    o = make()
    names = ("x", "g", "crs", "dgs")
    buf = bench.pack_arena(o, names, "cpu")
    mirror = buf.clone()
    before = {n: getattr(o, n).clone() for n in names}
    buf.zero_()
    for s, e in bench.arena_spans(buf, [getattr(o, n) for n in names]):
        buf[s:e].copy_(mirror[s:e])
    for n in names:
        assert torch.equal(getattr(o, n), before[n]), n


def test_tensor_piece_views_rows():
    """A row piece of a benchmark tensor: every row array (and the optimizer
    moments) becomes the view of rows [r0, r1) of the same storage, the
    per-tensor arrays (alpha, scratch) stay shared, the element count
    follows the rows."""
    o = make()
    o.case = types.SimpleNamespace(shared=False, adam=True)
    o.alpha = torch.zeros(1)
    o.moments = {"crs": (torch.rand(37, 4), torch.rand(37, 4))}
    o.n = o.x.numel()
    p = bench.tensor_piece(o, 5, 12)
    for n in ("x", "g", "crs", "dgs", "codes", "scales"):
        v, whole = getattr(p, n), getattr(o, n)
        assert v.shape[0] == 7 and v.data_ptr() == whole[5].data_ptr(), n
        assert torch.equal(v, whole[5:12]), n
    m, vv = p.moments["crs"]
    assert m.data_ptr() == o.moments["crs"][0][5].data_ptr() and vv.shape == (7, 4)
    assert p.alpha is o.alpha and p.n == 7 * 64
    assert o.x.shape[0] == 37 and o.n == 37 * 64      # the whole tensor is unchanged
