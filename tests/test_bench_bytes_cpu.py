"""CPU: the algorithmic bytes per element behind every GB/s figure and the
roofline numerator -- what each phase must move at minimum, counted from its
operands: x, y, g, gx at the element size; fp32 coefficients (and their
gradients) per element unless one set serves all rows; 0.5 byte of codes and
one scale byte per block; the NVFP4 alpha pass reads x once.  The bf16 /
sub-block-8 figures are the per-element table of the scope (fwd 4.625 /
4.75, bwd with gx 7.25 / 7.5, pack 3.156 / 3.3125, alpha +2)."""
import pytest

import bench


@pytest.mark.parametrize("fmt,fwd,bwd,pack", [("mxfp4", 4.625, 7.25, 3.15625), ("nvfp4", 4.75, 7.5, 3.3125)])
def test_bytes_per_element_bf16(fmt, fwd, bwd, pack):
    b = bench.bytes_per_elem(bench.Case(fmt=fmt), 2)
    assert b["fwd"] == pytest.approx(fwd) and b["bwd"] == pytest.approx(bwd) and b["pack"] == pytest.approx(pack)
    assert ("alpha" in b) == (fmt == "nvfp4")
    if fmt == "nvfp4":
        assert b["alpha"] == 2.0
    # the default step: alpha + fwd + bwd + pack = 17.5625 bytes per element
    if fmt == "nvfp4":
        assert sum(b.values()) == pytest.approx(17.5625)


def test_shared_rows_drop_the_coefficients():
    b = bench.bytes_per_elem(bench.Case(fmt="mxfp4", shared=True), 2)
    assert b["fwd"] == 4.0 and b["bwd"] == 6.0 and b["pack"] == pytest.approx(2.0 + 0.5 + 1 / 32)


def test_fp32_io_and_learned_scale_and_adamw():
    b = bench.bytes_per_elem(bench.Case(fmt="mxfp4"), 4)           # fp32 x, y, g, gx
    assert b["fwd"] == pytest.approx(8.625) and b["bwd"] == pytest.approx(13.25)
    s = bench.bytes_per_elem(bench.Case(fmt="nvfp4", sfp=True), 2)  # S^fp in, dL/dS^fp out: 4 / 16 each
    assert s["fwd"] == pytest.approx(4.75 + 0.25) and s["bwd"] == pytest.approx(7.5 + 0.5)
    a = bench.bytes_per_elem(bench.Case(fmt="nvfp4", adam=True), 2)
    # p, m, v in and out per learned value (0.75 B of coefficients per element), no gradient out
    assert a["bwd"] == pytest.approx(6.0 + 6 * 0.75)
