"""GPU parity of the tensor-core FP4 GEMM over focus_pack_mma exports.

Both operands are fake-quantized and exported on the GPU; the export must
equal the oracle's bit for bit, and D must match the oracle's binary64
contraction of the oracle's own export (oracle.fp4_gemm) within the fp32
accumulation bound

    |D - D_ref| <= (K / 16 + 8) * 2^-23 * sum_k |A[m, k] B[n, k]|  (+ 2^-23 |D_ref| for alpha)

(every product is exact in fp32; each accumulation step rounds at most once
by 2^-23 relative to the running magnitude).  A wrong scale, element or
block shifts D by far more."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_01847_gb300 import build as B
from paper_2608_01847_gb300 import focus as F
from paper_2608_01847_gb300 import workloads as W
from gpu_helpers import assert_bits_equal, assert_gemm_close, dev, gemm_bound, host

pytestmark = pytest.mark.gpu

FMT = {"mx": O.MXFP4, "nv": O.NVFP4}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    F.lib()


def operand(rows, k, seed, kind):
    """Seeded host operand: an activation (N(0,1), a few outlier channels)
    or a weight (Student-t(5) x 0.02), bf16."""
    if kind == "act":
        w = W.Workload("a", (W.TensorSpec("a", rows, k),), "bf16", ("nvfp4",), "activation", None, 1.0,
                       "channels", 4, 30.0, (0.9, 1.1), seed)
    else:
        w = W.Workload("w", (W.TensorSpec("w", rows, k),), "bf16", ("nvfp4",), "weight", 5.0, 0.02,
                       "entries", 0.001, 20.0, (0.9, 1.1), seed)
    x, _ = W.host_tensor(w, 0)
    return w, x


def export_both(x, fmt, crs):
    """GPU export (checked against the oracle's) and the oracle's export."""
    a = O.alpha(x) if fmt == O.NVFP4 else 0.0
    a_dev = torch.tensor([a], dtype=torch.float32, device="cuda")
    cd = dev(crs) if crs is not None else None
    codes, tiles = F.focus_pack_mma(dev(x), fmt, cd, None, a_dev)
    ref = O.fwd(x, fmt, crs=crs, alpha=a, want_y=False, want_codes=True)
    torch.cuda.synchronize()
    assert_bits_equal(host(codes), ref["codes"], "codes")
    assert_bits_equal(host(tiles), O.mma_scale_tiles(ref["scales"]), "scale tiles")
    return codes, tiles, a_dev, ref, a


def check_gemm(fmt, M, N, K, seed=0, crs=True):
    block = 32 if fmt == O.MXFP4 else 16
    wa, xa = operand(M, K, seed, "act")
    wb, xb = operand(N, K, seed + 1, "weight")
    ca = W.draw_coefs(wa, M * K // block, seed + 2).reshape(M, -1) if crs else None
    cb = W.draw_coefs(wb, N * K // block, seed + 3).reshape(N, -1) if crs else None
    ac, at, aa_dev, ra, aa = export_both(xa, fmt, ca)
    bc, bt, ab_dev, rb, ab = export_both(xb, fmt, cb)
    flag = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = F.focus_fp4_gemm(fmt, ac, at, bc, bt, aa_dev, ab_dev, timeout_flag=flag)
    torch.cuda.synchronize()
    assert int(flag.item()) == 0, "MMA wait gave up"
    ref = O.fp4_gemm(ra["codes"], ra["scales"], rb["codes"], rb["scales"], fmt, aa, ab)
    mag = O.fp4_gemm(ra["codes"] & 0x77, ra["scales"], rb["codes"] & 0x77, rb["scales"], fmt, aa, ab)
    assert_gemm_close(host(d), ref, mag, K)
    return d, ref


@pytest.mark.parametrize("fmt", ["mx", "nv"])
@pytest.mark.parametrize("M,N,K", [(128, 128, 64), (128, 128, 256), (256, 384, 512), (200, 130, 320),
                                   (1, 1, 64), (129, 257, 1024), (384, 128, 2560),
                                   (200, 132, 320), (130, 260, 512), (300, 520, 256),
                                   # several 256 x 256 pair tiles both ways; the last tile row and
                                   # column leave the second CTA of the pair without rows of A / B;
                                   # K of 13 steps ends in a one-step chunk
                                   (513, 770, 832),
                                   # K of 32, 96, 160: a last K step of 32 elements (zero codes
                                   # past K, the export's zeroed scale padding)
                                   (130, 260, 32), (129, 257, 96), (300, 520, 160)])
def test_fp4_gemm_parity(fmt, M, N, K):
    check_gemm(FMT[fmt], M, N, K, seed=M + N + K)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_fp4_gemm_without_coefficients(fmt):
    """c = 1: the export is plain RTN MXFP4 / NVFP4."""
    check_gemm(FMT[fmt], 256, 256, 512, seed=5, crs=False)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_fp4_gemm_degenerate_sizes(fmt):
    f = FMT[fmt]
    z = torch.zeros(16, dtype=torch.uint8, device="cuda")
    one = torch.ones(1, dtype=torch.float32, device="cuda")
    d = F.focus_fp4_gemm(f, torch.zeros((3, 0), dtype=torch.uint8, device="cuda"), z,
                         torch.zeros((5, 0), dtype=torch.uint8, device="cuda"), z, one, one,
                         d=torch.full((3, 5), 7.0, device="cuda"))
    torch.cuda.synchronize()
    assert torch.equal(d, torch.zeros_like(d))                       # K = 0: empty sums
    with pytest.raises(F.FocusError):   # K = 16: code rows off 16-byte boundaries, refused before launch
        F.focus_fp4_gemm(f, torch.zeros((4, 8), dtype=torch.uint8, device="cuda"), z,
                         torch.zeros((4, 8), dtype=torch.uint8, device="cuda"), z, one, one)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_export_read_by_library_gemm(fmt):
    """The export is what NVIDIA's own block-scaled FP4 GEMM (cuBLASLt,
    through torch._scaled_mm) reads: same product within bf16 output
    rounding.  Skipped where the installed torch has no FP4 path."""
    f = FMT[fmt]
    if not hasattr(torch, "float4_e2m1fn_x2"):
        pytest.skip("torch without float4_e2m1fn_x2")
    M, N, K = 256, 256, 512
    wa, xa = operand(M, K, 11, "act")
    wb, xb = operand(N, K, 12, "weight")
    ac, at, aa_dev, ra, aa = export_both(xa, f, None)
    bc, bt, ab_dev, rb, ab = export_both(xb, f, None)
    sdt = torch.float8_e8m0fnu if f == O.MXFP4 else torch.float8_e4m3fn
    try:
        out = torch._scaled_mm(ac.view(torch.float4_e2m1fn_x2), bc.view(torch.float4_e2m1fn_x2).t(),
                               at.view(sdt), bt.view(sdt), out_dtype=torch.bfloat16)
        torch.cuda.synchronize()
    except (RuntimeError, TypeError, NotImplementedError) as e:
        pytest.skip(f"library FP4 GEMM unavailable here: {str(e).splitlines()[0][:120]}")
    lib = out.float().cpu().numpy().astype(np.float64)
    if f == O.NVFP4:
        lib = lib * (float(np.float32(aa)) * float(np.float32(ab)))
    ref = O.fp4_gemm(ra["codes"], ra["scales"], rb["codes"], rb["scales"], f, aa, ab)
    mag = O.fp4_gemm(ra["codes"] & 0x77, ra["scales"], rb["codes"] & 0x77, rb["scales"], f, aa, ab)
    assert np.all(np.abs(lib - ref) <= 2.0 ** -7 * np.abs(ref) + 2.0 ** -18 * mag)


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_fp4_gemm_bf16_output(fmt):
    """bf16 output: the fp32 result rounded to nearest even (within one bf16
    rounding of the fp32 bound), and odd row pitches take the scalar path."""
    f = FMT[fmt]
    M, N, K = 192, 200, 768
    wa, xa = operand(M, K, 31, "act")
    wb, xb = operand(N, K, 32, "weight")
    ac, at, aa_dev, ra, aa = export_both(xa, f, None)
    bc, bt, ab_dev, rb, ab = export_both(xb, f, None)
    d32 = F.focus_fp4_gemm(f, ac, at, bc, bt, aa_dev, ab_dev)
    d16 = F.focus_fp4_gemm(f, ac, at, bc, bt, aa_dev, ab_dev, out_dtype=torch.bfloat16)
    wide = torch.zeros((M, N + 3), dtype=torch.bfloat16, device="cuda")
    F.focus_fp4_gemm(f, ac, at, bc, bt, aa_dev, ab_dev, d=wide[:, :N])
    torch.cuda.synchronize()
    assert torch.equal(d16, d32.to(torch.bfloat16))
    assert torch.equal(wide[:, :N], d16)
    assert torch.count_nonzero(wide[:, N:]) == 0


@pytest.mark.parametrize("fmt", ["mx", "nv"])
def test_fp4_gemm_full_size_sampled(fmt):
    """The benchmark's largest Qwen3-4B GEMM at full size (8192 tokens x
    gate_proj [9728, 2560]: 1216 tiles of 256 x 256 on 76 persistent CTA
    pairs, so every barrier of the ring, of the scale sets and of the
    accumulator wraps many times), with fp32
    and with bf16 output: D on 32 sampled rows x 32 sampled columns (first,
    last, random) against the oracle's contraction of the oracle's export of
    those rows, whose codes and scale bytes also match the GPU export."""
    f = FMT[fmt]
    M, N, K = 8192, 9728, 2560
    block = 32 if f == O.MXFP4 else 16
    _, xa = operand(M, K, 21, "act")
    _, xb = operand(N, K, 22, "weight")
    aa = O.alpha(xa) if f == O.NVFP4 else 0.0
    ab = O.alpha(xb) if f == O.NVFP4 else 0.0
    da, db = dev(xa), dev(xb)
    aa_dev = torch.tensor([aa], dtype=torch.float32, device="cuda")
    ab_dev = torch.tensor([ab], dtype=torch.float32, device="cuda")
    ac, at = F.focus_pack_mma(da, f, alpha=aa_dev)
    bc, bt = F.focus_pack_mma(db, f, alpha=ab_dev)
    # the same exports, row-major scale bytes (to compare sampled rows)
    ac2, as2 = F.focus_pack(da, f, alpha=aa_dev)
    bc2, bs2 = F.focus_pack(db, f, alpha=ab_dev)
    flag = torch.zeros(1, dtype=torch.int32, device="cuda")
    d32 = F.focus_fp4_gemm(f, ac, at, bc, bt, aa_dev, ab_dev, timeout_flag=flag)
    d16 = F.focus_fp4_gemm(f, ac, at, bc, bt, aa_dev, ab_dev, out_dtype=torch.bfloat16, timeout_flag=flag)
    torch.cuda.synchronize()
    assert int(flag.item()) == 0, "MMA wait gave up"
    rng = np.random.default_rng(7 + f)
    ma = np.unique(np.concatenate([[0, M - 1], rng.choice(M, 30, replace=False)]))
    nb = np.unique(np.concatenate([[0, N - 1], rng.choice(N, 30, replace=False)]))
    ra = O.fwd(xa[ma], f, alpha=aa, want_y=False, want_codes=True)
    rb = O.fwd(xb[nb], f, alpha=ab, want_y=False, want_codes=True)
    assert_bits_equal(host(ac2)[ma], ra["codes"], "A codes")
    assert_bits_equal(host(as2)[ma], ra["scales"], "A scale bytes")
    assert_bits_equal(host(bc2)[nb], rb["codes"], "B codes")
    assert_bits_equal(host(bs2)[nb], rb["scales"], "B scale bytes")
    assert torch.equal(ac, ac2) and torch.equal(bc, bc2)
    ref = O.fp4_gemm(ra["codes"], ra["scales"], rb["codes"], rb["scales"], f, aa, ab)
    mag = O.fp4_gemm(ra["codes"] & 0x77, ra["scales"], rb["codes"] & 0x77, rb["scales"], f, aa, ab)
    bound = gemm_bound(K, mag, ref)
    ia, ib = torch.from_numpy(ma).cuda(), torch.from_numpy(nb).cuda()
    got32 = host(d32[ia][:, ib]).astype(np.float64)
    got16 = host(d16[ia][:, ib].float()).astype(np.float64)
    assert np.all(np.abs(got32 - ref) <= bound), "fp32 output"
    # bf16 output: the fp32 result rounded once more (half an ulp of bf16)
    assert np.all(np.abs(got16 - ref) <= bound + 2.0 ** -8 * (np.abs(ref) + bound)), "bf16 output"
