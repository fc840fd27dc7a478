"""CPU oracle for the FOCUS FP4 fake-quantizer -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU legs of ``bench.py``
(the CPU baseline and ``--impl reference``) may import this package.  The product path (the CUDA library
under ``paper_2608_01847_gb300``) never imports it and shares no code with it.

The arithmetic lives in ``focus_oracle.c`` (plain scalar C, binary32 forward,
binary64 compensated gradient sums; see that file's header for the equations
it follows: FOCUS Sec. 3.1 Eq. 1-3, Sec. 3.2 Eq. 4-5, Sec. 3.3 Eq. 6-7,
Sec. 3.4 Eq. 8, Fig. 3(d)).  This module only builds it with gcc and marshals
numpy arrays into it.

Dtype codes: 0 = float32, 1 = bfloat16 (stored as uint16 bit patterns),
2 = IEEE binary16 (numpy float16).
Format codes: 0 = MXFP4 (block 32, E8M0), 1 = NVFP4 (block 16, E4M3 + alpha).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "focus_oracle.c")
_LIB = os.path.join(_HERE, "_build", "libfocus_oracle.so")

MXFP4, NVFP4 = 0, 1
F32, BF16, F16 = 0, 1, 2
STE_IDENTITY, STE_CLIPPED = 0, 1
MX_CEIL, MX_FLOOR = 0, 1

# -ffp-contract=off: no fused multiply-add may merge two binary32 roundings
# (GCC contracts by default on aarch64); no fast-math so IEEE semantics hold.
CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]


def build(force: bool = False) -> str:
    """Compile focus_oracle.c into ``_build/libfocus_oracle.so`` (idempotent)."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", *CFLAGS, _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB)
        i64, i32, p, f = ctypes.c_int64, ctypes.c_int, ctypes.c_void_p, ctypes.c_float
        L.focus_oracle_alpha.argtypes = [i32, i64, i64, i64, p, p]
        L.focus_oracle_fwd.argtypes = [i32, i32, i64, i64, i64, i32, i32, i32, i32,
                                       p, p, p, f, p, p, p, p]
        L.focus_oracle_bwd.argtypes = [i32, i32, i64, i64, i64, i32, i32, i32, i32, i32,
                                       p, p, p, f, p, p, p, p, p, p, p, p, p, p, p, p]
        L.focus_oracle_dequant.argtypes = [i32, i32, i64, i64, i32, p, p, f, p]
        L.focus_oracle_e2m1_code.argtypes = [f]
        L.focus_oracle_e2m1_value.argtypes = [i32]
        L.focus_oracle_e2m1_value.restype = f
        L.focus_oracle_e4m3_decode.argtypes = [ctypes.c_uint8]
        L.focus_oracle_e4m3_decode.restype = f
        L.focus_oracle_e4m3_encode.argtypes = [f]
        L.focus_oracle_e4m3_encode.restype = ctypes.c_uint8
        L.focus_oracle_e8m0_exponent.argtypes = [f, i32]
        L.focus_oracle_bf16_rne.argtypes = [f]
        L.focus_oracle_bf16_rne.restype = ctypes.c_uint16
        L.focus_oracle_e2m1_codes.argtypes = [p, i64, p]
        L.focus_oracle_e4m3_encodes.argtypes = [p, i64, p]
        L.focus_oracle_e8m0_exponents.argtypes = [p, i64, i32, p]
        L.focus_oracle_bf16_rnes.argtypes = [p, i64, p]
        L.focus_oracle_f16_rnes.argtypes = [p, i64, p]
        L.focus_oracle_f16_decodes.argtypes = [p, i64, p]
        _lib = L
    return _lib


class OracleError(RuntimeError):
    pass


def _ptr(a):
    return None if a is None else a.ctypes.data


def _check(rc):
    if rc == -1:
        raise OracleError("oracle: invalid argument")
    if rc == -2:
        raise OracleError("oracle: precondition violated (non-finite input or coefficient <= 0)")
    if rc != 0:
        raise OracleError(f"oracle: status {rc}")


def _dtype_code(x: np.ndarray) -> int:
    if x.dtype == np.float32:
        return F32
    if x.dtype == np.uint16:
        return BF16
    if x.dtype == np.float16:
        return F16
    raise TypeError("oracle inputs are float32, float16 or uint16 (bfloat16 bit patterns)")


def _c32(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.float32)


def default_block(fmt: int) -> int:
    return 32 if fmt == MXFP4 else 16


# --------------------------------------------------------------------------
# codecs, one value or a vector at a time
# --------------------------------------------------------------------------
def e2m1_codes(u) -> np.ndarray:
    u = np.ascontiguousarray(u, dtype=np.float32)
    out = np.empty(u.shape, np.uint8)
    lib().focus_oracle_e2m1_codes(_ptr(u), u.size, _ptr(out))
    return out


def e2m1_value(code: int) -> float:
    return lib().focus_oracle_e2m1_value(int(code))


def e4m3_decode(byte: int) -> float:
    return lib().focus_oracle_e4m3_decode(int(byte))


def e4m3_encode(r) -> np.ndarray:
    r = np.ascontiguousarray(r, dtype=np.float32)
    out = np.empty(r.shape, np.uint8)
    lib().focus_oracle_e4m3_encodes(_ptr(r), r.size, _ptr(out))
    return out


def e8m0_exponent(m, rule: int = MX_CEIL) -> np.ndarray:
    m = np.ascontiguousarray(m, dtype=np.float32)
    out = np.empty(m.shape, np.int32)
    lib().focus_oracle_e8m0_exponents(_ptr(m), m.size, int(rule), _ptr(out))
    return out


def bf16_rne(f) -> np.ndarray:
    f = np.ascontiguousarray(f, dtype=np.float32)
    out = np.empty(f.shape, np.uint16)
    lib().focus_oracle_bf16_rnes(_ptr(f), f.size, _ptr(out))
    return out


def f16_rne(f) -> np.ndarray:
    """binary32 -> binary16 bit patterns (round to nearest even)."""
    f = np.ascontiguousarray(f, dtype=np.float32)
    out = np.empty(f.shape, np.uint16)
    lib().focus_oracle_f16_rnes(_ptr(f), f.size, _ptr(out))
    return out


def f16_decode(h) -> np.ndarray:
    """binary16 bit patterns -> binary32 values."""
    h = np.ascontiguousarray(h, dtype=np.uint16)
    out = np.empty(h.shape, np.float32)
    lib().focus_oracle_f16_decodes(_ptr(h), h.size, _ptr(out))
    return out


# --------------------------------------------------------------------------
# tensor-level entry points
# --------------------------------------------------------------------------
def alpha(x: np.ndarray) -> float:
    """NVFP4 per-tensor scale alpha = fl(max|x| / 2688) (Eq. 2)."""
    x = np.ascontiguousarray(x)
    rows, cols = x.shape
    out = np.zeros(1, np.float32)
    _check(lib().focus_oracle_alpha(_dtype_code(x), rows, cols, cols, _ptr(x), _ptr(out)))
    return float(out[0])


def fwd(x, fmt, crs=None, dgs=None, alpha=0.0, block=None, sub=8, shared=False,
        mx_rule=MX_CEIL, want_y=True, want_scales=True, want_codes=False, sfp=None):
    """Fake-quant forward / export (Eq. 1-8, Fig. 3(d)).

    x: [rows, cols] float32 or uint16 (bf16 bits), contiguous.
    Returns dict with 'y' (same dtype as x), 'scales' uint8 [rows, cols/block],
    'codes' uint8 [rows, cols/2] (as requested).  sfp: optional learnable
    full-precision scales [rows, cols/block] (Eq. 4) replacing the absmax scale."""
    x = np.ascontiguousarray(x)
    rows, cols = x.shape
    block = block or default_block(fmt)
    crs, dgs, sfp = _c32(crs), _c32(dgs), _c32(sfp)
    out = {}
    y = np.empty_like(x) if want_y else None
    sc = np.zeros((rows, cols // block), np.uint8) if want_scales else None
    cd = np.zeros((rows, cols // 2), np.uint8) if want_codes else None
    _check(lib().focus_oracle_fwd(fmt, _dtype_code(x), rows, cols, cols, block, sub,
                                  int(bool(shared)), mx_rule, _ptr(x), _ptr(crs), _ptr(dgs),
                                  float(alpha), _ptr(sfp), _ptr(y), _ptr(sc), _ptr(cd)))
    if want_y:
        out["y"] = y
    if want_scales:
        out["scales"] = sc
    if want_codes:
        out["codes"] = cd
    return out


def bwd(x, g, fmt, crs=None, dgs=None, alpha=0.0, block=None, sub=8, shared=False,
        ste=STE_IDENTITY, mx_rule=MX_CEIL, want_gx=True, want_gcrs=True, want_gdgs=True,
        want_abs=False, want_f64=False, sfp=None, want_gsfp=False):
    """STE backward (Sec. 3.2; Eq. 6-8): input gradient and coefficient gradients.

    Returns dict with 'gx' (dtype of x), 'gcrs' float32 [rows or 1, cols/block],
    'gdgs' float32 [rows or 1, cols/sub], with want_abs the binary64
    term-magnitude sums 'gcrs_abs', 'gdgs_abs', and with want_f64 the
    gradients before their final rounding, 'gcrs64', 'gdgs64' (binary64).
    sfp: optional learnable scales (Eq. 4); want_gsfp adds 'gsfp' float32
    [rows, cols/block] (and 'gsfp_abs' with want_abs, 'gsfp64' with
    want_f64)."""
    x = np.ascontiguousarray(x)
    g = np.ascontiguousarray(g)
    assert g.dtype == x.dtype and g.shape == x.shape
    rows, cols = x.shape
    block = block or default_block(fmt)
    crs, dgs, sfp = _c32(crs), _c32(dgs), _c32(sfp)
    crow = 1 if shared else rows
    gs = np.zeros((rows, cols // block), np.float32) if want_gsfp else None
    gsa = np.zeros((rows, cols // block), np.float64) if (want_gsfp and want_abs) else None
    gx = np.empty_like(x) if want_gx else None
    gc = np.zeros((crow, cols // block), np.float32) if want_gcrs else None
    gd = np.zeros((crow, cols // sub), np.float32) if want_gdgs else None
    gca = np.zeros((crow, cols // block), np.float64) if (want_abs and want_gcrs) else None
    gda = np.zeros((crow, cols // sub), np.float64) if (want_abs and want_gdgs) else None
    gc64 = np.zeros((crow, cols // block), np.float64) if want_f64 else None
    gd64 = np.zeros((crow, cols // sub), np.float64) if want_f64 else None
    gs64 = np.zeros((rows, cols // block), np.float64) if (want_f64 and want_gsfp) else None
    _check(lib().focus_oracle_bwd(fmt, _dtype_code(x), rows, cols, cols, block, sub,
                                  int(bool(shared)), ste, mx_rule, _ptr(x), _ptr(crs),
                                  _ptr(dgs), float(alpha), _ptr(sfp), _ptr(g), _ptr(gx), _ptr(gc),
                                  _ptr(gd), _ptr(gs), _ptr(gca), _ptr(gda), _ptr(gsa), _ptr(gc64),
                                  _ptr(gd64), _ptr(gs64)))
    out = {}
    if want_gx:
        out["gx"] = gx
    if want_gcrs:
        out["gcrs"] = gc
        if want_abs:
            out["gcrs_abs"] = gca
    if want_gdgs:
        out["gdgs"] = gd
        if want_abs:
            out["gdgs_abs"] = gda
    if want_f64:
        out["gcrs64"], out["gdgs64"] = gc64, gd64
    if want_gsfp:
        out["gsfp"] = gs
        if want_abs:
            out["gsfp_abs"] = gsa
        if want_f64:
            out["gsfp64"] = gs64
    return out


# --------------------------------------------------------------------------
# AdamW (the optimizer of the paper's calibration, Sec. 4.1 "Implementation
# Details": AdamW with a constant learning rate, separate rates for the
# block scale and the relaxation coefficients; weights frozen, Sec. 4.4)
# --------------------------------------------------------------------------
def adamw(p, grad, m, v, lr, beta1, beta2, eps, weight_decay, step):
    """One AdamW step in binary64: decoupled weight decay (Loshchilov &
    Hutter), written with PyTorch's conventions (the paper's framework):

        p <- p * (1 - lr * weight_decay)
        m <- beta1 * m + (1 - beta1) * grad
        v <- beta2 * v + (1 - beta2) * grad^2
        p <- p - lr * (m / (1 - beta1^t)) / (sqrt(v / (1 - beta2^t)) + eps)

    `step` is t >= 1, the number of this update.  Hyper-parameters are taken
    as the binary32 values a caller passes to the device.  Returns the new
    (p, m, v) as float64 arrays; the inputs are not modified."""
    f = lambda a: float(np.float32(a))
    lr, beta1, beta2, eps, weight_decay = f(lr), f(beta1), f(beta2), f(eps), f(weight_decay)
    t = int(step)
    if t < 1:
        raise OracleError("AdamW step counts from 1")
    p = np.asarray(p, np.float64) * (1.0 - lr * weight_decay)
    g = np.asarray(grad, np.float64)
    m = beta1 * np.asarray(m, np.float64) + (1.0 - beta1) * g
    v = beta2 * np.asarray(v, np.float64) + (1.0 - beta2) * g * g
    mhat = m / (1.0 - beta1 ** t)
    vhat = v / (1.0 - beta2 ** t)
    p = p - lr * mhat / (np.sqrt(vhat) + eps)
    return p, m, v


def bwd_adamw(x, g, fmt, params, moments, hp, step, alpha=0.0, sub=8, shared=False,
              ste=STE_IDENTITY, mx_rule=MX_CEIL, want_gx=True):
    """The STE backward followed by one AdamW step on every learnable array.

    params: dict with any of 'crs', 'dgs', 'sfp' (float32 arrays; missing =
    not learned: coefficient 1 / absmax scale).  moments: dict name ->
    (m, v).  hp: dict lr_coef, lr_scale, beta1, beta2, eps, weight_decay
    (S^fp takes lr_scale, c_i and c_i^k take lr_coef).  The gradients are the
    oracle's binary64 sums before rounding.  Returns dict with 'gx' (if
    wanted), per learned name: 'grad' (float64), 'grad_abs', and the new
    'p', 'm', 'v' (float64)."""
    sfp = params.get("sfp")
    r = bwd(x, g, fmt, crs=params.get("crs"), dgs=params.get("dgs"), alpha=alpha, sub=sub,
            shared=shared, ste=ste, mx_rule=mx_rule, want_gx=want_gx, want_abs=True,
            want_f64=True, sfp=sfp, want_gsfp=sfp is not None)
    out = {"gx": r["gx"]} if want_gx else {}
    grads = {"crs": ("gcrs64", "gcrs_abs"), "dgs": ("gdgs64", "gdgs_abs"),
             "sfp": ("gsfp64", "gsfp_abs")}
    for name, (gk, ak) in grads.items():
        if params.get(name) is None:
            continue
        lr = hp["lr_scale"] if name == "sfp" else hp["lr_coef"]
        m, v = moments[name]
        pn, mn, vn = adamw(params[name], r[gk], m, v, lr, hp["beta1"], hp["beta2"], hp["eps"],
                           hp["weight_decay"], step)
        out[name] = {"grad": r[gk], "grad_abs": r[ak], "p": pn, "m": mn, "v": vn}
    return out


def dequant(codes, scales, fmt, alpha=0.0, block=None, dtype=F32):
    """Rebuild values from an export (codes + scale bytes [+ alpha])."""
    codes = np.ascontiguousarray(codes, dtype=np.uint8)
    scales = np.ascontiguousarray(scales, dtype=np.uint8)
    rows = codes.shape[0]
    cols = codes.shape[1] * 2
    block = block or default_block(fmt)
    y = np.empty((rows, cols), {F32: np.float32, BF16: np.uint16, F16: np.float16}[dtype])
    _check(lib().focus_oracle_dequant(fmt, dtype, rows, cols, block, _ptr(codes),
                                      _ptr(scales), float(alpha), _ptr(y)))
    return y


# --------------------------------------------------------------------------
# Deployment view: the exported FP4 operands of a block-scaled tensor-core
# GEMM (the hardware path the paper's "no inference overhead" rests on,
# Sec. 1 and Sec. 3.1; the export of Fig. 3(d))
# --------------------------------------------------------------------------
def mma_scale_tiles(scales):
    """Row-major scale bytes [R, C] -> the block-scaled MMA scale-factor
    layout: tiles of 128 rows x 4 columns (512 bytes) over the matrix padded
    with zero bytes to multiples of 128 x 4, tile (i, j) at (i * ceil(C/4) + j)
    * 512, row r / column c of a tile at (r % 32) * 16 + (r // 32) * 4 + c.
    Written out element by element."""
    scales = np.asarray(scales, np.uint8)
    R, C = scales.shape
    tr, tc = (R + 127) // 128, (C + 3) // 4
    out = np.zeros(tr * tc * 512, np.uint8)
    for r in range(R):
        for c in range(C):
            i, j = r // 128, c // 4
            rr, cc = r % 128, c % 4
            out[(i * tc + j) * 512 + (rr % 32) * 16 + (rr // 32) * 4 + cc] = scales[r, c]
    return out


def fp4_gemm(codes_a, scales_a, codes_b, scales_b, fmt, alpha_a=1.0, alpha_b=1.0, block=None):
    """D[m, n] = sum_k A[m, k] B[n, k] in binary64 for exported FP4 operands
    (codes [rows, K/2], element 2t in the low nibble; row-major scale bytes
    [rows, K/block]): A[m, k] = E2M1(code) * S(m, k / block) with S = 2^(byte
    - 127) for MXFP4 and E4M3(byte) for NVFP4, and D scaled by alpha_a *
    alpha_b for NVFP4 (the per-tensor scales, Eq. 2).  Dequantization
    through the oracle's own decoders; the contraction is numpy's matmul."""
    block = block or default_block(fmt)

    def dense(codes, scales):
        codes = np.asarray(codes, np.uint8)
        rows, half = codes.shape
        k = half * 2
        nib = np.empty((rows, k), np.int64)
        nib[:, 0::2] = codes & 15
        nib[:, 1::2] = codes >> 4
        val = np.array([e2m1_value(c) for c in range(16)], np.float64)[nib]
        sb = np.asarray(scales, np.uint8)
        if fmt == MXFP4:
            s = np.ldexp(1.0, sb.astype(np.int64) - 127)
        else:
            s = np.array([e4m3_decode(b) for b in range(256)], np.float64)[sb]
        return val * np.repeat(s, block, axis=1)

    d = dense(codes_a, scales_a) @ dense(codes_b, scales_b).T
    if fmt == NVFP4:
        d = d * (float(np.float32(alpha_a)) * float(np.float32(alpha_b)))
    return d
