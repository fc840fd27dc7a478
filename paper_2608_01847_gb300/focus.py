"""Python binding of libfocus_fq.so -- argument marshalling only.

Every function here has the name of the C entry point it calls (see
include/focus_fq.h for the semantics, layouts and error codes) and does no
arithmetic of its own: it turns torch CUDA tensors into device pointers, the
current torch stream into a cudaStream_t, allocates missing outputs with
torch (PyTorch is the device-memory provider), and raises FocusError on a
non-zero status.  There is no fallback: without the built library every call
raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libfocus_fq.so")

FOCUS_MXFP4, FOCUS_NVFP4 = 0, 1
FOCUS_F32, FOCUS_BF16, FOCUS_F16 = 0, 1, 2
FOCUS_STE_IDENTITY, FOCUS_STE_CLIPPED = 0, 1
FOCUS_MX_CEIL, FOCUS_MX_FLOOR = 0, 1
FOCUS_WS_ALPHA, FOCUS_WS_BWD = 0, 1

STATUS = {0: "FOCUS_OK", -1: "FOCUS_ERR_INVALID_ARG", -2: "FOCUS_ERR_UNSUPPORTED",
          -3: "FOCUS_ERR_MISALIGNED", -4: "FOCUS_ERR_WORKSPACE", -5: "FOCUS_ERR_CUDA"}

ENTRY_POINTS = ("focus_nvfp4_alpha", "focus_nvfp4_alpha_noalloc", "focus_fq_fwd", "focus_fq_bwd",
                "focus_fq_bwd_adamw", "focus_pack", "focus_pack_mma", "focus_mma_scale_bytes",
                "focus_fp4_gemm", "focus_nvfp4_alpha_group", "focus_group_workspace_bytes",
                "focus_fq_fwd_group", "focus_fq_bwd_group", "focus_pack_group",
                "focus_workspace_bytes", "focus_status_string", "focus_version")


class FocusError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = _lib.focus_status_string(status).decode() if _lib is not None else str(status)
        super().__init__(f"{where}: {STATUS.get(status, status)} ({msg})")


class focus_desc_t(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int64), ("cols", ctypes.c_int64), ("ld", ctypes.c_int64),
                ("dtype", ctypes.c_int32), ("fmt", ctypes.c_int32), ("block", ctypes.c_int32),
                ("sub_block", ctypes.c_int32), ("coef_shared_rows", ctypes.c_int32),
                ("ste", ctypes.c_int32), ("mx_rule", ctypes.c_int32)]


class focus_tensor_t(ctypes.Structure):
    _fields_ = [("desc", focus_desc_t)] + [(n, ctypes.c_void_p) for n in (
        "x", "g", "y", "gx", "crs", "dgs", "alpha", "sfp", "gcrs", "gdgs", "gsfp", "codes", "scale_bytes")]


FOCUS_MAX_GROUP = 16


class focus_adamw_t(ctypes.Structure):
    _fields_ = [("lr_coef", ctypes.c_float), ("lr_scale", ctypes.c_float),
                ("beta1", ctypes.c_float), ("beta2", ctypes.c_float), ("eps", ctypes.c_float),
                ("weight_decay", ctypes.c_float)]


class focus_adamw_state_t(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("m_crs", "v_crs", "m_dgs", "v_dgs", "m_sfp", "v_sfp")]


_lib: Optional[ctypes.CDLL] = None


def lib() -> ctypes.CDLL:
    """Load the in-tree library (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(LIB_PATH)
        P, D, SZ = ctypes.c_void_p, ctypes.POINTER(focus_desc_t), ctypes.c_size_t
        L.focus_nvfp4_alpha.argtypes = [D, P, P, P, SZ, P]
        L.focus_nvfp4_alpha_noalloc.argtypes = [D, P, P, P]
        L.focus_fq_fwd.argtypes = [D, P, P, P, P, P, P, P, P]
        L.focus_fq_bwd.argtypes = [D, P, P, P, P, P, P, P, P, P, P, P, SZ, P]
        L.focus_fq_bwd_adamw.argtypes = [D, P, P, P, P, P, P, P, ctypes.POINTER(focus_adamw_t),
                                         ctypes.POINTER(focus_adamw_state_t), P, P, P, P, P, SZ, P]
        L.focus_pack.argtypes = [D, P, P, P, P, P, P, P, P]
        L.focus_pack_mma.argtypes = [D, P, P, P, P, P, P, P, P]
        L.focus_mma_scale_bytes.argtypes = [D]
        L.focus_mma_scale_bytes.restype = SZ
        I32, I64 = ctypes.c_int32, ctypes.c_int64
        L.focus_fp4_gemm.argtypes = [I32, I64, I64, I64, P, P, P, P, P, P, P, I32, I64, P, P]
        T = ctypes.POINTER(focus_tensor_t)
        L.focus_nvfp4_alpha_group.argtypes = [T, ctypes.c_int, P, P, SZ, P]
        L.focus_group_workspace_bytes.argtypes = [T, ctypes.c_int]
        L.focus_group_workspace_bytes.restype = SZ
        for n in ("focus_fq_fwd_group", "focus_fq_bwd_group", "focus_pack_group"):
            getattr(L, n).argtypes = [T, ctypes.c_int, P]
            getattr(L, n).restype = ctypes.c_int
        L.focus_nvfp4_alpha_group.restype = ctypes.c_int
        L.focus_workspace_bytes.argtypes = [D, ctypes.c_int]
        L.focus_workspace_bytes.restype = SZ
        L.focus_status_string.argtypes = [ctypes.c_int]
        L.focus_status_string.restype = ctypes.c_char_p
        L.focus_version.restype = ctypes.c_int
        for n in ("focus_nvfp4_alpha", "focus_nvfp4_alpha_noalloc", "focus_fq_fwd", "focus_fq_bwd",
                  "focus_fq_bwd_adamw", "focus_pack", "focus_pack_mma", "focus_fp4_gemm"):
            getattr(L, n).restype = ctypes.c_int
        _lib = L
    return _lib


def block_of(fmt: int) -> int:
    return 32 if fmt == FOCUS_MXFP4 else 16


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return FOCUS_F32
    if t.dtype == torch.bfloat16:
        return FOCUS_BF16
    if t.dtype == torch.float16:
        return FOCUS_F16
    raise TypeError(f"unsupported dtype {t.dtype} (float32, bfloat16 or float16)")


def make_desc(x: torch.Tensor, fmt: int = FOCUS_MXFP4, sub_block: int = 8, shared: bool = False,
              ste: int = FOCUS_STE_IDENTITY, mx_rule: int = FOCUS_MX_CEIL,
              block: Optional[int] = None) -> focus_desc_t:
    if x.dim() != 2 or (x.shape[0] > 1 and x.shape[1] > 0 and x.stride(1) != 1):
        raise ValueError("x must be a 2-D tensor with unit stride along columns")
    rows, cols = x.shape
    ld = x.stride(0) if rows > 1 else cols
    return focus_desc_t(rows, cols, ld, _dtype_code(x), fmt, block or block_of(fmt),
                        sub_block, int(bool(shared)), ste, mx_rule)


def _like_x(x: torch.Tensor) -> torch.Tensor:
    """An output with x's exact shape and row pitch (the ABI's [rows, ld] layout)."""
    return torch.empty_strided(tuple(x.shape), tuple(x.stride()), dtype=x.dtype, device=x.device)


def _same_layout(x: torch.Tensor, t: Optional[torch.Tensor], name: str):
    if t is None:
        return
    if t.shape != x.shape or t.dtype != x.dtype or t.device != x.device or (
            x.shape[0] > 1 and t.stride() != x.stride()):
        raise ValueError(f"{name} must have x's shape, dtype, device and strides "
                         f"(got {tuple(t.shape)} {t.dtype} stride {t.stride()}, "
                         f"x is {tuple(x.shape)} {x.dtype} stride {x.stride()})")


def _dense(t: Optional[torch.Tensor], n: int, dtype, name: str):
    if t is None:
        return
    if not t.is_contiguous() or t.numel() != n or t.dtype != dtype:
        raise ValueError(f"{name} must be a contiguous {dtype} tensor of {n} elements")


def _p(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(device) -> ctypes.c_void_p:
    return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _check(rc: int, where: str):
    if rc != 0:
        raise FocusError(rc, where)


def _check_coefs(x, fmt, sub_block, shared, c, d):
    rows, cols = x.shape
    crow = 1 if shared else rows
    _dense(c, crow * (cols // block_of(fmt)), torch.float32, "block coefficients")
    _dense(d, crow * (cols // sub_block) if sub_block else 0, torch.float32,
           "sub-block coefficients")


def focus_workspace_bytes(desc: focus_desc_t, which: int) -> int:
    return int(lib().focus_workspace_bytes(ctypes.byref(desc), which))


def _workspace(desc, which, device, ws):
    n = focus_workspace_bytes(desc, which)
    if ws is None:
        ws = torch.empty(max(n, 16), dtype=torch.uint8, device=device)
    return ws, ws.numel() * ws.element_size()


def focus_nvfp4_alpha(x: torch.Tensor, alpha_out: Optional[torch.Tensor] = None,
                      ws: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Per-tensor NVFP4 scale alpha = max|x| / 2688 (Eq. 2) as a [1] fp32 tensor."""
    desc = make_desc(x, FOCUS_NVFP4)
    if alpha_out is None:
        alpha_out = torch.empty(1, dtype=torch.float32, device=x.device)
    ws, nb = _workspace(desc, FOCUS_WS_ALPHA, x.device, ws)
    _check(lib().focus_nvfp4_alpha(ctypes.byref(desc), _p(x), _p(alpha_out), _p(ws), nb,
                                   _stream(x.device)), "focus_nvfp4_alpha")
    return alpha_out


def focus_nvfp4_alpha_noalloc(x: torch.Tensor, alpha_out: torch.Tensor) -> torch.Tensor:
    """focus_nvfp4_alpha without a workspace, for callers that cannot allocate
    device memory: the partials live in the library's static device array.
    alpha_out must be given (a [1] fp32 CUDA tensor); nothing is allocated."""
    desc = make_desc(x, FOCUS_NVFP4)
    _check(lib().focus_nvfp4_alpha_noalloc(ctypes.byref(desc), _p(x), _p(alpha_out),
                                           _stream(x.device)), "focus_nvfp4_alpha_noalloc")
    return alpha_out


def _check_sfp(x, fmt, t, name):
    _dense(t, x.shape[0] * (x.shape[1] // block_of(fmt)), torch.float32, name)


def focus_fq_fwd(x, fmt, crs=None, dgs=None, alpha=None, *, sub_block=8, shared=False,
                 mx_rule=FOCUS_MX_CEIL, y=None, scale_bytes=None, want_scales=False, sfp=None):
    """y = Q_E2M1(x / S^q) * S^dq (Eq. 1-8); returns y, or (y, scale_bytes).
    sfp: optional learnable full-precision scales (Eq. 4)."""
    desc = make_desc(x, fmt, sub_block, shared, FOCUS_STE_IDENTITY, mx_rule)
    _check_coefs(x, fmt, sub_block, shared, crs, dgs)
    _check_sfp(x, fmt, sfp, "sfp")
    if y is None:
        y = _like_x(x)
    _same_layout(x, y, "y")
    if scale_bytes is None and want_scales:
        scale_bytes = torch.empty((x.shape[0], x.shape[1] // block_of(fmt)), dtype=torch.uint8,
                                  device=x.device)
    _dense(scale_bytes, x.shape[0] * (x.shape[1] // block_of(fmt)), torch.uint8, "scale_bytes")
    _check(lib().focus_fq_fwd(ctypes.byref(desc), _p(x), _p(crs), _p(dgs), _p(alpha), _p(sfp),
                              _p(y), _p(scale_bytes), _stream(x.device)), "focus_fq_fwd")
    return (y, scale_bytes) if (want_scales or scale_bytes is not None) else y


def focus_fq_bwd(x, g, fmt, crs=None, dgs=None, alpha=None, *, sub_block=8, shared=False,
                 ste=FOCUS_STE_IDENTITY, mx_rule=FOCUS_MX_CEIL, want_gx=True, want_gcrs=None,
                 want_gdgs=None, gx=None, gcrs=None, gdgs=None, ws=None, sfp=None,
                 want_gsfp=None, gsfp=None):
    """STE backward (Sec. 3.2): returns (gx, gcrs, gdgs) -- or (gx, gcrs, gdgs, gsfp)
    when the S^fp gradient is requested (by default when sfp is given); an
    unrequested output is None.  By default gcrs / gdgs are produced when
    crs / dgs are given."""
    desc = make_desc(x, fmt, sub_block, shared, ste, mx_rule)
    rows, cols = x.shape
    crow = 1 if shared else rows
    want_gcrs = (crs is not None) if want_gcrs is None else want_gcrs
    want_gdgs = (dgs is not None) if want_gdgs is None else want_gdgs
    _check_coefs(x, fmt, sub_block, shared, crs, dgs)
    _same_layout(x, g, "g")
    if gx is None and want_gx:
        gx = _like_x(x)
    _same_layout(x, gx, "gx")
    if gcrs is None and want_gcrs:
        gcrs = torch.empty((crow, cols // block_of(fmt)), dtype=torch.float32, device=x.device)
    if gdgs is None and want_gdgs:
        gdgs = torch.empty((crow, cols // sub_block), dtype=torch.float32, device=x.device)
    want_gsfp = (sfp is not None or gsfp is not None) if want_gsfp is None else want_gsfp
    if gsfp is None and want_gsfp:
        gsfp = torch.empty((rows, cols // block_of(fmt)), dtype=torch.float32, device=x.device)
    _check_sfp(x, fmt, sfp, "sfp")
    _check_sfp(x, fmt, gsfp, "gsfp")
    _check_coefs(x, fmt, sub_block, shared, gcrs, gdgs)
    ws, nb = _workspace(desc, FOCUS_WS_BWD, x.device, ws)
    _check(lib().focus_fq_bwd(ctypes.byref(desc), _p(x), _p(crs), _p(dgs), _p(alpha), _p(sfp),
                              _p(g), _p(gx), _p(gcrs), _p(gdgs), _p(gsfp), _p(ws), nb,
                              _stream(x.device)),
           "focus_fq_bwd")
    if want_gsfp:
        return gx, gcrs, gdgs, gsfp
    return gx, gcrs, gdgs


def focus_fq_bwd_adamw(x, g, fmt, step, hp, crs=None, dgs=None, sfp=None, moments=None,
                       alpha=None, *, sub_block=8, shared=False, ste=FOCUS_STE_IDENTITY,
                       mx_rule=FOCUS_MX_CEIL, want_gx=True, gx=None, gcrs=None, gdgs=None,
                       gsfp=None, ws=None):
    """STE backward fused with one AdamW step (Sec. 3.2, Sec. 4.1).

    crs / dgs / sfp: the learned arrays (fp32 CUDA tensors, updated in place;
    None = not learned).  moments: dict name -> (m, v) tensors shaped like the
    parameter ('crs', 'dgs', 'sfp'), updated in place.  step: int64 CUDA
    tensor holding t >= 1 (read only).  hp: dict with lr_coef, lr_scale,
    beta1, beta2, eps, weight_decay.  gcrs / gdgs / gsfp: optional gradient
    outputs.  Returns gx (or None)."""
    desc = make_desc(x, fmt, sub_block, shared, ste, mx_rule)
    moments = moments or {}
    _check_coefs(x, fmt, sub_block, shared, crs, dgs)
    _check_coefs(x, fmt, sub_block, shared, gcrs, gdgs)
    _check_sfp(x, fmt, sfp, "sfp")
    _check_sfp(x, fmt, gsfp, "gsfp")
    _same_layout(x, g, "g")
    if gx is None and want_gx:
        gx = _like_x(x)
    _same_layout(x, gx, "gx")
    if step.dtype != torch.int64 or step.numel() != 1 or step.device != x.device:
        raise ValueError("step must be a one-element int64 tensor on x's device")
    st = focus_adamw_state_t()
    for name, param in (("crs", crs), ("dgs", dgs), ("sfp", sfp)):
        if param is None:
            continue
        if name not in moments:
            raise ValueError(f"moments for {name} are missing")
        for k, t in zip("mv", moments[name]):
            _dense(t, param.numel(), torch.float32, f"{k}_{name}")
            setattr(st, f"{k}_{name}", t.data_ptr())
    h = focus_adamw_t(*(float(hp[k]) for k in ("lr_coef", "lr_scale", "beta1", "beta2", "eps",
                                                 "weight_decay")))
    ws, nb = _workspace(desc, FOCUS_WS_BWD, x.device, ws)
    _check(lib().focus_fq_bwd_adamw(ctypes.byref(desc), _p(x), _p(crs), _p(dgs), _p(alpha),
                                    _p(sfp), _p(g), _p(gx), ctypes.byref(h), ctypes.byref(st),
                                    _p(step), _p(gcrs), _p(gdgs), _p(gsfp), _p(ws), nb,
                                    _stream(x.device)),
           "focus_fq_bwd_adamw")
    return gx


def focus_pack(x, fmt, crs=None, dgs=None, alpha=None, *, sub_block=8, shared=False,
               mx_rule=FOCUS_MX_CEIL, codes=None, scale_bytes=None, sfp=None):
    """Export (Fig. 3(d)): returns (codes [rows, cols/2] uint8, scale bytes [rows, cols/B])."""
    desc = make_desc(x, fmt, sub_block, shared, FOCUS_STE_IDENTITY, mx_rule)
    rows, cols = x.shape
    if codes is None:
        codes = torch.empty((rows, cols // 2), dtype=torch.uint8, device=x.device)
    if scale_bytes is None:
        scale_bytes = torch.empty((rows, cols // block_of(fmt)), dtype=torch.uint8, device=x.device)
    _check_coefs(x, fmt, sub_block, shared, crs, dgs)
    _dense(codes, rows * cols // 2, torch.uint8, "codes")
    _dense(scale_bytes, rows * cols // block_of(fmt), torch.uint8, "scale_bytes")
    _check_sfp(x, fmt, sfp, "sfp")
    _check(lib().focus_pack(ctypes.byref(desc), _p(x), _p(crs), _p(dgs), _p(alpha), _p(sfp),
                            _p(codes), _p(scale_bytes), _stream(x.device)), "focus_pack")
    return codes, scale_bytes


def focus_mma_scale_bytes(desc: focus_desc_t) -> int:
    return int(lib().focus_mma_scale_bytes(ctypes.byref(desc)))


def focus_pack_mma(x, fmt, crs=None, dgs=None, alpha=None, *, sub_block=8, shared=False,
                   mx_rule=FOCUS_MX_CEIL, codes=None, scale_tiles=None, sfp=None):
    """Export for the block-scaled tensor-core MMA: returns (codes [rows, cols/2]
    uint8, scale tiles: focus_mma_scale_bytes uint8 in the 128 x 4 tile layout)."""
    desc = make_desc(x, fmt, sub_block, shared, FOCUS_STE_IDENTITY, mx_rule)
    rows, cols = x.shape
    n = focus_mma_scale_bytes(desc)
    if codes is None:
        codes = torch.empty((rows, cols // 2), dtype=torch.uint8, device=x.device)
    if scale_tiles is None:
        scale_tiles = torch.empty(max(n, 16), dtype=torch.uint8, device=x.device)
    _check_coefs(x, fmt, sub_block, shared, crs, dgs)
    _dense(codes, rows * cols // 2, torch.uint8, "codes")
    if not scale_tiles.is_contiguous() or scale_tiles.numel() < n or scale_tiles.dtype != torch.uint8:
        raise ValueError(f"scale_tiles must be a contiguous uint8 tensor of at least {n} bytes")
    _check_sfp(x, fmt, sfp, "sfp")
    _check(lib().focus_pack_mma(ctypes.byref(desc), _p(x), _p(crs), _p(dgs), _p(alpha), _p(sfp),
                                _p(codes), _p(scale_tiles), _stream(x.device)), "focus_pack_mma")
    return codes, scale_tiles


def focus_fp4_gemm(fmt, a_codes, a_tiles, b_codes, b_tiles, alpha_a=None, alpha_b=None, *, d=None,
                   out_dtype=torch.float32, timeout_flag=None):
    """D = A B^T on the block-scaled FP4 tensor cores from two focus_pack_mma
    exports (codes [M, K/2] and [N, K/2] uint8, their scale tiles); returns
    D [M, N] (fp32 or bf16).  alpha_a / alpha_b: NVFP4 per-tensor scales
    ([1] fp32)."""
    M, kh = a_codes.shape
    N, kh2 = b_codes.shape
    if kh != kh2:
        raise ValueError("A and B must have the same K")
    K = 2 * kh
    for t, name in ((a_codes, "a_codes"), (b_codes, "b_codes"), (a_tiles, "a_tiles"),
                    (b_tiles, "b_tiles")):
        if t.dtype != torch.uint8 or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous uint8 tensor")
    if d is None:
        d = torch.empty((M, N), dtype=out_dtype, device=a_codes.device)
    if d.dtype not in (torch.float32, torch.bfloat16) or d.dim() != 2 or d.shape[0] != M or \
            d.shape[1] != N or (M > 0 and N > 0 and d.stride(1) != 1):
        raise ValueError("d must be a [M, N] fp32 or bf16 tensor with unit column stride")
    dt = FOCUS_BF16 if d.dtype == torch.bfloat16 else FOCUS_F32
    _check(lib().focus_fp4_gemm(int(fmt), M, N, K, _p(a_codes), _p(a_tiles), _p(alpha_a),
                                _p(b_codes), _p(b_tiles), _p(alpha_b), _p(d), dt, max(d.stride(0), N),
                                _p(timeout_flag), _stream(a_codes.device)), "focus_fp4_gemm")
    return d


def focus_version() -> int:
    return int(lib().focus_version())


# ---------------------------------------------------------------------------
# group entry points: one launch for several tensors
# ---------------------------------------------------------------------------
_GROUP_FIELDS = ("x", "g", "y", "gx", "crs", "dgs", "alpha", "sfp", "gcrs", "gdgs", "gsfp", "codes",
                 "scale_bytes")


def _group_array(items, fmt, sub_block, ste=FOCUS_STE_IDENTITY, mx_rule=FOCUS_MX_CEIL):
    """ctypes array of focus_tensor_t from dicts of tensors (keys as the
    struct's fields).  The dicts are kept alive by the caller."""
    if len(items) > FOCUS_MAX_GROUP:
        raise ValueError(f"at most {FOCUS_MAX_GROUP} tensors per group")
    arr = (focus_tensor_t * max(1, len(items)))()
    for i, it in enumerate(items):
        x = it["x"]
        arr[i].desc = make_desc(x, fmt, sub_block, False, ste, mx_rule)
        for k in _GROUP_FIELDS:
            t = it.get(k)
            if t is not None:
                setattr(arr[i], k, t.data_ptr())
    return arr


def focus_nvfp4_alpha_group(xs, alpha_out=None, ws=None):
    """Per-tensor NVFP4 alpha (Eq. 2) of every tensor in xs, one launch pair;
    returns a [n] fp32 tensor."""
    items = [{"x": x} for x in xs]
    arr = _group_array(items, FOCUS_NVFP4, 16)
    dev_ = xs[0].device
    if alpha_out is None:
        alpha_out = torch.empty(len(xs), dtype=torch.float32, device=dev_)
    n = int(lib().focus_group_workspace_bytes(arr, len(xs)))
    if ws is None:
        ws = torch.empty(max(16, n), dtype=torch.uint8, device=dev_)
    _check(lib().focus_nvfp4_alpha_group(arr, len(xs), _p(alpha_out), _p(ws), ws.numel(), _stream(dev_)),
           "focus_nvfp4_alpha_group")
    return alpha_out


def focus_group_workspace_bytes(xs) -> int:
    arr = _group_array([{"x": x} for x in xs], FOCUS_NVFP4, 16)
    return int(lib().focus_group_workspace_bytes(arr, len(xs)))


def focus_fq_fwd_group(items, fmt, *, sub_block=8, mx_rule=FOCUS_MX_CEIL):
    """focus_fq_fwd for each dict of `items` (keys x, crs, dgs, alpha, sfp and
    optionally y, scale_bytes); allocates a missing y; returns the list of y."""
    for it in items:
        if it.get("y") is None:
            it["y"] = _like_x(it["x"])
        _same_layout(it["x"], it["y"], "y")
        _check_coefs(it["x"], fmt, sub_block, False, it.get("crs"), it.get("dgs"))
        _check_sfp(it["x"], fmt, it.get("sfp"), "sfp")
    arr = _group_array(items, fmt, sub_block, FOCUS_STE_IDENTITY, mx_rule)
    _check(lib().focus_fq_fwd_group(arr, len(items), _stream(items[0]["x"].device)), "focus_fq_fwd_group")
    return [it["y"] for it in items]


def focus_pack_group(items, fmt, *, sub_block=8, mx_rule=FOCUS_MX_CEIL):
    """focus_pack for each dict of `items`; allocates missing codes /
    scale_bytes; returns the list of (codes, scale_bytes)."""
    for it in items:
        x = it["x"]
        rows, cols = x.shape
        if it.get("codes") is None:
            it["codes"] = torch.empty((rows, cols // 2), dtype=torch.uint8, device=x.device)
        if it.get("scale_bytes") is None:
            it["scale_bytes"] = torch.empty((rows, cols // block_of(fmt)), dtype=torch.uint8, device=x.device)
        _dense(it["codes"], rows * cols // 2, torch.uint8, "codes")
        _dense(it["scale_bytes"], rows * cols // block_of(fmt), torch.uint8, "scale_bytes")
        _check_coefs(x, fmt, sub_block, False, it.get("crs"), it.get("dgs"))
        _check_sfp(x, fmt, it.get("sfp"), "sfp")
    arr = _group_array(items, fmt, sub_block, FOCUS_STE_IDENTITY, mx_rule)
    _check(lib().focus_pack_group(arr, len(items), _stream(items[0]["x"].device)), "focus_pack_group")
    return [(it["codes"], it["scale_bytes"]) for it in items]


def focus_fq_bwd_group(items, fmt, *, sub_block=8, ste=FOCUS_STE_IDENTITY, mx_rule=FOCUS_MX_CEIL):
    """focus_fq_bwd for each dict of `items` (keys x, g, crs, dgs, alpha, sfp
    and the outputs gx, gcrs, gdgs, gsfp, each allocated when the dict has
    the key with value None); returns the list of dicts."""
    for it in items:
        x = it["x"]
        rows, cols = x.shape
        _same_layout(x, it["g"], "g")
        if "gx" in it and it["gx"] is None:
            it["gx"] = _like_x(x)
        if "gcrs" in it and it["gcrs"] is None:
            it["gcrs"] = torch.empty((rows, cols // block_of(fmt)), dtype=torch.float32, device=x.device)
        if "gdgs" in it and it["gdgs"] is None:
            it["gdgs"] = torch.empty((rows, cols // sub_block), dtype=torch.float32, device=x.device)
        if "gsfp" in it and it["gsfp"] is None:
            it["gsfp"] = torch.empty((rows, cols // block_of(fmt)), dtype=torch.float32, device=x.device)
        _same_layout(x, it.get("gx"), "gx")
        _check_coefs(x, fmt, sub_block, False, it.get("crs"), it.get("dgs"))
        _check_coefs(x, fmt, sub_block, False, it.get("gcrs"), it.get("gdgs"))
        _check_sfp(x, fmt, it.get("sfp"), "sfp")
        _check_sfp(x, fmt, it.get("gsfp"), "gsfp")
    arr = _group_array(items, fmt, sub_block, ste, mx_rule)
    _check(lib().focus_fq_bwd_group(arr, len(items), _stream(items[0]["x"].device)), "focus_fq_bwd_group")
    return items
