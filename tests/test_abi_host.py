"""Host-side checks of the C ABI (no GPU needed).

The library must build for sm_103a, load, and export every entry point that
include/focus_fq.h declares -- and nothing else.  Argument errors must be
reported with the documented status before anything reaches the GPU, so the
calls below use placeholder pointer values that are never dereferenced.
"""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2608_01847_gb300 import build as B
from paper_2608_01847_gb300 import focus as F

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "focus_fq.h")


@pytest.fixture(scope="module")
def L():
    B.build()
    return F.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(focus_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_abi():
    assert declared_functions() == sorted(F.ENTRY_POINTS)


def test_exports_exactly_the_declared_symbols(L):
    for name in declared_functions():
        assert hasattr(L, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", B.LIB], capture_output=True, text=True,
                         check=True).stdout
    exported = sorted({ln.split()[-1] for ln in out.splitlines()
                       if ln.split() and ln.split()[-2] in ("T", "W")
                       and not ln.split()[-1].startswith("_")})
    assert exported == declared_functions()


def test_version_and_status_strings(L):
    assert F.focus_version() == 210
    for code in (0, -1, -2, -3, -4, -5):
        assert L.focus_status_string(code)
    assert L.focus_status_string(42) == b"unknown status"


def _desc(rows=4, cols=64, ld=None, dtype=1, fmt=0, block=None, sub=8, shared=0, ste=0, rule=0):
    return F.focus_desc_t(rows, cols, cols if ld is None else ld, dtype, fmt,
                          block if block is not None else (32 if fmt == 0 else 16), sub, shared,
                          ste, rule)


P = ctypes.c_void_p
ALIGNED = P(0x100000)       # placeholder device addresses: never dereferenced
ALIGNED2 = P(0x200000)
ODD = P(0x100008)           # 8-byte aligned only (rows and coefficient arrays need 16)
ODD8 = ODD


def fwd(L, d, x=ALIGNED, crs=None, dgs=None, alpha=ALIGNED2, y=ALIGNED2, sb=None, sfp=None):
    return L.focus_fq_fwd(ctypes.byref(d) if d is not None else None, x, crs, dgs, alpha, sfp, y,
                          sb, None)


@pytest.mark.parametrize("kw,status", [
    (dict(block=64), -2), (dict(fmt=1, block=32), -2), (dict(sub=3), -2), (dict(sub=32, fmt=1), -2),
    (dict(sub=64), -2), (dict(cols=48), -1), (dict(ld=60), -1), (dict(ld=68), -3),
    (dict(ld=76), -3), (dict(ld=72, dtype=0, rows=0), 0), (dict(ld=66, dtype=0), -3),
    # a row pitch of 16 (not 32) bytes passes the checks (shown on empty tensors,
    # which return before anything is launched)
    (dict(ld=72, rows=0), 0), (dict(ld=68, dtype=0, rows=0), 0),
    (dict(dtype=3), -1), (dict(dtype=2, rows=0), 0), (dict(dtype=2, ld=68), -3), (dict(fmt=2), -1), (dict(ste=3), -1), (dict(rule=2), -1),
    (dict(shared=2), -1), (dict(rows=-1), -1), (dict(rows=1 << 40, cols=1 << 20), -2),
])
def test_descriptor_rejections(L, kw, status):
    assert fwd(L, _desc(**kw)) == status


def test_null_and_alignment_rejections(L):
    assert fwd(L, None) == -1
    assert fwd(L, _desc(), x=None) == -1
    assert fwd(L, _desc(), y=None) == -1
    assert fwd(L, _desc(fmt=1), alpha=None) == -1                 # NVFP4 needs alpha
    assert fwd(L, _desc(), x=ODD) == -3
    assert fwd(L, _desc(), y=ODD) == -3
    assert fwd(L, _desc(), crs=ODD8) == -3
    assert fwd(L, _desc(rows=0)) == 0                             # empty: nothing to do
    d = _desc()
    assert L.focus_pack(ctypes.byref(d), ALIGNED, None, None, None, None, None, ALIGNED2,
                        None) == -1
    assert L.focus_pack(ctypes.byref(d), ALIGNED, None, None, None, None, P(0x100002), ALIGNED2,
                        None) == -3
    g = ALIGNED2
    assert L.focus_fq_bwd(ctypes.byref(d), ALIGNED, None, None, None, None, None, g, None, None,
                          None, None, 0, None) == -1              # g missing
    assert L.focus_fq_bwd(ctypes.byref(d), ALIGNED, None, None, None, None, g, ODD, None, None,
                          None, None, 0, None) == -3              # gx misaligned
    assert fwd(L, _desc(), sfp=P(0x100002)) == -3                 # S^fp must be 4-byte aligned
    assert fwd(L, _desc(shared=1), sfp=ALIGNED2) == -1            # S^fp is per row
    assert L.focus_fq_bwd(ctypes.byref(_desc(shared=1)), ALIGNED, None, None, None, None, g, None,
                          None, None, ALIGNED2, None, 0, None) == -1
    assert L.focus_nvfp4_alpha(ctypes.byref(d), ALIGNED, None, ALIGNED2, 1 << 20, None) == -1


def test_shared_backward_needs_workspace(L):
    d = _desc(rows=64, cols=256, shared=1)
    need = L.focus_workspace_bytes(ctypes.byref(d), F.FOCUS_WS_BWD)
    assert need > 0
    gc = ALIGNED2
    rc = L.focus_fq_bwd(ctypes.byref(d), ALIGNED, None, None, None, None, ALIGNED2, None, gc, None,
                        None, None, 0, None)
    assert rc == -4
    rc = L.focus_fq_bwd(ctypes.byref(d), ALIGNED, None, None, None, None, ALIGNED2, None, gc, None,
                        None, ALIGNED, need - 1, None)
    assert rc == -4
    assert L.focus_nvfp4_alpha(ctypes.byref(d), ALIGNED, ALIGNED2, None, 0, None) == -4


def test_workspace_queries(L):
    d = _desc(rows=64, cols=256, shared=0)
    assert L.focus_workspace_bytes(ctypes.byref(d), F.FOCUS_WS_BWD) == 0
    assert L.focus_workspace_bytes(ctypes.byref(d), F.FOCUS_WS_ALPHA) >= 4
    assert L.focus_workspace_bytes(ctypes.byref(d), 7) == 0
    assert L.focus_workspace_bytes(None, 0) == 0


def test_fastdiv_magic_numbers():
    """The invariant-divisor reciprocal used for row / column indices
    (Granlund-Montgomery) divides exactly for every 32-bit numerator."""
    import numpy as np
    rng = np.random.default_rng(0)
    for d in [1, 2, 3, 7, 64, 320, 1216, 3584, 4096, 65535, 1 << 20, (1 << 28) + 3]:
        l = 0
        while (1 << l) < d:
            l += 1
        m = ((1 << 32) * ((1 << l) - d)) // d + 1
        assert m < (1 << 32)
        n = np.concatenate([rng.integers(0, 1 << 32, 200000, dtype=np.uint64),
                            np.array([0, 1, d - 1, d, d + 1, (1 << 32) - 1], np.uint64)])
        n = n[n < (1 << 32)]
        t = (n * np.uint64(m)) >> np.uint64(32)
        q = (t + n) >> np.uint64(l)
        assert np.array_equal(q, n // np.uint64(d)), d


def adamw(L, d, hp, st, step=ALIGNED2, crs=ALIGNED, dgs=None, sfp=None, x=ALIGNED, g=ALIGNED2,
          gx=None, ws=None, nb=0):
    return L.focus_fq_bwd_adamw(ctypes.byref(d), x, crs, dgs, ALIGNED2, sfp, g, gx,
                                ctypes.byref(hp) if hp is not None else None,
                                ctypes.byref(st) if st is not None else None, step, None, None,
                                None, ws, nb, None)


def _hp(**kw):
    v = dict(lr_coef=5e-2, lr_scale=2e-2, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)
    v.update(kw)
    return F.focus_adamw_t(*(v[k] for k in ("lr_coef", "lr_scale", "beta1", "beta2", "eps",
                                            "weight_decay")))


def _st(**kw):
    st = F.focus_adamw_state_t()
    for i, n in enumerate(("m_crs", "v_crs", "m_dgs", "v_dgs", "m_sfp", "v_sfp")):
        setattr(st, n, kw.get(n, 0x300000 + 0x10000 * i))
    return st


@pytest.mark.parametrize("hp_kw,status", [
    (dict(lr_coef=-1.0), -1), (dict(lr_scale=float("nan")), -1), (dict(beta1=1.0), -1),
    (dict(beta2=-0.1), -1), (dict(eps=0.0), -1), (dict(eps=float("inf")), -1),
    (dict(weight_decay=-1e-3), -1), (dict(lr_coef=float("inf")), -1),
])
def test_adamw_hyperparameter_rejections(L, hp_kw, status):
    d = _desc(rows=0)      # nothing to compute: only the checks run
    assert adamw(L, d, _hp(**hp_kw), _st()) == status
    assert adamw(L, d, _hp(), _st()) == 0


def test_adamw_argument_rejections(L):
    d = _desc(rows=0)
    assert adamw(L, d, None, _st()) == -1                          # hyper-parameters missing
    assert adamw(L, d, _hp(), None) == -1                          # state missing
    assert adamw(L, d, _hp(), _st(), step=None) == -1              # step counter missing
    assert adamw(L, d, _hp(), _st(), step=P(0x100004)) == -3       # step is an int64
    assert adamw(L, d, _hp(), _st(m_crs=0)) == -1                  # moments of a learned array
    assert adamw(L, d, _hp(), _st(m_crs=0), crs=None) == 0         # ... not needed if not learned
    assert adamw(L, d, _hp(), _st(v_dgs=0x300008), dgs=ALIGNED) == -3
    assert adamw(L, d, _hp(), _st(m_sfp=0), sfp=ALIGNED) == -1
    assert adamw(L, _desc(rows=0, shared=1), _hp(), _st(), sfp=ALIGNED) == -1   # S^fp is per row
    assert adamw(L, _desc(), _hp(), _st(), x=ODD) == -3
    assert adamw(L, _desc(), _hp(), _st(), g=None) == -1
    assert adamw(L, _desc(fmt=1, block=32), _hp(), _st()) == -2
    d = _desc(rows=64, cols=256, shared=1)
    assert adamw(L, d, _hp(), _st()) == -4                         # shared rows need scratch


def _targ(rows=4, cols=64, dtype=1, fmt=1, shared=0, sub=8, x=ALIGNED, y=ALIGNED2, alpha=ALIGNED2):
    t = F.focus_tensor_t()
    t.desc = _desc(rows=rows, cols=cols, dtype=dtype, fmt=fmt, shared=shared, sub=sub)
    t.x, t.y, t.alpha = x.value, y.value, alpha.value
    t.g, t.codes, t.scale_bytes = ALIGNED2.value, ALIGNED2.value, ALIGNED2.value
    return t


def test_group_rejections(L):
    def fwd_group(*ts):
        arr = (F.focus_tensor_t * max(1, len(ts)))(*ts)
        return L.focus_fq_fwd_group(arr, len(ts), None)
    assert fwd_group() == 0                                             # nothing to do
    assert L.focus_fq_fwd_group(None, 1, None) == -1
    assert L.focus_fq_fwd_group(None, -1, None) == -1
    arr = (F.focus_tensor_t * 17)(*[_targ(rows=0) for _ in range(17)])
    assert L.focus_fq_fwd_group(arr, 17, None) == -2                   # more than FOCUS_MAX_GROUP
    assert fwd_group(_targ(rows=0), _targ(rows=0, dtype=0)) == -1      # element types differ
    assert fwd_group(_targ(rows=0), _targ(rows=0, sub=4)) == -1        # sub-block sizes differ
    assert fwd_group(_targ(rows=0), _targ(rows=0, fmt=0, sub=8)) == -1  # formats differ
    assert fwd_group(_targ(rows=0, shared=1)) == -1                    # shared coefficients
    assert fwd_group(_targ(x=ODD)) == -3
    assert fwd_group(_targ(alpha=P(0))) == -1                          # NVFP4 needs alpha
    assert fwd_group(_targ(y=P(0))) == -1
    assert fwd_group(_targ(rows=0), _targ(rows=0)) == 0                 # empty tensors are skipped
    arr = (F.focus_tensor_t * 2)(_targ(rows=64, cols=256), _targ(rows=8, cols=64))
    assert L.focus_group_workspace_bytes(arr, 2) >= 8
    assert L.focus_nvfp4_alpha_group(arr, 2, ALIGNED2, None, 0, None) == -4
    assert L.focus_nvfp4_alpha_group(arr, 2, None, ALIGNED, 1 << 20, None) == -1
