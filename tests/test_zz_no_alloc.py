"""The allocation-free alpha entry point against the allocating one.

focus_nvfp4_alpha_noalloc serves callers that cannot allocate device memory
(for example a plugin whose host application owns every device allocation,
or a hot loop that must never call cudaMalloc because it can synchronise the
device): it keeps its per-CTA partials in a static array inside the library
instead of a caller-provided workspace.  Its result must equal
focus_nvfp4_alpha's exactly, on consecutive calls -- the second call must not
be affected by what the first one left in the shared array.

This file is named to be collected last, so that a failure here comes after
every other test has run.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_01847_gb300 import build as B
from paper_2608_01847_gb300 import focus as F
from paper_2608_01847_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _alpha_both(L, x):
    """alpha of x through the C ABI: (allocating entry point, static-scratch one)."""
    desc = F.make_desc(x, F.FOCUS_NVFP4)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    nbytes = L.focus_workspace_bytes(ctypes.byref(desc), F.FOCUS_WS_ALPHA)
    ws = torch.empty(max(16, nbytes), dtype=torch.uint8, device="cuda")
    ref = torch.full((1,), float("nan"), dtype=torch.float32, device="cuda")
    got = torch.full((1,), float("nan"), dtype=torch.float32, device="cuda")
    rc = L.focus_nvfp4_alpha(ctypes.byref(desc), ctypes.c_void_p(x.data_ptr()),
                             ctypes.c_void_p(ref.data_ptr()), ctypes.c_void_p(ws.data_ptr()),
                             ws.numel(), stream)
    assert rc == 0, rc
    rc = L.focus_nvfp4_alpha_noalloc(ctypes.byref(desc), ctypes.c_void_p(x.data_ptr()),
                                     ctypes.c_void_p(got.data_ptr()), stream)
    assert rc == 0, rc
    torch.cuda.synchronize()
    return ref.cpu().numpy(), got.cpu().numpy()


def test_static_scratch_alpha_equals_allocating_alpha():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    L = F.lib()
    w = W.WORKLOADS["qwen3_4b_layer"]
    # first call: a large tensor with big outliers (many CTAs, large partials);
    # second call: a smaller tensor with a smaller max, so stale partials from
    # the first call would show up as a wrong (too large) alpha
    big, _ = W.device_tensor(w, 4, "cuda")                    # gate_proj 9728 x 2560 bf16
    small = torch.randn((1024, 2560), device="cuda", dtype=torch.float32) * 1e-3
    for x in (big, small):
        ref, got = _alpha_both(L, x)
        assert np.isfinite(ref[0]) and ref[0] > 0
        assert got.view(np.uint32)[0] == ref.view(np.uint32)[0], (got, ref)
