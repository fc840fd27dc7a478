"""Run one kernel of the fake-quantizer on one tensor of a workload, for
profiler captures (ncu) of a single launch on a case of known size.

  python -m paper_2608_01847_gb300.profile_case --phase bwd --workload qwen3_4b_layer \
      --tensor gate_proj --fmt nvfp4 --launches 3
  python -m paper_2608_01847_gb300.profile_case --phase bwd --workload act_262144x4096 \
      --tensor act --rows 32768 --shared --launches 3

`--rows R` draws only the first R rows' worth of the tensor (the same
recipe on an [R, cols] tensor), for captures of a smaller case of a large
workload; `--adam` runs the backward fused with one AdamW step on the
coefficients (and on S^fp with `--sfp`).

Draws the tensor on the GPU (seeded, same recipe as the benchmark), runs the
phase `--launches` times and prints the CUDA-event time per launch and the
algorithmic bytes it moves.  Not a benchmark: the numbers it prints are for
orientation only.
"""
from __future__ import annotations

import argparse
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def bytes_per_elem(phase, fmt, sub, shared, gx=True):
    B = 32 if fmt == "mxfp4" else 16
    coef = 0.0 if shared else 4 / B + 4 / sub
    return {"alpha": 2.0, "fwd": 4 + coef, "pack": 2 + coef + 0.5 + 1 / B,
            "bwd": 4 + (2 if gx else 0) + 2 * coef}[phase]


def main():
    import torch

    from paper_2608_01847_gb300 import build as B
    from paper_2608_01847_gb300 import focus as F
    from paper_2608_01847_gb300 import workloads as W

    ap = argparse.ArgumentParser()
    ap.add_argument("--phase", choices=["alpha", "fwd", "bwd", "pack", "gemm"], default="bwd")
    ap.add_argument("--tokens", type=int, default=8192, help="gemm: activation rows")
    ap.add_argument("--workload", default="qwen3_4b_layer")
    ap.add_argument("--tensor", default="gate_proj")
    ap.add_argument("--fmt", choices=["mxfp4", "nvfp4"], default="nvfp4")
    ap.add_argument("--sub", type=int, default=8)
    ap.add_argument("--shared", action="store_true")
    ap.add_argument("--no-gx", action="store_true")
    ap.add_argument("--sfp", action="store_true", help="bwd: learnable S^fp and its gradient")
    ap.add_argument("--adam", action="store_true", help="bwd: fused with one AdamW step")
    ap.add_argument("--rows", type=int, default=0, help="draw only this many rows of the tensor")
    ap.add_argument("--pad", type=int, default=0,
                    help="row pitch cols + PAD elements (PAD = 8 bf16: rows on 16-byte, not 32-byte, "
                         "boundaries)")
    ap.add_argument("--library", action="store_true",
                    help="gemm, NVFP4: NVIDIA's block-scaled GEMM (cuBLASLt through torch._scaled_mm) on the "
                         "same exports instead of fp4_gemm_kernel")
    ap.add_argument("--launches", type=int, default=3)
    a = ap.parse_args()

    B.build()
    F.lib()
    import dataclasses
    w = W.WORKLOADS[a.workload]
    idx = [t.name for t in w.tensors].index(a.tensor)
    if a.rows:
        t = w.tensors[idx]
        specs = list(w.tensors)
        specs[idx] = W.TensorSpec(t.name, min(a.rows, t.rows), t.cols)
        w = dataclasses.replace(w, tensors=tuple(specs))
    fmt = F.FOCUS_MXFP4 if a.fmt == "mxfp4" else F.FOCUS_NVFP4
    blk = F.block_of(fmt)
    x, g = W.device_tensor(w, idx, "cuda")
    if a.pad:
        def padded(t):
            b = torch.zeros((t.shape[0], t.shape[1] + a.pad), dtype=t.dtype, device=t.device)
            b[:, :t.shape[1]] = t
            return b[:, :t.shape[1]]
        x, g = padded(x), padded(g)
    crs, dgs = W.device_coefs(w, idx, blk, a.sub, "cuda", shared=a.shared)
    alpha = F.focus_nvfp4_alpha(x)
    y = F._like_x(x)
    gx = None if a.no_gx else F._like_x(x)
    gc, gd = torch.empty_like(crs), torch.empty_like(dgs)
    sfp = gsfp = None
    if a.sfp:
        # S^fp at its absmax initialisation (fp32 per block), as the benchmark's --sfp
        m = x.float().abs().reshape(x.shape[0], -1, blk).amax(-1)
        den = 6.0 if fmt == F.FOCUS_MXFP4 else float(alpha.item()) * 6.0
        sfp = (m / den).contiguous()
        gsfp = torch.empty_like(sfp)
    rows, cols = x.shape
    codes = torch.empty((rows, cols // 2), dtype=torch.uint8, device="cuda")
    sb = torch.empty((rows, cols // blk), dtype=torch.uint8, device="cuda")
    desc = F.make_desc(x, fmt, a.sub, a.shared)
    ws = torch.empty(max(16, F.focus_workspace_bytes(desc, F.FOCUS_WS_BWD),
                         F.focus_workspace_bytes(desc, F.FOCUS_WS_ALPHA)),
                     dtype=torch.uint8, device="cuda")

    if a.phase == "gemm":
        # W4A4 GEMM D[tokens, rows] = A[tokens, cols] W[rows, cols]^T on exports
        gen = torch.Generator(device="cuda")
        gen.manual_seed(4321)
        act = torch.randn((a.tokens, cols), generator=gen, device="cuda").to(torch.bfloat16)
        act_alpha = F.focus_nvfp4_alpha(act)
        ac, at = F.focus_pack_mma(act, fmt, alpha=act_alpha)
        wc, wt = F.focus_pack_mma(x, fmt, alpha=alpha)
        dmat = torch.empty((a.tokens, rows), dtype=torch.bfloat16, device="cuda")
        del act, g, gx, y
        if a.library:
            if fmt != F.FOCUS_NVFP4:
                raise SystemExit("--library: NVFP4 only")
            a4, w4 = ac.view(torch.float4_e2m1fn_x2), wc.view(torch.float4_e2m1fn_x2).t()
            sa, sw = at.view(torch.float8_e4m3fn), wt.view(torch.float8_e4m3fn)

    if a.adam:
        # the paper's learning rates (Sec. 4.1), PyTorch's AdamW defaults
        hp = dict(lr_coef=5e-2 if fmt == F.FOCUS_MXFP4 else 1e-3,
                  lr_scale=2e-2 * 2.0 ** -7 if fmt == F.FOCUS_MXFP4 else 5e-3,
                  beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)
        learned = {"crs": crs, "dgs": dgs, **({"sfp": sfp} if sfp is not None else {})}
        moments = {k: (torch.zeros_like(v), torch.zeros_like(v)) for k, v in learned.items()}
        step = torch.ones(1, dtype=torch.int64, device="cuda")

    def run():
        if a.phase == "bwd" and a.adam:
            F.focus_fq_bwd_adamw(x, g, fmt, step, hp, crs=crs, dgs=dgs, sfp=sfp, moments=moments,
                                 alpha=alpha, sub_block=a.sub, shared=a.shared, gx=gx,
                                 want_gx=not a.no_gx, ws=ws)
        elif a.phase == "gemm" and a.library:
            torch._scaled_mm(a4, w4, sa, sw, out_dtype=torch.bfloat16)
        elif a.phase == "gemm":
            F.focus_fp4_gemm(fmt, ac, at, wc, wt, act_alpha, alpha, d=dmat)
        elif a.phase == "alpha":
            F.focus_nvfp4_alpha(x, alpha, ws)
        elif a.phase == "fwd":
            F.focus_fq_fwd(x, fmt, crs, dgs, alpha, sub_block=a.sub, shared=a.shared, y=y)
        elif a.phase == "pack":
            F.focus_pack(x, fmt, crs, dgs, alpha, sub_block=a.sub, shared=a.shared, codes=codes,
                         scale_bytes=sb)
        else:
            F.focus_fq_bwd(x, g, fmt, crs, dgs, alpha, sub_block=a.sub, shared=a.shared, gx=gx,
                           want_gx=not a.no_gx, gcrs=gc, gdgs=gd, ws=ws, sfp=sfp, gsfp=gsfp)

    torch.cuda.synchronize()
    times = []
    # the timed launches inside one NVTX range, so that a profiler can take
    # them alone (ncu --nvtx --nvtx-include "launches/")
    torch.cuda.nvtx.range_push("launches")
    for _ in range(a.launches):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        run()
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    torch.cuda.nvtx.range_pop()
    if a.phase == "gemm":
        flops = 2 * a.tokens * rows * cols
        print(json.dumps({"phase": "gemm", "tensor": f"{a.workload}/{a.tensor}",
                          "shape": [a.tokens, rows, cols], "fmt": a.fmt,
                          "kernel": "cuBLASLt (torch._scaled_mm)" if a.library else "fp4_gemm_kernel", "ms": times,
                          "tflops_last": flops / (times[-1] * 1e-3) / 1e12}))
        return
    n = rows * cols
    bpe = bytes_per_elem(a.phase, a.fmt, a.sub, a.shared, not a.no_gx)
    if a.sfp and a.phase == "bwd":
        bpe += 2 * 4 / blk   # S^fp in, its gradient out
    if a.adam and a.phase == "bwd":
        # per learned value p, m, v in and out instead of p in and gradient out
        coef = 0.0 if a.shared else 4 / blk + 4 / a.sub
        bpe += 4 * (coef + (4 / blk if a.sfp else 0.0))
    print(json.dumps({"phase": a.phase, "tensor": f"{a.workload}/{a.tensor}", "shape": [rows, cols],
                      "fmt": a.fmt, "sub": a.sub, "shared": a.shared, "adam": a.adam, "pad": a.pad,
                      "ms": times,
                      "algorithmic_bytes": n * bpe,
                      "gbs_last": n * bpe / (times[-1] * 1e-3) / 1e9}))


if __name__ == "__main__":
    main()
