"""Benchmark of the FOCUS FP4 fake-quantizer hot path on GB300.

Default case: one step = one pass of the whole hot path over the W4A4
calibration activations of the paper's setup (Sec. 4.1: 128 sequences x
2048 tokens x hidden 4096 = 1.07 G bf16 elements, 2 GiB), NVFP4 (block 16,
E4M3 + a per-call fp32 alpha), per-block CRS and per-sub-block (8) DGS
coefficients:
  alpha (per tensor)  ->  fake-quant forward  ->  STE backward (input
  gradient + both coefficient gradients)  ->  export pack,
inputs resident in HBM.  The same workload under MXFP4 (block 32, E8M0) is
timed after it and reported under "other_format".  The step is captured once
as a CUDA graph: each tensor's phases chained on its own branch
(programmatic dependent launches), the tensors' branches side by side;
`--staged` joins all tensors between phases instead, `--group` runs each
phase as one group launch.  `value` is the algorithmic bytes of the step
(per-element figures in bytes_per_elem) over the step time.  The JSON line
also carries the phase split, the roofline of the dominant kernel, the
end-to-end figure (pinned host buffers, copies inside the timed region), the
CPU oracle baseline and the SM clocks sampled (NVML, read-only) during the
timed steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
                  [--workload NAME --fmt mxfp4|nvfp4 --shared --sfp --adam
                   --io f16 --sub B --staged --group --no-e2e --no-cpu-baseline]
  python bench.py --gemm [--fmt mxfp4] [--workload NAME] [--serial]

Other workloads (the Qwen3-4B layer, the Llama-3-8B block, the 70B layer
set, sweep tensors) are measured the same way with --workload.
`--impl reference` times the CPU oracle on a bounded sample of the same
workload.  `--gemm` times the W4A4 FP4 GEMMs of a layer's projections on
their exports (default: the Qwen3-4B layer x 8192 tokens), the independent
GEMMs of a step on parallel graph branches (--serial: one after another).

Under torchrun (N > 1) every rank runs the same workload on its own GPU
(replicas; no data-path collective), the step time is the max over ranks and
`value` sums all ranks' bytes (weak scaling).
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "fake-quant fwd+bwd GB/s and elems/s vs GB300 HBM peak; pack GB/s"
L2_BYTES = 129 * 1024 * 1024
# phase split: each phase captured this many times in one graph (the tensors
# joined between repetitions), so that a phase's time excludes the gap
# between graph replays
PHASE_REPS = 8


@dataclasses.dataclass(frozen=True)
class Case:
    workload: str = "act_262144x4096"
    fmt: str = "nvfp4"
    sub: int = 8
    shared: bool = False       # one coefficient set for all rows (activations)
    sfp: bool = False          # learnable full-precision scales S^fp (Eq. 4) and dL/dS^fp
    adam: bool = False         # backward fused with the AdamW step on c, c^k (and S^fp)
    io: str = ""               # element type of x, y, g, gx ("" = the workload's own)

    @property
    def block(self) -> int:
        return 16 if self.fmt == "nvfp4" else 32

    def phases(self):
        return (["alpha"] if self.fmt == "nvfp4" else []) + ["fwd", "bwd", "pack"]


def bytes_per_elem(case: Case, esz: int) -> dict:
    """Algorithmic bytes per element of each phase (what it must move at
    minimum): x, y, g, gx at `esz` bytes; fp32 coefficients in (and their
    gradients out) per element unless shared by all rows; codes 0.5 B, one
    scale byte per block."""
    coef = 0.0 if case.shared else 4.0 / case.block + 4.0 / case.sub
    sfp = 4.0 / case.block if case.sfp else 0.0     # S^fp in (and dL/dS^fp out)
    # fused AdamW: per learned value p, m, v in and p, m, v out; no gradient
    bwd_params = 6 * (coef + sfp) if case.adam else 2 * (coef + sfp)
    out = {"fwd": 2 * esz + coef + sfp, "bwd": 3 * esz + bwd_params,
           "pack": esz + coef + sfp + 0.5 + 1.0 / case.block}
    if case.fmt == "nvfp4":
        out["alpha"] = float(esz)
    return out


# DRAM traffic (read + write) of the dominant kernel of the default line,
# per element, from one ncu capture of that kernel on a smaller case of the
# same workload (DRAM bytes scale with the elements processed), keyed by
# (workload, format, phase), with the sha256 prefix of the kernel sources it
# was taken on.  Reported only while the sources are unchanged.
TRAFFIC = {
    # fq_block_kernel<1,1,8,2> on [32768, 4096] of the activations: 637.6 MB
    # read + 336.8 MB written for 134,217,728 elements
    # (profiles/fq_bwd_nvfp4_act_32768rows.txt)
    ("act_262144x4096", "nvfp4", "bwd"): {"sources": "42cba47e57d406a3", "bytes_per_elem": 7.2604},
}

# AdamW hyper-parameters of the fused optimizer: the paper's learning rates
# per format (Sec. 4.1: block scale / relaxation coefficients) and PyTorch's
# AdamW defaults, which the paper does not override.  S^fp is learned in the
# linear domain, where an MXFP4 block scale of these weights is about 2^-7;
# Adam's first steps move a parameter by about the learning rate, so the
# MXFP4 scale rate 2e-2 is applied relative to that magnitude.
ADAMW_HP = {"mxfp4": dict(lr_coef=5e-2, lr_scale=2e-2 * 2.0 ** -7, beta1=0.9, beta2=0.999,
                          eps=1e-8, weight_decay=0.01),
            "nvfp4": dict(lr_coef=1e-3, lr_scale=5e-3, beta1=0.9, beta2=0.999, eps=1e-8,
                          weight_decay=0.01)}


# the sources the default backward kernel is compiled from
BWD_SOURCES = ("fq_device.cuh", "fq_kernels.cuh", "fq_launch.h", "fq_inst_bwd_nv.cu")


def kernel_sources_sha() -> str:
    import hashlib
    h = hashlib.sha256()
    for f in sorted(os.path.join(ROOT, "paper_2608_01847_gb300", "csrc", n) for n in BWD_SOURCES):
        h.update(os.path.basename(f).encode())
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """SM clocks, power and throttle reasons of one GPU, sampled every
    `period_s` in a background thread while the benchmark runs, read-only:
    through NVML (the driver's libnvidia-ml, queried with ctypes), else by
    an nvidia-smi child process.  `mark(name)` stamps the host time of a
    moment of the run (after a device synchronize, so the stamps bracket the
    device work); `summary(a, b)` reduces the samples taken between two
    stamps."""
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")
    # NVML clock-event reason bits (nvml.h): SW power cap 0x4, HW slowdown
    # 0x8, SW thermal 0x20, HW thermal 0x40, HW power brake 0x80 (a HW slowdown)
    REASON_BITS = {"hw_slowdown": 0x8 | 0x80, "hw_thermal_slowdown": 0x40,
                   "sw_thermal_slowdown": 0x20, "sw_power_cap": 0x4}

    def __init__(self, index, uuid=None, period_s=0.01):
        self.index, self.uuid, self.period = index, uuid, period_s
        self.samples = []          # (host time, sm MHz, max sm MHz, power W, [reason names])
        self.marks = {}
        self.source = None
        self.error = None
        self._stop = None
        self._thread = None
        self._proc = None

    # -- NVML -------------------------------------------------------------
    def _nvml_open(self):
        import ctypes
        lib = ctypes.CDLL("libnvidia-ml.so.1")
        if lib.nvmlInit_v2() != 0:
            raise OSError("nvmlInit_v2 failed")
        h = ctypes.c_void_p()
        ok = False
        if self.uuid:
            ok = lib.nvmlDeviceGetHandleByUUID(("GPU-" + self.uuid).encode(), ctypes.byref(h)) == 0
        if not ok and lib.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(self.index), ctypes.byref(h)) != 0:
            lib.nvmlShutdown()
            raise OSError("no NVML handle for the device")
        reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            lib.nvmlDeviceGetCurrentClocksThrottleReasons
        return lib, h, reasons_fn

    def _nvml_loop(self, lib, h, reasons_fn):
        import ctypes
        clk, mx, pw, rs = ctypes.c_uint(), ctypes.c_uint(), ctypes.c_uint(), ctypes.c_ulonglong()
        try:
            while not self._stop.is_set():
                if (lib.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0 and
                        lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0 and
                        reasons_fn(h, ctypes.byref(rs)) == 0):
                    power = pw.value / 1000.0 if lib.nvmlDeviceGetPowerUsage(h, ctypes.byref(pw)) == 0 else None
                    names = [n for n, bit in self.REASON_BITS.items() if rs.value & bit]
                    self.samples.append((time.monotonic(), float(clk.value), float(mx.value), power, names))
                self._stop.wait(self.period)
        finally:
            lib.nvmlShutdown()

    # -- nvidia-smi ---------------------------------------------------------
    def _smi_loop(self):
        names = list(self.REASON_BITS)
        for ln in self._proc.stdout:
            f = [v.strip() for v in ln.split(",")]
            if len(f) < 7:
                continue
            try:
                power = float(f[2]) if f[2] not in ("", "[N/A]") else None
                self.samples.append((time.monotonic(), float(f[0]), float(f[1]), power,
                                     [n for n, v in zip(names, f[3:7]) if v.lower() == "active"]))
            except ValueError:
                continue

    def __enter__(self):
        import threading
        self._stop = threading.Event()
        try:
            lib, h, reasons_fn = self._nvml_open()
            self.source = "nvml"
            self._thread = threading.Thread(target=self._nvml_loop, args=(lib, h, reasons_fn), daemon=True)
        except (OSError, AttributeError) as e:
            self.error = f"nvml: {e}"
            try:
                self._proc = subprocess.Popen(
                    ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                     "--format=csv,noheader,nounits", "-lms", str(max(20, int(self.period * 1000)))],
                    stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True)
                self.source = "nvidia-smi"
                self._thread = threading.Thread(target=self._smi_loop, daemon=True)
            except OSError as e2:
                self.error += f"; nvidia-smi: {e2}"
        if self._thread is not None:
            self._thread.start()
        self.mark("start")
        return self

    def __exit__(self, *a):
        self.mark("end")
        if self._stop is not None:
            self._stop.set()
        if self._proc is not None:
            self._proc.terminate()
            try:
                _, err = self._proc.communicate(timeout=5)
                if not self.samples and err:
                    self.error = (self.error or "") + "; nvidia-smi: " + err.strip()[:200]
            except Exception:
                self._proc.kill()
        if self._thread is not None:
            self._thread.join(timeout=5)

    def mark(self, name):
        self.marks[name] = time.monotonic()

    def summary(self, a="start", b="end"):
        t0, t1 = self.marks.get(a, 0.0), self.marks.get(b, float("inf"))
        rows = [r for r in self.samples if t0 <= r[0] <= t1]
        out = {"source": self.source, "window": f"{a}..{b}", "samples": len(rows),
               "period_ms": round(self.period * 1e3, 1)}
        if not rows:
            out.update(sm_mhz=None, sm_max_mhz=None, reasons=["unavailable"])
            if self.error:
                out["error"] = self.error
            return out
        pw = [r[3] for r in rows if r[3] is not None]
        out.update(sm_mhz=statistics.median(r[1] for r in rows), sm_min_mhz=min(r[1] for r in rows),
                   sm_max_mhz=max(r[2] for r in rows),
                   reasons=sorted({n for r in rows for n in r[4]}),
                   power_w_max=round(max(pw), 1) if pw else None)
        return out


def device_uuid(device):
    """The CUDA device's UUID as NVML spells it after "GPU-", or None."""
    try:
        import torch
        u = str(torch.cuda.get_device_properties(device).uuid)
        return u if len(u) >= 32 else None
    except Exception:
        return None


# ----------------------------------------------------------------------------
# multi-rank timing (replicas: no data-path collective)
# ----------------------------------------------------------------------------
def max_over_ranks(ms: float, world: int, device=None) -> float:
    """The slowest rank's time: an all-reduce MAX of one scalar (the only
    collective of the benchmark; it is not part of the timed work)."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate_gbs(bytes_per_rank_step: float, world: int, max_ms_per_step: float) -> float:
    """Whole-job throughput under weak scaling: every rank processes the same
    bytes per step, the job's step time is the slowest rank's."""
    return world * bytes_per_rank_step / (max_ms_per_step * 1e-3) / 1e9


# ----------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------
ARENA_ALIGN = 256


def pack_arena(obj, names, device):
    """Moves the tensor attributes `names` of `obj` into one allocation on
    `device`, in that order, each at an ARENA_ALIGN-byte aligned offset, and
    returns the allocation (uint8); the attributes become views of it with
    their values, shapes and dtypes."""
    import torch
    arrs = [getattr(obj, n) for n in names]
    offs, end = [], 0
    for a in arrs:
        offs.append(end)
        end += -(-a.numel() * a.element_size() // ARENA_ALIGN) * ARENA_ALIGN
    buf = torch.empty(max(end, ARENA_ALIGN), dtype=torch.uint8, device=device)
    for n, a, off in zip(names, arrs, offs):
        v = buf[off:off + a.numel() * a.element_size()].view(a.dtype).view(a.shape)
        v.copy_(a)
        setattr(obj, n, v)
    return buf


def arena_spans(buf, arrays):
    """Byte ranges [start, end) of `buf` that cover `arrays` (views of it),
    neighbours merged (across their alignment padding): the copies that move
    those arrays between `buf` and a mirror of the same layout."""
    base, size = buf.data_ptr(), buf.numel()
    spans = []
    for s, e in sorted((a.data_ptr() - base, a.data_ptr() - base + a.numel() * a.element_size())
                       for a in arrays):
        if s < 0 or e > size:
            raise ValueError("array outside the arena")
        if spans and s - spans[-1][1] < ARENA_ALIGN:
            spans[-1][1] = max(spans[-1][1], e)
        else:
            spans.append([s, e])
    return [tuple(sp) for sp in spans]


class Tensor:
    """Device tensors of one projection (or activation) plus its outputs.
    The inputs a step takes from the host share one allocation, and so do
    the outputs it returns, so that the end-to-end step moves each tensor
    with one copy per direction."""

    def __init__(self, case: Case, w, idx, device, step=None):
        import torch
        from paper_2608_01847_gb300 import focus as F
        from paper_2608_01847_gb300 import workloads as W
        self.fmt = F.FOCUS_NVFP4 if case.fmt == "nvfp4" else F.FOCUS_MXFP4
        self.case = case
        self.x, self.g = W.device_tensor(w, idx, device)
        self.crs, self.dgs = W.device_coefs(w, idx, case.block, case.sub, device, shared=case.shared)
        rows, cols = self.x.shape
        self.n = rows * cols
        self.alpha = torch.zeros(1, dtype=torch.float32, device=device)
        self.y = torch.empty_like(self.x)
        self.gx = torch.empty_like(self.x)
        self.gcrs = torch.empty_like(self.crs)
        self.gdgs = torch.empty_like(self.dgs)
        self.codes = torch.empty((rows, cols // 2), dtype=torch.uint8, device=device)
        self.scales = torch.empty((rows, cols // case.block), dtype=torch.uint8, device=device)
        d = F.make_desc(self.x, self.fmt, case.sub, case.shared)
        self.ws_alpha = torch.empty(max(16, F.focus_workspace_bytes(d, F.FOCUS_WS_ALPHA)),
                                    dtype=torch.uint8, device=device)
        self.ws_bwd = torch.empty(max(16, F.focus_workspace_bytes(d, F.FOCUS_WS_BWD)),
                                  dtype=torch.uint8, device=device)
        self.sfp = self.gsfp = None
        if case.sfp:
            # S^fp initialised via absmax (Sec. 3.2), then moved by U(0.9, 1.1)
            m = self.x.float().abs().view(rows, cols // case.block, case.block).amax(-1)
            if case.fmt == "nvfp4":
                F.focus_nvfp4_alpha(self.x, self.alpha, self.ws_alpha)
                den = self.alpha * 6.0
            else:
                den = torch.full((1,), 6.0, device=device)
            gen = torch.Generator(device=device)
            gen.manual_seed(4242 + idx)
            jit = torch.rand(m.shape, generator=gen, device=device) * 0.2 + 0.9
            self.sfp = (m / den * jit).contiguous()
            self.gsfp = torch.empty_like(self.sfp)
        if case.adam:
            # two synthetic batches alternate, the second's output gradient
            # the negation of the first's, so that a fixed gradient does not
            # drive the parameters out of range over thousands of steps
            self.g_alt = -self.g
            in_names = ("g_alt", "x", "g")   # either batch's (x, g) is one span
        else:
            in_names = ("x", "g", "crs", "dgs") + (("sfp",) if case.sfp else ())
        out_names = ("y", "gx", "codes", "scales", "gcrs", "gdgs") + (("gsfp",) if case.sfp else ())
        self.in_buf = pack_arena(self, in_names, device)
        self.out_buf = pack_arena(self, out_names, device)
        if case.adam:
            # optimizer state resident in HBM; the paper's learning rates
            # (Sec. 4.1)
            self.step = step
            learned = {"crs": self.crs, "dgs": self.dgs}
            if self.sfp is not None:
                learned["sfp"] = self.sfp
            self.moments = {k: (torch.zeros_like(v), torch.zeros_like(v)) for k, v in learned.items()}
            self.hp = ADAMW_HP[case.fmt]

    def run(self, phase, parity=0):
        from paper_2608_01847_gb300 import focus as F
        c = self.case
        if phase == "bwd" and c.adam:
            F.focus_fq_bwd_adamw(self.x, self.g_alt if parity else self.g, self.fmt, self.step,
                                 self.hp, crs=self.crs, dgs=self.dgs, sfp=self.sfp,
                                 moments=self.moments, alpha=self.alpha, sub_block=c.sub,
                                 shared=c.shared, gx=self.gx, ws=self.ws_bwd)
            return
        if phase == "alpha":
            F.focus_nvfp4_alpha(self.x, self.alpha, self.ws_alpha)
        elif phase == "fwd":
            F.focus_fq_fwd(self.x, self.fmt, self.crs, self.dgs, self.alpha, sub_block=c.sub,
                           shared=c.shared, y=self.y, sfp=self.sfp)
        elif phase == "bwd":
            F.focus_fq_bwd(self.x, self.g, self.fmt, self.crs, self.dgs, self.alpha,
                           sub_block=c.sub, shared=c.shared, gx=self.gx, gcrs=self.gcrs,
                           gdgs=self.gdgs, ws=self.ws_bwd, sfp=self.sfp, gsfp=self.gsfp)
        else:
            F.focus_pack(self.x, self.fmt, self.crs, self.dgs, self.alpha, sub_block=c.sub,
                         shared=c.shared, codes=self.codes, scale_bytes=self.scales, sfp=self.sfp)

    def inputs(self, parity=0):
        """Device tensors a step reads from the host (end-to-end leg).  With
        the fused optimizer the parameters and moments stay in HBM."""
        if self.case.adam:
            return (self.x, self.g_alt if parity else self.g)
        return (self.x, self.g, self.crs, self.dgs) + ((self.sfp,) if self.sfp is not None else ())

    def outputs(self):
        """Device tensors a step returns to the host (end-to-end leg)."""
        if self.case.adam:
            return (self.y, self.gx, self.codes, self.scales)
        out = (self.y, self.gx, self.gcrs, self.gdgs, self.codes, self.scales)
        return out + ((self.gsfp,) if self.gsfp is not None else ())

    def launches(self, phase):
        return 2 if phase == "alpha" else (2 if (phase == "bwd" and self.case.shared) else 1)


class GroupRunner:
    """Every phase as one group launch over all tensors of the layer (the
    group entry points); outputs are the Tensor objects' own buffers."""

    def __init__(self, ts, case, device):
        import torch
        from paper_2608_01847_gb300 import focus as F
        self.ts, self.case = ts, case
        self.fmt = ts[0].fmt
        nv = case.fmt == "nvfp4"
        if nv:
            # one alpha array for the layer; each tensor reads its own entry
            self.alphas = torch.zeros(len(ts), dtype=torch.float32, device=device)
            for i, t in enumerate(ts):
                self.alphas[i:i + 1].copy_(t.alpha)
                t.alpha = self.alphas[i:i + 1]
            self.ws = torch.empty(max(16, F.focus_group_workspace_bytes([t.x for t in ts])),
                                  dtype=torch.uint8, device=device)
        common = lambda t: {"x": t.x, "crs": t.crs, "dgs": t.dgs, "alpha": t.alpha if nv else None,
                            "sfp": t.sfp}
        self.fwd = [dict(common(t), y=t.y) for t in ts]
        self.pack = [dict(common(t), codes=t.codes, scale_bytes=t.scales) for t in ts]
        self.bwd = []
        for t in ts:
            d = dict(common(t), g=t.g, gx=t.gx, gcrs=t.gcrs, gdgs=t.gdgs)
            if t.gsfp is not None:
                d["gsfp"] = t.gsfp
            self.bwd.append(d)

    def run(self, phase):
        from paper_2608_01847_gb300 import focus as F
        sub = self.case.sub
        if phase == "alpha":
            F.focus_nvfp4_alpha_group([t.x for t in self.ts], alpha_out=self.alphas, ws=self.ws)
        elif phase == "fwd":
            F.focus_fq_fwd_group(self.fwd, self.fmt, sub_block=sub)
        elif phase == "bwd":
            F.focus_fq_bwd_group(self.bwd, self.fmt, sub_block=sub)
        else:
            F.focus_pack_group(self.pack, self.fmt, sub_block=sub)

    @staticmethod
    def launches(phase):
        return 2 if phase == "alpha" else 1


class SeqGraph:
    """A CUDA graph of `body(stage)` for each stage, in order, on one stream."""

    def __init__(self, body, device, stages):
        import torch
        self.graph = torch.cuda.CUDAGraph()
        cap = torch.cuda.Stream(device)
        cap.wait_stream(torch.cuda.current_stream(device))
        with torch.cuda.graph(self.graph, stream=cap):
            for stage in stages:
                body(stage)
        torch.cuda.current_stream(device).wait_stream(cap)

    def replay(self):
        self.graph.replay()


class BranchGraph:
    """A CUDA graph of one or more stages run in order; in each stage the
    branches (one stream each) run `body(i, stage)` for every tensor i
    independently and join before the next stage."""

    def __init__(self, n, body, device, stages=(None,), before=None):
        import torch
        self.graph = torch.cuda.CUDAGraph()
        side = [torch.cuda.Stream(device) for _ in range(n)]
        cap = torch.cuda.Stream(device)
        cap.wait_stream(torch.cuda.current_stream(device))
        with torch.cuda.graph(self.graph, stream=cap):
            main = torch.cuda.current_stream(device)
            for stage in stages:
                if before is not None:
                    before(stage)
                for i, st in enumerate(side):
                    st.wait_stream(main)
                    with torch.cuda.stream(st):
                        body(i) if stage is None else body(i, stage)
                for st in side:
                    main.wait_stream(st)
        torch.cuda.current_stream(device).wait_stream(cap)

    def replay(self):
        self.graph.replay()


# arrays of a Tensor that hold one row (or one row's coefficients) per row
ROW_ARRAYS = ("x", "g", "g_alt", "y", "gx", "crs", "dgs", "sfp", "gcrs", "gdgs", "gsfp", "codes", "scales")
# outputs that only the forward-side phases (forward, pack) write
FRONT_OUTPUTS = ("y", "codes", "scales")


def tensor_piece(t, r0, r1):
    """Rows [r0, r1) of Tensor t: a shallow copy whose row arrays (and
    moments) are views of t's rows -- the C ABI computes a row range of a
    tensor exactly as the whole call would -- sharing t's alpha and scratch."""
    import copy
    p = copy.copy(t)
    for n in ROW_ARRAYS:
        a = getattr(t, n, None)
        if a is not None:
            setattr(p, n, a[r0:r1])
    if getattr(t, "moments", None) is not None:
        p.moments = {k: (m[r0:r1], v[r0:r1]) for k, (m, v) in t.moments.items()}
    p.n = (r1 - r0) * t.x.shape[1]
    return p


class StagedE2E:
    """End-to-end steps on two sets of device buffers, alternating between
    two streams.  A step is three graphs: its inputs copied from their
    pinned host mirror, each tensor's phases (one branch per tensor), its
    outputs copied to their pinned host mirror.  The input copies of
    consecutive steps run one after another, and so do the output copies,
    so that each direction of the full-duplex link carries one step at a
    time: step k's inputs cross while step k - 1's outputs return, and the
    phases run between them.  A set's next step follows its previous one on
    the set's stream, so no buffer is reused before its outputs have left.
    Only for steps that carry no state from one to the next (no fused
    optimizer): the two sets compute independently."""

    def __init__(self, sets, phases, device):
        import torch
        self.g_in, self.g_cmp, self.g_out = [], [], []
        for ts in sets:
            gi, gc, go = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
            cap = torch.cuda.Stream(device)
            cap.wait_stream(torch.cuda.current_stream(device))
            h2d = d2h = 0
            with torch.cuda.graph(gi, stream=cap):
                for t in ts:
                    for s, e in arena_spans(t.in_buf, t.inputs()):
                        t.in_buf[s:e].copy_(t.host_in[s:e], non_blocking=True)
                        h2d += e - s
            side = [torch.cuda.Stream(device) for _ in ts]
            with torch.cuda.graph(gc, stream=cap):
                main = torch.cuda.current_stream(device)
                for t, st in zip(ts, side):
                    st.wait_stream(main)
                    with torch.cuda.stream(st):
                        for ph in phases:
                            t.run(ph)
                for st in side:
                    main.wait_stream(st)
            with torch.cuda.graph(go, stream=cap):
                for t in ts:
                    for s, e in arena_spans(t.out_buf, t.outputs()):
                        t.host_out[s:e].copy_(t.out_buf[s:e], non_blocking=True)
                        d2h += e - s
            torch.cuda.current_stream(device).wait_stream(cap)
            self.g_in.append(gi)
            self.g_cmp.append(gc)
            self.g_out.append(go)
            self.h2d, self.d2h = h2d, d2h
        self.streams = [torch.cuda.Stream(device) for _ in sets]
        self.inputs_in = [torch.cuda.Event() for _ in sets]
        self.outputs_out = [torch.cuda.Event() for _ in sets]
        self.k = 0

    def fork(self, stream):
        for st in self.streams:
            st.wait_stream(stream)

    def join(self, stream):
        for st in self.streams:
            stream.wait_stream(st)

    def step(self):
        import torch
        n = len(self.streams)
        i, prev = self.k % n, (self.k - 1) % n
        st = self.streams[i]
        with torch.cuda.stream(st):
            if self.k > 0:
                st.wait_event(self.inputs_in[prev])
            self.g_in[i].replay()
            self.inputs_in[i].record(st)
            self.g_cmp[i].replay()
            if self.k > 0:
                st.wait_event(self.outputs_out[prev])
            self.g_out[i].replay()
            self.outputs_out[i].record(st)
        self.k += 1


class PipelineGraph:
    """End-to-end step as a graph of three chained streams: the H2D copies
    of each tensor's inputs, then its phases, then the D2H copies of its
    outputs (the inputs, and the outputs, of a tensor share an allocation
    mirrored by pinned host buffers of the same layout), so that one
    tensor's D2H overlaps the next one's H2D on the full-duplex link.

    A tensor of more than 2 * piece_elems elements (per-row coefficients) is
    moved and computed in row pieces of about piece_elems elements: the
    pieces' forward-side inputs (x and coefficients; NVFP4: all of x first,
    then the coefficients) first, then their upstream gradients; the forward
    and pack of a piece start once its rows have arrived (NVFP4: once all of
    x has, for the per-tensor alpha), its
    values, codes and scale bytes leave while the gradients still arrive,
    and its backward outputs follow its backward.  With the fused optimizer
    the phases keep their order (the pack reads the updated coefficients)."""

    def __init__(self, ts, phases, device, parity=0, before=None, piece_elems=1 << 27):
        import torch
        # the smallest tensor first (short pipeline fill: its H2D runs alone)
        # and the second smallest last (short drain: its D2H runs alone)
        order = sorted(range(len(ts)), key=lambda i: ts[i].n)
        order = order[:1] + order[2:] + order[1:2] if len(order) > 2 else order
        ts = [ts[i] for i in order]
        self.h2d = self.d2h = 0
        self.graph = torch.cuda.CUDAGraph()
        s_in, s_cmp, s_out = (torch.cuda.Stream(device) for _ in range(3))
        cap = torch.cuda.Stream(device)
        cap.wait_stream(torch.cuda.current_stream(device))

        def h2d(t, arrays):
            for s, e in arena_spans(t.in_buf, arrays):
                t.in_buf[s:e].copy_(t.host_in[s:e], non_blocking=True)
                self.h2d += e - s

        def d2h(t, arrays):
            for s, e in arena_spans(t.out_buf, arrays):
                t.host_out[s:e].copy_(t.out_buf[s:e], non_blocking=True)
                self.d2h += e - s

        with torch.cuda.graph(self.graph, stream=cap):
            main = torch.cuda.current_stream(device)
            if before is not None:
                before()
            for st in (s_in, s_cmp, s_out):
                st.wait_stream(main)
            for t in ts:
                rows = t.x.shape[0]
                n_p = 1 if t.case.shared else min(rows, t.n // piece_elems)
                if n_p < 2:
                    with torch.cuda.stream(s_in):
                        h2d(t, t.inputs(parity))
                    s_cmp.wait_stream(s_in)
                    with torch.cuda.stream(s_cmp):
                        for ph in phases:
                            t.run(ph, parity)
                    s_out.wait_stream(s_cmp)
                    with torch.cuda.stream(s_out):
                        d2h(t, t.outputs())
                    continue
                self._pieces(t, n_p, phases, parity, s_in, s_cmp, s_out, h2d, d2h)
            for st in (s_in, s_cmp, s_out):
                main.wait_stream(st)
        torch.cuda.current_stream(device).wait_stream(cap)

    @staticmethod
    def _pieces(t, n_p, phases, parity, s_in, s_cmp, s_out, h2d, d2h):
        import torch
        rows = t.x.shape[0]
        bounds = [rows * k // n_p for k in range(n_p + 1)]
        pcs = [tensor_piece(t, bounds[k], bounds[k + 1]) for k in range(n_p)]
        ids = lambda arrs: {id(a) for a in arrs}
        grad_in = ids((t.g_alt if parity else t.g,) if t.case.adam else (t.g,))
        work = [ph for ph in phases if ph != "alpha"]
        if t.case.adam:
            front, back = work[:work.index("bwd")], work[work.index("bwd"):]
        else:
            front, back = [ph for ph in work if ph != "bwd"], [ph for ph in work if ph == "bwd"]
        front_out = {n for n in FRONT_OUTPUTS if not t.case.adam or n == "y"}
        e_x, e_g, e_f, e_b = ([torch.cuda.Event() for _ in pcs] for _ in range(4))

        in_names = [n for n in ROW_ARRAYS if getattr(t, n, None) is not None and
                    id(getattr(t, n)) in ids(t.inputs(parity))]
        out_names = [n for n in ROW_ARRAYS if getattr(t, n, None) is not None and
                     id(getattr(t, n)) in ids(t.outputs())]
        fwd_in = [n for n in in_names if id(getattr(t, n)) not in grad_in]
        g_in = [n for n in in_names if id(getattr(t, n)) in grad_in]
        # NVFP4: every output waits for the per-tensor alpha, i.e. for all of
        # x, so x crosses first and the pieces' coefficients after it;
        # without alpha a piece's x and coefficients travel together
        x_first = "alpha" in phases and "x" in fwd_in
        e_xall = torch.cuda.Event()
        with torch.cuda.stream(s_in):
            if x_first:
                for p in pcs:
                    h2d(t, [p.x])
                e_xall.record()
            for p, e in zip(pcs, e_x):
                h2d(t, [getattr(p, n) for n in fwd_in if not (x_first and n == "x")])
                e.record()
            for p, e in zip(pcs, e_g):
                h2d(t, [getattr(p, n) for n in g_in])
                e.record()
        with torch.cuda.stream(s_cmp):
            if "alpha" in phases:
                s_cmp.wait_event(e_xall if x_first else e_x[-1])
                t.run("alpha", parity)
            for p, ex, ef in zip(pcs, e_x, e_f):
                s_cmp.wait_event(ex)
                for ph in front:
                    p.run(ph, parity)
                ef.record()
            for p, eg, eb in zip(pcs, e_g, e_b):
                s_cmp.wait_event(eg)
                for ph in back:
                    p.run(ph, parity)
                eb.record()
        with torch.cuda.stream(s_out):
            for p, ef in zip(pcs, e_f):
                s_out.wait_event(ef)
                d2h(t, [getattr(p, n) for n in out_names if n in front_out])
            for p, eb in zip(pcs, e_b):
                s_out.wait_event(eb)
                d2h(t, [getattr(p, n) for n in out_names if n not in front_out])

    def replay(self):
        self.graph.replay()


def gpu_arm(case, args, rank, world, device):
    import torch
    import torch.distributed as dist
    from paper_2608_01847_gb300 import focus as F
    from paper_2608_01847_gb300 import workloads as W

    F.lib()
    w = W.WORKLOADS[case.workload] if case.workload in W.WORKLOADS else W.sweep_workload(
        int(case.workload.split("_")[-1]))
    if case.io:
        w = dataclasses.replace(w, dtype=case.io)
    # the fused optimizer's step counter t, advanced on the device before
    # every backward phase (inside the captured graphs)
    step_t = torch.zeros(1, dtype=torch.int64, device=device) if case.adam else None
    ts = [Tensor(case, w, i, device, step_t) for i in range(len(w.tensors))]
    n_elem = sum(t.n for t in ts)
    esz = ts[0].x.element_size()
    stream = torch.cuda.current_stream(device)
    phases = case.phases()
    torch.cuda.synchronize(device)

    def before(stage):
        if step_t is not None and stage == "bwd":
            step_t.add_(1)

    # per-tensor launches on parallel graph branches (measured fastest on
    # GB300), or with --group the whole layer per phase in one group launch
    grouped = args.group and not (case.shared or case.adam) and len(ts) <= 16
    runner = GroupRunner(ts, case, device) if grouped else None

    # eager warm-up (resolves launch configurations), then capture each phase
    for ph in phases:
        before(ph)
        if grouped:
            runner.run(ph)
        else:
            for t in ts:
                t.run(ph)
    torch.cuda.synchronize(device)
    # Inputs that fit in L2 would stay there between back-to-back steps: then
    # every timed step (and phase) follows a write of twice the L2 size, and
    # the events bracket each step alone; the back-to-back figure is kept as
    # the "L2-resident" one.
    in_bytes = sum(t.x.numel() * t.x.element_size() * 2 for t in ts)
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=device) if in_bytes <= L2_BYTES else None

    # one graph per phase (for the phase split: PHASE_REPS repetitions, or
    # one per flushed replay) and one for the whole step; with the optimizer,
    # one of each per batch parity (alternating batches)
    parities = (0, 1) if case.adam else (0,)
    reps = 1 if flush is not None else PHASE_REPS
    if grouped:
        graphs = {ph: [SeqGraph(runner.run, device, (ph,) * reps)] for ph in phases}
        step_graphs = [SeqGraph(runner.run, device, phases)]
    else:
        graphs = {ph: [BranchGraph(len(ts), lambda i, st: ts[i].run(st[0], st[1]), device,
                                   stages=tuple((ph, (par + r) % len(parities)) for r in range(reps)),
                                   before=lambda st: before(st[0])) for par in parities]
                  for ph in phases}
        if args.staged:
            step_graphs = [BranchGraph(len(ts), lambda i, st, par=par: ts[i].run(st, par), device,
                                       stages=phases, before=before) for par in parities]
        else:
            # each tensor's phases chained on its own branch, no join between
            # phases (the tensors are independent); the optimizer's step
            # counter advances once, before the branches fork
            step_graphs = [BranchGraph(len(ts), lambda i, par=par: [ts[i].run(ph, par) for ph in phases],
                                       device, before=lambda _stage: before("bwd")) for par in parities]
    n_replay = [0]

    def step():
        step_graphs[n_replay[0] % len(parities)].replay()
        n_replay[0] += 1

    # clocks sampled from the warm-up to the end of the phase split; the
    # line's `clocks` covers the timed steps alone
    clk = ClockSampler(device.index if device.index is not None else 0, device_uuid(device))

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(device)

    def timed(run, n):
        """ms of n runs: back to back, or (flush) each after an L2 flush."""
        if flush is None:
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for k in range(n):
                run(k)
            b.record(stream)
            torch.cuda.synchronize(device)
            return a.elapsed_time(b)
        evs = []
        for k in range(n):
            flush.fill_(float(k))
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            run(k)
            b.record(stream)
            evs.append((a, b))
        torch.cuda.synchronize(device)
        return sum(a.elapsed_time(b) for a, b in evs)

    # ---- device-resident timing: K steps ----
    clk.__enter__()
    try:
        for _ in range(args.warmup):
            step()
        barrier()
        clk.mark("timed_start")
        total_ms = timed(lambda k: step(), args.steps)
        barrier()
        clk.mark("timed_end")
        # phase split: each phase graph replayed on its own, timed the same way
        phase_ms = {}
        n_split = max(1, min(args.steps, 100))
        for name, gph in graphs.items():
            phase_ms[name] = timed(lambda k: gph[k % len(parities)].replay(), n_split) * args.steps / n_split / reps
        torch.cuda.synchronize(device)
    finally:
        clk.__exit__()
    clocks = clk.summary("timed_start", "timed_end")
    clocks["run"] = {k: v for k, v in clk.summary().items() if k not in ("source", "period_ms")}
    total_ms = max_over_ranks(total_ms, world, device)
    l2_resident_ms = None
    if flush is not None:
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(args.steps):
            step()
        b.record(stream)
        torch.cuda.synchronize(device)
        l2_resident_ms = max_over_ranks(a.elapsed_time(b), world, device)

    res = dict(n_elem=n_elem, esz=esz, total_ms=total_ms, phase_ms=phase_ms, phase_reps=reps, clocks=clocks,
               l2_flushed=flush is not None, l2_resident_ms=l2_resident_ms,
               ntensors=len(ts), grouped=grouped,
               launches_per_step=(sum(GroupRunner.launches(ph) for ph in phases) if grouped else
                                  sum(t.launches(ph) for t in ts for ph in phases)))
    if args.no_e2e:
        return res

    # ---- end to end through the public API with pinned host buffers ----
    e2e_steps = max(4, min(args.steps, 20))
    e2e_steps += e2e_steps % 2
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for t in ts:
        t.host_in = t.in_buf.cpu().pin_memory()   # every batch's inputs
        t.host_out = torch.empty_like(t.out_buf, device="cpu").pin_memory()
    staged_used = not case.adam and (case.fmt == "nvfp4" or case.shared)
    if staged_used:
        # Steps without the fused optimizer are independent.  Where one step
        # cannot overlap its own input and output copies -- NVFP4, whose
        # outputs all wait for the whole of x (the per-tensor alpha), and
        # coefficients shared by all rows (one piece) -- two buffer sets let
        # step k's inputs cross the link while step k - 1 returns its outputs
        # (StagedE2E).  The second set reads the same pinned inputs and
        # writes its own pinned outputs.  (Per-row MXFP4 pipelines within
        # the step, and measured faster that way: 334 against 293 GB/s over
        # four alternating runs on one box; NVFP4 staged 313 against 298.)
        ts2 = [Tensor(case, w, i, device, None) for i in range(len(w.tensors))]
        for t, t2 in zip(ts, ts2):
            assert t2.in_buf.numel() == t.in_buf.numel() and t2.out_buf.numel() == t.out_buf.numel()
            t2.host_in = t.host_in
            t2.host_out = torch.empty_like(t2.out_buf, device="cpu").pin_memory()
        for ph in phases:   # eager warm-up of the second set's launch configurations
            for t2 in ts2:
                t2.run(ph)
        torch.cuda.synchronize(device)
        staged = StagedE2E([ts, ts2], phases, device)
        h2d, d2h = staged.h2d, staged.d2h
        staged.fork(stream)
        for _ in range(2):
            staged.step()
        staged.join(stream)
        barrier()
        e0.record(stream)
        staged.fork(stream)
        for _ in range(e2e_steps):
            staged.step()
        staged.join(stream)
        e1.record(stream)
        barrier()
    else:
        # One buffer set, each step a three-stage software pipeline captured
        # as one graph (an H2D chain, a compute chain, a D2H chain; tensor
        # k's D2H overlaps tensor k+1's H2D, and a large tensor moves in row
        # pieces).  With the fused optimizer a step updates the parameters
        # the next one reads, so steps cannot overlap.
        e2e_graphs = [PipelineGraph(ts, phases, device, par, before=lambda: before("bwd"))
                      for par in parities]
        h2d, d2h = e2e_graphs[-1].h2d, e2e_graphs[-1].d2h
        e2e_graphs[0].replay()
        if len(parities) > 1:
            e2e_graphs[1].replay()
        barrier()
        e0.record(stream)
        for k in range(e2e_steps):
            e2e_graphs[k % len(parities)].replay()
        e1.record(stream)
        barrier()
    e2e_ms = e0.elapsed_time(e1) / e2e_steps
    e2e_ms = max_over_ranks(e2e_ms, world, device)
    method = ("pinned host buffers, two device buffer sets: step k's inputs cross the host link while "
              "step k-1's outputs return (input, compute and output graphs per step)" if staged_used else
              "pinned host buffers, one device buffer set: one graph per step, H2D, compute and D2H "
              "chains pipelined over tensors and row pieces")
    res.update(e2e_ms=e2e_ms, h2d=h2d, d2h=d2h, e2e_method=method)
    return res


# ----------------------------------------------------------------------------
# oracle (CPU) runs: cpu_baseline leg and the reference arm
# ----------------------------------------------------------------------------
def oracle_step(case, samples):
    """One pass of the oracle's alpha, fwd, bwd, pack over host samples."""
    import numpy as np
    import oracle as O
    fmt = O.NVFP4 if case.fmt == "nvfp4" else O.MXFP4
    for x, g, crs, dgs, sfp in samples:
        a = O.alpha(x) if fmt == O.NVFP4 else 0.0
        kw = dict(crs=crs, dgs=dgs, alpha=a, sub=case.sub, shared=case.shared, sfp=sfp)
        O.fwd(x, fmt, want_scales=False, **kw)
        if case.adam:
            params = {k: v for k, v in (("crs", crs), ("dgs", dgs), ("sfp", sfp)) if v is not None}
            moments = {k: (np.zeros(v.shape, np.float32), np.zeros(v.shape, np.float32))
                       for k, v in params.items()}
            O.bwd_adamw(x, g, fmt, params, moments, ADAMW_HP[case.fmt], 1, alpha=a, sub=case.sub,
                        shared=case.shared)
        else:
            O.bwd(x, g, fmt, want_gsfp=sfp is not None, **kw)
        O.fwd(x, fmt, want_y=False, want_codes=True, **kw)


def oracle_samples(case, rows_per_tensor):
    import numpy as np
    from paper_2608_01847_gb300 import workloads as W
    w = W.WORKLOADS[case.workload]
    if case.io:
        w = dataclasses.replace(w, dtype=case.io)
    out = []
    for i in range(len(w.tensors)):
        x, g = W.host_tensor(w, i, rows=rows_per_tensor)
        crs, dgs = W.host_coefs(w, i, case.block, case.sub, shared=case.shared,
                                rows=rows_per_tensor)
        sfp = None
        if case.sfp:
            # absmax initialisation moved by U(0.9, 1.1), as on the device
            xf = W.bf16_bits_to_f32(x) if x.dtype == np.uint16 else x.astype(np.float32)
            m = np.abs(xf).reshape(x.shape[0], -1, case.block).max(-1)
            den = np.float32(6.0)
            if case.fmt == "nvfp4":
                den = np.float32(m.max() / np.float32(2688.0)) * np.float32(6.0)
            jit = np.random.default_rng(4242 + i).uniform(0.9, 1.1, m.shape).astype(np.float32)
            sfp = np.ascontiguousarray(m / den * jit, dtype=np.float32)
        out.append((x, g, crs, dgs, sfp))
    return out


def calibrate_oracle(case, target_s):
    """Rows per tensor so that one oracle step takes about target_s seconds."""
    probe = oracle_samples(case, 8)
    t0 = time.perf_counter()
    oracle_step(case, probe)
    dt = max(time.perf_counter() - t0, 1e-6)
    from paper_2608_01847_gb300 import workloads as W
    tensors = W.WORKLOADS[case.workload].tensors
    # at most 2^28 elements of the largest tensor (a bounded sample of the
    # 2 GiB activations; every layer's weights fit whole)
    most = min(max(t.rows for t in tensors), max(1, (1 << 28) // max(t.cols for t in tensors)))
    return max(1, min(int(8 * target_s / dt), most))


def sample_elems_and_bytes(case, samples):
    n = sum(s[0].size for s in samples)
    esz = samples[0][0].itemsize
    return n, n * sum(bytes_per_elem(case, esz).values())


# The oracle on every host core: worker k of P runs the oracle, unchanged,
# on rows [R k / P, R (k + 1) / P) of every sampled tensor.  The samples are
# drawn once, in this process, into shared memory that the workers map.  The
# pool is spawned, never forked.
_POOL = {}


def _pool_init(case, specs):
    from multiprocessing import shared_memory
    import numpy as np
    _POOL["case"] = case
    _POOL["shm"] = []
    samples = []
    for tensor in specs:
        arrays = []
        for spec in tensor:
            if spec is None:
                arrays.append(None)
                continue
            name, shape, dtype = spec
            shm = shared_memory.SharedMemory(name=name)
            _POOL["shm"].append(shm)
            arrays.append(np.ndarray(shape, dtype=dtype, buffer=shm.buf))
        samples.append(tuple(arrays))
    _POOL["samples"] = samples


def _row_slice(a, lo, hi, per_row):
    return a if (a is None or not per_row) else a[lo:hi]


def _pool_step(part):
    k, n_parts = part
    case = _POOL["case"]
    sl = []
    for x, g, crs, dgs, sfp in _POOL["samples"]:
        rows = x.shape[0]
        lo, hi = rows * k // n_parts, rows * (k + 1) // n_parts
        if hi > lo:
            sl.append((x[lo:hi], g[lo:hi], _row_slice(crs, lo, hi, not case.shared),
                       _row_slice(dgs, lo, hi, not case.shared), _row_slice(sfp, lo, hi, True)))
    oracle_step(case, sl)
    return k


class OraclePool:
    """The oracle over row slices of `samples` on `procs` spawned processes."""

    def __init__(self, case, samples, procs):
        import concurrent.futures as cf
        import multiprocessing as mp
        from multiprocessing import shared_memory
        import numpy as np
        self.procs = procs
        self.shm, specs = [], []
        for tensor in samples:
            spec = []
            for a in tensor:
                if a is None:
                    spec.append(None)
                    continue
                shm = shared_memory.SharedMemory(create=True, size=max(1, a.nbytes))
                self.shm.append(shm)
                np.ndarray(a.shape, dtype=a.dtype, buffer=shm.buf)[...] = a
                spec.append((shm.name, a.shape, a.dtype.str))
            specs.append(spec)
        self.pool = None
        try:
            self.pool = cf.ProcessPoolExecutor(procs, mp_context=mp.get_context("spawn"), initializer=_pool_init,
                                               initargs=(case, specs))
            self.step()   # every worker has started and mapped the samples
        except BaseException:
            self.close()
            raise

    def step(self):
        list(self.pool.map(_pool_step, [(k, self.procs) for k in range(self.procs)]))

    def close(self):
        if self.pool is not None:
            self.pool.shutdown()
            self.pool = None
        for shm in self.shm:
            shm.close()
            shm.unlink()
        self.shm = []

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()


def pool_fits(samples) -> bool:
    """The samples fit twice into the free shared-memory space (/dev/shm)."""
    need = sum(a.nbytes for t in samples for a in t if a is not None)
    try:
        st = os.statvfs("/dev/shm")
    except OSError:
        return False
    return 2 * need <= st.f_bavail * st.f_frsize


def host_cpu() -> str:
    """The host CPU as the OS names it (lscpu's model name, else the machine)."""
    import platform
    import subprocess
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.split(":")[0].strip() == "Model name":
                return f"{line.split(':', 1)[1].strip()} ({platform.machine()})"
    except (OSError, subprocess.SubprocessError):
        pass
    return platform.machine() or "unknown"


def host_cores() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return max(1, os.cpu_count() or 1)


def cpu_baseline(case, target_s=15.0):
    import oracle as O
    O.build()
    rows = calibrate_oracle(case, target_s)
    samples = oracle_samples(case, rows)
    n, nbytes = sample_elems_and_bytes(case, samples)
    t0 = time.perf_counter()
    oracle_step(case, samples)
    dt1 = time.perf_counter() - t0
    procs = host_cores() if pool_fits(samples) else 1
    if procs > 1:
        times = []
        with OraclePool(case, samples, procs) as pool:
            del samples
            while len(times) < 3 or sum(times) < 2.0:
                t0 = time.perf_counter()
                pool.step()
                times.append(time.perf_counter() - t0)
        dt = sorted(times)[len(times) // 2]
    else:
        times, dt = [dt1], dt1
    return {"value": round(nbytes / dt / 1e9, 6), "unit": "GB/s", "cores": procs, "kind": "oracle",
            "sample": f"first {rows} rows of each tensor of {case.workload} ({n} elements; "
                      f"{'+'.join(case.phases())}), row slices on {procs} processes, median of {len(times)} "
                      f"passes {dt:.2f} s",
            "elems_per_s": round(n / dt, 1), "cpu": host_cpu(),
            "single_thread": {"value": round(nbytes / dt1 / 1e9, 6), "unit": "GB/s", "cores": 1,
                              "seconds": round(dt1, 2)}}


def reference_arm(case, args):
    import oracle as O
    O.build()
    procs = host_cores()
    budget = 150.0 / max(1, args.steps + args.warmup)
    # single-thread seconds per step that the pool turns into about `budget`
    rows = calibrate_oracle(case, min(budget, 20.0) * procs)
    samples = oracle_samples(case, rows)
    n, nbytes = sample_elems_and_bytes(case, samples)
    if procs > 1 and pool_fits(samples):
        pool = OraclePool(case, samples, procs)
        del samples
        run, done = pool.step, pool.close
    else:
        if procs > 1:   # one core after all: a sample sized for one
            procs = 1
            rows = calibrate_oracle(case, min(budget, 20.0))
            samples = oracle_samples(case, rows)
            n, nbytes = sample_elems_and_bytes(case, samples)
        run, done = (lambda: oracle_step(case, samples)), (lambda: None)
    try:
        for _ in range(args.warmup):
            run()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            run()
        dt = (time.perf_counter() - t0) / max(1, args.steps)
    finally:
        done()
    value = nbytes / dt / 1e9
    return {"metric": METRIC, "value": round(value, 6), "unit": "GB/s", "impl": "reference",
            "n_gpus": 0, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(dt * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": {"workload": case.workload, "fmt": case.fmt, "sub_block": case.sub,
                       "shared_coefficients": case.shared, "learnable_sfp": case.sfp,
                       "fused_adamw": case.adam,
                       "sample_rows_per_tensor": rows,
                       "elements_per_step": n},
            "cpu_baseline": {"value": round(value, 6), "unit": "GB/s", "cores": procs, "kind": "oracle",
                             "sample": f"first {rows} rows of each tensor per step, CPU oracle "
                                       f"on row slices in {procs} processes", "cpu": host_cpu()},
            "e2e": {"value": round(value, 6), "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


# ----------------------------------------------------------------------------
# ----------------------------------------------------------------------------
# W4A4 GEMM on the exported operands (tensor cores)
# ----------------------------------------------------------------------------
GEMM_TOKENS = 8192          # activation rows: 4 sequences of 2048 tokens
FP4_PER_BF16 = 13.5 / 2.25  # nominal dense FP4 / BF16 tensor rate of GB300


def gemm_arm(args, device):
    """One step = the layer's projections as W4A4 GEMMs on their exports:
    D[T, out] = A[T, in] W[out, in]^T with A the activations and W the
    weights, both exported by focus_pack_mma (timed region: the GEMMs only,
    bf16 output)."""
    import torch
    from paper_2608_01847_gb300 import focus as F
    from paper_2608_01847_gb300 import workloads as W
    fmt = F.FOCUS_NVFP4 if args.fmt == "nvfp4" else F.FOCUS_MXFP4
    w = W.WORKLOADS[args.workload]
    gen = torch.Generator(device=device)
    gen.manual_seed(4321)
    acts, jobs, flops = {}, [], 0
    for i, t in enumerate(w.tensors):
        wx, _ = W.device_tensor(w, i, device)
        K = t.cols
        if K not in acts:
            a = torch.randn((GEMM_TOKENS, K), generator=gen, device=device).to(torch.bfloat16)
            aa = F.focus_nvfp4_alpha(a) if fmt == F.FOCUS_NVFP4 else None
            acts[K] = (*F.focus_pack_mma(a, fmt, alpha=aa), aa)
            del a
        wa = F.focus_nvfp4_alpha(wx) if fmt == F.FOCUS_NVFP4 else None
        wc, wt = F.focus_pack_mma(wx, fmt, alpha=wa)
        del wx
        d = torch.empty((GEMM_TOKENS, t.rows), dtype=torch.bfloat16, device=device)
        jobs.append((acts[K], (wc, wt, wa), d))
        flops += 2 * GEMM_TOKENS * t.rows * K
    flag = torch.zeros(1, dtype=torch.int32, device=device)

    def step():
        for (ac, at, aa), (wc, wt, wa), d in jobs:
            F.focus_fp4_gemm(fmt, ac, at, wc, wt, aa, wa, d=d, timeout_flag=flag)

    # the projections are independent: in the captured step each GEMM runs on
    # its own graph branch, so that one GEMM's last, partly filled wave of
    # tiles overlaps the next one's first
    side = [torch.cuda.Stream(device) for _ in jobs]

    def step_branches():
        main = torch.cuda.current_stream(device)
        for st, ((ac, at, aa), (wc, wt, wa), d) in zip(side, jobs):
            st.wait_stream(main)
            with torch.cuda.stream(st):
                F.focus_fp4_gemm(fmt, ac, at, wc, wt, aa, wa, d=d, timeout_flag=flag)
        for st in side:
            main.wait_stream(st)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(device)
    # the step's GEMMs as one CUDA graph (no host launch gaps between them)
    graph = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream(device)
    cap.wait_stream(torch.cuda.current_stream(device))
    with torch.cuda.graph(graph, stream=cap):
        (step if args.serial else step_branches)()
    torch.cuda.current_stream(device).wait_stream(cap)
    graph.replay()
    torch.cuda.synchronize(device)
    stream = torch.cuda.current_stream(device)
    with ClockSampler(device.index if device.index is not None else 0, device_uuid(device)) as clk:
        torch.cuda.synchronize(device)
        clk.mark("timed_start")
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            graph.replay()
        e1.record(stream)
        torch.cuda.synchronize(device)
        clk.mark("timed_end")
    ms = e0.elapsed_time(e1) / args.steps
    # dominant launch: the largest projection alone
    big = max(range(len(jobs)), key=lambda j: jobs[j][2].numel() * w.tensors[j].cols)
    (ac, at, aa), (wc, wt, wa), d = jobs[big]
    n_rep = max(3, min(args.steps, 50))
    e0.record(stream)
    for _ in range(n_rep):
        F.focus_fp4_gemm(fmt, ac, at, wc, wt, aa, wa, d=d, timeout_flag=flag)
    e1.record(stream)
    torch.cuda.synchronize(device)
    big_ms = e0.elapsed_time(e1) / n_rep
    big_flops = 2 * GEMM_TOKENS * w.tensors[big].rows * w.tensors[big].cols
    assert int(flag.item()) == 0, "a GEMM wait gave up"
    # context: NVIDIA's block-scaled GEMM (cuBLASLt through torch._scaled_mm)
    # on the same exports and the same largest projection, where the
    # installed torch has the FP4 path (NVFP4 only; alpha applied outside)
    library = None
    if fmt == F.FOCUS_NVFP4 and hasattr(torch, "float4_e2m1fn_x2"):
        try:
            a4, w4 = ac.view(torch.float4_e2m1fn_x2), wc.view(torch.float4_e2m1fn_x2).t()
            sa, sw = at.view(torch.float8_e4m3fn), wt.view(torch.float8_e4m3fn)
            for _ in range(3):
                torch._scaled_mm(a4, w4, sa, sw, out_dtype=torch.bfloat16)
            e0.record(stream)
            for _ in range(n_rep):
                torch._scaled_mm(a4, w4, sa, sw, out_dtype=torch.bfloat16)
            e1.record(stream)
            torch.cuda.synchronize(device)
            lib_ms = e0.elapsed_time(e1) / n_rep
            library = {"call": "torch._scaled_mm (cuBLASLt block-scaled NVFP4, bf16 out) on the same exports",
                       "kernel": w.tensors[big].name,
                       "tflops": round(big_flops / (lib_ms * 1e-3) / 1e12, 1)}
        except (RuntimeError, TypeError, NotImplementedError) as e:
            library = {"unavailable": str(e).splitlines()[0][:160]}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            bf16 = float(json.load(f)["bf16_tflops"])
        peak_kind = "measured bf16 burst x nominal FP4/BF16 ratio 6"
    except Exception:
        bf16, peak_kind = 1900.0, "fallback bf16 x nominal FP4/BF16 ratio 6"
    peak = bf16 * FP4_PER_BF16
    tflops = flops / (ms * 1e-3) / 1e12
    big_tflops = big_flops / (big_ms * 1e-3) / 1e12
    return {
        "metric": "W4A4 FP4 GEMM TFLOP/s on FOCUS exports", "value": round(tflops, 1), "unit": "TFLOP/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "e2m1", "data": "synthetic",
        "config": {"workload": f"{args.workload} projections x {GEMM_TOKENS} tokens", "fmt": args.fmt,
                   "gemms": [[GEMM_TOKENS, t.rows, t.cols] for t in w.tensors], "out": "bf16",
                   "launch": ("the GEMMs one after another in one captured graph (programmatic dependent "
                              "launches)" if args.serial else
                              "one captured graph, each GEMM on its own branch (independent projections)"),
                   "l2": "operands of one GEMM fit in L2 (weights <= 25 MB of codes); outputs stream"},
        "roofline": {"bound": "tensor", "kernel": f"fp4_gemm_kernel ({w.tensors[big].name})",
                     "achieved": round(big_tflops, 1), "peak": round(peak, 1), "peak_kind": peak_kind,
                     "unit": "TFLOP/s", "frac": round(big_tflops / peak, 4), "traffic": None},
        "clocks": clk.summary("timed_start", "timed_end"), "gpu_launches": args.steps * len(jobs),
        **({"library_reference": library} if library is not None else {}),
    }


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=500)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="focus", choices=["focus", "reference"])
    ap.add_argument("--workload", default=None,
                    help="default: act_262144x4096 (qwen3_4b_layer with --gemm)")
    ap.add_argument("--fmt", default="nvfp4", choices=["nvfp4", "mxfp4"])
    ap.add_argument("--sub", type=int, default=8)
    ap.add_argument("--shared", action="store_true", help="coefficients shared by all rows")
    ap.add_argument("--sfp", action="store_true",
                    help="learnable full-precision scales S^fp and their gradient")
    ap.add_argument("--adam", action="store_true",
                    help="backward fused with the AdamW step on the learned arrays")
    ap.add_argument("--io", default="", choices=["", "bf16", "f16", "f32"],
                    help="element type of x, y, g, gx (default: the workload's)")
    ap.add_argument("--staged", action="store_true",
                    help="step graph with a join of all tensors between phases (default: each "
                         "tensor's phases chained on its own branch)")
    ap.add_argument("--group", action="store_true",
                    help="one group launch per phase for all tensors instead of per-tensor launches")
    ap.add_argument("--serial", action="store_true",
                    help="--gemm: the step's GEMMs one after another on one stream instead of on graph branches")
    ap.add_argument("--gemm", action="store_true",
                    help="time the W4A4 FP4 GEMMs of the workload's projections on their exports")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    args = ap.parse_args()
    if args.workload is None:
        args.workload = "qwen3_4b_layer" if args.gemm else Case().workload
    case = Case(args.workload, args.fmt, args.sub, args.shared, args.sfp, args.adam, args.io)
    default_case = case == Case()

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(reference_arm(case, args)))
        return

    args.warmup = max(args.warmup, 3)
    import torch
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=device)
    from __graft_entry__ import build
    if rank == 0:
        build()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
        build()

    if args.gemm:
        if rank == 0:
            print(json.dumps(gemm_arm(args, device)))
        return
    r = gpu_arm(case, args, rank, world, device)
    # the default line also carries the other format on the same workload
    # (device-resident timing only)
    other = None
    if default_case:
        import gc
        gc.collect()
        torch.cuda.empty_cache()
        other_case = dataclasses.replace(case, fmt="mxfp4")
        other = (other_case, gpu_arm(other_case, argparse.Namespace(**{**vars(args), "no_e2e": True}), rank, world, device))
    if rank != 0:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return

    out = device_line(case, r, args, world, default_case)
    if other is not None:
        o = device_line(other[0], other[1], args, world, False)
        out["other_format"] = {k: o[k] for k in ("value", "unit", "ms_per_step", "elems_per_s", "fwd_bwd_gbs",
                                                 "pack_gbs", "phase_gbs", "phase_ms", "roofline", "clocks",
                                                 "gpu_launches")}
        out["other_format"]["config"] = {k: o["config"][k] for k in ("fmt", "sub_block", "coefficients",
                                                                     "bytes_per_elem")}
        out["gpu_launches"] += o["gpu_launches"]
    if "e2e_ms" in r:
        step_bytes = r["n_elem"] * sum(bytes_per_elem(case, r["esz"]).values())
        out["e2e"] = {"value": round(aggregate_gbs(step_bytes, world, r["e2e_ms"]), 2),
                      "unit": "GB/s", "h2d_bytes_per_step": r["h2d"], "d2h_bytes_per_step": r["d2h"]}
    if not args.no_cpu_baseline and world == 1:
        out["cpu_baseline"] = cpu_baseline(case)
    print(json.dumps(out))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def device_line(case, r, args, world, default_case):
    """The JSON line of one device-resident run (gpu_arm's result)."""
    peak, peak_kind = load_peaks()
    K = args.steps
    ms_step = r["total_ms"] / K
    bpe = bytes_per_elem(case, r["esz"])
    step_bytes = r["n_elem"] * sum(bpe.values())
    value = aggregate_gbs(step_bytes, world, ms_step)
    ph = {n: r["phase_ms"][n] / K for n in r["phase_ms"]}
    gbs = {n: r["n_elem"] * bpe[n] / (ph[n] * 1e-3) / 1e9 for n in ph}
    dom = max(ph, key=ph.get)
    fb_bytes = r["n_elem"] * (bpe["fwd"] + bpe["bwd"])
    traffic = None
    tr = TRAFFIC.get((case.workload, case.fmt, dom))
    if default_case and tr is not None and kernel_sources_sha() == tr["sources"]:
        traffic = round(tr["bytes_per_elem"] * r["n_elem"] / r["ntensors"])
    out = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": round(ms_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": case.workload, "tensors": r["ntensors"], "elements": r["n_elem"],
                   "fmt": case.fmt, "io_dtype": case.io or {4: "f32", 2: "bf16"}[r["esz"]],
                   "arithmetic": "binary32 (coefficient gradients in double-binary32)",
                   "sub_block": case.sub,
                   "coefficients": ("shared by all rows" if case.shared else
                                    "per-block CRS + per-sub-block DGS"),
                   "scales": "learnable S^fp (+ dL/dS^fp)" if case.sfp else "absmax",
                   "launch": "one group launch per phase" if r["grouped"] else
                             ("one launch per tensor and phase, tensors on parallel graph branches, "
                              "phases joined" if args.staged else
                              "one launch per tensor and phase, each tensor's phases chained on its "
                              "own graph branch (programmatic dependent launches)"),
                   "step": "+".join(case.phases()) + " over all tensors " +
                           ("(bwd: gx + AdamW on the learned arrays)" if case.adam else
                            "(bwd: gx + gcrs + gdgs)"),
                   "bytes_per_elem": round(sum(bpe.values()), 4),
                   "l2": (f"x+g = {r['n_elem'] * 2 * r['esz'] / 2**20:.0f} MiB fit in L2: L2 flushed "
                          "(2x its size written) before every timed step and phase, events around "
                          "each step" if r["l2_flushed"] else
                          f"inputs larger than L2: x+g = {r['n_elem'] * 2 * r['esz'] / 2**20:.0f} MiB"
                          " per step"),
                   "parallelism": f"replicas x{world}",
                   **({"e2e_method": r["e2e_method"]} if "e2e_method" in r else {}),
                   "phase_split": (f"each phase captured {r['phase_reps']} times in one graph (tensors joined "
                                   "between repetitions), timed per repetition" if r["phase_reps"] > 1 else
                                   "each phase graph timed per replay")},
        "elems_per_s": round(world * r["n_elem"] / (ms_step * 1e-3), 1),
        "fwd_bwd_gbs": round(fb_bytes / ((ph["fwd"] + ph["bwd"]) * 1e-3) / 1e9, 2),
        "pack_gbs": round(gbs["pack"], 2),
        "phase_gbs": {n: round(v, 2) for n, v in gbs.items()},
        "phase_ms": {n: round(v, 4) for n, v in ph.items()},
        "roofline": {"bound": "hbm", "kernel": f"fq_{dom}", "achieved": round(gbs[dom], 2),
                     "peak": peak, "peak_kind": peak_kind, "unit": "GB/s",
                     "frac": round(gbs[dom] / peak, 4), "traffic": traffic,
                     "traffic_unit": "bytes per launch (DRAM read + write)",
                     "algorithmic_bytes": round(r["n_elem"] * bpe[dom] / r["ntensors"])},
        "clocks": r["clocks"],
        "gpu_launches": K * r["launches_per_step"],
    }
    if r.get("l2_resident_ms"):
        out["l2_resident"] = {"value": round(aggregate_gbs(step_bytes, world, r["l2_resident_ms"] / K), 2),
                              "unit": "GB/s", "ms_per_step": round(r["l2_resident_ms"] / K, 4),
                              "note": "steps back to back, inputs left in L2 by the previous step"}
    return out


if __name__ == "__main__":
    main()
