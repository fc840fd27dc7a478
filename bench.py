"""Benchmark of the FOCUS FP4 fake-quantizer hot path on GB300.

One step = one pass of the whole hot path over the Qwen3-4B-shaped decoder
layer (7 bf16 projections, 100.9 M elements), NVFP4 (block 16, E4M3 + fp32
alpha), per-block CRS and per-sub-block (8) DGS coefficients:
  alpha (per tensor)  ->  fake-quant forward  ->  STE backward (input
  gradient + both coefficient gradients)  ->  export pack,
each phase over all 7 tensors before the next (as a calibration step runs
all forwards, then all backwards), inputs resident in HBM.  Each phase is
captured once as a CUDA graph (its 7 tensors on parallel branches) and a
step replays the four graphs in order.  `value` is the
algorithmic bytes of the step (per-element figures below) over the step time.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Under torchrun (N > 1) every rank runs the same workload on its own GPU
(replicas; no data-path collective), the step time is the max over ranks and
`value` sums all ranks' bytes (weak scaling).
"""
from __future__ import annotations

import argparse
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
WORKLOAD = "qwen3_4b_layer"
FMT_NAME = "nvfp4"
SUB = 8
L2_BYTES = 129 * 1024 * 1024

# Algorithmic bytes per element, bf16 I/O, fp32 coefficients, NVFP4 (B = 16),
# sub-block 8: what each phase must move at minimum.
BYTES_PER_ELEM = {
    "alpha": 2.0,                                 # read x
    "fwd": 2 + 2 + 4 / 16 + 4 / 8,                # x, y, c_i, c_i^k        = 4.75
    "bwd": 2 + 2 + 2 + 2 * (4 / 16 + 4 / 8),      # x, g, gx, (c, c^k) in+out = 7.5
    "pack": 2 + 4 / 16 + 4 / 8 + 0.5 + 1 / 16,    # x, c, c^k, codes, scales  = 3.3125
}
STEP_BYTES_PER_ELEM = sum(BYTES_PER_ELEM.values())

# DRAM traffic (read + write) of one backward phase (7 launches) of this
# benchmark, from an ncu launch list (gpu__time_duration, dram__bytes_read,
# dram__bytes_write; --cache-control none), and the sha256 prefix of the
# kernel sources it was taken on.  Reported only while they are unchanged.
BWD_TRAFFIC = {"sources": "7f8d1d796e157d46", "bytes_per_step": 762.1e6}


def kernel_sources_sha() -> str:
    import glob
    import hashlib
    h = hashlib.sha256()
    for f in sorted(glob.glob(os.path.join(ROOT, "paper_2608_01847_gb300", "csrc", "*"))):
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
    """nvidia-smi clocks / throttle reasons sampled during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        for ln in (self.out or "").splitlines():
            f = [s.strip() for s in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                rows.append((float(f[1]), float(f[2]), f[5:9], f[4]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i, v in enumerate(r[2]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# ----------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------
class Layer:
    """Device tensors of one projection plus its preallocated outputs."""

    def __init__(self, w, idx, device):
        import torch
        from paper_2608_01847_gb300 import focus as F
        from paper_2608_01847_gb300 import workloads as W
        self.x, self.g = W.device_tensor(w, idx, device)
        self.crs, self.dgs = W.device_coefs(w, idx, 16, SUB, device)
        rows, cols = self.x.shape
        self.n = rows * cols
        self.alpha = torch.empty(1, dtype=torch.float32, device=device)
        self.y = torch.empty_like(self.x)
        self.gx = torch.empty_like(self.x)
        self.gcrs = torch.empty_like(self.crs)
        self.gdgs = torch.empty_like(self.dgs)
        self.codes = torch.empty((rows, cols // 2), dtype=torch.uint8, device=device)
        self.scales = torch.empty((rows, cols // 16), dtype=torch.uint8, device=device)
        d = F.make_desc(self.x, F.FOCUS_NVFP4, SUB)
        self.ws = torch.empty(max(16, F.focus_workspace_bytes(d, F.FOCUS_WS_ALPHA)),
                              dtype=torch.uint8, device=device)


def phase_alpha(layers):
    from paper_2608_01847_gb300 import focus as F
    for L in layers:
        F.focus_nvfp4_alpha(L.x, L.alpha, L.ws)


def phase_fwd(layers):
    from paper_2608_01847_gb300 import focus as F
    for L in layers:
        F.focus_fq_fwd(L.x, F.FOCUS_NVFP4, L.crs, L.dgs, L.alpha, sub_block=SUB, y=L.y)


def phase_bwd(layers):
    from paper_2608_01847_gb300 import focus as F
    for L in layers:
        F.focus_fq_bwd(L.x, L.g, F.FOCUS_NVFP4, L.crs, L.dgs, L.alpha, sub_block=SUB, gx=L.gx,
                       gcrs=L.gcrs, gdgs=L.gdgs)


def phase_pack(layers):
    from paper_2608_01847_gb300 import focus as F
    for L in layers:
        F.focus_pack(L.x, F.FOCUS_NVFP4, L.crs, L.dgs, L.alpha, sub_block=SUB, codes=L.codes,
                     scale_bytes=L.scales)


PHASES = [("alpha", phase_alpha), ("fwd", phase_fwd), ("bwd", phase_bwd), ("pack", phase_pack)]
LAUNCHES_PER_TENSOR = {"alpha": 2, "fwd": 1, "bwd": 1, "pack": 1}


class PhaseGraph:
    """One phase (alpha, fwd, bwd or pack over all 7 tensors) captured as a
    CUDA graph whose 7 tensors run on parallel branches (one stream each), so
    small tensors fill the GPU alongside large ones."""

    def __init__(self, fn, layers, device):
        import torch
        self.graph = torch.cuda.CUDAGraph()
        side = [torch.cuda.Stream(device) for _ in layers]
        cap = torch.cuda.Stream(device)
        cap.wait_stream(torch.cuda.current_stream(device))
        with torch.cuda.graph(self.graph, stream=cap):
            main = torch.cuda.current_stream(device)
            for L, st in zip(layers, side):
                st.wait_stream(main)
                with torch.cuda.stream(st):
                    fn([L])
            for st in side:
                main.wait_stream(st)
        torch.cuda.current_stream(device).wait_stream(cap)

    def replay(self):
        self.graph.replay()


def gpu_arm(args, rank, world, device):
    import torch
    import torch.distributed as dist
    from paper_2608_01847_gb300 import focus as F
    from paper_2608_01847_gb300 import workloads as W

    F.lib()
    w = W.WORKLOADS[WORKLOAD]
    layers = [Layer(w, i, device) for i in range(len(w.tensors))]
    n_elem = sum(L.n for L in layers)
    stream = torch.cuda.current_stream(device)
    torch.cuda.synchronize(device)

    # eager warm-up (resolves launch configurations), then capture one step
    for name, fn in PHASES:
        fn(layers)
    torch.cuda.synchronize(device)
    graphs = [(name, PhaseGraph(fn, layers, device)) for name, fn in PHASES]

    def step():
        for _, gph in graphs:
            gph.replay()

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(device)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(device)

    # ---- device-resident timing: K graph replays; per-phase events ----
    phase_ms = {n: 0.0 for n, _ in PHASES}
    with ClockSampler(device.index if device.index is not None else 0) as clk:
        barrier()
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for k in range(args.steps):
            step()
        end.record(stream)
        barrier()
    total_ms = start.elapsed_time(end)
    # phase split: each phase graph replayed on its own, timed the same way
    n_split = max(1, min(args.steps, 100))
    for name, gph in graphs:
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(n_split):
            gph.replay()
        b.record(stream)
        torch.cuda.synchronize(device)
        phase_ms[name] = a.elapsed_time(b) * args.steps / n_split
    if world > 1:
        t = torch.tensor([total_ms], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())

    # ---- end to end through the public API with pinned host buffers ----
    e2e_steps = max(1, min(args.steps, 5))
    host_in = [(L.x.cpu().pin_memory(), L.g.cpu().pin_memory(), L.crs.cpu().pin_memory(),
                L.dgs.cpu().pin_memory()) for L in layers]
    host_out = [(torch.empty_like(L.y, device="cpu").pin_memory(),
                 torch.empty_like(L.gx, device="cpu").pin_memory(),
                 torch.empty_like(L.gcrs, device="cpu").pin_memory(),
                 torch.empty_like(L.gdgs, device="cpu").pin_memory(),
                 torch.empty_like(L.codes, device="cpu").pin_memory(),
                 torch.empty_like(L.scales, device="cpu").pin_memory()) for L in layers]
    h2d = sum(sum(t.numel() * t.element_size() for t in h) for h in host_in)
    d2h = sum(sum(t.numel() * t.element_size() for t in h) for h in host_out)

    def e2e_step():
        for L, (hx, hg, hc, hd) in zip(layers, host_in):
            L.x.copy_(hx, non_blocking=True)
            L.g.copy_(hg, non_blocking=True)
            L.crs.copy_(hc, non_blocking=True)
            L.dgs.copy_(hd, non_blocking=True)
        step()
        for L, outs in zip(layers, host_out):
            for h, d in zip(outs, (L.y, L.gx, L.gcrs, L.gdgs, L.codes, L.scales)):
                h.copy_(d, non_blocking=True)

    e2e_step()
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(e2e_steps):
        e2e_step()
    e1.record(stream)
    barrier()
    e2e_ms = e0.elapsed_time(e1) / e2e_steps
    if world > 1:
        t = torch.tensor([e2e_ms], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        e2e_ms = float(t.item())

    return dict(n_elem=n_elem, total_ms=total_ms, phase_ms=phase_ms, clocks=clk.summary(),
                e2e_ms=e2e_ms, h2d=h2d, d2h=d2h, ntensors=len(layers))


# ----------------------------------------------------------------------------
# oracle (CPU) runs: cpu_baseline leg and the reference arm
# ----------------------------------------------------------------------------
def oracle_step(samples):
    """One pass of alpha, fwd, bwd, pack of the oracle over host samples."""
    import oracle as O
    for x, g, crs, dgs in samples:
        a = O.alpha(x)
        O.fwd(x, O.NVFP4, crs=crs, dgs=dgs, alpha=a, sub=SUB, want_scales=False)
        O.bwd(x, g, O.NVFP4, crs=crs, dgs=dgs, alpha=a, sub=SUB)
        O.fwd(x, O.NVFP4, crs=crs, dgs=dgs, alpha=a, sub=SUB, want_y=False, want_codes=True)


def oracle_samples(rows_per_tensor):
    from paper_2608_01847_gb300 import workloads as W
    w = W.WORKLOADS[WORKLOAD]
    out = []
    for i in range(len(w.tensors)):
        x, g = W.host_tensor(w, i, rows=rows_per_tensor)
        crs, dgs = W.host_coefs(w, i, 16, SUB, rows=rows_per_tensor)
        out.append((x, g, crs, dgs))
    return out


def calibrate_oracle(target_s):
    """Rows per tensor so that one oracle step takes about target_s seconds."""
    probe = oracle_samples(8)
    t0 = time.perf_counter()
    oracle_step(probe)
    dt = max(time.perf_counter() - t0, 1e-6)
    rows = int(8 * target_s / dt)
    return max(1, min(rows, 1 << 20))


def cpu_baseline(target_s=15.0):
    import oracle as O
    O.build()
    rows = calibrate_oracle(target_s)
    samples = oracle_samples(rows)
    n = sum(s[0].size for s in samples)
    t0 = time.perf_counter()
    oracle_step(samples)
    dt = time.perf_counter() - t0
    return {"value": round(n * STEP_BYTES_PER_ELEM / dt / 1e9, 6), "unit": "GB/s", "cores": 1,
            "kind": "oracle",
            "sample": f"first {rows} rows of each of the 7 {WORKLOAD} projections "
                      f"({n} elements; alpha+fwd+bwd+pack, single thread), {dt:.1f} s",
            "elems_per_s": round(n / dt, 1)}


def reference_arm(args):
    import oracle as O
    O.build()
    budget = 150.0 / max(1, args.steps + args.warmup)
    rows = calibrate_oracle(min(budget, 20.0))
    samples = oracle_samples(rows)
    n = sum(s[0].size for s in samples)
    for _ in range(args.warmup):
        oracle_step(samples)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_step(samples)
    dt = (time.perf_counter() - t0) / max(1, args.steps)
    value = n * STEP_BYTES_PER_ELEM / dt / 1e9
    return {"metric": METRIC, "value": round(value, 6), "unit": "GB/s", "impl": "reference",
            "n_gpus": 0, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(dt * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": {"workload": WORKLOAD, "fmt": FMT_NAME, "io_dtype": "bf16", "sub_block": SUB,
                       "sample_rows_per_tensor": rows, "elements_per_step": n},
            "cpu_baseline": {"value": round(value, 6), "unit": "GB/s", "cores": 1, "kind": "oracle",
                             "sample": f"first {rows} rows of each projection per step, "
                                       f"single-threaded CPU oracle"},
            "e2e": {"value": round(value, 6), "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


# ----------------------------------------------------------------------------
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="focus", choices=["focus", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(reference_arm(args)))
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

    r = gpu_arm(args, rank, world, device)
    if rank != 0:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return

    peak, peak_kind = load_peaks()
    K = args.steps
    ms_step = r["total_ms"] / K
    step_bytes = r["n_elem"] * STEP_BYTES_PER_ELEM
    value = world * step_bytes / (ms_step * 1e-3) / 1e9
    ph = {n: r["phase_ms"][n] / K for n in r["phase_ms"]}
    gbs = {n: r["n_elem"] * BYTES_PER_ELEM[n] / (ph[n] * 1e-3) / 1e9 for n in ph}
    dom = max(ph, key=ph.get)
    achieved = gbs[dom]
    fb_bytes = r["n_elem"] * (BYTES_PER_ELEM["fwd"] + BYTES_PER_ELEM["bwd"])
    out = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": round(ms_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": WORKLOAD, "tensors": r["ntensors"], "elements": r["n_elem"],
                   "fmt": FMT_NAME, "io_dtype": "bf16", "sub_block": SUB,
                   "coefficients": "per-block CRS + per-sub-block DGS, U(0.9,1.1)",
                   "step": "alpha, fwd, bwd (gx + gcrs + gdgs), pack over all 7 tensors",
                   "bytes_per_elem": round(STEP_BYTES_PER_ELEM, 4),
                   "l2": f"inputs larger than L2: x+g = {r['n_elem'] * 4 / 2**20:.0f} MiB per step",
                   "parallelism": f"replicas x{world}"},
        "elems_per_s": round(world * r["n_elem"] / (ms_step * 1e-3), 1),
        "fwd_bwd_gbs": round(fb_bytes / ((ph["fwd"] + ph["bwd"]) * 1e-3) / 1e9, 2),
        "pack_gbs": round(gbs["pack"], 2),
        "phase_gbs": {n: round(v, 2) for n, v in gbs.items()},
        "phase_ms": {n: round(v, 4) for n, v in ph.items()},
        "roofline": {"bound": "hbm", "kernel": f"fq_{dom}", "achieved": round(achieved, 2),
                     "peak": peak, "peak_kind": peak_kind, "unit": "GB/s",
                     "frac": round(achieved / peak, 4),
                     "traffic": (BWD_TRAFFIC["bytes_per_step"]
                                 if dom == "bwd" and kernel_sources_sha() == BWD_TRAFFIC["sources"]
                                 else None),
                     "traffic_unit": "bytes per phase (7 launches)"},
        "clocks": r["clocks"],
        "e2e": {"value": round(world * step_bytes / (r["e2e_ms"] * 1e-3) / 1e9, 2), "unit": "GB/s",
                "h2d_bytes_per_step": r["h2d"], "d2h_bytes_per_step": r["d2h"]},
        "gpu_launches": K * r["ntensors"] * sum(LAUNCHES_PER_TENSOR.values()),
    }
    if not args.no_cpu_baseline and world == 1:
        out["cpu_baseline"] = cpu_baseline()
    print(json.dumps(out))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
