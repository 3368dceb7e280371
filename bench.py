#!/usr/bin/env python
"""Benchmark of the batched softmax with slice scheduling on GB300.

One step = one pass of the whole hot path over one batch: the scheduler's
persistent kernel pulls every patch of the workload and computes its row
softmax (bsm_softmax through the C ABI, plan cached after the first call;
the plan itself -- topology probe, address map, Sec. 4.1/4.2 steps -- is
built once up front, as the paper's scheduler builds its table once).

Default workload: fp32 softmax over the last dim of 384 slices of 512 x 512
(a 196608 x 512 tensor), values 3*N(0,1) from a fixed seed -- the shape of
the paper's SOFTMAX experiment (Sec. 6).  Inputs (805 MB with the output)
are larger than the 129 MB L2, so no flush is needed between steps.  A
working set under twice the L2 (--workload 1, 256 KB) is timed step by step
instead, with a buffer of twice the L2 written before every step.

Metric: GB/s of algorithmic traffic (every input element read once, every
output element written once) per step; also % of the measured HBM copy
peak and of the 8 TB/s nominal, and slices/s.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 2]
                  [--policy dynamic|cbmf_lb|minimax|rr|cbmf|whole_gpu] [--sweep]
                  [--impl reference]

--impl reference times the double-precision CPU oracle (the only other
implementation of the path) on this machine's host cores, each step a bounded
sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
METRIC = "batched softmax GB/s (read+write) and % of GB300 HBM peak; slices/sec"
KERNEL_SRC = os.path.join(ROOT, "paper_2002_07062_gb300", "csrc", "bsm_kernels.cu")
PROFILE_DIR = os.path.join(ROOT, "profiles")


def measured_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_hash() -> str:
    return hashlib.sha256(open(KERNEL_SRC, "rb").read()).hexdigest()[:16]


def profiled_traffic(workload_k):
    """DRAM bytes per launch of the softmax kernel on workload k (an int), or
    on the case a key names (e.g. "long_fp32_1024KiB"), in steady state
    (consecutive launches, caches not flushed) from a committed ncu summary
    taken on the current kernel source, else None."""
    import glob
    key = "workload%d" % workload_k if isinstance(workload_k, int) else str(workload_k)
    for path in sorted(glob.glob(os.path.join(PROFILE_DIR, "softmax_*.md"))):
        text = open(path).read()
        m_hash = re.search(r"kernel_source_sha256_16:\s*([0-9a-f]{16})", text)
        m_traf = re.search(r"dram_bytes_per_launch_%s:\s*([0-9]+)" % re.escape(key), text)
        if m_hash and m_traf and m_hash.group(1) == kernel_hash():
            return int(m_traf.group(1))
    return None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        time.sleep(0.25)
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        sm_sorted = sorted(sm)
        return {"sm_mhz": sm_sorted[len(sm_sorted) // 2], "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


COLL_DEVICE = "cuda"      # where the timing reduction's tensor lives (NCCL: the GPU)


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def reduce_max_ms(total_ms: float, device=None) -> float:
    """Largest timed-region duration over all ranks (the job's time)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([total_ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_gbs(world_size: int, bytes_per_step: int, steps: int, max_total_ms: float) -> float:
    """Whole-job throughput: every rank processed `steps` batches of
    `bytes_per_step` algorithmic bytes within the slowest rank's time."""
    return world_size * bytes_per_step * steps / (max_total_ms * 1e-3) / 1e9


def policy_code(name: str) -> int:
    from paper_2002_07062_gb300 import bsm
    return bsm.POLICIES[name]


def run_reference(args):
    """The oracle, as it stands, on the host cores: K timed steps, each a
    bounded sample of the workload."""
    import numpy as np
    from oracle import softmax as O
    from paper_2002_07062_gb300 import workload
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    w = workload.config(args.workload)
    cores = os.cpu_count() or 1
    # calibrate on one slice, then size a step so the whole run stays ~2 minutes
    one = workload.slice_sample(w, [0])
    t0 = time.perf_counter()
    O.softmax_batched(one.x, one.offsets, one.rows, one.cols, one.flags, want_f64=False,
                      nthreads=cores)
    t_one = max(time.perf_counter() - t0, 1e-4)
    budget = 120.0 / max(1, args.steps + args.warmup)
    n_sl = int(max(1, min(w.nslices, budget / t_one)))
    samp = workload.slice_sample(w, list(range(n_sl)))
    for _ in range(args.warmup):
        O.softmax_batched(samp.x, samp.offsets, samp.rows, samp.cols, samp.flags,
                          want_f64=False, nthreads=cores)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        O.softmax_batched(samp.x, samp.offsets, samp.rows, samp.cols, samp.flags,
                          want_f64=False, nthreads=cores)
    dt = (time.perf_counter() - t0) / args.steps
    gbs = samp.algorithmic_bytes / dt / 1e9
    line = {
        "impl": "reference", "metric": METRIC, "value": round(gbs, 3), "unit": "GB/s",
        "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(dt * 1e3, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "slices_per_step": n_sl},
        "slices_per_s": round(n_sl / dt, 3),
        "cpu_baseline": {"value": round(gbs, 3), "unit": "GB/s", "cores": cores,
                         "kind": "oracle",
                         "sample": "first %d of %d slices per step" % (n_sl, w.nslices)},
        "e2e": {"value": round(gbs, 3), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def cpu_baseline(w, seconds: float = 10.0):
    """Oracle throughput on a bounded sample of the workload (host cores): the
    first slices, as many as about `seconds` of work allows, repeated until
    at least 2 s have been timed (the whole workload is often much shorter)."""
    from oracle import softmax as O
    from paper_2002_07062_gb300 import workload
    cores = os.cpu_count() or 1
    one = workload.slice_sample(w, [0])
    t0 = time.perf_counter()
    O.softmax_batched(one.x, one.offsets, one.rows, one.cols, one.flags, want_f64=False,
                      nthreads=cores)
    t_one = max(time.perf_counter() - t0, 1e-4)
    n_sl = int(max(1, min(w.nslices, seconds / t_one)))
    samp = workload.slice_sample(w, list(range(n_sl)))
    passes, dt = 0, 0.0
    while dt < 2.0 and passes < 50:
        t0 = time.perf_counter()
        O.softmax_batched(samp.x, samp.offsets, samp.rows, samp.cols, samp.flags,
                          want_f64=False, nthreads=cores)
        dt += time.perf_counter() - t0
        passes += 1
    per = dt / passes
    # and on one core: the first slice(s), about a second
    n1 = int(max(1, min(n_sl, 1.0 / (t_one * cores))))
    samp1 = workload.slice_sample(w, list(range(n1)))
    t0 = time.perf_counter()
    O.softmax_batched(samp1.x, samp1.offsets, samp1.rows, samp1.cols, samp1.flags,
                      want_f64=False, nthreads=1)
    t1 = time.perf_counter() - t0
    return {"value": round(samp.algorithmic_bytes / per / 1e9, 4), "unit": "GB/s",
            "cores": cores, "kind": "oracle",
            "sample": "first %d of %d slices, %d passes, %.3f s per pass (double precision, "
                      "%d threads)" % (n_sl, w.nslices, passes, per, cores),
            "single_thread_value": round(samp1.algorithmic_bytes / t1 / 1e9, 4),
            "single_thread_sample": "first %d slices, one pass, 1 thread" % n1}


def bmm_cpu_baseline(w, seconds: float = 10.0):
    """The batched-product oracle (double-precision matrix product of the
    exactly converted bf16 operands) on a bounded sample of slices."""
    from oracle import bmm_oracle as O
    cores = os.cpu_count() or 1
    a1, b1 = w.operands([0])
    t0 = time.perf_counter()
    O.bmm_f64(a1, b1, 1, w.M, w.N, w.K)
    t_one = max(time.perf_counter() - t0, 1e-4)
    n_sl = int(max(1, min(w.B, seconds / 4 / t_one)))
    sl = list(range(n_sl))
    a, b = w.operands(sl)
    passes, dt = 0, 0.0
    while dt < 2.0 and passes < 20:
        t0 = time.perf_counter()
        O.bmm_f64(a, b, n_sl, w.M, w.N, w.K)
        dt += time.perf_counter() - t0
        passes += 1
    per = dt / passes
    frac = n_sl / w.B
    return {"value": round(w.algorithmic_bytes * frac / per / 1e9, 4), "unit": "GB/s",
            "cores": cores, "kind": "oracle",
            "tflops": round(w.flops * frac / per / 1e12, 5),
            "sample": "first %d of %d slices, %d passes, %.3f s per pass (float64 product, "
                      "numpy's BLAS threads; bf16 rounding of the result not timed)"
                      % (n_sl, w.B, passes, per)}


def profiled_bmm_traffic(k: int):
    """DRAM bytes per launch of the batched-product kernel for Sec. 6 shape k
    from the committed ncu summary, if it was taken on the current source."""
    path = os.path.join(PROFILE_DIR, "bmm_persistent_sec6_shapes.md")
    if not os.path.exists(path):
        return None
    text = open(path).read()
    m_hash = re.search(r"kernel_source_sha256_16:\s*([0-9a-f]{16})", text)
    m_traf = re.search(r"dram_bytes_per_launch_E%d:\s*([0-9]+)" % k, text)
    src = os.path.join(ROOT, "paper_2002_07062_gb300", "csrc", "bsm_bmm.cu")
    if not m_hash or not m_traf or \
            m_hash.group(1) != hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]:
        return None
    return int(m_traf.group(1))


def time_steps(fn, steps, stream, per_launch=False):
    """Run fn() `steps` times on `stream`; returns (total ms, per-step ms list).
    With per_launch, an event pair brackets every step -- which also keeps
    consecutive launches from overlapping, so the timed region uses one event
    pair around all steps."""
    import torch
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)] if per_launch else []
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for k in range(steps):
        if per_launch:
            ev[k][0].record(stream)
        fn()
        if per_launch:
            ev[k][1].record(stream)
    end.record(stream)
    end.synchronize()
    per = [a.elapsed_time(b) for a, b in ev] if per_launch else []
    return start.elapsed_time(end), per


L2_BYTES = 129 * 1000 * 1000          # GB300 L2


def time_steps_flushed(fn, steps, stream, flush_buf):
    """For working sets under twice the L2: before every step, write a buffer
    of twice the L2 on `stream` (evicting the previous step's data), then time
    the step alone with its own event pair.  Returns (sum of the step times in
    ms, per-step ms list)."""
    import torch
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    with torch.cuda.stream(stream):
        for k in range(steps):
            flush_buf.add_(1)
            ev[k][0].record(stream)
            fn()
            ev[k][1].record(stream)
    ev[-1][1].synchronize()
    per = [a.elapsed_time(b) for a, b in ev]
    return sum(per), per


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", type=int, default=2)
    ap.add_argument("--policy", default="dynamic")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--sweep", action="store_true",
                    help="also time every policy on workloads 2-5 (extra JSON lines)")
    ap.add_argument("--bmm", type=int, default=0, choices=[0, 1, 2],
                    help="time the Sec. 6 batched product 1 or 2 instead of the softmax")
    ap.add_argument("--long-rows", type=int, default=0,
                    help="time fp32 rows of this many elements (longer than a stage), 256 MiB in all")
    ap.add_argument("--die-check", action="store_true",
                    help="check the probed address -> die map: each die's SMs read only the "
                         "chunks it maps there (then the inverse, then a random map); one JSON line")
    ap.add_argument("--die-check-dump", default=None,
                    help="with --die-check: also save the maps and the raw probe matrix (.npy/.npz) here")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-workloads", action="store_true",
                    help="skip the other workloads, the policy ratios and the Sec. 6 products "
                         "(nested under 'workloads' in the JSON line)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--slices", type=int, default=0,
                    help="run only the first N slices of the workload (same shapes and values): a "
                         "smaller case of the same kernel, e.g. for a profiler capture of workload 4")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    if args.impl == "reference":
        return run_reference(args)

    import numpy as np
    import torch
    import __graft_entry__ as g
    from paper_2002_07062_gb300 import bsm, workload

    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist
        global COLL_DEVICE
        # one rank per GPU (a rank past the GPU count shares one: only the
        # gloo test of this path does that); the barrier and the max-reduce
        # of the timings go over NCCL (gloo when BSM_BENCH_DIST_BACKEND says so)
        torch.cuda.set_device(local % max(1, torch.cuda.device_count()))
        backend = os.environ.get("BSM_BENCH_DIST_BACKEND", "nccl")
        COLL_DEVICE = "cuda" if backend == "nccl" else "cpu"
        dist.init_process_group(backend)
    else:
        torch.cuda.set_device(0)
    if rank == 0 or ws == 1:
        g.build()
    if ws > 1:
        dist.barrier()
        g.build()
    dev = torch.cuda.current_device()

    if args.die_check:
        return run_die_check(bsm, dev, dump=args.die_check_dump)
    if args.bmm:
        return run_bmm(args, bsm, workload, ws, rank, dev)
    if args.long_rows:
        return run_long_rows(args, bsm, ws, rank, dev)

    w = workload.config(args.workload)
    if 0 < args.slices < w.nslices:
        w = workload.slice_sample(w, list(range(args.slices)))
    w = w.materialize()
    pol = policy_code(args.policy)
    xh = w.x
    x = torch.from_numpy(xh.view(np.int16) if w.dtype == workload.BF16 else xh).cuda()
    if w.dtype == workload.BF16:
        x = x.view(torch.bfloat16)
    y = torch.empty_like(x)
    stream = torch.cuda.Stream()
    uniform = w.uniform
    B, R, C = w.nslices, int(w.rows[0]), int(w.cols[0])

    def step():
        if uniform:
            bsm.bsm_softmax_ex(x, y, B, R, C, w.dtype, pol, w.flags, stream)
        else:
            bsm.bsm_softmax_ragged(x, y, w.offsets, w.rows, w.cols, w.dtype, pol, w.flags, stream)

    # plan once (cached), then the same plan's stats for the launch count
    with torch.cuda.stream(stream):
        step()
    stream.synchronize()
    plan = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, pol, offsets=w.offsets,
                               flags=w.flags)
    st = plan.stats()
    plan.close()
    launches_per_step = int(st["launches"])

    # a working set under twice the L2 (the small parity workload) is timed
    # step by step with the L2 flushed before each step; the others stream
    # more than the L2 holds at every step
    small = w.algorithmic_bytes < 2 * L2_BYTES
    flush_buf = torch.zeros(2 * L2_BYTES // 4, dtype=torch.int32, device="cuda") if small else None

    def timed(fn, n):
        if small:
            return time_steps_flushed(fn, n, stream, flush_buf)
        return time_steps(fn, n, stream)

    # the clock sampler starts first (it needs a moment), then the warm-up
    # steps, so that the timed steps follow busy ones instead of an idle gap
    with ClockSampler(dev) as clk:
        for _ in range(args.warmup):
            step()
        stream.synchronize()
        if ws > 1:
            dist.barrier()
        torch.cuda.synchronize()
        total_ms, _ = timed(step, args.steps)
    torch.cuda.synchronize()
    if ws > 1:
        dist.barrier()
        total_ms = reduce_max_ms(total_ms, device=COLL_DEVICE)
    status = bsm.bsm_device_status()
    # context on this very box: a plain device-to-device copy of the same
    # bytes (x into y: one read and one write of every element), timed the
    # same way; the roofline's peak stays the measured copy bandwidth
    copy_reps = 50

    def copy_step():
        with torch.cuda.stream(stream):
            y.copy_(x)
    for _ in range(3):
        copy_step()
    stream.synchronize()
    copy_ms, _ = timed(copy_step, copy_reps)
    ms = total_ms / args.steps
    bytes_step = w.algorithmic_bytes
    value = job_gbs(ws, bytes_step, args.steps, total_ms)
    peak, peak_src = measured_peak()
    # average duration of one launch of the kernel over the timed region (the
    # step is nothing but its launches)
    launch_ms = total_ms / (args.steps * launches_per_step)
    achieved = bytes_step / launches_per_step / (launch_ms * 1e-3) / 1e9
    # (a sample of the workload's slices has no profiled figure of its own)
    traffic = profiled_traffic(args.workload) if not args.slices else None

    out = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32" if w.dtype == workload.F32 else "bf16", "data": "synthetic",
        "config": {"workload": w.name, "policy": args.policy, "slices": B,
                   "rows": R if uniform else "ragged", "cols": C if uniform else "ragged",
                   "causal": bool(w.flags & 1), "seed": hex(w.seed),
                   "bytes_per_step": bytes_step,
                   "l2": ("working set %d KB under twice the L2: a %d MB buffer written before "
                          "every step, each step timed alone" % (bytes_step >> 10, 2 * L2_BYTES // 10**6)
                          if small else
                          "inputs larger than L2 (%d MB vs 129 MB), no flush" % (bytes_step >> 20)),
                   "parallelism": ("%d ranks, each its own batch of %d slices (weak scaling), "
                                   "no collective on the data path" % (ws, B)) if ws > 1 else "1 GPU"},
        "pct_of_measured_hbm": round(100 * value / ws / peak, 2),
        "pct_of_nominal_8tbs": round(100 * value / ws / NOMINAL_HBM_GBS, 2),
        "slices_per_s": round(ws * B / (ms * 1e-3), 1),
        "gpu_launches": launches_per_step * args.steps,
        "roofline": {"bound": "hbm", "achieved": round(achieved, 2), "peak": peak,
                     "unit": "GB/s", "frac": round(achieved / peak, 4), "traffic": traffic,
                     "peak_source": peak_src, "kernel": "softmax_persistent",
                     "launch_ms": round(launch_ms, 5)},
        "clocks": clk.summary(),
        "copy_context": {"GBps": round(bytes_step / (copy_ms / copy_reps * 1e-3) / 1e9, 2),
                         "what": "torch copy of x into y on the same stream (device to device), "
                                 "same bytes, mean of %d %s copies"
                                 % (copy_reps, "L2-flushed" if small else "back-to-back")},
        "plan": {k: st[k] for k in ("n_items", "n_die", "stage_bytes", "n_stages", "grid",
                                     "moved_items", "overlap_items", "tie_items", "L", "N",
                                     "map_chunk_bytes", "plan_ms", "steal")},
        "device_status": status,
    }

    if not args.no_e2e:
        # end to end through the host-buffer entry point: pinned host input and
        # output, every step copies x in and y out (overlapped in chunks)
        xp = torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
        xp.copy_(x.cpu())
        yp = torch.empty(y.shape, dtype=y.dtype, pin_memory=True)

        def e2e_step():
            if uniform:
                bsm.bsm_softmax_host(xp, yp, B, R, C, w.dtype, pol, w.flags, stream)
            else:
                raise SystemExit("e2e needs a uniform workload")

        for _ in range(3):
            e2e_step()
        stream.synchronize()
        if ws > 1:
            dist.barrier()
        e_ms, _ = time_steps(e2e_step, args.e2e_steps, stream, per_launch=False)
        if ws > 1:
            dist.barrier()
            e_ms = reduce_max_ms(e_ms, device=COLL_DEVICE)
        e_ms /= args.e2e_steps
        nb = x.numel() * x.element_size()
        out["e2e"] = {"value": round(ws * bytes_step / (e_ms * 1e-3) / 1e9, 2), "unit": "GB/s",
                      "h2d_bytes_per_step": nb, "d2h_bytes_per_step": nb,
                      "ms_per_step": round(e_ms, 4), "api": "bsm_softmax_host, pinned host buffers read and written by the kernel over the host link"}
        if ws == 1:
            # beside it, not the e2e figure: the same call on pageable host
            # buffers, which the library stages through its device buffers in
            # chunks (a device-to-host copy into pageable memory blocks the
            # host, so the host times these steps)
            import numpy as np
            xh = xp.view(torch.int32 if x.element_size() == 4 else torch.int16).numpy().copy()
            yh = np.empty_like(xh)
            bsm.bsm_softmax_host(xh, yh, B, R, C, w.dtype, pol, w.flags, stream)
            stream.synchronize()
            n_pg = 3
            t0 = time.perf_counter()
            for _ in range(n_pg):
                bsm.bsm_softmax_host(xh, yh, B, R, C, w.dtype, pol, w.flags, stream)
            stream.synchronize()
            pg_ms = (time.perf_counter() - t0) * 1e3 / n_pg
            out["e2e"]["pageable"] = {
                "value": round(bytes_step / (pg_ms * 1e-3) / 1e9, 2), "unit": "GB/s",
                "ms_per_step": round(pg_ms, 3), "steps": n_pg,
                "api": "bsm_softmax_host, pageable host buffers staged through device buffers in "
                       "48 MiB chunks (host clock)"}
    if not args.no_cpu_baseline and rank == 0 and ws == 1:
        out["cpu_baseline"] = cpu_baseline(w)

    if not args.no_workloads and ws == 1 and args.workload == 2 and args.policy == "dynamic":
        # the paper's policies against its round-robin baseline on this very
        # workload (Sec. 6 SOFTMAX table gives 1.08x for CBMF over RR, on
        # Intel NNP-T), then the other workloads and the Sec. 6 products
        out["policies"] = policy_ratios(bsm, w, x, y, stream)
        del x, y
        torch.cuda.empty_cache()
        out["workloads"] = other_workloads(bsm, workload, stream, dev)

    if rank == 0:
        print(json.dumps(out), flush=True)

    if args.sweep and rank == 0:
        sweep(args, bsm, workload, stream)
    if ws > 1:
        dist.destroy_process_group()
    return 0


def _softmax_tensors(w):
    import numpy as np
    import torch
    from paper_2002_07062_gb300 import workload
    xh = w.x.view(np.int16) if w.dtype == workload.BF16 else w.x
    x = torch.from_numpy(xh).cuda()
    if w.dtype == workload.BF16:
        x = x.view(torch.bfloat16)
    return x, torch.empty_like(x)


def _steps_for(fn, stream, target_s, lo=20, hi=20000, small=False, flush_buf=None):
    """Steps that fill about target_s seconds, from three calibration steps."""
    if small:
        t, _ = time_steps_flushed(fn, 3, stream, flush_buf)
    else:
        t, _ = time_steps(fn, 3, stream)
    per = max(t / 3, 1e-3)
    return int(min(hi, max(lo, target_s * 1e3 / per)))


def time_softmax(bsm, w, x, y, pol, stream, dev, target_s=1.0, clocks=True):
    """One softmax workload under one policy, timed like the main line:
    back-to-back steps under one event pair (working sets over twice the L2),
    or step by step after an L2 flush (smaller ones).  Returns a dict."""
    import torch
    from paper_2002_07062_gb300 import workload
    uniform = w.uniform
    B, R, C = w.nslices, int(w.rows[0]), int(w.cols[0])

    def step():
        if uniform:
            bsm.bsm_softmax_ex(x, y, B, R, C, w.dtype, pol, w.flags, stream)
        else:
            bsm.bsm_softmax_ragged(x, y, w.offsets, w.rows, w.cols, w.dtype, pol, w.flags, stream)
    with torch.cuda.stream(stream):
        step()
    stream.synchronize()
    plan = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, pol, offsets=w.offsets, flags=w.flags)
    st = plan.stats()
    plan.close()
    launches = int(st["launches"])
    small = w.algorithmic_bytes < 2 * L2_BYTES
    flush_buf = torch.zeros(2 * L2_BYTES // 4, dtype=torch.int32, device="cuda") if small else None
    for _ in range(5):
        step()
    stream.synchronize()
    steps = _steps_for(step, stream, target_s, small=small, flush_buf=flush_buf)
    torch.cuda.synchronize()
    if clocks:
        with ClockSampler(dev) as clk:
            for _ in range(3):
                step()
            torch.cuda.synchronize()
            total_ms, _ = (time_steps_flushed(step, steps, stream, flush_buf) if small
                           else time_steps(step, steps, stream))
    else:
        clk = None
        total_ms, _ = (time_steps_flushed(step, steps, stream, flush_buf) if small
                       else time_steps(step, steps, stream))
    ms = total_ms / steps
    gbs = w.algorithmic_bytes / (ms * 1e-3) / 1e9
    peak, peak_src = measured_peak()
    launch_ms = ms / max(1, launches)
    achieved = w.algorithmic_bytes / max(1, launches) / (launch_ms * 1e-3) / 1e9
    out = {"value": round(gbs, 2), "unit": "GB/s", "ms_per_step": round(ms, 5), "steps": steps,
           "dtype": "f32" if w.dtype == workload.F32 else "bf16",
           "slices_per_s": round(B / (ms * 1e-3), 1),
           "config": {"workload": w.name, "policy": bsm.POLICY_NAMES[pol],
                      "bytes_per_step": w.algorithmic_bytes,
                      "l2": ("working set %d KB under twice the L2: a %d MB buffer written before "
                             "every step, each step timed alone"
                             % (w.algorithmic_bytes >> 10, 2 * L2_BYTES // 10**6) if small else
                             "inputs larger than L2 (%d MB vs 129 MB), no flush"
                             % (w.algorithmic_bytes >> 20))},
           "gpu_launches": launches * steps,
           "roofline": {"bound": "hbm", "achieved": round(achieved, 2), "peak": peak,
                        "unit": "GB/s", "frac": round(achieved / peak, 4),
                        "traffic": None, "peak_source": peak_src,
                        "kernel": "softmax_persistent", "launch_ms": round(launch_ms, 5)},
           "device_status": bsm.bsm_device_status()}
    if clk is not None:
        out["clocks"] = clk.summary()
    return out


def policy_ratios(bsm, w, x, y, stream, target_s=0.5):
    """Every policy on the main workload (GB/s), and the ratios of the paper's
    policies to its round-robin baseline, beside the paper's own figure."""
    res = {}
    for name in ("whole_gpu", "rr", "dynamic", "cbmf", "cbmf_lb", "minimax"):
        r = time_softmax(bsm, w, x, y, bsm.POLICIES[name], stream, None, target_s=target_s,
                         clocks=False)
        res[name] = r["value"]
    rr = res["rr"]
    return {"GBps": res,
            "cbmf_over_rr": round(res["cbmf"] / rr, 4),
            "cbmf_lb_over_rr": round(res["cbmf_lb"] / rr, 4),
            "minimax_over_rr": round(res["minimax"] / rr, 4),
            "best_over_rr": round(max(res.values()) / rr, 4),
            "best": max(res, key=res.get),
            "paper_context": {"cbmf_over_rr": 1.08, "what": "HW utilization, CBMF over RR, "
                              "SOFTMAX on 384 slices of 512 x 512", "hardware": "Intel NNP-T",
                              "source": "Sec. 6, SOFTMAX table"}}


def time_bmm(bsm, workload, k, pol, stream, dev, target_s=1.0, clocks=True):
    """A Sec. 6 batched product on the tensor cores: operands resident,
    back-to-back launches, one event pair.  Returns a dict."""
    import numpy as np
    import torch
    w = workload.bmm_config(k)
    a_bits, bt_bits = w.operands()
    a = torch.from_numpy(a_bits.view(np.int16)).cuda()
    bt = torch.from_numpy(bt_bits.view(np.int16)).cuda()
    c = torch.empty(w.B * w.M * w.N, dtype=torch.int16, device="cuda")

    def step():
        bsm.bsm_bmm(a, bt, c, w.B, w.M, w.N, w.K, w.out_dtype, pol, stream)
    for _ in range(5):
        step()
    stream.synchronize()
    steps = _steps_for(step, stream, target_s)
    launches = w.B if pol == bsm.POLICY_WHOLE_GPU else 1
    torch.cuda.synchronize()
    clk = None
    if clocks:
        with ClockSampler(dev) as clk:
            for _ in range(3):
                step()
            stream.synchronize()
            total_ms, _ = time_steps(step, steps, stream)
    else:
        total_ms, _ = time_steps(step, steps, stream)
    ms = total_ms / steps
    gbs = w.algorithmic_bytes / (ms * 1e-3) / 1e9
    peak, peak_src = measured_peak()
    # cuBLAS on the same operands and stream, as context
    A3 = a.view(torch.bfloat16).view(w.B, w.M, w.K)
    B3 = bt.view(torch.bfloat16).view(w.B, w.N, w.K)
    with torch.cuda.stream(stream):
        def lib_step():
            torch.bmm(A3, B3.transpose(1, 2))
        for _ in range(3):
            lib_step()
        stream.synchronize()
        lib_ms = _median_ms(lib_step, 50, stream)
    out = {"value": round(gbs, 2), "unit": "GB/s", "ms_per_step": round(ms, 5), "steps": steps,
           "dtype": "bf16", "tflops": round(w.flops / (ms * 1e-3) / 1e12, 2),
           "config": {"workload": w.name, "policy": bsm.POLICY_NAMES[pol],
                      "bytes_per_step": w.algorithmic_bytes, "flops_per_step": w.flops,
                      "l2": "operands + product %d MB vs 129 MB L2, no flush"
                            % (w.algorithmic_bytes >> 20)},
           "gpu_launches": launches * steps,
           "roofline": {"bound": "hbm", "achieved": round(gbs, 2), "peak": peak, "unit": "GB/s",
                        "frac": round(gbs / peak, 4), "traffic": profiled_bmm_traffic(k),
                        "peak_source": peak_src, "kernel": "bmm_persistent",
                        "launch_ms": round(ms / launches, 5)},
           "torch_bmm_context_ms": round(lib_ms, 5),
           "vs_torch_bmm_time": round(ms / lib_ms, 4),
           "device_status": bsm.bsm_device_status()}
    if clk is not None:
        out["clocks"] = clk.summary()
    del a, bt, c
    return out


def other_workloads(bsm, workload, stream, dev):
    """The other softmax workloads (1, 3, 4, 5) under the default policy and
    both Sec. 6 batched products, each timed like the main line."""
    import torch
    res = {}
    for k in (1, 3, 4, 5):
        w = workload.config(k).materialize()
        x, y = _softmax_tensors(w)
        r = time_softmax(bsm, w, x, y, bsm.POLICY_DYNAMIC, stream, dev)
        r["roofline"]["traffic"] = profiled_traffic(k)
        res["workload%d" % k] = r
        del x, y, w
        torch.cuda.empty_cache()
    for k in (1, 2):
        res["bmm_E%d" % k] = time_bmm(bsm, workload, k, bsm.POLICY_DYNAMIC, stream, dev)
        torch.cuda.empty_cache()
    # rows longer than a shared-memory stage (256 MiB of input each)
    for C, dt, name in ((65536, workload.F32, "fp32_256KiB"), (262144, workload.F32, "fp32_1MiB"),
                        (1048576, workload.F32, "fp32_4MiB"), (65536, workload.BF16, "bf16_128KiB"),
                        (262144, workload.BF16, "bf16_512KiB"), (1048576, workload.BF16, "bf16_2MiB")):
        res["long_rows_" + name] = time_long_rows(bsm, C, dt, stream, dev)
        torch.cuda.empty_cache()
    return res


def sweep(args, bsm, workload, stream):
    """Policy-by-shape sweep: every policy on workloads 2-5 (median of 20)."""
    import numpy as np
    import torch
    for k in (2, 3, 4, 5):
        w = workload.config(k).materialize()
        xh = w.x.view(np.int16) if w.dtype == workload.BF16 else w.x
        x = torch.from_numpy(xh).cuda()
        if w.dtype == workload.BF16:
            x = x.view(torch.bfloat16)
        y = torch.empty_like(x)
        for name in ("whole_gpu", "rr", "dynamic", "cbmf", "cbmf_lb", "minimax"):
            reps = 3 if name == "whole_gpu" and k == 5 else 20
            # rows per patch: as many as fill a stage, or at most 64 / 16
            for rpi in (0, 64, 16):
                med = _sweep_cell(bsm, w, x, y, bsm.POLICIES[name], rpi, reps, stream)
                print(json.dumps({"sweep": True, "workload": w.name, "policy": name,
                                  "rows_per_patch": rpi or "stage", "ms": round(med, 4),
                                  "GBps": round(w.algorithmic_bytes / (med * 1e-3) / 1e9, 2),
                                  "slices_per_s": round(w.nslices / (med * 1e-3), 1)}),
                      flush=True)
        if k in (2, 3, 5):
            # backward pass on the same slices: read y and dy, write dx
            dy = torch.empty_like(x).normal_() if w.dtype == workload.F32 else \
                torch.empty_like(x).normal_()
            dx = torch.empty_like(x)
            bsm.bsm_softmax_ragged(x, y, w.offsets, w.rows, w.cols, w.dtype, bsm.POLICY_DYNAMIC,
                                   w.flags, stream)

            def bstep():
                bsm.bsm_softmax_backward_ragged(y, dy, dx, w.offsets, w.rows, w.cols, w.dtype,
                                                bsm.POLICY_DYNAMIC, stream)
            for _ in range(3):
                bstep()
            stream.synchronize()
            med = _median_ms(bstep, 20, stream)
            nbytes = 3 * w.numel * w.esize
            print(json.dumps({"sweep": True, "op": "backward", "workload": w.name,
                              "policy": "dynamic", "ms": round(med, 4),
                              "GBps": round(nbytes / (med * 1e-3) / 1e9, 2)}), flush=True)
            del dy, dx
        del x, y
        torch.cuda.empty_cache()
    long_row_sweep(bsm, workload, stream)
    bmm_sweep(bsm, workload, stream)


def _moved_factor(st, op="forward"):
    """Bytes a plan moves per algorithmic byte: rows split over groups of CTAs
    and rows staged whole read x once; rows streamed twice read it again
    (forward: 1.5, backward: 5/3 of the algorithmic bytes at most)."""
    if st["group_rows"] and st["group_rows"] == st["long_items"]:
        return 1.0
    return 1.5 if op == "forward" else 5 / 3


def long_row_sweep(bsm, workload, stream):
    """Rows longer than a shared-memory stage: GB/s of algorithmic traffic,
    forward (rows split over groups of CTAs, or streamed twice) and backward
    (streamed twice)."""
    import torch
    for dtype, name in ((workload.F32, "fp32"), (workload.BF16, "bf16")):
        tdt = torch.float32 if dtype == workload.F32 else torch.bfloat16
        es = 4 if dtype == workload.F32 else 2
        for C in (65536, 262144, 1048576):
            R = max(1, (256 << 20) // (C * es))        # 256 MiB of input
            x = torch.randn(R * C, device="cuda").to(tdt)
            y = torch.empty_like(x)
            plan = bsm.bsm_plan_create(x, y, [R], [C], dtype, bsm.POLICY_DYNAMIC)
            st = plan.stats()
            plan.close()

            def step():
                bsm.bsm_softmax(x, y, 1, R, C, dtype, bsm.POLICY_DYNAMIC, stream)
            for _ in range(3):
                step()
            stream.synchronize()
            med = _median_ms(step, 10, stream)
            alg = 2 * R * C * es
            print(json.dumps({"sweep": True, "op": "forward long rows", "workload":
                              "%s %d rows x %d (%d KiB rows)" % (name, R, C, C * es >> 10),
                              "policy": "dynamic", "ms": round(med, 4),
                              "GBps": round(alg / (med * 1e-3) / 1e9, 2),
                              "group_k": st["group_k"], "launches": st["launches"],
                              "moved_GBps": round(_moved_factor(st) * alg / (med * 1e-3) / 1e9, 2)}),
                  flush=True)
            dy = torch.randn(R * C, device="cuda").to(tdt)

            def bstep():
                bsm.bsm_softmax_backward(y, dy, x, 1, R, C, dtype, bsm.POLICY_DYNAMIC, stream)
            for _ in range(3):
                bstep()
            stream.synchronize()
            med = _median_ms(bstep, 10, stream)
            alg = 3 * R * C * es
            print(json.dumps({"sweep": True, "op": "backward long rows", "workload":
                              "%s %d rows x %d (%d KiB rows)" % (name, R, C, C * es >> 10),
                              "policy": "dynamic", "ms": round(med, 4),
                              "GBps": round(alg / (med * 1e-3) / 1e9, 2),
                              "moved_GBps": round(5 / 3 * alg / (med * 1e-3) / 1e9, 2)}), flush=True)
            del x, y, dy
            torch.cuda.empty_cache()


def time_long_rows(bsm, C, dtype, stream, dev, target_s=0.5):
    """Softmax of rows of C elements longer than a shared-memory stage, 256
    MiB of input, the default policy: one entry of the JSON line."""
    import torch
    from paper_2002_07062_gb300 import workload
    es = 4 if dtype == workload.F32 else 2
    R = max(1, (256 << 20) // (C * es))
    g = torch.Generator(device="cuda").manual_seed(0x2002070600 + C + dtype)
    x = torch.randn(R * C, device="cuda", generator=g)
    if dtype == workload.BF16:
        x = x.to(torch.bfloat16)
    y = torch.empty_like(x)
    plan = bsm.bsm_plan_create(x, y, [R], [C], dtype, bsm.POLICY_DYNAMIC)
    st = plan.stats()

    def step():
        plan.execute(stream)
    for _ in range(5):
        step()
    stream.synchronize()
    steps = _steps_for(step, stream, target_s)
    with ClockSampler(dev) as clk:
        for _ in range(3):
            step()
        stream.synchronize()
        total_ms, _ = time_steps(step, steps, stream)
    ms = total_ms / steps
    alg = 2 * R * C * es
    peak, peak_src = measured_peak()
    gbs = alg / (ms * 1e-3) / 1e9
    plan.close()
    kernel = "softmax_group" if st["group_rows"] else "softmax_persistent (long rows)"
    return {"value": round(gbs, 2), "unit": "GB/s", "ms_per_step": round(ms, 5), "steps": steps,
            "dtype": "f32" if dtype == workload.F32 else "bf16",
            "config": {"workload": "%s %d rows x %d (%d KiB rows), 256 MiB, random normal"
                                   % ("fp32" if dtype == workload.F32 else "bf16", R, C, C * es >> 10),
                       "policy": "dynamic", "bytes_per_step": alg,
                       "l2": "inputs larger than L2 (256 MiB vs 129 MB), no flush"},
            "plan": {"group_k": st["group_k"], "n_groups": st["n_groups"], "launches": st["launches"],
                     "stage_bytes": st["stage_bytes"]},
            "gpu_launches": int(st["launches"]) * steps,
            "roofline": {"bound": "hbm", "achieved": round(gbs, 2), "peak": peak, "unit": "GB/s",
                         "frac": round(gbs / peak, 4),
                         "traffic": profiled_traffic("long_%s_%dKiB" % ("fp32" if dtype == workload.F32
                                                                        else "bf16", C * es >> 10))
                         if st["launches"] == 1 else None,
                         "peak_source": peak_src,
                         "kernel": kernel, "launch_ms": round(ms / max(1, st["launches"]), 5),
                         "moved_bytes_per_step": int(_moved_factor(st) * alg)},
            "clocks": clk.summary(), "device_status": bsm.bsm_device_status()}


def run_bmm(args, bsm, workload, ws, rank, dev):
    """One JSON line for a Sec. 6 batched product on the tensor cores
    (operands resident, back-to-back launches, one event pair)."""
    import numpy as np
    import torch
    w = workload.bmm_config(args.bmm)
    a_bits, bt_bits = w.operands()
    a = torch.from_numpy(a_bits.view(np.int16)).cuda()
    bt = torch.from_numpy(bt_bits.view(np.int16)).cuda()
    c = torch.empty(w.B * w.M * w.N, dtype=torch.int16, device="cuda")
    stream = torch.cuda.Stream()
    pol = policy_code(args.policy)

    def step():
        bsm.bsm_bmm(a, bt, c, w.B, w.M, w.N, w.K, w.out_dtype, pol, stream)
    for _ in range(max(3, args.warmup)):
        step()
    stream.synchronize()
    launches = w.B if pol == bsm.POLICY_WHOLE_GPU else 1
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()
    with ClockSampler(dev) as clk:
        for _ in range(3):
            step()
        stream.synchronize()
        total_ms, _ = time_steps(step, args.steps, stream)
    torch.cuda.synchronize()
    if ws > 1:
        dist.barrier()
        total_ms = reduce_max_ms(total_ms, device=COLL_DEVICE)
    ms = total_ms / args.steps
    gbs = w.algorithmic_bytes / (ms * 1e-3) / 1e9          # per GPU (the roofline)
    peak, peak_src = measured_peak()
    out = {"metric": "batched matmul GB/s (operands read + product written)",
           "value": round(job_gbs(ws, w.algorithmic_bytes, args.steps, total_ms), 2),
           "unit": "GB/s", "n_gpus": ws, "steps": args.steps, "warmup": max(3, args.warmup),
           "ms_per_step": round(ms, 5), "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
           "config": {"workload": w.name, "policy": args.policy, "bytes_per_step": w.algorithmic_bytes,
                      "flops_per_step": w.flops,
                      "l2": "operands + product %d MB vs 129 MB L2, no flush" % (w.algorithmic_bytes >> 20)},
           "tflops": round(w.flops / (ms * 1e-3) / 1e12, 2),
           "gpu_launches": launches * args.steps,
           "roofline": {"bound": "hbm", "achieved": round(gbs, 2), "peak": peak, "unit": "GB/s",
                        "frac": round(gbs / peak, 4), "traffic": profiled_bmm_traffic(args.bmm),
                        "peak_source": peak_src,
                        "kernel": "bmm_persistent", "launch_ms": round(ms / launches, 5)},
           "clocks": clk.summary(), "device_status": bsm.bsm_device_status()}
    if not args.no_cpu_baseline and rank == 0 and ws == 1:
        out["cpu_baseline"] = bmm_cpu_baseline(w)
    if rank == 0:
        print(json.dumps(out), flush=True)
    return 0


def run_long_rows(args, bsm, ws, rank, dev):
    """One JSON line for fp32 rows longer than a shared-memory stage (256 MiB
    of input, dynamic policy): GB/s of algorithmic traffic (x read once, y
    written once) and of the bytes the two passes move (x read twice)."""
    import torch
    C = args.long_rows
    R = max(1, (256 << 20) // (4 * C))
    g = torch.Generator(device="cuda").manual_seed(0x2002070600 + C)
    x = torch.randn(R * C, device="cuda", generator=g)
    y = torch.empty_like(x)
    stream = torch.cuda.Stream()
    plan = bsm.bsm_plan_create(x, y, [R], [C], bsm.F32, bsm.POLICY_DYNAMIC)
    st = plan.stats()

    def step():
        plan.execute(stream)
    for _ in range(max(3, args.warmup)):
        step()
    stream.synchronize()
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()
    with ClockSampler(dev) as clk:
        for _ in range(3):
            step()
        stream.synchronize()
        total_ms, _ = time_steps(step, args.steps, stream)
    torch.cuda.synchronize()
    if ws > 1:
        dist.barrier()
        total_ms = reduce_max_ms(total_ms, device=COLL_DEVICE)
    ms = total_ms / args.steps
    alg = 2 * R * C * 4
    out = {"metric": "softmax of rows longer than a stage, GB/s (read+write)",
           "value": round(job_gbs(ws, alg, args.steps, total_ms), 2), "unit": "GB/s", "n_gpus": ws,
           "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": round(ms, 5),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
           "data": "synthetic", "config": {"workload": "fp32 %d rows x %d" % (R, C),
                                           "policy": "dynamic", "bytes_per_step": alg},
           "moved_GBps": round(_moved_factor(st) * alg / (ms * 1e-3) / 1e9, 2),
           "gpu_launches": int(st["launches"]) * args.steps,
           "plan": {k: st[k] for k in ("n_items", "long_items", "launches", "stage_bytes", "n_stages",
                                       "group_rows", "group_k", "n_groups")},
           "clocks": clk.summary(), "device_status": bsm.bsm_device_status()}
    plan.close()
    if rank == 0:
        print(json.dumps(out), flush=True)
    return 0


def run_die_check(bsm, dev, dump=None):
    """The Sec. 4.1 bank map on GB300 (address -> die, probed by latency),
    checked by its consequence: reading only the chunks mapped to the reader's
    own die.  For each grouping of the SMs -- the probe's dies, then the two
    halves of the %smid range, even / odd %smid, and even / odd TPC (pairs of
    %smid) -- a map of the buffer at 128 B (the L2 line) is taken by timing
    every line from an SM of each group, and die_check_kernel runs twice: each
    group's SMs read the lines mapped to their group, then the others.  A
    random map of the buffer (probe's grouping) is the control.  A profiler's
    lts__t_sectors_srcunit_ltcfabric / lts__t_sectors_srcunit_tex on these
    launches is the share of the traffic that crossed dies: near 0 and near 1
    for a grouping and map that match the chip, near 0.5 otherwise.  Also: how
    often the majority rule puts a 64 KiB patch on group 0, against what the
    map's group-0 share would give if every line were an independent draw."""
    import math
    import numpy as np
    import torch
    topo = bsm.bsm_topology_probe()
    if not topo["separable"]:
        print(json.dumps({"die_check": "topology not separable"}))
        return 0
    n_sm = topo["n_sm"]
    nbytes = 256 << 20                     # larger than the L2: every read streams from DRAM
    g = torch.Generator(device="cuda").manual_seed(0xD1E)
    buf = torch.randint(-2**31, 2**31 - 1, (nbytes // 4,), device="cuda", dtype=torch.int32,
                        generator=g)
    want = int(np.bitwise_xor.reduce(buf.cpu().numpy().view(np.uint32)))
    sm = np.arange(bsm.MAX_SM)
    probe = np.array(topo["sm_die"], np.int8)
    groupings = {"probe": probe,
                 "smid halves": np.where(sm < n_sm, (sm >= n_sm // 2).astype(np.int8), -1),
                 "smid parity": np.where(sm < n_sm, (sm % 2).astype(np.int8), -1),
                 "tpc parity": np.where(sm < n_sm, ((sm // 2) % 2).astype(np.int8), -1)}
    out = {"die_check": True, "buffer_bytes": nbytes, "sm_per_die": topo["sm_per_die"][:2],
           "granularity": topo["granularity"], "l_near": round(topo["l_near"], 1),
           "l_far": round(topo["l_far"], 1), "probe_grouping": "".join(
               str(int(v)) for v in probe[:n_sm]), "launches": []}
    lines = (64 << 10) // 128
    for name, grp in groupings.items():
        grp = grp.astype(np.int8)
        m = bsm.bsm_addr_group_map(buf, nbytes, 128, grp)
        m2 = bsm.bsm_addr_group_map(buf, nbytes, 128, grp)
        p = float(np.mean(m == 0))
        per = m.reshape(-1, lines)
        maj0 = float(np.mean((per == 0).sum(axis=1) > lines // 2))
        z = (0.5 - p) * math.sqrt(lines) / math.sqrt(max(p * (1 - p), 1e-12))
        entry = {"grouping": name, "share_group0": round(p, 5),
                 "agreement_of_two_maps": round(float(np.mean(m == m2)), 5),
                 "patches_64k_majority_group0": round(maj0, 4),
                 "binomial_prediction": round(0.5 * math.erfc(z / math.sqrt(2)), 4)}
        for inv in (False, True):
            got, ms = bsm.bsm_die_check_read(buf, nbytes, 128, m, invert=inv, sm_group=grp)
            entry["inverse" if inv else "map"] = {"ms": round(ms, 4), "covers_once": got == want}
        out["launches"].append(entry)
        if dump:
            np.save(os.path.join(dump, "map_%s.npy" % name.replace(" ", "_")), m)
    rnd = np.random.default_rng(7).integers(0, 2, nbytes // 128).astype(np.int8)
    got, ms = bsm.bsm_die_check_read(buf, nbytes, 128, rnd)
    out["launches"].append({"grouping": "probe", "random map": {"ms": round(ms, 4),
                                                               "covers_once": got == want}})
    if dump:
        # the raw probe matrix: cycles of an L2-hit load from every SM to 3072
        # lines (2048 consecutive, 1024 spread over 30 MiB) of the probe buffer
        off = np.concatenate([128 * np.arange(2048),
                              (1 << 20) + 30 * 1024 * np.arange(1024) + 128 * (np.arange(1024) % 8)])
        lat, seen = bsm.bsm_probe_latency(off, reps=8)
        np.savez(os.path.join(dump, "probe_matrix.npz"), lat=lat, seen=seen, off=off)
    out["device_status"] = bsm.bsm_device_status()
    print(json.dumps(out), flush=True)
    return 0

def _sweep_cell(bsm, w, x, y, pol, rpi, reps, stream):
    """Median ms of one policy on one workload, timed on a plan (one C call
    per execute, so that the host never paces the kernels); rpi > 0 caps the
    rows per patch, 0 lets patches fill a stage."""
    plan = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, pol, offsets=w.offsets,
                               flags=w.flags, rows_per_item=rpi)

    def step():
        plan.execute(stream)
    for _ in range(3):
        step()
    stream.synchronize()
    med = _median_ms(step, reps, stream)
    plan.close()
    return med


def _median_ms(fn, reps, stream, rounds=5):
    """Median over `rounds` of the mean time of `reps` back-to-back calls."""
    import numpy as np
    return float(np.median([time_steps(fn, reps, stream)[0] / reps for _ in range(rounds)]))


def bmm_sweep(bsm, workload, stream):
    """The batched products of Sec. 6 on the tensor cores under every policy,
    with torch.bmm (cuBLAS) on the same operands as context."""
    import torch
    for k in (1, 2):
        w = workload.bmm_config(k)
        a_bits, bt_bits = w.operands()
        import numpy as np
        a = torch.from_numpy(a_bits.view(np.int16)).cuda()
        bt = torch.from_numpy(bt_bits.view(np.int16)).cuda()
        c = torch.empty(w.B * w.M * w.N, dtype=torch.int16, device="cuda")
        for name in ("whole_gpu", "rr", "dynamic", "cbmf", "cbmf_lb", "minimax"):
            pol = bsm.POLICIES[name]

            def step():
                bsm.bsm_bmm(a, bt, c, w.B, w.M, w.N, w.K, w.out_dtype, pol, stream)
            for _ in range(3):
                step()
            stream.synchronize()
            med = _median_ms(step, 5 if name == "whole_gpu" else 50, stream)
            print(json.dumps({"sweep": True, "op": "bmm", "workload": w.name, "policy": name,
                              "ms": round(med, 5),
                              "GBps": round(w.algorithmic_bytes / (med * 1e-3) / 1e9, 2),
                              "TFLOPs": round(w.flops / (med * 1e-3) / 1e12, 2)}), flush=True)
        A3 = a.view(torch.bfloat16).view(w.B, w.M, w.K)
        B3 = bt.view(torch.bfloat16).view(w.B, w.N, w.K)
        with torch.cuda.stream(stream):
            def lib_step():
                torch.bmm(A3, B3.transpose(1, 2))
            for _ in range(3):
                lib_step()
            stream.synchronize()
            med = _median_ms(lib_step, 50, stream)
        print(json.dumps({"sweep": True, "op": "bmm", "workload": w.name,
                          "policy": "torch.bmm (cuBLAS), context only", "ms": round(med, 5),
                          "GBps": round(w.algorithmic_bytes / (med * 1e-3) / 1e9, 2),
                          "TFLOPs": round(w.flops / (med * 1e-3) / 1e12, 2)}), flush=True)
        del a, bt, c


if __name__ == "__main__":
    sys.exit(main())
