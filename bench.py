"""Benchmark of the signed-symmetric few-bit weight path on GB300.

One step = one pass of the whole hot path over one batch of synthetic input,
on Llama3-8B-shaped linear layers (q/o 4096x4096, k/v 1024x4096, gate/up
14336x4096, down 4096x14336), signed absmax grid, group 32:

  quantize  one layer's fresh fp32 weights (218.1M weights) at q = 4, 3, 2;
  GEMV      a batch-1 decode pass over a resident 32-layer packed stack at
            each of q = 4, 3, 2 (224 matrices, 9.2 GB of packed weights),
            launched per layer as a decoder can: {q,k,v} fused, o, {gate,up}
            fused, down (384 launches, programmatic dependent launch);
  GEMM      a 512-token prefill over the q=4 layer just quantized.

The headline value is the packed-weight GEMV throughput (algorithmic bytes:
codes + scales + x + y, per launch) in GB/s over the GEMV phases of the
timed steps; the quantizer (Gweights/s) and GEMM (TFLOP/s) are reported in
"phases".  Inputs are larger than L2 (the stack alone is 9.2 GB).  Each phase
is a CUDA graph; phases are timed with CUDA events on the launching stream.

`--impl reference` times the CPU oracle (the plain C reference the tests
check against) on the host cores on a bounded sample of the same workload.

Launch:  python bench.py [--gpus N] [--steps K] [--warmup W]
         torchrun --nproc-per-node N bench.py --gpus N ...   (one replica per GPU)
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

MEASURED_PEAKS = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0
QS = (4, 3, 2)
GROUP = 32
GEMM_M = 512
METRIC = ("packed-weight GEMV GB/s at batch 1 (Llama3-8B-shaped layers, q in {2,3,4}, "
          "group 32, signed symmetric); quantize Gweights/s and GEMM TFLOP/s in phases")


def peaks():
    try:
        with open(MEASURED_PEAKS) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), float(
            p.get("bf16_tflops_sustained", p["bf16_tflops"])), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS, 1700.0, "fallback"


def dist_info():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def reduce_max(values, device):
    """Element-wise max of `values` over all ranks (identity when the
    process group is absent or has one rank): every time the driver sees is
    the slowest rank's."""
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]


def job_rate(units_per_rank: float, world: int, steps: int, ms: float) -> float:
    """Whole-job throughput: the units all `world` replicas processed over
    `steps` steps, divided by the (max-over-ranks) time `ms`, per second."""
    return world * units_per_rank * steps / (ms * 1e-3)


def traffic_from_profiles(name: str):
    """dram bytes per launch recorded in profiles/<name> (line
    'traffic_bytes_per_launch: <int>'), or None."""
    path = os.path.join(ROOT, "profiles", name)
    try:
        for line in open(path):
            if line.strip().startswith("traffic_bytes_per_launch:"):
                v = line.split(":", 1)[1].strip()
                return None if v in ("", "null", "None") else float(v)
    except OSError:
        pass
    return None


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# ---------------------------------------------------------------------------
# workload
# ---------------------------------------------------------------------------

class Workload:
    def __init__(self, layers: int, seed_base: int = 0):
        import torch

        from paper_2607_08779_gb300 import inputs, sss

        self.torch, self.sss, self.inputs = torch, sss, inputs
        self.layers = layers
        self.shapes = list(inputs.LLAMA3_8B_LAYER.items())
        dev = "cuda"
        G = sss.GRID_SIGNED_SYM
        # resident packed stacks, one per q
        self.stack = {q: [[sss.empty_qtensor(n, k, q, GROUP, G) for _, (n, k) in self.shapes]
                          for _ in range(layers)] for q in QS}
        # fresh fp32 layers for the quantize phase (two, alternating), and
        # the packed outputs of that phase
        self.fresh = [[torch.empty((n, k), dtype=torch.float32, device=dev)
                       for _, (n, k) in self.shapes] for _ in range(2)]
        self.fresh_q = {q: [sss.empty_qtensor(n, k, q, GROUP, G) for _, (n, k) in self.shapes]
                        for q in QS}
        tmp = [torch.empty((n, k), dtype=torch.float32, device=dev) for _, (n, k) in self.shapes]
        for layer in range(layers):
            for mi, (name, (n, k)) in enumerate(self.shapes):
                inputs.student_t_weights_cuda(n, k, inputs.weight_seed(2, layer, mi) + seed_base,
                                              out=tmp[mi])
                for q in QS:
                    sss.sss_quantize(tmp[mi], q, GROUP, G, out=self.stack[q][layer][mi])
        for f in range(2):
            for mi, (name, (n, k)) in enumerate(self.shapes):
                inputs.student_t_weights_cuda(n, k, inputs.weight_seed(3, 100 + f, mi) + seed_base,
                                              out=self.fresh[f][mi])
        del tmp
        # activations and outputs
        ks = sorted({k for _, (n, k) in self.shapes})
        self.x = {k: inputs.normal_bf16_cuda((1, k), 7 + k + seed_base) for k in ks}
        self.X = {k: inputs.normal_bf16_cuda((GEMM_M, k), 11 + k + seed_base) for k in ks}
        self.y = [torch.empty((1, n), dtype=torch.float32, device=dev) for _, (n, k) in self.shapes]
        self.Y = [torch.empty((GEMM_M, n), dtype=torch.float32, device=dev)
                  for _, (n, k) in self.shapes]
        # one workspace per group of matrices sharing X (the GEMM phase runs
        # each group as one sss_gemm_multi call)
        idx = {name: i for i, (name, _) in enumerate(self.shapes)}
        self.ws = []
        for grp in self.GROUPS:
            need = sss.sss_gemm_multi_workspace_bytes([self.fresh_q[4][idx[nm]] for nm in grp],
                                                      GEMM_M)
            self.ws.append(torch.empty(max(need, 16), dtype=torch.uint8, device=dev))
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        torch.cuda.synchronize()

        # algorithmic work per step: per launch, the codes and scales of its
        # matrices, its activation vector once, and its outputs
        dims = dict(self.shapes)
        self.gemv_bytes = 0
        for q in QS:
            for grp in self.GROUPS:
                k = dims[grp[0]][1]
                self.gemv_bytes += 2 * k
                for nm in grp:
                    n = dims[nm][0]
                    self.gemv_bytes += n * k * q // 8 + 2 * n * (k // GROUP) + 4 * n
        self.gemv_bytes *= layers
        self.gemv_launches = layers * len(self.GROUPS) * len(QS)
        self.quant_weights = len(QS) * sum(n * k for _, (n, k) in self.shapes)
        self.quant_bytes = sum(4 * n * k + n * k * q // 8 + 2 * n * (k // GROUP)
                               for q in QS for _, (n, k) in self.shapes)
        self.gemm_flops = 2 * GEMM_M * sum(n * k for _, (n, k) in self.shapes)
        # quantize, GEMV, and per GEMM group the X conversion and the GEMM
        self.launches_per_step = (len(QS) * len(self.shapes) + self.gemv_launches
                                  + 2 * len(self.GROUPS))

    # -- phases (each captured once as a CUDA graph) --
    def quantize_phase(self, f: int):
        for q in QS:
            for mi in range(len(self.shapes)):
                self.sss.sss_quantize(self.fresh[f][mi], q, GROUP, self.sss.GRID_SIGNED_SYM,
                                      out=self.fresh_q[q][mi], dev_status=self.status)

    # one decode token through a layer: the launches a decoder can issue, in
    # its dependency order -- {q, k, v} share x, then o, then {gate, up}
    # share x, then down -- each a programmatic dependent launch (the
    # resident weights are not written by the preceding kernels)
    GROUPS = (("q_proj", "k_proj", "v_proj"), ("o_proj",), ("gate_proj", "up_proj"),
              ("down_proj",))

    def gemv_phase(self):
        sss = self.sss
        idx = {name: i for i, (name, _) in enumerate(self.shapes)}
        flags = sss.GEMV_PDL | sss.GEMV_WEIGHTS_READY
        for q in QS:
            for layer in range(self.layers):
                for grp in self.GROUPS:
                    mis = [idx[nm] for nm in grp]
                    k = self.shapes[mis[0]][1][1]
                    sss.sss_gemv_multi([self.stack[q][layer][mi] for mi in mis], self.x[k][0],
                                       ys=[self.y[mi][0] for mi in mis], flags=flags)

    # prefill of GEMM_M tokens through the layer's matrices, the ones that
    # share X in one launch: {q, k, v}, o, {gate, up}, down
    def gemm_phase(self):
        idx = {name: i for i, (name, _) in enumerate(self.shapes)}
        for gi, grp in enumerate(self.GROUPS):
            mis = [idx[nm] for nm in grp]
            k = self.shapes[mis[0]][1][1]
            self.sss.sss_gemm_multi([self.fresh_q[4][mi] for mi in mis], self.X[k],
                                    ys=[self.Y[mi] for mi in mis], workspace=self.ws[gi],
                                    dev_status=self.status)

    def capture(self):
        torch = self.torch
        # warm every kernel once outside capture
        self.quantize_phase(0)
        self.gemv_phase()
        self.gemm_phase()
        torch.cuda.synchronize()
        self.graphs = {}
        s = torch.cuda.Stream()
        for key, fn in (("q0", lambda: self.quantize_phase(0)), ("q1", lambda: self.quantize_phase(1)),
                        ("v", self.gemv_phase), ("m", self.gemm_phase)):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=s):
                fn()
            self.graphs[key] = g
        torch.cuda.synchronize()

    def step(self, s: int, ev):
        """Replay one step; ev = 4 events recorded around the phases."""
        ev[0].record()
        self.graphs["q%d" % (s % 2)].replay()
        ev[1].record()
        self.graphs["v"].replay()
        ev[2].record()
        self.graphs["m"].replay()
        ev[3].record()


def run_ours(args):
    import torch
    import torch.distributed as dist

    ws, rank, local = dist_info()
    if ws > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    from paper_2607_08779_gb300 import sss

    sss.load()
    hbm, bf16, bf16_sus, peak_kind = peaks()
    wl = Workload(args.layers, seed_base=rank * 7919)
    wl.capture()

    def barrier():
        torch.cuda.synchronize()
        if ws > 1:
            dist.barrier()
        torch.cuda.synchronize()

    nphase = 4
    for s in range(args.warmup):
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(nphase)]
        wl.step(s, ev)
    barrier()
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    events = []
    start = torch.cuda.Event(enable_timing=True)
    stop = torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.nvtx.range_push("bench_timed")  # lets a profiler select the timed steps
    start.record()
    for s in range(args.steps):
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(nphase)]
        wl.step(s, ev)
        events.append(ev)
    stop.record()
    torch.cuda.nvtx.range_pop()
    barrier()
    clocks = sampler.stop()
    total_ms = start.elapsed_time(stop)
    tq = sum(e[0].elapsed_time(e[1]) for e in events)
    tv = sum(e[1].elapsed_time(e[2]) for e in events)
    tm = sum(e[2].elapsed_time(e[3]) for e in events)
    status = int(wl.status.item())

    # the max over ranks of every time; the value counts all ranks' work
    total_ms, tq, tv, tm = reduce_max([total_ms, tq, tv, tm], "cuda")
    K = args.steps
    gemv_gbs = job_rate(wl.gemv_bytes, ws, K, tv) / 1e9
    quant_gws = job_rate(wl.quant_weights, ws, K, tq) / 1e9
    quant_gbs = job_rate(wl.quant_bytes, ws, K, tq) / 1e9
    gemm_tfs = job_rate(wl.gemm_flops, ws, K, tm) / 1e12

    e2e = None
    if not args.no_e2e:
        e2e = measure_e2e(wl, args, ws, barrier)

    # the dominant kernel by time is the GEMV: roofline against HBM
    per_gpu_gemv = gemv_gbs / ws
    # achieved = the phase's algorithmic bytes over its event-timed duration,
    # i.e. the mean bytes per launch over the mean launch duration; traffic
    # = the mean DRAM bytes per launch from the committed ncu summary
    roofline = {"bound": "hbm", "kernel": "gemv_stream_kernel (decode GEMV, batch 1)",
                "achieved": round(per_gpu_gemv, 1), "peak": hbm, "unit": "GB/s",
                "frac": round(per_gpu_gemv / hbm, 4), "peak_source": peak_kind,
                "traffic": traffic_from_profiles("gemv_stream_llama3_8b_b1.md"),
                "algorithmic_bytes_per_launch": wl.gemv_bytes // wl.gemv_launches,
                "mean_launch_us": round(tv / K / wl.gemv_launches * 1e3, 3)}
    cpu = None  # the oracle baseline runs on rank 0 of a single-GPU run only
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        try:
            cpu = cpu_baseline(wl, seconds=args.cpu_seconds,
                               cores=args.cpu_cores or host_cores())
        except Exception as e:  # noqa: BLE001 - the pool failed mid-run: one process
            print(f"oracle baseline on several cores failed ({e!r}); timing one process",
                  file=sys.stderr, flush=True)
            cpu = cpu_baseline(wl, seconds=args.cpu_seconds, cores=1)
    if rank == 0:
        line = {
            "metric": METRIC, "value": round(gemv_gbs, 1), "unit": "GB/s", "n_gpus": ws,
            "steps": K, "warmup": args.warmup, "ms_per_step": round(total_ms / K, 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f16", "data": "synthetic",
            "config": {"workload": "llama3-8b-shaped layers: 32-layer packed stack decode GEMV "
                                   "(batch 1) at q=4,3,2 + quantize of one fp32 layer at q=4,3,2 "
                                   "+ 512-token prefill GEMM at q=4",
                       "layers": args.layers, "q": list(QS), "group": GROUP,
                       "grid": "signed_symmetric", "batch": 1, "gemm_m": GEMM_M,
                       "decode_launches_per_layer": "{q,k,v} fused, o, {gate,up} fused, down; "
                                                    "programmatic dependent launch",
                       "accumulate": "f32", "parallelism": f"replicas x{ws}",
                       "l2": "inputs larger than L2 (9.2 GB packed stack read per step)"},
            "roofline": roofline,
            "phases": {
                "gemv": {"gbs": round(gemv_gbs, 1), "ms_per_step": round(tv / K, 4),
                         "frac_hbm": round(per_gpu_gemv / hbm, 4),
                         "launches_per_step": wl.gemv_launches},
                "quantize": {"gweights_per_s": round(quant_gws, 1), "gbs": round(quant_gbs, 1),
                             "frac_hbm": round(quant_gbs / ws / hbm, 4),
                             "ms_per_step": round(tq / K, 4)},
                "gemm": {"tflops": round(gemm_tfs, 1), "m": GEMM_M,
                         "frac_bf16_sustained": round(gemm_tfs / ws / bf16_sus, 4),
                         "ms_per_step": round(tm / K, 4)},
            },
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": wl.launches_per_step * K,
            "clocks": clocks,
            "device_status": status,
        }
        print(json.dumps(line), flush=True)
    if ws > 1:
        dist.barrier()
        dist.destroy_process_group()


def measure_e2e(wl, args, ws, barrier):
    """The step through the public API with HOST buffers.  The sss_* calls of
    each phase are captured once as CUDA graphs (their launches, issued
    through the C ABI) and replayed; inside the timed region, every step
    copies its inputs in from pinned host memory and reads its outputs back.

    value: the whole step (quantize one fresh fp32 layer, the decode GEMV
    over the stack, the prefill GEMM), its GEMV bytes over its time, so that
    it reads on the headline's scale.  The fresh layer is double-buffered:
    step s + 1's copy runs on a copy stream while step s computes, as a
    serving pipeline would overlap them; the small activation copies and
    the read-backs stay on the compute stream.  gemv_only: the decode GEMV
    phase alone, x copied in and y read back every step."""
    torch = wl.torch
    host_fresh = [f.cpu().pin_memory() for f in wl.fresh[0]]
    host_x = {k: v.cpu().pin_memory() for k, v in wl.x.items()}
    host_X = {k: v.cpu().pin_memory() for k, v in wl.X.items()}
    host_y = [y.cpu().pin_memory() for y in wl.y]
    host_Y = [Y.cpu().pin_memory() for Y in wl.Y]
    nb = lambda ts: sum(t.numel() * t.element_size() for t in ts)  # noqa: E731
    h2d_x = nb(host_x.values())
    d2h_y = nb(host_y)
    h2d = nb(host_fresh) + h2d_x + nb(host_X.values())
    d2h = d2h_y + nb(host_Y)
    steps = max(10, min(args.steps, 20))
    main = torch.cuda.current_stream()
    copy = torch.cuda.Stream()
    copied = [torch.cuda.Event(), torch.cuda.Event()]
    used = [torch.cuda.Event(), torch.cuda.Event()]

    def fresh_in(b):
        # into buffer b once the step that last quantized it is done
        copy.wait_event(used[b])
        with torch.cuda.stream(copy):
            for d, h in zip(wl.fresh[b], host_fresh):
                d.copy_(h, non_blocking=True)
        copied[b].record(copy)

    def x_in():
        for k in wl.x:
            wl.x[k].copy_(host_x[k], non_blocking=True)

    def y_out():
        for h, d in zip(host_y, wl.y):
            h.copy_(d, non_blocking=True)

    def run_steps(n):
        for b in (0, 1):
            used[b].record(main)
        fresh_in(0)
        for s in range(n):
            b = s % 2
            if s + 1 < n:
                fresh_in(1 - b)
            main.wait_event(copied[b])
            x_in()
            for k in wl.X:
                wl.X[k].copy_(host_X[k], non_blocking=True)
            wl.graphs["q%d" % b].replay()
            used[b].record(main)
            wl.graphs["v"].replay()
            wl.graphs["m"].replay()
            y_out()
            for h, d in zip(host_Y, wl.Y):
                h.copy_(d, non_blocking=True)

    def gemv_steps(n):
        for _ in range(n):
            x_in()
            wl.graphs["v"].replay()
            y_out()

    def timed(fn, n):
        fn(2)
        barrier()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        fn(n)
        b.record()
        barrier()
        return reduce_max([a.elapsed_time(b) / n], "cuda")[0]

    ms = timed(run_steps, steps)
    ms_v = timed(gemv_steps, steps)
    return {"value": round(job_rate(wl.gemv_bytes, ws, 1, ms) / 1e9, 1), "unit": "GB/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": round(ms, 4), "steps": steps,
            "scope": "whole step (quantize a fresh fp32 layer + decode GEMV over the stack + "
                     "prefill GEMM) with host copies; value = the step's GEMV bytes over its time",
            "api": "sss_* calls captured once as CUDA graphs, replayed each step; the fresh "
                   "layer's host copy for step s+1 overlaps step s on a copy stream",
            "gemv_only": {"value": round(job_rate(wl.gemv_bytes, ws, 1, ms_v) / 1e9, 1),
                          "unit": "GB/s", "h2d_bytes_per_step": h2d_x,
                          "d2h_bytes_per_step": d2h_y, "ms_per_step": round(ms_v, 4),
                          "steps": steps}}


def oracle_gemv_rate(codes, scales, n_rows, k, q, xbits, seconds):
    """GB/s of packed bytes the oracle GEMV processes on this host (one
    core), over as many row blocks as fit in `seconds`."""
    import oracle

    rows_per_call = 64
    row_bytes = k * q // 8 + 2 * (k // GROUP)
    done_rows, t0 = 0, time.perf_counter()
    r0 = 0
    while time.perf_counter() - t0 < seconds:
        r1 = min(n_rows, r0 + rows_per_call)
        oracle.gemv(codes[r0:r1], scales[r0:r1], None, r1 - r0, k, q, GROUP,
                    oracle.GRID_SIGNED_SYM, xbits)
        done_rows += r1 - r0
        r0 = 0 if r1 >= n_rows else r1
    el = time.perf_counter() - t0
    return done_rows * row_bytes / el / 1e9, done_rows, el


def _oracle_gemv_worker(job):
    return oracle_gemv_rate(*job)


def oracle_pool(cores: int):
    """A pool of `cores` spawned processes for the oracle baseline (spawned,
    so none inherits CUDA state), or None for one core or when the host
    cannot start one (the caller then measures one process and reports
    cores = 1)."""
    if cores <= 1:
        return None
    import multiprocessing as mp

    try:
        pool = mp.get_context("spawn").Pool(cores)
        pool.map(_noop, range(cores))
        return pool
    except Exception as e:  # noqa: BLE001 - reported, then one process
        print(f"oracle baseline: no process pool ({e!r}); timing one process",
              file=sys.stderr, flush=True)
        return None


def _noop(i):
    return i


def oracle_gemv_rate_cores(pool, cores, codes, scales, n_rows, k, q, xbits, seconds):
    """The unchanged oracle GEMV run in `cores` processes at once, each over
    the same row blocks for `seconds`: GB/s of packed bytes all of them
    processed over the longest one's time, the single-process GB/s of the
    first worker, the rows done and that time."""
    if pool is None:
        gbs, rows, el = oracle_gemv_rate(codes, scales, n_rows, k, q, xbits, seconds)
        return gbs, gbs, rows, el
    job = (codes, scales, n_rows, k, q, xbits, seconds)
    res = pool.map(_oracle_gemv_worker, [job] * cores)
    total = sum(g * e for g, _, e in res)
    wall = max(e for _, _, e in res)
    return total / wall, res[0][0], sum(r for _, r, _ in res), wall


def oracle_quantize_rate(w, q, seconds):
    """Weights per second the oracle quantizer (signed grid, group 32)
    processes on this host (one process) over repeated calls on `w`."""
    import oracle

    done, t0 = 0, time.perf_counter()
    while time.perf_counter() - t0 < seconds:
        oracle.quantize(w, q, GROUP, oracle.GRID_SIGNED_SYM)
        done += w.size
    el = time.perf_counter() - t0
    return done / el, done, el


def _oracle_quantize_worker(job):
    return oracle_quantize_rate(*job)


def oracle_gemm_rate(codes, scales, n_rows, k, q, xbits, seconds):
    """FLOP/s the oracle GEMM (dequantise a block of packed rows, then the
    fp64 matmul with the tokens xbits) sustains on this host (one process),
    over row blocks of the sample for `seconds`."""
    import oracle

    rows_per_call = 64
    m = xbits.shape[0]
    flops, t0, r0 = 0, time.perf_counter(), 0
    while time.perf_counter() - t0 < seconds:
        r1 = min(n_rows, r0 + rows_per_call)
        What = oracle.dequantize(codes, scales, None, n_rows, k, q, GROUP, oracle.GRID_SIGNED_SYM,
                                 rows=(r0, r1 - r0))
        oracle.matmul_f64(What, xbits)
        flops += 2 * (r1 - r0) * k * m
        r0 = 0 if r1 >= n_rows else r1
    el = time.perf_counter() - t0
    return flops / el, flops, el


def _oracle_gemm_worker(job):
    return oracle_gemm_rate(*job)


def host_cores() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return max(1, os.cpu_count() or 1)


def cpu_baseline(wl, seconds: float, cores: int):
    """The oracle's GEMV, as it stands, on the host cores, on a bounded
    sample of the same workload (rows of the layer-0 gate_proj at q=4); and
    beside it the oracle quantizer and the oracle GEMM on samples of their
    phases."""
    mi = [name for name, _ in wl.shapes].index("gate_proj")
    qt = wl.stack[4][0][mi]
    n, k = qt.n, qt.k
    codes = qt.codes[:4096].cpu().numpy()
    scales = qt.scales[:4096].cpu().numpy().view(np.uint16)
    xbits = wl.x[k].cpu().view(wl.torch.int16).numpy().view(np.uint16)
    # the quantize phase's oracle: rows of the fresh fp32 gate_proj at q=4
    wq = wl.fresh[0][mi][:256].cpu().numpy()
    # the GEMM phase's oracle: the same packed rows against 16 of its tokens
    gtok = 16
    Xs = wl.X[k][:gtok].cpu().view(wl.torch.int16).numpy().view(np.uint16)
    pool = oracle_pool(cores)
    if pool is None:
        cores = 1
    try:
        gbs, gbs1, rows, el = oracle_gemv_rate_cores(pool, cores, codes, scales, codes.shape[0],
                                                     k, 4, xbits, seconds)
        qsec = max(1.0, seconds / 2)
        gjob = (codes, scales, codes.shape[0], k, 4, Xs, qsec)
        if pool is None:
            qres = [oracle_quantize_rate(wq, 4, qsec)]
            gres = [oracle_gemm_rate(*gjob)]
        else:
            qres = pool.map(_oracle_quantize_worker, [(wq, 4, qsec)] * cores)
            gres = pool.map(_oracle_gemm_worker, [gjob] * cores)
    finally:
        if pool is not None:
            pool.close()
            pool.join()
    qwall = max(e for _, _, e in qres)
    qdone = sum(d for _, d, _ in qres)
    gwall = max(e for _, _, e in gres)
    gdone = sum(d for _, d, _ in gres)
    return {"value": round(gbs, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
            "single_core_value": round(gbs1, 4),
            "sample": f"{rows} rows of gate_proj (14336x4096) at q=4 g=32, batch 1: "
                      f"{cores} processes x {el:.1f} s of the single-threaded oracle GEMV (fp64)",
            "quantize": {"value": round(qdone / qwall / 1e9, 6), "unit": "Gweights/s",
                         "cores": cores, "single_core_value": round(qres[0][0] / 1e9, 6),
                         "sample": f"{qdone} weights: 256 rows of the fresh fp32 gate_proj "
                                   f"(256x4096) at q=4 g=32, signed grid, {cores} processes x "
                                   f"{qwall:.1f} s of the single-threaded oracle quantizer"},
            "gemm": {"value": round(gdone / gwall / 1e12, 9), "unit": "TFLOP/s", "cores": cores,
                     "single_core_value": round(gres[0][0] / 1e12, 9),
                     "sample": f"{gdone} FLOPs: blocks of 64 packed gate_proj rows at q=4 g=32 "
                               f"dequantised, then the fp64 matmul with {gtok} tokens of the "
                               f"prefill X; {cores} processes x {gwall:.1f} s of the "
                               f"single-threaded oracle GEMM"}}


def run_reference(args):
    """The oracle on the host cores, on the same metric; rank 0 only."""
    ws, rank, local = dist_info()
    if rank != 0:
        return
    import oracle
    from paper_2607_08779_gb300 import inputs

    oracle.build()
    n, k = inputs.LLAMA3_8B_LAYER["gate_proj"]
    rows = 1024
    W = inputs.student_t_weights(rows, k, inputs.weight_seed(2, 0, 4))
    packed = {}
    for q in QS:
        codes, scales, _, _, _ = oracle.quantize(W, q, GROUP, oracle.GRID_SIGNED_SYM)
        packed[q] = (codes, scales)
    xbits = inputs.normal_bf16_bits((1, k), 7)
    per_step = max(0.5, args.ref_seconds)
    cores = getattr(args, "cpu_cores", 0) or host_cores()
    pool = oracle_pool(cores)
    if pool is None:
        cores = 1
    try:
        for _ in range(args.warmup):
            oracle_gemv_rate_cores(pool, cores, *packed[4], rows, k, 4, xbits, 0.05)
        total_bytes, total_s, one_bytes = 0.0, 0.0, 0.0
        for s in range(args.steps):
            q = QS[s % len(QS)]
            gbs, gbs1, r, el = oracle_gemv_rate_cores(pool, cores, *packed[q], rows, k, q, xbits,
                                                      per_step)
            total_bytes += gbs * el * 1e9
            one_bytes += gbs1 * el * 1e9
            total_s += el
    finally:
        if pool is not None:
            pool.close()
            pool.join()
    value = total_bytes / total_s / 1e9
    line = {
        "metric": METRIC, "value": round(value, 4), "unit": "GB/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(total_s / args.steps * 1e3, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "impl": "reference",
        "config": {"workload": "llama3-8b-shaped layers: batch-1 GEMV over packed gate_proj "
                               "rows at q=4,3,2 (bounded sample per step)",
                   "group": GROUP, "grid": "signed_symmetric", "batch": 1},
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
                         "single_core_value": round(one_bytes / total_s / 1e9, 4),
                         "sample": f"{args.steps} steps x {per_step:.1f} s of the oracle GEMV in "
                                   f"{cores} processes over {rows} rows of gate_proj, "
                                   f"q cycling 4,3,2"},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_micro(args):
    """One operation on one Llama3-8B shape, cycling over `--rotate` distinct
    copies of its inputs (more than L2 in total), timed with CUDA events.
    Prints one JSON line (not the benchmark's headline line)."""
    import torch

    from paper_2607_08779_gb300 import inputs, sss

    torch.cuda.set_device(0)
    sss.load()
    names = args.matrices.split(",")
    shapes = [inputs.LLAMA3_8B_LAYER[nm] for nm in names]
    if args.rows:
        shapes = [(args.rows, kk) for _, kk in shapes]
    k = shapes[0][1]
    G = sss.GRID_ASYM if args.grid == "asym" else (
        sss.GRID_UNSIGNED_SYM if args.grid == "unsigned" else sss.GRID_SIGNED_SYM)
    q, g = args.q, args.group
    copies = []
    for c in range(args.rotate):
        mats = []
        for mi, (n, kk) in enumerate(shapes):
            w = inputs.student_t_weights_cuda(n, kk, 1000 * c + mi)
            if args.micro == "quantize":
                mats.append((w, sss.empty_qtensor(n, kk, q, g, G)))
            else:
                mats.append(sss.sss_quantize(w, q, g, G))
                del w
        copies.append(mats)
    rows_x = args.m if args.micro == "gemm" else (args.batch if args.micro == "gemv_single" else 1)
    x = inputs.normal_bf16_cuda((rows_x, k), 5)
    ys = [torch.empty((rows_x, n), dtype=torch.float32, device="cuda") for n, _ in shapes]
    ws = None
    if args.micro == "gemm":
        need = (sss.sss_gemm_multi_workspace_bytes(copies[0], args.m) if args.fuse else
                max(sss.sss_workspace_bytes(qt, args.m, sss.OP_GEMM) for qt in copies[0]))
        ws = torch.empty(max(need, 16), dtype=torch.uint8, device="cuda")

    def op(c):
        mats = copies[c % args.rotate]
        if args.micro == "gemv":
            sss.sss_gemv_multi(mats, x[0], ys=[y[0] for y in ys], flags=args.flags)
        elif args.micro == "gemv_single":
            for qt, y in zip(mats, ys):
                sss.sss_gemv(qt, x, y=y)
        elif args.micro == "gemm" and args.fuse:
            sss.sss_gemm_multi(mats, x, ys=ys, workspace=ws)
        elif args.micro == "gemm":
            for qt, y in zip(mats, ys):
                sss.sss_gemm(qt, x, y=y, workspace=ws)
        else:
            for w, qt in mats:
                sss.sss_quantize(w, q, g, G, out=qt)

    for c in range(3):
        op(c)
    torch.cuda.synchronize()
    # the timed loop is one CUDA graph, so host-side call overhead is excluded
    graph = torch.cuda.CUDAGraph()
    cs = torch.cuda.Stream()
    with torch.cuda.graph(graph, stream=cs):
        for c in range(args.iters):
            op(c)
    graph.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    graph.replay()
    b.record()
    torch.cuda.synchronize()
    us = a.elapsed_time(b) * 1e3 / args.iters
    nbytes = 0
    for (n, kk) in shapes:
        packed = n * kk * q // 8 + 2 * n * (kk // g) * (2 if G == sss.GRID_ASYM else 1)
        if args.micro == "quantize":
            nbytes += 4 * n * kk + packed
        elif args.micro == "gemm":
            nbytes += packed + 2 * args.m * kk + 4 * args.m * n
        else:
            nbytes += packed + 4 * n * rows_x
    if args.micro not in ("quantize", "gemm"):
        nbytes += 2 * k * rows_x
    flops = 2 * rows_x * sum(n * kk for n, kk in shapes)
    print(json.dumps({"micro": args.micro, "matrices": names, "q": q, "group": g, "rows_x": rows_x,
                      "grid": args.grid, "fused": bool(getattr(args, "fuse", False)),
                      "us_per_call": round(us, 3),
                      "gbs": round(nbytes / us / 1e3, 1), "tflops": round(flops / us / 1e6, 2),
                      "iters": args.iters, "rotate": args.rotate}), flush=True)


def _graph_time_us(fn, iters: int) -> float:
    """Mean µs per call of fn(i), i = 0..iters-1, captured in one CUDA graph
    and replayed once after a warm replay."""
    import torch

    for i in range(3):
        fn(i)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    cs = torch.cuda.Stream()
    with torch.cuda.graph(graph, stream=cs):
        for i in range(iters):
            fn(i)
    graph.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    graph.replay()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) * 1e3 / iters


def sweep_qwen3_quantize(args):
    """Weight quantization of a whole Qwen3-32B-shaped model (64 layers of
    q/k/v/o/gate/up/down, 31.2G weights), signed grid, q in {2, 3} x group
    in {32, 128}.  Each layer's fp32 weights are generated on the device into
    reused buffers (heavy-tailed, with outlier channels); every quantize
    launch is timed with CUDA events and the rate is weights over the sum of
    kernel times.  Prints one JSON line per (q, group) and a summary."""
    import torch

    from paper_2607_08779_gb300 import inputs, sss

    torch.cuda.set_device(0)
    sss.load()
    hbm, _, _, peak_kind = peaks()
    shapes = list(inputs.QWEN3_32B_LAYER.items())
    layers = args.layers if args.layers != 32 else inputs.QWEN3_32B_LAYERS
    variants = [(q, g) for q in (2, 3) for g in (32, 128)]
    G = sss.GRID_SIGNED_SYM
    w = [torch.empty((n, k), dtype=torch.float32, device="cuda") for _, (n, k) in shapes]
    outs = {v: [sss.empty_qtensor(n, k, v[0], v[1], G) for _, (n, k) in shapes] for v in variants}
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ms = {v: 0.0 for v in variants}
    weights = 0
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2 * len(variants))]
    for layer in range(layers):
        for mi, (_, (n, k)) in enumerate(shapes):
            inputs.student_t_weights_cuda(n, k, inputs.weight_seed(4, layer, mi), out=w[mi])
        weights += sum(n * k for _, (n, k) in shapes)
        for vi, v in enumerate(variants):
            ev[2 * vi].record()
            for mi in range(len(shapes)):
                sss.sss_quantize(w[mi], v[0], v[1], G, out=outs[v][mi], dev_status=status)
            ev[2 * vi + 1].record()
        torch.cuda.synchronize()
        for vi, v in enumerate(variants):
            ms[v] += ev[2 * vi].elapsed_time(ev[2 * vi + 1])
    summary = []
    for v in variants:
        q, g = v
        bpw = 4 + q / 8 + 2 / g
        gw = weights / (ms[v] * 1e-3) / 1e9
        line = {"sweep": "qwen3_32b_quantize", "layers": layers, "q": q, "group": g,
                "grid": "signed", "weights": weights, "kernel_ms": round(ms[v], 3),
                "gweights_per_s": round(gw, 1), "gbs": round(gw * bpw, 1),
                "frac_hbm": round(gw * bpw / hbm, 4), "peak_source": peak_kind,
                "device_status": int(status.item())}
        summary.append(line)
        print(json.dumps(line), flush=True)
    return summary


def sweep_grids(args):
    """The grid comparison on the 4096x4096 shape (heavy-tailed weights with
    outlier channels): unsigned symmetric vs signed symmetric vs min-max, at
    q in {2, 3, 4} and group 32 / 128.  Per format: the per-group l2 error of
    the stored (fp16-scale) dequantised weights (mean, p50, p99, fp64), the
    fraction of groups with |C_gamma| <= |C_-gamma| (symmetric grids), and
    the decode GEMV GB/s at batch 1 / 4 / 16, timed in a CUDA graph over more
    copies of the packed matrix than L2 holds."""
    import torch

    from paper_2607_08779_gb300 import inputs, sss

    torch.cuda.set_device(0)
    sss.load()
    hbm, _, _, peak_kind = peaks()
    n = k = 4096
    l2 = torch.cuda.get_device_properties(0).L2_cache_size
    W = inputs.student_t_weights_cuda(n, k, inputs.weight_seed(5, 0, 0))
    Wd = W.double()
    xs = {b: inputs.normal_bf16_cuda((b, k), 50 + b) for b in (1, 4, 16)}
    rows = []
    for gname, grid in (("unsigned", sss.GRID_UNSIGNED_SYM), ("signed", sss.GRID_SIGNED_SYM),
                        ("asym", sss.GRID_ASYM)):
        for q in (2, 3, 4):
            for g in (32, 128):
                cc = torch.zeros((n, k // g, 2), dtype=torch.uint8, device="cuda")
                st = torch.zeros(1, dtype=torch.int32, device="cuda")
                qt = sss.sss_quantize(W, q, g, grid, clip_counts=cc, dev_status=st)
                what = sss.sss_dequantize(qt)
                err = (Wd - what.double()).view(n, k // g, g).pow(2).sum(-1).sqrt().flatten()
                qs = torch.quantile(err.float(), torch.tensor([0.5, 0.99], device="cuda"))
                line = {"sweep": "grids", "grid": gname, "q": q, "group": g,
                        "l2_err_mean": float(err.mean()), "l2_err_p50": float(qs[0]),
                        "l2_err_p99": float(qs[1]),
                        "frac_groups_clip_self_le_other": (
                            None if grid == sss.GRID_ASYM else
                            float((cc[..., 0] <= cc[..., 1]).float().mean())),
                        "device_status": int(st.item())}
                packed = qt.codes.numel() + qt.scales.numel() * 2 + (
                    qt.mins.numel() * 2 if qt.mins is not None else 0)
                copies = max(4, -(-4 * l2 // packed))
                pool = [qt] + [sss.QTensor(qt.n, qt.k, q, g, grid, qt.codes.clone(),
                                           qt.scales.clone(),
                                           None if qt.mins is None else qt.mins.clone())
                               for _ in range(copies - 1)]
                for b, x in xs.items():
                    y = torch.empty((b, n), dtype=torch.float32, device="cuda")
                    need = sss.sss_workspace_bytes(qt, b, sss.OP_GEMV)
                    ws = torch.empty(max(need, 16), dtype=torch.uint8, device="cuda")
                    us = _graph_time_us(
                        lambda i: sss.sss_gemv(pool[i % copies], x, y=y, workspace=ws),
                        max(args.iters, 2 * copies))
                    nbytes = packed + 2 * b * k + 4 * b * n
                    line["gemv_b%d_us" % b] = round(us, 3)
                    line["gemv_b%d_gbs" % b] = round(nbytes / us / 1e3, 1)
                line["gemv_b1_frac_hbm"] = round(line["gemv_b1_gbs"] / hbm, 4)
                line["peak_source"] = peak_kind
                rows.append(line)
                print(json.dumps(line), flush=True)
                del pool
    return rows


def sweep_margins(args):
    """Cardinality margin against realised error gain (Remark
    rem:cardinality-margin) on every group of one Llama3-8B-shaped layer
    (heavy-tailed weights with outlier channels), group 32, q in {2, 3, 4}.

    Per group: gamma* is the sign the signed grid stored; the margin is
    m = |C_-gamma*| - |C_gamma*| from the signed quantizer's clip counts; the
    gain is g = ||w - Q_-gamma*(w)||^2 - ||w - Q_gamma*(w)||^2, both errors
    of the stored (fp16-scale) dequantised weights in fp64.  Q_+1 is the
    unsigned grid on w; Q_-1(w) = -Q_+1(-w), the unsigned grid on -w.
    Groups with M = 0 are left out."""
    import torch

    from paper_2607_08779_gb300 import inputs, sss

    torch.cuda.set_device(0)
    sss.load()
    g = 32
    rows = []
    for q in (2, 3, 4):
        tot = {"groups": 0, "m_ge0": 0, "m_gt0": 0, "m_gt0_g_gt0": 0, "m_lt0": 0,
               "m_lt0_g_gt0": 0, "m_eq0": 0, "m_eq0_g_gt0": 0, "g_gt0": 0}
        for mi, (name, (n, k)) in enumerate(inputs.LLAMA3_8B_LAYER.items()):
            w = inputs.student_t_weights_cuda(n, k, inputs.weight_seed(2, 0, mi))
            cc = torch.zeros((n, k // g, 2), dtype=torch.uint8, device="cuda")
            st = torch.zeros(1, dtype=torch.int32, device="cuda")
            qs = sss.sss_quantize(w, q, g, sss.GRID_SIGNED_SYM, clip_counts=cc, dev_status=st)
            qp = sss.sss_quantize(w, q, g, sss.GRID_UNSIGNED_SYM, dev_status=st)
            qm = sss.sss_quantize(-w, q, g, sss.GRID_UNSIGNED_SYM, dev_status=st)
            wd = w.double().view(n, k // g, g)
            e_plus = (wd - sss.sss_dequantize(qp).double().view(n, k // g, g)).pow(2).sum(-1)
            e_minus = (wd + sss.sss_dequantize(qm).double().view(n, k // g, g)).pow(2).sum(-1)
            s_bits = qs.scales.view(torch.int16)
            neg = (s_bits < 0)                    # stored sign bit: gamma* = -1
            live = (s_bits & 0x7FFF) != 0         # M > 0
            gain = torch.where(neg, e_plus - e_minus, e_minus - e_plus)
            m = cc[..., 1].int() - cc[..., 0].int()
            gp = gain > 0
            tot["groups"] += int(live.sum())
            tot["m_ge0"] += int((live & (m >= 0)).sum())
            tot["m_gt0"] += int((live & (m > 0)).sum())
            tot["m_gt0_g_gt0"] += int((live & (m > 0) & gp).sum())
            tot["m_lt0"] += int((live & (m < 0)).sum())
            tot["m_lt0_g_gt0"] += int((live & (m < 0) & gp).sum())
            tot["m_eq0"] += int((live & (m == 0)).sum())
            tot["m_eq0_g_gt0"] += int((live & (m == 0) & gp).sum())
            tot["g_gt0"] += int((live & gp).sum())
            if int(st.item()) != 0:
                tot["device_status"] = int(st.item())
            del w, wd, e_plus, e_minus, gain
        n_g = max(1, tot["groups"])
        line = {"sweep": "margins", "layer": "llama3_8b", "q": q, "group": g,
                "groups": tot["groups"],
                "frac_condition_m_ge0": round(tot["m_ge0"] / n_g, 5),
                "frac_m_gt0": round(tot["m_gt0"] / n_g, 5),
                "frac_gain_pos_given_m_gt0": round(tot["m_gt0_g_gt0"] / max(1, tot["m_gt0"]), 5),
                "frac_gain_pos_given_m_eq0": round(tot["m_eq0_g_gt0"] / max(1, tot["m_eq0"]), 5),
                "frac_gain_pos_given_m_lt0": round(tot["m_lt0_g_gt0"] / max(1, tot["m_lt0"]), 5),
                "frac_gain_pos": round(tot["g_gt0"] / n_g, 5),
                "device_status": tot.get("device_status", 0)}
        rows.append(line)
        print(json.dumps(line), flush=True)
    return rows


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--layers", type=int, default=32)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--cpu-cores", type=int, default=0,
                    help="processes for the oracle baseline (0 = every host core)")
    ap.add_argument("--ref-seconds", type=float, default=2.0)
    ap.add_argument("--micro", choices=["gemv", "gemv_single", "gemm", "quantize"])
    ap.add_argument("--matrices", default="gate_proj,up_proj")
    ap.add_argument("--q", type=int, default=4)
    ap.add_argument("--group", type=int, default=32)
    ap.add_argument("--grid", choices=["signed", "unsigned", "asym"], default="signed")
    ap.add_argument("--m", type=int, default=512)
    ap.add_argument("--batch", type=int, default=1, help="micro gemv_single: activation rows")
    ap.add_argument("--iters", type=int, default=50)
    ap.add_argument("--rotate", type=int, default=8)
    ap.add_argument("--flags", type=int, default=0)
    ap.add_argument("--fuse", action="store_true",
                    help="micro gemm: the matrices in one sss_gemm_multi call")
    ap.add_argument("--rows", type=int, default=0, help="micro: override every matrix's rows")
    ap.add_argument("--sweep", choices=["qwen3_quantize", "grids", "margins"],
                    help="measurement sweeps: whole-model quantization of Qwen3-32B shapes, "
                         "the unsigned / signed / min-max grid comparison, or the "
                         "cardinality margin against the realised l2 gain")
    args = ap.parse_args()
    if args.sweep == "qwen3_quantize":
        sweep_qwen3_quantize(args)
        return
    if args.sweep == "grids":
        sweep_grids(args)
        return
    if args.sweep == "margins":
        sweep_margins(args)
        return
    if args.micro:
        run_micro(args)
        return
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
