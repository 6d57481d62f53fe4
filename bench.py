#!/usr/bin/env python
"""MoCE layer forward benchmark on GB300.

One step = one MoCE forward (pooling, gate, softmax weights, routed mixing,
residual) over the whole batch of the ResNet-50 stage-1 bottleneck-entrance
projection (N=64, 56x56, C_in=256 -> 64 routed experts + 1 residual, k=16,
bf16 NHWC), on seeded synthetic inputs already resident in HBM. Supports are
packed once before timing (reported separately as pack_us).

Reported value: achieved algorithmic HBM bandwidth, GB/s = (x read once +
y written once + packed tables + gate parameters) / layer time, summed over
ranks and divided by the slowest rank's time. us_per_layer is the layer time.
Between timed steps the inputs rotate over enough copies that every step
reads x from HBM, not L2.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

--impl reference times the CPU oracle (the plain restatement of the paper's
equations) on the host cores, on a bounded sample of the same workload.
Multi-GPU (torchrun): every rank runs its own batch (weak scaling, no
collective on the data path).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

WORKLOAD = "rn50_stage1_reduce"
DATA = {"relu": "synthetic (seeded post-ReLU N(0,1); stands in for ImageNet activations)",
        "gelu": "synthetic (seeded GELU(N(0,1)); stands in for ViT-B token activations)"}
METRIC = "MoCE fwd µs/layer & achieved HBM GB/s (% of GB300 peak) vs dense 1×1 cuBLAS"
UNIT = "GB/s"
SEED = 0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20000)
    ap.add_argument("--warmup", type=int, default=200)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=WORKLOAD)
    ap.add_argument("--batch", type=int, default=None,
                    help="examples per layer instead of the workload's N (smaller profiling cases)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--path", default="auto",
                    help="kernel path of the forward (auto, stream, steps)")
    ap.add_argument("--d", type=int, default=32,
                    help="router rank of the input-conditioned variant (--op dynamic)")
    ap.add_argument("--op", choices=["forward", "backward", "train", "dynamic"], default="forward",
                    help="forward: the layer forward (the benchmark); backward: the layer's "
                         "gradients for an upstream gradient; train: TopK over the full "
                         "routing matrix and the coverage loss with its gradient; dynamic: "
                         "static against input-conditioned supports (Eq. dynamic)")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="CPU work budget of the oracle baseline leg")
    return ap.parse_args()


# ------------------------------------------------------------------ helpers


def dist_env():
    from paper_2608_23794_gb300 import dist as mdist
    info = mdist.rank_info()
    return info.rank, info.world, info.local_rank


def workload_bytes(cfg, n_resid: int) -> int:
    from paper_2608_23794_gb300 import costmodel
    return costmodel.layer_bytes(cfg.N, cfg.H, cfg.W, cfg.C_in, cfg.C_out, cfg.k,
                                 cfg.elem_bytes, n_resid)


# FP32 fused multiply-adds per second: 128 FP32 lanes per SM x the SM count x
# the maximum SM clock (the unit counts and clock of GB300's datasheet; the
# routed mix and the gate run on these lanes, not on tensor cores).
FP32_LANES_PER_SM = 128


def fp32_fma_peak(sms: int, mhz: float) -> float:
    return FP32_LANES_PER_SM * sms * mhz * 1e6


def sgemm_fma_rate(dev) -> float:
    """FP32 multiply-adds per second of cuBLAS SGEMM (8192^3 at the "highest" float32 matmul
    precision: no TF32), a measured check beside the derived FP32 peak."""
    import torch
    n = 8192
    g = torch.Generator(device=dev).manual_seed(0)
    a = torch.randn(n, n, device=dev, generator=g)
    b = torch.randn(n, n, device=dev, generator=g)
    c = torch.empty(n, n, device=dev)
    prec = torch.get_float32_matmul_precision()
    torch.set_float32_matmul_precision("highest")
    try:
        for _ in range(3):
            torch.matmul(a, b, out=c)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record()
        for _ in range(10):
            torch.matmul(a, b, out=c)
        e1.record()
        torch.cuda.synchronize()
    finally:
        torch.set_float32_matmul_precision(prec)
    return n ** 3 / (e0.elapsed_time(e1) * 1e-3 / 10)


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


def csrc_hash() -> str:
    """Hash of the CUDA sources' code: line comments and blank lines do not count, so a
    comment edit keeps a traffic record taken on the same code valid."""
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2608_23794_gb300", "csrc")
    for f in sorted(os.listdir(d)):
        with open(os.path.join(d, f), encoding="utf-8") as fh:
            lines = [ln.split("//", 1)[0].rstrip() for ln in fh]
        h.update(f.encode() + "\n".join(ln for ln in lines if ln).encode())
    return h.hexdigest()[:16]


def ncu_traffic(workload: str, kernel: str):
    """DRAM bytes per step from a committed ncu summary, if taken on the current kernels."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        d = json.load(f)
    rec = d.get(workload)
    if not rec or rec.get("csrc_hash") != csrc_hash() or rec.get("kernel", kernel) != kernel:
        return None
    return rec.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples taken while the timed region runs."""

    FIELDS = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.proc = None
        self.lines: list[str] = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)
        rows = []
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 10:
                continue
            if self.uuid and parts[1] != self.uuid:
                continue
            rows.append(parts)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        sm = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        mx = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = sorted({names[i] for r in rows for i in range(4) if r[6 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


def gpu_uuid(torch, dev):
    try:
        u = str(torch.cuda.get_device_properties(dev).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        return None


# ------------------------------------------------------------------ CPU oracle leg


def oracle_sample_run(lay, cfg, budget_s: float):
    """Time the oracle on a bounded sample of the workload, single-threaded; returns (GB/s,
    sample str, seconds per run, examples, rows)."""
    import numpy as np

    import oracle
    pidx, plog, resid = oracle.pack(lay.support_idx, lay.support_logits, cfg.C_in)
    args = (pidx, plog, resid, lay.W1, lay.b1, lay.w2, float(lay.b2[0]), cfg.tau_min, cfg.tau_max)
    # one example first, to size the sample
    t0 = time.perf_counter()
    oracle.forward(lay.x[:1], cfg.layout, *args)
    t_ex = max(time.perf_counter() - t0, 1e-6)
    n_ex = int(max(1, min(cfg.N, budget_s / t_ex)))
    h_rows = cfg.H
    if t_ex > budget_s and cfg.layout == "nhwc":
        h_rows = int(max(1, cfg.H * budget_s / t_ex))
    xs = np.ascontiguousarray(lay.x[:n_ex, :h_rows]) if cfg.layout == "nhwc" else lay.x[:n_ex]
    reps, times = 0, []
    start = time.perf_counter()
    while True:
        t0 = time.perf_counter()
        oracle.forward(xs, cfg.layout, *args)
        times.append(time.perf_counter() - t0)
        reps += 1
        if time.perf_counter() - start >= budget_s or reps >= 1000:
            break
    sub = cfg.replace(N=n_ex, H=h_rows)
    nbytes = workload_bytes(sub, len(resid))
    t = statistics.median(times)
    sample = (f"{n_ex} of {cfg.N} examples x {h_rows} of {cfg.H} rows, median of {reps} "
              f"single-threaded oracle runs")
    return nbytes / t / 1e9, sample, t, n_ex, h_rows


# ------------------------------------------------------------------ the oracle on every host core

_POOL = None  # in a worker: (layer, layout, oracle arguments)


def _pool_init(cfg, seed):
    """Worker start-up (spawned): the parent's seeded layer and packed tables, rebuilt."""
    global _POOL
    from paper_2608_23794_gb300 import synth
    import oracle
    lay = synth.make_layer(cfg, seed=seed)
    pidx, plog, resid = oracle.pack(lay.support_idx, lay.support_logits, cfg.C_in)
    _POOL = (lay, cfg.layout, (pidx, plog, resid, lay.W1, lay.b1, lay.w2, float(lay.b2[0]),
                               cfg.tau_min, cfg.tau_max))


def _pool_run(job):
    import numpy as np

    import oracle
    e0, e1, h = job
    lay, layout, args = _POOL
    x = lay.x[e0:e1, :h] if layout == "nhwc" else lay.x[e0:e1, :, :h]
    oracle.forward(np.ascontiguousarray(x), layout, *args)
    return e1 - e0


class OraclePool:
    """The oracle, as it stands, run on every host core: one spawned process per core (spawn,
    so it is safe after CUDA has started), each on a share of the sample's examples."""

    def __init__(self, cfg, seed: int, n_ex: int, h_rows: int):
        import multiprocessing as mp
        try:
            cores = len(os.sched_getaffinity(0))
        except AttributeError:
            cores = os.cpu_count() or 1
        self.procs = max(1, min(cores, n_ex))
        self.jobs = [(i * n_ex // self.procs, (i + 1) * n_ex // self.procs, h_rows)
                     for i in range(self.procs)]
        self.pool = mp.get_context("spawn").Pool(self.procs, initializer=_pool_init,
                                                 initargs=(cfg, seed))

    def run(self) -> float:
        """One pass over the sample; its wall time in seconds."""
        t0 = time.perf_counter()
        self.pool.map(_pool_run, self.jobs)
        return time.perf_counter() - t0

    def close(self):
        self.pool.close()
        self.pool.join()


def oracle_parallel_run(cfg, seed: int, n_ex: int, h_rows: int, budget_s: float):
    """Median wall time of one all-cores pass over n_ex examples x h_rows rows, and the
    number of processes."""
    pool = OraclePool(cfg, seed, n_ex, h_rows)
    try:
        pool.run()  # warm
        times, start = [], time.perf_counter()
        while True:
            times.append(pool.run())
            if time.perf_counter() - start >= budget_s or len(times) >= 200:
                break
    finally:
        pool.close()
    return statistics.median(times), pool.procs


def run_reference(args, cfg):
    """The reference arm: the CPU oracle, timed as it stands, on the host cores."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from paper_2608_23794_gb300 import synth
    import oracle
    oracle.build()
    lay = synth.make_layer(cfg, seed=SEED)
    pidx, plog, resid = oracle.pack(lay.support_idx, lay.support_logits, cfg.C_in)
    args_o = (pidx, plog, resid, lay.W1, lay.b1, lay.w2, float(lay.b2[0]), cfg.tau_min, cfg.tau_max)
    t0 = time.perf_counter()
    oracle.forward(lay.x[:1], cfg.layout, *args_o)
    t_ex = max(time.perf_counter() - t0, 1e-6)
    # each step is a bounded sample so that warmup + steps fit in about two minutes (sized
    # from one example on one core; the steps run on every core)
    per_step = 120.0 / max(1, args.steps + args.warmup)
    n_ex = int(max(1, min(cfg.N, per_step / t_ex)))
    h_rows = cfg.H if t_ex <= per_step else int(max(1, cfg.H * per_step / t_ex))
    pool = OraclePool(cfg, SEED, n_ex, h_rows)
    try:
        for _ in range(args.warmup):
            pool.run()
        dt = sum(pool.run() for _ in range(args.steps)) / max(1, args.steps)
    finally:
        pool.close()
    sub = cfg.replace(N=n_ex, H=h_rows)
    value = workload_bytes(sub, len(resid)) / dt / 1e9
    sample = (f"{n_ex} of {cfg.N} examples x {h_rows} of {cfg.H} rows per step, split over "
              f"{pool.procs} processes")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded; stands in for ImageNet activations)",
        "config": {"workload": cfg.name, "N": cfg.N, "H": cfg.H, "W": cfg.W, "C_in": cfg.C_in,
                   "C_out": cfg.C_out, "k": cfg.k, "sample": sample},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": pool.procs, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ our arm


def run_ours(args, cfg):
    import numpy as np
    import torch

    from paper_2608_23794_gb300 import build as moce_build
    from paper_2608_23794_gb300 import costmodel, moce, synth

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    moce_build.build()

    from paper_2608_23794_gb300 import dist as mdist
    lay = synth.make_layer(cfg, seed=mdist.shard_seed(SEED, rank))
    bits = torch.from_numpy(lay.x_bits.view(np.int16)).view(torch.bfloat16)
    cu = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).to(device=dev, dtype=dt)
    W1, b1, w2, b2 = (cu(lay.W1, torch.float32), cu(lay.b1, torch.float32),
                      cu(lay.w2, torch.float32), cu(lay.b2, torch.float32))
    sidx, slog = cu(lay.support_idx, torch.int32), cu(lay.support_logits, torch.float32)

    # one-time packing (Sec. 3.2: supports are static at inference)
    moce.moce_pack_supports(sidx, slog, cfg.C_in)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    packed = moce.moce_pack_supports(sidx, slog, cfg.C_in)
    e1.record()
    torch.cuda.synchronize()
    pack_us = e0.elapsed_time(e1) * 1e3

    # rotate input/output copies so that every timed step reads x from HBM
    props = torch.cuda.get_device_properties(dev)
    l2 = getattr(props, "L2_cache_size", 0) or 132 * 2**20
    x_bytes = bits.numel() * 2
    n_rot = max(2, int(np.ceil(3 * l2 / x_bytes)) + 1)
    xs = [bits.to(dev) for _ in range(n_rot)]
    ys = [torch.empty((cfg.N, cfg.H, cfg.W, cfg.C_out + 1), dtype=torch.bfloat16, device=dev)
          for _ in range(n_rot)]
    ws = moce.Workspace(cfg.N, cfg.H, cfg.W, cfg.C_in, cfg.C_out, cfg.k, device=dev)
    fwd = lambda i: moce.moce_forward(xs[i % n_rot], "nhwc", packed, W1, b1, w2, b2, cfg.tau_min,
                                      cfg.tau_max, ws=ws, y=ys[i % n_rot], path=args.path)
    launches_per_step = moce.moce_forward_launches(xs[0], "nhwc", cfg.C_out, cfg.k, path=args.path)
    kernel_name = moce.moce_forward_kernel(xs[0], "nhwc", cfg.C_out, cfg.k, path=args.path)

    for i in range(args.warmup):
        fwd(i)
    torch.cuda.synchronize()
    moce.moce_check_device_error(ws)

    K = args.steps
    t_begin, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(gpu_uuid(torch, dev))
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    t_begin.record()
    for i in range(K):
        fwd(i)
    t_end.record()
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    clocks = sampler.stop()
    moce.moce_check_device_error(ws)
    # the forward's own launch duration (roofline), in a separate loop with an
    # event pair around every launch (events between launches add gaps, so the
    # headline loop above has none)
    Kl = min(K, 2000)
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(Kl)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(Kl)]
    for i in range(Kl):
        starts[i].record()
        fwd(i)
        ends[i].record()
    torch.cuda.synchronize()
    moce.moce_check_device_error(ws)
    total_ms = t_begin.elapsed_time(t_end)
    launch_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    total_ms = mdist.max_over_ranks(total_ms, device=dev)
    ms_per_step = total_ms / K
    nbytes = workload_bytes(cfg, packed.n_resid)
    value = mdist.job_throughput(nbytes * K, world, total_ms * 1e-3) / 1e9

    # roofline of the forward (one launch on the stream path; on the step path
    # the event pair spans its launches): the binding one of the HBM floor
    # (algorithmic bytes at the measured copy bandwidth) and the FP32 floor
    # (routed + gate MACs at the FMA peak of the SM count and maximum clock)
    peaks, peak_src = measured_peaks()
    kern_s = statistics.mean(launch_ms) * 1e-3
    flops = costmodel.layer_flops(cfg.N, cfg.H, cfg.W, cfg.C_in, cfg.C_out, cfg.k,
                                  packed.n_resid)
    macs = flops["routed_macs"] + flops["gate_macs"]
    fma_peak = fp32_fma_peak(props.multi_processor_count, peaks.get("sm_max_mhz", 2070.0))
    hbm_floor = nbytes / (peaks["hbm_gbs"] * 1e9)
    fma_floor = macs / fma_peak
    kern_label = (kernel_name if launches_per_step == 1 else
                  f"{kernel_name} ({launches_per_step} launches)")
    if hbm_floor >= fma_floor:
        achieved = nbytes / kern_s / 1e9
        # the data sheet's figure beside the measured copy: memory clock x 2 transfers x 8192 bits
        nominal = peaks.get("mem_max_mhz", 3996.0) * 1e6 * 2 * 8192 / 8 / 1e9
        roofline = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                    "frac": achieved / peaks["hbm_gbs"],
                    "traffic": ncu_traffic(cfg.name, kernel_name),
                    "peak_source": f"{peak_src} (burst copy)", "kernel": kern_label,
                    "algorithmic_bytes_per_launch": nbytes,
                    "nominal_peak": nominal, "frac_of_nominal": achieved / nominal}
    else:
        achieved = macs / kern_s / 1e12
        roofline = {"bound": "alu", "achieved": achieved, "peak": fma_peak / 1e12,
                    "unit": "T FMA/s", "frac": achieved * 1e12 / fma_peak, "traffic": None,
                    "peak_source": f"derived: {FP32_LANES_PER_SM} FP32 lanes x "
                                   f"{props.multi_processor_count} SMs x "
                                   f"{peaks.get('sm_max_mhz', 2070.0):.0f} MHz",
                    "kernel": kern_label, "algorithmic_macs_per_launch": macs}
        sgemm = sgemm_fma_rate(dev)
        roofline["sgemm_check"] = {"value": sgemm / 1e12, "unit": "T FMA/s",
                                   "frac_of_derived_peak": sgemm / fma_peak,
                                   "what": "cuBLAS SGEMM 8192^3, no TF32"}
    floors = {"hbm_us": hbm_floor * 1e6, "fp32_fma_us": fma_floor * 1e6,
              "binding": roofline["bound"], "measured_us": kern_s * 1e6,
              "frac_of_binding": max(hbm_floor, fma_floor) / kern_s}

    # dense 1x1 comparator: cuBLAS bf16 GEMM [P x C_in] x [C_in x C_out]
    P = cfg.N * cfg.H * cfg.W
    Wd = torch.randn(cfg.C_in, cfg.C_out, device=dev, dtype=torch.bfloat16)
    outs = [torch.empty(P, cfg.C_out, device=dev, dtype=torch.bfloat16) for _ in range(n_rot)]
    for i in range(20):
        torch.matmul(xs[i % n_rot].view(P, cfg.C_in), Wd, out=outs[i % n_rot])
    torch.cuda.synchronize()
    Kd = min(K, 2000)
    e0.record()
    for i in range(Kd):
        torch.matmul(xs[i % n_rot].view(P, cfg.C_in), Wd, out=outs[i % n_rot])
    e1.record()
    torch.cuda.synchronize()
    dense_us = e0.elapsed_time(e1) * 1e3 / Kd
    dense_bytes = P * cfg.C_in * 2 + P * cfg.C_out * 2 + cfg.C_in * cfg.C_out * 2

    # end to end through the public API: pinned host x -> device, forward, y -> pinned host.
    # Pipelined across steps: a copy stream brings step i + 1's x into the other device buffer
    # while the compute stream runs step i's forward and reads its y back; every step's two
    # copies are inside the timed region.
    x_host = bits.pin_memory()
    y_host = [torch.empty(ys[0].shape, dtype=torch.bfloat16).pin_memory() for _ in range(2)]
    x_dev, y_dev = [xs[0], xs[1 % n_rot]], [ys[0], ys[1 % n_rot]]
    ws2 = [ws, moce.Workspace(cfg.N, cfg.H, cfg.W, cfg.C_in, cfg.C_out, cfg.k, device=dev)]
    cs, ks = torch.cuda.Stream(device=dev), torch.cuda.current_stream()
    ev_in = [torch.cuda.Event(), torch.cuda.Event()]
    ev_done = [torch.cuda.Event(), torch.cuda.Event()]

    def e2e_run(K):
        with torch.cuda.stream(cs):
            cs.wait_stream(ks)
            x_dev[0].copy_(x_host, non_blocking=True)
            ev_in[0].record(cs)
        for i in range(K):
            b, nb = i & 1, (i & 1) ^ 1
            if i + 1 < K:
                with torch.cuda.stream(cs):
                    if i >= 1:
                        cs.wait_event(ev_done[nb])  # step i - 1 no longer reads x_dev[nb]
                    x_dev[nb].copy_(x_host, non_blocking=True)
                    ev_in[nb].record(cs)
            ks.wait_event(ev_in[b])
            moce.moce_forward(x_dev[b], "nhwc", packed, W1, b1, w2, b2, cfg.tau_min, cfg.tau_max,
                              ws=ws2[b], y=y_dev[b], path=args.path)
            y_host[b].copy_(y_dev[b], non_blocking=True)
            ev_done[b].record(ks)

    Ke = max(3, min(K, 200))
    e2e_run(3)
    torch.cuda.synchronize()
    e0.record()
    e2e_run(Ke)
    e1.record()
    torch.cuda.synchronize()
    e2e_s = e0.elapsed_time(e1) * 1e-3 / Ke
    e2e_s = mdist.max_over_ranks(e2e_s, device=dev)
    e2e = {"value": mdist.job_throughput(nbytes, world, e2e_s) / 1e9, "unit": UNIT,
           "h2d_bytes_per_step": x_bytes, "d2h_bytes_per_step": y_host[0].numel() * 2,
           "us_per_layer": e2e_s * 1e6,
           "note": "step i + 1's x copy overlaps step i's forward and y copy (two streams)"}

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        gbs, sample, t_rep, n_ex, h_rows = oracle_sample_run(lay, cfg, args.cpu_seconds)
        # the same sample on every host core (one process per core, examples split)
        t_par, procs = oracle_parallel_run(cfg, mdist.shard_seed(SEED, rank), n_ex, h_rows,
                                           args.cpu_seconds)
        nb = workload_bytes(cfg.replace(N=n_ex, H=h_rows), packed.n_resid)
        cpu = {"value": nb / t_par / 1e9, "unit": UNIT, "cores": procs, "kind": "oracle",
               "sample": f"{n_ex} of {cfg.N} examples x {h_rows} of {cfg.H} rows split over "
                         f"{procs} processes, median of all-core passes",
               "single_thread": {"value": gbs, "cores": 1, "sample": sample}}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "us_per_layer": ms_per_step * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32", "data": DATA[cfg.activation],
            "config": {"workload": cfg.name, "N": cfg.N, "H": cfg.H, "W": cfg.W,
                       "C_in": cfg.C_in, "C_out": cfg.C_out, "k": cfg.k, "n_resid": packed.n_resid,
                       "path": kernel_name,
                       "storage_dtype": cfg.dtype, "layout": cfg.layout,
                       "l2": f"inputs rotate over {n_rot} copies ({n_rot * x_bytes / 2**20:.0f} MiB"
                             f" > 3x the {l2 / 2**20:.0f} MiB L2)",
                       "parallelism": f"batch shard x{world} (no collective)"},
            "roofline": roofline,
            "floors": floors,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": launches_per_step * K,
            "clocks": clocks,
            "pack_us": pack_us,
            "dense_cublas": {"us_per_layer": dense_us, "GB/s": dense_bytes / dense_us / 1e3,
                             "moce_speedup": dense_us / (ms_per_step * 1e3)},
            "macs": {"routed": flops["routed_macs"], "gate": flops["gate_macs"],
                     "dense_equiv": flops["dense_equiv_flops"] // 2},
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def run_train(args, cfg):
    """Support maintenance on the layer's routing matrix L [C_out, C_in] (Sec. 3.2 TopK, Sec. 3.4
    coverage loss and gradient): device time per call, GB/s of the algorithmic bytes, and the
    oracle on one host core beside it."""
    import numpy as np
    import torch

    from paper_2608_23794_gb300 import build as moce_build
    from paper_2608_23794_gb300 import moce

    torch.cuda.set_device(0)
    moce_build.build()
    R, C, k = cfg.C_out, cfg.C_in, cfg.k
    rng = np.random.default_rng(SEED)
    L = rng.standard_normal((R, C)).astype(np.float32)
    dL = torch.from_numpy(L).cuda()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(fn, reps):
        for _ in range(max(3, args.warmup)):
            fn()
        torch.cuda.synchronize()
        e0.record()
        for _ in range(reps):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / reps

    reps = max(10, min(args.steps, 2000))
    topk_us = timed(lambda: moce.moce_topk_supports(dL, k), reps)
    cov_us = timed(lambda: moce.moce_coverage_loss(dL, 1e-8), reps)
    cov_nograd_us = timed(lambda: moce.moce_coverage_loss(dL, 1e-8, grad=False), reps)
    topk_bytes = R * C * 4 + R * k * 8
    cov_bytes = 2 * R * C * 4  # L read once, the gradient written once
    cpu = None
    if not args.no_cpu_baseline:
        import oracle
        oracle.build()
        t0 = time.perf_counter()
        oracle.topk(L, k)
        t1 = time.perf_counter()
        oracle.coverage(L, 1e-8)
        t2 = time.perf_counter()
        cpu = {"topk_us": (t1 - t0) * 1e6, "coverage_us": (t2 - t1) * 1e6, "cores": 1,
               "kind": "oracle", "sample": f"the whole {R} x {C} routing matrix, one run"}
    peaks, _ = measured_peaks()
    line = {"metric": "MoCE support maintenance: TopK over the routing matrix + coverage loss and "
                      "gradient (µs per call, GB/s of algorithmic bytes)",
            "value": cov_bytes / cov_us / 1e3, "unit": UNIT, "n_gpus": 1, "steps": reps,
            "warmup": args.warmup, "higher_is_better": True, "dtype": "f32",
            "data": "synthetic (seeded N(0,1) routing logits)",
            "config": {"workload": cfg.name, "C_out": R, "C_in": C, "k": k, "op": "train"},
            "topk": {"us": topk_us, "GB/s": topk_bytes / topk_us / 1e3,
                     "note": "the call is synchronous (it validates): device time between events "
                             "includes the error-word copy"},
            "coverage_with_grad": {"us": cov_us, "GB/s": cov_bytes / cov_us / 1e3,
                                   "frac_of_hbm": cov_bytes / cov_us / 1e3 / peaks["hbm_gbs"]},
            "coverage_loss_only": {"us": cov_nograd_us},
            "gpu_launches": 6 * reps,
            "cpu_baseline": cpu}
    print(json.dumps(line), flush=True)


def run_backward(args, cfg):
    """The layer's backward with static supports (Sec. 3.2) at the workload's full size: device
    time per call (inputs rotated so every call reads x and dy from HBM), GB/s of the algorithmic
    bytes (x and dy read once, dx written once in fp32) against the HBM peak, and the oracle's
    backward on one host core over a sample of examples."""
    import numpy as np
    import torch

    from paper_2608_23794_gb300 import build as moce_build
    from paper_2608_23794_gb300 import moce, synth

    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    moce_build.build()
    lay = synth.make_layer(cfg, seed=SEED)
    dyv, dyb = synth.make_dy(cfg, seed=SEED)
    s = 2 if cfg.dtype == "bf16" else 4
    if cfg.dtype == "bf16":
        x = torch.from_numpy(lay.x_bits.view(np.int16)).view(torch.bfloat16)
        dy = torch.from_numpy(dyb.view(np.int16)).view(torch.bfloat16)
    else:
        x, dy = torch.from_numpy(lay.x), torch.from_numpy(dyv)
    cu = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).to(device=dev, dtype=dt)
    W1, b1, w2, b2 = (cu(lay.W1, torch.float32), cu(lay.b1, torch.float32),
                      cu(lay.w2, torch.float32), cu(lay.b2, torch.float32))
    packed = moce.moce_pack_supports(cu(lay.support_idx, torch.int32),
                                     cu(lay.support_logits, torch.float32), cfg.C_in)
    R, k, C = cfg.C_out, cfg.k, cfg.C_in
    M = cfg.N * cfg.H * cfg.W
    alg_bytes = M * C * s + M * (R + 1) * s + M * C * 4
    props = torch.cuda.get_device_properties(dev)
    l2 = getattr(props, "L2_cache_size", 0) or 132 * 2**20
    n_rot = max(2, int(np.ceil(3 * l2 / alg_bytes)) + 1)
    xs = [x.to(dev) for _ in range(n_rot)]
    dys = [dy.to(dev) for _ in range(n_rot)]
    f32 = dict(dtype=torch.float32, device=dev)
    outs = [moce.Gradients(torch.empty(x.shape, **f32), torch.empty((R, k), **f32),
                           torch.empty((k, k), **f32), torch.empty(k, **f32),
                           torch.empty(k, **f32), torch.empty(1, **f32)) for _ in range(n_rot)]
    ws = torch.empty(moce.moce_backward_workspace_bytes(cfg.N, cfg.H, cfg.W, C, R, k),
                     dtype=torch.uint8, device=dev)
    bwd = lambda i: moce.moce_backward(xs[i % n_rot], dys[i % n_rot], cfg.layout, packed, W1, b1,
                                       w2, b2, cfg.tau_min, cfg.tau_max, ws=ws,
                                       out=outs[i % n_rot])
    for i in range(max(3, args.warmup)):
        bwd(i)
    torch.cuda.synchronize()
    K = max(3, min(args.steps, 500))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(gpu_uuid(torch, dev))
    sampler.start()
    time.sleep(0.3)
    torch.cuda.synchronize()
    e0.record()
    for i in range(K):
        bwd(i)
    e1.record()
    torch.cuda.synchronize()
    clocks = sampler.stop()
    us = e0.elapsed_time(e1) * 1e3 / K
    peaks, _ = measured_peaks()
    gbs = alg_bytes / us / 1e3
    cpu = None
    if not args.no_cpu_baseline:
        import oracle
        oracle.build()
        pidx, plog, resid = oracle.pack(lay.support_idx, lay.support_logits, C)
        n_ex, spent = 0, 0.0
        while n_ex < cfg.N and spent < min(args.cpu_seconds, 20.0):
            t0 = time.perf_counter()
            oracle.backward(lay.x[n_ex:n_ex + 1], dyv[n_ex:n_ex + 1], cfg.layout, pidx, plog,
                            resid, lay.W1, lay.b1, lay.w2, float(lay.b2[0]), cfg.tau_min,
                            cfg.tau_max)
            spent += time.perf_counter() - t0
            n_ex += 1
        cpu = {"value": spent / n_ex * cfg.N * 1e6, "unit": "µs per backward (extrapolated)",
               "cores": 1, "kind": "oracle",
               "sample": f"{n_ex} of {cfg.N} examples, one core, scaled to the whole batch"}
    line = {"metric": "MoCE backward µs/layer (static supports) & GB/s of algorithmic bytes",
            "value": gbs, "unit": UNIT, "n_gpus": 1, "steps": K, "warmup": args.warmup,
            "ms_per_step": us / 1e3, "us_per_layer": us, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": DATA[cfg.activation],
            "config": {"workload": cfg.name, "N": cfg.N, "H": cfg.H, "W": cfg.W, "C_in": C,
                       "C_out": R, "k": k, "storage_dtype": cfg.dtype, "layout": cfg.layout,
                       "op": "backward", "l2": f"{n_rot} rotating input copies (> L2)"},
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": gbs / peaks["hbm_gbs"], "traffic": None,
                         "note": "whole backward call (all its kernels), algorithmic bytes "
                                 "x + dy + dx(fp32)"},
            "clocks": clocks, "gpu_launches": None, "cpu_baseline": cpu}
    print(json.dumps(line), flush=True)


def run_dynamic(args, cfg):
    """Static supports against the input-conditioned variant of Eq. (dynamic) on the same layer
    and inputs (Sec. 5 compares the two): device µs per call of the whole layer for each, and of
    the paper's "routing-and-gather" path, i.e. the static indexed mix against the dynamic
    router (hidden layer, rank-d logits, per-example TopK, U(X)) plus the per-example mix. The
    mix kernels fuse the gather with the aggregation, so both sides include the aggregation."""
    import numpy as np
    import torch

    from paper_2608_23794_gb300 import build as moce_build
    from paper_2608_23794_gb300 import moce, synth

    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    moce_build.build()
    d = args.d
    lay = synth.make_layer(cfg, seed=SEED)
    xv, xb = synth.make_dynamic_x(cfg, seed=SEED)
    rt = synth.make_router(cfg, d, seed=SEED)
    cu = lambda a, dt=torch.float32: torch.from_numpy(np.ascontiguousarray(a)).to(dev, dt)
    x = (torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16) if xb is not None
         else torch.from_numpy(xv))
    router = moce.DynamicRouter(cu(rt["L"]), cu(rt["Wh"]), cu(rt["bh"]), cu(rt["V"]), cu(rt["Q"]))
    gate = (cu(lay.W1), cu(lay.b1), cu(lay.w2), cu(lay.b2))
    N, R, k, C = cfg.N, cfg.C_out, cfg.k, cfg.C_in
    # the static layer selects TopK of the same routing matrix, packed once
    idx_t, lg_t = moce.moce_topk_supports(router.logits, k)
    packed = moce.moce_pack_supports(idx_t, lg_t, C)
    s_el = 2 if cfg.dtype == "bf16" else 4
    x_bytes = N * cfg.H * cfg.W * C * s_el
    props = torch.cuda.get_device_properties(dev)
    l2 = getattr(props, "L2_cache_size", 0) or 132 * 2**20
    n_rot = max(2, int(np.ceil(3 * l2 / x_bytes)) + 1)
    xs = [x.to(dev) for _ in range(n_rot)]
    shape_y = (N, cfg.H, cfg.W, R + 1) if cfg.layout == "nhwc" else (N, R + 1, cfg.H, cfg.W)
    ys = [torch.empty(shape_y, dtype=xs[0].dtype, device=dev) for _ in range(n_rot)]
    ws = moce.Workspace(N, cfg.H, cfg.W, C, R, k, device=dev)
    dws = torch.empty(moce.moce_dynamic_workspace_bytes(N, cfg.H, cfg.W, C, R, k, d),
                      dtype=torch.uint8, device=dev)
    sup = moce._empty_supports(N, R, k, C, dev)
    z = moce.moce_pool(xs[0], cfg.layout)
    _, a_static = moce.moce_gate(z, packed, *gate, cfg.tau_min, cfg.tau_max)
    a_dyn = torch.empty((N, R, k), dtype=torch.float32, device=dev)
    moce.moce_dynamic_supports(z, router, k, ws=dws, out=sup)
    resid_static = packed.resid_idx
    K = max(3, min(args.steps, 500))

    def timed(fn):
        for i in range(max(3, args.warmup)):
            fn(i)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for i in range(K):
            fn(i)
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / K

    sampler = ClockSampler(gpu_uuid(torch, dev))
    sampler.start()
    time.sleep(0.3)
    t_static = timed(lambda i: moce.moce_forward(xs[i % n_rot], cfg.layout, packed, *gate,
                                                 cfg.tau_min, cfg.tau_max, ws=ws,
                                                 y=ys[i % n_rot]))
    t_dyn = timed(lambda i: moce.moce_forward_dynamic(xs[i % n_rot], cfg.layout, router, k, *gate,
                                                      cfg.tau_min, cfg.tau_max, ws=dws,
                                                      y=ys[i % n_rot]))
    t_mix_static = timed(lambda i: moce.moce_mix(xs[i % n_rot], cfg.layout,
                                                 packed.packed_idx.view(R, k), a_static,
                                                 resid_static, packed.n_resid, ws,
                                                 y=ys[i % n_rot]))
    t_route = timed(lambda i: moce.moce_dynamic_supports(z, router, k, ws=dws, out=sup))
    t_mix_dyn = timed(lambda i: moce.moce_mix(xs[i % n_rot], cfg.layout, sup.sup_idx, a_dyn,
                                              sup.resid_idx, sup.n_resid, ws, y=ys[i % n_rot]))
    clocks = sampler.stop()
    rg_static = t_mix_static
    rg_dyn = t_route + t_mix_dyn
    line = {"metric": "MoCE static vs input-conditioned supports (Eq. dynamic): µs per layer and "
                      "routing-and-gather ratio",
            "value": rg_dyn / rg_static, "unit": "x (dynamic / static routing-and-gather time)",
            "n_gpus": 1, "steps": K, "warmup": args.warmup, "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": DATA[cfg.activation] +
            "; per-example channel means N(0, 0.25) so the router sees different descriptors",
            "config": {"workload": cfg.name, "N": N, "H": cfg.H, "W": cfg.W, "C_in": C,
                       "C_out": R, "k": k, "d": d, "storage_dtype": cfg.dtype,
                       "layout": cfg.layout, "op": "dynamic",
                       "l2": f"{n_rot} rotating input copies (> L2)"},
            "static": {"layer_us": t_static, "mix_us": t_mix_static},
            "dynamic": {"layer_us": t_dyn, "route_us": t_route, "mix_us": t_mix_dyn,
                        "route_note": "router hidden layer, rank-d logits of every (expert, "
                                      "channel), per-example TopK, U(X)"},
            "ratio_layer": t_dyn / t_static,
            "ratio_routing_and_gather": rg_dyn / rg_static,
            "paper_ratio_routing_and_gather": 13.5 / 1.9,
            "clocks": clocks, "gpu_launches": None}
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    from paper_2608_23794_gb300 import synth
    cfg = synth.CONFIGS[args.workload]
    if args.batch is not None:
        cfg = cfg.replace(N=args.batch)
    if args.op == "train":
        run_train(args, cfg)
        return
    if args.op == "backward":
        run_backward(args, cfg)
        return
    if args.op == "dynamic":
        run_dynamic(args, cfg)
        return
    if args.impl == "ours" and (cfg.dtype, cfg.layout) != ("bf16", "nhwc"):
        raise SystemExit(f"bench.py times bf16 NHWC layers; {cfg.name} is {cfg.dtype} {cfg.layout}")
    if args.impl == "reference":
        run_reference(args, cfg)
    else:
        run_ours(args, cfg)


if __name__ == "__main__":
    main()
