"""Benchmark: QuantEase layer quantization on GB300 (one JSON line on stdout).

Workload (default): the Falcon-180B-shaped MLP down projection, q = 14848 rows,
p = 59392 inputs, n = 65536 calibration tokens, bf16 W and X (synthetic,
seeded), 3 bits, 10 CD sweeps: the largest single-GPU layer of the paper's
workloads (Sigma alone is 14.1 GB, resident in HBM).  One step = build
Sigma = X X^T, then quantize the layer: the whole hot path, inputs resident in
HBM.  --config names any other workload of paper_2309_01885_gb300.inputs.

metric / unit: CD column-updates per second (q p^2 per sweep, summed over the
step's bit-widths) over the whole step including the Sigma build; the JSON line
also carries the layer quantize time, Sigma TFLOP/s and the CD-phase rate, and
the rooflines of the Sigma GEMM and of the CD sweep separately.

--impl reference times the fp64 CPU oracle (the reference arm) on a bounded
sample of the same workload (rows are independent given Sigma).

Multi-GPU (torchrun): every rank quantizes its own layer (weak scaling, no
collective on the data path); timing is the max over ranks.
"""
from __future__ import annotations

import argparse
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

METRIC = ("layer quantize time; CD column-updates/s (q·p²/s) and Σ TFLOP/s vs roofline")
UNIT = "q·p² column-updates/s"
DEFAULT_CONFIG = "falcon180b_down_14848x59392"
DTYPE = ("16-bit tensor-core products, fp32 accumulation (Σ: bf16 X x bf16 X; CD GEMMs fp32-accurate: Σ̄ in two row-scaled fp16 planes against operands exact in fp16, three bf16 planes otherwise; binary32 decisions, near-ties decided in double-float)")


def max_over_ranks(x: float, device) -> float:
    """The slowest rank's value of x (the job ends when its last replica ends); x itself on
    one rank or outside a process group."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: float, world: int, ms: float) -> float:
    """Whole-job units per second: every rank processes units_per_rank per step (weak
    scaling, independent layers) and the step takes the slowest rank's ms."""
    return units_per_rank * world / (ms / 1e3)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="qe", choices=["qe", "reference"])
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--cpu-rows", type=int, default=0,
                    help="oracle rows in the CPU sample (0 = about 10 s of host work)")
    ap.add_argument("--structured", action="store_true",
                    help="outlier workloads: keep whole columns (Sec. 4.3, structured outliers)")
    ap.add_argument("--dense-sweeps", type=int, default=0,
                    help="sweeps whose cross-block term uses the tensor-core GEMM (0 = the library's "
                         "adaptive schedule)")
    ap.add_argument("--group-size", type=int, default=0,
                    help="grouped grids: a scale and zero-point per row and group of this many columns")
    ap.add_argument("--relax", type=int, default=0,
                    help="relax heuristic period R (Sec. 3.2): sweeps t with t mod R = 0, t < iters, unquantized")
    ap.add_argument("--tokens", type=int, default=0,
                    help="override n (calibration tokens), for small profiling captures only")
    ap.add_argument("--rows", type=int, default=0,
                    help="override q (rows of W), for small profiling captures only")
    return ap.parse_args()


def plan_sweeps(iters, relax, dense):
    """The sweep schedule of qe_quantize_layer, mirrored: per sweep its kind and
    window ("first": classic sweep 1 + a residual refresh with the objective; "seq":
    a relaxed sweep or the one after it, three-plane changes; "dense": tensor-core
    window sweep; "list": change-list sweep), the residual refreshes without the
    objective, and the change-list launches (one per run of list sweeps, per 32)."""
    def relaxed(t):
        return relax > 0 and (t + 1) % relax == 0 and t + 1 < iters
    sweeps, refreshes, list_runs = [], 0, []
    t, src = 0, "w"
    if not relaxed(0):
        sweeps.append(("first", 0))
        t, src = 1, "codes"
    exact, chain = True, False
    while t < iters:
        if relaxed(t) or src != "codes":
            if not exact and not chain:
                refreshes += 1
                exact = True
            sweeps.append(("seq", -1 if exact else 1))
            src = "v" if relaxed(t) else "codes"
            t += 1
            exact, chain = False, True
            if src == "codes" and t < iters:
                refreshes += 1
                exact, chain = True, False
            continue
        tend = t
        while tend < iters and not relaxed(tend):
            tend += 1
        while t < tend and t < dense:
            sweeps.append(("dense", -1 if exact else 1))
            t += 1
            exact, chain = False, False
        while t < tend:
            te = min(tend, t + 32)
            list_runs.append(te - t)
            sweeps += [("list", 0)] * (te - t)
            t = te
            exact, chain = False, False
    return sweeps, refreshes, list_runs


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            m = json.load(fh)
        return dict(hbm=float(m["hbm_gbs"]), bf16=float(m["bf16_tflops"]),
                    bf16_sustained=float(m["bf16_tflops_sustained"]), source="measured")
    except (OSError, KeyError, ValueError):
        return dict(hbm=6800.0, bf16=1900.0, bf16_sustained=1700.0, source="fallback")


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
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
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax = float(parts[2])
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() in ("active", "1", "yes"):
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


# Committed DRAM-traffic figures (profiles/roofline_traffic.json): per kernel, the
# bytes one launch moved in one ncu capture, keyed by a hash of the sources the
# tensor-core GEMM is compiled from and launched by; null once those sources change.
TRAFFIC_SOURCES = ("qe_api.cu", "qe_common.cuh", "qe_gemm.cu", "qe_internal.h", "qe_kernels.h")


def traffic_sources_sha256() -> str:
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2309_01885_gb300", "csrc")
    for name in TRAFFIC_SOURCES:
        with open(os.path.join(csrc, name), "rb") as fh:
            h.update(name.encode() + b"\0" + fh.read())
    return h.hexdigest()


def traffic_record(key: str, workload: str):
    """(DRAM bytes per launch, note) of kernel `key` on `workload` from the committed ncu
    summary, if the kernel sources are unchanged since it was taken; else (None, why)."""
    path = os.path.join(ROOT, "profiles", "roofline_traffic.json")
    try:
        with open(path) as fh:
            rec = json.load(fh)
    except (OSError, ValueError):
        return None, "no committed capture"
    entry = rec.get(workload, {}).get(key)
    if not entry:
        return None, "no committed capture for this workload"
    if entry.get("sources_sha256") != traffic_sources_sha256():
        return None, "kernel sources changed since the capture"
    return entry.get("dram_bytes_per_launch"), entry.get("note", "")


def gemm_tiles_sigma(p):
    """Tiles of the Sigma GEMM that run (128 x 256, on or above the diagonal)."""
    return sum(1 for m0 in range(0, p, 128) for n0 in range(0, p, 256) if n0 + 256 > m0)


def tensor_peak(pk, clk):
    """The bf16 peak a kernel timed inside this run is held to: the burst figure when the
    sampled clocks stayed at their maximum with no power cap, else the sustained one."""
    if clk and not clk.get("reasons") and clk.get("sm_max_mhz") and clk["sm_mhz"] >= 0.97 * clk["sm_max_mhz"]:
        return pk["bf16"], f"{pk['source']} bf16 dense burst (MEASURED_PEAKS.json; clocks at max, no power cap)"
    return pk["bf16_sustained"], (f"{pk['source']} bf16 dense sustained (MEASURED_PEAKS.json; "
                                  f"clock reasons {clk.get('reasons') if clk else 'unsampled'})")


def roofline_tensor(kernel, flops, exec_flops, ms, launches, peak, peak_src, traffic, traffic_note, **extra):
    """A tensor-bound roofline entry: achieved = algorithmic flops / measured time."""
    if ms <= 0:
        return None
    achieved = flops / (ms / 1e3) / 1e12
    return {"bound": "tensor", "kernel": kernel, "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
            "frac": achieved / peak, "traffic": traffic, "traffic_note": traffic_note,
            "launches_per_step": launches, "ms_per_step": ms,
            "executed_tflops": exec_flops / (ms / 1e3) / 1e12 if exec_flops else None,
            "peak_source": peak_src, **extra}


def roofline_lists(bytes_per_launch, ms, launches, pk):
    """The change-list CD kernel against the HBM roofline.  Algorithmic bytes of one list
    sweep: the residual R (4 q p), the codes (q p) and fp32 Sigma_bar (4 p^2) read once;
    the gathers of Sigma_bar rows re-read it from L2 and are not counted."""
    if ms <= 0 or launches <= 0:
        return None
    achieved = bytes_per_launch * launches / (ms / 1e3) / 1e9
    return {"bound": "hbm", "kernel": "k_cd_rows_lists<256>", "achieved": achieved, "peak": pk["hbm"],
            "unit": "GB/s", "frac": achieved / pk["hbm"], "launches_per_step": launches, "ms_per_step": ms,
            "peak_source": f"{pk['source']} HBM copy bandwidth (MEASURED_PEAKS.json)"}


def oracle_rows(p, threads, target_s=10.0):
    """Rows of a CPU-oracle sample worth about target_s seconds on `threads` host threads
    (a row sweep costs p^2 column updates at roughly 3.5e8 per second per thread), in
    whole rounds of the threads."""
    per_thread = max(1, int(round(target_s * 3.5e8 / (p * p))))
    return threads * per_thread


def cpu_oracle_sample(W64, S, bits, rows, sweeps, threads=0):
    """Time Algorithm 1 of the fp64 oracle on a row sample (on `threads` host threads,
    0 = all); S binary64 or binary32 (promoted exactly); returns (units/s, seconds,
    threads used)."""
    import numpy as np
    import oracle
    O = oracle.get()
    s, z = O.grid(W64[:rows], bits)
    old = O.threads(threads)
    used = O.threads(0)
    try:
        t0 = time.perf_counter()
        O.alg1(np.ascontiguousarray(W64[:rows]), S, s, z, bits, sweeps)
        dt = time.perf_counter() - t0
    finally:
        O.threads(old)
    p = W64.shape[1]
    return rows * p * p * sweeps / dt, dt, used


def run_reference(args):
    """The reference arm: the fp64 CPU oracle, on a bounded sample per step."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import numpy as np
    from paper_2309_01885_gb300 import inputs
    import oracle
    O = oracle.get()
    cfg = inputs.CONFIGS[args.config]
    threads = O.threads(0)   # the OpenMP threads the oracle's row loops use
    rows = args.cpu_rows or oracle_rows(cfg.p, threads)
    rows = max(1, min(cfg.q, rows))
    W = inputs.layer_weights(rows, cfg.p, dtype=cfg.w_dtype, seed=cfg.seed, device="cpu").double().numpy()
    # Sigma from a few tokens: the oracle's CD cost depends on p, not on Sigma's values.
    # Wide layers: a binary32 Sigma (the oracle promotes it exactly, half the host
    # memory) from a numpy product of a 32-token X; this input is not timed.
    n_ref = 4096 if cfg.p <= 16384 else 32
    X = inputs.calib_inputs(cfg.p, n_ref, dtype=cfg.x_dtype, seed=cfg.seed, device="cpu",
                            heavy_frac=cfg.heavy_frac, heavy_mult=cfg.heavy_mult)
    if cfg.p <= 16384:
        S = O.sigma(X.double().numpy())
    else:
        X32 = X.float().numpy()
        S = X32 @ X32.T
    del X
    times = []
    for step in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        for b in cfg.bits:
            cpu_oracle_sample(W, S, b, rows, 1)
        dt = time.perf_counter() - t0
        if step >= args.warmup:
            times.append(dt)
    units = rows * cfg.p * cfg.p * len(cfg.bits)
    ms = 1e3 * sum(times) / len(times)
    value = units / (ms / 1e3)
    sample = (f"Algorithm 1 (fp64 oracle) on {rows} of {cfg.q} rows, 1 sweep per bit-width "
              f"{list(cfg.bits)}, p={cfg.p}, Sigma from {n_ref} tokens; rows are independent given Sigma")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": cfg.name, "q": cfg.q, "p": cfg.p, "n": cfg.n, "bits": list(cfg.bits),
                       "sweeps": cfg.iters},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def layer_schedule(q, p, iters, forms, relax, dense_opt, adaptive, grouped, outlier, structured,
                   w_planes, B=256):
    """Per layer (one quantize call): algorithmic and executed flops of the trailing
    GEMMs, residual refreshes besides P, the sweeps by form and the launches of our
    kernels, mirrored from the library's schedule.  forms: the library's record of each
    sweep's form (0 sequential, 1 dense, 2 lists)."""
    nblk = -(-p // B)
    blocks = [(b0, min(B, p - b0)) for b0 in range(0, p, B)]
    tri_flops = sum(2 * q * bw * b0 for b0, bw in blocks)     # columns left of each block
    win_flops = sum(2 * q * bw * p for b0, bw in blocks)      # the last p column visits
    if outlier:
        plan, extra, list_runs = [("first", 0)] + [("list", 0)] * (iters - 1), 0, []
    elif relax:
        plan, extra, list_runs = plan_sweeps(iters, relax, dense_opt or 1)
    else:
        plan, extra, list_runs = [], 0, []
        run = 0
        for t, f in enumerate(forms):
            if f == 0:
                plan.append(("first", 0))
            elif f == 1:
                plan.append(("dense", -1 if plan and plan[-1][0] == "first" else 1))
            else:
                plan.append(("list", 0))
            if f == 2 and not adaptive:
                run += 1
                if run == 32:
                    list_runs.append(run)
                    run = 0
            elif run:
                list_runs.append(run)
                run = 0
        if run:
            list_runs.append(run)
    trail_flops = trail_exec = 0
    for kind, window in plan:
        if kind in ("first", "seq", "dense"):
            f = win_flops if window == 1 else tri_flops
            trail_flops += f
            # integer changes of a window sweep: one fp16 plane x two fp16 planes of Sigma_bar
            # (2 products); real-valued or grouped changes: three bf16 planes (6 products)
            # the first sweep's real changes scaled into two fp16 planes: 3 products
            if grouped:
                npr = 6
            elif kind == "dense":
                npr = 2
            elif kind == "first":
                npr = 3
            else:
                npr = 6
            trail_exec += npr * f
    refreshes = (1 if plan[0][0] == "first" else 0) + extra
    # launches: set-up (grid, Sigma diagonal, Sigma_bar planes, 1/d, packed blocks,
    # Sigma_bar rows, [W planes], P, initial residual); sweep 1: nblk - 1 trailing GEMMs
    # + nblk in-block + residual GEMM + objective sum; a dense or sequential sweep:
    # trailing GEMMs (nblk - 1 when its window starts empty) + nblk in-block + objective
    # step, a dense one also nblk near-tie checks; fixed schedule: one list launch and
    # one objective prefix per run of <= 32 list sweeps; adaptive schedule: every sweep
    # after the first enqueues both forms (trailing GEMMs, in-block, near-tie checks,
    # objective step, list launch, objective prefix) and all but the last the two switch
    # kernels; an extra refresh: C - z + residual GEMM
    per = 8 + w_planes + 2 * extra
    if outlier:
        # selection (P_s: 3 radix digit passes + count, scan, emit; columns: + 2 norm
        # kernels + emit), start: copy, selection, scatter + row pointers, grid,
        # Sigma_bar set-up (5) + [W planes] + P, 64 power steps (+ fill, last, final),
        # SpMM refresh, initial residual; sweep 1 blocked (2 nblk - 1), later sweeps one
        # change-list launch and an objective prefix, sweep 1 a residual GEMM + objective
        # sum; per iteration: IHT target, selection, scatter + row pointers, SpMM, objective (2)
        sel = 9 if structured else 6
        per = (1 + sel + 2 + 1 + 6 + w_planes + 67 + 1 + 1 + (2 * nblk - 1) + 2 * (iters - 1) + 2
               + iters * (1 + sel + 2 + 1 + 2))
    elif adaptive:
        per += (nblk - 1) + nblk + 2
        for t in range(1, iters):
            per += (nblk - (1 if t == 1 else 0)) + 2 * nblk + 3 + (2 if t + 1 < iters else 0)
    else:
        per += 2 * len(list_runs)
        for kind, window in plan:
            if kind == "first":
                per += (nblk - 1) + nblk + 2
            elif kind in ("seq", "dense"):
                per += (nblk if window == 1 else nblk - 1) + nblk + 1 + (nblk if kind == "dense" else 0)
    counts = {k: sum(1 for kd, _ in plan if kd == k) for k in ("first", "seq", "dense", "list")}
    return dict(trail_flops=trail_flops, trail_exec=trail_exec, refreshes=refreshes, launches=per,
                sweeps_by_form=counts, plan=plan)


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    import numpy as np
    import torch
    import torch.distributed as dist
    from paper_2309_01885_gb300 import inputs, qe
    from paper_2309_01885_gb300.build import build_lib

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if rank == 0:
        build_lib()
    if world > 1:
        dist.barrier()
    qe.load()

    cfg = inputs.CONFIGS[args.config]
    import dataclasses
    if args.tokens:
        cfg = dataclasses.replace(cfg, n=args.tokens)
    if args.rows:
        cfg = dataclasses.replace(cfg, q=args.rows)
    q, p, n = cfg.q, cfg.p, cfg.n
    cfg_r = dataclasses.replace(cfg, seed=cfg.seed + rank)   # each rank owns a different layer
    W = cfg_r.weights("cuda")
    X = cfg_r.inputs("cuda")
    Sigma = torch.empty(p, p, dtype=torch.float32, device="cuda")
    outlier = cfg.s_budget > 0                    # the outlier-aware workload (Algorithm 4)
    grouped = 0 < args.group_size < p
    ws = torch.empty(qe.qe_workspace_size(q, p, outlier=outlier, group_size=args.group_size), dtype=torch.uint8,
                     device="cuda")

    def quantize(Wt, b, timer=None, forms=False):
        if outlier:
            return qe.qe_quantize_layer_outlier(Wt, Sigma, b, cfg.iters, cfg.s_budget, workspace=ws,
                                                structured=args.structured, timer=timer)
        return qe.qe_quantize_layer(Wt, Sigma, b, cfg.iters, workspace=ws, timer=timer,
                                    dense_sweeps=args.dense_sweeps, relax_period=args.relax,
                                    group_size=args.group_size, record_forms=forms)
    stream = torch.cuda.current_stream()
    nb = len(cfg.bits)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(nb + 2)]
          for _ in range(args.steps)]

    def step(events=None, timer=None):
        if events:
            events[0].record(stream)
        qe.qe_build_sigma(X, Sigma=Sigma)
        if events:
            events[1].record(stream)
        outs = []
        for k, b in enumerate(cfg.bits):
            outs.append(quantize(W, b, timer))
            if events:
                events[2 + k].record(stream)
        return outs

    for _ in range(args.warmup):
        step()
    st = qe.qe_sync_status()
    if st != qe.QE_OK:
        raise RuntimeError(f"device status {qe.qe_status_string(st)}")

    clocks = ClockSampler(local)
    clocks.start()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    # the kernels are timed by CUDA events that the library records around each of its
    # launches on this stream (the Sigma GEMM by the step's own events around qe_build_sigma,
    # whose only launch it is)
    nblk = (p + 255) // 256                    # default column block width 256
    kinds = [qe.QE_KERNEL_PINIT_GEMM, qe.QE_KERNEL_RESIDUAL_GEMM, qe.QE_KERNEL_TRAIL_GEMM,
             qe.QE_KERNEL_CD_BLOCK, qe.QE_KERNEL_CD_LISTS]
    cap_layer = 8 + 2 * nblk * (cfg.iters + 1) + 2 * cfg.iters
    dom = qe.Timer(kinds, capacity=args.steps * nb * cap_layer + 16)
    t_start.record(stream)
    outs = None
    for k in range(args.steps):
        outs = step(ev[k], dom)
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    total_ms = t_start.elapsed_time(t_end)
    sigma_ms = [e[0].elapsed_time(e[1]) for e in ev]
    cd_ms = [[e[1 + k].elapsed_time(e[2 + k]) for e in ev] for k in range(nb)]
    ms = max_over_ranks(total_ms / args.steps, "cuda")
    timed = {k: dom.read(k) for k in kinds}
    dom.close()

    # per-class breakdown of one extra, untimed step (events around every launch), which
    # also records the form each sweep took
    brk = qe.Timer(kinds, capacity=nb * cap_layer + 16)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    qe.qe_build_sigma(X, Sigma=Sigma)
    e1.record(stream)
    forms = []
    for b in cfg.bits:
        o = quantize(W, b, brk, forms=not outlier)
        forms.append(o["sweep_forms"].tolist() if "sweep_forms" in o else [])
    torch.cuda.synchronize()
    names = {qe.QE_KERNEL_PINIT_GEMM: "pinit_gemm", qe.QE_KERNEL_RESIDUAL_GEMM: "residual_gemm",
             qe.QE_KERNEL_TRAIL_GEMM: "trail_gemm", qe.QE_KERNEL_CD_BLOCK: "cd_block",
             qe.QE_KERNEL_CD_LISTS: "cd_lists"}
    breakdown = {"sigma_gemm": {"launches": 1, "ms": e0.elapsed_time(e1)}}
    for k, nm in names.items():
        n_, ms_ = brk.read(k)
        breakdown[nm] = {"launches": n_, "ms": ms_}
    brk.close()

    # the library's schedule, mirrored: adaptive when the fp32 Sigma_bar rows exceed
    # three quarters of L2 (and no fixed dense_sweeps is asked for)
    l2 = getattr(torch.cuda.get_device_properties(local), "L2_cache_size", 128 << 20)
    ld = -(-p // 64) * 64
    adaptive = (not outlier and not args.relax and args.dense_sweeps == 0 and 4 * p * ld > 0.75 * l2)
    w_planes = 0 if cfg.w_dtype == torch.bfloat16 else 1
    sched = [layer_schedule(q, p, cfg.iters, forms[k], args.relax, args.dense_sweeps, adaptive, grouped,
                            outlier, args.structured, w_planes) for k in range(nb)]

    units_per_step = q * p * p * cfg.iters * nb           # column updates per rank per step
    value = job_throughput(units_per_step, world, ms)
    sig_flops = p * (p + 1) * n                            # symmetric half of X X^T
    sigma_avg = statistics.mean(sigma_ms)
    cd_avg = [statistics.mean(x) for x in cd_ms]
    pk = peaks()
    peak_tc, peak_src = tensor_peak(pk, clk)

    result = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
              "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
              "vs_baseline": None, "dtype": DTYPE, "data": "synthetic",
              "config": {"workload": cfg.name, "q": q, "p": p, "n": n, "bits": list(cfg.bits),
                         "sweeps": cfg.iters, "parallelism": f"layer-replicas x{world}",
                         **({"relax_period": args.relax} if args.relax else {}),
                         **({"group_size": args.group_size} if grouped else {}),
                         **({"dense_sweeps": args.dense_sweeps} if args.dense_sweeps else {}),
                         "l2": "inputs larger than L2 (X is %.2f GiB)" % (p * n * 2 / 2**30),
                         **({"s_budget": cfg.s_budget,
                             "outliers": "columns" if args.structured else "entries"} if outlier else {})},
              "layer_quantize_ms": ms,
              "sigma_ms": sigma_avg,
              "sigma_tflops": sig_flops / (sigma_avg / 1e3) / 1e12,
              "sigma_dense_equiv_tflops": 2 * p * p * n / (sigma_avg / 1e3) / 1e12,
              "cd_ms": {str(b): v for b, v in zip(cfg.bits, cd_avg)},
              "cd_updates_per_s": units_per_step / (sum(cd_avg) / 1e3),
              "sweep_forms": {str(b): f for b, f in zip(cfg.bits, forms)},
              "sweeps_by_form": {str(b): sc["sweeps_by_form"] for b, sc in zip(cfg.bits, sched)},
              "clocks": clk}

    # ---- rooflines ------------------------------------------------------------------
    qpad, ppad, kpad = -(-q // 128) * 128, -(-p // 256) * 256, -(-p // 64) * 64
    # (1) the Sigma GEMM alone: p(p+1)n algorithmic flops (the symmetric half) over its
    #     own CUDA-event time; executed = the 128 x 256 tiles on or above the diagonal
    sig_exec = gemm_tiles_sigma(p) * 2 * 128 * 256 * n
    tr, tr_note = traffic_record("k_tc_gemm_sigma", cfg.name)
    r_sigma = roofline_tensor("k_tc_gemm<256> Sigma = X X^T", sig_flops, sig_exec, sigma_avg, 1, peak_tc, peak_src,
                              tr, tr_note)
    # (2) the CD sweep: K q p^2 column updates of 2 flops each per layer (one combined
    #     rank-1 update per column, Sec. 3.2) over the whole quantize calls (grid, P,
    #     residual refreshes, every sweep); the CD GEMMs (P, residual refreshes, trailing
    #     corrections) execute 3 or 6 bf16 plane products per algorithmic product
    cd_alg = 2.0 * q * p * p * cfg.iters * nb
    gemm_cd_ms = sum(timed[k][1] for k in kinds[:3]) / args.steps
    gemm_cd_launches = sum(timed[k][0] for k in kinds[:3]) // args.steps
    gemm_cd_alg = sum(2 * q * p * p * (1 + sc["refreshes"]) + sc["trail_flops"] for sc in sched)
    # P: bf16 W as one fp16 plane x two fp16 planes (2 products), fp32 W in three bf16 planes x
    # three (6); residual: C - z x two fp16 planes (2), grouped: 6
    p_prods = 2 if cfg.w_dtype == torch.bfloat16 else 6
    gemm_cd_exec = sum((p_prods + (6 if grouped else 2) * sc["refreshes"]) * 2 * qpad * ppad * kpad
                       + sc["trail_exec"] for sc in sched)
    r_cd = roofline_tensor("CD sweep (all kernels of the quantize calls)", cd_alg, None, sum(cd_avg), None,
                           peak_tc, peak_src, None, "per-kernel traffic under the gemm and list entries",
                           cd_gemm={"kernel": "k_tc_gemm<256> P, residual, trailing corrections",
                                    "ms_per_step": gemm_cd_ms, "launches_per_step": gemm_cd_launches,
                                    "algorithmic_tflops": gemm_cd_alg / (gemm_cd_ms / 1e3) / 1e12 if gemm_cd_ms else None,
                                    "executed_tflops": gemm_cd_exec / (gemm_cd_ms / 1e3) / 1e12 if gemm_cd_ms else None,
                                    "frac_executed": (gemm_cd_exec / (gemm_cd_ms / 1e3) / 1e12 / peak_tc)
                                    if gemm_cd_ms else None},
                           split_factor=("per algorithmic product: 2 fp16 products where one operand is exact in "
                                         "fp16 (window sweeps' integer changes, C - z, bf16 W), 3 for the first "
                                         "sweep's real changes, 6 bf16 products for relaxed sweeps and grouped "
                                         "grids; ceiling of the algorithmic fraction about 1/2"))
    # (3) k_tc_gemm<256> over all its launches in a step (Sigma + the CD GEMMs)
    gemm_ms = sigma_avg + gemm_cd_ms
    tr, tr_note = traffic_record("k_tc_gemm_step", cfg.name)
    r_gemm = roofline_tensor("k_tc_gemm<256> (Sigma, P, residual, trailing)", sig_flops + gemm_cd_alg,
                             sig_exec + gemm_cd_exec, gemm_ms, 1 + gemm_cd_launches, peak_tc, peak_src,
                             tr, tr_note)
    # (4) the change-list kernel against HBM (when lists ran)
    list_launches, list_ms = timed[qe.QE_KERNEL_CD_LISTS]
    n_list = sum(sc["sweeps_by_form"]["list"] for sc in sched)
    r_lists = None
    if n_list and list_ms > 0:
        lb = n_list * (4 * q * p + q * p + 4 * p * p)
        r_lists = roofline_lists(lb / max(1, n_list), list_ms / args.steps, n_list, pk)
    # the dominant kernel by time share is the line's roofline; the others sit beside it
    shares = {"k_tc_gemm": gemm_ms, "k_cd_rows_lists": list_ms / args.steps,
              "k_cd_block": timed[qe.QE_KERNEL_CD_BLOCK][1] / args.steps}
    top = max(shares, key=shares.get)
    result["roofline"] = dict(r_lists if (top == "k_cd_rows_lists" and r_lists) else r_gemm)
    result["roofline"]["sigma"] = r_sigma
    result["roofline"]["cd"] = r_cd
    if r_lists:
        result["roofline"]["lists"] = r_lists
    result["roofline"]["time_share"] = {k: v / ms for k, v in shares.items()}
    # ideal step: per phase max(algorithmic flops / tensor peak, algorithmic bytes / HBM), summed
    peak_f, hbm = peak_tc * 1e12, pk["hbm"] * 1e9
    cd_flops, cd_bytes = 2.0 * q * p * p * cfg.iters, 15.0 * q * p * cfg.iters   # ~15 B per coordinate per sweep
    ideal_s = (max(sig_flops / peak_f, 2.0 * p * n / hbm)
               + sum(max(2.0 * q * p * p * (1 + sc["refreshes"]) / peak_f, 12.0 * q * p * (1 + sc["refreshes"]) / hbm)
                     + max(cd_flops / peak_f, cd_bytes / hbm) for sc in sched))
    result["ideal"] = {"ms_per_step": ideal_s * 1e3, "frac": ideal_s * 1e3 / ms,
                       "model": ("per phase max(algorithmic flops / bf16 peak, algorithmic bytes / measured HBM): "
                                 "Sigma p(p+1)n flops vs X read once; per layer P and residual refreshes 2qp^2 "
                                 "flops each; CD 2qp^2 flops per sweep vs ~15 bytes per coordinate per sweep")}
    result["kernel_ms_per_step"] = breakdown
    # launches of our kernels per step (the schedule of qe_quantize_layer, mirrored)
    result["gpu_launches"] = args.steps * (1 + sum(sc["launches"] for sc in sched))

    # end to end through the C ABI with host buffers
    if not args.no_e2e:
        Xh = X.cpu().pin_memory()
        Wh = W.cpu().pin_memory()
        Wd = torch.empty_like(W)
        # X stays on the host: qe_build_sigma_host streams it in token chunks through
        # device buffers, one per chunk, so the next step's copies run while this step's
        # CD computes.  Copies that overlap more of the change-list sweeps (two steps'
        # worth of buffers, or one whole-X copy per step) measured slower: the copied
        # bytes pass through L2 and evict the Sigma_bar rows those sweeps gather.  At
        # least four chunks per step, each at most 65536 tokens.
        # fp32 X (the OPT-125m-sized layer) is copied whole and reduced on the device:
        # the streamed form takes bf16 chunks only.
        streamed = X.dtype == torch.bfloat16
        chunk = min(65536, max(8192, (n // 4) // 64 * 64)) if streamed else n
        staging = qe.sigma_host_staging(p, chunk, nbuf=max(2, -(-n // chunk))) if streamed else None
        Xd = None if streamed else torch.empty_like(X)
        host_out = [dict(codes=torch.empty(q, p, dtype=torch.uint8).pin_memory(),
                         scales=torch.empty(q).pin_memory(), zeros=torch.empty(q).pin_memory(),
                         obj=torch.empty(cfg.iters, dtype=torch.float64).pin_memory())
                    for _ in cfg.bits]

        def e2e_step():
            Wd.copy_(Wh, non_blocking=True)
            if streamed:
                qe.qe_build_sigma_host(Xh, Sigma, staging, chunk)
            else:
                Xd.copy_(Xh, non_blocking=True)
                qe.qe_build_sigma(Xd, Sigma=Sigma)
            for k, b in enumerate(cfg.bits):
                o = quantize(Wd, b)
                for key in ("codes", "scales", "zeros", "obj"):
                    host_out[k][key].copy_(o[key], non_blocking=True)

        e2e_step()                     # untimed: creates the copy stream and its events
        # a step's copies overlap the previous step's compute, which the first step
        # after the synchronize has not got: time at least 10 steps when steps are short
        e2e_steps = max(args.steps, 10) if ms < 1000 else max(args.steps, 3)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        e0.record(stream)
        for _ in range(e2e_steps):
            e2e_step()
        e1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, "cuda")
        h2d = X.numel() * X.element_size() + W.numel() * W.element_size()
        d2h = nb * (q * p + 4 * q + 4 * q + 8 * cfg.iters)
        result["e2e"] = {"value": job_throughput(units_per_step, world, e2e_ms), "unit": UNIT,
                         "ms_per_step": e2e_ms, "steps": e2e_steps, "h2d_bytes_per_step": h2d,
                         "d2h_bytes_per_step": d2h, "chunk_tokens": chunk}
        del Xh, Wh, Xd, staging, host_out

    st = qe.qe_sync_status()
    if st != qe.QE_OK:
        raise RuntimeError(f"device status {qe.qe_status_string(st)}")

    # CPU baseline: the fp64 oracle on a row sample of the same layer, given this
    # layer's binary32 Sigma (promoted exactly) (rank 0, N = 1 only)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        del X
        torch.cuda.empty_cache()
        threads = oracle.get().threads(0)
        rows = max(1, min(q, args.cpu_rows or oracle_rows(p, threads)))
        W64 = W[:rows].double().cpu().numpy()
        S32 = Sigma.cpu().numpy()
        rate, dt, threads = cpu_oracle_sample(W64, S32, cfg.bits[0], rows, 1)
        rows1 = max(1, rows // threads if rows >= threads else 1)
        rate1, dt1, _ = cpu_oracle_sample(W64, S32, cfg.bits[0], rows1, 1, threads=1)
        result["cpu_baseline"] = {
            "value": rate, "unit": "q·p² column-updates/s (CD only)", "cores": threads,
            "kind": "oracle",
            "sample": (f"Algorithm 1 (fp64 oracle) on {rows} of {q} rows x 1 sweep, {cfg.bits[0]}-bit, "
                       f"given this layer's Sigma; {dt:.1f} s"),
            "single_core": {"value": rate1, "cores": 1,
                            "sample": f"the same on {rows1} rows and one host thread; {dt1:.1f} s"}}
        result["obj_last"] = {str(b): float(o["obj"][-1].item()) for b, o in zip(cfg.bits, outs)}

    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
