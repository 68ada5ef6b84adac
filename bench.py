"""Benchmark: lane value+grad evaluations per second of the NDVM tape replay on GB300.

One step = the whole hot path over one batch: 200 seeded random-expression programs
(grammar + - * / exp log|x| sin pow-int, depth <= 6, 1-8 constants), each replayed
forward and in reverse over B = 4096 parameter lanes and 256 data points (MSE loss)
-- 819,200 lane value+grad evaluations.  Inputs are resident in HBM before the timed
region; L2 is flushed between timed steps.  Prints one JSON line: the headline
configuration's numbers, and under "configs" the same measurement of every other
configuration (exp-decay, logistic f64 and f32, the two Kalman filters, the 64-state
population), each with a bounded CPU-oracle baseline, and the 200 programs at 64 lanes
each (launch-bound) timed both as one call per program on the streams and as one
batched ndvm_value_and_grad_multi call.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
                    [--config C] [--dtype f32] [--only]

Under N processes (one per GPU) the population has N x 4096 lanes per program; rank r
replays lanes [4096 r, 4096 (r + 1)) of every program (weak scaling) and rank 0 gathers
the slices of loss and gradient on the host after the timed region.

--impl reference times the oracle (the plain CPU reference evaluator) on the host
cores instead, on a bounded sample of the same workload.
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

N_PROGRAMS, B_LANES, N_POINTS, SEED = 200, 4096, 256, 1234
METRIC = "lane value+grad evals/sec (fp64, 1 GB300) and % of FP64/HBM roofline"
UNIT = "lane-evals/s"

def measured_hbm_gbs():
    """HBM copy bandwidth measured on the GB300s, else the recipe's fallback."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "MEASURED_PEAKS.json hbm_gbs (measured copy)"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback 6.8 TB/s"


def kernel_sources_digest():
    """SHA-256 over the replay library's sources (names and bytes, sorted by name)."""
    import hashlib
    d = os.path.join(ROOT, "paper_2607_03574_gb300", "csrc")
    h = hashlib.sha256()
    for name in sorted(os.listdir(d)):
        path = os.path.join(d, name)
        if os.path.isfile(path):
            h.update(name.encode())
            with open(path, "rb") as f:
                h.update(f.read())
    return h.hexdigest()


def recorded_traffic(cfg: int, dtype: str, lanes: int, n_programs: int):
    """DRAM bytes (read + write) per replay launch from the committed ncu summary of this
    workload, if the library's sources are the ones it was taken from; else None."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    if rec.get("sources_sha256") != kernel_sources_digest() or dtype != "f64":
        return None
    if lanes or (cfg == 2 and n_programs != N_PROGRAMS):
        return None
    ent = rec.get("per_launch", {}).get(str(cfg))
    return None if ent is None else float(ent["dram_bytes"])


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(ms: float, device=None) -> float:
    """Step time of the whole job: the slowest rank's (no data-path collective exists)."""
    import torch
    import torch.distributed as dist
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size() == 1:
        return ms
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


class ClockSampler:
    """nvidia-smi clock/throttle samples taken during the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except (OSError, ValueError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

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
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


DEFAULT_LANES = {1: 64, 2: B_LANES, 3: 16384, 4: 8192, 5: 65536, 6: 1024}
DESCRIPTIONS = {1: "exp-decay y = a exp(-b t) + c: {B} lanes x 50 points, MSE",
                3: "logistic Euler (stack bytecode): {B} lanes x 1000 steps, 100 obs, MSE",
                4: "4-state constant-velocity Kalman NLL: {B} lanes x {T} steps",
                5: "8-state random stable Kalman NLL: {B} lanes x {T} steps",
                6: "64-state Kalman NLL population, 8-d observations: {B} lanes x {T} steps"}
DEFAULT_T = {4: 200, 5: 1000, 6: 50}


def population(args, cfg: int, world: int = 1, rank: int = 0, lanes_per_rank: int = 0):
    """(this rank's Workloads, description, lanes per program in the whole population).

    One seeded population of world x lanes_per_rank lanes per program (the generator's
    population at that size); this rank's Workloads hold its slice of the lanes
    (shard.lane_slice), the same programs and observations on every rank."""
    from dataclasses import replace

    from paper_2607_03574_gb300.shard import lane_slice
    B_rank = lanes_per_rank or DEFAULT_LANES[cfg]
    B_total = B_rank * world
    if cfg == 2:
        progs = W.random_exprs(n_programs=args.programs, B=B_total, n_points=N_POINTS, seed=SEED)
        desc = (f"random-expression programs: {len(progs)} programs x {B_total} lanes x {N_POINTS} points, MSE")
    else:
        T = (getattr(args, "T", 0) or DEFAULT_T[cfg]) if cfg in DEFAULT_T else None
        progs = [W.config(cfg, B=B_total, seed=SEED, **({"T": T} if T else {}))]
        desc = DESCRIPTIONS[cfg].format(B=B_total, T=T)
    lo, hi = lane_slice(B_total, world, rank)
    local = [replace(w, params=w.params[lo:hi]) for w in progs]
    return local, desc, B_total


def workload_for(args, seed=SEED):
    """(list of Workloads, description) of the configuration being measured, one process."""
    progs, desc, _ = population(args, args.config, 1, 0, args.lanes)
    return progs, f"{desc}, {args.dtype} value+grad"


def cpu_sample_lanes(args, progs):
    """Oracle lanes per program for a CPU sample of about 10-30 s on 16 cores."""
    if args.cpu_lanes:
        return min(args.cpu_lanes, progs[0].B)
    return 2048 if args.config == 2 else progs[0].B


def oracle_sample_time(progs, lanes_per_prog: int, nthreads: int, f32: bool = False, min_seconds: float = 0.0,
                       tile: bool = True):
    """Time the oracle on a bounded sample: `lanes_per_prog` lanes of every program,
    repeated until at least `min_seconds` have passed (small workloads)."""
    import oracle
    oracle.build()
    t0 = time.perf_counter()
    n = 0
    while True:
        for w in progs:
            p = w.params[:lanes_per_prog]
            if tile and len(p) < 1024:  # small populations: tile the lanes so thread start-up does not dominate
                p = np.resize(p, (1024, p.shape[1]))
            if f32:
                p = p.astype(np.float32).astype(np.float64)
            oracle.run(w.program, p, w.obs, frontend=w.frontend, nthreads=nthreads, f32=f32)
            n += len(p)
        if time.perf_counter() - t0 >= min_seconds:
            return n, time.perf_counter() - t0


def cpu_baseline(args, progs):
    """The oracle timed on the host cores: every core on a bounded sample (about 10-30 s
    of CPU work), and one core on a sample sized from that rate to take about 2 s."""
    cores = os.cpu_count() or 1
    f32 = args.dtype == "f32"
    lanes = cpu_sample_lanes(args, progs)
    oracle_sample_time(progs[:2], 2, cores, f32)
    n, dt = oracle_sample_time(progs, lanes, cores, f32, min_seconds=2.0)
    rate = n / dt
    per_core = rate / cores
    progs1 = progs[:max(1, min(len(progs), 8))]
    lanes1 = int(min(lanes, max(1, per_core * 2.0 / len(progs1))))
    n1, dt1 = oracle_sample_time(progs1, lanes1, 1, f32, min_seconds=0.5, tile=False)
    return {"value": rate, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{lanes} lanes of each of the {len(progs)} program(s), repeated to {n} lane evals ({dt:.1f} s)",
            "single_core": {"value": n1 / dt1, "unit": UNIT, "cores": 1,
                            "sample": f"{lanes1} lanes of each of {len(progs1)} program(s), repeated to {n1} lane "
                                      f"evals ({dt1:.1f} s)"}}


def bounded_cpu_baseline(progs, f32: bool, seconds: float = 2.0):
    """The oracle on every host core over a sample sized to take about `seconds`: a short
    probe on a few lanes gives the rate, which sizes the timed sample (a prefix of the
    population's lanes, the same for every program)."""
    cores = os.cpu_count() or 1
    probe = max(1, min(progs[0].B, cores))
    n, dt = oracle_sample_time(progs, probe, cores, f32, tile=False)
    lanes = int(min(progs[0].B, max(probe, (n / dt) * seconds / len(progs))))
    n, dt = oracle_sample_time(progs, lanes, cores, f32, tile=False)
    return {"value": n / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"the first {lanes} of {progs[0].B} lanes of each of the {len(progs)} program(s): "
                      f"{n} lane evals in {dt:.1f} s"}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    cores = os.cpu_count() or 1
    progs, workload = workload_for(args, SEED)
    lanes = min(args.ref_lanes, progs[0].B)
    f32 = args.dtype == "f32"
    for _ in range(args.warmup):
        oracle_sample_time(progs[:4], 2, cores, f32)
    ns, dts = [], []
    for _ in range(args.steps):  # a step: the sample, repeated to at least a second for small workloads
        n, dt = oracle_sample_time(progs, lanes, cores, f32, min_seconds=1.0)
        ns.append(n)
        dts.append(dt)
    ms = 1e3 * float(np.mean(dts))
    value = float(np.sum(ns)) / float(np.sum(dts))
    sample = (f"{lanes} lanes of each of the {len(progs)} program(s), whole data set "
              f"({int(np.mean(ns))} lane evals per step)")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": args.dtype, "data": "synthetic", "config": {"workload": workload, "sample": sample},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


NOMINAL_FP64_TFLOPS = 1.25  # GB300 nominal FP64 rate (context)
FP64_DFMA_PER_CLK_PER_SM = 2.0  # the FP64 pipe: 16 active cycles per 32-lane warp instruction (ncu)


def fp64_pipe_peak(sms: int) -> tuple[float, str]:
    """Peak FP64 rate from unit counts and clocks (flop/s, 2 per DFMA): 2 DFMA per clock
    per SM x SMs x the maximum SM clock (MEASURED_PEAKS.json sm_max_mhz, else 2070 MHz)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            mhz, src = float(json.load(f)["sm_max_mhz"]), "MEASURED_PEAKS.json sm_max_mhz"
    except (OSError, KeyError, ValueError):
        mhz, src = 2070.0, "GB300 maximum SM clock 2070 MHz"
    return (2.0 * FP64_DFMA_PER_CLK_PER_SM * sms * mhz * 1e6,
            f"FP64 pipe peak from unit counts: {FP64_DFMA_PER_CLK_PER_SM:g} DFMA/clk/SM x {sms} SMs x {mhz:g} MHz "
            f"({src}); ncu's FP64-pipe utilisation is relative to the same rate")


def measure(nd, dev, local_progs, B_total, cfg, dtype, args, world, rank, peaks, want_gather, batched=False):
    """Time one configuration: W warm-up steps, then K timed steps of a captured CUDA
    graph of one whole step (every program of this rank's slice), L2 flushed before
    each; then the same work end to end through the host-buffer entry point.  With
    `batched`, one step is one ndvm_value_and_grad_multi call over every program (end to
    end: pinned host copies in, the call, copies out) instead of one call per program on
    the streams.  Returns the measurement and, on rank 0 when want_gather, the population
    gathered from every rank's slice."""
    import torch

    tdt = torch.float32 if dtype == "f32" else torch.float64
    npdt = np.float32 if dtype == "f32" else np.float64
    progs = local_progs
    t0 = time.perf_counter()
    tapes = [nd.trace_build(w.program, w.frontend) for w in progs]
    trace_s = time.perf_counter() - t0
    params = [torch.tensor(w.params, dtype=tdt, device=dev) for w in progs]
    obs = [torch.tensor(w.obs, dtype=tdt, device=dev) for w in progs]
    loss = [torch.empty(w.B, dtype=tdt, device=dev) for w in progs]
    grad = [torch.empty_like(p) for p in params]
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)  # > 129 MB L2
    stream = torch.cuda.current_stream(dev)
    work = 0.0
    alg_bytes = 0.0  # saved intermediates written once and read once, params, loss, grad, obs
    esz = np.dtype(npdt).itemsize
    for tp, w in zip(tapes, progs):
        c = tp.cost()
        work += (c["work_fwd"] + c["work_rev"]) * w.B + c["work_shared"]
        alg_bytes += (2 * c["save_elems"] + 2 * w.P + 1) * esz * w.B + esz * w.obs.size

    # independent programs run on several streams so their kernels co-reside on the SMs
    n_streams = min(args.streams, len(tapes))
    side = [torch.cuda.Stream(dev) for _ in range(n_streams)]

    def step():
        cur = torch.cuda.current_stream(dev)  # the capture stream while a graph is captured
        if batched:
            nd.value_and_grad_multi(tapes, params, obs, loss=loss, grad=grad, stream=cur)
            return
        if n_streams <= 1:
            for k in range(len(tapes)):
                nd.value_and_grad(tapes[k], params[k], obs[k], loss=loss[k], grad=grad[k], stream=cur)
            return
        start = torch.cuda.Event()
        start.record(cur)
        done = []
        for j, s in enumerate(side):
            s.wait_event(start)
            for k in range(j, len(tapes), n_streams):
                nd.value_and_grad(tapes[k], params[k], obs[k], loss=loss[k], grad=grad[k], stream=s)
            e = torch.cuda.Event()
            e.record(s)
            done.append(e)
        for e in done:
            cur.wait_event(e)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    # the timed step replays a CUDA graph of one whole step (all programs, all streams):
    # host launch overhead is paid once at capture, as a deployed calibration loop would
    per_step_launches = 0
    graph = None
    if args.graph:
        l_cap = nd.launch_count()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            step()
        per_step_launches = nd.launch_count() - l_cap
        graph.replay()
        torch.cuda.synchronize()
    run_step = graph.replay if graph is not None else step

    clocks = ClockSampler(dev.index)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    l0 = nd.launch_count()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    wall0 = time.perf_counter()
    for i in range(args.steps):
        flush.zero_()
        ev[i][0].record(stream)
        run_step()
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    if world > 1:
        torch.distributed.barrier()
    launches = nd.launch_count() - l0 + per_step_launches * args.steps
    step_ms = [a.elapsed_time(b) for a, b in ev]
    ms = max_over_ranks(float(statistics.median(step_ms)), dev)
    ms_mean = max_over_ranks(float(np.mean(step_ms)), dev)
    clk = clocks.stop()
    lanes_per_step = sum(w.B for w in progs) * world
    value = lanes_per_step / (ms * 1e-3)
    for t in tapes:
        nd.check_device(t)

    gathered = None
    if want_gather and world > 1:
        from paper_2607_03574_gb300.shard import gather_lanes
        ok = True
        for k in range(len(tapes)):
            ll, gg = loss[k].double().cpu().numpy(), grad[k].double().cpu().numpy()
            gl = gather_lanes(ll, B_total, world, rank, group=args.host_group)
            gg_all = gather_lanes(gg, B_total, world, rank, group=args.host_group)
            if rank == 0:
                ok &= gl.shape == (B_total,) and gg_all.shape == (B_total, gg.shape[1])
                ok &= bool(np.array_equal(gl[: len(ll)], ll)) and bool(np.array_equal(gg_all[: len(gg)], gg))
        gathered = {"lanes_per_program": B_total, "programs": len(tapes), "rank0_slice_intact": bool(ok)}

    # ---- end to end through the host-buffer entry point (pinned host memory)
    hp = [torch.tensor(w.params, dtype=tdt).pin_memory().numpy() for w in progs]
    ho = [torch.tensor(w.obs, dtype=tdt).pin_memory().numpy() for w in progs]
    h2d = sum(a.nbytes for a in hp) + sum(a.nbytes for a in ho)
    d2h = sum(w.B * esz * (1 + w.P) for w in progs)
    hl = [torch.empty(w.B, dtype=tdt).pin_memory().numpy() for w in progs]
    hg = [torch.empty((w.B, w.P), dtype=tdt).pin_memory().numpy() for w in progs]

    if batched:
        # a batch caller's layout: every program's inputs packed in one pinned host buffer
        # and one device buffer (per-program views), likewise the outputs, so that one
        # copy moves each way
        def packed(shapes):
            n = sum(int(np.prod(sh)) for sh in shapes)
            h = torch.empty(n, dtype=tdt).pin_memory()
            d = torch.empty(n, dtype=tdt, device=dev)
            views, off = [], 0
            for sh in shapes:
                m = int(np.prod(sh))
                views.append((h[off:off + m].view(sh), d[off:off + m].view(sh)))
                off += m
            return h, d, views
        hin, din, vin = packed([tuple(w.params.shape) for w in progs] + [tuple(w.obs.shape) for w in progs])
        for (hv, _), a in zip(vin, [w.params for w in progs] + [w.obs for w in progs]):
            hv.copy_(torch.from_numpy(np.ascontiguousarray(a, dtype=npdt)))
        hout, dout, vout = packed([(w.B,) for w in progs] + [(w.B, w.P) for w in progs])
        n_p = len(progs)
        b_params, b_obs = [v[1] for v in vin[:n_p]], [v[1] for v in vin[n_p:]]
        b_loss, b_grad = [v[1] for v in vout[:n_p]], [v[1] for v in vout[n_p:]]

    def e2e_step():
        if batched:
            # one copy in, one batched call, one copy out, on one stream, then one wait
            cur = torch.cuda.current_stream(dev)
            din.copy_(hin, non_blocking=True)
            nd.value_and_grad_multi(tapes, b_params, b_obs, loss=b_loss, grad=b_grad, stream=cur)
            hout.copy_(dout, non_blocking=True)
            cur.synchronize()
            return
        # every program's copies and replay queued on the streams, then one wait
        for k in range(len(tapes)):
            nd.value_and_grad_host_async(tapes[k], hp[k], ho[k], hl[k], hg[k], stream=side[k % len(side)])
        for s in side:
            s.synchronize()

    e2e_step()
    e2e_times = []
    for _ in range(max(2, args.steps // 2)):
        t1 = time.perf_counter()
        e2e_step()
        e2e_times.append(time.perf_counter() - t1)
    e2e_value = lanes_per_step / float(np.median(e2e_times)) if world == 1 else None

    # ---- roofline of the replay kernel: the slower of the FP64 work at the FP64 pipe's
    # peak rate and the algorithmic bytes at the measured HBM bandwidth, against the
    # step's kernel time (all launches of a step; they overlap on the streams)
    pipe_peak, pipe_src, probe_peak = peaks
    achieved = 2.0 * work / (ms * 1e-3)  # flop/s (2 per DFMA-equivalent)
    hbm_gbs, hbm_src = measured_hbm_gbs()
    t_fp64, t_hbm = 2.0 * work / pipe_peak, alg_bytes / (hbm_gbs * 1e9)
    roofline = {
        "bound": "alu", "achieved": achieved / 1e12, "peak": pipe_peak / 1e12, "unit": "TFLOP/s",
        "frac": max(t_fp64, t_hbm) / (ms * 1e-3),
        "traffic": recorded_traffic(cfg, dtype, args.lanes or args.T, len(tapes)),
        "peak_source": pipe_src,
        "peak_probe": probe_peak / 1e12, "frac_of_probe": achieved / probe_peak,
        "probe_source": "DFMA stream measured in this process (8 chains/thread, 4x256 threads/SM): "
                        "ncu shows the FP64 pipe 84 % active there, one warp instruction per 19 cycles per SM",
        "nominal_peak": NOMINAL_FP64_TFLOPS, "frac_of_nominal": achieved / (NOMINAL_FP64_TFLOPS * 1e12),
        "work_dfma_per_step": work,
        "hbm_term": {"algorithmic_bytes_per_step": alg_bytes, "peak_gbs": hbm_gbs, "peak_source": hbm_src,
                     "ms_at_peak": 1e3 * t_hbm, "fp64_ms_at_peak": 1e3 * t_fp64,
                     "binds": "fp64" if t_fp64 >= t_hbm else "hbm"},
    }
    if t_hbm > t_fp64:
        roofline.update({"bound": "hbm", "achieved": alg_bytes / (ms * 1e-3) / 1e9, "peak": hbm_gbs, "unit": "GB/s"})
    if dtype == "f32":
        # the cost table counts FP64 work; the fp32 variant runs on the FP32 pipe, whose
        # rate is far higher, so no FP64 fraction describes it
        roofline.update({"frac": None, "frac_of_nominal": None, "frac_of_probe": None,
                         "note": "fp32 variant: the FP64 cost model does not apply; frac not reported"})
    out = {"value": value, "unit": UNIT, "ms_per_step": ms, "ms_per_step_mean": ms_mean,
           "step_ms": step_ms if world == 1 else None, "lanes_per_step": lanes_per_step,
           "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
           "gpu_launches": launches, "graph": graph is not None, "roofline": roofline, "clocks": clk,
           "wall_s_timed": wall, "trace_build_s": trace_s}
    if gathered is not None:
        out["gathered_on_rank0"] = gathered
    del tapes, params, obs, loss, grad, flush, graph
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return out


EXTRA = [(1, "f64"), (3, "f64"), (3, "f32"), (4, "f64"), (5, "f64"), (6, "f64")]
SMALL_LANES = 64  # lanes per program of the launch-bound batch measured both ways
PROBE_ITERS = 2000


def probe_costs():
    """Device time per call of every probed function, all SMs busy, and its ratio to a
    DFMA's (each probed call carries one FP64 add, which the ratio leaves in: subtract 1
    for the function alone).  With an ncu capture of the same launches (one per function,
    after one warm-up launch each), FP64-pipe instructions per call = the launch's
    smsp__inst_executed_pipe_fp64.sum x 32 / calls."""
    import torch
    import paper_2607_03574_gb300 as nd
    nd.load()
    torch.cuda.set_device(0)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    calls = 4 * PROBE_ITERS * sms * 4 * 256
    ns = {name: nd.measure_op_cost(name, PROBE_ITERS) for name in nd.PROBES}
    out = {"unit": "ns per call (device time, all SMs busy) and DFMA-equivalents (incl. one FP64 add)",
           "iters": PROBE_ITERS, "calls_per_launch": calls,
           "ns_per_call": ns, "dfma_equivalents": {k: v / ns["dfma"] for k, v in ns.items()}}
    print(json.dumps(out), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ndvm", choices=["ndvm", "reference"])
    ap.add_argument("--programs", type=int, default=N_PROGRAMS, help="programs per step (smaller for profiling)")
    ap.add_argument("--config", type=int, default=2, choices=[1, 2, 3, 4, 5, 6],
                    help="headline workload: 2 (default) random-expression programs; 1, 3, 4, 5 the other "
                         "configurations; 6 a 64-state Kalman population (block-cooperative lanes)")
    ap.add_argument("--dtype", default="f64", choices=["f64", "f32"])
    ap.add_argument("--only", action="store_true",
                    help="measure the headline configuration only (no per-configuration table)")
    ap.add_argument("--ref-lanes", type=int, default=256, help="oracle lanes per program per reference step")
    ap.add_argument("--cpu-lanes", type=int, default=0,
                    help="oracle lanes per program for cpu_baseline (default: 2048 for the random programs, "
                         "every lane otherwise)")
    ap.add_argument("--lanes", type=int, default=0, help="lanes per program and rank instead of the "
                                                         "configuration's (smaller cases for profiling)")
    ap.add_argument("--T", type=int, default=0, help="time steps of the Kalman configurations (4-6) instead of "
                                                     "theirs (smaller cases for profiling)")
    ap.add_argument("--streams", type=int, default=16, help="CUDA streams the programs are spread over")
    ap.add_argument("--no-graph", dest="graph", action="store_false",
                    help="launch every step from the host instead of replaying a captured CUDA graph")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--probe-costs", action="store_true",
                    help="print each library function's measured throughput cost in DFMA-equivalents and exit")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        return run_reference(args)
    if args.probe_costs:
        return probe_costs()

    import torch
    import paper_2607_03574_gb300 as nd

    rank, world, local = dist_env()
    args.host_group = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
        args.host_group = dist.new_group(backend="gloo")  # host-side gather of the lane slices
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    nd.load()
    pipe_peak, pipe_src = fp64_pipe_peak(torch.cuda.get_device_properties(dev).multi_processor_count)
    peaks = (pipe_peak, pipe_src, nd.measure_fp64_peak())

    progs, desc, B_total = population(args, args.config, world, rank, args.lanes)
    head = measure(nd, dev, progs, B_total, args.config, args.dtype, args, world, rank, peaks, True)
    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args, progs)

    configs = {}
    if not args.only and not args.lanes and not args.T:
        for cfg, dt in EXTRA:
            if (cfg, dt) == (args.config, args.dtype):
                continue
            p2, d2, bt2 = population(args, cfg, world, rank, 0)
            m = measure(nd, dev, p2, bt2, cfg, dt, args, world, rank, peaks, False)
            m["workload"] = f"{d2}, {dt} value+grad"
            if rank == 0 and not args.no_cpu_baseline:
                m["cpu_baseline"] = bounded_cpu_baseline(p2, dt == "f32")
            configs[f"{cfg}" if dt == "f64" else f"{cfg}_{dt}"] = m
        # small populations (64 lanes per program), where launches dominate: one call per
        # program on the streams against one batched call for all programs
        p2, d2, bt2 = population(args, 2, world, rank, SMALL_LANES)
        for key, bat in (("2_64lanes_streams", False), ("2_64lanes_batched", True)):
            m = measure(nd, dev, p2, bt2, 2, "f64", args, world, rank, peaks, False, batched=bat)
            m["workload"] = (f"{d2}, f64 value+grad, " +
                             ("ndvm_value_and_grad_multi: one call for every program" if bat else
                              f"one ndvm_value_and_grad call per program on {args.streams} streams"))
            configs[key] = m

    if rank == 0:
        cfg_key = {"workload": f"{desc}, {args.dtype} value+grad", "programs": len(progs),
                   "lanes_per_program": B_total, "lanes_per_rank": progs[0].B, "points": N_POINTS, "seed": SEED,
                   "l2": "flushed (256 MB write) before every timed step",
                   "parallelism": f"one population, lanes sliced across ranks (dp{world}); host gather on rank 0",
                   "streams": args.streams, "step_time": "median of the timed steps (max over ranks)"}
        line = {
            "metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": head["ms_per_step"], "ms_per_step_mean": head["ms_per_step_mean"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": args.dtype,
            "data": "synthetic", "config": cfg_key, "e2e": head["e2e"], "gpu_launches": head["gpu_launches"],
            "graph": head["graph"], "roofline": head["roofline"], "cpu_baseline": cpu, "clocks": head["clocks"],
            "wall_s_timed": head["wall_s_timed"], "trace_build_s": head["trace_build_s"],
            "step_ms": head["step_ms"],
        }
        if "gathered_on_rank0" in head:
            line["gathered_on_rank0"] = head["gathered_on_rank0"]
        if configs:
            line["configs"] = configs
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
