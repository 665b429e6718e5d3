"""Benchmark of the exact MPT solver (subset-splits evaluated per second).

One step = one exact solve of the whole hot path -- request-set scatter,
superset sums, the layered min-plus recurrence with argmins, the hierarchy
walk -- of one RAG-shaped instance with m = 28 requests (workload 4:
100k passages, 16 topical pools of 300, k = 20, Zipf(1.1) tail, seed 0),
through the C ABI.  Splits per solve = (3^m + 1)/2 - 2^m.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

N > 1 runs one process per GPU under torchrun; the path does not shard, so
every rank solves its own replica instance (seed = rank) and the whole-job
value is the sum of their splits over the slowest rank's time.

``--impl reference`` times the CPU oracle (the plain recurrence of Sec. 3.1)
on the host cores, on a bounded sample of the same workload.
"""

from __future__ import annotations

import argparse
import json
import math
import os
import platform
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "subset-splits evaluated/sec (≈3^m/2 per solve) and exact-MPT solve time at m=28"
WORKLOAD = 4
FULL_RUN_REQUESTS = 22  # context: the oracle's whole recurrence on the first 22 requests
# Each split is one 32-bit add and min, which the pair kernel issues as one
# instruction on the integer ALU pipe (ncu: its arithmetic runs on that pipe).
# The roofline peak is that instruction's rate measured on this GPU
# (mpt_alu_addmin_peak: every SM busy, nothing else in the loop).
OPS_PER_SPLIT = 1


def splits_per_solve(m: int) -> int:
    return (3 ** m + 1) // 2 - 2 ** m


def measured_peaks() -> dict:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except OSError:
        return {}


# ---------------------------------------------------------------------------
# distributed helpers (replicas; rank 0 prints)
# ---------------------------------------------------------------------------

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def init_dist(world: int, backend: str):
    import torch.distributed as dist

    if world > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend)
    return dist


def replica_seed(rank: int) -> int:
    """Instance seed of a replica: rank r solves workload 4 drawn with seed r."""
    return rank


def max_over_ranks(x: float, world: int, device=None) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist

    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


# ---------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines: list[str] = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
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

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# ---------------------------------------------------------------------------
# CPU oracle legs
# ---------------------------------------------------------------------------

_HOST_CORES = None


def host_cores() -> int:
    """OpenMP threads the oracle has on this host, read before any call
    that sets a smaller count (the setting persists in the process)."""
    global _HOST_CORES
    if _HOST_CORES is None:
        import oracle

        _HOST_CORES = oracle.max_threads()
    return _HOST_CORES


def oracle_sample(inst, m_sub: int, threads: int = 0):
    """The oracle's full recurrence on the first ``m_sub`` requests of the
    instance (all host cores, or ``threads`` of them)."""
    import oracle

    P = threads or host_cores()
    bits = np.ascontiguousarray(inst.bits[:m_sub])
    t0 = time.perf_counter()
    opt, F, wI, split = oracle.solve(inst.weights, bits, threads=P)
    dt = time.perf_counter() - t0
    return splits_per_solve(m_sub), dt, P


RUNS_PER_LAYER = 4
_TABLES: dict = {}


def stand_in_table(m: int) -> np.ndarray:
    """A 2^m int64 table of ones, kept for the next sample of the same size
    (the sampled work does not depend on the values, only on the table's size)."""
    if m not in _TABLES:
        _TABLES.clear()
        _TABLES[m] = np.ones(1 << m, dtype=np.int64)
    return _TABLES[m]


def next_same_size(S: int) -> int:
    """The next larger integer with the same number of set bits (Gosper)."""
    c = S & -S
    r = S + c
    return (((r ^ S) >> 2) // c) | r


def oracle_extrapolated(m: int, threads: int = 0, seed: int = 0, layer_splits: float = 4e8,
                        measure_cost: float = 3e9, wi_requests: int = 22, inst=None) -> dict:
    """The oracle's whole solve time for an m-request instance, extrapolated
    from samples of every layer of its recurrence (labelled as such).

    Layer k of the oracle's loop holds C(m, k) subsets of 2^(k-1) - 1 splits
    each (the table values only decide rare strict improvements, not the
    work), run in parallel over the subsets of the layer.  Each layer's
    sample -- runs of 8 consecutive k-subsets in the increasing order the
    oracle visits them, from seeded random starts, at least 4 per thread --
    goes through the oracle's own step (``oracle.dp_at``) on a table of the
    full 2^m size, and its measured splits/s prices the layer; a layer of at
    most 4 subsets per thread is run whole.  Layers whose sample would cost
    more than ``measure_cost`` splits are priced from the per-thread split
    time of the largest measured layer, in rounds of one subset per thread.
    The direct-intersection table w(I) (a single-threaded walk over all 2^m
    subsets) is timed on the first ``wi_requests`` requests and scaled by
    2^(m - wi_requests)."""
    import oracle

    P = threads or host_cores()
    table = stand_in_table(m)  # stands in for F and w(I)
    rng = np.random.default_rng(seed)
    total, measured, modelled, tau = 0.0, [], [], None
    for k in range(2, m + 1):
        per = (1 << (k - 1)) - 1
        count = math.comb(m, k)
        want = min(count, max(4 * P, math.ceil(layer_splits / per)), 4096)
        if want * per <= measure_cost or tau is None:
            if want == count:
                S = (1 << k) - 1
                sample = []
                while S < (1 << m):
                    sample.append(S)
                    S = next_same_size(S)
            else:
                sample = []
                run = max(8, want // RUNS_PER_LAYER)
                while len(sample) < want:
                    S = int(sum(1 << int(i) for i in rng.choice(m, size=k, replace=False)))
                    for _ in range(run):
                        if S >= (1 << m) or len(sample) >= want:
                            break
                        sample.append(S)
                        S = next_same_size(S)
            subsets = np.array(sample, dtype=np.uint64)
            t0 = time.perf_counter()
            oracle.dp_at(table, table, m, subsets, threads=P)
            dt = time.perf_counter() - t0
            layer = dt if len(sample) == count else count * dt / len(sample)
            tau = dt * min(P, len(sample)) / (len(sample) * per)
            measured.append(k)
        else:
            layer = math.ceil(count / P) * per * tau
            modelled.append(k)
        total += layer
    wi = None
    if inst is not None:
        sub = min(wi_requests, m)
        bits = np.ascontiguousarray(inst.bits[:sub])
        t0 = time.perf_counter()
        oracle.intersection_weights(inst.weights, bits)
        wi = (time.perf_counter() - t0) * 2.0 ** (m - sub)
        total += wi
    return {"m": m, "extrapolated_solve_s": total, "splits_per_s": splits_per_solve(m) / total, "threads": P,
            "layers_sampled": measured, "layers_priced_from_largest_sampled": modelled,
            "wI_walk_s": wi,
            "sample": (f"every layer k = 2..{m} of the oracle's recurrence sampled (>= 4 subsets per thread, "
                       f"runs of 8 consecutive k-subsets from seeded starts, ~{layer_splits:.0e} splits per "
                       "layer, small layers whole) through oracle.dp_at on a 2^m table; layer time = "
                       "C(m,k)(2^(k-1)-1) / sampled splits/s; w(I) walk timed on the first "
                       f"{min(wi_requests, m)} requests x 2^{m - min(wi_requests, m)}; EXTRAPOLATED, not a full run")}


def cpu_model() -> str:
    """The host CPU as the OS names it (model name, else the Arm part id)."""
    try:
        with open("/proc/cpuinfo") as f:
            info = f.read()
    except OSError:
        return platform.processor() or platform.machine()
    for key in ("model name", "Model", "CPU part"):
        for line in info.splitlines():
            if line.startswith(key):
                return f"{platform.machine()} {key}: {line.split(':', 1)[1].strip()}"
    return platform.machine()


def run_reference(args):
    world, rank, local = dist_env()
    if world > 1:
        init_dist(world, "gloo")
        if rank != 0:
            barrier(world)
            return
    from paper_2609_13692_gb300 import instances

    inst = instances.config(args.workload, seed=0)
    m = inst.m
    for w in range(args.warmup):
        oracle_extrapolated(m, seed=1000 + w)
    total_t, cores, last = 0.0, 1, None
    t_wall = 0.0
    for step in range(args.steps):
        t0 = time.perf_counter()
        last = oracle_extrapolated(m, seed=step, inst=inst if step == 0 else None)
        t_wall += time.perf_counter() - t0
        if step == 0:
            wi_s = last["wI_walk_s"]
        else:
            last["extrapolated_solve_s"] += wi_s
        total_t += last["extrapolated_solve_s"]
        cores = last["threads"]
    solve_s = total_t / args.steps
    rate = splits_per_solve(m) / solve_s
    full_m = min(FULL_RUN_REQUESTS, m)
    full_s, full_dt, _ = oracle_sample(inst, full_m)
    sample = (f"workload {args.workload} (m = {m}) per step: " + last["sample"] +
              f"; {1000 * t_wall / args.steps:.0f} ms of host time per step")
    line = {
        "impl": "reference", "metric": METRIC, "value": rate, "unit": "splits/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * solve_s,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
        "solve_time_s": solve_s, "solve_time_kind": "extrapolated from per-layer samples",
        "config": {"workload": instances.CONFIG_NAMES[args.workload], "m": m, "n": inst.n,
                   "splits_per_solve": splits_per_solve(m), "parallelism": "host cores"},
        "cpu_baseline": {"value": rate, "unit": "splits/s", "cores": cores, "kind": "oracle", "sample": sample,
                         "cpu": cpu_model(),
                         "full_run": {"value": full_s / full_dt, "sample": f"whole recurrence on the first "
                                      f"{full_m} requests ({full_s} splits, {full_dt:.1f} s)"}},
        "e2e": {"value": rate, "unit": "splits/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        barrier(world)


# ---------------------------------------------------------------------------
# GPU leg
# ---------------------------------------------------------------------------

def source_digest(rel: str) -> str:
    import hashlib

    with open(os.path.join(ROOT, rel), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def load_traffic_profile():
    """DRAM bytes per pair-kernel launch from a committed ncu summary, or None
    when the kernel source has changed since those counters were taken."""
    path = os.path.join(ROOT, "profiles", "k_dp_pairs_traffic.json")
    try:
        with open(path) as f:
            tr = json.load(f)
    except OSError:
        return None
    src = tr.get("source")
    if not src or tr.get("source_sha256_16") != source_digest(src):
        return None
    return tr


def measure_alu_peak(mpt, stream, device_index: int, tries: int = 3) -> dict:
    """The add-min peak of the integer ALU pipe measured on this GPU
    (mpt_alu_addmin_peak, best of ``tries``), with the SM clock sampled
    while it ran."""
    sampler = ClockSampler(device_index)
    sampler.start()
    rates = [mpt.mpt_alu_addmin_peak(1 << 43, stream) for _ in range(tries)]
    clocks = sampler.stop()
    return {"ops_per_s": max(rates), "runs": rates, "clocks": clocks}


def run_ours(args):
    import torch

    world, rank, local = dist_env()
    if world > 1:
        torch.cuda.set_device(local)
        init_dist(world, "nccl")
    else:
        torch.cuda.set_device(0)
    device = torch.device("cuda", torch.cuda.current_device())

    from paper_2609_13692_gb300 import build as B
    from paper_2609_13692_gb300 import instances, mpt

    if not B.LIB.exists():
        B.build()
    mpt.load()

    inst = instances.config(args.workload, seed=replica_seed(rank))
    if args.requests:
        # profiling a smaller case of the same workload: its first requests
        inst = instances.Instance(inst.weights, np.ascontiguousarray(inst.bits[:args.requests]),
                                  f"{inst.name}, first {args.requests} requests")
    m = inst.m
    splits = splits_per_solve(m)

    ctx = mpt.mpt_create(inst.weights, inst.bits)
    if args.dp_mode != "auto":
        mpt.mpt_set_dp_mode(ctx, args.dp_mode)
    if args.tables != "int64":
        mpt.mpt_set_tables(ctx, args.tables)
    mpt.mpt_set_profiling(ctx, True)
    ws = torch.empty(mpt.mpt_workspace_bytes(ctx), dtype=torch.uint8, device=device)
    stream = torch.cuda.current_stream()

    for _ in range(args.warmup):
        mpt.mpt_solve(ctx, ws, stream.cuda_stream)

    # ---- device-resident timed region: K solves of the resident instance ----
    clocks = ClockSampler(torch.cuda.current_device()) if rank == 0 else None
    prof_sum = {"ms_dp_pairs": 0.0, "splits_pairs": 0.0, "launches_pairs": 0, "launches_total": 0,
                "ms_dp_tiles": 0.0, "ms_zeta": 0.0, "ms_scatter": 0.0, "ms_walk": 0.0}
    opts = []
    barrier(world)
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        opts.append(mpt.mpt_solve(ctx, ws, stream.cuda_stream))
        p = mpt.mpt_get_profile(ctx)
        for k in prof_sum:
            prof_sum[k] += p[k]
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    clock_info = clocks.stop() if clocks else None
    local_ms = e0.elapsed_time(e1)
    max_ms = max_over_ranks(local_ms, world, device)
    value = world * splits * args.steps / (max_ms / 1000.0)
    dp_mode = {1: "blocked", 2: "general", 3: "wide"}.get(p["dp_mode"], "?")

    # ---- end to end through the C ABI with host buffers ----
    h2d = int(inst.weights.nbytes + inst.bits.nbytes)
    slots = int(sum(int(x).bit_count() for x in inst.bits.ravel()))
    d2h = 8 + 32 + 8 * (m + 1) + 8 * slots + 4 * m
    e2e_steps = max(1, args.steps)
    barrier(world)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        c2 = mpt.mpt_create(inst.weights, inst.bits)
        if args.dp_mode != "auto":
            mpt.mpt_set_dp_mode(c2, args.dp_mode)
        if args.tables != "int64":
            mpt.mpt_set_tables(c2, args.tables)
        mpt.mpt_solve(c2, ws, stream.cuda_stream)
        offs, chunks, dfs = mpt.mpt_layout(c2)
        mpt.mpt_destroy(c2)
    torch.cuda.synchronize()
    e2e_s = max_over_ranks(time.perf_counter() - t0, world, device)
    e2e_value = world * splits * e2e_steps / e2e_s

    if rank != 0:
        return

    # roofline of the dominant kernel (the pair kernel of the blocked DP)
    peaks = measured_peaks()
    if dp_mode in ("blocked", "wide") and prof_sum["ms_dp_pairs"] > 0:
        launches = max(1, prof_sum["launches_pairs"])
        avg_ms = prof_sum["ms_dp_pairs"] / launches
        ops_per_launch = OPS_PER_SPLIT * prof_sum["splits_pairs"] / launches
        achieved = ops_per_launch / (avg_ms / 1000.0) / 1e12
        tr = load_traffic_profile()
        # the pipe's add-min rate measured on this GPU, next to the nominal
        # SMs x 4 sub-partitions x 16 lanes per clock at the maximum SM clock
        alu = measure_alu_peak(mpt, stream.cuda_stream, torch.cuda.current_device())
        alu_peak = alu["ops_per_s"] / 1e12
        sms = torch.cuda.get_device_properties(device).multi_processor_count
        max_mhz = (clock_info or {}).get("sm_max_mhz") or 2070.0
        nominal = sms * 64 * max_mhz * 1e6 / 1e12
        run_mhz = (clock_info or {}).get("sm_mhz")
        probe_mhz = alu["clocks"].get("sm_mhz")
        wide = dp_mode == "wide"
        roofline = {"bound": "alu", "kernel": "k_dp_pairs_w" if wide else "k_dp_pairs", "achieved": achieved,
                    "peak": alu_peak, "unit": "Tops/s", "frac": achieved / alu_peak,
                    "traffic": None if wide or tr is None else tr.get("dram_bytes_per_launch"),
                    "traffic_source": None if wide or tr is None else
                    f"ncu capture summarised in profiles/k_dp_pairs_traffic.json ({tr.get('workload', '')}), "
                    "scaled to this workload's average launch; not measured by this run",
                    "ops_per_split": OPS_PER_SPLIT,
                    "peak_basis": "measured: mpt_alu_addmin_peak, independent add-min chains on every SM, "
                                  f"best of {len(alu['runs'])} ({', '.join(f'{r / 1e12:.2f}' for r in alu['runs'])} "
                                  f"Tops/s) at a median SM clock of {probe_mhz} MHz"
                                  + ("; 64-bit keys take several ALU instructions per split" if wide else ""),
                    "nominal_peak": nominal, "frac_of_nominal": achieved / nominal,
                    "nominal_basis": f"{sms} SMs x 64 integer-ALU-pipe lanes x {max_mhz / 1000:.3f} GHz",
                    "per_sm_clock": {"kernel_ops": achieved * 1e12 / (sms * run_mhz * 1e6) if run_mhz else None,
                                     "kernel_mhz": run_mhz,
                                     "peak_ops": alu["ops_per_s"] / (sms * probe_mhz * 1e6) if probe_mhz else None,
                                     "peak_mhz": probe_mhz, "nominal_ops": 64},
                    "share_of_step": prof_sum["ms_dp_pairs"] / (local_ms if local_ms > 0 else 1)}
    else:
        hbm = float(peaks.get("hbm_gbs", 6800.0))
        gbs = 16.0 * splits * args.steps / (local_ms / 1000.0) / 1e9
        roofline = {"bound": "hbm", "kernel": "k_dp_layer_*", "achieved": gbs, "peak": hbm, "unit": "GB/s",
                    "frac": gbs / hbm, "traffic": None, "bytes_per_split": 16}
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    # the naive recurrence reads 16 B per split at scattered subsets: against
    # the measured random-gather bandwidth of a table of this size
    gather_gbs = mpt.mpt_gather_bandwidth(min(m, 30), 1 << 28, stream.cuda_stream)
    gather_frac = (16.0 * value / world) / (gather_gbs * 1e9)

    # CPU baseline: the oracle, timed on this host on bounded samples of the
    # same workload (every layer of its recurrence), extrapolated to a whole
    # solve; beside it the m = 30 workload and one whole run at 22 requests
    cpu = None
    if not args.no_cpu_baseline and world == 1:
        t_cpu = time.perf_counter()
        ext = oracle_extrapolated(m, inst=inst)
        ext1 = oracle_extrapolated(m, threads=1, layer_splits=1e7, measure_cost=4e7)
        ext1["extrapolated_solve_s"] += ext["wI_walk_s"]
        ext1["splits_per_s"] = splits / ext1["extrapolated_solve_s"]
        cpu = {"value": ext["splits_per_s"], "unit": "splits/s", "cores": ext["threads"], "kind": "oracle",
               "sample": f"workload {args.workload} (m = {m}): " + ext["sample"],
               "extrapolated_solve_s": ext["extrapolated_solve_s"],
               "single_thread": {"value": ext1["splits_per_s"], "extrapolated_solve_s": ext1["extrapolated_solve_s"],
                                 "sample": "the same per-layer sampling with one thread (~1e7 splits per layer)"},
               "cpu": cpu_model()}
        if args.workload == WORKLOAD:
            inst30 = instances.config(5, seed=0)
            e30 = oracle_extrapolated(30, inst=inst30)
            e30_1 = oracle_extrapolated(30, threads=1, layer_splits=1e7, measure_cost=4e7)
            e30_1["extrapolated_solve_s"] += e30["wI_walk_s"]
            cpu["m30"] = {"workload": instances.CONFIG_NAMES[5], "extrapolated_solve_s": e30["extrapolated_solve_s"],
                          "splits_per_s": e30["splits_per_s"], "threads": e30["threads"],
                          "single_thread_extrapolated_solve_s": e30_1["extrapolated_solve_s"],
                          "sample": "the same per-layer sampling on the m = 30 workload"}
        s_sub, dt, _ = oracle_sample(inst, FULL_RUN_REQUESTS)
        sub = instances.Instance(inst.weights, np.ascontiguousarray(inst.bits[:FULL_RUN_REQUESTS]))
        e_sub = oracle_extrapolated(FULL_RUN_REQUESTS, inst=sub)
        cpu["full_run"] = {"value": s_sub / dt, "solve_s": dt,
                           "extrapolated_solve_s": e_sub["extrapolated_solve_s"],
                           "sample": f"whole oracle recurrence on the first {FULL_RUN_REQUESTS} of the {m} requests "
                                     f"({s_sub} splits, {dt:.1f} s), beside the per-layer extrapolation of the "
                                     "same run as a check of the method"}
        cpu["host_seconds"] = time.perf_counter() - t_cpu

    solve_s = max_ms / 1000.0 / args.steps
    line = {
        "metric": METRIC if m == 28 else METRIC.replace("m=28", f"m={m}"),
        "value": value,
        "unit": "splits/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": max_ms / args.steps,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": {"blocked": "u32", "wide": "u64"}.get(dp_mode, "int64"),
        "dtype_note": {"blocked": "exact: 32-bit packed integer keys, valid because the shared weight is below "
                                  "2^(32 - tile bits) (checked at mpt_create); int64 tables and OPT",
                       "wide": "exact: 64-bit packed integer keys (shared weight < 2^51); int64 tables and OPT"
                       }.get(dp_mode, "exact int64 arithmetic"),
        "data": "synthetic",
        "solve_time_s": solve_s,
        "config": {"workload": instances.CONFIG_NAMES[args.workload]
                   + (f" (first {args.requests} requests)" if args.requests else ""), "m": m, "n": inst.n,
                   "k": instances.CONFIGS[args.workload].get("k", m - 1), "seed": replica_seed(rank),
                   "splits_per_solve": splits, "dp_mode": dp_mode, "tables": args.tables,
                   "workspace_gib": round(ws.numel() / 2**30, 2),
                   "parallelism": "replicas" if world > 1 else "single GPU",
                   "l2": f"inputs larger than L2: the 2^{m}-entry tables span "
                         f"{(1 << m) * (16 if args.tables == 'lean' else 28) / 2**30:.2f} GiB (L2 129 MB), no flush",
                   "opt": opts[-1] if opts else None},
        "roofline": roofline,
        "gather_roofline_frac": gather_frac,
        "gather_roofline": {"measured_gbs": gather_gbs, "table": f"2^{min(m, 30)} int64 entries",
                            "bytes_per_split": 16, "vs_copy_peak_frac": (16.0 * value / world) / (hbm * 1e9)},
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_value, "unit": "splits/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "steps": e2e_steps, "path": "mpt_create(host arrays) + mpt_solve + mpt_layout(host arrays)"},
        "gpu_launches": int(prof_sum["launches_total"]),
        "stage_ms_per_step": {k: prof_sum[k] / args.steps for k in
                              ("ms_scatter", "ms_zeta", "ms_dp_pairs", "ms_dp_tiles", "ms_walk")},
        "clocks": clock_info,
    }
    print(json.dumps(line), flush=True)


def batch_groups(count: int, seed: int, n: int = 100_000, k: int = 8, m_lo: int = 8, m_hi: int = 13):
    """Request groups shaped like the paper's exact-solve groups (Sec. 7: at
    most 13 requests, k = 8 retrieved passages): each group draws its requests
    from one of 64 topical pools of 60 passages (80 %) or a uniform tail."""
    rng = np.random.default_rng(seed)
    mu = math.log(150.0) - 0.18
    weights = np.clip(np.rint(rng.lognormal(mu, 0.6, size=n)), 32, 512).astype(np.int64)
    pools = rng.choice(n, size=(64, 60), replace=False)
    groups = []
    for _ in range(count):
        m = int(rng.integers(m_lo, m_hi + 1))
        pool = pools[int(rng.integers(64))]
        reqs = []
        for _ in range(m):
            chosen = set()
            while len(chosen) < k:
                chosen.add(int(pool[int(rng.integers(60))]) if rng.random() < 0.8 else int(rng.integers(n)))
            reqs.append(sorted(chosen))
        groups.append(reqs)
    return weights, groups


def run_batch(args):
    """Batched small-instance solves (mpt_batch_*): instances and splits per second."""
    import torch

    from paper_2609_13692_gb300 import build as B
    from paper_2609_13692_gb300 import mpt

    torch.cuda.set_device(0)
    if not B.LIB.exists():
        B.build()
    m_lo, m_hi = (int(v) for v in args.batch_sizes.split("-"))
    weights, groups = batch_groups(args.batch_size, seed=0, m_lo=m_lo, m_hi=m_hi)
    ir, ro, ch = mpt.pack_batch(groups)
    ms = np.diff(ir)
    splits = int(sum((3 ** int(m) + 1) // 2 - 2 ** int(m) for m in ms))
    b = mpt.mpt_batch_create(weights, ir, ro, ch)
    ws = torch.empty(mpt.mpt_batch_workspace_bytes(b), dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        mpt.mpt_batch_solve(b, ws, stream.cuda_stream)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        mpt.mpt_batch_solve(b, ws, stream.cuda_stream)
    e1.record(stream)
    torch.cuda.synchronize()
    ms_step = e0.elapsed_time(e1) / args.steps
    line = {"mode": "batch", "metric": f"exact solves of request groups (m = {m_lo}..{m_hi}, k = 8) per second",
            "value": len(groups) / (ms_step / 1000.0), "unit": "instances/s", "splits_per_s": splits / (ms_step / 1000.0),
            "ms_per_step": ms_step, "steps": args.steps, "warmup": args.warmup, "batch": len(groups),
            "splits_per_step": splits, "note": "timed region includes the per-step input upload and result download"}
    if not args.no_cpu_baseline:
        import oracle

        sample = groups[:200]
        t0 = time.perf_counter()
        for reqs in sample:
            oracle.solve(weights, _pack(reqs, weights.shape[0]))
        dt = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": len(sample) / dt, "unit": "instances/s", "cores": oracle.max_threads(),
                                "kind": "oracle", "sample": f"first {len(sample)} groups, one oracle solve each"}
    print(json.dumps(line), flush=True)


def run_greedy(args):
    """Agglomerative hierarchy + spanning-tree bound on a trace-sized request
    set (m requests of k = 8 passages, the size of the paper's NFCorpus trace)."""
    import torch

    from paper_2609_13692_gb300 import build as B
    from paper_2609_13692_gb300 import mpt

    torch.cuda.set_device(0)
    if not B.LIB.exists():
        B.build()
    rng = np.random.default_rng(0)
    m, n = args.greedy_m, max(1200, int(args.greedy_m * 1.2))
    weights = np.clip(np.rint(rng.lognormal(math.log(150.0) - 0.18, 0.6, size=n)), 32, 512).astype(np.int64)
    pools = [rng.choice(n, size=60, replace=False) for _ in range(max(8, m // 15))]
    reqs = []
    for _ in range(m):
        pool = pools[int(rng.integers(len(pools)))]
        chosen = set()
        while len(chosen) < 8:
            chosen.add(int(pool[int(rng.integers(60))]) if rng.random() < 0.85 else int(rng.integers(n)))
        reqs.append(sorted(chosen))
    for _ in range(args.warmup):
        mpt.mpt_greedy(weights, reqs)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        g = mpt.mpt_greedy(weights, reqs)
    dt = (time.perf_counter() - t0) / args.steps
    total = int(sum(int(weights[x]) for r in reqs for x in r))
    line = {"mode": "greedy", "metric": "agglomerative hierarchy + layout + spanning-tree bound, wall time per call",
            "value": dt, "unit": "s", "higher_is_better": False, "m": m, "k": 8, "steps": args.steps,
            "no_sharing_cost": total, "greedy_cost": g.cost, "lower_bound": g.lower_bound,
            "greedy_fraction_of_no_sharing": g.cost / total, "bound_fraction_of_no_sharing": g.lower_bound / total,
            "note": "host arrays in and out, device buffers allocated inside the call",
            "gap_to_exact": greedy_gap_small_groups(mpt)}
    print(json.dumps(line), flush=True)


def greedy_gap_small_groups(mpt):
    """Greedy cost over the exact optimum (both on the GPU) for 72 synthetic
    RAG groups of m = 10..15 requests (12 seeds per size, topical pools with a
    Zipf tail), the shape of the paper's synthetic comparison; not timed."""
    from paper_2609_13692_gb300 import instances as I

    gaps = []
    for m in range(10, 16):
        for seed in range(12):
            inst = I.rag_pools(m, 2000, 4, 30, 8, 1.1, seed=1000 * m + seed)
            reqs = [[x for x in range(inst.weights.shape[0]) if (int(inst.bits[i, x >> 6]) >> (x & 63)) & 1]
                    for i in range(m)]
            exact = mpt.solve(inst.weights, inst.bits).opt
            greedy = mpt.mpt_greedy(inst.weights, reqs).cost
            gaps.append((greedy - exact) / exact)
    return {"instances": len(gaps), "m": "10-15", "k": 8, "avg": float(np.mean(gaps)), "worst": float(np.max(gaps)),
            "exact_hits": int(sum(1 for x in gaps if x == 0)),
            "paper_context": "2.6% average, 11% worst over its 72 synthetic instances (m = 10-15, Zipf pools)"}


def run_cache(args):
    """Wall time of the Thm 7 serving order (mpt_serve_order) and of the
    LRU radix-cache simulator (mpt_cache_costs, 10 capacities per call) on the
    greedy layout of an NFCorpus-shaped request stream."""
    import torch

    from paper_2609_13692_gb300 import build as B
    from paper_2609_13692_gb300 import instances
    from paper_2609_13692_gb300 import mpt

    torch.cuda.set_device(0)
    if not B.LIB.exists():
        B.build()
    if args.cache_m:
        # a longer stream of the same shape: pools scaled with the request count
        c = dict(instances.STREAMS["nfcorpus-shaped"])
        scale = args.cache_m / c["m"]
        weights, ranked = instances.rag_ranked(args.cache_m, int(c["n"] * scale), max(1, int(c["pools"] * scale)),
                                               c["pool_size"], c["k"], c["tail_s"], seed=0, w_mean=c["w_mean"],
                                               wmin=c["wmin"], wmax=c["wmax"])
    else:
        weights, ranked = instances.stream("nfcorpus-shaped", seed=0)
    n, m = len(weights), len(ranked)
    one = float(np.mean([sum(int(weights[x]) for x in q) for q in ranked]))
    caps = [int(round(f * one)) for f in (0.25, 0.5, 0.75, 0.9, 1, 4, 16, 64, 256, 1024)]
    layout = mpt.mpt_greedy(weights, ranked).perms if m <= 16384 else [list(r) for r in ranked]
    csr = mpt.to_csr(layout)
    arr = np.arange(m, dtype=np.int32)
    for _ in range(args.warmup):
        mpt.mpt_cache_costs(weights, csr, caps, arr)
        mpt.mpt_serve_order(n, csr)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        mpt.mpt_cache_costs(weights, csr, caps, arr)
    dt = (time.perf_counter() - t0) / args.steps
    t0 = time.perf_counter()
    for _ in range(args.steps):
        mpt.mpt_serve_order(n, csr)
    dt_order = (time.perf_counter() - t0) / args.steps
    line = {"mode": "cache", "metric": "LRU radix-cache simulator, 10 capacities per call, wall time",
            "value": dt, "unit": "s", "higher_is_better": False, "steps": args.steps, "warmup": args.warmup,
            "serve_order_s": dt_order,
            "workload": f"nfcorpus-shaped stream: m = {m} requests, k = 8, greedy layout"
                        + (" (scaled)" if args.cache_m else ""),
            "accesses": int(sum(len(q) for q in layout)),
            "note": "host arrays in and out, device buffers allocated inside each call"}
    print(json.dumps(line), flush=True)


def _pack(reqs, n):
    from paper_2609_13692_gb300 import instances

    return instances.pack_requests(reqs, n)


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--dp-mode", choices=["auto", "blocked", "general", "wide"], default="auto")
    ap.add_argument("--workload", type=int, default=WORKLOAD, choices=[1, 2, 3, 4, 5, 6, 7],
                    help="benchmark workload (default 4: m = 28); others are for profiling")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--requests", type=int, default=0,
                    help="solve only the workload's first M requests (smaller cases for ncu captures)")
    ap.add_argument("--tables", choices=["int64", "lean"], default="int64",
                    help="table layout of the exact solve (lean: one int32 table, F over w(I))")
    ap.add_argument("--mode", choices=["solve", "batch", "greedy", "cache"], default="solve",
                    help="solve: the m = 28 exact solve (default); batch: many small request groups; "
                         "greedy: agglomerative hierarchy on a trace-sized request set; "
                         "cache: serving order and radix-cache simulator timings on a request stream")
    ap.add_argument("--batch-size", type=int, default=20000)
    ap.add_argument("--batch-sizes", default="8-13", help="request-count range of the batched groups, e.g. 14-15")
    ap.add_argument("--greedy-m", type=int, default=3000)
    ap.add_argument("--cache-m", type=int, default=0,
                    help="cache mode: requests in a scaled stream (default: the 2,921-request stream)")
    args = ap.parse_args()
    if args.mode == "batch":
        run_batch(args)
        return
    if args.mode == "greedy":
        run_greedy(args)
        return
    if args.mode == "cache":
        run_cache(args)
        return
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
