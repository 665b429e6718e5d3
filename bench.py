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
ORACLE_SAMPLE_REQUESTS = 22  # reference arm: full oracle recurrence on the first 22 requests per step
CPU_BASELINE_REQUESTS = 23  # cpu_baseline: one run on the first 23 requests (10-30 s of CPU work)
# Each split is one 32-bit add and min, which the pair kernel issues as one
# instruction on the integer ALU pipe (ncu: its arithmetic runs on that pipe).
# The pipe peak (SMs x 4 sub-partitions x 16 lanes per clock at the maximum SM
# clock) is computed from the device where the roofline is reported.
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

def oracle_sample(inst, m_sub: int, threads: int = 0):
    """The oracle's full recurrence on the first ``m_sub`` requests of the
    instance (all host cores, or ``threads`` of them)."""
    import oracle

    bits = np.ascontiguousarray(inst.bits[:m_sub])
    t0 = time.perf_counter()
    opt, F, wI, split = oracle.solve(inst.weights, bits, threads=threads)
    dt = time.perf_counter() - t0
    return splits_per_solve(m_sub), dt, (threads or oracle.max_threads())


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

    inst = instances.config(WORKLOAD, seed=0)
    m_sub = args.ref_requests
    for _ in range(args.warmup):
        oracle_sample(inst, m_sub)
    total_splits, total_t, cores = 0, 0.0, 1
    for _ in range(args.steps):
        s, dt, cores = oracle_sample(inst, m_sub)
        total_splits += s
        total_t += dt
    rate = total_splits / total_t
    sample = (f"oracle recurrence (C, OpenMP over the subsets of each size) on the first {m_sub} of the "
              f"{inst.m} requests of workload {WORKLOAD}: {splits_per_solve(m_sub)} splits per step")
    line = {
        "impl": "reference", "metric": METRIC, "value": rate, "unit": "splits/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * total_t / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
        "config": {"workload": instances.CONFIG_NAMES[WORKLOAD], "m": inst.m, "n": inst.n, "sample_requests": m_sub,
                   "parallelism": "host cores"},
        "cpu_baseline": {"value": rate, "unit": "splits/s", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": rate, "unit": "splits/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        barrier(world)


# ---------------------------------------------------------------------------
# GPU leg
# ---------------------------------------------------------------------------

def load_traffic_profile():
    """DRAM bytes per pair-kernel launch from a committed ncu summary (or None)."""
    path = os.path.join(ROOT, "profiles", "k_dp_pairs_traffic.json")
    try:
        with open(path) as f:
            return json.load(f)
    except OSError:
        return None


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
    e2e_steps = max(1, min(args.steps, 3))
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
        # integer ALU pipe: SMs (from the device) x 4 sub-partitions x 16 lanes
        # per clock at the maximum SM clock nvidia-smi reports (2,070 MHz if
        # it reports none)
        sms = torch.cuda.get_device_properties(device).multi_processor_count
        max_mhz = (clock_info or {}).get("sm_max_mhz") or 2070.0
        alu_peak = sms * 64 * max_mhz * 1e6 / 1e12
        wide = dp_mode == "wide"
        roofline = {"bound": "alu", "kernel": "k_dp_pairs_w" if wide else "k_dp_pairs", "achieved": achieved,
                    "peak": alu_peak, "unit": "Tops/s", "frac": achieved / alu_peak,
                    "traffic": None if wide else (tr or {}).get("dram_bytes_per_launch"),
                    "ops_per_split": OPS_PER_SPLIT,
                    "peak_basis": f"{sms} SMs x 64 integer-ALU-pipe lanes x {max_mhz / 1000:.3f} GHz "
                                  "(one add-min per split" + ("; 64-bit keys take several ALU instructions "
                                                              "per split" if wide else "") + ")",
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

    # CPU baseline: the oracle, timed on this host, bounded sample
    cpu = None
    if not args.no_cpu_baseline and world == 1:
        s_sub, dt, cores = oracle_sample(inst, CPU_BASELINE_REQUESTS)
        s1, dt1, _ = oracle_sample(inst, 19, threads=1)
        cpu = {"value": s_sub / dt, "unit": "splits/s", "cores": cores, "kind": "oracle",
               "sample": f"full oracle recurrence on the first {CPU_BASELINE_REQUESTS} of the {m} requests "
                         f"({s_sub} splits, {dt:.1f} s)",
               "single_thread": {"value": s1 / dt1, "sample": f"first 19 requests ({s1} splits, {dt1:.1f} s)"},
               "cpu": cpu_model()}

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
        "data": "synthetic",
        "solve_time_s": solve_s,
        "config": {"workload": instances.CONFIG_NAMES[args.workload], "m": m, "n": inst.n,
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
    weights, groups = batch_groups(args.batch_size, seed=0)
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
    line = {"mode": "batch", "metric": "exact solves of request groups (m = 8..13, k = 8) per second",
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
    """Finite-cache study (Sec. 8) on the NFCorpus-shaped stream: prefill cost
    at many capacities per call, in arrival order, inside reorder windows and
    in Thm 7's order, for the production (relevance-order), greedy and pinned
    layouts."""
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
    mult = [0.25, 0.5, 0.75, 0.9, 1, 4, 16, 64, 256, 1024]
    caps = [int(round(f * one)) for f in mult]
    layouts = {"production": [list(r) for r in ranked]}
    if m <= 16384:  # the greedy hierarchy's limit
        layouts["greedy"] = mpt.mpt_greedy(weights, ranked).perms
        for t in (1, 2, 3):
            layouts[f"pin_top{t}"] = mpt.mpt_layout_pinned(weights, ranked, t, "greedy").strings
    total = int(sum(int(weights[x]) for q in ranked for x in q))
    arrival = list(range(m))
    g = layouts.get("greedy", layouts["production"])
    # timed: the C ABI calls on a CSR built once (host arrays in and out)
    g_csr = mpt.to_csr(g)
    arr = np.arange(m, dtype=np.int32)
    for _ in range(args.warmup):
        mpt.mpt_cache_costs(weights, g_csr, caps, arr)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        mpt.mpt_cache_costs(weights, g_csr, caps, arr)
    dt = (time.perf_counter() - t0) / args.steps
    t0 = time.perf_counter()
    for _ in range(args.steps):
        thm7 = mpt.mpt_serve_order(n, g_csr)
    dt_order = (time.perf_counter() - t0) / args.steps

    table = {}
    for name, strings in layouts.items():
        unb = None
        row = {}
        for label, order in (("arrival", arrival), ("thm7", mpt.mpt_serve_order(n, strings).tolist())):
            costs, unb = mpt.mpt_cache_costs(weights, strings, caps, order)
            row[label] = {f"{f}x": int(c) for f, c in zip(mult, costs)}
        row["unbounded"] = unb
        row["saving_vs_no_sharing"] = 1 - unb / total
        table[name] = row
    windows = {}
    for W in sorted({1, 128, 512, 2048, m}):
        order = mpt.mpt_serve_order(n, g, arrival, W).tolist()
        costs, unb = mpt.mpt_cache_costs(weights, g, caps[4:], order)
        windows["all" if W == m else str(W)] = {f"{f}x": round(c / unb - 1, 4) for f, c in zip(mult[4:], costs)}
    line = {"mode": "cache", "metric": "finite radix cache, prefill cost at 10 capacities per call",
            "value": dt, "unit": "s", "higher_is_better": False, "steps": args.steps,
            "timed_layout": "greedy" if "greedy" in layouts else "production",
            "workload": f"nfcorpus-shaped stream: m = {m} requests, k = 8, one request = {one:.0f} tokens"
                        + (" (scaled)" if args.cache_m else ""),
            "accesses": int(sum(len(q) for q in g)), "serve_order_s": dt_order,
            "capacities_in_requests": mult, "no_sharing_cost": total, "layouts": table,
            "window_excess_over_unbounded_greedy": windows,
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
    ap.add_argument("--ref-requests", type=int, default=ORACLE_SAMPLE_REQUESTS,
                    help="reference arm: requests of the workload in each step's oracle sample")
    ap.add_argument("--tables", choices=["int64", "lean"], default="int64",
                    help="table layout of the exact solve (lean: one int32 table, F over w(I))")
    ap.add_argument("--mode", choices=["solve", "batch", "greedy", "cache"], default="solve",
                    help="solve: the m = 28 exact solve (default); batch: many small request groups; "
                         "greedy: agglomerative hierarchy on a trace-sized request set; "
                         "cache: finite-cache study on a request stream")
    ap.add_argument("--batch-size", type=int, default=20000)
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
