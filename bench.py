#!/usr/bin/env python3
"""SkewAdam optimizer-step benchmark on GB300.

A step is one SkewAdam update (all tiers: factored second moments, backbone
momentum, exact router / vector second moments, update-RMS clipping, decoupled
weight decay, dithered bf16 write-back) over a synthetic parameter set shaped
like the paper's 6.78B-parameter MoE (App. B shapes: 6,784,327,680 bf16
parameters in 408 tensors). Weights ~ N(0, 0.02^2), gradients ~ N(0, 1e-3^2),
resident in HBM; 27.1 GB of weights + gradients per step (App. B shapes) is far larger than the
129 MiB L2, so no flush is needed between steps.

Reported (one JSON line, rank 0):
  value       -- parameters updated per second, whole job (all ranks);
  ms_per_step -- device time per step (CUDA events, max over ranks);
  hbm         -- algorithmic minimum bytes per step / step time, and its share
                 of the 8 TB/s nominal and of the measured copy bandwidth;
  roofline    -- the dominant kernel's algorithmic bytes / its event-timed
                 duration against the measured HBM copy peak, and its DRAM traffic
                 (the committed one-launch ncu record of the small workload, scaled
                 by algorithmic bytes; null once the kernel source has changed);
  kernels_ms  -- each launch's mean event-timed duration;
  step_spans  -- median / mean / min / max of the per-step times;
  e2e         -- the same metric through the C ABI with the gradients copied
                 in from pinned host memory and the weights read back each step
                 (the step run as --e2e-groups handles over runs of consecutive
                 tensors, so one group's copies overlap the others' steps), beside
                 the host link's own rates just before and after it;
  cpu_baseline-- one step of the CPU oracle over the whole workload (a sample only when it
                 would not fit the time or host-memory budget), its tensors spread over
                 the host's cores;
  clocks      -- SM clocks and throttle reasons sampled during the timed steps.
Multi-GPU (torchrun): every rank updates its own full parameter set (the step
has no cross-tensor coupling, so it shards by tensor with no collective);
scaling is weak.

--impl reference times the CPU oracle (the reference arm of this benchmark) on
the host cores instead: each step the whole workload when --steps + --warmup of
them fit --ref-seconds, else a sample of it; ms_per_step is the time of what ran.
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def parse():
    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=100)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="appb", help="shape set (appb = the paper's 6.78B App. B shapes)")
    p.add_argument("--seed", type=int, default=20260207)
    p.add_argument("--e2e-steps", type=int, default=8)
    p.add_argument("--e2e-groups", type=int, default=8, help="tensor groups of the end-to-end leg's pipeline")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-threads", type=int, default=0,
                   help="host threads of the CPU oracle (cpu_baseline and --impl reference); 0: one per core")
    p.add_argument("--cpu-seconds", type=float, default=30.0,
                   help="oracle time budget of the CPU baseline (a full step when it fits, else a sample)")
    p.add_argument("--ref-seconds", type=float, default=300.0, help="target total time of --impl reference")
    p.add_argument("--grad-scale", type=float, default=None,
                   help="step on gamma * G with gamma a device scalar (the trainer's global-norm clip inside the step)")
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(path))
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# ---------------------------------------------------------------------------
# nvidia-smi clock sampling during the timed region
# ---------------------------------------------------------------------------
CLOCK_Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
           "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
           "clocks_event_reasons.sw_power_cap")


def clocks_start(dev_index):
    f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
    try:
        p = subprocess.Popen(["nvidia-smi", f"--query-gpu={CLOCK_Q}", "--format=csv,noheader,nounits", "-lms", "100",
                              "-i", str(dev_index)], stdout=f, stderr=subprocess.DEVNULL)
    except Exception:
        p = None
    return p, f


def clocks_stop(handle):
    p, f = handle
    if p is None:
        return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
    p.terminate()
    try:
        p.wait(timeout=5)
    except Exception:
        p.kill()
    f.seek(0)
    sm, smax, reasons, pw = [], [], set(), []
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    for line in f.read().splitlines():
        c = [x.strip() for x in line.split(",")]
        if len(c) < 9:
            continue
        try:
            sm.append(float(c[1]))
            smax.append(float(c[2]))
            pw.append(float(c[3]))
        except ValueError:
            continue
        for n, v in zip(names, c[5:9]):
            if v.lower().startswith("active"):
                reasons.add(n)
    os.unlink(f.name)
    return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
            "reasons": sorted(reasons), "samples": len(sm), "power_w_max": max(pw) if pw else None}


# ---------------------------------------------------------------------------
# byte accounting
# ---------------------------------------------------------------------------
def policy_name(wl):
    from paper_2607_19058_gb300 import workloads as WL
    return {WL.POLICY_TIERED: "tiered", WL.POLICY_EXPERT_MOMENTUM: "expert_momentum",
            WL.POLICY_FACTORED_ROUTER: "factored_router", WL.POLICY_UNIFORM: "uniform",
            WL.POLICY_ADAFACTOR: "adafactor"}[wl.hp.policy]


def byte_model(opt, n_tensors):
    """Algorithmic minimum bytes of one step and of each kernel's own traffic."""
    N = N_mom = N_full = N_fact = N_nomom = N_row = N_rowm = 0
    rc = rc_row = 0
    for k in range(n_tensors):
        i = opt.info(k)
        E = max(1, i.stack)  # a stack of E matrices: rows / cols are one matrix's
        N += i.numel
        if i.momentum:
            N_mom += i.numel
        else:
            N_nomom += i.numel
        if i.kind == 0:
            N_full += i.numel
        elif i.rowpath:
            N_row += i.numel
            N_rowm += i.numel if i.momentum else 0
            rc_row += E * (i.rows + i.cols)
        else:
            N_fact += i.numel
            rc += E * (i.rows + i.cols)
    step_min = 6 * N + 8 * N_mom + 8 * N_full + 8 * (rc + rc_row)
    N_rest = N - N_row  # tensors of the strip / flat tiles
    kernels = {
        "k_sumsq": 2 * N_fact,                                   # read G of strip-path factored matrices
        "k_rowsq": 2 * N_row + 8 * N_rowm + 8 * rc_row,          # read G (and M r/w) of row-path matrices; R r/w
        "k_finalize": 8 * (rc + rc_row),                         # R, C read + write
        "k_rms": 2 * N_rest + 8 * (N_mom - N_rowm) + 8 * N_full,  # read G; M, v read + write
        "k_fallback": 0,                                          # runs only when a clamp may bind
        "k_apply": 4 * N_rest + 2 * (N_nomom - (N_row - N_rowm)) + 4 * (N_mom - N_rowm) + 4 * N_full,
        "k_apply_rows": 6 * N_row - 2 * N_rowm + 4 * N_rowm,     # W r/w and G (or the new M) read
    }
    return dict(N=N, N_mom=N_mom, N_full=N_full, rc=rc, step_min=step_min, kernels=kernels)


def recorded_traffic(kernel, alg_bytes, root=None):
    """DRAM bytes per launch of `kernel` from the committed ncu record, which is taken on
    the 558M-parameter `small` workload (a few GB on the device; profiles/dram_traffic_small.md,
    `traffic:` lines) and scaled to this launch by its algorithmic bytes (the kernel's
    traffic grows with the units it processes). None when there is no record or the kernel
    source has changed since the counters were taken (its SHA-256 differs)."""
    root = root or os.path.dirname(os.path.abspath(__file__))
    src = os.path.join(root, "paper_2607_19058_gb300", "csrc", "skew_kernels.cu")
    summ = os.path.join(root, "profiles", "dram_traffic_small.md")
    try:
        with open(src, "rb") as f:
            sha = hashlib.sha256(f.read()).hexdigest()
        lines = open(summ).read().splitlines()
    except OSError:
        return None
    for ln in lines:
        if not ln.startswith("traffic:"):
            continue
        kv = dict(x.split("=", 1) for x in ln[len("traffic:"):].split())
        if kv.get("kernel") == kernel and kv.get("source_sha256") == sha and int(kv.get("alg_bytes", 0)) > 0:
            return int(round(int(kv["per_launch"]) * alg_bytes / int(kv["alg_bytes"])))
    return None


# ---------------------------------------------------------------------------
# CPU oracle timing (reported baseline / reference arm)
# ---------------------------------------------------------------------------
def oracle_sample_specs(wl, target_params):
    """A sample of the workload with its tier mix: experts + backbone matrices + vectors + router."""
    specs = wl.specs
    ex = [k for k, s in enumerate(specs) if s.tier == 1]
    bb2 = [k for k, s in enumerate(specs) if s.tier == 0 and len(s.shape) == 2 and s.numel <= 20_000_000]
    vec = [k for k, s in enumerate(specs) if len(s.shape) == 1][:2]
    rt = [k for k, s in enumerate(specs) if s.tier == 2]
    chosen, tot = list(rt) + vec, sum(specs[k].numel for k in rt + vec)
    bi = ei = 0
    while tot < target_params and (bi < len(bb2) or ei < len(ex)):
        # keep roughly the paper's 5 % backbone / 95 % expert split
        nbb = sum(specs[k].numel for k in chosen if specs[k].tier == 0)
        if bi < len(bb2) and nbb < 0.05 * tot:
            k = bb2[bi]
            bi += 1
        elif ei < len(ex):
            k = ex[ei]
            ei += 1
        else:
            k = bb2[bi]
            bi += 1
        chosen.append(k)
        tot += specs[k].numel
    return chosen, tot


def mem_available():
    """MemAvailable of this host in bytes (None where /proc/meminfo is missing)."""
    try:
        for ln in open("/proc/meminfo"):
            if ln.startswith("MemAvailable:"):
                return int(ln.split()[1]) * 1024
    except OSError:
        pass
    return None


def gpu_numa(dev_index):
    """The NUMA node of GPU `dev_index` (sysfs, from its PCI address) and that node's CPUs;
    read-only queries. None values where the host does not say."""
    try:
        out = subprocess.run(["nvidia-smi", "--query-gpu=pci.bus_id", "--format=csv,noheader", "-i", str(dev_index)],
                             capture_output=True, text=True, timeout=30).stdout.strip()
        bus = out.lower()
        if bus.count(":") == 2 and len(bus.split(":")[0]) > 4:  # 00000009:01:00.0 -> 0009:01:00.0
            bus = bus[-12:]
        node = int(open(f"/sys/bus/pci/devices/{bus}/numa_node").read().strip())
        cpus = None
        if node >= 0:
            cpus = set()
            for part in open(f"/sys/devices/system/node/node{node}/cpulist").read().strip().split(","):
                lo, _, hi = part.partition("-")
                cpus.update(range(int(lo), int(hi or lo) + 1))
        return {"gpu_pci": bus, "gpu_numa_node": node, "node_cpus": sorted(cpus) if cpus else None}
    except Exception:
        return {"gpu_pci": None, "gpu_numa_node": None, "node_cpus": None}


def pages_by_node(ptr):
    """NUMA nodes holding the pages of the mapping that contains host address `ptr`
    (/proc/self/numa_maps), as {node: pages}; None where unavailable."""
    try:
        for ln in open("/proc/self/numa_maps"):
            f = ln.split()
            start = int(f[0], 16)
            # numa_maps gives only starts: take the last mapping starting at or below ptr
            if start <= ptr:
                best = f
            else:
                break
        return {int(x[1:x.index("=")]): int(x.split("=")[1]) for x in best if x.startswith("N") and "=" in x}
    except Exception:
        return None


def host_info():
    """The host the CPU oracle runs on: its logical CPU count and CPU model."""
    import platform
    model = None
    try:
        for ln in open("/proc/cpuinfo"):
            key = ln.split(":")[0].strip().lower()
            if key in ("model name", "cpu model", "hardware"):
                model = ln.split(":", 1)[1].strip()
                break
    except OSError:
        pass
    return {"nproc": os.cpu_count(), "cpu": model or platform.machine()}


_ORACLE_THREADS = None


def oracle_threads():
    """Host threads for the CPU oracle: the tensors of a step are independent, and the oracle
    is plain C called through ctypes (which releases the GIL), so a thread per core runs them
    side by side (--cpu-threads sets another count, e.g. 1 for a single-core baseline)."""
    return _ORACLE_THREADS or max(1, os.cpu_count() or 1)


def time_oracle(wl, tids, inputs, step, lr, seed, threads=1, states=None):
    """Wall time of one oracle step over tensors `tids` (inputs[k] = (w bits, g bits); w is
    updated in place), the tensors spread over `threads` host threads, largest first."""
    import concurrent.futures as cf
    import oracle as O
    from paper_2607_19058_gb300 import workloads as WL
    hpd = wl.hp
    ohp = O.hparams(hpd.beta1, hpd.beta2, hpd.eps, hpd.clip_d, hpd.weight_decay,
                    annealed=hpd.policy == WL.POLICY_ADAFACTOR)
    if states is None:
        states = {}
    for k in tids:
        if k not in states:
            states[k] = O.TensorState(wl.specs[k].shape, wl.specs[k].tier, hpd.policy, wl.specs[k].no_decay)
    O.lib()  # loaded before the threads start
    order = sorted(tids, key=lambda k: -wl.specs[k].numel)

    def one(k):
        w, g = inputs[k]
        O.tensor_step(w, g, states[k], k, ohp, step, lr, seed)

    t0 = time.perf_counter()
    if threads <= 1:
        for k in order:
            one(k)
    else:
        with cf.ThreadPoolExecutor(threads) as ex:
            list(ex.map(one, order))
    return time.perf_counter() - t0


def cpu_inputs(wl, tids, step=1, src=None, threads=1):
    """bf16 bit patterns (host numpy) of the weights and step-`step` gradients of `tids`:
    copied from the device tensors `src`, or drawn on the host."""
    import concurrent.futures as cf
    from paper_2607_19058_gb300 import workloads as WL

    def one(k):
        if src is not None:
            w, g = src[k]
            return k, (WL.bf16_bits(w).copy(), WL.bf16_bits(g).copy())
        return k, (WL.bf16_bits(WL.init_weight(wl, k, "cpu")).copy(), WL.bf16_bits(WL.grad(wl, k, step, "cpu")).copy())

    with cf.ThreadPoolExecutor(max(1, threads)) as ex:
        return dict(ex.map(one, tids))


def oracle_host_bytes(wl, tids):
    """Host memory an oracle step over `tids` holds: bf16 weights and gradients, the fp32
    state (its closed form) and the fp64 update of the tensors running at once (at most the
    largest ones)."""
    import oracle as O
    n = sum(wl.specs[k].numel for k in tids)
    big = sorted((wl.specs[k].numel for k in tids), reverse=True)[:oracle_threads()]
    state = O.state_bytes([(wl.specs[k].shape, wl.specs[k].tier) for k in tids], wl.hp.policy)
    return 4 * n + state + 8 * sum(big)


def calibrate_oracle_rate(wl):
    """Params/s of the oracle on a small expert-shaped tensor (to size the samples)."""
    import numpy as np
    import oracle as O
    O.build()
    n, m = 1024, 1024
    rng = np.random.default_rng(0)
    w = rng.integers(0, 2**16, n * m, dtype=np.uint16) & 0x3FFF
    g = rng.integers(0, 2**16, n * m, dtype=np.uint16) & 0x3AFF
    st = O.TensorState((n, m), O.TIER_EXPERT)
    ohp = O.hparams(0.9, 0.999, 1e-30, 1.0, 0.1)
    t0 = time.perf_counter()
    O.tensor_step(w, g, st, 0, ohp, 1, 1e-3, 1)
    return n * m / (time.perf_counter() - t0)


def oracle_plan(wl, budget_s, nsteps):
    """Tensors of each oracle step and how they were chosen: the whole workload when
    `nsteps` steps of it fit `budget_s` seconds on the host's threads and its inputs fit in
    host memory, else a sample with the tier mix kept, sized to the budget."""
    rate = calibrate_oracle_rate(wl) * oracle_threads() * 0.8
    avail = mem_available()
    full = list(range(len(wl.specs)))
    if wl.numel / rate * nsteps <= budget_s and (avail is None or oracle_host_bytes(wl, full) < 0.7 * avail):
        return full, wl.numel, "the whole workload"
    tids, tot = oracle_sample_specs(wl, max(1e6, rate * budget_s / max(1, nsteps)))
    return tids, tot, f"{len(tids)} of the {len(wl.specs)} tensors ({tot} of {wl.numel} params, tier mix kept)"


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2607_19058_gb300 import workloads as WL
    wl = WL.get(args.workload)
    threads = oracle_threads()
    tids, tot, what = oracle_plan(wl, args.ref_seconds, args.steps + args.warmup)
    inputs = cpu_inputs(wl, tids, threads=threads)
    states = {}
    for s in range(args.warmup):
        time_oracle(wl, tids, inputs, s + 1, wl.hp.lr, args.seed, threads, states)
    secs = [time_oracle(wl, tids, inputs, args.warmup + s + 1, wl.hp.lr, args.seed, threads, states)
            for s in range(args.steps)]
    value = tot * len(secs) / sum(secs)
    ms = 1e3 * sum(secs) / len(secs)
    desc = f"each step: {what}, on {threads} host threads (tensors spread over them)"
    out = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "params/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": wl.name, "params": wl.numel, "tensors": len(wl.specs), "policy": policy_name(wl),
                   "params_per_step": tot},
        "cpu_baseline": {"value": value, "unit": "params/s", "cores": threads, "kind": "oracle", "sample": desc,
                         "host": host_info()},
        "e2e": {"value": value, "unit": "params/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "note": "CPU oracle (plain fp64 C) on the host cores; ms_per_step is the measured time of the step it ran",
    }
    print(json.dumps(out))


METRIC = "SkewAdam optimizer step over the 6.78B-parameter MoE shape set: params/s (step ms, HBM GB/s)"


# ---------------------------------------------------------------------------
# Across ranks (one process per GPU; every rank steps its own full parameter set)
# ---------------------------------------------------------------------------
def max_over_ranks(x, world, device):
    """The largest `x` over the ranks (the job's time is its slowest rank's); `x` on one rank."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(world, params_per_rank, ms):
    """Whole-job parameters per second: every rank's parameters over the job's step time."""
    return world * params_per_rank / (ms * 1e-3)


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
def flat_views(wl, dev):
    """One device buffer holding every tensor of the workload (bf16, or fp32 for an fp32
    tensor) at 512-byte aligned offsets (as the allocator places separate tensors);
    returns it, the per-tensor views and their byte offsets (with the total last)."""
    import torch
    offs, total = [], 0
    for s in wl.specs:
        total = (total + 511) // 512 * 512
        offs.append(total)
        total += s.numel * (4 if s.fp32 else 2)
    buf = torch.empty(max(total, 1), dtype=torch.uint8, device=dev)
    views = [buf[o:o + s.numel * (4 if s.fp32 else 2)].view(s.dtype).view(s.shape) for o, s in zip(offs, wl.specs)]
    return buf, views, offs + [total]


def e2e_groups(offs, n_groups):
    """Splits the tensors (byte offsets `offs`, total last) into at most n_groups runs of
    consecutive tensors of about equal bytes: [(first, end), ...]."""
    total, n = offs[-1], len(offs) - 1
    bounds, k = [0], 0
    for gi in range(1, n_groups):
        while k < n and offs[k] < total * gi / n_groups:
            k += 1
        if bounds[-1] < k < n:
            bounds.append(k)
    bounds.append(n)
    return list(zip(bounds[:-1], bounds[1:]))


def run_ours(args):
    import torch
    import torch.distributed as dist
    from paper_2607_19058_gb300 import _build
    from paper_2607_19058_gb300 import skewadam as S
    from paper_2607_19058_gb300 import workloads as WL

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    _build.build()
    dev = torch.device("cuda", local)
    wl = WL.get(args.workload)
    hp = wl.hp
    # inputs resident in HBM before timing, one allocation per tensor (as a framework keeps
    # its parameters)
    W = [WL.init_weight(wl, k, dev) for k in range(len(wl.specs))]
    G = [WL.grad(wl, k, 1, dev) for k in range(len(wl.specs))]
    params = [(W[k], G[k], s.tier, S.F_NO_DECAY if s.no_decay else 0) for k, s in enumerate(wl.specs)]
    opt = S.SkewAdam(params, S.hparams(hp.beta1, hp.beta2, hp.eps, hp.clip_d, hp.weight_decay, hp.policy))
    bm = byte_model(opt, len(wl.specs))
    wg_bytes = sum(w.numel() * w.element_size() + g.numel() * g.element_size() for w, g in zip(W, G))
    stream = torch.cuda.current_stream()
    gscale = None if args.grad_scale is None else torch.tensor([args.grad_scale], dtype=torch.float32, device=dev)
    torch.cuda.synchronize()

    step = 0
    for _ in range(args.warmup):
        step += 1
        opt.step(step, hp.lr, args.seed, grad_scale=gscale)
    opt.sync_status()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    clk = clocks_start(vis.split(",")[local] if vis else local)
    S.skew_profile_begin(opt.h, args.steps)
    marks = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]  # step boundaries
    e0, e1 = marks[0], marks[-1]
    e0.record(stream)
    for i in range(args.steps):
        step += 1
        opt.step(step, hp.lr, args.seed, grad_scale=gscale)
        marks[i + 1].record(stream)
    torch.cuda.synchronize()
    clocks = clocks_stop(clk)
    opt.sync_status()
    names, rows = S.skew_profile_end(opt.h)
    ms = max_over_ranks(e0.elapsed_time(e1) / args.steps, world, dev)
    if world > 1:
        dist.barrier()

    # per-kernel live durations; per-step times between consecutive step boundaries
    kmean = {n: statistics.fmean(r[i] for r in rows) for i, n in enumerate(names)}
    spans = [marks[i].elapsed_time(marks[i + 1]) for i in range(args.steps)]
    step_stats = {"median_ms": statistics.median(spans), "mean_ms": statistics.fmean(spans),
                  "min_ms": min(spans), "max_ms": max(spans)} if spans else None
    dom = max(kmean, key=kmean.get)
    peak, peak_src = peaks()
    dom_bytes = bm["kernels"][dom]
    achieved = dom_bytes / (kmean[dom] * 1e-3) / 1e9
    step_gbs = bm["step_min"] / (ms * 1e-3) / 1e9

    # end to end through the C ABI with host buffers: every step copies all gradients in
    # from pinned host memory and all updated weights back out. The step has no coupling
    # across tensors, so this leg runs it as --e2e-groups handles over runs of consecutive
    # tensors, each a 512-byte aligned slice of one device buffer per kind: group g's
    # gradients come in (one copy), its step runs, its weights go out (one copy), while the
    # next group's gradients are already coming in. Each copy waits only for the step that
    # frees its buffer, so the host link stays busy in both directions.
    e2e = None
    # pinned host memory of this leg: gradients in and weights out, for every rank on this host
    host_need = wg_bytes * int(os.environ.get("LOCAL_WORLD_SIZE", "1"))
    host_avail = mem_available()
    if not args.no_e2e and args.e2e_steps > 0 and host_avail is not None and host_need > 0.8 * host_avail:
        e2e = {"value": None, "unit": "params/s",
               "skipped": f"host memory: {host_need / 1e9:.0f} GB of pinned buffers for the ranks on this host, "
                          f"{host_avail / 1e9:.0f} GB available"}
    elif not args.no_e2e and args.e2e_steps > 0:
        Wbuf, Wf, offs = flat_views(wl, dev)
        Gbuf, Gf, _ = flat_views(wl, dev)
        for k in range(len(wl.specs)):
            Wf[k].copy_(W[k])
            Gf[k].copy_(G[k])
        groups = e2e_groups(offs, max(1, args.e2e_groups))
        opts = [S.SkewAdam([(Wf[k], Gf[k], wl.specs[k].tier, S.F_NO_DECAY if wl.specs[k].no_decay else 0)
                            for k in range(k0, k1)],
                           S.hparams(hp.beta1, hp.beta2, hp.eps, hp.clip_d, hp.weight_decay, hp.policy))
                for k0, k1 in groups]
        spans = [(offs[k0], offs[k1] if k1 < len(wl.specs) else offs[-1]) for k0, k1 in groups]
        for _ in range(args.warmup):
            step += 1
            for o in opts:
                o.step(step, hp.lr, args.seed)
        # pinned buffers on the GPU's own NUMA node: allocate them from that node's CPUs
        # (pages land on the node of the thread that first touches them)
        numa = gpu_numa(vis.split(",")[local] if vis else local)
        prev_aff = os.sched_getaffinity(0) if hasattr(os, "sched_getaffinity") else None
        if numa["node_cpus"] and prev_aff is not None:
            try:
                os.sched_setaffinity(0, set(numa["node_cpus"]) & prev_aff or prev_aff)
            except OSError:
                pass
        hg = torch.empty(Gbuf.numel(), dtype=torch.uint8, pin_memory=True)
        hw = torch.empty(Wbuf.numel(), dtype=torch.uint8, pin_memory=True)
        hg.copy_(Gbuf)
        hw.copy_(Wbuf)
        numa["pinned_pages_by_node"] = {"grads": pages_by_node(hg.data_ptr()), "weights": pages_by_node(hw.data_ptr())}
        # the link alone: one copy each way, then both at once (4 GB or less), timed over
        # three rounds after an untimed one; taken before the end-to-end region and again
        # after it, since the link is shared (each host CPU serves two GPUs) and its rate
        # can change from one minute to the next
        nb = min(int(Gbuf.numel()), 4 << 30)
        s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)

        def link_rates():
            out = {}
            for name, dirs in (("h2d", ("in",)), ("d2h", ("out",)), ("both", ("in", "out"))):
                ta, tb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                for rep in range(4):
                    torch.cuda.synchronize()
                    if rep == 1:
                        ta.record(stream)
                    sts = [s_in if d == "in" else s_out for d in dirs]
                    for st_ in sts:          # both directions start together
                        st_.wait_stream(stream)
                    for d, st_ in zip(dirs, sts):
                        with torch.cuda.stream(st_):
                            if d == "in":
                                Gbuf[:nb].copy_(hg[:nb], non_blocking=True)
                            else:
                                hw[:nb].copy_(Wbuf[:nb], non_blocking=True)
                    for st_ in sts:
                        stream.wait_stream(st_)
                tb.record(stream)
                torch.cuda.synchronize()
                out[name + "_gbs"] = 3 * len(dirs) * nb / (ta.elapsed_time(tb) * 1e-3) / 1e9
            return out

        link = link_rates()
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        ev = lambda: torch.cuda.Event(enable_timing=False)
        stepped = [None] * len(groups)
        drained = [None] * len(groups)

        def e2e_steps(k):
            nonlocal step
            for _ in range(k):
                step += 1
                for gi, (lo, hi) in enumerate(spans):
                    if stepped[gi] is not None:
                        s_in.wait_event(stepped[gi])       # the group's last step has read its gradients
                    with torch.cuda.stream(s_in):
                        Gbuf[lo:hi].copy_(hg[lo:hi], non_blocking=True)
                    loaded = ev()
                    loaded.record(s_in)
                    stream.wait_event(loaded)
                    if drained[gi] is not None:
                        stream.wait_event(drained[gi])     # the group's last weights are back on the host
                    opts[gi].step(step, hp.lr, args.seed)
                    stepped[gi] = ev()
                    stepped[gi].record(stream)
                    s_out.wait_event(stepped[gi])
                    with torch.cuda.stream(s_out):
                        hw[lo:hi].copy_(Wbuf[lo:hi], non_blocking=True)
                    drained[gi] = ev()
                    drained[gi].record(s_out)

        # untimed warm-up of the whole leg, copies included: the first device access to
        # each page of freshly pinned host memory costs extra (about 190 ms for 2 x 12 GiB
        # here), which a step-only warm-up leaves inside the timed region
        e2e_steps(max(1, args.warmup))
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(s_in)
        e2e_steps(args.e2e_steps)
        b.record(s_out)
        torch.cuda.synchronize()
        # integrity of the leg: each group's first and last 16 MiB of updated weights in
        # host memory equal the device's, and its gradients on the device equal the host's
        chk = 16 << 20
        w_ok = g_ok = True
        checked = 0
        for lo, hi in spans:
            for a0, a1 in ((lo, min(hi, lo + chk)), (max(lo, hi - chk), hi)):
                w_ok &= bool(torch.equal(hw[a0:a1].to(dev), Wbuf[a0:a1]))
                g_ok &= bool(torch.equal(hg[a0:a1].to(dev), Gbuf[a0:a1]))
                checked += 2 * (a1 - a0)
        link_after = link_rates()
        e2e_ms = max_over_ranks(a.elapsed_time(b) / args.e2e_steps, world, dev)
        if prev_aff is not None:
            try:
                os.sched_setaffinity(0, prev_aff)
            except OSError:
                pass
        e2e = {"value": job_rate(world, bm["N"], e2e_ms), "unit": "params/s", "ms_per_step": e2e_ms,
               "h2d_bytes_per_step": int(Gbuf.numel()), "d2h_bytes_per_step": int(Wbuf.numel()),
               "h2d_gbs": Gbuf.numel() / (e2e_ms * 1e-3) / 1e9, "d2h_gbs": Wbuf.numel() / (e2e_ms * 1e-3) / 1e9,
               "verified": {"weights_back_equal": w_ok, "grads_in_equal": g_ok, "bytes_checked": checked},
               "link_alone": link, "link_alone_after": link_after, "numa": {k: v for k, v in numa.items() if k != "node_cpus"},
               "groups": len(groups),
               "path": f"skew_step via ctypes on {len(groups)} handles over runs of consecutive tensors; every "
                       "step copies all gradients in from pinned host memory and all updated weights back to "
                       "pinned host memory, one copy per direction per group, a group's copies beside the "
                       "other groups' steps"}
        for o in opts:
            o.sync_status()
            o.close()
        del hg, hw, Wf, Gf, Wbuf, Gbuf

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        threads = oracle_threads()
        tids, tot, what = oracle_plan(wl, args.cpu_seconds, 1)
        inputs = cpu_inputs(wl, tids, src={k: (W[k], G[k]) for k in tids}, threads=threads)
        secs = time_oracle(wl, tids, inputs, 1, hp.lr, args.seed, threads)
        del inputs
        cpu = {"value": tot / secs, "unit": "params/s", "cores": threads, "kind": "oracle", "host": host_info(),
               "ms_per_step": 1e3 * secs,
               "sample": f"one step of {what} in {secs:.1f} s, plain fp64 C, tensors spread over {threads} "
                         "host threads"}

    if rank == 0:
        out = {
            "metric": METRIC,
            "value": job_rate(world, bm["N"], ms), "unit": "params/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": wl.name, "params": bm["N"], "tensors": len(wl.specs), "policy": policy_name(wl),
                       "state_bytes": opt.state_bytes, "workspace_bytes": opt.workspace_bytes,
                       "l2": f"inputs larger than L2 ({wg_bytes / 1e9:.1f} GB of weights + grads vs 129 MiB), no flush",
                       "weights_grads": "bf16, W~N(0,0.02^2), G~N(0,1e-3^2)",
                       "grad_scale": args.grad_scale},
            "hbm": {"min_bytes_per_step": bm["step_min"], "achieved_gbs": step_gbs,
                    "frac_of_8tbs": step_gbs / NOMINAL_HBM_GBS, "frac_of_measured": step_gbs / peak,
                    "peak_gbs": peak, "peak_source": peak_src},
            "roofline": {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": recorded_traffic(dom, dom_bytes),
                         "traffic_source": "ncu DRAM bytes of one launch on the small workload, scaled by algorithmic bytes",
                         "algorithmic_bytes_per_launch": dom_bytes,
                         "launch_ms": kmean[dom], "peak_source": peak_src},
            "kernels_ms": kmean,
            "kernel_algorithmic_bytes": bm["kernels"],
            "step_spans": step_stats,
            "e2e": e2e,
            "cpu_baseline": cpu,
            "gpu_launches": args.steps * S.skew_launches_per_step(opt.h),
            "clocks": clocks,
        }
        print(json.dumps(out))
    opt.close()
    if world > 1:
        dist.destroy_process_group()


def main():
    global _ORACLE_THREADS
    args = parse()
    _ORACLE_THREADS = args.cpu_threads if args.cpu_threads > 0 else None
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
