"""Benchmark of the scheduler hot path on one window: prints ONE JSON line (rank 0).

A step is one ``ps_schedule_window`` call on the production-scale window (1024 instances x 16384
requests, the 1024-instance workload): the probe kernel (prefix-hit length of all R x I pairs), the
fused score kernel (latencies, admission sets and the independent per-request pick of all pairs)
and the greedy in-window assignment, with inputs resident in HBM.  ``value`` is request x instance
scorings per second over whole steps; ``decisions_per_s`` is R per step time.  ``e2e`` repeats the
step through the same C ABI with page-locked host buffers (host->device window copy and
device->host decisions inside the timed region).

Timing: CUDA events on the stream the library launches on, W untimed warm-up steps, K timed steps
between barrier + synchronize, max over ranks.  Inputs (1.8 GB of tables, 0.5 GB of chains) are
larger than L2, so no flush is needed between steps.

--impl reference times the oracle (the single-threaded C++ restatement of Algorithm 1) on this
host's cores on bounded prefixes of the same window, as the reference arm.

Multi-GPU (torchrun): each rank schedules its own instance pool and window (seed + rank): the
windows are independent problems, so there is no collective on the data path (weak scaling).
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "request×instance scorings/sec and scheduling decisions/sec at 1 GB300; % HBM roofline"
WORKLOADS = {
    0: "tiny window: 8 instances x 64 requests",
    1: "eval-scale window: 64 instances x 4096 requests",
    2: "production-scale window: 1024 instances x 16384 requests, 8192 Zipf(1.1) sessions, "
       "200K-block caches at 90% load factor",
    3: "long-context window: 256 instances x 2048 requests, prefixes 128K-1M tokens",
}


def _env_rank():
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def rank_seed(config: int, rank: int) -> int:
    """Seed of a rank's instance pool and window: each rank schedules an independent problem."""
    import workload as W
    return int(W.CONFIGS[config]["seed"]) + rank


def max_over_ranks(value: float, device) -> float:
    """The largest value over all ranks (the job is as slow as its slowest rank); identity when
    torch.distributed is not initialised."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(world: int, units_per_rank: int, ms_per_step: float) -> float:
    """Whole-job throughput (weak scaling): every rank processes units_per_rank per step and the
    step time is the slowest rank's."""
    return world * units_per_rank / (ms_per_step / 1000.0)


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        fd, self.path = tempfile.mkstemp(prefix="clocks_bench_", suffix=".csv")
        os.close(fd)

    def __enter__(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.dev}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if not os.path.exists(self.path):
            return None
        with open(self.path) as f:
            lines = f.readlines()
        os.remove(self.path)
        if self.proc is None:
            return None
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = max(mx, float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def probe_algorithmic_bytes(st: dict, I: int, with_tpf: bool) -> tuple[int, int]:
    """Bytes the two probe kernels' algorithm must move in one launch, from the library's own
    counters of that launch (ps_last_probe_stats): one 32-byte sector per table lookup (the least a
    random lookup can move), 8 B per chain block read (the key of a lookup, or a staged block), the
    earlier row's hits a derived row starts from (4 B per instance), and per pair the u32 hit and,
    when the greedy pass follows, the f32 T_pf written."""
    out_b = (4 + (4 if with_tpf else 0)) * I
    lookups = st["lookups_scratch"] + st["lookups_derived"]
    nbytes = (32 * lookups + 8 * st["chain_reads"] + out_b * (st["rows_scratch"] + st["rows_derived"])
              + 4 * I * st["rows_derived"])
    return int(nbytes), int(lookups)


def score_algorithmic_bytes(R: int, I: int, per_pair_outputs: bool) -> int:
    """Bytes the fused score kernel must move in one launch: the u32 hit of every pair read; with
    per-pair outputs the f32 TPOT, f32 TTFT and u8 class of every pair written; per request its
    prompt length and two targets read and its pick (i32) and path (u8) written; per instance its
    state (b, qr, B_max as i32; q, S, M_KV as i64) read."""
    per_pair = 4 + ((4 + 4 + 1) if per_pair_outputs else 0)
    return int(R * I * per_pair + R * (12 + 5) + I * 36)


def profile_figure(name: str, label: str):
    """A per-unit DRAM figure ("<label>: <number>") from a committed ncu summary under profiles/, or
    None when the summary is absent."""
    path = os.path.join(ROOT, "profiles", name)
    if not os.path.exists(path):
        return None
    for line in open(path):
        if line.startswith(label + ":"):
            return float(line.split(":", 1)[1])
    return None


def oracle_sample(wl, seconds: float, max_rows: int | None = None):
    """Oracle greedy over successive prefixes of the window until ~`seconds` of CPU time."""
    import workload as W
    from oracle import Oracle
    win = wl.window
    t0 = time.perf_counter()
    orc = Oracle(wl.instances.I, wl.model).load(wl.instances)
    load_s = time.perf_counter() - t0
    done, chunk, spent = 0, 4, 0.0
    while done < win.R and spent < seconds and (max_rows is None or done < max_rows):
        n = min(chunk, win.R - done)
        sub = W.Window(chain_off=win.chain_off[done:done + n + 1] - win.chain_off[done],
                       chain_hash=win.chain_hash[win.chain_off[done]:win.chain_off[done + n]],
                       prompt_tokens=win.prompt_tokens[done:done + n],
                       ttft_target=win.ttft_target[done:done + n], tpot_target=win.tpot_target[done:done + n],
                       session=win.session[done:done + n], out_tokens=win.out_tokens[done:done + n])
        t = time.perf_counter()
        orc.schedule(sub)
        spent += time.perf_counter() - t
        done += n
        chunk = min(chunk * 2, 256)
    return done, spent, load_s


def run_reference(args):
    rank, world, _ = _env_rank()
    if rank != 0:
        return
    import workload as W
    W.build()
    import oracle
    oracle.build()
    wl = W.generate(args.config)
    I, R = wl.instances.I, wl.window.R
    budget = max(5.0, 60.0 / max(1, args.steps + args.warmup))
    times, rows = [], []
    from oracle import Oracle
    orc = Oracle(I, wl.model).load(wl.instances)
    done = 0
    win = wl.window
    for k in range(args.warmup + args.steps):
        # each step: the oracle's greedy over the next requests of the window, about `budget` s
        t0 = time.perf_counter()
        n_done = 0
        while time.perf_counter() - t0 < budget and done < R:
            n = min(8, R - done)
            sub = W.Window(chain_off=win.chain_off[done:done + n + 1] - win.chain_off[done],
                           chain_hash=win.chain_hash[win.chain_off[done]:win.chain_off[done + n]],
                           prompt_tokens=win.prompt_tokens[done:done + n],
                           ttft_target=win.ttft_target[done:done + n], tpot_target=win.tpot_target[done:done + n],
                           session=win.session[done:done + n], out_tokens=win.out_tokens[done:done + n])
            orc.schedule(sub)
            done += n
            n_done += n
        if k >= args.warmup:
            times.append(time.perf_counter() - t0)
            rows.append(n_done)
    t = sum(times)
    value = sum(rows) * I / t if t > 0 else 0.0
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "scorings/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * t / max(1, args.steps),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32+u64",
            "data": "synthetic (seeded generator)",
            "decisions_per_s": sum(rows) / t if t > 0 else 0.0,
            "config": {"workload": WORKLOADS.get(args.config, str(args.config)), "instances": I,
                       "window_requests": R},
            "cpu_baseline": {"value": value, "unit": "scorings/s", "cores": 1, "kind": "oracle",
                             "sample": f"oracle greedy over the first {sum(rows)} requests of the window "
                                       f"(each decision scores all {I} instances)"},
            "e2e": {"value": value, "unit": "scorings/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def run_streaming(args):
    """Streaming workload (1024 instances, 1000-request windows, state carried across windows):
    per window one schedule, commit and advance (engine progress + leaf-first LRU eviction), with
    the window's arrays copied from page-locked host memory inside the timed region.  Windows are
    drawn by the generator outside the timed region (its cost is not the scheduler's): all before
    timing for short runs, each just before it is scheduled for long ones (more than 64 windows, whose
    pinned copies would not all fit).  The time of a window is the device time of its three calls
    (CUDA events around them); the run's time is their sum.  Prints one JSON line: decisions/s and the
    share of each kernel."""
    import torch
    import workload as W
    import paper_2609_33224_gb300 as P
    rank, world, local = _env_rank()
    torch.cuda.set_device(local)
    P.build()
    W.build()
    wl = W.generate(4, seed=rank_seed(4, rank))
    ins = wl.instances
    Rw = wl.window.R
    n_win = args.warmup + args.steps
    lazy = n_win > 64

    def pinned(w):
        view = {np.dtype(np.uint64): np.int64, np.dtype(np.uint32): np.int32}
        return W.Window(**{k: torch.from_numpy(np.ascontiguousarray(getattr(w, k)).view(
            view.get(getattr(w, k).dtype, getattr(w, k).dtype))).pin_memory() for k in w.__dataclass_fields__})

    if lazy:
        maxb = 8192 * Rw  # every chain is at most 8192 blocks (128K tokens)
        hwins = None
    else:
        wins = [wl.window] + [wl.next_window() for _ in range(n_win - 1)]
        maxb = max(int(w.chain_off[-1]) for w in wins)
        hwins = [pinned(w) for w in wins]
    stream = torch.cuda.current_stream()
    sched = P.Scheduler(ins.I, ins.cap_blocks, Rw, maxb, wl.model, table_load_factor=wl.table_load_factor,
                        device=local, stream=stream.cuda_stream, probe_mode=P.PS_PROBE_SEARCH, track_lru=True,
                        max_active_requests=512)
    sched.load_workload_instances(ins)
    sched.load_requests(wl.initial_requests())
    kern = {"probe": 0.0, "score": 0.0, "greedy": 0.0, "commit": 0.0, "advance": 0.0}
    paths = np.zeros(3, np.int64)
    ea, eb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    total_ms = 0.0
    with ClockSampler(local) as clk:
        for w in range(n_win):
            if lazy:
                hw = pinned(wl.window if w == 0 else wl.next_window())
            else:
                hw = hwins[w]
            torch.cuda.synchronize()
            e0.record(stream)
            out = sched.schedule_window(hw)
            sched.commit_window(last_use=w + 1)
            t = sched.timings()
            ea.record(stream)
            sched.advance_window(20.0, 1000, evict=True)
            eb.record(stream)
            e1.record(stream)
            torch.cuda.synchronize()
            if w >= args.warmup:
                total_ms += e0.elapsed_time(e1)
                for k in ("probe", "score", "greedy", "commit"):
                    kern[k] += max(0.0, t[k])
                kern["advance"] += ea.elapsed_time(eb)
                paths += np.bincount(out["path"].astype(np.int64), minlength=3)
    ms = max_over_ranks(total_ms / args.steps, f"cuda:{local}")
    km = {k: v / args.steps for k, v in kern.items()}
    cached = sched.cached_blocks()
    sched.close()
    line = {"metric": "streaming scheduling decisions/sec (schedule + commit + advance per window) at 1 GB300",
            "value": job_rate(world, Rw, ms), "unit": "decisions/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32+u64", "data": "synthetic (seeded generator)",
            "config": {"workload": "streaming: 1024 instances, 1000-request windows, 200K-block caches, "
                                   "LRU leaf-first eviction, 20 ms engine progress per window",
                       "window_requests": Rw, "windows_timed": args.steps,
                       "inputs": "page-locked host windows, copied inside the timed region",
                       "path_counts": paths.tolist()},
            "kernel_ms_per_window": km,
            "greedy_share": km["greedy"] / ms if ms > 0 else None,
            "advance_share": km["advance"] / ms if ms > 0 else None,
            "cached_blocks_after": {"min": int(cached.min()), "max": int(cached.max()),
                                    "capacity": int(np.max(ins.cap_blocks))},
            "scorings_per_s": job_rate(world, Rw * ins.I, ms),
            "clocks": clk.summary()}
    if rank == 0:
        print(json.dumps(line))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", type=int, default=2)
    ap.add_argument("--tpot", type=float, default=None)
    ap.add_argument("--cpu-seconds", type=float, default=20.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--probe-mode", type=int, default=1, choices=[0, 1])
    ap.add_argument("--window-requests", type=int, default=None,
                    help="smaller window of the same workload (profiler captures only; not a bench line)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
        return
    if args.config == 4:
        run_streaming(args)
        return

    import torch
    rank, world, local = _env_rank()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    import workload as W
    import paper_2609_33224_gb300 as P
    P.build()
    W.build()
    over = {} if args.tpot is None else {"tpot_target_ms": args.tpot}
    if args.window_requests:
        over["window_requests"] = args.window_requests
    wl = W.generate(args.config, seed=rank_seed(args.config, rank), **over)
    win, ins = wl.window, wl.instances
    I, R = ins.I, win.R
    nb = np.diff(win.chain_off).astype(np.int64)
    stream = torch.cuda.current_stream()
    sched = P.scheduler_for(wl, device=local, stream=stream.cuda_stream, probe_mode=args.probe_mode)

    def to_dev(a):
        a = np.ascontiguousarray(a)
        view = {np.dtype(np.uint64): np.int64, np.dtype(np.uint32): np.int32}.get(a.dtype, a.dtype)
        return torch.from_numpy(a.view(view)).to(f"cuda:{local}")

    dwin = W.Window(**{k: to_dev(getattr(win, k)) for k in win.__dataclass_fields__})

    def step():
        return sched.schedule_window(dwin, scores=("best", "path"), device_outputs=True)

    for _ in range(args.warmup):
        step()
    pstats = sched.probe_stats()  # the probe phase of the last schedule step (same window every step)
    probe_bytes, n_probes = probe_algorithmic_bytes(pstats, I, with_tpf=args.probe_mode == 1)
    dist_on = world > 1
    if dist_on:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    kern = {"probe": [], "score": [], "greedy": [], "relations": [], "probe_scratch": [], "probe_derived": []}
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        e0.record(stream)
        for _ in range(args.steps):
            out = step()
            t = sched.timings()
            for k in kern:
                kern[k].append(t[k])
        e1.record(stream)
        torch.cuda.synchronize()
    if dist_on:
        dist.barrier()
    ms = max_over_ranks(e0.elapsed_time(e1) / args.steps, f"cuda:{local}")
    path_counts = np.bincount(out["path"].cpu().numpy().astype(np.int64), minlength=3).tolist()

    # e2e: the same step through the C ABI with page-locked host inputs and host outputs, the window
    # in the shared-prefix form (each request's own blocks and a parent link, ps_window.parent: what a
    # gateway that tracks sessions sends; the library rebuilds the chains on the device), and again
    # with every chain sent whole.
    def pinned(w):
        return type(w)(**{k: torch.from_numpy(np.ascontiguousarray(getattr(w, k)).view(
            {np.dtype(np.uint64): np.int64, np.dtype(np.uint32): np.int32}.get(getattr(w, k).dtype,
                                                                               getattr(w, k).dtype))).pin_memory()
            for k in w.__dataclass_fields__})

    def e2e_time(hw):
        sched.schedule_window(hw, scores=("best", "path"))
        torch.cuda.synchronize()
        if dist_on:
            dist.barrier()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            sched.schedule_window(hw, scores=("best", "path"))
        torch.cuda.synchronize()
        return max_over_ranks(1000 * (time.perf_counter() - t0) / args.steps, f"cuda:{local}")

    twin = W.tree_window(win)
    own_blocks = int(twin.chain_off[-1])
    e2e_ms = e2e_time(pinned(twin))
    e2e_full_ms = e2e_time(pinned(win))
    h2d = int(8 * (R + 1) + 8 * own_blocks + 4 * R + 12 * R)
    h2d_full = int(8 * (R + 1) + 8 * nb.sum() + 12 * R)
    d2h = int(R * (4 + 1 + 4) + R * (4 + 1))

    # The scoring call alone (ps_score_window, rows A1-A6): every per-pair output (hits, TPOT, TTFT,
    # class) and the per-request pick written to device buffers, timed the same way.
    want = ("hits", "tpot", "ttft", "cls", "best", "path")
    for _ in range(args.warmup):
        sched.score_window(dwin, want=want, device_outputs=True)
    skern = {"probe": [], "score": [], "relations": [], "probe_scratch": [], "probe_derived": []}
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        sched.score_window(dwin, want=want, device_outputs=True)
        t = sched.timings()
        for k in skern:
            skern[k].append(t[k])
    e1.record(stream)
    torch.cuda.synchronize()
    score_call_ms = max_over_ranks(e0.elapsed_time(e1) / args.steps, f"cuda:{local}")
    skm = {k: float(np.mean(v)) for k, v in skern.items()}
    score_bytes = score_algorithmic_bytes(R, I, per_pair_outputs=True)
    score_achieved = score_bytes / (skm["score"] / 1000) / 1e9

    km = {k: float(np.mean(v)) for k, v in kern.items()}
    phases = {k: km[k] for k in ("probe", "score", "greedy")}
    dominant = max(phases, key=phases.get)
    peak, peak_src = _peaks()
    probe_ms = km["probe_scratch"] + max(0.0, km["probe_derived"])
    # DRAM traffic per unit from the committed ncu summaries of the production window (scaled by this
    # run's units; None for another workload, whose kernels those captures do not cover)
    prod = args.config == 2 and args.probe_mode == 1
    greedy_traffic = profile_figure("greedy_pipe_production_window_1024x8192.md", "DRAM bytes per request") if prod else None
    probe_traffic = profile_figure("probe_search_production_window_1024x16384.md", "DRAM bytes per lookup") if prod else None
    score_traffic = profile_figure("score_block_production_window_1024x16384.md", "DRAM bytes per request") if prod else None
    score_kernel = "score_block_kernel" if 256 < I <= 1024 else "score_rows_kernel"
    if dominant == "probe":
        achieved = probe_bytes / (probe_ms / 1000) / 1e9
        roof = {"bound": "hbm", "kernel": "probe_search_kernel + probe_derived_kernel", "achieved": achieved,
                "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "traffic": None if probe_traffic is None else probe_traffic * n_probes,
                "peak_source": peak_src, "algorithmic_bytes_per_launch": probe_bytes}
    else:
        # per decision: the request's hit and T_pf rows (8 B per instance) and its decision outputs
        greedy_bytes = int(R * (8 * I + 16))
        achieved = greedy_bytes / (km[dominant] / 1000) / 1e9
        roof = {"bound": "hbm", "kernel": "greedy_pipe_kernel" if args.probe_mode == 1 else "greedy_kernel",
                "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "traffic": (None if greedy_traffic is None or args.probe_mode != 1 else greedy_traffic * R),
                "peak_source": peak_src, "algorithmic_bytes_per_launch": greedy_bytes,
                "ns_per_decision": 1e6 * km[dominant] / R,
                "note": "serial per-request dependency chain decided on one SM: latency-bound, not "
                        "bandwidth-bound; traffic scaled by request count from the 8192-request ncu capture"}
    probe_achieved = probe_bytes / (probe_ms / 1000) / 1e9
    # the whole A2 phase: the relations pass exists only to serve the probe, so it is counted too
    a2_ms = probe_ms + max(0.0, km["relations"])
    a2_achieved = probe_bytes / (a2_ms / 1000) / 1e9 if a2_ms > 0 else None
    line = {"metric": METRIC, "value": job_rate(world, R * I, ms), "unit": "scorings/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32+u64", "data": "synthetic (seeded generator)",
            "decisions_per_s": job_rate(world, R, ms),
            "config": {"workload": WORKLOADS.get(args.config, str(args.config)), "instances": I,
                       "window_requests": R, "window_chain_blocks": int(nb.sum()),
                       "tpot_target_ms": float(win.tpot_target[0]), "probe": ("hinted per-lane search of rows without an earlier prefix in the window, the rest derived"
                                 if args.probe_mode == 1 else "linear 32-wide warp walk"), "probes_per_window": n_probes,
                       "l2": "inputs larger than L2 (no flush)", "path_counts": path_counts},
            "kernel_ms": km,
            "probe_roofline": {"kernels": "probe_search_kernel + probe_derived_kernel", "achieved": probe_achieved,
                               "unit": "GB/s", "peak": peak, "frac": probe_achieved / peak,
                               "frac_vs_8tbs": probe_achieved / 8000.0, "ms": probe_ms,
                               "algorithmic_bytes_per_launch": probe_bytes, "stats": pstats,
                               "traffic": None if probe_traffic is None else probe_traffic * n_probes,
                               "a2_phase": {"kernels": "relations_kernel + probe_search_kernel + probe_derived_kernel",
                                            "ms": a2_ms, "achieved": a2_achieved,
                                            "frac": None if a2_achieved is None else a2_achieved / peak}},
            "roofline": roof,
            "scoring_call": {"what": "ps_score_window with hits, TPOT, TTFT and class of every pair and the "
                                     "per-request pick written to device buffers",
                             "ms": score_call_ms, "scorings_per_s": job_rate(world, R * I, score_call_ms),
                             "kernel_ms": skm,
                             "score_roofline": {"bound": "hbm", "kernel": score_kernel,
                                                "achieved": score_achieved, "peak": peak, "unit": "GB/s",
                                                "frac": score_achieved / peak, "peak_source": peak_src,
                                                "algorithmic_bytes_per_launch": score_bytes,
                                                "traffic": (None if score_traffic is None
                                                            else score_traffic * R)}},
            "e2e": {"value": job_rate(world, R * I, e2e_ms), "unit": "scorings/s", "ms_per_step": e2e_ms,
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "window_form": f"shared-prefix: {own_blocks} own blocks of {int(nb.sum())}, parent links"},
            "e2e_full_chains": {"value": job_rate(world, R * I, e2e_full_ms), "unit": "scorings/s",
                                "ms_per_step": e2e_full_ms, "h2d_bytes_per_step": h2d_full,
                                "d2h_bytes_per_step": d2h},
            # per step: window validation, last-block table, relations, base, probe (scratch rows),
            # probe (derived rows), score, greedy
            "gpu_launches": 8 * args.steps,
            "clocks": clk.summary()}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        rows, spent, load_s = oracle_sample(wl, args.cpu_seconds)
        line["cpu_baseline"] = {"value": rows * I / spent, "unit": "scorings/s", "cores": 1, "kind": "oracle",
                                "sample": f"oracle greedy over the first {rows} of {R} requests "
                                          f"({rows * I} scorings, {spent:.1f} s; cache load {load_s:.1f} s untimed)",
                                "decisions_per_s": rows / spent}
    sched.close()
    if rank == 0:
        print(json.dumps(line))
    if dist_on:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
