"""Benchmark of the cold full-vocabulary mask step on GB300.

Workload (default): SQL SELECT-only projection, schema 200 x 30, vocabulary
V = 151,936 (seeded, BPE-like, ~3% multi-word tokens), batch B = 32 parser
configurations at prefixes of U[50, 2000] tokens, fp32 logits N(0, 3).

One step = the whole per-token hot path for one batch, through the C ABI:
  grid_advance_masks: the advance (out-of-place, one admitted token per row)
  fed inside the mask step's first kernel, then the mask step (allowed sets +
  EOS gate, trie walk, id-order packing, with the in-place -inf fill of the
  fp32 logits fused into the packing).  The same step as two calls
  (grid_advance, then grid_masks_apply) is timed beside it.
The standalone grid_apply_mask kernel is timed on its own for its HBM
roofline (fp32 headline batch; bf16 B=256 in the cold-schema line).
Steps rotate over 16 distinct pre-built batches (512 prefixes); their logits
(16 x 19.45 MB = 311 MB) exceed the 129 MB L2, so every step reads cold logits.

Prints one JSON line (rank 0).  ``--impl reference`` times the CPU oracle on a
bounded sample of the same workload instead.
"""
import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

N_BATCHES = 16
METRIC = "cold full-vocab masks/s (batch-32 mask step at V=151,936)"


MASK_KERNELS = ["k_row", "k_filter", "k_walk", "k_pack"]
COUNTERS = os.path.join(ROOT, "profiles", "counters_sql_select_only.json")
SMSP_PER_SM = 4  # warp schedulers per SM, each issuing at most one warp instruction per clock
LANES = 32       # a warp-wide shared-memory access serves 32 lanes in one pipe cycle


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def _source_sha():
    """Hash of the device sources without comments and blank lines, so that the
    committed counters stay valid across comment-only edits."""
    import hashlib
    import re
    h = hashlib.sha256()
    for f in ("grid_kernels.cu", "grid_device.cuh", "grid_state.cuh"):
        with open(os.path.join(ROOT, "paper_2607_11951_gb300", "csrc", f)) as fh:
            for line in fh:
                code = re.sub(r"//.*", "", line).strip()
                if code:
                    h.update(code.encode() + b"\n")
    return h.hexdigest()[:16]


def _counters(kernel):
    """Per-launch ncu counters of `kernel` on this workload, from the committed
    JSON summary, if they were taken on the current kernel sources."""
    try:
        with open(COUNTERS) as f:
            d = json.load(f)
        if d.get("source_sha") != _source_sha():
            return None
        k = d["kernels"][kernel]
        return {"inst": float(k["warp_inst_per_launch"]), "dram": float(k["dram_bytes_per_launch"])}
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    FIELDS = "clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown," \
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown," \
             "clocks_event_reasons.sw_power_cap"

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.rows = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) == 7:
                self.rows.append(parts)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=2)
        except Exception:
            self.proc.kill()
        sm = [float(r[0]) for r in self.rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in self.rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in self.rows for k in range(4) if r[3 + k].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(self.rows)}


def _gpu_index(local):
    """nvidia-smi index of this process's GPU (CUDA_VISIBLE_DEVICES applied)."""
    vis = os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",")
    vis = [v.strip() for v in vis if v.strip()]
    if local < len(vis) and vis[local].isdigit():
        return int(vis[local])
    return local


def max_over_ranks(ms, ws, device):
    """The slowest rank's time: every rank runs its own replica of the step
    (rows are independent; no collective on the data path), so the job takes
    as long as the slowest one.  A barrier follows so no rank runs ahead."""
    if ws <= 1:
        return ms
    import torch
    import torch.distributed as dist
    tt = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(tt, op=dist.ReduceOp.MAX)
    dist.barrier()
    return float(tt.item())


def replica_value(ws, B, steps, ms):
    """Whole-job masks/s: every rank's B rows per step, over the slowest time."""
    return ws * B * steps / (ms / 1e3)


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _oracle_pool(wl):
    import multiprocessing as mp
    from tests.harness import _init_worker
    cores = os.cpu_count() or 1
    ctx = mp.get_context("spawn")
    return ctx.Pool(cores, initializer=_init_worker, initargs=(wl["grammar"], wl["role"], wl["lexicons"])), cores


def _oracle_throughput(pool, cores, wl, rows, jobs_per_row, ids_per_job, seed):
    """Oracle mask throughput on the pool's workers: each job builds a
    configuration from its prefix (not timed) and computes the mask bits of a
    slice of token ids (timed inside the worker).  Returns (token checks per
    second over all workers, checks, worker-seconds)."""
    import numpy as np
    from tests.harness import _oracle_rows_timed
    V = len(wl["tokens"])
    rng = np.random.default_rng(seed)
    jobs = []
    for r in rows:
        ids = rng.choice(V, jobs_per_row * ids_per_job, replace=False)
        for part in np.array_split(ids, jobs_per_row):
            jobs.append((wl["prefixes"][r % len(wl["prefixes"])], wl["tokens"], wl["eos"], wl["specials"],
                         [int(x) for x in part]))
    checks, busy = 0, 0.0
    for bits, sec in pool.map(_oracle_rows_timed, jobs, chunksize=1):
        if bits is not None:
            checks += len(bits)
            busy += sec
    return checks / (busy / cores), checks, busy


def headline_config(B, V):
    """The workload named by both arms' lines."""
    return {"workload": "sql_select_only", "B": B, "V": V, "prefix_tokens": "U[50,2000]",
            "schema": "200 tables x 30 columns", "logits": "f32 N(0,3)",
            "batches": N_BATCHES, "l2": "rotating inputs: 16 logits batches = 311 MB > L2",
            "step": "grid_advance_masks (the advance inside the mask step, the logits fill fused)"}


def run_reference(args):
    """The CPU oracle as it stands, on the host cores: each step is a bounded
    sample of the headline workload (``--ref-tokens`` token ids of one
    configuration, split over a spawn pool of all cores), scaled to
    full-vocabulary masks per second."""
    ws, rank, _ = _dist()
    if rank != 0:
        return
    from workloads import configs
    wl = configs.sql_select_only()
    V = len(wl["tokens"])
    pool, cores = _oracle_pool(wl)
    per_job = max(1, args.ref_tokens // cores)
    times, checks = [], 0
    with pool:
        for k in range(args.warmup + args.steps):
            tps, n, _ = _oracle_throughput(pool, cores, wl, [k], cores, per_job, seed=k)
            if k >= args.warmup:
                times.append(n / tps)
                checks += n
    tot = sum(times)
    value = checks / V / tot
    B = wl["B"]
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "masks/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup,
            # the time of one batch-32 full-vocabulary step at the measured rate
            "ms_per_step": 1e3 * B / value, "sample_ms_per_step": 1e3 * tot / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u32",
            "data": "synthetic",
            "config": headline_config(B, V),
            "cpu_baseline": {"value": value, "unit": "masks/s", "cores": cores, "kind": "oracle",
                             "sample": "per step: %d random token ids of one configuration (rows rotate), split "
                                       "over %d spawn workers; worker time inside the mask only" %
                                       (per_job * cores, cores)},
            "e2e": {"value": value, "unit": "masks/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def cpu_baseline_sample(wl):
    """The oracle on a bounded sample of the workload: 4 configurations x
    48,000 random token ids over a spawn pool of all host cores, scaled to
    full-vocabulary masks per second."""
    V = len(wl["tokens"])
    pool, cores = _oracle_pool(wl)
    with pool:
        tps, n, busy = _oracle_throughput(pool, cores, wl, range(4), 2 * cores, 48000 // (2 * cores), seed=1)
    return {"value": tps / V, "unit": "masks/s", "cores": cores, "kind": "oracle",
            "sample": "4 configurations x 48,000 random token ids of the headline workload (%d checks, %.1f "
                      "worker-seconds inside the mask on %d spawn workers), scaled to full-vocabulary masks" %
                      (n, busy, cores)}


def _time_steps(fn, steps, warmup, stream):
    """Per-step device times (us) of fn(k) over `steps` steps after `warmup`."""
    import torch
    for k in range(warmup):
        fn(k)
    torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for k in range(steps):
        evs[k][0].record(stream)
        fn(warmup + k)
        evs[k][1].record(stream)
    torch.cuda.synchronize()
    return sorted(a.elapsed_time(b) * 1e3 for a, b in evs)


def _apply_alone(G, mask, logits, steps, stream):
    """Mean device time (us) of grid_apply_mask alone, launched back to back
    over rotating logits buffers (larger than L2 together)."""
    import torch
    for k in range(3):
        G.grid_apply_mask(mask, logits[k % len(logits)], stream)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for k in range(steps):
        G.grid_apply_mask(mask, logits[k % len(logits)], stream)
    b.record(stream)
    torch.cuda.synchronize()
    return a.elapsed_time(b) * 1e3 / steps


def _roof_apply(B, V, esz, us, label):
    hbm_peak, peak_kind = _peaks()
    W = (V + 31) // 32
    nbytes = B * W * 4 + B * V * esz  # the mask read once + every logit written once
    ach = nbytes / (us * 1e-6) / 1e9
    return {"kernel": label, "bound": "hbm", "achieved": ach, "peak": hbm_peak,
            "peak_kind": peak_kind + " copy bandwidth", "unit": "GB/s", "frac": ach / hbm_peak,
            "bytes_per_launch": nbytes, "us_per_launch": us,
            "timing": "back-to-back launches over rotating logits buffers (> L2), CUDA events"}


def run_sweep(args):
    """Flatness of the per-step cost (the paper's requirement R): grid_masks on
    B=32 configurations per cell, n in {100, 1k, 4k, 16k} prefix tokens x
    nesting depth in {1, 8, 32, 64}; p50 per cell and, per depth, the OLS slope
    of step time vs n.  One JSON line with the clocks sampled meanwhile."""
    import numpy as np
    import torch
    from paper_2607_11951_gb300 import grid as G
    from workloads import configs
    dev = torch.device("cuda", 0)
    stream = torch.cuda.current_stream()
    warmup = max(3, args.warmup)
    ns, depths = [100, 1000, 4000, 16000], [1, 8, 32, 64]
    first = configs.sql_sweep_cell(ns[0], depths[0])
    grammar = G.Grammar(first["grammar"], first["role"], first["lexicons"])
    vocab = G.Vocab(first["tokens"], first["eos"], first["specials"])
    spec = G.Spec(grammar, vocab)
    B, V = first["B"], len(first["tokens"])
    W = (V + 31) // 32
    mask = torch.zeros((B, W), dtype=torch.int32, device=dev)
    status = torch.zeros(B, dtype=torch.int32, device=dev)
    built = {}
    for d in depths:
        for n in ns:
            wl = configs.sql_sweep_cell(n, d)
            c = G.Configs(spec, B)
            tt = np.full((B, n), -1, dtype=np.int32)
            for i, p in enumerate(wl["prefixes"]):
                tt[i, :len(p)] = p
            G.grid_advance(spec.h, c.h, c.h, torch.from_numpy(tt).to(dev), status)
            torch.cuda.synchronize()
            assert (status.cpu().numpy() == 0).all(), (n, d, status)
            built[(n, d)] = c
    clk = ClockSampler(_gpu_index(0))
    clk.start()
    cells = {}
    for d in depths:
        for n in ns:
            c = built[(n, d)]
            t = _time_steps(lambda k: G.grid_masks(spec.h, c.h, mask, status, stream), args.steps, warmup, stream)
            assert (status.cpu().numpy() == 0).all(), (n, d, status)
            p50 = t[len(t) // 2]
            cells["%d,%d" % (n, d)] = {"p50_us": p50, "p99_us": t[min(len(t) - 1, int(0.99 * len(t)))],
                                      "masks_per_s": B / (p50 * 1e-6)}
    clocks = clk.stop()
    slopes = {}
    for d in depths:
        x = np.array(ns, dtype=np.float64)
        y = np.array([cells["%d,%d" % (n, d)]["p50_us"] for n in ns])
        slope = float(np.polyfit(x, y, 1)[0]) * 1000.0
        slopes[str(d)] = {"us_per_1k_tokens": slope, "p50_at_100": y[0], "p50_at_16k": y[-1]}
    worst = max(abs(v["us_per_1k_tokens"]) for v in slopes.values())
    print(json.dumps({"metric": "per-step cost flatness: max |OLS slope| of grid_masks p50 vs prefix length",
                      "value": worst, "unit": "us per 1k prefix tokens", "higher_is_better": False,
                      "n_gpus": 1, "steps": args.steps, "warmup": warmup, "dtype": "u32", "data": "synthetic",
                      "config": {"workload": "sql_sweep_cell", "B": B, "V": V, "grammar": "SQL admin",
                                 "schema": "200 x 30", "n": ns, "depth": depths,
                                 "step": "grid_masks, K steps per cell with events around each"},
                      "cells": cells, "ols_slope_by_depth": slopes, "clocks": clocks}), flush=True)


def run_cold(args):
    """Cold-schema specialization: grid_specialize (CI classes of every
    precomputed lexer state over V=151,936) for a fresh 1,000 x 50 schema,
    then B=256 steps (advance + masks with the bf16 logits fill fused) on its
    configurations, and the standalone bf16 mask apply at B=256."""
    import numpy as np
    import torch
    from paper_2607_11951_gb300 import grid as G
    from workloads import configs
    dev = torch.device("cuda", 0)
    stream = torch.cuda.current_stream()
    warmup = max(3, args.warmup)
    wl = configs.sql_cold_schema()
    B, V = wl["B"], len(wl["tokens"])
    W = (V + 31) // 32
    t0 = time.perf_counter()
    grammar = G.Grammar(wl["grammar"], wl["role"], wl["lexicons"])
    t1 = time.perf_counter()
    vocab = G.Vocab(wl["tokens"], wl["eos"], wl["specials"])
    t2 = time.perf_counter()
    spec_ms = []
    specs = []
    clk = ClockSampler(_gpu_index(0))
    clk.start()
    for k in range(4):  # the first includes one-time CUDA module set-up
        torch.cuda.synchronize()
        a = time.perf_counter()
        specs.append(G.Spec(grammar, vocab))
        torch.cuda.synchronize()
        spec_ms.append((time.perf_counter() - a) * 1e3)
    spec = specs[-1]
    status = torch.zeros(B, dtype=torch.int32, device=dev)
    mask = torch.zeros((B, W), dtype=torch.int32, device=dev)
    c = G.Configs(spec, B)
    n = max(len(p) for p in wl["prefixes"])
    tt = np.full((B, n), -1, dtype=np.int32)
    for i, p in enumerate(wl["prefixes"]):
        tt[i, :len(p)] = p
    G.grid_advance(spec.h, c.h, c.h, torch.from_numpy(tt).to(dev), status)
    G.grid_masks(spec.h, c.h, mask, status)
    torch.cuda.synchronize()
    assert (status.cpu().numpy() == 0).all(), status
    from tests.harness import unpack
    bits = unpack(mask.cpu().numpy().view(np.uint32), V)
    rng = np.random.default_rng(7)
    tok = torch.from_numpy(np.array([rng.choice(np.nonzero(bits[i])[0]) for i in range(B)], np.int32)).to(dev)
    scratch = G.Configs(spec, B)
    logits = [torch.from_numpy(configs.logits(200 + k, B, V)).to(dev).to(torch.bfloat16) for k in range(2)]

    def step(k):
        G.grid_advance_masks(spec.h, c.h, scratch.h, tok, mask, status, logits[k % 2], stream)

    t = _time_steps(step, args.steps, warmup, stream)
    apply_us = _apply_alone(G, mask, logits, args.steps, stream)
    clocks = clk.stop()
    p50 = t[len(t) // 2]
    print(json.dumps({"metric": "cold-schema specialization ms (fresh 1,000 x 50 schema, V=151,936)",
                      "value": sorted(spec_ms[1:])[1], "unit": "ms", "higher_is_better": False,
                      "n_gpus": 1, "steps": args.steps, "warmup": warmup, "dtype": "u32", "data": "synthetic",
                      "grid_specialize_ms": sorted(spec_ms[1:])[1], "grid_specialize_ms_first": spec_ms[0],
                      "grid_compile_ms": (t1 - t0) * 1e3, "grid_load_vocab_ms": (t2 - t1) * 1e3,
                      "spec": spec.info(), "step_p50_us": p50, "step_p99_us": t[min(len(t) - 1, int(0.99 * len(t)))],
                      "masks_per_s": B / (p50 * 1e-6),
                      "roofline_apply_bf16": _roof_apply(B, V, 2, apply_us, "k_apply<bf16> (grid_apply_mask)"),
                      "config": {"workload": "sql_cold_schema", "B": B, "V": V, "schema": "1,000 x 50",
                                 "logits": "bf16 N(0,3), 2 rotating batches = 156 MB > L2",
                                 "step": "grid_advance_masks"},
                      "clocks": clocks}), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--ref-tokens", type=int, default=8192)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--workload", default="headline", choices=["headline", "sweep", "cold"],
                    help="headline: the driver's line; sweep: per-step cost vs prefix length and nesting "
                         "(n in {100,1k,4k,16k} x depth in {1,8,32,64}); cold: specialization of a fresh "
                         "1,000 x 50 schema, then B=256 steps with bf16 logits")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    if args.workload == "sweep":
        return run_sweep(args)
    if args.workload == "cold":
        return run_cold(args)
    args.warmup = max(3, args.warmup)

    import numpy as np
    import torch
    ws, rank, local = _dist()
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if ws > 1 else 0)
    torch.cuda.set_device(dev)

    from paper_2607_11951_gb300 import grid as G
    from workloads import configs
    from tests.harness import unpack

    # ---- inputs (seeded, synthetic) ----
    batches = [configs.sql_select_only(prefix_seed=5000 + k) for k in range(N_BATCHES)]
    wl = batches[0]
    cpu_base = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu_base = cpu_baseline_sample(wl)
    B, V = wl["B"], len(wl["tokens"])
    W = (V + 31) // 32
    grammar = G.Grammar(wl["grammar"], wl["role"], wl["lexicons"])
    vocab = G.Vocab(wl["tokens"], wl["eos"], wl["specials"])
    spec = G.Spec(grammar, vocab)
    stream = torch.cuda.current_stream()
    cfgs, toks = [], []
    status = torch.zeros(B, dtype=torch.int32, device=dev)
    mask = torch.zeros((B, W), dtype=torch.int32, device=dev)
    rng = np.random.default_rng(42)
    for k, bw in enumerate(batches):
        c = G.Configs(spec, B)
        n = max(len(p) for p in bw["prefixes"])
        tt = np.full((B, n), -1, dtype=np.int32)
        for i, p in enumerate(bw["prefixes"]):
            tt[i, :len(p)] = p
        G.grid_advance(spec.h, c.h, c.h, torch.from_numpy(tt).to(dev), status)
        torch.cuda.synchronize()
        assert (status.cpu().numpy() == 0).all(), status
        G.grid_masks(spec.h, c.h, mask, status)
        torch.cuda.synchronize()
        assert (status.cpu().numpy() == 0).all(), status
        bits = unpack(mask.cpu().numpy().view(np.uint32), V)
        pick = np.array([rng.choice(np.nonzero(bits[i])[0]) for i in range(B)], dtype=np.int32)
        cfgs.append(c)
        toks.append(torch.from_numpy(pick).to(dev))
    scratch = G.Configs(spec, B)
    logits = [torch.from_numpy(configs.logits(100 + k, B, V)).to(dev) for k in range(N_BATCHES)]

    def step(k, ev=None):
        i = k % N_BATCHES
        if ev:
            ev[0].record(stream)
        G.grid_advance_masks(spec.h, cfgs[i].h, scratch.h, toks[i], mask, status, logits[i], stream)
        if ev:
            ev[1].record(stream)

    def step2(k):  # the same step as two calls
        i = k % N_BATCHES
        G.grid_advance(spec.h, cfgs[i].h, scratch.h, toks[i], status, stream)
        G.grid_masks_apply(spec.h, scratch.h, mask, status, logits[i], stream)

    for k in range(args.warmup):
        step(k)
    torch.cuda.synchronize()
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    # Passes of K steps each, back to back:
    #   A  the timed region of `value`: events only at its two ends
    #   B  per-step events around the call (p50/p99)
    #   C  events recorded by the library around each kernel of the mask step
    #   D  the standalone grid_apply_mask (its HBM roofline)
    #   E  one more pass with k_walk's work counters on (their counts only;
    #      counting slows the kernel, so no time is taken from this pass)
    # Events cost the GPU a little time each, so A carries none between steps.
    ev_b = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    ev_c = [[torch.cuda.Event(enable_timing=True) for _ in range(len(MASK_KERNELS) + 1)] for _ in range(args.steps)]
    for ev in ev_b + ev_c:  # create each event by a first record, before the library sees its handle
        for e in ev:
            e.record(stream)
    torch.cuda.synchronize()
    clk = ClockSampler(_gpu_index(local))
    clk.start()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    torch.cuda.nvtx.range_push("timed")
    t_start.record(stream)
    for k in range(args.steps):
        step(args.warmup + k)
    t_end.record(stream)
    torch.cuda.synchronize()
    torch.cuda.nvtx.range_pop()
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    total_ms = t_start.elapsed_time(t_end)
    for k in range(args.steps):  # pass B
        step(args.warmup + k, ev_b[k])
    for k in range(args.steps):  # pass C
        G.grid_configs_set_events(scratch.h, ev_c[k])
        step(args.warmup + k)
    torch.cuda.synchronize()
    G.grid_configs_set_events(scratch.h, [])
    # the two-call step (grid_advance, then grid_masks_apply), and the advance
    # alone, back to back
    sa_, sb_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sa_.record(stream)
    for k in range(args.steps):
        step2(args.warmup + k)
    sb_.record(stream)
    sa_.synchronize()
    sb_.synchronize()
    two_call_ms = sa_.elapsed_time(sb_) / args.steps
    sa_.record(stream)
    for k in range(args.steps):
        i = (args.warmup + k) % N_BATCHES
        G.grid_advance(spec.h, cfgs[i].h, scratch.h, toks[i], status, stream)
    sb_.record(stream)
    torch.cuda.synchronize()
    adv_alone_us = sa_.elapsed_time(sb_) * 1e3 / args.steps
    apply_us = _apply_alone(G, mask, logits, args.steps, stream)  # pass D
    # pass F: the same steps through the configuration-keyed mask cache (its
    # context-independent part read from entries filled by earlier steps; the
    # residue and EOS gate computed every step): the warm path beside the cold
    cache = G.Cache(spec, 1024)

    def warm_step(k):
        i = k % N_BATCHES
        G.grid_advance_masks(spec.h, cfgs[i].h, scratch.h, toks[i], mask, status, logits[i], stream, cache=cache)

    for k in range(N_BATCHES + args.warmup):
        warm_step(k)
    torch.cuda.synchronize()
    c0 = cache.stats()
    wa, wb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    wa.record(stream)
    for k in range(args.steps):
        warm_step(args.warmup + k)
    wb.record(stream)
    torch.cuda.synchronize()
    c1 = cache.stats()
    warm_ms = wa.elapsed_time(wb) / args.steps
    cache_line = {"ms_per_step": warm_ms, "masks_per_s": B / (warm_ms * 1e-3),
                  "hit_rate": (c1["hits"] - c0["hits"]) / max(1, c1["lookups"] - c0["lookups"]),
                  "entries_ready": c1["ready"],
                  "step": "grid_advance_masks through the cache (fused fp32 fill), cache warmed by one pass "
                          "over the 16 batches"}
    # pass G: independent batch-32 steps on 4 streams at once (each stream
    # with its own scratch, mask and status; no two streams on one batch at a
    # time): how much of the GPU one step leaves idle, beside the sequential
    # value above
    NS_ = 4
    strs = [torch.cuda.Stream(device=dev) for _ in range(NS_)]
    scr = [G.Configs(spec, B) for _ in range(NS_)]
    msk = [torch.zeros((B, W), dtype=torch.int32, device=dev) for _ in range(NS_)]
    sts = [torch.zeros(B, dtype=torch.int32, device=dev) for _ in range(NS_)]

    def conc_run(n):
        start = torch.cuda.Event(enable_timing=True)
        done = [torch.cuda.Event() for _ in range(NS_)]
        start.record(stream)
        for x in strs:
            x.wait_event(start)
        for k in range(n):
            j, i = k % NS_, k % N_BATCHES
            G.grid_advance_masks(spec.h, cfgs[i].h, scr[j].h, toks[i], msk[j], sts[j], logits[i], strs[j])
        for j in range(NS_):
            done[j].record(strs[j])
            stream.wait_event(done[j])
        end = torch.cuda.Event(enable_timing=True)
        end.record(stream)
        return start, end

    conc_run(N_BATCHES)
    torch.cuda.synchronize()
    ca, cb = conc_run(args.steps)
    torch.cuda.synchronize()
    conc_ms = ca.elapsed_time(cb)
    concurrent = {"streams": NS_, "masks_per_s": B * args.steps / (conc_ms * 1e-3),
                  "ms_per_step": conc_ms / args.steps,
                  "step": "grid_advance_masks, K steps dealt round-robin to the streams"}
    clocks = clk.stop()
    work = torch.zeros(6, dtype=torch.int64, device=dev)  # pass E
    G.grid_spec_set_work_counters(spec.h, work)
    for k in range(N_BATCHES):
        step(args.warmup + k)
    torch.cuda.synchronize()
    G.grid_spec_set_work_counters(spec.h, None)
    work = [int(x) / N_BATCHES for x in work.cpu().tolist()]
    total_ms = max_over_ranks(total_ms, ws, dev)
    per_step = [e[0].elapsed_time(e[1]) * 1e3 for e in ev_b]
    call_us = statistics.mean(per_step)
    kern_us = {}
    for j, name in enumerate(MASK_KERNELS):
        kern_us[name] = statistics.mean(e[j].elapsed_time(e[j + 1]) * 1e3 for e in ev_c)
    per_step.sort()
    p50 = per_step[len(per_step) // 2]
    p99 = per_step[min(len(per_step) - 1, int(math.ceil(0.99 * len(per_step))) - 1)]
    value = replica_value(ws, B, args.steps, total_ms)

    # ---- end to end through the public API with host buffers ----
    # Every step copies its token ids and logits from pinned host memory and
    # reads its mask and status back.  Three streams: a host-to-device stream brings
    # step k+1's inputs into the second of two device buffers while step k
    # computes, the compute stream waits for them before using them, and a
    # device-to-host stream reads each step's mask and status (double
    # buffered) while the next step computes.  The timed region starts before
    # the first copy and ends after the last read.
    e2e = None
    if not args.no_e2e:
        h_logits = [torch.from_numpy(configs.logits(100 + k, B, V)).pin_memory() for k in range(4)]
        h_toks = [t.cpu().pin_memory() for t in toks]
        h_mask = [torch.empty((B, W), dtype=torch.int32).pin_memory() for _ in range(2)]
        h_status = [torch.empty(B, dtype=torch.int32).pin_memory() for _ in range(2)]
        d_tok = [torch.empty(B, dtype=torch.int32, device=dev) for _ in range(2)]
        d_logits = [torch.empty((B, V), dtype=torch.float32, device=dev) for _ in range(2)]
        d_mask = [torch.empty((B, W), dtype=torch.int32, device=dev) for _ in range(2)]
        d_status = [torch.empty(B, dtype=torch.int32, device=dev) for _ in range(2)]
        h2d, d2h = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
        ev_in = [torch.cuda.Event() for _ in range(2)]    # step's inputs on the device
        ev_used = [torch.cuda.Event() for _ in range(2)]  # step's masking done: its input buffers are free
        ev_out = [torch.cuda.Event() for _ in range(2)]   # step's mask and status read back

        def copy_in(k):
            j = k % 2
            h2d.wait_event(ev_used[j])
            with torch.cuda.stream(h2d):
                d_tok[j].copy_(h_toks[k % N_BATCHES], non_blocking=True)
                d_logits[j].copy_(h_logits[k % 4], non_blocking=True)
            ev_in[j].record(h2d)

        def e2e_step(k, last):
            i, j = k % N_BATCHES, k % 2
            if not last:
                copy_in(k + 1)
            stream.wait_event(ev_in[j])
            stream.wait_event(ev_out[j])  # mask/status buffers of step k-2 read back
            G.grid_advance_masks(spec.h, cfgs[i].h, scratch.h, d_tok[j], d_mask[j], d_status[j], d_logits[j],
                                 stream)
            ev_used[j].record(stream)
            d2h.wait_event(ev_used[j])
            with torch.cuda.stream(d2h):
                h_mask[j].copy_(d_mask[j], non_blocking=True)
                h_status[j].copy_(d_status[j], non_blocking=True)
            ev_out[j].record(d2h)

        def run(n):
            for e in ev_used + ev_out:
                e.record(stream)
            copy_in(0)
            for k in range(n):
                e2e_step(k, k == n - 1)
            stream.wait_event(ev_out[(n - 1) % 2])

        run(args.warmup)
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        run(args.steps)
        b.record(stream)
        torch.cuda.synchronize()
        e_ms = a.elapsed_time(b)
        e_ms = max_over_ranks(e_ms, ws, dev)
        e2e = {"value": replica_value(ws, B, args.steps, e_ms), "unit": "masks/s",
               "h2d_bytes_per_step": B * 4 + B * V * 4, "d2h_bytes_per_step": B * W * 4 + B * 4,
               "overlap": "inputs of step k+1 copied in and outputs of step k read back on two copy streams "
                          "while step k computes (double-buffered)"}

    # ---- rooflines ----
    # mask apply: HBM-bound, write-mostly; algorithmic bytes = the mask read
    # once + every logit written once (the reject fill touches every sector)
    roof_apply = _roof_apply(B, V, 4, apply_us, "k_apply<f32> (grid_apply_mask)")
    ac = _counters("k_apply")
    roof_apply["traffic"] = ac["dram"] if ac else None
    # walk: its algorithmic work (lexer steps of byte walks, ACTION and GOTO
    # lookups of reduce chains, verdict-class events), each unit at least one
    # dependent shared-memory access by one lane: the ceiling is the shared-
    # memory pipe serving 32 lanes per clock per SM at the sampled clock.  The
    # issue-rate fraction (ncu warp instructions, committed with a source hash)
    # is given beside it.
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    mhz = clocks.get("sm_mhz") or 2070.0
    walk_us = kern_us["k_walk"]
    units = sum(work[:4])
    peak_units = sms * LANES * mhz * 1e6 / 1e9
    roof_walk = {"kernel": "k_walk (grid_advance_masks)", "bound": "alu",
                 "unit": "G work units/s (lexer steps + ACTION + GOTO lookups + verdict-class events)",
                 "achieved": units / (walk_us * 1e-6) / 1e9, "peak": peak_units,
                 "peak_kind": "derived: %d SMs x %d lanes of shared-memory pipe per clock x %.0f MHz sampled" %
                 (sms, LANES, mhz),
                 "work_per_launch": {"lexer_steps": work[0], "action_lookups": work[1], "goto_lookups": work[2],
                                     "verdict_class_events": work[3]},
                 "evaluated_per_launch": {"verdict_class_records": work[4], "byte_walked_spellings": work[5],
                                          "verdict_class_records_per_row": work[4] / B,
                                          "paper_class_verdicts_per_step": "143-150 (its own SQL bench and "
                                                                           "tokenizer, Sec. 4.2 / Sec. 8.2)"},
                 "traffic": None}
    roof_walk["frac"] = roof_walk["achieved"] / peak_units
    wc = _counters("k_walk")
    issue_peak = sms * SMSP_PER_SM * mhz * 1e6 / 1e9
    roof_walk["issue"] = {"unit": "G warp-inst/s", "peak": issue_peak,
                          "achieved": wc["inst"] / (walk_us * 1e-6) / 1e9 if wc else None,
                          "frac": wc["inst"] / (walk_us * 1e-6) / 1e9 / issue_peak if wc else None,
                          "counters": os.path.relpath(COUNTERS, ROOT) if wc else "stale or missing"}
    if wc:
        roof_walk["traffic"] = wc["dram"]
    dominant = max((k for k in kern_us), key=kern_us.get)
    roof = roof_walk if dominant == "k_walk" else roof_apply

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "masks/s", "n_gpus": ws, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "u32", "data": "synthetic",
                "config": headline_config(B, V),
                "p50_us": p50, "p99_us": p99,
                "token_checks_per_s": value * V,
                "call_us": {"grid_advance_masks": call_us},
                "two_call_step": {"ms_per_step": two_call_ms, "masks_per_s": B / (two_call_ms * 1e-3),
                                  "grid_advance_alone_us": adv_alone_us,
                                  "step": "grid_advance, then grid_masks_apply (the advance in its own kernel)"},
                "kernel_us": kern_us, "dominant_kernel": dominant,
                "roofline": roof, "roofline_apply": roof_apply, "cpu_baseline": cpu_base, "e2e": e2e,
                "mask_cache": cache_line, "concurrent_batches": concurrent,
                "gpu_launches": args.steps * len(MASK_KERNELS), "clocks": clocks,
                "timing": "value: K steps between two events; p50/p99 and call_us: a second pass of K "
                          "steps with events around each call; kernel_us: a third pass with events "
                          "around each kernel of the step (k_row includes the advance, k_pack the logits "
                          "fill); roofline_apply: the standalone grid_apply_mask, back to back"}
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
