#!/usr/bin/env python3
"""Benchmark of the HedgeSpec panoramic-feedback step on GB300.

One step = hs_feedback (alpha and e_len for every drafter, query and
position) + hs_learner_step (length loss, NormalHedge or Hedge update and
the next choice) on one batch of seeded synthetic logits already resident in
HBM.  Prints ONE JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
                  [--mode stochastic|greedy|topl|token] [--branch-l L]
                  [--impl ours|reference]

--mode topl runs the draft-tree feedback (Thm 2: the drafter proposes its L
most likely tokens as a node's children) with a stochastic target.
--mode token runs the stochastic feedback and then the token-level game with
delay through QFI-D: the chunk's verified tokens join the per-query stream,
the learner consumes every revealed token loss in token order, and the next
drafter is drawn from the weights with a caller-supplied uniform.

Timing: the K steps run as CUDA-graph replays on one stream, bracketed by
CUDA events after a barrier + synchronize; inputs rotate over enough buffer
sets (>= 2x the L2 size in total) that no call finds its logits in L2.  The
feedback path alone is timed the same way in a second region for the
roofline.  `e2e` repeats the step through the public API from pinned host
buffers, with the host->device copy of every step's logits and the
device->host read of its result (weights and choice) inside the timed region.
Under torchrun each rank runs its own queries (weak scaling, no collective on
the data path); value = all ranks' evaluations / the slowest rank's time.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = ("drafter-position-vocab evals/s and achieved HBM GB/s (% of GB300 peak) "
          "per hs_feedback")
DEFAULT_WORKLOAD = "long_session"
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--mode", choices=("stochastic", "greedy", "topl", "token"),
                    default="stochastic")
    ap.add_argument("--branch-l", type=int, default=10,
                    help="children per node of the draft tree (--mode topl)")
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=200)
    ap.add_argument("--clock-preload-s", type=float, default=1.5,
                    help="seconds of untimed step replays before the timed region, under "
                         "the clock sampler")
    ap.add_argument("--cpu-budget-s", type=float, default=8.0,
                    help="seconds of oracle work per CPU-baseline leg (1 thread, all cores)")
    ap.add_argument("--queries", type=int, default=0,
                    help="run the workload with this many queries B instead of its own (a "
                         "smaller case of the same kernels, for profiling)")
    ap.add_argument("--session", action="store_true",
                    help="long-session learner run: cumulative regret over the workload's rounds")
    ap.add_argument("--rounds", type=int, default=0, help="session rounds (0: the workload's)")
    return ap.parse_args()


# ---- clocks during the timed region -----------------------------------------

class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", self.gpu_id], stdout=self.out, stderr=subprocess.DEVNULL)
            self.t0 = time.time()
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self) -> dict | None:
        if self.proc is None:
            return None
        if time.time() - self.t0 < 0.35:
            time.sleep(0.35 - (time.time() - self.t0))
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
                except ValueError:
                    continue
        os.unlink(self.path)
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[j] for _, _, flags in rows for j, v in enumerate(flags)
                          if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows),
                "sm_max_mhz": max(r[1] for r in rows), "reasons": reasons,
                "samples": len(rows)}


def gpu_uuid(dev) -> str:
    import torch
    try:
        u = str(torch.cuda.get_device_properties(dev).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        return str(dev.index)


# ---- roofline inputs ----------------------------------------------------------

def measured_hbm_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


# the sources of the kernels a feedback call of each mode launches
KERNEL_SOURCES = {
    "stochastic": ("hs_common.cuh", "hs_feedback.cu", "hs_fused.cu", "hs_fused.h",
                   "hs_stream.cu", "hs_stream.h", "hs_twopass.cu", "hs_twopass.h"),
    "greedy": ("hs_common.cuh", "hs_feedback.cu", "hs_greedy.cu", "hs_greedy.h"),
    "topl": ("hs_common.cuh", "hs_feedback.cu", "hs_topl.cu", "hs_topl.h"),
    "token": ("hs_common.cuh", "hs_feedback.cu", "hs_fused.cu", "hs_fused.h", "hs_stream.cu",
              "hs_stream.h", "hs_twopass.cu", "hs_twopass.h", "hs_delayed.cu",
              "hs_learner_core.cuh"),
}


def kernel_source_hash(mode: str) -> str:
    """Hash of the kernel sources a feedback call of `mode` runs: a committed
    ncu summary counts only while the kernels it measured are unchanged."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2510_20064_gb300", "csrc")
    for name in KERNEL_SOURCES[mode]:
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + f.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str, mode: str):
    """DRAM bytes per feedback call from a committed ncu summary, if that
    summary was taken on the current kernel sources."""
    path = os.path.join(ROOT, "profiles", f"feedback_{workload}_{mode}.md")
    if not os.path.exists(path):
        return None
    fields = {}
    with open(path) as f:
        for line in f:
            if ":" in line and line.strip().startswith("- "):
                k, v = line.strip()[2:].split(":", 1)
                fields[k.strip()] = v.strip().strip("`")
    if fields.get("kernel_source_hash") != kernel_source_hash(mode):
        return None
    try:
        return int(fields["dram_bytes_per_call"])
    except (KeyError, ValueError):
        return None


# ---- CPU oracle baseline ------------------------------------------------------

def oracle_alpha(o, w, args):
    """The oracle's per-pair feedback for the bench's mode."""
    if args.mode == "topl":
        return lambda t, d: o.alpha_topl(t, d, w.temperature, False, args.branch_l)
    greedy = args.mode == "greedy"
    return lambda t, d: o.alpha_pair(t, d, w.temperature, greedy)


def host_cpu() -> dict:
    """The host's usable core count and CPU model (lscpu), recorded beside
    the oracle's timings."""
    try:
        cores = len(os.sched_getaffinity(0))
    except AttributeError:
        cores = os.cpu_count() or 1
    model = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                model = line.split(":", 1)[1].strip()
                break
    except (OSError, subprocess.SubprocessError):
        pass
    return {"nproc": cores, "model": model, "machine": os.uname().machine}


def oracle_tiles(w, d):
    """(target row, drafter rows) of every (b,k) tile of one input set, as
    the stored bytes the oracle reads."""
    from paper_2510_20064_gb300 import synth
    t_all = synth.storage_numpy(d["target"])
    path = d.get("path")
    path_np = None if path is None else path.cpu().numpy()
    B = d["drafter"].shape[1]
    for tile in range(B * w.P):
        b, k = divmod(tile, w.P)
        trow = t_all[b, path_np[b, k]] if path_np is not None else t_all[b, k]
        yield trow, synth.storage_numpy(d["drafter"][:, b, k])


def oracle_rate(w, tiles, args, threads: int, budget_s: float):
    """The fp64 C oracle as it stands, on whole (b,k) tiles cycled from
    `tiles`, on `threads` host threads for about budget_s seconds: each
    thread takes one drafter row at a time (rows in parallel, each row's sums
    sequential inside the oracle; ctypes releases the GIL during the call).
    Returns (evals/s, rows done, seconds)."""
    import concurrent.futures as cf
    import threading

    import oracle
    o = oracle.get()
    pair = oracle_alpha(o, w, args)
    rows = [(t, dr[i]) for t, dr in tiles for i in range(w.N)]
    lock = threading.Lock()
    counter = [0]
    t_start = time.perf_counter()
    deadline = t_start + budget_s

    def worker():
        done = 0
        while time.perf_counter() < deadline:
            with lock:
                j = counter[0]
                counter[0] += 1
            t, d = rows[j % len(rows)]
            pair(t, d)
            done += 1
        return done

    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        done = sum(ex.map(lambda _: worker(), range(threads)))
    elapsed = time.perf_counter() - t_start
    return done * w.V / elapsed, done, elapsed


def oracle_sample(w, sets, args):
    """The fp64 C oracle (as it stands) on whole (b,k) tiles of the first
    input set: once on 1 thread and once on every host core, each for
    --cpu-budget-s seconds."""
    host = host_cpu()
    tiles = []
    for tile in oracle_tiles(w, sets[0]):
        tiles.append(tile)
        if len(tiles) >= 4 * host["nproc"]:  # enough distinct rows to keep every core busy
            break
    v1, n1, s1 = oracle_rate(w, tiles, args, 1, args.cpu_budget_s)
    vall, nall, sall = oracle_rate(w, tiles, args, host["nproc"], args.cpu_budget_s)
    return {"value": vall, "unit": "evals/s", "cores": host["nproc"], "kind": "oracle",
            "value_1_core": v1, "host": host,
            "sample": f"{nall} drafter rows (all cores) and {n1} rows (1 core) cycling over "
                      f"{len(tiles)} (b,k) tiles x {w.N} drafters x V={w.V} of the {w.name} "
                      f"workload, fp64 C oracle, {sall:.1f} s / {s1:.1f} s"}


# ---- the benchmark -------------------------------------------------------------

def run_ours(args):
    import torch

    import paper_2510_20064_gb300 as hf
    from paper_2510_20064_gb300 import dist as hdist
    from paper_2510_20064_gb300 import synth

    rank, world, local = hdist.rank_info()
    assert torch.cuda.is_available(), "bench.py needs a GPU"
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    hdist.init("nccl", world)
    hf.lib()

    w = synth.WORKLOADS[args.workload]
    if args.queries:
        w = dataclasses.replace(w, B=args.queries, name=f"{w.name}_B{args.queries}")
    greedy = args.mode == "greedy"
    topl = args.mode == "topl"
    token = args.mode == "token"
    learner = hf.HS_HEDGE if w.learner == "hedge" else hf.HS_NORMALHEDGE
    N, B, P, V = w.N, w.B, w.P, w.V
    props = torch.cuda.get_device_properties(dev)
    l2 = getattr(props, "L2_cache_size", 0) or 129 * 2**20
    n_sets = max(2, math.ceil(2 * l2 / w.bytes_per_call))
    sets = [synth.make_inputs(w, rnd=s, device=dev, seed=hdist.rank_seed(w.seed_base, rank) + s)
            for s in range(n_sets)]
    if token:  # the uniforms of the sampled play are inputs, drawn per input set
        gen = torch.Generator(device=dev).manual_seed(hdist.rank_seed(w.seed_base, rank) + 99)
        for d in sets:
            d["uniforms"] = torch.rand(w.B, generator=gen, device=dev)

    stream = torch.cuda.Stream(device=dev)
    alpha = torch.empty(N, B, P, device=dev)
    e_len = torch.empty(N, B, device=dev)
    ws_bytes = (hf.hs_feedback_topl_workspace_size(N, B, P, V) if topl else
                hf.hs_feedback_workspace_size(N, B, P, V, synth.DTYPES[w.dtype], greedy))
    ws = torch.empty(max(ws_bytes, 1), dtype=torch.uint8, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    state = torch.zeros(N, B, device=dev)
    weights = torch.full((N, B), 1.0 / N, device=dev)
    sel = torch.zeros(B, dtype=torch.int32, device=dev)
    eta = w.eta if w.eta else math.sqrt(8 * math.log(max(N, 2)) / 2000)
    if token:
        K = P - 1
        ts = hf.TokenStream(N, B, K + 2 * P, dev)
        k_full = torch.full((B,), K, dtype=torch.int32, device=dev)  # no censoring: fixed K
        sel_arg = torch.zeros(B, dtype=torch.int32, device=dev)
        played = torch.zeros(B, device=dev)

    def feedback(d):
        if topl and "path" in d:
            hf.hs_feedback_topl_path(d["target"], d["path"], d["drafter"], args.branch_l,
                                     w.temperature, False, alpha=alpha, e_len=e_len,
                                     workspace=ws, dev_status=status, stream=stream)
        elif topl:
            hf.hs_feedback_topl(d["target"], d["drafter"], args.branch_l, w.temperature, False,
                                alpha=alpha, e_len=e_len, workspace=ws, dev_status=status,
                                stream=stream)
        elif "path" in d:
            hf.hs_feedback_path(d["target"], d["path"], d["drafter"], w.temperature, greedy,
                                alpha=alpha, e_len=e_len, workspace=ws, dev_status=status,
                                stream=stream)
        else:
            hf.hs_feedback(d["target"], d["drafter"], w.temperature, greedy, alpha=alpha,
                           e_len=e_len, workspace=ws, dev_status=status, stream=stream)

    def token_learner(d):
        # this chunk's verified tokens (played by sel) join the stream; QFI-D
        # catch-up on every revealed token loss; the next drafter is drawn
        hf.hs_token_append(ts, alpha, k_full, sel, dev_status=status, stream=stream)
        hf.hs_token_learner_step(ts, K, hf.HS_LOSS_LENGTH, learner, eta, state, weights, sel_arg,
                                 played_loss=played, dev_status=status, stream=stream)
        hf.hs_sample_select(weights, d["uniforms"], selected=sel, dev_status=status,
                            stream=stream)

    def step(d):
        feedback(d)
        if token:
            token_learner(d)
        else:
            hf.hs_learner_step(alpha, e_len, hf.HS_LOSS_LENGTH, learner, eta, state, weights,
                               sel, stream=stream)

    # eager warm-up, then graphs of whole steps and of feedback calls
    with torch.cuda.stream(stream):
        for s in range(max(args.warmup, 3)):
            step(sets[s % n_sets])
    stream.synchronize()
    per_graph = n_sets * max(1, math.ceil(32 / n_sets))

    def capture(fn, count):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for s in range(count):
                fn(sets[s % n_sets])
        return g

    def timed(fn, steps, preload_s=0.0):
        full, rem = divmod(steps, per_graph)
        g_full = capture(fn, per_graph) if full else None
        g_rem = capture(fn, rem) if rem else None
        g_any = g_full or g_rem
        with torch.cuda.stream(stream):
            for _ in range(2):  # graph warm-up
                g_any.replay()
        stream.synchronize()
        if preload_s > 0:
            # keep the GPU busy for preload_s right before the timed region,
            # so that the clock samples describe the kernels under load
            w0 = torch.cuda.Event(enable_timing=True)
            w1 = torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                w0.record(stream)
                g_any.replay()
                w1.record(stream)
            stream.synchronize()
            per_replay = max(w0.elapsed_time(w1) / 1e3, 1e-6)
            with torch.cuda.stream(stream):
                for _ in range(int(math.ceil(preload_s / per_replay))):
                    g_any.replay()
            stream.synchronize()
        hdist.barrier(world, dev)
        torch.cuda.synchronize(dev)
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):  # replay() launches on the current stream
            t0.record(stream)
            for _ in range(full):
                g_full.replay()
            if rem:
                g_rem.replay()
            t1.record(stream)
        torch.cuda.synchronize(dev)
        hdist.barrier(world, dev)
        return t0.elapsed_time(t1) / 1e3

    clocks = ClockSampler(gpu_uuid(dev))
    clocks.start()
    t_step = timed(step, args.steps, preload_s=args.clock_preload_s)
    clk = clocks.stop()
    if clk is not None:
        clk["window"] = (f"{args.clock_preload_s:.1f} s of step-graph replays right before the "
                         "timed region, then the timed region")
    t_fb = timed(feedback, args.steps)
    t_learn = timed(token_learner, args.steps) if token else None
    assert int(status.item()) == 0, hf.hs_status_string(int(status.item()))

    # ---- end to end through the public API from pinned host buffers ----
    host_sets = [{k: v.cpu().pin_memory() for k, v in d.items() if torch.is_tensor(v)}
                 for d in sets[:2]]
    dsts = {k: torch.empty_like(v, device=dev) for k, v in host_sets[0].items()}
    out_w = torch.empty(N, B).pin_memory()
    out_s = torch.empty(B, dtype=torch.int32).pin_memory()
    h2d = sum(v.numel() * v.element_size() for k, v in host_sets[0].items() if k != "sigma")
    d2h = out_w.numel() * 4 + out_s.numel() * 4
    e2e_steps = max(1, min(args.steps, args.e2e_steps))

    def e2e_step(s):
        hs = host_sets[s % 2]
        for k, v in hs.items():
            if k != "sigma":
                dsts[k].copy_(v, non_blocking=True)
        step(dsts)
        out_w.copy_(weights, non_blocking=True)
        out_s.copy_(sel, non_blocking=True)

    with torch.cuda.stream(stream):
        # warm-up over both host sets: the first copy out of a freshly pinned
        # buffer pays a one-time mapping cost of tens of milliseconds
        for s in range(2 * max(1, math.ceil(args.warmup / 2))):
            e2e_step(s)
        hdist.barrier(world, dev)
        torch.cuda.synchronize(dev)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for s in range(e2e_steps):
            e2e_step(s)
        e1.record(stream)
        torch.cuda.synchronize(dev)
    t_e2e = e0.elapsed_time(e1) / 1e3

    t_step = hdist.max_over_ranks(t_step, world, dev)
    t_fb = hdist.max_over_ranks(t_fb, world, dev)
    t_e2e = hdist.max_over_ranks(t_e2e, world, dev)
    if token:
        t_learn = hdist.max_over_ranks(t_learn, world, dev)
    evals_step = w.evals
    value = world * args.steps * evals_step / t_step
    peak, peak_src = measured_hbm_peak()
    fb_avg = t_fb / args.steps
    achieved = w.bytes_per_call / fb_avg / 1e9
    launches_step = (3 if token else 1) + (
        hf.hs_feedback_topl_kernel_count(N, B, P, V) if topl else
        hf.hs_feedback_kernel_count(N, B, P, V, synth.DTYPES[w.dtype], greedy))

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = oracle_sample(w, sets, args)
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "evals/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * t_step / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
            "data": "synthetic: seeded Zipf + Gaussian logits, drafter = target + noise "
                    "(no dataset, no trained weights)",
            "config": {"workload": w.name, "N": N, "B": B, "K": w.K, "V": V,
                       "temperature": None if greedy else w.temperature, "mode": args.mode,
                       "branch_l": args.branch_l if topl else None,
                       "learner": "hedge" if learner == hf.HS_HEDGE else "normalhedge",
                       "loss": "length", "l2": f"{n_sets} rotating input sets "
                       f"({n_sets * w.bytes_per_call / 2**20:.0f} MiB > 2x L2 {l2 / 2**20:.0f} MiB)",
                       "parallelism": f"queries sharded over {world} rank(s), no collective"},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "peak_source": peak_src,
                         "traffic": profiled_traffic(w.name, args.mode),
                         "kernel": "hs_feedback (all its kernels), timed alone",
                         "algorithmic_bytes_per_call": w.bytes_per_call,
                         "us_per_call": 1e6 * fb_avg},
            "cpu_baseline": cpu,
            "e2e": {"value": world * e2e_steps * evals_step / t_e2e, "unit": "evals/s",
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": e2e_steps},
            "gpu_launches": launches_step * args.steps,
            "clocks": clk,
        }
        if token:
            line["config"]["learner_path"] = ("token-level game with delay through QFI-D, "
                                              "length loss, K = P-1, sampled play")
            line["learner_us_per_step"] = 1e6 * t_learn / args.steps
        print(json.dumps(line), flush=True)
    hdist.finalize(world)


def run_reference(args):
    """The fp64 CPU oracle on every host core, same metric and config: each
    step is a bounded sample of the workload, enough whole (b,k) tiles for
    one drafter row per core, the rows run in parallel (ctypes releases the
    GIL during each oracle call)."""
    from paper_2510_20064_gb300 import dist as hdist
    rank, world, _ = hdist.rank_info()
    if rank != 0:
        return
    import concurrent.futures as cf

    import oracle
    from paper_2510_20064_gb300 import synth
    w = synth.WORKLOADS[args.workload]
    host = host_cpu()
    cores = host["nproc"]
    tiles_per_step = max(1, math.ceil(cores / w.N))
    d = synth.make_inputs(w, device="cpu", B=min(w.B, max(2, math.ceil(2 * tiles_per_step / w.P))))
    tiles = list(oracle_tiles(w, d))
    o = oracle.get()
    pair = oracle_alpha(o, w, args)

    def one(ex, s):
        rows = []
        for j in range(tiles_per_step):
            t, dr = tiles[(s * tiles_per_step + j) % len(tiles)]
            rows.extend((t, dr[i]) for i in range(w.N))
        list(ex.map(lambda td: pair(*td), rows))

    with cf.ThreadPoolExecutor(max_workers=cores) as ex:
        for s in range(args.warmup):
            one(ex, s)
        t0 = time.perf_counter()
        for s in range(args.steps):
            one(ex, args.warmup + s)
        t = time.perf_counter() - t0
    evals_step = tiles_per_step * w.N * w.V
    value = args.steps * evals_step / t
    sample = (f"each step = {tiles_per_step} (b,k) tile(s) of {w.name}: {tiles_per_step * w.N} "
              f"drafter rows x V={w.V}, fp64 C oracle, rows in parallel on {cores} threads")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "evals/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * t / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "N": w.N, "B": w.B, "K": w.K, "V": w.V,
                   "mode": args.mode, "branch_l": args.branch_l if args.mode == "topl" else None},
        "cpu_baseline": {"value": value, "unit": "evals/s", "cores": cores, "kind": "oracle",
                         "sample": sample, "host": host},
        "e2e": {"value": value, "unit": "evals/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def run_session(args):
    """Many verification rounds with fresh logits each round: feedback, then
    Hedge and NormalHedge side by side on the same losses; reports the mean
    over queries of the cumulative regret sum_t f_t[i_t] - min_i sum_t f_t[i]
    (Sec. 3.1) of each learner."""
    import torch

    import paper_2510_20064_gb300 as hf
    from paper_2510_20064_gb300 import synth
    w = synth.WORKLOADS["long_session" if args.workload == DEFAULT_WORKLOAD else args.workload]
    rounds = args.rounds or w.rounds
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    hf.lib()
    N, B, P = w.N, w.B, w.P
    eta = w.eta or math.sqrt(8 * math.log(max(N, 2)) / rounds)
    alpha = torch.empty(N, B, P, device=dev)
    e_len = torch.empty(N, B, device=dev)
    ws = torch.empty(max(1, hf.hs_feedback_workspace_size(N, B, P, w.V, synth.DTYPES[w.dtype],
                                                          False)), dtype=torch.uint8, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    learners = {}
    for name, kind in (("hedge", hf.HS_HEDGE), ("normalhedge", hf.HS_NORMALHEDGE)):
        learners[name] = dict(kind=kind, state=torch.zeros(N, B, device=dev),
                              weights=torch.full((N, B), 1.0 / N, device=dev),
                              sel=torch.zeros(B, dtype=torch.int32, device=dev),
                              played=torch.zeros(B, device=dev),
                              loss=torch.empty(N, B, device=dev))
    cum = torch.zeros(N, B, device=dev, dtype=torch.float64)
    t_fb = 0.0
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_start = time.time()
    for t in range(rounds):
        d = synth.make_inputs(w, rnd=t, device=dev)
        ev0.record()
        hf.hs_feedback(d["target"], d["drafter"], w.temperature, False, alpha=alpha, e_len=e_len,
                       workspace=ws, dev_status=status)
        for L in learners.values():
            hf.hs_learner_step(alpha, e_len, hf.HS_LOSS_LENGTH, L["kind"], eta, L["state"],
                               L["weights"], L["sel"], loss_out=L["loss"],
                               played_loss=L["played"])
        ev1.record()
        cum += learners["hedge"]["loss"].double()
        ev1.synchronize()
        t_fb += ev0.elapsed_time(ev1)
        del d
    assert int(status.item()) == 0, hf.hs_status_string(int(status.item()))
    best = cum.min(dim=0).values
    out = {"session": w.name, "rounds": rounds, "N": N, "B": B, "K": w.K, "V": w.V,
           "eta_hedge": eta, "ms_per_round_feedback_and_learners": t_fb / rounds,
           "wall_s": time.time() - t_start}
    for name, L in learners.items():
        reg = (L["played"].double() - best)
        out[f"{name}_regret_mean"] = float(reg.mean())
        out[f"{name}_regret_max"] = float(reg.max())
        out[f"{name}_final_choice_is_expert_frac"] = float(
            (L["sel"].long().cpu() == (torch.arange(B) + (rounds - 1) // 250) % N).float().mean())
    out["best_fixed_drafter_loss_mean"] = float(best.mean())
    print(json.dumps(out), flush=True)


def main():
    args = parse_args()
    if args.session:
        run_session(args)
        return
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
