"""Benchmark of the WAMachine hot path on GB300.

One timed step = one closed-loop control step on the 12-block d=768 DiT (1296 joint tokens,
10 native Euler steps, batch 1): Trajectory Remapping of the finished replan (executed shift 8
of 16 actions), an anticipatory prefix of 1 step under the predicted observation, Observation
Rebinding against the real observation (Eq. 4), and the remaining 2 steps with Residual
Rescaling, ending in one action chunk.  The first replan of the episode is a cold 10-step
sample (warm-up).  Synthetic inputs: weights N(0, 0.02) seed 0; observations follow
o' = 0.9 o + sqrt(0.19) N(0,1) with the prediction 0.9 o; fresh noise seed 1000+step.

Printed JSON line: `value` = action chunks/s with every input already resident in HBM;
`latency_ms` = per-control-step p50/p99 and the observation-to-action part (rebinding + the
steps after it); `cold` = a native cold 10-step sample; `e2e` = the same control loop through
the C ABI with pinned host buffers (host<->device copies inside the timed region);
`roofline` = the dominant kernel class (tcgen05 GEMM) against the measured bf16 peak;
`ablation` = the same control steps with the layer stack launched kernel by kernel instead of
replayed from CUDA graphs; `independent` = the separate video / action models of independent
execution, their continuations overlapped on two streams and in sequence; `cpu_baseline` = the float64 CPU oracle on the host cores for one
control step.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
Multi-GPU (torchrun): one replica per rank, no collective on the data path (the work is
independent episodes); the timed region is bracketed by barriers and the slowest rank counts.
"""
from __future__ import annotations

import argparse
import json
import math
import multiprocessing as mp
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "action chunks/sec & p50 control-step latency at 1 GB300; tensor-pipe % of peak"
WORKLOAD = "closed_loop"


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(hbm=p["hbm_gbs"], bf16=p["bf16_tflops"], bf16_sus=p["bf16_tflops_sustained"],
                    source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


TENSOR_CLASSES = ("gemm", "attn")


def slowest_rank_ms(ms: float, dist) -> float:
    """The job's time: the largest of the ranks' timed-region durations (all ranks get it)."""
    if dist is None:
        return ms
    import torch
    t = torch.tensor([ms], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t[0])


def job_throughput(units_per_rank: int, world: int, ms: float) -> float:
    """Whole-job throughput: the units every rank processed over the slowest rank's time."""
    return units_per_rank * world / (ms * 1e-3)


def kernel_table(prof: dict, units: int, peaks: dict) -> dict:
    """Per kernel class: time per unit, share, and achieved rate against the measured peak
    (TFLOP/s for the tensor-core classes, GB/s of algorithmic bytes for the HBM-bound ones)."""
    tot = sum(v["ms"] for v in prof.values())
    out = {}
    for k, v in prof.items():
        if v["launches"] == 0:
            continue
        row = {"ms_per_unit": v["ms"] / units, "share": v["ms"] / tot if tot else 0.0, "launches": v["launches"]}
        if v["ms"] > 0:
            if k in TENSOR_CLASSES:
                row["tflops"] = v["flops"] / (v["ms"] * 1e-3) / 1e12
                row["frac"] = row["tflops"] / peaks["bf16_sus"]
            else:
                row["gbs"] = v["bytes"] / (v["ms"] * 1e-3) / 1e9
                row["frac"] = row["gbs"] / peaks["hbm"]
        out[k] = row
    return out


def _gemm_traffic():
    """DRAM bytes per GEMM launch from the committed ncu summary, if the kernel source is
    unchanged since those counters were taken (else None)."""
    import hashlib
    import re
    summ = os.path.join(ROOT, "profiles", "gemm_tc_closed_loop.md")
    src = os.path.join(ROOT, "paper_2609_34608_gb300", "csrc", "gemm_tc.cu")
    try:
        text = open(summ).read()
        tb = int(re.search(r"traffic_bytes_per_launch: (\d+)", text).group(1))
        sha = re.search(r"kernel_source_sha1_prefix: ([0-9a-f]+)", text).group(1)
        cur = hashlib.sha1(open(src, "rb").read()).hexdigest()
    except (OSError, AttributeError, ValueError):
        return None
    return tb if cur.startswith(sha) else None


def _workload_config(cfg: dict) -> dict:
    return {
        "workload": "closed-loop control step (TR shift 8 + 1 anticipatory step + OR + 2 steps with RR) "
                    "of the 12-block d768 12-head bf16 DiT, 256 obs + 1024 video + 16x7 action tokens, "
                    "10 native Euler steps, batch 1",
        "n_layers": cfg["n_layers"], "d_model": cfg["d_model"], "tokens": cfg["n_obs"] + cfg["n_video"] + cfg["n_action"],
        "batch": 1, "steps_native": cfg["n_steps"], "warm_steps": cfg["n_steps"] - cfg["tr_entry_stage"],
        "rr_boundaries": [cfg["rr_q"], cfg["rr_s"], cfg["rr_e"]],
        "l2": "inputs larger than L2: 255 MB of bf16 weights are streamed by every denoising step",
    }


# ------------------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.proc = None
        self.path = tempfile.mktemp(suffix=".csv")
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={gpu_index}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
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
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------------------ CPU oracle
def _oracle_control_step_worker(q, cfg, seed, n_steps):
    """Time the float64 oracle on one warm control step (a bounded sample of the workload)."""
    from oracle import wam_oracle as O
    from paper_2609_34608_gb300 import inputs as I

    Wd = I.make_weights(cfg)
    ocfg = O.OracleConfig.from_dict(cfg)
    K = cfg["n_steps"]
    b0 = cfg["tr_entry_stage"]
    ep = O.OracleEpisode(Wd, ocfg)
    proc = I.ObsProcess(cfg, 1, seed=seed)
    rng = np.random.default_rng(seed)
    T = ocfg.traj_len
    # a finished previous replan (its stage-K and stage-r latents) to remap from
    ep.obs = proc.obs[0].astype(np.float64)
    ep.hist = {K: rng.standard_normal(T), b0: rng.standard_normal(T)}
    ep.hist_from, ep.stage, ep.finished = b0, K, True
    times = []
    for t in range(n_steps):
        pred, real = proc.predicted()[0], proc.step()[0]
        eps = I.make_fresh_eps(cfg, 1, t)[0]
        t0 = time.perf_counter()
        if ep.adapt(pred, cfg["shift"], eps) == O.ADAPT_TR_INIT:
            ep.advance(cfg.get("prefix_steps", 1))
        ep.adapt(real, 0, None)
        ep.advance(K - ep.stage)
        times.append(time.perf_counter() - t0)
    q.put(times)


def run_oracle_steps(cfg, n_steps, seed=0):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    ncpu = os.cpu_count() or 1
    os.environ.setdefault("OPENBLAS_NUM_THREADS", str(ncpu))
    os.environ.setdefault("OMP_NUM_THREADS", str(ncpu))
    p = ctx.Process(target=_oracle_control_step_worker, args=(q, cfg, seed, n_steps))
    p.start()
    times = q.get()
    p.join()
    return times, int(os.environ["OPENBLAS_NUM_THREADS"])


# ------------------------------------------------------------------------------ reference arm
def main_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    from paper_2609_34608_gb300 import inputs as I

    cfg = I.get_config(WORKLOAD)
    times, cores = run_oracle_steps(cfg, args.warmup + args.steps)
    timed = times[args.warmup:]
    total = sum(timed)
    value = len(timed) / total
    sample = "one full warm control step per timed step (3 denoising forwards + TR + OR), float64 oracle"
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "chunks/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * total / len(timed),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": _workload_config(cfg),
        "cpu_baseline": {"value": value, "unit": "chunks/s", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "chunks/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ------------------------------------------------------------------------------ our arm
def main_ours(args):
    import torch

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("gloo")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    # The CPU baseline process is spawned before any GPU work.
    cpu_times, cpu_cores = (None, None)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        from paper_2609_34608_gb300 import inputs as I0
        cpu_times, cpu_cores = run_oracle_steps(I0.get_config(WORKLOAD), 2)

    from paper_2609_34608_gb300 import _build
    from paper_2609_34608_gb300 import inputs as I
    from paper_2609_34608_gb300 import wam as W

    _build.build()
    cfg = I.get_config(WORKLOAD)
    K, b0, shift = cfg["n_steps"], cfg["tr_entry_stage"], cfg["shift"]
    stream = torch.cuda.Stream(dev)
    flat = torch.from_numpy(I.flatten_weights(I.make_weights(cfg))).to(dev)
    ctx = W.Context(cfg, flat, stream=stream.cuda_stream)
    del flat
    n_total = args.warmup + args.steps
    proc = I.ObsProcess(cfg, 1, seed=rank)
    first_obs = proc.obs.copy()
    host = []
    for t in range(n_total + 1):
        pred = proc.predicted()
        real = proc.step()
        host.append((pred, real, I.make_fresh_eps(cfg, 1, t)))
    with torch.cuda.stream(stream):
        dev_in = [tuple(torch.from_numpy(a).to(dev) for a in h) for h in host]
        pin_in = [tuple(torch.from_numpy(a).pin_memory() for a in h) for h in host]
        act_dev = torch.zeros((1, cfg["n_action"], cfg["action_dim"]), device=dev)
        act_host = torch.zeros((1, cfg["n_action"], cfg["action_dim"])).pin_memory()
        noise = torch.from_numpy(I.make_noise(cfg, 1)).to(dev)
        obs0 = torch.from_numpy(first_obs).to(dev)

    def control_step(inp, act, ev=None):
        pred, real, eps = inp
        s1 = ctx.adapt(st, pred, shift=shift, fresh_noise=eps)[0]
        if s1 == W.ADAPT_TR_INIT:
            ctx.continue_(st, 1)
        if ev is not None:
            ev.record(stream)
        s2 = ctx.adapt(st, real)[0]
        ctx.continue_(st, K - (b0 + 1 if s2 == W.ADAPT_REBIND_ACCEPT else b0), act)
        return s1, s2

    def barrier():
        torch.cuda.synchronize(dev)
        if dist is not None:
            dist.barrier()

    # ---- device-resident inputs -------------------------------------------------------
    st = ctx.state(1)
    with torch.cuda.stream(stream):
        ctx.sample_cold(st, obs0, noise, K, act_dev)
        for t in range(args.warmup):
            control_step(dev_in[t], act_dev)
    ctx.reset_stats()
    ev_s = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    ev_m = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    clocks = ClockSampler(local)
    barrier()
    with torch.cuda.stream(stream):
        ev_s[0].record(stream)
        for i in range(args.steps):
            control_step(dev_in[args.warmup + i], act_dev, ev_m[i])
            ev_s[i + 1].record(stream)
    barrier()
    clk = clocks.stop()
    stats = ctx.stats()
    total_ms = ev_s[0].elapsed_time(ev_s[-1])
    step_ms = [ev_s[i].elapsed_time(ev_s[i + 1]) for i in range(args.steps)]
    o2a_ms = [ev_m[i].elapsed_time(ev_s[i + 1]) for i in range(args.steps)]
    total_ms = slowest_rank_ms(total_ms, dist)

    # ---- end to end: pinned host inputs and outputs through the C ABI -----------------
    st_e = ctx.state(1)
    with torch.cuda.stream(stream):
        ctx.sample_cold(st_e, obs0, noise, K, act_dev)
        st, st_keep = st_e, st
        for t in range(min(args.warmup, 3)):
            control_step(pin_in[t], act_host)
    barrier()
    e0 = time.perf_counter()
    ev_e0, ev_e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        ev_e0.record(stream)
        for i in range(args.steps):
            control_step(pin_in[args.warmup + i], act_host)
        ev_e1.record(stream)
    barrier()
    e2e_wall = time.perf_counter() - e0
    e2e_ms = slowest_rank_ms(ev_e0.elapsed_time(ev_e1), dist)
    st = st_keep
    h2d = sum(a.numel() * 4 for a in pin_in[0])
    d2h = act_host.numel() * 4

    # ---- native cold 10-step sample for comparison -----------------------------------
    st_c = ctx.state(1)
    cold_ms = []
    with torch.cuda.stream(stream):
        for i in range(max(3, min(10, args.steps))):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            ctx.sample_cold(st_c, obs0, noise, K, act_dev)
            b.record(stream)
            cold_ms.append((a, b))
    torch.cuda.synchronize(dev)
    cold_ms = [a.elapsed_time(b) for a, b in cold_ms][1:]

    # ---- ablation: the same control steps with every kernel launched individually ------
    # (CUDA-graph replay of the layer stack off; the paper's Table 3 "Graph" switch)
    st = st_keep
    n_abl = min(args.steps, 50)
    ctx.set_graph_replay(False)
    a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        a0.record(stream)
        for i in range(n_abl):
            control_step(dev_in[args.warmup + i], act_dev)
        a1.record(stream)
    torch.cuda.synchronize(dev)
    ctx.set_graph_replay(True)
    abl_ms = a0.elapsed_time(a1) / n_abl

    # ---- kernel-class timing (CUDA events on the library's stream) --------------------
    st = st_keep
    ctx.profile_enable(True)
    nprof = min(args.steps, 20)
    with torch.cuda.stream(stream):
        for i in range(nprof):
            control_step(dev_in[args.warmup + i], act_dev)
    prof = ctx.profile_read()
    ctx.profile_enable(False)

    serving = serving_rr = independent = None
    if not args.no_serving:
        ctx.close()
        serving = run_serving(dev, stream, _peaks())
        serving_rr = run_serving(dev, stream, _peaks(), relax_gate=True)
    if not args.no_independent:
        independent = run_independent(dev)

    if rank != 0:
        return 0
    peaks = _peaks()
    g = prof["gemm"]
    gemm_tflops = g["flops"] / (g["ms"] * 1e-3) / 1e12 if g["ms"] > 0 else 0.0
    value = job_throughput(args.steps, world, total_ms)
    line = {
        "metric": METRIC, "value": value, "unit": "chunks/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": _workload_config(cfg),
        "latency_ms": {"p50": float(np.percentile(step_ms, 50)), "p99": float(np.percentile(step_ms, 99)),
                       "o2a_p50": float(np.percentile(o2a_ms, 50)), "o2a_p99": float(np.percentile(o2a_ms, 99))},
        "cold": {"ms_p50": float(np.percentile(cold_ms, 50)), "chunks_per_s": 1000.0 / float(np.percentile(cold_ms, 50)),
                 "what": "native cold 10-step sample of the same model, RR active after the first step"},
        "ablation": {"graph_replay_off": {"chunks_per_s": 1000.0 / abl_ms, "ms_per_step": abl_ms, "steps": n_abl,
                                          "what": "same control steps, every kernel launched individually"}},
        "reuse": {"r_rr": stats["n_reuse"] / max(1, stats["n_attempt"]), "f_skip": stats["b_skip"] / max(1, stats["b_dense"]),
                  "r_or": stats["n_bind"] / max(1, stats["n_start"]), "coverage": stats["n_bind"] / max(1, stats["n_noninitial"])},
        "roofline": {"bound": "tensor", "kernel": "tcgen05 GEMM (QKV / out / MLP projections)",
                     "achieved": gemm_tflops, "peak": peaks["bf16_sus"], "unit": "TFLOP/s",
                     "frac": gemm_tflops / peaks["bf16_sus"], "traffic": _gemm_traffic(),
                     "algorithmic_bytes_per_launch": g["bytes"] / max(1, g["launches"]),
                     "peak_source": f"{peaks['source']} sustained bf16"},
        "kernels": kernel_table(prof, nprof, peaks),
        "gpu_launches": int(stats["n_kernel_launches"]),
        "e2e": {"value": job_throughput(args.steps, world, e2e_ms), "unit": "chunks/s", "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(d2h), "wall_s": e2e_wall},
        "clocks": clk,
    }
    if serving is not None:
        line["serving"] = serving
        line["serving_rr_accept"] = serving_rr
    if independent is not None:
        line["independent"] = independent
    if cpu_times:
        ct = cpu_times[-1]
        line["cpu_baseline"] = {"value": 1.0 / ct, "unit": "chunks/s", "cores": cpu_cores, "kind": "oracle",
                                "sample": "one warm control step (TR + 1 prefix step + OR + 2 steps, RR), float64 "
                                          "oracle; best-effort second of two runs"}
    print(json.dumps(line))
    return 0


def run_serving(dev, stream, peaks, warm_batches=2, batches=3, relax_gate=False):
    """Batched serving: 32 independent episodes per batch on the 24-block d1024 DiT (2464 tokens);
    each batch mixes 16 fresh episodes (cold, 10 steps) and 16 warm continuations (TR shift 16,
    2 of 10 steps), run as one state so every step batches the active episodes.  With
    `relax_gate` the RR thresholds let every check pass (the injection path and the layer skip
    at scale; not the acceptance rate of any trained model)."""
    import torch

    from paper_2609_34608_gb300 import inputs as I
    from paper_2609_34608_gb300 import wam as W

    over = dict(rr_gamma_cos=-1.0, rr_gamma_fit=1e30) if relax_gate else {}
    cfg = I.get_config("serving", **over)
    B, K = cfg["batch"], cfg["n_steps"]
    flat = torch.from_numpy(I.flatten_weights(I.make_weights(cfg))).to(dev)
    ctx = W.Context(cfg, flat, stream=stream.cuda_stream)
    del flat
    half = B // 2
    entry = np.array([W.ENTRY_COLD] * half + [K - 2] * half, np.int32)
    shift = np.array([0] * half + [16] * half, np.int32)
    n_steps = np.array([K] * half + [2] * half, np.int32)
    with torch.cuda.stream(stream):
        obs = [torch.from_numpy(I.make_obs(cfg, B, seed=100 + i)).to(dev) for i in range(warm_batches + batches + 1)]
        eps = [torch.from_numpy(I.make_fresh_eps(cfg, B, i)).to(dev) for i in range(warm_batches + batches + 1)]
        act = torch.zeros((B, cfg["n_action"], cfg["action_dim"]), device=dev)
        st = ctx.state(B)
        ctx.sample_cold(st, obs[0], eps[0], K, act)

    def batch(i):
        ctx.adapt(st, obs[i], shift=shift, entry=entry, fresh_noise=eps[i])
        ctx.continue_(st, n_steps, act)

    with torch.cuda.stream(stream):
        for i in range(warm_batches):
            batch(1 + i)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for i in range(batches):
            batch(1 + warm_batches + i)
        e1.record(stream)
    torch.cuda.synchronize(dev)
    ms = e0.elapsed_time(e1) / batches
    ctx.reset_stats()
    ctx.profile_enable(True)
    with torch.cuda.stream(stream):
        batch(1)
    prof = ctx.profile_read()
    stats = ctx.stats()
    ctx.close()
    kt = kernel_table(prof, 1, peaks)
    res = {
        "workload": "24-block d1024 16-head bf16 DiT, 384 obs + 2048 video + 32x7 action tokens; batch of 32 "
                    "episodes: 16 cold (10 steps) + 16 warm (TR shift 16, 2 of 10 steps) per batch",
        "chunks_per_s": B / (ms * 1e-3), "ms_per_batch": ms, "batches": batches,
        "gemm_tflops": kt["gemm"]["tflops"], "attn_tflops": kt["attn"]["tflops"],
        "gemm_frac": kt["gemm"]["frac"], "attn_frac": kt["attn"]["frac"],
        "kernels_per_batch": kt,
        "reuse": {"r_rr": stats["n_reuse"] / max(1, stats["n_attempt"]),
                  "f_skip": stats["b_skip"] / max(1, stats["b_dense"])},
    }
    if relax_gate:
        res["workload"] += "; RR gate thresholds relaxed so every check passes"
    return res


def run_independent(dev, n_steps=50, warmup=5):
    """Independent execution (§3.3; the Fast-WAM-IDM profile of App. B.1): a video-only and an
    action-only 12-block d768 model, each with its own replan state, on its own stream.  One
    control step: the video branch remaps stage 5 to entry 4 (shifted schedule) and runs its
    2-step anticipatory prefix under the predicted observation; when the real observation
    arrives the video branch rebinds and finishes its 4 steps while the action branch remaps
    with the executed shift 8, enters stage 5 and runs 5 steps.  Timed twice: the two
    continuations through wam_continue_many (one host thread per context, overlapping on the
    GPU; the action stream has the higher priority), as two wam_continue calls in sequence, and
    in sequence with the action branch first (the shortest observation-to-action time).
    O2A = real observation to action chunk (for the concurrent call, when it returns: an upper
    bound, since the call returns once both branches are issued)."""
    import torch

    from paper_2609_34608_gb300 import inputs as I
    from paper_2609_34608_gb300 import wam as W

    cv, ca = I.get_config("idm_video"), I.get_config("idm_action")
    K = cv["n_steps"]
    # the action branch produces the chunk the robot waits for: its stream gets the higher
    # priority, so its blocks are scheduled first whenever both branches have work queued
    sv, sa = torch.cuda.Stream(dev), torch.cuda.Stream(dev, priority=-1)
    ctxs = []
    for cfg, s in ((cv, sv), (ca, sa)):
        flat = torch.from_numpy(I.flatten_weights(I.make_weights(cfg))).to(dev)
        ctxs.append(W.Context(cfg, flat, stream=s.cuda_stream))
        del flat
    vctx, actx = ctxs
    total = 3 * (warmup + n_steps) + 1
    proc = I.ObsProcess(cv, 1, seed=5)
    with torch.cuda.stream(sv):
        obs0 = torch.from_numpy(proc.obs.copy()).to(dev)
        inputs = []
        for t in range(total):
            pred, real = proc.predicted(), proc.step()
            inputs.append((torch.from_numpy(pred).to(dev), torch.from_numpy(real).to(dev),
                           torch.from_numpy(I.make_fresh_eps(cv, 1, t)).to(dev),
                           torch.from_numpy(I.make_fresh_eps(ca, 1, 500 + t)).to(dev)))
        vout = torch.zeros((1, cv["n_video"], cv["video_dim"]), device=dev)
        aout = torch.zeros((1, ca["n_action"], ca["action_dim"]), device=dev)
        vst, ast = vctx.state(1), actx.state(1)
        vctx.sample_cold(vst, obs0, torch.from_numpy(I.make_noise(cv, 1)).to(dev), K)
    with torch.cuda.stream(sa):
        actx.sample_cold(ast, obs0, torch.from_numpy(I.make_noise(ca, 1, seed=2)).to(dev), K)
    torch.cuda.synchronize(dev)
    b0v, pv = cv["tr_entry_stage"], cv["prefix_steps"]
    ev = lambda: torch.cuda.Event(enable_timing=True)

    def control_step(inp, mode, marks=None):
        pred, real, eps_v, eps_a = inp
        if marks is not None:
            marks[0].record(sv)
            sa.wait_event(marks[0])
        s1 = vctx.adapt(vst, pred, shift=0, fresh_noise=eps_v)[0]
        if s1 == W.ADAPT_TR_INIT:
            vctx.continue_(vst, pv)
        if marks is not None:
            marks[1].record(sv)          # the real observation arrives
            sa.wait_event(marks[1])
        actx.adapt(ast, real, shift=ca["shift"], fresh_noise=eps_a)
        s2 = vctx.adapt(vst, real)[0]
        kv = b0v + pv if s2 == W.ADAPT_REBIND_ACCEPT else b0v
        calls = [(vctx, vst, K - kv, None, vout), (actx, ast, K - ca["tr_entry_stage"], aout, None)]
        if mode == "concurrent":
            W.Context.continue_many(calls)
            if marks is not None:
                marks[2].record(sa)      # action chunk ready (recorded once the concurrent call returns)
        else:
            for c in (calls if mode == "sequential" else calls[::-1]):
                c[0].continue_(c[1], c[2], c[3], c[4])
                if marks is not None and c[0] is actx:
                    marks[2].record(sa)  # action chunk ready, before the other branch is issued
        if marks is not None:
            sv.wait_event(marks[2])
            marks[3].record(sv)          # both branches done

    res = {}
    t = 0
    for mode in ("concurrent", "sequential", "action_first"):
        for _ in range(warmup):
            control_step(inputs[t], mode)
            t += 1
        vctx.reset_stats()
        actx.reset_stats()
        torch.cuda.synchronize(dev)
        marks = [[ev() for _ in range(4)] for _ in range(n_steps)]
        for i in range(n_steps):
            control_step(inputs[t], mode, marks[i])
            t += 1
        torch.cuda.synchronize(dev)
        total_ms = marks[0][0].elapsed_time(marks[-1][3])
        step_ms = [m[0].elapsed_time(m[3]) for m in marks]
        o2a_ms = [m[1].elapsed_time(m[2]) for m in marks]
        res[mode] = {"chunks_per_s": n_steps / (total_ms * 1e-3), "ms_per_step": total_ms / n_steps,
                    "step_ms_p50": float(np.percentile(step_ms, 50)),
                    "o2a_ms_p50": float(np.percentile(o2a_ms, 50)),
                    "o2a_ms_p99": float(np.percentile(o2a_ms, 99))}
        if mode == "concurrent":
            for name, c in (("video", vctx), ("action", actx)):
                st = c.stats()
                res.setdefault("reuse", {})[name] = {
                    "r_rr": st["n_reuse"] / max(1, st["n_attempt"]), "f_skip": st["b_skip"] / max(1, st["b_dense"]),
                    "r_or": st["n_bind"] / max(1, st["n_start"])}
    vctx.close()
    actx.close()
    res["workload"] = ("independent execution (Fast-WAM-IDM profile): video-only 12-block d768 model "
                       "(256 obs + 1024 video tokens, shifted schedule s=5, stage 5 -> entry 4, 2+4 steps) and "
                       "action-only 12-block d768 model (256 obs + 16x7 action tokens, shift 8, entry 5, 5 steps), "
                       "batch 1, RR gates cos >= 0.80, fit <= 0.60; each on its own stream")
    res["steps"] = n_steps
    return res


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-serving", action="store_true", help="skip the batched serving section")
    ap.add_argument("--no-independent", action="store_true", help="skip the independent-execution section")
    args = ap.parse_args()
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")
    if args.impl == "reference":
        return main_reference(args)
    return main_ours(args)


if __name__ == "__main__":
    sys.exit(main())
