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
`roofline` = the dominant kernel class (tcgen05 GEMM) against the measured burst bf16 peak,
its time taken as its share of a profiled pass applied to the un-instrumented step;
`kernels` = every kernel class of the profiled pass; `ablation` = the paper's Table 3 variants
(w/o TR, w/o OR, w/o RR, w/o graph replay, native with and without graphs) and a labelled run
with a relaxed RR gate; `seeds` = the closed-loop rollout over seeds 0..3 (its own observation
process per seed), each seed's warm control steps against cold 10-step samples under the same
observations; `async_prefix` = the anticipatory prefix on a second stream during a modelled
action-execution window (O2A and GPU time per replan); `serving` = 32-episode batches of the 24-block d1024 model;
`bimanual` = the 28-block d1152 model (head dim 72, 4914 tokens, batch 8): cold 10 steps and
the warm sweep over 1..9 retained steps with shift 25; `independent` = the separate video /
action models of independent execution, their continuations overlapped on two streams and in
sequence; `cpu_baseline` = the float64 CPU oracle on the host cores continuing the GPU run's
cold sample (all cores; one core extrapolated from one forward).  `--cpu-plan` times the whole
CPU plan (latency cold sample end to end, serving / bimanual sample-steps) and exits.

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


def kernel_table(prof: dict, units: int, peaks: dict, tensor_peak: str = "bf16", step_ms: float | None = None) -> dict:
    """Per kernel class: time per unit, share, and achieved rate against the measured peak
    (TFLOP/s for the tensor-core classes, GB/s of algorithmic bytes for the HBM-bound ones).
    `tensor_peak` is "bf16" (burst: a step of a few ms) or "bf16_sus" (seconds-long runs).
    The profiled pass brackets every launch with CUDA events, which serialises launches that
    would otherwise overlap their prologues, so its spans add up to more than an un-instrumented
    unit; with `step_ms` (the un-instrumented time per unit) each class also gets its share of
    that time (`ms_in_step`, which sum to step_ms) and the rate over it (`*_in_step`)."""
    tot = sum(v["ms"] for v in prof.values())
    out = {}
    for k, v in prof.items():
        if v["launches"] == 0:
            continue
        row = {"ms_per_unit": v["ms"] / units, "share": v["ms"] / tot if tot else 0.0, "launches": v["launches"]}
        spans = [("", v["ms"] / units)]
        if step_ms is not None:
            row["ms_in_step"] = row["share"] * step_ms
            spans.append(("_in_step", row["ms_in_step"]))
        for suffix, ms in spans:
            if ms <= 0:
                continue
            if k in TENSOR_CLASSES:
                row["tflops" + suffix] = v["flops"] / units / (ms * 1e-3) / 1e12
                row["frac" + suffix] = row["tflops" + suffix] / peaks[tensor_peak]
            else:
                row["gbs" + suffix] = v["bytes"] / units / (ms * 1e-3) / 1e9
                row["frac" + suffix] = row["gbs" + suffix] / peaks["hbm"]
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

    def __init__(self, gpu_index: int, interval_ms: int = 25):
        """nvidia-smi polling every interval_ms; the timed region of a control-step run lasts tens of
        milliseconds, so the interval is short and start() waits for the first sample."""
        self.proc = None
        self.path = tempfile.mktemp(suffix=".csv")
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={gpu_index}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", str(interval_ms)], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def wait_first_sample(self, timeout_s: float = 5.0) -> bool:
        """Block until nvidia-smi has written its first sample (it takes a while to start)."""
        if self.proc is None:
            return False
        t0 = time.time()
        while time.time() - t0 < timeout_s:
            try:
                if os.path.getsize(self.path) > 0:
                    return True
            except OSError:
                pass
            if self.proc.poll() is not None:
                return False
            time.sleep(0.005)
        return False

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
def _oracle_episode_from(cfg, retained):
    """An oracle episode holding a finished replan: `retained` = dict of the stage latents
    ("hist": {stage: x}), the bound observation and the RR layer state (p_a, R_a), taken from a
    real cold sample; None draws a random finished replan (the reference arm's own stand-in)."""
    from oracle import wam_oracle as O
    from paper_2609_34608_gb300 import inputs as I

    Wd = I.make_weights(cfg)
    ocfg = O.OracleConfig.from_dict(cfg)
    K = cfg["n_steps"]
    ep = O.OracleEpisode(Wd, ocfg)
    if retained is None:
        rng = np.random.default_rng(0)
        T = ocfg.traj_len
        b0 = cfg["tr_entry_stage"]
        ep.hist = {K: rng.standard_normal(T), b0: rng.standard_normal(T)}
        ep.hist_from = b0
    else:
        ep.hist = {int(k): np.asarray(v, np.float64) for k, v in retained["hist"].items()}
        ep.hist_from = 0
        if retained.get("p_a") is not None:
            ep.layer = O.LayerState(p_a=np.asarray(retained["p_a"], np.float64),
                                    R_a=np.asarray(retained["R_a"], np.float64))
    ep.obs = np.asarray(retained["obs"] if retained is not None else np.zeros((cfg["n_obs"], cfg["d_model"])),
                        np.float64)
    ep.stage, ep.finished = K, True
    ep.x = ep.hist[K].copy()
    return ep


def _oracle_control_step_worker(q, cfg, seed, n_steps, retained):
    """Time the float64 oracle on warm control steps (a bounded sample of the workload)."""
    from oracle import wam_oracle as O
    from paper_2609_34608_gb300 import inputs as I

    ep = _oracle_episode_from(cfg, retained)
    K = cfg["n_steps"]
    proc = I.ObsProcess(cfg, 1, seed=seed)
    if retained is not None:
        proc.obs = np.asarray(retained["obs"], np.float32)[None]
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


def _oracle_forward_worker(q, cfg, n):
    """Time n float64 oracle denoising forwards (one sample-step each) of one episode."""
    from oracle import wam_oracle as O
    from paper_2609_34608_gb300 import inputs as I

    Wd = I.make_weights(cfg)
    ocfg = O.OracleConfig.from_dict(cfg)
    x, obs = I.make_noise(cfg, 1)[0], I.make_obs(cfg, 1)[0]
    times = []
    for _ in range(n):
        t0 = time.perf_counter()
        O.velocity(Wd, ocfg, x, obs, 0.5)
        times.append(time.perf_counter() - t0)
    q.put(times)


def _oracle_tiny_e2e_worker(q, cfg):
    """The tiny workload end to end: cold K-step sample, TR with the executed shift, warm
    continuation of the retained steps."""
    from oracle import wam_oracle as O
    from paper_2609_34608_gb300 import inputs as I

    Wd = I.make_weights(cfg)
    ocfg = O.OracleConfig.from_dict(cfg)
    K = cfg["n_steps"]
    t0 = time.perf_counter()
    ep = O.OracleEpisode(Wd, ocfg)
    ep.sample_cold(I.make_obs(cfg, 1)[0], I.make_noise(cfg, 1)[0], K)
    ep.adapt(I.make_obs(cfg, 1, seed=3)[0], cfg["shift"], I.make_fresh_eps(cfg, 1, 0)[0])
    ep.advance(K - ep.stage)
    q.put([time.perf_counter() - t0])


def _spawn(target, args, threads):
    """Run an oracle timing in a fresh (spawned) process with `threads` BLAS threads."""
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    keys = ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS")
    saved = {k: os.environ.get(k) for k in keys}
    for k in keys:
        os.environ[k] = str(threads)
    try:
        p = ctx.Process(target=target, args=(q,) + tuple(args))
        p.start()
        out = q.get()
        p.join()
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    return out


def run_oracle_steps(cfg, n_steps, seed=0, retained=None, threads=None):
    threads = threads or (os.cpu_count() or 1)
    return _spawn(_oracle_control_step_worker, (cfg, seed, n_steps, retained), threads), threads


def cpu_baseline(retained):
    """The oracle on the host cores, bounded to about a minute: two warm control steps of the
    benchmarked workload continuing a real cold sample (all cores), one denoising forward of
    that model on one core (a control step runs three), and the tiny workload end to end on
    all cores and on one core."""
    from paper_2609_34608_gb300 import inputs as I

    ncpu = os.cpu_count() or 1
    cfg = I.get_config(WORKLOAD)
    steps, _ = run_oracle_steps(cfg, 2, retained=retained, threads=ncpu)
    fwd1 = _spawn(_oracle_forward_worker, (cfg, 1), 1)
    tiny = I.get_config("tiny")
    t_all = _spawn(_oracle_tiny_e2e_worker, (tiny,), ncpu)
    t_one = _spawn(_oracle_tiny_e2e_worker, (tiny,), 1)
    per_step = statistics.mean(steps)
    return {
        "value": 1.0 / per_step, "unit": "chunks/s", "cores": ncpu, "kind": "oracle",
        "sample": "two warm control steps (TR + 1 prefix step + OR + 2 steps, RR) continuing the GPU run's "
                  "cold sample (its retained latents and layer state), float64 oracle, mean of the two",
        "step_s": steps,
        "one_core": {"forward_s": fwd1[0], "chunks_per_s_extrapolated": 1.0 / (3.0 * fwd1[0]),
                     "what": "one denoising forward of the same model on one core; a control step runs "
                             "three (TR and OR are below 1 % of it), so chunks/s is extrapolated"},
        "tiny_e2e_s": {"cores_all": t_all[0], "cores_1": t_one[0],
                       "what": "2-block d128 fp32 model: cold 8-step sample + TR (shift 1) + 4 warm steps"},
    }


def cpu_plan():
    """The full CPU plan (a few minutes on 16 cores): the tiny workload end to end and the latency
    model's cold 10-step sample end to end on all cores, one forward of the latency model on one
    core, and one sample-step of the serving and bimanual models on all cores, extrapolated to
    their batches (their one-core figures scale the all-core ones by the latency model's
    one-core / all-core ratio)."""
    from paper_2609_34608_gb300 import inputs as I

    ncpu = os.cpu_count() or 1
    out = {"cores": ncpu}
    tiny = I.get_config("tiny")
    out["tiny_e2e_s"] = {"all": _spawn(_oracle_tiny_e2e_worker, (tiny,), ncpu)[0],
                         "one": _spawn(_oracle_tiny_e2e_worker, (tiny,), 1)[0]}
    lat = I.get_config("latency")
    f_all = _spawn(_oracle_forward_worker, (lat, lat["n_steps"]), ncpu)
    f_one = _spawn(_oracle_forward_worker, (lat, 1), 1)
    out["latency_cold10"] = {"all_s": sum(f_all), "one_s_extrapolated": 10 * f_one[0],
                             "chunks_per_s_all": 1.0 / sum(f_all)}
    ratio = f_one[0] / (sum(f_all) / len(f_all))
    out["latency_cold10"]["one_core_over_all_cores"] = ratio
    for name in ("serving", "bimanual"):
        cfg = I.get_config(name)
        fa = _spawn(_oracle_forward_worker, (cfg, 1), ncpu)[0]
        fo = fa * ratio
        B, K = cfg["batch"], cfg["n_steps"]
        steps = B // 2 * K + B // 2 * 2 if name == "serving" else B * K
        out[name] = {"sample_step_s_all": fa, "sample_step_s_one_extrapolated": fo, "sample_steps_per_batch": steps,
                     "chunks_per_s_all_extrapolated": B / (steps * fa),
                     "chunks_per_s_one_extrapolated": B / (steps * fo)}
    return out


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

    from paper_2609_34608_gb300 import _build
    from paper_2609_34608_gb300 import inputs as I
    from paper_2609_34608_gb300 import wam as W

    _build.build()
    cfg = I.get_config(WORKLOAD)
    K, b0, shift = cfg["n_steps"], cfg["tr_entry_stage"], cfg["shift"]
    stream = torch.cuda.Stream(dev)
    flat = torch.from_numpy(I.flatten_weights(I.make_weights(cfg))).to(dev)
    ctx = W.Context(cfg, flat, stream=stream.cuda_stream)
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

    def control_step(inp, act, ev=None, c=None, s=None):
        c = c or ctx
        s = s or st
        pred, real, eps = inp
        s1 = c.adapt(s, pred, shift=shift, fresh_noise=eps)[0]
        if s1 == W.ADAPT_TR_INIT:
            c.continue_(s, cfg["prefix_steps"])
        if ev is not None:
            ev.record(stream)
        s2 = c.adapt(s, real)[0]
        c.continue_(s, K - (b0 + cfg["prefix_steps"] if s2 == W.ADAPT_REBIND_ACCEPT else b0), act)
        return s1, s2

    def barrier():
        torch.cuda.synchronize(dev)
        if dist is not None:
            dist.barrier()

    # ---- device-resident inputs -------------------------------------------------------
    st = ctx.state(1)
    with torch.cuda.stream(stream):
        ctx.sample_cold(st, obs0, noise, K, act_dev)
    torch.cuda.synchronize(dev)
    # the finished cold replan, kept for the CPU oracle baseline to continue from
    retained = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        retained = {"hist": {k: ctx.read(st, W.FIELD_X_STAGE, k)[0] for k in range(K + 1)},
                    "obs": first_obs[0], "p_a": ctx.read(st, W.FIELD_RR_P)[0], "R_a": ctx.read(st, W.FIELD_RR_R)[0]}
    with torch.cuda.stream(stream):
        for t in range(args.warmup):
            control_step(dev_in[t], act_dev)
    ctx.reset_stats()
    ev_s = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    ev_m = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    clocks = ClockSampler(local)
    clocks.wait_first_sample()
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
    rr_log = ctx.log(st)

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

    # ---- kernel-class timing (CUDA events on the library's stream) --------------------
    ctx.profile_enable(True)
    nprof = min(args.steps, 20)
    with torch.cuda.stream(stream):
        for i in range(nprof):
            control_step(dev_in[args.warmup + i], act_dev)
    prof = ctx.profile_read()
    ctx.profile_enable(False)

    # ---- Table 3 ablation of the mechanisms and the graph replay ----------------------
    ablation = None
    if not args.no_ablation:
        ablation = run_table3(ctx, flat, cfg, dev, stream, dev_in, obs0, noise, min(args.steps, 20))
    seeds = None
    if not args.no_seeds:
        seeds = run_seeds(ctx, cfg, dev, stream, min(args.steps, 200))
    async_prefix = None
    if not args.no_async:
        async_prefix = run_async_prefix(ctx, cfg, dev, stream, dev_in, obs0, noise, n=min(args.steps, 20))
    del flat

    serving = serving_rr = independent = bimanual = None
    if not args.no_serving:
        ctx.close()
        serving = run_serving(dev, stream, _peaks())
        serving_rr = run_serving(dev, stream, _peaks(), relax_gate=True)
    if not args.no_bimanual:
        ctx.close()
        bimanual = run_bimanual(dev, stream, _peaks())
    if not args.no_independent:
        independent = run_independent(dev)

    if rank != 0:
        return 0
    peaks = _peaks()
    kt = kernel_table(prof, nprof, peaks, step_ms=total_ms / args.steps)
    g = prof["gemm"]
    # The per-launch events of the profiled pass stretch every kernel (they serialise the
    # launches); the GEMM class's rate is taken from its share of that pass applied to the
    # un-instrumented step time.
    gemm_flops_step = g["flops"] / nprof
    gemm_ms_step = kt["gemm"]["ms_in_step"]
    gemm_tflops = kt["gemm"]["tflops_in_step"]
    value = job_throughput(args.steps, world, total_ms)
    accepted = [r for r in rr_log if r["rr_attempt"]]
    line = {
        "metric": METRIC, "value": value, "unit": "chunks/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": _workload_config(cfg),
        "latency_ms": {"p50": float(np.percentile(step_ms, 50)), "p99": float(np.percentile(step_ms, 99)),
                       "o2a_p50": float(np.percentile(o2a_ms, 50)), "o2a_p99": float(np.percentile(o2a_ms, 99))},
        "cold": {"ms_p50": float(np.percentile(cold_ms, 50)), "chunks_per_s": 1000.0 / float(np.percentile(cold_ms, 50)),
                 "what": "native cold 10-step sample of the same model, RR active after the first step"},
        "reuse": {"r_rr": stats["n_reuse"] / max(1, stats["n_attempt"]), "f_skip": stats["b_skip"] / max(1, stats["b_dense"]),
                  "r_or": stats["n_bind"] / max(1, stats["n_start"]), "coverage": stats["n_bind"] / max(1, stats["n_noninitial"]),
                  "rr_cos_last_step": [r["cos"] for r in accepted[-1:]],
                  "rr_fit_last_step": [r["fit"] for r in accepted[-1:]]},
        "roofline": {"bound": "tensor", "kernel": "tcgen05 GEMM (QKV / out / MLP projections)",
                     "achieved": gemm_tflops, "peak": peaks["bf16"], "unit": "TFLOP/s",
                     "frac": gemm_tflops / peaks["bf16"], "traffic": _gemm_traffic(),
                     "algorithmic_bytes_per_launch": g["bytes"] / max(1, g["launches"]),
                     "gemm_flops_per_step": gemm_flops_step, "gemm_ms_per_step": gemm_ms_step,
                     "method": "GEMM FLOPs of a control step / (GEMM share of the profiled pass x the timed step time)",
                     "event_timed_tflops": kt["gemm"]["tflops"],
                     "peak_source": f"{peaks['source']} burst bf16 (the timed unit is a step of a few ms)"},
        "kernels": kt,
        "gpu_launches": int(stats["n_kernel_launches"]),
        "e2e": {"value": job_throughput(args.steps, world, e2e_ms), "unit": "chunks/s", "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(d2h), "wall_s": e2e_wall},
        "clocks": clk,
    }
    if ablation is not None:
        line["ablation"] = ablation
    if seeds is not None:
        line["seeds"] = seeds
    if async_prefix is not None:
        line["async_prefix"] = async_prefix
    if serving is not None:
        line["serving"] = serving
        line["serving_rr_accept"] = serving_rr
    if bimanual is not None:
        line["bimanual"] = bimanual
    if independent is not None:
        line["independent"] = independent
    if retained is not None:
        line["cpu_baseline"] = cpu_baseline(retained)
    print(json.dumps(line))
    return 0


def run_table3(ctx, flat, cfg, dev, stream, dev_in, obs0, noise, n, warm=3):
    """The mechanisms of the paper's ablation (Table 3, App. C) on the benchmarked workload,
    each timed over n control steps: GPU ms per replan (all denoising work of the replan) and
    O2A ms (real observation to action chunk; App. A).
      full       TR + OR (1 anticipatory step) + RR, layer stack replayed from CUDA graphs
      wo_tr      every replan from fresh noise: 8 anticipatory steps under the prediction (the
                 same rebinding stage), OR, 2 steps under the real observation
      wo_or      TR, then all 3 retained steps under the real observation (no prefix)
      wo_rr      TR + OR, every step runs all layers
      wo_graph   TR + OR + RR, every kernel launched individually (RR decided on the host)
      native / native_graph   cold 10-step sample under the real observation, all layers
      host_branching   full, with the RR decision read back to the host every step instead of
                 taken on the device inside the step's graph
    plus `rr_relaxed`: the full variant with RR thresholds that let every check pass (on random
    weights the d768 model's consecutive probe residuals have cosine ~0.7, below every Table 7
    threshold, so this is the only way to time the reuse path here; not a trained model's rate)."""
    import torch

    from paper_2609_34608_gb300 import inputs as I
    from paper_2609_34608_gb300 import wam as W

    K, b0, shift, pre = cfg["n_steps"], cfg["tr_entry_stage"], cfg["shift"], cfg["prefix_steps"]
    ctx_norr = W.Context(dict(cfg, rr_policy=0), flat, stream=stream.cuda_stream)
    ctx_relax = W.Context(dict(cfg, rr_gamma_cos=-1.0, rr_gamma_fit=1e30), flat, stream=stream.cuda_stream)
    act = torch.zeros((1, cfg["n_action"], cfg["action_dim"]), device=dev)

    def step_full(c, s, inp, mark):
        pred, real, eps = inp
        if c.adapt(s, pred, shift=shift, fresh_noise=eps)[0] == W.ADAPT_TR_INIT:
            c.continue_(s, pre)
        mark.record(stream)
        s2 = c.adapt(s, real)[0]
        c.continue_(s, K - (b0 + pre if s2 == W.ADAPT_REBIND_ACCEPT else b0), act)

    def step_wo_tr(c, s, inp, mark):
        pred, real, eps = inp
        c.adapt(s, pred, entry=W.ENTRY_COLD, fresh_noise=eps)
        c.continue_(s, b0 + pre)
        mark.record(stream)
        s2 = c.adapt(s, real)[0]
        c.continue_(s, K - (b0 + pre if s2 == W.ADAPT_REBIND_ACCEPT else 0), act)

    def step_wo_or(c, s, inp, mark):
        pred, real, eps = inp
        mark.record(stream)
        c.adapt(s, real, shift=shift, fresh_noise=eps)
        c.continue_(s, K - b0, act)

    def step_native(c, s, inp, mark):
        pred, real, eps = inp
        mark.record(stream)
        c.sample_cold(s, real, eps, K, act)

    variants = [("full", ctx, True, step_full), ("wo_tr", ctx, True, step_wo_tr), ("wo_or", ctx, True, step_wo_or),
                ("wo_rr", ctx_norr, True, step_full), ("wo_graph", ctx, False, step_full),
                ("native_graph", ctx_norr, True, step_native), ("native", ctx_norr, False, step_native),
                ("rr_relaxed", ctx_relax, True, step_full), ("host_branching", ctx, True, step_full),
                ("rr_relaxed_host_branching", ctx_relax, True, step_full)]
    ev = lambda: torch.cuda.Event(enable_timing=True)
    out = {}
    for name, c, graphs, fn in variants:
        c.set_graph_replay(graphs)
        c.set_device_branching(not name.endswith("host_branching"))
        s = c.state(1)
        with torch.cuda.stream(stream):
            c.sample_cold(s, obs0, noise, K)
            for t in range(warm):
                fn(c, s, dev_in[t % len(dev_in)], ev())
        c.reset_stats()
        torch.cuda.synchronize(dev)
        marks = [(ev(), ev(), ev()) for _ in range(n)]
        with torch.cuda.stream(stream):
            for i in range(n):
                marks[i][0].record(stream)
                fn(c, s, dev_in[(warm + i) % len(dev_in)], marks[i][1])
                marks[i][2].record(stream)
        torch.cuda.synchronize(dev)
        gpu = [m[0].elapsed_time(m[2]) for m in marks]
        o2a = [m[1].elapsed_time(m[2]) for m in marks]
        stt = c.stats()
        out[name] = {"gpu_ms_per_replan": statistics.mean(gpu), "o2a_ms": statistics.mean(o2a),
                     "o2a_ms_p50": float(np.percentile(o2a, 50)), "chunks_per_s": 1000.0 / statistics.mean(gpu),
                     "r_rr": stt["n_reuse"] / max(1, stt["n_attempt"]),
                     "f_skip": stt["b_skip"] / max(1, stt["b_dense"]),
                     "r_or": stt["n_bind"] / max(1, stt["n_start"])}
        s.close()
        c.set_graph_replay(True)
        c.set_device_branching(True)
    ctx_norr.close()
    ctx_relax.close()
    out["steps"] = n
    out["what"] = ("Table 3 variants on the closed-loop workload (GPU = mean ms of one replan's work, O2A = real "
                   "observation to action chunk, both on the device clock); rr_relaxed = full with RR thresholds "
                   "that accept every check (labelled: random weights, not a trained model's acceptance)")
    return out


def run_seeds(ctx, cfg, dev, stream, n, seeds=(0, 1, 2, 3), warm=3):
    """The closed-loop rollout over several seeds: per seed, its own observation process
    (o' = 0.9 o + sqrt(0.19) N(0,1), prediction 0.9 o), initial noise and fresh-noise draws, one
    cold replan, then n control steps (TR shift, 1 anticipatory step, OR, the remaining steps with
    RR), each timed on the device; beside it the cold 10-step sample under the same real
    observations, so every seed reports warm versus cold."""
    import torch

    from paper_2609_34608_gb300 import inputs as I
    from paper_2609_34608_gb300 import wam as W

    K, b0, shift, pre = cfg["n_steps"], cfg["tr_entry_stage"], cfg["shift"], cfg["prefix_steps"]
    act = torch.zeros((1, cfg["n_action"], cfg["action_dim"]), device=dev)
    ev = lambda: torch.cuda.Event(enable_timing=True)
    out = {}
    for seed in seeds:
        proc = I.ObsProcess(cfg, 1, seed=seed)
        with torch.cuda.stream(stream):
            obs0 = torch.from_numpy(proc.obs.copy()).to(dev)
            noise = torch.from_numpy(I.make_noise(cfg, 1, seed=1 + seed)).to(dev)
            inp = []
            for t in range(warm + n):
                pred = proc.predicted()
                real = proc.step()
                eps = I.make_fresh_eps(cfg, 1, 100000 * seed + t)
                inp.append(tuple(torch.from_numpy(a).to(dev) for a in (pred, real, eps)))
        st, st_c = ctx.state(1), ctx.state(1)
        with torch.cuda.stream(stream):
            ctx.sample_cold(st, obs0, noise, K, act)
            for t in range(warm):
                pred, real, eps = inp[t]
                if ctx.adapt(st, pred, shift=shift, fresh_noise=eps)[0] == W.ADAPT_TR_INIT:
                    ctx.continue_(st, pre)
                s2 = ctx.adapt(st, real)[0]
                ctx.continue_(st, K - (b0 + pre if s2 == W.ADAPT_REBIND_ACCEPT else b0), act)
        ctx.reset_stats()
        torch.cuda.synchronize(dev)
        warm_ev = [(ev(), ev()) for _ in range(n)]
        cold_ev = [(ev(), ev()) for _ in range(n)]
        with torch.cuda.stream(stream):
            for i in range(n):
                pred, real, eps = inp[warm + i]
                warm_ev[i][0].record(stream)
                if ctx.adapt(st, pred, shift=shift, fresh_noise=eps)[0] == W.ADAPT_TR_INIT:
                    ctx.continue_(st, pre)
                s2 = ctx.adapt(st, real)[0]
                ctx.continue_(st, K - (b0 + pre if s2 == W.ADAPT_REBIND_ACCEPT else b0), act)
                warm_ev[i][1].record(stream)
        stt = ctx.stats()
        with torch.cuda.stream(stream):
            for i in range(n):
                pred, real, eps = inp[warm + i]
                cold_ev[i][0].record(stream)
                ctx.sample_cold(st_c, real, eps, K, act)
                cold_ev[i][1].record(stream)
        torch.cuda.synchronize(dev)
        w = [a.elapsed_time(b) for a, b in warm_ev]
        c = [a.elapsed_time(b) for a, b in cold_ev]
        out[f"seed_{seed}"] = {"chunks_per_s": 1000.0 * n / sum(w), "ms_p50": float(np.percentile(w, 50)),
                               "ms_p99": float(np.percentile(w, 99)),
                               "cold_chunks_per_s": 1000.0 * n / sum(c), "cold_ms_p50": float(np.percentile(c, 50)),
                               "speedup_vs_cold": sum(c) / sum(w),
                               "r_or": stt["n_bind"] / max(1, stt["n_start"]),
                               "r_rr": stt["n_reuse"] / max(1, stt["n_attempt"])}
        st.close()
        st_c.close()
        del inp
    out["steps_per_seed"] = n
    out["what"] = ("closed-loop rollout per seed (own observation process, noise and fresh-noise draws): n warm "
                   "control steps and, under the same real observations, n cold 10-step samples; device time")
    return out


def run_async_prefix(ctx, cfg, dev, stream, dev_in, obs0, noise, windows_ms=(0.0, 1.0, 3.0), n=20, warm=3):
    """Asynchronous execution (§3.2; App. B.3) with App. A's timing: the controller executes the
    previous action chunk for a modelled window while the anticipatory prefix of the next replan
    (TR + 1 step under the predicted observation) runs on a second stream; when the window ends
    the real observation arrives (t_obs), Observation Rebinding and the remaining steps run on the
    main stream, and the chunk is copied to pinned host memory (t_ready).  O2A = t_ready - t_obs
    on the host clock; GPU = the replan's device time (prefix + foreground, CUDA events)."""
    import torch

    from paper_2609_34608_gb300 import wam as W

    K, b0, shift, pre = cfg["n_steps"], cfg["tr_entry_stage"], cfg["shift"], cfg["prefix_steps"]
    s_pre = torch.cuda.Stream(dev)
    act = torch.zeros((1, cfg["n_action"], cfg["action_dim"])).pin_memory()
    ev = lambda: torch.cuda.Event(enable_timing=True)
    out = {}
    for wms in windows_ms:
        st = ctx.state(1)
        with torch.cuda.stream(stream):
            ctx.sample_cold(st, obs0, noise, K, act)
        torch.cuda.synchronize(dev)
        t_ready = time.perf_counter()
        o2a, gpu, hidden = [], [], 0
        for i in range(warm + n):
            pred, real, eps = dev_in[i % len(dev_in)]
            # the controller starts executing the chunk; the prefix runs meanwhile
            g0, g1, f0, f1 = ev(), ev(), ev(), ev()
            ready = torch.cuda.Event()
            ready.record(stream)
            s_pre.wait_event(ready)
            ctx.set_stream(s_pre.cuda_stream)
            g0.record(s_pre)
            if ctx.adapt(st, pred, shift=shift, fresh_noise=eps)[0] == W.ADAPT_TR_INIT:
                ctx.continue_(st, pre)
            g1.record(s_pre)
            ctx.set_stream(stream.cuda_stream)
            stream.wait_event(g1)
            while time.perf_counter() < t_ready + wms * 1e-3:
                pass
            t_obs = time.perf_counter()
            done_early = g1.query()
            f0.record(stream)
            s2 = ctx.adapt(st, real)[0]
            ctx.continue_(st, K - (b0 + pre if s2 == W.ADAPT_REBIND_ACCEPT else b0), act)   # returns with the chunk
            f1.record(stream)
            t_ready = time.perf_counter()
            if i >= warm:
                f1.synchronize()
                o2a.append((t_ready - t_obs) * 1e3)
                gpu.append(g0.elapsed_time(g1) + f0.elapsed_time(f1))
                hidden += 1 if done_early else 0
        st.close()
        out[f"window_{wms:g}ms"] = {"o2a_ms_p50": float(np.percentile(o2a, 50)), "o2a_ms_p99": float(np.percentile(o2a, 99)),
                                    "gpu_ms_per_replan": statistics.mean(gpu), "prefix_done_before_obs": hidden / n}
    out["what"] = ("anticipatory prefix (TR + 1 step under the prediction) on a second stream during a modelled "
                   "action-execution window; then OR + 2 steps on the main stream, chunk to pinned host memory. "
                   "O2A on the host clock from the end of the window; GPU = prefix + foreground device time")
    out["steps"] = n
    return out


def run_bimanual(dev, stream, peaks, n_cold=2):
    """The large bimanual model (28 blocks, d1152, 16 heads of dim 72; 768 obs + 4096 video +
    50 x 14 action tokens = 4914 tokens; batch 8): a 10-step cold sample of the batch, then the
    warm-continuation sweep over retained-step counts 1..9 with executed shift 25 (TR of the
    finished replan to entry stage K - n, then n steps; run from n = 9 down to 1)."""
    import torch

    from paper_2609_34608_gb300 import inputs as I
    from paper_2609_34608_gb300 import wam as W

    # retained stage = entry stage (r = b0), so that each replan of the sweep (n = 9 down to 1,
    # entry stage K - n rising) remaps a stage the previous replan produced
    cfg = I.get_config("bimanual", tr_retain_stage=-1)
    B, K = cfg["batch"], cfg["n_steps"]
    flat = torch.from_numpy(I.flatten_weights(I.make_weights(cfg))).to(dev)
    ctx = W.Context(cfg, flat, stream=stream.cuda_stream)
    del flat
    with torch.cuda.stream(stream):
        obs = torch.from_numpy(I.make_obs(cfg, B)).to(dev)
        noise = torch.from_numpy(I.make_noise(cfg, B)).to(dev)
        eps = [torch.from_numpy(I.make_fresh_eps(cfg, B, i)).to(dev) for i in range(K)]
        act = torch.zeros((B, cfg["n_action"], cfg["action_dim"]), device=dev)
        st = ctx.state(B)
        ctx.sample_cold(st, obs, noise, K, act)   # warm-up (also captures the layer graphs)
    ev = lambda: torch.cuda.Event(enable_timing=True)
    cold = []
    with torch.cuda.stream(stream):
        for _ in range(n_cold):
            a, b = ev(), ev()
            a.record(stream)
            ctx.sample_cold(st, obs, noise, K, act)
            b.record(stream)
            cold.append((a, b))
    torch.cuda.synchronize(dev)
    cold_ms = statistics.mean(a.elapsed_time(b) for a, b in cold)
    sweep = {}
    with torch.cuda.stream(stream):
        marks = []
        for n in range(K - 1, 0, -1):
            a, b = ev(), ev()
            a.record(stream)
            ctx.adapt(st, obs, shift=cfg["shift"], entry=K - n, fresh_noise=eps[n])
            ctx.continue_(st, n, act)
            b.record(stream)
            marks.append((n, a, b))
    torch.cuda.synchronize(dev)
    for n, a, b in marks:
        ms = a.elapsed_time(b)
        sweep[str(n)] = {"ms_per_batch": ms, "chunks_per_s": B / (ms * 1e-3)}
    ctx.profile_enable(True)
    with torch.cuda.stream(stream):
        ctx.sample_cold(st, obs, noise, K, act)
    prof = ctx.profile_read()
    ctx.profile_enable(False)
    ctx.close()
    kt = kernel_table(prof, 1, peaks, tensor_peak="bf16_sus")
    return {
        "workload": "28-block d1152 16-head (head dim 72) bf16 DiT, 768 obs + 4096 video + 50x14 action tokens, "
                    "batch 8; cold 10-step sample, then warm continuation of n = 1..9 retained steps after TR with "
                    "executed shift 25",
        "cold_ms_per_batch": cold_ms, "cold_chunks_per_s": B / (cold_ms * 1e-3),
        "warm_sweep": sweep,
        "gemm_tflops": kt["gemm"]["tflops"], "gemm_frac": kt["gemm"]["frac"],
        "attn_tflops": kt["attn"]["tflops"], "attn_frac": kt["attn"]["frac"],
        "kernels_per_cold_batch": kt,
        "peak_source": "measured sustained bf16 (a batch runs for seconds)",
    }


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
    kt = kernel_table(prof, 1, peaks, tensor_peak="bf16_sus")
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
    ap.add_argument("--no-bimanual", action="store_true", help="skip the large bimanual model section")
    ap.add_argument("--no-ablation", action="store_true", help="skip the Table 3 ablation section")
    ap.add_argument("--no-async", action="store_true", help="skip the asynchronous-prefix section")
    ap.add_argument("--no-seeds", action="store_true", help="skip the per-seed closed-loop rollouts")
    ap.add_argument("--cpu-plan", action="store_true",
                    help="only time the CPU oracle plan (all cores and one core; no GPU) and print it")
    args = ap.parse_args()
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")
    if args.cpu_plan:
        print(json.dumps({"cpu_plan": cpu_plan()}))
        return 0
    if args.impl == "reference":
        return main_reference(args)
    return main_ours(args)


if __name__ == "__main__":
    sys.exit(main())
