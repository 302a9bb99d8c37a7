"""Single-kernel timing through the C ABI (include/wam_ops.h), for kernel tuning and ncu captures.

    python -m paper_2609_34608_gb300.kernel_bench gemm M N K [--iters I] [--tile T --cluster C] [--epi E]
    python -m paper_2609_34608_gb300.kernel_bench attn B N H [--iters I] [--impl tc|mma] [--head-dim 64|72]
    python -m paper_2609_34608_gb300.kernel_bench step CONFIG [--batch B] [--rounds R] [--relax-gate]
    python -m paper_2609_34608_gb300.kernel_bench sweep CONFIG B1 B2 ... [--relax-gate]

Each invocation builds the library if needed, warms up, captures `iters` back-to-back launches in
a CUDA graph, times a replay with CUDA events and prints one JSON line (microseconds per launch
and algorithmic TFLOP/s: 2MNK for the GEMM, 4 B N^2 d for attention).

`sweep` runs one warm round (the profile's Trajectory Remapping, then its remaining steps) at
each batch size with the library's kernel-class timing on
(CUDA events on its stream) and prints, per size, the achieved algorithmic bandwidth of the
residual-stream and adaptation kernel classes (final layer + Euler, TR / OR adaptation, RR probe,
RR apply, LN) as fractions of the measured copy bandwidth.

`step` drives a named model configuration (inputs.NAMED_CONFIGS) through the library's public
calls with seeded synthetic inputs: a cold sample of all episodes, then R warm rounds, each a
Trajectory Remapping by the configuration's shift with Observation Rebinding to new observations
and a continuation of two steps (Residual Rescaling active; --relax-gate lets every RR check
pass, exercising the injection path).  It prints the cold and per-round times; its launches are
what the elementwise / adaptation profiles capture.
"""
from __future__ import annotations

import argparse
import json

import torch

from . import _build
from . import wam as W


def _time(fn, iters: int) -> float:
    """Microseconds per call of fn(stream): `iters` calls captured in one CUDA graph and replayed,
    so the host-side work of each op call (tensor-map encoding) is not in the measurement."""
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for _ in range(3):
            fn(side.cuda_stream)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        s = torch.cuda.current_stream().cuda_stream
        for _ in range(iters):
            fn(s)
    g.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    g.replay()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) * 1000.0 / iters


EPILOGUES = {"bf16": W.EPI_BF16, "gelu": W.EPI_GELU_BF16, "resid": W.EPI_RESID_F32}


def bench_gemm(M: int, N: int, K: int, iters: int, tile_n: int = 0, cluster: int = 0, epi: str = "bf16") -> dict:
    """One projection; tile_n / cluster = 0: the library's plan, else an explicit plan
    (wam_op_gemm_bf16_plan: tile width, 1 single CTAs, 2 multicast pairs, 3 two-SM MMA pairs)."""
    dev = torch.device("cuda")
    A = torch.randn(M, K, device=dev).to(torch.bfloat16)
    Wt = (torch.randn(N, K, device=dev) * 0.05).to(torch.bfloat16)
    e = EPILOGUES[epi]
    C = torch.zeros(M, N, device=dev, dtype=torch.float32 if e == W.EPI_RESID_F32 else torch.bfloat16)
    b = torch.zeros(N, device=dev)
    gate = torch.full((M, N), 0.5, device=dev) if e == W.EPI_RESID_F32 else None
    if tile_n == 0 and cluster == 0:
        fn = lambda st: W.op_gemm_bf16(A, Wt, b, C, M, N, K, e, gate=gate, gate_stride=N, rows_per_item=M,
                                       stream=st)
    else:
        fn = lambda st: W.op_gemm_bf16_plan(A, Wt, b, C, M, N, K, e, tile_n, 1, gate=gate, gate_stride=N,
                                            rows_per_item=M, stream=st, cluster=cluster)
    us = _time(fn, iters)
    return {"kernel": "gemm_tc", "M": M, "N": N, "K": K, "tile_n": tile_n, "cluster": cluster, "epi": epi,
            "us": us, "tflops": 2.0 * M * N * K / us / 1e6}


def bench_attn(B: int, N: int, H: int, iters: int, impl: str, head_dim: int = 64) -> dict:
    dev = torch.device("cuda")
    if head_dim != 64 and impl != "tc":
        raise ValueError("the mma.sync attention takes head dim 64 only")
    d = head_dim * H
    qkv = torch.randn(B * N, 3 * d, device=dev).to(torch.bfloat16)
    out = torch.empty(B * N, d, device=dev, dtype=torch.bfloat16)
    if impl == "tc":
        vt_ld = (N + 7) // 8 * 8
        vt = torch.randn(B * d, vt_ld, device=dev).to(torch.bfloat16)
        fn = lambda st: W.op_attention_tc(qkv, vt, out, B, N, d, H, stream=st)
    else:
        fn = lambda st: W.op_attention(qkv, out, B, N, d, H, "bf16", stream=st)
    us = _time(fn, iters)
    return {"kernel": f"attention_{impl}", "B": B, "N": N, "H": H, "head_dim": head_dim, "us": us,
            "tflops": 4.0 * B * N * N * d / us / 1e6}


def bench_step(name: str, batch: int, rounds: int, relax_gate: bool) -> dict:
    import numpy as np

    from . import inputs as I
    dev = torch.device("cuda")
    over = dict(rr_gamma_cos=-1.0, rr_gamma_fit=1e30) if relax_gate else {}
    cfg = I.get_config(name, batch=batch, **over)
    K = cfg["n_steps"]
    stream = torch.cuda.Stream()
    ctx = W.Context(cfg, I.flatten_weights(I.make_weights(cfg)), stream=stream.cuda_stream)
    st = ctx.state(batch)
    shift = np.full(batch, int(cfg["shift"]), np.int32)
    entry = np.full(batch, K - 2, np.int32)
    with torch.cuda.stream(stream):
        obs = [torch.from_numpy(I.make_obs(cfg, batch, seed=100 + i)).to(dev) for i in range(rounds + 1)]
        eps = [torch.from_numpy(I.make_fresh_eps(cfg, batch, i)).to(dev) for i in range(rounds + 1)]
        noise = torch.from_numpy(I.make_noise(cfg, batch)).to(dev)
        e = [torch.cuda.Event(enable_timing=True) for _ in range(rounds + 2)]
        e[0].record(stream)
        ctx.sample_cold(st, obs[0], noise, K)
        e[1].record(stream)
        for r in range(rounds):
            ctx.adapt(st, obs[r + 1], shift=shift, entry=entry, fresh_noise=eps[r + 1])
            ctx.continue_(st, np.full(batch, 2, np.int32))
            e[r + 2].record(stream)
    torch.cuda.synchronize()
    out = {"kind": "step", "config": name, "batch": batch, "cold_ms": e[0].elapsed_time(e[1]),
           "warm_round_ms": [e[r + 1].elapsed_time(e[r + 2]) for r in range(rounds)], "stats": ctx.stats()}
    ctx.close()
    return out


def bench_sweep(name: str, batches: list, relax_gate: bool) -> list:
    import json as _json
    import os

    import numpy as np

    from . import inputs as I
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    peaks_path = os.path.join(root, "MEASURED_PEAKS.json")
    hbm = _json.load(open(peaks_path))["hbm_gbs"] if os.path.exists(peaks_path) else 6800.0
    dev = torch.device("cuda")
    over = dict(rr_gamma_cos=-1.0, rr_gamma_fit=1e30) if relax_gate else {}
    out = []
    bmax = max(batches)
    cfg = I.get_config(name, batch=bmax, **over)
    K = cfg["n_steps"]
    stream = torch.cuda.Stream()
    ctx = W.Context(cfg, I.flatten_weights(I.make_weights(cfg)), stream=stream.cuda_stream, batch_max=bmax)
    for batch in batches:
        st = ctx.state(batch)
        shift = np.full(batch, int(cfg["shift"]), np.int32)
        b0 = int(cfg["tr_entry_stage"])  # the profile's entry stage (its retained stage is valid)
        with torch.cuda.stream(stream):
            obs = [torch.from_numpy(I.make_obs(cfg, batch, seed=100 + i)).to(dev) for i in range(3)]
            eps = [torch.from_numpy(I.make_fresh_eps(cfg, batch, i)).to(dev) for i in range(3)]
            noise = torch.from_numpy(I.make_noise(cfg, batch)).to(dev)
            ctx.sample_cold(st, obs[0], noise, K)
            ctx.adapt(st, obs[1], shift=shift, fresh_noise=eps[1])
            ctx.continue_(st, np.full(batch, K - b0, np.int32))
            ctx.profile_enable(True)
            ctx.adapt(st, obs[2], shift=shift, fresh_noise=eps[2])
            ctx.continue_(st, np.full(batch, K - b0, np.int32))
            prof = ctx.profile_read()
            ctx.profile_enable(False)
        row = {"config": name, "batch": batch}
        for k in ("final", "adapt", "rr_probe", "rr_apply", "norm"):
            v = prof[k]
            if v["ms"] > 0:
                gbs = v["bytes"] / (v["ms"] * 1e-3) / 1e9
                row[k] = {"launches": v["launches"], "us_per_launch": 1e3 * v["ms"] / max(1, v["launches"]),
                          "gbs": gbs, "frac": gbs / hbm}
        out.append(row)
        st.close()
    ctx.close()
    return out


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("kind", choices=["gemm", "attn", "step", "sweep"])
    ap.add_argument("dims", nargs="+")
    ap.add_argument("--iters", type=int, default=20)
    ap.add_argument("--impl", choices=["tc", "mma"], default="tc")
    ap.add_argument("--head-dim", type=int, choices=[64, 72], default=64)
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--rounds", type=int, default=1)
    ap.add_argument("--relax-gate", action="store_true")
    ap.add_argument("--tile", type=int, default=0, help="gemm: explicit tile width (0 = the library's plan)")
    ap.add_argument("--cluster", type=int, default=0, help="gemm: 1 single, 2 multicast pairs, 3 two-SM pairs")
    ap.add_argument("--epi", choices=sorted(EPILOGUES), default="bf16")
    a = ap.parse_args()
    _build.build()
    if a.kind == "gemm":
        print(json.dumps(bench_gemm(*map(int, a.dims), a.iters, a.tile, a.cluster, a.epi)))
    elif a.kind == "attn":
        print(json.dumps(bench_attn(*map(int, a.dims), a.iters, a.impl, a.head_dim)))
    elif a.kind == "sweep":
        for row in bench_sweep(a.dims[0], [int(b) for b in a.dims[1:]], a.relax_gate):
            print(json.dumps(row))
    else:
        print(json.dumps(bench_step(a.dims[0], a.batch, a.rounds, a.relax_gate)))


if __name__ == "__main__":
    main()
