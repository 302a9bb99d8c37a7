"""CUDA-graph replay of the layer stack changes launch overhead only: a cold sample followed by
warm continuations (Trajectory Remapping, Observation Rebinding, Residual Rescaling) gives
bit-identical latents, velocities and actions with replay on and off, in both precisions, with
the default RR gate (rejected episodes gathered through the middle layers) and with a relaxed
gate (every check passes: injection, the middle layers skipped)."""
import numpy as np
import pytest

from paper_2609_34608_gb300 import inputs as I
from paper_2609_34608_gb300 import wam as W

pytestmark = pytest.mark.gpu


def _run(cfg, replay, batch):
    Wd = I.make_weights(cfg)
    ctx = W.Context(cfg, I.flatten_weights(Wd))
    ctx.set_graph_replay(replay)
    K = cfg["n_steps"]
    st = ctx.state(batch)
    obs = I.make_obs(cfg, batch)
    ctx.sample_cold(st, obs, I.make_noise(cfg, batch), K)
    outs = [ctx.read(st, W.FIELD_X).copy()]
    entry = int(cfg["tr_entry_stage"])
    for r in range(3):   # repeated continuations: eager first use, capture, then replays
        new_obs = I.make_obs(cfg, batch, seed=50 + r)
        ctx.adapt(st, new_obs, shift=np.full(batch, int(cfg["shift"]), np.int32),
                  entry=np.full(batch, entry, np.int32), fresh_noise=I.make_fresh_eps(cfg, batch, r))
        act = np.zeros((batch, cfg["n_action"], cfg["action_dim"]), np.float32)
        ctx.continue_(st, np.full(batch, K - entry, np.int32), act)
        outs += [ctx.read(st, W.FIELD_X).copy(), ctx.read(st, W.FIELD_V_STEP, K - 1).copy(), act]
    stats = ctx.stats()
    ctx.close()
    return outs, stats


# head dim 64 for the bf16 path (tcgen05 attention), RR (1, 2, 3) over 4 layers
SMALL_BF16 = dict(n_layers=4, d_model=128, n_heads=2, n_obs=32, n_video=96, n_action=8, action_dim=7,
                  n_steps=6, precision="bf16", rr_policy=1, rr_q=1, rr_s=2, rr_e=3,
                  tr_entry_stage=3, tr_retain_stage=-1, shift=2)


@pytest.mark.parametrize("precision", ["fp32", "bf16"])
@pytest.mark.parametrize("relax", [False, True])
def test_graph_replay_is_bit_identical(wamlib, precision, relax):
    over = dict(rr_gamma_cos=-1.0, rr_gamma_fit=1e30) if relax else {}
    if precision == "bf16":
        cfg = I.get_config("tiny", batch=3, **SMALL_BF16, **over)
    else:
        cfg = I.get_config("tiny_rr", batch=3, **over)
    a, sa = _run(cfg, True, 3)
    b, sb = _run(cfg, False, 3)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    assert sa["n_reuse"] == sb["n_reuse"]
    if relax:
        assert sa["n_reuse"] > 0   # the injection path (middle layers skipped) ran


def _closed_loop_b1(cfg, device_branching, rounds=4):
    """Batch-1 closed loop: cold sample, then TR + one prefix step + OR + the rest, repeated."""
    Wd = I.make_weights(cfg)
    ctx = W.Context(cfg, I.flatten_weights(Wd))
    ctx.set_device_branching(device_branching)
    K, b0 = cfg["n_steps"], int(cfg["tr_entry_stage"])
    st = ctx.state(1)
    proc = I.ObsProcess(cfg, 1, seed=4)
    ctx.sample_cold(st, proc.obs.copy(), I.make_noise(cfg, 1), K)
    outs, logs = [], []
    for r in range(rounds):
        pred, real = proc.predicted(), proc.step()
        s1 = ctx.adapt(st, pred, shift=int(cfg["shift"]), fresh_noise=I.make_fresh_eps(cfg, 1, r))[0]
        if s1 == W.ADAPT_TR_INIT:
            ctx.continue_(st, 1)
            logs += ctx.log(st)
        ctx.adapt(st, real)
        act = np.zeros((1, cfg["n_action"], cfg["action_dim"]), np.float32)
        ctx.continue_(st, K - int(ctx.read(st, W.FIELD_META)[0][0]), act)
        logs += ctx.log(st)
        outs += [ctx.read(st, W.FIELD_X).copy(), act, ctx.read(st, W.FIELD_RR_P).copy()]
    stats = ctx.stats()
    ctx.close()
    return outs, logs, stats


@pytest.mark.parametrize("precision", ["fp32", "bf16"])
@pytest.mark.parametrize("gate", ["relaxed", "strict", "default"])
def test_device_branching_matches_host_branching(wamlib, precision, gate):
    """The RR decision taken on the device inside the step's graph (conditional middle layers)
    gives the same latents, actions, layer state, step log and reuse statistics as the host
    decision, on the accept path (relaxed gate), the reject path (strict gate) and a mix."""
    over = {"relaxed": dict(rr_gamma_cos=-1.0, rr_gamma_fit=1e30),
            "strict": dict(rr_gamma_cos=0.99999, rr_gamma_fit=1e-6), "default": {}}[gate]
    if precision == "bf16":
        cfg = I.get_config("tiny", **SMALL_BF16, **over)
    else:
        cfg = I.get_config("tiny_rr", **over)
    a, la, sa = _closed_loop_b1(cfg, True)
    b, lb, sb = _closed_loop_b1(cfg, False)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    assert la == lb
    for k in ("n_reuse", "n_attempt", "b_skip", "b_dense", "n_layer_evals", "n_bind"):
        assert sa[k] == sb[k], k
    if gate == "relaxed":
        assert sa["n_reuse"] == sa["n_attempt"] > 0
    if gate == "strict":
        assert sa["n_reuse"] == 0 and sa["n_attempt"] > 0
    assert sa["n_kernel_launches"] > 0


def test_prefix_on_second_stream_matches_one_stream(wamlib):
    """The anticipatory prefix (TR + one step under the prediction) issued on a second stream
    while the first is idle, ordered by events, gives the same replans as one stream."""
    import torch

    cfg = I.get_config("tiny", **SMALL_BF16)
    K, b0 = cfg["n_steps"], int(cfg["tr_entry_stage"])
    dev = torch.device("cuda")
    res = []
    for two in (False, True):
        main, side = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
        ctx = W.Context(cfg, I.flatten_weights(I.make_weights(cfg)), stream=main.cuda_stream)
        st = ctx.state(1)
        proc = I.ObsProcess(cfg, 1, seed=6)
        act = torch.zeros((1, cfg["n_action"], cfg["action_dim"])).pin_memory()
        ctx.sample_cold(st, proc.obs.copy(), I.make_noise(cfg, 1), K, act)
        outs = []
        for r in range(4):
            pred, real = proc.predicted(), proc.step()
            if two:
                ready = torch.cuda.Event()
                ready.record(main)
                side.wait_event(ready)
                ctx.set_stream(side.cuda_stream)
            s1 = ctx.adapt(st, pred, shift=int(cfg["shift"]), fresh_noise=I.make_fresh_eps(cfg, 1, r))[0]
            if s1 == W.ADAPT_TR_INIT:
                ctx.continue_(st, 1)
            if two:
                done = torch.cuda.Event()
                done.record(side)
                ctx.set_stream(main.cuda_stream)
                main.wait_event(done)
            s2 = ctx.adapt(st, real)[0]
            ctx.continue_(st, K - (b0 + 1 if s2 == W.ADAPT_REBIND_ACCEPT else b0), act)   # host output: synchronous
            outs += [act.numpy().copy(), ctx.read(st, W.FIELD_X).copy()]
        res.append((outs, ctx.stats()["n_reuse"]))
        ctx.close()
    for x, y in zip(res[0][0], res[1][0]):
        assert np.array_equal(x, y)
    assert res[0][1] == res[1][1]
