"""The fused row-chain launch (out-projection .. MLP .. next block's LN + QKV as one persistent
kernel) against the separate per-projection launches: the same arithmetic, so a cold sample and
warm continuations (TR, OR, RR with rejected episodes gathered through the middle layers, and with
a relaxed gate that injects) give bit-identical latents, velocities and actions either way; also
at the full size of the latency model."""
import numpy as np
import pytest

from paper_2609_34608_gb300 import inputs as I
from paper_2609_34608_gb300 import wam as W

pytestmark = pytest.mark.gpu

SMALL_BF16 = dict(n_layers=4, d_model=128, n_heads=2, n_obs=32, n_video=96, n_action=8, action_dim=7,
                  n_steps=6, precision="bf16", rr_policy=1, rr_q=1, rr_s=2, rr_e=3,
                  tr_entry_stage=3, tr_retain_stage=-1, shift=2)


def _run(cfg, fusion, batch, replans=3):
    Wd = I.make_weights(cfg)
    ctx = W.Context(cfg, I.flatten_weights(Wd))
    ctx.set_layer_fusion(fusion)
    K = cfg["n_steps"]
    st = ctx.state(batch)
    ctx.sample_cold(st, I.make_obs(cfg, batch), I.make_noise(cfg, batch), K)
    outs = [ctx.read(st, W.FIELD_X).copy(), ctx.read(st, W.FIELD_V_STEP, 0).copy()]
    entry = int(cfg["tr_entry_stage"])
    for r in range(replans):
        ctx.adapt(st, I.make_obs(cfg, batch, seed=50 + r), shift=np.full(batch, int(cfg["shift"]), np.int32),
                  entry=np.full(batch, entry, np.int32), fresh_noise=I.make_fresh_eps(cfg, batch, r))
        act = np.zeros((batch, cfg["n_action"], cfg["action_dim"]), np.float32)
        ctx.continue_(st, np.full(batch, K - entry, np.int32), act)
        outs += [ctx.read(st, W.FIELD_X).copy(), ctx.read(st, W.FIELD_V_STEP, K - 1).copy(), act]
    stats = ctx.stats()
    ctx.close()
    return outs, stats


@pytest.mark.parametrize("relax", [False, True])
def test_fused_chain_is_bit_identical_small(wamlib, relax):
    over = dict(rr_gamma_cos=-1.0, rr_gamma_fit=1e30) if relax else {}
    cfg = I.get_config("tiny", batch=3, **SMALL_BF16, **over)
    a, sa = _run(cfg, True, 3)
    b, sb = _run(cfg, False, 3)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    assert sa["n_reuse"] == sb["n_reuse"]
    assert sa["n_kernel_launches"] < sb["n_kernel_launches"]
    if relax:
        assert sa["n_reuse"] > 0


def test_fused_chain_is_bit_identical_latency_model(wamlib):
    cfg = I.get_config("latency")
    a, _ = _run(cfg, True, 1, replans=1)
    b, _ = _run(cfg, False, 1, replans=1)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
