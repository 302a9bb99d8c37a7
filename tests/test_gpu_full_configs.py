"""Parity at the full sizes of the batched-serving and bimanual models.

The oracle needs tens of seconds per float64 forward at these sizes, so each test checks a
few denoising steps of one episode with teacher forcing (the oracle evaluates the velocity at
the GPU's latent and replays its RR decision), plus properties that hold at any size: an
episode computed inside a batch equals the same episode computed alone.
"""
import numpy as np
import pytest

from oracle import wam_oracle as O
from paper_2609_34608_gb300 import inputs as I
from paper_2609_34608_gb300 import wam as W

pytestmark = pytest.mark.gpu

BF16_VEL_TOL = 2e-2


def _rel_l2(a, b):
    a = np.asarray(a, np.float64).ravel()
    b = np.asarray(b, np.float64).ravel()
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def _setup(name, batch):
    cfg = I.get_config(name, batch=batch)
    Wd = I.make_weights(cfg)
    ctx = W.Context(cfg, I.flatten_weights(Wd))
    return cfg, Wd, ctx


def _teacher_forced(cfg, Wd, ctx, st, obs, ep):
    ocfg = O.OracleConfig.from_dict(cfg)
    sig = O.schedule(cfg["n_steps"], cfg["sched_shift"])
    layer = None
    errs = []
    for rec in (r for r in ctx.log(st) if r["episode"] == ep):
        k = rec["stage"]
        x = ctx.read(st, W.FIELD_X_STAGE, k)[ep]
        v, layer, orec = O.velocity_rr(Wd, ocfg, x, obs, sig[k], layer, True,
                                       rec["rr_accept"] if rec["rr_attempt"] else None)
        assert orec.rr_attempt == rec["rr_attempt"]
        errs.append(_rel_l2(ctx.read(st, W.FIELD_V_STEP, k)[ep], v))
    return errs


def test_serving_model_two_steps_and_batch_consistency(wamlib):
    cfg, Wd, ctx = _setup("serving", 3)
    obs = I.make_obs(cfg, 3)
    noise = I.make_noise(cfg, 3)
    st = ctx.state(3)
    ctx.sample_cold(st, obs, noise, 2)                 # 2 of 10 steps: the second one gates RR
    errs = _teacher_forced(cfg, Wd, ctx, st, obs[0], 0)
    assert len(errs) == 2 and max(errs) <= BF16_VEL_TOL, errs
    x_batch = ctx.read(st, W.FIELD_X)
    st1 = ctx.state(1)
    ctx.sample_cold(st1, obs[2:3], noise[2:3], 2)
    assert np.allclose(ctx.read(st1, W.FIELD_X)[0], x_batch[2], rtol=1e-5, atol=1e-5)


def test_bimanual_model_one_step(wamlib):
    """Head dim 72 (the tcgen05 attention with the head padded to 80), 4914 joint tokens, 14-DoF
    actions."""
    cfg, Wd, ctx = _setup("bimanual", 1)
    obs = I.make_obs(cfg, 1)
    st = ctx.state(1)
    ctx.sample_cold(st, obs, I.make_noise(cfg, 1), 1)
    errs = _teacher_forced(cfg, Wd, ctx, st, obs[0], 0)
    assert len(errs) == 1 and errs[0] <= BF16_VEL_TOL, errs


def test_bimanual_model_warm_step_after_remap(wamlib):
    """The bimanual workload's warm path: a finished 10-step replan remapped with executed shift 25
    (half of the 50-step action horizon receives retained state, the rest fresh noise) into entry
    stage 9, then one RR-gated step, teacher-forced against the oracle (head dim 72, 4914 tokens)."""
    cfg, Wd, ctx = _setup("bimanual", 1)
    ocfg = O.OracleConfig.from_dict(cfg)
    K = cfg["n_steps"]
    sig = O.schedule(K, cfg["sched_shift"])
    obs = I.make_obs(cfg, 1)
    st = ctx.state(1)
    ctx.sample_cold(st, obs, I.make_noise(cfg, 1), K)
    r = cfg["tr_retain_stage"]
    x_bar, x_r = ctx.read(st, W.FIELD_X_STAGE, K)[0], ctx.read(st, W.FIELD_X_STAGE, r)[0]
    obs2 = I.make_obs(cfg, 1, seed=9)
    eps = I.make_fresh_eps(cfg, 1, 3)
    b0 = K - 1
    assert ctx.adapt(st, obs2, shift=cfg["shift"], entry=b0, fresh_noise=eps)[0] == W.ADAPT_TR_INIT
    want = O.tr_remap(ocfg, x_bar, x_r, sig[r], sig[b0], cfg["shift"], eps[0])
    got = ctx.read(st, W.FIELD_X_INIT)[0]
    ulp = np.spacing(np.abs(want).astype(np.float32)).astype(np.float64)
    assert np.all(np.abs(got.astype(np.float64) - want) <= ulp)
    # slots past the shifted horizon hold sigma_b0 * eps exactly
    V, ad = ocfg.video_len, cfg["action_dim"]
    tail = slice(V + (cfg["n_action"] - cfg["shift"]) * ad, None)
    assert np.array_equal(got[tail], (sig[b0] * eps[0][tail].astype(np.float64)).astype(np.float32))
    # the layer state the step's RR check compares against (left by the cold replan; TR keeps it)
    layer0 = O.LayerState(p_a=ctx.read(st, W.FIELD_RR_P)[0].astype(np.float64),
                          R_a=ctx.read(st, W.FIELD_RR_R)[0].astype(np.float64))
    ctx.continue_(st, 1)
    rec = ctx.log(st)[0]
    assert rec["stage"] == b0 and rec["rr_attempt"]
    v, _, orec = O.velocity_rr(Wd, ocfg, ctx.read(st, W.FIELD_X_STAGE, b0)[0], obs2[0], sig[b0], layer0, True,
                               rec["rr_accept"])
    assert orec.rr_attempt
    assert _rel_l2(ctx.read(st, W.FIELD_V_STEP, b0)[0], v) <= BF16_VEL_TOL
