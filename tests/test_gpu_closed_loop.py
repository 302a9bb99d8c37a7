"""Parity of the warm closed-loop control step (§3.1 Trajectory Remapping, §3.2 Observation
Rebinding, §3.3 Residual Rescaling, coordinated as in §3.4) against the CPU oracle, through the
C ABI, with every device reduction spanning several blocks.

* Full size (12 blocks, d=768, 1296 tokens, T = 16 496, bf16): the control step the benchmark
  times.  The TR direction RMS runs over 8 + 1 blocks of 2048 values (video, action), the OR
  score over 256 x 768 observation values (24 blocks of 8192), the RR probe sums over
  1280 x 768 and 16 x 768 values (120 + 2 blocks of 8192).  The oracle continues from the GPU's
  finished replan (its retained latents and layer state), so the remapped initialisation is
  compared value by value: within one float32 ulp of the float64 remap, and bit-exact in its
  index work (a zero-direction case).  Each later step is teacher-forced (rel-L2 <= 2e-2), the
  RR statistics are compared with the oracle's, and the oracle's free run gives the final
  actions (max-abs <= 5e-2).
* A float32 model whose trajectory, observation and probe reductions all span several blocks
  (video 4800 values, action 2100, observation 20 480, probe 58 880 / 38 400): free-running
  parity of three control steps at 1e-4, the OR status sequence and the RR decisions.
"""
import numpy as np
import pytest

from oracle import wam_oracle as O
from paper_2609_34608_gb300 import inputs as I
from paper_2609_34608_gb300 import wam as W

pytestmark = pytest.mark.gpu

FP32_TOL = 1e-4
BF16_VEL_TOL = 2e-2
BF16_ACT_TOL = 5e-2
RR_STAT_TOL = 2e-2   # cos / fit / alpha of a bf16 probe residual against the float64 one


def _rel_l2(a, b):
    a = np.asarray(a, np.float64).ravel()
    b = np.asarray(b, np.float64).ravel()
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


def _within_one_ulp(got, ref):
    ref = np.asarray(ref, np.float64)
    ulp = np.spacing(np.abs(ref).astype(np.float32)).astype(np.float64)
    return bool(np.all(np.abs(np.asarray(got, np.float64) - ref) <= ulp))


def _oracle_from_gpu_replan(Wd, ocfg, ctx, st, obs):
    """An oracle episode holding the GPU's finished replan: its stage latents, bound
    observation and retained RR layer state."""
    K = ocfg.n_steps
    ep = O.OracleEpisode(Wd, ocfg)
    ep.hist = {k: ctx.read(st, W.FIELD_X_STAGE, k)[0].astype(np.float64) for k in range(K + 1)}
    ep.hist_from, ep.stage, ep.finished = 0, K, True
    ep.x = ep.hist[K].copy()
    ep.obs = np.asarray(obs, np.float64).copy()
    ep.path, ep.path_steps, ep.kappa, ep.since_bind = "cold", K, 0, K
    if ocfg.rr_enabled:
        ep.layer = O.LayerState(p_a=ctx.read(st, W.FIELD_RR_P)[0].astype(np.float64),
                                R_a=ctx.read(st, W.FIELD_RR_R)[0].astype(np.float64))
    return ep


def _teacher_forced(Wd, ocfg, ctx, st, obs, layer):
    """Oracle velocity at each GPU latent of the latest call (replaying the GPU's RR decision),
    with the RR statistics of both sides."""
    sig = O.schedule(ocfg.n_steps, ocfg.sched_shift)
    out = []
    for rec in ctx.log(st):
        k = rec["stage"]
        x = ctx.read(st, W.FIELD_X_STAGE, k)[0]
        v, layer, orec = O.velocity_rr(Wd, ocfg, x, obs, sig[k], layer, True,
                                       rec["rr_accept"] if rec["rr_attempt"] else None)
        assert orec.rr_attempt == rec["rr_attempt"]
        out.append((rec, orec, _rel_l2(ctx.read(st, W.FIELD_V_STEP, k)[0], v)))
    return out, layer


def _check_rr_stats(rec, orec):
    if not rec["rr_attempt"]:
        return
    for br, chk in enumerate(orec.checks):
        assert abs(rec["cos"][br] - chk.cos) <= RR_STAT_TOL, (br, rec["cos"], chk)
        assert abs(rec["fit"][br] - chk.fit) <= RR_STAT_TOL, (br, rec["fit"], chk)
        assert abs(rec["alpha"][br] - chk.alpha) <= RR_STAT_TOL, (br, rec["alpha"], chk)


def test_closed_loop_control_step_full_size(wamlib):
    cfg = I.get_config("closed_loop")
    Wd = I.make_weights(cfg)
    ocfg = O.OracleConfig.from_dict(cfg)
    ctx = W.Context(cfg, I.flatten_weights(Wd))
    K, b0, shift = cfg["n_steps"], cfg["tr_entry_stage"], cfg["shift"]
    r = cfg["tr_retain_stage"]
    sig = O.schedule(K, cfg["sched_shift"])
    proc = I.ObsProcess(cfg, 1, seed=0)
    obs0 = proc.obs.copy()
    st = ctx.state(1)
    ctx.sample_cold(st, obs0, I.make_noise(cfg, 1), K)
    ep = _oracle_from_gpu_replan(Wd, ocfg, ctx, st, obs0[0])
    pred, real = proc.predicted(), proc.step()
    eps = I.make_fresh_eps(cfg, 1, 0)

    # Trajectory Remapping (Eqs. 1-2): the float64 remap of the same retained latents
    s1 = ctx.adapt(st, pred, shift=shift, fresh_noise=eps)[0]
    assert s1 == ep.adapt(pred[0], shift, eps[0]) == W.ADAPT_TR_INIT
    assert _within_one_ulp(ctx.read(st, W.FIELD_X_INIT)[0], ep.x_b0)

    # anticipatory prefix: one step under the predicted observation, RR gate against the
    # layer state of the cold replan
    ctx.continue_(st, cfg["prefix_steps"])
    tf, layer = _teacher_forced(Wd, ocfg, ctx, st, pred[0], ep.layer)
    for rec, orec, err in tf:
        assert err <= BF16_VEL_TOL, err
        _check_rr_stats(rec, orec)
    ep.advance(cfg["prefix_steps"], forced=[t[0]["rr_accept"] for t in tf])

    # Observation Rebinding (Eq. 4 and the kappa rule)
    S = O.or_score(ocfg, pred[0], real[0])
    s2 = ctx.adapt(st, real)[0]
    assert s2 == ep.adapt(real[0], 0, None)
    assert s2 == (W.ADAPT_REBIND_ACCEPT if S < cfg["or_tau"] else W.ADAPT_REBIND_RESTART)
    assert np.array_equal(ctx.read(st, W.FIELD_OBS)[0], real[0])

    # the rest of the replan under the real observation
    act = np.zeros((1, cfg["n_action"], cfg["action_dim"]), np.float32)
    n_rest = K - int(ctx.read(st, W.FIELD_META)[0][0])
    ctx.continue_(st, n_rest, act)
    tf, _ = _teacher_forced(Wd, ocfg, ctx, st, real[0], layer)
    assert len(tf) == n_rest
    for rec, orec, err in tf:
        assert err <= BF16_VEL_TOL, err
        _check_rr_stats(rec, orec)
    ep.advance(n_rest, forced=[t[0]["rr_accept"] for t in tf])
    assert np.max(np.abs(act[0] - ep.actions())) <= BF16_ACT_TOL

    # index work at full size: x^r = x_bar gives a zero direction, so every remapped slot is a
    # retained value moved by the shift and every uncovered slot sigma_b0 * eps, bit for bit
    T = ctx.T
    st2 = ctx.state(1)
    x_bar = (np.arange(T, dtype=np.float32) * 0.5 + 3.0)[None]
    eps2 = -1.0 - np.arange(T, dtype=np.float32)[None]
    ctx.write(st2, W.FIELD_X_STAGE, x_bar, index=K)
    ctx.write(st2, W.FIELD_X_STAGE, x_bar, index=r)
    meta = np.zeros((1, 8), np.int32)
    meta[:, 0], meta[:, 4] = K, 1
    ctx.write(st2, W.FIELD_META, meta)
    assert ctx.adapt(st2, pred, shift=shift, fresh_noise=eps2)[0] == W.ADAPT_TR_INIT
    want = O.tr_remap(ocfg, x_bar[0], x_bar[0], sig[r], sig[b0], shift, eps2[0])
    assert np.array_equal(ctx.read(st2, W.FIELD_X_INIT)[0], want.astype(np.float32))
    ctx.close()


MULTIBLOCK_FP32 = dict(n_obs=160, n_video=300, n_action=300, n_steps=8, tr_entry_stage=4,
                       tr_retain_stage=4, shift=3)


def test_multiblock_reductions_fp32_closed_loop(wamlib):
    cfg = I.get_config("tiny_rr", **MULTIBLOCK_FP32)
    Wd = I.make_weights(cfg)
    ocfg = O.OracleConfig.from_dict(cfg)
    ctx = W.Context(cfg, I.flatten_weights(Wd))
    K, shift = cfg["n_steps"], cfg["shift"]
    assert cfg["n_video"] * cfg["video_dim"] > 2 * 2048 and cfg["n_action"] * cfg["action_dim"] > 2048
    assert cfg["n_obs"] * cfg["d_model"] > 2 * 8192
    proc = I.ObsProcess(cfg, 1, seed=3)
    obs0 = proc.obs.copy()
    noise = I.make_noise(cfg, 1)
    st = ctx.state(1)
    act = np.zeros((1, cfg["n_action"], cfg["action_dim"]), np.float32)
    ctx.sample_cold(st, obs0, noise, K, act)
    ep = O.OracleEpisode(Wd, ocfg)
    ep.sample_cold(obs0[0], noise[0], K, forced=[r["rr_accept"] for r in ctx.log(st)])
    assert np.max(np.abs(act[0] - ep.actions())) <= FP32_TOL
    seq_gpu, seq_or, n_accept = [], [], 0
    for t in range(3):
        pred, real = proc.predicted(), proc.step()
        if t == 2:
            real = real + 2.0            # a surprise: the rebinding check fails and restarts
        eps = I.make_fresh_eps(cfg, 1, t)
        s1 = ctx.adapt(st, pred, shift=shift, fresh_noise=eps)[0]
        o1 = ep.adapt(pred[0], shift, eps[0])
        assert np.max(np.abs(ctx.read(st, W.FIELD_X_INIT)[0] - ep.x_b0)) <= FP32_TOL
        if s1 == W.ADAPT_TR_INIT:
            ctx.continue_(st, 1)
            log = ctx.log(st)
            ep.advance(1, forced=[r["rr_accept"] for r in log])
            n_accept += sum(r["rr_accept"] for r in log)
        s2 = ctx.adapt(st, real)[0]
        o2 = ep.adapt(real[0], 0, None)
        seq_gpu += [int(s1), int(s2)]
        seq_or += [o1, o2]
        n = K - int(ctx.read(st, W.FIELD_META)[0][0])
        ctx.continue_(st, n, act)
        log = ctx.log(st)
        ep.advance(n, forced=[r["rr_accept"] for r in log])
        n_accept += sum(r["rr_accept"] for r in log)
        for k in range(K - n, K):
            assert _rel_l2(ctx.read(st, W.FIELD_V_STEP, k)[0], ep.vhist[k]) <= FP32_TOL
        assert np.max(np.abs(act[0] - ep.actions())) <= FP32_TOL
    assert seq_gpu == seq_or
    assert W.ADAPT_REBIND_ACCEPT in seq_gpu and W.ADAPT_REBIND_RESTART in seq_gpu
    assert n_accept > 0   # the injection path ran with multi-block probe sums
    ctx.close()
