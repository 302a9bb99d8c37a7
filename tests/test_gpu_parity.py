"""End-to-end parity of the CUDA path (called through the C ABI) with the CPU oracle.

Tolerances (stated for the method in fp32 and bf16):
  fp32 precision mode: per-step velocity relative L2 <= 1e-4, final actions max-abs <= 1e-4;
  bf16 precision mode: per-step velocity relative L2 <= 2e-2 (oracle evaluated at the GPU's
  latent of that step), final actions max-abs <= 5e-2 (oracle run free);
  index work (which slot a remapped value comes from, which slots get fresh noise): bit-exact.
Residual-Rescaling decisions are floating-point threshold tests; the oracle replays the GPU's
decision and asserts agreement whenever the oracle's own margin exceeds 1e-3.
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


def rel_l2(a, b):
    a = np.asarray(a, dtype=np.float64).ravel()
    b = np.asarray(b, dtype=np.float64).ravel()
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


class Run:
    def __init__(self, name, batch=1, **over):
        self.cfg = I.get_config(name, **over)
        self.cfg["batch"] = batch
        self.Wd = I.make_weights(self.cfg)
        self.flat = I.flatten_weights(self.Wd)
        self.ocfg = O.OracleConfig.from_dict(self.cfg)
        self.K = self.cfg["n_steps"]
        self.sig = O.schedule(self.K, self.cfg["sched_shift"])
        self.ctx = W.Context(self.cfg, self.flat)
        self.acts = (self.cfg["n_action"], self.cfg["action_dim"])

    def actions(self, B):
        return np.zeros((B,) + self.acts, np.float32)


def forced(log, ep=0):
    return [r["rr_accept"] for r in log if r["episode"] == ep]


def teacher_forced(run, ctx, st, log, obs, layer=None, ep=0):
    """Oracle velocity at each GPU latent of the latest call, replaying the GPU's RR decision."""
    pairs = []
    for rec in (r for r in log if r["episode"] == ep):
        k = rec["stage"]
        x = ctx.read(st, W.FIELD_X_STAGE, k)[ep]
        if run.ocfg.rr_enabled:
            v, layer, orec = O.velocity_rr(run.Wd, run.ocfg, x, obs, run.sig[k], layer, True,
                                           rec["rr_accept"] if rec["rr_attempt"] else None)
            assert orec.rr_attempt == rec["rr_attempt"]
        else:
            v = O.velocity(run.Wd, run.ocfg, x, obs, run.sig[k])
        pairs.append((ctx.read(st, W.FIELD_V_STEP, k)[ep], v))
    return pairs, layer


def _cold_then_warm(run, vel_tol, act_tol, teacher=False):
    cfg, K = run.cfg, run.K
    obs = I.make_obs(cfg, 1)
    noise = I.make_noise(cfg, 1)
    obs2 = I.make_obs(cfg, 1, seed=3)
    eps = I.make_fresh_eps(cfg, 1, 0)
    ctx = run.ctx
    st = ctx.state(1)
    act = run.actions(1)
    ctx.sample_cold(st, obs, noise, K, act)
    log1 = ctx.log(st)
    assert [r["stage"] for r in log1] == list(range(K))
    if teacher:
        pairs, layer = teacher_forced(run, ctx, st, log1, obs[0])
        for g, o in pairs:
            assert rel_l2(g, o) <= vel_tol
    ep = O.OracleEpisode(run.Wd, run.ocfg)
    ep.sample_cold(obs[0], noise[0], K, forced=forced(log1))
    if not teacher:
        for k in range(K):
            assert rel_l2(ctx.read(st, W.FIELD_V_STEP, k)[0], ep.vhist[k]) <= vel_tol
    assert np.max(np.abs(act[0] - ep.actions())) <= act_tol

    b0 = cfg["tr_entry_stage"]
    status = ctx.adapt(st, obs2, shift=cfg["shift"], fresh_noise=eps)
    assert status[0] == ep.adapt(obs2[0], cfg["shift"], eps[0]) == O.ADAPT_TR_INIT
    assert np.max(np.abs(ctx.read(st, W.FIELD_X_INIT)[0] - ep.x_b0)) <= act_tol
    ctx.continue_(st, K - b0, act)
    log2 = ctx.log(st)
    assert [r["stage"] for r in log2] == list(range(b0, K))
    if teacher:
        pairs, _ = teacher_forced(run, ctx, st, log2, obs2[0], layer)
        for g, o in pairs:
            assert rel_l2(g, o) <= vel_tol
    ep.advance(K - b0, forced=forced(log2))
    if not teacher:
        for k in range(b0, K):
            assert rel_l2(ctx.read(st, W.FIELD_V_STEP, k)[0], ep.vhist[k]) <= vel_tol
    assert np.max(np.abs(act[0] - ep.actions())) <= act_tol
    return log1 + log2


def test_tiny_fp32_cold_then_warm(wamlib):
    _cold_then_warm(Run("tiny"), FP32_TOL, FP32_TOL)


def test_tiny_fp32_residual_rescaling(wamlib):
    run = Run("tiny_rr")
    log = _cold_then_warm(run, FP32_TOL, FP32_TOL)
    assert sum(r["rr_attempt"] for r in log) == len(log) - 1
    st = run.ctx.stats()
    assert st["n_attempt"] == len(log) - 1 and st["b_dense"] == len(log) * 6


SMALL_BF16 = dict(n_layers=4, d_model=128, n_heads=2, n_obs=32, n_video=96, n_action=8, action_dim=7,
                  n_steps=6, precision="bf16", rr_policy=1, rr_q=1, rr_s=2, rr_e=3,
                  tr_entry_stage=3, tr_retain_stage=-1, shift=2)


def test_small_bf16_teacher_forced_and_free_running(wamlib):
    _cold_then_warm(Run("tiny", **SMALL_BF16), BF16_VEL_TOL, BF16_ACT_TOL, teacher=True)


def test_small_bf16_video_fresh_mode_and_shifted_schedule(wamlib):
    run = Run("tiny", **dict(SMALL_BF16, tr_video_mode=1, sched_shift=5.0, rr_policy=0))
    _cold_then_warm(run, BF16_VEL_TOL, BF16_ACT_TOL, teacher=True)


def test_latency_config_full_size(wamlib):
    """12 blocks, d=768, 1296 tokens, 10 bf16 steps: every step teacher-forced, then free-running
    final actions."""
    run = Run("latency")
    cfg, K = run.cfg, run.K
    obs = I.make_obs(cfg, 1)
    noise = I.make_noise(cfg, 1)
    st = run.ctx.state(1)
    act = run.actions(1)
    run.ctx.sample_cold(st, obs, noise, K, act)
    log = run.ctx.log(st)
    pairs, _ = teacher_forced(run, run.ctx, st, log, obs[0])
    errs = [rel_l2(g, o) for g, o in pairs]
    assert max(errs) <= BF16_VEL_TOL, errs
    ep = O.OracleEpisode(run.Wd, run.ocfg)
    ep.sample_cold(obs[0], noise[0], K, forced=forced(log))
    assert np.max(np.abs(act[0] - ep.actions())) <= BF16_ACT_TOL


# ------------------------------------------------------------------ Trajectory Remapping
def _finished_state(run, B, x_bar, x_r, r):
    st = run.ctx.state(B)
    K = run.K
    run.ctx.write(st, W.FIELD_X_STAGE, x_bar, index=K)
    run.ctx.write(st, W.FIELD_X_STAGE, x_r, index=r)
    meta = np.zeros((B, 8), np.int32)
    meta[:, 0] = K      # stage
    meta[:, 4] = 1      # finished
    run.ctx.write(st, W.FIELD_META, meta)
    return st


def test_tr_slot_indices_are_bit_exact(wamlib):
    run = Run("tiny", batch=4)
    cfg, K, T = run.cfg, run.K, run.ctx.T
    B = 4
    x_bar = np.tile(np.arange(T, dtype=np.float32), (B, 1)) + 1000 * np.arange(B)[:, None]
    eps = -1.0 - np.tile(np.arange(T, dtype=np.float32), (B, 1))
    shifts = np.array([0, 1, 3, cfg["n_action"] + 2], np.int32)
    r = cfg["tr_entry_stage"]
    st = _finished_state(run, B, x_bar, x_bar, r)     # x^r == x_bar: zero direction
    status = run.ctx.adapt(st, I.make_obs(cfg, B), shift=shifts, fresh_noise=eps)
    assert list(status) == [W.ADAPT_TR_INIT] * B
    got = run.ctx.read(st, W.FIELD_X_INIT)
    for b in range(B):
        want = O.tr_remap(run.ocfg, x_bar[b], x_bar[b], run.sig[r], run.sig[r], int(shifts[b]), eps[b])
        assert np.array_equal(got[b], want.astype(np.float32))


def test_tr_values_match_oracle(wamlib):
    for mode in (0, 1):
        run = Run("tiny", batch=2, tr_video_mode=mode, tr_retain_stage=5, tr_entry_stage=3)
        cfg, K, T = run.cfg, run.K, run.ctx.T
        rng = np.random.default_rng(mode)
        x_bar = rng.standard_normal((2, T)).astype(np.float32)
        x_r = rng.standard_normal((2, T)).astype(np.float32)
        eps = rng.standard_normal((2, T)).astype(np.float32)
        st = _finished_state(run, 2, x_bar, x_r, 5)
        run.ctx.adapt(st, I.make_obs(cfg, 2), shift=[2, 0], fresh_noise=eps)
        got = run.ctx.read(st, W.FIELD_X_INIT)
        for b, s in enumerate((2, 0)):
            want = O.tr_remap(run.ocfg, x_bar[b], x_r[b], run.sig[5], run.sig[3], s, eps[b])
            assert np.allclose(got[b], want, rtol=2e-7, atol=1e-7)


def test_invariant_zero_shift_identity_normaliser_equals_plain_continuation(wamlib):
    run = Run("tiny", tr_normalize=0, tr_entry_stage=4)
    cfg, K = run.cfg, run.K
    obs, noise = I.make_obs(cfg, 1), I.make_noise(cfg, 1)
    st = run.ctx.state(1)
    a1, a2 = run.actions(1), run.actions(1)
    run.ctx.sample_cold(st, obs, noise, K, a1)
    x4 = run.ctx.read(st, W.FIELD_X_STAGE, 4)
    run.ctx.adapt(st, obs, shift=0, fresh_noise=I.make_fresh_eps(cfg, 1, 0))
    assert np.allclose(run.ctx.read(st, W.FIELD_X_INIT), x4, rtol=1.2e-7, atol=0)
    run.ctx.continue_(st, K - 4, a2)
    assert np.allclose(a2, a1, atol=1e-6)


def test_invariant_empty_target_set_equals_cold(wamlib):
    run = Run("tiny", tr_video_mode=1, tr_entry_stage=0)
    cfg, K = run.cfg, run.K
    obs, obs2 = I.make_obs(cfg, 1), I.make_obs(cfg, 1, seed=5)
    eps = I.make_fresh_eps(cfg, 1, 1)
    st = run.ctx.state(1)
    a_warm, a_cold = run.actions(1), run.actions(1)
    run.ctx.sample_cold(st, obs, I.make_noise(cfg, 1), K)
    run.ctx.adapt(st, obs2, shift=cfg["n_action"], fresh_noise=eps)
    run.ctx.continue_(st, K, a_warm)
    st2 = run.ctx.state(1)
    run.ctx.sample_cold(st2, obs2, eps, K, a_cold)
    assert np.array_equal(a_warm, a_cold)


# ------------------------------------------------------------------ Observation Rebinding
def test_rebinding_kappa_sequence_and_restart_match_oracle(wamlib):
    run = Run("tiny")
    cfg, K = run.cfg, run.K
    proc = I.ObsProcess(cfg, 1, seed=7)
    obs = proc.obs.copy()
    st = run.ctx.state(1)
    act = run.actions(1)
    run.ctx.sample_cold(st, obs, I.make_noise(cfg, 1), K, act)
    ep = O.OracleEpisode(run.Wd, run.ocfg)
    ep.sample_cold(obs[0], I.make_noise(cfg, 1)[0], K)
    seq_gpu, seq_or = [], []
    for t in range(7):
        pred = proc.predicted()
        real = proc.step()
        if t == 5:
            real = real + 3.0            # a surprise: the prediction fails the check
        eps = I.make_fresh_eps(cfg, 1, t)
        s1 = run.ctx.adapt(st, pred, shift=1, fresh_noise=eps)[0]
        o1 = ep.adapt(pred[0], 1, eps[0])
        if s1 == W.ADAPT_TR_INIT:
            run.ctx.continue_(st, 1)
            ep.advance(1)
        s2 = run.ctx.adapt(st, real)[0]
        o2 = ep.adapt(real[0], 0, None)
        seq_gpu += [int(s1), int(s2)]
        seq_or += [o1, o2]
        meta = run.ctx.read(st, W.FIELD_META)[0]
        run.ctx.continue_(st, K - int(meta[0]), act)
        ep.advance(K - ep.stage)
        assert np.max(np.abs(act[0] - ep.actions())) <= FP32_TOL
    assert seq_gpu == seq_or
    assert W.ADAPT_REBIND_RESTART in seq_gpu and W.ADAPT_TR_INIT_NO_PREFIX in seq_gpu
    s = run.ctx.stats()
    assert (s["n_start"], s["n_bind"], s["n_noninitial"]) == (ep.stats.n_start, ep.stats.n_bind,
                                                              ep.stats.n_noninitial)


# ------------------------------------------------------------------ batching
def test_mixed_cold_and_warm_batch_matches_per_episode_oracle(wamlib):
    run = Run("tiny_rr", batch=4)
    cfg, K = run.cfg, run.K
    B = 4
    obs = I.make_obs(cfg, B)
    noise = I.make_noise(cfg, B)
    st = run.ctx.state(B)
    run.ctx.sample_cold(st, obs, noise, K)
    log_cold = run.ctx.log(st)
    eps = I.make_fresh_eps(cfg, B, 0)
    obs2 = I.make_obs(cfg, B, seed=11)
    entry = np.array([W.ENTRY_COLD, W.ENTRY_COLD, K - 2, K - 2], np.int32)
    status = run.ctx.adapt(st, obs2, shift=[0, 0, 1, 3], entry=entry, fresh_noise=eps)
    assert list(status) == [W.ADAPT_COLD_INIT] * 2 + [W.ADAPT_TR_INIT] * 2
    act = run.actions(B)
    run.ctx.continue_(st, [K, K, 2, 2], act)
    log_mix = run.ctx.log(st)
    for b in range(B):
        ep = O.OracleEpisode(run.Wd, run.ocfg)
        ep.sample_cold(obs[b], noise[b], K, forced=forced(log_cold, b))
        if entry[b] == W.ENTRY_COLD:
            ep.adapt(obs2[b], 0, eps[b], entry_stage=O.ENTRY_COLD)
            ep.advance(K, forced=forced(log_mix, b))
        else:
            ep.adapt(obs2[b], [0, 0, 1, 3][b], eps[b], entry_stage=K - 2)
            ep.advance(2, forced=forced(log_mix, b))
        assert np.max(np.abs(act[b] - ep.actions())) <= FP32_TOL


# ------------------------------------------------------------------ failures are reported
def test_errors_are_status_codes(wamlib):
    run = Run("tiny")
    cfg, K = run.cfg, run.K
    st = run.ctx.state(1)
    with pytest.raises(W.WamError) as e:
        run.ctx.continue_(st, 1)                  # never started
    assert e.value.code == 2
    run.ctx.sample_cold(st, I.make_obs(cfg, 1), I.make_noise(cfg, 1), K)
    with pytest.raises(W.WamError) as e:
        run.ctx.continue_(st, 1)                  # finished replan must be adapted first
    assert e.value.code == 2
    run.ctx.adapt(st, I.make_obs(cfg, 1), shift=1, fresh_noise=I.make_fresh_eps(cfg, 1, 0))
    with pytest.raises(W.WamError) as e:
        run.ctx.adapt(st, I.make_obs(cfg, 1), shift=2)   # a rebind takes no shift
    assert e.value.code == 2
    with pytest.raises(W.WamError) as e:
        run.ctx.continue_(st, K)                  # past the last stage
    assert e.value.code == 1
    with pytest.raises(W.WamError) as e:
        run.ctx.adapt(st, I.make_obs(cfg, 1), shift=-1)
    assert e.value.code == 1
