"""Independent execution (§3.3; App. B.1-B.2, the Fast-WAM-IDM profile): a video-only and an
action-only model, each with its own replan state, schedule, TR stages and RR decisions,
advanced together by wam_continue_many on two streams.

Parity against the CPU oracle (one OracleEpisode per branch) with the tolerances of the joint
tests: fp32 per-step velocity relative L2 <= 1e-4; bf16 teacher-forced velocity <= 2e-2 and
free-running final actions max-abs <= 5e-2; RR decisions replayed into the oracle, which must
agree whenever its margin exceeds 1e-3.
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

SMALL_BF16 = dict(n_layers=4, n_heads=2, n_obs=32, precision="bf16", rr_q=1, rr_s=2, rr_e=3)


def rel_l2(a, b):
    a = np.asarray(a, dtype=np.float64).ravel()
    b = np.asarray(b, dtype=np.float64).ravel()
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


class Branch:
    """One branch model on its own stream, with its oracle counterpart."""

    def __init__(self, name, stream, **over):
        self.cfg = I.get_config(name, **over)
        self.Wd = I.make_weights(self.cfg)
        self.ocfg = O.OracleConfig.from_dict(self.cfg)
        self.K = self.cfg["n_steps"]
        self.sig = O.schedule(self.K, self.cfg["sched_shift"])
        self.stream = stream
        self.ctx = W.Context(self.cfg, I.flatten_weights(self.Wd), stream=stream.cuda_stream)
        self.st = self.ctx.state(1)
        self.ep = O.OracleEpisode(self.Wd, self.ocfg)
        self.tlayer = None  # RR layer state of the teacher-forced oracle evaluations
        # record slot of the model's single RR branch: 0 (obs + video rows) or 1 (action rows)
        self.slot = 0 if self.cfg["n_action"] == 0 else 1

    def stage(self):
        return int(self.ctx.read(self.st, W.FIELD_META)[0][0])

    def out(self):
        c = self.cfg
        if c["n_action"] == 0:
            return np.zeros((1, c["n_video"], c["video_dim"]), np.float32)
        return np.zeros((1, c["n_action"], c["action_dim"]), np.float32)

    def check_call(self, stages, tol, teacher=False, obs=None):
        """Compare the latest call's per-step velocities and RR records with the oracle, then
        advance the oracle with the GPU's RR decisions."""
        log = self.ctx.log(self.st)
        assert [r["stage"] for r in log] == stages
        for r in log:
            other = 1 - self.slot
            assert r["alpha"][other] == r["cos"][other] == r["fit"][other] == 0.0
        forced = [r["rr_accept"] for r in log]
        if teacher:
            layer = self.tlayer
            for r in log:
                k = r["stage"]
                x = self.ctx.read(self.st, W.FIELD_X_STAGE, k)[0]
                v, layer, orec = O.velocity_rr(self.Wd, self.ocfg, x, obs, self.sig[k], layer, True,
                                               r["rr_accept"] if r["rr_attempt"] else None)
                assert orec.rr_attempt == r["rr_attempt"]
                assert rel_l2(self.ctx.read(self.st, W.FIELD_V_STEP, k)[0], v) <= tol
            self.tlayer = layer
        n0 = len(self.ep.records)
        self.ep.advance(len(stages), forced=forced)
        for r, orec in zip(log, self.ep.records[n0:]):
            assert orec.rr_attempt == r["rr_attempt"] and orec.rr_accept == r["rr_accept"]
            if r["rr_attempt"] and not teacher:
                (chk,) = orec.checks
                assert r["alpha"][self.slot] == pytest.approx(chk.alpha, rel=1e-3)
                assert r["cos"][self.slot] == pytest.approx(chk.cos, abs=1e-3)
                assert r["fit"][self.slot] == pytest.approx(chk.fit, abs=1e-3)
            if not teacher:
                k = r["stage"]
                assert rel_l2(self.ctx.read(self.st, W.FIELD_V_STEP, k)[0], self.ep.vhist[k]) <= tol
        return log


def _pair(prefix, **over):
    import torch
    vid = Branch(f"{prefix}_video", torch.cuda.Stream(), **over)
    act = Branch(f"{prefix}_action", torch.cuda.Stream(), **over)
    return vid, act


def _control_loop(vid, act, n_replans, tol, act_tol, teacher=False, concurrent=True):
    """Cold first replan of both branches, then closed-loop replans: the video branch runs its
    anticipatory prefix under the predicted observation, rebinds to the real one and finishes;
    the action branch remaps with the executed shift under the real observation and finishes
    concurrently.  Returns the per-replan outputs (video latent, actions)."""
    K = vid.K
    proc = I.ObsProcess(vid.cfg, 1, seed=21)
    obs = proc.obs.copy()
    outs = []
    for br, seed in ((vid, 1), (act, 2)):
        noise = I.make_noise(br.cfg, 1, seed=seed)
        br.ctx.sample_cold(br.st, obs, noise, K)
        br.ep.cold_init(obs[0], noise[0])
        br.tlayer = None
        br.check_call(list(range(K)), tol, teacher, obs[0])
    for t in range(n_replans):
        pred, real = proc.predicted(), proc.step()
        eps_v = I.make_fresh_eps(vid.cfg, 1, t)
        eps_a = I.make_fresh_eps(act.cfg, 1, 100 + t)
        s = int(vid.ctx.adapt(vid.st, pred, shift=0, fresh_noise=eps_v)[0])
        assert s == vid.ep.adapt(pred[0], 0, eps_v[0])
        b0 = vid.cfg["tr_entry_stage"]
        if s == W.ADAPT_TR_INIT:
            p = vid.cfg["prefix_steps"]
            vid.ctx.continue_(vid.st, p)
            vid.check_call(list(range(b0, b0 + p)), tol, teacher, pred[0])
        s2 = int(vid.ctx.adapt(vid.st, real)[0])
        assert s2 == vid.ep.adapt(real[0], 0, None)
        sa = int(act.ctx.adapt(act.st, real, shift=act.cfg["shift"], fresh_noise=eps_a)[0])
        assert sa == act.ep.adapt(real[0], act.cfg["shift"], eps_a[0]) == W.ADAPT_TR_INIT
        kv, ka = vid.stage(), act.stage()
        assert ka == act.cfg["tr_entry_stage"]
        v_out, a_out = vid.out(), act.out()
        calls = [(vid.ctx, vid.st, K - kv, None, v_out), (act.ctx, act.st, K - ka, a_out, None)]
        if concurrent:
            status = W.Context.continue_many(calls)
            assert list(status) == [0, 0]
        else:
            for c in calls:
                c[0].continue_(c[1], c[2], c[3], c[4])
        vid.check_call(list(range(kv, K)), tol, teacher, real[0])
        act.check_call(list(range(ka, K)), tol, teacher, real[0])
        assert np.max(np.abs(a_out[0] - act.ep.actions())) <= act_tol
        assert np.max(np.abs(v_out[0].ravel() - vid.ep.hist[K])) <= act_tol
        outs.append((v_out.copy(), a_out.copy()))
    return outs


def test_independent_branches_fp32_match_oracle(wamlib):
    vid, act = _pair("tiny")
    _control_loop(vid, act, 4, FP32_TOL, FP32_TOL)
    sv, sa = vid.ctx.stats(), act.ctx.stats()
    # each branch decided reuse on its own, at every step after its first full one
    assert sv["n_attempt"] == vid.ep.stats.n_attempt > 0
    assert sa["n_attempt"] == act.ep.stats.n_attempt > 0
    assert (sv["n_reuse"], sa["n_reuse"]) == (vid.ep.stats.n_reuse, act.ep.stats.n_reuse)
    assert (sv["n_start"], sv["n_bind"]) == (vid.ep.stats.n_start, vid.ep.stats.n_bind)
    assert sa["n_start"] == 0


def test_independent_branches_small_bf16_teacher_forced(wamlib):
    vid, act = _pair("tiny", **SMALL_BF16)
    _control_loop(vid, act, 2, BF16_VEL_TOL, BF16_ACT_TOL, teacher=True)


def test_continue_many_equals_separate_calls_bitwise(wamlib):
    runs = []
    for concurrent in (False, True):
        vid, act = _pair("tiny", **SMALL_BF16)
        runs.append(_control_loop(vid, act, 3, BF16_VEL_TOL, BF16_ACT_TOL, concurrent=concurrent))
    for (v0, a0), (v1, a1) in zip(*runs):
        assert np.array_equal(v0, v1) and np.array_equal(a0, a1)


def test_idm_action_model_full_size(wamlib):
    """The 12-block d=768 action model (256 obs + 16 action tokens): cold 10 steps and a warm
    replan entering stage 5 with the horizon shifted by 8, every step teacher-forced, then the
    free-running final actions."""
    import torch
    br = Branch("idm_action", torch.cuda.Stream())
    cfg, K = br.cfg, br.K
    obs, obs2 = I.make_obs(cfg, 1), I.make_obs(cfg, 1, seed=3)
    noise, eps = I.make_noise(cfg, 1), I.make_fresh_eps(cfg, 1, 0)
    a = br.out()
    br.ctx.sample_cold(br.st, obs, noise, K, a)
    br.ep.cold_init(obs[0], noise[0])
    br.check_call(list(range(K)), BF16_VEL_TOL, True, obs[0])
    assert np.max(np.abs(a[0] - br.ep.actions())) <= BF16_ACT_TOL
    assert int(br.ctx.adapt(br.st, obs2, shift=cfg["shift"], fresh_noise=eps)[0]) == W.ADAPT_TR_INIT
    br.ep.adapt(obs2[0], cfg["shift"], eps[0])
    b0 = cfg["tr_entry_stage"]
    # remapped slots are bit-exact in index: the shifted part comes from the retained slots
    assert np.max(np.abs(br.ctx.read(br.st, W.FIELD_X_INIT)[0] - br.ep.x_b0)) <= BF16_ACT_TOL
    br.ctx.continue_(br.st, K - b0, a)
    br.check_call(list(range(b0, K)), BF16_VEL_TOL, True, obs2[0])
    assert np.max(np.abs(a[0] - br.ep.actions())) <= BF16_ACT_TOL


def test_continue_many_rejects_bad_arguments(wamlib):
    vid, act = _pair("tiny")
    with pytest.raises(W.WamError) as e:
        W.Context.continue_many([(vid.ctx, vid.st, 1), (vid.ctx, vid.st, 1)])
    assert e.value.code == 1
    with pytest.raises(W.WamError) as e:
        W.Context.continue_many([(vid.ctx, act.st, 1)])
    assert e.value.code == 1
