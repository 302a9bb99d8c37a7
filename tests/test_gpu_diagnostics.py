"""App. E state-continuity diagnostics computed by the library against the oracle: latent
similarity across consecutive replans, action RMSE, the per-layer hidden-state change of the full
forward at an episode's pending stage, and the residual-reuse output error E_out."""
import numpy as np
import pytest
import torch

from oracle import wam_oracle as O
from paper_2609_34608_gb300 import inputs as I
from paper_2609_34608_gb300 import wam as W

pytestmark = pytest.mark.gpu

SMALL_BF16 = dict(n_layers=4, d_model=128, n_heads=2, n_obs=32, n_video=96, n_action=8, action_dim=7,
                  n_steps=6, precision="bf16", rr_policy=1, rr_q=1, rr_s=2, rr_e=3,
                  tr_entry_stage=3, tr_retain_stage=-1, shift=2)


def test_similarity_and_action_rmse_vs_oracle(wamlib):
    cfg = I.get_config("tiny_rr")
    ctx = W.Context(cfg, I.flatten_weights(I.make_weights(cfg)))
    rng = np.random.default_rng(21)
    a = rng.standard_normal(4099).astype(np.float32)
    b = (0.8 * a + 0.3 * rng.standard_normal(4099)).astype(np.float32)
    for x, y in ((a, b), (torch.from_numpy(a).cuda(), torch.from_numpy(b).cuda())):   # host and device inputs
        cos, rel = ctx.diag_similarity(x, y)
        ocos, orel = O.latent_similarity(a, b)
        assert cos == pytest.approx(ocos, rel=1e-12) and rel == pytest.approx(orel, rel=1e-12)
    assert ctx.diag_similarity(a, a) == (pytest.approx(1.0, abs=1e-15), 0.0)
    acts_a = rng.standard_normal((16, 7)).astype(np.float32)
    acts_b = rng.standard_normal((16, 7)).astype(np.float32)
    assert ctx.diag_action_rmse(acts_a, acts_b, 6) == pytest.approx(O.action_rmse(acts_a, acts_b, dims=6), rel=1e-12)
    with pytest.raises(W.WamError):
        ctx.diag_action_rmse(acts_a, acts_b, 8)
    ctx.close()


@pytest.mark.parametrize("precision", ["fp32", "bf16"])
def test_layer_deltas_vs_oracle(wamlib, precision):
    cfg = I.get_config("tiny_rr", batch=2) if precision == "fp32" else I.get_config("tiny", batch=2, **SMALL_BF16)
    Wd = I.make_weights(cfg)
    ctx = W.Context(cfg, I.flatten_weights(Wd))
    st = ctx.state(2)
    obs = I.make_obs(cfg, 2)
    ctx.sample_cold(st, obs, I.make_noise(cfg, 2), 2)      # two of K steps: stage 2 pending
    x_before = ctx.read(st, W.FIELD_X).copy()
    ocfg = O.OracleConfig.from_dict(cfg)
    sig = O.schedule(cfg["n_steps"], cfg["sched_shift"])
    for ep in range(2):
        got = ctx.diag_layer_deltas(st, ep)
        want = O.layer_deltas(Wd, ocfg, x_before[ep], obs[ep], sig[2])
        tol = 1e-5 if precision == "fp32" else 3e-2
        assert np.allclose(got, want, rtol=tol, atol=0.0), (got, want)
    assert np.array_equal(ctx.read(st, W.FIELD_X), x_before)    # the state is left untouched
    ctx.sample_cold(st, obs, I.make_noise(cfg, 2), cfg["n_steps"])
    with pytest.raises(W.WamError):                               # finished: no pending stage
        ctx.diag_layer_deltas(st, 0)
    ctx.close()


@pytest.mark.parametrize("precision", ["fp32", "bf16"])
def test_reuse_error_vs_oracle(wamlib, precision):
    """App. E E_out at a pending stage against the oracle fed the GPU's retained layer state."""
    cfg = I.get_config("tiny_rr", batch=2) if precision == "fp32" else I.get_config("tiny", batch=2, **SMALL_BF16)
    Wd = I.make_weights(cfg)
    ctx = W.Context(cfg, I.flatten_weights(Wd))
    st = ctx.state(2)
    obs = I.make_obs(cfg, 2)
    ctx.sample_cold(st, obs, I.make_noise(cfg, 2), 3)      # three of K steps: RR state retained
    x_before = ctx.read(st, W.FIELD_X).copy()
    pa, ra = ctx.read(st, W.FIELD_RR_P).copy(), ctx.read(st, W.FIELD_RR_R).copy()
    ocfg = O.OracleConfig.from_dict(cfg)
    sig = O.schedule(cfg["n_steps"], cfg["sched_shift"])
    for ep in range(2):
        err, alphas = ctx.diag_reuse_error(st, ep)
        layer = O.LayerState(p_a=pa[ep].astype(np.float64), R_a=ra[ep].astype(np.float64))
        want, want_alpha = O.reuse_output_error(Wd, ocfg, x_before[ep], obs[ep], sig[3], layer)
        if precision == "fp32":
            assert err == pytest.approx(want, rel=1e-3, abs=1e-5)
            assert alphas == pytest.approx(want_alpha, rel=1e-4)
        else:
            assert err == pytest.approx(want, abs=3e-2)
            assert alphas == pytest.approx(want_alpha, abs=2e-2)
        assert err > 0.0
    assert np.array_equal(ctx.read(st, W.FIELD_X), x_before)    # the state is left untouched
    assert np.array_equal(ctx.read(st, W.FIELD_RR_P), pa) and np.array_equal(ctx.read(st, W.FIELD_RR_R), ra)
    ctx.sample_cold(st, obs, I.make_noise(cfg, 2), cfg["n_steps"])
    with pytest.raises(W.WamError) as e:                          # finished: no pending stage
        ctx.diag_reuse_error(st, 0)
    assert e.value.code == 2
    ctx.close()


def test_reuse_error_needs_a_retained_state_and_rr_boundaries(wamlib):
    cfg = I.get_config("tiny_rr")
    ctx = W.Context(cfg, I.flatten_weights(I.make_weights(cfg)))
    st = ctx.state(1)
    ctx.adapt(st, I.make_obs(cfg, 1), entry=W.ENTRY_COLD, fresh_noise=I.make_noise(cfg, 1))
    with pytest.raises(W.WamError) as e:                          # stage 0, nothing retained yet
        ctx.diag_reuse_error(st, 0)
    assert e.value.code == 2
    ctx.close()
    cfg = I.get_config("tiny")                                    # two blocks: no RR boundaries
    ctx = W.Context(cfg, I.flatten_weights(I.make_weights(cfg)))
    st = ctx.state(1)
    ctx.sample_cold(st, I.make_obs(cfg, 1), I.make_noise(cfg, 1), 2)
    with pytest.raises(W.WamError) as e:
        ctx.diag_reuse_error(st, 0)
    assert e.value.code == 1
    ctx.close()
