"""Checkpoint / resume of the per-episode state through wam_state_read / wam_state_write: a state
exported mid-replan and imported into a fresh state continues bit-identically (same kernels,
same inputs), including the retained RR layer state and the remapped init."""
import numpy as np
import pytest

from paper_2609_34608_gb300 import inputs as I
from paper_2609_34608_gb300 import wam as W

pytestmark = pytest.mark.gpu


def _export(ctx, st, K):
    out = {(W.FIELD_X, 0): ctx.read(st, W.FIELD_X), (W.FIELD_X_INIT, 0): ctx.read(st, W.FIELD_X_INIT),
           (W.FIELD_OBS, 0): ctx.read(st, W.FIELD_OBS), (W.FIELD_RR_P, 0): ctx.read(st, W.FIELD_RR_P),
           (W.FIELD_RR_R, 0): ctx.read(st, W.FIELD_RR_R), (W.FIELD_META, 0): ctx.read(st, W.FIELD_META)}
    for k in range(K + 1):
        out[(W.FIELD_X_STAGE, k)] = ctx.read(st, W.FIELD_X_STAGE, k)
    for k in range(K):
        out[(W.FIELD_V_STEP, k)] = ctx.read(st, W.FIELD_V_STEP, k)
    return out


@pytest.mark.parametrize("precision", ["fp32", "bf16"])
def test_exported_state_resumes_bit_identically(wamlib, precision):
    over = {} if precision == "fp32" else dict(precision="bf16", n_heads=2, n_obs=32, n_video=96)
    cfg = I.get_config("tiny_rr", batch=2, **over)
    K, b0 = cfg["n_steps"], cfg["tr_entry_stage"]
    ctx = W.Context(cfg, I.flatten_weights(I.make_weights(cfg)))
    st = ctx.state(2)
    ctx.sample_cold(st, I.make_obs(cfg, 2), I.make_noise(cfg, 2), K)
    ctx.adapt(st, I.make_obs(cfg, 2, seed=5), shift=[1, 3], fresh_noise=I.make_fresh_eps(cfg, 2, 0))
    ctx.continue_(st, 2)                                   # mid-replan: stage b0 + 2 pending
    saved = _export(ctx, st, K)
    st2 = ctx.state(2)
    for (field, index), value in saved.items():           # META last: it is validated on write
        if field != W.FIELD_META:
            ctx.write(st2, field, value, index=index)
    ctx.write(st2, W.FIELD_META, saved[(W.FIELD_META, 0)])
    assert all(np.array_equal(ctx.read(st2, f, i), v) for (f, i), v in saved.items())
    a1 = np.zeros((2, cfg["n_action"], cfg["action_dim"]), np.float32)
    a2 = np.zeros_like(a1)
    ctx.continue_(st, K - b0 - 2, a1)
    ctx.continue_(st2, K - b0 - 2, a2)
    assert np.array_equal(a1, a2)
    l1, l2 = ctx.log(st), ctx.log(st2)
    assert [(r["stage"], r["rr_attempt"], r["rr_accept"]) for r in l1] == \
        [(r["stage"], r["rr_attempt"], r["rr_accept"]) for r in l2]
    assert any(r["rr_attempt"] for r in l1)               # the retained layer state was used
    ctx.close()
