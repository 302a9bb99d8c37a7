"""The allocation-free remap entry point (wam_tr_remap_static) against the context path.

Callers that cannot allocate device memory (a control loop that forbids allocation after
start-up, or a host runtime that owns all device memory) remap through wam_tr_remap_static,
whose scratch is a fixed array inside the library.  Its output must match the remap that
wam_adapt_state computes for the same finished trajectories, on two calls in a row (the second
call sees the first call's leftovers in the shared array).  This file is collected last.
"""
import numpy as np
import pytest
import torch

from oracle import wam_oracle as O
from paper_2609_34608_gb300 import inputs as I
from paper_2609_34608_gb300 import wam as W

pytestmark = pytest.mark.gpu


def _context_remap(ctx, cfg, x_bar, x_r, eps, shift, r, b0):
    B = x_bar.shape[0]
    st = ctx.state(B)
    ctx.write(st, W.FIELD_X_STAGE, x_bar, index=cfg["n_steps"])
    ctx.write(st, W.FIELD_X_STAGE, x_r, index=r)
    meta = np.zeros((B, 8), np.int32)
    meta[:, 0] = cfg["n_steps"]
    meta[:, 4] = 1
    ctx.write(st, W.FIELD_META, meta)
    status = ctx.adapt(st, I.make_obs(cfg, B), shift=shift, entry=b0, fresh_noise=eps)
    assert list(status) == [W.ADAPT_TR_INIT] * B
    out = ctx.read(st, W.FIELD_X_INIT)
    st.close()
    return out


@pytest.mark.parametrize("video_mode", [0, 1])
def test_static_scratch_remap_matches_context_remap(wamlib, video_mode):
    B, r, b0 = 3, 5, 3
    cfg = I.get_config("tiny", batch=B, tr_retain_stage=r, tr_entry_stage=b0, tr_video_mode=video_mode)
    ctx = W.Context(cfg, I.flatten_weights(I.make_weights(cfg)))
    sig = O.schedule(cfg["n_steps"], cfg["sched_shift"])
    T = ctx.T
    dev = torch.device("cuda")
    for call, shift in enumerate((2, 0)):
        rng = np.random.default_rng(100 + call)
        x_bar, x_r, eps = (rng.standard_normal((B, T)).astype(np.float32) * (call + 1) for _ in range(3))
        expect = _context_remap(ctx, cfg, x_bar, x_r, eps, shift, r, b0)
        out = torch.full((B, T), float("nan"), device=dev)
        W.tr_remap_static(torch.from_numpy(x_bar).to(dev), torch.from_numpy(x_r).to(dev),
                          torch.from_numpy(eps).to(dev), out, B, cfg["n_video"], cfg["video_dim"],
                          cfg["n_action"], cfg["action_dim"], shift, sig[r], sig[b0], 1, video_mode)
        torch.cuda.synchronize()
        assert np.allclose(out.cpu().numpy(), expect, rtol=2e-7, atol=1e-7)
    ctx.close()


def test_static_scratch_rejects_oversized_batches(wamlib):
    dev = torch.device("cuda")
    x = torch.zeros((1, 4), device=dev)
    with pytest.raises(W.WamError) as e:
        # 5000 episodes x 2 branches x 1 chunk > 8192 partial sums
        W.tr_remap_static(x, x, x, x, 5000, 1, 2, 1, 2, 0, 0.5, 0.5)
    assert e.value.code == 6
