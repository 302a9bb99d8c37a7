"""The allocation-free remap entry point (wam_tr_remap_static).

Callers that cannot allocate device memory (a control loop that forbids allocation after
start-up, or a host runtime that owns all device memory) remap through wam_tr_remap_static,
whose scratch is a fixed array inside the library.  Its output must be bit-identical to the
remap that wam_adapt_state computes for the same finished trajectories, and within one float32
ulp of the float64 oracle's remap, on two calls in a row (the second call sees the first call's
leftovers in the shared array).  The trajectories span several 2048-value reduction blocks per
branch.  This file is collected last.
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
    if eps is None:
        eps = np.zeros_like(x_bar)  # the context path always takes a noise buffer
    status = ctx.adapt(st, I.make_obs(cfg, B), shift=shift, entry=b0, fresh_noise=eps)
    assert list(status) == [W.ADAPT_TR_INIT] * B
    out = ctx.read(st, W.FIELD_X_INIT)
    st.close()
    return out


def _within_one_ulp(out, ref):
    ref = np.asarray(ref, np.float64)
    ulp = np.spacing(np.abs(ref).astype(np.float32)).astype(np.float64)
    return np.all(np.abs(out.astype(np.float64) - ref) <= ulp)


# (n_video, n_action): one reduction block per branch, and several (video 300 x 16 = 4800
# values = 3 blocks of 2048, action 300 x 7 = 2100 values = 2 blocks)
@pytest.mark.parametrize("n_video,n_action", [(32, 8), (300, 300)])
@pytest.mark.parametrize("video_mode,normalize", [(0, 1), (1, 1), (0, 0)])
def test_static_scratch_remap_matches_context_remap_and_oracle(wamlib, n_video, n_action, video_mode, normalize):
    B, r, b0 = 3, 5, 3
    cfg = I.get_config("tiny", batch=B, n_video=n_video, n_action=n_action, tr_retain_stage=r,
                       tr_entry_stage=b0, tr_video_mode=video_mode, tr_normalize=normalize)
    ocfg = O.OracleConfig.from_dict(cfg)
    ctx = W.Context(cfg, I.flatten_weights(I.make_weights(cfg)))
    sig = O.schedule(cfg["n_steps"], cfg["sched_shift"])
    T = ctx.T
    dev = torch.device("cuda")
    # the second call takes no noise buffer where no slot needs one (shift 0, video remapped)
    calls = [(2, True), (0, video_mode == 1)]
    for call, (shift, with_eps) in enumerate(calls):
        rng = np.random.default_rng(100 + call)
        x_bar, x_r, eps = (rng.standard_normal((B, T)).astype(np.float32) * (call + 1) for _ in range(3))
        x_r[1] = x_bar[1]  # a zero direction: d = 0 when normalised
        eps_in = eps if with_eps else None
        expect = _context_remap(ctx, cfg, x_bar, x_r, eps_in, shift, r, b0)
        out = torch.full((B, T), float("nan"), device=dev)
        W.tr_remap_static(torch.from_numpy(x_bar).to(dev), torch.from_numpy(x_r).to(dev),
                          torch.from_numpy(eps).to(dev) if with_eps else None, out, B, cfg["n_video"],
                          cfg["video_dim"], cfg["n_action"], cfg["action_dim"], shift, sig[r], sig[b0],
                          normalize, video_mode)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        assert np.array_equal(got, expect)
        for b in range(B):
            ref = O.tr_remap(ocfg, x_bar[b], x_r[b], sig[r], sig[b0], shift, eps[b])
            assert _within_one_ulp(got[b], ref)
    ctx.close()


def test_static_scratch_rejects_oversized_batches(wamlib):
    dev = torch.device("cuda")
    x = torch.zeros((1, 4), device=dev)
    with pytest.raises(W.WamError) as e:
        # 5000 episodes x 2 branches x 1 chunk > 8192 partial sums
        W.tr_remap_static(x, x, x, x, 5000, 1, 2, 1, 2, 0, 0.5, 0.5)
    assert e.value.code == 6
    with pytest.raises(W.WamError) as e:
        # a trajectory longer than 2^31 - 1 values is rejected before any launch
        W.tr_remap_static(x, x, x, x, 1, 1 << 20, 1 << 12, 1, 2, 0, 0.5, 0.5)
    assert e.value.code == 1
