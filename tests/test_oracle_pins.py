"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test ties one oracle function to something other than itself: a value printed in the
paper (tests/golden/), a closed form, an invariant, a library routine computing the same
textbook operation, or brute force on tiny inputs.
"""
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as TF

from oracle import wam_oracle as O
from paper_2609_34608_gb300 import inputs as I
from tests.conftest import micro_config

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


def _setup(cfg_dict, seed=0, std=0.02):
    W = I.make_weights(cfg_dict, seed=seed, std=std)
    return W, O.OracleConfig.from_dict(cfg_dict)


# ----------------------------------------------------------------------------- schedule
def test_schedule_matches_fastwam_values_printed_in_paper():
    for n_steps, shift, stage, sigma in _golden("fastwam_schedule.txt"):
        sig = O.schedule(int(n_steps), float(shift))
        assert round(float(sig[int(stage)]), 5) == pytest.approx(float(sigma), abs=0.5e-5)


def test_linear_schedule_endpoints():
    sig = O.schedule(8, 1.0)
    assert sig[0] == 1.0 and sig[-1] == 0.0
    assert np.allclose(np.diff(sig), -1.0 / 8)


# ----------------------------------------------------------------------------- Euler
@pytest.mark.parametrize("shift", [1.0, 5.0])
def test_euler_constant_field_closed_form(shift):
    rng = np.random.default_rng(3)
    x0, v = rng.standard_normal(11), rng.standard_normal(11)
    xs = O.euler_integrate(x0, O.schedule(10, shift), lambda x, s: v)
    # sum of (sigma_{k+1} - sigma_k) telescopes to sigma_K - sigma_0 = -1
    assert np.allclose(xs[-1], x0 - v, atol=1e-14)


def test_euler_linear_field_product_form():
    sig = O.schedule(6, 1.0)
    a = 0.7
    xs = O.euler_integrate(np.array([2.0]), sig, lambda x, s: a * x)
    expect = 2.0 * np.prod([1.0 + a * (sig[k + 1] - sig[k]) for k in range(6)])
    assert xs[-1][0] == pytest.approx(expect, rel=1e-14)


# ----------------------------------------------------------------------------- attention
def _attention_bruteforce(q, k, v, n_heads):
    n, d = len(q), len(q[0])
    dh = d // n_heads
    out = [[0.0] * d for _ in range(n)]
    for h in range(n_heads):
        c0 = h * dh
        for i in range(n):
            logits = []
            for j in range(n):
                s = 0.0
                for c in range(dh):
                    s += q[i][c0 + c] * k[j][c0 + c]
                logits.append(s / math.sqrt(dh))
            mx = max(logits)
            w = [math.exp(x - mx) for x in logits]
            z = sum(w)
            for c in range(dh):
                out[i][c0 + c] = sum(w[j] * v[j][c0 + c] for j in range(n)) / z
    return np.array(out)


def test_attention_vs_bruteforce_loops():
    rng = np.random.default_rng(0)
    q, k, v = (rng.standard_normal((7, 8)) for _ in range(3))
    ref = _attention_bruteforce(q.tolist(), k.tolist(), v.tolist(), 2)
    assert np.allclose(O.attention(q, k, v, 2), ref, atol=1e-13)


def test_attention_vs_torch_sdpa():
    rng = np.random.default_rng(1)
    n, d, H = 13, 24, 3
    q, k, v = (rng.standard_normal((n, d)) for _ in range(3))
    t = lambda a: torch.from_numpy(a).reshape(n, H, d // H).permute(1, 0, 2)
    ref = TF.scaled_dot_product_attention(t(q), t(k), t(v)).permute(1, 0, 2).reshape(n, d)
    assert np.allclose(O.attention(q, k, v, H), ref.numpy(), atol=1e-12)


def test_attention_zero_queries_average_values():
    rng = np.random.default_rng(2)
    k, v = rng.standard_normal((5, 6)), rng.standard_normal((5, 6))
    out = O.attention(np.zeros((5, 6)), k, v, 3)
    assert np.allclose(out, np.broadcast_to(v.mean(axis=0), (5, 6)), atol=1e-14)


# ----------------------------------------------------------------------------- elementwise
def test_layer_norm_vs_torch():
    x = np.random.default_rng(4).standard_normal((5, 33)) * 3 + 1
    ref = TF.layer_norm(torch.from_numpy(x), (33,), eps=1e-6).numpy()
    assert np.allclose(O.layer_norm(x), ref, atol=1e-12)


def test_gelu_tanh_vs_torch_and_known_value():
    x = np.linspace(-6, 6, 101)
    ref = TF.gelu(torch.from_numpy(x), approximate="tanh").numpy()
    assert np.allclose(O.gelu_tanh(x), ref, atol=1e-14)
    assert O.gelu_tanh(np.array(1.0)) == pytest.approx(0.8411919906082768, abs=1e-15)


def test_silu_vs_torch():
    x = np.linspace(-8, 8, 77)
    assert np.allclose(O.silu(x), TF.silu(torch.from_numpy(x)).numpy(), atol=1e-15)


def test_timestep_features_at_zero_and_one_frequency():
    e0 = O.timestep_features(0.0)
    assert e0.shape == (256,) and np.all(e0[:128] == 1.0) and np.all(e0[128:] == 0.0)
    e = O.timestep_features(0.37)
    assert e[0] == pytest.approx(math.cos(370.0)) and e[128] == pytest.approx(math.sin(370.0))
    assert e[64] == pytest.approx(math.cos(370.0 * 10000 ** (-0.5)))


# ----------------------------------------------------------------------------- DiT layer
def _torch_block(W, cfg, h, l, mod):
    """The same adaLN-DiT block from torch library modules (float64)."""
    d = cfg.d_model
    p = f"layers.{l}."
    g = lambda n: torch.from_numpy(np.asarray(W[p + n], dtype=np.float64))
    mha = torch.nn.MultiheadAttention(d, cfg.n_heads, batch_first=True, dtype=torch.float64)
    with torch.no_grad():
        mha.in_proj_weight.copy_(g("qkv_w").T)
        mha.in_proj_bias.copy_(g("qkv_b"))
        mha.out_proj.weight.copy_(g("out_w").T)
        mha.out_proj.bias.copy_(g("out_b"))
        m = torch.from_numpy(mod)
        ht = torch.from_numpy(h)[None]
        x = TF.layer_norm(ht, (d,), eps=1e-6) * (1 + m[1]) + m[0]
        a, _ = mha(x, x, x, need_weights=False)
        ht = ht + m[2] * a
        x = TF.layer_norm(ht, (d,), eps=1e-6) * (1 + m[4]) + m[3]
        u = TF.gelu(TF.linear(x, g("up_w").T, g("up_b")), approximate="tanh")
        ht = ht + m[5] * TF.linear(u, g("down_w").T, g("down_b"))
    return ht[0].numpy()


def test_dit_layer_vs_torch_modules():
    cfgd = micro_config(d_model=24, n_heads=3)
    W, cfg = _setup(cfgd, std=0.2)
    rng = np.random.default_rng(5)
    h = rng.standard_normal((cfg.n_tokens, cfg.d_model))
    mod = rng.standard_normal((6, cfg.d_model)) * 0.5
    out = O.dit_layer(W, cfg, h, 1, mod)
    assert np.allclose(out, _torch_block(W, cfg, h, 1, mod), atol=1e-11)


def test_dit_layer_zero_gates_is_identity():
    W, cfg = _setup(micro_config(), std=0.3)
    rng = np.random.default_rng(6)
    h = rng.standard_normal((cfg.n_tokens, cfg.d_model))
    mod = rng.standard_normal((6, cfg.d_model))
    mod[2] = 0.0
    mod[5] = 0.0
    assert np.array_equal(O.dit_layer(W, cfg, h, 0, mod), h)


def test_conditioning_vs_torch_linear_chain():
    W, cfg = _setup(micro_config(), std=0.3)
    mods, fin = O.conditioning(W, cfg, 0.6)
    g = lambda n: torch.from_numpy(np.asarray(W[n], dtype=np.float64))
    e = torch.from_numpy(O.timestep_features(0.6))
    c = TF.linear(TF.silu(TF.linear(e, g("t_w1").T, g("t_b1"))), g("t_w2").T, g("t_b2"))
    m2 = TF.linear(TF.silu(c), g("layers.2.ada_w").T, g("layers.2.ada_b")).reshape(6, -1)
    assert np.allclose(mods[2], m2.numpy(), atol=1e-13)
    f = TF.linear(TF.silu(c), g("final_ada_w").T, g("final_ada_b")).reshape(2, -1)
    assert np.allclose(fin, f.numpy(), atol=1e-13)


def _torch_embed(W, cfg, x, obs):
    """Token embedding from torch library modules (float64): one nn.Linear per token group,
    concatenated, plus a learned position table looked up with nn.Embedding."""
    d = cfg.d_model
    g = lambda n: torch.from_numpy(np.asarray(W[n], dtype=np.float64))
    lin = {}
    for name, din in (("obs", d), ("vid", cfg.video_dim), ("act", cfg.action_dim)):
        m = torch.nn.Linear(din, d, dtype=torch.float64)
        with torch.no_grad():
            m.weight.copy_(g(name + "_w").T)
            m.bias.copy_(g(name + "_b"))
        lin[name] = m
    emb = torch.nn.Embedding(cfg.n_tokens, d, dtype=torch.float64)
    with torch.no_grad():
        emb.weight.copy_(g("pos"))
        xt = torch.from_numpy(np.asarray(x, dtype=np.float64))
        xv = xt[:cfg.video_len].reshape(cfg.n_video, cfg.video_dim)
        xa = xt[cfg.video_len:].reshape(cfg.n_action, cfg.action_dim)
        h = torch.cat([lin["obs"](torch.from_numpy(np.asarray(obs, dtype=np.float64))),
                       lin["vid"](xv), lin["act"](xa)], dim=0)
        h = h + emb(torch.arange(cfg.n_tokens))
    return h.numpy()


def _distinct_embedding_weights(W, rng):
    """Biases and positions of clearly different magnitudes, so that a dropped position term,
    a bias taken from the wrong group or rows of the wrong group all change the result."""
    W["obs_b"][:] = rng.standard_normal(W["obs_b"].shape) * 1.0
    W["vid_b"][:] = rng.standard_normal(W["vid_b"].shape) * 3.0 + 2.0
    W["act_b"][:] = rng.standard_normal(W["act_b"].shape) * 5.0 - 4.0
    W["pos"][:] = rng.standard_normal(W["pos"].shape) * 0.7


def test_embed_vs_torch_modules():
    W, cfg = _setup(micro_config(), std=0.3)
    rng = np.random.default_rng(11)
    _distinct_embedding_weights(W, rng)
    x = rng.standard_normal(cfg.traj_len)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    h = O.embed(W, cfg, x, obs)
    assert h.shape == (cfg.n_tokens, cfg.d_model)
    assert np.allclose(h, _torch_embed(W, cfg, x, obs), atol=1e-12)


def test_embed_zero_inputs_give_bias_plus_position_per_group():
    """Closed form: with zero trajectory and observation every row is its group's bias plus
    its own position row."""
    W, cfg = _setup(micro_config(), std=0.3)
    _distinct_embedding_weights(W, np.random.default_rng(12))
    h = O.embed(W, cfg, np.zeros(cfg.traj_len), np.zeros((cfg.n_obs, cfg.d_model)))
    No, Nv = cfg.n_obs, cfg.n_video
    pos = np.asarray(W["pos"], dtype=np.float64)
    for r in range(cfg.n_tokens):
        b = W["obs_b"] if r < No else (W["vid_b"] if r < No + Nv else W["act_b"])
        assert np.array_equal(h[r], np.asarray(b, dtype=np.float64) + pos[r])


def _torch_final(W, cfg, h, fin):
    """Final layer from torch library ops: layer_norm (no affine, eps 1e-6), adaLN modulation,
    then nn.Linear output heads on the video rows and on the action rows."""
    g = lambda n: torch.from_numpy(np.asarray(W[n], dtype=np.float64))
    d = cfg.d_model
    heads = {}
    for name, dout in (("vout", cfg.video_dim), ("aout", cfg.action_dim)):
        m = torch.nn.Linear(d, dout, dtype=torch.float64)
        with torch.no_grad():
            m.weight.copy_(g(name + "_w").T)
            m.bias.copy_(g(name + "_b"))
        heads[name] = m
    with torch.no_grad():
        f = torch.from_numpy(np.asarray(fin, dtype=np.float64))
        y = TF.layer_norm(torch.from_numpy(h), (d,), eps=1e-6) * (1 + f[1]) + f[0]
        a0, a1 = cfg.n_obs, cfg.n_obs + cfg.n_video
        vv = heads["vout"](y[a0:a1]).reshape(-1)
        va = heads["aout"](y[a1:]).reshape(-1)
    return torch.cat([vv, va]).numpy()


def test_final_velocity_vs_torch_modules():
    W, cfg = _setup(micro_config(), std=0.3)
    rng = np.random.default_rng(13)
    W["vout_b"][:] = rng.standard_normal(W["vout_b"].shape) * 2.0
    W["aout_b"][:] = rng.standard_normal(W["aout_b"].shape) * 2.0 - 3.0
    h = rng.standard_normal((cfg.n_tokens, cfg.d_model)) * 2.0 + 0.5
    # shift and scale of very different size and sign: a swapped pair, or a `scale` in place
    # of `1 + scale`, moves the result far outside the tolerance
    fin = np.stack([rng.standard_normal(cfg.d_model) * 4.0 + 3.0,
                    rng.standard_normal(cfg.d_model) * 0.3 - 0.6])
    v = O.final_velocity(W, cfg, h, fin)
    assert v.shape == (cfg.traj_len,)
    assert np.allclose(v, _torch_final(W, cfg, h, fin), atol=1e-11)


def test_final_velocity_closed_forms():
    """scale = -1 removes the normalised hidden state: every video row equals shift W_ov + b_ov
    and every action row shift W_oa + b_oa.  With scale = 0 and shift = 0 each row is
    LN(h) W + b, which for h = a row of +-c values (zero mean, unit variance after LN) is the
    signed column sum of W plus b."""
    W, cfg = _setup(micro_config(), std=0.3)
    rng = np.random.default_rng(14)
    d = cfg.d_model
    h = rng.standard_normal((cfg.n_tokens, d))
    shift = rng.standard_normal(d) * 2.0
    v = O.final_velocity(W, cfg, h, np.stack([shift, -np.ones(d)]))
    Wv, bv = np.asarray(W["vout_w"], np.float64), np.asarray(W["vout_b"], np.float64)
    Wa, ba = np.asarray(W["aout_w"], np.float64), np.asarray(W["aout_b"], np.float64)
    vv = v[:cfg.video_len].reshape(cfg.n_video, cfg.video_dim)
    va = v[cfg.video_len:].reshape(cfg.n_action, cfg.action_dim)
    assert np.allclose(vv, np.broadcast_to(shift @ Wv + bv, vv.shape), atol=1e-12)
    assert np.allclose(va, np.broadcast_to(shift @ Wa + ba, va.shape), atol=1e-12)
    sign = np.where(np.arange(d) % 2 == 0, 1.0, -1.0)
    h2 = np.broadcast_to(sign * 2.5, (cfg.n_tokens, d)).copy()
    v2 = O.final_velocity(W, cfg, h2, np.zeros((2, d)))
    ln = sign * (2.5 / math.sqrt(2.5 * 2.5 + 1e-6))
    assert np.allclose(v2[:cfg.video_len].reshape(cfg.n_video, -1),
                       np.broadcast_to(ln @ Wv + bv, (cfg.n_video, cfg.video_dim)), atol=1e-12)
    assert np.allclose(v2[cfg.video_len:].reshape(cfg.n_action, -1),
                       np.broadcast_to(ln @ Wa + ba, (cfg.n_action, cfg.action_dim)), atol=1e-12)


def test_velocity_is_token_permutation_equivariant_without_positions():
    cfgd = micro_config()
    W, cfg = _setup(cfgd, std=0.3)
    W["pos"][:] = 0.0
    rng = np.random.default_rng(7)
    x = rng.standard_normal(cfg.traj_len)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    v = O.velocity(W, cfg, x, obs, 0.4)
    pv = rng.permutation(cfg.n_video)
    pa = rng.permutation(cfg.n_action)
    xv = x[:cfg.video_len].reshape(cfg.n_video, -1)[pv].reshape(-1)
    xa = x[cfg.video_len:].reshape(cfg.n_action, -1)[pa].reshape(-1)
    po = rng.permutation(cfg.n_obs)
    v2 = O.velocity(W, cfg, np.concatenate([xv, xa]), obs[po], 0.4)
    vv = v[:cfg.video_len].reshape(cfg.n_video, -1)[pv].reshape(-1)
    va = v[cfg.video_len:].reshape(cfg.n_action, -1)[pa].reshape(-1)
    assert np.allclose(v2, np.concatenate([vv, va]), atol=1e-12)


def test_velocity_output_rows_match_token_rows():
    """Changing only the last action token's input changes its own output most directly:
    with zero attention weights on the output path the map is strictly per token."""
    cfgd = micro_config()
    W, cfg = _setup(cfgd, std=0.3)
    for l in range(cfg.n_layers):  # switch off both residual branches: tokens stay independent
        W[f"layers.{l}.ada_w"][:] = 0.0
        W[f"layers.{l}.ada_b"][:] = 0.0
    rng = np.random.default_rng(8)
    x = rng.standard_normal(cfg.traj_len)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    v = O.velocity(W, cfg, x, obs, 0.3)
    x2 = x.copy()
    x2[-1] += 1.0
    v2 = O.velocity(W, cfg, x2, obs, 0.3)
    changed = np.nonzero(np.abs(v2 - v) > 1e-14)[0]
    ad = cfg.action_dim
    assert set(changed.tolist()) <= set(range(cfg.traj_len - ad, cfg.traj_len))
    assert len(changed) > 0


# ----------------------------------------------------------------------------- TR
def test_rms_normaliser_has_unit_mean_square():
    v = np.random.default_rng(9).standard_normal(1000) * 7.3
    assert np.mean(O.normalize_rms(v) ** 2) == pytest.approx(1.0, abs=1e-14)
    assert np.all(O.normalize_rms(np.zeros(5)) == 0.0)


def test_tr_remap_slot_indices_bruteforce():
    cfgd = micro_config(tr_normalize=1)
    cfg = O.OracleConfig.from_dict(cfgd)
    T, V, ad = cfg.traj_len, cfg.video_len, cfg.action_dim
    x_bar = np.arange(T, dtype=np.float64)
    eps = -1.0 - np.arange(T, dtype=np.float64)
    for shift in range(0, cfg.n_action + 2):
        out = O.tr_remap(cfg, x_bar, x_bar, 0.5, 0.25, shift, eps)  # x^r == x_bar -> d = 0
        assert np.array_equal(out[:V], x_bar[:V])
        for j in range(cfg.n_action):
            for c in range(ad):
                src = j + shift
                want = x_bar[V + src * ad + c] if src < cfg.n_action else 0.25 * eps[V + j * ad + c]
                assert out[V + j * ad + c] == want


def test_tr_remap_closed_form_and_fresh_video_mode():
    cfgd = micro_config(tr_video_mode=1)
    cfg = O.OracleConfig.from_dict(cfgd)
    rng = np.random.default_rng(10)
    x_bar, x_r, eps = (rng.standard_normal(cfg.traj_len) for _ in range(3))
    out = O.tr_remap(cfg, x_bar, x_r, 0.6, 0.7, 0, eps)
    V = cfg.video_len
    assert np.array_equal(out[:V], 0.7 * eps[:V])
    u = (x_r[V:] - x_bar[V:]) / 0.6
    assert np.allclose(out[V:], x_bar[V:] + 0.7 * u / np.sqrt(np.mean(u * u)), atol=1e-14)


def test_tr_identity_normaliser_recovers_retained_latent():
    cfg = O.OracleConfig.from_dict(micro_config(tr_normalize=0))
    rng = np.random.default_rng(11)
    x_bar, x_r, eps = (rng.standard_normal(cfg.traj_len) for _ in range(3))
    out = O.tr_remap(cfg, x_bar, x_r, 0.4, 0.4, 0, eps)
    assert np.allclose(out, x_r, atol=1e-14)


def _episode(cfgd, std=0.3, seed=0):
    W, cfg = _setup(cfgd, std=std, seed=seed)
    return W, cfg, O.OracleEpisode(W, cfg)


def test_invariant_zero_shift_identity_rescale_equals_plain_continuation():
    cfgd = micro_config(tr_normalize=0, tr_entry_stage=2, tr_retain_stage=-1)
    W, cfg, ep = _episode(cfgd)
    rng = np.random.default_rng(12)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    noise = rng.standard_normal(cfg.traj_len)
    ep.sample_cold(obs, noise, cfg.n_steps)
    x2 = ep.hist[2].copy()
    final = ep.hist[cfg.n_steps].copy()
    assert ep.adapt(obs, 0, rng.standard_normal(cfg.traj_len)) == O.ADAPT_TR_INIT
    assert np.allclose(ep.x, x2, atol=1e-13)
    ep.advance(cfg.n_steps - 2)
    assert np.allclose(ep.hist[cfg.n_steps], final, atol=1e-12)


def test_invariant_empty_target_set_entry_zero_equals_cold():
    cfgd = micro_config(tr_video_mode=1, tr_entry_stage=0)
    W, cfg, ep = _episode(cfgd)
    rng = np.random.default_rng(13)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    ep.sample_cold(obs, rng.standard_normal(cfg.traj_len), cfg.n_steps)
    eps = rng.standard_normal(cfg.traj_len)
    obs2 = rng.standard_normal((cfg.n_obs, cfg.d_model))
    ep.adapt(obs2, cfg.n_action, eps)        # shift covers the whole action horizon
    assert np.array_equal(ep.x, eps)         # sigma_0 = 1: pure fresh noise
    warm = ep.advance(cfg.n_steps)
    cold = O.OracleEpisode(W, cfg).sample_cold(obs2, eps, cfg.n_steps)
    assert np.array_equal(warm, cold)


# ----------------------------------------------------------------------------- OR
def test_or_score_closed_forms():
    cfg = O.OracleConfig.from_dict(micro_config(n_obs=4, or_n_components=2,
                                                or_deltas=(2.0, 0.5, 1, 1),
                                                or_weights=(3.0, 1.0, 1, 1)))
    P = np.zeros((4, 16))
    R = np.zeros((4, 16))
    R[:2] = 1.0      # component 0: diff -1, / delta 2 -> e0 = 0.5
    R[2] = -0.25     # component 1: diffs 0.25 and 0.75, / delta 0.5 -> 0.5 and 1.5
    R[3] = -0.75     #   e1 = sqrt((0.25 + 2.25) / 2)
    e0, e1 = 0.5, math.sqrt(1.25)
    assert O.or_score(cfg, P, R) == pytest.approx(math.sqrt((3 * e0 ** 2 + e1 ** 2) / 4))
    assert O.or_score(cfg, R, R) == 0.0


def _kappa_run(cfgd, n_replans, real_offsets):
    W, cfg, ep = _episode(cfgd)
    rng = np.random.default_rng(14)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    ep.sample_cold(obs, rng.standard_normal(cfg.traj_len), cfg.n_steps)
    seq = []
    for t in range(n_replans):
        eps = rng.standard_normal(cfg.traj_len)
        st = ep.adapt(obs, 1, eps)
        seq.append(st)
        x_b0 = ep.x.copy()
        if st == O.ADAPT_TR_INIT:
            ep.advance(1)
        st2 = ep.adapt(obs + real_offsets[t], 0, None)
        seq.append(st2)
        if st2 == O.ADAPT_REBIND_RESTART:
            assert np.array_equal(ep.x, x_b0) and ep.stage == cfg.tr_entry_stage
        ep.advance(cfg.n_steps - ep.stage)
    return seq, ep


def test_kappa_cap_forces_refresh_and_skips_prefix():
    A, R, T, N, F = (O.ADAPT_REBIND_ACCEPT, O.ADAPT_REBIND_RESTART, O.ADAPT_TR_INIT,
                     O.ADAPT_TR_INIT_NO_PREFIX, O.ADAPT_REFRESH)
    seq, ep = _kappa_run(micro_config(or_tau=0.5, or_kappa_max=3), 6, [0.1] * 6)
    assert seq == [T, A, T, A, T, A, N, F, T, A, T, A]
    st = ep.stats.rates()
    assert ep.stats.n_start == 5 and ep.stats.n_bind == 5 and ep.stats.n_noninitial == 6
    assert st["r_or"] == 1.0 and st["coverage"] == pytest.approx(5 / 6)
    seq, _ = _kappa_run(micro_config(or_tau=0.5, or_kappa_max=3), 3, [0.1, 0.7, 0.1])
    assert seq == [T, A, T, R, T, A]


# ----------------------------------------------------------------------------- RR
@pytest.mark.parametrize("c", [0.5, 1.0, 1.1, 1.25, 2.0, -1.0])
def test_rr_scaled_probe_closed_form(c):
    cfg = O.OracleConfig.from_dict(micro_config())
    p_a = np.random.default_rng(15).standard_normal(200)
    chk = O.rr_check(c * p_a, p_a, cfg)
    alpha = min(max(c, 1.0), 1.25)
    assert chk.alpha == pytest.approx(alpha, abs=1e-14)
    assert chk.cos == pytest.approx(math.copysign(1.0, c), abs=1e-14)
    assert chk.fit == pytest.approx(abs(c - alpha) / abs(c), abs=1e-13)
    assert chk.passed == (chk.fit <= 0.40 and chk.cos >= 0.95)


def test_rr_gate_vs_bruteforce_loops():
    cfg = O.OracleConfig.from_dict(micro_config(rr_gamma_cos=0.5, rr_gamma_fit=0.9))
    rng = np.random.default_rng(16)
    for trial in range(20):
        p_a = rng.standard_normal(30).tolist()
        p_i = [a * 1.1 + 0.4 * rng.standard_normal() for a in p_a]
        n = len(p_a)
        num = sum(x * y for x, y in zip(p_i, p_a)) / n
        den = max(sum(y * y for y in p_a) / n, 1e-8)
        alpha = min(max(num / den, 1.0), 1.25)
        ni = math.sqrt(sum(x * x for x in p_i))
        na = math.sqrt(sum(y * y for y in p_a))
        cos = sum(x * y for x, y in zip(p_i, p_a)) / (ni * na)
        fit = math.sqrt(sum((x - alpha * y) ** 2 for x, y in zip(p_i, p_a))) / ni
        chk = O.rr_check(np.array(p_i), np.array(p_a), cfg)
        assert (chk.alpha, chk.cos, chk.fit) == pytest.approx((alpha, cos, fit), abs=1e-12)
        assert chk.passed == (cos >= 0.5 and fit <= 0.9)


def test_rr_zero_probe_fails_gate():
    cfg = O.OracleConfig.from_dict(micro_config())
    assert not O.rr_check(np.zeros(10), np.ones(10), cfg).passed
    assert not O.rr_check(np.ones(10), np.zeros(10), cfg).passed


def test_rr_reuse_on_identical_input_reproduces_full_forward():
    cfgd = micro_config(n_layers=6, rr_policy=1, rr_q=1, rr_s=2, rr_e=5)
    W, cfg = _setup(cfgd, std=0.3)
    rng = np.random.default_rng(17)
    x = rng.standard_normal(cfg.traj_len)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    full = O.velocity(W, cfg, x, obs, 0.5)
    v1, st, rec1 = O.velocity_rr(W, cfg, x, obs, 0.5, None, True)
    assert not rec1.rr_attempt and np.allclose(v1, full, atol=1e-13)
    v2, st2, rec2 = O.velocity_rr(W, cfg, x, obs, 0.5, st, True)
    assert rec2.rr_attempt and rec2.rr_accept and st2 is st
    for c in rec2.checks:
        assert c.alpha == 1.0 and c.cos == pytest.approx(1.0) and c.fit == pytest.approx(0.0, abs=1e-7)
    assert np.allclose(v2, full, atol=1e-12)


def test_rr_disabled_equals_full_forward():
    cfgd = micro_config(n_layers=6, rr_policy=0, rr_q=1, rr_s=2, rr_e=5)
    W, cfg, ep = _episode(cfgd)
    rng = np.random.default_rng(18)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    noise = rng.standard_normal(cfg.traj_len)
    out = ep.sample_cold(obs, noise, cfg.n_steps)
    sig = O.schedule(cfg.n_steps)
    xs = O.euler_integrate(noise, sig, lambda x, s: O.velocity(W, cfg, x, obs, s))
    assert np.array_equal(out, xs[-1])
    assert ep.stats.n_attempt == 0 and ep.stats.b_dense == 0


def test_rr_rejected_step_refreshes_state_and_counts():
    cfgd = micro_config(n_layers=6, rr_policy=1, rr_q=1, rr_s=2, rr_e=5,
                        rr_gamma_cos=1.1)       # unreachable: every check fails
    W, cfg, ep = _episode(cfgd)
    rng = np.random.default_rng(19)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    ep.sample_cold(obs, rng.standard_normal(cfg.traj_len), cfg.n_steps)
    assert ep.stats.n_attempt == cfg.n_steps - 1 and ep.stats.n_reuse == 0
    assert ep.stats.b_dense == cfg.n_steps * cfg.n_layers and ep.stats.b_skip == 0


def test_rr_layer_evaluation_counts_match_table6():
    for _, name, L, q, s, e, evaluated in (r for r in _golden("profiles.txt") if r[0] == "rr"):
        L, q, s, e = int(L), int(q), int(s), int(e)
        assert 0 < q < s < e < L
        assert L - (e - s) == int(evaluated)


def test_method_defaults_match_paper_tables():
    rows = _golden("profiles.txt")
    alpha = [r for r in rows if r[0] == "alpha"][0]
    d = I.METHOD_DEFAULTS
    assert (d["rr_alpha_min"], d["rr_alpha_max"], d["rr_eps"]) == tuple(float(a) for a in alpha[1:])
    motus = [r for r in rows if r[0] == "gate" and r[1] == "motus"][0]
    assert (d["rr_gamma_cos"], d["rr_gamma_fit"]) == (float(motus[2]), float(motus[3]))


def test_reuse_rates_definitions():
    s = O.Stats(n_attempt=8, n_reuse=6, b_skip=24, b_dense=96, n_start=5, n_bind=4, n_noninitial=9)
    r = s.rates()
    assert r == dict(r_rr=0.75, f_skip=0.25, r_or=0.8, coverage=4 / 9)


# ----------------------------------------------------------------------------- diagnostics (App. E)
def test_latent_similarity_closed_forms_and_bruteforce():
    rng = np.random.default_rng(11)
    a = rng.standard_normal(37)
    assert O.latent_similarity(a, a) == pytest.approx((1.0, 0.0), abs=1e-15)
    assert O.latent_similarity(2.0 * a, a) == pytest.approx((1.0, 1.0), abs=1e-15)
    assert O.latent_similarity(-a, a) == pytest.approx((-1.0, 2.0), abs=1e-15)
    e1, e2 = np.eye(4)[0] * 3.0, np.eye(4)[1] * 4.0
    assert O.latent_similarity(e1, e2) == pytest.approx((0.0, 5.0 / 4.0), abs=1e-15)   # 3-4-5 triangle
    b = rng.standard_normal(37)
    dot = sum(float(x) * float(y) for x, y in zip(a, b))
    na = math.sqrt(sum(float(x) ** 2 for x in a))
    nb = math.sqrt(sum(float(y) ** 2 for y in b))
    dd = math.sqrt(sum((float(x) - float(y)) ** 2 for x, y in zip(a, b)))
    cos, rel = O.latent_similarity(a, b)
    assert cos == pytest.approx(dot / (na * nb), rel=1e-13) and rel == pytest.approx(dd / nb, rel=1e-13)


def test_action_rmse_constant_offset_and_ignored_dims():
    rng = np.random.default_rng(12)
    b = rng.standard_normal((16, 7))
    assert O.action_rmse(b + 0.25, b, dims=6) == pytest.approx(0.25, abs=1e-15)
    a = b.copy()
    a[:, 6] += 9.0                     # only the dimension outside the first six differs
    assert O.action_rmse(a, b, dims=6) == 0.0
    assert O.action_rmse(a, b) == pytest.approx(9.0 / math.sqrt(7.0), abs=1e-12)


def _zero_gate_weights(W, cfg, which):
    d = cfg.d_model
    for l in range(cfg.n_layers):
        for g in which:   # modulation rows 2 (attention gate) and 5 (MLP gate)
            W[f"layers.{l}.ada_w"][:, g * d:(g + 1) * d] = 0.0
            W[f"layers.{l}.ada_b"][g * d:(g + 1) * d] = 0.0
    return W


def test_layer_deltas_zero_gates_and_gate_scaling():
    cfgd = micro_config()
    W, cfg = _setup(cfgd, std=0.2)
    rng = np.random.default_rng(13)
    x = rng.standard_normal(cfg.traj_len)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    Wz = _zero_gate_weights({k: v.copy() for k, v in W.items()}, cfg, (2, 5))
    assert O.layer_deltas(Wz, cfg, x, obs, 0.6) == [0.0] * cfg.n_layers
    # with the MLP gate zero a layer adds g1 * Attn(...): scaling the attention-gate weights by c
    # scales the first layer's change by |c|
    W1 = _zero_gate_weights({k: v.astype(np.float64) for k, v in W.items()}, cfg, (5,))   # exact scaling
    W2 = {k: v.copy() for k, v in W1.items()}
    d = cfg.d_model
    W2["layers.0.ada_w"][:, 2 * d:3 * d] *= -3.0
    W2["layers.0.ada_b"][2 * d:3 * d] *= -3.0
    d1 = O.layer_deltas(W1, cfg, x, obs, 0.6)[0]
    d2 = O.layer_deltas(W2, cfg, x, obs, 0.6)[0]
    assert d1 > 0.0 and d2 == pytest.approx(3.0 * d1, rel=1e-12)


# ----------------------------------------------------------------------------- independent execution
def test_independent_profiles_match_appendix_b():
    """The video / action pair follows the Fast-WAM-IDM profile of App. B.1-B.2: K = 10, the
    video branch remaps stage 5 (sigma 0.83333) to stage 4 (0.88235) on the shifted schedule and
    runs 2 + 4 steps, the action branch enters stage 5 for 5 steps, gates of Table 7."""
    rows = _golden("profiles.txt")
    gate = [r for r in rows if r[0] == "gate" and r[1] == "fastwam"][0]
    sched = {(int(r[2])): float(r[3]) for r in _golden("fastwam_schedule.txt")}
    for size in ("tiny", "idm"):
        v = I.get_config(f"{size}_video" if size == "idm" else "tiny_video")
        a = I.get_config(f"{size}_action" if size == "idm" else "tiny_action")
        steps_v = [r for r in rows if r[0] == "steps" and r[1] == "fastwam_video"][0]
        steps_a = [r for r in rows if r[0] == "steps" and r[1] == "fastwam_action"][0]
        assert v["n_action"] == 0 and a["n_video"] == 0
        assert v["n_steps"] == a["n_steps"] == int(steps_v[2]) == int(steps_a[2])
        sig = O.schedule(v["n_steps"], v["sched_shift"])
        assert round(sig[v["tr_retain_stage"]], 5) == sched[v["tr_retain_stage"]]
        assert round(sig[v["tr_entry_stage"]], 5) == sched[v["tr_entry_stage"]]
        assert (v["prefix_steps"], v["n_steps"] - v["tr_entry_stage"] - v["prefix_steps"]) == \
            (int(steps_v[3]), int(steps_v[4]))
        assert (a["prefix_steps"], a["n_steps"] - a["tr_entry_stage"]) == (int(steps_a[3]), int(steps_a[4]))
        for c in (v, a):
            assert (c["rr_gamma_cos"], c["rr_gamma_fit"]) == (float(gate[2]), float(gate[3]))


def test_single_branch_remap_is_the_joint_remap_of_its_branch():
    """App. B.1: video and action keep separate replan states, each normalised over its own
    trajectory; since Eq. 12 normalises per branch, a one-branch model remaps exactly the slice
    a joint model gives its branch."""
    joint = O.OracleConfig.from_dict(micro_config())
    vid = O.OracleConfig.from_dict(micro_config(n_action=0))
    act = O.OracleConfig.from_dict(micro_config(n_video=0))
    V = joint.video_len
    assert vid.traj_len == V and act.traj_len == joint.traj_len - V
    rng = np.random.default_rng(30)
    x_bar, x_r, eps = (rng.standard_normal(joint.traj_len) for _ in range(3))
    for shift in (0, 2, 7):
        out = O.tr_remap(joint, x_bar, x_r, 0.6, 0.8, shift, eps)
        assert np.array_equal(O.tr_remap(vid, x_bar[:V], x_r[:V], 0.6, 0.8, shift, eps[:V]), out[:V])
        assert np.array_equal(O.tr_remap(act, x_bar[V:], x_r[V:], 0.6, 0.8, shift, eps[V:]), out[V:])


def test_single_branch_rr_uses_one_factor_over_all_rows():
    """§3.3: a branch executed on its own decides reuse by itself, over all of its rows (one
    alpha, one check); a joint model checks observation + video and action rows separately.
    The probe residual is scaled by 1.1 on the first rows and 1.2 on the rest against the
    retained one, and alpha is checked against the least-squares ratio written out by loops."""
    for over, n_checks in ((dict(n_action=0), 1), (dict(n_video=0), 1), (dict(), 2)):
        cfgd = micro_config(n_layers=6, rr_policy=1, rr_q=1, rr_s=2, rr_e=5, rr_alpha_max=2.0, **over)
        W, cfg = _setup(cfgd, std=0.3)
        rng = np.random.default_rng(31)
        x = rng.standard_normal(cfg.traj_len)
        obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
        _, st, _ = O.velocity_rr(W, cfg, x, obs, 0.5, None, True)
        p_i = st.p_a
        half = cfg.n_tokens // 2
        scale = np.where(np.arange(cfg.n_tokens)[:, None] < half, 1.1, 1.2)
        crafted = O.LayerState(p_a=p_i / scale, R_a=st.R_a)
        _, _, rec = O.velocity_rr(W, cfg, x, obs, 0.5, crafted, True)
        assert rec.rr_attempt and len(rec.checks) == n_checks
        for (a, b), chk in zip(O.rr_branch_rows(cfg), rec.checks):
            pi = p_i[a:b].ravel().tolist()
            pa = crafted.p_a[a:b].ravel().tolist()
            num = sum(u * w for u, w in zip(pi, pa))
            den = sum(w * w for w in pa)
            assert chk.alpha == pytest.approx(min(max(num / den, 1.0), 2.0), rel=1e-12)
        if n_checks == 1:
            assert O.rr_branch_rows(cfg) == [(0, cfg.n_tokens)]
            assert 1.1 < rec.checks[0].alpha < 1.2


def test_single_branch_models_denoise_their_own_trajectory():
    """A video-only model outputs only video velocities and an action-only one only action
    velocities; with zero gates every layer is the identity, so each equals the output head
    applied to its own embedded tokens (the branches do not see each other)."""
    for over in (dict(n_action=0), dict(n_video=0)):
        cfgd = micro_config(**over)
        W, cfg = _setup(cfgd, std=0.3)
        W = _zero_gate_weights(W, cfg, (2, 5))
        rng = np.random.default_rng(32)
        x = rng.standard_normal(cfg.traj_len)
        obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
        v = O.velocity(W, cfg, x, obs, 0.3)
        assert v.shape == (cfg.traj_len,)
        _, fin = O.conditioning(W, cfg, 0.3)
        h = O.embed(W, cfg, x, obs)
        y = O.layer_norm(h) * (1.0 + fin[1]) + fin[0]
        a0, a1 = cfg.n_obs, cfg.n_obs + cfg.n_video
        want = np.concatenate([(y[a0:a1] @ W["vout_w"].astype(np.float64) + W["vout_b"]).ravel(),
                               (y[a1:] @ W["aout_w"].astype(np.float64) + W["aout_b"]).ravel()])
        assert np.allclose(v, want, atol=1e-12)


# ----------------------------------------------------------------------------- App. E reuse error
def test_reuse_output_error_zero_on_identical_inputs():
    """A layer state retained from the same inputs makes alpha = 1 and h_s + R_a = h_e: the
    reuse output equals the full one (Eq. 9 on identical inputs)."""
    cfgd = micro_config(n_layers=6, rr_policy=1, rr_q=1, rr_s=2, rr_e=5)
    W, cfg = _setup(cfgd, std=0.3)
    rng = np.random.default_rng(40)
    x = rng.standard_normal(cfg.traj_len)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    _, layer, _ = O.velocity_rr(W, cfg, x, obs, 0.5, None, True)
    err, alphas = O.reuse_output_error(W, cfg, x, obs, 0.5, layer)
    assert err < 1e-12 and alphas == [1.0, 1.0]


def test_reuse_output_error_bruteforce():
    """E_out against a direct evaluation: embed, layers [0, s), h_s + alpha_b R_a on each
    branch's rows with alpha_b the clamped least-squares ratio of Eq. 7 written out by loops,
    layers [e, L), output head; the state retained at another noise level."""
    cfgd = micro_config(n_layers=6, rr_policy=1, rr_q=1, rr_s=2, rr_e=5, rr_alpha_max=2.0)
    W, cfg = _setup(cfgd, std=0.3)
    rng = np.random.default_rng(41)
    x0, x1 = rng.standard_normal(cfg.traj_len), rng.standard_normal(cfg.traj_len)
    obs = rng.standard_normal((cfg.n_obs, cfg.d_model))
    _, layer, _ = O.velocity_rr(W, cfg, x0, obs, 0.7, None, True)
    err, alphas = O.reuse_output_error(W, cfg, x1, obs, 0.4, layer)
    mods, fin = O.conditioning(W, cfg, 0.4)
    h = O.embed(W, cfg, x1, obs)
    for l in range(cfg.rr_q):
        h = O.dit_layer(W, cfg, h, l, mods[l])
    h_q = h.copy()
    for l in range(cfg.rr_q, cfg.rr_s):
        h = O.dit_layer(W, cfg, h, l, mods[l])
    h_s = h.copy()
    split = cfg.n_obs + cfg.n_video
    for b, (a0, a1) in enumerate(((0, split), (split, cfg.n_tokens))):
        pi = (h_s[a0:a1] - h_q[a0:a1]).ravel().tolist()
        pa = layer.p_a[a0:a1].ravel().tolist()
        alpha = min(max(sum(u * v for u, v in zip(pi, pa)) / sum(v * v for v in pa), 1.0), 2.0)
        assert alphas[b] == pytest.approx(alpha, rel=1e-12)
        h[a0:a1] = h_s[a0:a1] + alpha * layer.R_a[a0:a1]
    for l in range(cfg.rr_e, cfg.n_layers):
        h = O.dit_layer(W, cfg, h, l, mods[l])
    y_reuse = O.final_velocity(W, cfg, h, fin)
    y_full = O.velocity(W, cfg, x1, obs, 0.4)
    want = np.linalg.norm(y_reuse - y_full) / np.linalg.norm(y_full)
    assert err == pytest.approx(want, rel=1e-12) and err > 1e-3
