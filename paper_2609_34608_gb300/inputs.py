"""Seeded synthetic inputs shared by the CUDA library's callers and by the CPU oracle.

This module only draws numbers and names shapes: it holds none of the method's
arithmetic.  Every array is drawn in float64 from numpy's PCG64 generator and cast to
float32, so both sides of a parity test receive identical bits.

Workloads (the paper evaluates trained third-party WAMs on LIBERO / RoboTwin 2.0,
none of which exists here; these synthetic shapes stand in for them):

* ``tiny``        2 blocks, d=128, 4 heads; 16 obs + 32 video (dim 16) + 8 action (7-DoF)
                  tokens; 8 Euler steps; fp32.  One cold sample, then a warm continuation
                  with executed shift 1 and 4 retained steps.
* ``latency``     12 blocks, d=768, 12 heads; 256 obs (2 views x 128) + 1024 video
                  (4 frames x 16x16, dim 16) + 16 action (7-DoF) tokens; 10 steps; bf16; B=1.
* ``closed_loop`` the ``latency`` model driven for 200 control steps; each step executes
                  8 of 16 actions; next obs = 0.9 prev + sqrt(0.19) N(0,1); warm
                  continuation of 3 of 10 steps (1 anticipatory + 2 real) vs cold 10.
* ``serving``     24 blocks, d=1024, 16 heads; B=32; 384 obs + 2048 video + 32 action
                  (7-DoF); 16 cold (10 steps) + 16 warm (2 of 10 steps).
* ``bimanual``    28 blocks, d=1152, 16 heads (head dim 72); B=8; 768 obs + 4096 video +
                  50 action (14-DoF); cold 10 + warm sweep over 1..9 retained steps, shift 25.
* ``tiny_video`` / ``tiny_action``, ``idm_video`` / ``idm_action``: independent execution, a
                  video-only and an action-only model with separate replan states (the
                  Fast-WAM-IDM profile), at the ``tiny_rr`` and ``latency`` sizes.

Weight tensors are N(0, 0.02) from seed 0 in the fixed order of ``weight_spec`` (the same
order the C header ``include/wam.h`` documents for the flat weight buffer).
"""
from __future__ import annotations

import math
from collections import OrderedDict

import numpy as np

# ---------------------------------------------------------------------------------------
# Model / method configurations (plain values; the method's profile constants come from
# the paper's appendix tables and are cited where they are consumed).
# ---------------------------------------------------------------------------------------

_MODEL_KEYS = ("n_layers", "d_model", "n_heads", "mlp_ratio", "n_obs", "n_video",
               "video_dim", "n_action", "action_dim")

NAMED_CONFIGS: dict[str, dict] = {
    "tiny": dict(
        n_layers=2, d_model=128, n_heads=4, mlp_ratio=4,
        n_obs=16, n_video=32, video_dim=16, n_action=8, action_dim=7,
        n_steps=8, precision="fp32", batch=1,
        tr_entry_stage=4, tr_retain_stage=4, shift=1,
        rr_policy=0, rr_q=0, rr_s=0, rr_e=0,
    ),
    # A six-block variant of ``tiny`` whose depth admits 0 < q < s < e < L.
    "tiny_rr": dict(
        n_layers=6, d_model=128, n_heads=4, mlp_ratio=4,
        n_obs=16, n_video=32, video_dim=16, n_action=8, action_dim=7,
        n_steps=8, precision="fp32", batch=1,
        tr_entry_stage=4, tr_retain_stage=4, shift=1,
        rr_policy=1, rr_q=1, rr_s=2, rr_e=5,
    ),
    "latency": dict(
        n_layers=12, d_model=768, n_heads=12, mlp_ratio=4,
        n_obs=256, n_video=1024, video_dim=16, n_action=16, action_dim=7,
        n_steps=10, precision="bf16", batch=1,
        tr_entry_stage=7, tr_retain_stage=7, shift=8,
        rr_policy=1, rr_q=2, rr_s=4, rr_e=8,
    ),
    "closed_loop": dict(
        n_layers=12, d_model=768, n_heads=12, mlp_ratio=4,
        n_obs=256, n_video=1024, video_dim=16, n_action=16, action_dim=7,
        n_steps=10, precision="bf16", batch=1,
        tr_entry_stage=7, tr_retain_stage=7, shift=8,
        rr_policy=1, rr_q=2, rr_s=4, rr_e=8,
        prefix_steps=1, control_steps=200, obs_rho=0.9,
    ),
    "serving": dict(
        n_layers=24, d_model=1024, n_heads=16, mlp_ratio=4,
        n_obs=384, n_video=2048, video_dim=16, n_action=32, action_dim=7,
        n_steps=10, precision="bf16", batch=32,
        tr_entry_stage=8, tr_retain_stage=8, shift=16,
        rr_policy=1, rr_q=2, rr_s=4, rr_e=20,
    ),
    "bimanual": dict(
        n_layers=28, d_model=1152, n_heads=16, mlp_ratio=4,
        n_obs=768, n_video=4096, video_dim=16, n_action=50, action_dim=14,
        n_steps=10, precision="bf16", batch=8,
        tr_entry_stage=5, tr_retain_stage=5, shift=25,
        rr_policy=1, rr_q=2, rr_s=4, rr_e=24,
    ),
    # Independent execution (§3.3; App. B.1 Fast-WAM-IDM profile): the video branch and the
    # action branch are separate models, each with its own replan state and RR decisions.
    # Video: shifted schedule s = 5, retained stage 5 remapped to entry stage 4 without a
    # temporal shift, 2 anticipatory + 4 real steps.  Action: linear schedule, enters stage 5
    # with the horizon shifted by the executed count, 5 steps under the real observation.  RR
    # thresholds of the Fast-WAM-IDM column of Table 7 (cos >= 0.80, fit <= 0.60).
    "tiny_video": dict(
        n_layers=6, d_model=128, n_heads=4, mlp_ratio=4,
        n_obs=16, n_video=32, video_dim=16, n_action=0, action_dim=7,
        n_steps=10, precision="fp32", batch=1, sched_shift=5.0,
        tr_entry_stage=4, tr_retain_stage=5, shift=0, prefix_steps=2,
        rr_policy=1, rr_q=1, rr_s=2, rr_e=5, rr_gamma_cos=0.80, rr_gamma_fit=0.60,
    ),
    "tiny_action": dict(
        n_layers=6, d_model=128, n_heads=4, mlp_ratio=4,
        n_obs=16, n_video=0, video_dim=16, n_action=8, action_dim=7,
        n_steps=10, precision="fp32", batch=1, sched_shift=1.0,
        tr_entry_stage=5, tr_retain_stage=5, shift=4, prefix_steps=0,
        rr_policy=1, rr_q=1, rr_s=2, rr_e=5, rr_gamma_cos=0.80, rr_gamma_fit=0.60,
    ),
    # The same pair at the size of the ``latency`` model: 12 blocks, d=768, 12 heads each;
    # video 256 obs + 1024 video tokens, action 256 obs + 16 action tokens (7-DoF).
    "idm_video": dict(
        n_layers=12, d_model=768, n_heads=12, mlp_ratio=4,
        n_obs=256, n_video=1024, video_dim=16, n_action=0, action_dim=7,
        n_steps=10, precision="bf16", batch=1, sched_shift=5.0,
        tr_entry_stage=4, tr_retain_stage=5, shift=0, prefix_steps=2,
        rr_policy=1, rr_q=2, rr_s=4, rr_e=8, rr_gamma_cos=0.80, rr_gamma_fit=0.60,
    ),
    "idm_action": dict(
        n_layers=12, d_model=768, n_heads=12, mlp_ratio=4,
        n_obs=256, n_video=0, video_dim=16, n_action=16, action_dim=7,
        n_steps=10, precision="bf16", batch=1, sched_shift=1.0,
        tr_entry_stage=5, tr_retain_stage=5, shift=8, prefix_steps=0,
        rr_policy=1, rr_q=2, rr_s=4, rr_e=8, rr_gamma_cos=0.80, rr_gamma_fit=0.60,
    ),
}

# Method constants shared by every profile: RR bounds and thresholds (App. B.2,
# Table 7 Motus column; alpha in [1, 1.25], eps = 1e-8) and the OR threshold / rebinding
# cap for one obs-token component compared at delta = 1 (the builder's synthetic
# reading of App. B.3: next-obs innovation RMS sqrt(0.19) ~ 0.436 < tau).
METHOD_DEFAULTS = dict(
    sched_shift=1.0, tr_normalize=1, tr_video_mode=0,
    rr_alpha_min=1.0, rr_alpha_max=1.25, rr_eps=1e-8,
    rr_gamma_cos=0.95, rr_gamma_fit=0.40,
    or_tau=0.5, or_kappa_max=3, or_n_components=1,
    or_deltas=(1.0, 1.0, 1.0, 1.0), or_weights=(1.0, 1.0, 1.0, 1.0),
)


def get_config(name: str, **overrides) -> dict:
    """Return a fresh dict: named workload values, method defaults, then overrides."""
    cfg = dict(METHOD_DEFAULTS)
    cfg.update(NAMED_CONFIGS[name])
    cfg.update(overrides)
    return cfg


def model_dims(cfg: dict) -> dict:
    return {k: int(cfg[k]) for k in _MODEL_KEYS}


def n_tokens(cfg: dict) -> int:
    return int(cfg["n_obs"]) + int(cfg["n_video"]) + int(cfg["n_action"])


def traj_len(cfg: dict) -> int:
    """Per-episode trajectory length: video values then action values."""
    return int(cfg["n_video"]) * int(cfg["video_dim"]) + int(cfg["n_action"]) * int(cfg["action_dim"])


# ---------------------------------------------------------------------------------------
# Weights
# ---------------------------------------------------------------------------------------

TIME_FEATURES = 256  # sinusoidal timestep features fed to the conditioning MLP


def weight_spec(cfg: dict) -> list[tuple[str, tuple[int, ...]]]:
    """Ordered (name, shape) list of every weight tensor.  Matrices are [in, out]."""
    L, d, r = int(cfg["n_layers"]), int(cfg["d_model"]), int(cfg["mlp_ratio"])
    vd, ad, N = int(cfg["video_dim"]), int(cfg["action_dim"]), n_tokens(cfg)
    spec = [
        ("obs_w", (d, d)), ("obs_b", (d,)),
        ("vid_w", (vd, d)), ("vid_b", (d,)),
        ("act_w", (ad, d)), ("act_b", (d,)),
        ("pos", (N, d)),
        ("t_w1", (TIME_FEATURES, d)), ("t_b1", (d,)),
        ("t_w2", (d, d)), ("t_b2", (d,)),
    ]
    for l in range(L):
        p = f"layers.{l}."
        spec += [
            (p + "ada_w", (d, 6 * d)), (p + "ada_b", (6 * d,)),
            (p + "qkv_w", (d, 3 * d)), (p + "qkv_b", (3 * d,)),
            (p + "out_w", (d, d)), (p + "out_b", (d,)),
            (p + "up_w", (d, r * d)), (p + "up_b", (r * d,)),
            (p + "down_w", (r * d, d)), (p + "down_b", (d,)),
        ]
    spec += [
        ("final_ada_w", (d, 2 * d)), ("final_ada_b", (2 * d,)),
        ("vout_w", (d, vd)), ("vout_b", (vd,)),
        ("aout_w", (d, ad)), ("aout_b", (ad,)),
    ]
    return spec


def weight_count(cfg: dict) -> int:
    return sum(math.prod(s) for _, s in weight_spec(cfg))


def make_weights(cfg: dict, seed: int = 0, std: float = 0.02) -> "OrderedDict[str, np.ndarray]":
    """All weights N(0, std^2), drawn tensor by tensor in ``weight_spec`` order."""
    rng = np.random.Generator(np.random.PCG64(seed))
    out: OrderedDict[str, np.ndarray] = OrderedDict()
    for name, shape in weight_spec(cfg):
        out[name] = (rng.standard_normal(shape) * std).astype(np.float32)
    return out


def flatten_weights(weights: "OrderedDict[str, np.ndarray]") -> np.ndarray:
    """One contiguous float32 buffer in ``weight_spec`` order (the C-ABI's layout)."""
    return np.ascontiguousarray(np.concatenate([w.reshape(-1) for w in weights.values()]),
                                dtype=np.float32)


# ---------------------------------------------------------------------------------------
# Per-call inputs
# ---------------------------------------------------------------------------------------

def _normal(seed: int, shape) -> np.ndarray:
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.standard_normal(shape).astype(np.float32)


def make_noise(cfg: dict, batch: int, seed: int = 1) -> np.ndarray:
    """Initial noise eps ~ N(0,1), shape [batch, T]."""
    return _normal(seed, (batch, traj_len(cfg)))


def make_obs(cfg: dict, batch: int, seed: int = 2) -> np.ndarray:
    """Already-encoded observation tokens ~ N(0,1), shape [batch, n_obs, d]."""
    return _normal(seed, (batch, int(cfg["n_obs"]), int(cfg["d_model"])))


def make_fresh_eps(cfg: dict, batch: int, step: int) -> np.ndarray:
    """Standard-normal draw for the uncovered slots of a remapped init, seed 1000+step."""
    return _normal(1000 + step, (batch, traj_len(cfg)))


class ObsProcess:
    """Synthetic environment: o' = rho * o + sqrt(1 - rho^2) * N(0,1) per token.

    ``predicted(o)`` is the AR(1) mean rho * o, the stand-in for the WAM's predicted
    future observation.
    """

    def __init__(self, cfg: dict, batch: int, seed: int, rho: float = 0.9):
        self.rho = float(rho)
        self.rng = np.random.Generator(np.random.PCG64(seed))
        self.shape = (batch, int(cfg["n_obs"]), int(cfg["d_model"]))
        self.obs = self.rng.standard_normal(self.shape).astype(np.float32)

    def step(self) -> np.ndarray:
        innov = self.rng.standard_normal(self.shape)
        nxt = self.rho * self.obs.astype(np.float64) + math.sqrt(1.0 - self.rho ** 2) * innov
        self.obs = nxt.astype(np.float32)
        return self.obs

    def predicted(self) -> np.ndarray:
        return (self.rho * self.obs.astype(np.float64)).astype(np.float32)
