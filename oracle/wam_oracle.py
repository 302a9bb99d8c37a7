"""Plain CPU oracle of the WAMachine denoising hot path (numpy, float64).

TEST INFRASTRUCTURE.  Only the test-suite, ``__graft_entry__.smoke()`` and the CPU-baseline /
reference legs of ``bench.py`` import this module.  The CUDA library never imports, links or
calls it, and the two share no code: the only common module is the seeded input generator,
which holds none of the method's arithmetic.

What it computes (paper: "Efficient World Action Model Inference with Adaptive Intermediate
States", arXiv 2609.34608):

* the DiT denoiser the method runs inside.  The paper cites DiT (§1) and never defines the
  network; the definition used here (token embedding, adaLN-modulated blocks, output heads) is
  written out in ``embed`` / ``dit_layer`` / ``final_velocity``,
* the Euler integration of the flow over the step schedule (§3.2 "native solver"; App. B.1,
  Table 5 and the Fast-WAM schedule values),
* Trajectory Remapping (§3.1, Eq. 1 direction, Eq. 2 remapped init; App. B.1 Eq. 12 unit-RMS
  normaliser),
* Observation Rebinding (§3.2, Eq. 4 consistency score and the kappa rule),
* Residual Rescaling (§3.3, Eqs. 5-9),
* the coordinating state machine (§3.4) and the reuse statistics (App. D.2, Eqs. 14-15),
* the state-continuity diagnostics (App. E): latent similarity across replans, action RMSE, the
  per-layer hidden-state change and the residual-reuse output error.

Precision: every array is promoted to float64 and every reduction is a float64 numpy reduction.

Parity status: each function is pinned by ``tests/test_oracle_pins.py`` against closed forms,
invariants, library routines, brute force on tiny inputs or values printed in the paper.  The
end-to-end action values of the synthetic DiT are not printed anywhere in the paper, so the
composite ``velocity`` is "parity unpinned" as a whole and pinned component by component.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

F64 = np.float64

# Adapt status codes (same meaning as the C header's WAM_ADAPT_* constants).
ADAPT_TR_INIT = 1
ADAPT_TR_INIT_NO_PREFIX = 2
ADAPT_COLD_INIT = 3
ADAPT_REBIND_ACCEPT = 4
ADAPT_REBIND_RESTART = 5
ADAPT_REFRESH = 6

ENTRY_COLD = -1  # entry-stage value that starts a fresh episode from noise at stage 0


@dataclass
class OracleConfig:
    n_layers: int
    d_model: int
    n_heads: int
    mlp_ratio: int
    n_obs: int
    n_video: int
    video_dim: int
    n_action: int
    action_dim: int
    n_steps: int
    sched_shift: float = 1.0
    tr_entry_stage: int = 0
    tr_retain_stage: int = -1          # -1: retain at the entry stage (r = b0)
    tr_normalize: int = 1
    tr_video_mode: int = 0             # 0: remap video without shift; 1: fresh noise
    rr_policy: int = 0                 # 0 off, 1 every path, 2 anticipatory path only
    rr_q: int = 0
    rr_s: int = 0
    rr_e: int = 0
    rr_alpha_min: float = 1.0
    rr_alpha_max: float = 1.25
    rr_eps: float = 1e-8
    rr_gamma_cos: float = 0.95
    rr_gamma_fit: float = 0.40
    or_tau: float = 0.5
    or_kappa_max: int = 3
    or_n_components: int = 1
    or_deltas: tuple = (1.0, 1.0, 1.0, 1.0)
    or_weights: tuple = (1.0, 1.0, 1.0, 1.0)

    @staticmethod
    def from_dict(d: dict) -> "OracleConfig":
        names = OracleConfig.__dataclass_fields__.keys()
        return OracleConfig(**{k: d[k] for k in names if k in d})

    @property
    def n_tokens(self) -> int:
        return self.n_obs + self.n_video + self.n_action

    @property
    def head_dim(self) -> int:
        return self.d_model // self.n_heads

    @property
    def video_len(self) -> int:
        return self.n_video * self.video_dim

    @property
    def traj_len(self) -> int:
        return self.video_len + self.n_action * self.action_dim

    @property
    def rr_enabled(self) -> bool:
        return self.rr_policy != 0 and 0 < self.rr_q < self.rr_s < self.rr_e < self.n_layers


# =========================================================================================
# Schedule and Euler integration
# =========================================================================================

def schedule(n_steps: int, shift: float = 1.0) -> np.ndarray:
    """Noise levels sigma_k, k = 0..K, for t_k = 1 - k/K.

    Linear flow time when shift == 1.  Otherwise the shifted schedule
    sigma = s t / (1 + (s - 1) t) whose values App. B.1 prints for Fast-WAM-IDM
    (stage 5 -> 0.83333, stage 4 -> 0.88235 with s = 5, K = 10).
    """
    k = np.arange(n_steps + 1, dtype=F64)
    t = 1.0 - k / n_steps
    return shift * t / (1.0 + (shift - 1.0) * t)


def euler_step(x: np.ndarray, v: np.ndarray, sigma_from: float, sigma_to: float) -> np.ndarray:
    """One explicit Euler step of dx/dsigma = v from sigma_from to sigma_to."""
    return x + (sigma_to - sigma_from) * v


def euler_integrate(x0, sigmas, velocity_fn):
    """Integrate from sigmas[0] to sigmas[-1]; returns every intermediate latent."""
    xs = [np.asarray(x0, dtype=F64)]
    for k in range(len(sigmas) - 1):
        v = velocity_fn(xs[-1], float(sigmas[k]))
        xs.append(euler_step(xs[-1], v, float(sigmas[k]), float(sigmas[k + 1])))
    return xs


# =========================================================================================
# DiT building blocks (builder-defined network; DiT is cited in §1)
# =========================================================================================

def timestep_features(sigma: float, n: int = 256) -> np.ndarray:
    """Sinusoidal features of 1000*sigma: cos then sin over n/2 frequencies 10000^(-j/(n/2))."""
    half = n // 2
    freqs = np.power(10000.0, -np.arange(half, dtype=F64) / half)
    arg = 1000.0 * float(sigma) * freqs
    return np.concatenate([np.cos(arg), np.sin(arg)])


def silu(x):
    return x / (1.0 + np.exp(-x))


def gelu_tanh(x):
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def layer_norm(x, eps: float = 1e-6):
    """Row-wise normalisation without affine parameters."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def softmax_rows(s):
    m = s.max(axis=-1, keepdims=True)
    p = np.exp(s - m)
    return p / p.sum(axis=-1, keepdims=True)


def attention(q, k, v, n_heads: int):
    """Full bidirectional multi-head attention; q, k, v are [N, d], head h owns columns
    h*dh .. (h+1)*dh.  Scale 1/sqrt(dh), no mask."""
    n, d = q.shape
    dh = d // n_heads
    out = np.empty_like(q, dtype=F64)
    for h in range(n_heads):
        sl = slice(h * dh, (h + 1) * dh)
        p = softmax_rows((q[:, sl] @ k[:, sl].T) / math.sqrt(dh))
        out[:, sl] = p @ v[:, sl]
    return out


def _w(W, name):
    return np.asarray(W[name], dtype=F64)


def conditioning(W, cfg: OracleConfig, sigma: float):
    """Per-layer modulations (shift1, scale1, gate1, shift2, scale2, gate2) and the final
    (shift, scale), all from the timestep embedding c of sigma."""
    e = timestep_features(sigma)
    c = silu(e @ _w(W, "t_w1") + _w(W, "t_b1")) @ _w(W, "t_w2") + _w(W, "t_b2")
    sc = silu(c)
    d = cfg.d_model
    mods = []
    for l in range(cfg.n_layers):
        m = sc @ _w(W, f"layers.{l}.ada_w") + _w(W, f"layers.{l}.ada_b")
        mods.append(m.reshape(6, d))
    fin = (sc @ _w(W, "final_ada_w") + _w(W, "final_ada_b")).reshape(2, d)
    return mods, fin


def embed(W, cfg: OracleConfig, x_traj, obs):
    """Joint token sequence [obs ; video ; action] embedded to width d, plus positions."""
    x_traj = np.asarray(x_traj, dtype=F64)
    xv = x_traj[: cfg.video_len].reshape(cfg.n_video, cfg.video_dim)
    xa = x_traj[cfg.video_len:].reshape(cfg.n_action, cfg.action_dim)
    h = np.concatenate([
        np.asarray(obs, dtype=F64) @ _w(W, "obs_w") + _w(W, "obs_b"),
        xv @ _w(W, "vid_w") + _w(W, "vid_b"),
        xa @ _w(W, "act_w") + _w(W, "act_b"),
    ], axis=0)
    return h + _w(W, "pos")


def dit_layer(W, cfg: OracleConfig, h, l: int, mod):
    """adaLN block: h += g1 * Attn(LN(h)(1+scale1)+shift1); h += g2 * MLP(LN(h)(1+scale2)+shift2)."""
    shift1, scale1, gate1, shift2, scale2, gate2 = mod
    p = f"layers.{l}."
    d = cfg.d_model
    x = layer_norm(h) * (1.0 + scale1) + shift1
    qkv = x @ _w(W, p + "qkv_w") + _w(W, p + "qkv_b")
    a = attention(qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:], cfg.n_heads)
    h = h + gate1 * (a @ _w(W, p + "out_w") + _w(W, p + "out_b"))
    x = layer_norm(h) * (1.0 + scale2) + shift2
    u = gelu_tanh(x @ _w(W, p + "up_w") + _w(W, p + "up_b"))
    return h + gate2 * (u @ _w(W, p + "down_w") + _w(W, p + "down_b"))


def final_velocity(W, cfg: OracleConfig, h, fin):
    """Modulated norm, then per-token output heads on the video and action rows."""
    shift, scale = fin
    y = layer_norm(h) * (1.0 + scale) + shift
    a0 = cfg.n_obs
    a1 = a0 + cfg.n_video
    vv = y[a0:a1] @ _w(W, "vout_w") + _w(W, "vout_b")
    va = y[a1:] @ _w(W, "aout_w") + _w(W, "aout_b")
    return np.concatenate([vv.reshape(-1), va.reshape(-1)])


def velocity(W, cfg: OracleConfig, x_traj, obs, sigma: float):
    """Full DiT forward without any reuse."""
    mods, fin = conditioning(W, cfg, sigma)
    h = embed(W, cfg, x_traj, obs)
    for l in range(cfg.n_layers):
        h = dit_layer(W, cfg, h, l, mods[l])
    return final_velocity(W, cfg, h, fin)


# =========================================================================================
# Residual Rescaling (§3.3)
# =========================================================================================

@dataclass
class RRCheck:
    alpha: float
    cos: float
    fit: float
    passed: bool
    margin: float  # signed distance to the nearer threshold (positive = pass side)


def rr_branch_rows(cfg: OracleConfig):
    """Token-row ranges of the branches whose rescaling factors and checks are separate.

    Joint execution (§3.3): observation + video rows form the video branch, action rows the
    action branch.  Independent execution (§3.3, the Fast-WAM-IDM profile of App. B.1) runs
    each branch as its own model (no action tokens, or no video tokens): that model is one
    branch, all of its rows.
    """
    if cfg.n_video == 0 or cfg.n_action == 0:
        return [(0, cfg.n_tokens)]
    a1 = cfg.n_obs + cfg.n_video
    return [(0, a1), (a1, cfg.n_tokens)]


def rr_check(p_i, p_a, cfg: OracleConfig) -> RRCheck:
    """Eq. 7 (least-squares rescale factor, clamped) and Eq. 8 (cosine and relative fit gate)."""
    p_i = np.asarray(p_i, dtype=F64).reshape(-1)
    p_a = np.asarray(p_a, dtype=F64).reshape(-1)
    num = np.mean(p_i * p_a)
    den = max(np.mean(p_a * p_a), cfg.rr_eps)
    alpha = min(max(num / den, cfg.rr_alpha_min), cfg.rr_alpha_max)
    ni = np.linalg.norm(p_i)
    na = np.linalg.norm(p_a)
    if ni == 0.0 or na == 0.0:
        return RRCheck(alpha, 0.0, math.inf, False, -math.inf)
    cos = float(np.dot(p_i, p_a) / (ni * na))
    fit = float(np.linalg.norm(p_i - alpha * p_a) / ni)
    passed = cos >= cfg.rr_gamma_cos and fit <= cfg.rr_gamma_fit
    margin = min(cos - cfg.rr_gamma_cos, cfg.rr_gamma_fit - fit)
    return RRCheck(float(alpha), cos, fit, passed, float(margin))


@dataclass
class LayerState:
    p_a: np.ndarray   # [N, d] probe residual h_s(a) - h_q(a), Eq. 5
    R_a: np.ndarray   # [N, d] middle residual h_e(a) - h_s(a), Eq. 5


@dataclass
class StepRecord:
    stage: int
    sigma: float
    v: np.ndarray
    rr_active: bool = False        # step belongs to an RR-enabled path
    rr_attempt: bool = False       # gate evaluated against a retained layer state
    rr_accept: bool = False        # middle layers skipped
    checks: list = field(default_factory=list)


def velocity_rr(W, cfg: OracleConfig, x_traj, obs, sigma: float, layer: LayerState | None,
                gate_allowed: bool, forced_accept: bool | None = None, margin_tol: float = 1e-3):
    """One DiT forward split at the RR boundaries 0 < q < s < e < L (§3.3).

    Returns (v, new_layer_state, record).  With ``gate_allowed`` and a retained layer state the
    probe residual p_i (Eq. 6) is checked per branch (Eqs. 7-8); if every branch passes, the
    middle layers are replaced by h_s + alpha R_a (Eq. 9) and the layer state is kept;
    otherwise the middle layers run from h_s and the state is refreshed with p_i and the new
    middle residual.  ``forced_accept`` replays a decision taken elsewhere: it must agree with
    the oracle's own decision whenever every branch's margin exceeds ``margin_tol``.
    """
    q, s, e, L = cfg.rr_q, cfg.rr_s, cfg.rr_e, cfg.n_layers
    mods, fin = conditioning(W, cfg, sigma)
    h = embed(W, cfg, x_traj, obs)
    for l in range(q):
        h = dit_layer(W, cfg, h, l, mods[l])
    h_q = h
    for l in range(q, s):
        h = dit_layer(W, cfg, h, l, mods[l])
    h_s = h
    p_i = h_s - h_q
    rec = StepRecord(stage=-1, sigma=sigma, v=None, rr_active=True)
    accept = False
    if gate_allowed and layer is not None:
        rec.rr_attempt = True
        rec.checks = [rr_check(p_i[a:b], layer.p_a[a:b], cfg) for a, b in rr_branch_rows(cfg)]
        accept = all(c.passed for c in rec.checks)
        if forced_accept is not None:
            decisive = all(abs(c.margin) > margin_tol for c in rec.checks)
            if decisive and bool(forced_accept) != accept:
                raise AssertionError(
                    f"RR decision mismatch with margins {[c.margin for c in rec.checks]}")
            accept = bool(forced_accept)
    if accept:
        h = h_s.copy()
        for (a, b), c in zip(rr_branch_rows(cfg), rec.checks):
            h[a:b] = h_s[a:b] + c.alpha * layer.R_a[a:b]
        new_layer = layer
    else:
        for l in range(s, e):
            h = dit_layer(W, cfg, h, l, mods[l])
        new_layer = LayerState(p_a=p_i, R_a=h - h_s)
    rec.rr_accept = accept
    for l in range(e, L):
        h = dit_layer(W, cfg, h, l, mods[l])
    return final_velocity(W, cfg, h, fin), new_layer, rec


# =========================================================================================
# Trajectory Remapping (§3.1)
# =========================================================================================

def normalize_rms(v):
    """Eq. 12: v / sqrt(mean(v^2)); an all-zero input stays zero."""
    v = np.asarray(v, dtype=F64)
    ms = np.mean(v * v)
    return v / math.sqrt(ms) if ms > 0.0 else np.zeros_like(v)


def tr_direction(x_r, x_bar, sigma_r: float, normalize: bool = True):
    """Eq. 1: d = N((x^r - x_bar) / sigma_r) for one branch's complete trajectory."""
    u = (np.asarray(x_r, dtype=F64) - np.asarray(x_bar, dtype=F64)) / sigma_r
    return normalize_rms(u) if normalize else u


def tr_remap(cfg: OracleConfig, x_bar, x_r, sigma_r: float, sigma_b0: float, shift: int, eps):
    """Eq. 2 for one episode's trajectory [video | action].

    Video: no temporal shift (every slot receives state), or fresh noise when
    ``tr_video_mode == 1`` (Motus profile, App. B.1).  Action: slot j receives the retained
    slot j + shift while that stays inside the horizon; the uncovered tail gets fresh noise.
    Fresh noise at level sigma_b0 is sigma_b0 * eps.  Each branch's direction is normalised over
    that branch alone, so a single-branch model of independent execution (App. B.1: video and
    action keep separate replan states) remaps exactly its part of the joint trajectory.
    """
    x_bar = np.asarray(x_bar, dtype=F64)
    x_r = np.asarray(x_r, dtype=F64)
    eps = np.asarray(eps, dtype=F64)
    V, Na, ad = cfg.video_len, cfg.n_action, cfg.action_dim
    norm = bool(cfg.tr_normalize)
    out = np.empty(cfg.traj_len, dtype=F64)
    if V == 0:
        pass  # action-only model (independent execution): no video branch
    elif cfg.tr_video_mode == 1:
        out[:V] = sigma_b0 * eps[:V]
    else:
        d_v = tr_direction(x_r[:V], x_bar[:V], sigma_r, norm)
        out[:V] = x_bar[:V] + sigma_b0 * d_v
    if Na == 0:
        return out  # video-only model (independent execution): no action branch
    d_a = tr_direction(x_r[V:], x_bar[V:], sigma_r, norm).reshape(Na, ad)
    xb_a = x_bar[V:].reshape(Na, ad)
    ea = eps[V:].reshape(Na, ad)
    oa = out[V:].reshape(Na, ad)
    for j in range(Na):
        src = j + shift
        if src < Na:
            oa[j] = xb_a[src] + sigma_b0 * d_a[src]
        else:
            oa[j] = sigma_b0 * ea[j]
    return out


# =========================================================================================
# Observation Rebinding (§3.2)
# =========================================================================================

def or_score(cfg: OracleConfig, predicted_obs, real_obs) -> float:
    """Eq. 4: per component RMSE of (prediction - observation)/delta_m, combined by a weighted
    root mean square.  Components are equal contiguous blocks of observation tokens."""
    P = np.asarray(predicted_obs, dtype=F64)
    O = np.asarray(real_obs, dtype=F64)
    M = cfg.or_n_components
    blk = cfg.n_obs // M
    num = 0.0
    den = 0.0
    for m in range(M):
        diff = (P[m * blk:(m + 1) * blk] - O[m * blk:(m + 1) * blk]) / cfg.or_deltas[m]
        e_m = math.sqrt(float(np.mean(diff * diff)))
        num += cfg.or_weights[m] * e_m * e_m
        den += cfg.or_weights[m]
    return math.sqrt(num / den)


# =========================================================================================
# Joint state machine (§3.4) and reuse statistics (App. D.2)
# =========================================================================================

@dataclass
class Stats:
    n_attempt: int = 0       # RR checks evaluated with a current probe
    n_reuse: int = 0         # accepted RR decisions that skipped the middle layers
    b_skip: int = 0          # skipped layer evaluations
    b_dense: int = 0         # full-depth layer count of RR-enabled steps
    n_start: int = 0         # anticipatory prefixes started
    n_bind: int = 0          # prefixes accepted and used
    n_noninitial: int = 0    # replans after the first

    def rates(self):
        """Eqs. 14-15."""
        div = lambda a, b: a / b if b else 0.0
        return dict(r_rr=div(self.n_reuse, self.n_attempt), f_skip=div(self.b_skip, self.b_dense),
                    r_or=div(self.n_bind, self.n_start),
                    coverage=div(self.n_bind, self.n_noninitial))


class OracleEpisode:
    """One episode's replan / denoising / layer state, mirroring the C-ABI's calls."""

    def __init__(self, W, cfg: OracleConfig):
        self.W = W
        self.cfg = cfg
        self.sig = schedule(cfg.n_steps, cfg.sched_shift)
        self.stats = Stats()
        self.stage = -1
        self.x = None
        self.hist: dict[int, np.ndarray] = {}
        self.hist_from = 0
        self.vhist: dict[int, np.ndarray] = {}
        self.obs = None
        self.finished = False
        self.x_b0 = None
        self.b0 = 0
        self.kappa = 0
        self.since_bind = 0
        self.path = "cold"
        self.path_steps = 0
        self.layer: LayerState | None = None
        self.records: list[StepRecord] = []

    # ---- cold start ---------------------------------------------------------------------
    def cold_init(self, obs, noise):
        """First replan: fresh noise at stage 0 (§3.1: the first replan starts from noise)."""
        self.x = np.asarray(noise, dtype=F64).copy()
        self.stage = 0
        self.hist = {0: self.x.copy()}
        self.hist_from = 0
        self.vhist = {}
        self.obs = np.asarray(obs, dtype=F64).copy()
        self.finished = False
        self.x_b0 = self.x.copy()
        self.b0 = 0
        self.kappa = 0
        self.since_bind = 0
        self.path = "cold"
        self.path_steps = 0
        self.layer = None
        return ADAPT_COLD_INIT

    def sample_cold(self, obs, noise, n_steps, forced=None):
        self.cold_init(obs, noise)
        return self.advance(n_steps, forced)

    # ---- adaptation ---------------------------------------------------------------------
    def adapt(self, new_obs, shift: int, eps, entry_stage: int | None = None):
        cfg = self.cfg
        if entry_stage == ENTRY_COLD:
            return self.cold_init(new_obs, eps)
        if self.finished:
            # Trajectory Remapping from the finished replan (Eqs. 1-2).
            b0 = cfg.tr_entry_stage if entry_stage is None else entry_stage
            r = b0 if cfg.tr_retain_stage < 0 else cfg.tr_retain_stage
            if not (0 <= b0 < cfg.n_steps and self.hist_from <= r < cfg.n_steps):
                raise ValueError("retained stage unavailable")
            x_bar = self.hist[cfg.n_steps]
            x_r = self.hist[r]
            self.x = tr_remap(cfg, x_bar, x_r, float(self.sig[r]), float(self.sig[b0]), shift, eps)
            self.x_b0 = self.x.copy()
            self.b0 = b0
            self.stage = b0
            self.hist[b0] = self.x.copy()
            self.hist_from = b0
            self.obs = np.asarray(new_obs, dtype=F64).copy()
            self.finished = False
            self.since_bind = 0
            self.path = "prefix"
            self.path_steps = 0
            self.stats.n_noninitial += 1
            if self.kappa >= cfg.or_kappa_max:
                # kappa reached its cap: the next replan refreshes and skips the prefix.
                return ADAPT_TR_INIT_NO_PREFIX
            return ADAPT_TR_INIT
        # Rebinding an in-flight replan to a new (real) condition (§3.2).
        if shift != 0:
            raise ValueError("rebinding takes no shift")
        new_obs = np.asarray(new_obs, dtype=F64)
        if self.since_bind == 0:
            # No anticipatory prefix ran: refresh under the real condition.
            self.obs = new_obs.copy()
            self.kappa = 0
            self.path = "refresh"
            self.path_steps = 0
            return ADAPT_REFRESH
        self.stats.n_start += 1
        S = or_score(cfg, self.obs, new_obs)
        if S < cfg.or_tau and self.kappa < cfg.or_kappa_max:
            self.obs = new_obs.copy()
            self.kappa += 1
            self.stats.n_bind += 1
            self.since_bind = 0
            return ADAPT_REBIND_ACCEPT
        # Restart from the remapped initialisation under the real condition.
        self.x = self.x_b0.copy()
        self.stage = self.b0
        self.hist[self.b0] = self.x.copy()
        self.obs = new_obs.copy()
        self.kappa = 0
        self.since_bind = 0
        self.path = "refresh"
        self.path_steps = 0
        return ADAPT_REBIND_RESTART

    # ---- denoising ----------------------------------------------------------------------
    def _gate_allowed(self) -> bool:
        cfg = self.cfg
        if cfg.rr_policy == 1:
            return True
        if cfg.rr_policy == 2:
            return self.path == "prefix" and self.path_steps >= 1
        return False

    def _rr_path(self) -> bool:
        cfg = self.cfg
        if not cfg.rr_enabled:
            return False
        return cfg.rr_policy == 1 or (cfg.rr_policy == 2 and self.path == "prefix")

    def advance(self, n_steps: int, forced=None):
        """Run n Euler steps from the current stage under the bound condition.

        ``forced`` optionally lists one RR decision per step to replay (see ``velocity_rr``).
        Returns the final trajectory when the replan reaches stage K, else None.
        """
        cfg = self.cfg
        if self.stage + n_steps > cfg.n_steps:
            raise ValueError("past the last stage")
        for i in range(n_steps):
            k = self.stage
            sig = float(self.sig[k])
            if self._rr_path():
                f = None if forced is None else forced[i]
                v, self.layer, rec = velocity_rr(self.W, cfg, self.x, self.obs, sig, self.layer,
                                                 self._gate_allowed(), f)
                self.stats.b_dense += cfg.n_layers
                if rec.rr_attempt:
                    self.stats.n_attempt += 1
                if rec.rr_accept:
                    self.stats.n_reuse += 1
                    self.stats.b_skip += cfg.rr_e - cfg.rr_s
            else:
                v = velocity(self.W, cfg, self.x, self.obs, sig)
                rec = StepRecord(stage=k, sigma=sig, v=v)
            rec.stage = k
            rec.v = v
            self.records.append(rec)
            self.vhist[k] = v
            self.x = euler_step(self.x, v, sig, float(self.sig[k + 1]))
            self.stage = k + 1
            self.hist[k + 1] = self.x.copy()
            self.since_bind += 1
            self.path_steps += 1
        if self.stage == cfg.n_steps:
            self.finished = True
            return self.x.copy()
        return None

    def actions(self):
        cfg = self.cfg
        return self.hist[cfg.n_steps][cfg.video_len:].reshape(cfg.n_action, cfg.action_dim)


def latent_similarity(x_t, x_prev):
    """App. E trajectory diagnostic: cosine similarity and relative L2 distance between the latent
    of the current replan x_t^r and the preceding replan's x_{t-1}^r at the same stage; the
    preceding latent is the reference of the relative distance."""
    a = np.asarray(x_t, dtype=F64).ravel()
    b = np.asarray(x_prev, dtype=F64).ravel()
    na, nb = float(np.linalg.norm(a)), float(np.linalg.norm(b))
    cos = float(a @ b) / (na * nb) if na > 0.0 and nb > 0.0 else 0.0
    dist = float(np.linalg.norm(a - b))
    rel = dist / nb if nb > 0.0 else (0.0 if dist == 0.0 else math.inf)
    return cos, rel


def layer_deltas(W, cfg: OracleConfig, x_traj, obs, sigma: float):
    """App. E layer diagnostic: relative L2 change of the hidden state across each layer of the
    full forward at sigma, Delta_l = ||h_{l+1} - h_l|| / ||h_l|| with h_0 the token embedding."""
    mods, _ = conditioning(W, cfg, sigma)
    h = embed(W, cfg, x_traj, obs)
    out = []
    for l in range(cfg.n_layers):
        h1 = dit_layer(W, cfg, h, l, mods[l])
        out.append(float(np.linalg.norm(h1 - h) / np.linalg.norm(h)))
        h = h1
    return out


def reuse_output_error(W, cfg: OracleConfig, x_traj, obs, sigma: float, layer: LayerState):
    """App. E residual-reuse diagnostic at one step: E_out = |y_reuse - y_full| / |y_full| on
    identical inputs, y_full the full forward and y_reuse the forward whose middle layers are
    replaced by h_s + alpha R_a (Eq. 9), alpha per branch from Eq. 7 against the retained layer
    state whatever the Eq. 8 checks say.  Returns (E_out, [alpha per branch])."""
    y_full = velocity(W, cfg, x_traj, obs, sigma)
    y_reuse, _, rec = velocity_rr(W, cfg, x_traj, obs, sigma, layer, True, forced_accept=True,
                                  margin_tol=math.inf)
    err = float(np.linalg.norm(y_reuse - y_full) / np.linalg.norm(y_full))
    return err, [c.alpha for c in rec.checks]


def action_rmse(a, b, dims=None):
    """App. E Eq. 17 diagnostic: RMSE over the first ``dims`` action dimensions."""
    a = np.asarray(a, dtype=F64)
    b = np.asarray(b, dtype=F64)
    if dims is not None:
        a, b = a[:, :dims], b[:, :dims]
    return math.sqrt(float(np.mean((a - b) ** 2)))
