"""Python binding of ``libwam_gb300.so`` (include/wam.h, include/wam_ops.h).

Argument marshalling only: every computation runs in the CUDA library.  Buffers may be numpy
arrays (host) or torch tensors (host or CUDA); they are passed by pointer.  The library must have
been built (``paper_2609_34608_gb300._build.build()``); loading fails loudly otherwise.
"""
from __future__ import annotations

import ctypes
import os
import re
import weakref

import numpy as np

from . import _build

# ---- constants (mirrors of include/wam.h) ------------------------------------------------
WAM_OK = 0
ERRORS = {1: "INVALID_ARG", 2: "BAD_STATE", 3: "OOM", 4: "CUDA", 5: "TIMEOUT", 6: "UNSUPPORTED"}
PREC = {"fp32": 0, "bf16": 1}
ENTRY_COLD = -1
ADAPT_TR_INIT, ADAPT_TR_INIT_NO_PREFIX, ADAPT_COLD_INIT = 1, 2, 3
ADAPT_REBIND_ACCEPT, ADAPT_REBIND_RESTART, ADAPT_REFRESH = 4, 5, 6
FIELD_X, FIELD_X_STAGE, FIELD_V_STEP, FIELD_X_INIT, FIELD_OBS, FIELD_RR_P, FIELD_RR_R, FIELD_META = range(8)
EPI_BF16, EPI_GELU_BF16, EPI_RESID_F32, EPI_F32 = 0, 1, 2, 3
KCLASSES = ["gemm", "attn", "norm", "cond", "adapt", "embed", "final", "rr_probe", "rr_apply"]


class WamError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{ERRORS.get(code, code)}: {msg}")
        self.code = code


class Config(ctypes.Structure):
    _fields_ = [
        ("n_layers", ctypes.c_int32), ("d_model", ctypes.c_int32), ("n_heads", ctypes.c_int32),
        ("mlp_ratio", ctypes.c_int32), ("n_obs", ctypes.c_int32), ("n_video", ctypes.c_int32),
        ("video_dim", ctypes.c_int32), ("n_action", ctypes.c_int32), ("action_dim", ctypes.c_int32),
        ("n_steps", ctypes.c_int32), ("precision", ctypes.c_int32), ("batch_max", ctypes.c_int32),
        ("sched_shift", ctypes.c_float),
        ("tr_entry_stage", ctypes.c_int32), ("tr_retain_stage", ctypes.c_int32),
        ("tr_normalize", ctypes.c_int32), ("tr_video_mode", ctypes.c_int32),
        ("rr_policy", ctypes.c_int32), ("rr_q", ctypes.c_int32), ("rr_s", ctypes.c_int32),
        ("rr_e", ctypes.c_int32),
        ("rr_alpha_min", ctypes.c_float), ("rr_alpha_max", ctypes.c_float), ("rr_eps", ctypes.c_float),
        ("rr_gamma_cos", ctypes.c_float), ("rr_gamma_fit", ctypes.c_float),
        ("or_tau", ctypes.c_float), ("or_kappa_max", ctypes.c_int32), ("or_n_components", ctypes.c_int32),
        ("or_deltas", ctypes.c_float * 4), ("or_weights", ctypes.c_float * 4),
    ]

    @classmethod
    def from_dict(cls, d: dict, batch_max: int | None = None) -> "Config":
        c = cls()
        for name, ctype in cls._fields_:
            if name == "precision":
                p = d.get("precision", "bf16")
                c.precision = PREC[p] if isinstance(p, str) else int(p)
            elif name == "batch_max":
                c.batch_max = int(batch_max if batch_max is not None else d.get("batch", 1))
            elif name in ("or_deltas", "or_weights"):
                vals = list(d.get(name, (1.0, 1.0, 1.0, 1.0)))[:4]
                getattr(c, name)[:] = [float(v) for v in vals] + [1.0] * (4 - len(vals))
            elif name in d:
                setattr(c, name, d[name])
            elif name == "tr_retain_stage":
                c.tr_retain_stage = -1
            elif name == "sched_shift":
                c.sched_shift = 1.0
        return c


class Stats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in (
        "n_attempt", "n_reuse", "b_skip", "b_dense", "n_start", "n_bind", "n_noninitial",
        "n_episode_steps", "n_layer_evals", "n_kernel_launches")]

    def as_dict(self) -> dict:
        return {n: int(getattr(self, n)) for n, _ in self._fields_}


class StepRecord(ctypes.Structure):
    _fields_ = [("episode", ctypes.c_int32), ("stage", ctypes.c_int32), ("rr_active", ctypes.c_int32),
                ("rr_attempt", ctypes.c_int32), ("rr_accept", ctypes.c_int32), ("pad_", ctypes.c_int32),
                ("alpha", ctypes.c_float * 2), ("cos", ctypes.c_float * 2), ("fit", ctypes.c_float * 2)]


class KClassTiming(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_int64), ("ms", ctypes.c_double), ("flops", ctypes.c_double),
                ("bytes", ctypes.c_double)]


_LIB = None
_vp = ctypes.c_void_p
_i32 = ctypes.c_int32


def lib() -> ctypes.CDLL:
    """Load the shared library once; raises if it has not been built."""
    global _LIB
    if _LIB is not None:
        return _LIB
    if not os.path.exists(_build.LIB_PATH):
        raise RuntimeError(f"{_build.LIB_PATH} is missing: build it with "
                           "`python -m paper_2609_34608_gb300._build` (nvcc, sm_103a)")
    L = ctypes.CDLL(_build.LIB_PATH)
    sig = {
        "wam_weight_count": (ctypes.c_size_t, [ctypes.POINTER(Config)]),
        "wam_create": (ctypes.c_int, [ctypes.POINTER(Config), _vp, ctypes.c_size_t, _vp, ctypes.POINTER(_vp)]),
        "wam_destroy": (None, [_vp]),
        "wam_last_error": (ctypes.c_char_p, [_vp]),
        "wam_set_stream": (ctypes.c_int, [_vp, _vp]),
        "wam_state_create": (ctypes.c_int, [_vp, _i32, ctypes.POINTER(_vp)]),
        "wam_state_destroy": (None, [_vp]),
        "wam_sample_cold": (ctypes.c_int, [_vp, _vp, _vp, _vp, _i32, _vp]),
        "wam_adapt_state": (ctypes.c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp]),
        "wam_continue": (ctypes.c_int, [_vp, _vp, _vp, _vp, _vp]),
        "wam_continue_many": (ctypes.c_int, [_i32, _vp, _vp, _vp, _vp, _vp, _vp]),
        "wam_get_stats": (ctypes.c_int, [_vp, ctypes.POINTER(Stats)]),
        "wam_reset_stats": (ctypes.c_int, [_vp]),
        "wam_state_log": (ctypes.c_int, [_vp, _vp, _i32, ctypes.POINTER(_i32)]),
        "wam_state_read": (ctypes.c_int, [_vp, _vp, _i32, _i32, _vp, ctypes.c_size_t]),
        "wam_state_write": (ctypes.c_int, [_vp, _vp, _i32, _i32, _vp, ctypes.c_size_t]),
        "wam_sync": (ctypes.c_int, [_vp]),
        "wam_profile_enable": (ctypes.c_int, [_vp, _i32]),
        "wam_profile_read": (ctypes.c_int, [_vp, _vp]),
        "wam_op_gemm_bf16": (ctypes.c_int, [_vp, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _vp, ctypes.c_int64, _i32, _vp]),
        "wam_op_gemm_f32": (ctypes.c_int, [_vp, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _vp, ctypes.c_int64, _i32, _vp]),
        "wam_op_gemm_bf16_plan": (ctypes.c_int, [_vp, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _vp, ctypes.c_int64, _i32,
                                                 _i32, _i32, _i32, _vp, ctypes.c_size_t, _vp]),
        "wam_op_gemm_workspace_bytes": (ctypes.c_size_t, []),
        "wam_op_gemm_plan": (ctypes.c_int, [_i32, _i32, _i32, _i32, _i32, _vp, _vp]),
        "wam_gemm_tile_width": (ctypes.c_int, [_vp, _i32, _i32, _i32, _i32]),
        "wam_set_graph_replay": (ctypes.c_int, [_vp, _i32]),
        "wam_set_layer_fusion": (ctypes.c_int, [_vp, _i32]),
        "wam_set_device_branching": (ctypes.c_int, [_vp, _i32]),
        "wam_profile_chain_trace": (ctypes.c_int, [_vp, _vp, _i32, ctypes.POINTER(_i32)]),
        "wam_diag_similarity": (ctypes.c_int, [_vp, _vp, _vp, ctypes.c_int64, _vp, _vp]),
        "wam_diag_action_rmse": (ctypes.c_int, [_vp, _vp, _vp, _i32, _i32, _i32, _vp]),
        "wam_diag_layer_deltas": (ctypes.c_int, [_vp, _vp, _i32, _vp]),
        "wam_diag_reuse_error": (ctypes.c_int, [_vp, _vp, _i32, _vp, _vp]),
        "wam_op_attention": (ctypes.c_int, [_vp, _vp, _i32, _i32, _i32, _i32, _i32, _vp]),
        "wam_op_ln_modulate": (ctypes.c_int, [_vp, _vp, _vp, ctypes.c_int64, _vp, _i32, _i32, _i32, _i32, _vp]),
        "wam_op_last_error": (ctypes.c_char_p, []),
        "wam_op_gemm_qkv_vt": (ctypes.c_int, [_vp, _vp, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _vp]),
        "wam_op_attention_tc": (ctypes.c_int, [_vp, _vp, _vp, _i32, _i32, _i32, _i32, _vp]),
        "wam_tr_remap_static": (ctypes.c_int, [_vp, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _i32, _i32,
                                               ctypes.c_double, ctypes.c_double, _i32, _i32, _vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _LIB = L
    return L


def header_functions() -> list[str]:
    """Names of every function declared in include/*.h."""
    names = []
    for h in ("wam.h", "wam_ops.h"):
        txt = open(os.path.join(_build.INCLUDE, h)).read()
        txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
        for line in txt.splitlines():
            if line.lstrip().startswith("#"):
                continue
            names += re.findall(r"\b(wam_\w+)\s*\(", line)
    return sorted(set(names))


def ptr(x) -> int | None:
    """Raw address of a numpy array or torch tensor (None passes NULL)."""
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("arrays must be C-contiguous")
        return x.ctypes.data
    if hasattr(x, "data_ptr"):
        if not x.is_contiguous():
            raise ValueError("tensors must be contiguous")
        return x.data_ptr()
    if isinstance(x, int):
        return x
    raise TypeError(f"unsupported buffer type {type(x)}")


def _i32_array(v, n: int):
    if v is None:
        return None
    a = np.ascontiguousarray(np.broadcast_to(np.asarray(v, dtype=np.int32), (n,)))
    return a


def weight_count(cfg: dict) -> int:
    c = Config.from_dict(cfg)
    return int(lib().wam_weight_count(ctypes.byref(c)))


class State:
    def __init__(self, ctx: "Context", batch: int):
        self.ctx = ctx
        self.batch = batch
        h = _vp()
        ctx._check(lib().wam_state_create(ctx.handle, batch, ctypes.byref(h)))
        self.handle = h
        ctx._states.add(self)

    def close(self):
        if self.handle:
            lib().wam_state_destroy(self.handle)
            self.handle = _vp()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Context:
    """One model + profile on the current CUDA device, bound to one stream."""

    def __init__(self, cfg: dict, weights, stream: int | None = None, batch_max: int | None = None):
        self.cfg = dict(cfg)
        self.config = Config.from_dict(cfg, batch_max)
        self.T = int(cfg["n_video"]) * int(cfg["video_dim"]) + int(cfg["n_action"]) * int(cfg["action_dim"])
        self.N = int(cfg["n_obs"]) + int(cfg["n_video"]) + int(cfg["n_action"])
        h = _vp()
        n = weights.numel() if hasattr(weights, "numel") else int(weights.size)
        code = lib().wam_create(ctypes.byref(self.config), ptr(weights), n, stream, ctypes.byref(h))
        if code != WAM_OK:
            raise WamError(code, "wam_create failed (see stderr)")
        self.handle = h
        self._states = weakref.WeakSet()

    def _check(self, code: int):
        if code != WAM_OK:
            raise WamError(code, lib().wam_last_error(self.handle).decode())

    def close(self):
        """Destroy every live state of this context, then the context itself."""
        if getattr(self, "handle", None):
            for st in list(getattr(self, "_states", ())):
                st.close()
            lib().wam_destroy(self.handle)
            self.handle = _vp()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_stream(self, stream: int | None):
        self._check(lib().wam_set_stream(self.handle, stream))

    def state(self, batch: int) -> State:
        return State(self, batch)

    def sample_cold(self, st: State, obs, noise, n_steps: int, actions_out=None):
        self._check(lib().wam_sample_cold(self.handle, st.handle, ptr(obs), ptr(noise), int(n_steps), ptr(actions_out)))

    def adapt(self, st: State, new_obs, shift=None, entry=None, fresh_noise=None) -> np.ndarray:
        status = np.zeros(st.batch, dtype=np.int32)
        sh = _i32_array(shift, st.batch)
        en = _i32_array(entry, st.batch)
        self._check(lib().wam_adapt_state(self.handle, st.handle, ptr(new_obs), ptr(sh), ptr(en),
                                          ptr(fresh_noise), ptr(status)))
        return status

    def continue_(self, st: State, n_steps, actions_out=None, video_out=None):
        n = _i32_array(n_steps, st.batch)
        self._check(lib().wam_continue(self.handle, st.handle, ptr(n), ptr(actions_out), ptr(video_out)))

    @staticmethod
    def continue_many(calls):
        """wam_continue_many: `calls` is a list of (context, state, n_steps, actions_out, video_out)
        on distinct contexts, advanced concurrently (one host thread each)."""
        n = len(calls)
        ctxs = (_vp * n)(*[c[0].handle.value for c in calls])
        states = (_vp * n)(*[c[1].handle.value for c in calls])
        steps = [_i32_array(c[2], c[1].batch) for c in calls]
        step_ptrs = (_vp * n)(*[s.ctypes.data for s in steps])
        outs_a = (_vp * n)(*[ptr(c[3]) if len(c) > 3 else None for c in calls])
        outs_v = (_vp * n)(*[ptr(c[4]) if len(c) > 4 else None for c in calls])
        status = np.zeros(n, dtype=np.int32)
        code = lib().wam_continue_many(n, ctxs, states, step_ptrs, outs_a, outs_v, status.ctypes.data)
        if code != WAM_OK:
            i = int(np.flatnonzero(status)[0]) if status.any() else 0
            calls[i][0]._check(code)
        return status

    def stats(self) -> dict:
        s = Stats()
        self._check(lib().wam_get_stats(self.handle, ctypes.byref(s)))
        return s.as_dict()

    def reset_stats(self):
        self._check(lib().wam_reset_stats(self.handle))

    def sync(self):
        self._check(lib().wam_sync(self.handle))

    def diag_similarity(self, a, b) -> tuple[float, float]:
        """App. E: (cosine, relative L2 against b) of two float32 vectors (host or device)."""
        c, r = ctypes.c_double(), ctypes.c_double()
        n = a.numel() if hasattr(a, "numel") else int(np.asarray(a).size)
        self._check(lib().wam_diag_similarity(self.handle, ptr(a), ptr(b), n, ctypes.byref(c), ctypes.byref(r)))
        return c.value, r.value

    def diag_action_rmse(self, a, b, dims: int = 6) -> float:
        """App. E Eq. 17: RMSE over the first `dims` values of each action row."""
        shape = tuple(a.shape)
        out = ctypes.c_double()
        self._check(lib().wam_diag_action_rmse(self.handle, ptr(a), ptr(b), int(np.prod(shape[:-1])), int(shape[-1]),
                                               int(dims), ctypes.byref(out)))
        return out.value

    def diag_layer_deltas(self, st: "State", episode: int) -> np.ndarray:
        """App. E: relative hidden-state change across each layer at the episode's pending stage."""
        out = np.zeros(int(self.cfg["n_layers"]), dtype=np.float64)
        self._check(lib().wam_diag_layer_deltas(self.handle, st.handle, int(episode), out.ctypes.data))
        return out

    def diag_reuse_error(self, st: "State", episode: int) -> tuple[float, list]:
        """App. E: output error of residual reuse against full computation at the episode's pending
        stage, and the Eq. 7 factor per branch."""
        e = ctypes.c_double()
        al = (ctypes.c_double * 2)()
        self._check(lib().wam_diag_reuse_error(self.handle, st.handle, int(episode), ctypes.byref(e), al))
        return e.value, [al[0], al[1]]

    def set_graph_replay(self, enable: bool):
        """CUDA-graph replay of the layer stack (default on); off launches every kernel."""
        self._check(lib().wam_set_graph_replay(self.handle, 1 if enable else 0))

    def set_device_branching(self, enable: bool):
        """RR decision of a single work item taken on the device inside the step's CUDA graph
        (default on); off reads the gate statistics back to the host every step."""
        self._check(lib().wam_set_device_branching(self.handle, 1 if enable else 0))

    def set_layer_fusion(self, enable: bool):
        """Fused row-chain launches between attentions (default off); off launches each kernel."""
        self._check(lib().wam_set_layer_fusion(self.handle, 1 if enable else 0))

    def gemm_tile_width(self, M: int, N: int, K: int, epilogue: int) -> int:
        """Output tile width the context uses for this GEMM shape (chosen from the shape alone)."""
        r = lib().wam_gemm_tile_width(self.handle, M, N, K, epilogue)
        if r < 0:
            self._check(r)
        return r

    def log(self, st: State) -> list[dict]:
        n = _i32()
        self._check(lib().wam_state_log(st.handle, None, 0, ctypes.byref(n)))
        recs = (StepRecord * max(1, n.value))()
        self._check(lib().wam_state_log(st.handle, recs, n.value, ctypes.byref(n)))
        out = []
        for r in recs[: n.value]:
            out.append(dict(episode=r.episode, stage=r.stage, rr_active=bool(r.rr_active),
                            rr_attempt=bool(r.rr_attempt), rr_accept=bool(r.rr_accept),
                            alpha=list(r.alpha), cos=list(r.cos), fit=list(r.fit)))
        return out

    def _field_shape(self, st: State, field: int):
        B, d = st.batch, int(self.cfg["d_model"])
        if field in (FIELD_X, FIELD_X_STAGE, FIELD_V_STEP, FIELD_X_INIT):
            return (B, self.T), np.float32
        if field == FIELD_OBS:
            return (B, int(self.cfg["n_obs"]), d), np.float32
        if field in (FIELD_RR_P, FIELD_RR_R):
            return (B, self.N, d), np.float32
        if field == FIELD_META:
            return (B, 8), np.int32
        raise ValueError(field)

    def read(self, st: State, field: int, index: int = 0) -> np.ndarray:
        shape, dt = self._field_shape(st, field)
        out = np.empty(shape, dtype=dt)
        self._check(lib().wam_state_read(self.handle, st.handle, field, index, ptr(out), out.nbytes))
        return out

    def write(self, st: State, field: int, value, index: int = 0):
        shape, dt = self._field_shape(st, field)
        a = np.ascontiguousarray(np.asarray(value, dtype=dt).reshape(shape))
        self._check(lib().wam_state_write(self.handle, st.handle, field, index, ptr(a), a.nbytes))

    def profile_enable(self, on: bool = True):
        self._check(lib().wam_profile_enable(self.handle, 1 if on else 0))

    def profile_chain_trace(self) -> np.ndarray:
        """Per-task records of the fused row-chain launches since profiling was enabled: a numpy
        structured array (launch, cta, kind, m, j, t_take, t_dep, t_epi0, t_epi1; times in ns)."""
        n = _i32()
        self._check(lib().wam_profile_chain_trace(self.handle, None, 0, ctypes.byref(n)))
        dt = np.dtype([("launch", "<i4"), ("cta", "<i4"), ("kind", "<i4"), ("m", "<i4"), ("j", "<i4"),
                       ("pad", "<i4"), ("t_take", "<u8"), ("t_dep", "<u8"), ("t_epi0", "<u8"), ("t_epi1", "<u8")])
        out = np.zeros(max(1, n.value), dtype=dt)
        self._check(lib().wam_profile_chain_trace(self.handle, out.ctypes.data, n.value, ctypes.byref(n)))
        return out[: n.value]

    def profile_read(self) -> dict:
        arr = (KClassTiming * len(KCLASSES))()
        self._check(lib().wam_profile_read(self.handle, arr))
        return {k: dict(launches=int(t.launches), ms=float(t.ms), flops=float(t.flops), bytes=float(t.bytes))
                for k, t in zip(KCLASSES, arr)}


# ---- kernel-level ops (wam_ops.h) -------------------------------------------------------
def _op_check(code: int):
    if code != WAM_OK:
        raise WamError(code, lib().wam_op_last_error().decode())


def op_gemm_bf16(A, Wt, bias, C, M, N, K, epilogue, gate=None, gate_stride=0, rows_per_item=1, stream=None):
    _op_check(lib().wam_op_gemm_bf16(ptr(A), ptr(Wt), ptr(bias), ptr(C), M, N, K, epilogue, ptr(gate),
                                     gate_stride, rows_per_item, stream))


def op_gemm_bf16_plan(A, Wt, bias, C, M, N, K, epilogue, tile_n, k_splits, workspace=None, gate=None,
                      gate_stride=0, rows_per_item=1, stream=None, cluster=0):
    """wam_op_gemm_bf16 with an explicit output tile width, K split and cluster size (0 = the
    library's rule, 1 = single CTAs, 2 = pairs sharing the A tile); workspace: a zero-filled device
    buffer of gemm_workspace_bytes() bytes, needed when k_splits > 1."""
    nbytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _op_check(lib().wam_op_gemm_bf16_plan(ptr(A), ptr(Wt), ptr(bias), ptr(C), M, N, K, epilogue, ptr(gate),
                                          gate_stride, rows_per_item, tile_n, k_splits, cluster, ptr(workspace),
                                          nbytes, stream))


def gemm_workspace_bytes():
    return int(lib().wam_op_gemm_workspace_bytes())


def gemm_plan(M, N, K, residual, num_sms):
    """The shape rule's plan for a bf16 projection (host only): (tile width, on CTA pairs)."""
    tn, pairs = _i32(), _i32()
    _op_check(lib().wam_op_gemm_plan(M, N, K, 1 if residual else 0, num_sms, ctypes.byref(tn), ctypes.byref(pairs)))
    return tn.value, bool(pairs.value)


def op_gemm_f32(A, Wt, bias, C, M, N, K, epilogue, gate=None, gate_stride=0, rows_per_item=1, stream=None):
    _op_check(lib().wam_op_gemm_f32(ptr(A), ptr(Wt), ptr(bias), ptr(C), M, N, K, epilogue, ptr(gate),
                                    gate_stride, rows_per_item, stream))


def op_attention(qkv, out, B, N, d, n_heads, precision="bf16", stream=None):
    _op_check(lib().wam_op_attention(ptr(qkv), ptr(out), B, N, d, n_heads, PREC[precision], stream))


def op_gemm_qkv_vt(A, Wt, bias, qkv, vt, M, d, rows_per_item, vt_ld, stream=None):
    _op_check(lib().wam_op_gemm_qkv_vt(ptr(A), ptr(Wt), ptr(bias), ptr(qkv), ptr(vt), M, d, rows_per_item, vt_ld,
                                       stream))


def op_attention_tc(qkv, vt, out, B, N, d, n_heads, stream=None):
    _op_check(lib().wam_op_attention_tc(ptr(qkv), ptr(vt), ptr(out), B, N, d, n_heads, stream))


def op_ln_modulate(h, shift, scale, mod_stride, out, M, d, rows_per_item, precision="bf16", stream=None):
    _op_check(lib().wam_op_ln_modulate(ptr(h), ptr(shift), ptr(scale), mod_stride, ptr(out), M, d,
                                       rows_per_item, PREC[precision], stream))


def tr_remap_static(x_bar, x_r, eps, out, batch, n_video, video_dim, n_action, action_dim, shift,
                    sigma_r, sigma_b0, normalize=1, video_mode=0, stream=None):
    """Trajectory Remapping without any device allocation (see include/wam_ops.h)."""
    _op_check(lib().wam_tr_remap_static(ptr(x_bar), ptr(x_r), ptr(eps), ptr(out), batch, n_video, video_dim,
                                        n_action, action_dim, shift, float(sigma_r), float(sigma_b0),
                                        normalize, video_mode, stream))
