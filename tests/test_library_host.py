"""Host-side checks of the CUDA library that need no GPU: it builds, loads, exports every
function include/*.h declares, agrees with the input generator on the weight layout, and
rejects invalid configurations before touching the device."""
import ctypes
import os

import pytest

from paper_2609_34608_gb300 import _build, inputs
from paper_2609_34608_gb300 import wam as W


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(_build.LIB_PATH):
        _build.build()
    return W.lib()


def test_every_header_function_is_exported(lib):
    names = W.header_functions()
    assert len(names) >= 20
    missing = [n for n in names if not hasattr(lib, n)]
    assert missing == []


@pytest.mark.parametrize("name", sorted(inputs.NAMED_CONFIGS))
def test_weight_count_matches_generator_layout(lib, name):
    cfg = inputs.get_config(name)
    assert W.weight_count(cfg) == inputs.weight_count(cfg)


def _create(cfg):
    c = W.Config.from_dict(cfg)
    h = ctypes.c_void_p()
    n = inputs.weight_count(cfg)
    buf = (ctypes.c_float * 1)()
    return W.lib().wam_create(ctypes.byref(c), buf, n, None, ctypes.byref(h))


@pytest.mark.parametrize("bad, code", [
    (dict(d_model=130), 1),                         # not a multiple of n_heads (4)
    (dict(rr_policy=1, rr_q=1, rr_s=1, rr_e=1), 1),  # boundaries not increasing
    (dict(tr_entry_stage=8), 1),                     # entry stage must be < K
    (dict(or_n_components=3), 1),                    # 3 does not divide 16 obs tokens
    (dict(batch=0), 1),                              # batch_max below 1
    (dict(d_model=96, n_heads=3), 6),                # width not a multiple of 128
    (dict(video_dim=32), 6),                         # output head wider than 16
    (dict(n_video=0, n_action=0), 1),                # a model needs video or action tokens
    (dict(n_action=-1), 1),                          # negative token count
])
def test_invalid_configs_are_rejected_before_device_work(lib, bad, code):
    cfg = inputs.get_config("tiny", **bad)
    assert _create(cfg) == code


def test_weight_buffer_size_is_checked(lib):
    cfg = inputs.get_config("tiny")
    c = W.Config.from_dict(cfg)
    h = ctypes.c_void_p()
    buf = (ctypes.c_float * 1)()
    assert lib.wam_create(ctypes.byref(c), buf, inputs.weight_count(cfg) - 1, None, ctypes.byref(h)) == 1
    assert lib.wam_create(ctypes.byref(c), None, inputs.weight_count(cfg), None, ctypes.byref(h)) == 1


def test_config_struct_matches_header_size(lib):
    # 12 ints + 1 float + 4 ints + 4 ints + 5 floats + 1 float + 2 ints + 8 floats = 37 x 4 bytes
    assert ctypes.sizeof(W.Config) == 37 * 4
    assert ctypes.sizeof(W.StepRecord) == 12 * 4


def test_every_header_function_has_a_binding_signature(lib):
    """The Python binding declares argument and result types for every function of include/*.h
    (no call goes through ctypes' default int conversion)."""
    W.lib()
    for name in W.header_functions():
        fn = getattr(lib, name)
        assert fn.argtypes is not None, name


# (rows, N, K, residual) -> (tile width, CTA pairs) on the 152 SMs of a GB300: the plans the shape
# rule gives the three models' projections.  One episode of the d768 model stays on single CTAs
# (its launches are bound by fixed costs); 32 serving episodes run 256-wide pairs; at 8 bimanual
# episodes N = 3456 / 1152 rule out 256-wide tiles, so the 128-wide tiles that fill four waves pair.
GEMM_PLANS = [
    ((1296, 768, 768, True), (64, False)),      # one episode: attention out-projection
    ((1296, 3072, 768, False), (128, False)),   # MLP up
    ((1296, 768, 3072, True), (64, False)),     # MLP down
    ((1296, 2304, 768, False), (128, False)),   # QKV
    ((78848, 3072, 1024, False), (256, True)),  # 32 serving episodes: QKV
    ((78848, 4096, 1024, False), (256, True)),  # MLP up
    ((78848, 1024, 4096, True), (256, True)),   # MLP down
    ((39312, 3456, 1152, False), (128, True)),  # 8 bimanual episodes: QKV
    ((39312, 1152, 4608, True), (128, True)),   # MLP down
    ((39312, 4608, 1152, False), (256, True)),  # MLP up
    ((272, 2304, 768, False), (128, False)),    # a small non-residual projection keeps 128-wide tiles
    ((272, 768, 768, True), (64, False)),       # ... and a small residual one takes 64-wide tiles
    ((78848, 1024, 192, False), (256, False)),  # K % 128 != 0: no pairs
]


@pytest.mark.parametrize("shape,plan", GEMM_PLANS)
def test_gemm_shape_rule(lib, shape, plan):
    M, N, K, resid = shape
    tile, pairs = W.gemm_plan(M, N, K, resid, 152)
    assert (tile, pairs) == plan
    assert N % tile == 0


def test_gemm_plan_query_rejects_bad_sizes(lib):
    for bad in ((0, 768, 768), (1296, 100, 768), (1296, 768, 96)):
        with pytest.raises(W.WamError):
            W.gemm_plan(*bad, True, 152)
