import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a GB300 and the built CUDA library")


def micro_config(**overrides):
    """A very small model for fast CPU tests of the oracle's logic."""
    from paper_2609_34608_gb300.inputs import METHOD_DEFAULTS
    cfg = dict(METHOD_DEFAULTS)
    cfg.update(n_layers=3, d_model=16, n_heads=2, mlp_ratio=4, n_obs=4, n_video=6,
               video_dim=4, n_action=5, action_dim=3, n_steps=4, precision="fp32", batch=1,
               tr_entry_stage=2, tr_retain_stage=-1, rr_policy=0, rr_q=0, rr_s=0, rr_e=0)
    cfg.update(overrides)
    return cfg


@pytest.fixture
def micro():
    return micro_config


def pytest_collection_modifyitems(config, items):
    """GPU tests need a CUDA device; on a machine without one they are skipped, never faked."""
    try:
        import torch
        has_gpu = torch.cuda.is_available()
    except Exception:
        has_gpu = False
    if has_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


@pytest.fixture(scope="session")
def wamlib():
    """The built CUDA library (built in-tree if stale)."""
    from paper_2609_34608_gb300 import _build
    from paper_2609_34608_gb300 import wam as W
    _build.build()
    return W.lib()
