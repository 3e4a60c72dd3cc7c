import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long CPU test")


@pytest.fixture(scope="session")
def micro_cfg():
    """A one-layer micro model small enough for scalar brute force."""
    return dict(name="micro", n_layers=1, d_model=8, n_heads=2, n_kv_heads=1, head_dim=4, ffn=12,
                vocab=16, mask_id=15, rope_theta=10000.0, norm_eps=1e-5,
                init_sigma=0.5, head_sigma=1.5, seed=7)
