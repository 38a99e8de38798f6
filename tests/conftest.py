import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running check")


def read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line)
    return rows


@pytest.fixture(scope="session")
def tiny_cfg():
    from paper_2609_37007_gb300.synth import TINY
    return TINY


@pytest.fixture(scope="session")
def tiny_model(tiny_cfg):
    from paper_2609_37007_gb300.synth import make_weights, weights_as_f32
    from oracle.model import Model
    return Model(tiny_cfg, weights_as_f32(tiny_cfg, make_weights(tiny_cfg)))
