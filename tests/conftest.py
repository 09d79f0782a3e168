import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running oracle case")


@pytest.fixture(scope="session")
def tiny_setup():
    """Tiny fp32 config, its weights (fp64 oracle view) and prompt."""
    import synth
    from oracle import chimera_oracle as co
    cfg = synth.get_config("tiny")
    w = synth.make_weights(cfg)
    return cfg, w, co.OracleWeights(w), synth.make_prompts(cfg)[0]
