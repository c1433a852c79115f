import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: full-size workload (minutes)")


def bf16_to_u16(t):
    """bf16 torch tensor -> numpy uint16 bit patterns (what the oracle accepts)."""
    import torch
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def oracle_weights(w):
    """synth.make_weights output -> oracle weight dict (bf16 bit patterns)."""
    return {
        "embed": bf16_to_u16(w["embed"]),
        "lm_head": bf16_to_u16(w["lm_head"]),
        "final_norm": bf16_to_u16(w["final_norm"]),
        "layers": [None if lw is None else {k: bf16_to_u16(v) for k, v in lw.items()} for lw in w["layers"]],
    }


@pytest.fixture(scope="session")
def tiny_weights():
    from paper_2609_26100_gb300 import synth
    return synth.make_weights(synth.TINY)


@pytest.fixture(scope="session")
def tiny_oracle_weights(tiny_weights):
    return oracle_weights(tiny_weights)
