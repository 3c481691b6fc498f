import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a); parity tests of the CUDA path")


def oracle_family(fam, base, experts, trim_scope=0):
    """Wrap a synthetic family's numpy data as an oracle.Family (group = tensor, or 0)."""
    import oracle

    bo, bl, bt = fam.block_table()
    groups = bt if trim_scope == 0 else np.zeros_like(bt)
    n_groups = len(fam.tensors) if trim_scope == 0 else 1
    return oracle.Family(fam.dtype, bo, bl, groups, n_groups, base, experts)


@pytest.fixture(scope="session")
def tiny_family():
    from paper_2605_29489_gb300 import synth

    fam = synth.tiny()
    base, experts = fam.host_arrays()
    return fam, base, experts
