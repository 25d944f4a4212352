import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and runs the CUDA library")
    config.addinivalue_line("markers", "slow: full-size workloads")
    # Build what the tests load: the oracle and the host generator always, the
    # CUDA library (cross-compiled; its import needs no GPU) too.
    from oracle.build import build as build_oracle
    from synth.build import build_host
    build_oracle()
    build_host()
    import importlib.util
    spec = importlib.util.spec_from_file_location(
        "_das_build", os.path.join(ROOT, "paper_2609_34538_gb300", "build.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    mod.build()


def pytest_collection_modifyitems(config, items):
    import torch
    if torch.cuda.is_available():
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)
