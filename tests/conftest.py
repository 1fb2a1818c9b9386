import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_addoption(parser):
    parser.addoption("--long", action="store_true", default=False,
                     help="also run the full-size checks of every output (the oracle recomputes "
                          "the whole batch: minutes of CPU work per test)")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a GB300 (sm_103a) GPU and the built libolive.so")
    config.addinivalue_line("markers", "slow: full-size parity case (minutes of CPU oracle work)")
    config.addinivalue_line("markers", "long: full-size check of every output; runs only with --long")


def pytest_collection_modifyitems(config, items):
    if not config.getoption("--long"):
        skip_long = pytest.mark.skip(reason="full-size check: pass --long")
        for item in items:
            if "long" in item.keywords:
                item.add_marker(skip_long)
    # GPU tests need CUDA; they are selected with -m gpu on the GPU machine.
    try:
        import torch
        has_cuda = torch.cuda.is_available()
    except Exception:  # pragma: no cover
        has_cuda = False
    if has_cuda:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)
