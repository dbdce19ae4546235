import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running on CPU")


def pytest_collection_modifyitems(config, items):
    # Keep file order (pytest default), but make sure files named test_zz_*
    # run after everything else even if collected from several directories.
    items.sort(key=lambda it: os.path.basename(str(it.fspath)).startswith("test_zz_"))
