import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built libjq.so")
    config.addinivalue_line("markers", "slow: long-running CPU test")
    config.addinivalue_line("markers", "late: parity cases of the newest kernels, run after all others")


def pytest_collection_modifyitems(config, items):
    # Long cases run last (stable sort: the order is otherwise unchanged), so that a slow case
    # cannot delay the rest, nor, under -x, keep them from running; the newest kernels' cases
    # come after those, so that under -x they cannot keep the established cases from running.
    items.sort(key=lambda item: 2 if item.get_closest_marker("late") is not None
               else int(item.get_closest_marker("slow") is not None))
