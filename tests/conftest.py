import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a GB300 (sm_103a) and the built CUDA library")
    config.addinivalue_line("markers", "slow: full-size case, minutes of CPU work")


import pytest  # noqa: E402


@pytest.fixture(autouse=True)
def _release_device_buffers():
    """Drop the device buffers a GPU test kept alive (tests/gpu_helpers.KEEP)."""
    yield
    mod = sys.modules.get("tests.gpu_helpers")
    if mod is not None:
        mod.KEEP.clear()
