import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device and the built libhilo")
    config.addinivalue_line("markers", "slow: long CPU test")


@pytest.fixture(autouse=True)
def _device_status_clean(request):
    """After every GPU test: no device-side wait ran out and (in the checks
    build) no index check failed, whether or not the test read the status."""
    yield
    if request.node.get_closest_marker("gpu") is None:
        return
    from paper_2606_13898_gb300 import hilo as H
    if H._lib is not None:
        H.hilo_sync_status()
