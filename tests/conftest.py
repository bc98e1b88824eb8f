import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")


@pytest.fixture(autouse=True)
def _device_status_clean(request):
    """After every GPU test: no bounded wait inside the tensor-core kernels gave up."""
    yield
    if request.node.get_closest_marker("gpu") is None:
        return
    from paper_2011_14504_gb300 import iq
    assert iq.iq_device_status() == 0
