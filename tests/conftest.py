import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
HERE = os.path.dirname(os.path.abspath(__file__))
if HERE not in sys.path:
    sys.path.insert(0, HERE)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    # A test run against another build of the library (the -DDART_DEBUG one):
    # the path is set before any test loads it.
    other = os.environ.get("DART_TEST_LIBRARY")
    if other:
        from paper_2608_13524_gb300 import dart
        dart.LIB_PATH = os.path.abspath(other)


@pytest.fixture(autouse=True)
def guarded_outputs(request):
    """GPU tests: every device output of the binding carries guard bytes on
    both sides, checked when the test ends."""
    if request.node.get_closest_marker("gpu") is None:
        yield
        return
    import canary
    from paper_2608_13524_gb300 import dart
    canary.reset()
    dart.set_output_allocator(canary.empty)
    try:
        yield
    finally:
        dart.set_output_allocator(None)
    import torch
    if torch.cuda.is_available():
        torch.cuda.synchronize()
        canary.check()
    canary.reset()
