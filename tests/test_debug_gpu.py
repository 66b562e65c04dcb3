"""The -DDART_DEBUG build of the library.

Its kernels check every data-dependent index (parent slots against the
previous depth's count, token ids against V, output positions against B)
before using it; a failed check skips the access and sets a status bit that
dart_status_sync returns as DART_ERR_BOUNDS.  Here: the report path works
(one check made to fail, touching no memory), and the small oracle parity
cases and the best-first constructions pass under the debug build with no
check failing (every one of those tests asserts dart_status_sync == OK).
"""
import os
import subprocess
import sys

import pytest
import torch

from workloads import Config, make_inputs
from parity import to_device

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def dart():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13524_gb300 import dart as d
    d.lib()
    return d


def small_handle(dart):
    cfg = Config("debug-probe", 2, 3000, 256, 3, 4, 4, 8, "bf16", 0.0, 77)
    dx = to_device(cfg, make_inputs(cfg))
    return dart.dart_init_head(cfg, dart.DART_BF16, dx["Wi"], dx["Wo"], dx["E"])


def test_bounds_report_of_this_build(dart):
    """Release: the check compiles away; debug (the test process below):
    DART_ERR_BOUNDS once, then cleared."""
    h = small_handle(dart)
    try:
        dart.dart_test_bounds_report(h)
        if dart.dart_debug_build():
            assert dart.dart_status_sync(h) == dart.DART_ERR_BOUNDS
        assert dart.dart_status_sync(h) == dart.DART_OK
    finally:
        dart.dart_destroy(h)


def test_debug_build_passes_the_parity_cases(dart):
    if os.environ.get("DART_TEST_LIBRARY"):
        pytest.skip("already the debug library's test process")
    assert not dart.dart_debug_build()
    from paper_2608_13524_gb300 import build
    lib = build.build(debug=True)
    env = dict(os.environ, DART_TEST_LIBRARY=lib)
    cmd = [sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-p", "no:cacheprovider",
           "tests/test_debug_gpu.py::test_bounds_report_of_this_build",
           "tests/test_debug_gpu.py::test_the_debug_library_is_loaded",
           "tests/test_parity_gpu.py::test_depthwise_parity",
           "tests/test_parity_gpu.py::test_build_tree_graph_matches_depthwise",
           "tests/test_parity_gpu.py::test_neg_inf_drafter_logits",
           "tests/test_parity_gpu.py::test_restricted_candidates_and_neg_inf",
           "tests/test_parity_gpu.py::test_fused_round_parity",
           "tests/test_parity_gpu.py::test_fused_round_neg_inf_and_states",
           "tests/test_heap_gpu.py::test_chain_ddtree_and_seq_heap_parity",
           "tests/test_heap_gpu.py::test_variants_and_algorithm1_on_one_handle",
           "tests/test_heap_gpu.py::test_dartree_fixed"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=1800)
    tail = (r.stdout[-4000:] + "\n" + r.stderr[-2000:]).strip()
    assert r.returncode == 0, tail
    summary = r.stdout.strip().splitlines()[-1]
    print(summary)
    assert " passed" in summary and "skipped" not in summary and "deselected" not in summary, summary


def test_the_debug_library_is_loaded(dart):
    if not os.environ.get("DART_TEST_LIBRARY"):
        pytest.skip("runs in the debug library's test process")
    assert dart.dart_debug_build()
