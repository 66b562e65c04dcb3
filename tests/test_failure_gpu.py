"""Failure detection on the GPU without a fault.

Every device-side wait of the library is bounded: a wait that runs out sets
the CTA's abort flag and a status bit, the other waits of the CTA give up as
soon as they see the flag, and dart_status_sync reports DART_ERR_TIMEOUT.
Here a wait is made to run out on purpose (an mbarrier nothing completes, a
short limit, no copy or MMA in flight) and the handle is then used again.
"""
import time

import numpy as np
import pytest
import torch

import oracle
from parity import compare_with_oracle, gpu_supertree, to_device, tol_of, tree_to_numpy
from workloads import Config, make_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dart():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13524_gb300 import dart as d
    d.lib()
    return d


def test_a_device_wait_that_runs_out_is_reported_and_the_handle_recovers(dart):
    cfg = Config("timeout", 2, 3000, 128, 4, 6, 6, 20, "bf16", 0.0, 77)
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    eng = dart.Dart(cfg, dx["Wi"], dx["Wo"], dx["E"])
    try:
        before = tree_to_numpy(eng.build_tree(dx["Dlog"], dx["h0"]))
        assert dart.dart_status_sync(eng.h) == dart.DART_OK
        limit_us = 200
        el = torch.full((2,), -1, dtype=torch.int64, device="cuda")
        t0 = time.perf_counter()
        dart.dart_test_wait_timeout(eng.h, limit_us, el)
        rc = dart.dart_status_sync(eng.h)
        wall = time.perf_counter() - t0
        assert rc == dart.DART_ERR_TIMEOUT
        e = el.cpu().numpy()
        # the short wait gave up after its limit, not much later
        assert limit_us * 1000 <= e[0] < 50_000_000, e
        # the other wait (the kernels' 2 s limit) returned on the abort flag
        assert 0 <= e[1] < 100_000_000, e
        assert wall < 1.5, wall
        # the status word was cleared by the read, and the context is intact
        assert dart.dart_status_sync(eng.h) == dart.DART_OK
        after = tree_to_numpy(eng.build_tree(dx["Dlog"], dx["h0"]))
        assert dart.dart_status_sync(eng.h) == dart.DART_OK
        for k in before:
            np.testing.assert_array_equal(after[k], before[k], err_msg=k)
        gst = gpu_supertree(dart, eng.h, cfg)
    finally:
        eng.close()
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    compare_with_oracle(cfg, ref, gst, after, tol_of(cfg), x=x)


def test_wait_probe_rejects_bad_limits(dart):
    cfg = Config("timeout-args", 1, 500, 64, 2, 2, 2, 4, "bf16", 0.0, 78)
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    eng = dart.Dart(cfg, dx["Wi"], dx["Wo"], dx["E"])
    try:
        for bad in (0, -5, 2_000_001):
            with pytest.raises(dart.DartError) as e:
                dart.dart_test_wait_timeout(eng.h, bad)
            assert e.value.code == dart.DART_ERR_INVALID
        assert dart.dart_status_sync(eng.h) == dart.DART_OK
    finally:
        eng.close()


def test_the_graph_cache_is_bounded_and_rotating_buffers_stay_correct(dart):
    """More distinct output pointer sets than the handle caches graphs for,
    used in rotation: every launch returns the same tree (evicted graphs are
    rebuilt on their next use)."""
    cfg = Config("graphs", 1, 2000, 128, 3, 4, 4, 10, "bf16", 1.0, 79)
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    eng = dart.Dart(cfg, dx["Wi"], dx["Wo"], dx["E"])
    try:
        ref = tree_to_numpy(eng.build_tree(dx["Dlog"], dx["h0"]))
        outs = [dart.alloc_tree_out(cfg) for _ in range(11)]
        for it in range(3):
            for t, o in outs:
                dart.dart_build_tree(eng.h, dx["Dlog"], dx["h0"], o)
        assert dart.dart_status_sync(eng.h) == dart.DART_OK
        for t, _ in outs:
            g = tree_to_numpy(t)
            for k in ref:
                np.testing.assert_array_equal(g[k], ref[k], err_msg=k)
    finally:
        eng.close()


def test_a_grid_barrier_that_runs_out_is_reported_and_the_fused_round_recovers(dart):
    """The fused round's grid barrier with a short limit and a block that
    never arrives (no copy or computation in flight): DART_ERR_TIMEOUT, the
    handle refuses rounds until the status is read, then the barrier is reset
    and the next round is the oracle's tree again."""
    # (V = 60000: the grid form of the fused round, whose barrier this is)
    cfg = Config("barrier-timeout", 1, 60000, 128, 4, 4, 4, 12, "f32", 0.0, 80, fused_round=1)
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    eng = dart.Dart(cfg, dx["Wi"], dx["Wo"], dx["E"])
    try:
        before = tree_to_numpy(eng.build_tree(dx["Dlog"], dx["h0"]))
        assert dart.dart_status_sync(eng.h) == dart.DART_OK
        t0 = time.perf_counter()
        dart.dart_test_barrier_timeout(eng.h, 300)
        with pytest.raises(dart.DartError) as e:
            eng.build_tree(dx["Dlog"], dx["h0"])
        assert e.value.code == dart.DART_ERR_STATE
        assert dart.dart_status_sync(eng.h) == dart.DART_ERR_TIMEOUT
        assert time.perf_counter() - t0 < 1.5
        assert dart.dart_status_sync(eng.h) == dart.DART_OK
        after = tree_to_numpy(eng.build_tree(dx["Dlog"], dx["h0"]))
        assert dart.dart_status_sync(eng.h) == dart.DART_OK
        for k in before:
            np.testing.assert_array_equal(after[k], before[k], err_msg=k)
        gst = gpu_supertree(dart, eng.h, cfg)
    finally:
        eng.close()
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    compare_with_oracle(cfg, ref, gst, after, tol_of(cfg), x=x)
    # a handle without the fused round has no barrier to probe
    cfg2 = cfg.replace(fused_round=2)
    eng = dart.Dart(cfg2, dx["Wi"], dx["Wo"], dx["E"])
    try:
        with pytest.raises(dart.DartError) as e:
            dart.dart_test_barrier_timeout(eng.h, 300)
        assert e.value.code == dart.DART_ERR_STATE
    finally:
        eng.close()
