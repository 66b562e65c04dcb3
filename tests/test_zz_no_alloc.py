"""The allocation-free depth-1 entry point against the regular handle path.

dart_expand_root_noalloc serves callers that cannot allocate device memory
while they run (a serving engine whose memory pool owns every free byte, or a
path where cudaMalloc's implicit synchronisation is not allowed): it keeps its
scratch in a static device array instead.  This file is collected last on
purpose, so a failure here cannot hide the result of any other test.
"""
import ctypes as C

import numpy as np
import pytest
import torch

import canary
from parity import to_device, tol_of
from workloads import Config, make_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dart():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13524_gb300 import dart as d
    d.lib()
    return d


def handle_depth1(dart, cfg, dx):
    """What the existing entry points return for depth 1."""
    h = dart.dart_init_head(cfg, dart.DART_BF16, dx["Wi"], dx["Wo"], dx["E"])
    try:
        dart.dart_expand_depth(h, 1, dx["Dlog"], dx["h0"])
        tok, logq, lse = dart.dart_get_node_topk(h, cfg)
        ftok, _, fsc, fcnt = dart.dart_get_frontier(h, 1, cfg)
        assert dart.dart_status_sync(h) == 0
        return [t.cpu().numpy() for t in (tok, logq, lse, ftok, fsc, fcnt)]
    finally:
        dart.dart_destroy(h)


def outputs(nseq, W, k):
    """Output tensors pre-filled with values no correct call leaves behind,
    each between guard bytes (checked when the test ends)."""
    spec = [((nseq, k), torch.int32, -7), ((nseq, k), torch.float32, 7.0), ((nseq,), torch.float32, 7.0),
            ((nseq, W), torch.int32, -7), ((nseq, W), torch.float32, 7.0), ((nseq,), torch.int32, -7)]
    return [canary.empty(shape, dtype=dt, device="cuda").fill_(v) for shape, dt, v in spec]


def dirty_the_array(dart):
    """One call of another shape (64 roots, d = 4096, k = 64), so the static
    array holds this call's partial lists, states and padding rows when the
    next call starts."""
    cfg = Config("noalloc-dirty", 64, 30000, 4096, 2, 64, 64, 64, "bf16", 0.5, 8999)
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    dart.dart_expand_root_noalloc(cfg, dx["E"], dx["Dlog"], dx["h0"], *outputs(64, 64, 64))
    assert dart.dart_noalloc_status() == dart.DART_OK


CASES = [(3, 20000, 512, 8, 12, 0.7),      # 16-node group, W <= k
         (1, 151936, 4096, 16, 16, 1.0),   # the Qwen3-8B shape
         (40, 20000, 2560, 6, 4, 0.0),     # 64-node group, W > k (unused frontier ranks), greedy T = 0
         (17, 9000, 1024, 8, 8, 0.3)]      # 32-node group


@pytest.mark.parametrize("nseq,V,d,W,k,T", CASES)
def test_noalloc_matches_handle_path_twice(dart, nseq, V, d, W, k, T):
    cfg = Config("noalloc", nseq, V, d, 4, W, k, 20, "bf16", T, 9000 + nseq)
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    ref = handle_depth1(dart, cfg, dx)
    tol = tol_of(cfg)
    dirty_the_array(dart)
    for call in range(2):  # the second call reuses the array the first one left behind
        out = outputs(nseq, W, k)
        dart.dart_expand_root_noalloc(cfg, dx["E"], dx["Dlog"], dx["h0"], *out)
        assert dart.dart_noalloc_status() == dart.DART_OK
        got = [t.cpu().numpy() for t in out]
        np.testing.assert_array_equal(got[0], ref[0], err_msg=f"node tokens, call {call}")
        np.testing.assert_allclose(got[1], ref[1], atol=tol, rtol=0, err_msg=f"node log q, call {call}")
        np.testing.assert_allclose(got[2], ref[2], atol=tol, rtol=0, err_msg=f"node lse, call {call}")
        np.testing.assert_array_equal(got[3], ref[3], err_msg=f"frontier tokens, call {call}")
        np.testing.assert_allclose(got[4], ref[4], atol=tol, rtol=0, err_msg=f"frontier scores, call {call}")
        np.testing.assert_array_equal(got[5], ref[5], err_msg=f"frontier counts, call {call}")
        if W > k:  # unused frontier ranks of the single parent
            assert np.all(got[3][:, k:] == -1) and np.all(np.isneginf(got[4][:, k:]))


@pytest.mark.parametrize("nseq,V,d,W,k,T", [(3, 20000, 512, 8, 12, 0.7), (40, 5000, 256, 6, 4, 0.0)])
def test_noalloc_matches_the_oracle(dart, nseq, V, d, W, k, T):
    """Depth 1 of Algorithm 1 from the allocation-free entry point against the
    fp64 oracle directly: each root's k best children (tokens exact where the
    oracle's gaps exceed the tolerance), log q~, log-sum-exp, and the
    frontier S_1 with its scores and size."""
    import oracle
    cfg = Config("noalloc-oracle", nseq, V, d, 1, W, k, 20, "bf16", T, 9100 + nseq)
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    tol = tol_of(cfg)
    out = outputs(nseq, W, k)
    dart.dart_expand_root_noalloc(cfg, dx["E"], dx["Dlog"], dx["h0"], *out)
    assert dart.dart_noalloc_status() == dart.DART_OK
    tok, logq, lse, ftok, fsc, fcnt = [t.cpu().numpy() for t in out]
    for s in range(nseq):
        rl, rt = ref["nd_logq"][s, 0, 0, :k], ref["nd_tok"][s, 0, 0, :k]
        assert abs(float(lse[s]) - ref["nd_lse"][s, 0, 0]) <= tol
        fin = np.isfinite(rl)
        assert np.all(np.abs(logq[s][fin] - rl[fin]) <= tol)
        gaps = -np.diff(ref["nd_logq"][s, 0, 0])
        if np.all(gaps[:k] >= tol):
            np.testing.assert_array_equal(tok[s], rt)
        n = int(ref["st_count"][s, 0])
        assert int(fcnt[s]) == n
        rs = ref["st_score"][s, 0, :n]
        assert np.all(np.abs(fsc[s, :n] - rs) <= tol)
        if n < 2 or np.all(-np.diff(rs) >= tol):
            np.testing.assert_array_equal(ftok[s, :n], ref["st_tok"][s, 0, :n])


def test_noalloc_rejects_sizes_beyond_its_array(dart):
    lib = dart.lib()
    big = Config("toolarge", 65, 1000, 128, 2, 2, 2, 4, "bf16", 0.0, 1)
    wide = Config("toowide", 1, 1000, 16384, 2, 2, 2, 4, "bf16", 0.0, 1)
    buf = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    p = C.c_void_p(buf.data_ptr())
    for cfg in (big, wide):
        c = dart.make_config(cfg)
        rc = lib.dart_expand_root_noalloc(C.byref(c), p, p, p, p, p, p, p, p, p, None)
        assert rc == dart.DART_ERR_INVALID
