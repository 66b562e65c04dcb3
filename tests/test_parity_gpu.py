"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle.

Every case, the full-size workloads included (Qwen3-8B and Qwen3-4B shapes,
batched serving, all sixteen points of the width / budget sweep, and the
candidate-restricted K = 64 shapes), is compared with a full oracle run:
exact topology where the oracle's rank gaps exceed the tolerance, path scores
within the tolerance, every depth after a near tie checked teacher-forced on
the GPU's own parents, and the pruned tree equal to the oracle's pruning of
the GPU's supertree.
"""
import numpy as np
import pytest
import torch

import oracle
from parity import compare_with_oracle, gpu_supertree, to_device, tol_of, tree_to_numpy
from workloads import BATCHED, NAMED, Q4B, Q8B, TOY, Config, make_inputs, sweep_configs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dart():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13524_gb300 import dart as d
    d.lib()
    return d


def C(name, nseq, V, d, L, W, k, B, wdtype="bf16", T=0.0, seed=1, **kw):
    return Config(name, nseq, V, d, L, W, k, B, wdtype, T, seed, **kw)


SMALL = [
    C("f32-small", 1, 1000, 128, 4, 4, 4, 10, "f32", 0.0, 11),
    C("f32-groups", 3, 1500, 64, 3, 12, 4, 20, "f32", 0.7, 12),
    C("bf16-small", 2, 1000, 128, 3, 4, 4, 7, "bf16", 1.0, 13),
    C("bf16-mid", 1, 5003, 512, 5, 8, 8, 24, "bf16", 0.0, 14),
    C("bf16-multitile", 1, 50000, 256, 4, 6, 7, 15, "bf16", 0.7, 15),
    C("bf16-groups", 4, 3000, 256, 3, 24, 24, 50, "bf16", 1.0, 16),
    C("bf16-N256", 8, 2000, 128, 3, 32, 8, 40, "bf16", 0.0, 17),
    C("bf16-k64", 1, 4000, 128, 3, 64, 64, 100, "bf16", 0.0, 18),
    C("bf16-d64", 1, 777, 64, 2, 3, 5, 4, "bf16", 0.0, 19),
    C("bf16-L1", 2, 900, 128, 1, 5, 9, 3, "bf16", 0.0, 20),
    C("bf16-chain", 1, 600, 128, 6, 1, 1, 6, "bf16", 0.0, 21),
    C("bf16-B1", 1, 600, 128, 4, 4, 4, 1, "bf16", 0.0, 22),
    C("bf16-Vk", 1, 8, 64, 4, 8, 8, 30, "bf16", 0.0, 23),
    C("bf16-beta0", 1, 1200, 128, 4, 6, 3, 11, "bf16", 0.0, 24, beta=0.0),
    C("bf16-kltW", 2, 1200, 128, 4, 9, 2, 25, "bf16", 0.0, 25, pos_offset=37),
    C("bf16-manytiles", 1, 320000, 128, 3, 8, 16, 20, "bf16", 1.0, 26),
    C("bf16-k64-many", 1, 200000, 64, 2, 64, 64, 80, "bf16", 0.0, 27),
    C("f32-manytiles", 2, 150000, 64, 3, 16, 16, 30, "f32", 0.0, 28),
    C("f32-d192", 2, 3000, 192, 4, 6, 4, 15, "f32", 0.5, 29),
    C("f32-d1024", 1, 2000, 1024, 3, 8, 8, 20, "f32", 0.0, 30),
    TOY,
]

# candidate-restricted scoring (Algorithm 1 with K = cand_k)
RESTRICTED = [
    C("cand-f32", 1, 3000, 128, 4, 4, 4, 10, "f32", 0.0, 51, cand_k=64),
    C("cand-bf16", 2, 20000, 256, 5, 8, 8, 24, "bf16", 1.0, 52, cand_k=64),
    C("cand-bf16-N256", 8, 5000, 128, 3, 32, 32, 60, "bf16", 0.0, 53, cand_k=64),
    C("cand-odd-K", 1, 4000, 192, 4, 6, 5, 20, "bf16", 0.7, 54, cand_k=37),
    C("cand-K1024", 1, 9000, 128, 3, 16, 16, 40, "bf16", 0.0, 55, cand_k=1024),
    C("cand-K=k", 2, 2500, 64, 4, 8, 8, 30, "bf16", 0.0, 56, cand_k=8),
    C("cand-K=V", 1, 300, 64, 3, 5, 5, 12, "f32", 0.0, 57, cand_k=300),
]


def run_depthwise(dart, cfg, dx):
    """Expands depth by depth, collecting node lists / frontiers / states."""
    h = dart.dart_init_head(cfg, dart.DART_BF16 if cfg.wdtype == "bf16" else dart.DART_F32,
                            dx["Wi"], dx["Wo"], dx["E"])
    per = []
    try:
        for dep in range(1, cfg.L + 1):
            dart.dart_expand_depth(h, dep, dx["Dlog"], dx["h0"])
            tok, lq, lse = dart.dart_get_node_topk(h, cfg)
            st = dart.dart_get_states(h, cfg)
            per.append(dict(tok=tok.cpu().numpy(), logq=lq.cpu().numpy(), lse=lse.cpu().numpy(),
                            states=st.cpu().numpy()))
        out_t, out = dart.alloc_tree_out(cfg)
        dart.dart_prune_and_emit(h, out)
        assert dart.dart_status_sync(h) == 0
        gst = gpu_supertree(dart, h, cfg)
        g = tree_to_numpy(out_t)
    finally:
        dart.dart_destroy(h)
    return per, gst, g


@pytest.mark.parametrize("cfg", SMALL + RESTRICTED, ids=[c.name for c in SMALL + RESTRICTED])
def test_depthwise_parity(dart, cfg):
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    per, gst, g = run_depthwise(dart, cfg, dx)
    tol = tol_of(cfg)
    rep = compare_with_oracle(cfg, ref, gst, g, tol, x=x)
    print(cfg.name, rep)
    # node-level lists and states while the frontiers agree exactly
    caps = cfg.caps()
    for dep in range(1, cfg.L + 1):
        if any(t[0] == s and (t[1] == "prune" or t[1] <= dep - 1) for s in range(cfg.nseq) for t in rep["near_tie"]):
            break
        P = caps[dep - 1]
        d = per[dep - 1]
        for s in range(cfg.nseq):
            npar = 1 if dep == 1 else int(ref["st_count"][s, dep - 2])
            for p in range(npar):
                row = s * P + p
                rl = ref["nd_logq"][s, dep - 1, p, :cfg.k]
                rt = ref["nd_tok"][s, dep - 1, p, :cfg.k]
                assert abs(float(d["lse"][row]) - ref["nd_lse"][s, dep - 1, p]) <= tol
                fin = np.isfinite(rl)
                assert np.all(np.abs(d["logq"][row][fin] - rl[fin]) <= tol)
                gaps = -np.diff(ref["nd_logq"][s, dep - 1, p])
                if np.all(gaps[:cfg.k] >= tol):
                    np.testing.assert_array_equal(d["tok"][row], rt)
        if dep < cfg.L:
            # states of the retained children vs teacher-forced oracle states
            stol = 5e-4 if cfg.wdtype == "bf16" else 2e-5
            for s in range(min(cfg.nseq, 2)):
                paths = oracle.node_paths(ref["st_tok"], ref["st_parent"], ref["st_count"], s, cfg.W)
                for r in range(min(int(ref["st_count"][s, dep - 1]), 4)):
                    hs = oracle.path_state(cfg, x["Wi"], x["Wo"], x["E"], x["h0"][s],
                                           np.array(paths[(dep - 1) * cfg.W + r], np.int32))
                    got = d["states"][s * caps[dep] + r]
                    assert np.max(np.abs(got - hs)) <= stol, (dep, s, r, np.max(np.abs(got - hs)))


GRAPH = SMALL[:6] + RESTRICTED[:3]


@pytest.mark.parametrize("cfg", GRAPH, ids=[c.name for c in GRAPH])
def test_build_tree_graph_matches_depthwise(dart, cfg):
    """dart_build_tree (one cached CUDA graph) equals the depth-by-depth
    calls, is deterministic across repeated launches, and the host-buffer
    variant returns the same tree.  (fp32: the graph of per-step launches;
    the fused round is compared with the oracle below.)"""
    cfg = cfg.replace(fused_round=2)
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    _, gst_ref, g_ref = run_depthwise(dart, cfg, dx)
    eng = dart.Dart(cfg, dx["Wi"], dx["Wo"], dx["E"])
    try:
        for it in range(3):
            out = eng.build_tree(dx["Dlog"], dx["h0"])
            torch.cuda.synchronize()
            g = tree_to_numpy(out)
            for k in g:
                np.testing.assert_array_equal(g[k], g_ref[k], err_msg=f"{k} (launch {it})")
        assert dart.dart_status_sync(eng.h) == 0
        ht, hout = dart.alloc_tree_out(cfg, pin=True)
        Dh = dx["Dlog"].cpu().pin_memory()
        h0h = dx["h0"].cpu().pin_memory()
        dart.dart_build_tree_host(eng.h, Dh, h0h, hout)
        for k in g_ref:
            np.testing.assert_array_equal(ht[k].numpy(), g_ref[k], err_msg=k)
    finally:
        eng.close()


# fp32 problems small enough for the fused round: one cluster per sequence
# where a block's share of E is small, else one cooperative grid (the V = 64K
# case; at most 32 nodes per depth)
FUSED = [c for c in SMALL if c.wdtype == "f32" and c.V <= 65536] + [
    C("f32-fused-nseq4", 4, 6000, 256, 5, 8, 8, 30, "f32", 0.7, 41),
    C("f32-fused-V64k", 1, 65536, 128, 3, 16, 16, 25, "f32", 0.0, 42),
    C("f32-fused-k32", 2, 4000, 64, 4, 16, 32, 40, "f32", 0.0, 43),
    C("f32-fused-L8W32", 1, 3000, 64, 8, 32, 8, 120, "f32", 0.3, 44),
    C("f32-fused-chain", 1, 2000, 128, 6, 1, 1, 6, "f32", 0.0, 45),
    C("f32-fused-B1", 2, 1500, 128, 4, 4, 4, 1, "f32", 0.0, 46, pos_offset=9),
    C("f32-fused-Vk", 1, 8, 64, 4, 8, 8, 30, "f32", 0.0, 47),
]


@pytest.mark.parametrize("cfg", FUSED, ids=[c.name for c in FUSED])
def test_fused_round_parity(dart, cfg):
    """The whole round as one kernel launch: the oracle's tree
    (compare_with_oracle), bit-identical on repeated launches and through the
    host-buffer entry point."""
    cfg = cfg.replace(fused_round=1)
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    eng = dart.Dart(cfg, dx["Wi"], dx["Wo"], dx["E"])
    try:
        assert dart.dart_launches_per_round(eng.h) == 1
        g = tree_to_numpy(eng.build_tree(dx["Dlog"], dx["h0"]))
        assert dart.dart_status_sync(eng.h) == 0
        gst = gpu_supertree(dart, eng.h, cfg)
        for it in range(2):
            again = tree_to_numpy(eng.build_tree(dx["Dlog"], dx["h0"]))
            for k in g:
                np.testing.assert_array_equal(again[k], g[k], err_msg=f"{k} (launch {it + 2})")
        ht, hout = dart.alloc_tree_out(cfg, pin=True)
        dart.dart_build_tree_host(eng.h, dx["Dlog"].cpu().pin_memory(), dx["h0"].cpu().pin_memory(), hout)
        assert dart.dart_status_sync(eng.h) == 0
        for k in g:
            np.testing.assert_array_equal(ht[k].numpy(), g[k], err_msg=k)
    finally:
        eng.close()
    compare_with_oracle(cfg, ref, gst, g, tol_of(cfg), x=x)


def test_fused_round_neg_inf_and_states(dart):
    """-inf drafter logits through the fused round, and the state hook after
    it: depth L's states equal the depth-by-depth path's within fp32
    rounding."""
    cfg = C("f32-fused-neginf", 2, 700, 128, 4, 6, 4, 40, "f32", 0.0, 48, fused_round=1)
    x = make_inputs(cfg)
    x["Dlog"][0, 1, 3:] = -np.inf      # depth 2 of seq 0: only tokens 0..2 possible
    x["Dlog"][1, 0, :] = -np.inf       # depth 1 of seq 1: no child at all
    x["Dlog"][1, 0, 5] = 0.0           #   ... except token 5
    dx = to_device(cfg, x)
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    per, _, _ = run_depthwise(dart, cfg, dx)
    eng = dart.Dart(cfg, dx["Wi"], dx["Wo"], dx["E"])
    try:
        g = tree_to_numpy(eng.build_tree(dx["Dlog"], dx["h0"]))
        assert dart.dart_status_sync(eng.h) == 0
        gst = gpu_supertree(dart, eng.h, cfg)
        st = dart.dart_get_states(eng.h, cfg).cpu().numpy()
    finally:
        eng.close()
    compare_with_oracle(cfg, ref, gst, g, tol_of(cfg), x=x)
    assert int(gst["st_count"][1, 0]) == 1 and int(gst["st_tok"][1, 0, 0]) == 5
    np.testing.assert_allclose(st, per[-1]["states"], rtol=0, atol=1e-4)


def test_fused_round_eligibility(dart):
    """fused_round = ON where the problem does not fit is refused at
    dart_init_head; AUTO then takes the per-step launches."""
    x = None
    for cfg in (C("f32-wide", 1, 1500, 64, 3, 40, 4, 20, "f32", 0.7, 12),          # W > 32
                C("f32-bigV", 1, 70000, 64, 2, 4, 4, 8, "f32", 0.0, 13),           # V > 65536, E slices > 512 KB
                C("bf16-small", 1, 1000, 128, 3, 4, 4, 8, "bf16", 0.0, 14)):        # bf16 weights
        x = make_inputs(cfg)
        dx = to_device(cfg, x)
        wd = dart.DART_BF16 if cfg.wdtype == "bf16" else dart.DART_F32
        with pytest.raises(dart.DartError) as e:
            dart.dart_init_head(cfg.replace(fused_round=1), wd, dx["Wi"], dx["Wo"], dx["E"])
        assert e.value.code == dart.DART_ERR_UNSUPPORTED
        h = dart.dart_init_head(cfg, wd, dx["Wi"], dx["Wo"], dx["E"])
        try:
            assert dart.dart_launches_per_round(h) > 1
        finally:
            dart.dart_destroy(h)


VARIANT_CFGS = [SMALL[2], SMALL[5], SMALL[6], RESTRICTED[1]]


@pytest.mark.parametrize("switch", [dict(head_split=2), dict(head_split_stream=2), dict(lmhead_ctas_per_sm=1),
                                    dict(lmhead_ctas_per_sm=2), dict(weights_tiled=2),
                                    dict(weights_tiled=2, head_split=2)],
                         ids=["unsplit", "same-stream", "lmhead-1cta", "lmhead-2cta", "row-major", "row-major-unsplit"])
@pytest.mark.parametrize("cfg", VARIANT_CFGS, ids=[c.name for c in VARIANT_CFGS])
def test_head_update_variants(dart, cfg, switch):
    """The variants behind the tuning fields of dart_config: the unsplit first
    head layer (gather of [h_p ; E[t_c]] and the full W_i GEMM, no table), the
    split layer's GEMM on the main stream, one or two LM-head CTAs per SM, and
    the caller's row-major weights streamed directly instead of tiled copies.
    Each matches the oracle, and the graph launch equals the depth-by-depth
    calls."""
    cfg = cfg.replace(**switch)
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    _, gst, g_ref = run_depthwise(dart, cfg, dx)
    compare_with_oracle(cfg, ref, gst, g_ref, tol_of(cfg), x=x)
    eng = dart.Dart(cfg, dx["Wi"], dx["Wo"], dx["E"])
    try:
        g = tree_to_numpy(eng.build_tree(dx["Dlog"], dx["h0"]))
        assert dart.dart_status_sync(eng.h) == 0
    finally:
        eng.close()
    for k in g_ref:
        np.testing.assert_array_equal(g[k], g_ref[k], err_msg=k)


def test_neg_inf_drafter_logits(dart):
    cfg = C("neginf", 2, 700, 128, 4, 6, 4, 40, "bf16", 0.0, 31)
    x = make_inputs(cfg)
    x["Dlog"][0, 1, 3:] = -np.inf      # depth 2 of seq 0: only tokens 0..2 possible
    x["Dlog"][1, 0, :] = -np.inf       # depth 1 of seq 1: no child at all
    x["Dlog"][1, 0, 5] = 0.0           #   ... except token 5
    dx = to_device(cfg, x)
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    _, gst, g = run_depthwise(dart, cfg, dx)
    compare_with_oracle(cfg, ref, gst, g, tol_of(cfg), x=x)
    assert int(gst["st_count"][1, 0]) == 1


def test_restricted_candidates_and_neg_inf(dart):
    """Restricted scoring with -inf drafter logits: C_d still holds K tokens
    (the -inf ones by token id), their children have probability zero and are
    never retained."""
    cfg = C("cand-neginf", 2, 700, 128, 4, 6, 4, 40, "bf16", 0.0, 58, cand_k=16)
    x = make_inputs(cfg)
    x["Dlog"][0, 1, 3:] = -np.inf      # depth 2 of seq 0: only tokens 0..2 possible
    x["Dlog"][1, 0, :] = -np.inf       # depth 1 of seq 1: no child at all
    x["Dlog"][1, 0, 5] = 0.0           #   ... except token 5
    dx = to_device(cfg, x)
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    _, gst, g = run_depthwise(dart, cfg, dx)
    compare_with_oracle(cfg, ref, gst, g, tol_of(cfg), x=x)
    assert int(gst["st_count"][1, 0]) == 1
    assert int(gst["st_tok"][1, 0, 0]) == 5


def test_call_order_and_argument_errors(dart):
    cfg = C("err", 1, 500, 64, 3, 2, 2, 4, "bf16", 0.0, 41)
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    h = dart.dart_init_head(cfg, dart.DART_BF16, dx["Wi"], dx["Wo"], dx["E"])
    try:
        out_t, out = dart.alloc_tree_out(cfg)
        with pytest.raises(dart.DartError) as e:
            dart.dart_expand_depth(h, 2, dx["Dlog"], dx["h0"])
        assert e.value.code == dart.DART_ERR_STATE
        with pytest.raises(dart.DartError) as e:
            dart.dart_prune_and_emit(h, out)
        assert e.value.code == dart.DART_ERR_STATE
        dart.dart_expand_depth(h, 1, dx["Dlog"], dx["h0"])
        with pytest.raises(dart.DartError) as e:
            dart.dart_expand_depth(h, 3, dx["Dlog"], dx["h0"])
        assert e.value.code == dart.DART_ERR_STATE
        with pytest.raises(dart.DartError) as e:
            dart.dart_expand_depth(h, 1, dx["Dlog"], None)   # anchor needed at depth 1
        assert e.value.code == dart.DART_ERR_INVALID
        dart.dart_expand_depth(h, 1, dx["Dlog"], dx["h0"])
        dart.dart_expand_depth(h, 2, dx["Dlog"], None)
        dart.dart_expand_depth(h, 3, dx["Dlog"], None)
        dart.dart_prune_and_emit(h, out)
        assert dart.dart_status_sync(h) == 0
    finally:
        dart.dart_destroy(h)


# ----------------------------------------------------------------- full size

_INPUTS = {}


def full_inputs(cfg):
    """Inputs of a full-size workload; the sixteen sweep points share theirs
    (same seed and shapes: W, k and B do not enter the generators)."""
    key = (cfg.seed, cfg.nseq, cfg.V, cfg.d, cfg.L, cfg.wdtype)
    if key not in _INPUTS:
        _INPUTS.clear()
        _INPUTS[key] = make_inputs(cfg)
    return _INPUTS[key]


def gpu_round(dart, cfg, x, dx):
    """One round in the launch configuration the benchmark times
    (dart_build_tree: the cached CUDA graph), with its supertree."""
    eng = dart.Dart(cfg, dx["Wi"], dx["Wo"], dx["E"])
    try:
        out = eng.build_tree(dx["Dlog"], dx["h0"])
        assert dart.dart_status_sync(eng.h) == 0
        g = tree_to_numpy(out)
        gst = gpu_supertree(dart, eng.h, cfg)
    finally:
        eng.close()
    return gst, g


def report(cfg, rep):
    print(f"{cfg.name}: bit_identical={rep['bit_identical']} arrays_exact={rep['arrays_exact']} "
          f"near_ties={rep['near_tie']} order_ties={rep['order_ties']} "
          f"depths_teacher_forced={rep['depths_teacher_forced']} max_score_err={rep['max_score_err']:.3g}")


FULL = [Q8B, Q4B, BATCHED, NAMED["qwen3-8b-k64"], NAMED["qwen3-4b-k64"], NAMED["batched-k64"]]


@pytest.mark.parametrize("cfg", FULL, ids=[c.name for c in FULL])
def test_full_size_oracle_parity(dart, cfg):
    """Full-size workloads, full oracle run, complete comparison."""
    x = full_inputs(cfg)
    dx = to_device(cfg, x)
    gst, g = gpu_round(dart, cfg, x, dx)
    del dx
    caps = cfg.caps()
    for s in range(cfg.nseq):
        assert list(gst["st_count"][s]) == caps[1:]
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    rep = compare_with_oracle(cfg, ref, gst, g, tol_of(cfg), x=x)
    report(cfg, rep)


@pytest.mark.parametrize("W", [8, 16, 32, 64])
def test_sweep_oracle_parity(dart, W):
    """The width / budget sweep at the Qwen3-4B shape: one oracle supertree per
    W (it does not depend on B), pruned and emitted by the oracle for every
    B in {32, 128, 512, 1024}; each GPU round (its own handle per point) is
    compared completely."""
    pts = [c for c in sweep_configs() if c.W == W]
    x = full_inputs(pts[0])
    dx = to_device(pts[0], x)
    big = max(pts, key=lambda c: c.B)
    sup = oracle.build_tree(big, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    for cfg in pts:
        gst, g = gpu_round(dart, cfg, x, dx)
        ref = {k: sup[k] for k in ("st_tok", "st_parent", "st_score", "st_count", "nd_lse", "nd_tok",
                                   "nd_logq", "fr_score")}
        pe = oracle.prune_emit(cfg, sup["st_tok"], sup["st_parent"], sup["st_score"], sup["st_count"])
        assert pe["rc"] == 0
        ref.update({k: pe[k] for k in ("tokens", "parents", "depths", "pos_ids", "scores", "n_nodes",
                                       "mask", "prune_gap")})
        rep = compare_with_oracle(cfg, ref, gst, g, tol_of(cfg), x=x)
        report(cfg, rep)


def test_handles_with_different_plans_coexist(dart):
    """Kernel attributes are process-wide: a handle created later with a
    smaller plan (here one LM-head CTA per SM, half as many partial lists to
    merge) must not break an earlier handle whose merge needs more shared
    memory.  Both give the oracle's tree (their vocabulary splits differ, so
    their fp32 sums may differ in the last bits)."""
    big = C("coexist", 1, 20000, 2560, 3, 32, 32, 40, "bf16", 0.0, 81, lmhead_ctas_per_sm=2)
    small = big.replace(lmhead_ctas_per_sm=1)
    x = make_inputs(big)
    dx = to_device(big, x)
    a = dart.Dart(big, dx["Wi"], dx["Wo"], dx["E"])
    b = dart.Dart(small, dx["Wi"], dx["Wo"], dx["E"])
    try:
        ga = tree_to_numpy(a.build_tree(dx["Dlog"], dx["h0"]))
        gb = tree_to_numpy(b.build_tree(dx["Dlog"], dx["h0"]))
        assert dart.dart_status_sync(a.h) == 0 and dart.dart_status_sync(b.h) == 0
        gst = gpu_supertree(dart, a.h, big)
        gstb = gpu_supertree(dart, b.h, small)
    finally:
        a.close()
        b.close()
    ref = oracle.build_tree(big, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    compare_with_oracle(big, ref, gst, ga, tol_of(big), x=x)
    compare_with_oracle(small, ref, gstb, gb, tol_of(big), x=x)


# the starting bound of the LM-head's top-k filters (topk_bound): forced on
# at every depth (1 node at depth 1 included); odd node counts per sequence
# (node blocks of fewer than 8), a vocabulary whose last seed chunks are
# empty, temperature, k = 64 with few nodes (128 seed rows), 64-node groups (32
# candidate slots, 4 accumulators) and 128-node groups
BOUND = [
    C("bound-k32-N64", 2, 6000, 256, 4, 32, 32, 60, "bf16", 0.0, 61),
    C("bound-odd-P", 3, 3001, 192, 3, 13, 40, 30, "bf16", 0.7, 62),
    C("bound-k64-W8", 1, 9000, 128, 3, 8, 64, 40, "bf16", 0.0, 63),
    C("bound-N128", 4, 4000, 128, 3, 32, 32, 70, "bf16", 1.0, 64),
    C("bound-k64-d512", 1, 30000, 512, 3, 64, 64, 90, "bf16", 0.0, 65),
]


@pytest.mark.parametrize("cfg", BOUND, ids=[c.name for c in BOUND])
def test_topk_bound_matches_the_oracle_and_changes_nothing(dart, cfg):
    """With the seed pass on, the tree equals the oracle's, and every emitted
    array (scores included) is bit-identical to the run without it: the bound
    only keeps logits below a node's k-th best out of the top-k merges."""
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    on = cfg.replace(topk_bound=1)
    _, gst, g = run_depthwise(dart, on, dx)
    print(cfg.name, compare_with_oracle(on, ref, gst, g, tol_of(cfg), x=x))
    _, gst_off, g_off = run_depthwise(dart, cfg.replace(topk_bound=2), dx)
    for k in g:
        np.testing.assert_array_equal(g[k], g_off[k], err_msg=k)
    for k in gst:
        np.testing.assert_array_equal(gst[k], gst_off[k], err_msg=k)
    eng = dart.Dart(on, dx["Wi"], dx["Wo"], dx["E"])
    try:
        out = eng.build_tree(dx["Dlog"], dx["h0"])
        torch.cuda.synchronize()
        assert dart.dart_status_sync(eng.h) == 0
        gg = tree_to_numpy(out)
        for k in g:
            np.testing.assert_array_equal(gg[k], g[k], err_msg=f"graph {k}")
    finally:
        eng.close()


def test_topk_bound_with_neg_inf_drafter_logits(dart):
    """Seed chunks whose drafter logits are all -inf give no seed score; a
    sequence with a single finite token at a depth still gets its one child."""
    cfg = C("bound-neginf", 2, 2000, 128, 4, 40, 40, 60, "bf16", 0.0, 66, topk_bound=1)
    x = make_inputs(cfg)
    x["Dlog"][0, 1, 300:] = -np.inf     # depth 2 of seq 0: tokens 0..299 only (most chunks empty)
    x["Dlog"][1, 0, :] = -np.inf        # depth 1 of seq 1: token 7 only
    x["Dlog"][1, 0, 7] = 0.0
    x["Dlog"][1, 2, ::2] = -np.inf      # depth 3 of seq 1: every other token
    dx = to_device(cfg, x)
    ref = oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    _, gst, g = run_depthwise(dart, cfg, dx)
    compare_with_oracle(cfg, ref, gst, g, tol_of(cfg), x=x)
    assert int(gst["st_count"][1, 0]) == 1
    _, gst_off, g_off = run_depthwise(dart, cfg.replace(topk_bound=2), dx)
    for k in g:
        np.testing.assert_array_equal(g[k], g_off[k], err_msg=k)


LAUNCH_CFGS = [SMALL[0], SMALL[0].replace(fused_round=2), SMALL[1], SMALL[2], SMALL[5], SMALL[19],
               RESTRICTED[1], RESTRICTED[0], BOUND[0].replace(topk_bound=1), BOUND[1]]


@pytest.mark.parametrize("cfg", LAUNCH_CFGS, ids=[f"{c.name}-{c.fused_round}-{c.topk_bound}" for c in LAUNCH_CFGS])
def test_launches_per_round_matches_the_profiled_round(dart, cfg):
    """dart_launches_per_round (the bench's kernel-launch count) equals the
    launches one profiled round brackets, kind by kind summed (every launch
    of a round is bracketed while profiling is on)."""
    x = make_inputs(cfg)
    dx = to_device(cfg, x)
    eng = dart.Dart(cfg, dx["Wi"], dx["Wo"], dx["E"])
    try:
        eng.build_tree(dx["Dlog"], dx["h0"])
        dart.dart_set_profiling(eng.h, True)
        dart.dart_profile_read_kinds(eng.h)
        eng.build_tree(dx["Dlog"], dx["h0"])
        kinds = dart.dart_profile_read_kinds(eng.h)
        dart.dart_set_profiling(eng.h, False)
        assert dart.dart_status_sync(eng.h) == 0
        counted = sum(n for _, n in kinds.values())
        assert counted == dart.dart_launches_per_round(eng.h), kinds
    finally:
        eng.close()
