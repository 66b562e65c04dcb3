"""The GPU-vs-oracle comparison rules of ``parity.py``, exercised on the CPU:
fed the oracle's own tree (in the layout the C ABI returns) they pass, and
fed a tree with a planted discrepancy they fail.  This shows the GPU parity
tests can tell a wrong tree from a right one."""
import numpy as np
import pytest

import oracle
from parity import check_structure, compare_with_oracle, tol_of, validate_frontier_teacher_forced
from workloads import Config, make_inputs

CFG = Config("checker", 2, 600, 64, 4, 6, 4, 14, "bf16", 0.0, 91)


@pytest.fixture(scope="module")
def case():
    x = make_inputs(CFG)
    ref = oracle.build_tree(CFG, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    tol = tol_of(CFG)
    # every rank gap of this case is far above the tolerance (exact comparison applies)
    assert np.all(ref["prune_gap"] > 10 * tol)
    return x, ref, tol


def as_gpu(ref):
    """The oracle's supertree and emitted tree in the dtypes the C ABI returns."""
    gst = dict(st_tok=ref["st_tok"].copy(), st_parent=ref["st_parent"].copy(),
               st_score=ref["st_score"].astype(np.float32), st_count=ref["st_count"].copy())
    g = {k: ref[k].copy() for k in ("tokens", "parents", "depths", "pos_ids", "n_nodes")}
    g["scores"] = ref["scores"].astype(np.float32)
    g["mask"] = ref["mask"].view(np.int64).copy()
    return gst, g


def test_the_oracle_tree_passes(case):
    x, ref, tol = case
    gst, g = as_gpu(ref)
    rep = compare_with_oracle(CFG, ref, gst, g, tol)
    assert rep["bit_identical"] and rep["arrays_exact"] and not rep["near_tie"]
    for s in range(CFG.nseq):
        for dep in (1, 2, CFG.L):
            validate_frontier_teacher_forced(CFG, x, gst, s, dep, tol / CFG.L)


def test_scores_within_the_tolerance_pass_and_beyond_it_fail(case):
    _, ref, tol = case
    gst, g = as_gpu(ref)
    gst["st_score"][0, 2, 1] += 0.5 * tol
    compare_with_oracle(CFG, ref, gst, g, tol)
    gst["st_score"][0, 2, 1] += 2.0 * tol
    with pytest.raises(AssertionError):
        compare_with_oracle(CFG, ref, gst, g, tol)


def test_a_wrong_frontier_token_fails(case):
    _, ref, tol = case
    gst, g = as_gpu(ref)
    t = gst["st_tok"][1, 1, 2]
    gst["st_tok"][1, 1, 2] = (t + 1) % CFG.V
    with pytest.raises(AssertionError):
        compare_with_oracle(CFG, ref, gst, g, tol)


def test_swapped_frontier_ranks_fail(case):
    _, ref, tol = case
    gst, g = as_gpu(ref)
    for key in ("st_tok", "st_parent", "st_score"):
        gst[key][0, 0, [0, 1]] = gst[key][0, 0, [1, 0]]
    with pytest.raises(AssertionError):
        compare_with_oracle(CFG, ref, gst, g, tol)


@pytest.mark.parametrize("plant", ["token", "parent", "mask_bit", "pos_id", "padding", "n_nodes"])
def test_a_wrong_emitted_tree_fails(case, plant):
    _, ref, tol = case
    gst, g = as_gpu(ref)
    n = int(g["n_nodes"][0])
    i = int(np.nonzero(g["parents"][0, :n] >= 0)[0][-1])  # a node below depth 1
    if plant == "token":
        g["tokens"][0, i] = (g["tokens"][0, i] + 1) % CFG.V
    elif plant == "parent":
        g["parents"][0, i] = -1
    elif plant == "mask_bit":
        g["mask"][0, i, 0] &= ~np.int64(1 << int(g["parents"][0, i]))
    elif plant == "pos_id":
        g["pos_ids"][0, i] += 1
    elif plant == "padding":
        g["tokens"][0, CFG.B - 1] = 0 if n < CFG.B else g["tokens"][0, CFG.B - 1]
        g["n_nodes"][0] = n - 1
    elif plant == "n_nodes":
        g["n_nodes"][1] -= 1
    with pytest.raises(AssertionError):
        compare_with_oracle(CFG, ref, gst, g, tol)


def test_structure_check_rejects_an_orphan_and_a_rising_score(case):
    _, ref, _ = case
    _, g = as_gpu(ref)
    check_structure(CFG, g)
    n = int(g["n_nodes"][0])
    i = int(np.nonzero(g["parents"][0, :n] >= 0)[0][-1])
    bad = {k: v.copy() for k, v in g.items()}
    bad["scores"][0, i] = bad["scores"][0, int(bad["parents"][0, i])] + 0.1   # child above its parent
    with pytest.raises(AssertionError):
        check_structure(CFG, bad)
    bad = {k: v.copy() for k, v in g.items()}
    bad["parents"][0, i] = i   # a node that is its own parent
    with pytest.raises(AssertionError):
        check_structure(CFG, bad)


def test_teacher_forced_check_rejects_a_child_outside_the_top_k(case):
    x, ref, tol = case
    gst, _ = as_gpu(ref)
    # replace a kept depth-2 child by its parent's (k+2)-th best child, with the oracle's score
    p = int(gst["st_parent"][0, 1, 0])
    from oracle import node_paths
    path = node_paths(ref["st_tok"], ref["st_parent"], ref["st_count"], 0, CFG.W)[p]
    tok, lq, _, _ = oracle.node_children(CFG, x["Wi"], x["Wo"], x["E"], x["Dlog"][0], x["h0"][0],
                                         np.array(path, np.int32), CFG.k + 2)
    gst["st_tok"][0, 1, 0] = tok[CFG.k + 1]
    gst["st_score"][0, 1, 0] = ref["st_score"][0, 0, p] + lq[CFG.k + 1] + CFG.beta
    with pytest.raises(AssertionError):
        validate_frontier_teacher_forced(CFG, x, gst, 0, 2, tol / CFG.L)
