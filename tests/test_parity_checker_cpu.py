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


def emitted_row(ref, s, node_id):
    """Row of the emitted tree holding supertree node `node_id` (None if pruned)."""
    path = oracle.node_paths(ref["st_tok"], ref["st_parent"], ref["st_count"], s, CFG.W)[node_id]
    for i in range(int(ref["n_nodes"][s])):
        p, j = [], i
        while j >= 0:
            p.append(int(ref["tokens"][s, j]))
            j = int(ref["parents"][s, j])
        if tuple(reversed(p)) == path:
            return i
    return None


def test_scores_within_the_tolerance_pass_and_beyond_it_fail(case):
    _, ref, tol = case
    gst, g = as_gpu(ref)
    i = emitted_row(ref, 0, 2 * CFG.W + 1)
    assert i is not None
    for step in (0.5 * tol, 2.0 * tol):
        gst["st_score"][0, 2, 1] += step
        g["scores"][0, i] = gst["st_score"][0, 2, 1]
        if step < tol:
            compare_with_oracle(CFG, ref, gst, g, tol)
    with pytest.raises(AssertionError):
        compare_with_oracle(CFG, ref, gst, g, tol)


def test_emitted_scores_must_be_the_supertree_scores(case):
    _, ref, tol = case
    gst, g = as_gpu(ref)
    g["scores"][0, 3] += 0.25 * tol      # within tolerance of the oracle, but not the GPU's own score
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


# ----------------------------------------------- after a near tie at a frontier cut

TIE = Config("checker-tie", 2, 600, 64, 6, 6, 4, 20, "bf16", 0.0, 194)
TIE_SEQ, TIE_DEPTH = 1, 2   # the oracle's W-th / (W+1)-th gap there is 9.2e-4, below the 2e-3 tolerance


def consistent_gpu_tree(cfg, gst):
    """An emitted tree consistent with a supertree (its own top-B pruning), so
    that a planted supertree mistake can only be caught by the frontier checks."""
    pe = oracle.prune_emit(cfg, gst["st_tok"], gst["st_parent"], gst["st_score"].astype(np.float64),
                           gst["st_count"])
    g = {k: pe[k].copy() for k in ("tokens", "parents", "depths", "pos_ids", "n_nodes")}
    g["scores"] = pe["scores"].astype(np.float32)
    g["mask"] = pe["mask"].view(np.int64).copy()
    return g


@pytest.fixture(scope="module")
def tie_case():
    x = make_inputs(TIE)
    ref = oracle.build_tree(TIE, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    fr = ref["fr_score"][TIE_SEQ, TIE_DEPTH - 1]
    gap = fr[TIE.W - 1] - fr[TIE.W]
    assert 0 < gap < tol_of(TIE) / 2
    # a tree that legitimately takes the other side of the tie: the oracle run on
    # inputs whose (W+1)-th candidate's drafter logit is raised by 2x the gap
    # (less than the tolerance), so every score moves by less than the tolerance
    xs = {k: v.copy() for k, v in x.items()}
    # the (W+1)-th candidate of depth 2: recompute the candidates of the depth-1 parents
    from parity import TeacherForced
    tf = TeacherForced(TIE, x, TIE_SEQ)
    paths = oracle.node_paths(ref["st_tok"], ref["st_parent"], ref["st_count"], TIE_SEQ, TIE.W)
    cands = []
    for p in range(int(ref["st_count"][TIE_SEQ, 0])):
        tok, lq = tf.children(paths[p], TIE.k)
        for j in range(TIE.k):
            cands.append((-(ref["st_score"][TIE_SEQ, 0, p] + lq[j] + TIE.beta), p, j, int(tok[j])))
    cands.sort()
    p_alt = cands[TIE.W]
    xs["Dlog"][TIE_SEQ, TIE_DEPTH - 1, p_alt[3]] += np.float32(2 * gap)
    alt = oracle.build_tree(TIE, xs["Wi"], xs["Wo"], xs["E"], xs["Dlog"], xs["h0"])
    gst = dict(st_tok=alt["st_tok"].copy(), st_parent=alt["st_parent"].copy(),
               st_score=alt["st_score"].astype(np.float32), st_count=alt["st_count"].copy())
    assert set(oracle.node_paths(gst["st_tok"], gst["st_parent"], gst["st_count"], TIE_SEQ, TIE.W).values()) != \
        set(paths.values())
    return x, ref, gst


def test_a_near_tie_divergence_is_checked_at_every_later_depth(tie_case):
    x, ref, gst = tie_case
    rep = compare_with_oracle(TIE, ref, gst, consistent_gpu_tree(TIE, gst), tol_of(TIE), x=x)
    assert [t[:2] for t in rep["near_tie"]] == [(TIE_SEQ, TIE_DEPTH)]
    assert rep["depths_teacher_forced"] == TIE.L - TIE_DEPTH + 1
    assert rep["max_score_err"] < tol_of(TIE)


def planted(tie_case, dep, how):
    x, ref, gst0 = tie_case
    from parity import TeacherForced
    gst = {k: v.copy() for k, v in gst0.items()}
    W, k = TIE.W, TIE.k
    s = TIE_SEQ
    tf = TeacherForced(TIE, x, s)
    gp = oracle.node_paths(gst["st_tok"], gst["st_parent"], gst["st_count"], s, W)
    r = int(gst["st_count"][s, dep - 1]) - 1          # the last kept child of this depth
    p = int(gst["st_parent"][s, dep - 1, r])
    ps = float(gst["st_score"][s, dep - 2, p])
    tok, lq = tf.children(gp[(dep - 2) * W + p], k + 2)
    if how == "outside_top_k1":                      # the parent's (k+2)-th child, scored by the oracle
        gst["st_tok"][s, dep - 1, r] = tok[k + 1]
        gst["st_score"][s, dep - 1, r] = ps + lq[k + 1] + TIE.beta
    elif how == "kth_cut":                           # the (k+1)-th child without a near tie at the k-th cut
        assert lq[k - 1] - lq[k] > 4 * tol_of(TIE)
        gst["st_tok"][s, dep - 1, r] = tok[k]
        gst["st_score"][s, dep - 1, r] = ps + lq[k] + TIE.beta
    elif how == "score":                             # a path score off by 3x the tolerance
        gst["st_score"][s, dep - 1, r] -= 3 * tol_of(TIE)
    elif how == "not_top_w":                         # a kept child swapped for a lower-ranked candidate
        npar = int(gst["st_count"][s, dep - 2])
        pool = []
        kept = {(int(gst["st_parent"][s, dep - 1, i]), int(gst["st_tok"][s, dep - 1, i]))
                for i in range(int(gst["st_count"][s, dep - 1]))}
        for q in range(npar):
            t2, l2 = tf.children(gp[(dep - 2) * W + q], k)
            for j in range(k):
                if (q, int(t2[j])) not in kept:
                    pool.append((float(gst["st_score"][s, dep - 2, q]) + l2[j] + TIE.beta, q, int(t2[j])))
        pool.sort(reverse=True)
        sc, q, t = pool[-1]                          # the lowest-scored unkept candidate
        assert sc < float(gst["st_score"][s, dep - 1, r]) - 4 * tol_of(TIE)
        gst["st_tok"][s, dep - 1, r] = t
        gst["st_parent"][s, dep - 1, r] = q
        gst["st_score"][s, dep - 1, r] = sc
    elif how == "count":                             # one child fewer than the candidates allow
        gst["st_count"][s, dep - 1] -= 1
        gst["st_tok"][s, dep - 1, r] = -1
        gst["st_score"][s, dep - 1, r] = -np.inf
        if dep < TIE.L:                              # keep later depths from referring to the dropped slot
            gst["st_count"][s, dep:] = 0
    return x, ref, gst


@pytest.mark.parametrize("how", ["outside_top_k1", "kth_cut", "score", "not_top_w", "count"])
@pytest.mark.parametrize("dep", [TIE_DEPTH + 1, TIE.L])
def test_a_wrong_frontier_after_a_near_tie_fails(tie_case, dep, how):
    """Mistakes planted after the divergence, at depths the oracle's own tree
    cannot be compared with (its frontiers differ), are still caught."""
    x, ref, gst = planted(tie_case, dep, how)
    with pytest.raises(AssertionError):
        compare_with_oracle(TIE, ref, gst, consistent_gpu_tree(TIE, gst), tol_of(TIE), x=x)


# ------------------------------------- best-first (pop-order) trees

HEAP = Config("checker-heap", 2, 500, 64, 4, 4, 4, 20, "bf16", 0.5, 93)


@pytest.fixture(scope="module")
def heap_case():
    x = make_inputs(HEAP)
    a = oracle.chain_ddtree(HEAP, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    b = oracle.seq_heap(HEAP, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    return x, a, b


def as_gpu_rows(ref):
    g = {k: ref[k].copy() for k in ("tokens", "parents", "depths", "pos_ids", "n_nodes")}
    g["scores"] = ref["scores"].astype(np.float32)
    g["mask"] = ref["mask"].view(np.int64).copy()
    return g


def scorers(x, a):
    from parity import chain_path_score, corrected_path_score
    return chain_path_score(HEAP, x, a["chain_tok"]), corrected_path_score(HEAP, x)


def test_oracle_pop_order_trees_pass(heap_case):
    from parity import compare_pop_order_tree
    x, a, b = heap_case
    sa, sb = scorers(x, a)
    for ref, sc in ((a, sa), (b, sb)):
        rep = compare_pop_order_tree(HEAP, ref, as_gpu_rows(ref), tol_of(HEAP), sc)
        assert rep["bit_identical"] and not rep["near_tie"]


@pytest.mark.parametrize("which", ["chain", "seq"])
@pytest.mark.parametrize("plant", ["token", "score", "swap", "mask", "padding", "count", "parent"])
def test_a_wrong_pop_order_tree_fails(heap_case, which, plant):
    from parity import compare_pop_order_tree
    x, a, b = heap_case
    ref = a if which == "chain" else b
    sc = scorers(x, a)[0 if which == "chain" else 1]
    g = as_gpu_rows(ref)
    tol = tol_of(HEAP)
    n = int(g["n_nodes"][0])
    i = int(np.nonzero(g["parents"][0, :n] >= 0)[0][-1])   # a node below depth 1
    if plant == "token":
        g["tokens"][0, i] = (g["tokens"][0, i] + 1) % HEAP.V
    elif plant == "score":
        g["scores"][0, n - 1] -= np.float32(3 * tol)
    elif plant == "swap":
        j = next(j for j in range(n - 1) if ref["scores"][0, j] - ref["scores"][0, j + 1] > tol
                 and g["parents"][0, j + 1] != j)
        for k in ("tokens", "parents", "depths", "pos_ids", "scores"):
            g[k][0, [j, j + 1]] = g[k][0, [j + 1, j]]
    elif plant == "mask":
        g["mask"][0, i, 0] &= ~np.int64(1 << int(g["parents"][0, i]))
    elif plant == "padding":
        g["tokens"][0, HEAP.B - 1] = 3 if n < HEAP.B else g["tokens"][0, HEAP.B - 1]
        g["n_nodes"][0] = n - 1
    elif plant == "count":
        g["n_nodes"][1] -= 1
    elif plant == "parent":
        g["parents"][0, i] = -1
        g["depths"][0, i] = 1
        g["pos_ids"][0, i] = HEAP.pos_offset + 1
    with pytest.raises(AssertionError):
        compare_pop_order_tree(HEAP, ref, g, tol, sc)
