"""Pins of the fp64 oracle against what the paper and mathematics fix.

Nothing here retypes the oracle's code: every check compares it with a
library routine, exhaustive enumeration, a closed form, or a structural
invariant the paper states (Lemma 1, prefix closure, monotone scores).
"""
import itertools

import numpy as np
import pytest
import torch

import oracle
from refs import (TorchHead, all_path_scores, child_logq, child_logq_restricted, ddtree_topB,
                  topK_candidates, weights64)
from workloads import TOY, Config, bf16_bits_to_f32, f32_to_bf16_bits, make_inputs


def tiny(**kw):
    base = dict(name="tiny", nseq=1, V=5, d=8, L=3, W=125, k=5, B=20, wdtype="f32",
                temperature=0.0, seed=77)
    base.update(kw)
    return Config(**base)


def rand_inputs(cfg, e_std=0.7, seed=None):
    """Seeded inputs with a large E so the correction head visibly matters."""
    g = np.random.Generator(np.random.PCG64(cfg.seed if seed is None else seed))
    d = cfg.d
    Wi = (g.standard_normal((d, 2 * d)) / np.sqrt(2 * d)).astype(np.float32)
    Wo = (g.standard_normal((d, d)) / np.sqrt(d)).astype(np.float32)
    E = (g.standard_normal((cfg.V, d)) * e_std).astype(np.float32)
    Dlog = (g.standard_normal((cfg.nseq, cfg.L, cfg.V)) * 1.5).astype(np.float32)
    h0 = g.standard_normal((cfg.nseq, d)).astype(np.float32)
    if cfg.wdtype == "bf16":
        Wi, Wo, E = f32_to_bf16_bits(Wi), f32_to_bf16_bits(Wo), f32_to_bf16_bits(E)
    return dict(Wi=Wi, Wo=Wo, E=E, Dlog=Dlog, h0=h0)


def run(cfg, x):
    return oracle.build_tree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])


# --------------------------------------------------------------- pieces

@pytest.mark.parametrize("wdtype", ["f32", "bf16"])
def test_head_matches_library_modules(wdtype):
    cfg = tiny(d=48, V=11, wdtype=wdtype)
    x = rand_inputs(cfg)
    ref = TorchHead(cfg, x["Wi"], x["Wo"], x["E"])
    g = np.random.Generator(np.random.PCG64(5))
    for tok in (0, 3, 10):
        hp = g.standard_normal(cfg.d)
        got = oracle.head(cfg, x["Wi"], x["Wo"], x["E"], hp, tok)
        want = ref(torch.from_numpy(hp), tok).numpy()
        np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)
        # RMSNorm without gain: mean square is 1 up to eps
        assert abs(np.mean(got ** 2) - 1.0) < 1e-5


@pytest.mark.parametrize("wdtype,cand_k", [("f32", 0), ("bf16", 0), ("f32", 3)])
def test_teacher_forced_helpers_match_torch(wdtype, cand_k):
    """The teacher-forced helpers the GPU parity tests use: the state after a
    path is the library-module head applied token by token from h_0; the
    Eq. 5 scores along a path and a prefix's children equal the torch
    log-softmax (over C_i for cand_k > 0) of the same states."""
    cfg = tiny(V=9, d=16, L=4, W=4, k=4, wdtype=wdtype, cand_k=cand_k, temperature=0.8)
    x = rand_inputs(cfg)
    head = TorchHead(cfg, x["Wi"], x["Wo"], x["E"])
    E64 = head.E
    path = np.array([4, 0, 7], np.int32)
    h = torch.from_numpy(x["h0"][0].astype(np.float64))
    states = [h]
    for t in path:
        h = head(h, int(t))
        states.append(h)
    for n in range(len(path) + 1):
        got = oracle.path_state(cfg, x["Wi"], x["Wo"], x["E"], x["h0"][0], path[:n])
        np.testing.assert_allclose(got, states[n].numpy(), rtol=0, atol=1e-12)
    want, acc = [], 0.0
    for i, t in enumerate(path):
        if cand_k:
            lq = child_logq_restricted(cfg, E64, x["Dlog"][0, i], states[i], topK_candidates(x["Dlog"][0, i], cand_k))
        else:
            lq = child_logq(cfg, E64, x["Dlog"][0, i], states[i])
        acc += float(lq[int(t)]) + cfg.beta
        want.append(acc)
    got = oracle.path_scores(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"][0], x["h0"][0], path)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)
    n = 2
    if cand_k:
        lq = child_logq_restricted(cfg, E64, x["Dlog"][0, n], states[n], topK_candidates(x["Dlog"][0, n], cand_k))
    else:
        lq = child_logq(cfg, E64, x["Dlog"][0, n], states[n])
    kk = 3
    tok, lqk, lse, allq = oracle.node_children(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"][0], x["h0"][0], path[:n], kk,
                                                want_all=True)
    lqn = lq.numpy()
    np.testing.assert_allclose(allq, lqn, rtol=0, atol=1e-12)
    np.testing.assert_array_equal(tok, np.lexsort((np.arange(cfg.V), -lqn))[:kk])
    np.testing.assert_allclose(lqk, lqn[tok], rtol=0, atol=1e-12)


def test_child_logits_and_log_softmax_match_torch():
    cfg = tiny(V=300, d=32, temperature=0.7)
    x = rand_inputs(cfg)
    h = np.random.Generator(np.random.PCG64(9)).standard_normal(cfg.d)
    z = oracle.child_logits(cfg, x["E"], x["Dlog"][0, 1], h)
    zt = (torch.from_numpy(x["Dlog"][0, 1].astype(np.float64))
          + weights64(cfg, x["E"]) @ torch.from_numpy(h)) / 0.7
    np.testing.assert_allclose(z, zt.numpy(), rtol=0, atol=1e-12)
    lq, lse = oracle.log_softmax(z)
    np.testing.assert_allclose(lq, child_logq(cfg, weights64(cfg, x["E"]), x["Dlog"][0, 1],
                                              torch.from_numpy(h)).numpy(), atol=1e-12)
    assert abs(np.exp(lq).sum() - 1.0) < 1e-12
    assert np.all(lq <= 0.0)
    assert abs(lse - float(torch.logsumexp(zt, 0))) < 1e-12


def test_log_softmax_clamp_and_neg_inf():
    # a single finite logit: log q = 0 exactly (clamped), others -inf
    z = np.array([-np.inf, 3.0, -np.inf])
    lq, lse = oracle.log_softmax(z)
    assert lq[1] == 0.0 and np.isneginf(lq[0]) and np.isneginf(lq[2]) and lse == 3.0
    lq, lse = oracle.log_softmax(np.full(4, -np.inf))
    assert np.all(np.isneginf(lq)) and np.isneginf(lse)


def test_topk_matches_lexsort_with_ties():
    g = np.random.Generator(np.random.PCG64(3))
    x = np.round(g.standard_normal(500), 1)          # many exact ties
    x[[7, 99]] = -np.inf
    for kk in (1, 5, 37, 500):
        want = np.lexsort((np.arange(x.size), -x))[:kk]   # value desc, index asc
        np.testing.assert_array_equal(oracle.topk(x, kk), want)


# ------------------------------------------------- brute force on tiny V/L

@pytest.mark.parametrize("temperature,beta", [(0.0, -0.2), (0.7, 0.0)])
def test_bruteforce_full_supertree(temperature, beta):
    """W = V^L, k = V: the supertree is every prefix; each node's score must
    equal an independent per-path recomputation, and the pruned tree must be
    the brute-force top-B."""
    cfg = tiny(temperature=temperature, beta=beta)
    x = rand_inputs(cfg)
    r = run(cfg, x)
    brute = all_path_scores(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"][0], x["h0"][0], cfg.L)
    paths = oracle.node_paths(r["st_tok"], r["st_parent"], r["st_count"], 0, cfg.W)
    assert len(paths) == len(brute) == 5 + 25 + 125
    for nid, p in paths.items():
        assert abs(r["st_score"][0].reshape(-1)[nid] - brute[p]) < 1e-12
    ranked = sorted(brute.items(), key=lambda kv: -kv[1])
    assert ranked[cfg.B - 1][1] - ranked[cfg.B][1] > 1e-9
    want = {p for p, _ in ranked[:cfg.B]}
    emitted = set()
    for i in range(r["n_nodes"][0]):
        path = []
        j = i
        while j >= 0:
            path.append(int(r["tokens"][0, j]))
            j = int(r["parents"][0, j])
        emitted.add(tuple(reversed(path)))
    assert emitted == want


@pytest.mark.parametrize("V,W,k", [(6, 4, 4), (6, 5, 2), (7, 3, 7)])
def test_bruteforce_beam_levels(V, W, k):
    """Each S_d is the top-W (by Eq. 5 score) among the per-node top-k
    children of S_{d-1}, every child scored by an independent recomputation.
    For k >= W this is the same as the top-W over all V children."""
    cfg = tiny(V=V, W=W, k=k, L=4, B=7, d=6, seed=11)
    x = rand_inputs(cfg)
    r = run(cfg, x)
    head = TorchHead(cfg, x["Wi"], x["Wo"], x["E"])
    E64 = head.E
    frontier = [((), 0.0, torch.from_numpy(x["h0"][0].astype(np.float64)))]
    for dep in range(1, cfg.L + 1):
        cands = []
        for pi, (path, s, h) in enumerate(frontier):
            lq = child_logq(cfg, E64, x["Dlog"][0, dep - 1], h).numpy()
            order = np.lexsort((np.arange(V), -lq))
            allowed = order[:k] if k < W else order   # k >= W: all children
            for t in allowed:
                cands.append((s + lq[t] + cfg.beta, path + (int(t),), h, int(t)))
        cands.sort(key=lambda c: -c[0])
        keep = cands[:W]
        got = [tuple(oracle.node_paths(r["st_tok"], r["st_parent"], r["st_count"], 0, W)
                     [(dep - 1) * W + j]) for j in range(int(r["st_count"][0, dep - 1]))]
        assert got == [c[1] for c in keep]
        np.testing.assert_allclose(r["st_score"][0, dep - 1, :len(keep)],
                                   [c[0] for c in keep], atol=1e-12)
        frontier = [(c[1], c[0], head(c[2], c[3])) for c in keep]


# ---------------------------------------------------------- special cases

def test_zero_E_is_ddtree_optimal_tree():
    """E = 0 makes q~ path independent (Sec. 3.3): scores reduce to
    sum_i log_softmax(Dlog_i)[u_i] + beta d, and with W, k >= B the pruned
    tree equals DDTree's best-first top-B prefixes."""
    cfg = tiny(V=40, d=16, L=5, W=12, k=12, B=12, beta=-0.2)
    x = rand_inputs(cfg)
    x["E"] = np.zeros_like(x["E"])
    r = run(cfg, x)
    rows = [torch.log_softmax(torch.from_numpy(x["Dlog"][0, i].astype(np.float64)), 0).numpy()
            + cfg.beta for i in range(cfg.L)]
    want = ddtree_topB(rows, cfg.B)
    got = {}
    for i in range(r["n_nodes"][0]):
        path, j = [], i
        while j >= 0:
            path.append(int(r["tokens"][0, j]))
            j = int(r["parents"][0, j])
        got[tuple(reversed(path))] = r["scores"][0, i]
    assert set(got) == {p for p, _ in want}
    for p, s in want:
        assert abs(got[p] - s) < 1e-12


def test_greedy_chain_W1_k1():
    """W = k = 1: the tree is the greedy corrected chain; each step is the
    argmax of a library log-softmax, the state advanced by the library head."""
    cfg = tiny(V=64, d=24, L=6, W=1, k=1, B=6, temperature=1.0)
    x = rand_inputs(cfg)
    r = run(cfg, x)
    head = TorchHead(cfg, x["Wi"], x["Wo"], x["E"])
    h = torch.from_numpy(x["h0"][0].astype(np.float64))
    s = 0.0
    for i in range(cfg.L):
        lq = child_logq(cfg, head.E, x["Dlog"][0, i], h)
        t = int(torch.argmax(lq))
        s += float(lq[t]) + cfg.beta
        assert r["tokens"][0, i] == t and r["parents"][0, i] == i - 1
        assert abs(r["scores"][0, i] - s) < 1e-12
        h = head(h, t)


def test_single_depth_is_topk_of_log_softmax():
    cfg = tiny(V=500, d=32, L=1, W=9, k=12, B=6)
    x = rand_inputs(cfg)
    r = run(cfg, x)
    lq = child_logq(cfg, weights64(cfg, x["E"]), x["Dlog"][0, 0],
                    torch.from_numpy(x["h0"][0].astype(np.float64)))
    vals, idx = torch.topk(lq, 6)
    np.testing.assert_array_equal(r["tokens"][0, :6], idx.numpy())
    np.testing.assert_allclose(r["scores"][0, :6], vals.numpy() + cfg.beta, atol=1e-12)
    assert np.all(r["parents"][0, :6] == -1) and np.all(r["depths"][0, :6] == 1)


# ------------------------------------------------------------ Lemma 1 etc.

def _check_tree_structure(cfg, r):
    """Prefix closure, monotone scores, depths, position ids and the ancestor
    mask (transitive closure of the parent relation, diagonal set)."""
    nw = (cfg.B + 63) // 64
    for s in range(cfg.nseq):
        n = int(r["n_nodes"][s])
        par = r["parents"][s]
        for i in range(n):
            p = int(par[i])
            assert -1 <= p < i
            if p >= 0:
                assert r["depths"][s, i] == r["depths"][s, p] + 1
                assert r["scores"][s, i] <= r["scores"][s, p]
            else:
                assert r["depths"][s, i] == 1
            assert r["pos_ids"][s, i] == cfg.pos_offset + r["depths"][s, i]
            anc = {i}
            j = p
            while j >= 0:
                anc.add(j)
                j = int(par[j])
            bits = {b for b in range(cfg.B) if (int(r["mask"][s, i, b // 64]) >> (b % 64)) & 1}
            assert bits == anc
            assert len(bits) == r["depths"][s, i]
        for i in range(n, cfg.B):
            assert r["tokens"][s, i] == -1 and r["parents"][s, i] == -2
            assert r["depths"][s, i] == 0 and np.all(r["mask"][s, i] == 0)
        assert r["mask"].shape[-1] == nw


@pytest.mark.parametrize("beta", [0.0, -0.2, -1.5])
def test_lemma1_heap_equals_topB(beta):
    cfg = tiny(V=9, d=12, L=6, W=7, k=4, B=19, beta=beta, nseq=3, pos_offset=100)
    x = rand_inputs(cfg)
    r = run(cfg, x)
    _check_tree_structure(cfg, r)
    for s in range(cfg.nseq):
        popped = oracle.heap_select(cfg, r["st_parent"], r["st_score"], r["st_count"], s)
        order = sorted(((r["st_score"][s].reshape(-1)[i], i) for dep in range(cfg.L)
                        for i in [dep * cfg.W + j for j in range(r["st_count"][s, dep])]),
                       key=lambda t: (-t[0], t[1]))
        sel = [i for _, i in order[:cfg.B]]
        assert set(popped.tolist()) == set(sel)


def test_lemma1_with_exact_ties():
    """Quantised drafter logits and E = 0 give many exactly tied scores; with
    the node-id tie-break the heap and the top-B still agree."""
    cfg = tiny(V=6, d=8, L=5, W=9, k=6, B=23, beta=0.0)
    x = rand_inputs(cfg)
    x["E"] = np.zeros_like(x["E"])
    x["Dlog"] = np.round(x["Dlog"]).astype(np.float32)
    x["Dlog"][:, :, 0] = x["Dlog"][:, :, 1]
    r = run(cfg, x)
    sc = r["st_score"][0].reshape(-1)
    ids = [dep * cfg.W + j for dep in range(cfg.L) for j in range(r["st_count"][0, dep])]
    vals = [sc[i] for i in ids]
    assert len(vals) - len(set(vals)) > 5          # there really are ties
    popped = oracle.heap_select(cfg, r["st_parent"], r["st_score"], r["st_count"], 0)
    top = sorted(ids, key=lambda i: (-sc[i], i))[:cfg.B]
    assert popped.tolist() == top                  # identical pop order too
    _check_tree_structure(cfg, r)


def test_positive_beta_breaks_heap_equivalence():
    """Lemma 1 needs beta <= 0: a hand-built supertree where a child
    outranks its parent makes top-B not prefix closed."""
    cfg = tiny(V=3, L=2, W=2, k=2, B=1, beta=0.5)
    st_tok = np.array([[[0, -1], [1, -1]]], np.int32)
    st_parent = np.array([[[-1, -1], [0, -1]]], np.int32)
    st_score = np.array([[[-0.1, -np.inf], [0.3, -np.inf]]])
    st_count = np.array([[1, 1]], np.int32)
    popped = oracle.heap_select(cfg, st_parent, st_score, st_count, 0)
    assert popped.tolist() == [0]                  # the heap can only pop the root child
    r = oracle.prune_emit(cfg, st_tok, st_parent, st_score, st_count)
    assert r["rc"] == -1                           # top-1 picked the orphan child


def test_prune_emit_hand_example():
    """A 6-node supertree with known answer: B = 4 keeps ids {0,1,2,4}."""
    cfg = tiny(V=10, L=3, W=2, k=2, B=4, beta=-0.2, pos_offset=7)
    st_tok = np.array([[[5, 6], [7, 8], [9, 1]]], np.int32)
    st_parent = np.array([[[-1, -1], [0, 1], [0, 1]]], np.int32)
    st_score = np.array([[[-0.3, -0.5], [-0.9, -0.6], [-1.2, -0.7]]])
    st_count = np.array([[2, 2, 2]], np.int32)
    r = oracle.prune_emit(cfg, st_tok, st_parent, st_score, st_count)
    assert r["rc"] == 0 and r["n_nodes"][0] == 4
    # selected ids by (score desc, id asc): 0(-0.3) 1(-0.5) 3(-0.6) 5(-0.7)
    np.testing.assert_array_equal(r["tokens"][0], [5, 6, 8, 1])
    np.testing.assert_array_equal(r["parents"][0], [-1, -1, 1, 2])
    np.testing.assert_array_equal(r["depths"][0], [1, 1, 2, 3])
    np.testing.assert_array_equal(r["pos_ids"][0], [8, 8, 9, 10])
    np.testing.assert_array_equal(r["mask"][0, :, 0], [0b1, 0b10, 0b110, 0b1110])
    assert abs(r["prune_gap"][0] - (-0.7 + 0.9)) < 1e-15


def test_frontier_ties_across_parents_by_parent_slot():
    """Exact score ties at the W-th cut, across parents (the reading of the
    frontier order: score desc, parent slot asc, rank in the parent's list
    asc).  With E = 0 the head has no effect and log q~ is the log-softmax of
    the drafter row.  Depth 1: row [2, 2, -5, -5] makes tokens 0 and 1 equal,
    so slots 0 and 1 carry the same path score, and the cut at W = 3 falls
    inside the tie {2, 3} (rank asc keeps token 2).  Depth 2: row [3, 0, 0, 0]
    gives both of those parents the same children's scores; the two best are
    (slot 0, token 0) and (slot 1, token 0), and the third comes from the tie
    group {tokens 1, 2, 3} x {slots 0, 1}: slot 0, token 1."""
    cfg = tiny(V=4, d=8, L=2, W=3, k=4, B=6, beta=-0.2)
    x = rand_inputs(cfg)
    x["E"][:] = 0.0
    x["Dlog"][0, 0] = [2.0, 2.0, -5.0, -5.0]
    x["Dlog"][0, 1] = [3.0, 0.0, 0.0, 0.0]
    r = run(cfg, x)
    np.testing.assert_array_equal(r["st_count"][0], [3, 3])
    np.testing.assert_array_equal(r["st_tok"][0, 0], [0, 1, 2])
    np.testing.assert_array_equal(r["st_tok"][0, 1], [0, 0, 1])
    np.testing.assert_array_equal(r["st_parent"][0, 1], [0, 1, 0])
    # the ties are exact, and the scores are the closed form of Eq. 5
    l1 = torch.log_softmax(torch.tensor([2.0, 2.0, -5.0, -5.0], dtype=torch.float64), 0).numpy()
    l2 = torch.log_softmax(torch.tensor([3.0, 0.0, 0.0, 0.0], dtype=torch.float64), 0).numpy()
    assert r["st_score"][0, 0, 0] == r["st_score"][0, 0, 1]
    assert r["st_score"][0, 1, 0] == r["st_score"][0, 1, 1]
    np.testing.assert_allclose(r["st_score"][0, 0], l1[[0, 1, 2]] - 0.2, atol=1e-12)
    np.testing.assert_allclose(r["st_score"][0, 1], [l1[0] + l2[0] - 0.4, l1[1] + l2[0] - 0.4, l1[0] + l2[1] - 0.4],
                               atol=1e-12)
    _check_tree_structure(cfg, r)


def test_neg_inf_children_are_never_retained():
    cfg = tiny(V=8, d=8, L=3, W=6, k=4, B=30)
    x = rand_inputs(cfg)
    x["Dlog"][0, 1, 2:] = -np.inf        # depth 2: only tokens 0, 1 possible
    r = run(cfg, x)
    c = r["st_count"][0]
    assert c[1] == min(cfg.W, 2 * c[0])
    assert set(r["st_tok"][0, 1, :c[1]].tolist()) <= {0, 1}
    assert np.all(np.isfinite(r["st_score"][0, 1, :c[1]]))
    _check_tree_structure(cfg, r)


def test_toy_config_structure():
    x = make_inputs(TOY)
    r = run(TOY, x)
    assert r["n_nodes"][0] == 16 and list(r["st_count"][0]) == [4, 4, 4, 4]
    _check_tree_structure(TOY, r)
    # teacher-forced helpers agree with the construction
    paths = oracle.node_paths(r["st_tok"], r["st_parent"], r["st_count"], 0, TOY.W)
    for nid in (0, 5, 15):
        p = paths[nid]
        sc = oracle.path_scores(TOY, x["Wi"], x["Wo"], x["E"], x["Dlog"][0], x["h0"][0], p)
        assert abs(sc[-1] - r["st_score"][0].reshape(-1)[nid]) < 1e-9
        tok, lq, lse, _ = oracle.node_children(TOY, x["Wi"], x["Wo"], x["E"], x["Dlog"][0],
                                               x["h0"][0], p[:-1], TOY.k + 1)
        dep = len(p)
        par = r["st_parent"][0, dep - 1, nid % TOY.W] if dep > 1 else 0
        np.testing.assert_array_equal(tok, r["nd_tok"][0, dep - 1, par])
        np.testing.assert_allclose(lq, r["nd_logq"][0, dep - 1, par], atol=1e-12)


def test_bf16_roundtrip_helper():
    x = np.array([1.0, 1.00390625, 1.005859375, -3.0e-3, 0.0], np.float32)
    b = f32_to_bf16_bits(x)
    y = bf16_bits_to_f32(b)
    # 1.00390625 is the exact midpoint 1 + 2^-8 -> rounds to even (1.0)
    assert y[0] == 1.0 and y[1] == 1.0 and y[2] == np.float32(1.0078125)
    assert abs(y[3] - x[3]) <= abs(x[3]) * 2 ** -8


def test_prune_tiebreak_inside_tied_group():
    """Budget cuts that fall inside a group of exactly tied scores: the
    emitted nodes must be the smallest ids of the group (ancestors first),
    matching both a library sort by (score desc, id asc) and the heap."""
    cfg0 = tiny(V=6, d=8, L=5, W=9, k=6, B=23, beta=0.0)
    x = rand_inputs(cfg0)
    x["E"] = np.zeros_like(x["E"])
    x["Dlog"] = np.round(x["Dlog"]).astype(np.float32)
    x["Dlog"][:, :, 0] = x["Dlog"][:, :, 1]
    r = run(cfg0, x)
    sc = r["st_score"][0].reshape(-1)
    ids = [dep * cfg0.W + j for dep in range(cfg0.L) for j in range(r["st_count"][0, dep])]
    order = sorted(ids, key=lambda i: (-sc[i], i))
    cuts = [b for b in range(1, len(order)) if sc[order[b - 1]] == sc[order[b]]]
    assert len(cuts) >= 3
    for B in cuts:
        cfg = cfg0.replace(B=B)
        e = oracle.prune_emit(cfg, r["st_tok"], r["st_parent"], r["st_score"], r["st_count"])
        assert e["rc"] == 0
        keep = sorted(order[:B])
        np.testing.assert_array_equal(e["tokens"][0, :B], r["st_tok"][0].reshape(-1)[keep])
        np.testing.assert_array_equal(e["depths"][0, :B], [i // cfg.W + 1 for i in keep])
        popped = oracle.heap_select(cfg, r["st_parent"], r["st_score"], r["st_count"], 0)
        assert sorted(popped.tolist()) == keep


# ------------------------------------- candidate-restricted scoring (K)

def _emitted_paths(r, s=0):
    out = {}
    for i in range(r["n_nodes"][s]):
        path, j = [], i
        while j >= 0:
            path.append(int(r["tokens"][s, j]))
            j = int(r["parents"][s, j])
        out[tuple(reversed(path))] = r["scores"][s, i]
    return out


def test_candidates_match_lexsort_with_ties():
    """C_d = TopK(L_d^base, K): the K largest base logits, ties by token asc."""
    cfg = tiny(V=300, cand_k=37)
    g = np.random.default_rng(5)
    row = np.round(g.standard_normal(cfg.V) * 2) .astype(np.float32) / 2  # many exact ties
    got = oracle.candidates(cfg, row)
    np.testing.assert_array_equal(got, topK_candidates(row, cfg.cand_k))
    assert np.all(np.diff(got) > 0)


def test_restricted_with_K_equal_V_is_full_vocabulary():
    """K = V restricts nothing: the tree equals the full-vocabulary tree."""
    cfg = tiny(V=50, d=12, L=4, W=6, k=6, B=15, temperature=0.8, seed=21)
    x = rand_inputs(cfg)
    full = run(cfg, x)
    rest = run(cfg.replace(cand_k=cfg.V), x)
    for key in ("st_tok", "st_parent", "st_count", "tokens", "parents", "depths", "mask", "n_nodes"):
        np.testing.assert_array_equal(full[key], rest[key])
    np.testing.assert_allclose(full["st_score"], rest["st_score"], atol=1e-12)
    np.testing.assert_allclose(full["nd_lse"], rest["nd_lse"], atol=1e-12)


@pytest.mark.parametrize("temperature,beta", [(0.0, -0.2), (0.9, 0.0)])
def test_restricted_bruteforce_full_supertree(temperature, beta):
    """V = 7, K = 3, W = K^L, k = K: the supertree is every path through the
    candidate sets; each node's score must equal an independent per-path
    recomputation with q~ renormalised over C_d (library log_softmax on the
    subset), and the pruned tree must be the brute-force top-B."""
    cfg = tiny(V=7, L=3, W=27, k=3, B=17, cand_k=3, temperature=temperature, beta=beta, seed=31)
    x = rand_inputs(cfg)
    r = run(cfg, x)
    brute = all_path_scores(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"][0], x["h0"][0], cfg.L)
    paths = oracle.node_paths(r["st_tok"], r["st_parent"], r["st_count"], 0, cfg.W)
    assert len(paths) == len(brute) == 3 + 9 + 27
    for nid, p in paths.items():
        assert abs(r["st_score"][0].reshape(-1)[nid] - brute[p]) < 1e-12
    ranked = sorted(brute.items(), key=lambda kv: -kv[1])
    assert ranked[cfg.B - 1][1] - ranked[cfg.B][1] > 1e-9
    assert set(_emitted_paths(r)) == {p for p, _ in ranked[:cfg.B]}


def test_restricted_beam_levels_and_normalisation():
    """Each S_d is the top-W of the K candidates of every node of S_{d-1},
    scored by an independent recomputation; q~ sums to one over C_d and is
    zero outside it."""
    cfg = tiny(V=60, d=10, L=4, W=5, k=5, B=9, cand_k=8, temperature=0.7, seed=41)
    x = rand_inputs(cfg)
    r = run(cfg, x)
    head = TorchHead(cfg, x["Wi"], x["Wo"], x["E"])
    frontier = [((), 0.0, torch.from_numpy(x["h0"][0].astype(np.float64)))]
    for dep in range(1, cfg.L + 1):
        cand = topK_candidates(x["Dlog"][0, dep - 1], cfg.cand_k)
        cands = []
        for path, s, h in frontier:
            lq = child_logq_restricted(cfg, head.E, x["Dlog"][0, dep - 1], h, cand).numpy()
            assert abs(np.exp(lq[cand]).sum() - 1.0) < 1e-12
            for t in cand:
                cands.append((s + lq[t] + cfg.beta, path + (int(t),), h, int(t)))
        cands.sort(key=lambda c: -c[0])
        keep = cands[:cfg.W]
        got = [tuple(oracle.node_paths(r["st_tok"], r["st_parent"], r["st_count"], 0, cfg.W)
                     [(dep - 1) * cfg.W + j]) for j in range(int(r["st_count"][0, dep - 1]))]
        assert got == [c[1] for c in keep]
        np.testing.assert_allclose(r["st_score"][0, dep - 1, :len(keep)], [c[0] for c in keep],
                                   atol=1e-12)
        frontier = [(c[1], c[0], head(c[2], c[3])) for c in keep]
    # the oracle's own per-node distribution: zero outside C_d, sums to one over it
    tok, lq, lse, lq_all = oracle.node_children(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"][0], x["h0"][0],
                                                np.array([], np.int32), cfg.k, want_all=True)
    cand = topK_candidates(x["Dlog"][0, 0], cfg.cand_k)
    outside = np.setdiff1d(np.arange(cfg.V), cand)
    assert np.all(np.isneginf(lq_all[outside]))
    assert abs(np.exp(lq_all[cand]).sum() - 1.0) < 1e-12
    assert set(tok.tolist()) <= set(cand.tolist())


def test_restricted_zero_E_is_ddtree_over_candidates():
    """E = 0: q~ is the base distribution renormalised over C_d, path
    independent, so with W, k >= B the pruned tree equals DDTree's best-first
    top-B over the restricted marginals."""
    cfg = tiny(V=80, d=16, L=5, W=12, k=12, B=12, cand_k=16, beta=-0.2, seed=51)
    x = rand_inputs(cfg)
    x["E"] = np.zeros_like(x["E"])
    r = run(cfg, x)
    rows = []
    for i in range(cfg.L):
        cand = topK_candidates(x["Dlog"][0, i], cfg.cand_k)
        row = np.full(cfg.V, -np.inf)
        row[cand] = torch.log_softmax(torch.from_numpy(x["Dlog"][0, i, cand].astype(np.float64)), 0).numpy()
        rows.append(row + cfg.beta)
    want = ddtree_topB(rows, cfg.B)
    got = _emitted_paths(r)
    assert set(got) == {p for p, _ in want}
    for p, s in want:
        assert abs(got[p] - s) < 1e-12


def test_restricted_tree_structure():
    """Prefix closure, monotone scores, depths, position ids and the mask hold
    in the restricted mode too, and every token lies in its depth's C_d."""
    cfg = tiny(V=200, d=16, L=6, W=6, k=6, B=20, cand_k=10, temperature=1.0, seed=61, nseq=2)
    x = rand_inputs(cfg)
    r = run(cfg, x)
    _check_tree_structure(cfg, r)
    for s in range(cfg.nseq):
        for i in range(r["n_nodes"][s]):
            dep = int(r["depths"][s, i])
            assert r["tokens"][s, i] in set(topK_candidates(x["Dlog"][s, dep - 1], cfg.cand_k).tolist())


# ------------------------------------ the two constructions of Table 2

def paths_of(r, s=0):
    """{token path: score} of an emitted tree, and the paths in row order."""
    out, order = {}, []
    for i in range(int(r["n_nodes"][s])):
        path, j = [], i
        while j >= 0:
            path.append(int(r["tokens"][s, j]))
            j = int(r["parents"][s, j])
        p = tuple(reversed(path))
        out[p] = float(r["scores"][s, i])
        order.append(p)
    return out, order


def check_pop_order_tree(cfg, r, s=0):
    """Rows in pop order: parents precede children, scores never increase
    along the rows (best-first), depths/positions/mask consistent, padding."""
    n = int(r["n_nodes"][s])
    for i in range(n):
        p = int(r["parents"][s, i])
        assert -1 <= p < i
        assert r["depths"][s, i] == (1 if p < 0 else r["depths"][s, p] + 1)
        assert r["pos_ids"][s, i] == cfg.pos_offset + r["depths"][s, i]
        if i:
            assert r["scores"][s, i] <= r["scores"][s, i - 1]
        anc, j = set(), i
        while j >= 0:
            anc.add(j)
            j = int(r["parents"][s, j])
        row = r["mask"][s, i]
        assert {b for b in range(cfg.B) if (int(row[b // 64]) >> (b % 64)) & 1} == anc
    for i in range(n, cfg.B):
        assert r["tokens"][s, i] == -1 and r["parents"][s, i] == -2 and not np.any(r["mask"][s, i])


def torch_chain(cfg, x, s=0):
    """The greedy corrected chain with the library head: per depth the
    clamped log-softmax row, its argmax token and its log-sum-exp."""
    head = TorchHead(cfg, x["Wi"], x["Wo"], x["E"])
    h = torch.from_numpy(x["h0"][s].astype(np.float64))
    Tp = cfg.temperature if cfg.temperature > 0 else 1.0
    rows, toks, lses = [], [], []
    K = int(getattr(cfg, "cand_k", 0))
    for i in range(cfg.L):
        if K > 0:
            cand = topK_candidates(x["Dlog"][s, i], K)
            lq = child_logq_restricted(cfg, head.E, x["Dlog"][s, i], h, cand)
            z = (torch.from_numpy(x["Dlog"][s, i].astype(np.float64))[torch.from_numpy(cand)] +
                 head.E[torch.from_numpy(cand)] @ h) / Tp
        else:
            lq = child_logq(cfg, head.E, x["Dlog"][s, i], h)
            z = (torch.from_numpy(x["Dlog"][s, i].astype(np.float64)) + head.E @ h) / Tp
        t = int(np.lexsort((np.arange(cfg.V), -lq.numpy()))[0])
        rows.append(lq.numpy())
        toks.append(t)
        lses.append(float(torch.logsumexp(z, 0)))
        h = head(h, t)
    return rows, toks, lses


@pytest.mark.parametrize("cand_k", [0, 4])
def test_chain_is_the_greedy_corrected_chain(cand_k):
    """Domino-chain + DDTree, step 1: the chain follows the argmax of the
    corrected distribution of its own prefix (library head and softmax)."""
    cfg = tiny(V=23, d=16, L=5, W=1, k=1, B=9, temperature=0.7, cand_k=cand_k)
    x = rand_inputs(cfg)
    r = oracle.chain_ddtree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    _, toks, lses = torch_chain(cfg, x)
    assert list(r["chain_tok"][0]) == toks
    np.testing.assert_allclose(r["chain_lse"][0], lses, rtol=0, atol=1e-12)


@pytest.mark.parametrize("beta", [0.0, -0.2])
@pytest.mark.parametrize("B", [1, 7, 40])
def test_chain_ddtree_bruteforce(beta, B):
    """Domino-chain + DDTree = the top-B prefixes, over every token path, of
    the sum of the chain-conditioned log-probabilities (+ beta d): exhaustive
    enumeration on V = 5, L = 3, and the rows come out best first."""
    cfg = tiny(V=5, d=8, L=3, W=1, k=1, B=B, beta=beta, temperature=1.3)
    x = rand_inputs(cfg)
    r = oracle.chain_ddtree(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    rows, _, _ = torch_chain(cfg, x)
    every = {}
    for n in range(1, cfg.L + 1):
        for p in itertools.product(range(cfg.V), repeat=n):
            every[p] = sum(rows[i][t] for i, t in enumerate(p)) + beta * n
    want = sorted(every.items(), key=lambda kv: -kv[1])[:B]
    got, _ = paths_of(r)
    assert set(got) == {p for p, _ in want}
    for p, sc in want:
        assert abs(got[p] - sc) < 1e-12
    check_pop_order_tree(cfg, r)


@pytest.mark.parametrize("cand_k", [0, 12])
def test_zero_E_chain_ddtree_and_seq_heap_are_ddtree(cand_k):
    """E = 0: the correction is path independent, so both Table 2
    constructions reduce to DDTree's best-first tree over the drafter's
    marginals (renormalised over C_d when restricted), in the same pop order."""
    cfg = tiny(V=40, d=16, L=5, W=1, k=1, B=25, beta=-0.2, cand_k=cand_k)
    x = rand_inputs(cfg)
    x["E"] = np.zeros_like(x["E"])
    rows = []
    for i in range(cfg.L):
        z = torch.from_numpy(x["Dlog"][0, i].astype(np.float64))
        if cand_k:
            cand = topK_candidates(x["Dlog"][0, i], cand_k)
            row = np.full(cfg.V, -np.inf)
            row[cand] = torch.log_softmax(z[torch.from_numpy(cand)], 0).numpy()
        else:
            row = torch.log_softmax(z, 0).numpy()
        rows.append(row + cfg.beta)
    want = ddtree_topB(rows, cfg.B)
    for fn in (oracle.chain_ddtree, oracle.seq_heap):
        r = fn(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
        got, order = paths_of(r)
        assert order == [p for p, _ in want]
        for p, sc in want:
            assert abs(got[p] - sc) < 1e-12
        check_pop_order_tree(cfg, r)


@pytest.mark.parametrize("beta,temperature", [(0.0, 0.0), (-0.2, 1.0), (-1.5, 0.6)])
def test_seq_heap_bruteforce(beta, temperature):
    """Sequential correction with heap = exact best-first under the corrected
    scores = the top-B of every token path by its Eq. 5 score, each path
    scored from the root on its own (library head), V = 5, L = 3."""
    cfg = tiny(V=5, d=8, L=3, W=1, k=1, B=30, beta=beta, temperature=temperature)
    x = rand_inputs(cfg)
    every = all_path_scores(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"][0], x["h0"][0], cfg.L)
    r = oracle.seq_heap(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    want = sorted(every.items(), key=lambda kv: -kv[1])[:cfg.B]
    got, _ = paths_of(r)
    assert set(got) == {p for p, _ in want}
    for p, sc in want:
        assert abs(got[p] - sc) < 1e-12
    check_pop_order_tree(cfg, r)
    # one corrected distribution per popped prefix above depth L, and the root's
    n_inner = int(np.sum((r["depths"][0, :r["n_nodes"][0]] < cfg.L) & (r["depths"][0, :r["n_nodes"][0]] > 0)))
    assert r["expansions"][0] == 1 + n_inner


def test_seq_heap_restricted_bruteforce():
    cfg = tiny(V=7, d=8, L=3, W=1, k=1, B=20, cand_k=3, temperature=0.9)
    x = rand_inputs(cfg)
    every = all_path_scores(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"][0], x["h0"][0], cfg.L)
    r = oracle.seq_heap(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    want = sorted(every.items(), key=lambda kv: -kv[1])[:cfg.B]
    got, _ = paths_of(r)
    assert set(got) == {p for p, _ in want}
    for p, sc in want:
        assert abs(got[p] - sc) < 1e-12


def test_seq_heap_equals_dartree_with_a_full_beam():
    """With a beam wide enough to hold every prefix (W = V^(L-1), k = V),
    Algorithm 1's supertree is the whole prefix tree and, by Lemma 1, its
    top-B pruning is the exact best-first tree of the sequential heap."""
    cfg = tiny(V=4, d=8, L=4, W=64, k=4, B=50, nseq=2, beta=-0.3, temperature=0.8)
    x = rand_inputs(cfg)
    a = run(cfg, x)
    b = oracle.seq_heap(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"], x["h0"])
    for s in range(cfg.nseq):
        pa, _ = paths_of(a, s)
        pb, _ = paths_of(b, s)
        assert set(pa) == set(pb)
        for p in pa:
            assert abs(pa[p] - pb[p]) < 1e-12
