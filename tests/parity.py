"""GPU-vs-oracle comparison helpers.

Rules (the contract of the parity tests):
  * path scores within `tol` (2e-3 for bf16 weights, 1e-5 for fp32);
  * topology compared as sets of token paths, required equal at every depth
    whose relevant oracle rank gap (frontier cut, or the k-th / (k+1)-th cut
    of a node whose k-th child is kept) is >= tol;
  * after a near tie every later depth of that sequence is checked against
    the oracle teacher-forced on the GPU's own parents: path scores within
    tol of the oracle's score of the same path, the kept set a valid top-W
    of the oracle's candidates (no depth escapes an oracle check);
  * the pruned and emitted tree always equals, bit for bit, the oracle's
    pruning and emission of the GPU's own supertree;
  * the emitted arrays (tokens, parents, depths, pos_ids, mask, n_nodes) are
    required bit-exact against the oracle's own tree when no oracle rank gap
    anywhere is below tol;
  * the GPU tree is always checked for structural validity.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle


def to_device(cfg, x, dev="cuda"):
    if cfg.wdtype == "bf16":
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev).view(torch.bfloat16)
    else:
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    return dict(Wi=t(x["Wi"]), Wo=t(x["Wo"]), E=t(x["E"]),
                Dlog=torch.from_numpy(x["Dlog"]).to(dev), h0=torch.from_numpy(x["h0"]).to(dev))


def tol_of(cfg):
    return 2e-3 if cfg.wdtype == "bf16" else 1e-5


def gpu_supertree(dart, h, cfg):
    st_tok = np.empty((cfg.nseq, cfg.L, cfg.W), np.int32)
    st_par = np.empty_like(st_tok)
    st_score = np.empty((cfg.nseq, cfg.L, cfg.W), np.float32)
    st_count = np.empty((cfg.nseq, cfg.L), np.int32)
    for dep in range(1, cfg.L + 1):
        tok, par, sc, cnt = dart.dart_get_frontier(h, dep, cfg)
        st_tok[:, dep - 1] = tok.cpu().numpy()
        st_par[:, dep - 1] = par.cpu().numpy()
        st_score[:, dep - 1] = sc.cpu().numpy()
        st_count[:, dep - 1] = cnt.cpu().numpy()
    return dict(st_tok=st_tok, st_parent=st_par, st_score=st_score, st_count=st_count)


def tree_to_numpy(t):
    return {k: v.cpu().numpy() for k, v in t.items()}


def emitted_paths(g, s):
    out = {}
    for i in range(int(g["n_nodes"][s])):
        path, j = [], i
        while j >= 0:
            path.append(int(g["tokens"][s, j]))
            j = int(g["parents"][s, j])
        out[tuple(reversed(path))] = float(g["scores"][s, i])
    return out


def check_structure(cfg, g):
    """Prefix closure, monotone scores, depths, position ids, ancestor mask
    and padding of an emitted tree."""
    nw = (cfg.B + 63) // 64
    for s in range(cfg.nseq):
        n = int(g["n_nodes"][s])
        assert 0 <= n <= cfg.B
        par = g["parents"][s]
        for i in range(n):
            p = int(par[i])
            assert -1 <= p < i, (s, i, p)
            if p >= 0:
                assert g["depths"][s, i] == g["depths"][s, p] + 1
                assert g["scores"][s, i] <= g["scores"][s, p]
            else:
                assert g["depths"][s, i] == 1
            assert g["pos_ids"][s, i] == cfg.pos_offset + g["depths"][s, i]
            assert np.isfinite(g["scores"][s, i])
            anc = {i}
            j = p
            while j >= 0:
                anc.add(j)
                j = int(par[j])
            row = g["mask"][s, i].view(np.uint64)
            bits = {b for b in range(cfg.B) if (int(row[b // 64]) >> (b % 64)) & 1}
            assert bits == anc, (s, i)
        for i in range(n, cfg.B):
            assert g["tokens"][s, i] == -1 and g["parents"][s, i] == -2
            assert g["depths"][s, i] == 0 and g["pos_ids"][s, i] == -1
            assert np.isneginf(g["scores"][s, i]) and not np.any(g["mask"][s, i])
        assert g["mask"].shape[-1] == nw


def relevant_gaps(cfg, ref, s, dep):
    """(cut gap, min adjacent gap among kept) of the oracle at this depth."""
    W, k = cfg.W, cfg.k
    fr = ref["fr_score"][s, dep - 1]
    cnt = int(ref["st_count"][s, dep - 1])
    cut = np.inf
    if cnt == W and np.isfinite(fr[W]):
        cut = fr[W - 1] - fr[W]
    # a node whose k-th child is kept: its k-th / (k+1)-th cut decides the set
    kx = ref["nd_tok"].shape[-1]
    if kx > k:
        for r in range(cnt):
            p = int(ref["st_parent"][s, dep - 1, r]) if dep > 1 else 0
            t = int(ref["st_tok"][s, dep - 1, r])
            if ref["nd_tok"][s, dep - 1, p, k - 1] == t:
                g = ref["nd_logq"][s, dep - 1, p, k - 1] - ref["nd_logq"][s, dep - 1, p, k]
                cut = min(cut, g)
    adj = np.diff(-fr[:cnt]) if cnt > 1 else np.array([np.inf])
    return cut, float(np.min(adj)) if adj.size else np.inf


def compare_with_oracle(cfg, ref, gst, g, tol, x=None):
    """Compares the GPU supertree `gst` and emitted tree `g` with the oracle
    run `ref`.  Returns a report dict; raises AssertionError on a mismatch
    the rank gaps do not excuse.

    Where a frontier legitimately differs at a near tie (oracle cut gap below
    `tol`), every later depth of that sequence is still checked against the
    oracle, teacher-forced on the GPU's own parents (`x` = the inputs is then
    required): each kept child's path score within `tol` of the oracle's
    score of the same path, and the kept set a valid top-W of the oracle's
    candidates.  The pruned tree of every sequence must equal, bit for bit,
    the oracle's pruning and emission of the GPU's own supertree."""
    rep = dict(near_tie=[], order_ties=0, arrays_exact=None, bit_identical=None,
               depths_teacher_forced=0, max_score_err=0.0)
    all_exact = True
    for s in range(cfg.nseq):
        rp = oracle.node_paths(ref["st_tok"], ref["st_parent"], ref["st_count"], s, cfg.W)
        gp = oracle.node_paths(gst["st_tok"], gst["st_parent"], gst["st_count"], s, cfg.W)
        sets_equal = True
        for dep in range(1, cfg.L + 1):
            rc = int(ref["st_count"][s, dep - 1])
            gc = int(gst["st_count"][s, dep - 1])
            r_paths = [rp[(dep - 1) * cfg.W + r] for r in range(rc)]
            g_paths = [gp[(dep - 1) * cfg.W + r] for r in range(gc)]
            cut, adj = relevant_gaps(cfg, ref, s, dep)
            if set(r_paths) != set(g_paths):
                assert cut < tol, f"seq {s} depth {dep}: frontier differs with oracle cut gap {cut}"
                rep["near_tie"].append((s, dep, float(cut)))
                sets_equal = False
                all_exact = False
                assert x is not None, "inputs needed to check the depths after a near tie"
                # oracle scores of the GPU's nodes above this depth (same paths as the oracle's)
                rs_all = {rp[i]: float(ref["st_score"][s, i // cfg.W, i % cfg.W]) for i in rp}
                known = {i: rs_all[gp[i]] for i in gp if i < (dep - 1) * cfg.W}
                tf = TeacherForced(cfg, x, s)
                for d2 in range(dep, cfg.L + 1):
                    e = validate_depth_teacher_forced(cfg, tf, gst, s, d2, tol, known)
                    rep["max_score_err"] = max(rep["max_score_err"], e)
                    rep["depths_teacher_forced"] += 1
                break
            rs = {p: ref["st_score"][s, dep - 1, r] for r, p in enumerate(r_paths)}
            for r, p in enumerate(g_paths):
                d = abs(float(gst["st_score"][s, dep - 1, r]) - rs[p])
                rep["max_score_err"] = max(rep["max_score_err"], d)
                assert d <= tol, f"seq {s} depth {dep} path score off by {d}"
            if adj < tol:
                rep["order_ties"] += 1
                all_exact = False
                for i in range(len(g_paths) - 1):
                    assert rs[g_paths[i]] >= rs[g_paths[i + 1]] - tol
            else:
                assert r_paths == g_paths, f"seq {s} depth {dep}: rank order differs"
        if sets_equal:
            if ref["prune_gap"][s] < tol:
                all_exact = False
                rep["near_tie"].append((s, "prune", float(ref["prune_gap"][s])))
            else:
                ge = emitted_paths(g, s)
                re_ = emitted_paths(ref, s)
                assert set(ge) == set(re_), f"seq {s}: pruned tree differs"
                for p, sc in ge.items():
                    assert abs(sc - re_[p]) <= tol
    check_prune_of_own_supertree(cfg, gst, g)
    keys = ("tokens", "parents", "depths", "pos_ids", "n_nodes")
    same = all(np.array_equal(g[k], ref[k]) for k in keys) and np.array_equal(
        g["mask"].view(np.uint64), ref["mask"])
    rep["bit_identical"] = bool(same)
    rep["arrays_exact"] = all_exact
    if all_exact:
        assert same, "emitted arrays differ although every oracle rank gap exceeds the tolerance"
        ok = np.isfinite(ref["scores"])
        assert np.max(np.abs(g["scores"][ok] - ref["scores"][ok]), initial=0.0) <= tol
    check_structure(cfg, g)
    return rep


def check_prune_of_own_supertree(cfg, gst, g):
    """The GPU's pruning and emission (a6-a8) must equal, bit for bit, the
    oracle's top-B pruning and emission of the GPU's own supertree: both rank
    the same float32 scores by (score desc, node id asc)."""
    pe = oracle.prune_emit(cfg, gst["st_tok"], gst["st_parent"],
                           np.asarray(gst["st_score"], np.float32).astype(np.float64), gst["st_count"])
    assert pe["rc"] == 0, "the GPU supertree is not prefix-closed under top-B"
    for k in ("tokens", "parents", "depths", "pos_ids", "n_nodes"):
        np.testing.assert_array_equal(g[k], pe[k], err_msg=f"emitted {k} != oracle pruning of the GPU supertree")
    np.testing.assert_array_equal(np.asarray(g["mask"]).view(np.uint64), pe["mask"],
                                  err_msg="emitted mask != oracle pruning of the GPU supertree")
    np.testing.assert_array_equal(np.asarray(g["scores"], np.float32).astype(np.float64), pe["scores"],
                                  err_msg="emitted scores != the GPU supertree's scores")


class TeacherForced:
    """The oracle evaluated on prefixes the GPU chose: the state of a prefix is
    the oracle's head applied token by token from h_0 (each prefix once), and
    its children are the oracle's corrected distribution at that state (over
    C_d when the candidate set is restricted)."""

    def __init__(self, cfg, x, s):
        self.cfg, self.x, self.s = cfg, x, s
        self.states = {(): np.asarray(x["h0"][s], np.float32).astype(np.float64)}

    def state(self, path):
        path = tuple(path)
        if path not in self.states:
            hp = self.state(path[:-1])
            self.states[path] = oracle.head(self.cfg, self.x["Wi"], self.x["Wo"], self.x["E"], hp, path[-1])
        return self.states[path]

    def children(self, path, kk):
        """(tokens[kk], log q~[kk]) of the kk best children by (log q~ desc, token asc)."""
        cfg = self.cfg
        row = self.x["Dlog"][self.s, len(path)]
        z = oracle.child_logits(cfg, self.x["E"], row, self.state(path))
        if int(getattr(cfg, "cand_k", 0)) > 0:
            cand = oracle.candidates(cfg, row)
            lq, _ = oracle.log_softmax(z[cand])
            idx = oracle.topk(lq, kk)
            return cand[idx], lq[idx]
        lq, _ = oracle.log_softmax(z)
        idx = oracle.topk(lq, kk)
        return idx.astype(np.int32), lq[idx]


def validate_depth_teacher_forced(cfg, tf, gst, s, dep, tol, known):
    """S_dep of the GPU against the oracle, teacher-forced on the GPU's own
    parents.  `known` maps GPU node ids of depth dep-1 (and above) to their
    oracle path scores and receives those of depth dep.  Checks: every kept
    child is one of its parent's k best children (the (k+1)-th only at a near
    tie of the k-th cut), its path score is within `tol` of the oracle's, the
    count is min(W, finite candidates), and the kept set is a top-W of the
    candidates up to 2 tol.  Returns the largest score difference."""
    W, k = cfg.W, cfg.k
    kk = min(k + 1, oracle.cand_count(cfg))
    gp = oracle.node_paths(gst["st_tok"], gst["st_parent"], gst["st_count"], s, W)
    npar = 1 if dep == 1 else int(gst["st_count"][s, dep - 2])
    cands = {}
    lists = {}
    for p in range(npar):
        path = () if dep == 1 else gp[(dep - 2) * W + p]
        ps = 0.0 if dep == 1 else known[(dep - 2) * W + p]
        tok, lq = tf.children(path, kk)
        lists[p] = lq
        for j in range(kk):
            cands[(p, int(tok[j]))] = (ps + float(lq[j]) + cfg.beta, j)
    gc = int(gst["st_count"][s, dep - 1])
    err = 0.0
    kept = set()
    for r in range(gc):
        t = int(gst["st_tok"][s, dep - 1, r])
        p = 0 if dep == 1 else int(gst["st_parent"][s, dep - 1, r])
        assert (p, t) in cands, f"seq {s} depth {dep}: kept child ({p},{t}) is not among the parent's top-(k+1)"
        sc, j = cands[(p, t)]
        if j == k:
            assert lists[p][k - 1] - lists[p][k] < 2 * tol, f"seq {s} depth {dep}: kept child outside the top-k"
        e = abs(float(gst["st_score"][s, dep - 1, r]) - sc)
        assert e <= tol, f"seq {s} depth {dep} rank {r}: path score off by {e}"
        err = max(err, e)
        kept.add((p, t))
        known[(dep - 1) * W + r] = sc
    finite = [c for c, (sc, j) in cands.items() if j < k and np.isfinite(sc)]
    assert gc == min(W, len(finite)), f"seq {s} depth {dep}: {gc} kept of {len(finite)} candidates"
    if gc:
        lo = min(cands[c][0] for c in kept)
        others = [sc for c, (sc, j) in cands.items() if c not in kept and j < k]
        if others:
            assert lo >= max(others) - 2 * tol, f"seq {s} depth {dep}: kept set is not a top-W"
    return err


def validate_frontier_teacher_forced(cfg, x, gst, s, dep, tol_step):
    """Checks S_dep of the GPU against the oracle given the GPU's own parents
    and their GPU scores: each kept child's score increment within tol_step of
    the oracle's log q~ + beta, and the kept set a valid top-W of the
    candidates (per-node top-k)."""
    known = {}
    if dep > 1:
        for r in range(int(gst["st_count"][s, dep - 2])):
            known[(dep - 2) * cfg.W + r] = float(gst["st_score"][s, dep - 2, r])
    validate_depth_teacher_forced(cfg, TeacherForced(cfg, x, s), gst, s, dep, tol_step, known)


# ----------------------------------------------- best-first constructions

def pop_order_paths(g, s):
    """[(token path, score)] of the emitted rows of sequence s, in row order."""
    out = []
    for i in range(int(g["n_nodes"][s])):
        path, j = [], i
        while j >= 0:
            path.append(int(g["tokens"][s, j]))
            j = int(g["parents"][s, j])
        out.append((tuple(reversed(path)), float(g["scores"][s, i])))
    return out


def check_pop_order_structure(cfg, g, s):
    """Rows in pop order: parents first, depth = parent's + 1, position ids,
    scores finite and non-increasing (exact: a child adds log q~ <= 0 and
    beta <= 0 to its parent's score), ancestor mask, padding."""
    n = int(g["n_nodes"][s])
    assert 0 <= n <= cfg.B
    par = g["parents"][s]
    for i in range(n):
        p = int(par[i])
        assert -1 <= p < i, (s, i, p)
        assert g["depths"][s, i] == (1 if p < 0 else g["depths"][s, p] + 1)
        assert 1 <= g["depths"][s, i] <= cfg.L
        assert g["pos_ids"][s, i] == cfg.pos_offset + g["depths"][s, i]
        assert np.isfinite(g["scores"][s, i])
        if i:
            assert g["scores"][s, i] <= g["scores"][s, i - 1], (s, i)
        anc, j = set(), i
        while j >= 0:
            anc.add(j)
            j = int(par[j])
        row = np.asarray(g["mask"][s, i]).view(np.uint64)
        assert {b for b in range(cfg.B) if (int(row[b // 64]) >> (b % 64)) & 1} == anc, (s, i)
    for i in range(n, cfg.B):
        assert g["tokens"][s, i] == -1 and g["parents"][s, i] == -2
        assert g["depths"][s, i] == 0 and g["pos_ids"][s, i] == -1
        assert np.isneginf(g["scores"][s, i]) and not np.any(g["mask"][s, i])


def compare_pop_order_tree(cfg, ref, g, tol, path_score):
    """A best-first tree of the GPU (rows in pop order) against the oracle's.
    path_score(s, path) is the oracle's score of any prefix, so a GPU path the
    oracle tree lacks is still checked.  Rules: the same node count; every
    GPU path scored within tol of the oracle's score of that path; the two
    node sets equal, or differing only across a near tie at the budget cut
    (each path only one side has scores within 2 tol of the cut); the rows in
    the oracle's order wherever the oracle's adjacent scores differ by >= tol;
    the structure of check_pop_order_structure."""
    rep = dict(near_tie=[], order_ties=0, bit_identical=None, max_score_err=0.0)
    for s in range(cfg.nseq):
        check_pop_order_structure(cfg, g, s)
        gp, rp = pop_order_paths(g, s), pop_order_paths(ref, s)
        assert len(gp) == len(rp) == int(ref["n_nodes"][s]), (s, len(gp), len(rp))
        rs = dict(rp)
        orc = {}
        for p, sc in gp:
            o = rs[p] if p in rs else path_score(s, p)
            orc[p] = o
            e = abs(sc - o)
            rep["max_score_err"] = max(rep["max_score_err"], e)
            assert e <= tol, f"seq {s} path {p}: score off by {e}"
        if set(orc) != set(rs):
            cut = rp[-1][1] if rp else np.inf
            for p in set(orc) - set(rs):
                assert orc[p] >= cut - 2 * tol, f"seq {s}: GPU path {p} below the oracle's cut"
            gcut = min(orc.values()) if orc else -np.inf
            for p in set(rs) - set(orc):
                assert rs[p] <= gcut + 2 * tol, f"seq {s}: oracle path {p} missing well above the GPU's cut"
            rep["near_tie"].append((s, float(cut)))
            continue
        gaps = [rp[i][1] - rp[i + 1][1] for i in range(len(rp) - 1)]
        if all(x >= tol for x in gaps):
            assert [p for p, _ in gp] == [p for p, _ in rp], f"seq {s}: pop order differs"
        else:
            rep["order_ties"] += 1
            for i in range(len(gp) - 1):
                assert orc[gp[i][0]] >= orc[gp[i + 1][0]] - 2 * tol
    keys = ("tokens", "parents", "depths", "pos_ids", "n_nodes")
    rep["bit_identical"] = bool(all(np.array_equal(g[k], ref[k]) for k in keys) and
                                np.array_equal(np.asarray(g["mask"]).view(np.uint64), ref["mask"]))
    return rep


def chain_path_score(cfg, x, chain):
    """path_score for Domino-chain + DDTree: a prefix scored with the oracle's
    distributions of the chain prefixes (`chain` [nseq][L] = the oracle's
    chain), sum_i log q~_i(u_i | chain_<i) + beta len."""
    rows = {}

    def row(s, i):
        if (s, i) not in rows:
            tf = TeacherForced(cfg, x, s)
            z = oracle.child_logits(cfg, x["E"], x["Dlog"][s, i], tf.state(tuple(int(t) for t in chain[s][:i])))
            rows[(s, i)] = oracle.log_softmax(z)[0]
        return rows[(s, i)]

    return lambda s, p: sum(float(row(s, i)[t]) for i, t in enumerate(p)) + cfg.beta * len(p)


def corrected_path_score(cfg, x):
    """path_score for the sequential search: the prefix's own corrected
    scores (Eq. 5 along the path, teacher-forced by the oracle)."""
    return lambda s, p: float(oracle.path_scores(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"][s], x["h0"][s],
                                                 np.array(p, np.int32))[-1])
