"""Pins of the tree-attention oracle (oracle/tree_attn.py) to facts that do
not come from the oracle itself (Sec. 3.3: a tree node attends to the
verified context and to its own root-to-node path).

* A branch of the tree is an ordinary causal sequence: for every node, the
  oracle equals causal attention over [context ; root-to-node path] computed
  by torch's scaled_dot_product_attention, with RoPE applied through the
  complex-exponential form (an independent formulation of the rotation).
* RoPE: equal to the complex form, identity at position 0, norm preserving,
  and q.k after rotation depends only on the position difference.
* Unit values give unit outputs (the weights are a probability vector);
  unused rows are zero.
* Relabelling the nodes permutes the outputs.
* A planted mistake (a sibling leaking into the path) fails the causal pin.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import tree_attn as ta
from workloads import random_tree


def rope_complex(x, pos, theta):
    """Rotation of the pairs (x[t], x[t + dh/2]) as complex numbers
    multiplied by exp(i * pos * theta^(-2t/dh))."""
    x = np.asarray(x, dtype=np.float64)
    dh = x.shape[-1]
    half = dh // 2
    z = x[..., :half] + 1j * x[..., half:]
    freq = np.exp(-np.log(theta) * (2.0 * np.arange(half) / dh))
    r = z * np.exp(1j * np.asarray(pos, dtype=np.float64)[..., None] * freq)
    return np.concatenate([r.real, r.imag], axis=-1)


def branch(parents, i):
    """Root-to-node path of node i written independently of the oracle: the
    ancestor set of i (i included) ordered by distance from the root."""
    anc = {int(i)}
    frontier = int(i)
    while int(parents[frontier]) >= 0:
        frontier = int(parents[frontier])
        anc.add(frontier)

    def dist(j):
        n = 0
        while int(parents[j]) >= 0:
            j = int(parents[j])
            n += 1
        return n
    return sorted(anc, key=dist)


def make_case(seed, nseq=2, B=12, C=5, Hq=4, Hkv=2, dh=8, L=4, W=4, fill=None, theta=1.0e4):
    g = np.random.Generator(np.random.PCG64(seed))
    q = g.standard_normal((nseq, B, Hq, dh))
    kt = g.standard_normal((nseq, B, Hkv, dh))
    vt = g.standard_normal((nseq, B, Hkv, dh))
    kc = g.standard_normal((nseq, C, Hkv, dh))
    vc = g.standard_normal((nseq, C, Hkv, dh))
    parents = np.empty((nseq, B), dtype=np.int32)
    depths = np.empty((nseq, B), dtype=np.int32)
    n_nodes = np.empty(nseq, dtype=np.int32)
    for s in range(nseq):
        n = B if fill is None else fill[s]
        parents[s], depths[s] = random_tree(B, L, W, n, g)
        n_nodes[s] = n
    return dict(q=q, k_tree=kt, v_tree=vt, k_ctx=kc, v_ctx=vc, parents=parents, depths=depths,
                n_nodes=n_nodes, theta=theta, scale=1.0 / np.sqrt(dh), C=C)


def causal_reference(case, pos_offset, path_fn):
    """Node i of sequence s = the last query of causal attention over the
    sequence [context ; path(i)] (torch SDPA, fp64)."""
    q, kt, vt, kc, vc = case["q"], case["k_tree"], case["v_tree"], case["k_ctx"], case["v_ctx"]
    nseq, B, Hq, dh = q.shape
    Hkv = kt.shape[2]
    G = Hq // Hkv
    out = np.zeros_like(q)
    for s in range(nseq):
        for i in range(int(case["n_nodes"][s])):
            path = path_fn(case["parents"][s], i)
            d = len(path)
            pos = pos_offset + np.arange(1, d + 1)
            keys = np.concatenate([kc[s], rope_complex(kt[s, path], pos[:, None], case["theta"])], axis=0)
            vals = np.concatenate([vc[s], vt[s, path]], axis=0)
            qs = rope_complex(q[s, path], pos[:, None], case["theta"])  # queries of the whole branch
            n_ctx = kc.shape[1]
            # queries only for the branch positions; the context rows are keys only
            Q = torch.from_numpy(qs.transpose(1, 0, 2))                       # [Hq, d, dh]
            K = torch.from_numpy(np.repeat(keys, G, axis=1).transpose(1, 0, 2))  # [Hq, n_ctx + d, dh]
            V = torch.from_numpy(np.repeat(vals, G, axis=1).transpose(1, 0, 2))
            allow = torch.ones((d, n_ctx + d), dtype=torch.bool)
            allow[:, n_ctx:] = torch.tril(torch.ones((d, d), dtype=torch.bool))
            o = torch.nn.functional.scaled_dot_product_attention(Q, K, V, attn_mask=allow,
                                                                 scale=float(case["scale"]))
            out[s, i] = o[:, -1].numpy()
    return out


def run_oracle(case, pos_offset):
    return ta.tree_attention(case["q"], case["k_tree"], case["v_tree"], case["k_ctx"], case["v_ctx"],
                             case["parents"], case["depths"], case["n_nodes"], pos_offset, case["theta"],
                             case["scale"])


@pytest.mark.parametrize("seed,kw", [(1, {}), (2, dict(C=0)), (3, dict(Hq=2, Hkv=2, W=2, L=6)),
                                     (4, dict(B=16, fill=[9, 16], C=3, L=5, W=5))])
def test_branch_is_a_causal_sequence(seed, kw):
    case = make_case(seed, **kw)
    off = case["C"] + 7
    got = run_oracle(case, off)
    ref = causal_reference(case, off, branch)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)
    for s in range(case["q"].shape[0]):
        assert np.all(got[s, int(case["n_nodes"][s]):] == 0.0)


def test_chain_tree_is_plain_causal_attention():
    case = make_case(5, B=6, L=6, W=1)
    assert list(case["parents"][0]) == [-1, 0, 1, 2, 3, 4]
    got = run_oracle(case, case["C"])
    ref = causal_reference(case, case["C"], branch)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)


def test_rope_matches_complex_form_and_is_relative():
    g = np.random.Generator(np.random.PCG64(11))
    x = g.standard_normal((5, 16))
    y = g.standard_normal((5, 16))
    pos = np.array([0, 1, 7, 300, 4099])
    for theta in (1.0e4, 1.0e6):
        np.testing.assert_allclose(ta.rope(x, pos, theta), rope_complex(x, pos, theta), atol=1e-10)
        np.testing.assert_allclose(ta.rope(x[0], 0, theta), x[0], atol=0)
        np.testing.assert_allclose(np.linalg.norm(ta.rope(x, pos, theta), axis=-1), np.linalg.norm(x, axis=-1),
                                   rtol=1e-13)
        for shift in (1, 13, 2048):
            a = np.sum(ta.rope(x, pos, theta) * ta.rope(y, pos[::-1], theta), axis=-1)
            b = np.sum(ta.rope(x, pos + shift, theta) * ta.rope(y, pos[::-1] + shift, theta), axis=-1)
            np.testing.assert_allclose(a, b, rtol=1e-9, atol=1e-9)


def test_unit_values_give_unit_outputs():
    case = make_case(6, B=10, fill=[7, 10], C=4)
    case["v_tree"] = np.ones_like(case["v_tree"])
    case["v_ctx"] = np.ones_like(case["v_ctx"])
    got = run_oracle(case, 4)
    for s, n in enumerate(case["n_nodes"]):
        np.testing.assert_allclose(got[s, :n], 1.0, atol=1e-14)
        assert np.all(got[s, n:] == 0.0)


def test_relabelling_permutes_outputs():
    case = make_case(7, nseq=1, B=10, C=3, L=4, W=4)
    n = 10
    g = np.random.Generator(np.random.PCG64(70))
    perm = g.permutation(n)          # old id i -> new id perm[i]
    inv = np.argsort(perm)
    p2 = dict(case)
    for key in ("q", "k_tree", "v_tree"):
        arr = case[key].copy()
        arr[0, perm] = case[key][0, np.arange(n)]
        p2[key] = arr
    par = np.full_like(case["parents"], -2)
    dep = np.zeros_like(case["depths"])
    for i in range(n):
        pi = case["parents"][0, i]
        par[0, perm[i]] = -1 if pi < 0 else perm[pi]
        dep[0, perm[i]] = case["depths"][0, i]
    p2["parents"], p2["depths"] = par, dep
    a = run_oracle(case, 3)
    b = run_oracle(p2, 3)
    np.testing.assert_allclose(b[0, perm], a[0], atol=1e-13)
    np.testing.assert_allclose(b[0], a[0, inv], atol=1e-13)


def test_planted_sibling_leak_fails_the_causal_pin(monkeypatch):
    case = make_case(8, nseq=1, B=12, C=2, L=3, W=6)

    def with_sibling(parents, i):
        path = branch(parents, i)
        sib = [j for j in range(len(parents)) if parents[j] == parents[i] and j != i and parents[j] != -2]
        return path[:-1] + sib[:1] + path[-1:] if sib else path

    monkeypatch.setattr(ta, "root_path", with_sibling)
    got = run_oracle(case, 2)
    ref = causal_reference(case, 2, branch)
    assert np.max(np.abs(got - ref)) > 1e-3
