"""The vocabulary-shard exchange of one node (oracle/shard.py), in one
process: the merged partials of G shards equal the unsharded log-softmax and
top-k of the oracle for G = 1, 2, 3, 7 (uneven shards, -inf logits, exact
ties across shard boundaries), and planted mistakes in copies of the module
fail that check."""
import importlib.util

import numpy as np
import pytest

import oracle
from oracle import shard
from workloads import Config

CFG = Config("vp", 1, 1003, 32, 2, 4, 7, 8, "f32", 0.7, 6)


def node_logits():
    g = np.random.Generator(np.random.PCG64(11))
    E = (g.standard_normal((CFG.V, CFG.d)) * 0.5).astype(np.float32)
    dlog = (g.standard_normal(CFG.V) * 2).astype(np.float32)
    dlog[[5, 900]] = -np.inf
    h = g.standard_normal(CFG.d)
    z = oracle.child_logits(CFG, E, dlog, h)
    # exact ties, more of them than k, straddling shard boundaries: the token
    # order decides both inside a shard and in the merge
    top = float(np.max(z[np.isfinite(z)]))
    z[[60, 61, 142, 143, 501, 502, 700, 858, 990]] = top + 1.0
    return z


def check(mod, z, G):
    parts = []
    for r in range(G):
        v0, v1 = r * CFG.V // G, (r + 1) * CFG.V // G
        parts.append(mod.shard_partials(z[v0:v1], v0, CFG.k))
    lse, lq, tk = mod.merge_partials(parts, CFG.k)
    ref_lq, ref_lse = oracle.log_softmax(z)
    ref_tk = oracle.topk(ref_lq, CFG.k)
    assert abs(lse - ref_lse) < 1e-12
    np.testing.assert_array_equal(tk, ref_tk)
    np.testing.assert_allclose(lq, ref_lq[ref_tk], atol=1e-12)


@pytest.mark.parametrize("G", [1, 2, 3, 7])
def test_sharded_merge_equals_unsharded(G):
    check(shard, node_logits(), G)


MUTANTS = [
    ("shard sums not rescaled to the common max",
     "ssum = float(sum(p[1] * np.exp(p[0] - m) for p in parts if np.isfinite(p[0])))",
     "ssum = float(sum(p[1] for p in parts if np.isfinite(p[0])))"),
    ("union ordered by token desc on ties",
     "order = np.lexsort((toks, -vals))[:k]",
     "order = np.lexsort((-toks, -vals))[:k]"),
    ("shard tokens not offset by the shard start",
     "return m, s, z[order], (order + v0).astype(np.int64)",
     "return m, s, z[order], order.astype(np.int64)"),
    ("shard top-k: ties by token desc",
     "order = np.lexsort((np.arange(z.size), -z))[:k]",
     "order = np.lexsort((-np.arange(z.size), -z))[:k]"),
]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_shard_mistake_fails(tmp_path, name, old, new):
    src = open(shard.__file__).read()
    assert src.count(old) == 1
    p = tmp_path / "shard_mut.py"
    p.write_text(src.replace(old, new))
    spec = importlib.util.spec_from_file_location("shard_mut", p)
    mut = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mut)
    z = node_logits()
    failed = 0
    for G in (1, 2, 3, 7):
        try:
            check(mut, z, G)
        except AssertionError:
            failed += 1
    assert failed, f"planted mistake passed: {name}"
