"""Vocabulary-parallel scoring of one node, written out plainly (fp64).

TEST INFRASTRUCTURE ONLY (see the package docstring).  The hot path shards
naturally over sequences (replicas, no exchange).  Its one natural exchange
step, for a vocabulary split over G devices, is the merge of per-shard
partials of the corrected child distribution (Algorithm 1, scoring step):
each shard g holds z[v] for its rows and produces
    m_g = max_v z[v],  s_g = sum_v exp(z[v] - m_g),  its k best (z, v),
and any rank reconstructs logsumexp(z) = m + log(sum_g s_g exp(m_g - m))
(m = max_g m_g) and the global k best children as the k best of the union,
ordered by (z desc, token asc).  log q~ = min(z - logsumexp, 0).
"""
from __future__ import annotations

import numpy as np


def shard_partials(z_shard: np.ndarray, v0: int, k: int):
    """(m, s, top-k values, top-k tokens) of one vocabulary shard whose first
    token is v0."""
    z = np.asarray(z_shard, dtype=np.float64)
    m = float(np.max(z)) if z.size else -np.inf
    s = float(np.sum(np.exp(z - m))) if np.isfinite(m) else 0.0
    order = np.lexsort((np.arange(z.size), -z))[:k]
    return m, s, z[order], (order + v0).astype(np.int64)


def merge_partials(parts, k: int):
    """Merge [(m, s, vals, toks), ...] from all shards: (lse, top-k log q~, tokens)."""
    ms = np.array([p[0] for p in parts])
    m = float(np.max(ms))
    if not np.isfinite(m):
        return -np.inf, np.full(k, -np.inf), np.full(k, -1)
    ssum = float(sum(p[1] * np.exp(p[0] - m) for p in parts if np.isfinite(p[0])))
    lse = m + np.log(ssum)
    vals = np.concatenate([p[2] for p in parts])
    toks = np.concatenate([p[3] for p in parts])
    order = np.lexsort((toks, -vals))[:k]
    return lse, np.minimum(vals[order] - lse, 0.0), toks[order]
