"""fp64 CPU oracle of the tree-attention verification consumer.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg may use this module; the product path never
imports it.  It shares no code with the CUDA path.

What it computes (Sec. 3.3 of the paper, "Tree Verification and DDTree"):
the draft tree is flattened and verified in one target forward pass in
which every tree node attends to the verified context and to the tokens on
its own root-to-node path.  The target model is not available, so the
oracle evaluates one attention layer of that pass on given Q / K / V:

    out[s, i, h] = softmax_j(scale * q_i . k_j) v_j
    j over the C context keys of sequence s and the tree nodes on the path
    from the root to i (i itself included),

with q_i and the tree keys rotated by RoPE (rotate-half form) at the
node's position pos_offset + depth(i); the context keys are a KV cache and
arrive rotated.  The path is found by walking parent indices, not from a
bitmask, and positions come from depths, so nothing here depends on the
emitted mask or position ids that the GPU consumes.

Parity status: pinned by ``tests/test_attn_oracle_pins.py`` (a branch is
an ordinary causal sequence: each node equals causal attention over
context + its path computed with torch's scaled_dot_product_attention;
RoPE equals the complex-exponential form and depends only on relative
positions; unit values give unit outputs; relabelling the nodes permutes
the outputs; a planted sibling leak fails).
"""
from __future__ import annotations

import numpy as np


def rope(x: np.ndarray, pos, theta: float) -> np.ndarray:
    """Rotate-half RoPE of x [..., dh] at integer position(s) pos (fp64).

    For t < dh/2, with inv_freq_t = theta^(-2t/dh) and a = pos * inv_freq_t:
    y[t] = x[t] cos a - x[t + dh/2] sin a,  y[t + dh/2] = x[t + dh/2] cos a + x[t] sin a.
    """
    x = np.asarray(x, dtype=np.float64)
    dh = x.shape[-1]
    half = dh // 2
    inv_freq = float(theta) ** (-2.0 * np.arange(half, dtype=np.float64) / dh)
    ang = np.asarray(pos, dtype=np.float64)[..., None] * inv_freq
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def root_path(parents: np.ndarray, i: int) -> list:
    """Tree indices on the path from the root to node i, i included
    (parent -1 = child of the root)."""
    path = []
    j = int(i)
    while j >= 0:
        path.append(j)
        j = int(parents[j])
    return path[::-1]


def tree_attention(q, k_tree, v_tree, k_ctx, v_ctx, parents, depths, n_nodes, pos_offset: int,
                   rope_theta: float, scale: float, rows=None) -> np.ndarray:
    """One tree-attention layer (see module docstring).

    q [nseq, B, Hq, dh]; k_tree, v_tree [nseq, B, Hkv, dh]; k_ctx, v_ctx
    [nseq, C, Hkv, dh] (k_ctx rotated); parents, depths [nseq, B];
    n_nodes [nseq].  Returns out [nseq, B, Hq, dh] float64 with zero rows
    for i >= n_nodes.  `rows`, a list of (s, i), restricts the evaluation to
    those tree rows (the others stay zero).
    """
    q = np.asarray(q, dtype=np.float64)
    k_tree = np.asarray(k_tree, dtype=np.float64)
    v_tree = np.asarray(v_tree, dtype=np.float64)
    k_ctx = np.asarray(k_ctx, dtype=np.float64)
    v_ctx = np.asarray(v_ctx, dtype=np.float64)
    nseq, B, Hq, dh = q.shape
    Hkv = k_tree.shape[2]
    G = Hq // Hkv
    out = np.zeros((nseq, B, Hq, dh), dtype=np.float64)
    want = None if rows is None else {(int(s), int(i)) for s, i in rows}
    for s in range(nseq):
        n = int(n_nodes[s])
        pos = pos_offset + np.asarray(depths[s], dtype=np.int64)
        for i in range(n):
            if want is not None and (s, i) not in want:
                continue
            path = root_path(parents[s], i)
            for h in range(Hq):
                g = h // G
                qi = rope(q[s, i, h], pos[i], rope_theta)
                kt = rope(k_tree[s, path, g], pos[path], rope_theta)
                keys = np.concatenate([k_ctx[s, :, g], kt], axis=0)
                vals = np.concatenate([v_ctx[s, :, g], v_tree[s, path, g]], axis=0)
                logits = scale * (keys @ qi)
                w = np.exp(logits - logits.max())
                out[s, i, h] = (w @ vals) / w.sum()
    return out
