"""Seeded synthetic workloads for DARTree draft-tree construction.

This module only draws random inputs.  It holds none of the method's
arithmetic, so both the CPU oracle and the CUDA path can consume exactly the
same bits without sharing any code that computes the tree.

The shapes follow the paper's experimental setting (Qwen3-4B / Qwen3-8B
vocabulary and hidden sizes, a 16-token draft block, the width / budget
ranges of the hyper-parameter study, Sec. 5.1 and Sec. 5.3).  The paper's
drafter, correction head and datasets are not available, so:

* the correction head is the fallback head
  h_c = RMSNorm(h_p + W_o . SiLU(W_i . [h_p ; E[t_c]])) with
  W_i ~ N(0, 1/(2d)), W_o ~ N(0, 1/d), E ~ N(0, 0.02^2) (the LM head is tied to E);
* drafter marginal logits are 3 . N(0,1) per position plus a spike at one
  seeded random token per position (+8 for the fp32 toy, +6 at positions 0-7
  and +3 at positions 8-15 for the bf16 shapes, mimicking decaying drafter
  confidence along the block);
* the anchor state h_0 ~ N(0,1).

bf16 weights are drawn in fp32 and rounded to nearest-even bf16; they are
returned as uint16 bit patterns.  Every array is generated from numpy's PCG64
with a fixed seed per (config, tensor, row chunk), so the values do not depend
on the number of threads used to draw them or on the machine.
"""
from __future__ import annotations

import concurrent.futures as _cf
import dataclasses
import os

import numpy as np

BETA_DEFAULT = -0.2      # depth bonus of the pruned variant (Sec. 5.1)
RMS_EPS = 1e-6


@dataclasses.dataclass(frozen=True)
class Config:
    name: str
    nseq: int
    V: int
    d: int
    L: int
    W: int
    k: int
    B: int
    wdtype: str            # "f32" or "bf16"
    temperature: float     # 0 = greedy scoring (no scaling)
    seed: int
    beta: float = BETA_DEFAULT
    rms_eps: float = RMS_EPS
    pos_offset: int = 0
    spike_early: float = 6.0   # positions 0..7
    spike_late: float = 3.0    # positions 8..
    cand_k: int = 0            # K of Algorithm 1 (candidate-set size); 0 = full vocabulary
    # library tuning switches (dart_config; 0 = the library's choice, 1 = on,
    # 2 = off): they change neither the inputs nor the tree
    head_split: int = 0
    head_split_stream: int = 0
    lmhead_ctas_per_sm: int = 0
    weights_tiled: int = 0
    head_weights_tiled: int = 0
    variants: int = 0          # extra constructions prepared by the handle (bit set)
    fused_round: int = 0       # fp32: the whole round as one cooperative kernel (where possible)
    topk_bound: int = 0        # bf16: a starting bound of each node's top-k filter before each LM-head

    def replace(self, **kw) -> "Config":
        return dataclasses.replace(self, **kw)

    @property
    def bpe(self) -> int:
        return 4 if self.wdtype == "f32" else 2

    def caps(self):
        """Maximum frontier size |S_d| for d = 0..L (|S_0| = 1)."""
        c = [1]
        for _ in range(self.L):
            c.append(min(self.W, c[-1] * self.k))
        return c

    def expansions_per_round(self) -> int:
        """Nodes whose children are scored in one round: sum_d nseq*|S_{d-1}|."""
        c = self.caps()
        return self.nseq * sum(c[:self.L])

    def lmhead_bytes_per_depth(self) -> int:
        """Algorithmic HBM bytes of one LM-head pass: E once + the drafter row."""
        return self.V * self.d * self.bpe + self.nseq * self.V * 4


# Base seed 2608 + index, in the order the workloads are listed.
TOY = Config("toy", 1, 4096, 256, 4, 4, 4, 16, "f32", 0.0, 2608,
             spike_early=8.0, spike_late=8.0)
Q4B = Config("qwen3-4b", 1, 151936, 2560, 16, 8, 8, 64, "bf16", 0.0, 2609)
Q8B = Config("qwen3-8b", 1, 151936, 4096, 16, 16, 16, 256, "bf16", 1.0, 2610)
SWEEP_BASE = Config("sweep", 1, 151936, 2560, 16, 8, 8, 32, "bf16", 0.0, 2611)
BATCHED = Config("batched", 8, 151936, 4096, 16, 32, 32, 512, "bf16", 1.0, 2612)


def sweep_configs():
    out = []
    for W in (8, 16, 32, 64):
        for B in (32, 128, 512, 1024):
            out.append(SWEEP_BASE.replace(name=f"sweep-W{W}-B{B}", W=W, k=W, B=B))
    return out


# The same shapes and inputs with Algorithm 1's candidate restriction at the
# paper's default K = 64 (Sec. 5.1).
RESTRICTED = [Q8B.replace(name="qwen3-8b-k64", cand_k=64), Q4B.replace(name="qwen3-4b-k64", cand_k=64),
              BATCHED.replace(name="batched-k64", cand_k=64)]

NAMED = {c.name: c for c in (TOY, Q4B, Q8B, BATCHED)}
for _c in sweep_configs() + RESTRICTED:
    NAMED[_c.name] = _c


# --------------------------------------------------------------------------
# bit helpers (no method arithmetic: only storage conversions)

def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (nearest even); returns uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    out = np.empty(u.shape, dtype=np.uint16)
    flat_u = u.reshape(-1)
    flat_o = out.reshape(-1)
    step = 1 << 24
    for s in range(0, flat_u.size, step):
        c = flat_u[s:s + step]
        r = (c >> np.uint32(16)) & np.uint32(1)
        flat_o[s:s + step] = ((c + np.uint32(0x7FFF) + r) >> np.uint32(16)).astype(np.uint16)
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# --------------------------------------------------------------------------
# generators

_ROWS_PER_CHUNK = 4096


def _normal_rows(seed: int, tag: int, rows: int, cols: int, std: float,
                 threads: int | None = None) -> np.ndarray:
    """rows x cols float32 N(0, std^2); chunk c of rows uses PCG64([seed, tag, c])."""
    out = np.empty((rows, cols), dtype=np.float32)
    nchunk = (rows + _ROWS_PER_CHUNK - 1) // _ROWS_PER_CHUNK

    def work(c):
        r0 = c * _ROWS_PER_CHUNK
        r1 = min(rows, r0 + _ROWS_PER_CHUNK)
        g = np.random.Generator(np.random.PCG64([seed, tag, c]))
        blk = out[r0:r1]
        g.standard_normal(out=blk, dtype=np.float32)
        blk *= np.float32(std)

    if threads is None:
        threads = min(32, os.cpu_count() or 1)
    if nchunk == 1 or threads <= 1:
        for c in range(nchunk):
            work(c)
    else:
        with _cf.ThreadPoolExecutor(threads) as ex:
            list(ex.map(work, range(nchunk)))
    return out


def make_weights(cfg: Config, zero_E: bool = False):
    """Fallback-head weights: W_i [d,2d], W_o [d,d], E [V,d] (tied LM head).

    Returned as float32 arrays for fp32 configs, uint16 bf16 bit patterns for
    bf16 configs.
    """
    d = cfg.d
    Wi = _normal_rows(cfg.seed, 1, d, 2 * d, (1.0 / (2 * d)) ** 0.5)
    Wo = _normal_rows(cfg.seed, 2, d, d, (1.0 / d) ** 0.5)
    if zero_E:
        E = np.zeros((cfg.V, d), dtype=np.float32)
    else:
        E = _normal_rows(cfg.seed, 3, cfg.V, d, 0.02)
    if cfg.wdtype == "bf16":
        return f32_to_bf16_bits(Wi), f32_to_bf16_bits(Wo), f32_to_bf16_bits(E)
    return Wi, Wo, E


def make_sequences(cfg: Config, rank: int = 0):
    """Per-sequence drafter logits Dlog [nseq, L, V] and anchors h0 [nseq, d].

    `rank` selects a disjoint block of sequences (seed cfg.seed*1000 +
    rank*nseq + s), so replicas on different GPUs build different trees."""
    Dlog = np.empty((cfg.nseq, cfg.L, cfg.V), dtype=np.float32)
    h0 = np.empty((cfg.nseq, cfg.d), dtype=np.float32)
    for s in range(cfg.nseq):
        g = np.random.Generator(np.random.PCG64(cfg.seed * 1000 + rank * cfg.nseq + s))
        h0[s] = g.standard_normal(cfg.d, dtype=np.float32)
        noise = g.standard_normal((cfg.L, cfg.V), dtype=np.float32)
        Dlog[s] = noise * np.float32(3.0)
        spikes = g.integers(0, cfg.V, size=cfg.L)
        for i in range(cfg.L):
            amp = cfg.spike_early if i < 8 else cfg.spike_late
            Dlog[s, i, spikes[i]] += np.float32(amp)
    return Dlog, h0


def make_inputs(cfg: Config, zero_E: bool = False, rank: int = 0):
    Wi, Wo, E = make_weights(cfg, zero_E=zero_E)
    Dlog, h0 = make_sequences(cfg, rank=rank)
    return dict(Wi=Wi, Wo=Wo, E=E, Dlog=Dlog, h0=h0)


# --------------------------------------------------------------------------
# tree-attention verification inputs (Sec. 3.3: one target forward pass over
# the flattened tree).  The target model is not available: one attention
# layer with Qwen3-4B/8B head geometry (32 query heads, 8 key/value heads,
# head dim 128, RoPE base 1e6) on N(0,1) queries, keys and values, and a
# verified context of C tokens whose keys are a (rotated) KV cache.  The
# tree is a random prefix tree shaped like DARTree's supertree: depth levels
# 1..L of at most W nodes, each node's parent drawn uniformly from the level
# above, ids in level order (a topological order, as emitted).

@dataclasses.dataclass(frozen=True)
class AttnConfig:
    name: str
    nseq: int
    B: int          # tree rows per sequence (the budget)
    C: int          # context keys per sequence
    L: int          # maximum depth
    W: int          # maximum nodes per depth level
    seed: int
    Hq: int = 32
    Hkv: int = 8
    dh: int = 128
    rope_theta: float = 1.0e6
    pos_offset: int = -1     # < 0: the context length C, so depth d sits at position C + d
    fill: float = 1.0        # fraction of the B rows used by the tree (n_nodes)

    def replace(self, **kw) -> "AttnConfig":
        return dataclasses.replace(self, **kw)

    @property
    def scale(self) -> float:
        return 1.0 / float(self.dh) ** 0.5

    @property
    def offset(self) -> int:
        return self.C if self.pos_offset < 0 else self.pos_offset


ATTN_Q8B = AttnConfig("verify-qwen3-8b", 1, 256, 2048, 16, 16, 2620)
ATTN_Q4B = AttnConfig("verify-qwen3-4b", 1, 64, 2048, 16, 8, 2621)
ATTN_BATCHED = AttnConfig("verify-batched", 8, 512, 2048, 16, 32, 2622)
ATTN_NAMED = {c.name: c for c in (ATTN_Q8B, ATTN_Q4B, ATTN_BATCHED)}


def random_tree(B: int, L: int, W: int, n: int, g: np.random.Generator):
    """parents [B] (-1: child of the root, -2: unused row) and depths [B]
    (0 for unused rows) of a random n-node prefix tree in level order."""
    parents = np.full(B, -2, dtype=np.int32)
    depths = np.zeros(B, dtype=np.int32)
    prev = [-1]
    i = 0
    d = 1
    while i < n and d <= L:
        cnt = min(W, n - i)
        if d == L:
            cnt = n - i  # the last level takes what is left
        picks = np.sort(g.integers(0, len(prev), size=cnt))
        level = []
        for pk in picks:
            parents[i] = prev[pk]
            depths[i] = d
            level.append(i)
            i += 1
        prev = level
        d += 1
    return parents, depths


def make_attn_inputs(cfg: AttnConfig):
    """Q, K, V of the tree rows and the context (uint16 bf16 bit patterns,
    N(0,1) before rounding) and the tree structure (parents, depths, n_nodes)."""
    g = np.random.Generator(np.random.PCG64([cfg.seed, 7]))

    def bf(*shape):
        return f32_to_bf16_bits(g.standard_normal(shape, dtype=np.float32))

    q = bf(cfg.nseq, cfg.B, cfg.Hq, cfg.dh)
    k_tree = bf(cfg.nseq, cfg.B, cfg.Hkv, cfg.dh)
    v_tree = bf(cfg.nseq, cfg.B, cfg.Hkv, cfg.dh)
    k_ctx = bf(cfg.nseq, cfg.C, cfg.Hkv, cfg.dh)
    v_ctx = bf(cfg.nseq, cfg.C, cfg.Hkv, cfg.dh)
    parents = np.empty((cfg.nseq, cfg.B), dtype=np.int32)
    depths = np.empty((cfg.nseq, cfg.B), dtype=np.int32)
    n_nodes = np.empty(cfg.nseq, dtype=np.int32)
    for s in range(cfg.nseq):
        n = max(0, min(cfg.B, int(round(cfg.fill * cfg.B)) - (s % 3 if cfg.fill < 1.0 else 0)))
        parents[s], depths[s] = random_tree(cfg.B, cfg.L, cfg.W, n, g)
        n_nodes[s] = int((parents[s] != -2).sum())
    return dict(q=q, k_tree=k_tree, v_tree=v_tree, k_ctx=k_ctx, v_ctx=v_ctx, parents=parents,
                depths=depths, n_nodes=n_nodes)
