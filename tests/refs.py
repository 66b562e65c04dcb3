"""Independent fp64 references used to pin the oracle.

These are built from library routines (torch.nn.Linear / SiLU / RMSNorm,
torch.log_softmax, torch.topk, Python's heapq) and from exhaustive
enumeration, never from the oracle's own code.
"""
from __future__ import annotations

import heapq
import itertools

import numpy as np
import torch
import torch.nn.functional as F

from workloads import bf16_bits_to_f32


def weights64(cfg, W):
    a = bf16_bits_to_f32(W) if cfg.wdtype == "bf16" else np.asarray(W, np.float32)
    return torch.from_numpy(a.astype(np.float64))


class TorchHead(torch.nn.Module):
    """Fallback correction head as a composition of library modules:
    RMSNorm(h_p + Linear_o(SiLU(Linear_i(cat[h_p, E[t]]))))."""

    def __init__(self, cfg, Wi, Wo, E):
        super().__init__()
        d = cfg.d
        self.E = weights64(cfg, E)
        self.lin_i = torch.nn.Linear(2 * d, d, bias=False, dtype=torch.float64)
        self.lin_o = torch.nn.Linear(d, d, bias=False, dtype=torch.float64)
        with torch.no_grad():
            self.lin_i.weight.copy_(weights64(cfg, Wi))
            self.lin_o.weight.copy_(weights64(cfg, Wo))
        self.act = torch.nn.SiLU()
        self.norm = torch.nn.RMSNorm(d, eps=cfg.rms_eps, elementwise_affine=False,
                                     dtype=torch.float64)

    @torch.no_grad()
    def forward(self, hp, tok):
        x = torch.cat([hp, self.E[tok]])
        return self.norm(hp + self.lin_o(self.act(self.lin_i(x))))


def child_logq(cfg, E64, dlog_row, h):
    """Clamped log-softmax of (Dlog + E h)/T' via torch (fp64)."""
    Tp = cfg.temperature if cfg.temperature > 0 else 1.0
    z = (torch.from_numpy(np.asarray(dlog_row, np.float64)) + E64 @ h) / Tp
    return torch.clamp(torch.log_softmax(z, dim=0), max=0.0)


def topK_candidates(dlog_row, K):
    """C = the K largest base logits, ties by token asc (numpy lexsort), as a
    sorted token array."""
    row = np.asarray(dlog_row, np.float64)
    order = np.lexsort((np.arange(row.size), -row))
    return np.sort(order[:K])


def child_logq_restricted(cfg, E64, dlog_row, h, cand):
    """Clamped log-softmax over the candidate subset only (torch fp64); a
    full-vocabulary tensor with -inf outside the subset."""
    Tp = cfg.temperature if cfg.temperature > 0 else 1.0
    idx = torch.from_numpy(np.asarray(cand, np.int64))
    z = (torch.from_numpy(np.asarray(dlog_row, np.float64))[idx] + E64[idx] @ h) / Tp
    out = torch.full((cfg.V,), float("-inf"), dtype=torch.float64)
    out[idx] = torch.clamp(torch.log_softmax(z, dim=0), max=0.0)
    return out


def all_path_scores(cfg, Wi, Wo, E, Dlog_seq, h0_seq, max_len):
    """Exhaustive enumeration: Eq. 5 score of every token path of length
    1..max_len, each recomputed from the root on its own (no shared state).
    With cfg.cand_k = K > 0 the paths run over the candidate sets C_i (the K
    largest base logits of position i) and q~ is renormalised over C_i."""
    head = TorchHead(cfg, Wi, Wo, E)
    E64 = head.E
    h0 = torch.from_numpy(np.asarray(h0_seq, np.float64))
    K = int(getattr(cfg, "cand_k", 0))
    cands = [topK_candidates(Dlog_seq[i], K) if K > 0 else np.arange(cfg.V) for i in range(max_len)]
    out = {}
    for n in range(1, max_len + 1):
        for path in itertools.product(*[[int(t) for t in cands[i]] for i in range(n)]):
            h = h0.clone()
            s = 0.0
            for i, t in enumerate(path):
                if K > 0:
                    lq = child_logq_restricted(cfg, E64, Dlog_seq[i], h, cands[i])
                else:
                    lq = child_logq(cfg, E64, Dlog_seq[i], h)
                s += float(lq[t]) + cfg.beta
                h = head(h, t)
            out[path] = s
    return out


def ddtree_topB(logq_rows, B):
    """DDTree best-first over path-independent marginals (Sec. 3.3): pop the
    best prefix, push its next sibling and its first child.  Marginal rows are
    log-probabilities; the prefix score is their sum (beta folded in by the
    caller).  Returns the popped token paths in pop order."""
    L = len(logq_rows)
    order = [np.argsort(-np.asarray(r), kind="stable") for r in logq_rows]
    srt = [np.asarray(r)[o] for r, o in zip(logq_rows, order)]
    # heap entries: (-score, ranks tuple)
    h = [(-float(srt[0][0]), (0,))]
    out = []
    while h and len(out) < B:
        negs, ranks = heapq.heappop(h)
        s = -negs
        path = tuple(int(order[i][r]) for i, r in enumerate(ranks))
        out.append((path, s))
        dep = len(ranks)
        last = ranks[-1]
        if last + 1 < len(srt[dep - 1]):
            sib = ranks[:-1] + (last + 1,)
            heapq.heappush(h, (-(s - float(srt[dep - 1][last]) + float(srt[dep - 1][last + 1])), sib))
        if dep < L:
            heapq.heappush(h, (-(s + float(srt[dep][0])), ranks + (0,)))
    return out
