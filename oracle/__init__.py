"""fp64 CPU oracle for DARTree draft-tree construction (ctypes wrapper).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg may use this package; the product path never
imports it.  It shares no code with the CUDA path.

The arithmetic lives in ``dart_oracle.c`` (Algorithm 1, Eq. 5, Lemma 1 of the
paper, and the two constructions Table 2 compares DARTree with: Domino-chain +
DDTree and sequential correction with heap; each function citing its
passage).  This file only builds the C
library and marshals numpy arrays.  ``cfg`` arguments are any object with the
fields V, d, L, W, k, B, nseq, pos_offset, wdtype ("f32"/"bf16"), beta,
temperature, rms_eps.

Parity status: every function is pinned by the CPU tests in
``tests/test_oracle_pins.py`` (brute-force enumeration on tiny vocabularies,
library routines for the head and the softmax, the E = 0 closed form, the
greedy chain, Lemma 1 heap equality, prefix closure, monotonicity and mask
structure).  The paper prints no numeric tree, so no value is pinned to a
printed example.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dart_oracle.c")
_LIB = os.path.join(_HERE, "libdart_oracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP when available)."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    # a private temporary per process, renamed into place atomically, so
    # processes that build at the same time never load a half-written file
    tmp = f"{_LIB}.{os.getpid()}.tmp"
    base = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", _SRC, "-o", tmp, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB)
    return _LIB


class _Cfg(C.Structure):
    _fields_ = [("V", C.c_int), ("d", C.c_int), ("L", C.c_int), ("W", C.c_int),
                ("k", C.c_int), ("B", C.c_int), ("nseq", C.c_int),
                ("pos_offset", C.c_int), ("wdtype", C.c_int), ("cand_k", C.c_int),
                ("beta", C.c_double), ("temperature", C.c_double),
                ("rms_eps", C.c_double)]


def _cfg(cfg) -> _Cfg:
    return _Cfg(int(cfg.V), int(cfg.d), int(cfg.L), int(cfg.W), int(cfg.k), int(cfg.B),
                int(cfg.nseq), int(cfg.pos_offset), 0 if cfg.wdtype == "f32" else 1,
                int(getattr(cfg, "cand_k", 0)), float(cfg.beta), float(cfg.temperature),
                float(cfg.rms_eps))


def lib():
    global _lib
    if _lib is None:
        build()
        _lib = C.CDLL(_LIB)
        _lib.orc_num_threads.restype = C.c_int
        _lib.orc_log_softmax.restype = C.c_double
        _lib.orc_node_children.restype = C.c_double
        for f in ("orc_build_tree", "orc_prune_emit", "orc_heap_select", "orc_chain_ddtree", "orc_seq_heap"):
            getattr(_lib, f).restype = C.c_int
    return _lib


def _p(a):
    return a.ctypes.data_as(C.c_void_p)


def _w(cfg, a):
    want = np.float32 if cfg.wdtype == "f32" else np.uint16
    a = np.ascontiguousarray(a)
    if a.dtype != want:
        raise TypeError(f"weights must be {want.__name__} for wdtype={cfg.wdtype}")
    return a


def num_threads() -> int:
    return int(lib().orc_num_threads())


# ------------------------------------------------------------------ pieces

def head(cfg, Wi, Wo, E, hp, tok):
    """Fallback correction head on one state (fp64)."""
    hp = np.ascontiguousarray(hp, dtype=np.float64)
    out = np.empty(cfg.d, dtype=np.float64)
    Wi, Wo, E = _w(cfg, Wi), _w(cfg, Wo), _w(cfg, E)
    lib().orc_head(C.byref(_cfg(cfg)), _p(Wi), _p(Wo), _p(E), _p(hp), C.c_int(int(tok)), _p(out))
    return out


def child_logits(cfg, E, dlog_row, h):
    E = _w(cfg, E)
    dlog_row = np.ascontiguousarray(dlog_row, dtype=np.float32)
    h = np.ascontiguousarray(h, dtype=np.float64)
    z = np.empty(cfg.V, dtype=np.float64)
    lib().orc_child_logits(C.byref(_cfg(cfg)), _p(E), _p(dlog_row), _p(h), _p(z))
    return z


def log_softmax(z):
    z = np.ascontiguousarray(z, dtype=np.float64)
    out = np.empty_like(z)
    lse = lib().orc_log_softmax(_p(z), C.c_int(z.size), _p(out))
    return out, float(lse)


def cand_count(cfg) -> int:
    """Entries scored per node: the candidate-set size K, or V (full vocabulary)."""
    K = int(getattr(cfg, "cand_k", 0))
    return K if K > 0 else int(cfg.V)


def candidates(cfg, dlog_row):
    """C_d = TopK(L_d^base, K) of Algorithm 1, sorted by token id."""
    dlog_row = np.ascontiguousarray(dlog_row, dtype=np.float32)
    out = np.empty(int(cfg.cand_k), dtype=np.int32)
    lib().orc_candidates(C.byref(_cfg(cfg)), _p(dlog_row), _p(out))
    return out


def topk(x, kk):
    x = np.ascontiguousarray(x, dtype=np.float64)
    idx = np.empty(kk, dtype=np.int32)
    lib().orc_topk(_p(x), C.c_int(x.size), C.c_int(kk), _p(idx))
    return idx


# ------------------------------------------------------------- Algorithm 1

def build_tree(cfg, Wi, Wo, E, Dlog, h0):
    """Algorithm 1 + pruning + emission for every sequence.  Returns a dict
    of numpy arrays (see ``orc_build_tree`` in dart_oracle.c)."""
    Wi, Wo, E = _w(cfg, Wi), _w(cfg, Wo), _w(cfg, E)
    Dlog = np.ascontiguousarray(Dlog, dtype=np.float32)
    h0 = np.ascontiguousarray(h0, dtype=np.float32)
    ns, L, W, B = cfg.nseq, cfg.L, cfg.W, cfg.B
    kx = min(cfg.k + 1, cand_count(cfg))
    nw = (B + 63) // 64
    r = dict(
        st_tok=np.empty((ns, L, W), np.int32), st_parent=np.empty((ns, L, W), np.int32),
        st_score=np.empty((ns, L, W), np.float64), st_count=np.empty((ns, L), np.int32),
        nd_lse=np.empty((ns, L, W), np.float64), nd_tok=np.empty((ns, L, W, kx), np.int32),
        nd_logq=np.empty((ns, L, W, kx), np.float64),
        fr_score=np.empty((ns, L, W + 1), np.float64),
        tokens=np.empty((ns, B), np.int32), parents=np.empty((ns, B), np.int32),
        depths=np.empty((ns, B), np.int32), pos_ids=np.empty((ns, B), np.int32),
        scores=np.empty((ns, B), np.float64), n_nodes=np.empty(ns, np.int32),
        mask=np.empty((ns, B, nw), np.uint64), prune_gap=np.empty(ns, np.float64))
    rc = lib().orc_build_tree(
        C.byref(_cfg(cfg)), _p(Wi), _p(Wo), _p(E), _p(Dlog), _p(h0),
        _p(r["st_tok"]), _p(r["st_parent"]), _p(r["st_score"]), _p(r["st_count"]),
        _p(r["nd_lse"]), _p(r["nd_tok"]), _p(r["nd_logq"]), _p(r["fr_score"]),
        _p(r["tokens"]), _p(r["parents"]), _p(r["depths"]), _p(r["pos_ids"]),
        _p(r["scores"]), _p(r["n_nodes"]), _p(r["mask"]), _p(r["prune_gap"]))
    if rc != 0:
        raise RuntimeError("oracle: a selected node has an unselected parent")
    return r


def prune_emit(cfg, st_tok, st_parent, st_score, st_count):
    """Top-B pruning and emission of a given supertree (scores in fp64)."""
    ns, B = cfg.nseq, cfg.B
    nw = (B + 63) // 64
    st_tok = np.ascontiguousarray(st_tok, np.int32)
    st_parent = np.ascontiguousarray(st_parent, np.int32)
    st_score = np.ascontiguousarray(st_score, np.float64)
    st_count = np.ascontiguousarray(st_count, np.int32)
    r = dict(tokens=np.empty((ns, B), np.int32), parents=np.empty((ns, B), np.int32),
             depths=np.empty((ns, B), np.int32), pos_ids=np.empty((ns, B), np.int32),
             scores=np.empty((ns, B), np.float64), n_nodes=np.empty(ns, np.int32),
             mask=np.empty((ns, B, nw), np.uint64), prune_gap=np.empty(ns, np.float64))
    rc = lib().orc_prune_emit(C.byref(_cfg(cfg)), _p(st_tok), _p(st_parent), _p(st_score),
                              _p(st_count), _p(r["tokens"]), _p(r["parents"]),
                              _p(r["depths"]), _p(r["pos_ids"]), _p(r["scores"]),
                              _p(r["n_nodes"]), _p(r["mask"]), _p(r["prune_gap"]))
    r["rc"] = rc
    return r


def heap_select(cfg, st_parent, st_score, st_count, s=0):
    """Best-first heap selection (Lemma 1); node ids in pop order."""
    st_parent = np.ascontiguousarray(st_parent, np.int32)
    st_score = np.ascontiguousarray(st_score, np.float64)
    st_count = np.ascontiguousarray(st_count, np.int32)
    out = np.empty(cfg.L * cfg.W, np.int32)
    n = lib().orc_heap_select(C.byref(_cfg(cfg)), _p(st_parent), _p(st_score),
                              _p(st_count), C.c_int(s), _p(out))
    return out[:n].copy()


# ------------------------------------------- heap-based constructions

def _tree_out(cfg):
    ns, B = cfg.nseq, cfg.B
    nw = (B + 63) // 64
    return dict(tokens=np.empty((ns, B), np.int32), parents=np.empty((ns, B), np.int32),
                depths=np.empty((ns, B), np.int32), pos_ids=np.empty((ns, B), np.int32),
                scores=np.empty((ns, B), np.float64), n_nodes=np.empty(ns, np.int32),
                mask=np.empty((ns, B, nw), np.uint64))


def chain_ddtree(cfg, Wi, Wo, E, Dlog, h0):
    """Domino-chain + DDTree (see ``orc_chain_ddtree``): the emitted tree in
    pop order plus the chain (chain_tok, chain_lse [nseq][L])."""
    Wi, Wo, E = _w(cfg, Wi), _w(cfg, Wo), _w(cfg, E)
    Dlog = np.ascontiguousarray(Dlog, dtype=np.float32)
    h0 = np.ascontiguousarray(h0, dtype=np.float32)
    r = _tree_out(cfg)
    r["chain_tok"] = np.empty((cfg.nseq, cfg.L), np.int32)
    r["chain_lse"] = np.empty((cfg.nseq, cfg.L), np.float64)
    lib().orc_chain_ddtree(C.byref(_cfg(cfg)), _p(Wi), _p(Wo), _p(E), _p(Dlog), _p(h0), _p(r["chain_tok"]),
                           _p(r["chain_lse"]), _p(r["tokens"]), _p(r["parents"]), _p(r["depths"]),
                           _p(r["pos_ids"]), _p(r["scores"]), _p(r["n_nodes"]), _p(r["mask"]))
    return r


def seq_heap(cfg, Wi, Wo, E, Dlog, h0):
    """Sequential correction with heap (see ``orc_seq_heap``): the emitted
    tree in pop order plus expansions [nseq] (children distributions computed)."""
    Wi, Wo, E = _w(cfg, Wi), _w(cfg, Wo), _w(cfg, E)
    Dlog = np.ascontiguousarray(Dlog, dtype=np.float32)
    h0 = np.ascontiguousarray(h0, dtype=np.float32)
    r = _tree_out(cfg)
    r["expansions"] = np.empty(cfg.nseq, np.int32)
    lib().orc_seq_heap(C.byref(_cfg(cfg)), _p(Wi), _p(Wo), _p(E), _p(Dlog), _p(h0), _p(r["tokens"]),
                       _p(r["parents"]), _p(r["depths"]), _p(r["pos_ids"]), _p(r["scores"]), _p(r["n_nodes"]),
                       _p(r["mask"]), _p(r["expansions"]))
    return r


# ------------------------------------------------- teacher-forced helpers

def path_state(cfg, Wi, Wo, E, h0_seq, path):
    Wi, Wo, E = _w(cfg, Wi), _w(cfg, Wo), _w(cfg, E)
    h0_seq = np.ascontiguousarray(h0_seq, np.float32)
    path = np.ascontiguousarray(path, np.int32)
    out = np.empty(cfg.d, np.float64)
    lib().orc_path_state(C.byref(_cfg(cfg)), _p(Wi), _p(Wo), _p(E), _p(h0_seq), _p(path),
                         C.c_int(path.size), _p(out))
    return out


def node_children(cfg, Wi, Wo, E, Dlog_seq, h0_seq, path, kk, want_all=False):
    """(tokens[kk], logq[kk], lse, logq_all or None) of the prefix ``path``."""
    Wi, Wo, E = _w(cfg, Wi), _w(cfg, Wo), _w(cfg, E)
    Dlog_seq = np.ascontiguousarray(Dlog_seq, np.float32)
    h0_seq = np.ascontiguousarray(h0_seq, np.float32)
    path = np.ascontiguousarray(path, np.int32)
    tok = np.empty(max(kk, 1), np.int32)
    lq = np.empty(max(kk, 1), np.float64)
    allq = np.empty(cfg.V, np.float64) if want_all else None
    lse = lib().orc_node_children(C.byref(_cfg(cfg)), _p(Wi), _p(Wo), _p(E), _p(Dlog_seq),
                                  _p(h0_seq), _p(path), C.c_int(path.size), C.c_int(kk),
                                  _p(tok), _p(lq), _p(allq) if want_all else None)
    return tok[:kk], lq[:kk], float(lse), allq


def path_scores(cfg, Wi, Wo, E, Dlog_seq, h0_seq, path):
    Wi, Wo, E = _w(cfg, Wi), _w(cfg, Wo), _w(cfg, E)
    Dlog_seq = np.ascontiguousarray(Dlog_seq, np.float32)
    h0_seq = np.ascontiguousarray(h0_seq, np.float32)
    path = np.ascontiguousarray(path, np.int32)
    out = np.empty(path.size, np.float64)
    lib().orc_path_scores(C.byref(_cfg(cfg)), _p(Wi), _p(Wo), _p(E), _p(Dlog_seq), _p(h0_seq),
                          _p(path), C.c_int(path.size), _p(out))
    return out


# ------------------------------------------------------- tree utilities

def node_paths(st_tok, st_parent, st_count, s, W):
    """Token path of every supertree node of sequence s, keyed by node id
    (id = (depth-1)*W + rank)."""
    paths = {}
    L = st_tok.shape[1]
    for dep in range(1, L + 1):
        for r in range(int(st_count[s, dep - 1])):
            tok = int(st_tok[s, dep - 1, r])
            if dep == 1:
                paths[r] = (tok,)
            else:
                pid = (dep - 2) * W + int(st_parent[s, dep - 1, r])
                paths[(dep - 1) * W + r] = paths[pid] + (tok,)
    return paths
