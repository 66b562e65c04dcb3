"""Thin ctypes binding of the DARTree C ABI (include/dart.h).

Argument marshalling only: every step of the construction runs in the CUDA
kernels of ``libdart.so``.  Functions keep the C names; tensors are passed by
``data_ptr()`` and streams by their CUDA handle.  There is no fallback: if the
library is missing, the first call into it raises.
"""
from __future__ import annotations

import ctypes as C
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libdart.so")

DART_OK = 0
DART_ERR_INVALID = -1
DART_ERR_CUDA = -2
DART_ERR_NOMEM = -3
DART_ERR_TIMEOUT = -4
DART_ERR_STATE = -5
DART_ERR_UNSUPPORTED = -6
DART_ERR_BOUNDS = -7
DART_F32 = 0
DART_BF16 = 1
DART_AUTO, DART_ON, DART_OFF = 0, 1, 2
DART_VARIANT_CHAIN_DDTREE = 1
DART_VARIANT_SEQ_HEAP = 2


class DartConfig(C.Structure):
    _fields_ = [("V", C.c_int), ("d", C.c_int), ("L", C.c_int), ("W", C.c_int), ("k", C.c_int),
                ("B", C.c_int), ("nseq", C.c_int), ("beta", C.c_float),
                ("temperature", C.c_float), ("rms_eps", C.c_float), ("pos_offset", C.c_int),
                ("cand_k", C.c_int), ("head_split", C.c_int), ("head_split_stream", C.c_int),
                ("lmhead_ctas_per_sm", C.c_int), ("weights_tiled", C.c_int), ("head_weights_tiled", C.c_int),
                ("variants", C.c_int), ("fused_round", C.c_int), ("topk_bound", C.c_int)]


class DartTreeOut(C.Structure):
    _fields_ = [("tokens", C.c_void_p), ("parents", C.c_void_p), ("depths", C.c_void_p),
                ("pos_ids", C.c_void_p), ("scores", C.c_void_p), ("n_nodes", C.c_void_p),
                ("mask", C.c_void_p)]


class DartAttnConfig(C.Structure):
    _fields_ = [("nseq", C.c_int), ("B", C.c_int), ("C", C.c_int), ("Hq", C.c_int), ("Hkv", C.c_int),
                ("dh", C.c_int), ("rope_theta", C.c_float), ("scale", C.c_float)]


class DartError(RuntimeError):
    def __init__(self, code, what):
        super().__init__(f"{what}: {status_string(code)} ({code})")
        self.code = code


_lib = None
_empty = torch.empty


def set_output_allocator(fn=None):
    """Allocator of the device output tensors this module creates (same
    signature as torch.empty; None restores torch.empty).  Tests pass one
    that surrounds every output with guard bytes."""
    global _empty
    _empty = torch.empty if fn is None else fn


def lib():
    """Loads libdart.so (raises if it was not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} not found: build it with __graft_entry__.build()")
        L = C.CDLL(LIB_PATH)
        vp, i, f = C.c_void_p, C.c_int, C.c_float
        sig = {
            "dart_init_head": (i, [C.POINTER(vp), C.POINTER(DartConfig), i, vp, vp, vp, vp]),
            "dart_expand_depth": (i, [vp, i, vp, vp, vp]),
            "dart_prune_and_emit": (i, [vp, C.POINTER(DartTreeOut), vp]),
            "dart_build_tree": (i, [vp, vp, vp, C.POINTER(DartTreeOut), vp]),
            "dart_build_tree_host": (i, [vp, vp, vp, C.POINTER(DartTreeOut), vp]),
            "dart_build_tree_fixed": (i, [vp, vp, vp, C.POINTER(DartTreeOut), vp]),
            "dart_build_chain_ddtree": (i, [vp, vp, vp, C.POINTER(DartTreeOut), vp]),
            "dart_build_seq_heap": (i, [vp, vp, vp, C.POINTER(DartTreeOut), vp]),
            "dart_get_chain": (i, [vp, vp, vp, vp]),
            "dart_get_frontier": (i, [vp, i, vp, vp, vp, vp, vp]),
            "dart_get_node_topk": (i, [vp, vp, vp, vp, C.POINTER(i), vp]),
            "dart_get_states": (i, [vp, vp, C.POINTER(i), vp]),
            "dart_status_sync": (i, [vp, vp]),
            "dart_test_wait_timeout": (i, [vp, i, vp, vp]),
            "dart_debug_build": (i, []),
            "dart_test_barrier_timeout": (i, [vp, i, vp]),
            "dart_test_bounds_report": (i, [vp, vp]),
            "dart_noalloc_status": (i, [vp]),
            "dart_set_profiling": (i, [vp, i]),
            "dart_profile_read": (i, [vp, C.POINTER(f), C.POINTER(i)]),
            "dart_profile_read_kinds": (i, [vp, vp, vp, i]),
            "dart_launches_per_round": (i, [vp]),
            "dart_expand_root_noalloc": (i, [C.POINTER(DartConfig), vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]),
            "dart_tree_attention_workspace": (C.c_size_t, [C.POINTER(DartAttnConfig)]),
            "dart_tree_attention": (i, [C.POINTER(DartAttnConfig), vp, vp, vp, vp, vp, vp, vp, vp, vp, vp,
                                        C.c_size_t, vp, vp]),
            "dart_tree_attention_timed": (i, [C.POINTER(DartAttnConfig), vp, vp, vp, vp, vp, vp, vp, vp, vp, vp,
                                              C.c_size_t, vp, C.POINTER(f), C.POINTER(f), vp]),
            "dart_ancestor_mask": (i, [vp, vp, i, i, vp, vp]),
            "dart_destroy": (None, [vp]),
            "dart_status_string": (C.c_char_p, [i]),
            "dart_version": (i, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def status_string(code: int) -> str:
    return lib().dart_status_string(int(code)).decode()


def _check(code, what):
    if code != DART_OK:
        raise DartError(code, what)


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return C.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def make_config(cfg) -> DartConfig:
    """From any object with V, d, L, W, k, B, nseq, beta, temperature,
    rms_eps, pos_offset and optionally cand_k (0: full vocabulary) and the
    tuning fields head_split, head_split_stream, lmhead_ctas_per_sm,
    weights_tiled, head_weights_tiled, variants, fused_round, topk_bound (0: the
    library's choice)."""
    g = lambda name: int(getattr(cfg, name, 0))
    return DartConfig(int(cfg.V), int(cfg.d), int(cfg.L), int(cfg.W), int(cfg.k), int(cfg.B),
                      int(cfg.nseq), float(cfg.beta), float(cfg.temperature), float(cfg.rms_eps),
                      int(cfg.pos_offset), g("cand_k"), g("head_split"), g("head_split_stream"),
                      g("lmhead_ctas_per_sm"), g("weights_tiled"), g("head_weights_tiled"), g("variants"),
                      g("fused_round"), g("topk_bound"))


def alloc_tree_out(cfg, device="cuda", pin=False):
    """Allocates the emitted-tree arrays; returns (dict of tensors, DartTreeOut)."""
    ns, B = cfg.nseq, cfg.B
    nw = (B + 63) // 64
    kw = dict(device=device)
    new = _empty
    if pin:
        kw = dict(device="cpu", pin_memory=True)
        new = torch.empty
    t = dict(tokens=new((ns, B), dtype=torch.int32, **kw),
             parents=new((ns, B), dtype=torch.int32, **kw),
             depths=new((ns, B), dtype=torch.int32, **kw),
             pos_ids=new((ns, B), dtype=torch.int32, **kw),
             scores=new((ns, B), dtype=torch.float32, **kw),
             n_nodes=new((ns,), dtype=torch.int32, **kw),
             mask=new((ns, B, nw), dtype=torch.int64, **kw))
    out = DartTreeOut(*(t[k].data_ptr() for k in
                        ("tokens", "parents", "depths", "pos_ids", "scores", "n_nodes", "mask")))
    return t, out


# ----------------------------------------------------------------- the ABI

def dart_init_head(cfg, wdtype, W_i, W_o, E, stream=None):
    """Returns an opaque handle (int).  W_i/W_o/E are device tensors of the
    weight dtype (torch.bfloat16 or torch.float32)."""
    h = C.c_void_p()
    c = make_config(cfg)
    _check(lib().dart_init_head(C.byref(h), C.byref(c), int(wdtype), _ptr(W_i), _ptr(W_o), _ptr(E),
                                _stream(stream)), "dart_init_head")
    return h


def dart_expand_depth(h, depth, drafter_logits, anchor_h=None, stream=None):
    _check(lib().dart_expand_depth(h, int(depth), _ptr(drafter_logits), _ptr(anchor_h),
                                   _stream(stream)), "dart_expand_depth")


def dart_prune_and_emit(h, out: DartTreeOut, stream=None):
    _check(lib().dart_prune_and_emit(h, C.byref(out), _stream(stream)), "dart_prune_and_emit")


def dart_build_tree(h, drafter_logits, anchor_h, out: DartTreeOut, stream=None):
    _check(lib().dart_build_tree(h, _ptr(drafter_logits), _ptr(anchor_h), C.byref(out),
                                 _stream(stream)), "dart_build_tree")


def dart_build_tree_fixed(h, drafter_logits, anchor_h, out: DartTreeOut, stream=None):
    """DARTree (fixed): every retained node emitted, no pruning (B >= sum |S_d|)."""
    _check(lib().dart_build_tree_fixed(h, _ptr(drafter_logits), _ptr(anchor_h), C.byref(out),
                                       _stream(stream)), "dart_build_tree_fixed")


def dart_build_chain_ddtree(h, drafter_logits, anchor_h, out: DartTreeOut, stream=None):
    """Domino-chain + DDTree (the handle needs DART_VARIANT_CHAIN_DDTREE)."""
    _check(lib().dart_build_chain_ddtree(h, _ptr(drafter_logits), _ptr(anchor_h), C.byref(out),
                                         _stream(stream)), "dart_build_chain_ddtree")


def dart_build_seq_heap(h, drafter_logits, anchor_h, out: DartTreeOut, stream=None):
    """Sequential correction with heap (the handle needs DART_VARIANT_SEQ_HEAP)."""
    _check(lib().dart_build_seq_heap(h, _ptr(drafter_logits), _ptr(anchor_h), C.byref(out),
                                     _stream(stream)), "dart_build_seq_heap")


def dart_get_chain(h, cfg, stream=None):
    """(chain tokens [nseq][L] int32, log-sum-exp [nseq][L] float) after
    dart_build_chain_ddtree."""
    tok = _empty((cfg.nseq, cfg.L), dtype=torch.int32, device="cuda")
    lse = _empty((cfg.nseq, cfg.L), dtype=torch.float32, device="cuda")
    _check(lib().dart_get_chain(h, _ptr(tok), _ptr(lse), _stream(stream)), "dart_get_chain")
    return tok, lse


def dart_build_tree_host(h, drafter_logits_host, anchor_host, out_host: DartTreeOut, stream=None):
    _check(lib().dart_build_tree_host(h, _ptr(drafter_logits_host), _ptr(anchor_host),
                                      C.byref(out_host), _stream(stream)), "dart_build_tree_host")


def dart_get_frontier(h, depth, cfg, stream=None):
    dev = "cuda"
    tok = _empty((cfg.nseq, cfg.W), dtype=torch.int32, device=dev)
    par = _empty(tok.shape, dtype=tok.dtype, device=tok.device)
    score = _empty((cfg.nseq, cfg.W), dtype=torch.float32, device=dev)
    count = _empty((cfg.nseq,), dtype=torch.int32, device=dev)
    _check(lib().dart_get_frontier(h, int(depth), _ptr(tok), _ptr(par), _ptr(score), _ptr(count),
                                   _stream(stream)), "dart_get_frontier")
    return tok, par, score, count


def dart_get_node_topk(h, cfg, stream=None):
    rows = C.c_int()
    _check(lib().dart_get_node_topk(h, None, None, None, C.byref(rows), _stream(stream)),
           "dart_get_node_topk")
    n = rows.value
    tok = _empty((n, cfg.k), dtype=torch.int32, device="cuda")
    logq = _empty((n, cfg.k), dtype=torch.float32, device="cuda")
    lse = _empty((n,), dtype=torch.float32, device="cuda")
    _check(lib().dart_get_node_topk(h, _ptr(tok), _ptr(logq), _ptr(lse), C.byref(rows),
                                    _stream(stream)), "dart_get_node_topk")
    return tok, logq, lse


def dart_get_states(h, cfg, stream=None):
    rows = C.c_int()
    _check(lib().dart_get_states(h, None, C.byref(rows), _stream(stream)), "dart_get_states")
    st = _empty((rows.value, cfg.d), dtype=torch.float32, device="cuda")
    _check(lib().dart_get_states(h, _ptr(st), C.byref(rows), _stream(stream)), "dart_get_states")
    return st


def dart_status_sync(h, stream=None):
    return int(lib().dart_status_sync(h, _stream(stream)))


def dart_test_barrier_timeout(h, limit_us, stream=None):
    _check(lib().dart_test_barrier_timeout(h, int(limit_us), _stream(stream)), "dart_test_barrier_timeout")


def dart_debug_build() -> bool:
    return bool(lib().dart_debug_build())


def dart_test_bounds_report(h, stream=None):
    _check(lib().dart_test_bounds_report(h, _stream(stream)), "dart_test_bounds_report")


def dart_test_wait_timeout(h, limit_us, elapsed_ns=None, stream=None):
    """Runs the bounded-wait probe (see dart.h); the next dart_status_sync
    returns DART_ERR_TIMEOUT.  elapsed_ns: optional int64 device tensor [2]."""
    _check(lib().dart_test_wait_timeout(h, int(limit_us), _ptr(elapsed_ns), _stream(stream)),
           "dart_test_wait_timeout")


def dart_set_profiling(h, enable):
    _check(lib().dart_set_profiling(h, int(bool(enable))), "dart_set_profiling")


def dart_profile_read(h):
    ms = C.c_float()
    n = C.c_int()
    _check(lib().dart_profile_read(h, C.byref(ms), C.byref(n)), "dart_profile_read")
    return float(ms.value), int(n.value)


KIND_NAMES = ("lmhead", "merge_select", "gather", "gemm_wi", "silu_split", "gemm_wo", "residual_norm",
              "prep_anchor", "prune_emit", "cand_topk", "cand_score", "gather_silu", "row_topk", "ddtree",
              "seqheap_step", "seqheap_emit", "round_f32", "l2_prefetch", "topk_bound")


def dart_profile_read_kinds(h):
    """{kind name: (total ms, launches)} since the last read."""
    n = len(KIND_NAMES)
    ms = (C.c_float * n)()
    cnt = (C.c_int * n)()
    _check(lib().dart_profile_read_kinds(h, C.cast(ms, C.c_void_p), C.cast(cnt, C.c_void_p), n),
           "dart_profile_read_kinds")
    return {KIND_NAMES[i]: (float(ms[i]), int(cnt[i])) for i in range(n)}


def dart_launches_per_round(h):
    return int(lib().dart_launches_per_round(h))


def dart_expand_root_noalloc(cfg, E, drafter_logits, anchor_h, node_tok, node_logq, node_lse, front_tok,
                             front_score, front_count, stream=None):
    """Depth-1 expansion without device allocation (outputs are caller tensors)."""
    c = make_config(cfg)
    _check(lib().dart_expand_root_noalloc(C.byref(c), _ptr(E), _ptr(drafter_logits), _ptr(anchor_h),
                                          _ptr(node_tok), _ptr(node_logq), _ptr(node_lse), _ptr(front_tok),
                                          _ptr(front_score), _ptr(front_count), _stream(stream)),
           "dart_expand_root_noalloc")


def dart_noalloc_status(stream=None):
    """DART_OK or DART_ERR_TIMEOUT for the most recent dart_expand_root_noalloc
    on the current device (synchronises the stream)."""
    return int(lib().dart_noalloc_status(_stream(stream)))


def dart_destroy(h):
    if h:
        lib().dart_destroy(h)


class Dart:
    """Owns one handle plus the weight tensors it borrows."""

    def __init__(self, cfg, W_i, W_o, E, stream=None):
        if W_i.dtype == torch.bfloat16:
            wd = DART_BF16
        elif W_i.dtype == torch.float32:
            wd = DART_F32
        else:
            raise TypeError("weights must be bfloat16 or float32")
        self.cfg = cfg
        self._keep = (W_i, W_o, E)
        self.h = dart_init_head(cfg, wd, W_i, W_o, E, stream)
        self.out_t, self.out = alloc_tree_out(cfg)

    def build_tree(self, drafter_logits, anchor_h, stream=None):
        dart_build_tree(self.h, drafter_logits, anchor_h, self.out, stream)
        return self.out_t

    def build_tree_fixed(self, drafter_logits, anchor_h, stream=None):
        dart_build_tree_fixed(self.h, drafter_logits, anchor_h, self.out, stream)
        return self.out_t

    def build_chain_ddtree(self, drafter_logits, anchor_h, stream=None):
        dart_build_chain_ddtree(self.h, drafter_logits, anchor_h, self.out, stream)
        return self.out_t

    def build_seq_heap(self, drafter_logits, anchor_h, stream=None):
        dart_build_seq_heap(self.h, drafter_logits, anchor_h, self.out, stream)
        return self.out_t

    def close(self):
        dart_destroy(self.h)
        self.h = None

    def __del__(self):
        try:
            if self.h:
                self.close()
        except Exception:
            pass


# ------------------------------------------- tree-attention verification (dart_verify.h)

def make_attn_config(nseq, B, C_ctx, Hq, Hkv, dh, rope_theta, scale) -> DartAttnConfig:
    return DartAttnConfig(int(nseq), int(B), int(C_ctx), int(Hq), int(Hkv), int(dh), float(rope_theta),
                          float(scale))


def dart_tree_attention_workspace(acfg: DartAttnConfig) -> int:
    return int(lib().dart_tree_attention_workspace(C.byref(acfg)))


def dart_tree_attention(acfg: DartAttnConfig, q, k_tree, v_tree, k_ctx, v_ctx, pos_ids, mask, n_nodes, out,
                        workspace, status=None, stream=None):
    """One tree-attention layer; every tensor is a caller-owned device tensor
    (bf16 q/k/v, int32 pos_ids/n_nodes, int64 mask, fp32 out, uint8 workspace)."""
    _check(lib().dart_tree_attention(C.byref(acfg), _ptr(q), _ptr(k_tree), _ptr(v_tree), _ptr(k_ctx),
                                     _ptr(v_ctx), _ptr(pos_ids), _ptr(mask), _ptr(n_nodes), _ptr(out),
                                     _ptr(workspace), C.c_size_t(workspace.numel() * workspace.element_size()),
                                     _ptr(status), _stream(stream)), "dart_tree_attention")


def dart_tree_attention_timed(acfg: DartAttnConfig, q, k_tree, v_tree, k_ctx, v_ctx, pos_ids, mask, n_nodes, out,
                              workspace, status=None, stream=None):
    """As dart_tree_attention, then synchronises; returns (ms of the RoPE
    pre-pass, ms of the attention kernel)."""
    a, b = C.c_float(), C.c_float()
    _check(lib().dart_tree_attention_timed(C.byref(acfg), _ptr(q), _ptr(k_tree), _ptr(v_tree), _ptr(k_ctx),
                                           _ptr(v_ctx), _ptr(pos_ids), _ptr(mask), _ptr(n_nodes), _ptr(out),
                                           _ptr(workspace),
                                           C.c_size_t(workspace.numel() * workspace.element_size()),
                                           _ptr(status), C.byref(a), C.byref(b), _stream(stream)),
           "dart_tree_attention_timed")
    return float(a.value), float(b.value)


def dart_ancestor_mask(parents, n_nodes, mask, stream=None):
    nseq, B = parents.shape
    _check(lib().dart_ancestor_mask(_ptr(parents), _ptr(n_nodes), int(nseq), int(B), _ptr(mask),
                                    _stream(stream)), "dart_ancestor_mask")


class TreeAttention:
    """Owns the workspace of one tree-attention shape."""

    def __init__(self, nseq, B, C_ctx, Hq=32, Hkv=8, dh=128, rope_theta=1.0e6, scale=None):
        self.cfg = make_attn_config(nseq, B, C_ctx, Hq, Hkv, dh, rope_theta,
                                    scale if scale is not None else dh ** -0.5)
        n = dart_tree_attention_workspace(self.cfg)
        if n == 0:
            raise DartError(DART_ERR_INVALID, "dart_tree_attention_workspace")
        self.workspace = _empty((n,), dtype=torch.uint8, device="cuda")
        c = self.cfg
        self.out = _empty((c.nseq, c.B, c.Hq, c.dh), dtype=torch.float32, device="cuda")

    def __call__(self, q, k_tree, v_tree, k_ctx, v_ctx, pos_ids, mask, n_nodes, status=None, stream=None):
        dart_tree_attention(self.cfg, q, k_tree, v_tree, k_ctx, v_ctx, pos_ids, mask, n_nodes, self.out,
                            self.workspace, status, stream)
        return self.out

    def timed(self, q, k_tree, v_tree, k_ctx, v_ctx, pos_ids, mask, n_nodes, status=None, stream=None):
        return dart_tree_attention_timed(self.cfg, q, k_tree, v_tree, k_ctx, v_ctx, pos_ids, mask, n_nodes,
                                         self.out, self.workspace, status, stream)
