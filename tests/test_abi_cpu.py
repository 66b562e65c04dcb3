"""C-ABI checks that need no GPU: the library loads, exports every function
declared in include/dart.h, and rejects bad arguments on the host before any
CUDA call is made."""
import ctypes as C
import os
import re

import pytest

from paper_2608_13524_gb300 import dart

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = []
    for h in os.listdir(os.path.join(ROOT, "include")):
        if h.endswith(".h"):
            txt = open(os.path.join(ROOT, "include", h)).read()
            txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
            names += re.findall(r"\b(dart_\w+)\s*\(", txt)
    return sorted(set(names))


def test_library_exports_every_declared_symbol():
    lib = C.CDLL(dart.LIB_PATH)
    names = declared_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/ but not exported"


def test_status_strings_and_version():
    assert dart.lib().dart_version() >= 1
    for code in range(0, -7, -1):
        s = dart.status_string(code)
        assert s and s != "unknown status"
    assert dart.status_string(-99) == "unknown status"


class Cfg:
    def __init__(self, **kw):
        base = dict(V=1000, d=128, L=4, W=4, k=4, B=16, nseq=1, beta=-0.2, temperature=0.0,
                    rms_eps=1e-6, pos_offset=0, cand_k=0)
        base.update(kw)
        self.__dict__.update(base)


BAD = [dict(V=0), dict(d=100), dict(d=32), dict(L=0), dict(W=0), dict(W=65), dict(k=0), dict(k=65),
       dict(V=10, k=11), dict(W=64, k=65), dict(L=17, W=64), dict(B=0), dict(B=1025), dict(nseq=0),
       dict(nseq=5, W=64), dict(beta=0.1), dict(beta=float("nan")), dict(temperature=-1.0),
       dict(rms_eps=0.0), dict(cand_k=3), dict(cand_k=-1), dict(cand_k=1001), dict(V=5000, cand_k=1025),
       dict(d=16448), dict(V=1 << 24), dict(L=1025, W=1), dict(temperature=float("inf")),
       dict(rms_eps=float("nan")), dict(head_split=3), dict(head_split=-1), dict(head_split_stream=3),
       dict(lmhead_ctas_per_sm=3), dict(lmhead_ctas_per_sm=-1), dict(variants=4), dict(variants=-1),
       dict(fused_round=3), dict(fused_round=-1), dict(topk_bound=3), dict(topk_bound=-1)]


@pytest.mark.parametrize("bad", BAD, ids=[str(b) for b in BAD])
def test_init_rejects_bad_config_on_host(bad):
    lib = dart.lib()
    h = C.c_void_p(1234)
    cfg = dart.make_config(Cfg(**bad))
    buf = (C.c_uint8 * 64)()
    p = C.cast(buf, C.c_void_p).value
    p = (p + 15) & ~15
    rc = lib.dart_init_head(C.byref(h), C.byref(cfg), dart.DART_BF16, p, p, p, None)
    assert rc == dart.DART_ERR_INVALID
    assert h.value is None  # *out is cleared on failure


def test_init_rejects_null_and_misaligned_weights():
    lib = dart.lib()
    cfg = dart.make_config(Cfg())
    h = C.c_void_p()
    buf = (C.c_uint8 * 64)()
    p = (C.cast(buf, C.c_void_p).value + 15) & ~15
    assert lib.dart_init_head(C.byref(h), C.byref(cfg), dart.DART_BF16, None, p, p, None) == dart.DART_ERR_INVALID
    assert lib.dart_init_head(C.byref(h), C.byref(cfg), dart.DART_BF16, p + 2, p, p, None) == dart.DART_ERR_INVALID
    assert lib.dart_init_head(C.byref(h), C.byref(cfg), 7, p, p, p, None) == dart.DART_ERR_INVALID
    assert lib.dart_init_head(None, C.byref(cfg), dart.DART_BF16, p, p, p, None) == dart.DART_ERR_INVALID


def test_null_handle_is_rejected():
    lib = dart.lib()
    out = dart.DartTreeOut()
    assert lib.dart_expand_depth(None, 1, None, None, None) == dart.DART_ERR_INVALID
    assert lib.dart_prune_and_emit(None, C.byref(out), None) == dart.DART_ERR_INVALID
    assert lib.dart_build_tree(None, None, None, C.byref(out), None) == dart.DART_ERR_INVALID
    assert lib.dart_status_sync(None, None) == dart.DART_ERR_INVALID
    lib.dart_destroy(None)  # no-op


ATTN_BAD = [dict(nseq=0), dict(B=0), dict(B=1025), dict(C_ctx=-1), dict(Hq=12, Hkv=8), dict(Hq=24, Hkv=8),
            dict(Hq=4, Hkv=8), dict(dh=64), dict(rope_theta=1.0), dict(rope_theta=float("inf")), dict(scale=0.0),
            dict(scale=float("nan"))]


def attn_cfg(**kw):
    base = dict(nseq=1, B=64, C_ctx=128, Hq=32, Hkv=8, dh=128, rope_theta=1.0e6, scale=128 ** -0.5)
    base.update(kw)
    return dart.make_attn_config(**base)


@pytest.mark.parametrize("bad", ATTN_BAD, ids=[str(b) for b in ATTN_BAD])
def test_tree_attention_rejects_bad_config_on_host(bad):
    lib = dart.lib()
    cfg = attn_cfg(**bad)
    assert lib.dart_tree_attention_workspace(C.byref(cfg)) == 0
    buf = (C.c_uint8 * 1024)()
    p = (C.cast(buf, C.c_void_p).value + 255) & ~255
    rc = lib.dart_tree_attention(C.byref(cfg), p, p, p, p, p, p, p, p, p, p, 1 << 40, None, None)
    assert rc == dart.DART_ERR_INVALID


def test_tree_attention_rejects_null_and_misaligned_pointers():
    lib = dart.lib()
    cfg = attn_cfg()
    buf = (C.c_uint8 * 1024)()
    p = (C.cast(buf, C.c_void_p).value + 255) & ~255
    args = [p] * 10
    for i in range(10):
        a = list(args)
        a[i] = None  # context K/V (3, 4) may be NULL only when C = 0
        assert lib.dart_tree_attention(C.byref(cfg), *a, 1 << 40, None, None) == dart.DART_ERR_INVALID
        a[i] = p + 8
        assert lib.dart_tree_attention(C.byref(cfg), *a, 1 << 40, None, None) == dart.DART_ERR_INVALID
    assert lib.dart_ancestor_mask(None, p, 1, 8, p, None) == dart.DART_ERR_INVALID
    assert lib.dart_ancestor_mask(p, p, 1, 0, p, None) == dart.DART_ERR_INVALID
    assert lib.dart_ancestor_mask(p, p, 0, 8, p, None) == dart.DART_ERR_INVALID
    assert lib.dart_ancestor_mask(p, p, 1, 1025, p, None) == dart.DART_ERR_INVALID


def test_tree_attention_rejects_a_small_workspace_on_host():
    lib = dart.lib()
    cfg = attn_cfg()
    need = lib.dart_tree_attention_workspace(C.byref(cfg))
    # rotated tree keys (bf16) and the (cos, sin) table of the tree positions
    assert need >= 1 * 64 * 8 * 128 * 2 + 1 * 64 * 64 * 8
    buf = (C.c_uint8 * 1024)()
    p = (C.cast(buf, C.c_void_p).value + 255) & ~255
    rc = lib.dart_tree_attention(C.byref(cfg), p, p, p, p, p, p, p, p, p, p, need - 1, None, None)
    assert rc == dart.DART_ERR_INVALID


def test_profiling_kind_names_match_the_header():
    """The binding names as many profiling kinds as dart_profile_read_kinds
    accepts (include/dart.h), and the kinds numbered there are in the same
    order (the last one: the starting bound of the top-k filters)."""
    hdr = open(os.path.join(ROOT, "include", "dart.h")).read()
    n = int(re.search(r"nkinds <= (\d+)", hdr).group(1))
    assert len(dart.KIND_NAMES) == n
    assert dart.KIND_NAMES[-1] == "topk_bound" and re.search(rf"{n - 1} the starting bound of the top-k filters", hdr)
    assert dart.KIND_NAMES[16] == "round_f32" and dart.KIND_NAMES[17] == "l2_prefetch"
