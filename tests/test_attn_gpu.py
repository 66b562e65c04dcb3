"""GPU parity of the tree-attention verification consumer (dart_verify.h)
against the fp64 oracle (oracle/tree_attn.py), through the C ABI.

The oracle walks parent indices and takes positions from depths; the GPU
side consumes an ancestor bitmask and position ids (built on the GPU by
dart_ancestor_mask, or emitted by dart_build_tree), so the two share only
the seeded inputs.

Tolerance (bf16 operands, fp32 accumulation, exact fp64 reference): the
rotated q and k are rounded to bf16 (unit roundoff u = 2^-8) and so is the
probability tile P fed to the tensor cores.  For N(0,1) inputs a logit
s = q.k / sqrt(dh) is perturbed by about sqrt(2 dh / 3) u / sqrt(dh) ~ 0.3 u
(rms), which moves an output by about that times the spread of the values
(~1), and the P rounding adds ~u/sqrt(3) times the weighted spread; the
rms error is therefore ~1e-3 and the maximum over 10^5..10^7 outputs a few
times 1e-3.  The tests require max |err| <= 2.5e-2 and rms <= 4e-3.
"""
import numpy as np
import pytest
import torch

import canary
from oracle import tree_attn as ta
from workloads import ATTN_BATCHED, ATTN_Q4B, ATTN_Q8B, AttnConfig, bf16_bits_to_f32, make_attn_inputs

pytestmark = pytest.mark.gpu

ATOL = 2.5e-2
RMS = 4e-3


@pytest.fixture(scope="module")
def dart():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13524_gb300 import dart as d
    d.lib()
    return d


def bf_dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def bf_val(bits):
    return bf16_bits_to_f32(bits).astype(np.float64)


def gpu_attention(dart, cfg: AttnConfig, x, mask=None, pos_ids=None, n_nodes=None):
    """Runs dart_tree_attention; the mask comes from dart_ancestor_mask of the
    parent array unless given."""
    dev = "cuda"
    par = torch.from_numpy(x["parents"]).to(dev)
    nn = torch.from_numpy(x["n_nodes"]).to(dev) if n_nodes is None else n_nodes
    if mask is None:
        mw = (cfg.B + 63) // 64
        mask = canary.empty((cfg.nseq, cfg.B, mw), dtype=torch.int64, device=dev)
        dart.dart_ancestor_mask(par, nn, mask)
    if pos_ids is None:
        dep = torch.from_numpy(x["depths"]).to(dev)
        pos_ids = torch.where(dep > 0, dep + cfg.offset, torch.full_like(dep, -1)).to(torch.int32)
    att = dart.TreeAttention(cfg.nseq, cfg.B, cfg.C, cfg.Hq, cfg.Hkv, cfg.dh, cfg.rope_theta, cfg.scale)
    status = torch.zeros(4, dtype=torch.int32, device=dev)
    kc = bf_dev(x["k_ctx"]) if cfg.C > 0 else None
    vc = bf_dev(x["v_ctx"]) if cfg.C > 0 else None
    out = att(bf_dev(x["q"]), bf_dev(x["k_tree"]), bf_dev(x["v_tree"]), kc, vc, pos_ids, mask, nn, status)
    torch.cuda.synchronize()
    assert int(status[0].item()) == 0
    return out.cpu().numpy().astype(np.float64), mask


def oracle_attention(cfg, x, rows=None):
    return ta.tree_attention(bf_val(x["q"]), bf_val(x["k_tree"]), bf_val(x["v_tree"]), bf_val(x["k_ctx"]),
                             bf_val(x["v_ctx"]), x["parents"], x["depths"], x["n_nodes"], cfg.offset,
                             cfg.rope_theta, cfg.scale, rows=rows)


def compare(cfg, x, got, ref, rows=None):
    if rows is None:
        rows = [(s, i) for s in range(cfg.nseq) for i in range(cfg.B)]
    err = np.array([np.abs(got[s, i] - ref[s, i]).max() for s, i in rows])
    sq = np.concatenate([(got[s, i] - ref[s, i]).ravel() ** 2 for s, i in rows])
    rms = float(np.sqrt(sq.mean()))
    print(f"{cfg.name}: max|err| {err.max():.3e} rms {rms:.3e} over {len(rows)} rows")
    assert err.max() <= ATOL, (cfg.name, float(err.max()))
    assert rms <= RMS, (cfg.name, rms)
    for s in range(cfg.nseq):
        assert np.all(got[s, int(x["n_nodes"][s]):] == 0.0)


def A(name, nseq, B, C, L=16, W=16, seed=1, **kw):
    return AttnConfig(name, nseq, B, C, L, W, 3000 + seed, **kw)


SMALL = [
    A("g4-c10", 1, 40, 10, L=4, W=12, seed=1),
    A("g4-tree-only", 2, 100, 0, L=6, W=20, seed=2, fill=0.8),
    A("g1-c130", 1, 64, 130, L=8, W=8, seed=3, Hq=8, Hkv=8),
    A("g8-c300", 1, 48, 300, L=5, W=10, seed=4, Hq=32, Hkv=4),
    A("g16-c77", 2, 24, 77, L=4, W=8, seed=5, Hq=16, Hkv=1),
    A("g2-c5", 1, 70, 5, L=10, W=7, seed=6, Hq=16, Hkv=8),
    A("deep-3-tree-tiles", 2, 300, 200, L=16, W=32, seed=7, fill=0.9),
    A("long-context-splits", 1, 16, 4000, L=4, W=4, seed=8),
    A("pos-offset", 1, 33, 64, L=5, W=8, seed=9, pos_offset=500, rope_theta=1.0e4),
]


@pytest.mark.parametrize("cfg", SMALL, ids=lambda c: c.name)
def test_attention_parity(dart, cfg):
    x = make_attn_inputs(cfg)
    got, _ = gpu_attention(dart, cfg, x)
    ref = oracle_attention(cfg, x)
    compare(cfg, x, got, ref)


def test_empty_and_single_node_trees(dart):
    cfg = A("empty-and-single", 3, 20, 9, L=3, W=5, seed=10)
    x = make_attn_inputs(cfg)
    x["parents"][0] = -2
    x["depths"][0] = 0
    x["n_nodes"][0] = 0
    x["parents"][1] = -2
    x["depths"][1] = 0
    x["parents"][1, 0] = -1
    x["depths"][1, 0] = 1
    x["n_nodes"][1] = 1
    got, _ = gpu_attention(dart, cfg, x)
    assert np.all(got[0] == 0.0)
    ref = oracle_attention(cfg, x)
    compare(cfg, x, got, ref)


def test_ancestor_mask_matches_paths(dart):
    cfg = A("mask", 3, 200, 0, L=16, W=24, seed=11, fill=0.95)
    x = make_attn_inputs(cfg)
    par = torch.from_numpy(x["parents"]).cuda()
    nn = torch.from_numpy(x["n_nodes"]).cuda()
    mw = (cfg.B + 63) // 64
    mask = canary.empty((cfg.nseq, cfg.B, mw), dtype=torch.int64, device="cuda")
    dart.dart_ancestor_mask(par, nn, mask)
    m = mask.cpu().numpy().view(np.uint64)
    for s in range(cfg.nseq):
        n = int(x["n_nodes"][s])
        for i in range(cfg.B):
            want = np.zeros(mw, dtype=np.uint64)
            if i < n:
                for j in ta.root_path(x["parents"][s], i):
                    want[j // 64] |= np.uint64(1) << np.uint64(j % 64)
            assert np.array_equal(m[s, i], want), (s, i)


def test_large_budget_sampled(dart):
    cfg = A("B1024", 1, 1024, 0, L=16, W=64, seed=12)
    x = make_attn_inputs(cfg)
    got, _ = gpu_attention(dart, cfg, x)
    g = np.random.Generator(np.random.PCG64(12))
    rows = [(0, int(i)) for i in sorted(set(g.integers(0, 1024, 64).tolist()) | {0, 127, 128, 1023})]
    ref = oracle_attention(cfg, x, rows)
    compare(cfg, x, got, ref, rows)


@pytest.mark.parametrize("cfg", [ATTN_Q8B, ATTN_Q4B, ATTN_BATCHED], ids=lambda c: c.name)
def test_full_size_sampled(dart, cfg):
    x = make_attn_inputs(cfg)
    got, _ = gpu_attention(dart, cfg, x)
    g = np.random.Generator(np.random.PCG64(cfg.seed))
    rows = set()
    for s in range(cfg.nseq):
        n = int(x["n_nodes"][s])
        rows |= {(s, int(i)) for i in g.integers(0, n, 6)} | {(s, 0), (s, n - 1)}
    rows = sorted(rows)
    ref = oracle_attention(cfg, x, rows)
    compare(cfg, x, got, ref, rows)


def test_deterministic(dart):
    cfg = A("det", 2, 128, 1500, L=8, W=16, seed=13)
    x = make_attn_inputs(cfg)
    a, _ = gpu_attention(dart, cfg, x)
    b, _ = gpu_attention(dart, cfg, x)
    assert np.array_equal(a, b)


def test_consumes_the_emitted_tree(dart):
    """dart_build_tree -> emitted mask + pos_ids -> dart_tree_attention, against
    the oracle's own tree (orc_build_tree) and path-walk attention."""
    import oracle
    from parity import to_device
    from workloads import Config, make_inputs
    ccfg = Config("e2e", 2, 5003, 512, 5, 8, 8, 24, "bf16", 0.0, 14, pos_offset=40)
    xin = make_inputs(ccfg)
    dx = to_device(ccfg, xin)
    h = dart.Dart(ccfg, dx["Wi"], dx["Wo"], dx["E"])
    t = h.build_tree(dx["Dlog"], dx["h0"])
    torch.cuda.synchronize()
    orc = oracle.build_tree(ccfg, xin["Wi"], xin["Wo"], xin["E"], xin["Dlog"], xin["h0"])
    emitted = {k: v.cpu().numpy() for k, v in t.items()}
    if float(orc["prune_gap"].min()) < 2e-3:
        pytest.skip("near tie in the oracle's pruning: topology not unique")
    for k in ("parents", "depths", "n_nodes"):
        assert np.array_equal(emitted[k], orc[k]), k
    acfg = AttnConfig("e2e-attn", ccfg.nseq, ccfg.B, 40, ccfg.L, ccfg.W, 3100, pos_offset=ccfg.pos_offset)
    x = make_attn_inputs(acfg)
    x["parents"] = orc["parents"].astype(np.int32)
    x["depths"] = orc["depths"].astype(np.int32)
    x["n_nodes"] = orc["n_nodes"].astype(np.int32)
    got, _ = gpu_attention(dart, acfg, x, mask=t["mask"], pos_ids=t["pos_ids"], n_nodes=t["n_nodes"])
    ref = oracle_attention(acfg, x)
    compare(acfg, x, got, ref)
    h.close()


def test_tolerance_detects_a_planted_mask_error(dart, monkeypatch):
    """The tolerance is tight enough to see one wrong key: an oracle with a
    sibling leaking into every path (planted on the CPU) fails it."""
    cfg = SMALL[1]
    x = make_attn_inputs(cfg)
    got, _ = gpu_attention(dart, cfg, x)
    honest = ta.root_path

    def with_sibling(parents, i):
        path = honest(parents, i)
        sib = [j for j in range(len(parents)) if parents[j] == parents[i] and j != i]
        return path[:-1] + sib[:1] + path[-1:] if sib else path

    monkeypatch.setattr(ta, "root_path", with_sibling)
    bad = oracle_attention(cfg, x)
    assert np.abs(got - bad).max() > 10 * ATOL
