"""The seeded synthetic workloads (CPU): the named shapes are the paper's
Qwen3-4B / Qwen3-8B settings, the width / budget sweep and the batched
serving shape; the draws are deterministic, follow the stated distributions
and give each replica rank its own sequences."""
import numpy as np
import pytest

from workloads import BATCHED, NAMED, Q4B, Q8B, TOY, make_sequences, make_weights, sweep_configs


def test_named_shapes():
    shape = lambda c: (c.nseq, c.V, c.d, c.L, c.W, c.k, c.B, c.wdtype)
    assert shape(TOY) == (1, 4096, 256, 4, 4, 4, 16, "f32") and TOY.temperature == 0.0
    assert shape(Q4B) == (1, 151936, 2560, 16, 8, 8, 64, "bf16") and Q4B.temperature == 0.0
    assert shape(Q8B) == (1, 151936, 4096, 16, 16, 16, 256, "bf16") and Q8B.temperature == 1.0
    assert shape(BATCHED) == (8, 151936, 4096, 16, 32, 32, 512, "bf16") and BATCHED.temperature == 1.0
    grid = {(c.W, c.B) for c in sweep_configs()}
    assert grid == {(W, B) for W in (8, 16, 32, 64) for B in (32, 128, 512, 1024)}
    for c in sweep_configs():
        assert (c.V, c.d, c.L, c.k, c.wdtype) == (151936, 2560, 16, c.W, "bf16")
    for name in ("qwen3-8b-k64", "qwen3-4b-k64", "batched-k64"):
        assert NAMED[name].cand_k == 64
    assert all(c.beta == -0.2 for c in NAMED.values())
    # pruning is the identity exactly where the budget covers the supertree
    assert sum(Q8B.caps()[1:]) == 256 == Q8B.B
    assert sum(Q4B.caps()[1:]) == 128 > Q4B.B
    assert sum(BATCHED.caps()[1:]) == 512 == BATCHED.B


def test_drafter_logits_and_anchors():
    D, h0 = make_sequences(Q4B)
    assert D.shape == (1, 16, 151936) and D.dtype == np.float32 and h0.shape == (1, 2560)
    D2, h02 = make_sequences(Q4B)
    assert np.array_equal(D, D2) and np.array_equal(h0, h02)          # deterministic
    assert abs(float(D.std()) - 3.0) < 0.01 and abs(float(D.mean())) < 0.01
    assert abs(float(h0.std()) - 1.0) < 0.05
    Dr, _ = make_sequences(Q4B, rank=1)
    assert not np.array_equal(D, Dr)                                  # replicas differ
    Db, hb = make_sequences(BATCHED.replace(V=1000, d=64))
    assert len({hb[s].tobytes() for s in range(8)}) == 8               # sequences differ


@pytest.mark.parametrize("wdtype", ["f32", "bf16"])
def test_weight_distributions(wdtype):
    from workloads import bf16_bits_to_f32
    c = Q8B.replace(V=20000, d=512, wdtype=wdtype)
    Wi, Wo, E = make_weights(c)
    f = (lambda a: a) if wdtype == "f32" else bf16_bits_to_f32
    Wi, Wo, E = f(Wi), f(Wo), f(E)
    assert Wi.shape == (512, 1024) and Wo.shape == (512, 512) and E.shape == (20000, 512)
    assert abs(float(Wi.std()) * np.sqrt(2 * 512) - 1.0) < 0.01
    assert abs(float(Wo.std()) * np.sqrt(512) - 1.0) < 0.01
    assert abs(float(E.std()) / 0.02 - 1.0) < 0.01
    Wi2, _, _ = make_weights(c)
    assert np.array_equal(f(Wi2), Wi)


@pytest.mark.parametrize("cfg,early,late", [(Q4B, 6.0, 3.0), (Q8B, 6.0, 3.0), (TOY, 8.0, 8.0)],
                         ids=["qwen3-4b", "qwen3-8b", "toy"])
def test_spike_heights(cfg, early, late):
    """The same seed with the spikes switched off differs from the real draw by
    exactly one lifted token per position: +6 at positions 0-7 and +3 at 8-15
    (+8 everywhere in the fp32 toy)."""
    c = cfg.replace(V=5000, d=64)
    D, _ = make_sequences(c)
    D0, _ = make_sequences(c.replace(spike_early=0.0, spike_late=0.0))
    diff = (D - D0)[0]
    for i in range(c.L):
        nz = np.nonzero(np.abs(diff[i]) > 1e-3)[0]
        assert nz.size == 1
        assert abs(float(diff[i, nz[0]]) - (early if i < 8 else late)) < 1e-5
