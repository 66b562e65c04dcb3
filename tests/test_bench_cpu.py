"""Host-side logic of the benchmark (CPU): the byte accounting and the
L2-residency rule it mirrors from the library's plan, which decide the
roofline kernel and its algorithmic bytes per launch, and the whole-job rate."""
import pytest

import bench
from workloads import NAMED


def test_first_head_layer_bytes_per_depth():
    q8 = NAMED["qwen3-8b"]
    # split first layer (the default): W_i[:, 0:d] only, d*d bf16 elements
    assert bench.split_head(q8)
    assert bench.wi_bytes_per_depth(q8) == 4096 * 4096 * 2
    # unsplit (dart_config.head_split = DART_OFF): all of W_i [d][2d]
    off = q8.replace(head_split=2)
    assert not bench.split_head(off)
    assert bench.wi_bytes_per_depth(off) == 4096 * 2 * 4096 * 2
    assert bench.split_head(q8.replace(head_split=1))
    # the fp32 toy never splits
    toy = NAMED["toy"]
    assert not bench.split_head(toy)
    assert bench.wi_bytes_per_depth(toy) == 2 * toy.d * toy.d * 4


@pytest.mark.parametrize("name,split,expect", [
    ("qwen3-8b-k64", True, (True, True)),     # 33.5 + 33.5 MB <= 72 MiB
    ("qwen3-4b-k64", True, (True, True)),     # 13 + 13 MB
    ("qwen3-8b-k64", False, (True, False)),   # W_i 67 MB alone
    ("qwen3-4b-k64", False, (True, True)),    # 26 + 13 MB
    ("batched-k64", True, (False, False)),    # 256 children: cluster GEMMs, nothing kept
    ("qwen3-8b", True, (False, False)),       # full vocabulary: the E stream evicts them
])
def test_kept_head_weights_mirrors_the_plan(name, split, expect):
    cfg = NAMED[name] if split else NAMED[name].replace(head_split=2)
    assert bench.kept_head_weights(cfg) == expect


def test_whole_job_rate_counts_every_rank():
    q8 = NAMED["qwen3-8b"]
    assert q8.expansions_per_round() == 241
    one = bench.whole_job_rate(q8.expansions_per_round(), 1, 3.45e-3)
    four = bench.whole_job_rate(q8.expansions_per_round(), 4, 3.45e-3)
    assert four == pytest.approx(4 * one)
    assert one == pytest.approx(241 / 3.45e-3)
