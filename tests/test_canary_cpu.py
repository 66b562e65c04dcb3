"""The guard-byte checker of the device outputs (run on host tensors)."""
import pytest
import torch

import canary


def test_untouched_guards_pass():
    canary.reset()
    t = canary.empty((3, 5), dtype=torch.int32, device="cpu")
    t.fill_(-1)  # the whole output may be written
    canary.check()


@pytest.mark.parametrize("where", ["after", "before"])
def test_a_write_outside_the_output_fails(where):
    canary.reset()
    t = canary.empty((4, 3), dtype=torch.float32, device="cpu")
    buf, n = canary._live[-1]
    assert t.data_ptr() == buf.data_ptr() + canary.PAD and t.data_ptr() % 16 == 0
    # one element past the end, or one before the start
    if where == "after":
        buf[canary.PAD + n] = 0
    else:
        buf[canary.PAD - 1] = 0
    with pytest.raises(AssertionError, match="end" if where == "after" else "start"):
        canary.check()
    canary.reset()
