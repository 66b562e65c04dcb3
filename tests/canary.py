"""Guard bytes around every device output the binding allocates.

Each output tensor is a view into a larger byte buffer whose first and last
PAD bytes hold PATTERN.  After a GPU test, check() confirms that no kernel
wrote outside the outputs it was given (a write one row or one element past
an output's end, or before its start, changes a guard byte).
"""
import math

import torch

PAD = 4096          # bytes on each side (keeps the output 16-byte aligned)
PATTERN = 0xA5
_live = []


def empty(shape, dtype=torch.float32, device="cuda", **kw):
    if kw:  # pinned host memory and other special allocations: unguarded
        return torch.empty(shape, dtype=dtype, device=device, **kw)
    if isinstance(shape, int):
        shape = (shape,)
    item = torch.empty((), dtype=dtype).element_size()
    n = math.prod(shape) * item
    buf = torch.full((PAD + n + PAD,), PATTERN, dtype=torch.uint8, device=device)
    _live.append((buf, n))
    return buf[PAD:PAD + n].view(dtype).view(tuple(shape))


def check():
    """Raises AssertionError naming the first output whose guard changed."""
    bad = []
    for i, (buf, n) in enumerate(_live):
        head, tail = buf[:PAD], buf[PAD + n:]
        if not (bool((head == PATTERN).all()) and bool((tail == PATTERN).all())):
            first = int(torch.nonzero(torch.cat([head, tail]) != PATTERN)[0])
            where = f"{PAD - first} bytes before its start" if first < PAD else f"{first - PAD} bytes past its end"
            bad.append(f"output {i} ({n} bytes): the guard byte {where} changed")
    _live.clear()
    assert not bad, "; ".join(bad)


def reset():
    _live.clear()
