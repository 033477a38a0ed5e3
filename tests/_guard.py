"""Output buffers with guard bands, for the GPU tests.

compute-sanitizer is not available on the GPU pool, so out-of-bounds writes are caught the
plain way: every output a test hands to the library is a view into a larger buffer whose
bands on both sides hold a sentinel byte pattern, and after the call the bands must be
unchanged.  The views stay 256-byte aligned (the library wants 16).
"""
from __future__ import annotations

import torch

GUARD_BYTES = 4096
SENTINEL = 0xA5


class Guarded:
    """A tensor of `shape`/`dtype` on `device` inside a buffer with GUARD_BYTES of sentinel
    bytes before and after it.  `.t` is the tensor (filled with `fill`); `.check()` asserts
    both bands are intact."""

    def __init__(self, shape, dtype, device, fill=None):
        shape = tuple(int(s) for s in shape)
        n = 1
        for s in shape:
            n *= s
        item = torch.empty((), dtype=dtype).element_size()
        self.nbytes = n * item
        body = (self.nbytes + 255) // 256 * 256
        self.buf = torch.full((GUARD_BYTES + body + GUARD_BYTES,), SENTINEL, dtype=torch.uint8,
                              device=device)
        self.t = self.buf[GUARD_BYTES:GUARD_BYTES + self.nbytes].view(dtype).view(shape)
        if fill is not None:
            self.t.fill_(fill)
        # the tail of the last 256-byte block after the tensor is part of the back band
        self.back_from = GUARD_BYTES + self.nbytes

    def check(self, what="output"):
        front = self.buf[:GUARD_BYTES]
        back = self.buf[self.back_from:]
        bad_f = int((front != SENTINEL).sum())
        bad_b = int((back != SENTINEL).sum())
        assert bad_f == 0 and bad_b == 0, \
            f"{what}: {bad_f} bytes written before and {bad_b} after the buffer"


def guarded(shape, dtype, device, fill=None) -> Guarded:
    return Guarded(shape, dtype, device, fill)


def check_all(*gs):
    for i, g in enumerate(gs):
        g.check(f"output {i}")
