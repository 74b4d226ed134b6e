"""Guarded device outputs for the GPU parity tests.

The output tensor handed to a kernel is a view into a larger allocation
whose margins (GUARD bytes before and after it) hold a sentinel pattern.
`check()` fails when any margin byte changed, that is when a kernel wrote
outside its output: the element-by-element comparison of the output itself
cannot see such a write.  GUARD keeps the view's base address aligned as the
allocation's.
"""
import numpy as np

GUARD = 4096


def _pattern(n):
    i = np.arange(n, dtype=np.int64)
    return ((i * 151 + 89) & 0xFF).astype(np.uint8)   # never all one value


class Guarded:
    def __init__(self, shape, dtype, device="cuda"):
        import torch
        self.shape = tuple(int(x) for x in shape)
        n = int(np.prod(self.shape)) * torch.empty((), dtype=dtype).element_size()
        self.n = n
        self.buf = torch.from_numpy(_pattern(GUARD + n + GUARD)).to(device)
        self.view = self.buf[GUARD:GUARD + n].view(dtype).view(self.shape)

    def check(self):
        host = self.buf.cpu().numpy()
        ref = _pattern(host.size)
        for name, sl in (("before", slice(0, GUARD)), ("after", slice(GUARD + self.n, None))):
            bad = np.flatnonzero(host[sl] != ref[sl])
            if bad.size:
                off = bad[0] - GUARD if name == "before" else bad[0]
                raise AssertionError(f"{bad.size} guard bytes {name} the output were written "
                                     f"(first at offset {off} from the {name} edge)")
