"""The guard-byte helper of the GPU out-of-bounds tests, on the CPU: a write
one byte before or after the guarded tensor, or anywhere in the guards, is
reported; writes inside it are not."""
import torch

from gpu_helpers import GUARD, Guarded


def test_guard_detects_writes_outside_the_tensor():
    for dtype, shape in ((torch.bfloat16, (2, 3, 5, 64)), (torch.float32, (7, 128)), (torch.uint8, (33,))):
        g = Guarded(shape, dtype, device="cpu")
        assert g.t.shape == torch.Size(shape) and g.t.dtype == dtype
        g.t.fill_(1)
        assert g.intact()
        for pos in (GUARD - 1, GUARD + g.nbytes, 0, len(g.buf) - 1):
            h = Guarded(shape, dtype, device="cpu")
            h.t.fill_(1)
            h.buf[pos] = 0
            assert not h.intact(), (dtype, shape, pos)
        assert g.t.data_ptr() - g.buf.data_ptr() == GUARD and g.t.data_ptr() % 256 == g.buf.data_ptr() % 256
