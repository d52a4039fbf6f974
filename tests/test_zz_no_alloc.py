"""strided_dense_attn_noalloc, the entry point for callers that cannot
allocate device memory, against strided_dense_attn on the same inputs, on
calls in a row, and the proof that its calls allocate nothing: the device's
free memory and the default memory pool (where stream-ordered allocations
come from) are unchanged across a call, including the pool's high-water mark,
which a transient allocation freed within the call would still raise.
Collected last: a failure here leaves every other test run."""
import ctypes

import pytest
import torch

from paper_2505_11254_gb300 import binding
from gpu_helpers import assert_close, rand_qkv

pytestmark = pytest.mark.gpu

# CUmemPool_attribute values (cuda.h)
_RESERVED_CURRENT, _USED_CURRENT, _USED_HIGH = 5, 7, 8


class _DefaultPool:
    """The current device's default memory pool, read through the driver API."""

    def __init__(self):
        self.cuda = ctypes.CDLL("libcuda.so.1")
        dev = ctypes.c_int()
        assert self.cuda.cuDeviceGet(ctypes.byref(dev), torch.cuda.current_device()) == 0
        self.pool = ctypes.c_void_p()
        assert self.cuda.cuDeviceGetDefaultMemPool(ctypes.byref(self.pool), dev) == 0

    def get(self, attr):
        v = ctypes.c_uint64()
        assert self.cuda.cuMemPoolGetAttribute(self.pool, attr, ctypes.byref(v)) == 0
        return v.value

    def reset_high(self):
        zero = ctypes.c_uint64(0)
        assert self.cuda.cuMemPoolSetAttribute(self.pool, _USED_HIGH, ctypes.byref(zero)) == 0


@pytest.mark.parametrize("d", [128, 64])
def test_noalloc_matches_workspace_entry_point_twice(d):
    B, Hq, Hkv, N, gamma = 1, 8, 2, 8192, 16
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=11 + d)
    info = binding.plan_info(B, Hq, Hkv, N, d, 4, 256, gamma)
    assert info["split_units"] > 0, "the shape must use the split-K scratch"
    ref = binding.strided_dense_attn(q, k, v, gamma)
    torch.cuda.synchronize()
    outs = [torch.full_like(ref, float("nan")) for _ in range(3)]
    pool = _DefaultPool()
    # Call 0 may load the library's code and data onto the device (lazy module
    # loading by the CUDA runtime, which places the fixed scratch); calls 1
    # and 2 must then leave every allocation as it was.
    for call in range(3):
        torch.cuda.synchronize()
        pool.reset_high()
        free0 = torch.cuda.mem_get_info()[0]
        used0, reserved0 = pool.get(_USED_CURRENT), pool.get(_RESERVED_CURRENT)
        binding.strided_dense_attn_noalloc(q, k, v, gamma, out=outs[call])
        assert binding.check() == binding.DA_OK
        if call > 0:
            assert torch.cuda.mem_get_info()[0] == free0, "device memory changed across the call"
            assert pool.get(_USED_HIGH) <= used0 and pool.get(_RESERVED_CURRENT) == reserved0, \
                "the call allocated from the default pool"
        assert_close(outs[call], ref.double().cpu().numpy(), "no-alloc call %d (d=%d)" % (call, d))


def test_noalloc_rejects_shapes_beyond_its_scratch():
    # The 32K-token Llama-3-8B-shaped layer splits its dense rows into more
    # partials than the 16 MiB scratch holds; the check runs before anything
    # is launched, so the pointers are never read.
    need = binding.strided_dense_workspace_size(1, 32, 8, 32768, 128, 64)
    assert need > (16 << 20)
    fake = ctypes.c_void_p(1 << 20)
    rc = binding.load().strided_dense_attn_noalloc(fake, fake, fake, fake, 1, 32, 8, 32768, 128, 64, None)
    assert rc == binding.DA_ERR_WORKSPACE
