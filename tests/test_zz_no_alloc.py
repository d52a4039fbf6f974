"""strided_dense_attn_noalloc, the entry point for callers that cannot
allocate device memory, against strided_dense_attn on the same inputs, on two
calls in a row.  Collected last: a failure here leaves every other test run."""
import ctypes

import pytest
import torch

from paper_2505_11254_gb300 import binding
from gpu_helpers import assert_close, rand_qkv

pytestmark = pytest.mark.gpu


def test_noalloc_matches_workspace_entry_point_twice():
    B, Hq, Hkv, N, d, gamma = 1, 8, 2, 8192, 128, 16
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=11)
    info = binding.plan_info(B, Hq, Hkv, N, d, 4, 256, gamma)
    assert info["split_units"] > 0, "the shape must use the split-K scratch"
    ref = binding.strided_dense_attn(q, k, v, gamma)
    torch.cuda.synchronize()
    for call in range(2):
        out = torch.full_like(ref, float("nan"))
        binding.strided_dense_attn_noalloc(q, k, v, gamma, out=out)
        assert binding.check() == binding.DA_OK
        assert_close(out, ref.double().cpu().numpy(), "no-alloc call %d" % call)


def test_noalloc_rejects_shapes_beyond_its_scratch():
    # The 32K-token Llama-3-8B-shaped layer splits its dense rows into more
    # partials than the 16 MiB scratch holds; the check runs before anything
    # is launched, so the pointers are never read.
    need = binding.strided_dense_workspace_size(1, 32, 8, 32768, 128, 64)
    assert need > (16 << 20)
    fake = ctypes.c_void_p(1 << 20)
    rc = binding.load().strided_dense_attn_noalloc(fake, fake, fake, fake, 1, 32, 8, 32768, 128, 64, None)
    assert rc == binding.DA_ERR_WORKSPACE
