"""Out-of-bounds writes, caught with guard bytes (the sanitizer tools are not
available here): every buffer a call writes -- the output, the workspace, the
fp32 sampled-row buffers, the decode output -- is placed inside a larger
allocation whose bytes before and after it hold a known pattern, and the
pattern must be intact after the call.  The inputs must be unchanged too
(except K, which the RoPE-fused prefill rotates in place by contract).
Shapes cover both sink + window kernels (one-CTA and two-CTA), ragged tails,
d = 64 and 128, gamma dividing 128 or not (the separate Delta pass), the
dense tail, smoothing, the three standalone entry points, row ranges and the
decode."""
import os

import pytest
import torch

from paper_2505_11254_gb300 import binding
from paper_2505_11254_gb300.flops import n_samples
from gpu_helpers import Guarded, guarded_ws, rand_qkv

pytestmark = pytest.mark.gpu


def kernel(pair):
    """DELTA_ATTN_PAIR for the block: '1' two-CTA wherever it applies, '0' one-CTA, None the library's choice."""
    class _K:
        def __enter__(self):
            self.old = os.environ.get("DELTA_ATTN_PAIR")
            if pair is None:
                os.environ.pop("DELTA_ATTN_PAIR", None)
            else:
                os.environ["DELTA_ATTN_PAIR"] = pair

        def __exit__(self, *exc):
            if self.old is None:
                os.environ.pop("DELTA_ATTN_PAIR", None)
            else:
                os.environ["DELTA_ATTN_PAIR"] = self.old
    return _K()


# (B, Hq, Hkv, N, d, n_sink, window, gamma)
SHAPES = [
    (2, 8, 2, 517, 128, 4, 100, 64),     # ragged, gamma divides 128
    (1, 4, 2, 1100, 128, 4, 600, 48),    # gamma 48: Delta in its own pass
    (1, 8, 8, 700, 64, 4, 300, 16),      # d = 64, GQA 1
    (1, 2, 1, 1, 128, 4, 512, 4),        # N = 1
    (1, 6, 2, 1300, 128, 17, 512, 3),    # GQA 3, 17 sinks, gamma 3
]


def _ids(c):
    return "B%d_H%d-%d_N%d_d%d_s%d_w%d_g%d" % c


@pytest.mark.parametrize("pair", ["0", "1"])
@pytest.mark.parametrize("shape", SHAPES, ids=_ids)
def test_prefill_writes_stay_in_bounds(shape, pair):
    B, Hq, Hkv, N, d, s, w, gamma = shape
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=sum(shape))
    q0, k0, v0 = q.clone(), k.clone(), v.clone()
    forms = [dict(), dict(mode="recompute"), dict(tail_dense=min(N, 77)), dict(smooth="linear")]
    for form in forms:
        o = Guarded((B, Hq, N, d), torch.bfloat16)
        ws = guarded_ws(binding.workspace_size(B, Hq, Hkv, N, d, s, w, gamma, form.get("mode", "delta"),
                                               form.get("tail_dense", 0), smooth=form.get("smooth", "none")))
        with kernel(pair):
            binding.delta_attn_prefill(q, k, v, s, w, gamma, out=o.t, workspace=ws.t, **form)
        assert binding.check() == binding.DA_OK
        assert o.intact(), "output guard overwritten (%s)" % form
        assert ws.intact(), "workspace guard overwritten (%s)" % form
        assert torch.isfinite(o.t.float()).all()
    assert torch.equal(q, q0) and torch.equal(k, k0) and torch.equal(v, v0)


@pytest.mark.parametrize("shape", SHAPES[:3], ids=_ids)
def test_standalone_writes_stay_in_bounds(shape):
    B, Hq, Hkv, N, d, s, w, gamma = shape
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=sum(shape) + 1)
    ns = n_samples(N, gamma)
    o = Guarded((B, Hq, N, d), torch.bfloat16)
    ss = Guarded((B, Hq, ns, d), torch.float32)
    ds = Guarded((B, Hq, ns, d), torch.float32)
    ws = guarded_ws(binding.strided_dense_workspace_size(B, Hq, Hkv, N, d, gamma))
    binding.sparse_window_attn(q, k, v, s, w, gamma, out=o.t, s_sampled=ss.t)
    binding.strided_dense_attn(q, k, v, gamma, out=ds.t, workspace=ws.t)
    o2 = Guarded((B, Hq, N, d), torch.bfloat16)
    binding.delta_apply(o.t, ss.t, ds.t, gamma, out=o2.t)
    assert binding.check() == binding.DA_OK
    for name, g in (("sparse rows", o), ("sampled sparse rows", ss), ("dense rows", ds), ("workspace", ws),
                    ("delta_apply output", o2)):
        assert g.intact(), "%s guard overwritten" % name


def test_row_range_and_decode_writes_stay_in_bounds():
    B, Hq, Hkv, N, d, s, w, gamma = 1, 8, 2, 2048, 128, 4, 300, 16
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=9)
    r0, n = 512, 768
    o = Guarded((B, Hq, n, d), torch.bfloat16)
    ws = guarded_ws(binding.workspace_size_rows(B, Hq, Hkv, N, d, s, w, gamma, r0, n))
    binding.delta_attn_prefill_rows(q[:, :, r0:r0 + n].contiguous(), k, v, s, w, gamma, r0, out=o.t, workspace=ws.t)
    assert binding.check() == binding.DA_OK
    assert o.intact() and ws.intact()
    qd = q[:, :, -1, :].contiguous()
    od = Guarded((B, Hq, d), torch.bfloat16)
    wsd = guarded_ws(binding.decode_workspace_size(B, Hq, Hkv, N, d))
    binding.decode(qd, k, v, out=od.t, workspace=wsd.t)
    assert binding.check() == binding.DA_OK
    assert od.intact() and wsd.intact()


def test_rope_prefill_writes_stay_in_bounds():
    B, Hq, Hkv, N, d, s, w, gamma = 1, 4, 2, 1500, 128, 4, 512, 64
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=10)
    table = binding.rope_table(N, d, 500000.0)
    kg = Guarded((B, Hkv, N, d), torch.bfloat16)
    kg.t.copy_(k)
    o = Guarded((B, Hq, N, d), torch.bfloat16)
    ws = guarded_ws(binding.workspace_size(B, Hq, Hkv, N, d, s, w, gamma))
    binding.delta_attn_prefill_rope(q, kg.t, v, s, w, gamma, table, out=o.t, workspace=ws.t)
    assert binding.check() == binding.DA_OK
    assert kg.intact() and o.intact() and ws.intact()
