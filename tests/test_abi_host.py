"""The C-ABI library builds, loads, exports every declared entry point and
rejects bad arguments on the host, before touching a GPU (CPU only)."""
import ctypes
import os
import re

import pytest

from paper_2505_11254_gb300 import binding

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "delta_attn.h")


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(\w+)\s*\(", text, flags=re.M)))


def test_library_exports_every_declared_symbol():
    lib = binding.load()
    names = _declared()
    assert len(names) >= 13
    for name in names:
        assert hasattr(lib, name), name
    assert set(names) == set(binding._SIGNATURES), "binding and header disagree"


def test_status_strings():
    for code in range(-6, 1):
        assert binding.status_string(code) not in ("", "unknown status")
    assert binding.status_string(42) == "unknown status"


_FAKE = 0x10000  # never dereferenced: validation fails first


def _prefill(**kw):
    a = dict(Q=_FAKE, K=_FAKE, V=_FAKE, O=_FAKE, B=1, Hq=4, Hkv=2, N=256, d=128, n_sink=4, window=64, gamma=16,
             ws=None, ws_bytes=0, stream=None)
    a.update(kw)
    return binding.load().delta_attn_prefill(a["Q"], a["K"], a["V"], a["O"], a["B"], a["Hq"], a["Hkv"], a["N"],
                                             a["d"], a["n_sink"], a["window"], a["gamma"], a["ws"],
                                             a["ws_bytes"], a["stream"])


@pytest.mark.parametrize("kw,status", [
    (dict(Q=None), binding.DA_ERR_INVALID_ARG),
    (dict(O=None), binding.DA_ERR_INVALID_ARG),
    (dict(Hq=3, Hkv=2), binding.DA_ERR_INVALID_ARG),
    (dict(N=0), binding.DA_ERR_INVALID_ARG),
    (dict(gamma=0), binding.DA_ERR_INVALID_ARG),
    (dict(window=0), binding.DA_ERR_INVALID_ARG),
    (dict(n_sink=-1), binding.DA_ERR_INVALID_ARG),
    (dict(B=0), binding.DA_ERR_INVALID_ARG),
    (dict(N=1 << 31), binding.DA_ERR_INVALID_ARG),
    (dict(d=96), binding.DA_ERR_UNSUPPORTED),
    (dict(d=256), binding.DA_ERR_UNSUPPORTED),
    (dict(K=_FAKE + 8), binding.DA_ERR_MISALIGNED),
    (dict(O=_FAKE + 2), binding.DA_ERR_MISALIGNED),
    (dict(ws=_FAKE + 4, ws_bytes=1 << 20), binding.DA_ERR_MISALIGNED),
])
def test_prefill_rejects_bad_arguments(kw, status):
    assert _prefill(**kw) == status


def test_other_entry_points_reject_bad_arguments():
    lib = binding.load()
    assert lib.sparse_window_attn(None, _FAKE, _FAKE, _FAKE, None, 1, 2, 2, 64, 64, 0, 8, 4, None) == \
        binding.DA_ERR_INVALID_ARG
    assert lib.sparse_window_attn(_FAKE, _FAKE, _FAKE, _FAKE, _FAKE + 4, 1, 2, 2, 64, 64, 0, 8, 4, None) == \
        binding.DA_ERR_MISALIGNED
    assert lib.strided_dense_attn(_FAKE, _FAKE, _FAKE, None, 1, 2, 2, 64, 64, 4, None, 0, None) == \
        binding.DA_ERR_INVALID_ARG
    assert lib.strided_dense_attn(_FAKE, _FAKE, _FAKE, _FAKE, 1, 2, 2, 64, 80, 4, None, 0, None) == \
        binding.DA_ERR_UNSUPPORTED
    assert lib.delta_apply(_FAKE, None, None, _FAKE, 1, 2, 64, 64, 4, None) == binding.DA_ERR_INVALID_ARG
    assert lib.delta_apply(_FAKE, None, _FAKE, _FAKE, 1, 2, 64, 64, 0, None) == binding.DA_ERR_INVALID_ARG
    assert lib.delta_attn_debug_mask(64, 0, 8, 10, 5, _FAKE, None) == binding.DA_ERR_INVALID_ARG
    assert lib.delta_attn_debug_timeout(0, None) == binding.DA_ERR_INVALID_ARG
    assert lib.delta_attn_debug_timeout(2_000_000_000, None) == binding.DA_ERR_INVALID_ARG
    sz = ctypes.c_size_t(0)
    assert lib.delta_attn_workspace_size(1, 2, 2, 64, 64, 0, 8, 0, ctypes.byref(sz)) == binding.DA_ERR_INVALID_ARG
    assert lib.delta_attn_workspace_size(1, 2, 2, 64, 64, 0, 8, 4, None) == binding.DA_ERR_INVALID_ARG


@pytest.mark.parametrize("mode,tail", [(2, 0), (-1, 0), (0, -1), (1, 257), (0, 1 << 40)])
def test_prefill_ex_rejects_bad_mode_and_tail(mode, tail):
    """Unknown output modes and dense tails outside [0, N] are rejected before
    any device call (N = 256 here)."""
    lib = binding.load()
    assert lib.delta_attn_prefill_ex(_FAKE, _FAKE, _FAKE, _FAKE, 1, 4, 2, 256, 128, 4, 64, 16, mode, tail, None, 0,
                                     None) == binding.DA_ERR_INVALID_ARG
    sz = ctypes.c_size_t(0)
    assert lib.delta_attn_workspace_size_ex(1, 4, 2, 256, 128, 4, 64, 16, mode, tail, ctypes.byref(sz)) == \
        binding.DA_ERR_INVALID_ARG


def test_decode_rejects_bad_arguments():
    """Eq. 2 decode: NULL or misaligned pointers, L < max_keys, max_keys < 1,
    Hq % Hkv != 0, G > 16 and an unsupported head dimension are rejected
    before any device call."""
    lib = binding.load()
    ok = dict(q=_FAKE, K=_FAKE, V=_FAKE, lens=None, O=_FAKE, B=1, Hq=8, Hkv=2, L=100, mk=100, d=128)

    def call(**kw):
        a = dict(ok)
        a.update(kw)
        return lib.delta_attn_decode(a["q"], a["K"], a["V"], a["lens"], a["O"], a["B"], a["Hq"], a["Hkv"], a["L"],
                                     a["mk"], a["d"], None, 0, None)
    assert call(q=None) == binding.DA_ERR_INVALID_ARG
    assert call(L=50) == binding.DA_ERR_INVALID_ARG
    assert call(mk=0) == binding.DA_ERR_INVALID_ARG
    assert call(Hq=7) == binding.DA_ERR_INVALID_ARG
    assert call(Hq=34, Hkv=2) == binding.DA_ERR_UNSUPPORTED
    assert call(d=96) == binding.DA_ERR_UNSUPPORTED
    assert call(K=_FAKE + 8) == binding.DA_ERR_MISALIGNED
    assert call(lens=_FAKE + 4) == binding.DA_ERR_MISALIGNED
    sz = ctypes.c_size_t(0)
    assert lib.delta_attn_decode_workspace_size(1, 8, 2, 0, 128, ctypes.byref(sz)) == binding.DA_ERR_INVALID_ARG
