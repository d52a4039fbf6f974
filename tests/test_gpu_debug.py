"""Bit-exact checks of the kernels' visibility predicate, row -> sample map and
work decomposition (debug dumps of the same device code the kernels run)."""
import numpy as np
import pytest

from paper_2505_11254_gb300 import binding
from paper_2505_11254_gb300.flops import n_samples

pytestmark = pytest.mark.gpu


def _w_set(i, n_sink, window):
    return {j for j in range(i + 1) if j < n_sink or j > i - window}


@pytest.mark.parametrize("N,n_sink,window", [(200, 4, 16), (130, 0, 1), (64, 70, 3), (300, 2, 300)])
def test_mask_bit_exact(N, n_sink, window):
    m = binding.debug_mask(N, n_sink, window, 0, N).cpu().numpy()
    for i in range(N):
        want = np.zeros(N, np.uint8)
        want[list(_w_set(i, n_sink, window))] = 1
        assert np.array_equal(m[i], want), i


@pytest.mark.parametrize("N,gamma", [(1000, 64), (257, 1), (100, 3), (5, 128)])
def test_rowmap_bit_exact(N, gamma):
    rows, sampled = binding.debug_rowmap(N, gamma)
    rows, sampled = rows.cpu().numpy(), sampled.cpu().numpy()
    i = np.arange(N)
    assert np.array_equal(rows, (i // gamma) * gamma)
    assert np.array_equal(sampled, (i % gamma == 0).astype(np.uint8))


SHAPES = [(1, 4, 1, 1000, 128, 4, 200, 16), (2, 8, 2, 3000, 64, 3, 256, 64), (1, 2, 2, 777, 128, 0, 64, 5),
          (1, 32, 8, 32768, 128, 4, 2048, 64)]


@pytest.mark.parametrize("shape", SHAPES)
def test_sparse_tiles_cover_exactly_the_sparse_set(shape):
    B, Hq, Hkv, N, d, s, w, gamma = shape
    info = binding.plan_info(*shape)
    idx = sorted({0, 1, info["ctas_sparse"] // 2, info["ctas_sparse"] - 1})
    for index in idx:
        wk = binding.debug_work(0, *shape, index)
        rows = [r for (r, _, _, ok) in wk["lanes"] if ok]
        need = set()
        for i in rows:
            need |= {j // 128 for j in _w_set(i, s, w)} if N <= 4000 else set()
        tiles = [t for t, _ in wk["tiles"]]
        assert len(tiles) == len(set(tiles)), "a key tile is visited twice"
        if N <= 4000:
            assert need <= set(tiles), "a visible key is never visited"
        for t, masked in wk["tiles"]:
            if not masked:  # every (row, key) pair of an unmasked tile is visible
                lo, hi = t * 128, t * 128 + 127
                assert hi <= min(rows) and lo > max(rows) - w


@pytest.mark.parametrize("shape", SHAPES + [(1, 32, 8, 131072, 128, 4, 2048, 64)])
def test_dense_units_partition_the_causal_range(shape):
    """The device decode of the split-K units: each M-tile's chunks tile its
    causal key range [0, last causal key] exactly once, split M-tiles' chunks
    hold distinct partial slots and share one ticket (checked for every M-tile
    whose chunks are all among the units read: all units up to 6000)."""
    B, Hq, Hkv, N, d, s, w, gamma = shape
    info = binding.plan_info(*shape)
    ns = n_samples(N, gamma)
    chunks, slots, tickets = {}, set(), {}
    for u in range(min(info["ctas_dense"], 6000)):
        wk = binding.debug_work(1, *shape, u)
        key = (wk["b"], wk["h0"], wk["r0"])
        tiles = [t for t, _ in wk["tiles"]]
        assert wk["chunk_idx"] not in chunks.setdefault(key, {}), "a chunk is held twice"
        chunks[key][wk["chunk_idx"]] = (wk["n_chunks"], tiles)
        if wk["n_chunks"] > 1:
            assert 0 <= wk["slot"] < info["split_units"] and wk["slot"] not in slots, "partial slot"
            slots.add(wk["slot"])
            assert tickets.setdefault(key, wk["ticket"]) == wk["ticket"], "one ticket per M-tile"
        lanes = [(row, smp, h) for (row, smp, h, ok) in wk["lanes"] if ok]
        assert lanes and max(r for r, _, _ in lanes) <= (ns - 1) * gamma
        assert all(r == smp * gamma for r, smp, _ in lanes)
        for t, masked in wk["tiles"]:
            if not masked:
                assert t * 128 + 127 <= min(r for r, _, _ in lanes)
    R = info["samples_per_head"]
    complete = 0
    for (b, h0, k0), got in chunks.items():
        n_chunks = next(iter(got.values()))[0]
        if len(got) < n_chunks:
            continue  # some of its units were not read
        complete += 1
        tiles = sorted(t for c in got.values() for t in c[1])
        k_last = min(k0 + R - 1, ns - 1)
        assert tiles == list(range(k_last * gamma // 128 + 1))
    assert complete > 0
    assert len(set(tickets.values())) == len(tickets), "M-tiles share a ticket"
