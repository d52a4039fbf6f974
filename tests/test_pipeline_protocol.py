"""The attention kernel's barrier protocol, run as an executable model over
random interleavings (`pipeline_model.py`): no parity wait may pass on the
wrong phase, no buffer may be refilled before its reader is done, and every
interleaving must finish.  Covered: the sink + window layout at d = 128 and
d = 64 (one or two Q buffers), with and without the RoPE rotation of each Q
tile, and the strided dense pass (the same layout, items through the queue).
Item lengths include one- and two-tile items and the long items of wide
windows, so the ring and buffer indices wrap at every offset.  Deliberately
broken protocols (a dropped wait each) must be caught, which shows that the
model sees what it is meant to.  The decode kernel's K/V ring is checked the
same way: the deployed eight- and four-stage rings over four consumer warps
pass, a six-stage ring (stages shared between warps) must be flagged.  The
two-CTA sink + window kernel (two heads of a row tile in a CTA pair, the
leader issuing every MMA) is modelled with both CTAs' roles; its mutants
drop one CTA's share of a barrier."""
import random

import pytest

from pipeline_model import MUTANTS, PAIR_MUTANTS, Layout, ModelError, run, run_decode_ring, run_pair

LAYOUTS = {
    "sink_window_d128": Layout(dense=False, nq=1),
    "sink_window_d64": Layout(dense=False, nq=2, nk=4, nv=4),
    "sink_window_d128_rope": Layout(dense=False, nq=1, rope=True),
    "sink_window_d64_rope": Layout(dense=False, nq=2, nk=4, nv=4, rope=True),
    "strided_dense_d128": Layout(dense=True),
    "strided_dense_d64": Layout(dense=True, nq=2, nk=4, nv=4),
    "strided_dense_d128_rope": Layout(dense=True, rope=True),
}


def _items(rnd):
    return [rnd.choice([1, 1, 2, 3, 4, 5, 6, 7, 18]) for _ in range(rnd.randint(0, 9))]


@pytest.mark.parametrize("name", sorted(LAYOUTS))
def test_protocol_holds_over_random_interleavings(name):
    rnd = random.Random(hash(name) & 0xffff)
    for r in range(300):
        tiles = _items(rnd)
        try:
            run(LAYOUTS[name], tiles, seed=r)
        except ModelError as e:
            pytest.fail("%s, items %s, seed %d: %s" % (name, tiles, r, e))


@pytest.mark.parametrize("mutant", MUTANTS)
def test_a_dropped_wait_is_caught(mutant):
    layouts = ([LAYOUTS["strided_dense_d128"], LAYOUTS["sink_window_d128"]] if mutant == "q_no_free_wait"
               else [LAYOUTS["sink_window_d128"], LAYOUTS["strided_dense_d128"]])
    rnd = random.Random(7)
    for r in range(400):
        tiles = _items(rnd) + [18, 3]
        for lay in layouts:
            try:
                run(lay, tiles, seed=r, mutant=mutant)
            except ModelError:
                return
    pytest.fail("mutant %s was not caught" % mutant)


@pytest.mark.parametrize("stages, warps", [(8, 4), (4, 4)])
def test_decode_ring_holds(stages, warps):
    rnd = random.Random(stages * 31 + warps)
    for r in range(500):
        n = rnd.randint(0, 40)
        try:
            run_decode_ring(n, stages, warps, seed=r)
        except ModelError as e:
            pytest.fail("%d stages, %d warps, %d chunks, seed %d: %s" % (stages, warps, n, r, e))


def test_decode_ring_with_shared_stages_is_caught():
    """Six stages over four warps: a stage's phases alternate between warps,
    so a parity wait can pass on a phase two behind."""
    rnd = random.Random(3)
    for r in range(500):
        try:
            run_decode_ring(rnd.randint(8, 40), 6, 4, seed=r)
        except ModelError:
            return
    pytest.fail("the shared-stage ring was not caught")


PAIR_LAYOUTS = {  # deployed: two Q buffers, five K and four V slots (of half tiles)
    "pair_sink_window_d128": Layout(dense=False, nq=2, nk=5, nv=4),
    "pair_sink_window_d128_rope": Layout(dense=False, nq=2, nk=5, nv=4, rope=True),
    "pair_sink_window_d128_nq1": Layout(dense=False, nq=1, nk=6, nv=5),
}


@pytest.mark.parametrize("name", sorted(PAIR_LAYOUTS))
def test_pair_protocol_holds_over_random_interleavings(name):
    rnd = random.Random(hash(name) & 0xffff)
    for r in range(300):
        tiles = _items(rnd)
        try:
            run_pair(PAIR_LAYOUTS[name], tiles, seed=r)
        except ModelError as e:
            pytest.fail("%s, items %s, seed %d: %s" % (name, tiles, r, e))


@pytest.mark.parametrize("mutant", PAIR_MUTANTS)
def test_pair_mutant_is_caught(mutant):
    rnd = random.Random(11)
    for r in range(400):
        tiles = _items(rnd) + [18, 3]
        for lay in (PAIR_LAYOUTS["pair_sink_window_d128"], PAIR_LAYOUTS["pair_sink_window_d128_rope"]):
            try:
                run_pair(lay, tiles, seed=r, mutant=mutant)
            except ModelError:
                return
    pytest.fail("mutant %s was not caught" % mutant)
