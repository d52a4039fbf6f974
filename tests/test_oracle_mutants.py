"""Each deliberately broken build of the oracle must fail at least one pin.

The mutants (ORACLE_MUTANT=n in oracle/delta_oracle.c) plant plausible
mistakes: an off-by-one sink bound, a window one key too wide, the wrong GQA
head mapping, a dropped 1/sqrt(d), a flipped Delta sign, the dense row taken
over the sparse set, Delta taken against the current row instead of the
sample, a transposed K operand, and three smoothing slips (EMA weights
swapped, the filter's velocity gain replaced by its position gain, the
interpolation weight one row ahead), and a decode that leaves out the new
token's own key, a RoPE rotation in the wrong direction, and Lemma 1's
bound taken with the largest |v_j| over every causal key instead of W(i).
All of this runs on the CPU.
"""
import os
import tempfile

import pytest

from oracle import build as obuild
import oracle_pins as P

MUTANTS = {
    1: "sink bound j <= n_sink",
    2: "window one key too wide",
    3: "GQA head h % Hkv",
    4: "dropped 1/sqrt(d)",
    5: "Delta sign flipped",
    6: "dense row over the sparse set",
    7: "Delta against row i instead of its sample",
    8: "K read transposed",
    9: "EMA weights swapped",
    10: "filter velocity corrected with alpha",
    11: "linear interpolation weight one row ahead",
    12: "decode without the new token's own key",
    13: "RoPE rotation in the wrong direction",
    14: "Lemma 1 bound with the max |v| over every causal key",
}

_tmp = tempfile.mkdtemp(prefix="oracle_mutants_")


@pytest.mark.parametrize("m", sorted(MUTANTS), ids=lambda m: MUTANTS[m])
def test_mutant_is_caught(m):
    lib = obuild.build(force=True, extra_flags=("-DORACLE_MUTANT=%d" % m,),
                       out=os.path.join(_tmp, "liboracle_m%d.so" % m))
    caught = []
    for pin in P.ALL_PINS:
        try:
            pin(lib=lib)
        except AssertionError:
            caught.append(pin.__name__)
    assert caught, "mutant %d (%s) passed every pin" % (m, MUTANTS[m])
