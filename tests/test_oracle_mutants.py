"""Every planted mistake in the oracle (ORACLE_MUTANT=n builds) fails a pin.

The mistakes are planted in the oracle, on the CPU, at compile time:
1 sqrt(G + eps) in the denominator, 2 the step uses the old state,
3 wrong sign of the step, 4 one step per occurrence, 5 earlier occurrences
dropped from the sum, 6 first Put occurrence wins, 7 init drops lo,
8 dedup reports last positions, 9 state_init ignored, 10 a new key is
inserted once per occurrence, 11 import drops the state.
"""
import pytest

import oracle
import oracle_pins

MUTANTS = list(range(1, 12))


@pytest.mark.parametrize("mutant", MUTANTS)
def test_mutant_is_caught(mutant, tmp_path):
    lib = oracle.load(mutant=mutant, out_dir=str(tmp_path))
    assert lib.oracle_mutant() == mutant
    failed = []
    for check in oracle_pins.ALL_CHECKS:
        try:
            check(lib)
        except AssertionError:
            failed.append(check.__name__)
        except Exception as e:  # NaN / overflow paths also count as caught
            failed.append(f"{check.__name__}:{type(e).__name__}")
    assert failed, f"mutant {mutant} passed every pin"
