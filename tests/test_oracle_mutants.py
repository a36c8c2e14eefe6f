"""Each planted mistake in the oracle (OR_MUTANT = n) must fail at least one pin.

The mistakes are the plausible ones: a transposed operand, a wrong RoPE sign or pairing,
a missing scale, residual or epsilon, a wrong GQA index, a dropped term, an off-by-one
position, embedding row or tree parent, a swapped concat or gate/up, a broken tie rule.
"""
import pytest

import oracle
import oracle_pins as pins

MUTANTS = [m for m in range(1, oracle.N_MUTANTS + 1) if m not in oracle._UNUSED_MUTANTS]


@pytest.fixture(scope="module")
def mutant_dir(tmp_path_factory):
    return str(tmp_path_factory.mktemp("mutants"))


@pytest.mark.parametrize("mutant", MUTANTS)
def test_mutant_is_caught(mutant, mutant_dir):
    orc = oracle.load(mutant, mutant_dir)
    caught = []
    for pin in pins.ALL_PINS:
        try:
            pin(orc)
        except AssertionError:
            caught.append(pin.__name__)
        except Exception as e:  # a crash-free mistake that raises elsewhere also counts
            caught.append(f"{pin.__name__}:{type(e).__name__}")
    assert caught, f"planted mistake {mutant} passed every pin"
