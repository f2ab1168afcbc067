"""Each planted mistake in the oracle (compiled with -DORACLE_MUTANT=n) must be
caught by at least one pin, so the pins constrain every step of the scorer."""
import pytest

from tests import oracle_pins as P

MUTANTS = {
    1: "verify token ignores its own key/value",
    2: "RoPE rotates the wrong way",
    3: "interleaved instead of contiguous query-head groups",
    4: "scores not scaled by 1/sqrt(hd)",
    5: "output projection transposed",
    6: "feed-forward output replaces the residual",
    7: "P(+) read from the '-' entry",
    8: "verify token placed at position L-1",
    9: "RMSNorm without eps",
    10: "gate not passed through SiLU",
    12: "all query heads read kv head 0",
    14: "gate and up exchanged",
    15: "adapter scale left out",
    16: "adapter term subtracted",
    17: "a verify token of a depth-k readout also sees the tokens after it",
    18: "q/k norm applied after RoPE",
    19: "the key norm takes the query norm's gain",
    21: "gradient: softmax backward without its -D term",
    22: "gradient: RoPE backward rotated the wrong way",
    23: "gradient: RMSNorm backward without its second term",
}


@pytest.mark.parametrize("mutant", sorted(MUTANTS))
def test_mutant_is_caught(mutant):
    caught = []
    for pin in P.ALL_PINS:
        try:
            pin(mutant)
        except AssertionError:
            caught.append(pin.__name__)
    assert caught, f"planted mistake {mutant} ({MUTANTS[mutant]}) passed every pin"
