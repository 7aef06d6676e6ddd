"""Pins of the oracle's binary16 rounding against numpy's IEEE float16 conversion.

The row/column scales and the pivot values are stored in FP16 (App. C.3 step 6,
App. D); the oracle rounds to binary16 from the format's definition.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def test_fp16_round_matches_numpy(oracle, rng):
    mags = 10.0 ** rng.uniform(-9, np.log10(65000), size=4000)
    xs = mags * rng.choice([-1.0, 1.0], size=mags.size)
    # exact ties between binary16 neighbours (round half to even)
    ties = (np.arange(1, 400, dtype=np.float64) + 0.5) * 2.0 ** -10
    for x in np.concatenate([xs, ties, -ties, [0.0, 2.0 ** -24, 2.0 ** -25, 3 * 2.0 ** -26]]):
        assert oracle.fp16_round(x) == float(np.float16(x)), x


def test_fp16_saturates(oracle):
    for x in (65504.0, 65519.0, 65520.0, 1e6, 3.4e38):
        assert oracle.fp16_round(x) == 65504.0
        assert oracle.fp16_round(-x) == -65504.0


def test_fp16_encode_decode_all_patterns(oracle):
    for h in range(0, 1 << 16, 7):
        v = np.array([h], np.uint16).view(np.float16)[0]
        if not np.isfinite(v):
            continue
        assert oracle.fp16_decode(h) == float(v)
        if h != 0x8000:
            assert oracle.fp16_encode(float(v)) == h
