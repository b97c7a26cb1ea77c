"""Pins of the oracle's fp32 -> bf16 round-to-nearest-even (CPU only).

Independent checks: torch's CPU conversion (a separate implementation) on
every non-NaN pattern of a structured set that covers all rounding cases of
every exponent, a nearest-value search in float64 that restates IEEE RNE as
"the closest bf16 value, ties to the even mantissa", and hand cases. Planted
mistakes in the oracle (ties away from zero, truncation, a dropped sign)
must fail the same checks.
"""
import numpy as np
import pytest
import torch

from oracle import cast as ocast


def structured_patterns(seed=0):
    g = np.random.default_rng(seed)
    hi_all = np.arange(1 << 16, dtype=np.uint32)
    lows = np.array([0, 1, 0x7FFF, 0x8000, 0x8001, 0xFFFF, 0x4000, 0xC000], dtype=np.uint32)
    lows = np.concatenate([lows, g.integers(0, 1 << 16, 24).astype(np.uint32)])
    a = ((hi_all[:, None] << 16) | lows[None, :]).reshape(-1)
    his = np.array([0x0000, 0x0001, 0x007F, 0x0080, 0x00FF, 0x3F80, 0x3F81, 0x3FFF, 0x7F7E, 0x7F7F,
                    0x7F80, 0x7FFF, 0x8000, 0x8001, 0x80FF, 0xBF80, 0xBF81, 0xFF7F, 0xFF80, 0xFFFF], dtype=np.uint32)
    his = np.concatenate([his, g.integers(0, 1 << 16, 44).astype(np.uint32)])
    b = ((his[:, None] << 16) | np.arange(1 << 16, dtype=np.uint32)[None, :]).reshape(-1)
    return np.concatenate([a, b])


def is_nan_pattern(u):
    return ((u >> 23) & 0xFF == 0xFF) & (u & 0x7FFFFF != 0)


def torch_bf16_bits(u):
    t = torch.from_numpy(u.view(np.int32).copy()).view(torch.float32).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def nearest_bf16_bits(u):
    """RNE restated as a value search: candidates are the bf16 values on both
    sides of x; pick the closer one, the even mantissa on a tie; a result past
    the largest finite value is infinity."""
    u = np.asarray(u, np.uint32)
    x = u.view(np.float32).astype(np.float64)
    lo_bits = (u >> 16).astype(np.uint32)
    hi_bits = lo_bits + 1
    lo_val = (lo_bits << 16).view(np.float32).astype(np.float64)
    mag_hi = hi_bits & 0x7FFF
    with np.errstate(over="ignore", invalid="ignore"):
        hi_val = (hi_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    # the pattern after the largest finite one is infinity: its place on the
    # unbounded-exponent scale is 2**128
    sgn = np.where(u >> 31 == 1, -1.0, 1.0)
    hi_val = np.where(mag_hi == 0x7F80, sgn * 2.0 ** 128, hi_val)
    d_lo = np.abs(x - lo_val)
    d_hi = np.abs(hi_val - x)
    pick_hi = (d_hi < d_lo) | ((d_hi == d_lo) & (lo_bits & 1 == 1))
    return np.where(pick_hi, hi_bits, lo_bits).astype(np.uint16)


def check_against_torch(fn, u):
    keep = ~is_nan_pattern(u)
    return np.array_equal(fn(u[keep]), torch_bf16_bits(u[keep]))


def check_against_search(fn, u):
    u = u[~is_nan_pattern(u)]
    u = u[((u >> 23) & 0xFF) != 0xFF]  # finite inputs
    return np.array_equal(fn(u), nearest_bf16_bits(u))


def check_nan(fn):
    g = np.random.default_rng(3)
    man = np.concatenate([np.array([1, 0x400000, 0x7FFFFF, 0x3FFFFF], np.uint32),
                          g.integers(1, 1 << 23, 2000).astype(np.uint32)])
    u = np.concatenate([0x7F800000 | man, 0xFF800000 | man]).astype(np.uint32)
    want = np.where(u >> 31 == 1, 0xFFC0, 0x7FC0).astype(np.uint16)
    return np.array_equal(fn(u), want)


HAND = [
    (0x3F800000, 0x3F80),  # 1.0 exact
    (0x3F808000, 0x3F80),  # tie, last kept bit even -> down
    (0x3F818000, 0x3F82),  # tie, last kept bit odd -> up
    (0x3F808001, 0x3F81),  # just above the tie
    (0x3F807FFF, 0x3F80),  # just below the tie
    (0xBF808001, 0xBF81),  # negative, magnitude rounds up
    (0x7F7FFFFF, 0x7F80),  # largest finite fp32 overflows to +inf
    (0x7F7F7FFF, 0x7F7F),  # stays at the largest finite bf16
    (0x7F7F8000, 0x7F80),  # tie at the top, odd -> inf
    (0x7F800000, 0x7F80),  # +inf
    (0xFF800000, 0xFF80),  # -inf
    (0x00000000, 0x0000),
    (0x80000000, 0x8000),  # -0 keeps its sign
    (0x00008000, 0x0000),  # subnormal tie to even zero
    (0x00018000, 0x0002),  # subnormal tie, odd -> up
    (0x00010001, 0x0001),  # subnormal, no flush to zero
    (0x007FFFFF, 0x0080),  # largest subnormal rounds to the smallest normal
    (0x7FC00000, 0x7FC0),  # quiet NaN
    (0x7F800001, 0x7FC0),  # signalling NaN -> quiet
    (0xFFFFFFFF, 0xFFC0),  # negative NaN keeps its sign
]


def check_hand(fn):
    u = np.array([a for a, _ in HAND], np.uint32)
    want = np.array([b for _, b in HAND], np.uint16)
    return np.array_equal(fn(u), want)


def test_hand_cases():
    assert check_hand(ocast.f32_bits_to_bf16_bits)


def test_structured_vs_torch():
    assert check_against_torch(ocast.f32_bits_to_bf16_bits, structured_patterns())


def test_random_vs_torch_and_value_search():
    g = np.random.default_rng(11)
    u = g.integers(0, 1 << 32, 1 << 21, dtype=np.uint64).astype(np.uint32)
    assert check_against_torch(ocast.f32_bits_to_bf16_bits, u)
    assert check_against_search(ocast.f32_bits_to_bf16_bits, u)


def test_structured_vs_value_search():
    assert check_against_search(ocast.f32_bits_to_bf16_bits, structured_patterns(1))


def test_nan_rule():
    assert check_nan(ocast.f32_bits_to_bf16_bits)


def test_bytes_wrapper_roundtrip():
    g = np.random.default_rng(5)
    x = g.standard_normal(1001).astype(np.float32)
    out = ocast.cast_bytes_f32_to_bf16(x.view(np.uint8))
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint8)
    assert np.array_equal(out, want)
    with pytest.raises(ValueError):
        ocast.cast_bytes_f32_to_bf16(np.zeros(6, np.uint8))


# -- planted mistakes: each must fail at least one of the checks above ----------

def _mut_ties_away(u):
    u = np.asarray(u, np.uint32).astype(np.uint64)
    nan = is_nan_pattern(u.astype(np.uint32))
    r = (u + 0x8000) >> 16
    return np.where(nan, 0x7FC0 | ((u >> 31) << 15), r).astype(np.uint16)


def _mut_truncate(u):
    u = np.asarray(u, np.uint32)
    nan = is_nan_pattern(u)
    return np.where(nan, 0x7FC0 | ((u >> 31) << 15), u >> 16).astype(np.uint16)


def _mut_nan_drops_sign(u):
    out = ocast.f32_bits_to_bf16_bits(u)
    u = np.asarray(u, np.uint32)
    return np.where(is_nan_pattern(u), 0x7FC0, out).astype(np.uint16)


def _mut_no_carry(u):
    # rounds up inside the mantissa only (drops the carry into the exponent)
    u = np.asarray(u, np.uint32).astype(np.uint64)
    out = ocast.f32_bits_to_bf16_bits(u.astype(np.uint32)).astype(np.uint64)
    t = u >> 16
    carried = (out & 0xFF80) != (t & 0xFF80)
    return np.where(carried & (t & 0x7F == 0x7F), t, out).astype(np.uint16)


@pytest.mark.parametrize("mutant", [_mut_ties_away, _mut_truncate, _mut_nan_drops_sign, _mut_no_carry])
def test_planted_mistakes_are_caught(mutant):
    u = structured_patterns()
    caught = (not check_hand(mutant)) or (not check_against_torch(mutant, u)) or (not check_nan(mutant)) \
        or (not check_against_search(mutant, u))
    assert caught
