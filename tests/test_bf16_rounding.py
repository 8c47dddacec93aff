"""The bf16 storage rounding handed to the oracle, pinned bit for bit.

workloads.bf16_bits / round_bf16 give the values the oracle receives for
the bf16 factor path (fp64 -> fp32 -> bf16, round-to-nearest-even at each
step).  They are checked here against torch's own float32 -> bfloat16
conversion, an implementation written elsewhere, on the cases where a
rounding routine typically goes wrong: exact ties of both parities,
subnormals, carries into the next binade, overflow to infinity, signed
zeros, infinities and NaN.  The library's own conversion is checked against
the same rule on the GPU (stored factors read back with get_term).
"""
import numpy as np
import pytest

from workloads import bf16_bits, round_bf16

torch = pytest.importorskip("torch")


def torch_bits(a64: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(np.asarray(a64, dtype=np.float64)).to(torch.float32).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def f32_from_bits(bits) -> np.ndarray:
    with np.errstate(invalid="ignore"):
        return np.asarray(bits, dtype=np.uint32).view(np.float32).astype(np.float64)


def test_random_values_at_every_scale():
    rng = np.random.default_rng(0)
    a = rng.standard_normal(200_000) * np.exp2(rng.integers(-140, 120, 200_000).astype(np.float64))
    assert np.array_equal(bf16_bits(a), torch_bits(a))


def test_exact_ties_round_to_even():
    rng = np.random.default_rng(1)
    hi = rng.integers(0, 1 << 16, 4096, dtype=np.uint32)
    hi = hi[(hi & 0x7F80) != 0x7F80]           # finite patterns only
    ties = (hi << 16) | 0x8000                 # exactly half way between two bf16 values
    a = f32_from_bits(ties)
    got = bf16_bits(a)
    assert np.array_equal(got, torch_bits(a))
    # the kept pattern is the even one of the two neighbours
    assert np.all(got & 1 == 0)
    # one unit below and above the tie round down and up
    below, above = f32_from_bits(ties - 1), f32_from_bits(ties + 1)
    assert np.array_equal(bf16_bits(below), (hi & 0xFFFF).astype(np.uint16))
    assert np.array_equal(bf16_bits(above), torch_bits(above))


def test_subnormals_and_signed_zero():
    rng = np.random.default_rng(2)
    sub = rng.integers(1, 1 << 23, 4096, dtype=np.uint32)
    bits = np.concatenate([sub, sub | 0x80000000, [0, 0x80000000, 0x00008000, 0x00018000, 0x007FFFFF]])
    a = f32_from_bits(bits.astype(np.uint32))
    assert np.array_equal(bf16_bits(a), torch_bits(a))
    assert bf16_bits(np.array([-0.0]))[0] == 0x8000


def test_carry_and_overflow():
    # mantissa all ones: rounding up carries into the exponent
    carry = f32_from_bits(np.array([0x3FFFFFFF, 0x3F7FFFFF, 0x007FFFFF, 0x7F7FFFFF, 0xFF7FFFFF,
                                    0x7F7F7FFF, 0x7F7F8000, 0x7F7F8001], dtype=np.uint32))
    got = bf16_bits(carry)
    assert np.array_equal(got, torch_bits(carry))
    assert got[3] == 0x7F80 and got[4] == 0xFF80        # FLT_MAX rounds to +-inf
    # fp64 values beyond the float32 range overflow in the first step
    big = np.array([1e39, -1e39, 3.5e38, 1e-50, -1e-50])
    assert np.array_equal(bf16_bits(big), torch_bits(big))


def test_infinities_and_nan():
    a = np.array([np.inf, -np.inf, np.nan, -np.nan])
    got = bf16_bits(a)
    assert got[0] == 0x7F80 and got[1] == 0xFF80
    assert np.all((got[2:] & 0x7FFF) > 0x7F80)               # still NaN
    assert np.array_equal(got[:2], torch_bits(a)[:2])
    payload = f32_from_bits(np.array([0x7F800001, 0x7FBFFFFF], dtype=np.uint32))  # NaN with a low payload only
    assert np.all((bf16_bits(payload) & 0x7FFF) > 0x7F80)    # not truncated to infinity


def test_double_rounding_goes_through_float32():
    # a float64 just above a bf16 tie that float32 rounds onto the tie itself
    # (then ties-to-even applies), as the library's fp64 -> fp32 -> bf16 does
    tie = 1.0 + 2.0 ** -8                     # half way between bf16 1.0 and 1.0078125
    a = np.array([tie + 2.0 ** -40, tie - 2.0 ** -40, 1.0 + 3 * 2.0 ** -8 + 2.0 ** -40])
    assert np.array_equal(bf16_bits(a), torch_bits(a))
    assert bf16_bits(a)[0] == 0x3F80          # rounded to the tie by float32, then to even


def test_round_bf16_values_are_the_patterns():
    rng = np.random.default_rng(3)
    a = rng.standard_normal(10_000)
    r = round_bf16(a)
    assert np.array_equal(np.asarray(r, np.float32).view(np.uint32) >> 16, bf16_bits(a).astype(np.uint32))
    assert np.all(np.abs(r - a) <= np.abs(a) * 2.0 ** -8)   # within half an ulp (2^-9 relative) plus fp32's
