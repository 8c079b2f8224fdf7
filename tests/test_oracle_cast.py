"""Pins for the oracle's float32 -> bfloat16 round-to-nearest-even cast.

The cast itself is implied by the paper (Section 7.4: the rollout holds
16-bit weights); the rounding mode and the NaN rule are the reading taken here.
The oracle uses a bit trick; these tests check it against things other than
that trick:

* a brute-force rounding by value: the two bfloat16 neighbours of |x| are
  found by magnitude, their distances to x are taken in float64 (exact: all
  three numbers have at most 24 significant bits and lie within a factor of
  two of each other, with 2^128 standing in for +inf), the nearer one wins
  and a tie goes to the even mantissa;
* PyTorch's own float32 -> bfloat16 conversion (a library RNE) on non-NaN
  inputs;
* the NaN properties the reading fixes: the result is a NaN (never an
  infinity), keeps the sign and the upper payload bits, and is quiet.
"""
import numpy as np
import pytest
import torch

import oracle
import synth


def brute_force_rne(bits: np.ndarray) -> np.ndarray:
    """Round float32 patterns to bfloat16 by comparing distances; NaNs excluded."""
    bits = bits.astype(np.uint32)
    sign = bits & np.uint32(0x80000000)
    mag = bits & np.uint32(0x7FFFFFFF)
    assert not np.any(mag > 0x7F800000), "brute force is for non-NaN inputs"
    x = mag.view(np.float32).astype(np.float64)
    # Largest bfloat16 magnitude <= |x| and the next one up (bfloat16 values are the
    # float32 values whose low 16 bits are zero; magnitudes are monotone in the bits).
    lo = mag & np.uint32(0xFFFF0000)
    hi = lo + np.uint32(0x10000)
    lo_v = lo.view(np.float32).astype(np.float64)
    hi_v = np.where(hi >= 0x7F800000, 2.0 ** 128, hi.view(np.float32).astype(np.float64))
    with np.errstate(invalid="ignore"):   # inf - inf for x = +-inf, which is exact anyway
        d_lo = x - lo_v
        d_hi = hi_v - x
    exact = mag == lo           # low half zero: representable as is (incl. +-inf, +-0)
    lo_even = ((lo >> 16) & 1) == 0
    pick_hi = (~exact) & ((d_hi < d_lo) | ((d_hi == d_lo) & ~lo_even))
    res = np.where(pick_hi, hi, lo)
    res = np.where(res >= 0x7F800000, np.uint32(0x7F800000), res)  # overflow -> inf
    return ((res | sign) >> 16).astype(np.uint16)


def structured_patterns() -> np.ndarray:
    """Every high half with low halves at, around and away from the rounding tie."""
    hi = np.arange(1 << 16, dtype=np.uint32) << 16
    lows = np.array([0x0000, 0x0001, 0x7FFF, 0x8000, 0x8001, 0xFFFF], dtype=np.uint32)
    return (hi[:, None] | lows[None, :]).ravel()


def is_nan(bits):
    return (bits & np.uint32(0x7FFFFFFF)) > np.uint32(0x7F800000)


def test_special_table_against_brute_force():
    sp = synth.special_table()
    finite = sp[~is_nan(sp)]
    np.testing.assert_array_equal(oracle.rne_bf16(finite), brute_force_rne(finite))


def test_named_cases():
    cases = {
        0x3F808000: 0x3F80,  # tie, even kept
        0x3F818000: 0x3F82,  # tie, odd rounds up
        0x7F7F8000: 0x7F80,  # tie at max bf16 finite (odd) -> +inf
        0x7F7F7FFF: 0x7F7F,  # below that tie stays finite
        0x00000001: 0x0000,  # tiny subnormal -> +0
        0x00018000: 0x0002,  # subnormal tie, odd -> up
        0x007FFFFF: 0x0080,  # largest subnormal -> smallest normal
        0x80000000: 0x8000,  # -0
        0xFF800000: 0xFF80,  # -inf
        0x7F800001: 0x7FC0,  # NaN with payload only in the low half stays NaN
        0xFFA00000: 0xFFE0,  # negative signalling NaN -> quiet, sign kept
    }
    got = oracle.rne_bf16(np.array(list(cases), dtype=np.uint32))
    np.testing.assert_array_equal(got, np.array(list(cases.values()), dtype=np.uint16))


def test_structured_against_brute_force():
    pats = structured_patterns()
    pats = pats[~is_nan(pats)]
    np.testing.assert_array_equal(oracle.rne_bf16(pats), brute_force_rne(pats))


def test_random_against_brute_force_and_torch():
    rng = np.random.default_rng(1234)
    pats = rng.integers(0, 1 << 32, size=2_000_000, dtype=np.uint64).astype(np.uint32)
    pats = pats[~is_nan(pats)]
    got = oracle.rne_bf16(pats)
    np.testing.assert_array_equal(got, brute_force_rne(pats))
    t = torch.from_numpy(pats.view(np.float32)).to(torch.bfloat16).view(torch.int16)
    np.testing.assert_array_equal(got, t.numpy().view(np.uint16))


def test_generated_values_against_torch():
    vals = synth.values_host(1_000_000, 4, seed=3)
    t = torch.from_numpy(vals.view(np.float32)).to(torch.bfloat16).view(torch.int16)
    np.testing.assert_array_equal(oracle.rne_bf16(vals), t.numpy().view(np.uint16))


def test_nan_properties():
    rng = np.random.default_rng(7)
    payload = rng.integers(1, 1 << 23, size=200_000, dtype=np.uint64).astype(np.uint32)
    sign = rng.integers(0, 2, size=payload.size, dtype=np.uint64).astype(np.uint32) << 31
    nans = sign | np.uint32(0x7F800000) | payload
    nans = np.concatenate([nans, np.array([0x7F800001, 0xFF800001, 0x7FFFFFFF, 0x7FC00000],
                                          dtype=np.uint32)])
    out = oracle.rne_bf16(nans).astype(np.uint32)
    assert np.all((out & 0x7FFF) > 0x7F80), "a NaN became an infinity or a number"
    assert np.all((out & 0x0040) != 0), "result is not quiet"
    np.testing.assert_array_equal(out >> 15, nans >> 31)              # sign kept
    np.testing.assert_array_equal(out & 0x3F, (nans >> 16) & 0x3F)    # upper payload kept


@pytest.mark.slow
def test_all_float32_patterns():
    """All 2^32 patterns: non-NaN against brute force, NaN against the stated properties."""
    step = 1 << 26
    for start in range(0, 1 << 32, step):
        pats = np.arange(start, start + step, dtype=np.uint64).astype(np.uint32)
        got = oracle.rne_bf16(pats)
        nan = is_nan(pats)
        np.testing.assert_array_equal(got[~nan], brute_force_rne(pats[~nan]))
        g = got[nan].astype(np.uint32)
        assert np.all((g & 0x7FFF) > 0x7F80) and np.all(g & 0x40)


# ---------------------------------------------------------------------------
# float32 -> float16 (IEEE binary16), the optional rollout type
# ---------------------------------------------------------------------------

def _f16_table():
    """Every finite non-negative binary16 value in bit order (which is value
    order), then 2^16 standing in for +inf (the next value of the top binade
    if the exponent range went on)."""
    bits = np.arange(0x7C00, dtype=np.uint16)
    vals = bits.view(np.float16).astype(np.float64)
    return np.append(vals, 65536.0), np.append(bits, np.uint16(0x7C00))


def brute_force_f16(bits: np.ndarray) -> np.ndarray:
    """Round float32 patterns to binary16 by value; NaNs excluded.  The two
    neighbours of |x| are found in the table; |x| is compared with their
    midpoint, which is exact in float64 (both have at most 11 significant
    bits), so no rounding enters the comparison.  A tie goes to the even
    pattern; anything from 2^16 up is the infinity."""
    bits = bits.astype(np.uint32)
    sign = ((bits >> 16) & 0x8000).astype(np.uint16)
    mag = bits & np.uint32(0x7FFFFFFF)
    assert not np.any(mag > 0x7F800000), "brute force is for non-NaN inputs"
    x = mag.view(np.float32).astype(np.float64)
    vals, pats = _f16_table()
    i = np.searchsorted(vals, np.minimum(x, 65536.0), side="right") - 1   # vals[i] <= |x|
    lo_v, lo_p = vals[i], pats[i]
    j = np.minimum(i + 1, len(vals) - 1)
    hi_v, hi_p = vals[j], pats[j]
    mid = (lo_v + hi_v) / 2
    pick_hi = (i < len(vals) - 1) & ((x > mid) | ((x == mid) & ((lo_p & 1) == 1)))
    return np.where(pick_hi, hi_p, lo_p).astype(np.uint16) | sign


def _f16_ties():
    """Every midpoint between neighbouring binary16 values (exact in float32),
    one float32 step either side of it, both signs."""
    vals, _ = _f16_table()
    mids = ((vals[:-1] + vals[1:]) / 2).astype(np.float32).view(np.uint32)
    pats = np.concatenate([mids, mids - 1, mids + 1])
    pats = pats[(pats & 0x7FFFFFFF) <= 0x7F800000]
    return np.concatenate([pats, pats | np.uint32(0x80000000)])


def test_f16_named_cases():
    cases = {
        0x3F800000: 0x3C00,  # 1.0
        0x477FE000: 0x7BFF,  # 65504, the largest finite
        0x477FEFFF: 0x7BFF,  # just under the overflow tie stays finite
        0x477FF000: 0x7C00,  # 65520: tie with an odd top value -> +inf
        0x38800000: 0x0400,  # 2^-14, the smallest normal
        0x387FFFFF: 0x0400,  # just under it rounds up to it
        0x33800000: 0x0001,  # 2^-24, the smallest subnormal
        0x33000000: 0x0000,  # 2^-25: tie between 0 and 2^-24 -> even 0
        0x33000001: 0x0001,  # just over that tie
        0x33C00000: 0x0002,  # 3 * 2^-25: tie between 1 and 2 (odd) -> 2
        0x00000001: 0x0000,  # a float32 subnormal -> +0
        0x80000000: 0x8000,  # -0
        0xFF800000: 0xFC00,  # -inf
        0x7FC00000: 0x7E00,  # quiet NaN
        0x7F800001: 0x7E00,  # NaN with payload only in the low bits stays NaN
        0xFFA02000: 0xFF01,  # negative signalling NaN -> quiet, sign and top payload kept
    }
    got = oracle.rne_f16(np.array(list(cases), dtype=np.uint32))
    np.testing.assert_array_equal(got, np.array(list(cases.values()), dtype=np.uint16))


def test_f16_ties_against_brute_force_and_numpy():
    pats = _f16_ties()
    got = oracle.rne_f16(pats)
    np.testing.assert_array_equal(got, brute_force_f16(pats))
    with np.errstate(over="ignore"):
        ref = pats.view(np.float32).astype(np.float16).view(np.uint16)
    np.testing.assert_array_equal(got, ref)


def test_f16_random_against_brute_force_and_numpy():
    rng = np.random.default_rng(16)
    pats = rng.integers(0, 1 << 32, size=2_000_000, dtype=np.uint64).astype(np.uint32)
    pats = pats[~is_nan(pats)]
    got = oracle.rne_f16(pats)
    np.testing.assert_array_equal(got, brute_force_f16(pats))
    with np.errstate(over="ignore"):
        ref = pats.view(np.float32).astype(np.float16).view(np.uint16)
    np.testing.assert_array_equal(got, ref)


def test_f16_nan_properties():
    rng = np.random.default_rng(17)
    payload = rng.integers(1, 1 << 23, size=200_000, dtype=np.uint64).astype(np.uint32)
    sign = rng.integers(0, 2, size=payload.size, dtype=np.uint64).astype(np.uint32) << 31
    nans = np.concatenate([sign | np.uint32(0x7F800000) | payload,
                           np.array([0x7F800001, 0xFF800001, 0x7FFFFFFF], dtype=np.uint32)])
    out = oracle.rne_f16(nans).astype(np.uint32)
    assert np.all((out & 0x7C00) == 0x7C00) and np.all(out & 0x03FF), "not a NaN"
    assert np.all(out & 0x0200), "result is not quiet"
    np.testing.assert_array_equal(out >> 15, nans >> 31)                  # sign kept
    np.testing.assert_array_equal(out & 0x01FF, (nans >> 13) & 0x01FF)   # top payload kept


def test_f16_from_every_bfloat16_pattern():
    """A bfloat16 source widens exactly and rounds like float32: all 2^16
    patterns against the brute force (numbers) and the NaN rule."""
    b = np.arange(1 << 16, dtype=np.uint32)
    L = oracle.Layout([("v", (1 << 16,), 2)], [("v", 0, [(0, 0, 1 << 16, 0, 1)])], n_shards=1,
                      tp=1, bucket_bytes=1 << 17, dst_dtype="f16")
    src = np.zeros(L.shard_bytes, np.uint8)
    src[:1 << 17] = b.astype(np.uint16).view(np.uint8)
    got = L.reshard_tensor(oracle.Source(shards=[src]), 0)
    wide = b << 16
    nan = is_nan(wide)
    np.testing.assert_array_equal(got[~nan], brute_force_f16(wide[~nan]))
    np.testing.assert_array_equal(got[nan], oracle.rne_f16(wide[nan]))
    assert np.all(got[nan].astype(np.uint32) & 0x0200)


@pytest.mark.slow
def test_f16_all_float32_patterns():
    """All 2^32 patterns: non-NaN against the brute force, NaN against the rule."""
    step = 1 << 26
    for start in range(0, 1 << 32, step):
        pats = np.arange(start, start + step, dtype=np.uint64).astype(np.uint32)
        got = oracle.rne_f16(pats)
        nan = is_nan(pats)
        np.testing.assert_array_equal(got[~nan], brute_force_f16(pats[~nan]))
        g = got[nan].astype(np.uint32)
        assert np.all((g & 0x7C00) == 0x7C00) and np.all(g & 0x0200)
