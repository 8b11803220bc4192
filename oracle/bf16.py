"""bf16 <-> float conversions of the oracle (test infrastructure only).

bfloat16 is the upper half of an IEEE-754 binary32: 1 sign bit, 8 exponent
bits, 7 fraction bits.  Upcasting appends 16 zero bits, which is exact.
Downcasting rounds a binary32 to the nearest bf16, ties to even
(IEEE-754 roundTiesToEven); NaN stays NaN.
"""
import numpy as np


def to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact value of bf16 bit patterns (uint16) as float64."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def from_f32(x) -> np.ndarray:
    """Round binary32 values to bf16 (ties to even); returns uint16 bit patterns."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    upper = u >> np.uint64(16)
    lower = u & np.uint64(0xFFFF)
    half = np.uint64(0x8000)
    round_up = (lower > half) | ((lower == half) & ((upper & np.uint64(1)) == np.uint64(1)))
    out = (upper + round_up.astype(np.uint64)).astype(np.uint32)
    nan = np.isnan(f)
    out = np.where(nan, (upper | np.uint64(0x40)).astype(np.uint32), out)
    return out.astype(np.uint16)


def from_f64(x) -> np.ndarray:
    """Round float64 values directly to bf16 (ties to even, no intermediate
    binary32 rounding); finite inputs only.  Returns uint16 bit patterns.

    The bf16 neighbour toward zero is found from the binary32 rounding (one
    step back when that rounded away from zero); the two neighbours differ by
    one bf16 ulp, so both distances to x are exact in float64."""
    x = np.asarray(x, dtype=np.float64)
    if not np.all(np.isfinite(x)):
        raise ValueError("from_f64 takes finite values")
    f = x.astype(np.float32)
    lo = (f.view(np.uint32) & np.uint32(0xFFFF0000))                # truncated to bf16
    lo_v = lo.view(np.float32).astype(np.float64)
    over = np.abs(lo_v) > np.abs(x)                                  # rounded away from zero: step back
    lo = np.where(over, lo - np.uint32(0x10000), lo).astype(np.uint32)
    lo_v = lo.view(np.float32).astype(np.float64)
    hi = (lo + np.uint32(0x10000)).astype(np.uint32)                 # next bf16 away from zero
    hi_v = hi.view(np.float32).astype(np.float64)
    d_lo, d_hi = np.abs(x - lo_v), np.abs(hi_v - x)
    lo16, hi16 = (lo >> np.uint32(16)).astype(np.uint16), (hi >> np.uint32(16)).astype(np.uint16)
    take_hi = (d_hi < d_lo) | ((d_hi == d_lo) & ((lo16 & np.uint16(1)) == 1))
    out = np.where(take_hi, hi16, lo16)
    return np.where(x == 0, np.where(np.signbit(x), np.uint16(0x8000), np.uint16(0)), out).astype(np.uint16)
