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
