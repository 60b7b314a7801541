"""Bit-level number formats used by the layer's inputs, decoded into float64.

TEST INFRASTRUCTURE: only tests/, __graft_entry__.smoke() and bench.py's CPU
baseline leg may import this package.  The product path never touches it.

The paper fixes 16-bit data for the MoE stage (ASAP Table 1, "Dsize = 16 bits");
the configuration it is evaluated on (DeepSeek-V3.2, Section 5.1) stores that
data as bfloat16.  The FP8 configuration uses OCP e4m3 ("e4m3fn": no infinities,
one NaN pattern per sign, maximum finite 448).

Everything here is written from the format definitions (sign, biased exponent,
fraction), not by reinterpreting bits as a wider float, so that the decoders can
be pinned against an independent library conversion.
"""
import numpy as np


def _bf16_fields_to_f64(bits):
    """bfloat16 bit patterns (uint16) -> float64, exactly, from the fields.

    Layout: 1 sign bit, 8 exponent bits (bias 127), 7 fraction bits.
    exponent 0      : subnormal, value = (-1)^s * 2^-126 * f/128
    exponent 1..254 : normal,    value = (-1)^s * 2^(e-127) * (1 + f/128)
    exponent 255    : inf (f == 0) or NaN (f != 0)
    """
    b = np.asarray(bits, dtype=np.uint16).astype(np.int64)
    sign = np.where((b >> 15) & 1, -1.0, 1.0)
    e = (b >> 7) & 0xFF
    f = (b & 0x7F).astype(np.float64)
    normal = np.ldexp(1.0 + f / 128.0, (e - 127).astype(np.int64))
    sub = np.ldexp(f / 128.0, -126)
    mag = np.where(e == 0, sub, normal)
    mag = np.where(e == 255, np.where(f == 0, np.inf, np.nan), mag)
    return sign * mag


_BF16_TABLE = None


def bf16_bits_to_f64(bits):
    """bfloat16 bit patterns (uint16) -> float64, exactly: a lookup in the
    table of all 65536 patterns decoded by ``_bf16_fields_to_f64``."""
    global _BF16_TABLE
    if _BF16_TABLE is None:
        _BF16_TABLE = _bf16_fields_to_f64(np.arange(65536, dtype=np.uint32).astype(np.uint16))
    return _BF16_TABLE[np.asarray(bits, dtype=np.uint16)]


def _e4m3_fields_to_f64(bits):
    """OCP e4m3fn bit patterns (uint8) -> float64, exactly, from the fields.

    Layout: 1 sign bit, 4 exponent bits (bias 7), 3 fraction bits.
    exponent 0     : subnormal, value = (-1)^s * 2^-6 * f/8
    exponent 1..15 : normal,    value = (-1)^s * 2^(e-7) * (1 + f/8)
    exponent 15 with f == 7 is NaN (the format has no infinities).
    """
    b = np.asarray(bits, dtype=np.uint8).astype(np.int64)
    sign = np.where((b >> 7) & 1, -1.0, 1.0)
    e = (b >> 3) & 0xF
    f = (b & 0x7).astype(np.float64)
    normal = np.ldexp(1.0 + f / 8.0, (e - 7).astype(np.int64))
    sub = np.ldexp(f / 8.0, -6)
    mag = np.where(e == 0, sub, normal)
    mag = np.where((e == 15) & (f == 7), np.nan, mag)
    return sign * mag


_E4M3_TABLE = None


def e4m3_bits_to_f64(bits):
    """OCP e4m3fn bit patterns (uint8) -> float64, exactly: a lookup in the
    table of all 256 patterns decoded by ``_e4m3_fields_to_f64``."""
    global _E4M3_TABLE
    if _E4M3_TABLE is None:
        _E4M3_TABLE = _e4m3_fields_to_f64(np.arange(256, dtype=np.uint8))
    return _E4M3_TABLE[np.asarray(bits, dtype=np.uint8)]


E4M3_MAX = 448.0


def round_to_e4m3_sat(v):
    """Round float64 values to the nearest e4m3fn value, ties to even, with
    saturation to +-448 (the largest finite magnitude) instead of NaN.

    Returns the rounded values as float64 (every result is exactly an e4m3
    value).  Normal binades [2^e, 2^(e+1)) for e in [-6, 8] hold 8 values
    spaced 2^(e-3); below 2^-6 the subnormal spacing is 2^-9.
    """
    v = np.asarray(v, dtype=np.float64)
    a = np.abs(v)
    with np.errstate(divide="ignore"):
        e = np.floor(np.log2(np.where(a > 0, a, 1.0)))
    # log2 of an exact power of two can land one binade low or high; fix up.
    e = np.where(np.ldexp(1.0, e.astype(np.int64)) > a, e - 1, e)
    e = np.where(np.ldexp(1.0, (e + 1).astype(np.int64)) <= a, e + 1, e)
    e = np.maximum(e, -6.0)  # subnormal range shares the 2^-6 spacing rule
    step = np.ldexp(1.0, (e - 3).astype(np.int64))
    q = a / step
    r = np.floor(q)
    frac = q - r
    up = (frac > 0.5) | ((frac == 0.5) & (np.fmod(r, 2.0) == 1.0))
    r = r + up
    out = np.minimum(r * step, E4M3_MAX)
    return np.copysign(out, v)
