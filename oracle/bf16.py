"""bf16 <-> float64, exactly (oracle; test infrastructure only).

The paper runs its forward pass in bfloat16 (Appendix "Run information", precision row).
bf16 is the top half of an IEEE-754 binary32: 1 sign bit, 8 exponent bits, 7 stored
mantissa bits.  Values are carried as ``uint16`` bit patterns.

``decode`` is exact (every bf16 value is a float64 value).  ``round_rne`` rounds a
float64 straight to bf16 with round-to-nearest, ties-to-even, in one step (no
intermediate binary32 rounding), by scaling to an 8-bit integer significand and
calling ``numpy.rint`` (which rounds half to even).
"""
import numpy as np

_MIN_NORMAL_EXP = -126          # smallest normal binary32/bf16 exponent
_SUBNORMAL_QUANTUM_EXP = -133   # bf16 subnormal spacing 2^-133 (7 stored bits)


def decode(bits):
    """uint16 bf16 bit patterns -> float64 (exact)."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    with np.errstate(invalid="ignore"):  # NaN payloads widen unchanged
        return b.view(np.float32).astype(np.float64)


def round_to_bf16_value(x):
    """Round float64 ``x`` to the nearest bf16 value (ties to even); returns float64.

    Normal range: x = m * 2^e with 0.5 <= |m| < 1, so x * 2^(8-e) carries the 8
    significant bits in its integer part; rint() rounds the rest half-to-even.
    Below the normal range the quantum is fixed at 2^-133.  Overflow rounds to inf
    when the rounded significand exceeds the largest finite bf16.
    """
    x = np.asarray(x, dtype=np.float64)
    out = np.empty_like(x)
    finite = np.isfinite(x)
    out[~finite] = x[~finite]
    xf = x[finite]
    m, e = np.frexp(xf)
    small = e - 1 < _MIN_NORMAL_EXP
    q = np.where(small, _SUBNORMAL_QUANTUM_EXP, e - 8)
    r = np.rint(np.ldexp(xf, -q))
    val = np.ldexp(r, q)
    val = np.where(np.abs(val) > 3.3895313892515355e38, np.copysign(np.inf, xf), val)
    out[finite] = val
    return out


def encode(x):
    """float64 -> uint16 bf16 bit patterns, round-to-nearest-even (exact, one rounding)."""
    v = round_to_bf16_value(x)
    # v is exactly representable in binary32 with the low 16 bits zero.
    b32 = v.astype(np.float32).view(np.uint32)
    return (b32 >> np.uint32(16)).astype(np.uint16)
