"""Rounding of exact (fp64) values to the weight storage dtype (test infrastructure only).

Each weight pass of the fused contract (Alg. 2 line "W_i <- W_i + eps U_i Z_i V_i^T",
fused over consecutive updates) computes the new weight exactly in fp64 and
rounds it ONCE to the dtype W is stored in, round-to-nearest, ties to even.
The paper's own runs stored fp16 weights (Sec. 5.x memory analysis, Table 6);
the workloads here use bf16 and fp32.
"""

import numpy as np

_BF16_MIN_EXP = -133       # bf16 subnormal quantum is 2^-133
_BF16_MAX = (2.0 - 2.0 ** -7) * 2.0 ** 127


def round_to_bf16(x):
    """Round fp64 values to the nearest bf16 value (RNE), returned as fp64.

    bf16 keeps 8 significant bits and fp32's exponent range.  For |x| in
    [2^E, 2^(E+1)) the spacing is 2^(E-7); below the normal range it is
    2^-133.  Rounding x / spacing to an integer with ties-to-even (np.rint)
    and scaling back is exact in fp64 because the spacing is a power of two.
    """
    x = np.asarray(x, dtype=np.float64)
    out = np.array(x, copy=True)
    fin = np.isfinite(x) & (x != 0.0)
    xf = x[fin]
    _, e = np.frexp(xf)                    # xf = f * 2^e, f in [0.5, 1)
    q_exp = np.maximum(e - 8, _BF16_MIN_EXP)
    q = np.ldexp(1.0, q_exp)
    y = np.rint(xf / q) * q
    y = np.where(np.abs(y) > _BF16_MAX, np.copysign(np.inf, y), y)
    out[fin] = y
    return out


def round_to_f32(x):
    """Round fp64 values to fp32 (RNE, numpy's cast), returned as fp64."""
    return np.asarray(x, dtype=np.float64).astype(np.float32).astype(np.float64)


def round_to(x, dtype):
    """Round to the storage dtype; "f64" leaves the value exact (used by pins)."""
    if dtype == "f64":
        return np.asarray(x, dtype=np.float64).copy()
    if dtype == "bf16":
        return round_to_bf16(x)
    if dtype == "f32":
        return round_to_f32(x)
    raise ValueError(f"unknown weight dtype {dtype!r}")


def bf16_ulp(x):
    """Spacing of bf16 numbers at |x| (the unit in the last place)."""
    x = np.abs(np.asarray(x, dtype=np.float64))
    _, e = np.frexp(np.where(x == 0.0, 2.0 ** -126, x))
    return np.ldexp(1.0, np.maximum(e - 8, _BF16_MIN_EXP))


def bf16_bits_to_f64(bits):
    """uint16 bf16 bit patterns -> fp64 values."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def f64_to_bf16_bits(x):
    """fp64 values that are exactly bf16-representable -> uint16 bit patterns."""
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    return (f.view(np.uint32) >> np.uint32(16)).astype(np.uint16)
