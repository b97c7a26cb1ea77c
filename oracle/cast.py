"""fp32 -> bf16 round-to-nearest-even on bit patterns (oracle).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU baseline / reference arm, never by the product path.

The paper has no cast; the fused cast on get is part of the store's statement
of the problem (get into a consumer buffer as bf16). IEEE-754
round-to-nearest, ties-to-even, written out on bit patterns:

* A finite float's magnitude is ordered like its bit pattern with the sign bit
  cleared, so the two bf16 neighbours of x are the pattern truncated to its
  upper 16 bits (toward zero) and that pattern plus one (away from zero; a
  mantissa carry moves into the exponent, and past the largest finite value it
  lands on infinity, which is the correct overflow).
* The dropped lower 16 bits tell which neighbour is nearer: above half of the
  bf16 spacing (0x8000) rounds away, below rounds toward zero, exactly half
  picks the neighbour whose last mantissa bit is 0 (even).
* Infinities have zero dropped bits and are kept. Subnormals follow the same
  rule (no flush to zero), so do signed zeros.
* NaN: the paper and IEEE-754 do not fix a payload. Reading taken here: a quiet
  NaN that keeps the sign, 0x7FC0 | sign << 15.

Pinned by ``tests/test_oracle_cast.py``: torch's CPU conversion (an
independent implementation) on all non-NaN patterns of a structured set, a
nearest-value search in float64 on random patterns, and hand cases.
"""
from __future__ import annotations

import numpy as np

BF16_QNAN = 0x7FC0


def f32_bits_to_bf16_bits(u: np.ndarray) -> np.ndarray:
    """uint32 fp32 bit patterns -> uint16 bf16 bit patterns, RNE."""
    u = np.asarray(u, dtype=np.uint32).astype(np.uint64)
    sign = u >> 31
    exponent = (u >> 23) & 0xFF
    mantissa = u & 0x7FFFFF
    is_nan = (exponent == 0xFF) & (mantissa != 0)

    toward_zero = u >> 16              # upper neighbour candidates, bit pattern
    dropped = u & 0xFFFF               # the 16 bits that do not fit
    half = 0x8000
    last_bit_odd = (toward_zero & 1) == 1
    away = (dropped > half) | ((dropped == half) & last_bit_odd)
    rounded = toward_zero + away.astype(np.uint64)

    out = np.where(is_nan, BF16_QNAN | (sign << 15), rounded)
    return out.astype(np.uint16)


def cast_bytes_f32_to_bf16(raw: np.ndarray) -> np.ndarray:
    """Little-endian fp32 bytes -> little-endian bf16 bytes (len must be a multiple of 4)."""
    raw = np.ascontiguousarray(raw, dtype=np.uint8)
    if raw.size % 4:
        raise ValueError("fp32 byte length must be a multiple of 4")
    return f32_bits_to_bf16_bits(raw.view("<u4")).astype("<u2").view(np.uint8)
