"""Oracle quantisers (test infrastructure; see ``oracle/__init__.py``).

Grouped asymmetric quantiser
----------------------------
Appendix C.3 of the paper describes it in one sentence: a scale and a zero
point per group of ``g`` elements, using all ``2^b`` levels (the KIVI / MLX
grouped scheme it benchmarks in Sec. 4).  The paper gives no formula, so the
reading used here (and by the CUDA path) is the usual one:

    mn    = min(x)            zero  = mn
    mx    = max(x)            levels = 2^b - 1
    scale = f32( f32(mx - mn) / levels )
    code  = clamp( rint( f32( f32(x - mn) / scale ) ), 0, levels )

Every arithmetic step is one IEEE-754 binary32 operation rounded to nearest
even (NumPy float32 arrays), so the codes and scales are reproducible
bit-for-bit by any implementation that performs the same operation sequence
without contraction.  ``rint`` rounds half to even.  A constant group
(mx == mn) stores scale 0 and all codes 0; it dequantises to ``zero`` exactly.

Dequantisation is carried out in float64: ``x_hat = code * scale + zero``.

Groups are either *per token* (``g`` consecutive channels of one token-head
row) or *per channel* (``g`` consecutive token positions of one channel, the
KIVI key layout).  For per-channel groups, positions after the last full
group stay unquantised (the "residual"; Tab. realized_bits counts such a
full-precision window).

Symmetric per-vector quantiser
------------------------------
Appendix C.3, the scheme the paper trains with: one scale per stored vector
(a 128-element token-head row), no zero point, ``q = 2^(b-1) - 1``,
``s = max|x| / q``, ``code = clip(round(x / s), -q, q)``, dequantise as
``code * s``.  The caption of Tab. realized_bits fixes the stored scale as
one bf16 per row; the paper does not say whether the codes are computed
with the scale before or after that rounding.  The reading used here (and by
the CUDA path) computes them with the stored scale, so that dequantisation
uses exactly the scale the codes were made for:

    s32  = f32( max|x| / q )            one binary32 division
    s    = bf16(s32)                    round to nearest even
    code = clip( rint( f32(x / s) ), -q, q )

A zero vector stores scale 0 and codes 0.
"""
from __future__ import annotations

import numpy as np

F32 = np.float32


def levels_for_bits(bits: int) -> int:
    """Number of steps of a ``bits``-bit unsigned code (2^b - 1)."""
    if bits not in (2, 4, 8):
        raise ValueError(f"grouped quantiser supports 2, 4 or 8 bits, got {bits}")
    return (1 << bits) - 1


def quantise_groups(x: np.ndarray, bits: int):
    """Quantise along the LAST axis of ``x`` (each row is one group).

    ``x`` is any float array; it is converted to float32 first (bf16 and fp32
    inputs convert exactly).  Returns ``(codes uint8, scale f32, zero f32)``
    with ``codes.shape == x.shape`` and ``scale.shape == zero.shape ==
    x.shape[:-1]``.
    """
    x = np.asarray(x, dtype=F32)
    lev = F32(levels_for_bits(bits))
    mn = x.min(axis=-1)
    mx = x.max(axis=-1)
    rng = (mx - mn).astype(F32)                 # one rounded f32 subtraction
    scale = (rng / lev).astype(F32)             # one rounded f32 division
    diff = (x - mn[..., None]).astype(F32)      # one rounded f32 subtraction
    safe = np.where(scale == 0, F32(1), scale).astype(F32)
    ratio = (diff / safe[..., None]).astype(F32)  # one rounded f32 division
    codes = np.clip(np.rint(ratio), F32(0), lev)
    codes = np.where(scale[..., None] == 0, F32(0), codes)
    return codes.astype(np.uint8), scale.astype(F32), mn.astype(F32)


def quantise_per_token(x: np.ndarray, bits: int, group: int):
    """Per-token groups: ``group`` consecutive channels of the last axis.

    ``x``: ``[..., D]`` with ``D % group == 0``.
    Returns ``codes [..., D] u8``, ``scale [..., D/group] f32``,
    ``zero [..., D/group] f32``.
    """
    x = np.asarray(x, dtype=F32)
    D = x.shape[-1]
    if D % group:
        raise ValueError("group must divide the channel count")
    xg = x.reshape(*x.shape[:-1], D // group, group)
    c, s, z = quantise_groups(xg, bits)
    return c.reshape(x.shape), s, z


def quantise_per_channel(x: np.ndarray, bits: int, group: int):
    """Per-channel groups: ``group`` consecutive positions of axis -2.

    ``x``: ``[..., T, D]``.  Positions ``[0, Tq)`` with ``Tq = group *
    floor(T / group)`` are quantised; the rest are returned unchanged as the
    residual.  Returns ``codes [..., Tq, D] u8``, ``scale [..., Tq/group, D]``,
    ``zero [..., Tq/group, D]`` and ``residual [..., T - Tq, D]`` (float32).
    """
    x = np.asarray(x, dtype=F32)
    T, D = x.shape[-2], x.shape[-1]
    nG = T // group
    Tq = nG * group
    xq = x[..., :Tq, :].reshape(*x.shape[:-2], nG, group, D)
    xq = np.swapaxes(xq, -1, -2)                # [..., nG, D, group]
    c, s, z = quantise_groups(xq, bits)         # c: [..., nG, D, group]
    c = np.swapaxes(c, -1, -2).reshape(*x.shape[:-2], Tq, D)
    return c, s, z, x[..., Tq:, :].copy()


def dequantise_per_token(codes, scale, zero, group: int) -> np.ndarray:
    """float64 ``code * scale + zero`` with per-token groups of ``group``."""
    c = np.asarray(codes, dtype=np.float64)
    D = c.shape[-1]
    s = np.repeat(np.asarray(scale, dtype=np.float64), group, axis=-1)
    z = np.repeat(np.asarray(zero, dtype=np.float64), group, axis=-1)
    assert s.shape[-1] == D
    return c * s + z


def dequantise_per_channel(codes, scale, zero, group: int, residual=None) -> np.ndarray:
    """float64 dequantisation of per-channel groups, residual appended."""
    c = np.asarray(codes, dtype=np.float64)
    s = np.repeat(np.asarray(scale, dtype=np.float64), group, axis=-2)
    z = np.repeat(np.asarray(zero, dtype=np.float64), group, axis=-2)
    out = c * s + z
    if residual is not None and residual.shape[-2] > 0:
        out = np.concatenate([out, np.asarray(residual, dtype=np.float64)], axis=-2)
    return out


def round_bf16(x) -> np.ndarray:
    """float32 -> nearest bfloat16 (ties to even), returned as float32.

    Integer arithmetic on the binary32 pattern: adding 0x7FFF plus the lowest
    kept bit and truncating the low 16 bits rounds to nearest, ties to even,
    for every finite value (subnormals included)."""
    u = np.asarray(x, dtype=F32).view(np.uint32).astype(np.uint64)
    r = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return r.astype(np.uint32).view(F32)


def sym_levels(bits: int) -> int:
    """q = 2^(b-1) - 1 of the symmetric quantiser (b = 2, 4 or 8)."""
    if bits not in (2, 4, 8):
        raise ValueError(f"symmetric quantiser supports 2, 4 or 8 bits, got {bits}")
    return (1 << (bits - 1)) - 1


def quantise_symmetric(x: np.ndarray, bits: int):
    """Paper's symmetric per-vector quantiser along the last axis.

    Returns ``(codes int8, scale f32)``; ``codes`` lie in ``[-q, q]`` with
    ``q = 2^(bits-1) - 1``; ``scale`` holds bf16 values (the stored scale).
    A zero vector stores scale 0 and codes 0.
    """
    x = np.asarray(x, dtype=F32)
    q = F32(sym_levels(bits))
    amax = np.abs(x).max(axis=-1)
    s = round_bf16((amax / q).astype(F32))       # one f32 division, then bf16
    safe = np.where(s == 0, F32(1), s).astype(F32)
    r = (x / safe[..., None]).astype(F32)         # one f32 division
    codes = np.clip(np.rint(r), -q, q)
    codes = np.where(s[..., None] == 0, F32(0), codes)
    return codes.astype(np.int8), s


def dequantise_symmetric(codes, scale) -> np.ndarray:
    """float64 ``code * scale`` (one scale per vector of the last axis)."""
    return np.asarray(codes, np.float64) * np.asarray(scale, np.float64)[..., None]
