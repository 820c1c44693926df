"""4-bit symmetric base-weight compression (Section 3, "Base model weights compression").

The paper fixes only "4-bit symmetric mode INT4" for every non-LoRA parameter,
embeddings included.  The readings taken here (group size 64 along the input
dimension, fp16 scales, restricted range [-7, 7]):

For every row n of W [rows, cols] and every group g of 64 consecutive columns:

    amax  = max |w|                          (fp32)
    s     = fp16_rne(min(amax / 7, 65504))   (fp32 division, then round to fp16;
                                              the min is fp16 saturation)
    q     = 0                                 if s == 0
          = clamp(rint(w / s), -7, 7)         otherwise (fp32 division, ties to even)
    u     = q + 8                             (offset-binary nibble, 1..15)

Storage: ``qpack`` uint8 [rows, cols/2] holds each run of 8 consecutive columns in one
little-endian 32-bit word, even columns in the low half-word and odd columns in the high
half-word: element 8w + 2j sits in bits 4j..4j+3 of word w and element 8w + 2j + 1 in bits
16 + 4j..16 + 4j + 3 (j = 0..3).  As bytes: (u0 | u2 << 4), (u4 | u6 << 4), (u1 | u3 << 4),
(u5 | u7 << 4).  ``scales[g, n]`` (fp16 [cols/64, rows], group-major).

Decode: ``deq = q * s`` — exact in fp32 (a 4-bit integer times an 11-bit
significand).  The GPU feeds its tensor cores the IEEE-half rounding
``fp16_rne(q * s)``; the function ``dequant_f16_bits`` states that value so the GPU's
operand can be compared bit for bit.

The code and scale decisions are taken in fp32 because that is the precision
the GPU kernel takes them in (a quantised code is an integer decided by
floating point, so both sides decide it in the same precision).
"""
from __future__ import annotations

import numpy as np

GROUP = 64
QMAX = 7
FP16_MAX = np.float32(65504.0)


def compress(W: np.ndarray, group: int = GROUP):
    """Quantise W (fp32 [rows, cols], cols % group == 0) -> (qpack uint8 [rows, cols/2], scales fp16 [cols/group, rows])."""
    W = np.ascontiguousarray(W, dtype=np.float32)
    rows, cols = W.shape
    if cols % group or group % 8:
        raise ValueError("cols must be a multiple of the group size")
    Wg = W.reshape(rows, cols // group, group)
    amax = np.abs(Wg).max(axis=2)                                   # fp32
    s16 = np.minimum(amax / np.float32(QMAX), FP16_MAX).astype(np.float16)
    sf = s16.astype(np.float32)
    with np.errstate(divide="ignore", invalid="ignore"):
        ratio = Wg / sf[:, :, None]                                 # fp32 division
    q = np.clip(np.rint(ratio), -QMAX, QMAX)
    q = np.where(sf[:, :, None] == 0, 0.0, q).astype(np.int8).reshape(rows, cols)
    u = (q.astype(np.int16) + 8).astype(np.uint8).reshape(rows, cols // 8, 8)
    words = np.stack([u[:, :, 0] | (u[:, :, 2] << 4), u[:, :, 4] | (u[:, :, 6] << 4),
                      u[:, :, 1] | (u[:, :, 3] << 4), u[:, :, 5] | (u[:, :, 7] << 4)], axis=2)
    qpack = np.ascontiguousarray(words.reshape(rows, cols // 2)).astype(np.uint8)
    scales = np.ascontiguousarray(s16.T)                            # [cols/group, rows]
    return qpack, scales


def unpack_codes(qpack: np.ndarray) -> np.ndarray:
    """Signed codes q (int8 [rows, cols]) from packed nibbles."""
    rows, half = qpack.shape
    b = qpack.reshape(rows, half // 4, 4).astype(np.int16)
    u = np.empty((rows, half // 4, 8), np.int16)
    for k, (lo, hi) in enumerate(((0, 2), (4, 6), (1, 3), (5, 7))):
        u[:, :, lo] = b[:, :, k] & 0x0F
        u[:, :, hi] = b[:, :, k] >> 4
    return (u - 8).astype(np.int8).reshape(rows, 2 * half)


def row_scales(scales: np.ndarray, group: int = GROUP) -> np.ndarray:
    """Per-element scale (fp32 [rows, cols]) from group-major fp16 scales [cols/group, rows]."""
    return np.repeat(scales.T.astype(np.float32), group, axis=1)


def dequant(qpack: np.ndarray, scales: np.ndarray, group: int = GROUP) -> np.ndarray:
    """deq = q * s as float64 [rows, cols] (the value the method defines; exact)."""
    return unpack_codes(qpack).astype(np.float64) * row_scales(scales, group).astype(np.float64)


def dequant_rows(qpack: np.ndarray, scales: np.ndarray, rows: np.ndarray, group: int = GROUP) -> np.ndarray:
    """deq of selected rows only (e.g. an embedding gather), float64 [len(rows), cols]."""
    q = unpack_codes(qpack[rows]).astype(np.float64)
    s = np.repeat(scales[:, rows].T.astype(np.float64), group, axis=1)
    return q * s


def dequant_f16_bits(qpack: np.ndarray, scales: np.ndarray, group: int = GROUP) -> np.ndarray:
    """uint16 bits of fp16_rne(q * s) [rows, cols]: the tensor-core operand value
    (numpy's float32 -> float16 conversion rounds to nearest, ties to even)."""
    deq32 = unpack_codes(qpack).astype(np.float32) * row_scales(scales, group)
    return deq32.astype(np.float16).view(np.uint16)


def f16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(bits, np.uint16).view(np.float16).astype(np.float64)
