"""Write-back formats of a refined layer (test infrastructure, like jarq_oracle).

TEST INFRASTRUCTURE: only the test-suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may use this module.

At termination the scales and codes define the returned weights, which are
cast to the model's weight dtype (App. E "Early stopping"); the codes
themselves are b-bit integers (Sec. 3.1).  Plain definitions:

* ``dequantize_cast``: what = s (q - z) exactly (float64 holds it: a 24-bit
  scale times an integer of at most 9 bits), then one round-to-nearest-even
  to float32, float16 or bfloat16.
* ``pack_codes``: each row's codes as one little-endian bit stream, code k in
  bits [k b, k b + b), cut into 32-bit words (the last word zero-padded).
"""
from __future__ import annotations

import numpy as np

from .jarq_oracle import dequantize


def round_to_bfloat16(x):
    """Round float64 values to the nearest bfloat16 (8 significant bits), ties
    to even, returned as float64.  Normal range only (weights)."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                    # x = m 2^e, 0.5 <= |m| < 1
    return np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)


def dequantize_cast(S, Q, Z, g: int, dtype: str):
    """The returned weights s (q - z) in ``dtype`` ("float32", "float16" or
    "bfloat16"; bfloat16 is returned as float64 values)."""
    w = dequantize(S, Q, Z, g)
    if dtype == "float32":
        return w.astype(np.float32)
    if dtype == "float16":
        return w.astype(np.float16)
    if dtype == "bfloat16":
        return round_to_bfloat16(w)
    raise ValueError(dtype)


def packed_words(din: int, bits: int) -> int:
    return (din * bits + 31) // 32


def pack_codes(Q, bits: int):
    """uint32 [dout][ceil(din b / 32)]: code k of a row in bits [k b, k b + b)
    of the row's little-endian bit stream."""
    Q = np.asarray(Q, dtype=np.uint64)
    dout, din = Q.shape
    nw = packed_words(din, bits)
    out = np.zeros((dout, nw), dtype=np.uint64)
    for k in range(din):
        pos = k * bits
        w, off = divmod(pos, 32)
        out[:, w] |= (Q[:, k] << np.uint64(off)) & np.uint64(0xFFFFFFFF)
        if off + bits > 32:                       # the code continues in the next word
            out[:, w + 1] |= Q[:, k] >> np.uint64(32 - off)
    return out.astype(np.uint32)


def unpack_codes(P, din: int, bits: int):
    """Inverse of ``pack_codes``."""
    P = np.asarray(P, dtype=np.uint64)
    dout = P.shape[0]
    mask = np.uint64((1 << bits) - 1)
    Q = np.zeros((dout, din), dtype=np.uint8)
    for k in range(din):
        pos = k * bits
        w, off = divmod(pos, 32)
        v = P[:, w] >> np.uint64(off)
        if off + bits > 32:
            v |= P[:, w + 1] << np.uint64(32 - off)
        Q[:, k] = (v & mask).astype(np.uint8)
    return Q
