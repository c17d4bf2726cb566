"""Bit-packed codes (Sec. 3.4, Table 1 storage model), plain Python.

TEST INFRASTRUCTURE ONLY (see the package docstring).

The paper stores each sub-codeword index in log2(K) bits.  Stream layout
used by the library: code i occupies stream bits [i*b, (i+1)*b), code bit t
at stream bit i*b + t; stream bit s is bit (s mod 8) of byte s // 8 (least
significant bit first).  b = bits_for(K) = ceil(log2 K), at least 1.
"""
from __future__ import annotations

import numpy as np


def bits_for(K: int) -> int:
    b = 1
    while (1 << b) < K:
        b += 1
    return b


def pack(codes, b: int) -> bytes:
    """Codes (ints < 2^b) -> the packed byte stream, ceil(n*b/8) bytes."""
    codes = [int(c) for c in np.asarray(codes).ravel()]
    out = bytearray((len(codes) * b + 7) // 8)
    for i, c in enumerate(codes):
        if c < 0 or c >= (1 << b):
            raise ValueError(f"code {c} does not fit {b} bits")
        for t in range(b):
            if (c >> t) & 1:
                s = i * b + t
                out[s // 8] |= 1 << (s % 8)
    return bytes(out)


def unpack(stream: bytes, n: int, b: int) -> np.ndarray:
    """The first n codes of a packed stream, as uint8."""
    data = bytes(stream)
    out = np.zeros(n, np.uint8)
    for i in range(n):
        c = 0
        for t in range(b):
            s = i * b + t
            c |= ((data[s // 8] >> (s % 8)) & 1) << t
        out[i] = c
    return out


def pack_rows(codes2d, b: int, pitch: int) -> bytes:
    """Each row packed on its own and zero-padded to `pitch` bytes (the FC
    kernels' row-aligned layout)."""
    rows = []
    for row in np.asarray(codes2d):
        r = pack(row, b)
        if len(r) > pitch:
            raise ValueError("pitch too small")
        rows.append(r + bytes(pitch - len(r)))
    return b"".join(rows)
