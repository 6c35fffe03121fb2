"""Independent pure-Python restatement of the byte codec (test infrastructure).

Written separately from ``tq_oracle.c`` (different language, different
derivation) so that the two can pin each other: here a byte is built by
Horner's rule from the most significant digit down and split by ``divmod``;
the C file accumulates powers of three upward and divides repeatedly.

Reading of the paper's "lattice-aware packing" ("Packing: From Quantization
to Serialization") used throughout: five trits per byte, digit = trit + 1,
first trit least significant; 128-trit groups are 25 full bytes plus a tail
byte with three trits and two pad digits equal to 1.
"""
from __future__ import annotations

TRITS_PER_BYTE = 5
GROUP = 128
GROUP_BYTES = 26


def encode(trits) -> int:
    """Five trits (first least significant) -> byte value 0..242."""
    trits = [int(t) for t in trits]
    assert len(trits) == TRITS_PER_BYTE
    v = 0
    for t in reversed(trits):  # Horner, most significant digit first
        assert t in (-1, 0, 1)
        v = v * 3 + (t + 1)
    return v


def decode(v: int):
    """Byte value -> five trits, or None if the byte is not a valid numeral."""
    if not 0 <= v < 3 ** TRITS_PER_BYTE:
        return None
    out = []
    for _ in range(TRITS_PER_BYTE):
        v, d = divmod(v, 3)
        out.append(d - 1)
    return out


def encode_group(trits) -> bytes:
    """128 trits -> 26 bytes (tail byte padded with trit 0)."""
    trits = [int(t) for t in trits]
    assert len(trits) == GROUP
    padded = trits + [0] * (GROUP_BYTES * TRITS_PER_BYTE - GROUP)
    return bytes(encode(padded[i:i + 5]) for i in range(0, len(padded), 5))


def decode_group(data: bytes):
    """26 bytes -> (128 trits, ok).  ok is False for invalid bytes or pads."""
    assert len(data) == GROUP_BYTES
    out, ok = [], True
    for b in data:
        t = decode(b)
        if t is None:
            ok = False
            t = [0] * 5
        out.extend(t)
    if any(out[GROUP:]):
        ok = False
    return out[:GROUP], ok
