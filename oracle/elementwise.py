"""CPU oracle of the element-wise four-mask ternary representation.

TEST INFRASTRUCTURE ONLY (like the rest of ``oracle/``): only ``tests/``,
``__graft_entry__.smoke()`` and bench.py's CPU legs may import it; it shares
no code with the CUDA library.

What it computes (paper, "Model and Representation": four disjoint salience
masks, num_mask = 4, orders = [2, 2, 1, 1], and the compact form
W-hat = (mu + alpha0 T0 + alpha1 T1) (.) M, T in {-1, 0, +1}):
    W[n, k] = mu[n, m] + alpha0[n, m] T0[n, k] + alpha1[n, m] T1[n, k],
    m = mask[n, k],
with one (mu, alpha0) pair per row and mask ("For each masked block, mu =
rowmean(W) ...": a masked block is read as one row's elements of one mask),
alpha1 only for the two masks of order 2 (masks 0 and 1) and T1 zero on the
elements of order-1 masks.  The linear layer is y[m][n] = sum_k W[n,k] x[m,k]
in fp64, with a[m][n] = sum_k |W[n,k] x[m,k]| for the tolerance.

Storage (the paper gives none; this library's reading):
  * mask plane: uint32 [N][K/16], the mask id of element (n, k) in bits
    2 (k mod 16) and 2 (k mod 16) + 1 of word [n][k / 16];
  * plane 1: T0 of every element in the group format's plane-1 layout
    (26 bytes per 128 elements, five trits per byte in base 3, digit = t + 1,
    first trit least significant, rows padded to 16 bytes) -- packed here by
    the C oracle's codec;
  * plane 2: per row, the T1 trits of the row's order-2 elements (mask 0 or
    1) in increasing k, five per byte in the same base-3 digit order, the
    row's last byte padded with digit 1 (t = 0); row n's bytes start at byte
    p2rowptr[n] (p2rowptr[N] = all bytes);
  * parameters: fp16 mu [N][4], alpha0 [N][4], alpha1 [N][2].

Data-error status bits (as the group format's): 1 bad code (T outside
{-1, 0, 1} or a mask id above 3), 2 T1 nonzero on an order-1 element, 4 byte
above 242, 8 a pad digit that is not 1.
"""
from __future__ import annotations

import numpy as np

from . import pack as _c_pack, unpack as _c_unpack  # the C oracle's group-format codec (plane 1)

ORDERS = (2, 2, 1, 1)
BAD_CODE, T1_OUTSIDE, BAD_BYTE, BAD_PAD = 1, 2, 4, 8


def half(bits) -> np.ndarray:
    """fp16 bit patterns -> float64 (exact)."""
    return np.ascontiguousarray(bits, dtype=np.uint16).view(np.float16).astype(np.float64)


# ---------------------------------------------------------------- mask plane
def pack_masks(mask: np.ndarray) -> np.ndarray:
    N, K = mask.shape
    assert K % 16 == 0
    m = mask.astype(np.uint64).reshape(N, K // 16, 16)
    shifts = (2 * np.arange(16, dtype=np.uint64))
    return (m << shifts).sum(axis=2).astype(np.uint32)


def unpack_masks(plane: np.ndarray, K: int) -> np.ndarray:
    N = plane.shape[0]
    w = plane.astype(np.uint64).reshape(N, K // 16, 1)
    shifts = (2 * np.arange(16, dtype=np.uint64)).reshape(1, 1, 16)
    return ((w >> shifts) & np.uint64(3)).reshape(N, K).astype(np.uint8)


# ------------------------------------------------------------------- plane 2
def order2(mask: np.ndarray) -> np.ndarray:
    """Whether each element's mask has order 2 (masks 0 and 1)."""
    return mask <= 1


def plane2_rowptr(mask: np.ndarray) -> np.ndarray:
    """Byte offsets of each row's plane-2 bytes: ceil(order-2 count / 5)."""
    counts = order2(mask).sum(axis=1).astype(np.int64)
    rp = np.zeros(mask.shape[0] + 1, np.int64)
    rp[1:] = np.cumsum((counts + 4) // 5)
    return rp.astype(np.int32)


def _pack_trits(t: np.ndarray) -> np.ndarray:
    """A row's trits, five per byte, base 3, first trit least significant,
    the last byte padded with digit 1."""
    n = t.size
    nb = (n + 4) // 5
    d = np.ones(nb * 5, np.int64)
    d[:n] = t.astype(np.int64) + 1
    d = d.reshape(nb, 5)
    return (d * (3 ** np.arange(5))).sum(axis=1).astype(np.uint8)


def _unpack_trits(b: np.ndarray, n: int):
    """(trits, status bits) of n trits from bytes b."""
    st = 0
    v = b.astype(np.int64)
    if (v > 242).any():
        st |= BAD_BYTE
    v = np.minimum(v, 242)
    d = (v.reshape(-1, 1) // (3 ** np.arange(5))) % 3
    d = d.reshape(-1)
    if (d[n:] != 1).any():
        st |= BAD_PAD
    return (d[:n] - 1).astype(np.int8), st


# --------------------------------------------------------------------- codec
def pack(T0: np.ndarray, T1: np.ndarray, mask: np.ndarray):
    """-> (mask plane, plane 1, p2rowptr, plane 2, status bits)."""
    N, K = T0.shape
    st = 0
    if (np.abs(T0.astype(np.int64)) > 1).any() or (np.abs(T1.astype(np.int64)) > 1).any() or (mask > 3).any():
        st |= BAD_CODE
    if (T1[~order2(mask)] != 0).any():
        st |= T1_OUTSIDE
    sal = np.zeros((N, (K // 128 + 31) // 32), np.uint32)
    rp0 = np.zeros(N + 1, np.int32)
    p1, _, st1 = _c_pack(N, K, np.clip(T0, -1, 1).astype(np.int8), None, sal, rp0)
    st |= st1
    rp = plane2_rowptr(np.minimum(mask, 3))
    p2 = np.zeros(int(rp[N]), np.uint8)
    for n in range(N):
        sel = order2(mask[n])
        p2[rp[n]:rp[n + 1]] = _pack_trits(np.clip(T1[n][sel], -1, 1))
    return pack_masks(np.minimum(mask, 3)), p1, rp, p2, st


def unpack(N: int, K: int, mplane: np.ndarray, p1: np.ndarray, rp: np.ndarray, p2: np.ndarray):
    """-> (T0, T1, mask, status bits)."""
    mask = unpack_masks(mplane, K)
    sal = np.zeros((N, (K // 128 + 31) // 32), np.uint32)
    T0, _, st = _c_unpack(N, K, p1, None, sal, np.zeros(N + 1, np.int32), want_t2=False)
    T1 = np.zeros((N, K), np.int8)
    for n in range(N):
        sel = order2(mask[n])
        t, s = _unpack_trits(p2[rp[n]:rp[n + 1]], int(sel.sum()))
        T1[n][sel] = t
        st |= s
    return T0, T1, mask, st


# ------------------------------------------------------- correction index
# A structure derived from a packed weight (this library's, no counterpart
# in the paper), like the group format's second-plane index: the elements of
# masks 0..2 of every row, block by block of IDX_BLOCK elements along K, in
# increasing k, each as one uint16 entry
#     (k mod IDX_BLOCK) | code << 11,  code = 9 q + 3 (T0 + 1) + (T1 + 1),
# with int32 offsets[n * nb + b] of row n's block b (nb = ceil(K / IDX_BLOCK),
# offsets[N nb] = all entries).  Everything the masks 0..2 add to the
# mask-3 form of a row is in its entries.  A block of 2048 elements makes an
# entry's 11 offset bits and 5 code bits (27 codes) fill its 16 bits.
IDX_BLOCK = 2048
IDX_SHIFT = 11


def correction_index(T0: np.ndarray, T1: np.ndarray, mask: np.ndarray):
    """-> (offsets int32 [N nb + 1], entries uint16)."""
    N, K = mask.shape
    nb = (K + IDX_BLOCK - 1) // IDX_BLOCK
    rows, cols = np.nonzero(mask != 3)  # row-major: increasing k within a row
    counts = np.bincount(rows * nb + cols // IDX_BLOCK, minlength=N * nb)
    offsets = np.zeros(N * nb + 1, np.int64)
    offsets[1:] = np.cumsum(counts)
    q = mask[rows, cols].astype(np.int64)
    code = 9 * q + 3 * (T0[rows, cols].astype(np.int64) + 1) + (T1[rows, cols].astype(np.int64) + 1)
    entries = (cols % IDX_BLOCK) | (code << IDX_SHIFT)
    return offsets.astype(np.int32), entries.astype(np.uint16)


def decode_index(N: int, K: int, offsets, entries):
    """-> (mask, T0, T1) with mask 3 and zero codes wherever no entry is."""
    nb = (K + IDX_BLOCK - 1) // IDX_BLOCK
    mask = np.full((N, K), 3, np.uint8)
    T0 = np.zeros((N, K), np.int8)
    T1 = np.zeros((N, K), np.int8)
    e = entries.astype(np.int64)
    for n in range(N):
        for b in range(nb):
            for v in e[offsets[n * nb + b]:offsets[n * nb + b + 1]]:
                k, code = b * IDX_BLOCK + (v & (IDX_BLOCK - 1)), v >> IDX_SHIFT
                mask[n, k], T0[n, k], T1[n, k] = code // 9, (code // 3) % 3 - 1, code % 3 - 1
    return mask, T0, T1


# -------------------------------------------------------------------- linear
def dense_rows(K: int, mplane, p1, rp, p2, mu, a0, a1, rows):
    """fp64 W rows decoded from the packed bytes (the paper's compact form)."""
    sub = lambda a: np.ascontiguousarray(a[rows])
    T0, T1, mask, st = unpack(len(rows), K, sub(mplane), sub(p1),
                              _rows_rp(rp, rows), _rows_p2(rp, p2, rows))
    assert st == 0, st
    mu_, a0_ = half(mu)[rows], half(a0)[rows]
    a1_ = np.concatenate([half(a1)[rows], np.zeros((len(rows), 2))], axis=1)
    r = np.arange(len(rows))[:, None]
    return mu_[r, mask] + a0_[r, mask] * T0 + a1_[r, mask] * T1


def _rows_rp(rp, rows):
    lens = (rp[1:] - rp[:-1])[rows].astype(np.int64)
    out = np.zeros(len(rows) + 1, np.int32)
    out[1:] = np.cumsum(lens)
    return out


def _rows_p2(rp, p2, rows):
    return np.concatenate([p2[rp[n]:rp[n + 1]] for n in rows]) if len(rows) else np.zeros(0, np.uint8)


def linear(x_bits: np.ndarray, K: int, mplane, p1, rp, p2, mu, a0, a1, rows=None, block=256):
    """fp64 y[m][r] and a[m][r] = sum_k |x W| for the selected rows (all if
    None), W reconstructed from the packed bytes and a naive matmul."""
    N = mplane.shape[0]
    rows = np.arange(N) if rows is None else np.asarray(rows)
    x = half(x_bits)  # [M][K]
    y = np.zeros((x.shape[0], len(rows)))
    a = np.zeros_like(y)
    for i in range(0, len(rows), block):
        W = dense_rows(K, mplane, p1, rp, p2, mu, a0, a1, rows[i:i + block])
        y[:, i:i + block] = x @ W.T
        a[:, i:i + block] = np.abs(x) @ np.abs(W).T
    return y, a
