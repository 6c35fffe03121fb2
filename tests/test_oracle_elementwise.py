"""Pins of the element-wise four-mask oracle (oracle/elementwise.py) against
what the paper and the mathematics fix, with no GPU: the mask plane's bit
positions and plane 2's bytes worked by hand, the row offsets' closed form,
lossless round trips and the rejection of invalid inputs, the reduction to
the group format (C oracle) when every element is in mask 3, an exact
rational case by brute force over every element, one-hot activations,
zero codes, and the independence of order-1 masks from alpha1; the
correction index's entries worked by hand, its offsets closed form, its
lossless decoding and, on exact rational data, the mask-3 form of every
element plus the sum over the index's entries equal to the definition."""
import numpy as np
import pytest

import oracle
import workloads as wl
from oracle import elementwise as ew


def _bits(v):
    return np.asarray(v, np.float16).view(np.uint16)


def test_mask_plane_bit_positions():
    mask = np.zeros((2, 32), np.uint8)
    mask[0, 5] = 2   # bits 10..11 of word 0
    mask[0, 17] = 3  # bits 2..3 of word 1
    mask[1, 15] = 1  # bits 30..31 of word 0 of row 1
    p = ew.pack_masks(mask)
    assert p.tolist() == [[2 << 10, 3 << 2], [1 << 30, 0]]
    assert np.array_equal(ew.unpack_masks(p, 32), mask)


def test_plane2_bytes_by_hand():
    # order-2 trits (1, -1, 0, 1, 1, -1): digits (2, 0, 1, 2, 2) -> 2 + 9 + 54 + 162 = 227,
    # then (0, pad 1, 1, 1, 1) -> 0 + 3 + 9 + 27 + 81 = 120
    assert ew._pack_trits(np.array([1, -1, 0, 1, 1, -1])).tolist() == [227, 120]
    t, st = ew._unpack_trits(np.array([227, 120], np.uint8), 6)
    assert st == 0 and t.tolist() == [1, -1, 0, 1, 1, -1]


def test_plane2_rowptr_closed_form():
    mask = np.full((4, 128), 3, np.uint8)
    mask[1, :1] = 0
    mask[2, 10:15] = 1
    mask[3, 0:6] = 0
    assert ew.plane2_rowptr(mask).tolist() == [0, 0, 1, 2, 4]


@pytest.mark.parametrize("N,K", [(1, 128), (7, 256), (33, 1152), (64, 4096)])
def test_round_trip(N, K):
    w = wl.gen_ew_weights(N, K, config=1, proj=N)
    mp, p1, rp, p2, st = ew.pack(w.T0, w.T1, w.mask)
    assert st == 0
    T0, T1, m, st = ew.unpack(N, K, mp, p1, rp, p2)
    assert st == 0
    assert np.array_equal(T0, w.T0) and np.array_equal(T1, w.T1) and np.array_equal(m, w.mask)


def test_invalid_inputs_rejected():
    w = wl.gen_ew_weights(3, 128, config=1)
    T1 = w.T1.copy()
    k = int(np.argwhere(w.mask[0] >= 2)[0][0])
    T1[0, k] = 1
    assert ew.pack(w.T0, T1, w.mask)[4] & ew.T1_OUTSIDE
    T0 = w.T0.copy()
    T0[1, 3] = 2
    assert ew.pack(T0, w.T1, w.mask)[4] & ew.BAD_CODE
    mp, p1, rp, p2, _ = ew.pack(w.T0, w.T1, w.mask)
    bad = p2.copy()
    bad[0] = 243
    assert ew.unpack(3, 128, mp, p1, rp, bad)[3] & ew.BAD_BYTE
    # a row whose order-2 count is not a multiple of 5: its last byte's pad digits must be 1
    mask = np.full((1, 128), 3, np.uint8)
    mask[0, :3] = 0
    T = np.zeros((1, 128), np.int8)
    mp, p1, rp, p2, st = ew.pack(T, T, mask)
    assert st == 0 and p2.tolist() == [1 + 3 + 9 + 27 + 81]
    assert ew.unpack(1, 128, mp, p1, rp, np.array([1 + 3 + 9 + 27], np.uint8))[3] & ew.BAD_PAD


def test_all_mask3_reduces_to_group_format():
    """Every element in mask 3: W = mu_3 + alpha0_3 T0, the group format's
    s1 T1 + off with s1 = alpha0_3 and off = mu_3 in every group; the group
    format's C oracle (pinned on its own) gives the same y."""
    N, K, M = 20, 640, 3
    w = wl.gen_ew_weights(N, K, config=2)
    mask = np.full((N, K), 3, np.uint8)
    T1 = np.zeros_like(w.T1)
    mp, p1, rp, p2, st = ew.pack(w.T0, T1, mask)
    assert st == 0
    x = wl.gen_x(M, K, config=2)
    y, a = ew.linear(x, K, mp, p1, rp, p2, w.mu, w.a0, w.a1)
    G = K // 128
    s1 = np.repeat(w.a0[:, 3:4], G, axis=1)
    off = np.repeat(w.mu[:, 3:4], G, axis=1)
    sal = np.zeros((N, 1), np.uint32)
    gp1, _, st = oracle.pack(N, K, w.T0, None, sal, np.zeros(N + 1, np.int32))
    assert st == 0 and np.array_equal(gp1, p1)
    y_g, a_g = oracle.linear(M, N, K, gp1, None, sal, s1, off, None, x)
    np.testing.assert_allclose(y, y_g, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(a, a_g, rtol=1e-12, atol=1e-12)


def test_exact_rational_brute_force():
    """Dyadic parameters and small integer activations: every product and sum
    is exact in fp64, so the oracle must equal a sum over every element with
    its own mask's mu, alpha0 and (order 2 only) alpha1 exactly."""
    rng = np.random.default_rng(5)
    N, K = 3, 128
    mask = rng.integers(0, 4, (N, K)).astype(np.uint8)
    T0 = rng.integers(-1, 2, (N, K)).astype(np.int8)
    T1 = (rng.integers(-1, 2, (N, K)) * (mask <= 1)).astype(np.int8)
    mu = rng.integers(-8, 9, (N, 4)) / 64.0
    a0 = rng.integers(1, 9, (N, 4)) / 16.0
    a1 = rng.integers(1, 9, (N, 2)) / 32.0
    x = rng.integers(-3, 4, (2, K)).astype(np.float64)
    mp, p1, rp, p2, st = ew.pack(T0, T1, mask)
    assert st == 0
    y, _ = ew.linear(_bits(x), K, mp, p1, rp, p2, _bits(mu), _bits(a0), _bits(a1))
    for m in range(2):
        for n in range(N):
            want = 0.0
            for k in range(K):
                q = mask[n, k]
                wv = mu[n, q] + a0[n, q] * T0[n, k]
                if q <= 1:
                    wv += a1[n, q] * T1[n, k]
                want += wv * x[m, k]
            assert y[m, n] == want


def test_one_hot_columns():
    N, K = 9, 256
    w = wl.gen_ew_weights(N, K, config=3)
    mp, p1, rp, p2, st = ew.pack(w.T0, w.T1, w.mask)
    h = lambda b: ew.half(b)
    for k in (0, 77, 128, 255):
        x = np.zeros((1, K), np.float16)
        x[0, k] = 1.0
        y, _ = ew.linear(x.view(np.uint16), K, mp, p1, rp, p2, w.mu, w.a0, w.a1)
        for n in range(N):
            q = w.mask[n, k]
            want = h(w.mu[n, q]) + h(w.a0[n, q]) * w.T0[n, k] + (h(w.a1[n, q]) * w.T1[n, k] if q <= 1 else 0.0)
            assert y[0, n] == want


def test_zero_codes_give_mask_means():
    N, K, M = 5, 384, 2
    w = wl.gen_ew_weights(N, K, config=4)
    Z = np.zeros((N, K), np.int8)
    mp, p1, rp, p2, _ = ew.pack(Z, Z, w.mask)
    x = wl.gen_x(M, K, config=4)
    y, _ = ew.linear(x, K, mp, p1, rp, p2, w.mu, w.a0, w.a1)
    xf = ew.half(x)
    for n in range(N):
        want = sum(ew.half(w.mu[n, q]) * xf[:, w.mask[n] == q].sum(axis=1) for q in range(4))
        np.testing.assert_allclose(y[:, n], want, rtol=1e-12, atol=1e-12)


def test_order1_masks_ignore_alpha1_and_mu_is_per_mask():
    N, K = 6, 512
    w = wl.gen_ew_weights(N, K, config=5)
    mask = np.where(w.mask <= 1, 2, w.mask).astype(np.uint8)  # only order-1 masks
    T1 = np.zeros_like(w.T1)
    mp, p1, rp, p2, _ = ew.pack(w.T0, T1, mask)
    x = wl.gen_x(1, K, config=5)
    y0, _ = ew.linear(x, K, mp, p1, rp, p2, w.mu, w.a0, w.a1)
    y1, _ = ew.linear(x, K, mp, p1, rp, p2, w.mu, w.a0, _bits(np.full((N, 2), 8.0)))
    assert np.array_equal(y0, y1)
    # raising mu of mask 2 by d adds d * (sum of x over the row's mask-2 elements)
    mu2 = ew.half(w.mu).copy()
    mu2[:, 2] += 0.25
    mu2_bits = _bits(mu2)
    y2, _ = ew.linear(x, K, mp, p1, rp, p2, mu2_bits, w.a0, w.a1)
    xf = ew.half(x)[0]
    for n in range(N):
        d = (ew.half(mu2_bits)[n, 2] - ew.half(w.mu)[n, 2]) * xf[mask[n] == 2].sum()
        np.testing.assert_allclose(y2[0, n] - y0[0, n], d, rtol=1e-9, atol=1e-12)


def test_index_entries_by_hand():
    # row 0: k = 3 mask 0 (T0 = 1, T1 = -1), k = 2060 mask 2 (T0 = -1); row 1: k = 5 mask 1 (T0 = 0, T1 = 1)
    N, K = 2, 2176
    mask = np.full((N, K), 3, np.uint8)
    T0 = np.zeros((N, K), np.int8)
    T1 = np.zeros((N, K), np.int8)
    mask[0, 3], T0[0, 3], T1[0, 3] = 0, 1, -1
    mask[0, 2060], T0[0, 2060] = 2, -1
    mask[1, 5], T1[1, 5] = 1, 1
    off, ent = ew.correction_index(T0, T1, mask)
    # nb = 2 blocks of 2048 per row; code = 9 q + 3 (T0 + 1) + (T1 + 1) in bits 11..15
    assert off.tolist() == [0, 1, 2, 3, 3]
    assert ent.tolist() == [3 | (0 + 6 + 0) << 11, 12 | (18 + 0 + 1) << 11, 5 | (9 + 3 + 2) << 11]


@pytest.mark.parametrize("N,K", [(1, 128), (7, 2048), (33, 1152), (16, 4224)])
def test_index_offsets_and_decoding(N, K):
    w = wl.gen_ew_weights(N, K, config=6, proj=N)
    off, ent = ew.correction_index(w.T0, w.T1, w.mask)
    nb = (K + 2047) // 2048
    want = [int((w.mask[n, b * 2048:(b + 1) * 2048] != 3).sum()) for n in range(N) for b in range(nb)]
    assert np.array_equal(np.diff(off), want) and off[0] == 0
    m, T0, T1 = ew.decode_index(N, K, off, ent)
    sel = w.mask != 3
    assert np.array_equal(m, np.where(sel, w.mask, 3))
    assert np.array_equal(T0[sel], w.T0[sel]) and np.array_equal(T1[sel], w.T1[sel])


def test_index_correction_plus_mask3_form_is_exact():
    """Dyadic parameters and small integer activations: the mask-3 form of
    every element (mu_3 + alpha0_3 T0) plus, over the index's entries,
    (mu_q - mu_3) + (alpha0_q - alpha0_3) T0 + alpha1_q T1 times x equals the
    oracle's linear exactly."""
    rng = np.random.default_rng(11)
    N, K = 4, 4096 + 128
    mask = rng.choice(4, size=(N, K), p=[0.05, 0.1, 0.15, 0.7]).astype(np.uint8)
    T0 = rng.integers(-1, 2, (N, K)).astype(np.int8)
    T1 = (rng.integers(-1, 2, (N, K)) * (mask <= 1)).astype(np.int8)
    mu = rng.integers(-8, 9, (N, 4)) / 64.0
    a0 = rng.integers(1, 9, (N, 4)) / 16.0
    a1 = rng.integers(1, 9, (N, 2)) / 32.0
    x = rng.integers(-3, 4, (2, K)).astype(np.float64)
    mp, p1, rp, p2, st = ew.pack(T0, T1, mask)
    assert st == 0
    y, _ = ew.linear(_bits(x), K, mp, p1, rp, p2, _bits(mu), _bits(a0), _bits(a1))
    off, ent = ew.correction_index(T0, T1, mask)
    nb = (K + 2047) // 2048
    a1x = np.concatenate([a1, np.zeros((N, 2))], axis=1)
    for n in range(N):
        base = (mu[n, 3] + a0[n, 3] * T0[n].astype(np.float64)) @ x.T
        corr = np.zeros(2)
        for b in range(nb):
            for v in ent[off[n * nb + b]:off[n * nb + b + 1]].astype(np.int64):
                k, code = b * 2048 + (v & 2047), v >> 11
                q, t0, t1 = code // 9, (code // 3) % 3 - 1, code % 3 - 1
                corr += ((mu[n, q] - mu[n, 3]) + (a0[n, q] - a0[n, 3]) * t0 + a1x[n, q] * t1) * x[:, k]
        assert np.array_equal(base + corr, y[:, n])
