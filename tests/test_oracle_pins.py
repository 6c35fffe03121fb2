"""Pins of the CPU oracle against facts fixed by the paper and by mathematics.

None of these compare the oracle with itself: the byte codec is pinned by
numpy's base-3 conversion, an independent pure-Python codec and exhaustive
enumeration; fp16 decoding by numpy's float16; the linear by closed forms of
special cases (paper eq. W-hat per group), brute-force trit read-out through
decimal place values, exact rational arithmetic and numpy's float64 matmul.
"""
import itertools
import os
from fractions import Fraction

import numpy as np
import pytest

import workloads as wl
from oracle import codec as pycodec

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def base3_digits(v, n=5):
    s = np.base_repr(v, 3).rjust(n, "0")
    return [int(c) for c in reversed(s)]  # least significant first


# ------------------------------------------------------------------ codec
def test_byte_codec_exhaustive(oracle_mod):
    """All 3^5 five-trit tuples <-> bytes 0..242: a bijection that agrees with
    numpy.base_repr and the independent Python codec (paper eq. b_T: five
    trits fit a byte because 3^5 = 243 <= 256)."""
    seen = set()
    for tup in itertools.product((-1, 0, 1), repeat=5):
        v = oracle_mod.encode_byte(tup)
        assert v == pycodec.encode(tup)
        assert base3_digits(v) == [t + 1 for t in tup]
        seen.add(v)
    assert seen == set(range(243))
    for v in range(256):
        t, st = oracle_mod.decode_byte(v)
        if v < 243:
            assert st == 0
            assert list(t) == pycodec.decode(v) == [d - 1 for d in base3_digits(v)]
        else:
            assert st == oracle_mod.BAD_BYTE and pycodec.decode(v) is None
    # closed forms: all -1 -> 0, all 0 -> (3^5-1)/2 = 121, all +1 -> 3^5-1
    assert oracle_mod.encode_byte([-1] * 5) == 0
    assert oracle_mod.encode_byte([0] * 5) == 121
    assert oracle_mod.encode_byte([1] * 5) == 242


def test_tail_byte_all_27(oracle_mod):
    """The 26th byte of a group holds trits 125..127 and two pad digits = 1."""
    N, K = 1, 128
    sal = np.zeros((1, 1), np.uint32)
    rp = np.zeros(2, np.int32)
    for tup in itertools.product((-1, 0, 1), repeat=3):
        T = np.zeros((N, K), np.int8)
        T[0, 125:128] = tup
        p1, _, st = oracle_mod.pack(N, K, T, None, sal, rp)
        assert st == 0
        b = int(p1[0, 25])
        assert base3_digits(b) == [t + 1 for t in tup] + [1, 1]
        assert all(x == 121 for x in p1[0, :25])  # all-zero trits
        assert all(x == 0 for x in p1[0, 26:])    # row pad bytes
        assert bytes(p1[0, :26]) == pycodec.encode_group(list(T[0]))


def test_row_bytes_and_sizes(oracle_mod):
    # 26 bytes per 128-trit group, rows padded to 16 bytes
    assert [oracle_mod.row_bytes(K) for K in (1024, 2560, 4096, 9728, 12288)] == [208, 528, 832, 1984, 2496]
    assert oracle_mod.row_bytes(100) == 0
    assert [oracle_mod.sal_words(K) for K in (128, 4096, 4224, 12288)] == [1, 1, 2, 3]


def packed_bytes(N, K, nnz):
    G = K // 128
    return (N * (((26 * G) + 15) // 16 * 16) + 2 * 2 * N * G + 4 * N * ((G + 31) // 32)
            + 26 * nnz + 2 * nnz + 4 * (N + 1))


def test_packed_size_accounting():
    """Bits/weight of the format: 1.625 bits per trit-plane weight
    (26 bytes / 128 trits) against log2(3) = 1.585 (paper eq. b_T) and the
    per-step byte count of the Qwen3-8B linear decode step."""
    assert 26 * 8 / 128 == 1.625 and 1.625 > np.log2(3)
    total = sum(packed_bytes(p.N, p.K, round(0.1 * p.N * (p.K // 128))) for p in wl.config_projections(2))
    assert total == 1_792_241_424
    weights = sum(p.N * p.K for p in wl.config_projections(2))
    assert weights == 6_945_767_424
    assert packed_bytes(512, 1024, 0) == 126_980


def test_fp16_decode_all_patterns(oracle_mod):
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ref = bits.view(np.float16).astype(np.float64)
    got = np.array([oracle_mod.half_to_double(int(b)) for b in bits])
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan], ref[~nan])


@pytest.mark.parametrize("N,K,frac", [(3, 128, 0.0), (7, 384, 0.3), (64, 1024, 0.1), (5, 4224, 0.5)])
def test_pack_unpack_roundtrip(oracle_mod, N, K, frac):
    w = wl.gen_weights(N, K, frac, config=9, proj=N)
    rp, st = oracle_mod.rowptr(N, K, w.sal)
    assert st == 0 and rp[N] == w.nnz
    assert np.array_equal(rp[1:], np.cumsum(w.sal_dense.sum(axis=1)))
    p1, p2, st = oracle_mod.pack(N, K, w.T1, w.T2, w.sal, rp)
    assert st == 0
    T1, T2, st = oracle_mod.unpack(N, K, p1, p2, w.sal, rp)
    assert st == 0
    assert np.array_equal(T1, w.T1) and np.array_equal(T2, w.T2)
    # every group re-decoded by the independent codec
    for n in range(N):
        for g in range(K // 128):
            t, ok = pycodec.decode_group(bytes(p1[n, 26 * g:26 * g + 26]))
            assert ok and t == list(w.T1[n, 128 * g:128 * g + 128])
    salient = [(n, g) for n in range(N) for g in range(K // 128) if w.sal_dense[n, g]]
    for j, (n, g) in enumerate(salient):
        t, ok = pycodec.decode_group(bytes(p2[j]))
        assert ok and t == list(w.T2[n, 128 * g:128 * g + 128])


def test_unpack_validation(oracle_mod):
    N, K = 4, 256
    w = wl.gen_weights(N, K, 0.25, config=9, proj=77)
    rp, _ = oracle_mod.rowptr(N, K, w.sal)
    p1, p2, _ = oracle_mod.pack(N, K, w.T1, w.T2, w.sal, rp)
    bad = p1.copy(); bad[1, 3] = 243
    assert oracle_mod.unpack(N, K, bad, p2, w.sal, rp)[2] == oracle_mod.BAD_BYTE
    bad = p1.copy(); bad[2, 25] = 0          # tail byte with pad digits 0
    assert oracle_mod.unpack(N, K, bad, p2, w.sal, rp)[2] == oracle_mod.BAD_PAD
    bad = p1.copy(); bad[0, 60] = 1          # row pad byte (52..63) nonzero
    assert oracle_mod.unpack(N, K, bad, p2, w.sal, rp)[2] == oracle_mod.BAD_PAD
    rp_bad = rp.copy(); rp_bad[2] += 1
    assert oracle_mod.unpack(N, K, p1, p2, w.sal, rp_bad)[2] & oracle_mod.BAD_ROWPTR
    T1 = w.T1.copy(); T1[0, 0] = 2
    assert oracle_mod.pack(N, K, T1, w.T2, w.sal, rp)[2] == oracle_mod.BAD_CODE
    T2 = w.T2.copy()
    n, g = np.argwhere(~w.sal_dense)[0]
    T2[n, 128 * g + 5] = 1
    assert oracle_mod.pack(N, K, w.T1, T2, w.sal, rp)[2] == oracle_mod.T2_OUTSIDE


# ----------------------------------------------------------------- linear
def oracle_linear(oracle_mod, w, x, M, rows=None, nthreads=2):
    rp, _ = oracle_mod.rowptr(w.N, w.K, w.sal)
    p1, p2, st = oracle_mod.pack(w.N, w.K, w.T1, w.T2, w.sal, rp)
    assert st == 0
    return oracle_mod.linear(M, w.N, w.K, p1, p2, w.sal, w.s1, w.off, w.s2, x, rows=rows, nthreads=nthreads)


def f16(a):
    return np.asarray(a, np.float64).astype(np.float16).view(np.uint16)


def test_linear_zero_codes_is_offset_sum(oracle_mod):
    """mu != 0: zero trits still carry the offset (paper "E2M-ATQ": a zero
    count is not a ternary test because mu != 0).  T1 = T2 = 0 gives
    y = sum_g off_g * sum_{k in g} x_k."""
    N, K, M = 6, 512, 3
    w = wl.gen_weights(N, K, 0.3, config=9, proj=3)
    w.T1[:] = 0
    w.T2[:] = 0
    x = wl.gen_x(M, K, config=9)
    y, _ = oracle_linear(oracle_mod, w, x, M)
    xs = wl.half_bits_to_float(x).reshape(M, K // 128, 128).sum(axis=2)
    off = wl.half_bits_to_float(w.off)
    assert np.allclose(y, xs @ off.T, rtol=1e-12, atol=1e-15)


def test_linear_zero_params_is_exact_zero(oracle_mod):
    N, K, M = 5, 384, 2
    w = wl.gen_weights(N, K, 0.5, config=9, proj=4)
    w.s1[:] = 0; w.off[:] = 0; w.s2[:] = 0
    y, a = oracle_linear(oracle_mod, w, wl.gen_x(M, K, config=9), M)
    assert np.all(y == 0) and np.all(a == 0)


def test_linear_one_hot_reads_one_weight(oracle_mod):
    """x = e_k picks column k: y[n] = s1[n,g] T1[n,k] (off = 0, no salience).
    N != K so a transposed operand would read the wrong element."""
    N, K = 9, 256
    w = wl.gen_weights(N, K, 0.0, config=9, proj=5)
    w.off[:] = 0
    rp, _ = oracle_mod.rowptr(N, K, w.sal)
    p1, p2, _ = oracle_mod.pack(N, K, w.T1, w.T2, w.sal, rp)
    s1 = wl.half_bits_to_float(w.s1)
    for k in (0, 1, 4, 5, 124, 125, 127, 128, 200, 255):
        x = np.zeros((1, K)); x[0, k] = 1.0
        y, _ = oracle_mod.linear(1, N, K, p1, p2, w.sal, w.s1, w.off, w.s2, f16(x))
        assert np.array_equal(y[0], s1[:, k // 128] * w.T1[:, k])


def test_linear_brute_force_byte_readout(oracle_mod):
    """Every byte value at several byte slots of a group, read back through
    the linear: with s1 = 1, off = 0 and x = 1, 3, 9, 27, 81 on the byte's five
    columns, y = sum_i t_i 3^i is the byte's balanced-ternary value, which is
    v - 121 (121 = the numeral of five zero trits) and unique per byte."""
    K = 128
    N = 243
    for slot in (0, 7, 24):
        p1 = np.zeros((N, 32), np.uint8)
        p1[:, :25] = 121
        p1[:, 25] = 1 + 3 + 9 + 27 + 81  # tail: three zero trits, pads 1
        p1[:, slot] = np.arange(243, dtype=np.uint8)
        sal = np.zeros((N, 1), np.uint32)
        s1 = f16(np.ones((N, 1)))
        off = f16(np.zeros((N, 1)))
        x = np.zeros((1, K)); x[0, 5 * slot:5 * slot + 5] = [1, 3, 9, 27, 81]
        y, a = oracle_mod.linear(1, N, K, p1, None, sal, s1, off, None, f16(x))
        assert np.array_equal(y[0], np.arange(243) - 121)
        for v in range(243):
            assert a[0, v] == sum(abs(d - 1) * 3 ** i for i, d in enumerate(base3_digits(v)))


def test_linear_second_plane_own_scale(oracle_mod):
    """s1 = off = 0: only salient groups contribute, each with its own s2 in
    (n, g) order.  Distinct powers of two as s2 expose a wrong index."""
    N, K, M = 4, 512, 1
    G = K // 128
    w = wl.gen_weights(N, K, 0.5, config=9, proj=6)
    w.s1[:] = 0; w.off[:] = 0
    w.s2 = f16(2.0 ** -np.arange(w.nnz))
    x = f16(np.ones((M, K)))
    y, _ = oracle_linear(oracle_mod, w, x, M)
    j = 0
    want = np.zeros(N)
    for n in range(N):
        for g in range(G):
            if w.sal_dense[n, g]:
                want[n] += 2.0 ** -j * w.T2[n, 128 * g:128 * g + 128].sum()
                j += 1
    assert np.array_equal(y[0], want)


def test_linear_exact_rational(oracle_mod):
    """fp64 result within rounding of the exact rational value."""
    N, K, M = 3, 256, 2
    w = wl.gen_weights(N, K, 0.5, config=9, proj=8)
    x = wl.gen_x(M, K, config=9, proj=8)
    y, a = oracle_linear(oracle_mod, w, x, M)
    F = lambda b: Fraction(float(np.array([b], np.uint16).view(np.float16)[0]))
    G = K // 128
    j = 0
    sidx = {}
    for n in range(N):
        for g in range(G):
            if w.sal_dense[n, g]:
                sidx[(n, g)] = j; j += 1
    for m in range(M):
        for n in range(N):
            tot = Fraction(0)
            for k in range(K):
                g = k // 128
                wv = F(w.s1[n, g]) * int(w.T1[n, k]) + F(w.off[n, g])
                if w.sal_dense[n, g]:
                    wv += F(w.s2[sidx[(n, g)]]) * int(w.T2[n, k])
                tot += wv * F(x[m, k])
            assert abs(float(tot) - y[m, n]) <= 1e-13 * a[m, n]


def test_linear_matches_numpy_matmul(oracle_mod):
    """Cross-check with numpy's float64 matmul on W built from the codes."""
    N, K, M = 40, 1024, 3
    w = wl.gen_weights(N, K, 0.1, config=9, proj=9)
    x = wl.gen_x(M, K, config=9, proj=9)
    y, a = oracle_linear(oracle_mod, w, x, M)
    s1 = np.repeat(wl.half_bits_to_float(w.s1), 128, axis=1)
    off = np.repeat(wl.half_bits_to_float(w.off), 128, axis=1)
    s2d = np.zeros((N, K // 128))
    s2d[w.sal_dense] = wl.half_bits_to_float(w.s2)
    W = s1 * w.T1 + off + np.repeat(s2d, 128, axis=1) * w.T2
    xd = wl.half_bits_to_float(x)
    assert np.allclose(y, xd @ W.T, rtol=0, atol=1e-12 * np.abs(a).max())
    assert np.allclose(a, np.abs(xd[:, None, :] * W[None]).sum(-1), rtol=1e-12)


def test_linear_linearity_and_group_scaling(oracle_mod):
    N, K, M = 8, 512, 1
    w = wl.gen_weights(N, K, 0.2, config=9, proj=10)
    rng = np.random.default_rng(5)
    x1 = rng.integers(-8, 9, (M, K)).astype(np.float64)  # exact in fp16, and so are sums
    x2 = rng.integers(-8, 9, (M, K)).astype(np.float64)
    y1, _ = oracle_linear(oracle_mod, w, f16(x1), M)
    y2, _ = oracle_linear(oracle_mod, w, f16(x2), M)
    y12, a12 = oracle_linear(oracle_mod, w, f16(x1 + x2), M)
    assert np.all(np.abs(y12 - (y1 + y2)) <= 1e-12 * (a12 + 1))
    # doubling one group's s1 changes only that group's T1 contribution
    w2 = wl.gen_weights(N, K, 0.2, config=9, proj=10)
    w2.s1[2, 1] = f16([2 * wl.half_bits_to_float(w.s1[2:3, 1:2])[0, 0]])[0]
    y_b, _ = oracle_linear(oracle_mod, w2, f16(x1), M)
    contrib = wl.half_bits_to_float(w.s1[2:3, 1:2])[0, 0] * (w.T1[2, 128:256] * x1[0, 128:256]).sum()
    diff = y_b - y1
    assert abs(diff[0, 2] - contrib) <= 1e-12 * max(1.0, abs(contrib))
    assert np.all(diff[0, np.arange(N) != 2] == 0)


def test_linear_row_subset(oracle_mod):
    N, K, M = 30, 640, 2
    w = wl.gen_weights(N, K, 0.3, config=9, proj=11)
    x = wl.gen_x(M, K, config=9, proj=11)
    y, a = oracle_linear(oracle_mod, w, x, M)
    rows = np.array([29, 0, 7, 7, 13])
    ys, as_ = oracle_linear(oracle_mod, w, x, M, rows=rows, nthreads=3)
    assert np.array_equal(ys, y[:, rows]) and np.array_equal(as_, a[:, rows])


def test_golden_fixture(oracle_mod):
    """Regression pin: values written by tests/golden/make_golden.py (which
    calls only the oracle), checked against the oracle as it stands."""
    here = os.path.join(os.path.dirname(__file__), "golden", "small_linear.txt")
    lines = [l.split() for l in open(here) if l.strip() and not l.startswith("#")]
    N, K, M = map(int, lines[0])
    w = wl.gen_weights(N, K, 0.25, config=8, proj=1)
    x = wl.gen_x(M, K, config=8, proj=1)
    y, _ = oracle_linear(oracle_mod, w, x, M)
    want = np.array([[float(v) for v in l] for l in lines[1:]])
    assert np.array_equal(y, want)
