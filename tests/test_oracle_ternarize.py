"""Pins of the E2M-ATQ ternarizer oracle (paper "Conversion Pipeline",
"E2M-ATQ") against facts that do not come from the oracle itself:

* closed forms: weights built as mu + a T0 (+ b T1) from dyadic values, which
  every step of the method must give back exactly (the threshold 0.75 times
  the mean absolute deviation separates a from 0 and from b; the
  least-squares scales of exact data are the generating scales);
* exact symmetries of round-to-nearest arithmetic: negating the weights
  negates mu and the supports and keeps the scales and the salience;
  scaling by a power of two scales mu and the scales and keeps the supports;
* the alternating refinement converges to the least-squares fit of w on
  [1, T0, T1], computed by numpy.linalg.lstsq in float64, and never raises
  the float64 squared error;
* salience is the top-nnz energy set, checked against Python's sorted();
* the output planes and parameters, packed by the C oracle and read back by
  its fp64 linear layer, reconstruct mu + alpha0 T0 + alpha1 T1 per block.
"""
import numpy as np
import pytest

import workloads as wl
from oracle import ternarize as tz

F32 = np.float32


def dyadic_blocks(rng, B, two_plane):
    """Blocks w = mu + a T0 (+ b T1 on the zeros of T0), every value a
    multiple of 1/64 below 2 in magnitude (exact in fp16 and in every float32
    partial sum).  T0 and T1 have as many +1 as -1, so the block mean is mu."""
    mu = rng.integers(-16, 17, B) / 64.0
    a = rng.integers(16, 33, B) / 64.0        # 1/4 .. 1/2
    b = np.where(two_plane, rng.integers(2, 5, B) / 64.0, 0.0)  # 1/32 .. 1/16
    T0 = np.zeros((B, 128), np.int8)
    T1 = np.zeros((B, 128), np.int8)
    for i in range(B):
        perm = rng.permutation(128)
        h = int(rng.integers(16, 33))          # h entries +1 and h entries -1
        T0[i, perm[:h]] = 1
        T0[i, perm[h:2 * h]] = -1
        if two_plane[i]:
            q = int(rng.integers(8, 17))
            T1[i, perm[2 * h:2 * h + q]] = 1
            T1[i, perm[2 * h + q:2 * h + 2 * q]] = -1
    w = mu[:, None] + a[:, None] * T0 + b[:, None] * T1
    bits = w.astype(np.float16)
    assert np.array_equal(bits.astype(np.float64), w)  # exactly representable
    return bits.view(np.uint16), mu, a, b, T0, T1


@pytest.mark.parametrize("sweeps", [0, 4])
def test_closed_form_one_plane(sweeps):
    """w = mu + a T0 exactly: the first support is T0, the offset mu, the
    scale a, the residual energy 0 (E2M-ATQ, eqs. for mu, Delta0 and T0 and
    the least-squares scale), and refinement leaves them unchanged."""
    rng = np.random.default_rng(1)
    B = 64
    bits, mu, a, _, T0, _ = dyadic_blocks(rng, B, np.zeros(B, bool))
    W = bits.reshape(4, 16 * 128)  # 4 rows of 16 groups
    r = tz.ternarize(W, nnz=0, sweeps=sweeps)
    assert np.array_equal(r["T1"].reshape(B, 128), T0)
    assert not r["T2"].any() and not r["sal"].any()
    assert np.array_equal(r["mu"].ravel(), mu.astype(F32))
    assert np.array_equal(r["alpha0"].ravel(), a.astype(F32))
    assert np.array_equal(r["E"].ravel(), np.zeros(B, F32))
    assert np.array_equal(r["off"].ravel(), mu.astype(np.float16).view(np.uint16))
    assert np.array_equal(r["s1"].ravel(), a.astype(np.float16).view(np.uint16))


@pytest.mark.parametrize("sweeps", [0, 3])
def test_closed_form_two_planes_and_salience(sweeps):
    """w = mu + a T0 + b T1 with T1 on zeros of T0: the blocks with b > 0 are
    exactly the ones with residual energy (b^2 |T1|), so with nnz = their count
    they alone are salient, and the residual's support and least-squares
    scale give back T1 and b.  With three more salient slots the ties at
    energy 0 go to the lowest block ids, whose second plane is empty."""
    rng = np.random.default_rng(2)
    B = 96
    two = rng.random(B) < 0.25
    bits, mu, a, b, T0, T1 = dyadic_blocks(rng, B, two)
    W = bits.reshape(6, 16 * 128)
    nnz = int(two.sum())
    r = tz.ternarize(W, nnz=nnz, sweeps=sweeps)
    assert np.array_equal(r["salient"].ravel(), two)
    assert np.array_equal(r["T1"].reshape(B, 128), T0)
    assert np.array_equal(r["T2"].reshape(B, 128), T1)
    assert np.array_equal(r["mu"].ravel(), mu.astype(F32))
    assert np.array_equal(r["alpha0"].ravel(), a.astype(F32))
    assert np.array_equal(r["alpha1"].ravel(), b.astype(F32))
    assert np.array_equal(r["s2"], b[two].astype(np.float16).view(np.uint16))
    assert np.array_equal(r["E"].ravel(), (b * b * np.abs(T1).sum(1)).astype(F32))
    # three more slots: the three lowest ids among the zero-energy blocks
    r3 = tz.ternarize(W, nnz=nnz + 3, sweeps=sweeps)
    extra = np.flatnonzero(~two)[:3]
    want = two.copy()
    want[extra] = True
    assert np.array_equal(r3["salient"].ravel(), want)
    assert not r3["T2"].reshape(B, 128)[extra].any()
    assert np.array_equal(r3["alpha1"].ravel()[extra], np.zeros(3, F32))


def test_negation_symmetry():
    """Round to nearest even is odd-symmetric, so -W gives -mu, -T0, -T1 and
    the same scales, energies and salience, bit for bit."""
    W = wl.gen_dense_weights(24, 640, proj=3)
    neg = W ^ np.uint16(0x8000)
    r, q = tz.ternarize(W, nnz=12, sweeps=4), tz.ternarize(neg, nnz=12, sweeps=4)
    assert np.array_equal(q["T1"], -r["T1"]) and np.array_equal(q["T2"], -r["T2"])
    assert np.array_equal(q["mu"], -r["mu"])
    for k in ("alpha0", "alpha1", "E", "sal", "s1", "s2"):
        assert np.array_equal(q[k], r[k]), k
    assert np.array_equal(q["off"], r["off"] ^ np.uint16(0x8000))


def test_power_of_two_scaling():
    """Scaling every weight by 4 (exact in fp16 and float32 away from the
    extremes) scales mu and the scales by 4 and the energies by 16 and keeps
    supports and salience."""
    W = wl.gen_dense_weights(16, 512, proj=4)
    W4 = (W.view(np.float16).astype(np.float64) * 4).astype(np.float16)
    assert np.array_equal(W4.astype(np.float64), W.view(np.float16).astype(np.float64) * 4)
    r, q = tz.ternarize(W, nnz=7, sweeps=4), tz.ternarize(W4.view(np.uint16), nnz=7, sweeps=4)
    for k in ("T1", "T2", "sal"):
        assert np.array_equal(q[k], r[k]), k
    for k in ("mu", "alpha0", "alpha1"):
        assert np.array_equal(q[k], r[k] * F32(4)), k
    assert np.array_equal(q["E"], r["E"] * F32(16))


def _lstsq_fit(w, t0, t1):
    cols = [np.ones(128), t0.astype(np.float64)]
    if t1.any():
        cols.append(t1.astype(np.float64))
    A = np.stack(cols, 1)
    keep = [0] + [j for j in range(1, A.shape[1]) if A[:, j].any()]
    coef = np.zeros(3)
    sol = np.linalg.lstsq(A[:, keep], w, rcond=None)[0]
    for j, c in zip(keep, sol):
        coef[j] = c
    return coef


def test_refinement_converges_to_least_squares():
    """With the supports fixed, many alternating sweeps reach the float64
    least-squares (mu, alpha0, alpha1) of w on [1, T0, T1]."""
    N, K = 8, 1024
    W = wl.gen_dense_weights(N, K, proj=5)
    r = tz.ternarize(W, nnz=20, sweeps=200)
    w = W.view(np.float16).astype(np.float64).reshape(N * K // 128, 128)
    T0 = r["T1"].reshape(-1, 128)
    T1 = r["T2"].reshape(-1, 128)
    got = np.stack([r["mu"].ravel(), r["alpha0"].ravel(), r["alpha1"].ravel()], 1).astype(np.float64)
    for i in range(w.shape[0]):
        want = _lstsq_fit(w[i], T0[i], T1[i])
        np.testing.assert_allclose(got[i], want, rtol=2e-4, atol=2e-6, err_msg=f"block {i}")


def test_refinement_never_raises_error():
    """Each sweep minimises the squared error over one parameter exactly, so
    the float64 error of the fit is non-increasing over sweeps (up to the
    float32 rounding of the parameters)."""
    W = wl.gen_dense_weights(6, 768, proj=6)
    w = W.view(np.float16).astype(np.float64).reshape(-1, 128)
    prev = None
    for s in range(6):
        r = tz.ternarize(W, nnz=9, sweeps=s)
        fit = (r["mu"].reshape(-1, 1) + r["alpha0"].reshape(-1, 1) * r["T1"].reshape(-1, 128)
               + r["alpha1"].reshape(-1, 1) * r["T2"].reshape(-1, 128))
        err = ((w - fit) ** 2).sum(1)
        if prev is not None:
            assert np.all(err <= prev * (1 + 1e-5) + 1e-12)
        prev = err


def test_salience_is_top_energy():
    """The salient set is the nnz largest energies, ties by lower block id,
    checked with Python's sorted() over (energy, id) pairs."""
    W = wl.gen_dense_weights(32, 384, proj=7)
    W[5] = W[4]  # duplicate rows: equal energies
    W[9] = W[4]
    for nnz in (0, 1, 17, 50, 96):
        r = tz.ternarize(W, nnz=nnz, sweeps=1)
        E = [float(v) for v in r["E"].ravel()]
        want = set(sorted(range(len(E)), key=lambda i: (-E[i], i))[:nnz])
        assert set(np.flatnonzero(r["salient"].ravel())) == want
        assert int(r["sal"].astype(np.uint64).sum() > 0) == int(nnz > 0)


def test_degenerate_blocks():
    """A constant block has no support (its centred values are all 0), scale
    0, offset the constant; all-zero weights with every block salient give
    all-zero planes and scales."""
    W = np.zeros((2, 256), np.float16)
    W[0, :128] = 0.375
    W[1, 128:] = -2.0
    r = tz.ternarize(W.view(np.uint16), nnz=4, sweeps=4)
    assert not r["T1"].any() and not r["T2"].any()
    assert np.array_equal(r["mu"], np.array([[0.375, 0], [0, -2.0]], F32))
    assert not r["alpha0"].any() and not r["alpha1"].any()
    assert r["salient"].all() and r["s2"].size == 4 and not r["s2"].any()


def test_output_reconstructs_through_packed_oracle(oracle_mod):
    """The ternarizer's output is a valid packed weight: the C oracle packs
    it, and its fp64 linear layer with identity activations returns
    fp16(mu) + fp16(alpha0) T0 + fp16(alpha1) T1 for every weight."""
    N, K = 5, 256
    W = wl.gen_dense_weights(N, K, proj=8)
    r = tz.ternarize(W, nnz=3, sweeps=4)
    rp, st = oracle_mod.rowptr(N, K, r["sal"])
    assert st == 0 and rp[N] == 3
    p1, p2, st = oracle_mod.pack(N, K, r["T1"], r["T2"], r["sal"], rp)
    assert st == 0
    x = np.eye(K, dtype=np.float16).view(np.uint16)
    y, _ = oracle_mod.linear(K, N, K, p1, p2, r["sal"], r["s1"], r["off"], r["s2"], x, nthreads=1)
    h = lambda b: b.view(np.float16).astype(np.float64)
    s2d = np.zeros(N * K // 128)
    s2d[r["salient"].ravel()] = h(r["s2"])
    rep = lambda v: np.repeat(v.reshape(N, K // 128), 128, axis=1)
    want = rep(h(r["off"])) + rep(h(r["s1"])) * r["T1"] + rep(s2d) * r["T2"]
    np.testing.assert_array_equal(y.T, want)


@pytest.mark.parametrize("second", [False, True])
def test_threshold_factor_boundary(second):
    """The factor 0.75 of the thresholds (E2M-ATQ, eq. for Delta0; the second
    support reuses it).  A zero-mean block of 32 entries each at +u, -u, +v u,
    -v u (0 < v < 1) has mean |value| (1 + v) u / 2, so its inner entries are
    in the support iff v u > 0.75 (1 + v) u / 2, i.e. v > 0.6: v = 38/64 is
    out, v = 39/64 is in (a factor f moves the boundary to f / (2 - f):
    0.7 puts both in, 0.8 both out).  For the second support 16 entries each
    at +u, -u, +v u, -v u (u = 1/64) sit on the 64 zeros of a first plane of
    scale 1/2, whose least-squares scale they do not disturb; the residual's
    mean |value| is then (1 + v) u / 4 and the boundary v > 0.75 / 3.25
    (0.2308): v = 14/64 is out, v = 15/64 is in (0.7 puts both in, 0.8 both
    out)."""
    rng = np.random.default_rng(9)
    blocks, want = [], []
    lo, hi, bound = (14 / 64, 15 / 64, 0.75 / 3.25) if second else (38 / 64, 39 / 64, 0.6)
    for v in (lo, hi):
        for _ in range(4):
            perm = rng.permutation(128)
            pat = np.zeros(128)
            q = 16 if second else 32
            u = 1 / 64 if second else 1.0
            pat[perm[:q]], pat[perm[q:2 * q]] = u, -u
            pat[perm[2 * q:3 * q]], pat[perm[3 * q:4 * q]] = v * u, -v * u
            inner = np.zeros(128, np.int8)
            if v > bound:
                inner[perm[2 * q:3 * q]], inner[perm[3 * q:4 * q]] = 1, -1
            outer = np.zeros(128, np.int8)
            outer[perm[:q]], outer[perm[q:2 * q]] = 1, -1
            if second:
                t0 = np.zeros(128, np.int8)
                t0[perm[64:96]], t0[perm[96:]] = 1, -1
                w = 0.5 * t0 + pat
                want.append((t0, outer + inner))
            else:
                w = pat
                want.append((outer + inner, np.zeros(128, np.int8)))
            blocks.append(w)
    W = np.asarray(blocks).astype(np.float16)
    assert np.array_equal(W.astype(np.float64), np.asarray(blocks))
    r = tz.ternarize(W.view(np.uint16).reshape(2, 4 * 128), nnz=8 if second else 0, sweeps=0)
    for i, (t0, t1) in enumerate(want):
        assert np.array_equal(r["T1"].reshape(8, 128)[i], t0), i
        assert np.array_equal(r["T2"].reshape(8, 128)[i], t1), i


def test_moment_form_of_the_sweeps():
    """The GPU runs each refinement sweep on seven moments of the block (n0,
    n1, sum T0, sum T1, sum T0 T1, sum w, sum w T0, sum w T1) instead of
    passes over the weights.  In float64 the two forms are the same
    coordinate updates: they agree to rounding on every block, salient or not."""
    W = wl.gen_dense_weights(12, 1024, proj=13)
    r = tz.ternarize(W, nnz=25, sweeps=0)
    w = W.view(np.float16).astype(np.float64).reshape(-1, 128)
    T0 = r["T1"].reshape(-1, 128).astype(np.float64)
    T1 = r["T2"].reshape(-1, 128).astype(np.float64)
    mu = r["mu"].ravel().astype(np.float64)
    a0 = r["alpha0"].ravel().astype(np.float64)
    a1 = r["alpha1"].ravel().astype(np.float64)
    n0, n1 = np.abs(T0).sum(1), np.abs(T1).sum(1)
    safe = lambda v, n: np.where(n > 0, v / np.maximum(n, 1), 0.0)
    # passes over the weights (the oracle's order of updates)
    pm, p0, p1 = mu.copy(), a0.copy(), a1.copy()
    # moments
    z0, z1, z01 = T0.sum(1), T1.sum(1), (T0 * T1).sum(1)
    sw, sw0, sw1 = w.sum(1), (w * T0).sum(1), (w * T1).sum(1)
    mm, m0, m1 = mu.copy(), a0.copy(), a1.copy()
    # the second plane's first scale: least squares of r = w - mu - alpha0 T0 on T1
    r_first = safe(((w - mu[:, None] - a0[:, None] * T0) * T1).sum(1), n1)
    np.testing.assert_allclose(safe(sw1 - mu * z1 - a0 * z01, n1), r_first, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(r_first, a1, rtol=1e-5, atol=1e-9)  # the oracle's float32 value
    for _ in range(4):
        pm = (w - p0[:, None] * T0 - p1[:, None] * T1).mean(1)
        p0 = safe(((w - pm[:, None] - p1[:, None] * T1) * T0).sum(1), n0)
        p1 = safe(((w - pm[:, None] - p0[:, None] * T0) * T1).sum(1), n1)
        mm = (sw - m0 * z0 - m1 * z1) / 128
        m0 = safe(sw0 - mm * z0 - m1 * z01, n0)
        m1 = safe(sw1 - mm * z1 - m0 * z01, n1)
    assert r["salient"].sum() == 25
    np.testing.assert_allclose(mm, pm, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(m0, p0, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(m1, p1, rtol=1e-12, atol=1e-15)
