"""CPU oracle of the E2M-ATQ ternarizer (paper "Conversion Pipeline", subsection
"E2M-ATQ", and "Model and Representation", eq. for W-hat).

TEST INFRASTRUCTURE ONLY: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU legs of ``bench.py`` may import it; the CUDA library never calls it.

What it computes, for every masked block (this library's block is one row n
and one group g of 128 consecutive columns, the per-group reading used by the
packed format), with w the block's 128 fp16 weights read as float32:

1. mu = rowmean(w), Wc = w - mu                      (E2M-ATQ, mean and centring)
2. Delta0 = 0.75 * rowmean(|Wc|)                     (E2M-ATQ, first threshold)
3. T0 = +1 where Wc > Delta0, -1 where Wc < -Delta0, else 0   (first support)
4. alpha0 = sum(Wc * T0) / sum(T0^2), 0 for an empty support  (least-squares
   scale of the support, mu held fixed)
5. residual R = Wc - alpha0 * T0; its energy E = sum(R^2)
6. salience: the `nnz` blocks of the projection with the largest E get a
   second plane (ties: lower block id n * G + g first)
7. on those blocks the residual is quantized like the weights were:
   Delta1 = 0.75 * rowmean(|R|), T1 from R at Delta1, alpha1 = sum(R * T1) /
   sum(T1^2); other blocks have T1 = 0 and alpha1 = 0
8. alternating refinement with the supports fixed, `sweeps` times:
   mu <- mean(w - alpha0 T0 - alpha1 T1), then alpha0 <- least squares of
   w - mu - alpha1 T1 on T0, then alpha1 <- least squares of w - mu - alpha0 T0
   on T1 (salient blocks only)
9. stored: offset = fp16(mu), scale1 = fp16(alpha0), scale2 = fp16(alpha1),
   plane-1 trits = T0, plane-2 trits = T1 (the packed format calls them T1 and
   T2).

Readings where the paper is silent (each also listed with the library's
design notes): the block is (row, group of 128); the second support uses the
first support's threshold rule on the residual; salience is the top-`nnz`
residual energy after the first plane; the refinement order is mu, alpha0,
alpha1 and the sweep count is a parameter (4 by default).

Precision.  The supports and the salience set are integer decisions taken
from floating-point values, so this oracle and the CUDA kernels take them in
the same arithmetic: IEEE float32, round to nearest even, no fused
multiply-add, every sum over a block accumulated in index order 0..127
starting from +0, a mean as the sum times 1/128, and the fp16 outputs
rounded to nearest even from float32.  numpy's float32 element-wise
operations are exactly these operations, one rounding each.
"""
from __future__ import annotations

import numpy as np

GROUP = 128
F32 = np.float32
INV_GROUP = F32(1.0 / GROUP)  # exact power of two
THRESH = F32(0.75)


def _sum_in_order(v: np.ndarray) -> np.ndarray:
    """Row sums of v (blocks, 128) in float32, columns added in index order from +0."""
    s = np.zeros(v.shape[0], F32)
    for i in range(v.shape[1]):
        s = np.add(s, v[:, i], dtype=F32)
    return s


def _times_trit(v: np.ndarray, t: np.ndarray) -> np.ndarray:
    """v * t for t in {-1, 0, +1}: v, -v or +0 (exact)."""
    return np.where(t > 0, v, np.where(t < 0, -v, F32(0))).astype(F32)


def _trit_times(a: np.ndarray, t: np.ndarray) -> np.ndarray:
    """Per-block scale a times trits t: a, -a or +0 per element (exact)."""
    a = a[:, None]
    return np.where(t > 0, a, np.where(t < 0, -a, F32(0))).astype(F32)


def _support(v: np.ndarray, delta: np.ndarray) -> np.ndarray:
    """Ternary support of v at per-block threshold delta (E2M-ATQ, eq. for T0)."""
    t = np.zeros(v.shape, np.int8)
    d = delta[:, None]
    t[v > d] = 1
    t[v < -d] = -1
    return t


def _ls_scale(v: np.ndarray, t: np.ndarray, n: np.ndarray) -> np.ndarray:
    """Least-squares scale of v on support t: sum(v t) / sum(t^2), 0 if the support is empty."""
    num = _sum_in_order(_times_trit(v, t))
    den = n.astype(F32)
    out = np.zeros_like(num)
    np.divide(num, den, out=out, where=n > 0)
    return out.astype(F32)


def first_plane(w: np.ndarray):
    """Steps 1-5 for blocks w (B, 128) float32.

    Returns mu, delta0, T0, alpha0, E (E as float32)."""
    w = np.asarray(w, F32)
    mu = np.multiply(_sum_in_order(w), INV_GROUP, dtype=F32)
    c = np.subtract(w, mu[:, None], dtype=F32)
    delta0 = np.multiply(THRESH, np.multiply(_sum_in_order(np.abs(c)), INV_GROUP, dtype=F32), dtype=F32)
    t0 = _support(c, delta0)
    n0 = np.abs(t0).sum(axis=1)
    a0 = _ls_scale(c, t0, n0)
    r = np.subtract(c, _trit_times(a0, t0), dtype=F32)
    e = _sum_in_order(np.multiply(r, r, dtype=F32))
    return mu, delta0, t0, a0, e


def select_salient(e: np.ndarray, nnz: int) -> np.ndarray:
    """Step 6: boolean mask of the nnz blocks with the largest E, ties by lower id.

    Compared as the float32 bit patterns, which order non-negative floats
    like their values (a NaN energy, from a non-finite weight, sorts first)."""
    e = np.ascontiguousarray(e, F32)
    keys = e.view(np.uint32).astype(np.int64)
    ids = np.arange(e.size, dtype=np.int64)
    order = np.lexsort((ids, -keys))  # primary: key descending; secondary: id ascending
    sal = np.zeros(e.size, bool)
    sal[order[:nnz]] = True
    return sal


def ternarize_blocks(w: np.ndarray, salient: np.ndarray, sweeps: int):
    """Steps 1-5, 7 and 8 for blocks w (B, 128) whose salience is given.

    Returns dict with float32 mu, alpha0, alpha1, int8 T0, T1 (B, 128) and E."""
    w = np.asarray(w, F32)
    mu, delta0, t0, a0, e = first_plane(w)
    n0 = np.abs(t0).sum(axis=1)
    c = np.subtract(w, mu[:, None], dtype=F32)
    r = np.subtract(c, _trit_times(a0, t0), dtype=F32)
    delta1 = np.multiply(THRESH, np.multiply(_sum_in_order(np.abs(r)), INV_GROUP, dtype=F32), dtype=F32)
    t1 = _support(r, delta1)
    t1[~salient] = 0
    n1 = np.abs(t1).sum(axis=1)
    a1 = _ls_scale(r, t1, n1)
    for _ in range(sweeps):
        u = np.subtract(np.subtract(w, _trit_times(a0, t0), dtype=F32), _trit_times(a1, t1), dtype=F32)
        mu = np.multiply(_sum_in_order(u), INV_GROUP, dtype=F32)
        c = np.subtract(w, mu[:, None], dtype=F32)
        a0 = _ls_scale(np.subtract(c, _trit_times(a1, t1), dtype=F32), t0, n0)
        a1 = _ls_scale(np.subtract(c, _trit_times(a0, t0), dtype=F32), t1, n1)
    return {"mu": mu, "alpha0": a0, "alpha1": a1, "T0": t0, "T1": t1, "E": e}


def _f16_bits(v: np.ndarray) -> np.ndarray:
    return np.asarray(v, F32).astype(np.float16).view(np.uint16)


def ternarize(W_bits: np.ndarray, nnz: int, sweeps: int = 4, row_chunk: int = 1024):
    """The whole projection: W_bits uint16 fp16 patterns [N][K], K % 128 == 0.

    Returns dict: T1, T2 int8 [N][K] (T2 zero outside salient groups),
    sal uint32 [N][ceil(G/32)], s1, off uint16 [N][G], s2 uint16 [nnz] in
    (row, group) order, and the float32 internals mu, alpha0, alpha1, E [N][G]."""
    W_bits = np.ascontiguousarray(W_bits, np.uint16)
    N, K = W_bits.shape
    assert K % GROUP == 0 and N >= 1
    G = K // GROUP
    assert 0 <= nnz <= N * G
    blocks = W_bits.view(np.float16).reshape(N * G, GROUP)
    # pass 1: energies of the whole projection
    e = np.empty(N * G, F32)
    step = row_chunk * G
    for b0 in range(0, N * G, step):
        e[b0:b0 + step] = first_plane(blocks[b0:b0 + step].astype(F32))[4]
    sal = select_salient(e, nnz)
    # pass 2: planes and refined parameters
    out = {k: np.empty(N * G, F32) for k in ("mu", "alpha0", "alpha1")}
    T1 = np.empty((N * G, GROUP), np.int8)
    T2 = np.empty((N * G, GROUP), np.int8)
    for b0 in range(0, N * G, step):
        r = ternarize_blocks(blocks[b0:b0 + step].astype(F32), sal[b0:b0 + step], sweeps)
        for k in out:
            out[k][b0:b0 + step] = r[k]
        T1[b0:b0 + step] = r["T0"]
        T2[b0:b0 + step] = r["T1"]
    SW = (G + 31) // 32
    salw = np.zeros((N, SW), np.uint32)
    sal2 = sal.reshape(N, G)
    for g in range(G):
        salw[:, g // 32] |= sal2[:, g].astype(np.uint32) << np.uint32(g % 32)
    return {
        "T1": T1.reshape(N, K), "T2": T2.reshape(N, K), "sal": salw,
        "s1": _f16_bits(out["alpha0"]).reshape(N, G), "off": _f16_bits(out["mu"]).reshape(N, G),
        "s2": _f16_bits(out["alpha1"][sal]),
        "mu": out["mu"].reshape(N, G), "alpha0": out["alpha0"].reshape(N, G),
        "alpha1": out["alpha1"].reshape(N, G), "E": e.reshape(N, G), "salient": sal2,
    }
