"""GPU parity of tq_ternarize (E2M-ATQ, paper "Conversion Pipeline") against
the float32 oracle: salience, rowptr and both packed planes bit for bit (both
sides take every decision in IEEE float32 with sums in index order); the
fp16 offsets and scales within one fp16 unit in the last place (the GPU runs
the refinement sweeps on each block's moments, the oracle in passes over the
weights: the same updates, rounded differently in float32)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from oracle import ternarize as tz

pytestmark = pytest.mark.gpu


def _host(t, dtype):
    return t.contiguous().cpu().numpy().view(dtype)


def assert_f16_within_ulp(got, want, what):
    """fp16 bit patterns at most one fp16 ulp apart; on large arrays at least
    98 % identical.

    Where the 98 % comes from: the two sides compute each parameter in float32
    from sums of one 128-weight block, in different orders. The worst-case
    relative error of a 128-term float32 sum is about 128 x 2^-24 = 2^-17. The
    two fp16 roundings differ only if the float32 value lies that close to an
    fp16 rounding midpoint. Midpoints are at least 2^-11 apart relative to the
    value, so a flip happens for at most 2^-17 / 2^-11 = 2^-6 (about 1.6 %) of
    well-conditioned values. The 2 % gate adds a small margin for the sweeps'
    few further operations."""
    g = got.view(np.float16).astype(np.float64)
    w = want.view(np.float16).astype(np.float64)
    ulp = np.spacing(np.maximum(np.abs(g), np.abs(w)).astype(np.float16)).astype(np.float64)
    bad = np.abs(g - w) > ulp
    if bad.any():
        i = np.flatnonzero(bad.ravel())[0]
        raise AssertionError(f"{what}: {bad.sum()} values more than 1 ulp apart, first {g.ravel()[i]} vs {w.ravel()[i]}")
    if got.size >= 1000:
        assert (got == want).mean() >= 0.98, f"{what}: {(got == want).mean():.4f} bit-identical"


def compare(W_bits, nnz, sweeps, index=False):
    """Ternarize on the GPU and with the oracle; assert the integer outputs
    equal and the fp16 parameters within one ulp."""
    from paper_2609_09240_gb300 import tq
    N, K = W_bits.shape
    Wd = torch.from_numpy(np.ascontiguousarray(W_bits).view(np.float16)).cuda()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    pw = tq.ternarize(Wd, nnz, sweeps=sweeps, d_status=st, index=index)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    r = tz.ternarize(W_bits, nnz, sweeps=sweeps)
    rp, s = oracle.rowptr(N, K, r["sal"])
    assert s == 0
    p1, p2, s = oracle.pack(N, K, r["T1"], r["T2"], r["sal"], rp)
    assert s == 0
    sal = _host(pw.salience, np.uint32)
    if not np.array_equal(sal, r["sal"]):
        bad = np.argwhere(sal != r["sal"])[0]
        raise AssertionError(f"salience differs first at word {tuple(bad)}")
    assert np.array_equal(_host(pw.rowptr, np.int32), rp)
    assert_f16_within_ulp(_host(pw.offset, np.uint16), r["off"], "offset")
    assert_f16_within_ulp(_host(pw.scale1, np.uint16), r["s1"], "scale1")
    g1 = _host(pw.plane1, np.uint8)
    if not np.array_equal(g1, p1):
        bad = np.argwhere(g1 != p1)[0]
        raise AssertionError(f"plane 1 differs first at {tuple(bad)}")
    if nnz:
        assert np.array_equal(_host(pw.plane2, np.uint8)[:nnz], p2), "plane 2"
        assert_f16_within_ulp(_host(pw.scale2, np.uint16)[:nnz], r["s2"], "scale2")
    return pw, r


@pytest.mark.parametrize("N,K,frac", [(1, 128, 0.0), (1, 128, 1.0), (37, 384, 0.1), (256, 1024, 0.1),
                                      (300, 2560, 0.1), (130, 4224, 0.25), (64, 12288, 0.1), (97, 640, 1.0)])
@pytest.mark.parametrize("sweeps", [0, 4])
def test_ternarize_parity(N, K, frac, sweeps):
    W = wl.gen_dense_weights(N, K, config=9, proj=N + K)
    compare(W, int(round(frac * N * (K // 128))), sweeps)


def test_ternarize_ties_in_energy():
    """Duplicated rows and constant blocks give equal energies across the
    selection boundary: the lower block ids win on both sides."""
    W = wl.gen_dense_weights(40, 1024, config=9, proj=1)
    W[7] = W[3]
    W[8] = W[3]
    W[20:30] = np.float16(0.25).view(np.uint16)  # constant blocks: energy 0
    G = 8
    for nnz in (3, 31 * G + 5, 32 * G, 34 * G + 2):
        compare(W, nnz, 4)


def test_ternarize_degenerate():
    """All-zero weights, every block salient: zero planes and scales."""
    W = np.zeros((9, 256), np.uint16)
    pw, r = compare(W, 18, 4)
    assert not r["T1"].any()


def test_ternarize_full_size_gate_projection():
    """A Qwen3-8B gate projection (12288 x 4096, 10 % salient groups, four
    refinement sweeps) in one call, every output compared."""
    W = wl.gen_dense_weights(12288, 4096, config=9, proj=100)
    compare(W, int(round(0.1 * 12288 * 32)), 4, index=True)


def test_ternarize_then_linear():
    """The ternarized weight runs through the decode path like any packed
    weight: tq_linear against the fp64 oracle on the oracle's own planes."""
    import gpu_helpers as H
    from paper_2609_09240_gb300 import tq
    N, K = 520, 2560
    W = wl.gen_dense_weights(N, K, config=9, proj=2)
    nnz = int(round(0.1 * N * K / 128))
    pw, r = compare(W, nnz, 4, index=True)
    x = wl.gen_x(3, K, config=9, proj=2)
    y = tq.tq_linear_f32out(H.dev(x), pw)
    H.device_status_ok()
    rp, _ = oracle.rowptr(N, K, r["sal"])
    p1, p2, _ = oracle.pack(N, K, r["T1"], r["T2"], r["sal"], rp)
    y_ref, a_ref = oracle.linear(3, N, K, p1, p2, r["sal"], r["s1"], r["off"], r["s2"], x)
    H.assert_close(y.cpu().numpy(), y_ref, a_ref)


def test_ternarize_nonfinite_weight_flagged():
    """An inf weight sets TQ_DATA_BAD_WEIGHT; the call still completes."""
    from paper_2609_09240_gb300 import tq
    W = wl.gen_dense_weights(8, 256, config=9, proj=3).view(np.float16).copy()
    W[2, 77] = np.inf
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    tq.ternarize(torch.from_numpy(W).cuda(), 2, d_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & 32


def test_ternarize_argument_errors():
    import ctypes
    from paper_2609_09240_gb300 import tq
    L = tq.lib()
    N, K = 16, 256
    W = torch.zeros((N, K), dtype=torch.float16, device="cuda")
    p1 = torch.empty((N, tq.tq_row_bytes(K)), dtype=torch.uint8, device="cuda")
    sal = torch.empty((N, 1), dtype=torch.int32, device="cuda")
    rp = torch.empty(N + 1, dtype=torch.int32, device="cuda")
    p2 = torch.empty((32, 26), dtype=torch.uint8, device="cuda")
    s = torch.empty((N, 2), dtype=torch.float16, device="cuda")
    s2 = torch.empty(32, dtype=torch.float16, device="cuda")
    nb = tq.tq_ternarize_workspace_bytes(N, K)
    ws = tq.workspace(nb, "cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    P = lambda t: ctypes.c_void_p(t.data_ptr())
    strm = tq._stream(None)
    call = lambda **kw: L.tq_ternarize(kw.get("N", N), K, kw.get("W", P(W)), kw.get("nnz", 4), kw.get("sweeps", 4),
                                       P(p1), P(sal), P(rp), P(p2), P(s), P(s), P(s2), kw.get("ws", P(ws)),
                                       kw.get("nb", nb), P(st), strm)
    assert call(nnz=33) == -2           # more salient blocks than blocks
    assert call(nnz=-1) == -2
    assert call(sweeps=65) == -2
    assert call(nb=nb - 1) == -2        # workspace too small
    assert call(W=None) == -1
    assert call(ws=None) == -1
    Wb = torch.zeros(N * K + 8, dtype=torch.float16, device="cuda")[1:N * K + 1]
    assert call(W=ctypes.c_void_p(Wb.data_ptr())) == -3
    assert call() == 0
    torch.cuda.synchronize()
