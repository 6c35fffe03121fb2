"""GPU parity of the element-wise four-mask representation (orders [2, 2, 1,
1]) against the fp64 oracle (oracle/elementwise.py): tq_ew_rowptr / tq_ew_pack
bytes equal the oracle's packing bit for bit and tq_ew_unpack inverts them;
tq_ew_linear satisfies |y - y_ref| <= 2e-3 * sum_k |W x| per element on
ragged shapes, 1..40 tokens (decode and prefill paths under the mask-3 pass)
and Qwen3-8B projection shapes (sampled rows); tq_ew_linear_batched meets
the same bound on mixed batches and on a Qwen3-8B layer's seven
projections; the correction index equals the oracle's bit for bit, reports
offsets that do not match the mask plane, and the linear through it meets
the bound on every path above, alone and mixed with index-less weights in
one batched call."""
import ctypes

import numpy as np
import pytest
import torch

import workloads as wl
from oracle import elementwise as ew

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    import gpu_helpers
    return gpu_helpers


def _pack(H, w):
    from paper_2609_09240_gb300 import tq
    return tq.pack_ew_weight(H.dev(w.T0), H.dev(w.T1), H.dev(w.mask), H.dev(w.mu), H.dev(w.a0), H.dev(w.a1))


def _np(t, dtype):
    return np.ascontiguousarray(t.cpu().numpy()).view(dtype)


@pytest.mark.parametrize("N,K", [(1, 128), (37, 256), (300, 1152), (129, 4096), (64, 12288)])
def test_codec_bit_exact(H, N, K):
    from paper_2609_09240_gb300 import tq
    w = wl.gen_ew_weights(N, K, config=12, proj=N)
    mp, p1, rp, p2, st = ew.pack(w.T0, w.T1, w.mask)
    assert st == 0
    g = _pack(H, w)
    torch.cuda.synchronize()
    assert np.array_equal(_np(g.p2rowptr, np.int32), rp)
    assert np.array_equal(_np(g.mask, np.uint32), mp)
    assert np.array_equal(_np(g.plane1, np.uint8), p1)
    assert np.array_equal(_np(g.plane2, np.uint8)[:rp[N]], p2)
    T0, T1, m = tq.tq_ew_unpack(g)
    torch.cuda.synchronize()
    assert np.array_equal(T0.cpu().numpy(), w.T0) and np.array_equal(T1.cpu().numpy(), w.T1)
    assert np.array_equal(m.cpu().numpy(), w.mask)


def test_codec_coverage_extremes(H):
    """Rows with no order-2 element, rows entirely of mask 0, and order-2
    counts of every residue mod 5."""
    N, K = 10, 256
    w = wl.gen_ew_weights(N, K, config=13)
    mask = np.full((N, K), 3, np.uint8)
    mask[1] = 0
    for r in range(2, 7):
        mask[r, : (r - 2) + 5 * r] = 1
    mask[7, ::2] = 2
    T1 = (w.T1 * 0 + wl._trits(np.random.default_rng(3), (N, K))) * (mask <= 1)
    T1 = T1.astype(np.int8)
    mp, p1, rp, p2, st = ew.pack(w.T0, T1, mask)
    assert st == 0
    w2 = wl.EwWeights(N, K, w.T0, T1, mask, w.mu, w.a0, w.a1)
    g = _pack(H, w2)
    torch.cuda.synchronize()
    assert np.array_equal(_np(g.p2rowptr, np.int32), rp)
    assert np.array_equal(_np(g.plane2, np.uint8)[:rp[N]], p2)


def test_codec_flags_bad_data(H):
    from paper_2609_09240_gb300 import tq
    N, K = 4, 256
    w = wl.gen_ew_weights(N, K, config=14)
    dev = lambda a: H.dev(a)
    # T1 nonzero on an order-1 element
    T1 = w.T1.copy()
    k = int(np.argwhere(w.mask[0] >= 2)[0][0])
    T1[0, k] = -1
    with pytest.raises(tq.TQError):
        tq.pack_ew_weight(dev(w.T0), dev(T1), dev(w.mask), dev(w.mu), dev(w.a0), dev(w.a1))
    # a mask id above 3
    mask = w.mask.copy()
    mask[2, 5] = 7
    with pytest.raises(tq.TQError):
        tq.pack_ew_weight(dev(w.T0), dev(w.T1), dev(mask), dev(w.mu), dev(w.a0), dev(w.a1))
    # a plane-2 byte above 242 is reported by unpack
    g = _pack(H, w)
    g.plane2[0] = 250
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    tq.tq_ew_unpack(g, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & 4


@pytest.mark.parametrize("M,N,K", [(1, 512, 1024), (2, 300, 2560), (5, 129, 4224), (16, 1000, 640), (40, 256, 1152),
                                   (1, 1, 128)])
@pytest.mark.parametrize("f32", [False, True])
def test_linear_parity(H, M, N, K, f32):
    from paper_2609_09240_gb300 import tq
    w = wl.gen_ew_weights(N, K, config=15, proj=M + N)
    xb = wl.gen_x(M, K, config=15, proj=M + N)
    mp, p1, rp, p2, st = ew.pack(w.T0, w.T1, w.mask)
    assert st == 0
    y_ref, a_ref = ew.linear(xb, K, mp, p1, rp, p2, w.mu, w.a0, w.a1)
    y = tq.tq_ew_linear(H.dev(xb), _pack(H, w), f32=f32)
    H.device_status_ok()
    H.assert_close(y.float().cpu().numpy().astype(np.float64), y_ref, a_ref)


@pytest.mark.parametrize("N,K", [(4096, 4096), (12288, 4096), (4096, 12288)])
def test_linear_qwen3_8b_shapes_sampled_rows(H, N, K):
    from paper_2609_09240_gb300 import tq
    w = wl.gen_ew_weights(N, K, config=16, proj=N // 1024)
    xb = wl.gen_x(1, K, config=16, proj=N // 1024)
    mp, p1, rp, p2, st = ew.pack(w.T0, w.T1, w.mask)
    assert st == 0
    rows = np.sort(np.random.default_rng(N).choice(N, size=64, replace=False))
    y_ref, a_ref = ew.linear(xb, K, mp, p1, rp, p2, w.mu, w.a0, w.a1, rows=rows)
    y = tq.tq_ew_linear(H.dev(xb), _pack(H, w))
    H.device_status_ok()
    H.assert_close(y.float().cpu().numpy()[:, rows].astype(np.float64), y_ref, a_ref)


@pytest.mark.parametrize("M", [1, 2, 5, 16])
def test_batched_parity_mixed_shapes(H, M):
    from paper_2609_09240_gb300 import tq
    shapes = [(512, 1024), (37, 256), (300, 2560), (129, 4224), (1, 128)]
    items, refs = [], []
    for i, (N, K) in enumerate(shapes):
        w = wl.gen_ew_weights(N, K, config=17, proj=i)
        xb = wl.gen_x(M, K, config=17, proj=i)
        mp, p1, rp, p2, st = ew.pack(w.T0, w.T1, w.mask)
        assert st == 0
        refs.append(ew.linear(xb, K, mp, p1, rp, p2, w.mu, w.a0, w.a1))
        items.append((_pack(H, w), H.dev(xb), torch.empty((M, N), dtype=torch.float16, device="cuda")))
    b = tq.EwBatch(M, items)
    tq.tq_ew_linear_batched(b)
    H.device_status_ok()
    for (_, _, y), (y_ref, a_ref) in zip(items, refs):
        H.assert_close(y.float().cpu().numpy().astype(np.float64), y_ref, a_ref)


def test_batched_qwen3_8b_layer_sampled_rows(H):
    """The seven projections of a Qwen3-8B layer in one batched call, M = 1,
    64 sampled rows of each against the oracle; the same problems through
    tq_ew_linear one by one agree within the bound as well."""
    from paper_2609_09240_gb300 import tq
    items, refs, singles = [], [], []
    for p in wl.config_projections(4):
        w = wl.gen_ew_weights(p.N, p.K, config=18, proj=p.proj)
        xb = wl.gen_x(1, p.K, config=18, proj=p.proj)
        mp, p1, rp, p2, st = ew.pack(w.T0, w.T1, w.mask)
        assert st == 0
        rows = np.sort(np.random.default_rng(p.proj).choice(p.N, size=64, replace=False))
        refs.append((rows, ew.linear(xb, p.K, mp, p1, rp, p2, w.mu, w.a0, w.a1, rows=rows)))
        g = _pack(H, w)
        x = H.dev(xb)
        items.append((g, x, torch.empty((1, p.N), dtype=torch.float16, device="cuda")))
        singles.append(tq.tq_ew_linear(x, g))
    tq.tq_ew_linear_batched(tq.EwBatch(1, items))
    H.device_status_ok()
    for (_, _, y), ys, (rows, (y_ref, a_ref)) in zip(items, singles, refs):
        H.assert_close(y.float().cpu().numpy()[:, rows].astype(np.float64), y_ref, a_ref)
        H.assert_close(ys.float().cpu().numpy()[:, rows].astype(np.float64), y_ref, a_ref)


def test_batched_rejects_bad_arguments(H):
    from paper_2609_09240_gb300 import tq
    w = _pack(H, wl.gen_ew_weights(64, 256, config=19))
    x = torch.zeros((17, 256), dtype=torch.float16, device="cuda")
    y = torch.empty((17, 64), dtype=torch.float16, device="cuda")
    with pytest.raises(tq.TQError):
        tq.EwBatch(17, [(w, x, y)])  # M > 16: no batched workspace
    b = tq.EwBatch(1, [(w, x[:1], y[:1])])
    b.arr[0].x = b.arr[0].x + 2  # misaligned activations
    with pytest.raises(tq.TQError):
        tq.tq_ew_linear_batched(b)


def _indexed(H, w):
    from paper_2609_09240_gb300 import tq
    return tq.ew_index(_pack(H, w))


@pytest.mark.parametrize("N,K", [(1, 128), (37, 1024), (300, 1152), (129, 4224), (64, 12288)])
def test_index_bit_exact(H, N, K):
    w = wl.gen_ew_weights(N, K, config=20, proj=N)
    off, ent = ew.correction_index(w.T0, w.T1, w.mask)
    g = _indexed(H, w)
    torch.cuda.synchronize()
    assert np.array_equal(_np(g.idx_off, np.int32), off)
    assert np.array_equal(_np(g.idx, np.uint16)[:off[-1]], ent)


def test_index_reports_offsets_that_do_not_match(H):
    from paper_2609_09240_gb300 import tq
    N, K = 16, 2048
    a = _indexed(H, wl.gen_ew_weights(N, K, config=21, proj=0))
    b = _pack(H, wl.gen_ew_weights(N, K, config=21, proj=1))
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    idx = torch.zeros_like(a.idx)
    s_ = b.struct()
    assert tq.lib().tq_ew_index_fill(N, K, ctypes.byref(s_), a.idx_off.data_ptr(), idx.data_ptr(), st.data_ptr(),
                                     None) == 0
    torch.cuda.synchronize()
    assert int(st.item()) & 0x10  # TQ_DATA_BAD_ROWPTR


@pytest.mark.parametrize("M,N,K", [(1, 512, 1024), (2, 300, 2560), (5, 129, 4224), (16, 1000, 640), (40, 256, 1152),
                                   (1, 1, 128)])
@pytest.mark.parametrize("f32", [False, True])
def test_linear_parity_indexed(H, M, N, K, f32):
    from paper_2609_09240_gb300 import tq
    w = wl.gen_ew_weights(N, K, config=22, proj=M + N)
    xb = wl.gen_x(M, K, config=22, proj=M + N)
    mp, p1, rp, p2, st = ew.pack(w.T0, w.T1, w.mask)
    y_ref, a_ref = ew.linear(xb, K, mp, p1, rp, p2, w.mu, w.a0, w.a1)
    y = tq.tq_ew_linear(H.dev(xb), _indexed(H, w), f32=f32)
    H.device_status_ok()
    H.assert_close(y.float().cpu().numpy().astype(np.float64), y_ref, a_ref)


@pytest.mark.parametrize("M", [1, 3])
def test_batched_mixed_indexed_and_plain(H, M):
    """Problems with and without a correction index in one batched call (the
    two correction kernels share the call)."""
    from paper_2609_09240_gb300 import tq
    shapes = [(512, 4096), (300, 1152), (1024, 12288), (37, 256)]
    items, refs = [], []
    for i, (N, K) in enumerate(shapes):
        w = wl.gen_ew_weights(N, K, config=23, proj=i)
        xb = wl.gen_x(M, K, config=23, proj=i)
        mp, p1, rp, p2, st = ew.pack(w.T0, w.T1, w.mask)
        rows = np.arange(N) if N <= 512 else np.sort(np.random.default_rng(i).choice(N, 64, replace=False))
        refs.append((rows, ew.linear(xb, K, mp, p1, rp, p2, w.mu, w.a0, w.a1, rows=rows)))
        g = _indexed(H, w) if i % 2 == 0 else _pack(H, w)
        items.append((g, H.dev(xb), torch.empty((M, N), dtype=torch.float16, device="cuda")))
    tq.tq_ew_linear_batched(tq.EwBatch(M, items))
    H.device_status_ok()
    for (_, _, y), (rows, (y_ref, a_ref)) in zip(items, refs):
        H.assert_close(y.float().cpu().numpy()[:, rows].astype(np.float64), y_ref, a_ref)


@pytest.mark.parametrize("N,K", [(4096, 4096), (12288, 4096), (4096, 12288)])
def test_linear_indexed_qwen3_8b_shapes_sampled_rows(H, N, K):
    from paper_2609_09240_gb300 import tq
    w = wl.gen_ew_weights(N, K, config=24, proj=N // 1024)
    xb = wl.gen_x(1, K, config=24, proj=N // 1024)
    mp, p1, rp, p2, st = ew.pack(w.T0, w.T1, w.mask)
    rows = np.sort(np.random.default_rng(N + 1).choice(N, size=64, replace=False))
    y_ref, a_ref = ew.linear(xb, K, mp, p1, rp, p2, w.mu, w.a0, w.a1, rows=rows)
    y = tq.tq_ew_linear(H.dev(xb), _indexed(H, w))
    H.device_status_ok()
    H.assert_close(y.float().cpu().numpy()[:, rows].astype(np.float64), y_ref, a_ref)
