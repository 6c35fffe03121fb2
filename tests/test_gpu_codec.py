"""GPU codec parity: tq_salience_rowptr / tq_pack / tq_unpack against the CPU
oracle, bit-exact (paper "Packing": lossless re-encoding of the discrete
supports)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl

pytestmark = pytest.mark.gpu

SHAPES = [(1, 128, 0.0), (3, 128, 1.0), (7, 384, 0.3), (130, 1024, 0.1), (33, 2560, 0.1),
          (17, 4224, 0.5), (5, 9728, 0.1), (64, 12288, 0.1), (512, 1024, 0.0)]


@pytest.fixture(scope="module")
def H():
    import gpu_helpers
    return gpu_helpers


@pytest.mark.parametrize("N,K,frac", SHAPES)
def test_pack_unpack_bit_exact(H, N, K, frac):
    from paper_2609_09240_gb300 import tq
    w = wl.gen_weights(N, K, frac, config=7, proj=N + K)
    rp_o, st = oracle.rowptr(N, K, w.sal)
    assert st == 0
    p1_o, p2_o, st = oracle.pack(N, K, w.T1, w.T2, w.sal, rp_o)
    assert st == 0
    pw = H.pack_on_gpu(w)
    torch.cuda.synchronize()
    assert np.array_equal(pw.rowptr.cpu().numpy(), rp_o)
    assert pw.nnz == w.nnz
    assert np.array_equal(pw.plane1.cpu().numpy(), p1_o)
    if w.nnz:
        assert np.array_equal(pw.plane2.cpu().numpy()[:w.nnz], p2_o)
    # unpack the GPU bytes
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    T1 = torch.full((N, K), 7, dtype=torch.int8, device="cuda")
    T2 = torch.full((N, K), 7, dtype=torch.int8, device="cuda")
    tq.tq_unpack(N, K, pw.plane1, pw.plane2 if w.nnz else None, pw.salience, pw.rowptr, T1, T2, status)
    assert int(status.item()) == 0
    assert np.array_equal(T1.cpu().numpy(), w.T1)
    assert np.array_equal(T2.cpu().numpy(), w.T2)


@pytest.mark.parametrize("N,K,offset", [(37, 1024, 1), (9, 4224, 3), (3, 49280, 0)])
def test_pack_unpack_unstaged_paths(H, N, K, offset):
    """Code arrays that are not 16-byte aligned (offset into a larger buffer),
    or rows longer than the row-staged kernels take (K > 49152), go through
    the per-byte kernels; both must match the oracle bit for bit."""
    from paper_2609_09240_gb300 import tq
    w = wl.gen_weights(N, K, 0.2, config=7, proj=N + 3 * K)
    rp, st = oracle.rowptr(N, K, w.sal)
    p1_o, p2_o, st = oracle.pack(N, K, w.T1, w.T2, w.sal, rp)
    assert st == 0

    def codes(a):
        # a copy of a at `offset` bytes into a device buffer
        buf = torch.zeros(a.size + 16, dtype=torch.int8, device="cuda")
        v = buf[offset:offset + a.size]
        v.copy_(torch.from_numpy(np.ascontiguousarray(a).reshape(-1)))
        return v

    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    p1 = torch.empty((N, tq.tq_row_bytes(K)), dtype=torch.uint8, device="cuda")
    p2 = torch.empty((max(int(rp[N]), 1), 26), dtype=torch.uint8, device="cuda")
    tq.tq_pack(N, K, codes(w.T1), codes(w.T2), H.dev(w.sal), H.dev(rp), p1, p2, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert np.array_equal(p1.cpu().numpy(), p1_o)
    assert np.array_equal(p2.cpu().numpy()[:int(rp[N])], p2_o)
    T1 = codes(np.full(N * K, 7, np.int8))
    T2 = codes(np.full(N * K, 7, np.int8))
    tq.tq_unpack(N, K, p1, p2, H.dev(w.sal), H.dev(rp), T1, T2, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert np.array_equal(T1.cpu().numpy().reshape(N, K), w.T1)
    assert np.array_equal(T2.cpu().numpy().reshape(N, K), w.T2)


def test_unpack_reports_corruption_like_oracle(H):
    from paper_2609_09240_gb300 import tq
    N, K = 9, 512
    w = wl.gen_weights(N, K, 0.25, config=7, proj=1)
    rp, _ = oracle.rowptr(N, K, w.sal)
    p1, p2, _ = oracle.pack(N, K, w.T1, w.T2, w.sal, rp)
    cases = []
    b = p1.copy(); b[3, 10] = 250; cases.append((b, p2, rp, w.sal))
    b = p1.copy(); b[4, 25] = 0; cases.append((b, p2, rp, w.sal))             # tail pads 0
    b = p1.copy(); b[2, 26 * 4 + 3] = 99; cases.append((b, p2, rp, w.sal))    # row pad (104..111)
    q = p2.copy(); q[1, 7] = 255; cases.append((p1, q, rp, w.sal))            # plane-2 byte
    r = rp.copy(); r[5] += 1; r[6:] += 1; cases.append((p1, p2, r, w.sal))    # rowptr off by one
    for ci, (p1c, p2c, rpc, salc) in enumerate(cases):
        _, _, st_o = oracle.unpack(N, K, p1c, p2c, salc, rpc)
        assert st_o != 0
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        T1 = torch.empty((N, K), dtype=torch.int8, device="cuda")
        T2 = torch.empty((N, K), dtype=torch.int8, device="cuda")
        p2d = H.dev(np.vstack([p2c, np.zeros((1, 26), np.uint8)]))  # room for an over-long rowptr
        tq.tq_unpack(N, K, H.dev(p1c), p2d, H.dev(salc), H.dev(rpc), T1, T2, status)
        st = int(status.item())
        if ci == len(cases) - 1:
            # inconsistent rowptr: the GPU indexes plane 2 through rowptr (the
            # oracle recounts the salience bits), so besides BAD_ROWPTR it may
            # also flag what it finds in the records it was pointed at
            assert st & oracle.BAD_ROWPTR and not st & ~(oracle.BAD_ROWPTR | oracle.BAD_PAD | oracle.BAD_BYTE)
        else:
            assert st == st_o, (st, st_o)


def test_pack_reports_bad_codes_like_oracle(H):
    from paper_2609_09240_gb300 import tq
    N, K = 6, 256
    w = wl.gen_weights(N, K, 0.3, config=7, proj=2)
    rp, _ = oracle.rowptr(N, K, w.sal)
    T1 = w.T1.copy(); T1[1, 17] = 3
    T2 = w.T2.copy()
    n, g = np.argwhere(~w.sal_dense)[0]
    T2[n, 128 * g + 9] = -1
    for t1, t2 in ((T1, w.T2), (w.T1, T2), (T1, T2)):
        _, _, st_o = oracle.pack(N, K, t1, t2, w.sal, rp)
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        p1 = torch.empty((N, tq.tq_row_bytes(K)), dtype=torch.uint8, device="cuda")
        p2 = torch.empty((int(rp[N]), 26), dtype=torch.uint8, device="cuda")
        tq.tq_pack(N, K, H.dev(t1), H.dev(t2), H.dev(w.sal), H.dev(rp), p1, p2, status)
        assert int(status.item()) == st_o != 0


def test_rowptr_pad_bits(H):
    from paper_2609_09240_gb300 import tq
    N, K = 4, 640  # G = 5: bits 5..31 of each word are pad
    sal = np.zeros((N, 1), np.uint32)
    sal[:, 0] = [0b10101, 0b1, 0, 0b11111]
    rp_o, st_o = oracle.rowptr(N, K, sal)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    rp = torch.empty(N + 1, dtype=torch.int32, device="cuda")
    tq.tq_salience_rowptr(N, K, H.dev(sal), rp, status)
    assert np.array_equal(rp.cpu().numpy(), rp_o) and int(status.item()) == st_o == 0
    sal[2, 0] = 1 << 7
    rp_o, st_o = oracle.rowptr(N, K, sal)
    status.zero_()
    tq.tq_salience_rowptr(N, K, H.dev(sal), rp, status)
    assert np.array_equal(rp.cpu().numpy(), rp_o) and int(status.item()) == st_o == oracle.BAD_PAD


def test_large_rowptr(H):
    from paper_2609_09240_gb300 import tq
    N, K = 50_000, 4096
    rng = np.random.default_rng(1)
    sal = rng.integers(0, 2 ** 32, (N, 1), dtype=np.uint64).astype(np.uint32)
    rp_o, _ = oracle.rowptr(N, K, sal)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    rp = torch.empty(N + 1, dtype=torch.int32, device="cuda")
    tq.tq_salience_rowptr(N, K, H.dev(sal), rp, status)
    assert np.array_equal(rp.cpu().numpy(), rp_o)


def plane2_index_model(N, K, sal, rp, p2, s2_bits, cap, slot_off):
    """The index's bytes as tq.h lays them out, built with numpy from the
    oracle's plane 2: (colptr int32 [G + 1], slots uint8 [cap][32])."""
    G = K // 128
    bits = ((sal[:, np.arange(G) // 32] >> (np.arange(G) % 32)) & 1).astype(bool)  # [N][G]
    rank = np.cumsum(bits, axis=1) - bits  # salient groups of the row before g
    counts = bits.sum(axis=0)
    colptr = np.concatenate([[0], np.cumsum((counts + 15) // 16 * 16)]).astype(np.int64)
    logical = np.zeros((cap, 32), np.uint8)
    logical[:, 28:32] = 0xFF  # row -1 in the empty entries
    for g in range(G):
        rows = np.nonzero(bits[:, g])[0]
        j = rp[rows].astype(np.int64) + rank[rows, g]
        e = colptr[g] + np.arange(rows.size)
        o = 2 * ((g % 8) & 1)
        logical[e, :] = 0
        logical[e, o:o + 26] = p2[j]
        s2b = s2_bits[j].astype("<u2").view(np.uint8).reshape(-1, 2)
        so = 0 if o else 26
        logical[e, so:so + 2] = s2b
        logical[e, 28:32] = rows.astype("<i4").view(np.uint8).reshape(-1, 4)
    words = logical.reshape(cap, 8, 4)
    slots = words[:, [0, 4, 1, 5, 2, 6, 3, 7], :].reshape(cap, 32)
    return colptr, slots


@pytest.mark.parametrize("N,K,frac", [s for s in SHAPES if s[2] > 0] + [(1000, 41088, 0.05), (37, 1152, 1.0)])
def test_plane2_index_bit_exact(H, N, K, frac):
    """The group-ordered second-plane index: per group, its salient rows in
    order, each with its record (at the group's window alignment), s2 and row;
    groups padded to 16 entries with empty slots; bit for bit."""
    from paper_2609_09240_gb300 import tq
    w = wl.gen_weights(N, K, frac, config=7, proj=3 * N + K)
    rp, st = oracle.rowptr(N, K, w.sal)
    assert st == 0
    _, p2, st = oracle.pack(N, K, w.T1, w.T2, w.sal, rp)
    assert st == 0
    nnz = int(rp[N])
    s2_bits = np.ascontiguousarray(w.s2).view(np.uint16)
    idx = tq.tq_plane2_index(N, K, H.dev(w.sal), H.dev(rp), nnz, H.dev(p2), H.dev(s2_bits)).cpu().numpy()
    L = tq.lib()
    cap = int(L.tq_plane2_index_capacity(K, nnz))
    so = int(L.tq_plane2_index_slot_offset(K))
    assert idx.size * 4 == so + 32 * cap
    colptr, slots = plane2_index_model(N, K, w.sal, rp, p2, s2_bits, cap, so)
    np.testing.assert_array_equal(idx[:K // 128 + 1], colptr)
    got = idx.view(np.uint8)[so:].reshape(cap, 32)
    bad = np.nonzero((got != slots).any(axis=1))[0]
    assert bad.size == 0, f"{bad.size} slots differ; first {bad[0]}: {got[bad[0]]} vs {slots[bad[0]]}"
