"""Parity at full size, in the launch configuration bench.py times: the
whole Qwen3-8B decode step (36 layers x 7 projections, 252 problems, one
tq_linear_batched call) for M = 1, 2, 4, 8 and 16.

The oracle sees no byte the CUDA path produced.  Each projection's codes,
salience and fp16 parameters are drawn by the seeded generator on the
device; they are copied to the host, the oracle computes rowptr and packs
plane 1 and plane 2 itself, and the GPU's tq_pack output must equal those
bytes for all 252 projections.  The linear check then feeds the oracle its
own packed bytes: a seeded sample of rows of every projection of layers 0,
17 and 35 (every token), against |y - y_ref| <= 2e-3 * sum_k |W x|."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

REF_LAYERS = (0, 17, 35)


@pytest.fixture(scope="module")
def H():
    import gpu_helpers
    return gpu_helpers


def _np(t, dtype):
    return np.ascontiguousarray(t.detach().cpu().numpy()).view(dtype)


@pytest.fixture(scope="module")
def step():
    """The packed step (device) and, for the reference layers, the oracle's
    own packed bytes and the drawn parameters (host)."""
    import bench
    import oracle
    dev = torch.device("cuda", 0)
    ref, checked = {}, []

    def on_codes(p, g, pw):
        N, K = p.N, p.K
        sal = _np(g["sal"], np.uint32)
        T1 = _np(g["T1"], np.int8)
        T2 = _np(g["T2"], np.int8)
        rp, st = oracle.rowptr(N, K, sal)
        assert st == 0
        p1, p2, st = oracle.pack(N, K, T1, T2, sal, rp)
        assert st == 0
        nnz = int(rp[N])
        assert nnz == pw.nnz == g["nnz"]
        # bytes of the GPU's packing against the oracle's, every projection
        assert np.array_equal(_np(pw.rowptr, np.int32), rp), (p.layer, p.name)
        assert np.array_equal(_np(pw.plane1, np.uint8), p1), (p.layer, p.name)
        if nnz:
            assert np.array_equal(_np(pw.plane2[:nnz], np.uint8), p2), (p.layer, p.name)
        checked.append((p.layer, p.proj))
        if p.layer in REF_LAYERS:
            s2 = _np(g["s2"], np.uint16) if nnz else None
            ref[(p.layer, p.proj)] = (p1, p2 if nnz else None, sal, _np(g["s1"], np.uint16),
                                      _np(g["off"], np.uint16), s2)

    items, _, _, packed_bytes, _ = bench.build_step(1, dev, seed0=0, on_codes=on_codes)
    assert len(items) == 252 and len(checked) == 252 and packed_bytes == 1792241424
    return [pw for pw, _, _ in items], ref


@pytest.mark.parametrize("M", [1, 2, 4, 8, 16])
def test_qwen3_8b_step_sampled_rows(H, step, M):
    import oracle
    import workloads as wl
    from paper_2609_09240_gb300 import tq
    dev = torch.device("cuda", 0)
    pws, ref = step
    projs = wl.config_projections(2)
    items = []
    for p, pw in zip(projs, pws):
        x = wl.gen_x_torch(M, p.K, dev, 1000 * M + p.layer * 16 + p.proj)
        y = torch.full((M, p.N), float("nan"), dtype=torch.float16, device=dev)
        items.append((pw, x, y))
    tq.tq_linear_batched(tq.Batch(M, items))
    torch.cuda.synchronize()
    H.device_status_ok()
    rng = np.random.default_rng(M)
    for i, p in enumerate(projs):
        if p.layer not in REF_LAYERS:
            continue
        pw, x, y = items[i]
        p1, p2, sal, s1, off, s2 = ref[(p.layer, p.proj)]
        rows = np.sort(rng.choice(p.N, size=24, replace=False)).astype(np.int32)
        y_ref, a_ref = oracle.linear(M, p.N, p.K, p1, p2, sal, s1, off, s2, _np(x, np.uint16), rows=rows)
        yg = y.float().cpu().numpy()[:, rows].astype(np.float64)
        H.assert_close(yg, y_ref, a_ref)
    # every output of every projection was written (no NaN left)
    for pw, _, y in items:
        assert not torch.isnan(y).any()
