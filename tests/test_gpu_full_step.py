"""Parity at full size, in the launch configuration bench.py times: the
whole Qwen3-8B decode step (36 layers x 7 projections, 252 problems, one
tq_linear_batched call) for M = 1 and M = 16.  The packed planes are copied
back to the host and the fp64 oracle computes a seeded sample of rows of
every projection of a few layers (every token), against the tolerance
|y - y_ref| <= 2e-3 * sum_k |W x|."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    import gpu_helpers
    return gpu_helpers


def _host(t, dtype):
    return t.detach().cpu().numpy().view(dtype)


@pytest.mark.parametrize("M", [1, 16])
def test_qwen3_8b_step_sampled_rows(H, M):
    import bench
    import oracle
    from paper_2609_09240_gb300 import tq
    dev = torch.device("cuda", 0)
    items, x_all, y_all, packed_bytes, n_weights = bench.build_step(M, dev, seed0=0)
    assert len(items) == 252 and packed_bytes == 1792241424
    batch = tq.Batch(M, items)
    tq.tq_linear_batched(batch)
    torch.cuda.synchronize()
    H.device_status_ok()
    rng = np.random.default_rng(M)
    # layers 0, 17 and 35: all seven projection shapes, 24 sampled rows each
    for idx in [i for layer in (0, 17, 35) for i in range(7 * layer, 7 * layer + 7)]:
        pw, x, y = items[idx]
        rows = np.sort(rng.choice(pw.N, size=24, replace=False)).astype(np.int32)
        nnz = int(pw.nnz)
        y_ref, a_ref = oracle.linear(
            M, pw.N, pw.K, _host(pw.plane1, np.uint8), _host(pw.plane2[:nnz], np.uint8) if nnz else None,
            _host(pw.salience, np.uint32), _host(pw.scale1, np.uint16), _host(pw.offset, np.uint16),
            _host(pw.scale2[:nnz], np.uint16) if nnz else None, _host(x, np.uint16), rows=rows)
        yg = y.float().cpu().numpy()[:, rows].astype(np.float64)
        H.assert_close(yg, y_ref, a_ref)
