"""tq_linear_static (the allocation-free entry point): same results as
tq_linear with a caller workspace, on two calls in a row; oversize calls are
rejected before anything runs.  Collected last (file name) so that it also
runs after every other GPU test in the same process."""
import ctypes

import numpy as np
import pytest

import workloads as wl

TOL = 2e-3  # the linear-layer tolerance of the parity tests


@pytest.fixture(scope="module")
def H():
    import gpu_helpers
    return gpu_helpers


def test_oversize_call_is_rejected_without_gpu():
    from paper_2609_09240_gb300 import tq
    L = tq.lib()
    # K = 512 Ki inputs needs far more than the 1 MiB scratch; rejected
    # before any pointer is looked at or any CUDA call is made
    assert tq.tq_workspace_bytes(8, 64, 1 << 19) > tq.STATIC_SCRATCH_BYTES
    assert L.tq_linear_static(8, 64, 1 << 19, None, None, None, None) == -9
    assert L.tq_linear_static(0, 64, 4096, None, None, None, None) == -2
    assert b"SCRATCH" in L.tq_status_str(-9)


@pytest.mark.gpu
@pytest.mark.parametrize("M,N,K,frac", [(1, 512, 1024, 0.0), (3, 200, 4224, 0.1), (8, 4096, 4096, 0.1),
                                        (16, 1024, 2560, 0.1)])
def test_static_matches_workspace_path_twice(H, M, N, K, frac):
    import torch
    from paper_2609_09240_gb300 import tq
    w = wl.gen_weights(N, K, frac, config=7, proj=M)
    xb = wl.gen_x(M, K, config=7, proj=M)
    pw = H.pack_on_gpu(w)
    x = H.dev(xb)
    assert tq.tq_workspace_bytes(M, N, K) <= tq.STATIC_SCRATCH_BYTES
    y_ws = tq.tq_linear(x, pw).float().cpu().numpy()
    y1 = tq.tq_linear_static(x, pw).float().cpu().numpy()
    y2 = tq.tq_linear_static(x, pw).float().cpu().numpy()
    H.device_status_ok()
    # reference magnitudes from the oracle set the tolerance scale
    _, a_ref = H.oracle_ref(w, xb)
    for y in (y1, y2):
        err = np.abs(y.astype(np.float64) - y_ws)
        assert (err <= 2 * TOL * a_ref).all(), float((err / np.maximum(a_ref, 1e-300)).max())
