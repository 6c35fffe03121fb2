"""tq_linear_static (the allocation-free entry point): on two calls in a row
its output matches the fp64 oracle within the parity tests' tolerance, as
tq_linear's with a caller workspace does; oversize calls are
rejected before anything runs.  The cases cover the decode path with and
without the second-plane index (the latter runs more than 8 tokens as two
passes over the scratch) and the prefill path (M > 16, which needs no
workspace).  Collected last (file name), so that it also runs after every
other GPU test in the same process."""
import numpy as np
import pytest

import workloads as wl

TOL = 2e-3  # |y - y_ref| <= TOL * sum_k |W x|, the linear-layer tolerance of the parity tests


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
@pytest.mark.parametrize("M,N,K,frac,index", [
    (1, 512, 1024, 0.0, True),
    (3, 200, 4224, 0.1, True),
    (8, 4096, 4096, 0.1, True),
    (16, 1024, 2560, 0.1, True),
    (12, 300, 1280, 0.1, False),   # no index: tokens 0..7, then 8..11, over the same scratch
    (40, 256, 640, 0.2, True),     # prefill path
])
def test_static_matches_oracle_twice(H, M, N, K, frac, index):
    from paper_2609_09240_gb300 import tq
    w = wl.gen_weights(N, K, frac, config=7, proj=M)
    xb = wl.gen_x(M, K, config=7, proj=M)
    pw = H.pack_on_gpu(w, index=index)
    x = H.dev(xb)
    assert tq.tq_workspace_bytes(M, N, K) <= tq.STATIC_SCRATCH_BYTES
    y_ref, a_ref = H.oracle_ref(w, xb)
    y_ws = tq.tq_linear(x, pw).cpu().numpy()
    y1 = tq.tq_linear_static(x, pw).cpu().numpy()
    y2 = tq.tq_linear_static(x, pw).cpu().numpy()
    H.device_status_ok()
    for y in (y_ws, y1, y2):
        H.assert_close(y.astype(np.float32), y_ref, a_ref, tol=TOL)
