"""The failure path on the GPU without a fault: a bounded wait that nothing
completes runs out, the device status word reports it, and the context keeps
working (a linear call afterwards matches the oracle)."""
import ctypes
import time

import pytest
import torch

import workloads as wl

pytestmark = pytest.mark.gpu


def test_bounded_wait_runs_out_and_reports():
    import gpu_helpers as H
    from paper_2609_09240_gb300 import tq
    tq.tq_get_device_status(clear=True)
    r = torch.full((1,), 7, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    t0 = time.time()
    assert tq.lib().tq_wait_selftest(ctypes.c_void_p(r.data_ptr()), tq._stream(None)) == 0
    torch.cuda.synchronize()
    dt = time.time() - t0
    assert int(r.item()) == 0            # the wait gave up
    assert tq.tq_get_device_status(clear=True) & 1
    assert 1.5 < dt < 60, dt             # after about its 2 s limit
    # the context is intact
    w = wl.gen_weights(256, 1024, 0.1, config=6, proj=5)
    x = wl.gen_x(2, 1024, config=6, proj=5)
    y = tq.tq_linear_f32out(H.dev(x), H.pack_on_gpu(w))
    H.device_status_ok()
    y_ref, a_ref = H.oracle_ref(w, x)
    H.assert_close(y.cpu().numpy(), y_ref, a_ref)


def test_sequence_barrier_wait_runs_out_and_reports():
    """The dependency-ordered sequence kernel's problem barrier, made to wait
    for one CTA more than were launched: its bounded wait runs out (no
    fault), the status word reports the timeout, every CTA leaves, and a
    normal sequence afterwards matches the oracle."""
    import gpu_helpers as H
    from paper_2609_09240_gb300 import tq
    shapes = [(512, 1024), (300, 2560)]
    items, refs = [], []
    for i, (N, K) in enumerate(shapes):
        w = wl.gen_weights(N, K, 0.1, config=11, proj=i)
        xb = wl.gen_x(1, K, config=11, proj=i)
        refs.append(H.oracle_ref(w, xb))
        items.append((H.pack_on_gpu(w), H.dev(xb), torch.empty((1, N), dtype=torch.float16, device="cuda")))
    batch = tq.Batch(1, items)
    tq.tq_get_device_status(clear=True)
    torch.cuda.synchronize()
    t0 = time.time()
    tq.tq_sequence_selftest(batch)
    torch.cuda.synchronize()
    dt = time.time() - t0
    assert tq.tq_get_device_status(clear=True) & 1
    assert 1.5 < dt < 60, dt
    tq.tq_linear_sequence(batch)
    H.device_status_ok()
    for (_, _, y), (y_ref, a_ref) in zip(items, refs):
        H.assert_close(y.float().cpu().numpy(), y_ref, a_ref)
