"""Shared helpers of the GPU parity tests: move seeded inputs to the device,
pack them with the library, and compute the oracle's reference."""
import numpy as np
import torch

import oracle
import workloads as wl
from paper_2609_09240_gb300 import tq

TOL = 2e-3  # |y_gpu - y_ref| <= TOL * sum_k |W x| per element (fp32 accumulation)


def dev(a: np.ndarray, dtype=None):
    if a.dtype == np.uint16:
        a = a.view(np.float16)
    elif a.dtype == np.uint32:
        a = a.view(np.int32)
    t = torch.from_numpy(np.ascontiguousarray(a)).cuda()
    return t if dtype is None else t.to(dtype)


def pack_on_gpu(w: wl.Weights, index=True) -> tq.PackedWeight:
    return tq.pack_weight(dev(w.T1), dev(w.T2), dev(w.sal), dev(w.s1), dev(w.off),
                          dev(w.s2) if w.nnz else None, index=index)


def oracle_ref(w: wl.Weights, x_bits: np.ndarray, rows=None, nthreads=None):
    rp, st = oracle.rowptr(w.N, w.K, w.sal)
    assert st == 0
    p1, p2, st = oracle.pack(w.N, w.K, w.T1, w.T2, w.sal, rp)
    assert st == 0
    return oracle.linear(x_bits.shape[0], w.N, w.K, p1, p2, w.sal, w.s1, w.off, w.s2, x_bits,
                         rows=rows, nthreads=nthreads)


def device_status_ok():
    torch.cuda.synchronize()
    st = tq.tq_get_device_status(clear=True)
    assert st == 0, f"device status {st:#x} (a bounded wait ran out)"


def assert_close(y_gpu: np.ndarray, y_ref: np.ndarray, a_ref: np.ndarray, tol=TOL):
    err = np.abs(y_gpu.astype(np.float64) - y_ref)
    bound = tol * a_ref
    bad = err > bound
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(
            f"{bad.sum()} of {bad.size} outputs out of tolerance; first at {tuple(i)}: "
            f"gpu={y_gpu[tuple(i)]!r} ref={y_ref[tuple(i)]!r} err={err[tuple(i)]:.3e} bound={bound[tuple(i)]:.3e}")
    return float((err / np.maximum(a_ref, 1e-300)).max())
