"""GPU linear parity: tq_linear / tq_linear_f32out / tq_linear_batched
against the fp64 CPU oracle, |y - y_ref| <= 2e-3 * sum_k |W x| per element."""
import numpy as np
import pytest
import torch

import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    import gpu_helpers
    return gpu_helpers


def run_case(H, N, K, frac, M, f32, proj=0, config=6, index=True):
    from paper_2609_09240_gb300 import tq
    w = wl.gen_weights(N, K, frac, config=config, proj=proj)
    x = wl.gen_x(M, K, config=config, proj=proj)
    y_ref, a_ref = H.oracle_ref(w, x)
    pw = H.pack_on_gpu(w, index=index)
    xd = H.dev(x)
    y = (tq.tq_linear_f32out if f32 else tq.tq_linear)(xd, pw)
    H.device_status_ok()
    yg = y.float().cpu().numpy().astype(np.float64)
    return H.assert_close(yg, y_ref, a_ref)


@pytest.mark.parametrize("M", [1, 2, 3, 4, 8, 16])
@pytest.mark.parametrize("f32", [False, True])
def test_config0_single_linear(H, M, f32):
    run_case(H, 512, 1024, 0.0, M, f32)


@pytest.mark.parametrize("N,K,frac", [(1, 128, 0.0), (1, 128, 1.0), (129, 256, 0.5), (200, 2560, 0.1),
                                      (77, 4224, 0.1), (300, 9728, 0.1), (128, 12288, 0.1)])
@pytest.mark.parametrize("M", [1, 2, 5, 16])
def test_ragged_shapes(H, N, K, frac, M):
    run_case(H, N, K, frac, M, f32=False, proj=N)


@pytest.mark.parametrize("M", [17, 40])
def test_m_above_skinny(H, M):
    run_case(H, 130, 1024, 0.1, M, f32=True, proj=3)


@pytest.mark.parametrize("idx", range(7))
def test_config1_qwen3_4b_layer(H, idx):
    name, N, K = wl.QWEN3_4B[idx]
    run_case(H, N, K, 0.1, 1, f32=False, proj=idx, config=1)


def test_zero_codes_offset_only(H):
    """All-zero codes: the output is the offset term alone (zero trits still
    carry the offset, paper "E2M-ATQ" on mu != 0)."""
    from paper_2609_09240_gb300 import tq
    N, K, M = 256, 1024, 2
    w = wl.gen_weights(N, K, 0.1, config=6, proj=9)
    w.T1[:] = 0
    w.T2[:] = 0
    x = wl.gen_x(M, K, config=6, proj=9)
    y_ref, a_ref = H.oracle_ref(w, x)
    y = tq.tq_linear_f32out(H.dev(x), H.pack_on_gpu(w))
    H.assert_close(y.cpu().numpy(), y_ref, a_ref)


def test_batched_layer(H):
    from paper_2609_09240_gb300 import tq
    items, refs = [], []
    for i, (name, N, K) in enumerate(wl.QWEN3_4B):
        w = wl.gen_weights(N, K, 0.1, config=1, proj=i)
        x = wl.gen_x(1, K, config=1, proj=i)
        refs.append(H.oracle_ref(w, x))
        items.append((H.pack_on_gpu(w), H.dev(x), torch.empty((1, N), dtype=torch.float16, device="cuda")))
    b = tq.Batch(1, items)
    tq.tq_linear_batched(b)
    H.device_status_ok()
    for (pw, xd, y), (y_ref, a_ref) in zip(items, refs):
        H.assert_close(y.float().cpu().numpy(), y_ref, a_ref)


def test_argument_errors(H):
    from paper_2609_09240_gb300 import tq
    import ctypes
    w = wl.gen_weights(64, 256, 0.0, config=6, proj=11)
    pw = H.pack_on_gpu(w)
    x = torch.zeros((1, 256), dtype=torch.float16, device="cuda")
    y = torch.empty((1, 64), dtype=torch.float16, device="cuda")
    ws = tq.workspace(tq.tq_workspace_bytes(1, 64, 256), "cuda")
    L = tq.lib()
    s = tq._stream(None)
    ws_ = pw.struct()
    P = lambda t: ctypes.c_void_p(t.data_ptr())
    n = ws.numel()
    assert L.tq_linear(0, 64, 256, ctypes.byref(ws_), P(x), P(y), P(ws), n, s) == -2
    assert L.tq_linear(1, 64, 200, ctypes.byref(ws_), P(x), P(y), P(ws), n, s) == -2
    assert L.tq_linear(1, 64, 256, None, P(x), P(y), P(ws), n, s) == -1
    assert L.tq_linear(1, 64, 256, ctypes.byref(ws_), P(x), P(y), None, n, s) == -1
    assert L.tq_linear(1, 64, 256, ctypes.byref(ws_), P(x), P(y), P(ws), 16, s) == -2  # workspace too small
    xb = torch.zeros(300, dtype=torch.float16, device="cuda")[1:257]
    assert L.tq_linear(1, 64, 256, ctypes.byref(ws_), ctypes.c_void_p(xb.data_ptr()), P(y), P(ws), n, s) == -3
    wb = torch.empty(n + 256, dtype=torch.uint8, device="cuda")[16:]
    assert L.tq_linear(1, 64, 256, ctypes.byref(ws_), P(x), P(y), ctypes.c_void_p(wb.data_ptr()), n, s) == -3
    ws_.group = 64
    assert L.tq_linear(1, 64, 256, ctypes.byref(ws_), P(x), P(y), P(ws), n, s) == -2


@pytest.mark.parametrize("index", [False, True])
@pytest.mark.parametrize("M", [1, 3, 12])
def test_long_rows_second_plane(H, M, index):
    """321 groups per row: without the index, more salience words than the
    span kernel of the second plane stages, so the per-tile kernel runs it
    (12 tokens as two passes); with the index, the indexed kernel."""
    run_case(H, 96, 321 * 128, 0.1, M, f32=True, proj=21, index=index)


def test_batched_many_row_lengths(H):
    """A batch with more distinct plane-1 row lengths than tensor-map
    templates per launch runs as consecutive sub-batches."""
    from paper_2609_09240_gb300 import tq
    items, refs = [], []
    for i in range(11):
        N, K = 64 + 32 * i, 128 * (i + 1)
        w = wl.gen_weights(N, K, 0.2, config=6, proj=30 + i)
        x = wl.gen_x(1, K, config=6, proj=30 + i)
        refs.append(H.oracle_ref(w, x))
        items.append((H.pack_on_gpu(w), H.dev(x), torch.empty((1, N), dtype=torch.float16, device="cuda")))
    b = tq.Batch(1, items)
    tq.tq_linear_batched(b)
    H.device_status_ok()
    for (pw, xd, y), (y_ref, a_ref) in zip(items, refs):
        H.assert_close(y.float().cpu().numpy(), y_ref, a_ref)


@pytest.mark.parametrize("index", [True, False])
@pytest.mark.parametrize("M", [1, 3])
def test_batched_max_problems(H, M, index):
    """A batch of TQ_MAX_BATCH problems, all with a second plane: the last
    problems' descriptors sit at the far end of the kernels' parameter
    space, which every per-problem read has to reach."""
    from paper_2609_09240_gb300 import tq
    shapes = [(48, 256), (80, 640), (48, 640), (80, 256)]
    items, refs = [], []
    for i in range(tq.TQ_MAX_BATCH):
        N, K = shapes[i % 4]
        w = wl.gen_weights(N, K, 0.3, config=8, proj=i)
        x = wl.gen_x(M, K, config=8, proj=i)
        refs.append(H.oracle_ref(w, x))
        items.append((H.pack_on_gpu(w, index=index), H.dev(x), torch.empty((M, N), dtype=torch.float16, device="cuda")))
    b = tq.Batch(M, items)
    tq.tq_linear_batched(b)
    H.device_status_ok()
    for i, ((pw, xd, y), (y_ref, a_ref)) in enumerate(zip(items, refs)):
        try:
            H.assert_close(y.float().cpu().numpy(), y_ref, a_ref)
        except AssertionError as e:
            raise AssertionError(f"problem {i}: {e}") from None


@pytest.mark.parametrize("N,K,frac", [(1, 128, 1.0), (129, 256, 0.5), (300, 9728, 0.1), (700, 4096, 0.3)])
@pytest.mark.parametrize("M", [1, 3, 8, 9, 10, 12])
def test_second_plane_without_index(H, N, K, frac, M):
    """Weights packed without the second-plane index: the span kernel groups
    the records itself (more than 8 tokens then run as two passes of at most
    8, the indexed path takes up to 16 in one pass; a second pass of one or
    two tokens stays on the general kernels, whose layout the workspace
    holds)."""
    run_case(H, N, K, frac, M, f32=True, proj=40 + N, index=False)


@pytest.mark.parametrize("index", [False, True])
@pytest.mark.parametrize("M", [1, 4])
def test_second_plane_scale2_two_byte_aligned(H, M, index):
    """s2 is only required to be 2-byte aligned: a view starting 2 bytes
    into an allocation, read by the span kernel or copied into the
    group-ordered index."""
    from paper_2609_09240_gb300 import tq
    N, K = 300, 4096
    w = wl.gen_weights(N, K, 0.2, config=6, proj=77)
    x = wl.gen_x(M, K, config=6, proj=77)
    y_ref, a_ref = H.oracle_ref(w, x)
    pw = H.pack_on_gpu(w, index=False)
    buf = torch.empty(pw.nnz + 1, dtype=torch.float16, device="cuda")
    buf[1:] = pw.scale2[:pw.nnz]
    pw.scale2 = buf[1:]
    assert pw.scale2.data_ptr() % 4 == 2
    if index:
        pw.p2index = tq.tq_plane2_index(N, K, pw.salience, pw.rowptr, pw.nnz, pw.plane2, pw.scale2)
    y = tq.tq_linear_f32out(H.dev(x), pw)
    H.device_status_ok()
    H.assert_close(y.cpu().numpy(), y_ref, a_ref)


def test_two_host_threads(H):
    """tq_linear from two host threads at once, different shapes and token
    counts, each on its own stream and workspace: launch parameters are kept
    per host thread, so neither call ever runs with the other's sizes or
    pointers.  Every result of 40 calls per thread matches the oracle."""
    import threading

    from paper_2609_09240_gb300 import tq
    cases = [(1, 1024, 4096, 0.1, 11), (5, 300, 2560, 0.2, 12)]
    prepared = []
    for M, N, K, frac, proj in cases:
        w = wl.gen_weights(N, K, frac, config=6, proj=proj)
        xb = wl.gen_x(M, K, config=6, proj=proj)
        y_ref, a_ref = H.oracle_ref(w, xb)
        prepared.append((H.pack_on_gpu(w), H.dev(xb), y_ref, a_ref))
    torch.cuda.synchronize()
    results = [[], []]
    errors = []

    def worker(i):
        try:
            pw, x, _, _ = prepared[i]
            s = torch.cuda.Stream()
            ws = tq.workspace(tq.tq_workspace_bytes(x.shape[0], pw.N, pw.K), x.device)
            with torch.cuda.stream(s):
                for _ in range(40):
                    results[i].append(tq.tq_linear(x, pw, ws=ws, stream=s).clone())
            s.synchronize()
        except Exception as e:  # reported on the main thread
            errors.append(e)

    th = [threading.Thread(target=worker, args=(i,)) for i in range(2)]
    for t in th:
        t.start()
    for t in th:
        t.join()
    assert not errors, errors
    H.device_status_ok()
    for i, (_, _, y_ref, a_ref) in enumerate(prepared):
        assert len(results[i]) == 40
        for y in results[i]:
            H.assert_close(y.float().cpu().numpy(), y_ref, a_ref)


@pytest.mark.parametrize("M", [1, 2])
@pytest.mark.parametrize("f32", [False, True])
def test_one_group_per_lane_stage_shapes(H, M, f32):
    """The M <= 2 kernel's 4-group stages and 256-row tiles: group counts of
    every residue mod 4 and mod 8 (scales by tensor copy only when G % 8 ==
    0), tiles cut short by N, in one batch whose tiles straddle problems."""
    from paper_2609_09240_gb300 import tq
    shapes = [(257, 128 * 9), (511, 128 * 10), (256, 128 * 11), (300, 128 * 12), (1, 128 * 16), (640, 128 * 3),
              (513, 128 * 6)]
    items, refs = [], []
    for i, (N, K) in enumerate(shapes):
        w = wl.gen_weights(N, K, 0.15, config=6, proj=40 + i)
        xb = wl.gen_x(M, K, config=6, proj=40 + i)
        refs.append(H.oracle_ref(w, xb))
        pw = H.pack_on_gpu(w, index=(i % 2 == 0))
        x = H.dev(xb)
        if f32:
            y = tq.tq_linear_f32out(x, pw)
            H.device_status_ok()
            H.assert_close(y.cpu().numpy().astype(np.float64), *refs[-1])
        items.append((pw, x, torch.full((M, N), float("nan"), dtype=torch.float16, device=x.device)))
    if not f32:
        tq.tq_linear_batched(tq.Batch(M, items))
        H.device_status_ok()
        for (pw, x, y), (y_ref, a_ref) in zip(items, refs):
            H.assert_close(y.float().cpu().numpy().astype(np.float64), y_ref, a_ref)


@pytest.mark.parametrize("M,N,K,frac,index", [
    (1, 1024, 4096, 0.1, True),    # k/v shape: 4 tiles x 4 stages, every stage its own CTA
    (1, 4096, 12288, 0.1, True),   # down shape: 16 tiles x 12 stages, 9 CTAs per tile
    (1, 200, 4224, 0.2, False),    # 1 tile, 5 stages (the last of one group), second plane without index
    (2, 300, 9728, 0.1, True),     # two tokens: 2 tiles x 19 four-group stages
    (2, 1, 640, 1.0, True),        # one row, every group salient
])
def test_split_tiles_single_call(H, M, N, K, frac, index):
    """One tq_linear call on a projection with fewer 256-row tiles than SMs:
    each tile's stages are shared by several CTAs, which add partial sums
    into the fp32 workspace; the last to arrive writes y.  Checked against the
    oracle on two calls in a row (the counters restart every call)."""
    from paper_2609_09240_gb300 import tq
    w = wl.gen_weights(N, K, frac, config=6, proj=60 + M + N % 7)
    xb = wl.gen_x(M, K, config=6, proj=60 + M + N % 7)
    y_ref, a_ref = H.oracle_ref(w, xb)
    pw = H.pack_on_gpu(w, index=index)
    x = H.dev(xb)
    ws = tq.workspace(tq.tq_workspace_bytes(M, N, K), x.device)
    for _ in range(2):
        y = tq.tq_linear_f32out(x, pw, ws=ws)
        H.device_status_ok()
        H.assert_close(y.cpu().numpy().astype(np.float64), y_ref, a_ref)
