"""tq_linear_sequence, the dependency-ordered decode step (each problem
complete before the next starts, one persistent launch): parity with the
fp64 oracle, |y - y_ref| <= 2e-3 * sum_k |W x|, on mixed shapes and on one
Qwen3-8B layer with q/k/v and gate/up fused into single weights (the order a
model runs them: qkv, o, gate/up, down), over two calls in a row (the
barrier counter restarts every call).  The oracle packs its own bytes from
the same seeded codes."""
import numpy as np
import pytest
import torch

import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    import gpu_helpers
    return gpu_helpers


def _run(H, shapes, frac, config, rows_per=None):
    from paper_2609_09240_gb300 import tq
    items, refs = [], []
    for i, (N, K) in enumerate(shapes):
        w = wl.gen_weights(N, K, frac, config=config, proj=i)
        xb = wl.gen_x(1, K, config=config, proj=i)
        rows = None
        if rows_per is not None and N > rows_per:
            rows = np.sort(np.random.default_rng(N + i).choice(N, size=rows_per, replace=False)).astype(np.int32)
        refs.append((rows,) + H.oracle_ref(w, xb, rows=rows))
        items.append((H.pack_on_gpu(w), H.dev(xb), torch.full((1, N), float("nan"), dtype=torch.float16,
                                                             device="cuda")))
    batch = tq.Batch(1, items)
    for _ in range(2):
        for _, _, y in items:
            y.fill_(float("nan"))
        tq.tq_linear_sequence(batch)
        H.device_status_ok()
        for (pw, x, y), (rows, y_ref, a_ref) in zip(items, refs):
            yg = y.float().cpu().numpy().astype(np.float64)
            assert not np.isnan(yg).any()
            H.assert_close(yg if rows is None else yg[:, rows], y_ref, a_ref)


def test_sequence_mixed_shapes(H):
    # ragged rows and groups, a problem smaller than one tile, K of one group
    shapes = [(300, 1024), (1024, 2560), (129, 4224), (2000, 640), (64, 128), (700, 9728)]
    _run(H, shapes, 0.1, config=8)


def test_sequence_no_second_plane(H):
    _run(H, [(512, 1024), (256, 2048), (1000, 1152)], 0.0, config=8)


def test_sequence_qwen3_8b_layer_fused(H):
    """q/k/v concatenated (6144 x 4096), o, gate/up concatenated
    (24576 x 4096), down: sampled rows of each against the oracle."""
    shapes = [(6144, 4096), (4096, 4096), (24576, 4096), (4096, 12288)]
    _run(H, shapes, 0.1, config=9, rows_per=48)


def test_sequence_matches_batched(H):
    """The same problems through tq_linear_batched (independent) and
    tq_linear_sequence (in order) agree within the tolerance."""
    from paper_2609_09240_gb300 import tq
    shapes = [(1024, 4096), (4096, 4096), (640, 2560)]
    items_b, items_s, refs = [], [], []
    for i, (N, K) in enumerate(shapes):
        w = wl.gen_weights(N, K, 0.1, config=10, proj=i)
        xb = wl.gen_x(1, K, config=10, proj=i)
        refs.append(H.oracle_ref(w, xb))
        pw, x = H.pack_on_gpu(w), H.dev(xb)
        items_b.append((pw, x, torch.empty((1, N), dtype=torch.float16, device="cuda")))
        items_s.append((pw, x, torch.empty((1, N), dtype=torch.float16, device="cuda")))
    tq.tq_linear_batched(tq.Batch(1, items_b))
    tq.tq_linear_sequence(tq.Batch(1, items_s))
    H.device_status_ok()
    for (_, _, yb), (_, _, ys), (y_ref, a_ref) in zip(items_b, items_s, refs):
        H.assert_close(yb.float().cpu().numpy(), y_ref, a_ref)
        H.assert_close(ys.float().cpu().numpy(), y_ref, a_ref)
