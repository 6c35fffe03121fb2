"""GPU parity of the prefill tile path (M > 16 tokens: weight tiles
dequantized to fp16 and multiplied on the tensor cores) against the fp64 CPU
oracle, |y - y_ref| <= 2e-3 * sum_k |W x| per element.  Every token count
takes the kernel fed by tensor copies of x (ragged counts included).  The
full-size case
is the Qwen3-8B prefill shape (M = 2048 tokens) checked on sampled rows."""
import numpy as np
import pytest
import torch

import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def H():
    import gpu_helpers
    return gpu_helpers


@pytest.mark.parametrize("M,N,K,frac,f32", [
    (17, 512, 1024, 0.0, False),    # barely past the decode path, one ragged token tile
    (129, 256, 1024, 0.1, True),    # two token tiles, the second with one token
    (200, 300, 4224, 0.1, False),   # odd group count, ragged rows and tokens
    (256, 520, 2560, 1.0, False),   # every group salient
    (64, 1, 128, 0.5, True),        # one row, one group
    (24, 257, 640, 0.3, True),      # smallest token multiple of 8 past the decode path; a one-row second row tile
    (264, 384, 1152, 0.2, False),   # a second token tile of 8 tokens; odd group count
])
def test_prefill_small(H, M, N, K, frac, f32):
    from paper_2609_09240_gb300 import tq
    w = wl.gen_weights(N, K, frac, config=4, proj=(M * 7 + N) % 97)
    xb = wl.gen_x(M, K, config=4, proj=(M * 7 + N) % 97)
    y_ref, a_ref = H.oracle_ref(w, xb)
    pw = H.pack_on_gpu(w)
    x = H.dev(xb)
    y = (tq.tq_linear_f32out(x, pw) if f32 else tq.tq_linear(x, pw)).float().cpu().numpy()
    H.device_status_ok()
    H.assert_close(y, y_ref, a_ref)


PROJ = {"q": 0, "k": 1, "v": 2, "o": 3, "gate": 4, "up": 5, "down": 6}


@pytest.mark.parametrize("name,N,K,nrows", [("k", 1024, 4096, 48), ("down", 4096, 12288, 24),
                                            ("q", 4096, 4096, 32), ("gate", 12288, 4096, 48)])
def test_prefill_qwen3_8b_shape_sampled_rows(H, name, N, K, nrows):
    """M = 2048 tokens through one Qwen3-8B projection shape; the oracle
    checks a seeded sample of rows (every token) across all row tiles.  q
    (as o: 4096 x 4096), gate (as up: 12288 x 4096, more than one wave of
    SMs) and down run 512-token tiles; k runs 256-token tiles."""
    from paper_2609_09240_gb300 import tq
    M = 2048
    w = wl.gen_weights(N, K, 0.1, config=4, layer=0, proj=PROJ[name])
    xb = wl.gen_x(M, K, config=4, layer=0, proj=PROJ[name])
    pw = H.pack_on_gpu(w)
    y = tq.tq_linear(H.dev(xb), pw).float().cpu().numpy()
    H.device_status_ok()
    rows = np.sort(np.random.default_rng(4).choice(N, size=nrows, replace=False)).astype(np.int32)
    y_ref, a_ref = H.oracle_ref(w, xb, rows=rows)
    H.assert_close(y[:, rows], y_ref, a_ref)


@pytest.mark.parametrize("M,N,K,wide", [(2048, 2560, 640, True), (2048, 1024, 640, False), (300, 10240, 256, True),
                                        (700, 19584, 384, True)])
def test_prefill_tile_widths_sampled_rows(H, M, N, K, wide):
    """Both token-tile widths of the tensor-copy kernel: 512 tokens per CTA
    when 256-token tiles would need more than one wave of SMs (2560 rows at
    M = 2048; 10240 rows at M = 300, whose second token half holds 44
    tokens; 19584 rows at M = 700, a ragged second 512-token tile), 256
    tokens when twice as many CTAs still fit one wave (1024 rows); sampled
    rows of every 128-row tile."""
    from paper_2609_09240_gb300 import tq
    w = wl.gen_weights(N, K, 0.2, config=4, layer=1, proj=N % 89)
    xb = wl.gen_x(M, K, config=4, layer=1, proj=N % 89)
    pw = H.pack_on_gpu(w)
    y = tq.tq_linear(H.dev(xb), pw).float().cpu().numpy()
    H.device_status_ok()
    rng = np.random.default_rng(N)
    rows = np.sort(np.concatenate([t * 128 + rng.choice(min(128, N - t * 128), size=min(2, N - t * 128), replace=False)
                                   for t in range((N + 127) // 128)])).astype(np.int32)
    y_ref, a_ref = H.oracle_ref(w, xb, rows=rows)
    H.assert_close(y[:, rows], y_ref, a_ref)


@pytest.mark.parametrize("M", [40, 300])
def test_prefill_batched_mixed_shapes(H, M):
    """tq_linear_batched at a prefill M: problems of different N and K in one
    launch (the longest K first), every row against the oracle."""
    from paper_2609_09240_gb300 import tq
    shapes = [(300, 1152), (129, 4224), (512, 640), (64, 128), (1000, 256)]
    items, refs = [], []
    for i, (N, K) in enumerate(shapes):
        w = wl.gen_weights(N, K, 0.2, config=4, layer=2, proj=i)
        xb = wl.gen_x(M, K, config=4, layer=2, proj=i)
        refs.append(H.oracle_ref(w, xb))
        items.append((H.pack_on_gpu(w), H.dev(xb), torch.empty((M, N), dtype=torch.float16, device="cuda")))
    tq.tq_linear_batched(tq.Batch(M, items))
    H.device_status_ok()
    for (_, _, y), (y_ref, a_ref) in zip(items, refs):
        H.assert_close(y.float().cpu().numpy(), y_ref, a_ref)


def test_prefill_batched_more_than_one_launch(H):
    """18 problems: two launches of at most 16 problems each."""
    from paper_2609_09240_gb300 import tq
    M = 64
    items, refs = [], []
    for i in range(18):
        N, K = 32 + 8 * i, 128 * (1 + i % 3)
        w = wl.gen_weights(N, K, 0.1, config=4, layer=3, proj=i)
        xb = wl.gen_x(M, K, config=4, layer=3, proj=i)
        refs.append(H.oracle_ref(w, xb))
        items.append((H.pack_on_gpu(w), H.dev(xb), torch.empty((M, N), dtype=torch.float16, device="cuda")))
    tq.tq_linear_batched(tq.Batch(M, items))
    H.device_status_ok()
    for (_, _, y), (y_ref, a_ref) in zip(items, refs):
        H.assert_close(y.float().cpu().numpy(), y_ref, a_ref)


def test_prefill_batched_qwen3_8b_layer_sampled_rows(H):
    """One Qwen3-8B layer's seven projections at M = 2048 in one batched
    call; 16 seeded rows of each against the oracle (every token)."""
    from paper_2609_09240_gb300 import tq
    M = 2048
    items, checks = [], []
    for p in wl.config_projections(4):
        w = wl.gen_weights(p.N, p.K, 0.1, config=4, layer=0, proj=p.proj)
        xb = wl.gen_x(M, p.K, config=4, layer=0, proj=p.proj)
        rows = np.sort(np.random.default_rng(p.proj).choice(p.N, size=16, replace=False)).astype(np.int32)
        checks.append((w, xb, rows))
        items.append((H.pack_on_gpu(w), H.dev(xb), torch.empty((M, p.N), dtype=torch.float16, device="cuda")))
    tq.tq_linear_batched(tq.Batch(M, items))
    H.device_status_ok()
    for (_, _, y), (w, xb, rows) in zip(items, checks):
        y_ref, a_ref = H.oracle_ref(w, xb, rows=rows)
        H.assert_close(y.float().cpu().numpy()[:, rows], y_ref, a_ref)
