"""GPU side of the provenance checks: tq_dequantize (W-hat as fp16, paper
"Model and Representation", eq. for W-hat per group) bit-exact against a
numpy float32 statement of the same formula; the "measurable weight change"
report of a ternarized projection against the oracle's; and a container
round trip back to the device that runs the decode path bit-identically."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from oracle import ternarize as tz

pytestmark = pytest.mark.gpu

F32 = np.float32


def what_formula(w: wl.Weights):
    """fp16((s1 t1 + off) + s2 t2) with float32 sums, for every weight."""
    G = w.K // 128
    rep = lambda v: np.repeat(v.reshape(w.N, G), 128, axis=1)
    s1 = rep(w.s1.view(np.float16).astype(F32))
    off = rep(w.off.view(np.float16).astype(F32))
    s2d = np.zeros(w.N * G, F32)
    s2d[w.sal_dense.ravel()] = w.s2.view(np.float16).astype(F32)
    s2 = rep(s2d)
    a = np.where(w.T1 > 0, s1, np.where(w.T1 < 0, -s1, F32(0))).astype(F32)
    b = np.where(w.T2 > 0, s2, np.where(w.T2 < 0, -s2, F32(0))).astype(F32)
    return np.add(np.add(a, off, dtype=F32), b, dtype=F32).astype(np.float16)


@pytest.mark.parametrize("N,K,frac", [(1, 128, 1.0), (77, 4224, 0.3), (300, 2560, 0.1)])
def test_dequantize_bit_exact(N, K, frac):
    import gpu_helpers as H
    from paper_2609_09240_gb300 import tq
    w = wl.gen_weights(N, K, frac, config=10, proj=N)
    pw = H.pack_on_gpu(w, index=False)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    Wh = tq.tq_dequantize(pw, d_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(Wh.cpu().numpy().view(np.uint16), what_formula(w).view(np.uint16))


def test_provenance_of_ternarized_weight():
    """The ternarized projection differs measurably from its source (paper
    "Provenance safeguards"), by the relative RMSE the oracle's parameters
    give in float64."""
    from paper_2609_09240_gb300 import tq
    N, K = 512, 2560
    W = wl.gen_dense_weights(N, K, config=10, proj=7)
    nnz = int(round(0.1 * N * K / 128))
    Wd = torch.from_numpy(W.view(np.float16)).cuda()
    rep = tq.provenance(Wd, tq.ternarize(Wd, nnz, index=False))
    r = tz.ternarize(W, nnz)
    G = K // 128
    h = lambda b: b.view(np.float16).astype(np.float64)
    s2d = np.zeros(N * G)
    s2d[r["salient"].ravel()] = h(r["s2"])
    R = lambda v: np.repeat(v.reshape(N, G), 128, axis=1)
    Wh = R(h(r["off"])) + R(h(r["s1"])) * r["T1"] + R(s2d) * r["T2"]
    src = h(W)
    want = np.sqrt(((Wh - src) ** 2).sum() / (src ** 2).sum())
    assert not rep["identical"] and rep["changed_fraction"] > 0.9
    assert abs(rep["rel_rmse"] - want) <= 2e-3 * want, (rep, want)


def test_container_round_trip_to_device():
    """Ternarize, serialize from the device, read back with the key check:
    every packed field (and the rebuilt second-plane index) bit-identical,
    and the decode path's outputs equal up to the order of its float32
    atomic additions of second-plane partial sums."""
    import gpu_helpers as H
    from paper_2609_09240_gb300 import tq
    N, K = 1000, 4096
    W = wl.gen_dense_weights(N, K, config=10, proj=8)
    Wd = torch.from_numpy(W.view(np.float16)).cuda()
    pw = tq.ternarize(Wd, int(round(0.1 * N * K / 128)))
    h = tq.fnv1a64(Wd)
    buf = tq.container_write([("layers.3.o", pw, h)])
    out = tq.container_read(buf.tobytes(), expected=["layers.3.o"], device="cuda")
    pw2, h2 = out["layers.3.o"]
    assert h2 == h == tq.fnv1a64(W)
    nnz = pw.nnz
    for k in ("plane1", "salience", "rowptr", "scale1", "offset"):
        assert torch.equal(getattr(pw, k).view(torch.uint8), getattr(pw2, k).view(torch.uint8)), k
    assert pw2.nnz == nnz
    assert torch.equal(pw.plane2[:nnz], pw2.plane2[:nnz]) and torch.equal(pw.scale2[:nnz], pw2.scale2[:nnz])
    # the index's colptr and slots (the alignment gap between them is not part of it)
    G, so = K // 128, tq.lib().tq_plane2_index_slot_offset(K) // 4
    assert torch.equal(pw.p2index[:G + 1], pw2.p2index[:G + 1])
    assert torch.equal(pw.p2index[so:], pw2.p2index[so:])
    x = H.dev(wl.gen_x(3, K, config=10, proj=8))
    y1 = tq.tq_linear_f32out(x, pw)
    y2 = tq.tq_linear_f32out(x, pw2)
    H.device_status_ok()
    torch.testing.assert_close(y1, y2, rtol=1e-5, atol=1e-5)


def test_convert_pipeline():
    """tq.convert: ternarize, provenance and container for a small model;
    reading it back with the expected keys gives the same packed weights."""
    from paper_2609_09240_gb300 import tq
    shapes = {"layers.0.q": (256, 512), "layers.0.down": (128, 1024), "layers.1.k": (64, 512)}
    Ws = {n: torch.from_numpy(wl.gen_dense_weights(N, K, config=10, proj=i).view(np.float16)).cuda()
          for i, (n, (N, K)) in enumerate(shapes.items())}
    buf, reps = tq.convert(Ws)
    assert set(reps) == set(shapes) and all(0.1 < r["rel_rmse"] < 0.9 for r in reps.values())
    out = tq.container_read(buf.tobytes(), expected=list(shapes), device="cuda", index=False)
    for n, W in Ws.items():
        pw, h = out[n]
        assert h == tq.fnv1a64(W)
        ref = tq.ternarize(W, pw.nnz, index=False)
        assert torch.equal(ref.plane1, pw.plane1) and torch.equal(ref.salience, pw.salience)
