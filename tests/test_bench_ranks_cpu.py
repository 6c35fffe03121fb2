"""The bench's multi-rank arithmetic on two gloo ranks (CPU): every rank
ends with the slowest rank's time, and the whole-job rate counts the units
of all replicas over that time."""
import os

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench

    ms = bench.max_over_ranks(10.0 + 5.0 * rank, dist, "cpu")
    out[rank] = (ms, bench.whole_job_rate(1.5e9, world, ms))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_and_rate_gloo():
    port = 29500 + os.getpid() % 2000
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank, args=(2, port, out), nprocs=2, join=True)
        res = dict(out)
    assert res[0][0] == res[1][0] == 15.0
    assert res[0][1] == pytest.approx(2 * 1.5e9 / 15e-3 / 1e9)


def test_single_process_passthrough():
    import bench

    assert bench.max_over_ranks(3.25, None, "cpu") == 3.25
    assert bench.whole_job_rate(1.79e9, 1, 0.73) == pytest.approx(1.79e9 / 0.73e-3 / 1e9)


def test_kernel_hash_ignores_comments(tmp_path, monkeypatch):
    """The key of the committed traffic summary: a // comment or blank line
    added to a decode source keeps it, a changed line of code does not."""
    import shutil

    import bench

    csrc = tmp_path / "paper_2609_09240_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for f in bench.DECODE_SOURCES:
        shutil.copy(os.path.join(bench.ROOT, "paper_2609_09240_gb300", "csrc", f), csrc / f)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h0 = bench.kernel_hash()
    src = csrc / "tq_gemv_g4.cu"
    text = src.read_text()
    src.write_text("// a note\n\n" + text.replace("\n", "  // trailing\n", 1))
    assert bench.kernel_hash() == h0
    src.write_text(text.replace("kP2rTiles = 8;", "kP2rTiles = 9;", 1))
    assert "kP2rTiles = 9;" in src.read_text() and bench.kernel_hash() != h0
