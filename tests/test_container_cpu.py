"""The packed-weight container (host code of libtq.so, no GPU): round trip,
the paper's provenance checks ("Provenance safeguards": zero missing or
unexpected keys, no malformed packed tensors) and corruption detection.
Packed fields come from the C oracle's packer, so the container is checked
against an independent producer of the format."""
import numpy as np
import pytest

import oracle
import workloads as wl


@pytest.fixture(scope="module")
def tq():
    from paper_2609_09240_gb300 import tq as m
    m.lib()
    return m


def packed_fields(N, K, frac, proj):
    w = wl.gen_weights(N, K, frac, config=10, proj=proj)
    rp, st = oracle.rowptr(N, K, w.sal)
    assert st == 0
    p1, p2, st = oracle.pack(N, K, w.T1, w.T2, w.sal, rp)
    assert st == 0
    return dict(N=N, K=K, nnz=w.nnz, plane1=p1, salience=w.sal.view(np.int32), rowptr=rp, plane2=p2,
                scale1=w.s1.view(np.float16), offset=w.off.view(np.float16),
                scale2=w.s2.view(np.float16) if w.nnz else None)


ENTRIES = [("layers.0.q", 40, 384, 0.1, 1), ("layers.0.k", 7, 4224, 0.3, 2), ("layers.0.v", 1, 128, 0.0, 3),
           ("layers.1.down", 33, 2560, 1.0, 4)]


def build(tq, entries=ENTRIES):
    ws = [(name, packed_fields(N, K, f, p), 1000 + p) for name, N, K, f, p in entries]
    return ws, tq.container_write(ws)


def test_fnv1a64_published_vectors(tq):
    """FNV-1a 64 test vectors published with the algorithm."""
    assert tq.fnv1a64(np.frombuffer(b"", np.uint8)) == 0xCBF29CE484222325
    assert tq.fnv1a64(np.frombuffer(b"a", np.uint8)) == 0xAF63DC4C8601EC8C
    assert tq.fnv1a64(np.frombuffer(b"foobar", np.uint8)) == 0x85944171F73967E8


def test_round_trip(tq):
    ws, buf = build(tq)
    assert bytes(buf[:8]) == b"TQPACK01"
    out = tq.container_read(buf.tobytes(), expected=[e[0] for e in ENTRIES])
    assert list(out) == [e[0] for e in ENTRIES]
    for name, f, h in ws:
        g, gh = out[name]
        assert gh == h and (g["N"], g["K"], g["nnz"]) == (f["N"], f["K"], f["nnz"])
        for k in ("plane1", "salience", "rowptr", "scale1", "offset"):
            assert np.array_equal(g[k].view(np.uint8), np.ascontiguousarray(f[k]).view(np.uint8)), (name, k)
        if f["nnz"]:
            assert np.array_equal(g["plane2"], f["plane2"]) and np.array_equal(g["scale2"], f["scale2"])


def test_keys_missing_and_unexpected(tq):
    """Zero missing / unexpected state keys (paper "Provenance safeguards")."""
    _, buf = build(tq)
    names = [e[0] for e in ENTRIES]
    with pytest.raises(tq.TQError, match="1 missing, 0 unexpected"):
        tq.container_read(buf, expected=names + ["layers.2.q"])
    with pytest.raises(tq.TQError, match="0 missing, 1 unexpected"):
        tq.container_read(buf, expected=names[1:])
    with pytest.raises(tq.TQError, match="1 missing, 1 unexpected"):
        tq.container_read(buf, expected=names[:-1] + ["layers.1.up"])


@pytest.mark.parametrize("name", ["", "x" * 128])
def test_bad_names_rejected(tq, name):
    with pytest.raises(tq.TQError) as e:
        tq.container_write([(name, packed_fields(4, 128, 0.0, 9), 0)])
    assert e.value.code == tq.TQ_ERR_KEY


def test_duplicate_names_rejected(tq):
    f = packed_fields(4, 128, 0.0, 9)
    with pytest.raises(tq.TQError) as e:
        tq.container_write([("a", f, 0), ("a", f, 0)])
    assert e.value.code == tq.TQ_ERR_KEY


def test_empty_container(tq):
    buf = tq.container_write([])
    assert buf.nbytes == 64 and tq.container_read(buf, expected=[]) == {}


def test_every_corrupted_byte_region_is_detected(tq):
    """A flipped bit in the header, the table, any field of any entry or the
    alignment padding between fields makes reading fail (hash mismatch or
    nonzero padding); a truncated or extended buffer too."""
    ws, buf = build(tq)
    rng = np.random.default_rng(0)
    # header and table
    for pos in (3, 12, 40, 64 + 130, 64 + 384 * 2 + 200):
        bad = buf.copy()
        bad[pos] ^= 0x10
        with pytest.raises(tq.TQError) as e:
            tq.container_read(bad)
        assert e.value.code == tq.TQ_ERR_FORMAT, pos
    # fields: positions inside each nonempty field of each entry
    data0 = 64 + 384 * len(ENTRIES)
    for pos in sorted(rng.choice(np.arange(data0, buf.nbytes), 40, replace=False)):
        bad = buf.copy()
        bad[pos] ^= 0x01
        try:
            tq.container_read(bad)
        except tq.TQError as e:
            assert e.code == tq.TQ_ERR_FORMAT
        else:
            raise AssertionError(f"a flipped bit at {pos} ({'field' if _inside_field(buf, pos) else 'padding'}) went unnoticed")
    for n in (buf.nbytes - 1, buf.nbytes + 16):
        cut = np.zeros(n, np.uint8)
        cut[:min(n, buf.nbytes)] = buf[:min(n, buf.nbytes)]
        with pytest.raises(tq.TQError):
            tq.container_read(cut)


def _inside_field(buf, pos):
    count = int(buf[12:16].view(np.uint32)[0])
    for i in range(count):
        e = buf[64 + 384 * i: 64 + 384 * (i + 1)]
        f = e[160:160 + 168].view(np.uint64).reshape(7, 3)
        for off, nb, _ in f:
            if off <= pos < off + nb:
                return True
    return False


def _rewrite(tq, f):
    return tq.container_write([("w", f, 0)])


def test_malformed_packed_tensors_rejected(tq):
    """Fields with valid hashes but invalid content (paper "Provenance
    safeguards": malformed packed tensors): a byte > 242, a tail pad digit
    != 1, a nonzero row pad byte, rowptr disagreeing with the salience map,
    a salience bit past the last group."""
    base = packed_fields(6, 4224, 0.3, 11)  # 33 groups: 858 bytes + 6 pad bytes per row
    assert tq.container_read(_rewrite(tq, base))["w"][0]["nnz"] == base["nnz"]

    def case(mut, code):
        f = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in base.items()}
        mut(f)
        with pytest.raises(tq.TQError) as e:
            tq.container_read(_rewrite(tq, f))
        assert e.value.code == code

    case(lambda f: f["plane1"].__setitem__((2, 7), 243), -5)
    case(lambda f: f["plane1"].__setitem__((0, 25), 121 - 81), -5)       # tail pad digit 0
    case(lambda f: f["plane1"].__setitem__((4, 860), 1), -5)             # row pad byte
    case(lambda f: f["plane2"].__setitem__((0, 3), 250), -5)
    case(lambda f: f["rowptr"].__setitem__(3, f["rowptr"][3] + 1), -6)
    case(lambda f: f["salience"].__setitem__((1, 1), f["salience"][1, 1] | np.int32(1 << 5)), -6)


def test_write_rejects_inconsistent_shapes(tq):
    f = packed_fields(4, 256, 0.0, 12)
    f["nnz"] = 9  # more than N * G
    with pytest.raises(tq.TQError):
        tq.container_write([("w", f, 0)])


def test_file_round_trip(tq, tmp_path):
    """A container saved to a file and loaded back with the key check."""
    ws, buf = build(tq)
    path = tmp_path / "model.tqpack"
    n = tq.save_container(str(path), ws)
    assert n == buf.nbytes == path.stat().st_size
    out = tq.load_container(str(path), expected=[e[0] for e in ENTRIES])
    for name, f, h in ws:
        g, gh = out[name]
        assert gh == h and np.array_equal(g["plane1"], f["plane1"])
    data = bytearray(path.read_bytes())
    data[-3] ^= 0xFF  # inside the last entry's last field
    path.write_bytes(bytes(data))
    with pytest.raises(tq.TQError):
        tq.load_container(str(path))
