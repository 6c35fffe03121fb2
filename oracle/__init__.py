"""CPU oracle of the packed ternary (W1.58A16) linear layer.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline / reference leg of ``bench.py`` may import this package.
The CUDA library never imports, links or calls it, and it imports nothing
from the CUDA library: the two share no code.

``tq_oracle.c`` is the plain C implementation (own byte decoder, fp16 -> fp64
conversion, dense fp64 row reconstruction per the paper's eq. W-hat read per
group of 128, naive dot products); ``codec.py`` is an independent pure-Python
restatement of the byte codec used to cross-check the C codec.

Every function here is exact or fp64; see the module docstrings of the C file
for the paper passages each part follows.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tq_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libtq_oracle.so")
_lock = threading.Lock()
_lib = None

# data-error bits (same meaning as the library's, re-declared here)
BAD_CODE = 1
T2_OUTSIDE = 2
BAD_BYTE = 4
BAD_PAD = 8
BAD_ROWPTR = 16

GROUP = 128
GROUP_BYTES = 26


def build(force: bool = False) -> str:
    """Compile the C oracle with gcc into oracle/_build (plain -O2, portable)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.run(
            ["gcc", "-O2", "-std=c11", "-Wall", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm", "-lpthread"],
            check=True,
        )
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            path = build()
            L = ctypes.CDLL(path)
            c_p = ctypes.c_void_p
            L.tqo_row_bytes.restype = ctypes.c_longlong
            L.tqo_row_bytes.argtypes = [ctypes.c_int]
            L.tqo_sal_words.restype = ctypes.c_longlong
            L.tqo_sal_words.argtypes = [ctypes.c_int]
            L.tqo_half_to_double.restype = ctypes.c_double
            L.tqo_half_to_double.argtypes = [ctypes.c_uint16]
            L.tqo_encode_byte.restype = ctypes.c_int
            L.tqo_encode_byte.argtypes = [c_p]
            L.tqo_decode_byte.restype = ctypes.c_int
            L.tqo_decode_byte.argtypes = [ctypes.c_int, c_p]
            L.tqo_rowptr.restype = ctypes.c_uint
            L.tqo_rowptr.argtypes = [ctypes.c_int, ctypes.c_int, c_p, c_p]
            L.tqo_pack.restype = ctypes.c_uint
            L.tqo_pack.argtypes = [ctypes.c_int, ctypes.c_int, c_p, c_p, c_p, c_p, c_p, c_p]
            L.tqo_unpack.restype = ctypes.c_uint
            L.tqo_unpack.argtypes = [ctypes.c_int, ctypes.c_int, c_p, c_p, c_p, c_p, c_p, c_p]
            L.tqo_linear_rows.restype = ctypes.c_int
            L.tqo_linear_rows.argtypes = [ctypes.c_int] * 3 + [c_p] * 8 + [ctypes.c_int, c_p, c_p, ctypes.c_int]
            _lib = L
    return _lib


def _ptr(a):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


def row_bytes(K: int) -> int:
    return int(lib().tqo_row_bytes(K))


def sal_words(K: int) -> int:
    return int(lib().tqo_sal_words(K))


def half_to_double(bits: int) -> float:
    return float(lib().tqo_half_to_double(bits))


def encode_byte(trits) -> int:
    t = np.ascontiguousarray(np.asarray(trits, dtype=np.int8))
    assert t.shape == (5,)
    return int(lib().tqo_encode_byte(_ptr(t)))


def decode_byte(v: int):
    t = np.zeros(5, np.int8)
    st = int(lib().tqo_decode_byte(int(v), _ptr(t)))
    return t, st


def rowptr(N: int, K: int, sal: np.ndarray):
    sal = np.ascontiguousarray(sal, dtype=np.uint32)
    rp = np.zeros(N + 1, np.int32)
    st = int(lib().tqo_rowptr(N, K, _ptr(sal), _ptr(rp)))
    return rp, st


def pack(N: int, K: int, T1: np.ndarray, T2, sal: np.ndarray, rp: np.ndarray):
    """Returns (plane1 [N][row_bytes] u8, plane2 [nnz][26] u8, status bits)."""
    T1 = np.ascontiguousarray(T1, dtype=np.int8)
    T2 = None if T2 is None else np.ascontiguousarray(T2, dtype=np.int8)
    sal = np.ascontiguousarray(sal, dtype=np.uint32)
    rp = np.ascontiguousarray(rp, dtype=np.int32)
    nnz = int(rp[N])
    p1 = np.zeros((N, row_bytes(K)), np.uint8)
    p2 = np.zeros((max(nnz, 0), GROUP_BYTES), np.uint8)
    st = int(lib().tqo_pack(N, K, _ptr(T1), _ptr(T2), _ptr(sal), _ptr(rp), _ptr(p1), _ptr(p2) if nnz > 0 else None))
    return p1, p2, st


def unpack(N: int, K: int, plane1: np.ndarray, plane2, sal: np.ndarray, rp: np.ndarray, want_t2: bool = True):
    """Returns (T1, T2 or None, status bits)."""
    plane1 = np.ascontiguousarray(plane1, dtype=np.uint8)
    p2 = None if plane2 is None or plane2.size == 0 else np.ascontiguousarray(plane2, dtype=np.uint8)
    sal = np.ascontiguousarray(sal, dtype=np.uint32)
    rp = np.ascontiguousarray(rp, dtype=np.int32)
    T1 = np.zeros((N, K), np.int8)
    T2 = np.zeros((N, K), np.int8) if want_t2 else None
    st = int(lib().tqo_unpack(N, K, _ptr(plane1), _ptr(p2), _ptr(sal), _ptr(rp), _ptr(T1), _ptr(T2)))
    return T1, T2, st


def linear(M, N, K, plane1, plane2, sal, s1, off, s2, x, rows=None, nthreads=None):
    """fp64 y[m][r] and a[m][r] = sum_k |x W| for the selected rows (all if None).

    s1, off: fp16 bit patterns (uint16) [N][G]; s2: uint16 [nnz]; x: uint16 [M][K].
    """
    if nthreads is None:
        nthreads = os.cpu_count() or 1
    plane1 = np.ascontiguousarray(plane1, dtype=np.uint8)
    p2 = None if plane2 is None or plane2.size == 0 else np.ascontiguousarray(plane2, dtype=np.uint8)
    sal = np.ascontiguousarray(sal, dtype=np.uint32)
    s1 = np.ascontiguousarray(s1, dtype=np.uint16)
    off = np.ascontiguousarray(off, dtype=np.uint16)
    s2 = None if s2 is None or np.asarray(s2).size == 0 else np.ascontiguousarray(s2, dtype=np.uint16)
    x = np.ascontiguousarray(x, dtype=np.uint16)
    if rows is None:
        rws, nrows = None, N
    else:
        rws = np.ascontiguousarray(rows, dtype=np.int32)
        nrows = int(rws.size)
    y = np.zeros((M, nrows), np.float64)
    a = np.zeros((M, nrows), np.float64)
    rc = lib().tqo_linear_rows(
        M, N, K, _ptr(plane1), _ptr(p2), _ptr(sal), _ptr(s1), _ptr(off), _ptr(s2), _ptr(x),
        _ptr(rws), nrows, _ptr(y), _ptr(a), int(nthreads),
    )
    if rc != 0:
        raise RuntimeError(f"oracle linear failed: {rc}")
    return y, a
