"""Thin ctypes binding of the C ABI in include/tq.h.

Argument marshalling only: every step of the computation runs in the CUDA
kernels of libtq.so.  Tensors are torch CUDA tensors (torch supplies device
memory and streams); there is no CPU fallback and a missing library raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass

import numpy as np
import torch

from . import build as _build

TQ_GROUP = 128
TQ_GROUP_BYTES = 26
TQ_MAX_SKINNY_M = 16
TQ_MAX_BATCH = 256

TQ_OK = 0
STATUS_NAMES = {0: "TQ_OK", -1: "TQ_ERR_NULL", -2: "TQ_ERR_SHAPE", -3: "TQ_ERR_ALIGN", -4: "TQ_ERR_CODE",
                -5: "TQ_ERR_BYTE", -6: "TQ_ERR_SALIENCE", -7: "TQ_ERR_CUDA", -8: "TQ_ERR_TIMEOUT",
                -9: "TQ_ERR_SCRATCH", -10: "TQ_ERR_FORMAT", -11: "TQ_ERR_KEY"}
TQ_ERR_FORMAT, TQ_ERR_KEY = -10, -11
DATA_BAD_CODE, DATA_T2_OUTSIDE, DATA_BAD_BYTE, DATA_BAD_PAD, DATA_BAD_ROWPTR, DATA_BAD_WEIGHT = 1, 2, 4, 8, 16, 32

_lock = threading.Lock()
_lib = None


class TQError(RuntimeError):
    def __init__(self, code, where):
        super().__init__(f"{where}: {STATUS_NAMES.get(code, code)}")
        self.code = code


class tq_weight(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int32), ("K", ctypes.c_int32), ("group", ctypes.c_int32),
                ("plane1", ctypes.c_void_p), ("salience", ctypes.c_void_p), ("rowptr", ctypes.c_void_p),
                ("plane2", ctypes.c_void_p), ("scale1", ctypes.c_void_p), ("offset", ctypes.c_void_p),
                ("scale2", ctypes.c_void_p), ("nnz", ctypes.c_int64), ("p2index", ctypes.c_void_p)]


class tq_problem(ctypes.Structure):
    _fields_ = [("w", tq_weight), ("x", ctypes.c_void_p), ("y", ctypes.c_void_p)]


class tq_ew_weight(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int32), ("K", ctypes.c_int32), ("mask", ctypes.c_void_p), ("plane1", ctypes.c_void_p),
                ("p2rowptr", ctypes.c_void_p), ("plane2", ctypes.c_void_p), ("mu", ctypes.c_void_p),
                ("alpha0", ctypes.c_void_p), ("alpha1", ctypes.c_void_p), ("idx_off", ctypes.c_void_p),
                ("idx", ctypes.c_void_p)]


class tq_ew_problem(ctypes.Structure):
    _fields_ = [("w", tq_ew_weight), ("x", ctypes.c_void_p), ("y", ctypes.c_void_p)]


class tq_host_weight(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("N", ctypes.c_int32), ("K", ctypes.c_int32), ("nnz", ctypes.c_int64),
                ("plane1", ctypes.c_void_p), ("salience", ctypes.c_void_p), ("rowptr", ctypes.c_void_p),
                ("plane2", ctypes.c_void_p), ("scale1", ctypes.c_void_p), ("offset", ctypes.c_void_p),
                ("scale2", ctypes.c_void_p), ("source_hash", ctypes.c_uint64)]


def lib_path() -> str:
    return _build.LIB


def lib():
    """Load libtq.so (building it first if stale).  Raises if unavailable."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.build()
            if not os.path.exists(path):
                raise RuntimeError(f"CUDA library missing: {path}")
            L = ctypes.CDLL(path)
            vp, i32 = ctypes.c_void_p, ctypes.c_int32
            L.tq_row_bytes.restype = ctypes.c_size_t
            L.tq_row_bytes.argtypes = [i32]
            L.tq_sal_words.restype = ctypes.c_size_t
            L.tq_sal_words.argtypes = [i32]
            L.tq_salience_rowptr.restype = ctypes.c_int
            L.tq_salience_rowptr.argtypes = [i32, i32, vp, vp, vp, vp]
            L.tq_pack.restype = ctypes.c_int
            L.tq_pack.argtypes = [i32, i32, vp, vp, vp, vp, vp, vp, vp, vp]
            i64 = ctypes.c_int64
            L.tq_plane2_index_bytes.restype = ctypes.c_size_t
            L.tq_plane2_index_bytes.argtypes = [i32, i32, i64]
            L.tq_plane2_index_capacity.restype = ctypes.c_size_t
            L.tq_plane2_index_capacity.argtypes = [i32, i64]
            L.tq_plane2_index_slot_offset.restype = ctypes.c_size_t
            L.tq_plane2_index_slot_offset.argtypes = [i32]
            L.tq_plane2_index.restype = ctypes.c_int
            L.tq_plane2_index.argtypes = [i32, i32, vp, vp, i64, vp, vp, vp, vp]
            L.tq_unpack.restype = ctypes.c_int
            L.tq_unpack.argtypes = [i32, i32, vp, vp, vp, vp, vp, vp, vp, vp]
            sz = ctypes.c_size_t
            L.tq_workspace_bytes.restype = sz
            L.tq_workspace_bytes.argtypes = [i32, i32, i32]
            L.tq_batched_workspace_bytes.restype = sz
            L.tq_batched_workspace_bytes.argtypes = [i32, i32, ctypes.POINTER(tq_problem)]
            L.tq_linear.restype = ctypes.c_int
            L.tq_linear.argtypes = [i32, i32, i32, ctypes.POINTER(tq_weight), vp, vp, vp, sz, vp]
            L.tq_linear_f32out.restype = ctypes.c_int
            L.tq_linear_f32out.argtypes = [i32, i32, i32, ctypes.POINTER(tq_weight), vp, vp, vp, sz, vp]
            L.tq_linear_static.restype = ctypes.c_int
            L.tq_linear_static.argtypes = [i32, i32, i32, ctypes.POINTER(tq_weight), vp, vp, vp]
            L.tq_linear_batched.restype = ctypes.c_int
            L.tq_linear_batched.argtypes = [i32, i32, ctypes.POINTER(tq_problem), vp, sz, vp]
            EW = ctypes.POINTER(tq_ew_weight)
            L.tq_ew_rowptr.restype = ctypes.c_int
            L.tq_ew_rowptr.argtypes = [i32, i32, vp, vp, vp, vp]
            L.tq_ew_pack.restype = ctypes.c_int
            L.tq_ew_pack.argtypes = [i32, i32] + [vp] * 8 + [vp]
            L.tq_ew_unpack.restype = ctypes.c_int
            L.tq_ew_unpack.argtypes = [i32, i32] + [vp] * 8 + [vp]
            L.tq_ew_index_offsets.restype = ctypes.c_int
            L.tq_ew_index_offsets.argtypes = [i32, i32, vp, vp, vp]
            L.tq_ew_index_fill.restype = ctypes.c_int
            L.tq_ew_index_fill.argtypes = [i32, i32, EW, vp, vp, vp, vp]
            L.tq_ew_workspace_bytes.restype = sz
            L.tq_ew_workspace_bytes.argtypes = [i32, i32, i32]
            L.tq_ew_linear.restype = ctypes.c_int
            L.tq_ew_linear.argtypes = [i32, i32, i32, EW, vp, vp, vp, sz, vp]
            L.tq_ew_linear_f32out.restype = ctypes.c_int
            L.tq_ew_linear_f32out.argtypes = [i32, i32, i32, EW, vp, vp, vp, sz, vp]
            L.tq_ew_batched_workspace_bytes.restype = sz
            L.tq_ew_batched_workspace_bytes.argtypes = [i32, i32, ctypes.POINTER(tq_ew_problem)]
            L.tq_ew_linear_batched.restype = ctypes.c_int
            L.tq_ew_linear_batched.argtypes = [i32, i32, ctypes.POINTER(tq_ew_problem), vp, sz, vp]
            L.tq_linear_sequence.restype = ctypes.c_int
            L.tq_linear_sequence.argtypes = [i32, i32, ctypes.POINTER(tq_problem), vp, sz, vp]
            L.tq_sequence_selftest.restype = ctypes.c_int
            L.tq_sequence_selftest.argtypes = [i32, ctypes.POINTER(tq_problem), vp, sz, vp]
            L.tq_ternarize_workspace_bytes.restype = sz
            L.tq_ternarize_workspace_bytes.argtypes = [i32, i32]
            L.tq_ternarize.restype = ctypes.c_int
            L.tq_ternarize.argtypes = [i32, i32, vp, i64, i32] + [vp] * 8 + [sz, vp, vp]
            L.tq_dequantize.restype = ctypes.c_int
            L.tq_dequantize.argtypes = [i32, i32, ctypes.POINTER(tq_weight), vp, vp, vp]
            L.tq_fnv1a64.restype = ctypes.c_uint64
            L.tq_fnv1a64.argtypes = [vp, sz]
            HW = ctypes.POINTER(tq_host_weight)
            L.tq_container_bytes.restype = sz
            L.tq_container_bytes.argtypes = [i32, HW]
            L.tq_container_write.restype = ctypes.c_int
            L.tq_container_write.argtypes = [i32, HW, vp, sz]
            L.tq_container_count.restype = ctypes.c_int
            L.tq_container_count.argtypes = [vp, sz, ctypes.POINTER(ctypes.c_int32)]
            L.tq_container_find.restype = ctypes.c_int
            L.tq_container_find.argtypes = [vp, sz, ctypes.c_char_p, ctypes.POINTER(ctypes.c_int32)]
            L.tq_container_entry.restype = ctypes.c_int
            L.tq_container_entry.argtypes = [vp, sz, i32, HW]
            L.tq_container_check_keys.restype = ctypes.c_int
            L.tq_container_check_keys.argtypes = [vp, sz, i32, ctypes.POINTER(ctypes.c_char_p),
                                                  ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int32)]
            L.tq_wait_selftest.restype = ctypes.c_int
            L.tq_wait_selftest.argtypes = [vp, vp]
            L.tq_get_device_status.restype = ctypes.c_int
            L.tq_get_device_status.argtypes = [ctypes.POINTER(ctypes.c_uint32), ctypes.c_int]
            L.tq_status_str.restype = ctypes.c_char_p
            L.tq_status_str.argtypes = [ctypes.c_int]
            _lib = L
    return _lib


def _p(t):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError("expected a torch tensor")
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor (device memory)")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(code, where):
    if code != TQ_OK:
        raise TQError(code, where)


def tq_row_bytes(K: int) -> int:
    return int(lib().tq_row_bytes(K))


def tq_sal_words(K: int) -> int:
    return int(lib().tq_sal_words(K))


def tq_get_device_status(clear: bool = True) -> int:
    """Synchronous read of the library's device status word (0 = no bounded
    wait ran out)."""
    v = ctypes.c_uint32(0)
    _check(lib().tq_get_device_status(ctypes.byref(v), 1 if clear else 0), "tq_get_device_status")
    return int(v.value)


def tq_status_str(code: int) -> str:
    return lib().tq_status_str(code).decode()


def tq_salience_rowptr(N, K, sal, rowptr, d_status, stream=None):
    _check(lib().tq_salience_rowptr(N, K, _p(sal), _p(rowptr), _p(d_status), _stream(stream)), "tq_salience_rowptr")


def tq_pack(N, K, T1, T2, sal, rowptr, plane1, plane2, d_status, stream=None):
    _check(lib().tq_pack(N, K, _p(T1), _p(T2), _p(sal), _p(rowptr), _p(plane1), _p(plane2), _p(d_status),
                         _stream(stream)), "tq_pack")


def tq_unpack(N, K, plane1, plane2, sal, rowptr, T1, T2, d_status, stream=None):
    _check(lib().tq_unpack(N, K, _p(plane1), _p(plane2), _p(sal), _p(rowptr), _p(T1), _p(T2), _p(d_status),
                           _stream(stream)), "tq_unpack")


def tq_plane2_index(N, K, sal, rowptr, nnz, plane2, scale2, stream=None):
    """The group-ordered second-plane index of a weight (int32 device tensor), see tq.h."""
    nbytes = int(lib().tq_plane2_index_bytes(N, K, nnz))
    if nbytes == 0:
        raise TQError(-2, "tq_plane2_index_bytes")
    idx = torch.empty(nbytes // 4, dtype=torch.int32, device=sal.device)
    _check(lib().tq_plane2_index(N, K, _p(sal), _p(rowptr), nnz, _p(plane2), _p(scale2), _p(idx), _stream(stream)),
           "tq_plane2_index")
    return idx


@dataclass
class PackedWeight:
    """Device tensors of one packed projection (the fields of tq_weight)."""
    N: int
    K: int
    plane1: torch.Tensor   # uint8 [N][row_bytes]
    salience: torch.Tensor  # int32 (uint32 bits) [N][sal_words]
    rowptr: torch.Tensor   # int32 [N+1]
    plane2: torch.Tensor | None   # uint8 [nnz][26]
    scale1: torch.Tensor   # fp16 [N][G]
    offset: torch.Tensor   # fp16 [N][G]
    scale2: torch.Tensor | None   # fp16 [nnz]
    nnz: int
    p2index: torch.Tensor | None = None  # int32, tq_plane2_index (optional)

    def struct(self) -> tq_weight:
        w = tq_weight()
        w.N, w.K, w.group = self.N, self.K, TQ_GROUP
        w.plane1 = self.plane1.data_ptr()
        w.salience = self.salience.data_ptr()
        w.rowptr = self.rowptr.data_ptr()
        w.plane2 = self.plane2.data_ptr() if self.plane2 is not None and self.nnz > 0 else None
        w.scale1 = self.scale1.data_ptr()
        w.offset = self.offset.data_ptr()
        w.scale2 = self.scale2.data_ptr() if self.scale2 is not None and self.nnz > 0 else None
        w.nnz = self.nnz
        w.p2index = self.p2index.data_ptr() if self.p2index is not None and self.nnz > 0 else None
        return w

    def packed_bytes(self) -> int:
        """Bytes of the packed representation read by the linear kernels."""
        t = [self.plane1, self.salience, self.rowptr, self.scale1, self.offset]
        if self.nnz:
            t += [self.plane2, self.scale2]
        return sum(x.numel() * x.element_size() for x in t)


def pack_weight(T1, T2, sal, s1, off, s2, stream=None, check=True, index=True) -> PackedWeight:
    """Pack device int8 codes + fp16 params with tq_salience_rowptr + tq_pack
    (and, unless index=False, the second-plane index).

    Reads nnz back to the host (one synchronization) to size plane 2."""
    N, K = T1.shape
    dev = T1.device
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    rowptr = torch.empty(N + 1, dtype=torch.int32, device=dev)
    tq_salience_rowptr(N, K, sal, rowptr, status, stream)
    nnz = int(rowptr[N].item())
    plane1 = torch.empty((N, tq_row_bytes(K)), dtype=torch.uint8, device=dev)
    plane2 = torch.empty((max(nnz, 1), TQ_GROUP_BYTES), dtype=torch.uint8, device=dev)
    tq_pack(N, K, T1, T2 if nnz > 0 else None, sal, rowptr, plane1, plane2 if nnz > 0 else None, status, stream)
    if check:
        st = int(status.item())
        if st:
            raise TQError(-4, f"tq_pack data status {st:#x}")
    if s2 is None or nnz == 0:
        s2 = torch.zeros(1, dtype=torch.float16, device=dev)
    p2index = tq_plane2_index(N, K, sal, rowptr, nnz, plane2, s2, stream) if index and nnz > 0 else None
    return PackedWeight(N, K, plane1, sal, rowptr, plane2, s1, off, s2, nnz, p2index)


def tq_ternarize_workspace_bytes(N: int, K: int) -> int:
    return int(lib().tq_ternarize_workspace_bytes(N, K))


def ternarize(W, nnz: int, sweeps: int = 4, d_status=None, ws=None, stream=None, index=True) -> PackedWeight:
    """E2M-ATQ ternarization (tq_ternarize) of fp16 W [N][K] on the device
    into a packed weight with nnz salient groups (and, unless index=False,
    its second-plane index).  d_status: optional int32 device word the data
    status is OR-ed into (else a fresh one, not read)."""
    N, K = W.shape
    dev = W.device
    G = K // TQ_GROUP
    plane1 = torch.empty((N, tq_row_bytes(K)), dtype=torch.uint8, device=dev)
    sal = torch.empty((N, tq_sal_words(K)), dtype=torch.int32, device=dev)
    rowptr = torch.empty(N + 1, dtype=torch.int32, device=dev)
    plane2 = torch.empty((max(nnz, 1), TQ_GROUP_BYTES), dtype=torch.uint8, device=dev)
    s1 = torch.empty((N, G), dtype=torch.float16, device=dev)
    off = torch.empty((N, G), dtype=torch.float16, device=dev)
    s2 = torch.empty(max(nnz, 1), dtype=torch.float16, device=dev)
    if ws is None:
        ws = workspace(tq_ternarize_workspace_bytes(N, K), dev)
    if d_status is None:
        d_status = torch.zeros(1, dtype=torch.int32, device=dev)
    _check(lib().tq_ternarize(N, K, _p(W), nnz, sweeps, _p(plane1), _p(sal), _p(rowptr),
                              _p(plane2) if nnz > 0 else None, _p(s1), _p(off), _p(s2) if nnz > 0 else None,
                              _p(ws), ws.numel(), _p(d_status), _stream(stream)), "tq_ternarize")
    p2index = tq_plane2_index(N, K, sal, rowptr, nnz, plane2, s2, stream) if index and nnz > 0 else None
    return PackedWeight(N, K, plane1, sal, rowptr, plane2, s1, off, s2, nnz, p2index)


def tq_dequantize(w: PackedWeight, out=None, d_status=None, stream=None):
    """W-hat of a packed weight as dense fp16 [N][K] on the device."""
    if out is None:
        out = torch.empty((w.N, w.K), dtype=torch.float16, device=w.plane1.device)
    if d_status is None:
        d_status = torch.zeros(1, dtype=torch.int32, device=w.plane1.device)
    ws_ = w.struct()
    _check(lib().tq_dequantize(w.N, w.K, ctypes.byref(ws_), _p(out), _p(d_status), _stream(stream)), "tq_dequantize")
    return out


def provenance(W_source, w: PackedWeight, stream=None) -> dict:
    """The paper's "measurable weight change" check of a packed weight
    against its fp16 source (both on the device): relative RMSE of W-hat,
    the fraction of weights whose fp16 value changed, and whether W-hat is
    bit-identical to the source (which a real ternarization never is)."""
    Wh = tq_dequantize(w, stream=stream)
    src = W_source.float()
    err = (Wh.float() - src).pow(2).sum().sqrt() / src.pow(2).sum().sqrt().clamp_min(1e-30)
    changed = (Wh.view(torch.int16) != W_source.view(torch.int16)).float().mean()
    return {"rel_rmse": float(err), "changed_fraction": float(changed), "identical": bool(changed == 0)}


# ---------------------------------------------------------------- container
FIELDS = ("plane1", "salience", "rowptr", "plane2", "scale1", "offset", "scale2")


def fnv1a64(a) -> int:
    """FNV-1a 64 of a host array's bytes (or of a device tensor, copied to the host)."""
    if isinstance(a, torch.Tensor):
        a = a.detach().contiguous().cpu().numpy()
    a = np.ascontiguousarray(a)
    return int(lib().tq_fnv1a64(a.ctypes.data_as(ctypes.c_void_p), a.nbytes))


def _aligned_bytes(n: int, align: int = 16) -> np.ndarray:
    raw = np.empty(n + align, np.uint8)
    off = (-raw.ctypes.data) % align
    return raw[off:off + n]


def _host_fields(w) -> dict:
    """Host numpy copies of a weight's seven fields (PackedWeight or dict of arrays)."""
    if isinstance(w, PackedWeight):
        nnz = w.nnz
        d = {"plane1": w.plane1, "salience": w.salience, "rowptr": w.rowptr, "scale1": w.scale1, "offset": w.offset,
             "plane2": w.plane2[:nnz] if nnz else None, "scale2": w.scale2[:nnz] if nnz else None}
        d = {k: (None if v is None else v.detach().contiguous().cpu().numpy()) for k, v in d.items()}
        return dict(N=w.N, K=w.K, nnz=nnz, **d)
    return dict(w)


def container_write(entries) -> np.ndarray:
    """Serialize [(name, weight, source_hash), ...] (weight: PackedWeight or a
    dict with N, K, nnz and the seven host fields) into a 16-byte aligned
    uint8 array, ready to be written to a file."""
    hs = (tq_host_weight * max(len(entries), 1))()
    keep = []
    for i, (name, w, src_hash) in enumerate(entries):
        f = _host_fields(w)
        h = hs[i]
        nb = name.encode()
        keep.append(nb)
        h.name, h.N, h.K, h.nnz, h.source_hash = nb, int(f["N"]), int(f["K"]), int(f["nnz"]), int(src_hash)
        for k in FIELDS:
            a = f.get(k)
            if a is not None and a.size:
                a = np.ascontiguousarray(a)
                keep.append(a)
                setattr(h, k, a.ctypes.data_as(ctypes.c_void_p))
            else:
                setattr(h, k, None)
    n = int(lib().tq_container_bytes(len(entries), hs))
    if n == 0:
        raise TQError(-2, "tq_container_bytes")
    buf = _aligned_bytes(n)
    _check(lib().tq_container_write(len(entries), hs, buf.ctypes.data_as(ctypes.c_void_p), n), "tq_container_write")
    return buf


def container_read(data, expected=None, device=None, index=True):
    """Check and unpack a container.  `data`: bytes or a uint8 array.  With
    `expected` (list of names) the key check runs first and raises on any
    missing or unexpected name.  Returns {name: (weight, source_hash)}; the
    weight is a dict of host numpy arrays (device None) or a PackedWeight on
    `device` (with its second-plane index unless index=False)."""
    buf = _aligned_bytes(len(data))
    buf[:] = np.frombuffer(data, np.uint8) if not isinstance(data, np.ndarray) else data.view(np.uint8)
    p, n = buf.ctypes.data_as(ctypes.c_void_p), buf.nbytes
    L = lib()
    if expected is not None:
        names = (ctypes.c_char_p * max(len(expected), 1))(*[e.encode() for e in expected])
        miss, extra = ctypes.c_int32(0), ctypes.c_int32(0)
        rc = L.tq_container_check_keys(p, n, len(expected), names, ctypes.byref(miss), ctypes.byref(extra))
        if rc == TQ_ERR_KEY:
            raise TQError(rc, f"container keys: {miss.value} missing, {extra.value} unexpected")
        _check(rc, "tq_container_check_keys")
    cnt = ctypes.c_int32(0)
    _check(L.tq_container_count(p, n, ctypes.byref(cnt)), "tq_container_count")
    out = {}
    for i in range(cnt.value):
        h = tq_host_weight()
        _check(L.tq_container_entry(p, n, i, ctypes.byref(h)), f"tq_container_entry {i}")
        N, K, nnz = h.N, h.K, h.nnz
        G = K // TQ_GROUP
        shapes = {"plane1": ((N, tq_row_bytes(K)), np.uint8), "salience": ((N, tq_sal_words(K)), np.int32),
                  "rowptr": ((N + 1,), np.int32), "plane2": ((nnz, TQ_GROUP_BYTES), np.uint8),
                  "scale1": ((N, G), np.float16), "offset": ((N, G), np.float16), "scale2": ((nnz,), np.float16)}
        f = {}
        for k, (shape, dt) in shapes.items():
            ptr = getattr(h, k)
            cnt_el = int(np.prod(shape))
            if not ptr or cnt_el == 0:
                f[k] = np.zeros(shape, dt)
                continue
            off = ptr - buf.ctypes.data
            f[k] = buf[off:off + cnt_el * np.dtype(dt).itemsize].view(dt).reshape(shape).copy()
        name = h.name.decode()
        if device is None:
            out[name] = (dict(N=N, K=K, nnz=nnz, **f), int(h.source_hash))
            continue
        t = {k: torch.from_numpy(v).to(device) for k, v in f.items()}
        plane2 = t["plane2"] if nnz else torch.zeros((1, TQ_GROUP_BYTES), dtype=torch.uint8, device=device)
        s2 = t["scale2"] if nnz else torch.zeros(1, dtype=torch.float16, device=device)
        p2i = tq_plane2_index(N, K, t["salience"], t["rowptr"], nnz, plane2, s2) if index and nnz else None
        out[name] = (PackedWeight(N, K, t["plane1"], t["salience"], t["rowptr"], plane2, t["scale1"], t["offset"],
                                  s2, nnz, p2i), int(h.source_hash))
    return out


def save_container(path, entries) -> int:
    """container_write(entries) into the file at `path` (written to a
    temporary name, then renamed, so a reader never sees a partial file).
    Returns the bytes written."""
    buf = container_write(entries)
    tmp = f"{path}.tmp{os.getpid()}"
    with open(tmp, "wb") as f:
        f.write(buf.tobytes())
    os.replace(tmp, path)
    return buf.nbytes


def load_container(path, expected=None, device=None, index=True):
    """container_read of the file at `path` (every check of the reader applies)."""
    with open(path, "rb") as f:
        data = f.read()
    return container_read(data, expected=expected, device=device, index=index)


def convert(weights, salient_fraction: float = 0.1, sweeps: int = 4, stream=None):
    """The paper's conversion pipeline from E2M-ATQ to serialization, for a
    dict {name: fp16 [N][K] device tensor}: each projection ternarized
    (round(salient_fraction * N * K / 128) salient groups), its provenance
    checked (it must differ from the source), and all of them written into
    one container, each with its source's FNV-1a 64 fingerprint.  Returns
    (container bytes as a uint8 array, {name: provenance report})."""
    entries, reports = [], {}
    for name, W in weights.items():
        N, K = W.shape
        st = torch.zeros(1, dtype=torch.int32, device=W.device)
        pw = ternarize(W, int(round(salient_fraction * N * K / TQ_GROUP)), sweeps=sweeps, d_status=st,
                       stream=stream, index=False)
        rep = provenance(W, pw, stream=stream)
        status = int(st.item())
        if status:
            raise TQError(-4, f"tq_ternarize {name}: data status {status:#x}")
        if rep["identical"]:
            raise TQError(-4, f"{name}: the packed weight reproduces its source exactly (not ternarized)")
        reports[name] = rep
        entries.append((name, pw, fnv1a64(W)))
    return container_write(entries), reports


def tq_workspace_bytes(M: int, N: int, K: int) -> int:
    return int(lib().tq_workspace_bytes(M, N, K))


def workspace(nbytes: int, device) -> torch.Tensor:
    """Device scratch for the decode path (torch allocations are 256-byte aligned)."""
    t = torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)
    assert t.data_ptr() % 256 == 0
    return t


def tq_linear(x, w: PackedWeight, y=None, ws=None, stream=None):
    """y = x W^T, fp16.  x: fp16 [M][K] on the device; ws: optional workspace."""
    M, K = x.shape
    assert K == w.K and x.dtype == torch.float16
    if y is None:
        y = torch.empty((M, w.N), dtype=torch.float16, device=x.device)
    if ws is None:
        ws = workspace(tq_workspace_bytes(M, w.N, K), x.device)
    ws_ = w.struct()
    _check(lib().tq_linear(M, w.N, K, ctypes.byref(ws_), _p(x), _p(y), _p(ws), ws.numel(), _stream(stream)),
           "tq_linear")
    return y


def tq_linear_f32out(x, w: PackedWeight, y=None, ws=None, stream=None):
    M, K = x.shape
    assert K == w.K and x.dtype == torch.float16
    if y is None:
        y = torch.empty((M, w.N), dtype=torch.float32, device=x.device)
    if ws is None:
        ws = workspace(tq_workspace_bytes(M, w.N, K), x.device)
    ws_ = w.struct()
    _check(lib().tq_linear_f32out(M, w.N, K, ctypes.byref(ws_), _p(x), _p(y), _p(ws), ws.numel(),
                                  _stream(stream)), "tq_linear_f32out")
    return y


STATIC_SCRATCH_BYTES = 1 << 20  # TQ_STATIC_SCRATCH_BYTES


def tq_linear_static(x, w: PackedWeight, y=None, stream=None):
    """y = x W^T, fp16, with the library's own device scratch (no workspace
    argument, nothing allocated by the call except y when y is None)."""
    M, K = x.shape
    assert K == w.K and x.dtype == torch.float16
    if y is None:
        y = torch.empty((M, w.N), dtype=torch.float16, device=x.device)
    ws_ = w.struct()
    _check(lib().tq_linear_static(M, w.N, K, ctypes.byref(ws_), _p(x), _p(y), _stream(stream)), "tq_linear_static")
    return y


class Batch:
    """A prepared tq_problem array (host memory) and its device workspace."""

    def __init__(self, M, items, device=None):
        self.M = M
        self.items = list(items)  # (PackedWeight, x, y); keeps tensors alive
        self.arr = (tq_problem * len(self.items))()
        for i, (w, x, y) in enumerate(self.items):
            self.arr[i].w = w.struct()
            self.arr[i].x = x.data_ptr()
            self.arr[i].y = y.data_ptr()
        nbytes = int(lib().tq_batched_workspace_bytes(M, len(self.items), self.arr))
        if nbytes == 0:
            raise TQError(-2, "tq_batched_workspace_bytes")
        dev = device if device is not None else self.items[0][1].device
        self.ws = workspace(nbytes, dev)


def tq_linear_batched(batch: Batch, stream=None):
    _check(lib().tq_linear_batched(batch.M, len(batch.items), batch.arr, _p(batch.ws), batch.ws.numel(),
                                   _stream(stream)), "tq_linear_batched")


def tq_linear_sequence(batch: Batch, stream=None):
    """The batch's problems in order, each complete before the next starts
    (one persistent launch; M must be 1)."""
    _check(lib().tq_linear_sequence(batch.M, len(batch.items), batch.arr, _p(batch.ws), batch.ws.numel(),
                                    _stream(stream)), "tq_linear_sequence")


def tq_sequence_selftest(batch: Batch, stream=None):
    """Runs the sequence kernel with a problem barrier that cannot complete
    (its bounded wait runs out; the device status then reports the timeout)."""
    _check(lib().tq_sequence_selftest(len(batch.items), batch.arr, _p(batch.ws), batch.ws.numel(), _stream(stream)),
           "tq_sequence_selftest")


# ------------------------------------------------ element-wise four masks
@dataclass
class EwWeight:
    """Device tensors of one projection in the element-wise four-mask form
    (the fields of tq_ew_weight)."""
    N: int
    K: int
    mask: torch.Tensor      # int32 (uint32 bits) [N][K/16]
    plane1: torch.Tensor    # uint8 [N][row_bytes]
    p2rowptr: torch.Tensor  # int32 [N+1]
    plane2: torch.Tensor    # uint8 [max(p2rowptr[N], 1)]
    mu: torch.Tensor        # fp16 [N][4]
    alpha0: torch.Tensor    # fp16 [N][4]
    alpha1: torch.Tensor    # fp16 [N][2]
    idx_off: torch.Tensor | None = None  # int32 [N nb + 1] (nb = ceil(K / 2048)), correction index (ew_index)
    idx: torch.Tensor | None = None      # int16 (uint16 bits) entries

    def struct(self) -> tq_ew_weight:
        w = tq_ew_weight()
        w.N, w.K = self.N, self.K
        w.mask, w.plane1, w.p2rowptr = self.mask.data_ptr(), self.plane1.data_ptr(), self.p2rowptr.data_ptr()
        w.plane2 = self.plane2.data_ptr()
        w.mu, w.alpha0, w.alpha1 = self.mu.data_ptr(), self.alpha0.data_ptr(), self.alpha1.data_ptr()
        if self.idx_off is not None:
            w.idx_off, w.idx = self.idx_off.data_ptr(), self.idx.data_ptr()
        return w

    def index_bytes(self) -> int:
        """Bytes of the correction index (0 without one)."""
        if self.idx_off is None:
            return 0
        return self.idx_off.numel() * 4 + int(self.idx_off[-1].item()) * 2

    def packed_bytes(self) -> int:
        t = [self.mask, self.plane1, self.p2rowptr, self.mu, self.alpha0, self.alpha1]
        return sum(x.numel() * x.element_size() for x in t) + int(self.p2rowptr[-1].item())


def pack_ew_weight(T0, T1, mask_ids, mu, a0, a1, stream=None, check=True) -> EwWeight:
    """Pack device int8 T0, T1 [N][K] and uint8 mask ids with tq_ew_rowptr +
    tq_ew_pack (one synchronization, to size plane 2)."""
    N, K = T0.shape
    dev = T0.device
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    rp = torch.empty(N + 1, dtype=torch.int32, device=dev)
    _check(lib().tq_ew_rowptr(N, K, _p(mask_ids), _p(rp), _p(status), _stream(stream)), "tq_ew_rowptr")
    nb = int(rp[N].item())
    mplane = torch.empty((N, K // 16), dtype=torch.int32, device=dev)
    plane1 = torch.empty((N, tq_row_bytes(K)), dtype=torch.uint8, device=dev)
    plane2 = torch.empty(max(nb, 1), dtype=torch.uint8, device=dev)
    _check(lib().tq_ew_pack(N, K, _p(T0), _p(T1), _p(mask_ids), _p(rp), _p(mplane), _p(plane1), _p(plane2),
                            _p(status), _stream(stream)), "tq_ew_pack")
    if check:
        st = int(status.item())
        if st:
            raise TQError(-4, f"tq_ew_pack data status {st:#x}")
    return EwWeight(N, K, mplane, plane1, rp, plane2, mu, a0, a1)


def ew_index(w: EwWeight, stream=None, check=True) -> EwWeight:
    """The weight with its correction index built (tq_ew_index_offsets +
    tq_ew_index_fill; one synchronization, to size the entries)."""
    import dataclasses
    dev = w.plane1.device
    nb = (w.K + 2047) // 2048
    off = torch.empty(w.N * nb + 1, dtype=torch.int32, device=dev)
    _check(lib().tq_ew_index_offsets(w.N, w.K, _p(w.mask), _p(off), _stream(stream)), "tq_ew_index_offsets")
    ne = int(off[-1].item())
    idx = torch.empty(max(ne, 1), dtype=torch.int16, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    s = w.struct()
    _check(lib().tq_ew_index_fill(w.N, w.K, ctypes.byref(s), _p(off), _p(idx), _p(status), _stream(stream)),
           "tq_ew_index_fill")
    if check:
        st = int(status.item())
        if st:
            raise TQError(-4, f"tq_ew_index_fill data status {st:#x}")
    return dataclasses.replace(w, idx_off=off, idx=idx)


def tq_ew_unpack(w: EwWeight, status=None, stream=None):
    """-> (T0, T1, mask ids) on the device."""
    dev = w.plane1.device
    if status is None:
        status = torch.zeros(1, dtype=torch.int32, device=dev)
    T0 = torch.empty((w.N, w.K), dtype=torch.int8, device=dev)
    T1 = torch.empty((w.N, w.K), dtype=torch.int8, device=dev)
    m = torch.empty((w.N, w.K), dtype=torch.uint8, device=dev)
    _check(lib().tq_ew_unpack(w.N, w.K, _p(w.mask), _p(w.plane1), _p(w.p2rowptr), _p(w.plane2), _p(T0), _p(T1), _p(m),
                              _p(status), _stream(stream)), "tq_ew_unpack")
    return T0, T1, m


def tq_ew_linear(x, w: EwWeight, y=None, ws=None, stream=None, f32=False):
    """y = x W-hat^T for the element-wise form (fp16, or fp32 with f32=True)."""
    M, K = x.shape
    assert K == w.K and x.dtype == torch.float16
    if y is None:
        y = torch.empty((M, w.N), dtype=torch.float32 if f32 else torch.float16, device=x.device)
    if ws is None:
        ws = workspace(int(lib().tq_ew_workspace_bytes(M, w.N, K)), x.device)
    s = w.struct()
    fn = lib().tq_ew_linear_f32out if f32 else lib().tq_ew_linear
    _check(fn(M, w.N, K, ctypes.byref(s), _p(x), _p(y), _p(ws), ws.numel(), _stream(stream)), "tq_ew_linear")
    return y


class EwBatch:
    """A prepared tq_ew_problem array (host memory) and its device workspace."""

    def __init__(self, M, items, device=None):
        self.M = M
        self.items = list(items)  # (EwWeight, x, y); keeps tensors alive
        self.arr = (tq_ew_problem * len(self.items))()
        for i, (w, x, y) in enumerate(self.items):
            self.arr[i].w = w.struct()
            self.arr[i].x = x.data_ptr()
            self.arr[i].y = y.data_ptr()
        nbytes = int(lib().tq_ew_batched_workspace_bytes(M, len(self.items), self.arr))
        if nbytes == 0:
            raise TQError(-2, "tq_ew_batched_workspace_bytes")
        dev = device if device is not None else self.items[0][1].device
        self.ws = workspace(nbytes, dev)


def tq_ew_linear_batched(batch: EwBatch, stream=None):
    _check(lib().tq_ew_linear_batched(batch.M, len(batch.items), batch.arr, _p(batch.ws), batch.ws.numel(),
                                      _stream(stream)), "tq_ew_linear_batched")
