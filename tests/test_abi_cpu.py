"""CPU checks of the C-ABI library: it builds for sm_103a, loads, and exports
every entry point declared in include/tq.h (no compute calls without a GPU)."""
import ctypes
import os
import re
import subprocess

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "tq.h")).read()
    return sorted(set(re.findall(r"TQ_API\s+[\w\s\*]*?\b(tq_\w+)\s*\(", text)))


def test_header_declares_the_abi():
    names = declared_symbols()
    for want in ("tq_pack", "tq_unpack", "tq_linear", "tq_linear_f32out", "tq_linear_batched",
                 "tq_salience_rowptr", "tq_row_bytes", "tq_sal_words", "tq_status_str",
                 "tq_workspace_bytes", "tq_batched_workspace_bytes", "tq_get_device_status"):
        assert want in names


def test_library_loads_and_exports_every_symbol():
    from paper_2609_09240_gb300 import build, tq
    path = build.build()
    L = ctypes.CDLL(path)
    for name in declared_symbols():
        assert hasattr(L, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (tq_\w+)", out))
    assert set(declared_symbols()) <= exported
    assert tq.tq_row_bytes(2560) == 528 and tq.tq_row_bytes(100) == 0
    assert tq.tq_sal_words(4224) == 2
    assert "ALIGN" in tq.tq_status_str(-3)


def test_host_side_argument_errors_without_gpu():
    """Shape and null checks return before any CUDA call."""
    from paper_2609_09240_gb300 import tq
    L = tq.lib()
    assert L.tq_salience_rowptr(0, 128, None, None, None, None) == -2
    assert L.tq_salience_rowptr(4, 100, None, None, None, None) == -2
    assert L.tq_salience_rowptr(4, 128, None, None, None, None) == -1
    assert L.tq_pack(4, 128, None, None, None, None, None, None, None, None) == -1
    assert L.tq_unpack(4, 130, None, None, None, None, None, None, None, None) == -2
    assert L.tq_linear(1, 4, 128, None, None, None, None, 0, None) == -1
    assert L.tq_linear_batched(0, 1, None, None, 0, None) == -2
    assert L.tq_linear_batched(17, 1, None, None, 0, None) == -1  # M > 16: the prefill path, null problems
    assert L.tq_linear_batched(1, 0, None, None, 0, None) == -2
    # ternarizer: shape, count and null checks come before anything touches the device
    assert L.tq_ternarize(0, 128, None, 0, 4, *[None] * 8, 0, None, None) == -2
    assert L.tq_ternarize(4, 128, None, 5, 4, *[None] * 8, 0, None, None) == -2   # nnz > N * G
    assert L.tq_ternarize(4, 128, None, 1, 65, *[None] * 8, 0, None, None) == -2  # sweeps > 64
    assert L.tq_ternarize(4, 128, None, 1, 4, *[None] * 8, 0, None, None) == -1
    assert tq.tq_ternarize_workspace_bytes(0, 128) == 0 and tq.tq_ternarize_workspace_bytes(4, 100) == 0
    assert L.tq_dequantize(4, 128, None, None, None, None) == -1
    # stats (16 B) and keys (4 B) per block, the select state, one word per 1024 salience words
    assert tq.tq_ternarize_workspace_bytes(4096, 4096) == 2097152 + 524288 + 4352 + 256
    # M <= 8: activation fragments (320 B per group and token), C/S (64 B per
    # group), second-plane partials (4 B per row and token), each 256-padded,
    # and a 512-byte slot for the tensor maps of plane 1, s1 and off
    pad = lambda b: (b + 255) // 256 * 256
    mma = lambda M, N, K: pad(K // 128 * 320 * M) + pad(K // 128 * 64) + pad(N * M * 4) + 512
    # M <= 2 adds the one-group-per-lane kernel's operands: per stage (8
    # groups for one token, 4 for two) two slices of activation slots (33 or
    # 18 chunks of 64 B), then 64 B of C/S
    # and 16 arrival counters per 256-row tile (tiles shared by several CTAs)
    def g4(M, N, K):
        sg = 8 if M == 1 else 4
        nst = (K // 128 + sg - 1) // sg
        return pad(nst * 2 * (33 if sg == 8 else 18) * 64) + pad(nst * 64) + pad((N + 255) // 256 * 64)
    assert tq.tq_workspace_bytes(1, 4096, 4096) == mma(1, 4096, 4096) + g4(1, 4096, 4096) == 29184 + 16896 + 256 + 1024
    assert tq.tq_workspace_bytes(1, 300, 1152) == mma(1, 300, 1152) + g4(1, 300, 1152)
    assert tq.tq_workspace_bytes(2, 300, 1152) == mma(2, 300, 1152) + g4(2, 300, 1152)
    assert tq.tq_workspace_bytes(5, 100, 1024) == mma(5, 100, 1024)
    # 8 < M <= 16: C/S for two 8-token tiles (128 B per group);
    # M > 16: the prefill tile path needs no workspace (256 bytes are asked for)
    mma16 = lambda M, N, K: pad(K // 128 * 320 * M) + pad(K // 128 * 128) + pad(N * M * 4) + 512
    assert tq.tq_workspace_bytes(16, 4096, 4096) == mma16(16, 4096, 4096)
    assert tq.tq_workspace_bytes(9, 300, 1152) == mma16(9, 300, 1152)
    assert tq.tq_workspace_bytes(40, 64, 4096) == 256
    assert tq.tq_workspace_bytes(1, 4096, 100) == 0
    # second-plane index: int32 colptr[G + 1] padded to 128 bytes, then 32-byte slots for
    # up to nnz + 15 G entries (each group padded to 16), rounded up to 16 entries
    L = tq.lib()
    assert L.tq_plane2_index_slot_offset(4096) == 256  # 33 x 4 = 132 -> 256
    assert L.tq_plane2_index_slot_offset(128) == 128
    assert L.tq_plane2_index_capacity(4096, 13) == 496  # 13 + 15 x 32 = 493 -> 496
    assert L.tq_plane2_index_capacity(4096, 0) == 480
    assert L.tq_plane2_index_bytes(100, 4096, 13) == 256 + 32 * 496
    assert L.tq_plane2_index_bytes(100, 4096, 100 * 32 + 1) == 0  # more records than groups
    assert L.tq_plane2_index_bytes(100, 4000, 13) == 0  # K not a multiple of 128
    assert tq.tq_workspace_bytes(1, 0, 4096) == 0


def test_elementwise_workspace_formulas():
    """tq_ew_workspace_bytes = the views of the plane-1 pass (s1 and off
    [N][G] fp16, zero salience words, zero rowptr) and its fp32 result, each
    256-padded, plus the decode path's workspace; the batched form sums the
    views and results of every problem and then every problem's decode-path
    workspace, and refuses M > 16."""
    from paper_2609_09240_gb300 import tq
    L = tq.lib()
    pad = lambda b: (b + 255) // 256 * 256

    def parts(M, N, K):
        G, W = K // 128, (K // 128 + 31) // 32
        return 2 * pad(N * G * 2) + pad(N * W * 4) + pad((N + 1) * 4) + pad(M * N * 4)
    for M, N, K in ((1, 4096, 4096), (2, 300, 1152), (5, 129, 4224), (40, 256, 1152)):
        assert L.tq_ew_workspace_bytes(M, N, K) == parts(M, N, K) + tq.tq_workspace_bytes(M, N, K)
    assert L.tq_ew_workspace_bytes(1, 4096, 100) == 0 and L.tq_ew_workspace_bytes(0, 64, 128) == 0
    shapes = [(4096, 4096), (1024, 4096), (4096, 12288)]
    arr = (tq.tq_ew_problem * 3)()
    for i, (N, K) in enumerate(shapes):
        arr[i].w.N, arr[i].w.K = N, K
    for M in (1, 2, 16):
        want = sum(parts(M, N, K) + tq.tq_workspace_bytes(M, N, K) for N, K in shapes)
        assert L.tq_ew_batched_workspace_bytes(M, 3, arr) == want
    assert L.tq_ew_batched_workspace_bytes(17, 3, arr) == 0
    arr[1].w.K = 100
    assert L.tq_ew_batched_workspace_bytes(1, 3, arr) == 0


def test_binding_argument_counts_match_the_header():
    """Every function the ctypes binding declares takes as many arguments as
    its prototype in include/tq.h."""
    import os
    import re

    from paper_2609_09240_gb300 import tq
    L = tq.lib()
    text = open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "tq.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    protos = dict(re.findall(r"TQ_API\s+[\w\s\*]*?\b(tq_\w+)\s*\(([^)]*)\)", text))
    checked = 0
    for name, params in protos.items():
        fn = getattr(L, name)
        if fn.argtypes is None:
            continue
        n = 0 if params.strip() in ("", "void") else params.count(",") + 1
        assert len(fn.argtypes) == n, (name, len(fn.argtypes), n)
        checked += 1
    assert checked >= 25
