"""The C ABI: the library loads, exports every symbol include/dart.h declares,
and rejects bad arguments on the host before launching anything (so these
run without a GPU)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    import torch  # noqa: F401  (loads the CUDA runtime libdart.so links against)

    from paper_2608_02032_gb300 import binding, build

    build.build()
    return binding.lib()


def _declared():
    src = open(os.path.join(ROOT, "include", "dart.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dart_[a-z_0-9]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(L):
    names = _declared()
    assert {"dart_chunk_scan", "dart_sma_forward", "dart_decode_step"} <= set(names)
    for n in names:
        assert hasattr(L, n), f"{n} declared in dart.h but not exported"


def test_binding_covers_the_header():
    from paper_2608_02032_gb300 import binding

    assert set(binding.EXPORTED) == set(_declared())


def test_status_strings(L):
    for s in range(7):
        assert L.dart_status_string(s)
    assert b"unknown" in L.dart_status_string(99)


def _dims(**kw):
    from paper_2608_02032_gb300 import binding as B

    base = dict(batch=1, seqlen=512, nheads=2, ngroups=1, headdim=64, dstate=128, chunk=128,
                dtype=B.DART_BF16, eps=1e-6)
    base.update(kw)
    return B.make_dims(**base)


def test_workspace_sizes(L):
    from paper_2608_02032_gb300 import binding as B

    d = _dims()
    M = 512 // 128
    cum = 1 * 2 * M * 128 * 4
    dh = 1 * M * 2 * 128 * 64 * 4
    assert B.dart_workspace_size(d, B.DART_OP_CHUNK_SCAN) == cum + dh
    # bf16 tensor-core path: 96 KiB of pre-swizzled operands per (memory, head pair) + per-memory scales
    ops = 1 * M * 1 * 96 * 1024
    assert B.dart_workspace_size(d, B.DART_OP_SMA_FORWARD) == ops + (1 * M * 2 * 4 + 255) // 256 * 256
    # fp32 inputs take the CUDA-core path: one inverse RMS per memory row
    d32 = _dims(dtype=B.DART_F32)
    assert B.dart_workspace_size(d32, B.DART_OP_SMA_FORWARD) == (1 * M * 2 * 128 * 4 + 255) // 256 * 256
    assert B.dart_workspace_size(d, B.DART_OP_DECODE_STEP) == 0
    assert B.dart_workspace_size(_dims(headdim=48), B.DART_OP_CHUNK_SCAN) == 0


FAKE = 1 << 20  # a 16-byte aligned address that is never dereferenced: validation fails first


def _scan(L, d, ptrs=None, ws=FAKE, ws_bytes=1 << 40):
    v = ctypes.c_void_p
    p = ptrs or [FAKE] * 7
    return L.dart_chunk_scan(ctypes.byref(d), *[v(x) for x in p], None, None, v(ws), ws_bytes, None)


@pytest.mark.parametrize("kw,code", [
    (dict(batch=0), 1), (dict(seqlen=-4), 1), (dict(nheads=3, ngroups=2), 1), (dict(eps=0.0), 1),
    (dict(dtype=7), 1), (dict(headdim=48), 2), (dict(dstate=256), 2), (dict(chunk=96), 2),
    (dict(chunk=512, seqlen=1024), 2),
])
def test_bad_dims_rejected(L, kw, code):
    assert _scan(L, _dims(**kw)) == code


def test_ragged_length(L):
    """L % S != 0: the forward calls take it with a workspace that holds zero-padded
    copies of the token tensors (L = 500, S = 128 runs as 512 tokens); the backward
    calls refuse it."""
    from paper_2608_02032_gb300 import binding as B

    d, d512 = _dims(seqlen=500), _dims(seqlen=512)
    al = lambda v: (v + 255) // 256 * 256
    rows = 512  # Bsz 1 x 512 padded tokens; H 2, P 64, G 1, N 128, bf16 inputs, fp32 outputs
    copies = al(rows * 2 * 64 * 2) + al(rows * 2 * 4) + 2 * al(rows * 128 * 2) + al(rows * 2 * 64 * 4)
    assert B.dart_workspace_size(d, B.DART_OP_CHUNK_SCAN) == copies + B.dart_workspace_size(d512, B.DART_OP_CHUNK_SCAN)
    assert B.dart_workspace_size(d, B.DART_OP_SMA_FORWARD) > B.dart_workspace_size(d512, B.DART_OP_SMA_FORWARD)
    assert _scan(L, d, ws_bytes=100) == 3  # valid sizes, workspace too small
    v = ctypes.c_void_p
    assert L.dart_chunk_scan_backward(ctypes.byref(d), *[v(FAKE)] * 12, v(FAKE), 1 << 40, None) == 2
    assert B.dart_workspace_size(d, B.DART_OP_SCAN_BACKWARD) == 0


def test_null_and_misaligned_pointers_rejected(L):
    d = _dims()
    assert _scan(L, d, [FAKE] * 6 + [0]) == 1
    assert _scan(L, d, [FAKE + 8] + [FAKE] * 6) == 1
    assert _scan(L, d, ws=0) == 3
    assert _scan(L, d, ws=FAKE + 16) == 3
    assert _scan(L, d, ws_bytes=100) == 3
    assert L.dart_chunk_scan(None, *[None] * 10, 0, None) == 1


def test_decode_validation(L):
    from paper_2608_02032_gb300 import binding as B

    d = _dims(seqlen=1)
    v = ctypes.c_void_p
    args = [v(FAKE)] * 12  # state .. lse
    # pos / S beyond the cache capacity
    assert L.dart_decode_step(ctypes.byref(d), 4 * 128, 3, v(FAKE), *args, None, 0, None) == 1
    assert L.dart_decode_step(ctypes.byref(d), -1, 3, v(FAKE), *args, None, 0, None) == 1
    bad = list(args)
    bad[3] = v(FAKE + 4)
    assert L.dart_decode_step(ctypes.byref(d), 5, 3, v(FAKE), *bad, None, 0, None) == 1
    assert B.STATUS_NAMES[1] == "DART_ERR_INVALID_ARG"


def test_prefill_host_validation_and_workspace(L):
    """The host-buffer prefill: its workspace holds the device copies and one head
    group's scan and SMA workspaces; missing buffers or a short workspace are refused
    before any copy or launch."""
    from paper_2608_02032_gb300 import binding as B

    v = ctypes.c_void_p
    d = _dims(nheads=32)  # G = 1, H = 32: eight groups of 4 heads
    need = B.dart_workspace_size(d, B.DART_OP_PREFILL_HOST)
    one = _dims(nheads=4)  # the device sizes of one group of 4 heads
    per_group_inputs = 512 * 4 * 64 * 2
    assert need > 8 * per_group_inputs
    assert need > B.dart_workspace_size(one, B.DART_OP_CHUNK_SCAN)
    assert B.dart_workspace_size(_dims(headdim=48), B.DART_OP_PREFILL_HOST) == 0
    # beyond 64 groups the problem runs as one group (still a valid size)
    assert B.dart_workspace_size(_dims(nheads=1024), B.DART_OP_PREFILL_HOST) > 0
    host = [v(FAKE)] * 9  # X .. Y (never dereferenced: validation fails first)
    assert L.dart_prefill_host(ctypes.byref(d), *host, v(FAKE * 256), need - 256, None) == 3
    assert L.dart_prefill_host(ctypes.byref(d), *host, v(FAKE * 256 + 16), need, None) == 3
    bad = list(host)
    bad[4] = None
    assert L.dart_prefill_host(ctypes.byref(d), *bad, v(FAKE * 256), need, None) == 1
    assert L.dart_prefill_host(ctypes.byref(_dims(chunk=96)), *host, v(FAKE * 256), need, None) == 2


def test_noalloc_rejects_problems_beyond_its_scratch(L):
    """2^20 memory rows is the fixed limit; one more row is refused before any launch."""
    v = ctypes.c_void_p
    ok = _dims(batch=1, seqlen=2 ** 20 // (2 * 128) * 128, nheads=2, chunk=128)  # exactly 2^20 rows
    big = _dims(batch=2, seqlen=2 ** 20 // (2 * 128) * 128, nheads=2, chunk=128)
    assert L.dart_sma_forward_noalloc(ctypes.byref(big), *[v(FAKE)] * 9, None) == 6
    assert L.dart_sma_forward_noalloc(ctypes.byref(ok), *[v(FAKE)] * 6, v(0), v(FAKE), v(FAKE),
                                      None) == 1  # a NULL output is still caught first
    assert L.dart_sma_forward_noalloc(ctypes.byref(_dims(headdim=48)), *[v(FAKE)] * 9, None) == 2
