"""The C ABI without a GPU: the library builds and loads, exports every
function include/mosa.h declares, and rejects invalid arguments before
touching CUDA (these calls return before any runtime call, so they run on a
machine with no device)."""
import ctypes
import os
import re

import pytest

from paper_2505_00315_gb300 import _binding as B

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "mosa.h")
FAKE = ctypes.c_void_p(0x100000)   # never dereferenced: validation fails first


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mosa_[a-z_]+)\s*\(", text)))


def test_header_and_binding_agree():
    assert declared_functions() == sorted(B.EXPORTED)


def test_library_exports_every_declared_function():
    lib = B.load()
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_status_strings():
    for code in range(6):
        assert B.status_string(code).startswith("MOSA_")
    assert "unknown" in B.status_string(99)


def shape(**kw):
    base = dict(B=2, T=64, d=32, H=3, hp=32, k=8, dtype=B.MOSA_BF16, first_token=0)
    base.update(kw)
    return B.MosaShape(*[base[n] for n in ("B", "T", "d", "H", "hp", "k", "dtype", "first_token")])


@pytest.mark.parametrize("kw,ok", [
    ({}, True), (dict(k=64), True), (dict(k=65), False), (dict(k=0), False),
    (dict(B=0), False), (dict(T=-1), False), (dict(hp=48), False), (dict(d=12), False),
    (dict(dtype=7), False), (dict(T=70000, k=8), False), (dict(hp=128, dtype=B.MOSA_F32), True),
    (dict(first_token=1), True), (dict(first_token=1, k=1), True), (dict(first_token=2), False),
    (dict(first_token=-1), False),
])
def test_workspace_bytes_validates_shape(kw, ok):
    n = B.mosa_workspace_bytes(shape(**kw))
    assert (n > 0) == ok


def test_workspace_grows_with_problem():
    assert B.mosa_workspace_bytes(shape(B=4)) > B.mosa_workspace_bytes(shape(B=2))
    # intermediates take 4 bytes per element for either input dtype
    assert B.mosa_workspace_bytes(shape(dtype=B.MOSA_F32)) == B.mosa_workspace_bytes(shape())


def call_forward(s, ws=FAKE, ws_bytes=1 << 40, null_at=None):
    ptrs = [FAKE] * 10
    if null_at is not None:
        ptrs[null_at] = None
    return B.load().mosa_forward(ctypes.byref(s), *ptrs[:6], ptrs[6], ptrs[7], ptrs[8], None,
                                 ws, ws_bytes, None)


def test_forward_rejects_invalid_shape_and_pointers():
    assert call_forward(shape(k=65)) == B.MOSA_ERR_INVALID_ARG
    assert call_forward(shape(hp=40)) == B.MOSA_ERR_UNSUPPORTED
    for i in range(9):
        assert call_forward(shape(), null_at=i) == B.MOSA_ERR_INVALID_ARG
    assert B.load().mosa_forward(None, *[FAKE] * 9, None, FAKE, 1 << 40, None) == \
        B.MOSA_ERR_INVALID_ARG


def test_forward_rejects_bad_workspace():
    s = shape()
    need = B.mosa_workspace_bytes(s)
    assert call_forward(s, ws=None) == B.MOSA_ERR_WORKSPACE
    assert call_forward(s, ws=ctypes.c_void_p(0x100010)) == B.MOSA_ERR_WORKSPACE  # misaligned
    assert call_forward(s, ws_bytes=need - 1) == B.MOSA_ERR_WORKSPACE


def test_backward_and_indices_entry_reject_before_launch():
    L = B.load()
    s = shape()
    args = [FAKE] * 15
    assert L.mosa_backward(ctypes.byref(shape(k=100)), *args, FAKE, 1 << 40, None) == \
        B.MOSA_ERR_INVALID_ARG
    args[9] = None   # dY
    assert L.mosa_backward(ctypes.byref(s), *args, FAKE, 1 << 40, None) == B.MOSA_ERR_INVALID_ARG
    assert L.mosa_backward(ctypes.byref(s), *[FAKE] * 15, None, 1 << 40, None) == \
        B.MOSA_ERR_WORKSPACE
    assert L.mosa_forward_with_indices(ctypes.byref(s), *[FAKE] * 7, None, FAKE, 1 << 40,
                                       None) == B.MOSA_ERR_INVALID_ARG


def test_topk_rejects_bad_sizes():
    L = B.load()
    assert L.mosa_topk(4, 10, 11, FAKE, FAKE, FAKE, None) == B.MOSA_ERR_INVALID_ARG
    assert L.mosa_topk(0, 10, 1, FAKE, FAKE, FAKE, None) == B.MOSA_ERR_INVALID_ARG
    assert L.mosa_topk(4, 10, 3, None, FAKE, FAKE, None) == B.MOSA_ERR_INVALID_ARG
    assert L.mosa_topk(1, 70000, 3, FAKE, FAKE, FAKE, None) == B.MOSA_ERR_UNSUPPORTED


def test_check_status_rejects_bad_arguments():
    L = B.load()
    assert L.mosa_check_status(ctypes.byref(shape(k=0)), FAKE, None) == B.MOSA_ERR_INVALID_ARG
    assert L.mosa_check_status(ctypes.byref(shape()), None, None) == B.MOSA_ERR_WORKSPACE


@pytest.mark.parametrize("T,rho,k", [
    # Sec. 3.5: k = max(floor(T / rho), 2); a 10-token input at rho = 64 keeps 2
    (10, 64, 2), (1024, 8, 128), (1024, 64, 16), (130, 64, 2), (191, 64, 2), (192, 64, 3),
    (8192, 32, 256),
    # at most T tokens exist; no k for an empty input or rho < 1
    (1, 64, 1), (2, 64, 2), (0, 8, 0), (100, 0, 0),
])
def test_adaptive_k(T, rho, k):
    assert B.mosa_adaptive_k(T, rho) == k


def hshape(H_dense=2, window=0, **kw):
    return B.MosaHybridShape(shape(**kw), H_dense, window)


@pytest.mark.parametrize("H_dense,window,kw,ok", [
    (2, 0, {}, True), (2, 16, {}, True), (2, 64, {}, True), (0, 0, {}, True), (1, 1, {}, True),
    (2, 24, {}, False),              # local blocks must tile the sequence
    (2, 65, {}, False), (2, -1, {}, False), (-1, 0, {}, False),
    (2, 0, dict(k=65), False), (2, 0, dict(hp=48), False), (2, 0, dict(first_token=1), True),
])
def test_hybrid_workspace_bytes_validates_shape(H_dense, window, kw, ok):
    assert (B.mosa_hybrid_workspace_bytes(hshape(H_dense, window, **kw)) > 0) == ok


def test_hybrid_workspace_holds_both_head_groups():
    s = shape()
    sparse = B.mosa_workspace_bytes(s)
    assert B.mosa_hybrid_workspace_bytes(hshape(0)) == sparse
    dense = B.mosa_hybrid_workspace_bytes(hshape(2))
    assert dense > sparse
    assert B.mosa_hybrid_workspace_bytes(hshape(4)) > dense
    assert B.mosa_hybrid_workspace_bytes(hshape(2, window=64)) == dense   # w = T is dense
    # local heads keep every token too, in blocks: no fewer rows than dense heads
    assert B.mosa_hybrid_workspace_bytes(hshape(2, window=16)) > sparse


def test_hybrid_entries_reject_before_launch():
    L = B.load()
    fwd = [FAKE] * 14            # X, W_r, W_q..W_o, D_q..D_o, Y, I, r_sel, r_full
    assert L.mosa_hybrid_forward(ctypes.byref(hshape(window=24)), *fwd, FAKE, 1 << 40, None) \
        == B.MOSA_ERR_UNSUPPORTED
    assert L.mosa_hybrid_forward(None, *fwd, FAKE, 1 << 40, None) == B.MOSA_ERR_INVALID_ARG
    for i in range(13):
        a = list(fwd)
        a[i] = None
        assert L.mosa_hybrid_forward(ctypes.byref(hshape()), *a, FAKE, 1 << 40, None) == \
            B.MOSA_ERR_INVALID_ARG, i
    # without dense heads their weights may be NULL: validation reaches the workspace
    a = list(fwd)
    a[6:10] = [None] * 4
    assert L.mosa_hybrid_forward(ctypes.byref(hshape(0)), *a, None, 1 << 40, None) == \
        B.MOSA_ERR_WORKSPACE
    need = B.mosa_hybrid_workspace_bytes(hshape())
    assert L.mosa_hybrid_forward(ctypes.byref(hshape()), *fwd, FAKE, need - 1, None) == \
        B.MOSA_ERR_WORKSPACE
    bwd = [FAKE] * 23            # ..., I, r_sel, dY, dX, dW_r..dW_o, dD_q..dD_o
    for i in range(23):
        a = list(bwd)
        a[i] = None
        assert L.mosa_hybrid_backward(ctypes.byref(hshape()), *a, FAKE, 1 << 40, None) == \
            B.MOSA_ERR_INVALID_ARG, i
    assert L.mosa_hybrid_backward(ctypes.byref(hshape()), *bwd, None, 1 << 40, None) == \
        B.MOSA_ERR_WORKSPACE


def test_timeline_mode_switch_validates_its_argument():
    lib = B.load()
    assert lib.mosa_profile_timeline(2) == B.MOSA_ERR_INVALID_ARG
    assert lib.mosa_profile_timeline(-1) == B.MOSA_ERR_INVALID_ARG
    assert lib.mosa_profile_timeline(1) == B.MOSA_OK
    assert lib.mosa_profile_timeline(0) == B.MOSA_OK
    start = (ctypes.c_double * 16)()
    end = (ctypes.c_double * 16)()
    s = shape()
    # invalid pointers are rejected before any CUDA call
    assert lib.mosa_profile_timeline_read(ctypes.byref(s), None, start, end, 16) == 0
    assert lib.mosa_profile_timeline_read(None, FAKE, start, end, 16) == 0
