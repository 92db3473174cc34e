"""ctypes binding of libmosa (include/mosa.h).

Argument marshalling only: every step of the layer runs in the library's
CUDA kernels.  Torch supplies device memory and the current stream.  There
is no fallback: if the library cannot be built or loaded, or no CUDA device
is present, the calls raise.
"""
from __future__ import annotations

import ctypes
import os
import threading

from . import build as _build

MOSA_OK = 0
MOSA_ERR_INVALID_ARG = 1
MOSA_ERR_UNSUPPORTED = 2
MOSA_ERR_CUDA = 3
MOSA_ERR_DEVICE_TIMEOUT = 4
MOSA_ERR_WORKSPACE = 5
MOSA_ERR_RANGE = 6
MOSA_F32 = 0
MOSA_BF16 = 1

#: Every function include/mosa.h declares.
EXPORTED = ("mosa_status_string", "mosa_workspace_bytes", "mosa_forward",
            "mosa_forward_with_indices", "mosa_backward", "mosa_topk", "mosa_check_status",
            "mosa_kernel_launches", "mosa_profile_stages", "mosa_profile_read",
            "mosa_stage_name", "mosa_stage_engine", "mosa_route_noalloc", "mosa_adaptive_k",
            "mosa_hybrid_workspace_bytes", "mosa_hybrid_forward", "mosa_hybrid_backward",
            "mosa_profile_spans", "mosa_profile_timeline", "mosa_profile_timeline_read",
            "mosa_profile_spans_copy")


class MosaShape(ctypes.Structure):
    """mosa_shape: B sequences of T tokens of width d, H heads of size hp, k
    tokens per head, storage dtype (MOSA_F32 or MOSA_BF16), first_token (1:
    every head keeps token 0 and selects k-1 more, Sec. 3.2)."""
    _fields_ = [("B", ctypes.c_int32), ("T", ctypes.c_int32), ("d", ctypes.c_int32),
                ("H", ctypes.c_int32), ("hp", ctypes.c_int32), ("k", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("first_token", ctypes.c_int32),
                ("rope", ctypes.c_int32)]

    def astuple(self):
        return (self.B, self.T, self.d, self.H, self.hp, self.k, self.dtype, self.first_token,
                self.rope)


class MosaHybridShape(ctypes.Structure):
    """mosa_hybrid_shape: the MoSA heads' shape plus H_dense dense heads
    (window = 0) or local heads attending within blocks of ``window`` tokens
    (Sec. 2.2 hybridization, Sec. 3.4)."""
    _fields_ = [("sparse", MosaShape), ("H_dense", ctypes.c_int32), ("window", ctypes.c_int32)]


class MosaError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {status_string(code)}")


_lock = threading.Lock()
_lib = None


def lib_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load libmosa.so (building it first if needed) and declare signatures."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.build() if build_if_missing else _build.LIB
        if not os.path.exists(path):
            raise RuntimeError(f"libmosa is not built ({path}); run paper_2505_00315_gb300.build")
        L = ctypes.CDLL(path)
        vp, sz, i32 = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int32
        sp = ctypes.POINTER(MosaShape)
        L.mosa_status_string.argtypes = [ctypes.c_int]
        L.mosa_status_string.restype = ctypes.c_char_p
        L.mosa_workspace_bytes.argtypes = [sp]
        L.mosa_workspace_bytes.restype = sz
        L.mosa_forward.argtypes = [sp] + [vp] * 6 + [vp] * 4 + [vp, sz, vp]
        L.mosa_forward.restype = ctypes.c_int
        L.mosa_forward_with_indices.argtypes = [sp] + [vp] * 5 + [vp, vp, vp] + [vp, sz, vp]
        L.mosa_forward_with_indices.restype = ctypes.c_int
        L.mosa_backward.argtypes = [sp] + [vp] * 6 + [vp, vp, vp] + [vp] * 6 + [vp, sz, vp]
        L.mosa_backward.restype = ctypes.c_int
        L.mosa_topk.argtypes = [i32, i32, i32, vp, vp, vp, vp]
        L.mosa_topk.restype = ctypes.c_int
        L.mosa_check_status.argtypes = [sp, vp, vp]
        L.mosa_check_status.restype = ctypes.c_int
        L.mosa_kernel_launches.argtypes = []
        L.mosa_kernel_launches.restype = ctypes.c_ulonglong
        L.mosa_profile_stages.argtypes = [ctypes.c_uint32]
        L.mosa_profile_stages.restype = ctypes.c_int
        L.mosa_profile_read.argtypes = [ctypes.POINTER(ctypes.c_double),
                                        ctypes.POINTER(ctypes.c_int32), i32]
        L.mosa_profile_read.restype = i32
        L.mosa_profile_spans.argtypes = [sp, vp, ctypes.POINTER(ctypes.c_double), i32]
        L.mosa_profile_spans.restype = i32
        L.mosa_profile_spans_copy.argtypes = [sp, vp, vp, vp]
        L.mosa_profile_spans_copy.restype = ctypes.c_int
        L.mosa_profile_timeline.argtypes = [i32]
        L.mosa_profile_timeline.restype = ctypes.c_int
        L.mosa_profile_timeline_read.argtypes = [sp, vp, ctypes.POINTER(ctypes.c_double),
                                                 ctypes.POINTER(ctypes.c_double), i32]
        L.mosa_profile_timeline_read.restype = i32
        L.mosa_stage_name.argtypes = [i32]
        L.mosa_stage_name.restype = ctypes.c_char_p
        L.mosa_route_noalloc.argtypes = [sp, vp, vp, vp, vp, vp]
        L.mosa_route_noalloc.restype = ctypes.c_int
        L.mosa_stage_engine.argtypes = [sp, i32]
        L.mosa_stage_engine.restype = i32
        L.mosa_adaptive_k.argtypes = [i32, i32]
        L.mosa_adaptive_k.restype = i32
        hp_ = ctypes.POINTER(MosaHybridShape)
        L.mosa_hybrid_workspace_bytes.argtypes = [hp_]
        L.mosa_hybrid_workspace_bytes.restype = sz
        L.mosa_hybrid_forward.argtypes = [hp_] + [vp] * 10 + [vp] * 4 + [vp, sz, vp]
        L.mosa_hybrid_forward.restype = ctypes.c_int
        L.mosa_hybrid_backward.argtypes = [hp_] + [vp] * 10 + [vp, vp, vp] + [vp] * 10 + [vp, sz, vp]
        L.mosa_hybrid_backward.restype = ctypes.c_int
        _lib = L
        return L


def status_string(code: int) -> str:
    return load().mosa_status_string(int(code)).decode()


def _check(code: int, where: str) -> None:
    if code != MOSA_OK:
        raise MosaError(code, where)


# ---------------------------------------------------------------- torch glue

def _torch():
    import torch
    return torch


def _dtype_code(t) -> int:
    torch = _torch()
    if t.dtype == torch.float32:
        return MOSA_F32
    if t.dtype == torch.bfloat16:
        return MOSA_BF16
    raise TypeError(f"unsupported storage dtype {t.dtype} (float32 or bfloat16)")


def _dev(t, name: str, dtype=None):
    torch = _torch()
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor (libmosa runs on the GPU only)")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    torch = _torch()
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def make_shape(X, W_q, k: int, first_token: bool = False, rope: bool = False) -> MosaShape:
    B, T, d = X.shape
    H, d2, hp = W_q.shape
    if d2 != d:
        raise ValueError("W_q must be [H, d, hp] with the d of X")
    return MosaShape(B, T, d, H, hp, int(k), _dtype_code(X), 1 if first_token else 0,
                     1 if rope else 0)


def mosa_adaptive_k(T: int, rho: int) -> int:
    """Tokens per head for a T-token input at sparsity rho (Sec. 3.5):
    max(floor(T / rho), 2), at most T; 0 for T < 1 or rho < 1."""
    return int(load().mosa_adaptive_k(int(T), int(rho)))


def mosa_workspace_bytes(shape: MosaShape) -> int:
    return int(load().mosa_workspace_bytes(ctypes.byref(shape)))


def alloc_workspace(shape: MosaShape, device=None):
    """A torch uint8 device buffer of mosa_workspace_bytes(shape) bytes."""
    torch = _torch()
    n = mosa_workspace_bytes(shape)
    if n == 0:
        raise MosaError(MOSA_ERR_INVALID_ARG, "mosa_workspace_bytes")
    return torch.empty(n, dtype=torch.uint8, device=device or "cuda")


def _same(ref, *ts):
    for name, t in ts:
        if t.dtype != ref.dtype:
            raise TypeError(f"{name} must have the storage dtype {ref.dtype}")


def _shapes(**named):
    """Check each tensor's shape: name=(tensor, expected shape).  The library
    sees plain pointers, so a wrong shape here would mean out-of-range
    accesses there; None tensors are skipped."""
    for name, (t, want) in named.items():
        if t is not None and tuple(t.shape) != tuple(want):
            raise ValueError(f"{name} must have shape {tuple(want)}, got {tuple(t.shape)}")


def _layer_shapes(X, W_r, W_q, W_k, W_v, W_o, k=None, I=None, r_sel=None, dY=None):
    """Shapes of the layer's inputs against X [B,T,d] and W_q [H,d,hp]."""
    if X.dim() != 3 or W_q.dim() != 3:
        raise ValueError("X must be [B, T, d] and W_q [H, d, hp]")
    B, T, d = X.shape
    H, _, hp = W_q.shape
    _shapes(W_q=(W_q, (H, d, hp)), W_r=(W_r, (d, H)), W_k=(W_k, (H, d, hp)),
            W_v=(W_v, (H, d, hp)), W_o=(W_o, (H, hp, d)), dY=(dY, (B, T, d)))
    if k is not None:
        _shapes(I=(I, (B, H, k)), r_sel=(r_sel, (B, H, k)))
    return B, T, d, H, hp


def mosa_forward(X, W_r, W_q, W_k, W_v, W_o, k: int, workspace=None, want_r_full=False,
                 out=None, stream=None, first_token: bool = False, rope: bool = False):
    """Forward pass (Sec. 2.2).  Returns (Y, I, r_sel, r_full or None, workspace).

    ``out`` may hold preallocated "Y", "I", "r_sel" (and "r_full") tensors.
    With ``first_token`` every head keeps token 0 and selects k-1 more
    (Sec. 3.2); with ``rope`` Q and K are rotated at the tokens' original
    positions (Sec. 2.2), and the backward must be given ``rope`` too."""
    torch = _torch()
    _layer_shapes(X, W_r, W_q, W_k, W_v, W_o)
    shape = make_shape(X, W_q, k, first_token, rope)
    _same(X, ("W_r", W_r), ("W_q", W_q), ("W_k", W_k), ("W_v", W_v), ("W_o", W_o))
    B, T, d, H = shape.B, shape.T, shape.d, shape.H
    dev = X.device
    out = out or {}
    _shapes(Y=(out.get("Y"), (B, T, d)), I=(out.get("I"), (B, H, k)),
            r_sel=(out.get("r_sel"), (B, H, k)), r_full=(out.get("r_full"), (B, H, T)))
    Y = out.get("Y") if out.get("Y") is not None else torch.empty((B, T, d), dtype=torch.float32, device=dev)
    I = out.get("I") if out.get("I") is not None else torch.empty((B, H, k), dtype=torch.int32, device=dev)
    rs = out.get("r_sel") if out.get("r_sel") is not None else torch.empty((B, H, k), dtype=torch.float32, device=dev)
    rf = None
    if want_r_full:
        rf = out.get("r_full") if out.get("r_full") is not None else torch.empty((B, H, T), dtype=torch.float32, device=dev)
    if workspace is None:
        workspace = alloc_workspace(shape, dev)
    rc = load().mosa_forward(ctypes.byref(shape), _dev(X, "X"), _dev(W_r, "W_r"), _dev(W_q, "W_q"),
                             _dev(W_k, "W_k"), _dev(W_v, "W_v"), _dev(W_o, "W_o"),
                             _dev(Y, "Y", torch.float32), _dev(I, "I", torch.int32),
                             _dev(rs, "r_sel", torch.float32),
                             None if rf is None else _dev(rf, "r_full", torch.float32),
                             _dev(workspace, "workspace"), workspace.numel(), _stream(stream))
    _check(rc, "mosa_forward")
    return Y, I, rs, rf, workspace


def mosa_forward_with_indices(X, W_q, W_k, W_v, W_o, I, r_sel, workspace=None, out=None,
                              stream=None, rope: bool = False):
    """Forward with caller-chosen token sets (e.g. the fixed-sparse case of
    Sec. 3.1).  Returns (Y, workspace)."""
    torch = _torch()
    B_, T_, d_, H_, _ = _layer_shapes(X, None, W_q, W_k, W_v, W_o, k=I.shape[-1], I=I,
                                      r_sel=r_sel)
    _shapes(Y=((out or {}).get("Y"), (B_, T_, d_)))
    shape = make_shape(X, W_q, I.shape[-1], rope=rope)
    _same(X, ("W_q", W_q), ("W_k", W_k), ("W_v", W_v), ("W_o", W_o))
    B, T, d = shape.B, shape.T, shape.d
    Y = (out or {}).get("Y")
    if Y is None:
        Y = torch.empty((B, T, d), dtype=torch.float32, device=X.device)
    if workspace is None:
        workspace = alloc_workspace(shape, X.device)
    rc = load().mosa_forward_with_indices(
        ctypes.byref(shape), _dev(X, "X"), _dev(W_q, "W_q"), _dev(W_k, "W_k"), _dev(W_v, "W_v"),
        _dev(W_o, "W_o"), _dev(I, "I", torch.int32), _dev(r_sel, "r_sel", torch.float32),
        _dev(Y, "Y", torch.float32), _dev(workspace, "workspace"), workspace.numel(),
        _stream(stream))
    _check(rc, "mosa_forward_with_indices")
    return Y, workspace


def mosa_backward(X, W_r, W_q, W_k, W_v, W_o, I, r_sel, dY, workspace, out=None, stream=None,
                  rope: bool = False):
    """Backward pass; returns a dict with dX, dW_r, dW_q, dW_k, dW_v, dW_o (fp32).
    ``rope`` must match the forward's."""
    torch = _torch()
    _layer_shapes(X, W_r, W_q, W_k, W_v, W_o, k=I.shape[-1], I=I, r_sel=r_sel, dY=dY)
    shape = make_shape(X, W_q, I.shape[-1], rope=rope)
    _same(X, ("W_r", W_r), ("W_q", W_q), ("W_k", W_k), ("W_v", W_v), ("W_o", W_o), ("dY", dY))
    dev = X.device
    g = dict(out or {})
    f32 = torch.float32
    for name, like in (("dX", X), ("dW_r", W_r), ("dW_q", W_q), ("dW_k", W_k), ("dW_v", W_v),
                       ("dW_o", W_o)):
        if g.get(name) is None:
            g[name] = torch.empty(like.shape, dtype=f32, device=dev)
        else:
            _shapes(**{name: (g[name], like.shape)})
    rc = load().mosa_backward(
        ctypes.byref(shape), _dev(X, "X"), _dev(W_r, "W_r"), _dev(W_q, "W_q"), _dev(W_k, "W_k"),
        _dev(W_v, "W_v"), _dev(W_o, "W_o"), _dev(I, "I", torch.int32),
        _dev(r_sel, "r_sel", f32), _dev(dY, "dY"), _dev(g["dX"], "dX", f32),
        _dev(g["dW_r"], "dW_r", f32), _dev(g["dW_q"], "dW_q", f32), _dev(g["dW_k"], "dW_k", f32),
        _dev(g["dW_v"], "dW_v", f32), _dev(g["dW_o"], "dW_o", f32),
        _dev(workspace, "workspace"), workspace.numel(), _stream(stream))
    _check(rc, "mosa_backward")
    return g


def mosa_topk(scores, k: int, out=None, stream=None):
    """TopK alone over the last dim of fp32 ``scores`` [..., T]; returns (I, r_sel)."""
    torch = _torch()
    T = scores.shape[-1]
    rows = scores.numel() // T if T else 0
    lead = tuple(scores.shape[:-1])
    I = (out or {}).get("I")
    rs = (out or {}).get("r_sel")
    if I is None:
        I = torch.empty(lead + (k,), dtype=torch.int32, device=scores.device)
    if rs is None:
        rs = torch.empty(lead + (k,), dtype=torch.float32, device=scores.device)
    _shapes(I=(I, lead + (k,)), r_sel=(rs, lead + (k,)))
    rc = load().mosa_topk(rows, T, int(k), _dev(scores, "scores", torch.float32),
                          _dev(I, "I", torch.int32), _dev(rs, "r_sel", torch.float32),
                          _stream(stream))
    _check(rc, "mosa_topk")
    return I, rs


def mosa_check_status(shape: MosaShape, workspace, stream=None) -> int:
    """Synchronizes the stream, returns and clears the device status code."""
    return int(load().mosa_check_status(ctypes.byref(shape), _dev(workspace, "workspace"),
                                        _stream(stream)))


# ------------------------------------------------------------ measurement

def mosa_kernel_launches() -> int:
    """Kernels the library has launched since it was loaded."""
    return int(load().mosa_kernel_launches())


def mosa_profile_stages(mask: int) -> None:
    """Turn CUDA-event timing on for the stages in ``mask`` (0 = off)."""
    _check(load().mosa_profile_stages(int(mask)), "mosa_profile_stages")


def mosa_stage_name(stage: int) -> str:
    return load().mosa_stage_name(int(stage)).decode()


def mosa_profile_read() -> dict:
    """{stage name: (total ms, timed launches)} since the last read; resets."""
    L = load()
    n = 16
    ms = (ctypes.c_double * n)()
    cnt = (ctypes.c_int32 * n)()
    m = L.mosa_profile_read(ms, cnt, n)
    return {mosa_stage_name(i): (ms[i], cnt[i]) for i in range(min(m, n))}


def mosa_profile_spans(shape: MosaShape, workspace) -> dict:
    """{stage name: ms} from the first CTA start to the last CTA end of each
    stage's kernels in the last layer call with ``workspace`` (only stages
    timed with mosa_profile_stages; -1 where none recorded).  Waits for the
    device."""
    L = load()
    n = 16
    ms = (ctypes.c_double * n)()
    m = L.mosa_profile_spans(ctypes.byref(shape), ctypes.c_void_p(workspace.data_ptr()), ms, n)
    return {mosa_stage_name(i): ms[i] for i in range(min(m, n))}


def mosa_profile_spans_copy(shape: MosaShape, workspace, dst) -> None:
    """Enqueue on the current stream a copy of the workspace's 32 kernel-span
    slots (int64 [start, end] per stage) into the device tensor ``dst``
    (at least 32 int64); no wait."""
    torch = _torch()
    if dst.dtype != torch.int64 or dst.numel() < 32 or not dst.is_cuda or not dst.is_contiguous():
        raise ValueError("dst must be a contiguous CUDA int64 tensor of at least 32 elements")
    _check(load().mosa_profile_spans_copy(ctypes.byref(shape), ctypes.c_void_p(workspace.data_ptr()),
                                          ctypes.c_void_p(dst.data_ptr()),
                                          ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)),
           "mosa_profile_spans_copy")


def mosa_profile_timeline(on: bool) -> None:
    """Timeline mode: later layer calls record every stage's kernel span
    (first CTA start, last CTA end) without per-stage events or resets."""
    _check(load().mosa_profile_timeline(1 if on else 0), "mosa_profile_timeline")


def mosa_profile_timeline_read(shape: MosaShape, workspace) -> dict:
    """{stage name: (start us, end us)} of the last forward and backward calls
    with ``workspace`` in timeline mode, from the earliest recorded start;
    stages without a record are left out.  Waits for the device."""
    L = load()
    n = 16
    a = (ctypes.c_double * n)()
    b = (ctypes.c_double * n)()
    m = L.mosa_profile_timeline_read(ctypes.byref(shape), ctypes.c_void_p(workspace.data_ptr()),
                                     a, b, n)
    return {mosa_stage_name(i): (a[i], b[i]) for i in range(min(m, n)) if a[i] >= 0}


_ENGINES = {0: "simt", 1: "tensor", 2: "mem"}


def mosa_stage_engine(shape: MosaShape, stage: int) -> int:
    return int(load().mosa_stage_engine(ctypes.byref(shape), int(stage)))


def stage_impl(shape: MosaShape) -> dict:
    """{stage name: "simt" | "tensor" | "mem"} for this shape."""
    out = {}
    for i in range(32):
        if mosa_stage_name(i) == "unknown":
            break
        e = mosa_stage_engine(shape, i)
        if e >= 0:
            out[mosa_stage_name(i)] = _ENGINES[e]
    return out


def mosa_route_noalloc(X, W_r, k: int, hp: int = 64, out=None, stream=None,
                       first_token: bool = False):
    """Router + TopK with no workspace (the library's own 4 MiB score array);
    returns (I, r_sel).  For callers that cannot allocate device memory; the
    output tensors may be passed preallocated in ``out``."""
    torch = _torch()
    B, T, d = X.shape
    H = W_r.shape[1]
    shape = MosaShape(B, T, d, H, int(hp), int(k), _dtype_code(X), 1 if first_token else 0)
    _same(X, ("W_r", W_r))
    _shapes(W_r=(W_r, (d, H)))
    I = (out or {}).get("I")
    rs = (out or {}).get("r_sel")
    if I is None:
        I = torch.empty((B, H, k), dtype=torch.int32, device=X.device)
    if rs is None:
        rs = torch.empty((B, H, k), dtype=torch.float32, device=X.device)
    _shapes(I=(I, (B, H, k)), r_sel=(rs, (B, H, k)))
    rc = load().mosa_route_noalloc(ctypes.byref(shape), _dev(X, "X"), _dev(W_r, "W_r"),
                                   _dev(I, "I", torch.int32), _dev(rs, "r_sel", torch.float32),
                                   _stream(stream))
    _check(rc, "mosa_route_noalloc")
    return I, rs


# ------------------------------------------------------------ hybrid layers

def _hybrid_shapes(X, W_r, W_q, W_k, W_v, W_o, D_q, D_k, D_v, D_o, **kw):
    """Shapes of a hybrid call: the MoSA heads' as _layer_shapes, and the dense
    heads' D_q, D_k, D_v [H_dense, d, hp], D_o [H_dense, hp, d]."""
    B, T, d, H, hp = _layer_shapes(X, W_r, W_q, W_k, W_v, W_o, **kw)
    if D_q.dim() != 3:
        raise ValueError("D_q must be [H_dense, d, hp]")
    Hd = D_q.shape[0]
    _shapes(D_q=(D_q, (Hd, d, hp)), D_k=(D_k, (Hd, d, hp)), D_v=(D_v, (Hd, d, hp)),
            D_o=(D_o, (Hd, hp, d)))


def make_hybrid_shape(X, W_q, k: int, H_dense: int, window: int = 0,
                      first_token: bool = False, rope: bool = False) -> MosaHybridShape:
    return MosaHybridShape(make_shape(X, W_q, k, first_token, rope), int(H_dense), int(window))


def mosa_hybrid_workspace_bytes(shape: MosaHybridShape) -> int:
    return int(load().mosa_hybrid_workspace_bytes(ctypes.byref(shape)))


def alloc_hybrid_workspace(shape: MosaHybridShape, device=None):
    """A torch uint8 device buffer of mosa_hybrid_workspace_bytes(shape) bytes."""
    torch = _torch()
    n = mosa_hybrid_workspace_bytes(shape)
    if n == 0:
        raise MosaError(MOSA_ERR_INVALID_ARG, "mosa_hybrid_workspace_bytes")
    return torch.empty(n, dtype=torch.uint8, device=device or "cuda")


def mosa_hybrid_forward(X, W_r, W_q, W_k, W_v, W_o, D_q, D_k, D_v, D_o, k: int,
                        window: int = 0, workspace=None, out=None, stream=None,
                        first_token: bool = False, rope: bool = False):
    """Hybrid layer forward (Sec. 2.2 hybridization, Sec. 3.4): the MoSA heads
    plus the dense heads D_q, D_k, D_v [H_dense,d,hp], D_o [H_dense,hp,d]
    (local heads with ``window`` > 0), summed into Y.  Returns
    (Y, I, r_sel, workspace)."""
    torch = _torch()
    _hybrid_shapes(X, W_r, W_q, W_k, W_v, W_o, D_q, D_k, D_v, D_o)
    shape = make_hybrid_shape(X, W_q, k, D_q.shape[0], window, first_token, rope)
    _same(X, ("W_r", W_r), ("W_q", W_q), ("W_k", W_k), ("W_v", W_v), ("W_o", W_o),
          ("D_q", D_q), ("D_k", D_k), ("D_v", D_v), ("D_o", D_o))
    B, T, d, H = X.shape[0], X.shape[1], X.shape[2], W_q.shape[0]
    dev = X.device
    out = out or {}
    _shapes(Y=(out.get("Y"), (B, T, d)), I=(out.get("I"), (B, H, k)),
            r_sel=(out.get("r_sel"), (B, H, k)))
    Y = out.get("Y") if out.get("Y") is not None else torch.empty((B, T, d), dtype=torch.float32, device=dev)
    I = out.get("I") if out.get("I") is not None else torch.empty((B, H, k), dtype=torch.int32, device=dev)
    rs = out.get("r_sel") if out.get("r_sel") is not None else torch.empty((B, H, k), dtype=torch.float32, device=dev)
    if workspace is None:
        workspace = alloc_hybrid_workspace(shape, dev)
    rc = load().mosa_hybrid_forward(
        ctypes.byref(shape), _dev(X, "X"), _dev(W_r, "W_r"), _dev(W_q, "W_q"), _dev(W_k, "W_k"),
        _dev(W_v, "W_v"), _dev(W_o, "W_o"), _dev(D_q, "D_q"), _dev(D_k, "D_k"), _dev(D_v, "D_v"),
        _dev(D_o, "D_o"), _dev(Y, "Y", torch.float32), _dev(I, "I", torch.int32),
        _dev(rs, "r_sel", torch.float32), None, _dev(workspace, "workspace"), workspace.numel(),
        _stream(stream))
    _check(rc, "mosa_hybrid_forward")
    return Y, I, rs, workspace


def mosa_hybrid_backward(X, W_r, W_q, W_k, W_v, W_o, D_q, D_k, D_v, D_o, I, r_sel, dY,
                         workspace, window: int = 0, out=None, stream=None,
                         rope: bool = False):
    """Hybrid layer backward; returns a dict with dX (both head groups),
    dW_r, dW_q, dW_k, dW_v, dW_o (MoSA heads) and dD_q, dD_k, dD_v, dD_o
    (dense heads), fp32.  ``window`` and ``rope`` must match the forward's."""
    torch = _torch()
    _hybrid_shapes(X, W_r, W_q, W_k, W_v, W_o, D_q, D_k, D_v, D_o, k=I.shape[-1], I=I,
                   r_sel=r_sel, dY=dY)
    shape = make_hybrid_shape(X, W_q, I.shape[-1], D_q.shape[0], window, rope=rope)
    _same(X, ("W_r", W_r), ("W_q", W_q), ("W_k", W_k), ("W_v", W_v), ("W_o", W_o),
          ("D_q", D_q), ("D_k", D_k), ("D_v", D_v), ("D_o", D_o), ("dY", dY))
    dev = X.device
    g = dict(out or {})
    f32 = torch.float32
    for name, like in (("dX", X), ("dW_r", W_r), ("dW_q", W_q), ("dW_k", W_k), ("dW_v", W_v),
                       ("dW_o", W_o), ("dD_q", D_q), ("dD_k", D_k), ("dD_v", D_v),
                       ("dD_o", D_o)):
        if g.get(name) is None:
            g[name] = torch.empty(like.shape, dtype=f32, device=dev)
        else:
            _shapes(**{name: (g[name], like.shape)})
    grads = [_dev(g[n], n, f32) for n in ("dX", "dW_r", "dW_q", "dW_k", "dW_v", "dW_o", "dD_q",
                                          "dD_k", "dD_v", "dD_o")]
    rc = load().mosa_hybrid_backward(
        ctypes.byref(shape), _dev(X, "X"), _dev(W_r, "W_r"), _dev(W_q, "W_q"), _dev(W_k, "W_k"),
        _dev(W_v, "W_v"), _dev(W_o, "W_o"), _dev(D_q, "D_q"), _dev(D_k, "D_k"), _dev(D_v, "D_v"),
        _dev(D_o, "D_o"), _dev(I, "I", torch.int32), _dev(r_sel, "r_sel", f32), _dev(dY, "dY"),
        *grads, _dev(workspace, "workspace"), workspace.numel(), _stream(stream))
    _check(rc, "mosa_hybrid_backward")
    return g
