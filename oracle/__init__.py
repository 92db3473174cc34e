"""Plain CPU oracle for the MoSA layer (arXiv 2505.00315, Sec. 2.1-2.2).

TEST INFRASTRUCTURE ONLY.  Only the test suite, ``__graft_entry__.smoke()``
and the benchmark's CPU-baseline leg may import this package.  The product
library never loads it and shares no code with it.

The arithmetic lives in ``mosa_oracle.c`` (fp64, explicit loops, OpenMP over
independent loops); this module only compiles it with gcc and marshals numpy
arrays through ctypes.  Every function takes and returns float64 arrays in the
paper's row-major layouts:

    X [B,T,d]; W_r [d,H]; W_q, W_k, W_v [H,d,h']; W_o [H,h',d];
    Y, dY, dX [B,T,d]; I [B,H,k] int32 ascending; r_sel [B,H,k]; r_full [B,H,T].

Parity status of each function is recorded beside its pins in
``tests/test_oracle_pins.py``; all of them are pinned.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
# A test may point the oracle at a modified copy of its source (to check that
# the pins catch planted mistakes); that copy's library is built beside it.
_SRC = os.environ.get("MOSA_ORACLE_SRC") or os.path.join(_HERE, "mosa_oracle.c")
_LIB = (os.path.splitext(_SRC)[0] + ".so" if os.environ.get("MOSA_ORACLE_SRC")
        else os.path.join(_HERE, "_build", "liboracle.so"))
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``mosa_oracle.c`` into ``oracle/_build/liboracle.so`` with gcc."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-Wall", "-Wextra",
           "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            d = ctypes.POINTER(ctypes.c_double)
            i32 = ctypes.POINTER(ctypes.c_int32)
            u8 = ctypes.POINTER(ctypes.c_ubyte)
            c_int = ctypes.c_int
            lib.oracle_num_threads.restype = c_int
            lib.oracle_set_num_threads.argtypes = [c_int]
            lib.oracle_router.argtypes = [c_int, c_int, c_int, c_int, d, d, d]
            lib.oracle_topk.argtypes = [c_int, c_int, d, i32, d]
            lib.oracle_topk.restype = c_int
            lib.oracle_topk_first.argtypes = [c_int, c_int, d, i32, d]
            lib.oracle_topk_first.restype = c_int
            lib.oracle_forward.argtypes = [c_int] * 6 + [d] * 6 + [d, i32, d, d, u8, u8, c_int,
                                                                    c_int]
            lib.oracle_forward.restype = c_int
            lib.oracle_forward_indices.argtypes = [c_int] * 6 + [d] * 6 + [i32, d, d, u8, u8, c_int]
            lib.oracle_forward_indices.restype = c_int
            lib.oracle_backward.argtypes = ([c_int] * 6 + [d] * 6 + [i32, d] + [d] * 6 +
                                            [u8, u8, c_int])
            lib.oracle_backward.restype = c_int
            lib.oracle_dense_forward.argtypes = [c_int] * 6 + [d] * 5 + [d, u8, u8, c_int]
            lib.oracle_dense_forward.restype = c_int
            lib.oracle_dense_backward.argtypes = ([c_int] * 6 + [d] * 6 + [d] * 5 +
                                                  [u8, u8, c_int])
            lib.oracle_dense_backward.restype = c_int
            _lib = lib
    return _lib


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _ptr(a: np.ndarray | None, ctype=ctypes.c_double):
    if a is None:
        return None
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def _mask(sel, n):
    if sel is None:
        return None
    m = np.zeros(n, dtype=np.uint8)
    m[np.asarray(sel, dtype=np.int64)] = 1
    return m


def num_threads() -> int:
    """Threads the oracle's OpenMP loops use."""
    return int(_load().oracle_num_threads())


def set_num_threads(n: int) -> None:
    _load().oracle_set_num_threads(int(n))


def _dims(X, Wq):
    B, T, d = X.shape
    H, d2, hp = Wq.shape
    assert d2 == d
    return B, T, d, H, hp


def router(X, Wr) -> np.ndarray:
    """r_full[b,h,t] = sigma(X[b,t,:] . W_r[:,h])  (Sec. 2.2, router)."""
    X, Wr = _f64(X), _f64(Wr)
    B, T, d = X.shape
    H = Wr.shape[1]
    out = np.empty((B, H, T), dtype=np.float64)
    _load().oracle_router(B, T, d, H, _ptr(X), _ptr(Wr), _ptr(out))
    return out


def topk(r_row, k: int, first_token: bool = False):
    """TopK over one row of scores (Sec. 2.2): full sort by (-score, index),
    first k kept, returned in ascending index order with their scores.  With
    ``first_token`` (Sec. 3.2) token 0 is always kept and the other k-1 are the
    TopK of tokens 1..T-1."""
    r_row = _f64(r_row).reshape(-1)
    T = r_row.shape[0]
    I = np.empty(k, dtype=np.int32)
    rs = np.empty(k, dtype=np.float64)
    fn = _load().oracle_topk_first if first_token else _load().oracle_topk
    if fn(T, k, _ptr(r_row), _ptr(I, ctypes.c_int32), _ptr(rs)) != 0:
        raise ValueError("oracle_topk: invalid arguments")
    return I, rs


def forward(X, Wr, Wq, Wk, Wv, Wo, k: int, batches=None, heads=None, first_token=False,
            rope=False):
    """MoSA layer forward (Sec. 2.2, Eq. mosa_mha).  Returns (Y, I, r_sel, r_full).

    ``batches`` / ``heads`` restrict the computed units (b,h); Y[b] is exact
    for a batch whose every head is computed.  ``first_token``: every head
    keeps token 0 and selects k-1 more (Sec. 3.2).  ``rope``: Q and K rotated
    at the tokens' original positions (Sec. 2.2, positional encodings)."""
    X, Wr, Wq, Wk, Wv, Wo = map(_f64, (X, Wr, Wq, Wk, Wv, Wo))
    B, T, d, H, hp = _dims(X, Wq)
    Y = np.zeros((B, T, d))
    I = np.zeros((B, H, k), dtype=np.int32)
    rs = np.zeros((B, H, k))
    rf = np.zeros((B, H, T))
    bm, hm = _mask(batches, B), _mask(heads, H)
    rc = _load().oracle_forward(B, T, d, H, hp, k, _ptr(X), _ptr(Wr), _ptr(Wq), _ptr(Wk),
                                _ptr(Wv), _ptr(Wo), _ptr(Y), _ptr(I, ctypes.c_int32), _ptr(rs),
                                _ptr(rf), _ptr(bm, ctypes.c_ubyte), _ptr(hm, ctypes.c_ubyte),
                                1 if first_token else 0, 1 if rope else 0)
    if rc != 0:
        raise ValueError("oracle_forward failed (bad arguments or out of memory)")
    return Y, I, rs, rf


def forward_indices(X, Wr, Wq, Wk, Wv, Wo, I, r_sel=None, batches=None, heads=None,
                    rope=False):
    """Forward with the token sets I fixed.  If ``r_sel`` is None the scores
    are sigma(X W_r)[I] (TopK held constant); otherwise they are used as given
    (e.g. ones, for the fixed-sparse special case of Sec. 3.1)."""
    X, Wr, Wq, Wk, Wv, Wo = map(_f64, (X, Wr, Wq, Wk, Wv, Wo))
    B, T, d, H, hp = _dims(X, Wq)
    I = np.ascontiguousarray(I, dtype=np.int32)
    k = I.shape[-1]
    rs = None if r_sel is None else _f64(r_sel)
    Y = np.zeros((B, T, d))
    bm, hm = _mask(batches, B), _mask(heads, H)
    rc = _load().oracle_forward_indices(B, T, d, H, hp, k, _ptr(X), _ptr(Wr), _ptr(Wq),
                                        _ptr(Wk), _ptr(Wv), _ptr(Wo),
                                        _ptr(I, ctypes.c_int32), _ptr(rs), _ptr(Y),
                                        _ptr(bm, ctypes.c_ubyte), _ptr(hm, ctypes.c_ubyte),
                                        1 if rope else 0)
    if rc != 0:
        raise ValueError("oracle_forward_indices failed")
    return Y


def backward(X, Wr, Wq, Wk, Wv, Wo, I, dY, batches=None, heads=None, rope=False):
    """Gradients of sum(Y * dY) for the token sets I (TopK held constant).
    Returns a dict with dX, dWr, dWq, dWk, dWv, dWo."""
    X, Wr, Wq, Wk, Wv, Wo, dY = map(_f64, (X, Wr, Wq, Wk, Wv, Wo, dY))
    B, T, d, H, hp = _dims(X, Wq)
    I = np.ascontiguousarray(I, dtype=np.int32)
    k = I.shape[-1]
    g = {"dX": np.zeros((B, T, d)), "dWr": np.zeros((d, H)), "dWq": np.zeros((H, d, hp)),
         "dWk": np.zeros((H, d, hp)), "dWv": np.zeros((H, d, hp)), "dWo": np.zeros((H, hp, d))}
    bm, hm = _mask(batches, B), _mask(heads, H)
    rc = _load().oracle_backward(B, T, d, H, hp, k, _ptr(X), _ptr(Wr), _ptr(Wq), _ptr(Wk),
                                 _ptr(Wv), _ptr(Wo), _ptr(I, ctypes.c_int32), _ptr(dY),
                                 _ptr(g["dX"]), _ptr(g["dWr"]), _ptr(g["dWq"]), _ptr(g["dWk"]),
                                 _ptr(g["dWv"]), _ptr(g["dWo"]), _ptr(bm, ctypes.c_ubyte),
                                 _ptr(hm, ctypes.c_ubyte), 1 if rope else 0)
    if rc != 0:
        raise ValueError("oracle_backward failed")
    return g


def dense_forward(X, Dq, Dk, Dv, Do, window: int = 0, batches=None, heads=None, rope=False):
    """Dense heads of a hybrid layer (Sec. 2.2, hybridization): causal
    multi-head attention over all T tokens (Sec. 2.1, Eq. mha), no router.
    ``window`` > 0: local heads (Sec. 3.4), token i sees token j iff j <= i and
    both lie in the same block of ``window`` positions.  Returns Y [B,T,d]."""
    X, Dq, Dk, Dv, Do = map(_f64, (X, Dq, Dk, Dv, Do))
    B, T, d, H, hp = _dims(X, Dq)
    Y = np.zeros((B, T, d))
    bm, hm = _mask(batches, B), _mask(heads, H)
    rc = _load().oracle_dense_forward(B, T, d, H, hp, int(window), _ptr(X), _ptr(Dq), _ptr(Dk),
                                      _ptr(Dv), _ptr(Do), _ptr(Y), _ptr(bm, ctypes.c_ubyte),
                                      _ptr(hm, ctypes.c_ubyte), 1 if rope else 0)
    if rc != 0:
        raise ValueError("oracle_dense_forward failed")
    return Y


def dense_backward(X, Dq, Dk, Dv, Do, dY, window: int = 0, batches=None, heads=None,
                   rope=False):
    """Gradients of sum(Y * dY) for the dense (or local) heads of
    ``dense_forward``.  Returns a dict with dX, dWq, dWk, dWv, dWo."""
    X, Dq, Dk, Dv, Do, dY = map(_f64, (X, Dq, Dk, Dv, Do, dY))
    B, T, d, H, hp = _dims(X, Dq)
    g = {"dX": np.zeros((B, T, d)), "dWq": np.zeros((H, d, hp)), "dWk": np.zeros((H, d, hp)),
         "dWv": np.zeros((H, d, hp)), "dWo": np.zeros((H, hp, d))}
    bm, hm = _mask(batches, B), _mask(heads, H)
    rc = _load().oracle_dense_backward(B, T, d, H, hp, int(window), _ptr(X), _ptr(Dq), _ptr(Dk),
                                       _ptr(Dv), _ptr(Do), _ptr(dY), _ptr(g["dX"]),
                                       _ptr(g["dWq"]), _ptr(g["dWk"]), _ptr(g["dWv"]),
                                       _ptr(g["dWo"]), _ptr(bm, ctypes.c_ubyte),
                                       _ptr(hm, ctypes.c_ubyte), 1 if rope else 0)
    if rc != 0:
        raise ValueError("oracle_dense_backward failed")
    return g


def hybrid_forward(X, Wr, Wq, Wk, Wv, Wo, Dq, Dk, Dv, Do, k: int, window: int = 0,
                   batches=None, first_token=False, rope=False):
    """Hybrid layer (Sec. 2.2, hybridization): the MoSA heads plus the dense
    (or local) heads, outputs summed as every head's is (Eq. mha).  Returns
    (Y, I, r_sel, r_full) with I, r_sel, r_full those of the MoSA heads."""
    Y, I, rs, rf = forward(X, Wr, Wq, Wk, Wv, Wo, k, batches=batches,
                           first_token=first_token, rope=rope)
    Y = Y + dense_forward(X, Dq, Dk, Dv, Do, window, batches=batches, rope=rope)
    return Y, I, rs, rf


def hybrid_backward(X, Wr, Wq, Wk, Wv, Wo, Dq, Dk, Dv, Do, I, dY, window: int = 0,
                    batches=None, rope=False):
    """Gradients of the hybrid layer: dX summed over both head groups; dWr,
    dWq, dWk, dWv, dWo of the MoSA heads; dDq, dDk, dDv, dDo of the dense
    heads."""
    g = backward(X, Wr, Wq, Wk, Wv, Wo, I, dY, batches=batches, rope=rope)
    gd = dense_backward(X, Dq, Dk, Dv, Do, dY, window, batches=batches, rope=rope)
    g["dX"] = g["dX"] + gd["dX"]
    for n in ("q", "k", "v", "o"):
        g["dD" + n] = gd["dW" + n]
    return g
