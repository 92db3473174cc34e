"""Seeded synthetic MoSA workloads shared by the tests, the oracle checks and
the benchmark.

This module draws random inputs and nothing else: it holds none of the
layer's arithmetic (no sigmoid, no attention; logits are ranked only to plant
the router margin described below, never to choose the layer's tokens), so
the CPU oracle and the CUDA library can both be fed from it without sharing
code.

Shapes follow the paper's language-model workloads (Sec. 3, implementation
details: T=1024, hidden sizes 512/1024, head size 64; Sec. 3.4: T up to 8192
with hidden size 1024).  C4 text, the tokenizer and trained weights are not
used: activations and weights are Gaussian stand-ins.

Planted router margin.  Bit-exact comparison of the selected indices needs a
clear gap between the k-th and (k+1)-th router score of every (batch, head)
row.  With i.i.d. Gaussian inputs the expected gap at these sizes is below
1e-3, so a seed search cannot find one.  Instead the generator
  1. draws X0 ~ N(0,1) and W_r ~ N(0,1/d) (rounded to the storage dtype),
  2. forms the logits L0 = X0 W_r with a plain matrix product,
  3. ranks each (b,h) column of L0 with a stable argsort and builds
     G[b,t,h] = delta for the k highest-ranked tokens, else 0,
  4. sets X = X0 + G pinv(W_r)  (W_r has full column rank for H <= d, so
     X W_r = L0 + G exactly before rounding), and rounds X to the dtype.
The logit gap then exceeds delta minus the rounding noise (about 1e-3).
Only library primitives (matmul, argsort, pinv) are used for this.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

PLANT_DELTA = 0.05


@dataclass(frozen=True)
class MosaConfig:
    """One MoSA layer problem: B sequences of T tokens of width d, H heads of
    size hp (the paper's h'), k tokens per head, in ``dtype`` storage."""
    name: str
    B: int
    T: int
    d: int
    H: int
    hp: int
    k: int
    dtype: str = "bf16"          # "f32" or "bf16" storage; accumulation is fp32
    backward: bool = True
    seed: int = 0
    first_token: bool = False    # every head keeps token 0 and selects k-1 more
    rope: bool = False           # rotary position encoding of Q and K
    note: str = field(default="", compare=False)

    @property
    def tokens(self) -> int:
        return self.B * self.T

    def with_(self, **kw) -> "MosaConfig":
        d = dict(self.__dict__)
        d.update(kw)
        return MosaConfig(**d)


def _c5(H: int, k: int) -> MosaConfig:
    return MosaConfig(f"B4_T4096_d1024_H{H}_k{k}", B=4, T=4096, d=1024, H=H, hp=64, k=k, seed=5,
                      note="sparsity sweep at B4 T4096 d1024, per-layer attention work "
                           "roughly constant")


CONFIGS: dict[str, MosaConfig] = {
    c.name: c for c in [
        MosaConfig("f32_B1_T256_d128_H4_k64", B=1, T=256, d=128, H=4, hp=32, k=64, dtype="f32",
                   backward=False, seed=0, note="single layer, forward, fp32"),
        MosaConfig("B8_T1024_d512_H16_k128", B=8, T=1024, d=512, H=16, hp=64, k=128, seed=1,
                   note="forward+backward, bf16, sparsity 8"),
        MosaConfig("B16_T1024_d1024_H64_k64", B=16, T=1024, d=1024, H=64, hp=64, k=64, seed=2,
                   note="many small heads, sparsity 16"),
        MosaConfig("B2_T8192_d1024_H32_k256", B=2, T=8192, d=1024, H=32, hp=64, k=256, seed=3,
                   note="long sequence, sparsity 32"),
    ] + [_c5(H, k) for H, k in [(8, 2048), (16, 1024), (32, 512), (64, 256), (128, 128),
                                (256, 64)]]
}

#: The configuration the headline throughput is quoted on: the one with the
#: most work per step (163.8 GFLOP forward + backward).
BENCH_CONFIG = "B4_T4096_d1024_H8_k2048"


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even), returned as
    float32 holding exactly representable bf16 values."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    bits = a.view(np.uint32).astype(np.uint64)
    bits = (bits + 0x7FFF + ((bits >> 16) & 1)) & 0xFFFF0000
    return bits.astype(np.uint32).view(np.float32)


def to_storage(a: np.ndarray, dtype: str) -> np.ndarray:
    a = np.asarray(a, dtype=np.float32)
    return round_to_bf16(a) if dtype == "bf16" else np.ascontiguousarray(a)


def make_inputs(cfg: MosaConfig, seed: int | None = None, plant: bool = True,
                delta: float = PLANT_DELTA) -> dict[str, np.ndarray]:
    """Draw X, W_r, W_q, W_k, W_v, W_o and dY for ``cfg`` as float32 arrays whose
    values are exactly representable in ``cfg.dtype``.

    X ~ N(0,1) [B,T,d]; W_r ~ N(0,1/d) [d,H]; W_q, W_k, W_v ~ N(0,1/d) [H,d,hp];
    W_o ~ N(0,1/d) [H,hp,d]; dY ~ N(0,1) [B,T,d].  One generator, one draw per
    tensor in that fixed order.  With ``plant`` the router margin described in
    the module docstring is added to X."""
    rng = np.random.default_rng(cfg.seed if seed is None else seed)
    B, T, d, H, hp, k = cfg.B, cfg.T, cfg.d, cfg.H, cfg.hp, cfg.k
    s = 1.0 / np.sqrt(d)
    X0 = rng.standard_normal((B, T, d), dtype=np.float32)
    Wr = to_storage(rng.standard_normal((d, H), dtype=np.float32) * s, cfg.dtype)
    Wq = to_storage(rng.standard_normal((H, d, hp), dtype=np.float32) * s, cfg.dtype)
    Wk = to_storage(rng.standard_normal((H, d, hp), dtype=np.float32) * s, cfg.dtype)
    Wv = to_storage(rng.standard_normal((H, d, hp), dtype=np.float32) * s, cfg.dtype)
    Wo = to_storage(rng.standard_normal((H, hp, d), dtype=np.float32) * s, cfg.dtype)
    dY = to_storage(rng.standard_normal((B, T, d), dtype=np.float32), cfg.dtype)
    X0 = to_storage(X0, cfg.dtype)
    if plant:
        X = plant_margin(X0, Wr, k, delta, cfg.first_token)
    else:
        X = X0
    X = to_storage(X, cfg.dtype)
    return {"X": X, "Wr": Wr, "Wq": Wq, "Wk": Wk, "Wv": Wv, "Wo": Wo, "dY": dY}


def make_dense_weights(cfg: MosaConfig, H_dense: int, seed: int | None = None
                       ) -> dict[str, np.ndarray]:
    """Weights of the dense (or local) heads of a hybrid layer (Sec. 2.2,
    hybridization): D_q, D_k, D_v ~ N(0,1/d) [H_dense,d,hp] and D_o ~ N(0,1/d)
    [H_dense,hp,d], rounded to ``cfg.dtype``; one generator seeded with
    ``cfg.seed + 1000`` (or ``seed``), one draw per tensor in that order."""
    rng = np.random.default_rng(cfg.seed + 1000 if seed is None else seed)
    d, hp = cfg.d, cfg.hp
    s = 1.0 / np.sqrt(d)
    out = {}
    for name, shape in (("Dq", (H_dense, d, hp)), ("Dk", (H_dense, d, hp)),
                        ("Dv", (H_dense, d, hp)), ("Do", (H_dense, hp, d))):
        out[name] = to_storage(rng.standard_normal(shape, dtype=np.float32) * s, cfg.dtype)
    return out


def plant_margin(X0: np.ndarray, Wr: np.ndarray, k: int, delta: float,
                 first_token: bool = False) -> np.ndarray:
    """Return X0 + G pinv(W_r) where G raises the k highest logits of every
    (b, head) column of X0 W_r by ``delta`` (float64 arithmetic, float32 result).
    With ``first_token`` the raised set is token 0 and the k-1 highest of the
    other tokens (the set the selection then keeps)."""
    B, T, d = X0.shape
    H = Wr.shape[1]
    Wr64 = Wr.astype(np.float64)
    pinv = np.linalg.pinv(Wr64)                       # [H, d]
    Xout = np.empty_like(X0)
    for b in range(B):
        L0 = X0[b].astype(np.float64) @ Wr64          # [T, H]
        G = np.zeros((T, H))
        cols = np.arange(H)[None, :]
        if first_token:
            order = np.argsort(-L0[1:], axis=0, kind="stable") + 1   # tokens 1..T-1
            G[0, :] = delta
            G[order[:k - 1, :], cols] = delta
        else:
            order = np.argsort(-L0, axis=0, kind="stable")  # per column, highest first
            G[order[:k, :], cols] = delta
        Xout[b] = (X0[b].astype(np.float64) + G @ pinv).astype(np.float32)
    return Xout


def fixed_sparse_indices(B: int, H: int, T: int, k: int) -> np.ndarray:
    """I = [0, rho, 2 rho, ..., T - rho] for every (b, h), rho = T / k: the fixed
    sparse attention of Sec. 3.1 written as a MoSA index set."""
    if T % k:
        raise ValueError("fixed sparse attention needs k | T")
    rho = T // k
    row = np.arange(0, T, rho, dtype=np.int32)
    return np.ascontiguousarray(np.broadcast_to(row, (B, H, k)))
