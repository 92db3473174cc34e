"""Precision audit of the bf16 path's intermediates (analysis script, not a
test; writes the table recorded in the design notes).

The layer (Sec. 2.2, Eq. mosa_mha, forward and backward) is restated in fp64
torch on the CPU, on the seeded benchmark inputs, once exactly and once for
each intermediate rounded (alone) to bf16 or to fp16 where it is produced:
Q, K, V, the attention probabilities P, AR = diag(r) A, dA, dS and the three
input-side gradients dQ|dK|dV; plus two sets rounded together (the attention
operands Q, K, V, P, dA, dS in fp16, the set the k > 128 kernels keep at one
MMA per product, the same set in bf16, and all eight in fp16).  For every output (Y, dX and the
weight gradients) it reports the relative L2 and the largest absolute error
against the exact result, to be read against the comparison rule for bf16
storage (2e-2 relative L2, 5e-2 absolute per element).  Run:

    python tests/precision_audit.py [--only LABEL] [workload ...]   (default:
    the four bf16 benchmark workloads and every variant; a few minutes each on
    eight cores)
"""
from __future__ import annotations

import math
import os
import sys

import numpy as np
import torch

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
from paper_2505_00315_gb300 import workloads as W  # noqa: E402

F64 = torch.float64
OUTPUTS = ("Y", "dX", "dWr", "dWq", "dWk", "dWv", "dWo")
SINGLE = ("Q", "K", "V", "P", "AR", "dA", "dS", "dQKV")
ATTN_SET = ("Q", "K", "V", "P", "dA", "dS")


def rounder(names, dtype):
    names = set(names)
    def R(name, t):
        return t.to(dtype).to(F64) if name in names else t
    return R


def layer(x, k, R):
    """Forward + backward of the layer in fp64 with the rounding hook R."""
    t = lambda a: torch.from_numpy(np.asarray(a, np.float64))
    X, Wr, Wq, Wk, Wv, Wo, dY = (t(x[n]) for n in ("X", "Wr", "Wq", "Wk", "Wv", "Wo", "dY"))
    B, T, d = X.shape
    H, _, hp = Wq.shape
    out = {"Y": torch.zeros(B, T, d, dtype=F64), "dX": torch.zeros(B, T, d, dtype=F64),
           "dWr": torch.zeros(d, H, dtype=F64), "dWq": torch.zeros_like(Wq),
           "dWk": torch.zeros_like(Wk), "dWv": torch.zeros_like(Wv), "dWo": torch.zeros_like(Wo)}
    mask = torch.ones(k, k, dtype=torch.bool).tril()
    sc = 1.0 / math.sqrt(hp)
    for b in range(B):
        r_all = torch.sigmoid(X[b] @ Wr)                          # [T, H]
        I = torch.topk(r_all.T, k, dim=1).indices.sort(dim=1).values   # [H, k] ascending
        r = torch.gather(r_all.T, 1, I)                           # [H, k]
        Xs = X[b][I]                                              # [H, k, d]
        Q = R("Q", Xs @ Wq)
        K = R("K", Xs @ Wk)
        V = R("V", Xs @ Wv)
        S = (Q @ K.transpose(1, 2)) * sc
        S = S.masked_fill(~mask, float("-inf"))
        P = R("P", torch.softmax(S, dim=-1))
        A = P @ V
        AR = R("AR", r[..., None] * A)
        out["Y"][b].index_add_(0, I.reshape(-1), (AR @ Wo).reshape(-1, d))
        dYs = dY[b][I]                                            # [H, k, d]
        G = dYs @ Wo.transpose(1, 2)                              # [H, k, hp]
        dA = R("dA", r[..., None] * G)
        D = (AR * G).sum(-1)                                      # r <A, G>
        dlogit = D * (1 - r)
        dP = dA @ V.transpose(1, 2)
        dS = R("dS", P * (dP - D[..., None]))
        dQ = R("dQKV", (dS @ K) * sc)
        dK = R("dQKV", (dS.transpose(1, 2) @ Q) * sc)
        dV = R("dQKV", P.transpose(1, 2) @ dA)
        dXs = (dQ @ Wq.transpose(1, 2) + dK @ Wk.transpose(1, 2) + dV @ Wv.transpose(1, 2)
               + dlogit[..., None] * Wr.T[:, None, :])
        out["dX"][b].index_add_(0, I.reshape(-1), dXs.reshape(-1, d))
        out["dWq"] += Xs.transpose(1, 2) @ dQ
        out["dWk"] += Xs.transpose(1, 2) @ dK
        out["dWv"] += Xs.transpose(1, 2) @ dV
        out["dWo"] += AR.transpose(1, 2) @ dYs
        out["dWr"] += (Xs.transpose(1, 2) @ dlogit[..., None]).squeeze(-1).T
    return out


def audit(name, only=()):
    cfg = W.CONFIGS[name]
    x = W.make_inputs(cfg)
    exact = layer(x, cfg.k, lambda n, a: a)
    rows = []
    variants = [(f"{n} {p}", rounder([n], dt)) for p, dt in (("bf16", torch.bfloat16),
                                                                ("fp16", torch.float16))
                for n in SINGLE]
    variants += [("Q,K,V,P,dA,dS fp16", rounder(ATTN_SET, torch.float16)),
                 ("Q,K,V,P,dA,dS bf16", rounder(ATTN_SET, torch.bfloat16)),
                 ("all eight fp16", rounder(SINGLE, torch.float16))]
    if only:
        variants = [v for v in variants if v[0] in only]
    for label, R in variants:
        got = layer(x, cfg.k, R)
        errs = {}
        for o in OUTPUTS:
            e = got[o] - exact[o]
            errs[o] = (float(e.norm() / exact[o].norm()), float(e.abs().max()))
        rows.append((label, errs))
        worst_rel = max(v[0] for v in errs.values())
        worst_abs = max(v[1] for v in errs.values())
        ok = worst_rel < 2e-2 and worst_abs < 5e-2
        print(f"{name} | {label:20s} | worst rel-L2 {worst_rel:.2e} ({max(errs, key=lambda o: errs[o][0])}) "
              f"| worst max-abs {worst_abs:.2e} ({max(errs, key=lambda o: errs[o][1])}) | "
              f"{'passes' if ok else 'FAILS'}", flush=True)
    return rows


if __name__ == "__main__":
    torch.set_num_threads(os.cpu_count() or 8)
    args = sys.argv[1:]
    only = ()
    if args[:1] == ["--only"]:
        only, args = (args[1],), args[2:]
    names = args or ["B8_T1024_d512_H16_k128", "B16_T1024_d1024_H64_k64",
                             "B2_T8192_d1024_H32_k256", "B4_T4096_d1024_H8_k2048"]
    for n in names:
        audit(n, only)
