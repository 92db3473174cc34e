"""FLOP model of the MoSA layer.

``head_flops_dense`` / ``head_flops_mosa`` / ``model_forward_flops`` restate
App. A (and Sec. 3.2, "FLOPs Calculation"): a product of [i,j] and [j,k]
matrices counts 2ijk FLOPs; a dense head costs 8hh'T + 4h'T^2, a MoSA head
8hh'k + 4h'k^2 + 2hT + h'k, a feed-forward block 16h^2T.  ``isoflop_heads``
picks the largest head count whose model does not exceed the dense baseline,
as App. C describes.

``layer_work`` gives the algorithmic work of one MoSA layer as this library
executes it, per kernel, with causal attention counted exactly
(k(k+1)/2 allowed query-key pairs per head) instead of the paper's 4h'k^2.
These are the numerators of the reported roofline fractions.
"""
from __future__ import annotations


def head_flops_dense(h: int, hp: int, T: int) -> int:
    """App. A: Q, K, V, O mappings 8hh'T plus attention 4h'T^2."""
    return 8 * h * hp * T + 4 * hp * T * T


def head_flops_mosa(h: int, hp: int, T: int, k: int) -> int:
    """App. A: mappings on k tokens 8hh'k, attention 4h'k^2, routing 2hT + h'k."""
    return 8 * h * hp * k + 4 * hp * k * k + 2 * h * T + hp * k


def model_forward_flops(layers: int, h: int, hp: int, T: int, n_dense: int, n_mosa: int,
                        k: int) -> int:
    """App. A: l H_dense FLOP_dense + l H_mosa FLOP_mosa + 16 l h^2 T."""
    return (layers * n_dense * head_flops_dense(h, hp, T)
            + layers * n_mosa * head_flops_mosa(h, hp, T, k)
            + 16 * layers * h * h * T)


def isoflop_heads(layers: int, h: int, hp: int, T: int, n_heads_dense_baseline: int,
                  rho: int, n_dense: int) -> int:
    """Largest number of MoSA heads (with ``n_dense`` dense heads kept) whose
    forward FLOPs do not exceed the dense baseline's (App. C)."""
    budget = model_forward_flops(layers, h, hp, T, n_heads_dense_baseline, 0, 0)
    if rho == 1:
        return 0
    k = T // rho
    fixed = model_forward_flops(layers, h, hp, T, n_dense, 0, k)
    return (budget - fixed) // (layers * head_flops_mosa(h, hp, T, k))


def layer_work(B: int, T: int, d: int, H: int, hp: int, k: int, elem_bytes: int = 2,
               causal: bool = True) -> dict:
    """Algorithmic FLOPs and HBM bytes of one MoSA layer, per step of the
    forward (F1-F5) and backward (B1-B4) pass, summed over all B*H units.

    FLOPs: router 2dT per (b,h); projections 6dh'k; causal attention
    2h'k(k+1) forward and 5h'k(k+1) backward; output 2h'dk; output backward
    4h'dk; input backward 6dh'k + 2dk; weight backward 6dh'k + 2dk.
    ``causal=False`` counts attention as the paper does (App. A: 4h'k^2
    forward, not halved for the mask) and 10h'k^2 backward.
    Bytes (minimum, each operand touched once): see the per-entry comments."""
    U = B * H
    e = elem_bytes
    causal = hp * k * (k + 1) if causal else 2 * hp * k * k
    w = {
        "router": {"flops": 2 * d * T * U,
                   # read X once, write r [B,H,T] fp32
                   "bytes": B * T * d * e + d * H * e + B * H * T * 4},
        "select": {"flops": 0,
                   # read r once, write I (int32) and r_sel (fp32)
                   "bytes": B * H * T * 4 + 2 * B * H * k * 4},
        "qkv": {"flops": 6 * d * hp * k * U,
                # gathered rows of X, the three projection weights, Q/K/V out
                "bytes": U * k * d * e + 3 * H * d * hp * e + 3 * U * k * hp * e},
        "attn_fwd": {"flops": 2 * causal * U,
                     "bytes": 3 * U * k * hp * e + 2 * U * k * hp * e + U * k * 4},
        "out": {"flops": 2 * hp * d * k * U,
                # read scaled A and W_o; fp32 reduction into Y[B,T,d]
                "bytes": U * k * hp * e + H * hp * d * e + U * k * d * 4},
        # G = dY[I] W_o^T and the row terms (dr, dA, D, dlogit)
        "out_bwd": {"flops": 2 * hp * d * k * U,
                    "bytes": U * k * d * e + H * hp * d * e + 2 * U * k * hp * e},
        # dW_o = (diag(r) A)^T dY[I]
        "dwo": {"flops": 2 * hp * d * k * U,
                "bytes": U * k * d * e + U * k * hp * e + H * hp * d * 4},
        "attn_bwd": {"flops": 5 * causal * U,
                     "bytes": 6 * U * k * hp * e + 3 * U * k * hp * e},
        "in_bwd": {"flops": (6 * d * hp * k + 2 * d * k) * U,
                   "bytes": 3 * U * k * hp * e + 3 * H * d * hp * e + U * k * d * 4},
        "w_bwd": {"flops": (6 * d * hp * k + 2 * d * k) * U,
                  "bytes": U * k * d * e + 3 * U * k * hp * e + 3 * H * d * hp * 4 + d * H * 4},
    }
    # F3 + F4 + F5 in one kernel (k <= 128): the three steps' FLOPs; bytes as
    # those steps minus the Q/K/V and scaled-A round trips they no longer make
    # (Q/K/V, A, AR and lse are still written once for the backward)
    w["fwd_unit"] = {"flops": w["qkv"]["flops"] + w["attn_fwd"]["flops"] + w["out"]["flops"],
                     "bytes": U * k * d * e + 3 * H * d * hp * e + H * hp * d * e
                              + 3 * U * k * hp * e + 2 * U * k * hp * e + U * k * 4
                              + U * k * d * 4}
    # B1 (G and row terms) + B2 in one kernel (k <= 128): the two steps' FLOPs;
    # bytes: gathered dY, W_o, A, Q/K/V in, dQ|dK|dV out
    w["bwd_unit"] = {"flops": w["out_bwd"]["flops"] + w["attn_bwd"]["flops"],
                     "bytes": U * k * d * e + H * hp * d * e + U * k * hp * 4 + 3 * U * k * hp * e
                              + 3 * U * k * hp * e}
    fwd = ("router", "select", "qkv", "attn_fwd", "out")
    bwd = ("out_bwd", "dwo", "attn_bwd", "in_bwd", "w_bwd")
    w["forward_flops"] = sum(w[s]["flops"] for s in fwd)
    w["backward_flops"] = sum(w[s]["flops"] for s in bwd)
    return w


def hybrid_work(B: int, T: int, d: int, H: int, hp: int, k: int, H_dense: int,
                window: int = 0, elem_bytes: int = 2, causal: bool = True) -> dict:
    """``layer_work`` of a hybrid layer (Sec. 2.2, hybridization; Sec. 3.4):
    the MoSA heads plus H_dense dense heads over all T tokens (window 0) or
    local heads over blocks of ``window`` tokens, per step, summed.  The dense
    heads have no router: no F1 work, their token lists are written once
    (8 bytes per row), and no dlogit terms in B3/B4."""
    w = layer_work(B, T, d, H, hp, k, elem_bytes, causal)
    if H_dense <= 0:
        return w
    blk = window if window else T
    Bd = B * (T // blk)
    dn = layer_work(Bd, blk, d, H_dense, hp, blk, elem_bytes, causal)
    rows = Bd * H_dense * blk
    dn["router"] = {"flops": 0, "bytes": 0}
    dn["select"] = {"flops": 0, "bytes": 2 * rows * 4}
    for s in ("in_bwd", "w_bwd"):
        dn[s] = dict(dn[s], flops=dn[s]["flops"] - 2 * d * blk * Bd * H_dense)
    dn["w_bwd"]["bytes"] -= d * H_dense * 4
    out = {}
    for s, v in w.items():
        if isinstance(v, dict):
            out[s] = {"flops": v["flops"] + dn[s]["flops"], "bytes": v["bytes"] + dn[s]["bytes"]}
    fwd = ("router", "select", "qkv", "attn_fwd", "out")
    bwd = ("out_bwd", "dwo", "attn_bwd", "in_bwd", "w_bwd")
    out["forward_flops"] = sum(out[s]["flops"] for s in fwd)
    out["backward_flops"] = sum(out[s]["flops"] for s in bwd)
    return out
