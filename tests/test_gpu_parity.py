"""GPU parity: libmosa (through its C ABI) against the fp64 CPU oracle.

Indices are compared bit-exactly; floats within the stated tolerances
(fp32 storage: 1e-4 relative L2; bf16 storage: 2e-2 relative L2 and 5e-2
max-abs).  Small cases are compared element by element in full; the full
workload sizes are compared on sampled units the oracle computes exactly
(every head of one sequence for Y and dX, every sequence of one head for the
weight gradients) plus every selected index.
"""
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2505_00315_gb300 as mosa
from paper_2505_00315_gb300 import workloads as W
from _gpu import assert_close, run_layer, to_dev
from _util import sigmoid_gap

pytestmark = pytest.mark.gpu


def weights(x):
    return x["Wr"], x["Wq"], x["Wk"], x["Wv"], x["Wo"]


# ------------------------------------------------------------ TopK alone ----

def score_rows(kind, rows, T, rng, k=1):
    if kind == "uniform":
        return rng.random((rows, T), dtype=np.float32)
    if kind == "ties":
        return rng.choice(np.array([0.125, 0.25, 0.5, 0.75], np.float32), size=(rows, T))
    if kind == "equal":
        return np.full((rows, T), 0.5, np.float32)
    if kind == "signed":      # negatives, both zeros, sub-normals
        v = rng.standard_normal((rows, T)).astype(np.float32)
        v[:, ::7] = 0.0
        v[:, 3::11] = -0.0
        v[:, 5::13] = np.float32(1e-42)
        return v
    if kind == "split":       # the k kept scores alone in the first radix byte's bin
        v = (0.25 + 0.01 * rng.random((rows, T))).astype(np.float32)
        for r in range(rows):
            v[r, rng.choice(T, size=k, replace=False)] += np.float32(1.25)
        return v
    if kind == "gap":         # router-like scores around 1/2, a 1e-3 gap after the k-th
        v = 0.5 + 0.05 * rng.standard_normal((rows, T))
        for r in range(rows):
            top = np.argsort(-v[r], kind="stable")[:k]
            v[r, top] += 1e-3
        return v.astype(np.float32)
    raise ValueError(kind)


# ("split" and "gap" let the radix passes stop early, after the first byte or
# after two or three, as router scores with a planted margin do)
@pytest.mark.parametrize("kind", ["uniform", "ties", "equal", "signed", "split", "gap"])
@pytest.mark.parametrize("T,k", [(1, 1), (7, 3), (1000, 1), (1024, 128), (1025, 1025),
                                 (4096, 64), (8192, 4000), (65536, 257)])
def test_topk_bit_exact(kind, T, k):
    rng = np.random.default_rng(T * 31 + k)
    rows = 3 if T > 10000 else 5
    s = score_rows(kind, rows, T, rng, k)
    I, rs = mosa.mosa_topk(torch.from_numpy(s).cuda(), k)
    I, rs = I.cpu().numpy(), rs.cpu().numpy()
    for r in range(rows):
        Iref, _ = oracle.topk(s[r].astype(np.float64), k)
        np.testing.assert_array_equal(I[r], Iref)
        np.testing.assert_array_equal(rs[r].view(np.uint32), s[r][Iref].view(np.uint32))


# ---------------------------------------------------- small full parity ----

SMALL = [
    W.CONFIGS["f32_B1_T256_d128_H4_k64"],
    W.MosaConfig("ragged_f32", B=2, T=300, d=136, H=3, hp=32, k=77, dtype="f32", seed=11),
    W.MosaConfig("ragged_bf16", B=2, T=300, d=136, H=3, hp=64, k=77, dtype="bf16", seed=12),
    W.MosaConfig("k_eq_T_bf16", B=2, T=96, d=64, H=2, hp=64, k=96, dtype="bf16", seed=13),
    W.MosaConfig("k1_f32", B=3, T=50, d=16, H=5, hp=16, k=1, dtype="f32", seed=14),
    W.MosaConfig("hp128_bf16", B=1, T=200, d=256, H=2, hp=128, k=130, dtype="bf16", seed=15),
    W.MosaConfig("hp16_f32", B=2, T=129, d=24, H=7, hp=16, k=65, dtype="f32", seed=16),
    # k <= 64: several sequences of a head share one 128-row attention tile
    W.MosaConfig("pack2_oddB_bf16", B=3, T=200, d=64, H=2, hp=64, k=64, dtype="bf16", seed=17),
    W.MosaConfig("pack4_bf16", B=5, T=100, d=64, H=3, hp=64, k=32, dtype="bf16", seed=18),
    W.MosaConfig("pack2_k50_bf16", B=5, T=120, d=64, H=2, hp=64, k=50, dtype="bf16", seed=19),
    # k <= 128 with weights large against X (3 H h' > 2 B T): dQ|dK|dV stay
    # bf16 pairs for the input- and weight-gradient products
    W.MosaConfig("pairs_bf16", B=1, T=160, d=64, H=4, hp=64, k=48, dtype="bf16", seed=20),
    W.MosaConfig("pack42_k3_bf16", B=5, T=40, d=32, H=2, hp=64, k=3, dtype="bf16", seed=20),
    # k > 128: several 128-query tiles and 128-key blocks, full and ragged
    W.MosaConfig("largek_bf16", B=1, T=512, d=128, H=3, hp=64, k=384, dtype="bf16", seed=21),
    W.MosaConfig("largek_ragged_bf16", B=2, T=600, d=64, H=2, hp=64, k=300, dtype="bf16", seed=22),
]


@pytest.fixture(params=["default", "unfused", "fused_bwd", "rowmajor", "tokenmajor", "simt"])
def kernel_path(request, monkeypatch):
    """Run a test on the default kernels (tensor cores where the shape allows,
    the fused forward for k <= 128, the token-major output and input-gradient
    products for k > 128 where the heads keep a large share of the tokens),
    again with the forward as three separate kernels, again with the fused
    backward switched on, again with the row-major (scatter-add) products
    only, again with the token-major products wherever they apply, and again
    with the CUDA-core kernels forced."""
    monkeypatch.delenv("MOSA_FORCE_SIMT", raising=False)
    monkeypatch.delenv("MOSA_FUSED_FWD", raising=False)
    monkeypatch.delenv("MOSA_FUSED_BWD", raising=False)
    monkeypatch.delenv("MOSA_HEADSUM", raising=False)
    if request.param == "rowmajor":
        monkeypatch.setenv("MOSA_HEADSUM", "0")
    elif request.param == "tokenmajor":
        monkeypatch.setenv("MOSA_HEADSUM", "1")
    elif request.param == "simt":
        monkeypatch.setenv("MOSA_FORCE_SIMT", "1")
    elif request.param == "unfused":
        monkeypatch.setenv("MOSA_FUSED_FWD", "0")
    elif request.param == "fused_bwd":
        monkeypatch.setenv("MOSA_FUSED_BWD", "1")
    return request.param


@pytest.mark.parametrize("cfg", SMALL, ids=lambda c: c.name)
def test_small_forward_backward_full_parity(cfg, kernel_path):
    x = W.make_inputs(cfg)
    Y, I, rs, rf = oracle.forward(x["X"], *weights(x), k=cfg.k)
    assert sigmoid_gap(rf, cfg.k) > 1e-3
    g = run_layer(cfg, x, backward=True)
    np.testing.assert_array_equal(g["I"], I)
    assert_close("r_full", g["r_full"], rf, cfg.dtype)
    assert_close("r_sel", g["r_sel"], rs, cfg.dtype)
    assert_close("Y", g["Y"], Y, cfg.dtype)
    untouched = np.ones((cfg.B, cfg.T), bool)
    for b in range(cfg.B):
        untouched[b, I[b].ravel()] = False
    assert (g["Y"][untouched] == 0).all()
    ref = oracle.backward(x["X"], *weights(x), I=I, dY=x["dY"])
    for name in ("dX", "dWr", "dWq", "dWk", "dWv", "dWo"):
        gname = name[:2] + "_" + name[2:].lower() if name != "dX" else "dX"
        assert_close(name, g[gname], ref[name], cfg.dtype)


# ------------------------------------ first token always kept (Sec. 3.2) ----

FIRST = [
    W.MosaConfig("first_bf16", B=3, T=200, d=64, H=2, hp=64, k=64, dtype="bf16", seed=31,
                 first_token=True),
    W.MosaConfig("first_pack_bf16", B=5, T=90, d=32, H=3, hp=64, k=30, dtype="bf16", seed=32,
                 first_token=True),
    W.MosaConfig("first_k1_bf16", B=2, T=50, d=32, H=3, hp=64, k=1, dtype="bf16", seed=33,
                 first_token=True),
    W.MosaConfig("first_f32", B=2, T=129, d=24, H=3, hp=32, k=40, dtype="f32", seed=34,
                 first_token=True),
    W.MosaConfig("first_largek_bf16", B=1, T=400, d=64, H=2, hp=64, k=200, dtype="bf16",
                 seed=35, first_token=True),
]


@pytest.mark.parametrize("cfg", FIRST, ids=lambda c: c.name)
def test_first_token_forward_backward_parity(cfg, kernel_path):
    x = W.make_inputs(cfg)
    Y, I, rs, rf = oracle.forward(x["X"], *weights(x), k=cfg.k, first_token=True)
    if cfg.k > 1:
        assert sigmoid_gap(rf[..., 1:], cfg.k - 1) > 1e-3
    g = run_layer(cfg, x, backward=True)
    assert (g["I"][:, :, 0] == 0).all()
    np.testing.assert_array_equal(g["I"], I)
    assert_close("r_sel", g["r_sel"], rs, cfg.dtype)
    assert_close("Y", g["Y"], Y, cfg.dtype)
    ref = oracle.backward(x["X"], *weights(x), I=I, dY=x["dY"])
    for name in ("dX", "dWr", "dWq", "dWk", "dWv", "dWo"):
        gname = name[:2] + "_" + name[2:].lower() if name != "dX" else "dX"
        assert_close(name, g[gname], ref[name], cfg.dtype)


def test_first_token_long_rows_unstaged_select():
    # rows longer than the TopK kernel stages in shared memory (16384 scores)
    cfg = W.MosaConfig("first_long", B=1, T=20000, d=64, H=2, hp=64, k=300, dtype="bf16",
                       seed=36, first_token=True)
    x = W.make_inputs(cfg)
    X, Wr = to_dev(x["X"], "bf16"), to_dev(x["Wr"], "bf16")
    I, rs = mosa.mosa_route_noalloc(X, Wr, cfg.k, first_token=True)
    rf = oracle.router(x["X"], x["Wr"])
    assert sigmoid_gap(rf[..., 1:], cfg.k - 1) > 1e-3
    I = I.cpu().numpy()
    for h in range(cfg.H):
        Iref, _ = oracle.topk(rf[0, h], cfg.k, first_token=True)
        np.testing.assert_array_equal(I[0, h], Iref)


# ------------------------------------------- RoPE at the original positions ----

ROPE = [
    W.MosaConfig("rope_bf16", B=3, T=200, d=64, H=2, hp=64, k=64, dtype="bf16", seed=41,
                 rope=True),
    W.MosaConfig("rope_largek_bf16", B=2, T=600, d=64, H=2, hp=64, k=300, dtype="bf16",
                 seed=42, rope=True),
    W.MosaConfig("rope_far_bf16", B=1, T=20000, d=64, H=2, hp=64, k=64, dtype="bf16", seed=43,
                 rope=True),
    W.MosaConfig("rope_f32", B=2, T=129, d=24, H=3, hp=32, k=40, dtype="f32", seed=44,
                 rope=True),
    W.MosaConfig("rope_hp16_f32", B=2, T=90, d=16, H=2, hp=16, k=33, dtype="f32", seed=45,
                 rope=True),
    W.MosaConfig("rope_first_bf16", B=2, T=150, d=32, H=2, hp=64, k=50, dtype="bf16", seed=46,
                 rope=True, first_token=True),
]


@pytest.mark.parametrize("cfg", ROPE, ids=lambda c: c.name)
def test_rope_forward_backward_parity(cfg, kernel_path):
    x = W.make_inputs(cfg)
    Y, I, rs, rf = oracle.forward(x["X"], *weights(x), k=cfg.k, first_token=cfg.first_token,
                                  rope=True)
    g = run_layer(cfg, x, backward=True)
    np.testing.assert_array_equal(g["I"], I)
    assert_close("Y", g["Y"], Y, cfg.dtype)
    ref = oracle.backward(x["X"], *weights(x), I=I, dY=x["dY"], rope=True)
    for name in ("dX", "dWr", "dWq", "dWk", "dWv", "dWo"):
        gname = name[:2] + "_" + name[2:].lower() if name != "dX" else "dX"
        assert_close(name, g[gname], ref[name], cfg.dtype)


# ------------------------- hybrid layer: MoSA heads beside dense heads ----

@pytest.mark.parametrize("rope", [False, True])
def test_hybrid_mosa_plus_dense_heads(rope):
    # Sec. 2.2 (hybridization): MoSA heads and dense heads in one layer, their
    # outputs summed; a dense head is the index-given forward with I = 0..T-1
    # and unit scores
    cfg = W.MosaConfig("hybrid", B=2, T=128, d=64, H=4, hp=64, k=32, dtype="bf16", seed=51,
                       rope=rope)
    dense = W.MosaConfig("hybrid_dense", B=2, T=128, d=64, H=2, hp=64, k=128, dtype="bf16",
                         seed=52, rope=rope)
    x = W.make_inputs(cfg)
    xd = W.make_inputs(dense, plant=False)
    Ym, I, _, _ = oracle.forward(x["X"], *weights(x), k=cfg.k, rope=rope)
    Idense = np.broadcast_to(np.arange(cfg.T, dtype=np.int32), (cfg.B, dense.H, cfg.T)).copy()
    ones = np.ones((cfg.B, dense.H, cfg.T))
    Yd = oracle.forward_indices(x["X"], xd["Wr"], xd["Wq"], xd["Wk"], xd["Wv"], xd["Wo"],
                                I=Idense, r_sel=ones, rope=rope)
    X = to_dev(x["X"], "bf16")
    Wm = [to_dev(x[n], "bf16") for n in ("Wr", "Wq", "Wk", "Wv", "Wo")]
    Wd = [to_dev(xd[n], "bf16") for n in ("Wq", "Wk", "Wv", "Wo")]
    Yg, Ig, _, _, _ = mosa.mosa_forward(X, *Wm, cfg.k, rope=rope)
    Ydg, _ = mosa.mosa_forward_with_indices(
        X, *Wd, torch.tensor(Idense, device="cuda"),
        torch.ones((cfg.B, dense.H, cfg.T), dtype=torch.float32, device="cuda"), rope=rope)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(Ig.cpu().numpy(), I)
    assert_close("Y", (Yg + Ydg).cpu().numpy(), Ym + Yd, "bf16")


# --------------- hybrid layer entry (Sec. 2.2 hybridization, Sec. 3.4) ----

# (config, dense heads, window): window 0 = dense causal heads over all T
# tokens, w > 0 = local heads within blocks of w tokens
HYBRID = [
    (W.MosaConfig("hyb_dense_bf16", B=2, T=256, d=128, H=4, hp=64, k=64, dtype="bf16",
                  seed=53), 2, 0),
    (W.MosaConfig("hyb_local64_rope_bf16", B=2, T=256, d=128, H=4, hp=64, k=32, dtype="bf16",
                  seed=54, rope=True), 3, 64),
    (W.MosaConfig("hyb_local128_first_rope_bf16", B=2, T=384, d=64, H=2, hp=64, k=48,
                  dtype="bf16", seed=55, rope=True, first_token=True), 2, 128),
    (W.MosaConfig("hyb_dense_rope_f32", B=2, T=96, d=48, H=3, hp=32, k=24, dtype="f32", seed=56,
                  rope=True), 2, 0),
    (W.MosaConfig("hyb_local40_f32", B=1, T=120, d=40, H=2, hp=16, k=30, dtype="f32", seed=57),
     1, 40),
]


def run_hybrid(cfg, x, xd, window):
    dt = cfg.dtype
    X, Wr, Wq, Wk, Wv, Wo = (to_dev(x[n], dt) for n in ("X", "Wr", "Wq", "Wk", "Wv", "Wo"))
    D = [to_dev(xd[n], dt) for n in ("Dq", "Dk", "Dv", "Do")]
    Y, I, rs, ws = mosa.mosa_hybrid_forward(X, Wr, Wq, Wk, Wv, Wo, *D, cfg.k, window=window,
                                            first_token=cfg.first_token, rope=cfg.rope)
    out = {"Y": Y, "I": I}
    out.update(mosa.mosa_hybrid_backward(X, Wr, Wq, Wk, Wv, Wo, *D, I, rs, to_dev(x["dY"], dt),
                                         ws, window=window, rope=cfg.rope))
    torch.cuda.synchronize()
    assert mosa.mosa_check_status(mosa.make_shape(X, Wq, cfg.k), ws) == 0
    return {k: v.cpu().numpy() for k, v in out.items()}


HYB_GRADS = (("dX", "dX"), ("dWr", "dW_r"), ("dWq", "dW_q"), ("dWk", "dW_k"), ("dWv", "dW_v"),
             ("dWo", "dW_o"), ("dDq", "dD_q"), ("dDk", "dD_k"), ("dDv", "dD_v"),
             ("dDo", "dD_o"))


@pytest.mark.parametrize("case", HYBRID, ids=lambda c: c[0].name)
def test_hybrid_entry_forward_backward_parity(case, kernel_path):
    cfg, H_dense, window = case
    x = W.make_inputs(cfg)
    xd = W.make_dense_weights(cfg, H_dense)
    Y, I, _, _ = oracle.hybrid_forward(x["X"], *weights(x), xd["Dq"], xd["Dk"], xd["Dv"],
                                       xd["Do"], k=cfg.k, window=window,
                                       first_token=cfg.first_token, rope=cfg.rope)
    ref = oracle.hybrid_backward(x["X"], *weights(x), xd["Dq"], xd["Dk"], xd["Dv"], xd["Do"],
                                 I=I, dY=x["dY"], window=window, rope=cfg.rope)
    g = run_hybrid(cfg, x, xd, window)
    np.testing.assert_array_equal(g["I"], I)
    assert_close("Y", g["Y"], Y, cfg.dtype)
    for name, gname in HYB_GRADS:
        assert_close(name, g[gname], ref[name], cfg.dtype)


def test_hybrid_entry_paper_sizes_sampled():
    # the IsoFLOP hybrids of Sec. 3.2 keep 4 dense heads beside the MoSA
    # heads (here at B8 T1024 d512 H16 k128); the long-sequence models of
    # Sec. 3.4 pair 60 MoSA heads (k = 64) with 4 local heads at T = 2048,
    # d = 1024 (block of 512 tokens).  Y and dX of the last sequence, exact in
    # the oracle for that sequence alone.
    for cfg, H_dense, window in (
            (W.MosaConfig("hyb_isoflop", B=8, T=1024, d=512, H=16, hp=64, k=128, dtype="bf16",
                          seed=58, rope=True, first_token=True), 4, 0),
            (W.MosaConfig("hyb_long", B=1, T=2048, d=1024, H=60, hp=64, k=64, dtype="bf16",
                          seed=59, rope=True), 4, 512)):
        x = W.make_inputs(cfg)
        xd = W.make_dense_weights(cfg, H_dense)
        g = run_hybrid(cfg, x, xd, window)
        b0 = cfg.B - 1
        Y, I, _, _ = oracle.hybrid_forward(x["X"], *weights(x), xd["Dq"], xd["Dk"], xd["Dv"],
                                           xd["Do"], k=cfg.k, window=window, batches=[b0],
                                           first_token=cfg.first_token, rope=cfg.rope)
        np.testing.assert_array_equal(g["I"][b0], I[b0])
        assert_close("Y", g["Y"][b0], Y[b0], cfg.dtype)
        ref = oracle.hybrid_backward(x["X"], *weights(x), xd["Dq"], xd["Dk"], xd["Dv"],
                                     xd["Do"], I=I, dY=x["dY"], window=window, batches=[b0],
                                     rope=cfg.rope)
        assert_close("dX", g["dX"][b0], ref["dX"][b0], cfg.dtype)
        if cfg.B == 1:
            for name, gname in HYB_GRADS[1:]:
                assert_close(name, g[gname], ref[name], cfg.dtype)


# ------------------------------------------------ full workload sizes ----

FULL = [c for c in W.CONFIGS.values() if c.dtype == "bf16"]


@pytest.mark.parametrize("cfg", FULL, ids=lambda c: c.name)
def test_full_size_sampled_parity(cfg):
    x = W.make_inputs(cfg)
    g = run_layer(cfg, x, backward=True)
    # Every selected index, bit-exact, from the oracle's full score table.
    rf = oracle.router(x["X"], x["Wr"])
    assert sigmoid_gap(rf, cfg.k) > 1e-3
    for b in range(cfg.B):
        for h in range(cfg.H):
            Iref, rsref = oracle.topk(rf[b, h], cfg.k)
            np.testing.assert_array_equal(g["I"][b, h], Iref)
    assert_close("r_full", g["r_full"], rf, cfg.dtype)
    # Y and dX of sequence 0 (all heads), exact in the oracle.
    b0 = cfg.B - 1
    Y, I, _, _ = oracle.forward(x["X"], *weights(x), k=cfg.k, batches=[b0])
    assert_close("Y[b]", g["Y"][b0], Y[b0], cfg.dtype)
    gb = oracle.backward(x["X"], *weights(x), I=g["I"], dY=x["dY"], batches=[b0])
    assert_close("dX[b]", g["dX"][b0], gb["dX"][b0], cfg.dtype)
    # Weight gradients of one head (all sequences), exact in the oracle.
    h0 = cfg.H // 2
    gh = oracle.backward(x["X"], *weights(x), I=g["I"], dY=x["dY"], heads=[h0])
    for name in ("dWq", "dWk", "dWv", "dWo"):
        assert_close(name + "[h]", g[name[:2] + "_" + name[2:].lower()][h0], gh[name][h0],
                     cfg.dtype)
    assert_close("dWr[:,h]", g["dW_r"][:, h0], gh["dWr"][:, h0], cfg.dtype)


# --------------------------------------------------- indices entry point ----

@pytest.mark.parametrize("dtype,hp", [("f32", 32), ("bf16", 32), ("bf16", 64)])
def test_fixed_sparse_indices_entry(dtype, hp, kernel_path):
    cfg = W.MosaConfig("fixed", B=2, T=512, d=64, H=4, hp=hp, k=64, dtype=dtype, seed=21)
    x = W.make_inputs(cfg, plant=False)
    I = W.fixed_sparse_indices(cfg.B, cfg.H, cfg.T, cfg.k)
    ones = np.ones((cfg.B, cfg.H, cfg.k), np.float32)
    ref = oracle.forward_indices(x["X"], *weights(x), I=I, r_sel=ones)
    Xd, Wq, Wk, Wv, Wo = (to_dev(x[n], dtype) for n in ("X", "Wq", "Wk", "Wv", "Wo"))
    Y, ws = mosa.mosa_forward_with_indices(Xd, Wq, Wk, Wv, Wo, torch.from_numpy(I).cuda(),
                                           torch.from_numpy(ones).cuda())
    assert mosa.mosa_check_status(mosa.make_shape(Xd, Wq, cfg.k), ws) == 0
    assert_close("Y", Y.cpu().numpy(), ref, dtype)


def test_invalid_indices_are_flagged_not_followed():
    cfg = W.MosaConfig("bad", B=1, T=64, d=32, H=2, hp=32, k=8, dtype="f32", seed=22)
    x = W.make_inputs(cfg, plant=False)
    I = W.fixed_sparse_indices(cfg.B, cfg.H, cfg.T, cfg.k).copy()
    I[0, 1, 3] = 10_000          # out of range
    I[0, 0, 5] = I[0, 0, 4]      # not strictly ascending
    Xd, Wq, Wk, Wv, Wo = (to_dev(x[n], "f32") for n in ("X", "Wq", "Wk", "Wv", "Wo"))
    rs = torch.ones((1, 2, 8), device="cuda")
    Y, ws = mosa.mosa_forward_with_indices(Xd, Wq, Wk, Wv, Wo, torch.from_numpy(I).cuda(), rs)
    shape = mosa.make_shape(Xd, Wq, cfg.k)
    assert mosa.mosa_check_status(shape, ws) == 1          # MOSA_ERR_INVALID_ARG
    assert torch.isfinite(Y).all()
    assert mosa.mosa_check_status(shape, ws) == 0          # cleared by the read


@pytest.mark.parametrize("which", ["Wo", "Wq", "X"])
def test_fp16_copy_beyond_range_is_reported(which):
    # k > 128 on the tensor cores keeps fp16 copies of X, W_q|W_k|W_v and W_o:
    # a bf16 value beyond the fp16 range in any of them is reported as
    # MOSA_ERR_RANGE after the layer's forward and backward
    cfg = W.MosaConfig("range", B=1, T=512, d=128, H=8, hp=64, k=256, dtype="bf16", seed=23)
    x = W.make_inputs(cfg)
    names = ("X", "Wr", "Wq", "Wk", "Wv", "Wo")
    shape = mosa.make_shape(to_dev(x["X"], "bf16"), to_dev(x["Wq"], "bf16"), cfg.k, True)
    dY = to_dev(x["dY"], "bf16")

    def layer(inp):
        a = [to_dev(inp[n], "bf16") for n in names]
        _, I, rs, _, ws = mosa.mosa_forward(*a, cfg.k, first_token=True)
        mosa.mosa_backward(*a, I, rs, dY, ws)
        return mosa.mosa_check_status(shape, ws)

    bad = dict(x)
    bad[which] = x[which].copy()
    bad[which].flat[5] = 1.0e5
    assert layer(bad) == 6                                  # MOSA_ERR_RANGE
    assert layer(x) == 0


def test_status_word_maps_to_error_codes():
    # A bounded device wait that gives up sets the timeout bit in the
    # workspace status word; here the bits are written from the host (no
    # kernel waits or faults) and the read maps them to error codes, timeout
    # first, and clears the word.
    X = torch.zeros((1, 16, 32), dtype=torch.float32, device="cuda")
    Wq = torch.zeros((2, 32, 32), dtype=torch.float32, device="cuda")
    shape = mosa.make_shape(X, Wq, 4)
    ws = mosa.alloc_workspace(shape)
    ws.zero_()
    for word, code in ((2, 4), (3, 4), (1, 1), (0, 0)):   # timeout, both, bad index, none
        ws[:4].copy_(torch.tensor(list(word.to_bytes(4, "little")), dtype=torch.uint8))
        assert mosa.mosa_check_status(shape, ws) == code, word
        assert mosa.mosa_check_status(shape, ws) == 0      # cleared by the read
        assert int(ws[:4].sum().item()) == 0


def test_workspace_reuse_gives_same_result():
    cfg = W.CONFIGS["B8_T1024_d512_H16_k128"].with_(B=2)
    x = W.make_inputs(cfg)
    a = run_layer(cfg, x)
    b = run_layer(cfg, x)
    np.testing.assert_array_equal(a["I"], b["I"])
    for n in ("Y", "dX", "dW_q", "dW_o", "dW_r"):
        np.testing.assert_allclose(a[n], b[n], rtol=1e-5, atol=1e-6)


@pytest.mark.parametrize("name", ["largek_bf16", "pack2_oddB_bf16"])
def test_stage_kernel_spans_inside_event_windows(name):
    # The kernel spans (first CTA start to last CTA end, stamped by the kernels
    # themselves) of every tensor-core stage lie inside that stage's CUDA-event
    # window, and timing leaves the results unchanged.
    cfg = next(c for c in SMALL if c.name == name)
    x = W.make_inputs(cfg)
    plain = run_layer(cfg, x)
    dt = cfg.dtype
    X, Wr, Wq, Wk, Wv, Wo = (to_dev(x[n], dt) for n in ("X", "Wr", "Wq", "Wk", "Wv", "Wo"))
    dY = to_dev(x["dY"], dt)
    shape = mosa.make_shape(X, Wq, cfg.k)
    impl = mosa.stage_impl(shape)
    mosa.mosa_profile_read()
    mosa.mosa_profile_stages(0xFFFF)
    try:
        Y, I, rs, _, ws = mosa.mosa_forward(X, Wr, Wq, Wk, Wv, Wo, cfg.k)
        g = mosa.mosa_backward(X, Wr, Wq, Wk, Wv, Wo, I, rs, dY, ws)
        torch.cuda.synchronize()
        events = mosa.mosa_profile_read()
        spans = mosa.mosa_profile_spans(shape, ws)
        slots = torch.zeros(32, dtype=torch.int64, device="cuda")
        mosa.mosa_profile_spans_copy(shape, ws, slots)
        torch.cuda.synchronize()
    finally:
        mosa.mosa_profile_stages(0)
    # the device-side copy holds the same slots the synchronous read decoded
    # (slots decoded as the library does: unsigned, start all ones or end 0 or
    # end before start mean no record; unused slots hold whatever was there)
    sl = slots.cpu().numpy()
    m64 = (1 << 64) - 1
    for i in range(12):
        name = mosa.mosa_stage_name(i)
        a, b = int(sl[2 * i]) & m64, int(sl[2 * i + 1]) & m64
        if a != m64 and b != 0 and b >= a:
            assert abs((b - a) * 1e-6 - spans[name]) < 1e-9, (name, a, b, spans[name])
        else:
            assert spans[name] == -1.0, (name, spans[name])
    assert mosa.mosa_check_status(shape, ws) == 0
    np.testing.assert_array_equal(I.cpu().numpy(), plain["I"])
    np.testing.assert_allclose(Y.float().cpu().numpy(), plain["Y"], rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(g["dX"].float().cpu().numpy(), plain["dX"], rtol=1e-5, atol=1e-6)
    tensor = [s for s, e in impl.items() if e == "tensor" and events[s][1] > 0]
    assert tensor
    for s in tensor:
        assert 0.0 < spans[s] <= events[s][0] + 0.02, (s, spans[s], events[s])


@pytest.mark.parametrize("name", ["largek_bf16", "pack2_oddB_bf16"])
def test_timeline_mode_orders_the_stages_and_leaves_results_unchanged(name):
    # Timeline mode stamps every stage's kernel span with no events between
    # the kernels: each stage on the caller's stream starts after the one
    # before it ends (the early-launch wait holds its CTAs until then), every
    # tensor-core stage has a record, and the results are those of a plain run.
    cfg = next(c for c in SMALL if c.name == name)
    x = W.make_inputs(cfg)
    plain = run_layer(cfg, x)
    dt = cfg.dtype
    X, Wr, Wq, Wk, Wv, Wo = (to_dev(x[n], dt) for n in ("X", "Wr", "Wq", "Wk", "Wv", "Wo"))
    dY = to_dev(x["dY"], dt)
    shape = mosa.make_shape(X, Wq, cfg.k)
    impl = mosa.stage_impl(shape)
    mosa.mosa_profile_timeline(True)
    try:
        Y, I, rs, _, ws = mosa.mosa_forward(X, Wr, Wq, Wk, Wv, Wo, cfg.k)
        g = mosa.mosa_backward(X, Wr, Wq, Wk, Wv, Wo, I, rs, dY, ws)
        torch.cuda.synchronize()
        tl = mosa.mosa_profile_timeline_read(shape, ws)
    finally:
        mosa.mosa_profile_timeline(False)
    assert mosa.mosa_check_status(shape, ws) == 0
    np.testing.assert_array_equal(I.cpu().numpy(), plain["I"])
    np.testing.assert_allclose(Y.float().cpu().numpy(), plain["Y"], rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(g["dX"].float().cpu().numpy(), plain["dX"], rtol=1e-5, atol=1e-6)
    fwd = ["fwd_unit"] if cfg.k <= 128 else ["qkv", "attn_fwd", "out"]
    for s in fwd + ["select", "out_bwd", "attn_bwd", "in_bwd", "w_bwd", "dwo"]:
        assert s in tl, (s, tl)
    if impl.get("router") == "tensor":
        assert "router" in tl, tl
    main = [s for s in ("router", "select", "qkv", "attn_fwd", "out", "fwd_unit", "out_bwd",
                        "attn_bwd", "in_bwd") if s in tl]
    for a, b in zip(main, main[1:]):
        assert tl[b][0] >= tl[a][1] - 0.5, (a, b, tl)
    assert min(v[0] for v in tl.values()) == 0.0


def test_router_wait_limit_gives_up_then_next_call_is_exact(monkeypatch):
    # The router GEMM's main-loop waits get a 1 us limit: its epilogue waits
    # for the whole 128-block K loop (d = 8192), gives up, stops the producer
    # and the MMA issuer, lets the copies and MMAs in flight finish, and the
    # status word reads MOSA_ERR_DEVICE_TIMEOUT.  The same workspace then gives
    # the oracle's results on the next (normal) call.
    cfg = W.MosaConfig("router_wait_bf16", B=1, T=256, d=8192, H=8, hp=64, k=32, dtype="bf16",
                       seed=41)
    x = W.make_inputs(cfg)
    Y, I, rs, rf = oracle.forward(x["X"], *weights(x), k=cfg.k)
    assert sigmoid_gap(rf, cfg.k) > 1e-3
    X, Wr, Wq, Wk, Wv, Wo = (to_dev(x[n], cfg.dtype) for n in ("X", "Wr", "Wq", "Wk", "Wv", "Wo"))
    shape = mosa.make_shape(X, Wq, cfg.k)
    assert mosa.stage_impl(shape)["router"] == "tensor"
    _, _, _, rf0, ws = mosa.mosa_forward(X, Wr, Wq, Wk, Wv, Wo, cfg.k, want_r_full=True)
    torch.cuda.synchronize()
    assert mosa.mosa_check_status(shape, ws) == 0
    monkeypatch.setenv("MOSA_GRAPHS", "0")
    monkeypatch.setenv("MOSA_TEST_ROUTER_WAIT_NS", "1000")
    mosa.mosa_forward(X, Wr, Wq, Wk, Wv, Wo, cfg.k, workspace=ws, want_r_full=True,
                      out={"r_full": rf0})
    torch.cuda.synchronize()
    assert mosa.mosa_check_status(shape, ws) == 4          # MOSA_ERR_DEVICE_TIMEOUT
    monkeypatch.delenv("MOSA_TEST_ROUTER_WAIT_NS")
    monkeypatch.delenv("MOSA_GRAPHS")
    Yg, Ig, rsg, rfg, _ = mosa.mosa_forward(X, Wr, Wq, Wk, Wv, Wo, cfg.k, workspace=ws,
                                            want_r_full=True)
    torch.cuda.synchronize()
    assert mosa.mosa_check_status(shape, ws) == 0
    np.testing.assert_array_equal(Ig.cpu().numpy(), I)
    assert_close("r_full", rfg.cpu().numpy(), rf, cfg.dtype)
    assert_close("r_sel", rsg.cpu().numpy(), rs, cfg.dtype)
    assert_close("Y", Yg.cpu().numpy(), Y, cfg.dtype)


def test_token_major_products_equal_row_major_at_full_size(monkeypatch):
    # B4 T4096 d1024 H8 k2048, every head keeping half the tokens: Y and dX
    # from the token-major products (each head's rows of a token tile summed
    # in TMEM, written once) and from the row-major products (each head's rows
    # scatter-added) are the same sums in another order.
    cfg = W.CONFIGS["B4_T4096_d1024_H8_k2048"]
    x = W.make_inputs(cfg)
    monkeypatch.setenv("MOSA_HEADSUM", "1")
    a = run_layer(cfg, x)
    monkeypatch.setenv("MOSA_HEADSUM", "0")
    b = run_layer(cfg, x)
    np.testing.assert_array_equal(a["I"], b["I"])
    from _util import rel_l2
    for n in ("Y", "dX"):
        assert rel_l2(a[n], b[n]) < 1e-5, n
        assert np.abs(a[n] - b[n]).max() < 1e-4, n
