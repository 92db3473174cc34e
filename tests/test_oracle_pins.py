"""Pins for the CPU oracle: each check ties it to something other than itself.

  - TopK against brute force (a full stable sort) with crafted ties.
  - k = T: the layer reduces to dense causal multi-head attention (Sec. 2.1,
    Eq. mha) with each token's output scaled by its router score, checked
    against torch's float64 scaled_dot_product_attention (a library routine).
  - Fixed sparse attention (Sec. 3.1): I = [0, rho, ...], r = 1 is dense causal
    attention on X[::rho], scattered back.
  - H = 1, k = 1 closed form: the only row is r x W^V W^O.
  - Invariants: indices unique / ascending / in range, untouched rows zero,
    per-head support, order of I irrelevant, batches independent, Y linear
    in W^O.
  - Backward: central finite differences of sum(Y * dY) with TopK held
    constant, and torch float64 autograd through a gather / einsum / scatter
    restatement of the forward (the operations Sec. 2.2 names).
  - Sampled evaluation (batch/head masks) agrees with the full evaluation.
  - The App. A FLOP model reproduces the paper's printed head counts.
"""
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from paper_2505_00315_gb300 import flops
from paper_2505_00315_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def small(B, T, d, H, hp, k, seed=0, plant=True, dtype="f32"):
    cfg = W.MosaConfig("t", B=B, T=T, d=d, H=H, hp=hp, k=k, dtype=dtype, seed=seed)
    return cfg, W.make_inputs(cfg, plant=plant)


def weights(x):
    return x["Wr"], x["Wq"], x["Wk"], x["Wv"], x["Wo"]


# ---------------------------------------------------------------- TopK ----

def brute_topk(row, k):
    order = sorted(range(len(row)), key=lambda t: (-row[t], t))[:k]
    return sorted(order)


@pytest.mark.parametrize("seed", range(20))
def test_topk_matches_full_sort(seed):
    rng = np.random.default_rng(seed)
    T = int(rng.integers(1, 60))
    k = int(rng.integers(1, T + 1))
    if seed % 3 == 0:
        row = rng.choice([0.1, 0.25, 0.5, 0.75], size=T)      # heavy ties
    elif seed % 3 == 1:
        row = rng.random(T)
    else:
        row = np.round(rng.random(T), 1)                         # ties at threshold
    I, rs = oracle.topk(row, k)
    assert list(I) == brute_topk(list(row), k)
    np.testing.assert_array_equal(rs, row[I])


def test_topk_all_equal_takes_lowest_indices():
    I, _ = oracle.topk(np.full(17, 0.3), 5)
    assert list(I) == [0, 1, 2, 3, 4]


def test_topk_threshold_ties_prefer_lower_index():
    row = np.array([0.9, 0.5, 0.2, 0.5, 0.5, 0.1, 0.5])
    I, rs = oracle.topk(row, 3)
    assert list(I) == [0, 1, 3]
    np.testing.assert_array_equal(rs, [0.9, 0.5, 0.5])


def test_topk_k_equals_T_and_bad_k():
    row = np.random.default_rng(1).random(9)
    I, _ = oracle.topk(row, 9)
    assert list(I) == list(range(9))
    with pytest.raises(ValueError):
        oracle.topk(row, 10)
    with pytest.raises(ValueError):
        oracle.topk(row, 0)


# Sec. 3.2: every head keeps the first token and selects k-1 more by score.

@pytest.mark.parametrize("seed", range(16))
def test_topk_first_token_matches_definition(seed):
    rng = np.random.default_rng(100 + seed)
    T = int(rng.integers(1, 60))
    k = int(rng.integers(1, T + 1))
    row = rng.choice([0.1, 0.25, 0.5, 0.75], size=T) if seed % 2 else rng.random(T)
    I, rs = oracle.topk(row, k, first_token=True)
    rest = sorted(range(1, T), key=lambda t: (-row[t], t))[:k - 1]
    assert list(I) == [0] + sorted(rest)
    np.testing.assert_array_equal(rs, row[I])


def test_topk_first_token_special_cases():
    row = np.array([0.1, 0.9, 0.5, 0.9, 0.2, 0.9])
    assert list(oracle.topk(row, 1, first_token=True)[0]) == [0]
    assert list(oracle.topk(row, 6, first_token=True)[0]) == list(range(6))
    # token 0 would lose the plain TopK: it is kept anyway, ties below go to lower indices
    assert list(oracle.topk(row, 3, first_token=True)[0]) == [0, 1, 3]
    assert list(oracle.topk(row, 3)[0]) == [1, 3, 5]
    # token 0 already the largest: both rules agree
    top = np.array([0.95, 0.2, 0.7, 0.1, 0.6])
    for k in range(1, 6):
        assert list(oracle.topk(top, k, first_token=True)[0]) == list(oracle.topk(top, k)[0])


def test_forward_first_token_is_forward_on_its_token_sets():
    cfg = W.MosaConfig("first", B=2, T=40, d=16, H=3, hp=8, k=6, dtype="f32", seed=7,
                       first_token=True)
    x = W.make_inputs(cfg)
    w = [x[n] for n in ("Wr", "Wq", "Wk", "Wv", "Wo")]
    Y, I, rs, rf = oracle.forward(x["X"], *w, k=cfg.k, first_token=True)
    assert (I[:, :, 0] == 0).all()
    for b in range(cfg.B):
        for h in range(cfg.H):
            Iref, rsref = oracle.topk(rf[b, h], cfg.k, first_token=True)
            np.testing.assert_array_equal(I[b, h], Iref)
            np.testing.assert_array_equal(rs[b, h], rsref)
    Y2 = oracle.forward_indices(x["X"], *w, I=I)
    np.testing.assert_allclose(Y, Y2, rtol=0, atol=1e-12)


def test_planted_margin_with_first_token():
    cfg = W.MosaConfig("first", B=2, T=300, d=64, H=4, hp=16, k=37, dtype="bf16", seed=9,
                       first_token=True)
    x = W.make_inputs(cfg)
    rf = oracle.router(x["X"], x["Wr"])
    s = -np.sort(-rf[..., 1:], axis=-1)
    assert float(np.min(s[..., cfg.k - 2] - s[..., cfg.k - 1])) > 1e-3


# ----------------------------------------------------- forward reductions ----

def dense_causal_mha_scaled(X, Wr, Wq, Wk, Wv, Wo):
    """Eq. (mha) with causal mask via torch SDPA, each head's output row t
    scaled by sigma(X_t W^r_h) before W^O (k = T special case of Sec. 2.2)."""
    Xt = torch.tensor(X, dtype=torch.float64)
    Y = torch.zeros_like(Xt)
    for h in range(Wq.shape[0]):
        q = Xt @ torch.tensor(Wq[h], dtype=torch.float64)
        kk = Xt @ torch.tensor(Wk[h], dtype=torch.float64)
        v = Xt @ torch.tensor(Wv[h], dtype=torch.float64)
        a = F.scaled_dot_product_attention(q, kk, v, is_causal=True)
        r = torch.sigmoid(Xt @ torch.tensor(Wr[:, h], dtype=torch.float64))
        Y += r[..., None] * (a @ torch.tensor(Wo[h], dtype=torch.float64))
    return Y.numpy()


@pytest.mark.parametrize("shape", [(2, 12, 8, 3, 4), (1, 7, 5, 2, 3), (3, 16, 16, 1, 8)])
def test_k_equals_T_is_dense_causal_mha(shape):
    B, T, d, H, hp = shape
    _, x = small(B, T, d, H, hp, T, seed=3, plant=False)
    Y, I, rs, rf = oracle.forward(x["X"], *weights(x), k=T)
    assert (I == np.arange(T)[None, None, :]).all()
    np.testing.assert_array_equal(rs, rf)
    ref = dense_causal_mha_scaled(x["X"], *weights(x))
    np.testing.assert_allclose(Y, ref, rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("rho", [2, 4, 8])
def test_fixed_sparse_is_dense_attention_on_strided_tokens(rho):
    B, T, d, H, hp = 2, 32, 8, 3, 4
    k = T // rho
    _, x = small(B, T, d, H, hp, k, seed=4, plant=False)
    I = W.fixed_sparse_indices(B, H, T, k)
    Y = oracle.forward_indices(x["X"], *weights(x), I=I, r_sel=np.ones((B, H, k)))
    Xs = torch.tensor(x["X"][:, ::rho, :], dtype=torch.float64)
    ref = torch.zeros((B, T, d), dtype=torch.float64)
    for h in range(H):
        q = Xs @ torch.tensor(x["Wq"][h], dtype=torch.float64)
        kk = Xs @ torch.tensor(x["Wk"][h], dtype=torch.float64)
        v = Xs @ torch.tensor(x["Wv"][h], dtype=torch.float64)
        a = F.scaled_dot_product_attention(q, kk, v, is_causal=True)
        ref[:, ::rho, :] += a @ torch.tensor(x["Wo"][h], dtype=torch.float64)
    np.testing.assert_allclose(Y, ref.numpy(), rtol=1e-11, atol=1e-12)


def test_single_head_single_token_closed_form():
    B, T, d, hp = 2, 9, 6, 4
    _, x = small(B, T, d, 1, hp, 1, seed=5, plant=False)
    Y, I, rs, rf = oracle.forward(x["X"], *weights(x), k=1)
    X64 = x["X"].astype(np.float64)
    for b in range(B):
        t = int(np.argmax(rf[b, 0]))          # argmax returns the first maximum
        assert I[b, 0, 0] == t
        expect = np.zeros((T, d))
        expect[t] = rs[b, 0, 0] * (X64[b, t] @ x["Wv"][0].astype(np.float64)
                                   @ x["Wo"][0].astype(np.float64))
        np.testing.assert_allclose(Y[b], expect, rtol=1e-12, atol=1e-14)


# ------------------------------------------------------------ invariants ----

@pytest.fixture(scope="module")
def mid_case():
    cfg, x = small(3, 64, 16, 5, 8, 12, seed=6)
    Y, I, rs, rf = oracle.forward(x["X"], *weights(x), k=cfg.k)
    return cfg, x, Y, I, rs, rf


def test_indices_unique_ascending_in_range(mid_case):
    cfg, _, _, I, rs, rf = mid_case
    assert I.min() >= 0 and I.max() < cfg.T
    assert (np.diff(I, axis=-1) > 0).all()
    np.testing.assert_array_equal(rs, np.take_along_axis(rf, I.astype(np.int64), axis=-1))


def test_selected_scores_dominate_rest(mid_case):
    cfg, _, _, I, _, rf = mid_case
    for b in range(cfg.B):
        for h in range(cfg.H):
            sel = np.zeros(cfg.T, bool)
            sel[I[b, h]] = True
            assert rf[b, h, sel].min() >= rf[b, h, ~sel].max()


def test_unselected_rows_are_zero(mid_case):
    cfg, _, Y, I, _, _ = mid_case
    for b in range(cfg.B):
        touched = np.zeros(cfg.T, bool)
        touched[I[b].ravel()] = True
        assert (Y[b, ~touched] == 0).all()
        assert np.abs(Y[b, touched]).sum(axis=1).min() > 0


def test_per_head_support(mid_case):
    cfg, x, _, I, _, _ = mid_case
    for h in range(cfg.H):
        Yh, _, _, _ = oracle.forward(x["X"], *weights(x), k=cfg.k, heads=[h])
        for b in range(cfg.B):
            outside = np.ones(cfg.T, bool)
            outside[I[b, h]] = False
            assert (Yh[b, outside] == 0).all()


def test_heads_sum(mid_case):
    """Eq. (mosa_mha): the layer is the sum of the single-head layers."""
    cfg, x, Y, _, _, _ = mid_case
    acc = np.zeros_like(Y)
    for h in range(cfg.H):
        acc += oracle.forward(x["X"], *weights(x), k=cfg.k, heads=[h])[0]
    np.testing.assert_allclose(acc, Y, rtol=1e-12, atol=1e-13)


def test_order_of_indices_is_irrelevant(mid_case):
    cfg, x, Y, I, rs, _ = mid_case
    rng = np.random.default_rng(0)
    perm = np.stack([np.stack([rng.permutation(cfg.k) for _ in range(cfg.H)])
                     for _ in range(cfg.B)])
    Ip = np.take_along_axis(I, perm, axis=-1)
    rp = np.take_along_axis(rs, perm, axis=-1)
    Yp = oracle.forward_indices(x["X"], *weights(x), I=Ip, r_sel=rp)
    np.testing.assert_allclose(Yp, Y, rtol=1e-12, atol=1e-13)


def test_batches_independent(mid_case):
    cfg, x, Y, _, _, _ = mid_case
    X2 = x["X"].copy()
    X2[1] = np.random.default_rng(9).standard_normal(X2[1].shape)
    Y2, _, _, _ = oracle.forward(X2, *weights(x), k=cfg.k)
    np.testing.assert_allclose(Y2[0], Y[0], rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(Y2[2], Y[2], rtol=1e-13, atol=1e-15)
    assert not np.allclose(Y2[1], Y[1])


def test_linear_in_output_weights(mid_case):
    cfg, x, Y, _, _, _ = mid_case
    Wo2 = np.random.default_rng(2).standard_normal(x["Wo"].shape) * 0.1
    Ya = oracle.forward(x["X"], x["Wr"], x["Wq"], x["Wk"], x["Wv"], Wo2, k=cfg.k)[0]
    Yb = oracle.forward(x["X"], x["Wr"], x["Wq"], x["Wk"], x["Wv"], x["Wo"] + Wo2, k=cfg.k)[0]
    np.testing.assert_allclose(Yb, Y + Ya, rtol=1e-10, atol=1e-12)


def test_sampled_units_match_full(mid_case):
    cfg, x, Y, I, _, _ = mid_case
    Yb = oracle.forward(x["X"], *weights(x), k=cfg.k, batches=[1])[0]
    np.testing.assert_allclose(Yb[1], Y[1], rtol=1e-13, atol=1e-15)
    assert (Yb[0] == 0).all()
    dY = x["dY"]
    g = oracle.backward(x["X"], *weights(x), I=I, dY=dY)
    gh = oracle.backward(x["X"], *weights(x), I=I, dY=dY, heads=[2])
    for name in ("dWq", "dWk", "dWv", "dWo"):
        np.testing.assert_allclose(gh[name][2], g[name][2], rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(gh["dWr"][:, 2], g["dWr"][:, 2], rtol=1e-12, atol=1e-14)
    gb = oracle.backward(x["X"], *weights(x), I=I, dY=dY, batches=[0])
    np.testing.assert_allclose(gb["dX"][0], g["dX"][0], rtol=1e-12, atol=1e-14)


def test_planted_margin_gives_clear_gap():
    for B, T, d, H, k in [(2, 256, 64, 8, 32), (1, 1024, 128, 16, 64)]:
        cfg, x = small(B, T, d, H, 16, k, seed=11, dtype="bf16")
        rf = oracle.router(x["X"], x["Wr"])
        s = -np.sort(-rf, axis=-1)
        assert (s[..., k - 1] - s[..., k]).min() > 1e-3


# -------------------------------------------------------------- backward ----

def loss_fixed_I(x, I, overrides=None):
    p = dict(x)
    if overrides:
        p.update(overrides)
    Y = oracle.forward_indices(p["X"], p["Wr"], p["Wq"], p["Wk"], p["Wv"], p["Wo"], I=I)
    return float(np.sum(Y * x["dY"].astype(np.float64)))


@pytest.mark.parametrize("seed", [0, 1])
def test_backward_matches_finite_differences(seed):
    cfg, x = small(2, 10, 6, 2, 4, 4, seed=20 + seed, plant=False)
    x = {n: v.astype(np.float64) for n, v in x.items()}
    _, I, _, _ = oracle.forward(x["X"], *weights(x), k=cfg.k)
    g = oracle.backward(x["X"], *weights(x), I=I, dY=x["dY"])
    eps = 1e-6
    for name, gname in [("X", "dX"), ("Wr", "dWr"), ("Wq", "dWq"), ("Wk", "dWk"),
                        ("Wv", "dWv"), ("Wo", "dWo")]:
        base = x[name]
        num = np.zeros_like(base)
        it = np.nditer(base, flags=["multi_index"])
        for _ in it:
            idx = it.multi_index
            plus, minus = base.copy(), base.copy()
            plus[idx] += eps
            minus[idx] -= eps
            num[idx] = (loss_fixed_I(x, I, {name: plus}) - loss_fixed_I(x, I, {name: minus})) / (2 * eps)
        scale = max(np.abs(num).max(), 1e-3)
        assert np.abs(num - g[gname]).max() / scale < 1e-6, name


def rope_complex(Z, pos):
    """RoPE as complex multiplication: the first h'/2 entries of each row of Z
    [..., k, h'] read as h'/4 complex numbers (2p + i (2p+1)), each multiplied
    by exp(i pos theta_p), theta_p = 10000^(-2p / (h'/2)); the rest unchanged."""
    hp = Z.shape[-1]
    half = hp // 2
    p = torch.arange(half // 2, dtype=torch.float64)
    theta = 10000.0 ** (-2.0 * p / half)
    ang = pos[..., None].to(torch.float64) * theta
    zc = torch.view_as_complex(Z[..., :half].reshape(*Z.shape[:-1], half // 2, 2).contiguous())
    rot = torch.view_as_real(zc * torch.polar(torch.ones_like(ang), ang))
    return torch.cat([rot.reshape(*Z.shape[:-1], half), Z[..., half:]], dim=-1)


def torch_restatement(X, Wr, Wq, Wk, Wv, Wo, I, rope=False):
    """Forward written with gather / einsum / scatter_add on float64 tensors."""
    B, T, d = X.shape
    H, _, hp = Wq.shape
    k = I.shape[-1]
    idx = I.long()
    logits = torch.einsum("btc,ch->bht", X, Wr)
    r_sel = torch.gather(torch.sigmoid(logits), 2, idx)                      # [B,H,k]
    Xs = torch.gather(X[:, None].expand(B, H, T, d), 2, idx[..., None].expand(B, H, k, d))
    Q = torch.einsum("bhkc,hcp->bhkp", Xs, Wq)
    K = torch.einsum("bhkc,hcp->bhkp", Xs, Wk)
    V = torch.einsum("bhkc,hcp->bhkp", Xs, Wv)
    if rope:
        Q, K = rope_complex(Q, idx), rope_complex(K, idx)
    S = torch.einsum("bhip,bhjp->bhij", Q, K) / np.sqrt(hp)
    allowed = idx[..., :, None] >= idx[..., None, :]
    S = S.masked_fill(~allowed, float("-inf"))
    A = torch.einsum("bhij,bhjp->bhip", torch.softmax(S, dim=-1), V)
    Xo = r_sel[..., None] * torch.einsum("bhip,hpc->bhic", A, Wo)
    Y = torch.zeros(B, T, d, dtype=X.dtype)
    Y.scatter_add_(1, idx.reshape(B, H * k)[..., None].expand(B, H * k, d),
                   Xo.reshape(B, H * k, d))
    return Y


def test_backward_matches_torch_autograd():
    cfg, x = small(2, 40, 12, 3, 8, 9, seed=30)
    _, I, _, _ = oracle.forward(x["X"], *weights(x), k=cfg.k)
    ts = {n: torch.tensor(v, dtype=torch.float64, requires_grad=(n != "dY"))
          for n, v in x.items()}
    Y = torch_restatement(ts["X"], ts["Wr"], ts["Wq"], ts["Wk"], ts["Wv"], ts["Wo"],
                          torch.tensor(I))
    Yo = oracle.forward_indices(x["X"], *weights(x), I=I)
    np.testing.assert_allclose(Y.detach().numpy(), Yo, rtol=1e-11, atol=1e-12)
    (Y * ts["dY"]).sum().backward()
    g = oracle.backward(x["X"], *weights(x), I=I, dY=x["dY"])
    for name in ("X", "Wr", "Wq", "Wk", "Wv", "Wo"):
        np.testing.assert_allclose(g["d" + name], ts[name].grad.numpy(), rtol=1e-10,
                                   atol=1e-11, err_msg=name)


# ------------------------------------------------------------ FLOP model ----

def read_golden():
    heads, models = [], {}
    with open(os.path.join(GOLDEN, "isoflop_table.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            p = line.split()
            if p[0] == "heads":
                heads.append((p[1], p[2], p[3:]))
            else:
                models[p[1]] = dict(layers=int(p[2]), h=int(p[3]), hp=int(p[4]),
                                    heads=int(p[5]), gflops=float(p[6]))
    return heads, models


def test_flop_model_reproduces_dense_totals():
    _, models = read_golden()
    for name, m in models.items():
        total = flops.model_forward_flops(m["layers"], m["h"], m["hp"], 1024, m["heads"], 0, 0)
        if name == "Medium":
            assert round(total / 1e9, 2) == 439.70    # printed 430.70: read as a typo
        else:
            assert round(total / 1e9, 2) == m["gflops"], name


def test_flop_model_reproduces_isoflop_head_counts():
    heads, models = read_golden()
    for name, kind, row in heads:
        m = models[name]
        for rho, printed in zip([1, 2, 4, 8, 16, 32, 64, 128, 256], row):
            if printed == "-":
                continue
            n = flops.isoflop_heads(m["layers"], m["h"], m["hp"], 1024, m["heads"], rho,
                                    n_dense=4 if kind == "MoSA" else 0)
            assert n == int(printed), (name, kind, rho)


def test_layer_work_matches_head_formula_without_causal_halving():
    """With the paper's 4h'k^2 attention count, the per-head forward work of
    layer_work equals the App. A MoSA head cost minus the h'k scaling term."""
    B, T, d, H, hp, k = 2, 1024, 512, 4, 64, 128
    w = flops.layer_work(B, T, d, H, hp, k)
    mine = w["forward_flops"] - w["attn_fwd"]["flops"] + 4 * hp * k * k * B * H
    paper = flops.head_flops_mosa(d, hp, T, k) * B * H - hp * k * B * H
    assert mine == paper


# ------------------------------------------------ RoPE (Sec. 2.2) ----

@pytest.mark.parametrize("hp", [4, 8, 16])
def test_rope_forward_backward_match_complex_restatement(hp):
    cfg, x = small(2, 40, 12, 3, hp, 9, seed=40 + hp)
    _, I, _, _ = oracle.forward(x["X"], *weights(x), k=cfg.k)
    ts = {n: torch.tensor(v, dtype=torch.float64, requires_grad=(n != "dY"))
          for n, v in x.items()}
    Y = torch_restatement(ts["X"], ts["Wr"], ts["Wq"], ts["Wk"], ts["Wv"], ts["Wo"],
                          torch.tensor(I), rope=True)
    Yo = oracle.forward_indices(x["X"], *weights(x), I=I, rope=True)
    np.testing.assert_allclose(Y.detach().numpy(), Yo, rtol=1e-11, atol=1e-12)
    (Y * ts["dY"]).sum().backward()
    g = oracle.backward(x["X"], *weights(x), I=I, dY=x["dY"], rope=True)
    for name in ("X", "Wr", "Wq", "Wk", "Wv", "Wo"):
        np.testing.assert_allclose(g["d" + name], ts[name].grad.numpy(), rtol=1e-10,
                                   atol=1e-11, err_msg=name)


def test_rope_changes_only_through_positions():
    # the rotation is a function of the original positions: the same token set
    # with RoPE differs from the set without it, and k = T with RoPE equals
    # dense causal attention on rotated queries and keys (positions 0..T-1)
    B, T, d, H, hp = 1, 24, 16, 2, 8
    _, x = small(B, T, d, H, hp, T, seed=5, plant=False)
    Y, I, rs, rf = oracle.forward(x["X"], *weights(x), k=T, rope=True)
    Y0, _, _, _ = oracle.forward(x["X"], *weights(x), k=T)
    assert np.abs(Y - Y0).max() > 1e-3
    Xt = torch.tensor(x["X"], dtype=torch.float64)
    ref = torch.zeros_like(Xt)
    pos = torch.arange(T)
    for h in range(H):
        q = rope_complex(Xt @ torch.tensor(x["Wq"][h], dtype=torch.float64), pos)
        kk = rope_complex(Xt @ torch.tensor(x["Wk"][h], dtype=torch.float64), pos)
        v = Xt @ torch.tensor(x["Wv"][h], dtype=torch.float64)
        a = F.scaled_dot_product_attention(q, kk, v, is_causal=True)
        r = torch.sigmoid(Xt @ torch.tensor(x["Wr"][:, h], dtype=torch.float64))
        ref += r[..., None] * (a @ torch.tensor(x["Wo"][h], dtype=torch.float64))
    np.testing.assert_allclose(Y, ref.numpy(), rtol=1e-10, atol=1e-12)


# ---------------------------------- hybrid layers (Sec. 2.2 hybridization, Sec. 3.4) ----

def dense_heads_sdpa(X, Dq, Dk, Dv, Do, window=0, rope=False):
    """Eq. (mha) over all T tokens with torch's SDPA and an explicit boolean
    mask: query i sees key j iff j <= i and, for a window w > 0, floor(i/w) =
    floor(j/w).  float64 tensors in and out, differentiable."""
    T = X.shape[1]
    pos = torch.arange(T)
    allowed = pos[:, None] >= pos[None, :]
    if window:
        allowed = allowed & ((pos[:, None] // window) == (pos[None, :] // window))
    Y = torch.zeros_like(X)
    for h in range(Dq.shape[0]):
        q, kk, v = X @ Dq[h], X @ Dk[h], X @ Dv[h]
        if rope:
            q, kk = rope_complex(q, pos), rope_complex(kk, pos)
        Y = Y + F.scaled_dot_product_attention(q, kk, v, attn_mask=allowed) @ Do[h]
    return Y


def dense_inputs(B, T, d, H, hp, Hd, seed):
    cfg, x = small(B, T, d, H, hp, max(1, T // 4), seed=seed)
    x.update(W.make_dense_weights(cfg, Hd))
    return cfg, x


@pytest.mark.parametrize("window,rope", [(0, False), (0, True), (4, False), (5, True),
                                         (18, False)])
def test_dense_heads_match_sdpa_forward_and_autograd(window, rope):
    # T = 18 with w = 4 or 5 leaves a shorter last block
    _, x = dense_inputs(2, 18, 12, 2, 8, 3, seed=50 + window)
    D = [x[n] for n in ("Dq", "Dk", "Dv", "Do")]
    ts = {n: torch.tensor(x[n], dtype=torch.float64, requires_grad=(n != "dY"))
          for n in ("X", "Dq", "Dk", "Dv", "Do", "dY")}
    Y = dense_heads_sdpa(ts["X"], ts["Dq"], ts["Dk"], ts["Dv"], ts["Do"], window, rope)
    Yo = oracle.dense_forward(x["X"], *D, window=window, rope=rope)
    np.testing.assert_allclose(Yo, Y.detach().numpy(), rtol=1e-11, atol=1e-12)
    (Y * ts["dY"]).sum().backward()
    g = oracle.dense_backward(x["X"], *D, dY=x["dY"], window=window, rope=rope)
    for name, tname in (("dX", "X"), ("dWq", "Dq"), ("dWk", "Dk"), ("dWv", "Dv"),
                        ("dWo", "Do")):
        np.testing.assert_allclose(g[name], ts[tname].grad.numpy(), rtol=1e-10, atol=1e-11,
                                   err_msg=name)


def test_local_window_one_is_the_value_path():
    # w = 1: each token sees only itself, softmax of one entry is 1, so
    # Y = sum_h X D_v[h] D_o[h] whatever the queries and keys
    _, x = dense_inputs(2, 11, 8, 1, 4, 3, seed=60)
    Y = oracle.dense_forward(x["X"], x["Dq"], x["Dk"], x["Dv"], x["Do"], window=1, rope=True)
    X64 = x["X"].astype(np.float64)
    ref = sum(X64 @ x["Dv"][h].astype(np.float64) @ x["Do"][h].astype(np.float64)
              for h in range(3))
    np.testing.assert_allclose(Y, ref, rtol=1e-12, atol=1e-13)


def test_local_heads_are_blockwise_dense_heads_with_rope():
    # RoPE scores depend on position differences only, so local heads at the
    # original positions equal dense heads run on each block as its own
    # sequence from position 0 (the form the CUDA library computes them in)
    B, T, w = 2, 24, 8
    _, x = dense_inputs(B, T, 16, 1, 8, 2, seed=61)
    D = [x[n] for n in ("Dq", "Dk", "Dv", "Do")]
    Y = oracle.dense_forward(x["X"], *D, window=w, rope=True)
    Xb = x["X"].reshape(B * T // w, w, -1)
    Yb = oracle.dense_forward(Xb, *D, window=0, rope=True).reshape(B, T, -1)
    np.testing.assert_allclose(Y, Yb, rtol=1e-10, atol=1e-12)
    g = oracle.dense_backward(x["X"], *D, dY=x["dY"], window=w, rope=True)
    gb = oracle.dense_backward(Xb, *D, dY=x["dY"].reshape(B * T // w, w, -1), rope=True)
    np.testing.assert_allclose(g["dX"], gb["dX"].reshape(B, T, -1), rtol=1e-10, atol=1e-12)
    for n in ("dWq", "dWk", "dWv", "dWo"):
        np.testing.assert_allclose(g[n], gb[n], rtol=1e-10, atol=1e-12, err_msg=n)
    # and they differ from dense heads over the whole sequence
    assert np.abs(Y - oracle.dense_forward(x["X"], *D, rope=True)).max() > 1e-3


@pytest.mark.parametrize("window,rope", [(0, False), (6, True)])
def test_hybrid_layer_matches_torch_restatement(window, rope):
    cfg, x = dense_inputs(2, 24, 12, 3, 8, 2, seed=62 + window)
    Y, I, _, _ = oracle.hybrid_forward(x["X"], *weights(x), x["Dq"], x["Dk"], x["Dv"], x["Do"],
                                       k=cfg.k, window=window, rope=rope)
    names = ("X", "Wr", "Wq", "Wk", "Wv", "Wo", "Dq", "Dk", "Dv", "Do")
    ts = {n: torch.tensor(x[n], dtype=torch.float64, requires_grad=True) for n in names}
    Yt = (torch_restatement(ts["X"], ts["Wr"], ts["Wq"], ts["Wk"], ts["Wv"], ts["Wo"],
                            torch.tensor(I), rope=rope) +
          dense_heads_sdpa(ts["X"], ts["Dq"], ts["Dk"], ts["Dv"], ts["Do"], window, rope))
    np.testing.assert_allclose(Y, Yt.detach().numpy(), rtol=1e-11, atol=1e-12)
    (Yt * torch.tensor(x["dY"], dtype=torch.float64)).sum().backward()
    g = oracle.hybrid_backward(x["X"], *weights(x), x["Dq"], x["Dk"], x["Dv"], x["Do"], I=I,
                               dY=x["dY"], window=window, rope=rope)
    for n in names:
        np.testing.assert_allclose(g["d" + n], ts[n].grad.numpy(), rtol=1e-10, atol=1e-11,
                                   err_msg=n)


def test_hybrid_work_adds_dense_and_local_heads():
    # dense heads: every token, causal attention over T, no router terms;
    # local heads of w tokens: B*T/w sequences of w tokens
    B, T, d, H, hp, k, Hd = 2, 64, 32, 3, 16, 8, 2
    base = flops.layer_work(B, T, d, H, hp, k)
    assert flops.hybrid_work(B, T, d, H, hp, k, 0) == base
    for w, n_seq in ((0, B), (16, B * T // 16)):
        blk = w or T
        h = flops.hybrid_work(B, T, d, H, hp, k, Hd, w)
        U = n_seq * Hd
        assert h["router"] == base["router"]
        assert h["attn_fwd"]["flops"] - base["attn_fwd"]["flops"] == 2 * hp * blk * (blk + 1) * U
        assert h["qkv"]["flops"] - base["qkv"]["flops"] == 6 * d * hp * blk * U
        assert h["in_bwd"]["flops"] - base["in_bwd"]["flops"] == 6 * d * hp * blk * U
        assert h["w_bwd"]["flops"] - base["w_bwd"]["flops"] == 6 * d * hp * blk * U
        assert h["forward_flops"] == sum(h[s]["flops"] for s in
                                         ("router", "select", "qkv", "attn_fwd", "out"))


def test_paper_count_matches_app_a_head_formula():
    # with attention not halved for the mask, the layer's forward FLOPs are
    # App. A's MoSA head cost per (b, h) minus its h'k scaling term, which the
    # library's count leaves out
    B, T, d, H, hp, k = 2, 1024, 512, 16, 64, 128
    w = flops.layer_work(B, T, d, H, hp, k, causal=False)
    assert w["forward_flops"] + B * H * hp * k == B * H * flops.head_flops_mosa(d, hp, T, k)
    assert w["attn_bwd"]["flops"] == 10 * hp * k * k * B * H
    c = flops.layer_work(B, T, d, H, hp, k)
    assert c["attn_fwd"]["flops"] == 2 * hp * k * (k + 1) * B * H < w["attn_fwd"]["flops"]
