"""The binding's shape checks on CPU tensors: valid inputs pass every check
and stop at the first device-only step ("must be a CUDA tensor"); each
mis-shaped tensor stops at its shape check, before any pointer reaches the
library (which sees plain pointers and could not tell)."""
import pytest
import torch

from paper_2505_00315_gb300 import _binding as mb

B, T, d, H, hp, k, Hd = 2, 64, 48, 3, 32, 8, 2   # d != hp: W_o [H,hp,d] differs from [H,d,hp]
bf = torch.bfloat16


def layer(**over):
    t = {"X": torch.zeros(B, T, d, dtype=bf), "W_r": torch.zeros(d, H, dtype=bf),
         "W_q": torch.zeros(H, d, hp, dtype=bf), "W_k": torch.zeros(H, d, hp, dtype=bf),
         "W_v": torch.zeros(H, d, hp, dtype=bf), "W_o": torch.zeros(H, hp, d, dtype=bf),
         "D_q": torch.zeros(Hd, d, hp, dtype=bf), "D_k": torch.zeros(Hd, d, hp, dtype=bf),
         "D_v": torch.zeros(Hd, d, hp, dtype=bf), "D_o": torch.zeros(Hd, hp, d, dtype=bf),
         "I": torch.zeros(B, H, k, dtype=torch.int32), "r_sel": torch.zeros(B, H, k),
         "dY": torch.zeros(B, T, d, dtype=bf)}
    t.update(over)
    return t


def forward(t, out=None):
    return mb.mosa_forward(t["X"], t["W_r"], t["W_q"], t["W_k"], t["W_v"], t["W_o"], k, out=out)


def with_indices(t, out=None):
    return mb.mosa_forward_with_indices(t["X"], t["W_q"], t["W_k"], t["W_v"], t["W_o"], t["I"],
                                        t["r_sel"], out=out)


def backward(t, out=None):
    return mb.mosa_backward(t["X"], t["W_r"], t["W_q"], t["W_k"], t["W_v"], t["W_o"], t["I"],
                            t["r_sel"], t["dY"], torch.zeros(16, dtype=torch.uint8), out=out)


def hybrid_forward(t, out=None):
    return mb.mosa_hybrid_forward(t["X"], t["W_r"], t["W_q"], t["W_k"], t["W_v"], t["W_o"],
                                  t["D_q"], t["D_k"], t["D_v"], t["D_o"], k, window=16, out=out)


def hybrid_backward(t, out=None):
    return mb.mosa_hybrid_backward(t["X"], t["W_r"], t["W_q"], t["W_k"], t["W_v"], t["W_o"],
                                   t["D_q"], t["D_k"], t["D_v"], t["D_o"], t["I"], t["r_sel"],
                                   t["dY"], torch.zeros(16, dtype=torch.uint8), window=16,
                                   out=out)


CALLS = {"forward": forward, "with_indices": with_indices, "backward": backward,
         "hybrid_forward": hybrid_forward, "hybrid_backward": hybrid_backward}


@pytest.mark.parametrize("call", list(CALLS))
def test_valid_shapes_reach_the_device_step(call):
    with pytest.raises(ValueError, match="must be a CUDA tensor"):
        CALLS[call](layer())


BAD = {
    "W_r": torch.zeros(d, H + 1, dtype=bf), "W_k": torch.zeros(H, d, hp + 1, dtype=bf),
    "W_v": torch.zeros(H + 1, d, hp, dtype=bf), "W_o": torch.zeros(H, d, hp, dtype=bf),
    "dY": torch.zeros(B, T + 1, d, dtype=bf), "r_sel": torch.zeros(B, H, k + 1),
    "D_k": torch.zeros(Hd, d, hp + 1, dtype=bf), "D_o": torch.zeros(Hd, d, hp, dtype=bf),
}
USES = {"forward": ("W_r", "W_k", "W_v", "W_o"),
        "with_indices": ("W_k", "W_v", "W_o", "r_sel"),
        "backward": ("W_r", "W_k", "W_v", "W_o", "dY", "r_sel"),
        "hybrid_forward": ("W_r", "W_k", "W_o", "D_k", "D_o"),
        "hybrid_backward": ("W_r", "W_o", "dY", "r_sel", "D_k", "D_o")}


@pytest.mark.parametrize("call,name", [(c, n) for c, ns in USES.items() for n in ns])
def test_each_misshaped_input_is_refused(call, name):
    with pytest.raises(ValueError, match=f"{name} must have shape"):
        CALLS[call](layer(**{name: BAD[name]}))


@pytest.mark.parametrize("call,outs", [
    ("forward", {"Y": torch.zeros(B, T, d + 1)}),
    ("forward", {"I": torch.zeros(B, H, k + 1, dtype=torch.int32)}),
    ("with_indices", {"Y": torch.zeros(B, T - 1, d)}),
    ("backward", {"dW_o": torch.zeros(H, d, hp)}),
    ("backward", {"dX": torch.zeros(B, T, d + 8)}),
    ("hybrid_forward", {"r_sel": torch.zeros(B, H + 1, k)}),
    ("hybrid_backward", {"dD_o": torch.zeros(Hd, d, hp)}),
])
def test_misshaped_outputs_are_refused(call, outs):
    with pytest.raises(ValueError, match="must have shape"):
        CALLS[call](layer(), out=outs)


def test_valid_outputs_pass():
    outs = {"Y": torch.zeros(B, T, d), "I": torch.zeros(B, H, k, dtype=torch.int32),
            "r_sel": torch.zeros(B, H, k), "r_full": torch.zeros(B, H, T)}
    with pytest.raises(ValueError, match="must be a CUDA tensor"):
        forward(layer(), out=outs)
    grads = {"dX": torch.zeros(B, T, d), "dW_r": torch.zeros(d, H),
             "dW_q": torch.zeros(H, d, hp), "dW_k": torch.zeros(H, d, hp),
             "dW_v": torch.zeros(H, d, hp), "dW_o": torch.zeros(H, hp, d),
             "dD_q": torch.zeros(Hd, d, hp), "dD_k": torch.zeros(Hd, d, hp),
             "dD_v": torch.zeros(Hd, d, hp), "dD_o": torch.zeros(Hd, hp, d)}
    with pytest.raises(ValueError, match="must be a CUDA tensor"):
        hybrid_backward(layer(), out=grads)


def test_topk_and_route_outputs():
    with pytest.raises(ValueError, match="I must have shape"):
        mb.mosa_topk(torch.zeros(4, 50), 5, out={"I": torch.zeros(4, 6, dtype=torch.int32)})
    with pytest.raises(ValueError, match="must be a CUDA tensor"):
        mb.mosa_topk(torch.zeros(4, 50), 5)
    with pytest.raises(ValueError, match="W_r must have shape"):
        mb.mosa_route_noalloc(torch.zeros(B, T, d, dtype=bf), torch.zeros(d + 8, H, dtype=bf), k)
