"""Helpers for the GPU parity tests: move seeded numpy inputs to the device,
run the library through its binding, compare against the oracle."""
import numpy as np
import torch

from _util import max_abs, rel_l2
import paper_2505_00315_gb300 as mosa

#: Tolerances stated by the layer's comparison rules: fp32 storage must match
#: the fp64 oracle to 1e-4 relative L2; bf16 storage (fp32 accumulation) to
#: 2e-2 relative L2 and 5e-2 absolute per element.
TOL = {"f32": {"rel_l2": 1e-4, "max_abs": None}, "bf16": {"rel_l2": 2e-2, "max_abs": 5e-2}}


def torch_dtype(dtype: str):
    return torch.bfloat16 if dtype == "bf16" else torch.float32


def to_dev(a: np.ndarray, dtype: str):
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda").to(torch_dtype(dtype))


def run_layer(cfg, x, backward=True):
    """Forward (and backward) on the GPU; returns numpy outputs."""
    dt = cfg.dtype
    X, Wr, Wq, Wk, Wv, Wo = (to_dev(x[n], dt) for n in ("X", "Wr", "Wq", "Wk", "Wv", "Wo"))
    Y, I, rs, rf, ws = mosa.mosa_forward(X, Wr, Wq, Wk, Wv, Wo, cfg.k, want_r_full=True,
                                         first_token=cfg.first_token, rope=cfg.rope)
    out = {"Y": Y, "I": I, "r_sel": rs, "r_full": rf}
    if backward:
        dY = to_dev(x["dY"], dt)
        out.update(mosa.mosa_backward(X, Wr, Wq, Wk, Wv, Wo, I, rs, dY, ws, rope=cfg.rope))
    torch.cuda.synchronize()
    st = mosa.mosa_check_status(mosa.make_shape(X, Wq, cfg.k), ws)
    assert st == 0, f"device status {st}"
    return {k: v.cpu().numpy() for k, v in out.items()}


def assert_close(name, got, ref, dtype):
    tol = TOL[dtype]
    e = rel_l2(got, ref)
    assert e < tol["rel_l2"], f"{name}: rel L2 {e:.3e} >= {tol['rel_l2']}"
    if tol["max_abs"] is not None:
        m = max_abs(got, ref)
        assert m < tol["max_abs"], f"{name}: max abs {m:.3e} >= {tol['max_abs']}"
    return e
