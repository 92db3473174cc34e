"""mosa_route_noalloc: routing for callers that cannot allocate device memory.

Some callers cannot give the library a workspace: a host application that
owns the device heap and hands out nothing after start-up, a plug-in that
only sees its inputs and outputs, a loop that may never trigger cudaMalloc's
device-wide synchronisation.  For them the entry point keeps the router
scores in a fixed 4 MiB array inside the library.  These tests call it
through the C ABI and check that it selects exactly what mosa_forward
selects and what the oracle selects, on two calls in a row (the second must
not see the first's scores), and that it refuses problems larger than its
array.  The file is
named to be collected last."""
import ctypes

import numpy as np
import pytest
import torch

import paper_2505_00315_gb300 as mosa
from paper_2505_00315_gb300 import _binding as B
from paper_2505_00315_gb300 import workloads as W


def test_refuses_problems_beyond_its_array():
    # B*H*T = 4*256*4096 > 2^20 scores: rejected before any CUDA call.
    s = B.MosaShape(4, 4096, 1024, 256, 64, 64, B.MOSA_BF16)
    fake = ctypes.c_void_p(0x100000)
    assert B.load().mosa_route_noalloc(ctypes.byref(s), fake, fake, fake, fake, None) == \
        B.MOSA_ERR_UNSUPPORTED
    s = B.MosaShape(1, 64, 64, 2, 64, 65, B.MOSA_BF16)     # k > T
    assert B.load().mosa_route_noalloc(ctypes.byref(s), fake, fake, fake, fake, None) == \
        B.MOSA_ERR_INVALID_ARG


@pytest.mark.gpu
def test_matches_forward_and_oracle_on_two_calls_in_a_row():
    import oracle
    from _util import sigmoid_gap
    cases = [W.CONFIGS["B8_T1024_d512_H16_k128"],
             W.MosaConfig("second", B=3, T=500, d=136, H=5, hp=64, k=77, dtype="bf16", seed=31)]
    for cfg in cases:
        x = W.make_inputs(cfg)
        dev = {n: torch.from_numpy(x[n]).cuda().to(torch.bfloat16) for n in x}
        _, I_ref, rs_ref, _, _ = mosa.mosa_forward(dev["X"], dev["Wr"], dev["Wq"], dev["Wk"],
                                                   dev["Wv"], dev["Wo"], cfg.k)
        I, rs = mosa.mosa_route_noalloc(dev["X"], dev["Wr"], cfg.k, hp=cfg.hp)
        torch.cuda.synchronize()
        I, rs = I.cpu().numpy(), rs.cpu().numpy()
        # the same router kernel as mosa_forward: identical indices and scores
        np.testing.assert_array_equal(I, I_ref.cpu().numpy())
        np.testing.assert_array_equal(rs.view(np.uint32), rs_ref.cpu().numpy().view(np.uint32))
        # and the oracle's selection (its k-th / (k+1)-th score gap is planted)
        rf = oracle.router(x["X"], x["Wr"])
        assert sigmoid_gap(rf, cfg.k) > 1e-3
        for b in range(cfg.B):
            for h in range(cfg.H):
                Iref, rsref = oracle.topk(rf[b, h], cfg.k)
                np.testing.assert_array_equal(I[b, h], Iref)
                np.testing.assert_allclose(rs[b, h], rsref, rtol=1e-5, atol=0)
