"""The allocation-free router (buddy_route_noalloc) against buddy_route.

buddy_route_noalloc serves callers that cannot allocate device memory (and so
cannot create a context): its scratch is a static device array inside the
library.  Two calls in a row with different inputs must each match the
context-based router, which also shows that the shared scratch carries no
stale state from the previous call.  This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import parity as P
from workloads import configs as C
from workloads import device as D
from workloads import synth

pytestmark = pytest.mark.gpu


def test_noalloc_router_matches_context_router_twice():
    import paper_2606_09514_gb300 as pkg
    from paper_2606_09514_gb300 import binding as B

    w = C.scaled(C.T_QWEN, ctx=[1, 2, 63, 64, 65, 129, 300, 7, 1000, 17, 256, 5], k=[1, 5, 3, 2, 4, 5, 1, 2, 3, 4, 5, 1],
                 name="t-qwen-noalloc")
    dw = D.build(w, prior=True)
    s = w.shape
    Bn, L, Lm = w.batch, s.n_layers, s.l_mid
    dev = "cuda"
    for call in range(2):
        h1 = synth.h_in(s, 1234 + call, 0, range(Bn), dev) * (2.0 + call)
        k = dw.k if call == 0 else torch.flip(dw.k, [0]).contiguous()
        outs = []
        for noalloc in (False, True):
            sel = torch.full((Bn, Lm), -7, dtype=torch.int32, device=dev)
            mask = torch.full((Bn, L), 9, dtype=torch.uint8, device=dev)
            sc = torch.full((Bn, Lm), float("nan"), device=dev)
            if noalloc:
                flags = torch.full((1,), -1, dtype=torch.int32, device=dev)
                pkg.binding.buddy_route_noalloc(s, dw.dm, dw.kv.pool_sum, dw.kv.len, h1, k, sel, mask, sc,
                                                flags, prior=dw.prior, omega=0.1)
                torch.cuda.synchronize()
                assert int(flags.item()) == 0
            else:
                dw.ctx.buddy_route(dw.kv, h1, k, sel, mask, sc)
                torch.cuda.synchronize()
                assert dw.ctx.buddy_device_status() == 0
            outs.append((sel.cpu().numpy(), mask.cpu().numpy(), sc.cpu().numpy()))
        (s0, m0, c0), (s1, m1, c1) = outs
        np.testing.assert_allclose(c1, c0, rtol=0, atol=P.ROUTE_MARGIN / 4)
        np.testing.assert_array_equal(s1, s0)
        np.testing.assert_array_equal(m1, m0)
        np.testing.assert_array_equal(m1.sum(1), k.cpu().numpy() + 2)

    # a budget outside [1, L-2] (seen only by the device): the flags word says
    # so, nothing else is written, and the next valid call is not held up by
    # the abort word this call left in the shared scratch
    bad = dw.k.clone()
    bad[4] = 0
    sel = torch.full((Bn, Lm), -7, dtype=torch.int32, device=dev)
    mask = torch.full((Bn, L), 9, dtype=torch.uint8, device=dev)
    sc = torch.full((Bn, Lm), 123.0, device=dev)
    flags = torch.full((1,), -1, dtype=torch.int32, device=dev)
    h1 = synth.h_in(s, 77, 0, range(Bn), dev)
    pkg.binding.buddy_route_noalloc(s, dw.dm, dw.kv.pool_sum, dw.kv.len, h1, bad, sel, mask, sc, flags,
                                    prior=dw.prior, omega=0.1)
    torch.cuda.synchronize()
    assert int(flags.item()) == B.BUDDY_DEV_BAD_BUDGET
    assert torch.all(sel == -7) and torch.all(mask == 9) and torch.all(sc == 123.0)
    flags.fill_(-1)
    pkg.binding.buddy_route_noalloc(s, dw.dm, dw.kv.pool_sum, dw.kv.len, h1, dw.k, sel, mask, sc, flags,
                                    prior=dw.prior, omega=0.1)
    sel2 = torch.empty_like(sel)
    mask2 = torch.empty_like(mask)
    sc2 = torch.empty_like(sc)
    dw.ctx.buddy_route(dw.kv, h1, dw.k, sel2, mask2, sc2)
    torch.cuda.synchronize()
    assert int(flags.item()) == 0
    np.testing.assert_array_equal(sel.cpu().numpy(), sel2.cpu().numpy())
    np.testing.assert_array_equal(mask.cpu().numpy(), mask2.cpu().numpy())
    np.testing.assert_allclose(sc.cpu().numpy(), sc2.cpu().numpy(), rtol=0, atol=P.ROUTE_MARGIN / 4)

    # sizes beyond the static scratch are rejected before any launch
    big = torch.zeros(300, s.d_model, device=dev)
    lib = B.load_library()
    dmw = B.buddy_dm_weights(dw.dm["w1"].data_ptr(), dw.dm["b1"].data_ptr(), dw.dm["w2"].data_ptr(),
                             dw.dm["b2"].data_ptr(), None, 0.0)
    rc = lib.buddy_route_noalloc(s.n_layers, s.d_model, s.n_q_heads, s.n_kv_heads, s.head_dim, 300,
                                 ctypes.byref(dmw), 300, ctypes.c_void_p(big.data_ptr()),
                                 ctypes.c_void_p(dw.kv.len.data_ptr()), ctypes.c_void_p(big.data_ptr()),
                                 ctypes.c_void_p(dw.k.data_ptr()), None, None, None, None, None)
    assert rc == B.BUDDY_ERR_RANGE
