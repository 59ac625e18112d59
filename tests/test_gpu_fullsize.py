"""GPU parity at the benchmark workloads' full sizes, in the launch configuration
bench.py times (CUDA graph, programmatic dependent launch).

One decode step per workload.  The oracle evaluates the first layer and the
router for every sequence (routes checked with the near-tie rule, compaction
bit-exact for every layer) and the full routed depth for a few sampled
sequences (hidden state and the K/V written at the new position), streaming
their caches one layer at a time.
"""
import numpy as np
import pytest
import torch

import parity as P
from oracle import adapter as A
from oracle import buddy_oracle as O
from workloads import configs as C
from workloads import device as D
from workloads import synth

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

CASES = [
    (C.C2_LLAMA3_B1, [0]),
    (C.C3_LLAMA3_B64, [0, 37]),
    (C.C4_LLAMA2_13B, [0, 31]),
    (C.C5_QWEN_B256, [0, 129, 255]),
]


@pytest.mark.parametrize("w,sampled", CASES, ids=[c[0].name for c in CASES])
def test_fullsize_step_parity(w, sampled):
    s = w.shape
    dev = "cuda"
    dw = D.build(w, extra_steps=2, use_graph=True)
    B, L, Lm = w.batch, s.n_layers, s.l_mid
    h_in = synth.workload_h_in(w, 0, dev)
    h_out = torch.empty(B, s.d_model, device=dev)
    mask = torch.empty(B, L, dtype=torch.uint8, device=dev)
    rows = torch.empty(L, B, dtype=torch.int32, device=dev)
    count = torch.empty(L, dtype=torch.int32, device=dev)
    scores = torch.empty(B, Lm, device=dev)
    dw.ctx.buddy_decode_step(dw.kv, h_in, dw.k, h_out, mask, rows, count, scores)
    torch.cuda.synchronize()
    assert dw.ctx.buddy_device_status() == 0
    g_mask = mask.cpu().numpy()
    g_sel = P.sel_from_mask(g_mask)
    # K/V the GPU wrote at the new position, for the sampled sequences
    n0 = w.contexts()
    g_kv = {(l, i): (dw.kv.view("k", l, i)[:, int(n0[i]), :].float().cpu().numpy(),
                     dw.kv.view("v", l, i)[:, int(n0[i]), :].float().cpu().numpy())
            for l in range(L) for i in sampled}
    g_h = h_out.cpu().numpy()
    g_scores = scores.cpu().numpy()
    g_rows, g_count = rows.cpu().numpy(), count.cpu().numpy()
    dw.ctx.close()
    del dw
    torch.cuda.empty_cache()

    model = A.build_model(s, w.seed, layer_source=lambda l: synth.layer_weights(s, w.seed, l, dev),
                          dm_source=lambda: synth.dm_weights(s, w.seed, dev), cache_layers=1)
    st = A.lazy_state(s, w.seed, n0, gen_device=dev)
    k = w.budgets()
    route = O.first_layer_and_route(model, st, A.to_f64(h_in), k)
    st.drop(0)
    sel, fails, adopted = P.adopt_routes(route.scores, route.sel, g_sel, k)
    assert not fails, fails[:5]
    route.sel = sel
    np.testing.assert_allclose(g_scores, route.scores, rtol=0, atol=P.ROUTE_MARGIN / 4)
    np.testing.assert_array_equal(g_mask.sum(1), k + 2)
    res = O.routed_layers(model, st, route, seqs=sampled)
    for l in range(L):
        assert g_count[l] == len(res.rows[l]), l
        assert g_rows[l, : g_count[l]].tolist() == res.rows[l], l
    for i in sampled:
        e = P.max_rel_err(g_h[i], res.h_out[i])
        print(f"{w.name}: sequence {i} hidden max rel err {e:.3e}; adopted near-ties {adopted}")
        assert e < P.HIDDEN_TOL[s.dtype], (i, e)
        for l in range(L):
            gk, gv = g_kv[(l, i)]
            ok, ov = res.kv_new[(l, i)]
            if g_mask[i, l]:
                assert P.max_rel_err(gk, ok) < P.KV_TOL[s.dtype] and P.max_rel_err(gv, ov) < P.KV_TOL[s.dtype], (l, i)
            else:
                assert not gk.any() and not gv.any(), (l, i)
