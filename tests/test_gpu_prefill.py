"""GPU parity of the routed prefill (buddy_prefill) against the oracle's
prefill: prompts of 1..300 tokens appended after ragged cached contexts (so
M-tiles and attention tiles have ragged tails, and causal attention crosses
the cache/prompt boundary), both head dimensions, q/k/v bias, the router
variants (K + V feature, context layer, Budget Predictor, masked skip-KV).

Checked: routes (near-tie rule), every token's final hidden state, the K/V
every layer stored at every prompt position (zeros where skipped; nothing in
the masked variant), positions, the pooled context; then decode steps on the
state the prefill left, against the oracle continuing from its own state.
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

pytestmark = pytest.mark.gpu

CASES = [
    (C.scaled(C.T_GQA, ctx=[0, 5, 130, 0, 64, 1, 299, 17, 40], k=[1, 4, 2, 3, 1, 4, 2, 3, 4], name="pf-gqa"),
     [1, 63, 64, 65, 130, 7, 200, 33, 2]),
    (C.scaled(C.T_QWEN, ctx=[0, 100, 257, 3], k=[1, 5, 3, 2], name="pf-qwen"), [129, 1, 66, 300]),
    (C.scaled(C.T_VARIANTS[1], ctx=[0, 65, 3, 200, 9], k=[0, 2, 0, 4, 1], name="pf-kv-c1-pred"), [70, 1, 128, 5, 40]),
    (C.scaled(C.T_VARIANTS[2], ctx=[0, 65, 3, 200, 9, 31], k=[1, 2, 3, 4, 1, 2], name="pf-masked"),
     [70, 1, 128, 5, 40, 64]),
]


def run_prefill_parity(w, lengths, decode_steps=2):
    s = w.shape
    dev = "cuda"
    B, L, T = w.batch, s.n_layers, int(sum(lengths))
    masked = s.skip_kv == "masked"
    dw = D.build(w, extra_steps=max(lengths) + decode_steps + 2, max_prefill_tokens=T)
    model, st = P.oracle_for(dw)
    k = w.budgets()
    x = synth.prompt_inputs(s, w.seed, lengths, dev)
    h_out = torch.empty(T, s.d_model, device=dev)
    mask = torch.empty(B, L, dtype=torch.uint8, device=dev)
    scores = torch.empty(B, s.n_cand, device=dev)
    base_before = (dw.kv.layer_len.cpu().numpy().copy() if masked
                   else np.tile(dw.kv.len.cpu().numpy(), (L, 1)))
    dw.ctx.buddy_prefill(dw.kv, lengths, x, dw.k, h_out, mask, scores)
    torch.cuda.synchronize()
    assert dw.ctx.buddy_device_status() == 0
    g_mask = mask.cpu().numpy()
    off = np.concatenate([[0], np.cumsum(lengths)])
    prompts = [A.to_f64(x[off[i]:off[i + 1]]) for i in range(B)]
    info = {}

    def override(rr):
        sel, ks, fails, n = P.adopt(model, rr, g_mask, k)
        info["fails"], info["k"] = fails, ks
        return sel

    res = O.prefill(model, st, prompts, k, override_sel=override)
    assert not info["fails"], info["fails"]
    np.testing.assert_allclose(scores.cpu().numpy(), res.scores, rtol=0, atol=P.ROUTE_MARGIN / 2)
    np.testing.assert_array_equal(g_mask.sum(1), np.asarray(info["k"]) + s.ctx_layer + 2)
    np.testing.assert_array_equal(g_mask, res.mask)
    g_h = h_out.cpu().numpy()
    worst = 0.0
    tol = P.HIDDEN_TOL[s.dtype]
    for i in range(B):
        for t in range(lengths[i]):
            e = P.max_rel_err(g_h[off[i] + t], res.h_out[i][t])
            worst = max(worst, e)
            assert e < tol, (i, t, e)
    # K/V at every prompt position of every layer
    for l in range(L):
        for i in range(B):
            p0 = int(base_before[l, i])
            gk = dw.kv.view("k", l, i)[:, p0:p0 + lengths[i], :].float().cpu().numpy()
            gv = dw.kv.view("v", l, i)[:, p0:p0 + lengths[i], :].float().cpu().numpy()
            if g_mask[i, l]:
                ok, ov = res.kv_new[(l, i)]
                for t in range(lengths[i]):
                    assert P.max_rel_err(gk[:, t], ok[t]) < P.KV_TOL[s.dtype], (l, i, t)
                    assert P.max_rel_err(gv[:, t], ov[t]) < P.KV_TOL[s.dtype], (l, i, t)
            elif not masked:
                assert not gk.any() and not gv.any(), (l, i)
    np.testing.assert_array_equal(dw.kv.len.cpu().numpy(), np.asarray(st.n))
    if masked:
        for l in range(L):
            np.testing.assert_array_equal(dw.kv.layer_len[l].cpu().numpy(), [st.length(l, i) for i in range(B)])
    # the pooled context is the sum of the planner feature over every position
    # the context layer's cache holds (as stored on the GPU: the oracle's own
    # entries may differ from them by a bf16 rounding, covered by the routes)
    c = s.ctx_layer
    pool = dw.kv.pool_sum.cpu().numpy().astype(np.float64)
    n_c = (dw.kv.layer_len[c] if masked else dw.kv.len).cpu().numpy()
    for i in range(B):
        Kg = dw.kv.view("k", c, i)[:, :int(n_c[i]), :].double().cpu().numpy().transpose(1, 0, 2)
        Vg = dw.kv.view("v", c, i)[:, :int(n_c[i]), :].double().cpu().numpy().transpose(1, 0, 2)
        ref = O.planner_feature(model.shape, Kg, Vg).sum(axis=0).reshape(-1)
        np.testing.assert_allclose(pool[i], ref, rtol=1e-5, atol=1e-4)
    # decode steps continue from the prefilled state
    hd_out = torch.empty(B, s.d_model, device=dev)
    for step in range(decode_steps):
        h_in = synth.workload_h_in(w, 100 + step, dev)
        dw.ctx.buddy_decode_step(dw.kv, h_in, dw.k, hd_out, mask)
        torch.cuda.synchronize()
        assert dw.ctx.buddy_device_status() == 0
        g_mask = mask.cpu().numpy()

        def override_d(rr):
            sel, ks, fails, n = P.adopt(model, rr, g_mask, k)
            info["fails"] = fails
            return sel

        r = O.decode_step(model, st, A.to_f64(h_in), k, override_sel=override_d)
        assert not info["fails"], info["fails"]
        g = hd_out.cpu().numpy()
        for i in range(B):
            e = P.max_rel_err(g[i], r.h_out[i])
            worst = max(worst, e)
            assert e < tol, ("decode", step, i, e)
    print(f"{w.name}: prefill of {T} tokens + {decode_steps} decode steps, worst hidden max rel err {worst:.3e}")
    return worst


@pytest.mark.parametrize("w,lengths", CASES, ids=[c[0].name for c in CASES])
def test_prefill_parity(w, lengths):
    run_prefill_parity(w, lengths)


def test_prefill_rejects_bad_budget_and_writes_nothing():
    w, lengths = CASES[0]
    dw = D.build(w, extra_steps=max(lengths) + 2, max_prefill_tokens=sum(lengths))
    x = synth.prompt_inputs(w.shape, w.seed, lengths, "cuda")
    h_out = torch.full((sum(lengths), w.shape.d_model), 7.0, device="cuda")
    len0 = dw.kv.len.clone()
    k0 = [t.clone() for t in dw.kv.k]
    bad = dw.k.clone()
    bad[2] = w.shape.n_cand + 1
    import paper_2606_09514_gb300 as pkg
    with pytest.raises(pkg.BuddyError) as e:
        dw.ctx.buddy_prefill(dw.kv, lengths, x, bad, h_out)
    assert e.value.code == pkg.binding.BUDDY_ERR_DEVICE
    assert dw.ctx.buddy_device_status() & pkg.binding.BUDDY_DEV_BAD_BUDGET
    assert torch.all(h_out == 7.0) and torch.equal(dw.kv.len, len0)
    assert all(torch.equal(a, b) for a, b in zip(k0, dw.kv.k))
    # over the token bound: rejected on the host
    with pytest.raises(pkg.BuddyError):
        dw.ctx.buddy_prefill(dw.kv, lengths + [1], torch.cat([x, x[:1]]), torch.cat([dw.k, dw.k[:1]]), h_out)
