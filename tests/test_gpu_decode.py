"""GPU parity: libbuddy's decode step (through the C ABI) against the oracle.

Small workloads that span several GEMM tiles with ragged tails, contexts 0..1000
(including n_i = 0 and chunk boundaries), budgets 1..L_mid, GQA groups 1..4,
qkv bias on/off, fp32 and bf16.  Multi-step runs are free-running on both
sides; the near-tie rule is the only place the oracle takes a GPU decision.
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


def run_parity(w, steps=None, use_graph=False, prior=False, check_kv=True):
    dw = D.build(w, use_graph=use_graph, prior=prior)
    model, st = P.oracle_for(dw)
    s = w.shape
    B, L, Lm = w.batch, s.n_layers, s.n_cand
    masked = s.skip_kv == "masked"
    dev = "cuda"
    h_out = torch.empty(B, s.d_model, device=dev)
    mask = torch.empty(B, L, dtype=torch.uint8, device=dev)
    rows = torch.empty(L, B, dtype=torch.int32, device=dev)
    count = torch.empty(L, dtype=torch.int32, device=dev)
    scores = torch.empty(B, Lm, device=dev)
    k = w.budgets()
    tol = P.HIDDEN_TOL[s.dtype]
    worst = 0.0
    adopted_total = 0
    for t in range(steps or w.steps):
        n_before = list(st.n)
        ll_before = dw.kv.layer_len.cpu().numpy().copy() if masked else None
        h_in = synth.workload_h_in(w, t, dev)
        dw.ctx.buddy_decode_step(dw.kv, h_in, dw.k, h_out, mask, rows, count, scores)
        torch.cuda.synchronize()
        assert dw.ctx.buddy_device_status() == 0
        g_mask = mask.cpu().numpy()
        info = {}

        def override(rr):
            sel, ks, fails, n = P.adopt(model, rr, g_mask, k)
            info["fails"], info["n"], info["k"] = fails, n, ks
            return sel

        res = O.decode_step(model, st, A.to_f64(h_in), k, override_sel=override)
        assert not info["fails"], info["fails"]
        adopted_total += info["n"]
        # scores agree well inside the near-tie margin
        np.testing.assert_allclose(scores.cpu().numpy(), res.scores, rtol=0, atol=P.ROUTE_MARGIN / 2)
        # exactly k routed layers + the always-executed ones
        np.testing.assert_array_equal(g_mask.sum(1), np.asarray(info["k"]) + s.ctx_layer + 2)
        # compaction: bit-exact
        g_count = count.cpu().numpy()
        g_rows = rows.cpu().numpy()
        for l in range(L):
            assert g_count[l] == len(res.rows[l]), (t, l)
            assert g_rows[l, : g_count[l]].tolist() == res.rows[l], (t, l)
        # hidden states
        g_h = h_out.cpu().numpy()
        for i in range(B):
            e = P.max_rel_err(g_h[i], res.h_out[i])
            worst = max(worst, e)
            assert e < tol, (t, i, e)
        # KV written this step: real entries match, skipped layers hold zeros
        # (zero variant) or nothing (masked variant: the layer's length grows
        # only where it executed)
        if check_kv:
            for l in range(L):
                for i in range(B):
                    pos = int(ll_before[l, i]) if masked else n_before[i]
                    gk = dw.kv.view("k", l, i)[:, pos, :].float().cpu().numpy()
                    gv = dw.kv.view("v", l, i)[:, pos, :].float().cpu().numpy()
                    if g_mask[i, l]:
                        ok, ov = res.kv_new[(l, i)]
                        assert P.max_rel_err(gk, ok) < P.KV_TOL[s.dtype] and P.max_rel_err(gv, ov) < P.KV_TOL[s.dtype]
                    elif not masked:
                        assert not gk.any() and not gv.any()
            if masked:
                np.testing.assert_array_equal(dw.kv.layer_len.cpu().numpy(), ll_before + g_mask.T)
    # positions advanced by one per step
    np.testing.assert_array_equal(dw.kv.len.cpu().numpy(), np.asarray(st.n))
    if masked:
        for l in range(L):
            np.testing.assert_array_equal(dw.kv.layer_len[l].cpu().numpy(), [st.length(l, i) for i in range(B)])
    return worst, adopted_total


@pytest.mark.parametrize("w", [C.T_F32, C.C1_TINY], ids=lambda w: w.name)
def test_decode_parity_f32(w):
    worst, _ = run_parity(w, steps=2)
    assert worst < 1e-4


@pytest.mark.parametrize("w", [C.T_GQA, C.T_QWEN], ids=lambda w: w.name)
def test_decode_parity_bf16(w):
    worst, _ = run_parity(w)
    assert worst < 2e-2


# Batch sizes at the mode boundaries of the bf16 path: up to 8 rows the QKV
# and gate/up GEMMs normalise in-kernel panels and the last K split applies
# the epilogue, above 8 a fixup kernel does; up to 16 rows the router's first
# layer is one CTA per hidden unit, above it a packed tiled GEMM; above 128
# rows the GEMMs take two M-tiles.
@pytest.mark.parametrize("base,batch", [(C.T_QWEN, 8), (C.T_QWEN, 9), (C.T_QWEN, 16), (C.T_QWEN, 17),
                                        (C.T_QWEN, 128), (C.T_QWEN, 129), (C.T_GQA, 8), (C.T_GQA, 17)],
                         ids=lambda v: v.shape.name if hasattr(v, "shape") else str(v))
def test_decode_parity_batch_boundaries(base, batch):
    if base.ctx_kind == "list":   # the listed contexts and budgets, repeated to the batch
        ctx = [base.ctx_args[i % len(base.ctx_args)] for i in range(batch)]
        k = [base.k_args[i % len(base.k_args)] for i in range(batch)]
        w = C.scaled(base, ctx=ctx, k=k, name=f"{base.name}-b{batch}")
    else:
        w = C.scaled(base, batch=batch, name=f"{base.name}-b{batch}")
    assert w.batch == batch
    worst, _ = run_parity(w, steps=2)
    assert worst < 2e-2


def test_decode_parity_prior_and_graph():
    run_parity(C.T_GQA, steps=2, use_graph=True, prior=True)


def test_full_budget_every_layer_executes():
    w = C.scaled(C.T_QWEN, k=[C.T_QWEN.shape.l_mid] * C.T_QWEN.batch, name="t-qwen-dense")
    run_parity(w, steps=1)


def test_budget_one_and_batch_one():
    w = C.scaled(C.T_GQA, ctx=[77], k=[1], name="t-gqa-b1")
    run_parity(w, steps=3)


def test_decode_parity_three_rows_graph_prior():
    """Three rows (a single 16-row MMA tile, most of it padding) with bias,
    RoPE partners, ragged contexts, the prior and the graph."""
    w = C.scaled(C.T_QWEN, ctx=[0, 129, 700], k=[1, 5, 3], name="t-qwen-b3")
    worst, _ = run_parity(w, steps=3, use_graph=True, prior=True)
    assert worst < 2e-2


@pytest.mark.parametrize("w", C.T_VARIANTS, ids=lambda w: w.name)
def test_decode_parity_router_variants(w):
    """K and K+V planner features, a context layer c > 0 with the Budget
    Predictor choosing some budgets, and the masked skip-KV variant."""
    worst, _ = run_parity(w)
    assert worst < P.HIDDEN_TOL[w.shape.dtype]


def test_router_variants_graph_prior():
    run_parity(C.T_VARIANTS[1], steps=2, use_graph=True, prior=True)
    run_parity(C.T_VARIANTS[2], steps=2, use_graph=True, prior=True)


def test_graph_replay_equals_direct_launches():
    w = C.T_GQA
    outs = []
    for g in (False, True):
        dw = D.build(w, use_graph=g)
        h_out = torch.empty(w.batch, w.shape.d_model, device="cuda")
        mask = torch.empty(w.batch, w.shape.n_layers, dtype=torch.uint8, device="cuda")
        res = []
        for t in range(3):
            dw.ctx.buddy_decode_step(dw.kv, synth.workload_h_in(w, t, "cuda"), dw.k, h_out, mask)
            res.append((h_out.clone(), mask.clone()))
        torch.cuda.synchronize()
        outs.append(res)
    for (a, ma), (b, mb) in zip(*outs):
        assert torch.equal(ma, mb)
        assert torch.equal(a, b)


def test_route_entry_point_matches_oracle_router():
    """buddy_route alone: pool over the cached first-layer V (including the
    newest token, already appended), Decision Module, top-k."""
    w = C.T_QWEN
    dw = D.build(w, prior=True)
    s = w.shape
    B, Lm = w.batch, s.l_mid
    h1 = synth.h_in(s, 99, 0, range(B), "cuda") * 3.0
    sel = torch.empty(B, Lm, dtype=torch.int32, device="cuda")
    mask = torch.empty(B, s.n_layers, dtype=torch.uint8, device="cuda")
    sc = torch.empty(B, Lm, device="cuda")
    # the router needs len >= 1: sequences with n_i = 0 get one appended position
    ctxs = w.contexts()
    empty = [i for i in range(B) if ctxs[i] == 0]
    for i in empty:
        ids = torch.tensor([i], dtype=torch.int32, device="cuda")
        K = synth.kv_block(s, w.seed, "k", 0, i, 0, 1, "cuda").unsqueeze(0)
        V = synth.kv_block(s, w.seed, "v", 0, i, 0, 1, "cuda").unsqueeze(0)
        dw.ctx.buddy_kv_append(dw.kv, 0, ids, K, V, advance=True)
    dw.ctx.buddy_route(dw.kv, h1, dw.k, sel, mask, sc)
    torch.cuda.synchronize()
    assert dw.ctx.buddy_device_status() == 0
    model, _ = P.oracle_for(dw)
    sh = model.shape
    lens = dw.kv.len.cpu().numpy()
    o_sel, o_sc = [], []
    for i in range(B):
        V0 = A.to_f64(synth.kv_block(s, w.seed, "v", 0, i, 0, int(lens[i]), "cuda"))
        x = np.concatenate([O.expand_kv_heads(O.pool_context(V0), sh), A.to_f64(h1[i])])
        sc_i = O.decision_scores(model.dm, x)
        o_sc.append(sc_i)
        o_sel.append(O.top_k_layers(sc_i, int(w.budgets()[i])))
    o_sc = np.array(o_sc)
    np.testing.assert_allclose(sc.cpu().numpy(), o_sc, rtol=0, atol=1e-5)
    g_sel = [[int(v) for v in row if v >= 0] for row in sel.cpu().numpy()]
    _, fails, _ = P.adopt_routes(o_sc, o_sel, g_sel, w.budgets())
    assert not fails
    np.testing.assert_array_equal(mask.cpu().numpy().sum(1), w.budgets() + 2)


def test_kv_append_pool_is_full_sum():
    w = C.T_GQA
    dw = D.build(w)
    s = w.shape
    pool = dw.kv.pool_sum.cpu().numpy().astype(np.float64)
    for i in range(w.batch):
        n = int(w.contexts()[i])
        V0 = A.to_f64(synth.kv_block(s, w.seed, "v", 0, i, 0, n, "cuda")) if n else np.zeros((0, s.n_kv_heads, s.head_dim))
        ref = V0.sum(0).reshape(-1)
        np.testing.assert_allclose(pool[i], ref, rtol=1e-5, atol=1e-4)
    np.testing.assert_array_equal(dw.kv.len.cpu().numpy(), w.contexts())


def test_device_checks_write_nothing():
    w = C.T_GQA
    dw = D.build(w)
    s = w.shape
    B = w.batch
    h_in = synth.workload_h_in(w, 0, "cuda")
    h_out = torch.full((B, s.d_model), 7.0, device="cuda")
    k0 = [t.clone() for t in dw.kv.k]
    len0 = dw.kv.len.clone()
    pool0 = dw.kv.pool_sum.clone()
    bad = dw.k.clone()
    bad[3] = s.l_mid + 1
    dw.ctx.buddy_decode_step(dw.kv, h_in, bad, h_out)
    flags = dw.ctx.buddy_device_status()
    assert flags & 1
    assert torch.all(h_out == 7.0)
    assert torch.equal(dw.kv.len, len0) and torch.equal(dw.kv.pool_sum, pool0)
    assert all(torch.equal(a, b) for a, b in zip(k0, dw.kv.k))
    # a position beyond capacity
    dw.kv.len[5] = int(dw.caps[5])
    dw.ctx.buddy_decode_step(dw.kv, h_in, dw.k, h_out)
    assert dw.ctx.buddy_device_status() & 2
    assert torch.all(h_out == 7.0)
    # the context stays usable: a valid call succeeds afterwards
    dw.kv.len.copy_(len0)
    dw.ctx.buddy_decode_step(dw.kv, h_in, dw.k, h_out)
    assert dw.ctx.buddy_device_status() == 0
    assert not torch.all(h_out == 7.0)


def test_misaligned_buffers_rejected_on_host():
    """Hidden-state buffers and caches are accessed with 16-byte vectors: a
    pointer off by 4 bytes is rejected before any launch (nothing written)."""
    import paper_2606_09514_gb300 as pkg
    w = C.T_GQA
    dw = D.build(w)
    s = w.shape
    B = w.batch
    h_in = synth.workload_h_in(w, 0, "cuda")
    flat = torch.full((B * s.d_model + 4,), 7.0, device="cuda")
    h_off = flat[1:1 + B * s.d_model].view(B, s.d_model)   # data_ptr() % 16 == 4
    assert h_off.data_ptr() % 16 == 4
    len0 = dw.kv.len.clone()
    with pytest.raises(pkg.binding.BuddyError) as e:
        dw.ctx.buddy_decode_step(dw.kv, h_in, dw.k, h_off)
    assert e.value.code == pkg.binding.BUDDY_ERR_ARG
    in_off = torch.empty(B * s.d_model + 4, device="cuda")[1:1 + B * s.d_model].view(B, s.d_model)
    in_off.copy_(h_in)
    h_out = torch.empty(B, s.d_model, device="cuda")
    with pytest.raises(pkg.binding.BuddyError) as e:
        dw.ctx.buddy_decode_step(dw.kv, in_off, dw.k, h_out)
    assert e.value.code == pkg.binding.BUDDY_ERR_ARG
    torch.cuda.synchronize()
    assert torch.all(flat == 7.0) and torch.equal(dw.kv.len, len0)
    # the context stays usable
    dw.ctx.buddy_decode_step(dw.kv, h_in, dw.k, h_out)
    assert dw.ctx.buddy_device_status() == 0


def test_gemm_wait_limit_runs_out_and_context_recovers():
    """With a wait limit far below the time a TMA stage takes, the GEMMs give
    up: the step reports BUDDY_DEV_TIMEOUT.  Restoring the limit, the same
    step from the same state equals a fresh context's result (the arrival
    counters were re-armed)."""
    import paper_2606_09514_gb300 as pkg
    for w in (C.T_GQA, C.scaled(C.T_QWEN, ctx=[5, 300, 64], k=[1, 3, 5], name="t-qwen-b3-timeout")):
        s = w.shape
        h_in = synth.workload_h_in(w, 0, "cuda")
        ref = D.build(w)
        h_ref = torch.empty(w.batch, s.d_model, device="cuda")
        ref.ctx.buddy_decode_step(ref.kv, h_in, ref.k, h_ref)
        torch.cuda.synchronize()
        assert ref.ctx.buddy_device_status() == 0
        dw = D.build(w)
        len0, pool0 = dw.kv.len.clone(), dw.kv.pool_sum.clone()
        h_out = torch.empty(w.batch, s.d_model, device="cuda")
        dw.ctx.buddy_set_wait_limit(1)
        dw.ctx.buddy_decode_step(dw.kv, h_in, dw.k, h_out)
        torch.cuda.synchronize()
        assert dw.ctx.buddy_device_status() & pkg.binding.BUDDY_DEV_TIMEOUT
        dw.ctx.buddy_set_wait_limit(0)
        dw.kv.len.copy_(len0)
        dw.kv.pool_sum.copy_(pool0)
        dw.ctx.buddy_decode_step(dw.kv, h_in, dw.k, h_out)
        torch.cuda.synchronize()
        assert dw.ctx.buddy_device_status() == 0
        assert torch.equal(h_out, h_ref)
        ref.ctx.close()
        dw.ctx.close()


def test_host_buffer_entry_matches_device_entry():
    w = C.T_GQA
    outs = []
    for host in (False, True):
        dw = D.build(w)
        h_in = synth.workload_h_in(w, 0, "cuda")
        if host:
            hh = h_in.cpu().pin_memory()
            kh = dw.k.cpu().pin_memory()
            oh = torch.empty(w.batch, w.shape.d_model).pin_memory()
            mh = torch.empty(w.batch, w.shape.n_layers, dtype=torch.uint8).pin_memory()
            dw.ctx.buddy_decode_step_host(dw.kv, hh, kh, oh, mh)
            outs.append((oh.clone(), mh.clone()))
        else:
            o = torch.empty(w.batch, w.shape.d_model, device="cuda")
            m = torch.empty(w.batch, w.shape.n_layers, dtype=torch.uint8, device="cuda")
            dw.ctx.buddy_decode_step(dw.kv, h_in, dw.k, o, m)
            outs.append((o.cpu(), m.cpu()))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])


def test_generator_identical_on_cpu_and_gpu():
    s = C.LLAMA3_8B
    for kind, ids, n, start in [("w_q", (3,), 100003, 77), ("k_cache", (0, 5), 65536, 1 << 20),
                                ("h_in", (2, 1), 4096, 0)]:
        key = synth.stream_key(0, kind, *ids)
        a = synth.normal((n,), key, 0.02, torch.bfloat16, "cpu", start=start)
        b = synth.normal((n,), key, 0.02, torch.bfloat16, "cuda", start=start).cpu()
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
        a = synth.normal((n,), key, 1.0, torch.float32, "cpu", start=start)
        b = synth.normal((n,), key, 1.0, torch.float32, "cuda", start=start).cpu()
        assert torch.equal(a.view(torch.int32), b.view(torch.int32))
