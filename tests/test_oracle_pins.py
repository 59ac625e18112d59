"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test ties an oracle function to something other than itself: a value the
paper prints, a closed form, an invariant of the method, or a textbook
library routine (torch float64) computing the same definition another way.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch
import torch.nn.functional as Fnn

from oracle import adapter as A
from oracle import buddy_oracle as O
from workloads import configs as C
from workloads import cost

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _gold(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def _tiny_shape(dtype="f32", n_q=4, n_kv=2, hd=8, L=5, d=None, F=24, r=16):
    d = d or n_q * hd
    return O.Shape(L, d, n_q, n_kv, hd, F, r, dtype, 1e-5, 1e4)


def _rand_layer(sh, rng, bias=True):
    d, qd, kvd, F = sh.d_model, sh.n_q_heads * sh.head_dim, sh.n_kv_heads * sh.head_dim, sh.ffn_dim
    g = lambda *s: rng.standard_normal(s) * 0.3
    return O.LayerWeights(attn_norm=1 + 0.1 * rng.standard_normal(d), w_q=g(qd, d), w_k=g(kvd, d),
                          w_v=g(kvd, d), w_o=g(d, qd), ffn_norm=1 + 0.1 * rng.standard_normal(d),
                          w_gate=g(F, d), w_up=g(F, d), w_down=g(d, F),
                          b_q=g(qd) if bias else None, b_k=g(kvd) if bias else None,
                          b_v=g(kvd) if bias else None)


# ---------------------------------------------------------------------------
# Paper-printed values
# ---------------------------------------------------------------------------
def test_paper_flops_example():
    g = _gold("dm_flops_overhead.json")
    p = g["params"]
    assert cost.paper_f_dm(p["B"], p["T"], p["d"], p["r"], p["L"], p["I"]) == g["F_DM"]
    assert cost.paper_f_layer(p["T"], p["d"], p["d_c"]) == g["F_layer"]
    for b, v in g["F_model"].items():
        assert cost.paper_f_model(Fraction(b), p["L"], p["T"], p["d"], p["d_c"]) == v
    for b, v in g["rho"].items():
        rho = cost.paper_rho(Fraction(b), p["B"], p["T"], p["d"], p["d_c"], p["r"], p["L"], p["I"])
        assert float(f"{rho:.{g['rho_printed_digits']}g}") == pytest.approx(v, rel=1e-12)


def test_budget_to_k_paper_settings():
    g = _gold("budget_k.json")
    for c in g["cases"]:
        L = c["L"]
        assert c["removed"] + c["k"] + 2 == L
        assert O.budget_to_k(c["b"], L) == c["k"]
        # Eq. 3 round trip: b = (k+2)/L maps back to the same k
        assert O.budget_to_k(O.k_to_budget(c["k"], L), L) == c["k"]
    # clamping to the action space {1..L_mid}
    assert O.budget_to_k(0.0, 32) == 1
    assert O.budget_to_k(1.0, 32) == 30
    assert O.budget_to_k(2.0, 32) == 30


def test_topk_golden_cases():
    for c in _gold("topk_cases.json")["cases"]:
        assert O.top_k_layers(np.array(c["scores"]), c["k"]) == c["sel"], c


def test_topk_matches_stable_argsort():
    rng = np.random.default_rng(5)
    for _ in range(300):
        n = int(rng.integers(1, 40))
        s = rng.integers(-4, 5, size=n).astype(np.float64) / 4.0   # many ties
        k = int(rng.integers(1, n + 1))
        ref = np.argsort(-s, kind="stable")[:k] + 1
        assert O.top_k_layers(s, k) == sorted(ref.tolist())


# ---------------------------------------------------------------------------
# Number formats
# ---------------------------------------------------------------------------
def test_bf16_round_matches_torch():
    rng = np.random.default_rng(0)
    x = rng.standard_normal(200000).astype(np.float32) * np.float32(10.0) ** rng.integers(-8, 8, 200000)
    # exact ties between two bf16 neighbours, both parities
    base = rng.standard_normal(1000).astype(np.float32)
    bits = (base.view(np.uint32) & 0xFFFF0000) | 0x8000
    x = np.concatenate([x, bits.astype(np.uint32).view(np.float32), np.float32([0.0, -0.0, 1e38, -3e38])])
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    got = O.round_to_bf16(x.astype(np.float64))
    np.testing.assert_array_equal(got, ref)


def test_bf16_decode_matches_torch():
    bits = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16)
    t = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    got = O.bf16_bits_to_f64(bits)
    fin = np.isfinite(t)
    np.testing.assert_array_equal(got[fin], t[fin])
    assert np.array_equal(np.isnan(got), np.isnan(t))


# ---------------------------------------------------------------------------
# Layer building blocks vs library routines / closed forms
# ---------------------------------------------------------------------------
def test_rms_norm_matches_torch():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((7, 96)) * 3
    g = rng.standard_normal(96)
    ref = Fnn.rms_norm(torch.from_numpy(x), (96,), torch.from_numpy(g), eps=1e-5).numpy()
    np.testing.assert_allclose(O.rms_norm(x, g, 1e-5), ref, rtol=1e-13, atol=1e-13)


def test_rope_equals_complex_rotation():
    rng = np.random.default_rng(2)
    hd, theta = 16, 10000.0
    x = rng.standard_normal((3, hd))
    for pos in (0, 1, 7, 1234, 8191):
        z = x[:, : hd // 2] + 1j * x[:, hd // 2:]
        freq = theta ** (-np.arange(0, hd, 2) / hd)
        r = z * np.exp(1j * pos * freq)
        ref = np.concatenate([r.real, r.imag], axis=-1)
        np.testing.assert_allclose(O.rope(x, pos, theta), ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_array_equal(O.rope(x, 0, theta), x)


def test_rope_relative_position_property():
    rng = np.random.default_rng(3)
    q, k = rng.standard_normal(32), rng.standard_normal(32)
    a = O.rope(q, 100, 5e5) @ O.rope(k, 37, 5e5)
    b = O.rope(q, 100 + 911, 5e5) @ O.rope(k, 37 + 911, 5e5)
    assert a == pytest.approx(b, rel=1e-10)
    # not trivially position-independent
    c = O.rope(q, 101, 5e5) @ O.rope(k, 37, 5e5)
    assert abs(a - c) > 1e-3


def test_decode_attention_matches_sdpa_gqa():
    rng = np.random.default_rng(4)
    n_q, n_kv, hd, n = 6, 2, 16, 23
    q = rng.standard_normal((n_q, hd))
    K = rng.standard_normal((n, n_kv, hd))
    V = rng.standard_normal((n, n_kv, hd))
    got = O.decode_attention(q, K, V, n_q // n_kv)
    tq = torch.from_numpy(q)[:, None, :]                          # [H, 1, hd]
    tk = torch.from_numpy(K).permute(1, 0, 2).repeat_interleave(n_q // n_kv, 0)
    tv = torch.from_numpy(V).permute(1, 0, 2).repeat_interleave(n_q // n_kv, 0)
    ref = Fnn.scaled_dot_product_attention(tq, tk, tv)[:, 0, :].numpy()
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_attention_over_zero_filled_keys_is_mean_of_values():
    # Zero K rows (skipped-layer positions, Sec. 6) take part with logit 0.
    rng = np.random.default_rng(5)
    V = rng.standard_normal((9, 1, 8))
    V[3] = 0.0
    out = O.decode_attention(rng.standard_normal((2, 8)), np.zeros((9, 1, 8)), V, 2)
    np.testing.assert_allclose(out, np.repeat(V.mean(axis=0), 2, axis=0), rtol=1e-13, atol=1e-15)


def _textbook_layer_prefill(sh, W, X):
    """A Llama decoder layer over a whole sequence with torch float64 routines
    (F.rms_norm, F.linear, causal SDPA, complex-rotation RoPE)."""
    T = X.shape[0]
    hd = sh.head_dim
    t = lambda a: torch.from_numpy(np.asarray(a))
    x = t(X)
    xn = Fnn.rms_norm(x, (sh.d_model,), t(W.attn_norm), eps=sh.rms_eps)
    q = Fnn.linear(xn, t(W.w_q), None if W.b_q is None else t(W.b_q))
    k = Fnn.linear(xn, t(W.w_k), None if W.b_k is None else t(W.b_k))
    v = Fnn.linear(xn, t(W.w_v), None if W.b_v is None else t(W.b_v))
    freq = t(sh.rope_theta ** (-np.arange(0, hd, 2) / hd))
    rot = torch.exp(1j * torch.arange(T, dtype=torch.float64)[:, None] * freq[None, :])  # [T, hd/2]

    def rope_c(a, H):
        a = a.view(T, H, hd)
        z = torch.complex(a[..., : hd // 2], a[..., hd // 2:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], -1)

    q, k, v = rope_c(q, sh.n_q_heads), rope_c(k, sh.n_kv_heads), v.view(T, sh.n_kv_heads, hd)
    rep = sh.n_q_heads // sh.n_kv_heads
    att = Fnn.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1).repeat_interleave(rep, 0),
                                           v.transpose(0, 1).repeat_interleave(rep, 0), is_causal=True)
    att = att.transpose(0, 1).reshape(T, -1)
    h = x + Fnn.linear(att, t(W.w_o))
    xn2 = Fnn.rms_norm(h, (sh.d_model,), t(W.ffn_norm), eps=sh.rms_eps)
    h = h + Fnn.linear(Fnn.silu(Fnn.linear(xn2, t(W.w_gate))) * Fnn.linear(xn2, t(W.w_up)), t(W.w_down))
    return h.numpy(), k.numpy(), v.numpy()


@pytest.mark.parametrize("n_q,n_kv,bias", [(4, 2, True), (4, 4, False), (6, 2, True)])
def test_decoder_layer_decode_equals_causal_prefill(n_q, n_kv, bias):
    """Decoding token n against the cache of tokens 0..n-1 (Eq. 9) reproduces
    row n of a causal full-sequence pass of the textbook layer."""
    rng = np.random.default_rng(6)
    sh = _tiny_shape(n_q=n_q, n_kv=n_kv)
    W = _rand_layer(sh, rng, bias)
    T = 11
    X = rng.standard_normal((T, sh.d_model))
    H, Kt, Vt = _textbook_layer_prefill(sh, W, X)
    for n in (0, 1, T - 1):
        h, k_t, v_t = O.decoder_layer(sh, W, X[n], Kt[:n], Vt[:n], n)
        np.testing.assert_allclose(h, H[n], rtol=1e-11, atol=1e-11)
        np.testing.assert_allclose(k_t, Kt[n], rtol=1e-11, atol=1e-11)
        np.testing.assert_allclose(v_t, Vt[n], rtol=1e-11, atol=1e-11)


def test_decoder_layer_bf16_rounds_only_stored_tensors():
    # With bf16 storage, K_t and V_t are bf16 values and the output stays close
    # to the unrounded layer (relative error at the bf16 level, not worse).
    rng = np.random.default_rng(7)
    sh32 = _tiny_shape()
    sh16 = _tiny_shape(dtype="bf16")
    W = _rand_layer(sh32, rng)
    K, V = rng.standard_normal((5, 2, 8)), rng.standard_normal((5, 2, 8))
    h = rng.standard_normal(sh32.d_model)
    a, ka, va = O.decoder_layer(sh32, W, h, K, V, 5)
    b, kb, vb = O.decoder_layer(sh16, W, h, K, V, 5)
    np.testing.assert_array_equal(O.round_to_bf16(kb), kb)
    np.testing.assert_array_equal(O.round_to_bf16(vb), vb)
    err = np.max(np.abs(a - b)) / np.max(np.abs(a))
    assert 1e-6 < err < 2e-2


def test_first_layer_keeps_activations_unrounded():
    """round_act=False rounds only the stored K/V: with the same stored K/V the
    bf16 layer equals the unrounded (f32-shape) layer."""
    rng = np.random.default_rng(11)
    sh32, sh16 = _tiny_shape(), _tiny_shape(dtype="bf16")
    W = _rand_layer(sh32, rng)
    K, V = rng.standard_normal((5, 2, 8)), rng.standard_normal((5, 2, 8))
    h = rng.standard_normal(sh32.d_model)
    b, kb, vb = O.decoder_layer(sh16, W, h, K, V, 5, round_act=False)
    np.testing.assert_array_equal(O.round_to_bf16(kb), kb)
    # recompute the f32 layer with the same (rounded) new K/V appended
    xn = O.rms_norm(h, W.attn_norm, sh32.rms_eps)
    q = O.rope((W.w_q @ xn + W.b_q).reshape(4, 8), 5, sh32.rope_theta)
    att = O.decode_attention(q, np.concatenate([K, kb[None]]), np.concatenate([V, vb[None]]), 2).reshape(-1)
    x = h + W.w_o @ att
    xn2 = O.rms_norm(x, W.ffn_norm, sh32.rms_eps)
    ref = x + W.w_down @ (O.silu(W.w_gate @ xn2) * (W.w_up @ xn2))
    np.testing.assert_allclose(b, ref, rtol=1e-12, atol=1e-12)
    a, _, _ = O.decoder_layer(sh16, W, h, K, V, 5, round_act=True)
    assert np.max(np.abs(a - b)) > 0


def test_dm_matches_torch_mlp():
    rng = np.random.default_rng(8)
    d2, r, Lm = 24, 10, 7
    dm = O.DecisionModule(w1=rng.standard_normal((r, d2)), b1=rng.standard_normal(r),
                          w2=rng.standard_normal((Lm, r)), b2=rng.standard_normal(Lm),
                          prior=rng.standard_normal(Lm), omega=0.1)
    mlp = torch.nn.Sequential(torch.nn.Linear(d2, r), torch.nn.SiLU(), torch.nn.Linear(r, Lm)).double()
    with torch.no_grad():
        mlp[0].weight.copy_(torch.from_numpy(dm.w1)); mlp[0].bias.copy_(torch.from_numpy(dm.b1))
        mlp[2].weight.copy_(torch.from_numpy(dm.w2)); mlp[2].bias.copy_(torch.from_numpy(dm.b2))
    x = rng.standard_normal(d2)
    ref = mlp(torch.from_numpy(x)).detach().numpy() + 0.1 * dm.prior
    np.testing.assert_allclose(O.decision_scores(dm, x), ref, rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------------------
# KV-aware planner
# ---------------------------------------------------------------------------
def test_pool_closed_forms():
    n_kv, hd = 2, 4
    for n in (0, 1, 5, 100):
        V = np.arange(n + 1, dtype=np.float64)[:, None, None] * np.ones((1, n_kv, hd)) * 0.5
        np.testing.assert_allclose(O.pool_context(V), np.full(n_kv * hd, 0.5 * n / 2), rtol=0, atol=1e-12)
        c = np.full((n + 1, n_kv, hd), 3.25)
        np.testing.assert_array_equal(O.pool_context(c), np.full(n_kv * hd, 3.25))


def test_expand_kv_heads_order():
    sh = _tiny_shape(n_q=6, n_kv=2, hd=2)
    g = np.array([1.0, 2.0, 3.0, 4.0])      # head0 = (1,2), head1 = (3,4)
    np.testing.assert_array_equal(O.expand_kv_heads(g, sh), [1, 2, 1, 2, 1, 2, 3, 4, 3, 4, 3, 4])


def test_router_pools_newest_token_with_cache():
    """With SiLU driven into its linear regime, s' is linear in the router
    input; reading the pool back shows mean over the n cached positions AND
    the newest token's V (Sec. 4.3), concatenated before H_1."""
    rng = np.random.default_rng(9)
    sh = _tiny_shape(n_q=4, n_kv=2, hd=4, L=2 + 16, d=16)
    d, Lm = sh.d_model, sh.l_mid
    W0 = _rand_layer(sh, rng)
    big = 60.0
    w1 = np.zeros((2 * d, 2 * d)); w1[np.arange(2 * d), np.arange(2 * d)] = 1.0
    w2 = np.zeros((Lm, 2 * d)); w2[np.arange(Lm), np.arange(Lm)] = 1.0     # s_j = x_j (pool part)
    dm = O.DecisionModule(w1=w1, b1=np.full(2 * d, big), w2=w2, b2=np.full(Lm, -big))
    model = O.Model(sh, lambda l: W0, dm)
    n = 6
    st = O.KVState([n])
    st.set(0, 0, rng.standard_normal((n, 2, 4)), np.zeros((n, 2, 4)))
    rr = O.first_layer_and_route(model, st, rng.standard_normal((1, d)), [3])
    v_t = rr.kv0_new[0][1].reshape(-1)
    expect = O.expand_kv_heads(v_t / (n + 1), sh)[:Lm]
    np.testing.assert_allclose(rr.scores[0], expect, rtol=0, atol=1e-9)


# ---------------------------------------------------------------------------
# Method invariants on generated workloads
# ---------------------------------------------------------------------------
def _run(w, steps=1, override=None, k=None):
    model = A.build_model(w.shape, w.seed)
    st = A.build_state(w.shape, w.seed, w.contexts())
    kk = w.budgets() if k is None else k
    out = []
    for t in range(steps):
        out.append(O.decode_step(model, st, A.workload_inputs(w, t), kk, override_sel=override))
    return model, st, out


def test_exactly_k_layers_executed_first_last_always():
    w = C.T_F32
    _, _, (res,) = _run(w)
    k = w.budgets()
    np.testing.assert_array_equal(res.mask.sum(axis=1), k + 2)
    assert res.mask[:, 0].all() and res.mask[:, -1].all()
    for i, s in enumerate(res.sel):
        assert len(s) == k[i] and all(1 <= l <= w.shape.n_layers - 2 for l in s)


def test_full_budget_equals_dense_model():
    """k = L_mid executes every block: Eq. 1 with M = 1 (bit-exact)."""
    w = C.T_F32
    model = A.build_model(w.shape, w.seed)
    st = A.build_state(w.shape, w.seed, w.contexts())
    h = A.workload_inputs(w, 0)
    dense = O.dense_decode_step(model, st, h)
    res = O.decode_step(model, st, h, [w.shape.l_mid] * w.batch)
    for i in range(w.batch):
        np.testing.assert_array_equal(res.h_out[i], dense[i])


def test_skipped_layers_are_identity_and_store_zero_kv():
    w = C.T_F32
    model = A.build_model(w.shape, w.seed)
    st = A.build_state(w.shape, w.seed, w.contexts())
    h = A.workload_inputs(w, 0)
    n0 = list(st.n)
    res = O.decode_step(model, st, h, w.budgets())
    sh = model.shape
    for i in range(w.batch):
        # the routed result is the composition of the executed blocks only
        x = h[i].astype(np.float64)
        st_ref = A.build_state(w.shape, w.seed, w.contexts(), seqs=[i])
        for l in [0] + res.sel[i] + [sh.n_layers - 1]:
            K, V = st_ref.get(l, i)
            x, _, _ = O.decoder_layer(sh, model.layer(l), x, K, V, n0[i], round_act=(l != 0))
        np.testing.assert_array_equal(res.h_out[i], x)
        for l in range(sh.n_layers):
            K, V = st.get(l, i)
            assert K.shape[0] == n0[i] + 1
            if res.mask[i, l]:
                assert np.any(K[-1] != 0) and np.any(V[-1] != 0)
            else:
                assert not np.any(K[-1]) and not np.any(V[-1])


def test_compaction_rows_are_ascending_and_complete():
    w = C.T_GQA
    rng = np.random.default_rng(10)
    L = w.shape.n_layers
    sel = [sorted(rng.choice(np.arange(1, L - 1), size=int(rng.integers(1, L - 1)), replace=False).tolist())
           for _ in range(w.batch)]
    rows = O.compaction(sel, L)
    assert rows[0] == list(range(w.batch)) and rows[-1] == list(range(w.batch))
    for l in range(1, L - 1):
        assert rows[l] == sorted(rows[l])
        assert set(rows[l]) == {i for i in range(w.batch) if l in sel[i]}


def test_rerouting_every_decode_step():
    """Routes are recomputed each step from that step's state (Sec. 4.3,
    'Recompute'): different inputs at the same state give different sets, and
    a multi-step run changes sets across steps."""
    w = C.T_F32
    model = A.build_model(w.shape, w.seed)
    st = A.build_state(w.shape, w.seed, w.contexts())
    k = w.budgets()
    r1 = O.first_layer_and_route(model, st, A.workload_inputs(w, 0), k)
    r2 = O.first_layer_and_route(model, st, A.workload_inputs(w, 1), k)
    assert r1.sel != r2.sel
    assert not np.allclose(r1.scores, r2.scores)
    # the state advanced by one step changes the scores for the same input
    O.decode_step(model, st, A.workload_inputs(w, 0), k)
    r3 = O.first_layer_and_route(model, st, A.workload_inputs(w, 0), k)
    assert not np.allclose(r1.scores, r3.scores)


def test_cache_grows_by_one_position_per_step():
    w = C.T_F32
    _, st, res = _run(w, steps=2)
    n0 = w.contexts()
    for i in range(w.batch):
        assert st.n[i] == n0[i] + 2
        for l in range(w.shape.n_layers):
            K, V = st.get(l, i)
            assert K.shape[0] == n0[i] + 2
            np.testing.assert_array_equal(K[-1], res[1].kv_new[(l, i)][0])
            np.testing.assert_array_equal(V[-2], res[0].kv_new[(l, i)][1])


def test_budget_out_of_range_rejected():
    w = C.T_F32
    model = A.build_model(w.shape, w.seed)
    st = A.build_state(w.shape, w.seed, w.contexts())
    with pytest.raises(ValueError):
        O.first_layer_and_route(model, st, A.workload_inputs(w, 0), [0] * w.batch)
    with pytest.raises(ValueError):
        O.first_layer_and_route(model, st, A.workload_inputs(w, 0), [w.shape.l_mid + 1] * w.batch)
