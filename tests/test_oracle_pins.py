"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test ties an oracle function to something other than itself: a value the
paper prints, a closed form, an invariant of the method, or a textbook
library routine (torch float64) computing the same definition another way.
"""
import dataclasses
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
    with np.errstate(invalid="ignore"):   # the NaN patterns (signalling ones among them)
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


def _textbook_layer_prefill(sh, W, X, kv_cast=None, attn_mask=None):
    """A Llama decoder layer over a whole sequence with torch float64 routines
    (F.rms_norm, F.linear, causal SDPA, complex-rotation RoPE).  kv_cast, if
    given, is applied to the keys and values (their storage type)."""
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
    if kv_cast is not None:
        k, v = kv_cast(k), kv_cast(v)
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
        h, k_t, v_t = O.decoder_layer(sh, W, X[n][None], [(Kt[:n], Vt[:n])], [n])
        np.testing.assert_allclose(h[0], H[n], rtol=1e-11, atol=1e-11)
        np.testing.assert_allclose(k_t[0], Kt[n], rtol=1e-11, atol=1e-11)
        np.testing.assert_allclose(v_t[0], Vt[n], rtol=1e-11, atol=1e-11)


def test_bf16_cache_is_the_only_rounding():
    """A bf16 shape stores its new K/V as bfloat16 (torch's round-to-nearest-
    even) and computes everything else in float64: decoding token n equals
    the textbook float64 causal pass whose keys and values are cast to bf16,
    to float64 rounding error."""
    rng = np.random.default_rng(7)
    sh = _tiny_shape(dtype="bf16", n_q=6, n_kv=2)
    W = _rand_layer(sh, rng, True)
    T = 9
    X = rng.standard_normal((T, sh.d_model))
    cast = lambda a: a.to(torch.bfloat16).to(torch.float64)
    H, Kt, Vt = _textbook_layer_prefill(sh, W, X, kv_cast=cast)
    for n in (0, 4, T - 1):
        h, k_t, v_t = O.decoder_layer(sh, W, X[n][None], [(Kt[:n], Vt[:n])], [n])
        np.testing.assert_array_equal(k_t[0], Kt[n])
        np.testing.assert_array_equal(v_t[0], Vt[n])
        np.testing.assert_allclose(h[0], H[n], rtol=1e-11, atol=1e-11)
    # and the rounding is really there: the unrounded textbook layer differs
    H32, _, _ = _textbook_layer_prefill(sh, W, X)
    assert np.max(np.abs(H32[T - 1] - H[T - 1])) > 1e-6


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


def _linear_readback_model(sh, rng, W0):
    """A model whose Decision Module is linear in its input (SiLU driven into
    its linear regime by a large bias that the second layer removes), with
    s_j = x_j: the scores read back the first n_cand entries of the pooled
    half of the router input."""
    d, Lm = sh.d_model, sh.n_cand
    big = 60.0
    w1 = np.zeros((2 * d, 2 * d)); w1[np.arange(2 * d), np.arange(2 * d)] = 1.0
    w2 = np.zeros((Lm, 2 * d)); w2[np.arange(Lm), np.arange(Lm)] = 1.0
    dm = O.DecisionModule(w1=w1, b1=np.full(2 * d, big), w2=w2, b2=np.full(Lm, -big))
    return O.Model(sh, lambda l: W0, dm)


@pytest.mark.parametrize("feature", ["v", "k", "kv"])
@pytest.mark.parametrize("ctx_layer", [0, 1])
def test_router_pools_newest_token_with_cache(feature, ctx_layer):
    """Reading the pool back through a linear DM shows the mean over the n
    cached positions AND the newest token's entry of the context layer's cache
    (Sec. 4.3): V, K (as cached, after RoPE) or their element-wise sum K + V
    (Sec. 5.4), concatenated before the hidden state."""
    rng = np.random.default_rng(9)
    sh = dataclasses.replace(_tiny_shape(n_q=4, n_kv=2, hd=4, L=2 + 16 + ctx_layer, d=16),
                             feature=feature, ctx_layer=ctx_layer)
    W0 = _rand_layer(sh, rng)
    model = _linear_readback_model(sh, rng, W0)
    n = 6
    st = O.KVState([n])
    Kc = {l: rng.standard_normal((n, 2, 4)) for l in range(ctx_layer + 1)}
    Vc = {l: rng.standard_normal((n, 2, 4)) for l in range(ctx_layer + 1)}
    for l in range(ctx_layer + 1):
        st.set(l, 0, Kc[l], Vc[l])
    rr = O.first_layers_and_route(model, st, rng.standard_normal((1, sh.d_model)), [3])
    k_t, v_t = rr.kv_new[(ctx_layer, 0)]
    K = np.concatenate([Kc[ctx_layer], k_t[None]])
    V = np.concatenate([Vc[ctx_layer], v_t[None]])
    F = {"v": V, "k": K, "kv": K + V}[feature]
    expect = O.expand_kv_heads(F.sum(axis=0).reshape(-1) / (n + 1), sh)[:sh.n_cand]
    np.testing.assert_allclose(rr.scores[0], expect, rtol=0, atol=1e-9)
    # the selection names layers c+1 .. L-2
    assert all(ctx_layer + 1 <= l <= sh.n_layers - 2 for l in rr.sel[0]) and len(rr.sel[0]) == 3


def test_router_hidden_half_is_state_after_context_layer():
    """The second half of the router input is the newest token's hidden state
    after layer c: with a DM reading x[d + j], the scores equal H_{c+1}."""
    rng = np.random.default_rng(12)
    for c in (0, 2):
        sh = dataclasses.replace(_tiny_shape(n_q=4, n_kv=2, hd=4, L=12, d=16), ctx_layer=c)
        d, Lm = sh.d_model, sh.n_cand
        W = [_rand_layer(sh, rng) for _ in range(sh.n_layers)]
        big = 60.0
        w1 = np.zeros((2 * d, 2 * d)); w1[np.arange(2 * d), np.arange(2 * d)] = 1.0
        w2 = np.zeros((Lm, 2 * d)); w2[np.arange(Lm), d + np.arange(Lm)] = 1.0
        dm = O.DecisionModule(w1=w1, b1=np.full(2 * d, big), w2=w2, b2=np.full(Lm, -big))
        model = O.Model(sh, lambda l: W[l], dm)
        st = O.KVState([5])
        for l in range(sh.n_layers):
            st.set(l, 0, rng.standard_normal((5, 2, 4)), rng.standard_normal((5, 2, 4)))
        x = rng.standard_normal((1, d))
        h = x.copy()
        for l in range(c + 1):
            h, _, _ = O.decoder_layer(sh, W[l], h, [st.get(l, 0)], [5])
        rr = O.first_layers_and_route(model, st, x, [2])
        np.testing.assert_allclose(rr.scores[0], h[0, :Lm], rtol=0, atol=1e-9)


def test_budget_predictor_matches_torch_policy():
    """k^ = argmax of a Linear-SiLU-Linear categorical policy over
    A = {1..n_cand} (Sec. 4.4, Eq. 3), ties to the smaller k; b^ = (k^+2)/L."""
    rng = np.random.default_rng(13)
    d2, r, Lm = 20, 9, 11
    bp = O.BudgetPredictor(w1=rng.standard_normal((r, d2)), b1=rng.standard_normal(r),
                           w2=rng.standard_normal((Lm, r)), b2=rng.standard_normal(Lm))
    mlp = torch.nn.Sequential(torch.nn.Linear(d2, r), torch.nn.SiLU(), torch.nn.Linear(r, Lm)).double()
    with torch.no_grad():
        mlp[0].weight.copy_(torch.from_numpy(bp.w1)); mlp[0].bias.copy_(torch.from_numpy(bp.b1))
        mlp[2].weight.copy_(torch.from_numpy(bp.w2)); mlp[2].bias.copy_(torch.from_numpy(bp.b2))
    seen = set()
    for _ in range(200):
        x = rng.standard_normal(d2) * 3
        pi = torch.softmax(mlp(torch.from_numpy(x)), -1).detach()
        ref = int(torch.argmax(pi)) + 1
        assert O.predict_k(bp, x) == ref
        seen.add(ref)
    assert len(seen) > 2       # the policy is input-dependent
    # ties go to the smaller k
    tie = O.BudgetPredictor(w1=np.zeros((1, 2)), b1=np.zeros(1), w2=np.zeros((5, 1)),
                            b2=np.array([0.0, 2.0, 1.0, 2.0, 2.0]))
    assert O.predict_k(tie, np.zeros(2)) == 2
    assert O.k_to_budget(O.predict_k(tie, np.zeros(2)), 32) == 4 / 32


def test_predicted_budget_drives_selection():
    """A sequence without a budget (k = 0) executes exactly k^ routed layers,
    the top-k^ of its scores; a sequence with one ignores the predictor."""
    w = C.T_PRED
    model = A.build_model(w.shape, w.seed)
    st = A.build_state(w.shape, w.seed, w.contexts())
    k = w.budgets()
    assert (k == 0).any() and (k > 0).any()
    rr = O.first_layers_and_route(model, st, A.workload_inputs(w, 0), k)
    sh = model.shape
    for i in range(w.batch):
        K, V = st.get(sh.ctx_layer, i)
        kt, vt = rr.kv_new[(sh.ctx_layer, i)]
        x = O.router_input(sh, np.concatenate([K, kt[None]]), np.concatenate([V, vt[None]]), rr.h[i])
        want = O.predict_k(model.predictor, x) if k[i] == 0 else int(k[i])
        assert rr.k[i] == want and len(rr.sel[i]) == want
        assert rr.sel[i] == O.top_k_layers(rr.scores[i], want, sh.first_candidate)
    assert len({rr.k[i] for i in range(w.batch) if k[i] == 0}) > 1


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
        x = h[i][None].astype(np.float64)
        st_ref = A.build_state(w.shape, w.seed, w.contexts(), seqs=[i])
        for l in [0] + res.sel[i] + [sh.n_layers - 1]:
            x, _, _ = O.decoder_layer(sh, model.layer(l), x, [st_ref.get(l, i)], [n0[i]])
        # (the step runs each layer on all its rows at once: equal to rounding)
        np.testing.assert_allclose(res.h_out[i], x[0], rtol=1e-12, atol=1e-12)
        for l in range(sh.n_layers):
            K, V = st.get(l, i)
            assert K.shape[0] == n0[i] + 1
            if res.mask[i, l]:
                assert np.any(K[-1] != 0) and np.any(V[-1] != 0)
            else:
                assert not np.any(K[-1]) and not np.any(V[-1])


def test_masked_skip_attends_only_executed_positions():
    """Masked variant (Sec. 6): a skipped layer stores nothing, so its later
    attention is the zero-filled cache's attention with the skipped positions
    masked out (torch SDPA with a boolean mask over the zero-filled cache)."""
    rng = np.random.default_rng(14)
    sh = _tiny_shape(n_q=4, n_kv=2)
    W = _rand_layer(sh, rng)
    n = 10
    K = rng.standard_normal((n, 2, 8))
    V = rng.standard_normal((n, 2, 8))
    skipped = [2, 3, 7]
    K[skipped] = 0.0
    V[skipped] = 0.0
    keep = [p for p in range(n) if p not in skipped]
    x = rng.standard_normal((1, sh.d_model))
    hm, km, vm = O.decoder_layer(sh, W, x, [(K[keep], V[keep])], [n])
    # reference: textbook attention for the query at position n, mask over [cache; new]
    t = lambda a: torch.from_numpy(np.asarray(a))
    xn = Fnn.rms_norm(t(x), (sh.d_model,), t(W.attn_norm), eps=sh.rms_eps)
    q = O.rope(Fnn.linear(xn, t(W.w_q), t(W.b_q)).numpy().reshape(4, 8), n, sh.rope_theta)
    Kall = np.concatenate([K, km])
    Vall = np.concatenate([V, vm])
    allowed = torch.ones(1, n + 1, dtype=torch.bool)
    allowed[0, skipped] = False
    att = Fnn.scaled_dot_product_attention(t(q)[:, None, :], t(Kall).permute(1, 0, 2).repeat_interleave(2, 0),
                                           t(Vall).permute(1, 0, 2).repeat_interleave(2, 0),
                                           attn_mask=allowed)[:, 0, :].reshape(1, -1)
    h = t(x) + Fnn.linear(att, t(W.w_o))
    xn2 = Fnn.rms_norm(h, (sh.d_model,), t(W.ffn_norm), eps=sh.rms_eps)
    h = h + Fnn.linear(Fnn.silu(Fnn.linear(xn2, t(W.w_gate))) * Fnn.linear(xn2, t(W.w_up)), t(W.w_down))
    np.testing.assert_allclose(hm, h.numpy(), rtol=1e-11, atol=1e-11)
    # the zero-filled variant differs (the zeros take part with logit 0)
    hz, _, _ = O.decoder_layer(sh, W, x, [(K, V)], [n])
    assert np.max(np.abs(hz - hm)) > 1e-6


def test_masked_skip_cache_lengths_and_full_budget():
    """In the masked variant a layer's cache grows only when it executes; at
    k = n_cand nothing is skipped and both variants agree bit-exactly."""
    wz = C.T_F32
    wm = C.with_shape(wz, skip_kv="masked")
    for k_all in (None, wz.shape.n_cand):
        outs = []
        for w in (wz, wm):
            model = A.build_model(w.shape, w.seed)
            st = A.build_state(w.shape, w.seed, w.contexts())
            kk = w.budgets() if k_all is None else [k_all] * w.batch
            res = [O.decode_step(model, st, A.workload_inputs(w, t), kk) for t in range(2)]
            outs.append((res, st))
        (rz, sz), (rm, sm) = outs
        if k_all is not None:
            for i in range(wz.batch):
                np.testing.assert_array_equal(rz[1].h_out[i], rm[1].h_out[i])
        else:
            n0 = wz.contexts()
            for i in range(wz.batch):
                for l in range(wz.shape.n_layers):
                    execs = int(rm[0].mask[i, l]) + int(rm[1].mask[i, l])
                    assert sm.length(l, i) == n0[i] + execs
                    assert sz.length(l, i) == n0[i] + 2
            assert any(not np.array_equal(rz[1].h_out[i], rm[1].h_out[i]) for i in range(wz.batch))


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
    r1 = O.first_layers_and_route(model, st, A.workload_inputs(w, 0), k)
    r2 = O.first_layers_and_route(model, st, A.workload_inputs(w, 1), k)
    assert r1.sel != r2.sel
    assert not np.allclose(r1.scores, r2.scores)
    # the state advanced by one step changes the scores for the same input
    O.decode_step(model, st, A.workload_inputs(w, 0), k)
    r3 = O.first_layers_and_route(model, st, A.workload_inputs(w, 0), k)
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
        O.first_layers_and_route(model, st, A.workload_inputs(w, 0), [0] * w.batch)
    with pytest.raises(ValueError):
        O.first_layers_and_route(model, st, A.workload_inputs(w, 0), [w.shape.l_mid + 1] * w.batch)


# ---------------------------------------------------------------------------
# Prefill with routing (Sec. 4.1; App. E "Prefill vs. Decode")
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_prefill_layer_equals_textbook_causal_pass(dtype):
    """T new tokens after n cached ones: rows n..T-1 of the textbook causal
    pass over all T tokens (keys and values cast to the cache type)."""
    rng = np.random.default_rng(15)
    sh = _tiny_shape(dtype=dtype, n_q=6, n_kv=2)
    W = _rand_layer(sh, rng, True)
    T = 13
    X = rng.standard_normal((T, sh.d_model))
    cast = (lambda a: a.to(torch.bfloat16).to(torch.float64)) if dtype == "bf16" else None
    H, Kt, Vt = _textbook_layer_prefill(sh, W, X, kv_cast=cast)
    for n in (0, 5):
        h, k, v = O.prefill_layer(sh, W, X[n:], Kt[:n], Vt[:n], n)
        np.testing.assert_allclose(h, H[n:], rtol=1e-11, atol=1e-11)
        np.testing.assert_array_equal(k, Kt[n:]) if dtype == "bf16" else np.testing.assert_allclose(
            k, Kt[n:], rtol=1e-11, atol=1e-11)


def _prompts(w, lengths, seed=21):
    rng = np.random.default_rng(seed)
    return [rng.standard_normal((t, w.shape.d_model)) for t in lengths]


@pytest.mark.parametrize("variant", ["zero", "masked-c1-kv"])
def test_routed_prefill_equals_decoding_the_prompt_with_the_route_fixed(variant):
    """A routed prefill equals decoding the prompt token by token (Eq. 9) with
    the prefill's route held fixed (the 'Reuse' strategy of Sec. 5.3): same
    hidden states for every token, same caches."""
    w = C.T_F32 if variant == "zero" else C.with_shape(C.T_F32, skip_kv="masked", ctx_layer=1, feature="kv",
                                                       n_layers=7)
    model = A.build_model(w.shape, w.seed)
    lengths = [5, 1, 9, 3, 6, 2]
    prompts = _prompts(w, lengths)
    st = A.build_state(w.shape, w.seed, w.contexts())
    st0 = A.build_state(w.shape, w.seed, w.contexts())
    k = w.budgets()
    pr = O.prefill(model, st, prompts, k)
    assert [len(s) for s in pr.sel] == list(k)
    for i in range(w.batch):
        st_i = O.KVState([w.contexts()[i]])          # sequence i alone
        for l in range(w.shape.n_layers):
            st_i.set(l, 0, *st0.get(l, i))
        for t in range(lengths[i]):
            r = O.decode_step(model, st_i, prompts[i][t][None], [k[i]], override_sel=lambda rr: [pr.sel[i]])
            np.testing.assert_allclose(r.h_out[0], pr.h_out[i][t], rtol=1e-10, atol=1e-10)
        for l in range(w.shape.n_layers):
            Ka, Va = st.get(l, i)
            Kb, Vb = st_i.get(l, 0)
            assert Ka.shape == Kb.shape
            np.testing.assert_allclose(Ka, Kb, rtol=1e-10, atol=1e-10)
            np.testing.assert_allclose(Va, Vb, rtol=1e-10, atol=1e-10)
        assert st.n[i] == w.contexts()[i] + lengths[i]


def test_prefill_route_reads_the_pooled_prompt_and_last_token():
    """The prefill route of a prompt pools the context layer's cache over the
    cached positions and every prompt token, and takes the last prompt
    token's hidden state after layer c."""
    rng = np.random.default_rng(16)
    sh = _tiny_shape(n_q=4, n_kv=2, hd=4, L=2 + 16, d=16)
    W0 = _rand_layer(sh, rng)
    model = _linear_readback_model(sh, rng, W0)
    n, T = 4, 7
    st = O.KVState([n])
    Kc, Vc = rng.standard_normal((n, 2, 4)), rng.standard_normal((n, 2, 4))
    for l in range(sh.n_layers):
        st.set(l, 0, Kc, Vc)
    X = rng.standard_normal((T, sh.d_model))
    pr = O.prefill(model, st, [X], [3])
    H1, kn, vn = O.prefill_layer(sh, W0, X, Kc, Vc, n)
    V = np.concatenate([Vc, vn])
    expect = O.expand_kv_heads(V.sum(axis=0).reshape(-1) / (n + T), sh)[:sh.n_cand]
    np.testing.assert_allclose(pr.scores[0], expect, rtol=0, atol=1e-9)
    # a DM reading the hidden half x[d + j]: the last token after layer 0
    d, Lm = sh.d_model, sh.n_cand
    model.dm.w2 = np.zeros((Lm, 2 * d))
    model.dm.w2[np.arange(Lm), d + np.arange(Lm)] = 1.0
    st = O.KVState([n])
    for l in range(sh.n_layers):
        st.set(l, 0, Kc, Vc)
    pr = O.prefill(model, st, [X], [3])
    np.testing.assert_allclose(pr.scores[0], H1[-1, :Lm], rtol=0, atol=1e-9)


def test_prefill_skipped_layers_store_zeros_at_every_prompt_position():
    w = C.T_F32
    model = A.build_model(w.shape, w.seed)
    st = A.build_state(w.shape, w.seed, w.contexts())
    lengths = [3, 4, 1, 2, 5, 2]
    pr = O.prefill(model, st, _prompts(w, lengths), w.budgets())
    n0 = w.contexts()
    for i in range(w.batch):
        for l in range(w.shape.n_layers):
            K, V = st.get(l, i)
            assert K.shape[0] == n0[i] + lengths[i]
            new = K[n0[i]:]
            assert (not new.any()) == (not pr.mask[i, l])
