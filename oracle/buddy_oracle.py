"""CPU oracle for BUDDY's budget-routed decode step (and its prefill routing).

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute this module; only tests/, __graft_entry__.smoke() and bench.py's
cpu_baseline / reference legs use it.  It shares no code with the CUDA path.

What it computes (plain numpy, float64 arithmetic):

  * Layer skipping (Sec. 3.1, Eq. 1): an executed block adds F_l(H) to the
    residual, a skipped block is the identity.
  * First and last blocks always execute; the L_mid = L - 2 middle blocks are
    the candidates (Sec. 4.2.1).  With a context layer c > 0 (App. D,
    "Ablation on the Start Layer") blocks 0..c all execute and the candidates
    are c+1 .. L-2.
  * KV-aware planner (Sec. 4.3): the context layer's cache, with the newest
    token's entry appended, is mean-pooled over positions.  The pooled feature
    G_t is the value states (default, Sec. 5 "Hyper-parameters"), the key
    states, or their element-wise sum (Sec. 5.4, "Hidden-State Features").  It
    is expanded to width d by repeating each KV head over its query-head group
    and concatenated with the newest token's hidden state after layer c.
  * Decision Module (Sec. 4.2.3, App. C.1): Linear -> SiLU -> Linear gives one
    score per candidate layer; a prior p~ is fused as s' = s + omega * p~
    (Eq. 2).
  * Deterministic top-k (Eq. 2): the k highest s' execute; equal scores are
    broken by the lower layer index.  Softmax is monotone, so ranking s' gives
    the same set.
  * Budget Predictor (Sec. 4.4): a categorical policy over A = {1..L_mid}
    from the same router input; k^ = argmax (ties to the smaller k) replaces
    the budget of sequences that give none (k = 0 here).
  * Grouping by mask (App. C.1): block l runs on the sequences that selected it.
  * Skipped layers store zero K and V at the new position (Sec. 6,
    "Limitations"), so every layer's cache grows by one position per step;
    the masked variant (the "more efficient KV-cache strategies" Sec. 6 leaves
    to future work) stores nothing, so a layer's attention reads only the
    positions at which that layer executed.
  * Decoder block and KV cache (App. E "Background", Eq. 9): Llama-style block
    — RMSNorm, Q/K/V projections (optional bias), rotate-half RoPE at the
    token's position, grouped-query attention over [K_cache; K_t],
    [V_cache; V_t], output projection, RMSNorm, SwiGLU MLP d -> F -> d.
  * Prefill (Sec. 4.1, App. E "Prefill vs. Decode"): the prompt's tokens pass
    the first blocks with causal attention, one route is chosen per prompt
    from the pooled prompt context and the last prompt token's hidden state,
    and the selected blocks run on all of that prompt's tokens.

Precision.  Every operation is float64.  The only rounding is that of the KV
cache: for "bf16" shapes the K and V a block writes are stored as bfloat16
(round to nearest even), the storage type of the cache, and read back from
it.  Inputs (weights, prefilled caches, hidden states) are the bf16 / fp32
values of the seeded generator, converted exactly.

Parity status: pinned by tests/test_oracle_pins.py (closed forms, invariants,
library reductions, paper-printed values); routed hidden-state *values* on
random weights have no independent reference beyond those pins.
"""
from __future__ import annotations

import dataclasses
from typing import Callable, Dict, List, Optional, Sequence

import numpy as np


# ---------------------------------------------------------------------------
# Number formats
# ---------------------------------------------------------------------------
def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact value of bfloat16 bit patterns (uint16) as float64."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bfloat16 (ties to even), via float32; returns float64."""
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


# ---------------------------------------------------------------------------
# Model description
# ---------------------------------------------------------------------------
@dataclasses.dataclass
class Shape:
    n_layers: int
    d_model: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn_dim: int
    dm_hidden: int
    dtype: str            # "f32" | "bf16": storage type of the KV cache
    rms_eps: float
    rope_theta: float
    feature: str = "v"    # planner feature G_t: "v", "k" or "kv" (element-wise sum)
    ctx_layer: int = 0    # c: layers 0..c always run; the planner reads layer c's cache
    skip_kv: str = "zero"  # "zero": skipped layers store zero K/V; "masked": they store nothing

    @property
    def l_mid(self) -> int:
        return self.n_layers - 2

    @property
    def first_candidate(self) -> int:
        return self.ctx_layer + 1

    @property
    def n_cand(self) -> int:
        """Number of routed layers: c+1 .. L-2."""
        return self.n_layers - 2 - self.ctx_layer

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    def store(self, x: np.ndarray) -> np.ndarray:
        """Value of a K/V entry as the cache stores it."""
        return round_to_bf16(x) if self.dtype == "bf16" else np.asarray(x, dtype=np.float64)


@dataclasses.dataclass
class LayerWeights:
    """float64 copies of one decoder layer, nn.Linear layout [out, in]."""
    attn_norm: np.ndarray
    w_q: np.ndarray
    w_k: np.ndarray
    w_v: np.ndarray
    w_o: np.ndarray
    ffn_norm: np.ndarray
    w_gate: np.ndarray
    w_up: np.ndarray
    w_down: np.ndarray
    b_q: Optional[np.ndarray] = None
    b_k: Optional[np.ndarray] = None
    b_v: Optional[np.ndarray] = None


@dataclasses.dataclass
class DecisionModule:
    w1: np.ndarray        # [r, 2d]
    b1: np.ndarray        # [r]
    w2: np.ndarray        # [n_cand, r]
    b2: np.ndarray        # [n_cand]
    prior: Optional[np.ndarray] = None   # p~ [n_cand]
    omega: float = 0.0


@dataclasses.dataclass
class BudgetPredictor:
    """Categorical policy over A = {1..n_cand} (Sec. 4.4), Linear-SiLU-Linear."""
    w1: np.ndarray        # [r_p, 2d]
    b1: np.ndarray        # [r_p]
    w2: np.ndarray        # [n_cand, r_p]
    b2: np.ndarray        # [n_cand]


@dataclasses.dataclass
class Model:
    shape: Shape
    layer: Callable[[int], LayerWeights]   # float64 weights of layer l, 0-based
    dm: DecisionModule
    predictor: Optional[BudgetPredictor] = None


class KVState:
    """Per-(layer, sequence) caches with room to grow.

    n[i] is the number of tokens of sequence i (the position of its next
    token).  The cache of (layer l, sequence i) holds `length(l, i)` entries
    [length, n_kv, hd] float64 (stored values); it equals n[i] unless the
    masked skip variant left some positions out.  An optional loader supplies
    a cache on first use (positions 0..n_i-1 as prefilled), so that large
    workloads can be evaluated one layer at a time; `drop(l)` forgets a
    layer's caches."""

    def __init__(self, n_ctx: Sequence[int], loader: Optional[Callable[[int, int], tuple]] = None):
        self.n = [int(v) for v in n_ctx]
        self.loader = loader
        self._buf: Dict[tuple, list] = {}      # (l, i) -> [K, V, length]

    def set(self, layer: int, seq: int, K: np.ndarray, V: np.ndarray):
        K = np.asarray(K, np.float64)
        V = np.asarray(V, np.float64)
        assert K.shape == V.shape and K.ndim == 3
        n = K.shape[0]
        cap = max(16, 2 * n)
        Kb = np.empty((cap,) + K.shape[1:])
        Vb = np.empty((cap,) + K.shape[1:])
        Kb[:n], Vb[:n] = K, V
        self._buf[(layer, seq)] = [Kb, Vb, n]

    def _entry(self, layer: int, seq: int):
        if (layer, seq) not in self._buf:
            if self.loader is None:
                raise KeyError((layer, seq))
            K, V = self.loader(layer, seq)
            self.set(layer, seq, K, V)
        return self._buf[(layer, seq)]

    def get(self, layer: int, seq: int):
        """(K, V) of the stored positions, [length, n_kv, hd] views."""
        Kb, Vb, n = self._entry(layer, seq)
        return Kb[:n], Vb[:n]

    def length(self, layer: int, seq: int) -> int:
        return self._entry(layer, seq)[2]

    def append(self, layer: int, seq: int, k: np.ndarray, v: np.ndarray):
        """Append entries k, v [t, n_kv, hd] (or [n_kv, hd] for one)."""
        e = self._entry(layer, seq)
        k = np.asarray(k, np.float64)
        v = np.asarray(v, np.float64)
        if k.ndim == 2:
            k, v = k[None], v[None]
        n, t = e[2], k.shape[0]
        if n + t > e[0].shape[0]:
            cap = max(2 * e[0].shape[0], n + t)
            for j in (0, 1):
                nb = np.empty((cap,) + e[j].shape[1:])
                nb[:n] = e[j][:n]
                e[j] = nb
        e[0][n:n + t] = k
        e[1][n:n + t] = v
        e[2] = n + t

    def drop(self, layer: int):
        for key in [k for k in self._buf if k[0] == layer]:
            del self._buf[key]

    def has(self, layer: int, seq: int) -> bool:
        return (layer, seq) in self._buf or self.loader is not None


# ---------------------------------------------------------------------------
# Building blocks of the Llama-style layer (App. E "Background"; Sec. 5 models)
# ---------------------------------------------------------------------------
def rms_norm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm: x / sqrt(mean(x^2) + eps) * gain, over the last axis."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * gain


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def linear(x: np.ndarray, w: np.ndarray, b: Optional[np.ndarray] = None) -> np.ndarray:
    """nn.Linear: x @ w^T (+ b), rows of x independent."""
    y = x @ w.T
    return y if b is None else y + b


def rope(x: np.ndarray, pos: int, theta: float) -> np.ndarray:
    """Rotary embedding, rotate-half convention, on [..., hd]: the pair
    (x_j, x_{j+hd/2}) is rotated by angle pos * theta^(-2j/hd)."""
    hd = x.shape[-1]
    half = hd // 2
    j = np.arange(half, dtype=np.float64)
    ang = float(pos) * np.power(float(theta), -2.0 * j / hd)
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def softmax(z: np.ndarray) -> np.ndarray:
    e = np.exp(z - np.max(z, axis=-1, keepdims=True))
    return e / np.sum(e, axis=-1, keepdims=True)


def decode_attention(q: np.ndarray, K: np.ndarray, V: np.ndarray, group: int,
                     k_t: Optional[np.ndarray] = None, v_t: Optional[np.ndarray] = None) -> np.ndarray:
    """Attn(Q_t, [K_cache; K_t], [V_cache; V_t]) for one token (Eq. 9).
    q [n_q, hd]; K, V [n, n_kv, hd] the cached positions; k_t, v_t [n_kv, hd]
    the token's own entry (appended as the last position when given).  Query
    head h reads KV head h // group."""
    n_q, hd = q.shape
    out = np.empty_like(q)
    for g in range(n_q // group):
        qg = q[g * group:(g + 1) * group]                    # [G, hd]
        logits = qg @ K[:, g, :].T / np.sqrt(hd)             # [G, n]
        if k_t is not None:
            logits = np.concatenate([logits, (qg @ k_t[g])[:, None] / np.sqrt(hd)], axis=1)
        p = softmax(logits)
        o = p[:, :K.shape[0]] @ V[:, g, :]
        if v_t is not None:
            o = o + p[:, K.shape[0]:] * v_t[g][None, :]
        out[g * group:(g + 1) * group] = o
    return out


def qkv_project(sh: Shape, W: LayerWeights, H: np.ndarray, pos: Sequence[int]):
    """RMSNorm, Q/K/V projections and RoPE for rows H [m, d] at token positions
    pos[j].  Returns q [m, n_q, hd] and the stored k, v [m, n_kv, hd]."""
    m = H.shape[0]
    hd = sh.head_dim
    xn = rms_norm(H, W.attn_norm, sh.rms_eps)
    q = linear(xn, W.w_q, W.b_q).reshape(m, sh.n_q_heads, hd)
    k = linear(xn, W.w_k, W.b_k).reshape(m, sh.n_kv_heads, hd)
    v = linear(xn, W.w_v, W.b_v).reshape(m, sh.n_kv_heads, hd)
    for j in range(m):
        q[j] = rope(q[j], pos[j], sh.rope_theta)
        k[j] = rope(k[j], pos[j], sh.rope_theta)
    return q, sh.store(k), sh.store(v)


def block_tail(sh: Shape, W: LayerWeights, H: np.ndarray, attn: np.ndarray) -> np.ndarray:
    """Output projection + residual, then RMSNorm + SwiGLU MLP + residual."""
    H = H + linear(attn, W.w_o)
    xn2 = rms_norm(H, W.ffn_norm, sh.rms_eps)
    return H + linear(silu(linear(xn2, W.w_gate)) * linear(xn2, W.w_up), W.w_down)


def decoder_layer(sh: Shape, W: LayerWeights, H: np.ndarray, caches: Sequence[tuple], pos: Sequence[int]):
    """One executed block for m independent decode tokens (one per sequence).
    H [m, d]; caches[j] = (K, V) [n_j, n_kv, hd] the row's stored positions;
    pos[j] the token's position.  Returns (H + F_l(H), k, v) with k, v
    [m, n_kv, hd] the entries to store."""
    H = np.atleast_2d(np.asarray(H, dtype=np.float64))
    q, k, v = qkv_project(sh, W, H, pos)
    attn = np.stack([decode_attention(q[j], caches[j][0], caches[j][1], sh.group, k[j], v[j]).reshape(-1)
                     for j in range(H.shape[0])])
    return block_tail(sh, W, H, attn), k, v


def prefill_layer(sh: Shape, W: LayerWeights, X: np.ndarray, K_cache: np.ndarray, V_cache: np.ndarray,
                  p0: int):
    """One executed block over T new tokens of one sequence (causal): token t
    at position p0 + t attends to the n cached positions and new tokens 0..t.
    Returns (X + F_l(X), k, v) with k, v [T, n_kv, hd] as stored."""
    X = np.asarray(X, dtype=np.float64)
    T = X.shape[0]
    q, k, v = qkv_project(sh, W, X, [p0 + t for t in range(T)])
    attn = np.empty((T, sh.n_q_heads * sh.head_dim))
    for t in range(T):
        Kt = np.concatenate([K_cache, k[:t + 1]], axis=0)
        Vt = np.concatenate([V_cache, v[:t + 1]], axis=0)
        attn[t] = decode_attention(q[t], Kt, Vt, sh.group).reshape(-1)
    return block_tail(sh, W, X, attn), k, v


# ---------------------------------------------------------------------------
# Router: KV-aware planner + Decision Module + top-k (Sec. 4.2, 4.3) and the
# Budget Predictor (Sec. 4.4)
# ---------------------------------------------------------------------------
def planner_feature(sh: Shape, K: np.ndarray, V: np.ndarray) -> np.ndarray:
    """Per-position feature of the context layer's cache: V, K or K + V."""
    if sh.feature == "v":
        return V
    if sh.feature == "k":
        return K
    if sh.feature == "kv":
        return K + V
    raise ValueError(sh.feature)


def pool_context(F: np.ndarray) -> np.ndarray:
    """G_t: arithmetic mean over positions of the feature F [n, n_kv, hd]
    (the cache including the newest token) -> [n_kv * hd]."""
    return np.mean(F, axis=0).reshape(-1)


def expand_kv_heads(g: np.ndarray, sh: Shape) -> np.ndarray:
    """Repeat each KV head over its query-head group: width n_kv*hd -> d
    (query head h uses KV head h // group)."""
    g = g.reshape(sh.n_kv_heads, sh.head_dim)
    return np.repeat(g, sh.group, axis=0).reshape(-1)


def router_input(sh: Shape, K: np.ndarray, V: np.ndarray, h: np.ndarray) -> np.ndarray:
    """x = [G_t expanded to d ; h] (width 2d) from the context layer's cache
    (newest token included) and the newest token's hidden state after it."""
    return np.concatenate([expand_kv_heads(pool_context(planner_feature(sh, K, V)), sh), h])


def decision_scores(dm: DecisionModule, x: np.ndarray) -> np.ndarray:
    """s' = W2 SiLU(W1 x + b1) + b2 + omega * p~  (App. C.1; Eq. 2)."""
    s = dm.w2 @ silu(dm.w1 @ x + dm.b1) + dm.b2
    if dm.prior is not None:
        s = s + dm.omega * dm.prior
    return s


def predictor_logits(bp: BudgetPredictor, x: np.ndarray) -> np.ndarray:
    """Logits of pi(k | G_t) over k = 1..n_cand (Sec. 4.4)."""
    return bp.w2 @ silu(bp.w1 @ x + bp.b1) + bp.b2


def predict_k(bp: BudgetPredictor, x: np.ndarray) -> int:
    """k^ = argmax_k pi(k | G_t) (Eq. 3); softmax is monotone, so the argmax
    of the logits; ties go to the smaller k."""
    return int(np.argmax(predictor_logits(bp, x))) + 1


def top_k_layers(scores: np.ndarray, k: int, first: int = 1) -> List[int]:
    """Candidate layers first, first+1, ... (scores[j] belongs to layer
    first + j) with the k largest scores; ties go to the lower index.
    Returned ascending."""
    order = sorted(range(len(scores)), key=lambda j: (-scores[j], j))
    return sorted(j + first for j in order[:k])


def budget_to_k(b: float, L: int, fixed: int = 2) -> int:
    """k = round(b * L) - 2 (Eq. 2), clamped to the action space {1..L-2}
    (Sec. 4.4).  Python's round() ties to even.  `fixed` is the number of
    always-executed layers (2, or c + 2 with a context layer c: App. C.2's I)."""
    return int(min(max(round(b * L) - fixed, 1), L - fixed))


def k_to_budget(k: int, L: int, fixed: int = 2) -> float:
    """b = (k + 2) / L (Eq. 3): the +2 counts the first and last blocks."""
    return (k + fixed) / L


# ---------------------------------------------------------------------------
# The decode step
# ---------------------------------------------------------------------------
@dataclasses.dataclass
class RouteResult:
    h: np.ndarray                  # [B, d] hidden state after the context layer c
    scores: np.ndarray             # [B, n_cand] s'
    k: List[int]                   # budget used per sequence (given or predicted)
    sel: List[List[int]]           # per sequence, ascending executed routed layers
    kv_new: Dict[tuple, tuple]     # (layer <= c, seq) -> (k_t, v_t) written
    x: Optional[np.ndarray] = None  # [B, 2d] router inputs


@dataclasses.dataclass
class StepResult:
    h_out: Dict[int, np.ndarray]   # sequence -> final hidden state [d]
    scores: np.ndarray
    k: List[int]
    sel: List[List[int]]
    mask: np.ndarray               # [B, L] uint8
    rows: List[List[int]]          # per layer: ascending active sequences
    kv_new: Dict[tuple, tuple]     # (layer, seq) -> (k_t, v_t) as stored (zeros if skipped, zero mode)


def route(model: Model, x: np.ndarray, k: int):
    """Scores, budget and selection of one sequence from its router input."""
    sh = model.shape
    s = decision_scores(model.dm, x)
    kk = int(k)
    if kk == 0:
        if model.predictor is None:
            raise ValueError("budget 0 needs a Budget Predictor")
        kk = predict_k(model.predictor, x)
    if not 1 <= kk <= sh.n_cand:
        raise ValueError(f"budget k={k} outside [1, {sh.n_cand}]")
    return s, kk, top_k_layers(s, kk, sh.first_candidate)


def first_layers_and_route(model: Model, st: KVState, h_in: np.ndarray, k: Sequence[int]) -> RouteResult:
    """Layers 0..c on every sequence, then the router on every sequence."""
    sh = model.shape
    B = h_in.shape[0]
    c = sh.ctx_layer
    H = np.asarray(h_in, dtype=np.float64).copy()
    kv_new = {}
    for l in range(c + 1):
        H, kn, vn = decoder_layer(sh, model.layer(l), H, [st.get(l, i) for i in range(B)], st.n)
        for i in range(B):
            kv_new[(l, i)] = (kn[i], vn[i])
    scores = np.empty((B, sh.n_cand))
    ks, sel, xs = [], [], []
    for i in range(B):
        K, V = st.get(c, i)
        kt, vt = kv_new[(c, i)]
        x = router_input(sh, np.concatenate([K, kt[None]]), np.concatenate([V, vt[None]]), H[i])
        scores[i], kk, si = route(model, x, k[i])
        ks.append(kk)
        sel.append(si)
        xs.append(x)
    return RouteResult(H, scores, ks, sel, kv_new, np.stack(xs))


def compaction(sel: Sequence[Sequence[int]], L: int, first: int = 1) -> List[List[int]]:
    """Grouping by mask: for every layer, the ascending list of sequences that
    execute it (all sequences for layers < first and the last layer)."""
    B = len(sel)
    rows = [list(range(B)) for _ in range(first)]
    for l in range(first, L - 1):
        rows.append([i for i in range(B) if l in sel[i]])
    rows.append(list(range(B)))
    return rows


def routed_layer(model: Model, st: KVState, l: int, h: Dict[int, np.ndarray], executes: Sequence[int],
                 seqs: Sequence[int], pos: Dict[int, int]) -> Dict[tuple, tuple]:
    """Layer l for the sequences `seqs`: those in `executes` run the block on
    their hidden state h[i] (updated in place) at token position pos[i]; the
    others keep h[i] (identity).  Appends each sequence's entry to the layer's
    cache (zeros for skipped ones in the zero variant, nothing in the masked
    one) and returns the entries written."""
    sh = model.shape
    run = [i for i in seqs if i in set(executes)]
    out = {}
    if run:
        H, kn, vn = decoder_layer(sh, model.layer(l), np.stack([h[i] for i in run]),
                                  [st.get(l, i) for i in run], [pos[i] for i in run])
        for j, i in enumerate(run):
            h[i] = H[j]
            out[(l, i)] = (kn[j], vn[j])
    zeros = np.zeros((sh.n_kv_heads, sh.head_dim))
    for i in seqs:
        if (l, i) not in out and sh.skip_kv == "zero":
            out[(l, i)] = (zeros, zeros)
    for (ll, i), (kt, vt) in out.items():
        st.append(ll, i, kt, vt)
    return out


def decode_step(model: Model, st: KVState, h_in: np.ndarray, k: Sequence[int],
                override_sel: Optional[Callable[[RouteResult], List[List[int]]]] = None,
                seqs: Optional[Sequence[int]] = None) -> StepResult:
    """One budget-routed decode step for the batch; advances the state.
    `override_sel` lets a caller replace selected sets (the near-tie rule);
    `seqs` restricts the (independent) per-sequence work after the router to
    a subset; layers 0..c, the routing and the compaction cover the batch."""
    sh = model.shape
    L, c = sh.n_layers, sh.ctx_layer
    B = h_in.shape[0]
    rr = first_layers_and_route(model, st, h_in, k)
    if override_sel is not None:
        rr.sel = override_sel(rr)
    seqs = list(range(B)) if seqs is None else sorted(int(s) for s in seqs)
    for (l, i), (kt, vt) in rr.kv_new.items():
        st.append(l, i, kt, vt)
    rows = compaction(rr.sel, L, sh.first_candidate)
    mask = np.zeros((B, L), dtype=np.uint8)
    for l in range(L):
        mask[rows[l], l] = 1
    h = {i: rr.h[i].copy() for i in seqs}
    pos = {i: st.n[i] for i in seqs}
    kv_new = dict(rr.kv_new)
    for l in range(c + 1, L):
        kv_new.update(routed_layer(model, st, l, h, rows[l], seqs, pos))
        if st.loader is not None:
            st.drop(l)
    for i in range(B):
        st.n[i] += 1
    return StepResult(h, rr.scores, rr.k, rr.sel, mask, rows, kv_new)


def dense_decode_step(model: Model, st: KVState, h_in: np.ndarray) -> Dict[int, np.ndarray]:
    """The unrouted model: every layer on every sequence (Eq. 1 with M = 1).
    Does not modify the state."""
    sh = model.shape
    B = h_in.shape[0]
    H = np.asarray(h_in, dtype=np.float64)
    for l in range(sh.n_layers):
        H, _, _ = decoder_layer(sh, model.layer(l), H, [st.get(l, i) for i in range(B)], st.n)
    return {i: H[i] for i in range(B)}


# ---------------------------------------------------------------------------
# Prefill with routing (Sec. 4.1; App. E "Prefill vs. Decode")
# ---------------------------------------------------------------------------
@dataclasses.dataclass
class PrefillResult:
    h_out: Dict[int, np.ndarray]   # sequence -> [T_i, d] final hidden states of its tokens
    scores: np.ndarray             # [B, n_cand]
    k: List[int]
    sel: List[List[int]]
    mask: np.ndarray               # [B, L]
    kv_new: Dict[tuple, tuple]     # (layer, seq) -> (K [T_i or 0, n_kv, hd], V) as stored


def prefill(model: Model, st: KVState, prompts: Sequence[np.ndarray], k: Sequence[int],
            override_sel: Optional[Callable[[RouteResult], List[List[int]]]] = None) -> PrefillResult:
    """Routed prefill of one prompt per sequence (prompts[i] [T_i, d], T_i >= 1,
    appended after the n_i cached positions).  Layers 0..c run on every token;
    each sequence is routed once from its pooled context-layer cache (prompt
    included) and its last token's hidden state after layer c; the selected
    blocks run on all of its tokens (grouping by mask); skipped blocks store
    zero K/V at every new position (zero variant) or nothing (masked).
    Advances n_i by T_i."""
    sh = model.shape
    L, c = sh.n_layers, sh.ctx_layer
    B = len(prompts)
    X = {i: np.asarray(prompts[i], dtype=np.float64).copy() for i in range(B)}
    T = {i: X[i].shape[0] for i in range(B)}
    kv_new: Dict[tuple, tuple] = {}

    def run_layer(l, i):
        W = model.layer(l)
        K, V = st.get(l, i)
        X[i], kn, vn = prefill_layer(sh, W, X[i], K, V, st.n[i])
        st.append(l, i, kn, vn)
        kv_new[(l, i)] = (kn, vn)

    for l in range(c + 1):
        for i in range(B):
            run_layer(l, i)
    scores = np.empty((B, sh.n_cand))
    ks, sel, xs = [], [], []
    for i in range(B):
        K, V = st.get(c, i)
        x = router_input(sh, K, V, X[i][-1])
        scores[i], kk, si = route(model, x, k[i])
        ks.append(kk)
        sel.append(si)
        xs.append(x)
    rr = RouteResult(np.stack([X[i][-1] for i in range(B)]), scores, ks, sel, {}, np.stack(xs))
    if override_sel is not None:
        sel = override_sel(rr)
    rows = compaction(sel, L, sh.first_candidate)
    mask = np.zeros((B, L), dtype=np.uint8)
    for l in range(L):
        mask[rows[l], l] = 1
    for l in range(c + 1, L):
        for i in range(B):
            if mask[i, l]:
                run_layer(l, i)
            elif sh.skip_kv == "zero":
                z = np.zeros((T[i], sh.n_kv_heads, sh.head_dim))
                st.append(l, i, z, z)
                kv_new[(l, i)] = (z, z)
    for i in range(B):
        st.n[i] += T[i]
    return PrefillResult(X, scores, ks, sel, mask, kv_new)
