"""CPU oracle for BUDDY's budget-routed decode step.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute this module; only tests/, __graft_entry__.smoke() and bench.py's
cpu_baseline / reference legs use it.  It shares no code with the CUDA path.

What it computes (plain numpy, float64 arithmetic, one sequence at a time):

  * Layer skipping (Sec. 3.1, Eq. 1): an executed block adds F_l(H) to the
    residual, a skipped block is the identity.
  * First and last blocks always execute; the L_mid = L - 2 middle blocks are
    the candidates (Sec. 4.2.1).
  * KV-aware planner (Sec. 4.3): the first layer's V cache, with the newest
    token's V appended, is mean-pooled over positions; value states are the
    default feature (Sec. 5 "Hyper-parameters").  The pooled vector is expanded
    to width d by repeating each KV head over its query-head group and
    concatenated with the newest token's hidden state after layer 0.
  * Decision Module (Sec. 4.2.3, App. C.1): Linear -> SiLU -> Linear gives one
    score per middle layer; a prior p~ is fused as s' = s + omega * p~ (Eq. 2).
  * Deterministic top-k (Eq. 2): the k middle layers with the largest s'
    execute; equal scores are broken by the lower layer index.  Softmax is
    monotone, so ranking s' gives the same set.
  * Grouping by mask (App. C.1): block l runs on the sequences that selected it.
  * Skipped layers store zero K and V at the new position (Sec. 6,
    "Limitations"), so every layer's cache grows by one position per step.
  * Decoder block and KV cache (App. "Background", Eq. 9): Llama-style block —
    RMSNorm, Q/K/V projections (optional bias), rotate-half RoPE, grouped-query
    attention over [K_cache; K_t], [V_cache; V_t], output projection, RMSNorm,
    SwiGLU MLP d -> F -> d.

Precision.  The paper runs its model in bfloat16 (Sec. 5 "Hyper-parameters").
For "bf16" shapes the oracle rounds exactly where a bf16 model stores a
tensor: the K/V written to the cache and, in every layer but the first, the
normalised GEMM inputs, the attention output and the SwiGLU product
(round-to-nearest-even through fp32).  The first layer, whose output is the
router's input, keeps its activations unrounded: rounding there makes the
layer output jump by ~1e-3 when an input moves by ~1e-7 (a flipped bf16
rounding of one element changes every SwiGLU product it feeds), and the
routing decision would then not be a function of the mathematics.
Everything else — projections, attention scores and softmax, residual
stream, Decision Module — is float64.  "f32" shapes round nothing.

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


def round_to_f32(x: np.ndarray) -> np.ndarray:
    return np.asarray(x, dtype=np.float64).astype(np.float32).astype(np.float64)


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
    dtype: str            # "f32" | "bf16"
    rms_eps: float
    rope_theta: float

    @property
    def l_mid(self):
        return self.n_layers - 2

    @property
    def group(self):
        return self.n_q_heads // self.n_kv_heads

    def store(self, x: np.ndarray) -> np.ndarray:
        """Value of a tensor as the model stores it (see module docstring)."""
        return round_to_bf16(x) if self.dtype == "bf16" else x


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
    w2: np.ndarray        # [L_mid, r]
    b2: np.ndarray        # [L_mid]
    prior: Optional[np.ndarray] = None   # p~ [L_mid]
    omega: float = 0.0


@dataclasses.dataclass
class Model:
    shape: Shape
    layer: Callable[[int], LayerWeights]   # float64 weights of layer l, 0-based
    dm: DecisionModule


class KVState:
    """Per-(layer, sequence) caches.  kv[(l, i)] = (K, V), each [n, n_kv, hd]
    float64 holding the stored values of positions 0..n-1.  An optional
    `loader(l, i)` supplies caches on first use (and `drop` forgets them), so
    that large workloads can be evaluated one layer at a time."""

    def __init__(self, n_ctx: Sequence[int], loader: Optional[Callable[[int, int], tuple]] = None):
        self.n = [int(v) for v in n_ctx]          # n_i: cached positions per sequence
        self.kv: Dict[tuple, tuple] = {}
        self.loader = loader

    def set(self, layer: int, seq: int, K: np.ndarray, V: np.ndarray):
        assert K.shape[0] == self.n[seq] and V.shape == K.shape
        self.kv[(layer, seq)] = (np.asarray(K, np.float64), np.asarray(V, np.float64))

    def get(self, layer: int, seq: int):
        if (layer, seq) not in self.kv and self.loader is not None:
            K, V = self.loader(layer, seq)
            self.set(layer, seq, K, V)
        return self.kv[(layer, seq)]

    def drop(self, layer: int):
        for key in [k for k in self.kv if k[0] == layer]:
            del self.kv[key]

    def has(self, layer: int, seq: int) -> bool:
        return (layer, seq) in self.kv or self.loader is not None


# ---------------------------------------------------------------------------
# Building blocks of the Llama-style layer (App. "Background"; Sec. 5 models)
# ---------------------------------------------------------------------------
def rms_norm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm: x / sqrt(mean(x^2) + eps) * gain, over the last axis."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * gain


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


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
    e = np.exp(z - np.max(z))
    return e / np.sum(e)


def decode_attention(q: np.ndarray, K: np.ndarray, V: np.ndarray, group: int) -> np.ndarray:
    """Attn(Q_t, [K_cache; K_t], [V_cache; V_t]) for one token (Eq. 9).
    q [n_q, hd]; K, V [n+1, n_kv, hd]; query head h reads KV head h // group."""
    n_q, hd = q.shape
    out = np.empty_like(q)
    for h in range(n_q):
        g = h // group
        logits = K[:, g, :] @ q[h] / np.sqrt(hd)
        out[h] = softmax(logits) @ V[:, g, :]
    return out


def decoder_layer(sh: Shape, W: LayerWeights, h: np.ndarray, K_cache: np.ndarray,
                  V_cache: np.ndarray, pos: int, round_act: bool = True):
    """One executed block for one token at position `pos` = number of cached
    positions.  Returns (h + F_l(h), K_t, V_t) with K_t, V_t [n_kv, hd] as stored.
    round_act=False keeps the GEMM inputs unrounded (the first layer)."""
    hd = sh.head_dim
    act = sh.store if round_act else (lambda x: x)
    xn = act(rms_norm(h, W.attn_norm, sh.rms_eps))
    q = W.w_q @ xn
    k = W.w_k @ xn
    v = W.w_v @ xn
    if W.b_q is not None:
        q, k, v = q + W.b_q, k + W.b_k, v + W.b_v
    q = rope(q.reshape(sh.n_q_heads, hd), pos, sh.rope_theta)
    k = rope(k.reshape(sh.n_kv_heads, hd), pos, sh.rope_theta)
    k_t = sh.store(k)
    v_t = sh.store(v.reshape(sh.n_kv_heads, hd))
    K = np.concatenate([K_cache, k_t[None]], axis=0)
    V = np.concatenate([V_cache, v_t[None]], axis=0)
    attn = act(decode_attention(q, K, V, sh.group).reshape(-1))
    h = h + W.w_o @ attn
    xn2 = act(rms_norm(h, W.ffn_norm, sh.rms_eps))
    a = act(silu(W.w_gate @ xn2) * (W.w_up @ xn2))
    h = h + W.w_down @ a
    return h, k_t, v_t


# ---------------------------------------------------------------------------
# Router: KV-aware planner + Decision Module + top-k (Sec. 4.2, 4.3)
# ---------------------------------------------------------------------------
def pool_context(V0: np.ndarray) -> np.ndarray:
    """G_t from the first layer's value cache including the newest token:
    arithmetic mean over positions of V0 [n+1, n_kv, hd] -> [n_kv * hd]."""
    return np.mean(V0, axis=0).reshape(-1)


def expand_kv_heads(g: np.ndarray, sh: Shape) -> np.ndarray:
    """Repeat each KV head over its query-head group: width n_kv*hd -> d
    (query head h uses KV head h // group)."""
    g = g.reshape(sh.n_kv_heads, sh.head_dim)
    return np.repeat(g, sh.group, axis=0).reshape(-1)


def decision_scores(dm: DecisionModule, x: np.ndarray) -> np.ndarray:
    """s' = W2 SiLU(W1 x + b1) + b2 + omega * p~  (App. C.1; Eq. 2)."""
    s = dm.w2 @ silu(dm.w1 @ x + dm.b1) + dm.b2
    if dm.prior is not None:
        s = s + dm.omega * dm.prior
    return s


def top_k_layers(scores: np.ndarray, k: int) -> List[int]:
    """Middle layers (1-based block ids 1..L_mid, i.e. 0-based layers 1..L-2)
    with the k largest scores; ties go to the lower index.  Returned ascending."""
    order = sorted(range(len(scores)), key=lambda j: (-scores[j], j))
    return sorted(j + 1 for j in order[:k])


def budget_to_k(b: float, L: int) -> int:
    """k = round(b * L) - 2 (Eq. 2), clamped to the action space {1..L_mid}
    (Sec. 4.4).  Python's round() ties to even."""
    return int(min(max(round(b * L) - 2, 1), L - 2))


def k_to_budget(k: int, L: int) -> float:
    """b = (k + 2) / L (Eq. 3): the +2 counts the first and last blocks."""
    return (k + 2) / L


# ---------------------------------------------------------------------------
# The decode step
# ---------------------------------------------------------------------------
@dataclasses.dataclass
class RouteResult:
    h1: np.ndarray                 # [B, d] hidden state after layer 0
    scores: np.ndarray             # [B, L_mid] s'
    sel: List[List[int]]           # per sequence, ascending executed middle layers
    kv0_new: List[tuple]           # per sequence (K_t, V_t) written to layer 0


@dataclasses.dataclass
class StepResult:
    h_out: Dict[int, np.ndarray]   # sequence -> final hidden state [d]
    scores: np.ndarray
    sel: List[List[int]]
    mask: np.ndarray               # [B, L] uint8
    rows: List[List[int]]          # per layer: ascending active sequences
    kv_new: Dict[tuple, tuple]     # (layer, seq) -> (K_t, V_t) as stored (zeros if skipped)


def first_layer_and_route(model: Model, st: KVState, h_in: np.ndarray, k: Sequence[int]) -> RouteResult:
    """Layer 0 on every sequence, then the router on every sequence."""
    sh = model.shape
    B = h_in.shape[0]
    W0 = model.layer(0)
    h1 = np.empty_like(h_in, dtype=np.float64)
    kv0 = []
    for i in range(B):
        K, V = st.get(0, i)
        h1[i], k_t, v_t = decoder_layer(sh, W0, h_in[i].astype(np.float64), K, V, st.n[i], round_act=False)
        kv0.append((k_t, v_t))
    scores = np.empty((B, sh.l_mid))
    sel = []
    for i in range(B):
        V0 = np.concatenate([st.get(0, i)[1], kv0[i][1][None]], axis=0)
        x = np.concatenate([expand_kv_heads(pool_context(V0), sh), h1[i]])
        scores[i] = decision_scores(model.dm, x)
        if not (1 <= int(k[i]) <= sh.l_mid):
            raise ValueError(f"budget k={k[i]} outside [1, {sh.l_mid}]")
        sel.append(top_k_layers(scores[i], int(k[i])))
    return RouteResult(h1, scores, sel, kv0)


def compaction(sel: Sequence[Sequence[int]], L: int) -> List[List[int]]:
    """Grouping by mask: for every layer, the ascending list of sequences that
    execute it (all sequences for the first and last layers)."""
    B = len(sel)
    rows = [list(range(B))]
    for l in range(1, L - 1):
        rows.append([i for i in range(B) if l in sel[i]])
    rows.append(list(range(B)))
    return rows


def routed_layers(model: Model, st: KVState, route: RouteResult,
                  seqs: Optional[Sequence[int]] = None) -> StepResult:
    """Middle and last layers on the routed subsets, then the step advance.
    `seqs` restricts the (independent) per-sequence work to a subset; the
    routing and compaction still cover the whole batch."""
    sh = model.shape
    B = route.h1.shape[0]
    L = sh.n_layers
    seqs = list(range(B)) if seqs is None else sorted(int(s) for s in seqs)
    rows = compaction(route.sel, L)
    mask = np.zeros((B, L), dtype=np.uint8)
    for l in range(L):
        mask[rows[l], l] = 1
    kv_new = {(0, i): route.kv0_new[i] for i in range(B)}
    h = {i: route.h1[i].copy() for i in seqs}
    zeros = np.zeros((sh.n_kv_heads, sh.head_dim))
    for l in range(1, L):
        W = None
        for i in seqs:
            if mask[i, l]:
                if W is None:
                    W = model.layer(l)
                K, V = st.get(l, i)
                h[i], k_t, v_t = decoder_layer(sh, W, h[i], K, V, st.n[i])
                kv_new[(l, i)] = (k_t, v_t)
            else:
                kv_new[(l, i)] = (zeros.copy(), zeros.copy())
        if st.loader is not None:
            st.drop(l)
    return StepResult(h, route.scores, route.sel, mask, rows, kv_new)


def advance(st: KVState, res: StepResult, seqs: Optional[Sequence[int]] = None):
    """Append the step's K_t, V_t (real or zero) to every cache and n_i += 1."""
    B = len(st.n)
    seqs = list(range(B)) if seqs is None else seqs
    for (l, i), (k_t, v_t) in res.kv_new.items():
        if st.has(l, i):
            K, V = st.get(l, i)
            st.kv[(l, i)] = (np.concatenate([K, k_t[None]]), np.concatenate([V, v_t[None]]))
    for i in range(B):
        st.n[i] += 1


def decode_step(model: Model, st: KVState, h_in: np.ndarray, k: Sequence[int],
                override_sel: Optional[Callable[[RouteResult], List[List[int]]]] = None,
                seqs: Optional[Sequence[int]] = None) -> StepResult:
    """One budget-routed decode step for the batch; advances the state.
    `override_sel` lets a caller replace selected sets (the near-tie rule)."""
    route = first_layer_and_route(model, st, h_in, k)
    if override_sel is not None:
        route.sel = override_sel(route)
    res = routed_layers(model, st, route, seqs)
    advance(st, res, seqs)
    return res


def dense_decode_step(model: Model, st: KVState, h_in: np.ndarray) -> Dict[int, np.ndarray]:
    """The unrouted model: every layer on every sequence (Eq. 1 with M = 1).
    Does not modify the state."""
    sh = model.shape
    out = {}
    for i in range(h_in.shape[0]):
        h = h_in[i].astype(np.float64)
        for l in range(sh.n_layers):
            K, V = st.get(l, i)
            h, _, _ = decoder_layer(sh, model.layer(l), h, K, V, st.n[i], round_act=(l != 0))
        out[i] = h
    return out
