"""Cost accounting for the budget-routed decode step (harness arithmetic).

Two things live here:

1. The paper's analytic overhead model (App. C.2 "Inference overhead"):
   F_DM = 2BTdr + 2BTr(L-I), F_layer = 8Td^2 + 4T^2 d + 4Td d_c,
   F_model(b) = b L F_layer, rho(b) = F_DM / F_model(b).

2. The algorithmic bytes and FLOPs of one realised decode step, used as the
   roofline numerator: the union of executed layers' weights, the KV actually
   read (every executed (sequence, layer) pair reads n_i + 1 positions of K
   and V), the KV written (one position per sequence and layer, real or zero),
   the Decision Module weights, the pooled running sums and the step's hidden
   states in and out.
"""
from __future__ import annotations

from fractions import Fraction
from typing import Sequence

import numpy as np

from .configs import ModelShape


# ---------------------------------------------------------------------------
# 1. Paper's overhead model (App. C.2)
# ---------------------------------------------------------------------------
def paper_f_dm(B: int, T: int, d: int, r: int, L: int, I: int) -> int:
    return 2 * B * T * d * r + 2 * B * T * r * (L - I)


def paper_f_layer(T: int, d: int, d_c: int) -> int:
    return 8 * T * d * d + 4 * T * T * d + 4 * T * d * d_c


def paper_f_model(b: Fraction, L: int, T: int, d: int, d_c: int) -> Fraction:
    return Fraction(b) * L * paper_f_layer(T, d, d_c)


def paper_rho(b: Fraction, B: int, T: int, d: int, d_c: int, r: int, L: int, I: int) -> float:
    return float(Fraction(paper_f_dm(B, T, d, r, L, I)) / paper_f_model(b, L, T, d, d_c))


# ---------------------------------------------------------------------------
# 2. Algorithmic cost of one realised step
# ---------------------------------------------------------------------------
def layer_weight_bytes(s: ModelShape) -> int:
    """Projection weights (storage dtype) plus fp32 norm gains and biases."""
    b = s.layer_params * s.elem_bytes + 2 * s.d_model * 4
    if s.qkv_bias:
        b += s.qkv_dim * 4
    return b


def dm_bytes(s: ModelShape) -> int:
    r, d, Lm = s.dm_hidden, s.d_model, s.l_mid
    return (r * 2 * d + r + Lm * r + 2 * Lm) * 4


def step_cost(s: ModelShape, mask: np.ndarray, n_ctx: Sequence[int]) -> dict:
    """mask [B, L] (1 = executed), n_ctx[i] = cached positions before the step."""
    mask = np.asarray(mask, dtype=bool)
    B, L = mask.shape
    n = np.asarray(n_ctx, dtype=np.int64)
    kv_row = s.kv_dim * s.elem_bytes                    # one position of K (or V)
    used = mask.any(axis=0)
    w_union = int(used.sum()) * layer_weight_bytes(s)
    kv_read = int(2 * kv_row * ((n + 1)[:, None] * mask).sum())
    kv_write = int(2 * kv_row * B * L)
    small = dm_bytes(s) + B * s.kv_dim * 4 * 2 + B * s.d_model * 4 * 2
    exec_pairs = int(mask.sum())
    attn_flops = int(4 * s.n_q_heads * s.head_dim * ((n + 1)[:, None] * mask).sum())
    flops = 2 * s.layer_params * exec_pairs + attn_flops \
        + 2 * B * (2 * s.d_model * s.dm_hidden + s.dm_hidden * s.l_mid)
    return {"bytes": w_union + kv_read + kv_write + small, "weight_bytes": w_union,
            "kv_read_bytes": kv_read, "kv_write_bytes": kv_write, "other_bytes": small,
            "flops": flops, "exec_pairs": exec_pairs, "layers_used": int(used.sum())}


def prefill_cost(s: ModelShape, mask: np.ndarray, lengths: Sequence[int], n0: Sequence[int]) -> dict:
    """Algorithmic FLOPs and bytes of one routed prefill: every executed
    (prompt, layer) pair runs its T_i tokens through the projections
    (2 * layer_params FLOPs per token) and causal attention (token t attends
    to n0_i + t + 1 positions: 4 * n_q * hd FLOPs per position); bytes are
    the union of executed layers' weights, the K/V written and read once,
    and the hidden states in and out."""
    mask = np.asarray(mask, dtype=bool)
    B, L = mask.shape
    T = np.asarray(lengths, dtype=np.int64)
    n0 = np.asarray(n0, dtype=np.int64)
    pairs_tok = int((T[:, None] * mask).sum())
    # sum over tokens t of (n0 + t + 1) = T n0 + T (T + 1) / 2
    att_pos = (T * n0 + T * (T + 1) // 2)[:, None] * mask
    flops = 2 * s.layer_params * pairs_tok + int(4 * s.n_q_heads * s.head_dim * att_pos.sum())
    kv_row = s.kv_dim * s.elem_bytes
    w_union = int(mask.any(axis=0).sum()) * layer_weight_bytes(s)
    kv = int(2 * kv_row * ((T + n0)[:, None] * mask).sum())
    hid = int(T.sum()) * s.d_model * 4 * 2
    return {"flops": flops, "bytes": w_union + kv + hid, "tokens": int(T.sum()), "gemm_flops":
            2 * s.layer_params * pairs_tok}


def roofline_seconds(cost: dict, hbm_gbs: float, tflops: float) -> float:
    return max(cost["bytes"] / (hbm_gbs * 1e9), cost["flops"] / (tflops * 1e12))
