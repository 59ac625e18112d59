"""Seeded synthetic inputs shared byte-for-byte by the GPU path and the oracle.

Every value is a pure function of (seed, tensor kind, ids, flat index), so any
slice of any tensor can be regenerated on any device: the oracle can draw the KV
cache of one sequence without materialising the whole batch, and the GPU side
can fill 100 GB of cache without a host round trip.

Generator (integer-exact, hence identical on CPU and CUDA):
  * word(c) = H(H((c + a) mod 2^32) XOR b), H = the public-domain "lowbias32"
    integer finaliser (xor-shift / multiply rounds), (a, b) a per-stream key;
  * two words per element give four 16-bit uniforms u1..u4; their sum S follows
    the Irwin-Hall(4) law (mean 131070, std 37837.23), a close, bounded
    (|z| <= 3.46) approximation of a normal draw;
  * value = fp32(S - 131070) * fp32(sigma / 37837.23) (one correctly rounded
    fp32 multiply), then round-to-nearest-even to bf16 for bf16 tensors.

No part of the routed decode computation lives here.
"""
from __future__ import annotations

import math
from typing import Dict, Sequence

import torch

from .configs import ModelShape, Workload

_M32 = 0xFFFFFFFF
_IH_MEAN = 4 * 65535 // 2            # 131070
_IH_STD = math.sqrt(4 * (65536.0 ** 2 - 1.0) / 12.0)
_CHUNK_CPU = 1 << 18     # cache-sized chunks on the host
_CHUNK_GPU = 1 << 25

KIND = {"w_q": 1, "w_k": 2, "w_v": 3, "w_o": 4, "w_gate": 5, "w_up": 6, "w_down": 7,
        "b_q": 8, "b_k": 9, "b_v": 10, "attn_norm": 11, "ffn_norm": 12,
        "dm_w1": 20, "dm_b1": 21, "dm_w2": 22, "dm_b2": 23, "prior": 24,
        "bp_w1": 25, "bp_b1": 26, "bp_w2": 27, "bp_b2": 28,
        "k_cache": 30, "v_cache": 31, "h_in": 40}

WEIGHT_STD = 0.02
NORM_GAIN_STD = 0.1


def _h32_int(x: int) -> int:
    x &= _M32
    x ^= x >> 16
    x = (x * 0x7FEB352D) & _M32
    x ^= x >> 15
    x = (x * 0x846CA68B) & _M32
    x ^= x >> 16
    return x


def stream_key(seed: int, kind: str, *ids: int):
    """Per-stream key pair (a, b) from the seed, the tensor kind and integer ids."""
    h = _h32_int(0x9E3779B9 ^ (seed & _M32))
    for v in (KIND[kind],) + tuple(int(i) for i in ids):
        h = _h32_int(h ^ (v & _M32))
        h = _h32_int((h + 0x632BE5AB) & _M32)
    a = h
    b = _h32_int(h ^ 0x5BD1E995)
    return a, b


def _mul32(x: torch.Tensor, c: int) -> torch.Tensor:
    # (x * c) mod 2^32 on int64 without overflow: split c into 16-bit halves.
    lo, hi = c & 0xFFFF, c >> 16
    return (x * lo + (((x * hi) & 0xFFFF) << 16)) & _M32


def _h32(x: torch.Tensor) -> torch.Tensor:
    x = x ^ (x >> 16)
    x = _mul32(x, 0x7FEB352D)
    x = x ^ (x >> 15)
    x = _mul32(x, 0x846CA68B)
    x = x ^ (x >> 16)
    return x


def _word(c: torch.Tensor, key) -> torch.Tensor:
    a, b = key
    return _h32(_h32((c + a) & _M32) ^ b)


def fill_normal_(out: torch.Tensor, key, sigma: float, mean: float = 0.0, start: int = 0):
    """Fill contiguous `out` (float32 or bfloat16) with the stream's elements
    start .. start+numel-1 in flat (row-major) order."""
    assert out.is_contiguous()
    flat = out.view(-1)
    n = flat.numel()
    dev = out.device
    scale = torch.tensor(sigma / _IH_STD, dtype=torch.float32, device=dev)
    shift = torch.tensor(mean, dtype=torch.float32, device=dev)
    chunk = _CHUNK_GPU if dev.type == "cuda" else _CHUNK_CPU
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        c = torch.arange(start + s, start + e, dtype=torch.int64, device=dev) * 2
        w0 = _word(c, key)
        w1 = _word(c + 1, key)
        S = (w0 & 0xFFFF) + (w0 >> 16) + (w1 & 0xFFFF) + (w1 >> 16)
        v = (S - _IH_MEAN).to(torch.float32) * scale
        if mean != 0.0:
            v = v + shift
        flat[s:e].copy_(v.to(out.dtype))
    return out


def normal(shape, key, sigma: float, dtype, device, mean: float = 0.0, start: int = 0):
    t = torch.empty(tuple(shape), dtype=dtype, device=device)
    return fill_normal_(t, key, sigma, mean=mean, start=start)


def storage_dtype(shape: ModelShape):
    return torch.float32 if shape.dtype == "f32" else torch.bfloat16


# --------------------------------------------------------------------------
# Workload tensors
# --------------------------------------------------------------------------
def layer_weights(shape: ModelShape, seed: int, layer: int, device="cpu") -> Dict[str, torch.Tensor]:
    """Decoder-layer weights in nn.Linear layout [out, in] (storage dtype);
    norm gains and biases are fp32."""
    dt = storage_dtype(shape)
    d, F, qd, kvd = shape.d_model, shape.ffn_dim, shape.q_dim, shape.kv_dim
    g = lambda kind, shp, dtype=dt, sigma=WEIGHT_STD, mean=0.0: normal(
        shp, stream_key(seed, kind, layer), sigma, dtype, device, mean=mean)
    w = {
        "w_q": g("w_q", (qd, d)), "w_k": g("w_k", (kvd, d)), "w_v": g("w_v", (kvd, d)),
        "w_o": g("w_o", (d, qd)),
        "w_gate": g("w_gate", (F, d)), "w_up": g("w_up", (F, d)), "w_down": g("w_down", (d, F)),
    }
    if shape.random_norm:
        w["attn_norm"] = g("attn_norm", (d,), torch.float32, NORM_GAIN_STD, 1.0)
        w["ffn_norm"] = g("ffn_norm", (d,), torch.float32, NORM_GAIN_STD, 1.0)
    else:
        w["attn_norm"] = torch.ones(d, dtype=torch.float32, device=device)
        w["ffn_norm"] = torch.ones(d, dtype=torch.float32, device=device)
    if shape.qkv_bias:
        w["b_q"] = g("b_q", (qd,), torch.float32)
        w["b_k"] = g("b_k", (kvd,), torch.float32)
        w["b_v"] = g("b_v", (kvd,), torch.float32)
    return w


def dm_weights(shape: ModelShape, seed: int, device="cpu") -> Dict[str, torch.Tensor]:
    """Decision Module (Linear 2d->r, SiLU, Linear r->n_cand), fp32."""
    d, r, Lm = shape.d_model, shape.dm_hidden, shape.n_cand
    g = lambda kind, shp: normal(shp, stream_key(seed, kind), WEIGHT_STD, torch.float32, device)
    return {"w1": g("dm_w1", (r, 2 * d)), "b1": g("dm_b1", (r,)),
            "w2": g("dm_w2", (Lm, r)), "b2": g("dm_b2", (Lm,))}


def predictor_weights(shape: ModelShape, seed: int, device="cpu") -> Dict[str, torch.Tensor]:
    """Budget Predictor (Linear 2d->r_p, SiLU, Linear r_p->n_cand), fp32.  Its
    second layer is drawn wider (sigma 0.5) so that the argmax varies across
    inputs instead of being fixed by the bias."""
    d, r, Lm = shape.d_model, shape.predictor_hidden, shape.n_cand
    g = lambda kind, shp, sd=WEIGHT_STD: normal(shp, stream_key(seed, kind), sd, torch.float32, device)
    return {"w1": g("bp_w1", (r, 2 * d)), "b1": g("bp_b1", (r,)),
            "w2": g("bp_w2", (Lm, r), 0.5), "b2": g("bp_b2", (Lm,))}


def prior(shape: ModelShape, seed: int, device="cpu") -> torch.Tensor:
    """An arbitrary normalised prior vector p~ over the routed layers (fp32)."""
    return normal((shape.n_cand,), stream_key(seed, "prior"), 1.0, torch.float32, device)


def kv_block(shape: ModelShape, seed: int, which: str, layer: int, seq: int,
             pos0: int, n_pos: int, device="cpu") -> torch.Tensor:
    """Prefilled cache entries of one sequence: positions pos0..pos0+n_pos-1,
    layout [n_pos, n_kv, hd] (storage dtype), values N(0,1)."""
    assert which in ("k", "v")
    key = stream_key(seed, "k_cache" if which == "k" else "v_cache", layer, seq)
    kvd = shape.kv_dim
    return normal((n_pos, shape.n_kv_heads, shape.head_dim), key, 1.0, storage_dtype(shape),
                  device, start=pos0 * kvd)


def h_in(shape: ModelShape, seed: int, step: int, seqs: Sequence[int], device="cpu") -> torch.Tensor:
    """Step input hidden states [len(seqs), d] fp32, N(0,1), one stream per (step, seq)."""
    out = torch.empty(len(seqs), shape.d_model, dtype=torch.float32, device=device)
    for r, s in enumerate(seqs):
        fill_normal_(out[r], stream_key(seed, "h_in", step, int(s)), 1.0)
    return out


def prompt_inputs(shape: ModelShape, seed: int, lengths: Sequence[int], device="cpu") -> torch.Tensor:
    """Input hidden states of one prompt per sequence, [sum(lengths), d] fp32
    N(0,1), sequence by sequence; one stream per (sequence, token)."""
    out = torch.empty(int(sum(lengths)), shape.d_model, dtype=torch.float32, device=device)
    r = 0
    for i, n in enumerate(lengths):
        for t in range(int(n)):
            fill_normal_(out[r], stream_key(seed, "h_in", 1 << 20 | i, t), 1.0)
            r += 1
    return out


def workload_h_in(w: Workload, step: int, device="cpu") -> torch.Tensor:
    return h_in(w.shape, w.seed, step, range(w.batch), device)
