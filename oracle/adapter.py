"""Builds oracle inputs from the shared seeded generator (test infrastructure).

Converts generator tensors (bf16 / fp32 torch tensors, on any device) to the
float64 numpy arrays the oracle consumes.  The conversion is exact: bf16 and
fp32 values are representable in float64.  Nothing here computes the method.
"""
from __future__ import annotations

import functools
from typing import Dict, Optional, Sequence

import numpy as np
import torch

from workloads import synth
from workloads.configs import ModelShape, Workload

from . import buddy_oracle as O


def to_f64(t: torch.Tensor) -> np.ndarray:
    """Exact float64 copy of a bf16 / fp32 tensor (converted where it lives)."""
    if t.is_cuda:
        return t.detach().to(torch.float64).cpu().numpy()
    t = t.detach().contiguous()
    if t.dtype == torch.bfloat16:
        return O.bf16_bits_to_f64(t.view(torch.int16).numpy().view(np.uint16))
    if t.dtype == torch.float32:
        return t.numpy().astype(np.float64)
    raise TypeError(t.dtype)


def oracle_shape(s: ModelShape) -> O.Shape:
    return O.Shape(s.n_layers, s.d_model, s.n_q_heads, s.n_kv_heads, s.head_dim, s.ffn_dim,
                   s.dm_hidden, s.dtype, s.rms_eps, s.rope_theta, feature=s.feature,
                   ctx_layer=s.ctx_layer, skip_kv=s.skip_kv)


def layer_from_tensors(w: Dict[str, torch.Tensor]) -> O.LayerWeights:
    f = lambda name: to_f64(w[name]) if name in w and w[name] is not None else None
    return O.LayerWeights(attn_norm=f("attn_norm"), w_q=f("w_q"), w_k=f("w_k"), w_v=f("w_v"),
                          w_o=f("w_o"), ffn_norm=f("ffn_norm"), w_gate=f("w_gate"),
                          w_up=f("w_up"), w_down=f("w_down"), b_q=f("b_q"), b_k=f("b_k"),
                          b_v=f("b_v"))


def build_model(shape: ModelShape, seed: int, *, layer_source=None, dm_source=None,
                prior: Optional[torch.Tensor] = None, omega: float = 0.0,
                cache_layers: int = 4, predictor_source=None) -> O.Model:
    """Oracle model for a generated workload.  `layer_source(l)` may supply the
    generator's tensors (e.g. already generated on the GPU and copied back);
    by default they are generated on the host."""
    src = layer_source or (lambda l: synth.layer_weights(shape, seed, l, "cpu"))

    @functools.lru_cache(maxsize=cache_layers)
    def layer(l: int) -> O.LayerWeights:
        return layer_from_tensors(src(l))

    dmw = dm_source() if dm_source is not None else synth.dm_weights(shape, seed, "cpu")
    dm = O.DecisionModule(w1=to_f64(dmw["w1"]), b1=to_f64(dmw["b1"]), w2=to_f64(dmw["w2"]),
                          b2=to_f64(dmw["b2"]),
                          prior=None if prior is None else to_f64(prior), omega=float(omega))
    bp = None
    if shape.predictor_hidden > 0:
        pw = predictor_source() if predictor_source is not None else synth.predictor_weights(shape, seed, "cpu")
        bp = O.BudgetPredictor(w1=to_f64(pw["w1"]), b1=to_f64(pw["b1"]), w2=to_f64(pw["w2"]),
                               b2=to_f64(pw["b2"]))
    return O.Model(oracle_shape(shape), layer, dm, bp)


def build_state(shape: ModelShape, seed: int, n_ctx: Sequence[int],
                layers: Optional[Sequence[int]] = None,
                seqs: Optional[Sequence[int]] = None, gen_device: str = "cpu") -> O.KVState:
    """Prefilled caches (positions 0..n_i-1) for the given layers and sequences.
    `gen_device` only chooses where the generator runs (values are identical)."""
    st = O.KVState(n_ctx)
    layers = range(shape.n_layers) if layers is None else layers
    seqs = range(len(n_ctx)) if seqs is None else seqs
    for l in layers:
        for i in seqs:
            n = int(n_ctx[i])
            K = to_f64(synth.kv_block(shape, seed, "k", l, i, 0, n, gen_device))
            V = to_f64(synth.kv_block(shape, seed, "v", l, i, 0, n, gen_device))
            st.set(l, i, K, V)
    return st


def lazy_state(shape: ModelShape, seed: int, n_ctx: Sequence[int], gen_device: str = "cpu") -> O.KVState:
    """KV state whose caches are generated on first use, one (layer, sequence)
    at a time, and dropped by the oracle after each layer."""
    def load(l, i):
        n = int(n_ctx[i])
        K = to_f64(synth.kv_block(shape, seed, "k", l, i, 0, n, gen_device))
        V = to_f64(synth.kv_block(shape, seed, "v", l, i, 0, n, gen_device))
        return K, V
    return O.KVState(n_ctx, loader=load)


def workload_inputs(w: Workload, step: int) -> np.ndarray:
    return to_f64(synth.workload_h_in(w, step))
