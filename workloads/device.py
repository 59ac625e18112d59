"""Materialises a workload on the GPU through libbuddy's public API.

Weights, Decision Module, prefilled KV caches (written with buddy_kv_append)
and per-step inputs all come from the seeded generator in `synth`; nothing
here computes any part of the routed decode step.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional

import numpy as np
import torch

from . import synth
from .configs import Workload


@dataclasses.dataclass
class DeviceWorkload:
    w: Workload
    ctx: object            # paper_2606_09514_gb300.Context
    kv: object             # paper_2606_09514_gb300.KVCache
    layers: List[dict]     # packed device weights
    dm: dict
    k: torch.Tensor        # [B] int32 budgets (device)
    contexts: np.ndarray
    caps: np.ndarray
    prior: Optional[torch.Tensor] = None


def build(w: Workload, device="cuda", extra_steps: int = 8, max_batch: Optional[int] = None,
          prior: bool = False, omega: float = 0.1, use_graph: bool = False,
          gen_device: Optional[str] = None, max_prefill_tokens: int = 0) -> DeviceWorkload:
    """gen_device: where the generator runs ("cpu": every tensor is drawn on
    the host and copied to `device` once; default: on `device`)."""
    import paper_2606_09514_gb300 as pkg

    s = w.shape
    dt = synth.storage_dtype(s)
    gd = gen_device or device
    mv = lambda t: t.to(device)
    ctxs = w.contexts()
    caps = ctxs + w.steps + extra_steps + 1
    ctx = pkg.Context.for_shape(s, max_batch=max_batch or w.batch, max_pos=int(caps.max()),
                                max_prefill_tokens=max_prefill_tokens)
    layers = [pkg.pack_layer({k: mv(v) for k, v in synth.layer_weights(s, w.seed, l, gd).items()})
              for l in range(s.n_layers)]
    dm = {k: mv(v) for k, v in synth.dm_weights(s, w.seed, gd).items()}
    pr = mv(synth.prior(s, w.seed, gd)) if prior else None
    ctx.buddy_set_weights(layers, dm, prior=pr, omega=omega if prior else 0.0)
    if s.predictor_hidden > 0:
        ctx.buddy_set_budget_predictor({k: mv(v) for k, v in synth.predictor_weights(s, w.seed, gd).items()})
    ctx.buddy_set_options(use_graph)
    kv = pkg.KVCache(s.n_layers, s.n_kv_heads, s.head_dim, caps.tolist(), dt, device, masked=s.skip_kv == "masked")
    prefill(ctx, kv, w, ctxs, device, gd)
    k = torch.tensor(w.budgets(), dtype=torch.int32, device=device)
    return DeviceWorkload(w, ctx, kv, layers, dm, k, ctxs, caps, pr)


def prefill(ctx, kv, w: Workload, ctxs, device="cuda", gen_device: Optional[str] = None):
    """Writes positions 0..n_i-1 of every layer with buddy_kv_append, one call
    per (layer, sequence); the last layer's call advances len_i."""
    s = w.shape
    gd = gen_device or device
    for i in range(w.batch):
        n = int(ctxs[i])
        ids = torch.tensor([i], dtype=torch.int32, device=device)
        for l in range(s.n_layers):
            if n > 0:
                K = synth.kv_block(s, w.seed, "k", l, i, 0, n, gd).unsqueeze(0).to(device)
                V = synth.kv_block(s, w.seed, "v", l, i, 0, n, gd).unsqueeze(0).to(device)
            else:
                K = V = torch.empty(1, 0, s.n_kv_heads, s.head_dim, dtype=synth.storage_dtype(s),
                                    device=device)
            ctx.buddy_kv_append(kv, l, ids, K, V, advance=(l == s.n_layers - 1))
