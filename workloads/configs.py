"""Model shapes and decode workloads for the budget-routed decode step.

A workload is a model shape (layers, widths, heads, Decision Module width) plus a
batch description (contexts n_i, per-sequence budgets k_i, number of decode
steps).  Nothing here computes any part of the method: these are plain records
and a seeded draw of the per-sequence metadata (contexts and budgets).

Shapes follow the public model families the paper evaluates (Sec. 5 "Settings":
Llama3-8B, Llama2-7B/13B-class, Qwen2.5-7B); the Decision Module is the
two-layer MLP of App. C.1 with hidden width r.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional

import numpy as np


@dataclasses.dataclass(frozen=True)
class ModelShape:
    name: str
    n_layers: int          # L (first and last always execute, Sec. 4.2.1)
    d_model: int           # d
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn_dim: int           # F (SwiGLU intermediate width)
    dm_hidden: int         # r (Decision Module hidden width, App. C.1)
    dtype: str             # "f32" or "bf16": storage type of weights, KV and GEMM inputs
    rms_eps: float
    rope_theta: float
    qkv_bias: bool = False
    random_norm: bool = False   # test shapes draw RMSNorm gains instead of using 1
    # router variants (Sec. 4.3, Sec. 5.4 ablations, Sec. 6)
    feature: str = "v"          # planner feature: "v", "k" or "kv" (K + V)
    ctx_layer: int = 0          # c: layers 0..c always run, the planner reads layer c
    skip_kv: str = "zero"       # "zero" (zero-filled K/V at skipped layers) or "masked"
    predictor_hidden: int = 0   # Budget Predictor hidden width (0: no predictor)

    @property
    def l_mid(self) -> int:
        return self.n_layers - 2

    @property
    def n_cand(self) -> int:
        """Routed candidate layers c+1 .. L-2."""
        return self.n_layers - 2 - self.ctx_layer

    @property
    def first_candidate(self) -> int:
        return self.ctx_layer + 1

    @property
    def kv_dim(self) -> int:
        return self.n_kv_heads * self.head_dim

    @property
    def q_dim(self) -> int:
        return self.n_q_heads * self.head_dim

    @property
    def qkv_dim(self) -> int:
        return (self.n_q_heads + 2 * self.n_kv_heads) * self.head_dim

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    @property
    def layer_params(self) -> int:
        """Backbone parameters of one decoder layer (projections only)."""
        d, F = self.d_model, self.ffn_dim
        return d * self.qkv_dim + self.q_dim * d + 2 * F * d + F * d


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    shape: ModelShape
    batch: int
    steps: int
    seed: int
    # context-length recipe
    ctx_kind: str                 # "fixed" | "uniform" | "lognormal" | "list"
    ctx_args: tuple
    # budget recipe
    k_kind: str                   # "fixed" | "choice" | "uniform" | "list"
    k_args: tuple
    description: str = ""

    def contexts(self) -> np.ndarray:
        """Prefilled context length n_i per sequence (int64, seeded)."""
        return _draw_meta(self)[0]

    def budgets(self) -> np.ndarray:
        """Per-sequence budget k_i in [1, n_cand], or 0 where the Budget
        Predictor chooses it (int64, seeded)."""
        return _draw_meta(self)[1]

    def capacities(self, extra_steps: int = 0) -> np.ndarray:
        """KV capacity per sequence: room for every decode step plus slack."""
        return self.contexts() + self.steps + extra_steps + 1


def _draw_meta(w: Workload):
    """Seeded draw of contexts then budgets (draw order: contexts, budgets)."""
    rng = np.random.default_rng(np.random.SeedSequence([w.seed, 0x6B7564]))
    B = w.batch
    if w.ctx_kind == "fixed":
        ctx = np.full(B, int(w.ctx_args[0]), dtype=np.int64)
    elif w.ctx_kind == "uniform":
        lo, hi = w.ctx_args
        ctx = rng.integers(lo, hi + 1, size=B, dtype=np.int64)
    elif w.ctx_kind == "lognormal":
        median, sigma, lo, hi = w.ctx_args
        z = rng.standard_normal(B)
        ctx = np.clip(np.rint(median * np.exp(sigma * z)), lo, hi).astype(np.int64)
    elif w.ctx_kind == "list":
        ctx = np.asarray(w.ctx_args, dtype=np.int64)
        assert ctx.shape == (B,)
    else:
        raise ValueError(w.ctx_kind)
    Lm = w.shape.n_cand
    if w.k_kind == "fixed":
        k = np.full(B, int(w.k_args[0]), dtype=np.int64)
    elif w.k_kind == "choice":
        k = rng.choice(np.asarray(w.k_args, dtype=np.int64), size=B)
    elif w.k_kind == "uniform":
        lo, hi = w.k_args
        k = rng.integers(lo, hi + 1, size=B, dtype=np.int64)
    elif w.k_kind == "list":
        k = np.asarray(w.k_args, dtype=np.int64)
        assert k.shape == (B,)
    else:
        raise ValueError(w.k_kind)
    ok = (k >= 1) & (k <= Lm)
    if w.shape.predictor_hidden > 0:
        ok |= k == 0
    assert np.all(ok), "budgets must lie in [1, n_cand] (0: predicted)"
    return ctx, k


# --------------------------------------------------------------------------
# Model shapes
# --------------------------------------------------------------------------
TINY_F32 = ModelShape("tiny-f32", 8, 256, 4, 4, 64, 688, 128, "f32", 1e-5, 1e4)
LLAMA3_8B = ModelShape("llama3-8b", 32, 4096, 32, 8, 128, 14336, 256, "bf16", 1e-5, 5e5)
LLAMA2_13B = ModelShape("llama2-13b", 40, 5120, 40, 40, 128, 13824, 256, "bf16", 1e-5, 1e4)
QWEN25_7B = ModelShape("qwen2.5-7b", 28, 3584, 28, 4, 128, 18944, 256, "bf16", 1e-6, 1e6,
                       qkv_bias=True)

# Small shapes for parity tests: several GEMM tiles with ragged tails (d and F not
# multiples of 128, N of QKV not a multiple of 128), GQA groups 3 and 4, both
# head dims, bias on/off, random RMSNorm gains.
SMALL_GQA_BF16 = ModelShape("small-gqa-bf16", 6, 576, 9, 3, 64, 1472, 64, "bf16", 1e-5, 1e4,
                            random_norm=True)
SMALL_QWEN_BF16 = ModelShape("small-qwen-bf16", 7, 768, 6, 2, 128, 2048, 96, "bf16", 1e-6, 1e6,
                             qkv_bias=True, random_norm=True)
SMALL_F32 = ModelShape("small-f32", 5, 320, 5, 1, 64, 832, 48, "f32", 1e-5, 1e4,
                       qkv_bias=True, random_norm=True)

# --------------------------------------------------------------------------
# Decode workloads
# --------------------------------------------------------------------------
C1_TINY = Workload("tiny-f32-b4", TINY_F32, batch=4, steps=1, seed=0,
                   ctx_kind="fixed", ctx_args=(128,), k_kind="fixed", k_args=(3,),
                   description="8 layers, d=256, MHA 4x64, F=688, fp32, B=4, ctx 128, k=3 of 6")
C2_LLAMA3_B1 = Workload("llama3-8b-b1", LLAMA3_8B, batch=1, steps=64, seed=0,
                        ctx_kind="fixed", ctx_args=(2048,), k_kind="fixed", k_args=(15,),
                        description="Llama-3-8B shape, bf16, B=1, ctx 2048, k=15 of 30, 64 steps")
C3_LLAMA3_B64 = Workload("llama3-8b-b64-mixed", LLAMA3_8B, batch=64, steps=32, seed=0,
                         ctx_kind="uniform", ctx_args=(512, 4096),
                         k_kind="choice", k_args=(8, 15, 23, 30),
                         description="Llama-3-8B shape, bf16, B=64, ctx U[512,4096], k in {8,15,23,30}")
C4_LLAMA2_13B = Workload("llama2-13b-b32", LLAMA2_13B, batch=32, steps=32, seed=0,
                         ctx_kind="fixed", ctx_args=(4096,), k_kind="fixed", k_args=(23,),
                         description="Llama-2-13B shape (MHA), bf16, B=32, ctx 4096, k=23 of 38")
C5_QWEN_B256 = Workload("qwen2.5-7b-b256", QWEN25_7B, batch=256, steps=16, seed=0,
                        ctx_kind="lognormal", ctx_args=(2048, 0.5, 512, 8192),
                        k_kind="uniform", k_args=(6, 26),
                        description="Qwen2.5-7B shape, bf16 + qkv bias, B=256, ctx lognormal "
                                    "median 2048 sigma 0.5 clip [512,8192], k U{6..26}")

FULL_WORKLOADS = [C1_TINY, C2_LLAMA3_B1, C3_LLAMA3_B64, C4_LLAMA2_13B, C5_QWEN_B256]

# Small parity workloads (oracle finishes in seconds).  Contexts include n_i = 0
# (the new token is the only position), 1, and values that are not multiples of
# the attention chunk; budgets include k = 1 and k = L_mid.
T_GQA = Workload("t-gqa-bf16", SMALL_GQA_BF16, batch=37, steps=3, seed=1,
                 ctx_kind="uniform", ctx_args=(0, 300), k_kind="uniform", k_args=(1, 4))
T_QWEN = Workload("t-qwen-bf16", SMALL_QWEN_BF16, batch=19, steps=3, seed=2,
                  ctx_kind="list",
                  ctx_args=(0, 1, 2, 63, 64, 65, 127, 128, 129, 255, 256, 257, 511, 700, 5, 17,
                            1000, 333, 90),
                  k_kind="list", k_args=(1, 5, 3, 2, 4, 5, 1, 1, 2, 3, 4, 5, 5, 2, 3, 1, 4, 2, 3))
T_F32 = Workload("t-small-f32", SMALL_F32, batch=6, steps=2, seed=3,
                 ctx_kind="list", ctx_args=(0, 7, 64, 129, 31, 300),
                 k_kind="list", k_args=(1, 2, 3, 3, 2, 1))

# Three-layer models with the benchmark shapes' per-layer sizes, for kernel
# profiling captures that must stay small on the device.
P_LLAMA3_3L_B1 = Workload("llama3-8b-3layer-b1", dataclasses.replace(LLAMA3_8B, name="llama3-8b-3layer", n_layers=3),
                          batch=1, steps=16, seed=0, ctx_kind="fixed", ctx_args=(2048,),
                          k_kind="fixed", k_args=(1,))
P_QWEN_3L_B256 = Workload("qwen2.5-7b-3layer-b256",
                          dataclasses.replace(QWEN25_7B, name="qwen2.5-7b-3layer", n_layers=3),
                          batch=256, steps=8, seed=0, ctx_kind="lognormal", ctx_args=(2048, 0.5, 512, 8192),
                          k_kind="fixed", k_args=(1,))

# Routed prefill: 16 prompts of 128..1024 tokens (seeded), fresh sequences,
# budget k = 15 of 30 (the 50% column of the paper's speed table).
PF_LLAMA3_B16 = Workload("llama3-8b-prefill-b16", LLAMA3_8B, batch=16, steps=1, seed=0,
                         ctx_kind="fixed", ctx_args=(0,), k_kind="fixed", k_args=(15,),
                         description="Llama-3-8B shape, bf16, 16 prompts of U[128,1024] tokens, k=15 of 30")


# Three-layer model with the same per-layer sizes, 4 prompts: kernel captures.
P_PF_LLAMA3_3L_B4 = Workload("llama3-8b-3layer-prefill-b4",
                             dataclasses.replace(LLAMA3_8B, name="llama3-8b-3layer", n_layers=3),
                             batch=4, steps=1, seed=0, ctx_kind="fixed", ctx_args=(0,), k_kind="fixed",
                             k_args=(1,))


def prompt_lengths(w: Workload, lo: int = 128, hi: int = 1024) -> np.ndarray:
    """Seeded prompt lengths U[lo, hi] of a prefill workload."""
    rng = np.random.default_rng(np.random.SeedSequence([w.seed, 0x7066]))
    return rng.integers(lo, hi + 1, size=w.batch, dtype=np.int64)


# Router variants on the small shapes: K and K + V planner features, a context
# layer c > 0, the masked skip-KV variant, and the Budget Predictor (budget 0 =
# predicted).
T_PRED = Workload("t-small-f32-pred", dataclasses.replace(SMALL_F32, name="small-f32-pred", predictor_hidden=24),
                  batch=6, steps=2, seed=3, ctx_kind="list", ctx_args=(0, 7, 64, 129, 31, 300),
                  k_kind="list", k_args=(0, 2, 0, 3, 0, 0))
T_VARIANTS = [
    Workload("t-gqa-bf16-k", dataclasses.replace(SMALL_GQA_BF16, name="small-gqa-bf16-k", feature="k"),
             batch=37, steps=3, seed=1, ctx_kind="uniform", ctx_args=(0, 300), k_kind="uniform", k_args=(1, 4)),
    Workload("t-qwen-bf16-kv-c1-pred",
             dataclasses.replace(SMALL_QWEN_BF16, name="small-qwen-bf16-kv-c1-pred", feature="kv", ctx_layer=1,
                                 predictor_hidden=40),
             batch=19, steps=3, seed=2, ctx_kind="list",
             ctx_args=(0, 1, 2, 63, 64, 65, 127, 128, 129, 255, 256, 257, 511, 700, 5, 17, 1000, 333, 90),
             k_kind="list", k_args=(1, 0, 3, 2, 4, 0, 1, 0, 2, 3, 4, 0, 4, 2, 3, 1, 0, 2, 3)),
    Workload("t-gqa-bf16-masked", dataclasses.replace(SMALL_GQA_BF16, name="small-gqa-bf16-masked", skip_kv="masked"),
             batch=37, steps=3, seed=1, ctx_kind="uniform", ctx_args=(0, 300), k_kind="uniform", k_args=(1, 4)),
    Workload("t-small-f32-masked-c2-kv",
             dataclasses.replace(SMALL_F32, name="small-f32-masked-c2-kv", skip_kv="masked", ctx_layer=2,
                                 feature="kv", n_layers=7),
             batch=6, steps=2, seed=3, ctx_kind="list", ctx_args=(0, 7, 64, 129, 31, 300),
             k_kind="list", k_args=(1, 2, 3, 3, 2, 1)),
]

BY_NAME = {w.name: w for w in FULL_WORKLOADS + [T_GQA, T_QWEN, T_F32, T_PRED, P_LLAMA3_3L_B1, P_QWEN_3L_B256,
                                                PF_LLAMA3_B16, P_PF_LLAMA3_3L_B4] + T_VARIANTS}


def with_shape(w: Workload, name: Optional[str] = None, **shape_changes) -> Workload:
    """The same workload on a shape with some fields changed (router variants)."""
    sh = dataclasses.replace(w.shape, name=w.shape.name + "-" + "-".join(f"{k}{v}" for k, v in shape_changes.items()),
                             **shape_changes)
    return dataclasses.replace(w, shape=sh, name=name or f"{w.name}-{sh.name}")


def scaled(w: Workload, *, batch: Optional[int] = None, steps: Optional[int] = None,
           ctx: Optional[List[int]] = None, k: Optional[List[int]] = None,
           name: Optional[str] = None) -> Workload:
    """Same model shape with an explicit batch, contexts or budgets."""
    B = batch if batch is not None else (len(ctx) if ctx is not None else w.batch)
    kw = dict(name=name or f"{w.name}-custom", shape=w.shape, batch=B,
              steps=steps if steps is not None else w.steps, seed=w.seed,
              ctx_kind=w.ctx_kind, ctx_args=w.ctx_args, k_kind=w.k_kind, k_args=w.k_args)
    if ctx is not None:
        kw["ctx_kind"], kw["ctx_args"] = "list", tuple(int(c) for c in ctx)
    if k is not None:
        kw["k_kind"], kw["k_args"] = "list", tuple(int(v) for v in k)
    return Workload(**kw)

