"""The seeded input recipe: the five benchmark workloads carry the shapes,
batches, context and budget distributions and step counts they are stated
with, and the generator's draws have the stated moments and bounds."""
import numpy as np
import torch

from workloads import configs as C
from workloads import synth


def _shape(s, L, d, nq, nkv, hd, F, r, dtype, eps, theta, bias=False):
    assert (s.n_layers, s.d_model, s.n_q_heads, s.n_kv_heads, s.head_dim, s.ffn_dim, s.dm_hidden) == \
        (L, d, nq, nkv, hd, F, r)
    assert s.dtype == dtype and s.rms_eps == eps and s.rope_theta == theta and s.qkv_bias == bias
    assert s.n_cand == L - 2 and s.feature == "v" and s.ctx_layer == 0 and s.skip_kv == "zero"


def test_benchmark_workload_shapes():
    _shape(C.C1_TINY.shape, 8, 256, 4, 4, 64, 688, 128, "f32", 1e-5, 1e4)
    _shape(C.C2_LLAMA3_B1.shape, 32, 4096, 32, 8, 128, 14336, 256, "bf16", 1e-5, 5e5)
    _shape(C.C3_LLAMA3_B64.shape, 32, 4096, 32, 8, 128, 14336, 256, "bf16", 1e-5, 5e5)
    _shape(C.C4_LLAMA2_13B.shape, 40, 5120, 40, 40, 128, 13824, 256, "bf16", 1e-5, 1e4)
    _shape(C.C5_QWEN_B256.shape, 28, 3584, 28, 4, 128, 18944, 256, "bf16", 1e-6, 1e6, bias=True)
    assert [(w.batch, w.steps) for w in C.FULL_WORKLOADS] == [(4, 1), (1, 64), (64, 32), (32, 32), (256, 16)]


def test_benchmark_workload_contexts_and_budgets():
    for w, ctx, k in ((C.C1_TINY, 128, 3), (C.C2_LLAMA3_B1, 2048, 15), (C.C4_LLAMA2_13B, 4096, 23)):
        assert np.all(w.contexts() == ctx) and np.all(w.budgets() == k)
    n, k = C.C3_LLAMA3_B64.contexts(), C.C3_LLAMA3_B64.budgets()
    assert n.min() >= 512 and n.max() <= 4096 and len(np.unique(n)) > 50
    assert set(k.tolist()) == {8, 15, 23, 30}
    n, k = C.C5_QWEN_B256.contexts(), C.C5_QWEN_B256.budgets()
    assert n.min() >= 512 and n.max() <= 8192
    assert 1800 <= np.median(n) <= 2300                    # lognormal around 2048
    z = np.log(n[(n > 512) & (n < 8192)] / 2048.0)
    assert 0.4 < z.std() < 0.6                             # sigma 0.5 in log space
    assert k.min() >= 6 and k.max() <= 26 and len(np.unique(k)) == 21
    # the draw is a pure function of the seed
    assert np.array_equal(C.C5_QWEN_B256.contexts(), n) and np.array_equal(C.C5_QWEN_B256.budgets(), k)


def test_generator_moments_bounds_and_slices():
    key = synth.stream_key(0, "k_cache", 3, 7)
    x = synth.normal((1 << 20,), key, 1.0, torch.float32, "cpu").double().numpy()
    assert abs(x.mean()) < 5e-3 and abs(x.std() - 1.0) < 5e-3      # mean 0, sigma 1
    assert np.abs(x).max() <= 2.0 * 65535 / synth._IH_STD + 1e-6    # Irwin-Hall(4): |z| <= 3.46
    assert np.abs(x).max() > 3.0
    # a slice regenerated from its start offset is the same values
    part = synth.normal((1000,), key, 1.0, torch.float32, "cpu", start=12345).double().numpy()
    assert np.array_equal(part, x[12345:13345])
    # bf16 storage is the rounded fp32 value
    b = synth.normal((4096,), key, 1.0, torch.bfloat16, "cpu")
    assert torch.equal(b, torch.from_numpy(x[:4096].astype(np.float32)).to(torch.bfloat16))
    # distinct streams are uncorrelated
    y = synth.normal((1 << 20,), synth.stream_key(0, "v_cache", 3, 7), 1.0, torch.float32, "cpu").double().numpy()
    assert abs(np.corrcoef(x, y)[0, 1]) < 5e-3
