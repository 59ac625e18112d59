"""The roofline numerator (workloads/cost.py) against an enumeration of the
tensors one routed decode step (or prefill) must move, built matrix by matrix
from the model's dimensions and sequence by sequence from the mask."""
import numpy as np

from workloads import configs as C
from workloads import cost

SHAPE = C.ModelShape("cost-tiny", n_layers=6, d_model=32, n_q_heads=4, n_kv_heads=2, head_dim=8, ffn_dim=48,
                     dm_hidden=8, dtype="bf16", rms_eps=1e-5, rope_theta=1e4, qkv_bias=True)


def _matrices(s):
    d, F, hd = s.d_model, s.ffn_dim, s.head_dim
    return {"q": (s.n_q_heads * hd, d), "k": (s.n_kv_heads * hd, d), "v": (s.n_kv_heads * hd, d),
            "o": (d, s.n_q_heads * hd), "gate": (F, d), "up": (F, d), "down": (d, F)}


def _mask(rng, B, L):
    m = rng.integers(0, 2, size=(B, L)).astype(np.uint8)
    m[:, 0] = m[:, -1] = 1
    m[:, 2] = 0            # a middle layer that no sequence selected
    return m


def test_step_cost_equals_enumeration():
    s = SHAPE
    rng = np.random.default_rng(7)
    B, L = 5, s.n_layers
    mask = _mask(rng, B, L)
    n = rng.integers(0, 40, size=B)
    e = s.elem_bytes
    mats = _matrices(s)
    weights = flops = kv_read = kv_write = 0
    for l in range(L):
        if mask[:, l].any():
            weights += sum(a * b for a, b in mats.values()) * e
            weights += 2 * s.d_model * 4                                  # the two RMSNorm gains (fp32)
            weights += (s.n_q_heads + 2 * s.n_kv_heads) * s.head_dim * 4  # q/k/v bias (fp32)
        for i in range(B):
            kv_write += 2 * s.n_kv_heads * s.head_dim * e                # K and V at the new position
            if mask[i, l]:
                positions = n[i] + 1
                kv_read += 2 * positions * s.n_kv_heads * s.head_dim * e
                flops += sum(2 * a * b for a, b in mats.values())
                flops += s.n_q_heads * positions * s.head_dim * 2 * 2   # q.K and p.V per query head
    Lm = L - 2
    dm = (s.dm_hidden * 2 * s.d_model + s.dm_hidden + Lm * s.dm_hidden + Lm + Lm) * 4   # W1 b1 W2 b2 prior
    flops += B * 2 * (s.dm_hidden * 2 * s.d_model + Lm * s.dm_hidden)
    small = dm + 2 * B * s.n_kv_heads * s.head_dim * 4 + 2 * B * s.d_model * 4   # pool sums, h in / out
    got = cost.step_cost(s, mask, n)
    assert got["weight_bytes"] == weights
    assert got["kv_read_bytes"] == kv_read
    assert got["kv_write_bytes"] == kv_write
    assert got["bytes"] == weights + kv_read + kv_write + small
    assert got["flops"] == flops
    assert got["layers_used"] == L - 1 and got["exec_pairs"] == int(mask.sum())


def test_prefill_cost_equals_token_by_token_sum():
    s = SHAPE
    rng = np.random.default_rng(3)
    B, L = 4, s.n_layers
    mask = _mask(rng, B, L)
    T = rng.integers(1, 30, size=B)
    n0 = rng.integers(0, 20, size=B)
    mats = _matrices(s)
    flops = 0
    for i in range(B):
        for l in range(L):
            if not mask[i, l]:
                continue
            for t in range(T[i]):
                flops += sum(2 * a * b for a, b in mats.values())
                flops += 4 * s.n_q_heads * s.head_dim * (n0[i] + t + 1)   # causal: the cache and tokens 0..t
    got = cost.prefill_cost(s, mask, T, n0)
    assert got["flops"] == flops
    assert got["tokens"] == int(T.sum())


def test_roofline_takes_the_larger_bound():
    c = {"bytes": 6.8e9, "flops": 1.0e12}
    assert cost.roofline_seconds(c, 6800.0, 1000.0) == 1e-3      # 1 ms of HBM vs 1 ms of tensor
    assert cost.roofline_seconds({"bytes": 6.8e9, "flops": 2e12}, 6800.0, 1000.0) == 2e-3
