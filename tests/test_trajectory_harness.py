"""The layer-major trajectory harness (tests/trajectory.py) computes what the
oracle's step-by-step decode computes: same routes, hidden states and K/V."""
import numpy as np
import pytest

import trajectory as T
from oracle import adapter as A
from oracle import buddy_oracle as O
from workloads import configs as C


@pytest.mark.parametrize("w", [C.T_QWEN, C.T_PRED, C.T_VARIANTS[3]], ids=lambda w: w.name)
def test_layer_major_equals_step_by_step(w):
    s = w.shape
    model = A.build_model(s, w.seed)
    n0, k = w.contexts(), w.budgets()
    S = 3
    sampled = [0, 2, w.batch - 1]
    h_in = [A.workload_inputs(w, t) for t in range(S)]
    ev = T.evaluate(model, n0, k, h_in, sampled,
                    lambda layers, seqs: A.build_state(s, w.seed, n0, layers=layers, seqs=seqs))
    st = A.build_state(s, w.seed, n0)
    for t in range(S):
        r = O.decode_step(model, st, h_in[t], k)
        np.testing.assert_allclose(ev["scores"][t], r.scores, rtol=1e-12, atol=1e-12)
        assert ev["sel"][t] == r.sel and ev["k"][t] == r.k
        for i in sampled:
            np.testing.assert_allclose(ev["H"][i][t], r.h_out[i], rtol=1e-11, atol=1e-11)
            for l in range(s.n_layers):
                o = ev["kv"][(l, i)][t]
                if (l, i) in r.kv_new:
                    np.testing.assert_allclose(o[0], r.kv_new[(l, i)][0], rtol=1e-11, atol=1e-11)
                    np.testing.assert_allclose(o[1], r.kv_new[(l, i)][1], rtol=1e-11, atol=1e-11)
                else:
                    assert o is None
