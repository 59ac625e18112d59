"""Layer-major evaluation of a decode trajectory with the oracle's building
blocks (test harness).

A decode step's block l at sequence i depends on the step's hidden state
after block l-1 and on block l's cache, which holds the entries of the
earlier steps.  So a whole trajectory can be evaluated one block at a time:
the projections of all (sequence, step) rows of a block at once (rows are
independent), the attention of each step in step order against the cache as
it grows (Eq. 9), then the block's tail.  Every value is the one the oracle's
step-by-step decode computes; only the order of independent work differs, so
that each block's float64 weights are materialised once per trajectory
(tests/test_trajectory_harness.py checks the equality).
"""
from __future__ import annotations

from typing import Callable, Dict, List, Optional, Sequence

import numpy as np

import parity as P
from oracle import buddy_oracle as O


def layer_over_trajectory(sh, W, st, l, X, execs, pos0, skip_zero):
    """Block l for every (sequence i, step t): X[i] [S, d] inputs per step,
    execs[i][t] whether step t executes the block, pos0[i] the position of
    step 0.  Returns the outputs (identity where skipped) and the entries
    written per step (zeros for skipped steps in the zero variant, None where
    nothing is stored)."""
    seqs = sorted(X)
    S = X[seqs[0]].shape[0]
    run = [(i, t) for i in seqs for t in range(S) if execs[i][t]]
    out = {i: X[i].copy() for i in seqs}
    written = {i: [None] * S for i in seqs}
    if run:
        Hr = np.stack([X[i][t] for i, t in run])
        q, k, v = O.qkv_project(sh, W, Hr, [pos0[i] + t for i, t in run])
        j_of = {it: j for j, it in enumerate(run)}
        attn = np.empty((len(run), sh.n_q_heads * sh.head_dim))
    zero = np.zeros((sh.n_kv_heads, sh.head_dim))
    for i in seqs:
        for t in range(S):
            if execs[i][t]:
                j = j_of[(i, t)]
                Kc, Vc = st.get(l, i)
                attn[j] = O.decode_attention(q[j], Kc, Vc, sh.group, k[j], v[j]).reshape(-1)
                st.append(l, i, k[j], v[j])
                written[i][t] = (k[j], v[j])
            elif skip_zero:
                st.append(l, i, zero, zero)
                written[i][t] = (zero, zero)
    if run:
        Ho = O.block_tail(sh, W, Hr, attn)
        for j, (i, t) in enumerate(run):
            out[i][t] = Ho[j]
    return out, written


def evaluate(model, n0: Sequence[int], k: Sequence[int], h_in: List[np.ndarray], sampled: Sequence[int],
             state_for: Callable[[Sequence[int], Optional[Sequence[int]]], O.KVState],
             gpu_masks: Optional[List[np.ndarray]] = None) -> dict:
    """The trajectory of len(h_in) decode steps from caches of n0[i] positions.

    state_for(layers, seqs) returns a fresh oracle state with the prefilled
    caches of those layers (and sequences; None = all).  Layers 0..c and the
    router run for every sequence; the routed layers for `sampled`.  With
    gpu_masks the near-tie rule adopts the GPU's sets.  Returns per step the
    scores, budgets used, selections and near-tie failures, and for the
    sampled sequences the final hidden states H[i] [S, d] and the entries
    written kv[(l, i)][t]."""
    sh = model.shape
    B, L, S, c = len(n0), sh.n_layers, len(h_in), sh.ctx_layer
    first = sh.first_candidate
    st = state_for(range(c + 1), None)
    X = {i: np.stack([h_in[t][i] for t in range(S)]) for i in range(B)}
    ex_all = {i: [True] * S for i in range(B)}
    kv = {}
    for l in range(c + 1):
        X, wr = layer_over_trajectory(sh, model.layer(l), st, l, X, ex_all, n0, True)
        for i in sampled:
            kv[(l, i)] = wr[i]
    out = {"scores": [], "k": [], "sel": [], "fails": [], "adopted": 0}
    for t in range(S):
        scores = np.empty((B, sh.n_cand))
        sel, ks = [], []
        for i in range(B):
            Kc, Vc = st.get(c, i)
            n = int(n0[i]) + t + 1          # the cache up to and including step t
            x = O.router_input(sh, Kc[:n], Vc[:n], X[i][t])
            scores[i], kk, si = O.route(model, x, k[i])
            sel.append(si)
            ks.append(kk)
        if gpu_masks is not None:
            g_sel = P.sel_from_mask(gpu_masks[t], first)
            sel, fails, na = P.adopt_routes(scores, sel, g_sel, ks, first)
            out["fails"] += [f"step {t}: {f}" for f in fails]
            out["adopted"] += na
        out["scores"].append(scores)
        out["k"].append(ks)
        out["sel"].append(sel)
    st = None
    H = {i: X[i] for i in sampled}
    for l in range(c + 1, L):
        stl = state_for([l], sampled)
        execs = {i: [l == L - 1 or l in out["sel"][t][i] for t in range(S)] for i in sampled}
        H, wr = layer_over_trajectory(sh, model.layer(l), stl, l, H, execs, n0, sh.skip_kv == "zero")
        for i in sampled:
            kv[(l, i)] = wr[i]
    out["H"] = H
    out["kv"] = kv
    return out
