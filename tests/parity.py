"""Parity rules between the GPU path and the oracle.

* Routes: the GPU's selected set must equal the oracle's, except when the
  oracle's k-th and (k+1)-th scores differ by less than ROUTE_MARGIN: then the
  oracle adopts the GPU's set, provided every layer on which the two sets
  differ has an oracle score within ROUTE_MARGIN of the k-th score.
* Hidden states: per sequence, max_j |g_j - o_j| / max_j |o_j| below
  HIDDEN_TOL[dtype].
* Compaction indices (rows/count): bit-exact against the oracle's grouping of
  the (adopted) selections.
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

import numpy as np

ROUTE_MARGIN = 1e-3
HIDDEN_TOL = {"f32": 1e-4, "bf16": 2e-2}
# K/V written at the new position derive from the same layer's hidden state:
# same normwise-by-max bound
KV_TOL = HIDDEN_TOL


def adopt_routes(o_scores: np.ndarray, o_sel: Sequence[Sequence[int]], g_sel: Sequence[Sequence[int]],
                 k: Sequence[int], first: int = 1) -> Tuple[List[List[int]], List[str], int]:
    """Returns (sets the oracle continues with, failures, number adopted).
    o_scores[i][j] belongs to layer first + j; k[i] is the budget the
    sequence used (the set sizes decide it where k[i] is 0, i.e. predicted)."""
    out, fails, adopted = [], [], 0
    for i, (os_, gs) in enumerate(zip(o_sel, g_sel)):
        os_, gs = sorted(int(x) for x in os_), sorted(int(x) for x in gs)
        if os_ == gs:
            out.append(os_)
            continue
        s = np.asarray(o_scores[i], dtype=np.float64)
        ki = int(k[i]) if int(k[i]) > 0 else len(os_)
        srt = np.sort(s)[::-1]
        if len(gs) != ki or ki >= len(s):
            fails.append(f"seq {i}: gpu {gs} vs oracle {os_} (k={ki})")
            out.append(os_)
            continue
        kth = srt[ki - 1]
        gap = srt[ki - 1] - srt[ki]
        diff = set(os_) ^ set(gs)
        near = all(abs(s[l - first] - kth) < ROUTE_MARGIN for l in diff)
        if gap < ROUTE_MARGIN and near:
            out.append(gs)
            adopted += 1
        else:
            fails.append(f"seq {i}: gpu {gs} vs oracle {os_}, gap {gap:.3g}")
            out.append(os_)
    return out, fails, adopted


def adopt_budgets(o_k: Sequence[int], g_k: Sequence[int], logits: Sequence[np.ndarray],
                  given: Sequence[int]) -> Tuple[List[int], List[str]]:
    """Budgets the oracle continues with.  Where the Budget Predictor chose
    (given[i] == 0) and the GPU's k^ differs from the oracle's, the oracle
    adopts it if both are within ROUTE_MARGIN of the largest oracle logit (a
    near-tie of the argmax, the same rule as for the layer ranking)."""
    out, fails = [], []
    for i, (ok, gk) in enumerate(zip(o_k, g_k)):
        if ok == gk:
            out.append(ok)
            continue
        if int(given[i]) == 0 and logits[i] is not None:
            lg = np.asarray(logits[i], dtype=np.float64)
            top = lg.max()
            if 1 <= gk <= len(lg) and top - lg[gk - 1] < ROUTE_MARGIN and top - lg[ok - 1] < ROUTE_MARGIN:
                out.append(gk)
                continue
        fails.append(f"seq {i}: gpu budget {gk} vs oracle {ok} (given {given[i]})")
        out.append(ok)
    return out, fails


def max_rel_err(g: np.ndarray, o: np.ndarray) -> float:
    g = np.asarray(g, dtype=np.float64)
    o = np.asarray(o, dtype=np.float64)
    return float(np.max(np.abs(g - o)) / max(np.max(np.abs(o)), 1e-30))


def sel_from_mask(mask: np.ndarray, first: int = 1) -> List[List[int]]:
    L = mask.shape[1]
    return [[l for l in range(first, L - 1) if mask[i, l]] for i in range(mask.shape[0])]


def oracle_for(dw, gen_device="cuda"):
    """Oracle model and state of a device workload (tests/GPU only)."""
    from oracle import adapter as A
    from workloads import synth
    w = dw.w
    s = w.shape
    model = A.build_model(s, w.seed, layer_source=lambda l: synth.layer_weights(s, w.seed, l, gen_device),
                          dm_source=lambda: synth.dm_weights(s, w.seed, gen_device),
                          prior=dw.prior, omega=0.1 if dw.prior is not None else 0.0,
                          cache_layers=s.n_layers,
                          predictor_source=lambda: synth.predictor_weights(s, w.seed, gen_device))
    st = A.build_state(s, w.seed, w.contexts(), gen_device=gen_device)
    return model, st


def adopt(model, rr, g_mask, k_given):
    """Near-tie rules: the oracle takes the GPU's budget where the Budget
    Predictor's argmax is a near-tie, then the GPU's set where the layer
    ranking is.  Returns (sets, budgets, failures, adopted)."""
    from oracle import buddy_oracle as O
    first = model.shape.first_candidate
    g_sel = sel_from_mask(g_mask, first)
    g_k = [len(x) for x in g_sel]
    logits = [O.predictor_logits(model.predictor, rr.x[i]) if model.predictor is not None else None
              for i in range(len(g_sel))]
    ks, fails_k = adopt_budgets(rr.k, g_k, logits, k_given)
    o_sel = [rr.sel[i] if ks[i] == rr.k[i] else O.top_k_layers(rr.scores[i], ks[i], first)
             for i in range(len(ks))]
    sel, fails, n = adopt_routes(rr.scores, o_sel, g_sel, ks, first)
    return sel, ks, fails_k + fails, n
