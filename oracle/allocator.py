"""Oracle: the allocation rule (test infrastructure).

Problem Statement: maximise the tokens generated per second subject to a budget on the drop
in generation quality relative to the unquantised model.  The Combined Configurations section
measures every candidate mask and keeps the fastest one whose quality is preserved.

Here a candidate is feasible when its Top-1 agreement with the bf16 path is at least
``min_top1`` and its perplexity delta is at most ``max_ppl_delta``; among the feasible
candidates the rule returns the one with the smallest per-token latency (equivalently the
largest speedup); ties go to the mask with fewer INT8 sublayers, then to the earlier
candidate.  The all-bf16 mask is feasible by definition (agreement 1, delta 0).
"""
from __future__ import annotations


def choose(candidates, min_top1: float = 0.989, max_ppl_delta: float = 0.01):
    """candidates: sequence of dicts with keys name, latency (any time unit), top1, ppl_delta,
    n_int8.  Returns the chosen candidate's index."""
    best = None
    for idx, c in enumerate(candidates):
        if not (c["top1"] >= min_top1 and c["ppl_delta"] <= max_ppl_delta):
            continue
        key = (c["latency"], c["n_int8"], idx)
        if best is None or key < best[0]:
            best = (key, idx)
    return None if best is None else best[1]


def greedy_order(gain, top1, ppl_delta, min_top1: float = 0.989, max_ppl_delta: float = 0.01):
    """Allocation per sublayer (below the paper's groups; its title names this granularity, its
    search stops at groups): rank the sublayers whose own single-sublayer mask is faster than
    all-bf16 (gain > 0) and meets the budget by itself, by latency gain per unit of quality cost,
    where the cost adds the Top-1 loss and the perplexity increase, each as a fraction of its
    budget.  Highest ratio first; equal ratios keep the lower index first.  All arithmetic in
    Python floats (double precision)."""
    t_scale = max(1e-6, 1.0 - float(min_top1))
    p_scale = max(1e-6, float(max_ppl_delta))
    ranked = []
    for i, (g, t, p) in enumerate(zip(gain, top1, ppl_delta)):
        g, t, p = float(g), float(t), float(p)
        if not g > 0.0 or not (t >= min_top1 and p <= max_ppl_delta):
            continue
        cost = max(0.0, 1.0 - t) / t_scale + max(0.0, p) / p_scale
        ranked.append((-(g / (cost + 1e-3)), i))
    ranked.sort()
    return [i for _, i in ranked]


def greedy_select(order, feasible):
    """Add the ranked sublayers one at a time, keeping each one only while feasible(set) still
    holds for the cumulative set; returns the accepted sublayers in order of acceptance."""
    chosen = []
    for i in order:
        if feasible(chosen + [i]):
            chosen.append(i)
    return chosen
