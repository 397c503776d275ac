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
