"""The library's allocation rule (w8a8_choose_mask, host code) against the oracle's rule: on the
paper's combined-configuration table and on random candidate sets (CPU, no GPU needed)."""
import json
import math
import os

import numpy as np
import pytest

from oracle import allocator, masks


@pytest.fixture(scope="module")
def B():
    from paper_2608_28003_gb300 import build
    build.build()
    from paper_2608_28003_gb300 import binding
    return binding


def test_library_rule_reproduces_paper_choice(B, golden_dir):
    gold = json.load(open(os.path.join(golden_dir, "paper_combined_table.json")))
    lat, t1, pd, n8 = [], [], [], []
    for r in gold["rows"]:
        ok = r["quality"] in ("reference", "good", "excellent")
        lat.append(1.0 / r["speedup"])
        t1.append(1.0 if ok else 0.5)
        pd.append(0.0 if ok else 1.0)
        n8.append(masks.PAPER_CONFIGS[r["name"]].n_int8_sublayers())
    names = [r["name"] for r in gold["rows"]]
    assert names[B.choose_mask(lat, t1, pd, n8)] == gold["chosen_quality_preserved"]
    assert names[B.choose_mask(lat, t1, pd, n8, 0.0, 1e30)] == gold["fastest_any_quality"]


def test_library_rule_matches_oracle_on_random_sets(B):
    g = np.random.default_rng(0)
    for trial in range(300):
        n = int(g.integers(1, 20))
        lat = np.round(g.uniform(0.5, 1.0, n), 2).astype(np.float32)  # rounded: ties happen
        t1 = g.choice([0.97, 0.985, 0.989, 0.99, 1.0], n).astype(np.float32)
        pd = g.choice([0.0, 0.005, 0.01, 0.02], n).astype(np.float32)
        n8 = g.integers(0, 53, n).astype(np.int32)
        cands = [{"latency": float(lat[i]), "top1": float(t1[i]), "ppl_delta": float(pd[i]), "n_int8": int(n8[i])}
                 for i in range(n)]
        want = allocator.choose(cands, min_top1=float(np.float32(0.989)), max_ppl_delta=float(np.float32(0.01)))
        got = B.choose_mask(lat.tolist(), t1.tolist(), pd.tolist(), n8.tolist(), 0.989, 0.01)
        assert got == (-1 if want is None else want), trial


def test_library_candidate_masks_equal_paper_groups(B):
    ours = B.candidate_masks()
    ref = list(masks.candidate_masks().items())
    assert [n for n, _ in ours] == [n for n, _ in ref]
    assert [bits for _, bits in ours] == [m.bits() for _, m in ref]


def test_library_greedy_order_matches_oracle_on_random_sets(B):
    g = np.random.default_rng(1)
    mt, mp = float(np.float32(0.989)), float(np.float32(0.01))
    for trial in range(300):
        n = int(g.integers(1, 54))
        gain = np.round(g.uniform(-1.0, 4.0, n), 1).astype(np.float32)  # rounded: equal ratios happen
        t1 = g.choice([0.95, 0.985, 0.989, 0.995, 1.0], n).astype(np.float32)
        pd = g.choice([-0.001, 0.0, 0.004, 0.01, 0.02], n).astype(np.float32)
        want = allocator.greedy_order(gain.tolist(), t1.tolist(), pd.tolist(), mt, mp)
        got = B.greedy_order(gain.tolist(), t1.tolist(), pd.tolist(), mt, mp)
        assert got == want, trial


def test_greedy_order_pins(B):
    mt, mp = float(np.float32(0.99)), float(np.float32(0.01))
    for rule in (lambda *a: allocator.greedy_order(*a, mt, mp), lambda *a: B.greedy_order(*a, mt, mp)):
        # zero quality cost: by gain alone; no gain, or a single that breaks the budget: left out
        assert rule([1.0, 3.0, 2.0, 0.0, -1.0, 5.0], [1.0, 1.0, 1.0, 1.0, 1.0, 0.9],
                    [0.0] * 6) == [1, 2, 0]
        # a small gain at no cost outranks a large gain that spends most of the budget
        assert rule([1.0, 10.0], [1.0, 0.991], [0.0, 0.0]) == [0, 1]
        # equal ratios: the lower index first
        assert rule([2.0, 2.0, 2.0], [1.0, 1.0, 1.0], [0.0, 0.0, 0.0]) == [0, 1, 2]
        # a perplexity decrease is not a negative cost
        assert rule([1.0, 1.0], [1.0, 1.0], [-0.5, 0.0]) == [0, 1]


def test_greedy_select_is_feasible_and_maximal():
    """With costs that add up (a monotone budget), the selection is feasible, keeps the ranked
    order, and no rejected item fits beside the final set (it did not fit beside a subset of it)."""
    g = np.random.default_rng(2)
    for _ in range(200):
        n = int(g.integers(1, 9))
        cost = g.uniform(0.0, 0.6, n)
        order = [int(i) for i in g.permutation(n)]
        feasible = lambda s: sum(cost[i] for i in s) <= 1.0  # noqa: E731
        got = allocator.greedy_select(order, feasible)
        assert feasible(got)
        assert got == [i for i in order if i in got]
        assert all(not feasible(got + [j]) for j in order if j not in got)
