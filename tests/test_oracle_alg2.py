"""Pins of the oracle's literal Alg. 2 victim loop (Eq. 6-8 and the tie rule)
against an independent water-filling closed form (``_util.alg2_closed_form``)
and a hand-derived example."""
import numpy as np
import pytest

import oracle as O
from _util import alg2_closed_form


def test_hand_example():
    """P = (5, 3), decrements (2, 1), keys g0 = (10, 30, 50), g1 = (20, 40, 60).
    Loop: g0 (P0 5->3); tie 3/3, heads 30 vs 20 -> g1 (P1 3->2); g0 (3->1);
    g1 (2->1); tie 1/1, heads 50 vs 60 -> g0."""
    Q = [[10, 30, 50], [20, 40, 60]]
    assert O.alg2_loop([5, 3], [2, 1], 0, Q, 5) == [(0, 0), (1, 0), (0, 1), (1, 1), (0, 2)]
    # eps = 1: only values > 1 are eligible (5, 3 of g0; 3, 2 of g1), then the
    # global fallback takes the smallest remaining keys, 50 then 60.
    assert O.alg2_loop([5, 3], [2, 1], 1, Q, 6) == [(0, 0), (1, 0), (0, 1), (1, 1), (0, 2), (1, 2)]
    # no indebted group: pure global order by key
    assert O.alg2_loop([0, 0], [1, 1], 0, Q, 3) == [(0, 0), (1, 0), (0, 1)]


@pytest.mark.parametrize("seed", range(300))
def test_random_instances_with_ties(seed):
    rng = np.random.default_rng(seed)
    G = int(rng.integers(1, 7))
    delta = [int(x) for x in rng.choice([1, 2, 3, 6], size=G)]
    P = [int(x) for x in rng.integers(0, 6, size=G) * 6]  # common grid: frequent ties
    eps = int(rng.choice([0, 0, 1, 5]))
    sizes = rng.integers(0, 7, size=G)
    keys = rng.permutation(10 * (sizes.sum() + 1))[: sizes.sum()]
    Q, k = [], 0
    for g in range(G):
        Q.append(sorted(int(x) for x in keys[k:k + sizes[g]]))
        k += sizes[g]
    m = int(rng.integers(0, sizes.sum() + 1))
    assert O.alg2_loop(P, delta, eps, Q, m) == alg2_closed_form(P, delta, eps, Q, m)
