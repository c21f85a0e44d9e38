"""Brute force on pools of at most 8 blocks.

Every trace of two steps over a small prompt alphabet (one or two requests per
step, pools of 1-3 blocks), and random multi-step traces over two groups and
pools of 2-8 blocks, for every policy.  After every step the invariants of
``_util.check_step`` hold; for lru the victims are exactly the oldest unpinned
blocks and for prefixshield they equal the water-filling closed form of Alg. 2.
"""
import itertools

import numpy as np
import pytest

import oracle as O
from _util import check_step, make_step, obj_tokens

X, Y = obj_tokens("X"), obj_tokens("Y")
PROMPTS = [X, Y, np.concatenate([X, Y]), np.concatenate([Y, X]), np.concatenate([X, X])]
STEPS = [(p,) for p in range(5)] + list(itertools.product(range(5), repeat=2))


@pytest.mark.parametrize("policy", ["lru", "s3fifo", "prefixshield"])
@pytest.mark.parametrize("N", [1, 2, 3])
def test_exhaustive_two_step_traces(policy, N):
    prm = O.Params(rho=(1.0,), beta=(1.0,))
    for s1 in STEPS:
        for s2 in STEPS:
            oc = O.OracleCache(N, 16, 1, policy, prm)
            for t, s in enumerate((s1, s2)):
                g, o, tk, _ = make_step([PROMPTS[i] for i in s])
                before = oc.export()
                r = oc.step(t + 1, g, o, tk)
                check_step(oc, before, oc.export(), (g, o, tk, t + 1), r, policy)


@pytest.mark.parametrize("policy", ["lru", "s3fifo", "prefixshield"])
def test_random_multi_step_traces(policy):
    rng = np.random.default_rng(17)
    alphabet = [obj_tokens(n) for n in "ABCD"]
    for trial in range(150):
        N = int(rng.integers(2, 9))
        oc = O.OracleCache(N, 16, 2, policy, O.Params(rho=(1.0,), beta=(2.0,)))
        now = 0
        for t in range(int(rng.integers(3, 9))):
            R = int(rng.integers(0, 4))
            prompts, groups = [], []
            for _ in range(R):
                L = int(rng.integers(0, 4))
                prompts.append(np.concatenate([alphabet[int(rng.integers(0, 4))] for _ in range(L)] +
                                              [np.zeros(int(rng.integers(0, 3)), np.int32)]))
                groups.append(int(rng.integers(0, 2)))
            now += int(rng.integers(0, 2))
            g, o, tk, _ = make_step(prompts, groups)
            before = oc.export()
            r = oc.step(now, g, o, tk)
            check_step(oc, before, oc.export(), (g, o, tk, now), r, policy)
