"""Pins of the oracle's read-only cached-prefix probe: the number of leading
full blocks of each prompt that are resident in the prompt's group
(n_cached of Alg. 1), without any change of state.  Expected values are
derived by hand; the probe must also agree with the next step's hit counts
for requests that share nothing within the step."""
import numpy as np

import oracle as O
from _util import make_step, obj_tokens


def _params():
    return O.Params(rho=(100.0,), beta=(100.0,))


def test_probe_counts_leading_resident_blocks_per_group():
    oc = O.OracleCache(64, 16, 2, "prefixshield", _params())
    A = obj_tokens("A", blocks=4)
    B = obj_tokens("B", blocks=2)
    # group 0 caches A (4 blocks) and A's first two blocks followed by B
    g, o, t, _ = make_step([A, np.concatenate([A[:32], B])], [0, 0])
    assert oc.step(1, g, o, t)["status"] == 0
    before = oc.export()
    queries = [
        (A, 0, 4),                                   # whole prompt cached
        (np.concatenate([A, B]), 0, 4),              # cached prefix, then a miss
        (np.concatenate([A[:32], B]), 0, 4),         # the second prompt: 2 + 2 blocks
        (np.concatenate([A[:32], B[16:]]), 0, 2),    # diverges at block 2
        (B, 0, 0),                                   # B's key differs as a first block
        (A, 1, 0),                                   # another group's namespace
        (A[:40], 0, 2),                              # a partial third block is not counted
    ]
    g, o, t, _ = make_step([q for q, _, _ in queries], [grp for _, grp, _ in queries])
    got = oc.cached_prefix(g, o, t)
    assert got.tolist() == [w for _, _, w in queries]
    after = oc.export()
    for k in before:
        a, b = before[k], after[k]
        if isinstance(a, tuple):
            assert all(np.array_equal(x, y) for x, y in zip(a, b)), k
        elif isinstance(a, np.ndarray):
            assert np.array_equal(a, b), k
        else:
            assert a == b, k


def test_probe_equals_the_next_steps_hits_without_in_step_sharing():
    from paper_2608_01657_gb300 import workloads as W
    steps = W.fuzz_steps(61, 2, 1, 40, docs_per_group=3, doc_blocks=8, fresh_max_blocks=4)
    oc = O.OracleCache(40, 16, 2, "prefixshield", _params())
    for st in steps:
        want = oc.cached_prefix(st.groups, st.offsets, st.tokens)
        r = oc.step(st.now, st.groups, st.offsets, st.tokens)
        # one request a step: no in-step sharing, so hits = the probe's count
        assert r["hit_blocks"].tolist() == want.tolist()
