"""Pins of the batch grant rule (reading A3 of the step): claimed keys are
ranked in (request, position) order and only the first `avail` ranks are
materialized; a request's in-step hits are the granted run of keys that
earlier requests of the step claimed; a request whose run stops at an
ungranted key admits nothing; the allocated ids (ascending) pair with the
granted keys in (request, position) order.  Both steps below start from an
empty pool, so avail = N and nothing is evicted; the expected values are
derived by hand.
"""
import numpy as np

import oracle as O
from _util import make_step, obj_tokens

P = obj_tokens("P", blocks=3)
Q = obj_tokens("Q", blocks=1)
S = obj_tokens("S", blocks=3)
T = obj_tokens("T", blocks=1)


def _stat(oc, name):
    return int(oc.stats()[:, O.STAT_NAMES.index(name)].sum())


def test_ranks_past_avail_are_not_materialized():
    """N = 5.  r0 = P (claims ranks 0-2), r1 = P + Q (P hits in step; Q is
    rank 3), r2 = S (ranks 4-6).  avail = 5: r0 gets 3, r1 gets 1 (Q) and 3
    in-step hits, r2 gets S's first block only; ids 0-4 in that order."""
    oc = O.OracleCache(5, 16, 1, "prefixshield", O.Params(rho=(100.0,), beta=(100.0,)))
    g, o, t, _ = make_step([P, np.concatenate([P, Q]), S])
    r = oc.step(1, g, o, t)
    assert r["status"] == 0
    assert r["hit_blocks"].tolist() == [0, 3, 0]
    assert r["admitted_blocks"].tolist() == [3, 1, 1]
    assert r["admitted_offsets"].tolist() == [0, 3, 4, 5]
    assert r["admitted_ids"].tolist() == [0, 1, 2, 3, 4]
    assert len(r["evicted_ids"]) == 0 and len(r["invalidated_ids"]) == 0
    assert _stat(oc, "ungranted_blocks") == 2 and _stat(oc, "instep_hit_blocks") == 3
    # the charges are the granted blocks only (I1): 100 - 5 blocks
    assert int(oc.export()["B"][0, 0]) == 95 << 20
    # S's second and third blocks were never cached: a later S hits one block
    g, o, t, _ = make_step([S])
    r = oc.step(2, g, o, t)
    assert r["hit_blocks"].tolist() == [1]


def test_a_run_that_stops_at_an_ungranted_key_admits_nothing():
    """N = 4.  r0 = P (ranks 0-2), r1 = S (ranks 3-5), r2 = S + T: its first
    three keys are r1's claims, of which only S's first (rank 3) is granted,
    so e_2 = 1 < 3 and r2 admits nothing (T would be rank 6 anyway)."""
    oc = O.OracleCache(4, 16, 1, "prefixshield", O.Params(rho=(100.0,), beta=(100.0,)))
    g, o, t, _ = make_step([P, S, np.concatenate([S, T])])
    r = oc.step(1, g, o, t)
    assert r["status"] == 0
    assert r["admitted_blocks"].tolist() == [3, 1, 0]
    assert r["hit_blocks"].tolist() == [0, 0, 1]
    assert r["admitted_offsets"].tolist() == [0, 3, 4, 4]
    assert r["admitted_ids"].tolist() == [0, 1, 2, 3]
    assert _stat(oc, "ungranted_blocks") == 2 + 1 and _stat(oc, "instep_hit_blocks") == 1
