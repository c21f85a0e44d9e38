"""Exact pin of the orphan rule (Alg. 1 counts only the leading cached
prefix), derived by hand.

A resident key past a request's first miss cannot be reached by lookup: its
block is dropped, freed and reported as invalidated (not evicted), and the
key is materialized again as new.  The scenario below makes a chain with two
holes (a miss at h with resident keys at h + 1 and h + 3), a chain whose very
first block is missing (h = 0), and a later request of the same step that
contains one of those orphans again (reported once).  Its holes come from the
retention classes: blocks admitted under a prefix id that is later proven
and promoted to Reuse outlive their Probationary parents (Eq. 9 order).

No request of a step can pin an orphan: chained keys make a key at position
m resident-reachable only through its own prefix, so a request that hits it
would have hit the missing parent too.

Pool N = 11, block size 16, groups 0 and 1, rho = beta = 1000 blocks (nobody
is ever in debt, so reclamation is the global (class, stamp) fallback).
Chains in group 0: X = x0..x5, V = v0 v1; in group 1: Y = y0..y5.

  S1  [X0:3 p=1] [V0:1 p=21]   admit x0 x1 x2 v0 -> ids 0 1 2 3 (Probationary:
                               first admission of each prefix id)
  S2  [X0:4 p=2] [V0:2 p=22]   hit 3 / 1; admit x3 -> 4, v1 -> 5 (Prob)
  S3  [X0:5 p=3]               admit x4 -> 6 (Prob)
  S4  [X0:6 p=4]               admit x5 -> 7 (Prob)
  S5  [X0:4 p=2] [V0:2 p=22]   proven: x3 and v1 (their blocks carry p) -> Reuse
  S6  [X0:6 p=4]               proven: x5 -> Reuse; every x restamped, deeper
                               blocks older (x5 < x4 < ... < x0)
  S7  [Y0:6 group 1 p=31]      3 free ids (8 9 10), 3 victims: the three
                               smallest (class, stamp) = Probationary v0 (S5
                               stamp), then x4, x2 (S6) -> evicted 2 3 6;
                               allocated 2 3 6 8 9 10 -> y0..y5
  S8  rA [X0:6 p=4]  h = 2 (x2 gone): x3 (id 4) and x5 (id 7) are orphans
      rC [V0:2 p=22] h = 0 (v0 gone): v1 (id 5) is an orphan
      rD [X0:4 p=4]  h = 2: x3 again (one invalidation)
      invalidated 4 5 7; pins x0 x1, so avail = 11 - 2 = 9 and the claims
      rA 4 (x2..x5), rC 2, rD 0 (x2 x3 owned by rA) are all granted;
      free = 11 - 8 = 3 (ids 4 5 7), 3 victims: y5 y4 y3 (ids 10 9 8, the
      oldest of the Probationary y's); allocated 4 5 7 8 9 10 paired in
      (request, position) order: x2 x3 x4 x5 v0 v1; rD's x2 x3 are in-step
      hits (owner rA granted), so hits are 2, 0, 4.
"""
import numpy as np

import oracle as O
from _util import make_step, obj_tokens


def _chain(name, blocks):
    return obj_tokens(name, blocks=blocks)


def test_orphans_are_invalidated_exactly():
    X, V, Y = _chain("X", 6), _chain("V", 2), _chain("Y", 6)
    kw = dict(rho=(1000.0,), beta=(1000.0,))
    oc = O.OracleCache(11, 16, 2, "prefixshield", O.Params(**kw))

    def step(now, reqs):
        prompts = [t[: 16 * nb] for t, nb, _, _ in reqs]
        g, o, t, _ = make_step(prompts, [grp for _, _, grp, _ in reqs])
        p = np.array([pid for _, _, _, pid in reqs], np.uint64)
        r = oc.step(now, g, o, t, None, p)
        assert r["status"] == 0
        return r

    r = step(1, [(X, 3, 0, 1), (V, 1, 0, 21)])
    assert r["admitted_ids"].tolist() == [0, 1, 2, 3]
    r = step(2, [(X, 4, 0, 2), (V, 2, 0, 22)])
    assert r["hit_blocks"].tolist() == [3, 1] and r["admitted_ids"].tolist() == [4, 5]
    assert step(3, [(X, 5, 0, 3)])["admitted_ids"].tolist() == [6]
    assert step(4, [(X, 6, 0, 4)])["admitted_ids"].tolist() == [7]
    step(5, [(X, 4, 0, 2), (V, 2, 0, 22)])
    step(6, [(X, 6, 0, 4)])
    e = oc.export()
    assert e["klass"][[4, 5, 7]].tolist() == [2, 2, 2]          # x3, v1, x5: Reuse
    assert e["klass"][[0, 1, 2, 3, 6]].tolist() == [0] * 5       # x0 x1 x2 v0 x4: Probationary
    r = step(7, [(Y, 6, 1, 31)])
    assert r["evicted_ids"].tolist() == [2, 3, 6]
    assert r["admitted_ids"].tolist() == [2, 3, 6, 8, 9, 10]
    assert r["invalidated_ids"].tolist() == []
    before = oc.stats()
    r = step(8, [(X, 6, 0, 4), (V, 2, 0, 22), (X, 4, 0, 4)])
    assert r["invalidated_ids"].tolist() == [4, 5, 7]
    assert r["evicted_ids"].tolist() == [8, 9, 10]
    assert r["hit_blocks"].tolist() == [2, 0, 4]
    assert r["admitted_blocks"].tolist() == [4, 2, 0]
    assert r["admitted_ids"].tolist() == [4, 5, 7, 8, 9, 10]
    d = oc.stats() - before
    inv = O.STAT_NAMES.index("invalidated_blocks")
    ev = O.STAT_NAMES.index("evicted_blocks")
    res = O.STAT_NAMES.index("resident_blocks")
    assert d[:, inv].tolist() == [3, 0]
    assert d[:, ev].tolist() == [0, 3]
    assert d[:, res].tolist() == [6 - 3, -3]                    # group 0: -3 orphans +6 admitted
    e = oc.export()
    assert e["resident"].sum() == 11
    # the re-materialized x3 is a new block: admitted this step under p = 4
    assert e["prefix"][5] == 4 and e["key"][5] != 0
