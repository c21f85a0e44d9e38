"""Pins of the oracle's StaticQuota baseline (Sec. V-A): a fixed, equal
partition of the pool per group (Q = floor(N / G) blocks) with no
cross-group borrowing; inside its partition a group reclaims its own least
recently released blocks.

* G = 1: one partition of the whole pool, i.e. exactly the LRU policy.
* One single-block request per step: per-group textbook LRU of capacity Q
  (collections.OrderedDict per group).
* The borrowing trace (Table III): with one group idle, the active group
  holds at most Q = 255 of 511 blocks, while lru and prefixshield borrow
  the whole pool.
* Invariants after every step of fuzz traces: no group above its quota,
  evictions only from a group whose new blocks overflow its free share, and
  those evictions are its oldest unpinned blocks.
"""
from collections import OrderedDict

import numpy as np
import pytest

import oracle as O
from paper_2608_01657_gb300 import workloads as W
from _util import obj_tokens, make_step


def _params(**kw):
    base = dict(rho=(2.0,), beta=(6.0,))
    base.update(kw)
    return O.Params(**base)


def _same(a, b, label):
    for k in a:
        if isinstance(a[k], np.ndarray):
            assert np.array_equal(a[k], b[k]), f"{label}: {k} differs"
        else:
            assert a[k] == b[k], f"{label}: {k} differs"


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_one_group_is_lru(seed):
    steps = W.fuzz_steps(seed, 1, 4, 40, docs_per_group=4, doc_blocks=6, fresh_max_blocks=3)
    q = O.OracleCache(24, 16, 1, "staticquota", _params())
    l = O.OracleCache(24, 16, 1, "lru", _params())
    for k, st in enumerate(steps):
        _same(q.step(st.now, st.groups, st.offsets, st.tokens), l.step(st.now, st.groups, st.offsets, st.tokens),
              f"step {k}")
    assert np.array_equal(q.stats(), l.stats())


@pytest.mark.parametrize("N,G", [(6, 2), (9, 3), (7, 2)])
def test_single_block_requests_are_per_group_lru(N, G):
    Q = N // G
    rng = np.random.default_rng(N * 10 + G)
    orc = O.OracleCache(N, 16, G, "staticquota", _params())
    ref = [OrderedDict() for _ in range(G)]
    for t in range(300):
        g = int(rng.integers(G))
        sym = f"g{g}-{int(rng.integers(Q + 3))}"
        grp, offs, toks, _ = make_step([obj_tokens(sym)], groups=[g])
        res = orc.step(t, grp, offs, toks)
        hit = sym in ref[g]
        if hit:
            ref[g].move_to_end(sym)
        else:
            evicted = len(ref[g]) == Q
            if evicted:
                ref[g].popitem(last=False)
            ref[g][sym] = True
            assert len(res["evicted_ids"]) == int(evicted), f"t={t}"
        assert int(res["hit_blocks"][0]) == int(hit), f"t={t}"
    e = orc.export()
    for g in range(G):
        assert int(((e["resident"] == 1) & (e["group"] == g)).sum()) == len(ref[g])


def test_borrowing_trace_is_capped_at_one_share():
    """Table III: the active borrower holds one equal share under StaticQuota
    and the whole pool under the work-conserving policies."""
    N, G = 511, 2
    peak = {}
    for policy in ("staticquota", "lru", "prefixshield"):
        orc = O.OracleCache(N, 16, G, policy, _params(rho=(64.0,), beta=(4096.0,)))
        occ = []
        for t in range(40):
            prompts = [obj_tokens(f"borrow-{t}-{j}", blocks=4) for j in range(8)]
            grp, offs, toks, _ = make_step(prompts, groups=[0] * 8)
            assert orc.step(t, grp, offs, toks)["status"] == 0
            e = orc.export()
            occ.append(int(((e["resident"] == 1) & (e["group"] == 0)).sum()))
        peak[policy] = max(occ)
    assert peak["staticquota"] == N // G
    assert peak["lru"] == N and peak["prefixshield"] == N


@pytest.mark.parametrize("seed,N,G", [(4, 30, 3), (5, 40, 2), (6, 17, 4)])
def test_quota_invariants_on_fuzz(seed, N, G):
    Q = N // G
    steps = W.fuzz_steps(seed, G, 5, 60, docs_per_group=3, doc_blocks=6, fresh_max_blocks=3, empty_every=11)
    orc = O.OracleCache(N, 16, G, "staticquota", _params())
    for k, st in enumerate(steps):
        before = orc.export()
        s0 = orc.stats()
        res = orc.step(st.now, st.groups, st.offsets, st.tokens)
        assert res["status"] == 0
        after = orc.export()
        d = orc.stats() - s0
        res_g = [int(((after["resident"] == 1) & (after["group"] == g)).sum()) for g in range(G)]
        assert max(res_g) <= Q, f"step {k}: a group holds more than its quota"
        ev = res["evicted_ids"]
        # a group evicts exactly what its new blocks overflow: admitted minus
        # the free part of its partition (after its invalidations)
        for g in range(G):
            held = int(((before["resident"] == 1) & (before["group"] == g)).sum()) - int(d[g, 9])
            want = max(0, int(d[g, 6]) - (Q - held))
            assert int(d[g, 8]) == want, f"step {k} group {g}: {int(d[g, 8])} evicted, {want} overflow"
        ev = res["evicted_ids"]
        if len(ev) == 0:
            continue
        # groups whose blocks were evicted, and how many each
        egroups, counts = np.unique(before["group"][ev], return_counts=True)
        # blocks hit in the step are pinned: same content, stamp moved to this
        # step (a reclaimed id holds other content afterwards)
        touched = (after["key"] == before["key"]) & (after["stamp"] != before["stamp"])
        for g, cnt in zip(egroups, counts):
            cand = np.where((before["resident"] == 1) & (before["group"] == g) & ~touched)[0]
            cand = cand[~np.isin(cand, res["invalidated_ids"])]
            oldest = cand[np.argsort(before["stamp"][cand], kind="stable")][:cnt]
            assert set(oldest.tolist()) == set(ev[before["group"][ev] == g].tolist()), f"step {k} group {g}"
