"""Pins of the oracle's replacement policies.

* LRU: hand-traced golden trace, and reduction to textbook LRU
  (collections.OrderedDict) when every step carries one single-block request.
* S3-FIFO: hand-traced golden trace of the published algorithm under the
  readings of its batch form stated in the trace file's header.
* PrefixShield: a hand-derived Alg. 2 example where debt directs reclamation
  to the indebted group even though its blocks are newer (Eq. 6-8).
* Chain release order: a request releases its blocks tail first.
"""
from collections import OrderedDict

import numpy as np
import pytest

import oracle as O
from _util import make_step, obj_tokens, params_line, parse_trace

BIG = dict(rho=(1000.0,), beta=(1000.0,))


def _keymap(oc, names):
    seed = oc.params.hash_seed
    return {int(O.chain_keys(seed, 0, oc.bs, obj_tokens(n, oc.bs))[0]): n for n in names}


def _run_trace(policy, fname, extra):
    steps, final = parse_trace(fname)
    pr = params_line(fname)
    names = sorted({n for reqs, _, _ in steps for n in reqs})
    oc = O.OracleCache(pr["N"], 16, 1, policy, O.Params(**BIG, **extra))
    k2n = _keymap(oc, names)
    for si, (reqs, hits, ev) in enumerate(steps):
        before = oc.export()
        g, o, t, _ = make_step([obj_tokens(n) for n in reqs])
        r = oc.step(si + 1, g, o, t)
        assert r["status"] == 0
        assert list(r["hit_blocks"]) == hits, f"step {si + 1}"
        got = sorted(k2n[int(before["key"][b])] for b in r["evicted_ids"])
        assert got == sorted(ev), f"step {si + 1}: evicted {got}, want {ev}"
    return oc, k2n, final


def test_lru_hand_trace():
    oc, k2n, final = _run_trace("lru", "lru_hand_trace.txt", {})
    st = oc.export()
    res = sorted(k2n[int(k)] for k, r in zip(st["key"], st["resident"]) if r)
    assert res == sorted(final["final resident"])


def test_s3fifo_hand_trace():
    pr = params_line("s3fifo_hand_trace.txt")
    oc, k2n, final = _run_trace("s3fifo", "s3fifo_hand_trace.txt",
                                dict(s3_small_pct=pr["small_pct"], s3_freq_cap=pr["freq_cap"],
                                     s3_move_min_freq=pr["move_min_freq"]))
    st = oc.export()
    res = [(int(st["s3seq"][b]), k2n[int(st["key"][b])], int(st["s3q"][b]), int(st["freq"][b]))
           for b in range(oc.N) if st["resident"][b]]
    res.sort()
    small = [f"{n}:{f}" for _, n, q, f in res if q == 0]
    main = [f"{n}:{f}" for _, n, q, f in res if q == 1]
    assert small == final["final small"]
    assert main == final["final main"]
    gg, gk, gs = st["ghost"]
    ghost = [k2n[int(k)] for _, k in sorted(zip(gs, gk))]
    assert ghost == final["final ghost"]


@pytest.mark.parametrize("N,seed", [(3, 0), (5, 1), (8, 2)])
def test_lru_reduces_to_textbook_lru(N, seed):
    rng = np.random.default_rng(seed)
    names = [f"o{i}" for i in range(2 * N + 2)]
    oc = O.OracleCache(N, 16, 1, "lru", O.Params(**BIG))
    k2n = _keymap(oc, names)
    ref = OrderedDict()
    for s in range(300):
        x = names[int(rng.integers(0, len(names)))]
        before = oc.export()
        g, o, t, _ = make_step([obj_tokens(x)])
        r = oc.step(s + 1, g, o, t)
        hit = x in ref
        ev = []
        if hit:
            ref.move_to_end(x)
        else:
            if len(ref) == N:
                ev.append(ref.popitem(last=False)[0])
            ref[x] = True
        assert int(r["hit_blocks"][0]) == int(hit)
        assert [k2n[int(before["key"][b])] for b in r["evicted_ids"]] == ev


def test_lru_releases_a_chain_tail_first():
    # A 3-block prompt admitted on an empty pool, then a new 1-block prompt:
    # the deepest block of the chain is the least recently released.
    oc = O.OracleCache(3, 16, 1, "lru", O.Params(**BIG))
    p = obj_tokens("P", blocks=3)
    g, o, t, _ = make_step([p])
    r1 = oc.step(1, g, o, t)
    assert list(r1["admitted_ids"]) == [0, 1, 2]  # position order, ascending ids
    g, o, t, _ = make_step([obj_tokens("Q")])
    r2 = oc.step(2, g, o, t)
    assert list(r2["evicted_ids"]) == [2]


def test_prefixshield_hand_example_directs_reclamation_to_debt():
    """Two groups, N = 4, rho = 1 block/tick, beta = 2 blocks.

    t=1  victim (g0) admits V = [v0 v1] into ids 0,1: balance 2-2 = 0, first
         admission -> Probationary.
    t=2  victim replays V: q=1, admitted, D_g0 = 0 after refill -> both
         promoted to Reuse, stamps refreshed (v1 older: released first).
    t=3  attacker (g1) admits A = [a0 a1] into ids 2,3: balance 0, Prob.
    t=3  attacker sends 3 fresh blocks; the pool is full, so 3 victims.
         Charge: B_g1 = 0 - 3 -> D~_g1 = 3 blocks, delta = 1 block (Eq. 8).
         Alg. 2: g1 is the only indebted candidate owner: a1 (P 3->2),
         a0 (P 2->1); g1 has no candidates left, so the global fallback takes
         the oldest Reuse block, v1.  Evicted ids {1, 2, 3}; under LRU the
         three oldest stamps v1, v0, a1 -> ids {0, 1, 3}.
    """
    want = {"prefixshield": [1, 2, 3], "lru": [0, 1, 3]}
    for pol, ev in want.items():
        oc = O.OracleCache(4, 16, 2, pol, O.Params(rho=(1.0,), beta=(2.0,)))
        V = obj_tokens("V", blocks=2)
        A = obj_tokens("A", blocks=2)
        F = obj_tokens("F", blocks=3)
        r = oc.step(1, *make_step([V], [0])[:3]); assert list(r["admitted_ids"]) == [0, 1]
        r = oc.step(2, *make_step([V], [0])[:3]); assert list(r["hit_blocks"]) == [2]
        st = oc.export(); assert list(st["klass"][:2]) == [2, 2]
        r = oc.step(3, *make_step([A], [1])[:3]); assert list(r["admitted_ids"]) == [2, 3]
        r = oc.step(3, *make_step([F], [1])[:3])
        assert list(r["evicted_ids"]) == ev, pol
        assert list(r["admitted_ids"]) == [1, 2, 3] if pol == "prefixshield" else [0, 1, 3]
        assert int(r["debt_raw"][1]) == 3 << 20 and int(r["debt_raw"][0]) == 0
        assert int(r["debt_norm"][1]) == 3 << 20


def test_no_segmentation_flag_uses_recency_inside_the_group():
    """Same as above but with a Reuse block in the indebted group: with
    segmentation the group's Prob block goes first; without, the older one."""
    for flags, want in ((0, "new"), (O.FLAG_NO_SEGMENTATION, "old")):
        oc = O.OracleCache(3, 16, 1, "prefixshield", O.Params(rho=(1.0,), beta=(1.0,), flags=flags))
        X = obj_tokens("X")  # 1 block, admitted t=1 (Prob), promoted t=2 (Reuse)
        Y = obj_tokens("Y")
        oc.step(1, *make_step([X])[:3])
        oc.step(2, *make_step([X])[:3])
        assert oc.export()["klass"][0] == 2
        oc.step(2, *make_step([Y])[:3])                      # id 1, Prob, balance -> -1
        oc.step(2, *make_step([obj_tokens("Z")])[:3])        # id 2, Prob, balance -> -2
        r = oc.step(2, *make_step([obj_tokens("W")])[:3])    # one victim from g0 (in debt)
        # segmented: Prob first -> the older Prob block Y (id 1); unsegmented:
        # plain recency -> X (id 0, stamped at t=2 before Y and Z)
        assert list(r["evicted_ids"]) == ([1] if want == "new" else [0])


def test_normalized_debt_and_decrements_with_three_contracts():
    """Eq. 5 and Eq. 8 with the paper's three contract tiers (rho 64, 40, 16
    blocks a tick, beta 256, 192, 128), hand-derived in fixed point.

    Tick 1: group A (contract rho 40) admits 217 blocks: B = 192 - 217 = -25;
    group B (contract rho 16 = rho_min) admits 134: B = -6.  Eq. 5:
      D~_A = floor(25 * 2^20 * 16 / 40) = 10 * 2^20,   D~_B = 6 * 2^20.
    Eq. 8 (rho_max over the indebted contracts of each group):
      delta_A = floor(2^20 * 16 / 40) = 419430,        delta_B = 2^20.
    The pool (351 blocks) is then full.  Still at tick 1 (no refill), group C
    (contract rho 64, no debt) admits 20 fresh blocks: 20 victims.  Alg. 2
    takes the larger projected score each time: A while 10485760 - k*419430
    exceeds 6291456 (k = 0..10: 11 victims, the last at 6291460), then B,
    A, A, B, A, A, A (4194310 > 4194304), B, A: 17 from A and 3 from B.
    Raw instead of normalized debt, or the ratio inverted, changes the split.
    """
    prm = O.Params(rho=(64.0, 40.0, 16.0), beta=(256.0, 192.0, 128.0), contract_of_group=[1, 2, 0])
    oc = O.OracleCache(351, 16, 3, "prefixshield", prm)
    g, o, t, _ = make_step([obj_tokens("A", blocks=217), obj_tokens("B", blocks=134)], [0, 1])
    r = oc.step(1, g, o, t)
    assert r["status"] == 0 and list(r["admitted_blocks"]) == [217, 134]
    assert [int(x) for x in r["debt_raw"]] == [25 << 20, 6 << 20, 0]
    assert [int(x) for x in r["debt_norm"]] == [10 << 20, 6 << 20, 0]
    before = oc.export()
    g, o, t, _ = make_step([obj_tokens("C", blocks=20)], [2])
    r = oc.step(1, g, o, t)
    assert r["status"] == 0 and int(r["admitted_blocks"][0]) == 20
    owners = before["group"][r["evicted_ids"]]
    assert (int((owners == 0).sum()), int((owners == 1).sum()), int((owners == 2).sum())) == (17, 3, 0)


def test_gate_reads_debt_before_the_request_charge_class_after():
    """Reading A14 (OnRequest, OnTouch, OnCacheFullBlocks in that order),
    derived by hand.  beta = 4, rho = 1, all at tick 1 (no refill):
      step 1: P (2 blocks) admitted: B = 2, class Prob (first admission);
      step 2: P + X (X = 3 new blocks): P is proven (q = 1, admitted) and the
        gate reads D before this request's charge (0): both P blocks are
        promoted.  Then the charge: B = 2 - 3 = -1, so X's blocks are Prob
        (B < -eps) and the raw debt is 1 block.
    A gate that read the debt after the charge would hold P back; a class
    taken from the balance before the charge would make X Normal."""
    oc = O.OracleCache(64, 16, 1, "prefixshield", O.Params(rho=(1.0,), beta=(4.0,)))
    P, X = obj_tokens("P", blocks=2), obj_tokens("X", blocks=3)
    r = oc.step(1, *make_step([P])[:3])
    assert r["admitted_ids"].tolist() == [0, 1]
    r = oc.step(1, *make_step([np.concatenate([P, X])])[:3])
    assert r["hit_blocks"].tolist() == [2] and r["admitted_blocks"].tolist() == [3]
    s = oc.stats()[0]
    assert (int(s[O.STAT_NAMES.index("promotions")]), int(s[O.STAT_NAMES.index("gated_reuses")])) == (2, 0)
    e = oc.export()
    assert e["klass"][:2].tolist() == [2, 2]      # P: Reuse
    assert e["klass"][2:5].tolist() == [0, 0, 0]  # X: Probationary
    assert int(r["debt_raw"][0]) == 1 << 20


def test_history_includes_earlier_requests_of_the_same_step():
    """Reading A13, derived by hand: one step, r0 = P (2 new blocks, first
    admission: Prob, B = 4 - 2 = 2), then r1 = P: its two keys are r0's
    granted claims (in-step hits).  r1's q counts r0's request (q = 1) and
    P counts as admitted by r0, so r1's touch is proven; the gate reads
    D = 0 and both new blocks are promoted: they enter the pool as Reuse."""
    oc = O.OracleCache(64, 16, 1, "prefixshield", O.Params(rho=(1.0,), beta=(4.0,)))
    P = obj_tokens("P", blocks=2)
    r = oc.step(1, *make_step([P, P])[:3])
    assert r["hit_blocks"].tolist() == [0, 2] and r["admitted_blocks"].tolist() == [2, 0]
    s = oc.stats()[0]
    assert int(s[O.STAT_NAMES.index("instep_hit_blocks")]) == 2
    assert (int(s[O.STAT_NAMES.index("promotions")]), int(s[O.STAT_NAMES.index("gated_reuses")])) == (2, 0)
    assert oc.export()["klass"][:2].tolist() == [2, 2]
    assert int(r["debt_raw"][0]) == 0
