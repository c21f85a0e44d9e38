"""Pins of the S3-FIFO batch closed form (``_s3fifo_closed_form.s3_batch``),
the arithmetic the CUDA library's parallel S3-FIFO kernels implement:

* against the oracle, step by step: from the oracle's state before a step and
  the step's pinned blocks and victim count, the closed form must predict the
  oracle's victims, every surviving block's queue, sequence number and
  frequency, the ghost's entries and counters, and both queues' order after
  the step;
* against the published loop on random small instances, ties, pins and
  every parameter corner included.
"""
import random

import numpy as np
import pytest

import oracle as O
from paper_2608_01657_gb300 import workloads as W
from _s3fifo_closed_form import s3_batch, s3_loop
from _util import chain_keys_of


def _pinned(oc, before, st):
    keys = chain_keys_of(oc.params.hash_seed, (st.groups, st.offsets, st.tokens), oc.bs)
    where = {(int(before["group"][b]), int(before["key"][b])): b for b in range(oc.N) if before["resident"][b]}
    pinned = set()
    for i, g in enumerate(st.groups):
        for key in keys[i]:
            b = where.get((int(g), int(key)))
            if b is None:
                break
            pinned.add(b)
    return pinned


def _check_trace(N, G, steps, params):
    orc = O.OracleCache(N, 16, G, "s3fifo", params)
    cap, mm = params.s3_freq_cap, params.s3_move_min_freq
    S_cap = max(1, N * params.s3_small_pct // 100)
    ghost_cap = N - S_cap
    applied = 0
    for k, st in enumerate(steps):
        before = orc.export()
        res = orc.step(st.now, st.groups, st.offsets, st.tokens, st.contracts, st.prefixes)
        assert res["status"] == 0
        after = orc.export()
        pinned = _pinned(orc, before, st)
        inval = set(res["invalidated_ids"].tolist())
        live = [b for b in range(N) if before["resident"][b] and b not in inval]
        S = sorted((b for b in live if before["s3q"][b] == 0), key=lambda b: before["s3seq"][b])
        M = sorted((b for b in live if before["s3q"][b] == 1), key=lambda b: before["s3seq"][b])
        f = {b: min(int(before["freq"][b]), cap) for b in live}
        E = res["evicted_ids"].tolist()
        out = s3_batch(S, M, f, pinned, len(E), cap, mm, S_cap, before["s3_ctr"])
        if out is None:
            continue
        applied += 1
        assert out["victims"] == set(E), f"step {k}: victims"
        # ghost: the small-queue victims' keys pushed in order, the oldest trimmed
        ghost = {(int(g), int(key)): int(q) for g, key, q in zip(*before["ghost"])}
        gctr = before["ghost_ctr"]
        for b in out["small_victims"]:
            gctr += 1
            ghost[(int(before["group"][b]), int(before["key"][b]))] = gctr
        for key in sorted(ghost, key=ghost.get)[: max(0, len(ghost) - ghost_cap)]:
            del ghost[key]
        # insertions in rank order: a ghost hit enters the main queue
        ctr = out["ctr_end"]
        ins = {0: [], 1: []}
        for b in res["admitted_ids"].tolist():
            key = (int(after["group"][b]), int(after["key"][b]))
            ctr += 1
            q = 1 if key in ghost else 0
            ghost.pop(key, None)
            ins[q].append(b)
            assert after["s3q"][b] == q and after["s3seq"][b] == ctr, f"step {k}: inserted block {b}"
        assert after["s3_ctr"] == ctr and after["ghost_ctr"] == gctr, f"step {k}: counters"
        assert {(int(g), int(key)): int(q) for g, key, q in zip(*after["ghost"])} == ghost, f"step {k}: ghost"
        for b in live:
            if b in out["victims"]:
                continue
            want_seq = out["seq"].get(b, before["s3seq"][b])
            assert after["s3seq"][b] == want_seq, f"step {k}: sequence number of {b}"
            assert after["s3q"][b] == (1 if b in out["seq"] else before["s3q"][b]), f"step {k}: queue of {b}"
            if b in out["freq"]:
                assert after["freq"][b] == out["freq"][b], f"step {k}: frequency of {b}"
            elif b not in pinned:
                assert after["freq"][b] == before["freq"][b], f"step {k}: frequency of {b}"
        res_after = [b for b in range(N) if after["resident"][b]]
        for q, want in ((0, out["new_small"] + ins[0]), (1, out["new_main"] + ins[1])):
            got = sorted((b for b in res_after if after["s3q"][b] == q), key=lambda b: after["s3seq"][b])
            assert got == want, f"step {k}: order of queue {q}"
    return applied


# min_applied: steps (of 60) the closed form must cover.  A small queue of
# 100% leaves the main queue mostly empty, where the sequential loop applies.
@pytest.mark.parametrize("seed,N,G,R,pct,cap,mm,min_applied", [
    (1, 24, 2, 3, 10, 3, 2, 50), (2, 40, 3, 6, 10, 3, 2, 50), (3, 64, 4, 8, 10, 3, 2, 50),
    (4, 12, 1, 2, 10, 3, 2, 50), (5, 30, 3, 5, 50, 3, 2, 30), (6, 30, 3, 5, 10, 3, 1, 50),
    (7, 48, 3, 6, 10, 5, 3, 50), (8, 48, 3, 6, 100, 3, 2, 5),
])
def test_closed_form_matches_the_oracle_step_by_step(seed, N, G, R, pct, cap, mm, min_applied):
    steps = W.fuzz_steps(seed, G, R, 60, docs_per_group=3, doc_blocks=7, fresh_max_blocks=2,
                         now_stride=2, empty_every=9)
    params = O.Params(rho=(2.0,), beta=(6.0,), s3_small_pct=pct, s3_freq_cap=cap, s3_move_min_freq=mm)
    assert _check_trace(N, G, steps, params) >= min_applied


def test_closed_form_matches_the_oracle_on_a_configured_workload():
    wl = W.make_workload(5, seed=2)
    sp = wl.spec
    params = O.Params(rho=sp.rho, beta=sp.beta)
    assert _check_trace(sp.capacity_blocks, sp.num_groups, list(wl.steps(40)), params) >= 40


def test_closed_form_matches_the_loop_on_random_instances():
    rnd = random.Random(7)
    applied = 0
    for _ in range(20000):
        nS, nM = rnd.randint(0, 12), rnd.randint(0, 12)
        ids = list(range(nS + nM))
        rnd.shuffle(ids)
        S, M = ids[:nS], ids[nS:]
        cap = rnd.choice([1, 2, 3, 3, 3, 5, 15])
        mm = rnd.randint(1, cap + 1)
        f = {b: rnd.randint(0, cap) for b in ids}
        pinned = {b for b in ids if rnd.random() < rnd.choice([0, 0.2, 0.5])}
        m = rnd.randint(0, len(ids) - len(pinned))
        S_cap, ctr0 = rnd.randint(1, 10), rnd.randint(0, 100)
        out = s3_batch(S, M, f, pinned, m, cap, mm, S_cap, ctr0)
        if out is None:
            continue
        applied += 1
        V, small_v, seq, f2, ctr = s3_loop(S, M, f, pinned, m, cap, mm, S_cap, ctr0)
        assert out["victims"] == V and out["small_victims"] == small_v and out["ctr_end"] == ctr
        for b in ids:
            if b not in V:
                assert out["seq"].get(b) == seq.get(b)
                assert out["freq"].get(b, f[b]) == f2[b]
        moved = sorted((b for b in seq if b not in V), key=seq.get)
        assert out["new_main"][len(out["new_main"]) - len(moved):] == moved
    assert applied > 15000


def test_closed_form_hand_example():
    """Small queue [a, b, c, d] (f = 0, 2, 0, 1, capacity 2, threshold 2), main
    [x, y] (f = 1, 0), m = 3, counter 10.  D = 4 - 2 = 2: eviction 1 pops a
    (victim); eviction 2 starts after 1 pop (<= D), pops b (moved, seq 11) and
    c (victim); eviction 3 starts after 3 pops (> D): main phase over
    [x, y, b] with f = (1, 0, 2): round 0 visits x (reinserted, f 0, seq 12),
    y (victim).  So victims a, c, y; the main queue is [b, x] by sequence."""
    f = {"a": 0, "b": 2, "c": 0, "d": 1, "x": 1, "y": 0}
    out = s3_batch(["a", "b", "c", "d"], ["x", "y"], f, set(), 3, 3, 2, 2, 10)
    assert out["victims"] == {"a", "c", "y"} and out["small_victims"] == ["a", "c"]
    assert out["seq"] == {"b": 11, "x": 12} and out["freq"] == {"x": 0}
    assert out["new_small"] == ["d"] and out["new_main"] == ["b", "x"] and out["ctr_end"] == 12
