"""The delayed-replay trace (the debt-gate ablation of Sec. V-D) on the oracle,
with the three contracts of Sec. V-A (critical 64/256, standard 40/192,
best-effort 16/128 blocks).

The trace's numbers follow from Eq. 1-3 and Alg. 1 by hand:
* the attacker's burst (tick 7) charges 192 blocks against a full 128-block
  bucket: 64 blocks of debt, repaid by refill 16 a tick, so the debt is
  64 - 16 k at tick 7 + k and zero from tick 11 on (Proposition 1);
* its replay touches 192 blocks that are proven (q = 1, admitted) and still
  Prob, so all 192 are gated while debt is outstanding (replay at tick 8,
  zero wait, or tick 9, half the designed wait) and all 192 are promoted
  without the gate, or with it at tick 11 (the designed clearance time);
* under the neutral pressure that follows, the gated attacker blocks stay
  in the first retention segment and are reclaimed before any of the
  victim's promoted blocks, while the ungated variant reclaims victim
  blocks; once the replay waits out the clearance time the two variants
  are the same cache.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_01657_gb300 import workloads as W

V, A, NEU = W.DelayedReplay.VICTIM, W.DelayedReplay.ATTACKER, W.DelayedReplay.NEUTRAL
PROB, REUSE = 0, 2
FP = 1 << 20


def _run(wait, flags):
    wl = W.make_workload(6, seed=5, wait=wait)
    sp = wl.spec
    orc = O.OracleCache(sp.capacity_blocks, sp.block_size, sp.num_groups, "prefixshield",
                        O.Params(rho=sp.rho, beta=sp.beta, contract_of_group=list(sp.contract_of_group),
                                 flags=flags))
    out = dict(steps=[], evicted_groups=[], victim_hits=[], debt=[])
    for st in wl.steps():
        before = orc.export()
        s0 = orc.stats()
        r = orc.step(st.now, st.groups, st.offsets, st.tokens)
        assert r["status"] == 0
        d = orc.stats() - s0
        out["steps"].append((st, r, d))
        out["evicted_groups"].append(before["group"][r["evicted_ids"]])
        out["debt"].append(int(r["debt_raw"][A]))
        if st.index > wl.replay_step:
            out["victim_hits"].append(int(r["hit_blocks"][1]))
        if st.index == wl.replay_step:
            out["replay"] = (d, orc.export())
    out["wl"] = wl
    out["final"] = orc.export()
    return out


def test_trace_shape():
    wl = W.make_workload(6, seed=5, wait=1)
    steps = list(wl.steps())
    assert len(steps) == wl.num_steps == 13
    assert [s.now for s in steps] == list(range(1, 14))
    burst = steps[W.DelayedReplay.BURST_STEP]
    assert burst.groups.tolist() == [A, A] and burst.num_tokens == 2 * 1536
    assert steps[7].num_requests == 0
    replay = steps[wl.replay_step]
    assert np.array_equal(replay.tokens, burst.tokens)


@pytest.mark.parametrize("wait", [0, 1, 3])
def test_debt_follows_proposition_1(wait):
    r = _run(wait, 0)
    wl = r["wl"]
    for st, res, _ in r["steps"][W.DelayedReplay.BURST_STEP:wl.replay_step + 1]:
        k = st.now - 7
        assert int(res["debt_raw"][A]) == max(0, 64 - 16 * k) * FP, f"tick {st.now}"
    # the victim's three 96-block admissions stay inside its 256-block bucket
    for st, res, _ in r["steps"][:6]:
        assert int(res["debt_raw"][V]) == 0


@pytest.mark.parametrize("wait", [0, 1])
def test_gate_holds_every_eligible_block_while_in_debt(wait):
    gated = _run(wait, 0)
    d, e = gated["replay"]
    assert (int(d[A, O.STAT_NAMES.index("promotions")]), int(d[A, O.STAT_NAMES.index("gated_reuses")])) == (0, 192)
    assert int(d[A, O.STAT_NAMES.index("hit_blocks")]) == 192 and int(d[A, O.STAT_NAMES.index("admitted_blocks")]) == 0
    atk = (e["resident"] == 1) & (e["group"] == A)
    assert atk.sum() == 192 and set(e["klass"][atk].tolist()) == {PROB}

    ungated = _run(wait, O.FLAG_NO_DEBT_GATE)
    d, e = ungated["replay"]
    assert (int(d[A, O.STAT_NAMES.index("promotions")]), int(d[A, O.STAT_NAMES.index("gated_reuses")])) == (192, 0)
    atk = (e["resident"] == 1) & (e["group"] == A)
    assert set(e["klass"][atk].tolist()) == {REUSE}
    # the accounting is the same: the gate changes only the class
    assert [x for x in gated["debt"][:ungated["wl"].replay_step + 1]] == \
        [x for x in ungated["debt"][:ungated["wl"].replay_step + 1]]


@pytest.mark.parametrize("wait", [0, 1])
def test_pressure_reclaims_the_attacker_not_the_victim(wait):
    gated, ungated = _run(wait, 0), _run(wait, O.FLAG_NO_DEBT_GATE)
    p0 = gated["wl"].replay_step + 1
    # first pressure step: the same demand either way (96 new neutral blocks,
    # the victim's prefix still whole), 511 - 480 = 31 free, so 65 victims
    first_g, first_u = gated["evicted_groups"][p0], ungated["evicted_groups"][p0]
    assert len(first_g) == len(first_u) == 65
    assert (first_g == A).all()
    # ungated: Alg. 2 takes the attacker's projected debt first (its rate is
    # the smallest, so one block repays one block of debt: x = 64 - 16 k at
    # tick 7 + k), then the global (class, recency) order, where the
    # victim's promoted blocks are older than the attacker's promoted ones
    x_att = 64 - 16 * (9 + wait - 7)
    assert (int((first_u == A).sum()), int((first_u == V).sum())) == (x_att, 65 - x_att)
    ev_g = np.concatenate(gated["evicted_groups"][p0:])
    ev_u = np.concatenate(ungated["evicted_groups"][p0:])
    assert int((ev_g == V).sum()) == 0
    assert int((ev_g == A).sum()) > int((ev_u == A).sum())
    # the victim keeps every hot prefix under the gate and loses some without it
    assert gated["victim_hits"] == [96] * len(gated["victim_hits"])
    assert sum(ungated["victim_hits"]) < sum(gated["victim_hits"])


def test_variants_converge_at_the_designed_clearance_time():
    gated, ungated = _run(3, 0), _run(3, O.FLAG_NO_DEBT_GATE)
    d, _ = gated["replay"]
    assert int(d[A, O.STAT_NAMES.index("promotions")]) == 192 and int(d[A, O.STAT_NAMES.index("gated_reuses")]) == 0
    for (st, rg, _), (_, ru, _) in zip(gated["steps"], ungated["steps"]):
        for k in rg:
            if isinstance(rg[k], np.ndarray):
                assert np.array_equal(rg[k], ru[k]), f"step {st.index}: {k}"
    for k in gated["final"]:
        assert np.array_equal(gated["final"][k], ungated["final"][k]), k
