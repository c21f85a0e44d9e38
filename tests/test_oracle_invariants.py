"""Pins of the oracle against what the paper fixes.

* Invariants after every step of adversarial fuzz traces and of the tiny
  one-touch trace, for every policy (``_util.check_step``): I1 (Sec. III-A),
  work conservation (Sec. III-E), fixed ownership (Sec. II-C), debt >= 0, and
  the lru / prefixshield victim sets against an independent closed form.
* Proposition 1 (quiescent debt clearance), exactly at the predicted tick.
* I2 (no debt laundering through reuse, Eq. 4) and its release after clearance.
* Creation within the refill rate never accrues debt (Sec. V-D sweep, ratio < 1).
* Work-conserving borrowing: an idle peer leaves the whole pool to the active
  group (Sec. V-C).
* A batch of requests equals the same requests one per step (the batch
  reading of Alg. 1), when no block is reclaimed.
* Error handling leaves the state untouched.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_01657_gb300 import workloads as W
from _util import check_step, make_step, obj_tokens

POLICIES = ("lru", "s3fifo", "prefixshield")


def _run_checked(oc, steps, policy):
    for st in steps:
        before = oc.export()
        r = oc.step(st.now, st.groups, st.offsets, st.tokens, st.contracts, st.prefixes)
        after = oc.export()
        check_step(oc, before, after, (st.groups, st.offsets, st.tokens, st.now, st.contracts), r, policy)


@pytest.mark.parametrize("policy", POLICIES)
@pytest.mark.parametrize("seed,N,G,R", [(1, 24, 2, 3), (2, 40, 3, 6), (3, 64, 4, 8), (4, 12, 1, 2)])
def test_invariants_fuzz(policy, seed, N, G, R):
    steps = W.fuzz_steps(seed, G, R, 40, docs_per_group=3, doc_blocks=6, fresh_max_blocks=2)
    oc = O.OracleCache(N, 16, G, policy, O.Params(rho=(2.0,), beta=(6.0,)))
    _run_checked(oc, steps, policy)


@pytest.mark.parametrize("policy", POLICIES)
def test_invariants_fuzz_contracts_prefixes_flags(policy):
    steps = W.fuzz_steps(7, 3, 5, 40, docs_per_group=3, doc_blocks=6, with_contracts=3,
                         with_prefixes=True, now_stride=3, empty_every=7)
    for flags in (0, O.FLAG_NO_SEGMENTATION, O.FLAG_NO_DEBT_GATE):
        oc = O.OracleCache(30, 16, 3, policy,
                           O.Params(rho=(4.0, 2.5, 1.0), beta=(16.0, 12.0, 8.0), flags=flags,
                                    contract_of_group=[0, 1, 2]))
        _run_checked(oc, steps, policy)


@pytest.mark.parametrize("policy", POLICIES)
def test_invariants_tiny_one_touch(policy):
    wl = W.make_workload(0, seed=3)
    sp = wl.spec
    oc = O.OracleCache(sp.capacity_blocks, sp.block_size, sp.num_groups, policy, O.Params(rho=sp.rho, beta=sp.beta))
    _run_checked(oc, list(wl.steps(20)), policy)


@pytest.mark.parametrize("policy,contracts", [("prefixshield", 2), ("s3fifo", 0), ("lru", 2)])
def test_orphans_are_invalidated_not_evicted(policy, contracts):
    # A resident block whose parent was reclaimed cannot be reached by lookup;
    # a request that misses the parent drops it (invalidated, not evicted).
    # prefixshield: a request under another contract promotes only the blocks
    # whose (g, c, p) matches, so a child can outrank its parent.  S3-FIFO's
    # frequency rule reorders chains too.  Under lru a parent is always more
    # recent than its child, so orphans never occur.
    seen = 0
    steps = W.fuzz_steps(11, 2, 4, 120, docs_per_group=2, doc_blocks=8, fresh_max_blocks=1,
                         with_contracts=contracts)
    oc = O.OracleCache(20, 16, 2, policy, O.Params(rho=(1.0, 2.0), beta=(3.0, 3.0)))
    for st in steps:
        before = oc.export()
        r = oc.step(st.now, st.groups, st.offsets, st.tokens, st.contracts)
        check_step(oc, before, oc.export(), (st.groups, st.offsets, st.tokens, st.now, st.contracts), r, policy)
        seen += len(r["invalidated_ids"])
    assert (seen > 0) == (policy != "lru")
    assert oc.stats()[:, O.STAT_NAMES.index("invalidated_blocks")].sum() == seen


@pytest.mark.parametrize("rho_blocks,burst", [(3.0, 20), (2.5, 16), (0.75, 9)])
def test_proposition1_quiescent_clearance(rho_blocks, burst):
    beta = 4.0
    oc = O.OracleCache(256, 16, 1, "prefixshield", O.Params(rho=(rho_blocks,), beta=(beta,)))
    r = oc.step(1, *make_step([obj_tokens("burst", blocks=burst)])[:3])
    unit = 1 << 20
    d0 = (burst - int(beta)) * unit
    assert int(r["debt_raw"][0]) == d0
    rho = int(round(rho_blocks * unit))
    tau = -(-d0 // rho)  # ceil(d0 / rho): the first tick with zero debt
    for k in range(1, tau + 3):
        r = oc.step(1 + k, *make_step([])[:3])
        want = max(0, d0 - rho * k)
        assert int(r["debt_raw"][0]) == want
        assert (int(r["debt_raw"][0]) == 0) == (k >= tau)


def test_i2_gate_blocks_promotion_until_clearance():
    """An attacker admits a 10-block prefix with debt, replays it while in
    debt (all 10 eligible touches gated, none promoted), then replays after
    the designed clearance time (all 10 promoted)."""
    for flags, expect_early in ((0, (0, 10)), (O.FLAG_NO_DEBT_GATE, (10, 0))):
        oc = O.OracleCache(64, 16, 1, "prefixshield", O.Params(rho=(1.0,), beta=(2.0,), flags=flags))
        P = obj_tokens("attack", blocks=10)
        r = oc.step(1, *make_step([P])[:3])
        assert int(r["debt_raw"][0]) == 8 << 20
        r = oc.step(2, *make_step([P])[:3])   # replay in debt (7 blocks after refill)
        s = oc.stats()[0]
        assert (int(s[O.STAT_NAMES.index("promotions")]), int(s[O.STAT_NAMES.index("gated_reuses")])) == expect_early
        assert int(r["admitted_blocks"][0]) == 0 and int(r["hit_blocks"][0]) == 10  # replay charges 0
        assert int(r["debt_raw"][0]) == 7 << 20
        if flags == 0:
            assert set(oc.export()["klass"][:10].tolist()) == {0}
            r = oc.step(2 + 7, *make_step([P])[:3])  # exactly at clearance
            s = oc.stats()[0]
            assert int(r["debt_raw"][0]) == 0
            assert int(s[O.STAT_NAMES.index("promotions")]) == 10
            assert set(oc.export()["klass"][:10].tolist()) == {2}


def test_creation_within_refill_never_accrues_debt():
    oc = O.OracleCache(4096, 16, 1, "prefixshield", O.Params(rho=(5.0,), beta=(5.0,)))
    for t in range(1, 60):
        r = oc.step(t, *make_step([obj_tokens(f"fresh{t}", blocks=5)])[:3])
        assert int(r["debt_raw"][0]) == 0 and int(r["admitted_blocks"][0]) == 5
    r = oc.step(60, *make_step([obj_tokens("over", blocks=6)])[:3])
    assert int(r["debt_raw"][0]) == 1 << 20


@pytest.mark.parametrize("policy", POLICIES)
def test_work_conserving_borrowing(policy):
    # group 1 idle: group 0 alone may fill every block, and nothing is evicted
    # while free blocks remain.
    N = 64
    oc = O.OracleCache(N, 16, 2, policy, O.Params(rho=(1.0,), beta=(1.0,)))
    total = 0
    for t in range(1, 20):
        r = oc.step(t, *make_step([obj_tokens(f"b{t}", blocks=5)], [0])[:3])
        total += 5
        assert len(r["evicted_ids"]) == max(0, total - N) - max(0, total - 5 - N)
    s = oc.stats()
    assert s[0, O.STAT_NAMES.index("resident_blocks")] == N
    assert s[1, O.STAT_NAMES.index("resident_blocks")] == 0


def test_in_step_sharing_charges_once():
    oc = O.OracleCache(64, 16, 1, "prefixshield", O.Params(rho=(100.0,), beta=(100.0,)))
    P = obj_tokens("shared", blocks=4)
    Q = np.concatenate([P, obj_tokens("tail", blocks=2)])
    r = oc.step(1, *make_step([P, Q, P])[:3])
    assert list(r["admitted_blocks"]) == [4, 2, 0]
    assert list(r["hit_blocks"]) == [0, 4, 4]
    s = oc.stats()[0]
    assert s[O.STAT_NAMES.index("instep_hit_blocks")] == 8
    assert int(oc.export()["B"][0, 0]) == (100 - 6) << 20


def test_batch_equals_one_request_per_step_without_reclamation():
    steps = W.fuzz_steps(5, 2, 6, 6, docs_per_group=2, doc_blocks=5)
    prm = O.Params(rho=(3.0,), beta=(9.0,))
    batch = O.OracleCache(4096, 16, 2, "prefixshield", prm)
    seq = O.OracleCache(4096, 16, 2, "prefixshield", prm)
    for st in steps:
        rb = batch.step(st.now, st.groups, st.offsets, st.tokens)
        hits, adm = [], []
        for i in range(st.num_requests):
            o0, o1 = st.offsets[i], st.offsets[i + 1]
            r = seq.step(st.now, st.groups[i:i + 1], np.array([0, o1 - o0]), st.tokens[o0:o1])
            hits.append(int(r["hit_blocks"][0]))
            adm.append(int(r["admitted_blocks"][0]))
        assert list(rb["hit_blocks"]) == hits and list(rb["admitted_blocks"]) == adm
        a, b = batch.export(), seq.export()
        for k in ("resident", "key", "group", "contract", "prefix", "klass", "acc", "freq"):
            assert np.array_equal(a[k], b[k]), k
        assert np.array_equal(np.argsort(a["stamp"], kind="stable"), np.argsort(b["stamp"], kind="stable"))
        assert np.array_equal(a["B"], b["B"])
    # every counter agrees except the split of hits into in-step and resident
    keep = [k for k in range(13) if O.STAT_NAMES[k] != "instep_hit_blocks"]
    assert np.array_equal(batch.stats()[:, keep], seq.stats()[:, keep])


def test_errors_leave_state_unchanged():
    oc = O.OracleCache(32, 16, 2, "prefixshield", O.Params(rho=(1.0,), beta=(2.0,), history_capacity=3))
    oc.step(5, *make_step([obj_tokens("a", blocks=2)], [0])[:3])
    snap = oc.export()
    g, o, t, _ = make_step([obj_tokens("b", blocks=2)], [0])
    assert oc.step(4, g, o, t)["status"] == O.ERR_CLOCK
    assert oc.step(5, np.array([2], np.int32), o, t)["status"] == O.ERR_INVALID_ARG
    assert oc.step(5, g, np.array([1, 32]), t)["status"] == O.ERR_INVALID_ARG
    assert oc.step(5, g, np.array([0, 32]), t, contracts=np.array([1], np.int32))["status"] == O.ERR_INVALID_ARG
    assert oc.step(5, g, o, t, prefixes=np.array([0], np.uint64))["status"] == O.ERR_INVALID_ARG
    after = oc.export()
    for k in ("resident", "key", "stamp", "klass"):
        assert np.array_equal(snap[k], after[k])
    assert np.array_equal(snap["B"], after["B"]) and snap["step"] == after["step"]
    # history capacity: three prefixes fit, the fourth is a sticky capacity error
    prompts = [obj_tokens(x, blocks=1) for x in ("p", "q", "r")]
    assert oc.step(6, *make_step(prompts[:2], [0, 1])[:3])["status"] == 0
    assert oc.step(6, *make_step(prompts[2:], [1])[:3])["status"] == O.ERR_CAPACITY
    assert oc.step(7, *make_step([])[:3])["status"] == O.ERR_CAPACITY
    oc.clear_status()
    assert oc.step(7, *make_step([])[:3])["status"] == 0


def test_params_validation():
    L = O.lib()
    import ctypes as C
    good = O.Params(rho=(1.0, 2.0), beta=(1.0, 1.0)).to_c(4)
    assert L.orc_check_params(16, 16, 4, 2, C.byref(good)) == 0
    for mut in (dict(rho=(0.0,)), dict(beta=(-1.0,)), dict(s3_small_pct=0), dict(history_capacity=0),
                dict(rho=(1.0, 2.0 ** 21), beta=(1.0, 1.0))):
        kw = dict(rho=(1.0,), beta=(1.0,)); kw.update(mut)
        p = O.Params(**kw).to_c(4)
        assert L.orc_check_params(16, 16, 4, 2, C.byref(p)) == O.ERR_INVALID_ARG, mut
    assert L.orc_check_params(16, 15, 4, 2, C.byref(good)) == O.ERR_INVALID_ARG  # odd block size
