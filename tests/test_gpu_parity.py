"""GPU-vs-oracle parity of the prefix-cache step, through the C ABI.

The CUDA library and the CPU oracle run the same seeded steps; every output
(hit and admitted counts, CSR offsets, admitted / evicted / invalidated ids,
raw and normalized debt) must match bit for bit after every step, and so must
the exported policy state (per-block key, owner, contract, prefix id, class,
recency stamp, access count, frequency; balances; clock; history) and the
per-group statistics.  Everything here is integer or fixed-point arithmetic,
so the tolerance is zero.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_01657_gb300 import workloads as W
from _util import compare_outputs, compare_state

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _pair(N, bs, G, policy, params_kw, max_requests, max_tokens):
    from paper_2608_01657_gb300 import binding as B
    gpu = B.Cache(N, bs, G, policy, B.Params(**params_kw), max_requests=max_requests, max_tokens=max_tokens)
    orc = O.OracleCache(N, bs, G, policy, O.Params(**params_kw))
    return gpu, orc


def _run(gpu, orc, steps, state_every=1, s3=False, label="", graph=True):
    dev = torch.device("cuda")
    gpu.set_graph(graph)
    for k, st in enumerate(steps):
        g = torch.from_numpy(st.groups).to(dev)
        o = torch.from_numpy(st.offsets).to(dev)
        t = torch.from_numpy(st.tokens if st.num_tokens else np.zeros(4, np.int32)).to(dev)
        c = None if st.contracts is None else torch.from_numpy(st.contracts).to(dev)
        p = None if st.prefixes is None else torch.from_numpy(st.prefixes.view(np.int64)).to(dev)
        rc = gpu.step(st.now, g, o, t, c, p)
        assert rc == 0, f"{label} step {k}: launch rc {rc}"
        assert gpu.uses_graph() == graph, f"{label} step {k}: graph replay is {gpu.uses_graph()}"
        got = gpu.fetch(st.num_requests)
        want = orc.step(st.now, st.groups, st.offsets, st.tokens, st.contracts, st.prefixes)
        compare_outputs(got, want, f"{label} step {k}")
        if state_every and (k % state_every == 0 or k == len(steps) - 1):
            compare_state(gpu.export(), orc.export(), f"{label} step {k}", s3=s3 or gpu.policy == "s3fifo")
    assert np.array_equal(gpu.stats(), orc.stats()), f"{label}: stats differ"


GPU_POLICIES = ["lru", "s3fifo", "prefixshield", "staticquota"]


@pytest.mark.parametrize("policy", GPU_POLICIES)
@pytest.mark.parametrize("seed,N,G,R,contracts,prefixes,flags", [
    (1, 24, 2, 3, 0, False, 0),
    (2, 40, 3, 6, 0, False, 0),
    (3, 64, 4, 8, 3, True, 0),
    (4, 12, 1, 2, 0, False, 0),
    (5, 30, 3, 5, 3, True, 1),
    (6, 30, 3, 5, 3, True, 2),
    (11, 20, 2, 4, 2, False, 0),
])
def test_parity_fuzz(policy, seed, N, G, R, contracts, prefixes, flags):
    steps = W.fuzz_steps(seed, G, R, 60, docs_per_group=3, doc_blocks=7, fresh_max_blocks=2,
                         with_contracts=contracts, with_prefixes=prefixes, now_stride=2, empty_every=9)
    kw = dict(rho=(2.0, 1.5, 1.0), beta=(6.0, 5.0, 4.0), flags=flags, contract_of_group=[g % 3 for g in range(G)])
    gpu, orc = _pair(N, 16, G, policy, kw, max_requests=R, max_tokens=4096)
    _run(gpu, orc, steps, label=f"fuzz{seed}/{policy}")


@pytest.mark.parametrize("policy,fname", [("lru", "lru_hand_trace.txt"), ("s3fifo", "s3fifo_hand_trace.txt")])
def test_parity_hand_traces(policy, fname):
    """The hand-traced golden traces, GPU against oracle (which the traces pin)."""
    from _util import make_step, obj_tokens, params_line, parse_trace
    steps, _ = parse_trace(fname)
    pr = params_line(fname)
    kw = dict(rho=(1000.0,), beta=(1000.0,))
    if policy == "s3fifo":
        kw.update(s3_small_pct=pr["small_pct"], s3_freq_cap=pr["freq_cap"], s3_move_min_freq=pr["move_min_freq"])
    gpu, orc = _pair(pr["N"], 16, 1, policy, kw, max_requests=4, max_tokens=256)
    seq = []
    for si, (reqs, _, _) in enumerate(steps):
        g, o, t, _ = make_step([obj_tokens(n) for n in reqs])
        seq.append(W.Step(index=si, now=si + 1, groups=g, offsets=o, tokens=t))
    _run(gpu, orc, seq, label=fname)


@pytest.mark.parametrize("bs", [2, 4, 8, 32, 64])
def test_parity_block_sizes(bs):
    steps = W.fuzz_steps(21, 2, 4, 25, block_size=bs, docs_per_group=3, doc_blocks=40, fresh_max_blocks=40)
    gpu, orc = _pair(200, bs, 2, "prefixshield", dict(rho=(8.0,), beta=(40.0,)), max_requests=4,
                     max_tokens=4 * 90 * bs)
    _run(gpu, orc, steps, label=f"bs{bs}")


@pytest.mark.parametrize("policy", GPU_POLICIES)
def test_parity_tiny_one_touch(policy):
    wl = W.make_workload(0, seed=1)
    sp = wl.spec
    gpu, orc = _pair(sp.capacity_blocks, sp.block_size, sp.num_groups, policy, dict(rho=sp.rho, beta=sp.beta),
                     max_requests=sp.requests_per_step, max_tokens=sp.requests_per_step * 1100)
    _run(gpu, orc, list(wl.steps()), state_every=5, label=f"cfg0/{policy}")


@pytest.mark.parametrize("policy", GPU_POLICIES)
@pytest.mark.parametrize("cfg,nsteps,rps", [(1, 40, None), (1, 60, 8), (2, 40, None), (2, 40, 8), (3, 30, None),
                                           (5, 120, None)])
def test_parity_configs(policy, cfg, nsteps, rps):
    wl = W.make_workload(cfg, seed=2, requests_per_step=rps)
    sp = wl.spec
    steps = list(wl.steps(nsteps))
    maxT = max(s.num_tokens for s in steps)
    kw = dict(rho=sp.rho, beta=sp.beta)
    if sp.contract_of_group is not None:
        kw["contract_of_group"] = list(sp.contract_of_group)
    gpu, orc = _pair(sp.capacity_blocks, sp.block_size, sp.num_groups, policy, kw,
                     max_requests=sp.requests_per_step, max_tokens=maxT)
    _run(gpu, orc, steps, state_every=10, label=f"cfg{cfg}/{policy}")


@pytest.mark.parametrize("policy", GPU_POLICIES)
@pytest.mark.parametrize("flags", [0, O.FLAG_INDEXED_QUEUES])
def test_parity_two_pass_replay(policy, flags):
    """The two-pass replay trace (Sec. V-B) shortened to 24 fresh attacker
    prompts replayed once, 8 requests a step, so the second pass runs: every
    step of both passes equals the oracle, and the oracle's replayed attacker
    prompts hit the cache (except under StaticQuota, whose cap on the
    attacker's partition leaves nothing to replay)."""
    if flags and policy == "s3fifo":
        pytest.skip("s3fifo keeps its own queues")
    wl = W.make_workload(2, seed=2, requests_per_step=8, attacker_prompts=24)
    sp = wl.spec
    steps = list(wl.steps())
    gpu, orc = _pair(sp.capacity_blocks, sp.block_size, sp.num_groups, policy,
                     dict(rho=sp.rho, beta=sp.beta, flags=flags), max_requests=sp.requests_per_step,
                     max_tokens=max(s.num_tokens for s in steps))
    dev = torch.device("cuda")
    seen = replay_hits = 0
    for k, st in enumerate(steps):
        rc = gpu.step(st.now, torch.from_numpy(st.groups).to(dev), torch.from_numpy(st.offsets).to(dev),
                      torch.from_numpy(st.tokens).to(dev))
        assert rc == 0
        want = orc.step(st.now, st.groups, st.offsets, st.tokens)
        compare_outputs(gpu.fetch(st.num_requests), want, f"replay/{policy} step {k}")
        for i, g in enumerate(st.groups):
            if g == 1:
                seen += 1
                if seen > 24:
                    replay_hits += int(want["hit_blocks"][i])
    compare_state(gpu.export(), orc.export(), f"replay/{policy}", s3=policy == "s3fifo")
    assert np.array_equal(gpu.stats(), orc.stats())
    assert seen == 48
    assert (replay_hits == 0) if policy == "staticquota" else (replay_hits > 0)


@pytest.mark.parametrize("policy", GPU_POLICIES)
@pytest.mark.parametrize("wait,flags", [(0, 0), (0, O.FLAG_NO_DEBT_GATE), (1, 0), (3, 0), (3, O.FLAG_NO_DEBT_GATE),
                                        (0, O.FLAG_NO_SEGMENTATION)])
def test_parity_delayed_replay(policy, wait, flags):
    """The delayed-replay trace with three contracts (critical, standard,
    best-effort): burst into debt, gated or ungated replay, neutral pressure."""
    wl = W.make_workload(6, seed=4, wait=wait)
    sp = wl.spec
    steps = list(wl.steps())
    kw = dict(rho=sp.rho, beta=sp.beta, contract_of_group=list(sp.contract_of_group), flags=flags)
    gpu, orc = _pair(sp.capacity_blocks, sp.block_size, sp.num_groups, policy, kw,
                     max_requests=sp.requests_per_step, max_tokens=2 * 1536)
    _run(gpu, orc, steps, label=f"cfg6/w{wait}/f{flags}/{policy}")


QUEUE_POLICIES = ["lru", "prefixshield", "staticquota"]
IQ = O.FLAG_INDEXED_QUEUES


@pytest.mark.parametrize("policy", QUEUE_POLICIES)
@pytest.mark.parametrize("seed,N,G,R,contracts,prefixes,flags", [
    (1, 24, 2, 3, 0, False, 0),
    (2, 40, 3, 6, 0, False, 0),
    (3, 64, 4, 8, 3, True, 0),
    (4, 12, 1, 2, 0, False, 0),
    (5, 30, 3, 5, 3, True, 1),
    (6, 30, 3, 5, 3, True, 2),
    (11, 20, 2, 4, 2, False, 0),
])
def test_parity_queues_fuzz(policy, seed, N, G, R, contracts, prefixes, flags):
    """Victims from the indexed queues over long fuzz traces.  The token
    bound is the trace's own, so the logs' buffers are small and every log is
    compacted many times."""
    steps = W.fuzz_steps(seed, G, R, 240, docs_per_group=3, doc_blocks=7, fresh_max_blocks=2,
                         with_contracts=contracts, with_prefixes=prefixes, now_stride=2, empty_every=9)
    kw = dict(rho=(2.0, 1.5, 1.0), beta=(6.0, 5.0, 4.0), flags=flags | IQ, contract_of_group=[g % 3 for g in range(G)])
    gpu, orc = _pair(N, 16, G, policy, kw, max_requests=R, max_tokens=max(16, max(st.num_tokens for st in steps)))
    _run(gpu, orc, steps, state_every=7, label=f"queues/fuzz{seed}/{policy}")


@pytest.mark.parametrize("policy", QUEUE_POLICIES)
@pytest.mark.parametrize("flags", [0, 1, 2])
def test_parity_queues_many_groups(policy, flags):
    """37 groups (114 logs), three contracts, ragged requests: many logs
    share each scan, layout and compaction."""
    G = 37
    steps = W.fuzz_steps(17, G, 12, 120, docs_per_group=2, doc_blocks=6, fresh_max_blocks=3,
                         with_contracts=3, now_stride=2, empty_every=13)
    kw = dict(rho=(2.0, 1.5, 1.0), beta=(6.0, 5.0, 4.0), flags=flags | IQ, contract_of_group=[g % 3 for g in range(G)])
    gpu, orc = _pair(180, 16, G, policy, kw, max_requests=12, max_tokens=max(st.num_tokens for st in steps))
    _run(gpu, orc, steps, state_every=9, label=f"queues/groups{G}/f{flags}/{policy}")


@pytest.mark.parametrize("policy", QUEUE_POLICIES)
def test_parity_queues_direct_launches(policy):
    """The indexed queues launched kernel by kernel (their second scan round
    and the compaction then run as kernels that find nothing to do)."""
    steps = W.fuzz_steps(12, 3, 5, 120, docs_per_group=3, doc_blocks=7, fresh_max_blocks=3, empty_every=7)
    kw = dict(rho=(2.0,), beta=(6.0,), flags=IQ)
    gpu, orc = _pair(30, 16, 3, policy, kw, max_requests=5, max_tokens=max(st.num_tokens for st in steps))
    _run(gpu, orc, steps, state_every=5, label=f"queues/direct/{policy}", graph=False)


@pytest.mark.parametrize("policy", QUEUE_POLICIES)
@pytest.mark.parametrize("cfg,nsteps,rps,wait,flags", [(1, 60, 8, 0, 0), (3, 30, None, 0, 0), (5, 120, None, 0, 0),
                                                       (6, None, None, 0, 0), (6, None, None, 1, 2)])
def test_parity_queues_configs(policy, cfg, nsteps, rps, wait, flags):
    wl = W.make_workload(cfg, seed=2, requests_per_step=rps, wait=wait)
    sp = wl.spec
    steps = list(wl.steps(nsteps))
    kw = dict(rho=sp.rho, beta=sp.beta, flags=flags | IQ)
    if sp.contract_of_group is not None:
        kw["contract_of_group"] = list(sp.contract_of_group)
    gpu, orc = _pair(sp.capacity_blocks, sp.block_size, sp.num_groups, policy, kw,
                     max_requests=sp.requests_per_step, max_tokens=max(st.num_tokens for st in steps))
    _run(gpu, orc, steps, state_every=10, label=f"queues/cfg{cfg}/{policy}")


@pytest.mark.parametrize("policy", QUEUE_POLICIES)
@pytest.mark.parametrize("cfg,nsteps,rps", [(1, 60, None), (3, 30, None)])
def test_parity_queues_second_round(policy, cfg, nsteps, rps):
    """First scan rounds of one chunk: every take longer than 1024 live
    entries, or behind dead ones, finishes in the second round."""
    wl = W.make_workload(cfg, seed=3, requests_per_step=rps)
    sp = wl.spec
    steps = list(wl.steps(nsteps))
    kw = dict(rho=sp.rho, beta=sp.beta, flags=IQ | O.FLAG_QUEUE_SHORT_WINDOWS)
    gpu, orc = _pair(sp.capacity_blocks, sp.block_size, sp.num_groups, policy, kw,
                     max_requests=sp.requests_per_step, max_tokens=max(st.num_tokens for st in steps))
    _run(gpu, orc, steps, state_every=10, label=f"queues/short/cfg{cfg}/{policy}")
    assert orc.stats()[:, O.STAT_NAMES.index("evicted_blocks")].sum() > 1024


def test_parity_queues_alg2_ties():
    """Eq. 7's tie rule with the tie candidates read from the queues."""
    G = 6
    steps = W.fuzz_steps(31, G, 6, 120, docs_per_group=2, doc_blocks=6, fresh_max_blocks=3)
    for flags in (0, 1):
        kw = dict(rho=(1.0,), beta=(2.0,), flags=flags | IQ)
        gpu, orc = _pair(36, 16, G, "prefixshield", kw, max_requests=6, max_tokens=4096)
        _run(gpu, orc, steps, label=f"queues/ties/f{flags}")


@pytest.mark.parametrize("flags", [0, O.FLAG_INDEXED_QUEUES])
def test_parity_three_contract_tiers(flags):
    """The paper's contract tiers with debts whose fixed-point decrements are
    not whole blocks (Eq. 5, Eq. 8): the hand-derived scenario of the oracle
    pins, then fuzz steps on the same pool."""
    from _util import make_step, obj_tokens
    kw = dict(rho=(64.0, 40.0, 16.0), beta=(256.0, 192.0, 128.0), contract_of_group=[1, 2, 0], flags=flags)
    gpu, orc = _pair(351, 16, 3, "prefixshield", kw, max_requests=4, max_tokens=217 * 16 + 134 * 16)
    seq = []
    g, o, t, _ = make_step([obj_tokens("A", blocks=217), obj_tokens("B", blocks=134)], [0, 1])
    seq.append(W.Step(index=0, now=1, groups=g, offsets=o, tokens=t))
    g, o, t, _ = make_step([obj_tokens("C", blocks=20)], [2])
    seq.append(W.Step(index=1, now=1, groups=g, offsets=o, tokens=t))
    for k, st in enumerate(W.fuzz_steps(23, 3, 4, 40, docs_per_group=3, doc_blocks=40, fresh_max_blocks=30)):
        seq.append(W.Step(index=2 + k, now=2 + k, groups=st.groups, offsets=st.offsets, tokens=st.tokens))
    _run(gpu, orc, seq, state_every=5, label=f"tiers/f{flags}")


@pytest.mark.parametrize("flags", [0, O.FLAG_INDEXED_QUEUES])
def test_parity_hand_derived_corners(flags):
    """The hand-derived oracle pins of the grant rule, the hook order inside a
    request and history within a step, replayed through the GPU step."""
    from _util import make_step, obj_tokens
    P, Q, S, T, X = (obj_tokens(n, blocks=b) for n, b in (("P", 3), ("Q", 1), ("S", 3), ("T", 1), ("X", 3)))
    P2 = obj_tokens("P2", blocks=2)
    cases = [
        (5, 100.0, [[P, np.concatenate([P, Q]), S], [S]]),       # ranks past avail
        (4, 100.0, [[P, S, np.concatenate([S, T])]]),            # a run stopped by an ungranted key
        (64, 4.0, [[P2], [np.concatenate([P2, X])]]),            # gate before the charge, class after
        (64, 4.0, [[P2, P2]]),                                   # history within a step
    ]
    for ci, (N, beta, steps) in enumerate(cases):
        kw = dict(rho=(1.0,) if beta == 4.0 else (100.0,), beta=(beta,), flags=flags)
        gpu, orc = _pair(N, 16, 1, "prefixshield", kw, max_requests=3, max_tokens=2048)
        seq = []
        for k, prompts in enumerate(steps):
            g, o, t, _ = make_step(prompts)
            seq.append(W.Step(index=k, now=1, groups=g, offsets=o, tokens=t))
        _run(gpu, orc, seq, label=f"corner{ci}/f{flags}")


@pytest.mark.parametrize("policy", GPU_POLICIES)
@pytest.mark.parametrize("flags", [0, O.FLAG_INDEXED_QUEUES])
def test_parity_orphan_scenario(policy, flags):
    """The hand-derived orphan scenario of the oracle pins (a chain with two
    holes, a chain with no first block, a later request holding an orphan
    again), replayed through the GPU step with its explicit prefix ids."""
    from _util import make_step, obj_tokens
    if flags and policy == "s3fifo":
        pytest.skip("s3fifo keeps its own queues")
    X, V, Y = obj_tokens("X", blocks=6), obj_tokens("V", blocks=2), obj_tokens("Y", blocks=6)
    plan = [[(X, 3, 0, 1), (V, 1, 0, 21)], [(X, 4, 0, 2), (V, 2, 0, 22)], [(X, 5, 0, 3)], [(X, 6, 0, 4)],
            [(X, 4, 0, 2), (V, 2, 0, 22)], [(X, 6, 0, 4)], [(Y, 6, 1, 31)],
            [(X, 6, 0, 4), (V, 2, 0, 22), (X, 4, 0, 4)]]
    seq = []
    for k, reqs in enumerate(plan):
        g, o, t, _ = make_step([tk[: 16 * nb] for tk, nb, _, _ in reqs], [grp for _, _, grp, _ in reqs])
        seq.append(W.Step(k, k + 1, g, o, t, None, np.array([pid for _, _, _, pid in reqs], np.uint64)))
    gpu, orc = _pair(11, 16, 2, policy, dict(rho=(1000.0,), beta=(1000.0,), flags=flags), max_requests=3,
                     max_tokens=12 * 16)
    _run(gpu, orc, seq, label=f"orphans/{policy}/f{flags}")


def test_parity_alg2_ties():
    """Groups with equal debt and equal decrements force Eq. 7's tie rule."""
    G = 6
    steps = W.fuzz_steps(31, G, 6, 50, docs_per_group=2, doc_blocks=6, fresh_max_blocks=3)
    kw = dict(rho=(1.0,), beta=(2.0,))
    gpu, orc = _pair(36, 16, G, "prefixshield", kw, max_requests=6, max_tokens=4096)
    _run(gpu, orc, steps, label="ties")


def test_invalid_inputs_leave_state_unchanged():
    gpu, orc = _pair(32, 16, 2, "prefixshield", dict(rho=(1.0,), beta=(2.0,), history_capacity=3),
                     max_requests=4, max_tokens=512)
    dev = torch.device("cuda")
    from _util import make_step, obj_tokens

    def both(now, prompts, groups, contracts=None, prefixes=None, offsets=None):
        g, o, t, _ = make_step(prompts, groups)
        if offsets is not None:
            o = np.asarray(offsets, np.int64)
        rc = gpu.step(now, torch.from_numpy(g).to(dev), torch.from_numpy(o).to(dev),
                      torch.from_numpy(t if len(t) else np.zeros(4, np.int32)).to(dev),
                      None if contracts is None else torch.from_numpy(np.asarray(contracts, np.int32)).to(dev),
                      None if prefixes is None else torch.from_numpy(np.asarray(prefixes, np.int64)).to(dev))
        assert rc == 0
        got = gpu.fetch(len(g))
        want = orc.step(now, g, o, t, None if contracts is None else np.asarray(contracts, np.int32),
                        None if prefixes is None else np.asarray(prefixes, np.uint64))
        compare_outputs(got, want, f"now={now}")
        return got["status"]

    A = obj_tokens("a", blocks=2)
    assert both(5, [A], [0]) == 0
    snap = gpu.export()
    assert both(4, [A], [0]) == O.ERR_CLOCK
    assert both(5, [A], [2]) == O.ERR_INVALID_ARG
    assert both(5, [A], [0], offsets=[1, 32]) == O.ERR_INVALID_ARG
    assert both(5, [A], [0], contracts=[1]) == O.ERR_INVALID_ARG
    assert both(5, [A], [0], prefixes=[0]) == O.ERR_INVALID_ARG
    compare_state(gpu.export(), snap, "after invalid steps")
    compare_state(gpu.export(), orc.export(), "after invalid steps vs oracle")
    P = [obj_tokens(x) for x in "pqr"]
    assert both(6, P[:2], [0, 1]) == 0
    assert both(6, P[2:], [1]) == O.ERR_CAPACITY
    assert both(7, [], []) == O.ERR_CAPACITY
    gpu.clear_status(); orc.clear_status()
    assert both(7, [], []) == 0


@pytest.mark.parametrize("N", [40, 70000])
def test_step_host_matches_step(N):
    """The host-buffer entry point (staging copies in the workspace) against
    the oracle; the larger pool spans several id-list compaction chunks."""
    from paper_2608_01657_gb300 import binding as B
    steps = W.fuzz_steps(41, 3, 5, 30, docs_per_group=3, doc_blocks=6)
    kw = dict(rho=(2.0,), beta=(6.0,))
    a = B.Cache(N, 16, 3, "prefixshield", B.Params(**kw), max_requests=5, max_tokens=2048)
    orc = O.OracleCache(N, 16, 3, "prefixshield", O.Params(**kw))
    for st in steps:
        out = a.step_host(st.now, st.groups, st.offsets, st.tokens)
        assert out["rc"] == 0
        cnt = out["counts"]
        got = {"status": int(cnt[3]), "hit_blocks": out["hit_blocks"][:st.num_requests],
               "admitted_blocks": out["admitted_blocks"][:st.num_requests],
               "admitted_offsets": out["admitted_offsets"][:st.num_requests + 1],
               "admitted_ids": out["admitted_ids"][:cnt[0]], "evicted_ids": out["evicted_ids"][:cnt[1]],
               "invalidated_ids": out["invalidated_ids"][:cnt[2]], "debt_raw": out["debt_raw"],
               "debt_norm": out["debt_norm"]}
        compare_outputs(got, orc.step(st.now, st.groups, st.offsets, st.tokens), f"step {st.index}")


@pytest.mark.parametrize("policy", ["lru", "prefixshield"])
def test_parity_host_pipelined(policy):
    """ps_step_host_async on alternating slots, two steps in flight: every
    output equals the oracle's; unpinned output buffers are refused."""
    from paper_2608_01657_gb300 import binding as B
    steps = W.fuzz_steps(43, 3, 5, 40, docs_per_group=3, doc_blocks=6, with_contracts=3, empty_every=7)
    kw = dict(rho=(2.0, 1.5, 1.0), beta=(6.0, 5.0, 4.0), contract_of_group=[0, 1, 2])
    a = B.Cache(40, 16, 3, policy, B.Params(**kw), max_requests=5, max_tokens=2048)
    orc = O.OracleCache(40, 16, 3, policy, O.Params(**kw))
    outs = [B.host_outputs(5, a.max_blocks, 3, pinned=True) for _ in range(2)]

    def pinned(x):
        return torch.from_numpy(np.ascontiguousarray(x)).pin_memory().numpy()

    host = [(st, pinned(st.groups), pinned(st.offsets), pinned(st.tokens if st.num_tokens else np.zeros(4, np.int32)),
             pinned(st.contracts)) for st in steps]

    def check(j):
        st = host[j][0]
        assert a.step_host_wait(j % 2) == 0
        out = outs[j % 2]
        cnt = out["counts"]
        got = {"status": int(cnt[3]), "hit_blocks": out["hit_blocks"][:st.num_requests],
               "admitted_blocks": out["admitted_blocks"][:st.num_requests],
               "admitted_offsets": out["admitted_offsets"][:st.num_requests + 1],
               "admitted_ids": out["admitted_ids"][:cnt[0]], "evicted_ids": out["evicted_ids"][:cnt[1]],
               "invalidated_ids": out["invalidated_ids"][:cnt[2]], "debt_raw": out["debt_raw"],
               "debt_norm": out["debt_norm"]}
        compare_outputs(got, orc.step(st.now, st.groups, st.offsets, st.tokens, st.contracts), f"step {st.index}")

    for k, (st, g, o, t, c) in enumerate(host):
        assert a.step_host_async(k % 2, st.now, g, o, t, outs[k % 2], contracts=c) == 0
        if k >= 1:
            check(k - 1)
    check(len(host) - 1)
    assert np.array_equal(a.stats(), orc.stats())
    # output buffers a kernel cannot write are refused before anything is enqueued
    st = steps[0]
    plain = B.host_outputs(5, a.max_blocks, 3, pinned=False)
    assert a.step_host_async(0, st.now + 1000, host[0][1], host[0][2], host[0][3], plain) == B.PS_ERR_INVALID_ARG


_SCALE = {}


def _scale_steps(n):
    if n not in _SCALE:
        wl = W.make_workload(4, seed=1)
        _SCALE[n] = (wl.spec, list(wl.steps(n)))
    return _SCALE[n]


@pytest.mark.parametrize("policy", GPU_POLICIES)
def test_parity_scale_full_size(policy):
    """The benchmarked configuration itself (64 groups, 1,048,576 blocks,
    4096 requests per step), from the empty pool through the fill and into
    steady-state reclamation: every output of every step and the complete
    final state equal the oracle's."""
    spec, steps = _scale_steps(9)
    maxT = max(s.num_tokens for s in steps)
    gpu, orc = _pair(spec.capacity_blocks, spec.block_size, spec.num_groups, policy,
                     dict(rho=spec.rho, beta=spec.beta, history_capacity=1 << 20),
                     max_requests=spec.requests_per_step, max_tokens=maxT)
    _run(gpu, orc, steps, state_every=4, label=f"scale/{policy}")
    assert orc.stats()[:, O.STAT_NAMES.index("evicted_blocks")].sum() > 0  # reclamation was exercised


@pytest.mark.parametrize("policy", ["lru", "prefixshield"])
def test_parity_queues_scale_full_size(policy):
    """The benchmarked configuration with victims from the indexed queues:
    every output of every step and the final state equal the oracle's."""
    spec, steps = _scale_steps(9)
    maxT = max(s.num_tokens for s in steps)
    gpu, orc = _pair(spec.capacity_blocks, spec.block_size, spec.num_groups, policy,
                     dict(rho=spec.rho, beta=spec.beta, history_capacity=1 << 20, flags=IQ),
                     max_requests=spec.requests_per_step, max_tokens=maxT)
    _run(gpu, orc, steps, state_every=4, label=f"queues/scale/{policy}")
    assert orc.stats()[:, O.STAT_NAMES.index("evicted_blocks")].sum() > 0


@pytest.mark.parametrize("policy", GPU_POLICIES)
def test_cached_prefix_probe(policy):
    """ps_cached_prefix (read-only) equals the oracle's leading-resident count
    before every step, leaves the state untouched, and equals the step's own
    hit counts for requests without in-step sharing."""
    steps = W.fuzz_steps(51, 3, 6, 40, docs_per_group=3, doc_blocks=40, fresh_max_blocks=30)
    gpu, orc = _pair(150, 16, 3, policy, dict(rho=(3.0,), beta=(9.0,)), max_requests=6, max_tokens=8192)
    dev = torch.device("cuda")
    for st in steps:
        g = torch.from_numpy(st.groups).to(dev)
        o = torch.from_numpy(st.offsets).to(dev)
        t = torch.from_numpy(st.tokens if st.num_tokens else np.zeros(4, np.int32)).to(dev)
        before = gpu.export()
        cnt, status = gpu.cached_prefix(g, o, t)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        want = orc.cached_prefix(st.groups, st.offsets, st.tokens)
        assert np.array_equal(cnt[: st.num_requests].cpu().numpy(), want)
        compare_state(gpu.export(), before, "probe must not change state")
        assert gpu.step(st.now, g, o, t) == 0
        got = gpu.fetch(st.num_requests)
        ref = orc.step(st.now, st.groups, st.offsets, st.tokens)
        compare_outputs(got, ref, f"step {st.index}")
    # a bad group id is reported, not a fault
    g = torch.tensor([7], dtype=torch.int32, device=dev)
    o = torch.tensor([0, 32], dtype=torch.int64, device=dev)
    t = torch.zeros(32, dtype=torch.int32, device=dev)
    _, status = gpu.cached_prefix(g, o, t)
    assert int(status.item()) == O.ERR_INVALID_ARG


@pytest.mark.parametrize("policy", GPU_POLICIES)
def test_parity_graph_replay_streams_and_timing(policy):
    """The step replays one captured graph: steps of every size (empty ones
    included) on a side stream, stage timing switched on and off (which
    captures the step again), with every output and the state checked."""
    steps = W.fuzz_steps(21, 3, 6, 48, docs_per_group=3, doc_blocks=7, fresh_max_blocks=2,
                         with_contracts=3, with_prefixes=True, now_stride=2, empty_every=5)
    kw = dict(rho=(2.0, 1.5, 1.0), beta=(6.0, 5.0, 4.0), contract_of_group=[0, 1, 2])
    gpu, orc = _pair(40, 16, 3, policy, kw, max_requests=6, max_tokens=4096)
    dev = torch.device("cuda")
    side = torch.cuda.Stream()
    for k, st in enumerate(steps):
        if k % 7 == 3:
            gpu.set_stage_timing(k % 14 == 3)
        with torch.cuda.stream(side):
            g = torch.from_numpy(st.groups).to(dev)
            o = torch.from_numpy(st.offsets).to(dev)
            t = torch.from_numpy(st.tokens if st.num_tokens else np.zeros(4, np.int32)).to(dev)
            c = torch.from_numpy(st.contracts).to(dev)
            p = torch.from_numpy(st.prefixes.view(np.int64)).to(dev)
            assert gpu.step(st.now, g, o, t, c, p, stream=side) == 0
            assert gpu.uses_graph()
        got = gpu.fetch(st.num_requests, stream=side)
        want = orc.step(st.now, st.groups, st.offsets, st.tokens, st.contracts, st.prefixes)
        compare_outputs(got, want, f"graph/{policy} step {k}")
        if k % 7 == 3 and k % 14 == 3:
            ms, launches = gpu.stage_times()
            assert launches > 0 and np.all(ms >= 0)
    compare_state(gpu.export(), orc.export(), f"graph/{policy}", s3=policy == "s3fifo")
    assert np.array_equal(gpu.stats(), orc.stats())


def test_parity_long_split_list():
    """A select whose split list is longer than one CTA finishes in shared
    memory: one indebted group holds 12,001 Probationary and 12,000 Normal
    candidates, and 5,425 victims fall inside the Probationary class, so the
    first digit (the class byte) leaves the whole class on the list."""
    rng = np.random.default_rng(77)
    steps = []
    for k, (pid, nb) in enumerate([(7, 1), (7, 12000), (9, 12000), (11, 6000)]):
        toks = rng.integers(0, W.VOCAB, size=nb * 16, dtype=np.int32)
        steps.append(W.Step(k, k, np.zeros(1, np.int32), np.array([0, nb * 16], np.int64), toks,
                            None, np.array([pid], np.uint64)))
    gpu, orc = _pair(24576, 16, 2, "prefixshield", dict(rho=(1.0,), beta=(13000.0,)),
                     max_requests=1, max_tokens=12000 * 16)
    _run(gpu, orc, steps, label="long list")
    assert int(gpu.stats()[0][8]) == 5425  # evicted blocks of group 0


@pytest.mark.parametrize("policy", GPU_POLICIES)
def test_parity_kernel_by_kernel(policy):
    """The same step launched kernel by kernel (no graph), stage timing on and
    off, matches the oracle too."""
    steps = W.fuzz_steps(23, 3, 6, 40, docs_per_group=3, doc_blocks=7, fresh_max_blocks=2,
                         with_contracts=3, with_prefixes=True, now_stride=2, empty_every=5)
    kw = dict(rho=(2.0, 1.5, 1.0), beta=(6.0, 5.0, 4.0), contract_of_group=[0, 1, 2])
    gpu, orc = _pair(40, 16, 3, policy, kw, max_requests=6, max_tokens=4096)
    gpu.set_graph(False)
    dev = torch.device("cuda")
    for k, st in enumerate(steps):
        if k % 10 == 5:
            gpu.set_stage_timing(k % 20 == 5)
        g = torch.from_numpy(st.groups).to(dev)
        o = torch.from_numpy(st.offsets).to(dev)
        t = torch.from_numpy(st.tokens if st.num_tokens else np.zeros(4, np.int32)).to(dev)
        c = torch.from_numpy(st.contracts).to(dev)
        p = torch.from_numpy(st.prefixes.view(np.int64)).to(dev)
        assert gpu.step(st.now, g, o, t, c, p) == 0
        assert not gpu.uses_graph()
        compare_outputs(gpu.fetch(st.num_requests),
                        orc.step(st.now, st.groups, st.offsets, st.tokens, st.contracts, st.prefixes),
                        f"direct/{policy} step {k}")
    compare_state(gpu.export(), orc.export(), f"direct/{policy}", s3=policy == "s3fifo")
    assert np.array_equal(gpu.stats(), orc.stats())


def test_parity_staticquota_borrowing_trace():
    """The borrowing trace (Table III) on the GPU: one group idle, the other
    capped at its equal share, every output and the state as the oracle's."""
    from _util import obj_tokens, make_step
    N, G = 511, 2
    gpu, orc = _pair(N, 16, G, "staticquota", dict(rho=(64.0,), beta=(4096.0,)), max_requests=8, max_tokens=8 * 64)
    steps = []
    for t in range(40):
        grp, offs, toks, _ = make_step([obj_tokens(f"borrow-{t}-{j}", blocks=4) for j in range(8)], groups=[0] * 8)
        steps.append(W.Step(t, t, grp, offs, toks))
    _run(gpu, orc, steps, state_every=5, label="borrowing")
    e = gpu.export()
    assert int(((e["resident"] == 1) & (e["group"] == 0)).sum()) == N // G
