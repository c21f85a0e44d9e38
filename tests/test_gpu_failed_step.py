"""A step that fails on the device leaves the pool exactly as it was.

Alg. 1's hooks change state only for requests that go ahead.  A step whose
new (group, prefix id) history entries would exceed the history capacity is
found out only on the device, after the lookup has pinned its cached
prefixes, claimed its new keys and installed its new history entries; all of
that must be undone.  Each case below steps the GPU and the oracle through:
steps that fill the history to capacity, a non-empty step that fails (with
pins, claims and a new entry), the sticky error, ps_clear_status on both
sides, the failed batch again without its new entry (same keys, same
blocks), a second failing step, and 25 more steps, comparing every output
and the complete state (history included) after each one.  Outputs,
state and statistics are integers: bit-exact.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_01657_gb300 import workloads as W
from _util import compare_outputs, compare_state

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

G, DOCS = 2, 3
HELD = (1, 1000 * 1 + DOCS)  # the (group, prefix id) kept out until the failing step


def _pairs(st):
    return [(int(g), int(p)) for g, p in zip(st.groups, st.prefixes)]


def _keep(st, keep):
    """The step with only the requests i where keep[i] (same token content)."""
    idx = [i for i, k in enumerate(keep) if k]
    pieces = [st.tokens[st.offsets[i]:st.offsets[i + 1]] for i in idx]
    offs = np.zeros(len(idx) + 1, np.int64)
    for j, p in enumerate(pieces):
        offs[j + 1] = offs[j] + len(p)
    toks = np.concatenate(pieces).astype(np.int32) if pieces else np.zeros(0, np.int32)
    return W.Step(st.index, st.now, st.groups[idx].copy(), offs, toks, None, st.prefixes[idx].copy())


def _without_held(st):
    return _keep(st, [pair != HELD for pair in _pairs(st)])


@pytest.mark.parametrize("policy,flags", [("prefixshield", 0), ("lru", 0), ("s3fifo", 0), ("staticquota", 0),
                                          ("prefixshield", O.FLAG_INDEXED_QUEUES), ("lru", O.FLAG_INDEXED_QUEUES)])
def test_failed_step_leaves_no_trace(policy, flags):
    from paper_2608_01657_gb300 import binding as B
    steps = W.fuzz_steps(61, G, 6, 80, docs_per_group=DOCS, doc_blocks=7, fresh_max_blocks=3, with_prefixes=True,
                         now_stride=2)
    kw = dict(rho=(2.0,), beta=(6.0,), history_capacity=G * DOCS - 1, flags=flags)
    gpu = B.Cache(40, 16, G, policy, B.Params(**kw), max_requests=6, max_tokens=4096)
    orc = O.OracleCache(40, 16, G, policy, O.Params(**kw))
    dev = torch.device("cuda")
    s3 = policy == "s3fifo"

    def both(st, label):
        t = st.tokens if st.num_tokens else np.zeros(4, np.int32)
        rc = gpu.step(st.now, torch.from_numpy(st.groups).to(dev), torch.from_numpy(st.offsets).to(dev),
                      torch.from_numpy(t).to(dev), None, torch.from_numpy(st.prefixes.view(np.int64)).to(dev))
        assert rc == 0, label
        got = gpu.fetch(st.num_requests)
        want = orc.step(st.now, st.groups, st.offsets, st.tokens, None, st.prefixes)
        compare_outputs(got, want, label)
        compare_state(gpu.export(), orc.export(), label, s3=s3)
        return want["status"]

    # the history fills up with every pair but the held one
    for k in range(15):
        assert both(_without_held(steps[k]), f"fill {k}") == 0
    assert len(orc.export()["history"][0]) == G * DOCS - 1

    # the failing batch: the held pair plus at least three other requests,
    # some with a cached prefix (pins) and some with new blocks (claims)
    fail_k = next(k for k in range(15, len(steps))
                  if HELD in _pairs(steps[k]) and sum(p != HELD for p in _pairs(steps[k])) >= 3)
    st = steps[fail_k]
    ex = orc.export()
    h = orc.cached_prefix(st.groups, st.offsets, st.tokens)
    n = np.diff(st.offsets) // 16
    assert h.sum() > 0 and (n - h).sum() > 0
    before = gpu.export()
    assert both(st, "failing step") == O.ERR_CAPACITY
    compare_state(gpu.export(), before, "the failed step changed the pool")
    compare_state(gpu.export(), ex, "the failed step changed the pool (oracle)")

    # sticky until cleared
    empty = W.Step(fail_k, st.now, np.zeros(0, np.int32), np.zeros(1, np.int64), np.zeros(0, np.int32), None,
                   np.zeros(0, np.uint64))
    assert both(empty, "sticky") == O.ERR_CAPACITY
    gpu.clear_status()
    orc.clear_status()

    # the same batch without the held pair: the same keys, pins and claims
    assert both(_without_held(st), "retried step") == 0
    # the held pair fails again (its entry was not left behind), then 25 steps
    again = next(k for k in range(fail_k + 1, len(steps)) if HELD in _pairs(steps[k]))
    assert both(steps[again], "second failing step") == O.ERR_CAPACITY
    gpu.clear_status()
    orc.clear_status()
    for k in range(fail_k + 1, fail_k + 26):
        assert both(_without_held(steps[k]), f"after {k}") == 0
    assert np.array_equal(gpu.stats(), orc.stats())


def test_undersized_output_buffers_are_refused():
    """Output capacities below what a step may write are refused before
    anything is enqueued (device and host entry points)."""
    from paper_2608_01657_gb300 import binding as B
    steps = W.fuzz_steps(62, 2, 4, 3, docs_per_group=2, doc_blocks=5)
    gpu = B.Cache(40, 16, 2, "prefixshield", B.Params(rho=(2.0,), beta=(6.0,)), max_requests=4, max_tokens=1024)
    orc = O.OracleCache(40, 16, 2, "prefixshield", O.Params(rho=(2.0,), beta=(6.0,)))
    dev = torch.device("cuda")
    st = steps[0]
    g, o = torch.from_numpy(st.groups).to(dev), torch.from_numpy(st.offsets).to(dev)
    t = torch.from_numpy(st.tokens).to(dev)
    L = B.load()
    import ctypes as C
    for field, value in (("ids_capacity", gpu.max_blocks - 1), ("req_capacity", st.num_requests - 1)):
        out = B.step_out(gpu.out)
        setattr(out, field, value)
        rc = L.ps_step(gpu._h, None, st.now, st.num_requests, B._ptr(g), B._ptr(o), B._ptr(t), None, None,
                       C.byref(out))
        assert rc == B.PS_ERR_INVALID_ARG, field
        host = B.host_outputs(st.num_requests, gpu.max_blocks, 2)
        ho = B.step_out(host)
        setattr(ho, field, value)
        rc = L.ps_step_host(gpu._h, None, st.now, st.num_requests, B._ptr(st.groups), B._ptr(st.offsets),
                            B._ptr(st.tokens), None, None, C.byref(ho))
        assert rc == B.PS_ERR_INVALID_ARG, field
    # nothing ran: the first real step still equals the oracle's first step
    for k, s in enumerate(steps):
        assert gpu.step(s.now, torch.from_numpy(s.groups).to(dev), torch.from_numpy(s.offsets).to(dev),
                        torch.from_numpy(s.tokens).to(dev)) == 0
        compare_outputs(gpu.fetch(s.num_requests), orc.step(s.now, s.groups, s.offsets, s.tokens), f"step {k}")
    compare_state(gpu.export(), orc.export(), "after refused calls")
