"""GPU-vs-oracle parity of the S3-FIFO baseline (Sec. V-A; Yang et al.,
SOSP 2023) under the library's execution choices and its parameter range.

The library computes a step's S3-FIFO evictions in closed form in parallel
and replays the published one-at-a-time loop on one device thread where the
closed form does not apply; the ghost FIFO is compacted into a second ring
when it lacks room.  Two test flags force the rarer paths on small pools
(every step sequential; a compaction on every step).  Every output and the
whole S3-FIFO state (queue, sequence number and frequency of every block,
the ghost's entries and counters) must equal the oracle's after every step.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_01657_gb300 import workloads as W
from _util import compare_outputs, compare_state

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

S3C, S3S = O.FLAG_S3_COMPACT_GHOST, O.FLAG_S3_SEQUENTIAL


def _run(N, G, R, steps, params_kw, label, max_tokens=4096):
    from paper_2608_01657_gb300 import binding as B
    gpu = B.Cache(N, 16, G, "s3fifo", B.Params(**params_kw), max_requests=R, max_tokens=max_tokens)
    orc = O.OracleCache(N, 16, G, "s3fifo", O.Params(**params_kw))
    dev = torch.device("cuda")
    for k, st in enumerate(steps):
        g = torch.from_numpy(st.groups).to(dev)
        o = torch.from_numpy(st.offsets).to(dev)
        t = torch.from_numpy(st.tokens if st.num_tokens else np.zeros(4, np.int32)).to(dev)
        c = None if st.contracts is None else torch.from_numpy(st.contracts).to(dev)
        p = None if st.prefixes is None else torch.from_numpy(st.prefixes.view(np.int64)).to(dev)
        assert gpu.step(st.now, g, o, t, c, p) == 0, f"{label} step {k}"
        want = orc.step(st.now, st.groups, st.offsets, st.tokens, st.contracts, st.prefixes)
        compare_outputs(gpu.fetch(st.num_requests), want, f"{label} step {k}")
        compare_state(gpu.export(), orc.export(), f"{label} step {k}", s3=True)
    assert np.array_equal(gpu.stats(), orc.stats()), f"{label}: stats differ"
    return orc


def _fuzz(seed, G, R, n=60):
    return W.fuzz_steps(seed, G, R, n, docs_per_group=3, doc_blocks=7, fresh_max_blocks=2,
                        with_contracts=0, with_prefixes=False, now_stride=2, empty_every=9)


@pytest.mark.parametrize("flags", [S3C, S3S, S3C | S3S])
@pytest.mark.parametrize("seed,N,G,R", [(1, 24, 2, 3), (3, 64, 4, 8), (5, 30, 3, 5), (11, 20, 2, 4), (7, 200, 4, 12)])
def test_s3fifo_execution_choices(flags, seed, N, G, R):
    """The sequential kernel on every step, the ghost compacted on every step,
    and both: the same results as the oracle."""
    orc = _run(N, G, R, _fuzz(seed, G, R), dict(rho=(2.0,), beta=(6.0,), flags=flags), f"s3/{flags}/{seed}")
    assert orc.stats()[:, O.STAT_NAMES.index("evicted_blocks")].sum() > 0


@pytest.mark.parametrize("pct,cap,mm", [
    (10, 20, 2),   # a frequency cap above the closed form's 16 bins: the sequential kernel
    (10, 15, 3),   # the largest cap the closed form takes
    (50, 3, 2),    # a small queue of half the pool
    (100, 3, 2),   # no ghost at all: every push is trimmed at once
    (10, 3, 1),    # any touch moves a block to the main queue
    (10, 3, 4),    # a threshold above the cap: nothing ever moves
    (30, 1, 1),
])
@pytest.mark.parametrize("seed,N,G,R", [(2, 40, 3, 6), (9, 96, 4, 10)])
def test_s3fifo_parameters(pct, cap, mm, seed, N, G, R):
    kw = dict(rho=(2.0,), beta=(6.0,), s3_small_pct=pct, s3_freq_cap=cap, s3_move_min_freq=mm)
    orc = _run(N, G, R, _fuzz(seed, G, R), kw, f"s3p/{pct}/{cap}/{mm}/{seed}")
    assert orc.stats()[:, O.STAT_NAMES.index("evicted_blocks")].sum() > 0


@pytest.mark.parametrize("cfg,nsteps,rps", [(1, 40, None), (5, 120, None), (3, 30, None)])
def test_s3fifo_configs_compacting(cfg, nsteps, rps):
    """Configured workloads with the ghost compacted on every step."""
    wl = W.make_workload(cfg, seed=2, requests_per_step=rps)
    sp = wl.spec
    steps = list(wl.steps(nsteps))
    kw = dict(rho=sp.rho, beta=sp.beta, flags=S3C)
    if sp.contract_of_group is not None:
        kw["contract_of_group"] = list(sp.contract_of_group)
    from paper_2608_01657_gb300 import binding as B
    gpu = B.Cache(sp.capacity_blocks, sp.block_size, sp.num_groups, "s3fifo", B.Params(**kw),
                  max_requests=sp.requests_per_step, max_tokens=max(s.num_tokens for s in steps))
    orc = O.OracleCache(sp.capacity_blocks, sp.block_size, sp.num_groups, "s3fifo", O.Params(**kw))
    dev = torch.device("cuda")
    for k, st in enumerate(steps):
        assert gpu.step(st.now, torch.from_numpy(st.groups).to(dev), torch.from_numpy(st.offsets).to(dev),
                        torch.from_numpy(st.tokens).to(dev)) == 0
        want = orc.step(st.now, st.groups, st.offsets, st.tokens)
        compare_outputs(gpu.fetch(st.num_requests), want, f"cfg{cfg}/s3c step {k}")
        if k % 10 == 0 or k == len(steps) - 1:
            compare_state(gpu.export(), orc.export(), f"cfg{cfg}/s3c step {k}", s3=True)
    assert np.array_equal(gpu.stats(), orc.stats())
