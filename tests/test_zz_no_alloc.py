"""ps_cached_prefix_noalloc against ps_cached_prefix, through the C ABI.

The no-allocation variant serves callers that may not allocate device memory
(graph-capture regions, foreign allocators, query-only threads): it keeps its
scratch in a fixed array inside the library instead of the handle's
workspace.  Its counts must equal the workspace variant's exactly (integers:
tolerance zero) on two calls in a row, over a pool that earlier steps filled.
This file is collected last so that a failure here cannot hide another test.
"""
import numpy as np
import pytest

from paper_2608_01657_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def test_noalloc_probe_matches_workspace_probe():
    from paper_2608_01657_gb300 import binding as B
    dev = torch.device("cuda")
    steps = W.fuzz_steps(61, 3, 6, 30, docs_per_group=3, doc_blocks=40, fresh_max_blocks=30)
    cache = B.Cache(150, 16, 3, "prefixshield", B.Params(rho=(3.0,), beta=(9.0,)), max_requests=6,
                    max_tokens=8192)
    for st in steps[:20]:  # fill the pool through the regular step
        assert cache.step(st.now, torch.from_numpy(st.groups).to(dev), torch.from_numpy(st.offsets).to(dev),
                          torch.from_numpy(st.tokens if st.num_tokens else np.zeros(4, np.int32)).to(dev)) == 0
    torch.cuda.synchronize()
    calls = 0
    for st in steps[20:]:
        if st.num_requests == 0:
            continue
        g = torch.from_numpy(st.groups).to(dev)
        o = torch.from_numpy(st.offsets).to(dev)
        t = torch.from_numpy(st.tokens).to(dev)
        want, wst = cache.cached_prefix(g, o, t)
        out = torch.full((st.num_requests,), -1, dtype=torch.int32, device=dev)
        status = torch.full((1,), 99, dtype=torch.int32, device=dev)
        assert cache.cached_prefix_noalloc(g, o, t, out, status) == 0
        torch.cuda.synchronize()
        assert int(wst.item()) == 0 and int(status.item()) == 0
        assert torch.equal(out, want[: st.num_requests])
        assert int(want.sum().item()) > 0  # the pool does hold prefixes
        calls += 1
        if calls == 2:
            break
    assert calls == 2


def test_noalloc_probe_rejects_oversized_batches():
    """More requests than the handle takes are refused as ps_cached_prefix
    refuses them (invalid argument); more than the fixed scratch holds (4096)
    on a handle that takes them is a capacity error."""
    from paper_2608_01657_gb300 import binding as B
    dev = torch.device("cuda")
    for max_requests, R, want in ((8, 9, B.PS_ERR_INVALID_ARG), (5000, 4097, B.PS_ERR_CAPACITY)):
        cache = B.Cache(64, 16, 2, "lru", B.Params(rho=(3.0,), beta=(9.0,)), max_requests=max_requests,
                        max_tokens=1024)
        g = torch.zeros(R, dtype=torch.int32, device=dev)
        o = torch.zeros(R + 1, dtype=torch.int64, device=dev)
        t = torch.zeros(4, dtype=torch.int32, device=dev)
        out = torch.zeros(R, dtype=torch.int32, device=dev)
        status = torch.zeros(1, dtype=torch.int32, device=dev)
        assert cache.cached_prefix_noalloc(g, o, t, out, status) == want
        if max_requests == 8:
            with pytest.raises(RuntimeError):
                cache.cached_prefix(g, o, t)


def test_noalloc_probe_block_limit_on_a_larger_handle():
    """On a handle whose per-step bound exceeds the fixed scratch (131072 full
    blocks), a call of exactly 131072 blocks equals ps_cached_prefix, and one
    block more makes the status an invalid-argument error."""
    from paper_2608_01657_gb300 import binding as B
    dev = torch.device("cuda")
    limit = 131072
    cache = B.Cache(4096, 16, 2, "lru", B.Params(rho=(3.0,), beta=(9.0,)), max_requests=4,
                    max_tokens=(limit + 64) * 16)
    rng = np.random.default_rng(5)
    head = rng.integers(0, W.VOCAB, size=64 * 16, dtype=np.int32)
    g1 = torch.zeros(1, dtype=torch.int32, device=dev)
    assert cache.step(1, g1, torch.tensor([0, head.size], dtype=torch.int64, device=dev),
                      torch.from_numpy(head).to(dev)) == 0
    for extra, ok in ((0, True), (1, False)):
        nb = limit + extra
        toks = np.concatenate([head, rng.integers(0, W.VOCAB, size=(nb - 64) * 16, dtype=np.int32)])
        o = torch.tensor([0, toks.size], dtype=torch.int64, device=dev)
        t = torch.from_numpy(toks).to(dev)
        out = torch.full((1,), -1, dtype=torch.int32, device=dev)
        status = torch.full((1,), 99, dtype=torch.int32, device=dev)
        assert cache.cached_prefix_noalloc(g1, o, t, out, status) == 0
        want, wst = cache.cached_prefix(g1, o, t)
        torch.cuda.synchronize()
        assert int(wst.item()) == 0 and int(want[0].item()) == 64
        if ok:
            assert int(status.item()) == 0 and int(out[0].item()) == 64
        else:
            assert int(status.item()) == B.PS_ERR_INVALID_ARG
