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
    from paper_2608_01657_gb300 import binding as B
    dev = torch.device("cuda")
    cache = B.Cache(64, 16, 2, "lru", B.Params(rho=(3.0,), beta=(9.0,)), max_requests=8, max_tokens=1024)
    R = 4097
    g = torch.zeros(R, dtype=torch.int32, device=dev)
    o = torch.zeros(R + 1, dtype=torch.int64, device=dev)
    t = torch.zeros(4, dtype=torch.int32, device=dev)
    out = torch.zeros(R, dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    assert cache.cached_prefix_noalloc(g, o, t, out, status) == B.PS_ERR_CAPACITY
