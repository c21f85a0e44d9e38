"""The C-ABI library builds for sm_103a, loads without a GPU, and exports
every entry point that include/prefixshield.h declares (no compute calls)."""
import ctypes
import os
import re
import shutil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            txt = open(os.path.join(ROOT, "include", fn)).read()
            txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
            names |= set(re.findall(r"\b(ps_[a-z_0-9]+)\s*\(", txt))
    return sorted(names)


@pytest.fixture(scope="module")
def lib():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("no nvcc")
    from paper_2608_01657_gb300 import build
    return ctypes.CDLL(build.build())


def test_header_declares_the_step_api():
    d = _declared()
    for n in ("ps_workspace_bytes", "ps_create", "ps_step", "ps_step_host", "ps_stats", "ps_destroy"):
        assert n in d


def test_library_exports_every_declared_symbol(lib):
    missing = [n for n in _declared() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_covers_every_declared_symbol():
    from paper_2608_01657_gb300 import binding
    assert set(binding.EXPORTED) == set(_declared())


def test_workspace_size_is_host_computable(lib):
    from paper_2608_01657_gb300 import binding as B
    L = B.load()
    p = B.Params(rho=(2000.0,), beta=(6000.0,)).to_c(64)
    n = L.ps_workspace_bytes(1 << 20, 16, 64, ctypes.byref(p), 4096, 12_000_000)
    assert n > 0 and n % 256 == 0
    assert L.ps_workspace_bytes(1 << 20, 15, 64, ctypes.byref(p), 4096, 12_000_000) == 0  # odd block size
    assert L.ps_workspace_bytes(0, 16, 64, ctypes.byref(p), 4096, 12_000_000) == 0


def test_queue_flags_grow_the_workspace_by_the_log_buffers(lib):
    """PS_FLAG_INDEXED_QUEUES adds two buffers of 16 (N + max_tokens / bs)
    entries of 12 bytes (block id, stamp) plus per-step scratch."""
    from paper_2608_01657_gb300 import binding as B
    L = B.load()
    N, bs, G, R, T = 1 << 16, 16, 8, 256, 1 << 20
    base = B.Params(rho=(2.0,), beta=(6.0,)).to_c(G)
    q = B.Params(rho=(2.0,), beta=(6.0,), flags=B.PS_FLAG_INDEXED_QUEUES).to_c(G)
    n0 = L.ps_workspace_bytes(N, bs, G, ctypes.byref(base), R, T)
    n1 = L.ps_workspace_bytes(N, bs, G, ctypes.byref(q), R, T)
    P = 16 * (N + T // bs)
    assert n1 - n0 >= 2 * 12 * P
    assert n1 - n0 < 2 * 12 * P + (16 << 20)


def test_host_calls_refuse_bad_arguments_before_any_device_work(lib):
    """Null handles and out-of-range slots return PS_ERR_INVALID_ARG."""
    from paper_2608_01657_gb300 import binding as B
    L = B.load()
    assert L.ps_step_host_wait(None, 0) == B.PS_ERR_INVALID_ARG
    assert L.ps_step_host_async(None, None, 0, 1, 0, None, None, None, None, None, None) == B.PS_ERR_INVALID_ARG
    assert L.ps_step_host(None, None, 1, 0, None, None, None, None, None, None) == B.PS_ERR_INVALID_ARG
    assert L.ps_step(None, None, 1, 0, None, None, None, None, None, None) == B.PS_ERR_INVALID_ARG


def test_flag_and_status_constants_match_the_header():
    """The binding's and the oracle wrapper's PS_FLAG_* values are the
    header's (the oracle ignores the execution-choice flags, but tests pass
    the same bits to both sides)."""
    import oracle as O
    from paper_2608_01657_gb300 import binding as B
    txt = open(os.path.join(ROOT, "include", "prefixshield.h")).read()
    flags = {m.group(1): int(m.group(2)) for m in re.finditer(r"#define\s+PS_FLAG_([A-Z0-9_]+)\s+(\d+)u", txt)}
    assert flags, "no PS_FLAG_ definitions found"
    for name, value in flags.items():
        assert getattr(B, "PS_FLAG_" + name) == value, name
        assert getattr(O, "FLAG_" + name) == value, name
    assert len(set(flags.values())) == len(flags) and all(v & (v - 1) == 0 for v in flags.values())
    status = dict(re.findall(r"\b(PS_OK|PS_ERR_[A-Z_]+)\s*=\s*(-?\d+)", txt))
    for name in ("PS_OK", "PS_ERR_INVALID_ARG", "PS_ERR_CAPACITY", "PS_ERR_CLOCK", "PS_ERR_CUDA"):
        assert getattr(B, name) == int(status[name]), name


def test_s3fifo_layout_grows_with_the_pool_and_the_step(lib):
    """The S3-FIFO queue arrays and ghost rings are carved for every policy:
    the workspace grows with N (queue regions, ghost map and rings) and with
    max_tokens / bs (a step's pushes are room in the ghost ring)."""
    from paper_2608_01657_gb300 import binding as B
    L = B.load()
    p = B.Params(rho=(2.0,), beta=(6.0,)).to_c(4)
    a = L.ps_workspace_bytes(1 << 16, 16, 4, ctypes.byref(p), 64, 1 << 16)
    b = L.ps_workspace_bytes(1 << 17, 16, 4, ctypes.byref(p), 64, 1 << 16)
    c = L.ps_workspace_bytes(1 << 16, 16, 4, ctypes.byref(p), 64, 1 << 22)
    assert a > 0 and b > a and c > a
    # two buffers of two queue regions of N u32 ids: at least 16 B a block more
    assert b - a >= 16 * (1 << 16)
