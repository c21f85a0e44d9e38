"""Thin ctypes binding of ``libprefixshield.so`` (C ABI: include/prefixshield.h).

Argument marshalling only: torch provides device memory and streams, every
stage of a step runs in the library's CUDA kernels.  ``load()`` raises when
the library has not been built; nothing here falls back to a CPU path.
"""
from __future__ import annotations

import ctypes as C
import os
from dataclasses import dataclass
from typing import Optional, Sequence

import numpy as np

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libprefixshield.so")

PS_MAX_CONTRACTS = 8
PS_MAX_GROUPS = 1024
PS_NUM_STATS = 15
STAT_NAMES = (
    "requests", "prompt_tokens", "full_blocks", "hit_blocks", "instep_hit_blocks",
    "hit_tokens", "admitted_blocks", "ungranted_blocks", "evicted_blocks",
    "invalidated_blocks", "promotions", "gated_reuses", "resident_blocks",
    "debt_raw", "debt_norm",
)
POLICIES = {"lru": 0, "s3fifo": 1, "prefixshield": 2, "staticquota": 3}
PS_OK, PS_ERR_INVALID_ARG, PS_ERR_CAPACITY, PS_ERR_CLOCK, PS_ERR_CUDA = 0, -1, -2, -3, -4
PS_FLAG_NO_SEGMENTATION, PS_FLAG_NO_DEBT_GATE, PS_FLAG_INDEXED_QUEUES, PS_FLAG_QUEUE_SHORT_WINDOWS = 1, 2, 4, 8
PS_FLAG_S3_COMPACT_GHOST, PS_FLAG_S3_SEQUENTIAL = 16, 32

EXPORTED = ("ps_workspace_bytes", "ps_create", "ps_step", "ps_step_host", "ps_step_host_async",
            "ps_step_host_wait", "ps_stats", "ps_clear_status",
            "ps_reset", "ps_destroy", "ps_status_string", "ps_export_state", "ps_export_history",
            "ps_export_ghost", "ps_set_stage_timing", "ps_get_stage_times", "ps_cached_prefix",
            "ps_cached_prefix_noalloc", "ps_uses_graph", "ps_set_graph")
PS_NUM_STAGES = 11
STAGE_NAMES = ("validate", "hash_lookup", "claims", "grant_instep", "meter", "touch_gate", "select",
               "take_lists", "evict", "insert", "commit")


class PsParams(C.Structure):
    _fields_ = [
        ("num_contracts", C.c_int32),
        ("fp_shift", C.c_int32),
        ("epsilon_fp", C.c_int64),
        ("rho_fp", C.c_int64 * PS_MAX_CONTRACTS),
        ("beta_fp", C.c_int64 * PS_MAX_CONTRACTS),
        ("contract_of_group", C.c_int32 * PS_MAX_GROUPS),
        ("hash_seed", C.c_uint64),
        ("s3_small_pct", C.c_int32),
        ("s3_freq_cap", C.c_int32),
        ("s3_move_min_freq", C.c_int32),
        ("pad0", C.c_int32),
        ("history_capacity", C.c_int64),
        ("flags", C.c_uint32),
        ("pad1", C.c_uint32),
    ]


OUT_ARRAYS = ("hit_blocks", "admitted_blocks", "admitted_offsets", "admitted_ids", "evicted_ids",
              "invalidated_ids", "counts", "debt_raw", "debt_norm")


class PsStepOut(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in OUT_ARRAYS] + [
        ("ids_capacity", C.c_int64), ("req_capacity", C.c_int32), ("pad", C.c_int32)]


def step_out(arrays: dict) -> PsStepOut:
    """The C output descriptor of a dict of arrays (device tensors or host
    numpy arrays): pointers, and the id lists' and per-request arrays' sizes."""
    def n(k):
        a = arrays.get(k)
        return 0 if a is None else int(a.shape[0])
    o = PsStepOut(**{k: _ptr(arrays.get(k)) for k in OUT_ARRAYS})
    o.ids_capacity = min(n("admitted_ids"), n("evicted_ids"), n("invalidated_ids"))
    o.req_capacity = min(n("hit_blocks"), n("admitted_blocks"), max(0, n("admitted_offsets") - 1))
    return o


class PsStateView(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in (
        "resident", "key", "group", "contract", "prefix", "klass", "stamp", "acc", "freq", "s3q", "s3seq",
        "balances")] + [("t_prev", C.c_int64), ("step", C.c_uint64), ("s3_ctr", C.c_uint64),
                        ("ghost_ctr", C.c_uint64)]


_lib = None


def load():
    """Load the CUDA library (built by ``paper_2608_01657_gb300.build``)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2608_01657_gb300.build.build()")
    L = C.CDLL(LIB_PATH)
    vp, i32, i64, u64, sz = C.c_void_p, C.c_int32, C.c_int64, C.c_uint64, C.c_size_t
    L.ps_workspace_bytes.restype = sz
    L.ps_workspace_bytes.argtypes = [i64, i32, i32, C.POINTER(PsParams), i32, i64]
    L.ps_create.restype = i32
    L.ps_create.argtypes = [C.POINTER(vp), i64, i32, i32, i32, C.POINTER(PsParams), vp, sz, i32, i64, vp]
    L.ps_step.restype = i32
    L.ps_step.argtypes = [vp, vp, i64, i32, vp, vp, vp, vp, vp, C.POINTER(PsStepOut)]
    L.ps_step_host.restype = i32
    L.ps_step_host.argtypes = [vp, vp, i64, i32, vp, vp, vp, vp, vp, C.POINTER(PsStepOut)]
    L.ps_step_host_async.restype = i32
    L.ps_step_host_async.argtypes = [vp, vp, i32, i64, i32, vp, vp, vp, vp, vp, C.POINTER(PsStepOut)]
    L.ps_step_host_wait.restype = i32
    L.ps_step_host_wait.argtypes = [vp, i32]
    L.ps_stats.restype = i32
    L.ps_stats.argtypes = [vp, vp, vp]
    L.ps_clear_status.restype = i32
    L.ps_clear_status.argtypes = [vp, vp]
    L.ps_reset.restype = i32
    L.ps_reset.argtypes = [vp, vp]
    L.ps_destroy.restype = None
    L.ps_destroy.argtypes = [vp]
    L.ps_status_string.restype = C.c_char_p
    L.ps_status_string.argtypes = [i32]
    L.ps_export_state.restype = i32
    L.ps_export_state.argtypes = [vp, vp, C.POINTER(PsStateView)]
    L.ps_export_history.restype = i64
    L.ps_export_history.argtypes = [vp, vp, vp, vp, vp, vp, i64]
    L.ps_export_ghost.restype = i64
    L.ps_export_ghost.argtypes = [vp, vp, vp, vp, vp, i64]
    L.ps_cached_prefix.restype = i32
    L.ps_cached_prefix.argtypes = [vp, vp, i32, vp, vp, vp, vp, vp]
    L.ps_cached_prefix_noalloc.restype = i32
    L.ps_cached_prefix_noalloc.argtypes = [vp, vp, i32, vp, vp, vp, vp, vp]
    L.ps_set_stage_timing.restype = i32
    L.ps_set_stage_timing.argtypes = [vp, i32]
    L.ps_get_stage_times.restype = i32
    L.ps_get_stage_times.argtypes = [vp, vp, i32, vp]
    L.ps_uses_graph.restype = i32
    L.ps_uses_graph.argtypes = [C.c_void_p]
    L.ps_set_graph.restype = i32
    L.ps_set_graph.argtypes = [C.c_void_p, i32]
    _lib = L
    return L


@dataclass
class Params:
    """Policy parameters in blocks; converted to fixed point (2^fp_shift)."""
    rho: Sequence[float] = (1.0,)
    beta: Sequence[float] = (1.0,)
    contract_of_group: Optional[Sequence[int]] = None
    epsilon_fp: int = 0
    fp_shift: int = 20
    hash_seed: int = 0x5EED
    s3_small_pct: int = 10
    s3_freq_cap: int = 3
    s3_move_min_freq: int = 2
    history_capacity: int = 1 << 20
    flags: int = 0
    rho_fp: Optional[Sequence[int]] = None
    beta_fp: Optional[Sequence[int]] = None

    def to_c(self, G: int) -> PsParams:
        p = PsParams()
        nc = len(self.rho if self.rho_fp is None else self.rho_fp)
        p.num_contracts = nc
        p.fp_shift = self.fp_shift
        p.epsilon_fp = self.epsilon_fp
        unit = 1 << self.fp_shift
        for c in range(nc):
            p.rho_fp[c] = int(self.rho_fp[c]) if self.rho_fp is not None else int(round(self.rho[c] * unit))
            p.beta_fp[c] = int(self.beta_fp[c]) if self.beta_fp is not None else int(round(self.beta[c] * unit))
        cog = self.contract_of_group or [0] * G
        for g in range(G):
            p.contract_of_group[g] = int(cog[g])
        p.hash_seed = self.hash_seed & ((1 << 64) - 1)
        p.s3_small_pct = self.s3_small_pct
        p.s3_freq_cap = self.s3_freq_cap
        p.s3_move_min_freq = self.s3_move_min_freq
        p.history_capacity = self.history_capacity
        p.flags = self.flags
        return p


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream_ptr(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


class Cache:
    """One multi-tenant block pool on the current CUDA device."""

    def __init__(self, capacity_blocks: int, block_size: int, num_groups: int, policy: str, params: Params,
                 max_requests: int, max_tokens: int, stream=None):
        import torch
        L = load()
        self.N, self.bs, self.G = int(capacity_blocks), int(block_size), int(num_groups)
        self.policy, self.params = policy, params
        self.max_requests, self.max_tokens = int(max_requests), int(max_tokens)
        self.max_blocks = self.max_tokens // self.bs
        self._p = params.to_c(self.G)
        self.C = self._p.num_contracts
        nbytes = L.ps_workspace_bytes(self.N, self.bs, self.G, C.byref(self._p), self.max_requests, self.max_tokens)
        if nbytes == 0:
            raise ValueError("invalid cache parameters")
        dev = torch.device("cuda", torch.cuda.current_device())
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        R, B, G = self.max_requests, max(1, self.max_blocks), self.G
        i32 = dict(dtype=torch.int32, device=dev)
        self.out = {
            "hit_blocks": torch.empty(max(1, R), **i32),
            "admitted_blocks": torch.empty(max(1, R), **i32),
            "admitted_offsets": torch.empty(R + 1, **i32),
            "admitted_ids": torch.empty(B, **i32),
            "evicted_ids": torch.empty(B, **i32),
            "invalidated_ids": torch.empty(B, **i32),
            "counts": torch.zeros(4, **i32),
            "debt_raw": torch.empty(G, dtype=torch.int64, device=dev),
            "debt_norm": torch.empty(G, dtype=torch.int64, device=dev),
        }
        self._out = step_out(self.out)
        h = C.c_void_p()
        rc = L.ps_create(C.byref(h), self.N, self.bs, self.G, POLICIES[policy], C.byref(self._p),
                         _ptr(self.workspace), nbytes, self.max_requests, self.max_tokens, _stream_ptr(stream))
        if rc != PS_OK:
            raise RuntimeError(f"ps_create failed: {L.ps_status_string(rc).decode()} ({rc})")
        self._h = h

    def close(self):
        if getattr(self, "_h", None):
            load().ps_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- the step ---------------------------------------------------------
    def step(self, now: int, groups, offsets, tokens, contracts=None, prefixes=None, stream=None) -> int:
        """Enqueue one step on device tensors; results land in ``self.out``."""
        R = int(groups.shape[0])
        return load().ps_step(self._h, _stream_ptr(stream), int(now), R, _ptr(groups), _ptr(offsets), _ptr(tokens),
                              _ptr(contracts), _ptr(prefixes), C.byref(self._out))

    def cached_prefix(self, groups, offsets, tokens, out=None, status=None, stream=None):
        """Read-only probe: leading resident full blocks of each prompt (device
        tensors in, device int32 counts out).  Returns (counts, status tensor)."""
        import torch
        R = int(groups.shape[0])
        if out is None:
            out = torch.empty(max(1, R), dtype=torch.int32, device=groups.device)
        if status is None:
            status = torch.zeros(1, dtype=torch.int32, device=groups.device)
        rc = load().ps_cached_prefix(self._h, _stream_ptr(stream), R, _ptr(groups), _ptr(offsets), _ptr(tokens),
                                     _ptr(out), _ptr(status))
        if rc != PS_OK:
            raise RuntimeError(f"ps_cached_prefix failed ({rc})")
        return out, status

    def cached_prefix_noalloc(self, groups, offsets, tokens, out, status, stream=None) -> int:
        """The same probe with the library's fixed scratch array: allocates
        nothing (the caller supplies ``out`` and ``status``).  Returns the rc."""
        R = int(groups.shape[0])
        return load().ps_cached_prefix_noalloc(self._h, _stream_ptr(stream), R, _ptr(groups), _ptr(offsets),
                                               _ptr(tokens), _ptr(out), _ptr(status))

    def step_host(self, now: int, groups, offsets, tokens, contracts=None, prefixes=None, stream=None,
                  out: Optional[dict] = None) -> dict:
        """The end-to-end call: host (ideally pinned) inputs and outputs."""
        R = int(len(groups))
        if out is None:
            out = host_outputs(R, self.max_blocks, self.G)
        o = step_out(out)
        rc = load().ps_step_host(self._h, _stream_ptr(stream), int(now), R, _ptr(groups), _ptr(offsets),
                                 _ptr(tokens), _ptr(contracts), _ptr(prefixes), C.byref(o))
        out["rc"] = rc
        return out

    def step_host_async(self, slot: int, now: int, groups, offsets, tokens, out: dict, contracts=None,
                        prefixes=None, stream=None) -> int:
        """Pipelined end-to-end call: enqueue a step from host buffers on
        staging slot 0 or 1 and return at once.  ``out`` must come from
        ``host_outputs(..., pinned=True)``; inputs and ``out`` must stay
        alive and unchanged until ``step_host_wait(slot)``."""
        R = int(len(groups))
        o = step_out(out)
        out["_keep"] = (o, groups, offsets, tokens, contracts, prefixes)
        return load().ps_step_host_async(self._h, _stream_ptr(stream), int(slot), int(now), R, _ptr(groups),
                                         _ptr(offsets), _ptr(tokens), _ptr(contracts), _ptr(prefixes), C.byref(o))

    def step_host_wait(self, slot: int) -> int:
        """Wait for the step on ``slot``; returns its status."""
        return load().ps_step_host_wait(self._h, int(slot))

    def fetch(self, R: int, stream=None) -> dict:
        """Copy the last step's outputs to host numpy arrays (synchronizes)."""
        import torch
        torch.cuda.current_stream().synchronize() if stream is None else stream.synchronize()
        counts = self.out["counts"].cpu().numpy()
        res = {"status": int(counts[3])}
        if counts[3] != PS_OK:
            return res
        res["hit_blocks"] = self.out["hit_blocks"][:R].cpu().numpy()
        res["admitted_blocks"] = self.out["admitted_blocks"][:R].cpu().numpy()
        res["admitted_offsets"] = self.out["admitted_offsets"][: R + 1].cpu().numpy()
        res["admitted_ids"] = self.out["admitted_ids"][: counts[0]].cpu().numpy()
        res["evicted_ids"] = self.out["evicted_ids"][: counts[1]].cpu().numpy()
        res["invalidated_ids"] = self.out["invalidated_ids"][: counts[2]].cpu().numpy()
        res["debt_raw"] = self.out["debt_raw"].cpu().numpy()
        res["debt_norm"] = self.out["debt_norm"].cpu().numpy()
        return res

    def stats(self, stream=None) -> np.ndarray:
        s = np.zeros((self.G, PS_NUM_STATS), np.int64)
        rc = load().ps_stats(self._h, _stream_ptr(stream), _ptr(s))
        if rc not in (PS_OK, PS_ERR_CAPACITY):
            raise RuntimeError(f"ps_stats failed ({rc})")
        return s

    def set_stage_timing(self, enable: bool = True):
        rc = load().ps_set_stage_timing(self._h, int(enable))
        if rc != PS_OK:
            raise RuntimeError(f"ps_set_stage_timing failed ({rc})")

    def set_graph(self, enable: bool = True):
        """Replay the step as one CUDA graph (default) or launch kernel by kernel."""
        rc = load().ps_set_graph(self._h, int(enable))
        if rc != PS_OK:
            raise RuntimeError(f"ps_set_graph failed ({rc})")

    def uses_graph(self) -> bool:
        """True once the step replays one captured CUDA graph."""
        rc = load().ps_uses_graph(self._h)
        if rc < 0:
            raise RuntimeError(f"ps_uses_graph failed ({rc})")
        return rc == 1

    def stage_times(self):
        """(per-stage ms of the last timed step, kernel launches of that step)."""
        ms = np.zeros(PS_NUM_STAGES, np.float32)
        nl = np.zeros(1, np.int32)
        n = load().ps_get_stage_times(self._h, _ptr(ms), PS_NUM_STAGES, _ptr(nl))
        if n < 0:
            raise RuntimeError(f"ps_get_stage_times failed ({n})")
        return ms[:n].copy(), int(nl[0])

    def clear_status(self, stream=None):
        return load().ps_clear_status(self._h, _stream_ptr(stream))

    def reset(self, stream=None):
        return load().ps_reset(self._h, _stream_ptr(stream))

    def export(self, stream=None) -> dict:
        N = self.N
        d = {
            "resident": np.zeros(N, np.uint8), "key": np.zeros(N, np.uint64),
            "group": np.zeros(N, np.int32), "contract": np.zeros(N, np.int32),
            "prefix": np.zeros(N, np.uint64), "klass": np.zeros(N, np.int32),
            "stamp": np.zeros(N, np.uint64), "acc": np.zeros(N, np.uint32),
            "freq": np.zeros(N, np.int32), "s3q": np.zeros(N, np.int32),
            "s3seq": np.zeros(N, np.uint64),
        }
        B = np.zeros(self.G * self.C, np.int64)
        v = PsStateView(**{k: _ptr(d[k]) for k in d}, balances=_ptr(B))
        rc = load().ps_export_state(self._h, _stream_ptr(stream), C.byref(v))
        if rc != PS_OK:
            raise RuntimeError(f"ps_export_state failed ({rc})")
        d["B"] = B.reshape(self.G, self.C)
        d["t_prev"], d["step"], d["s3_ctr"], d["ghost_ctr"] = int(v.t_prev), int(v.step), int(v.s3_ctr), int(v.ghost_ctr)
        L = load()
        n = L.ps_export_history(self._h, _stream_ptr(stream), None, None, None, None, 0)
        hg, hp = np.zeros(n, np.int32), np.zeros(n, np.uint64)
        hr, ha = np.zeros(n, np.uint64), np.zeros(n, np.uint8)
        L.ps_export_history(self._h, _stream_ptr(stream), _ptr(hg), _ptr(hp), _ptr(hr), _ptr(ha), n)
        o = np.lexsort((hp, hg))
        d["history"] = (hg[o], hp[o], hr[o], ha[o])
        n = L.ps_export_ghost(self._h, _stream_ptr(stream), None, None, None, 0)
        gg, gk, gs = np.zeros(n, np.int32), np.zeros(n, np.uint64), np.zeros(n, np.uint64)
        L.ps_export_ghost(self._h, _stream_ptr(stream), _ptr(gg), _ptr(gk), _ptr(gs), n)
        o = np.lexsort((gk, gg))
        d["ghost"] = (gg[o], gk[o], gs[o])
        return d


def host_outputs(R: int, max_blocks: int, G: int, pinned: bool = False) -> dict:
    """Host buffers for ``Cache.step_host`` (optionally page-locked)."""
    import torch

    def buf(n, dt):
        t = torch.empty(max(1, n), dtype=dt, pin_memory=pinned)
        return t.numpy()

    return {
        "hit_blocks": buf(R, torch.int32), "admitted_blocks": buf(R, torch.int32),
        "admitted_offsets": buf(R + 1, torch.int32), "admitted_ids": buf(max_blocks, torch.int32),
        "evicted_ids": buf(max_blocks, torch.int32), "invalidated_ids": buf(max_blocks, torch.int32),
        "counts": buf(4, torch.int32), "debt_raw": buf(G, torch.int64), "debt_norm": buf(G, torch.int64),
    }
