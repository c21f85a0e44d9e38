"""ctypes binding of the CPU oracle.

TEST INFRASTRUCTURE ONLY: the plain, sequential statement of the PrefixShield
prefix-cache step (``prefixshield_oracle.cpp``).  Only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may use
it; the CUDA library never does.  This module defines its own parameter block
and output layout and imports nothing from the CUDA package.
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass, field
from typing import Optional, Sequence

import numpy as np

from .build import build_oracle

MAX_CONTRACTS = 8
MAX_GROUPS = 1024
NUM_STATS = 15
STAT_NAMES = (
    "requests", "prompt_tokens", "full_blocks", "hit_blocks", "instep_hit_blocks",
    "hit_tokens", "admitted_blocks", "ungranted_blocks", "evicted_blocks",
    "invalidated_blocks", "promotions", "gated_reuses", "resident_blocks",
    "debt_raw", "debt_norm",
)
POLICIES = {"lru": 0, "s3fifo": 1, "prefixshield": 2, "staticquota": 3}
OK, ERR_INVALID_ARG, ERR_CAPACITY, ERR_CLOCK = 0, -1, -2, -3
FLAG_NO_SEGMENTATION, FLAG_NO_DEBT_GATE = 1, 2
# the CUDA library's indexed-queue victim selection: same victims, ignored here
FLAG_INDEXED_QUEUES = 4
FLAG_QUEUE_SHORT_WINDOWS = 8
# the CUDA library's S3-FIFO execution choices: same results, ignored here
FLAG_S3_COMPACT_GHOST = 16
FLAG_S3_SEQUENTIAL = 32


class OrcParams(C.Structure):
    _fields_ = [
        ("num_contracts", C.c_int32),
        ("fp_shift", C.c_int32),
        ("epsilon_fp", C.c_int64),
        ("rho_fp", C.c_int64 * MAX_CONTRACTS),
        ("beta_fp", C.c_int64 * MAX_CONTRACTS),
        ("contract_of_group", C.c_int32 * MAX_GROUPS),
        ("hash_seed", C.c_uint64),
        ("s3_small_pct", C.c_int32),
        ("s3_freq_cap", C.c_int32),
        ("s3_move_min_freq", C.c_int32),
        ("pad0", C.c_int32),
        ("history_capacity", C.c_int64),
        ("flags", C.c_uint32),
        ("pad1", C.c_uint32),
    ]


class OrcOut(C.Structure):
    _fields_ = [
        ("hit_blocks", C.c_void_p),
        ("admitted_blocks", C.c_void_p),
        ("admitted_offsets", C.c_void_p),
        ("admitted_ids", C.c_void_p),
        ("evicted_ids", C.c_void_p),
        ("invalidated_ids", C.c_void_p),
        ("debt_raw", C.c_void_p),
        ("debt_norm", C.c_void_p),
        ("n_admitted", C.c_int32),
        ("n_evicted", C.c_int32),
        ("n_invalidated", C.c_int32),
        ("status", C.c_int32),
    ]


_lib = None


def lib():
    global _lib
    if _lib is None:
        L = C.CDLL(build_oracle())
        vp, i32, i64, u64 = C.c_void_p, C.c_int32, C.c_int64, C.c_uint64
        L.orc_check_params.restype = i32
        L.orc_check_params.argtypes = [i64, i32, i32, i32, C.POINTER(OrcParams)]
        L.orc_create.restype = vp
        L.orc_create.argtypes = [i64, i32, i32, i32, C.POINTER(OrcParams)]
        L.orc_destroy.argtypes = [vp]
        L.orc_step.restype = i32
        L.orc_step.argtypes = [vp, i64, i32, vp, vp, vp, vp, vp, C.POINTER(OrcOut)]
        L.orc_clear_status.argtypes = [vp]
        L.orc_cached_prefix.argtypes = [vp, i32, vp, vp, vp, vp]
        L.orc_stats.argtypes = [vp, vp]
        L.orc_export_blocks.argtypes = [vp] + [vp] * 11
        L.orc_export_ledger.argtypes = [vp, vp, vp, vp, vp, vp]
        L.orc_export_history.restype = i64
        L.orc_export_history.argtypes = [vp, vp, vp, vp, vp]
        L.orc_export_ghost.restype = i64
        L.orc_export_ghost.argtypes = [vp, vp, vp, vp]
        L.orc_splitmix64_next.restype = u64
        L.orc_splitmix64_next.argtypes = [C.POINTER(C.c_uint64)]
        L.orc_mix64.restype = u64
        L.orc_mix64.argtypes = [u64]
        L.orc_nh.restype = u64
        L.orc_nh.argtypes = [vp, i32, vp, i32]
        L.orc_chain_keys.restype = i64
        L.orc_chain_keys.argtypes = [u64, i32, i32, vp, i64, vp]
        L.orc_make_stamp.restype = u64
        L.orc_make_stamp.argtypes = [u64, u64, u64, u64]
        L.orc_alg2_loop.restype = i64
        L.orc_alg2_loop.argtypes = [i32, vp, vp, i64, vp, vp, i64, vp, vp]
        _lib = L
    return _lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


@dataclass
class Params:
    """Policy parameters; rates and balances are in blocks (scaled by 2^fp_shift inside)."""
    rho: Sequence[float] = (1.0,)           # refill per accounting tick, per contract (Eq. 1)
    beta: Sequence[float] = (1.0,)          # burst capacity per contract (Eq. 1)
    contract_of_group: Optional[Sequence[int]] = None
    epsilon_fp: int = 0
    fp_shift: int = 20
    hash_seed: int = 0x5EED
    s3_small_pct: int = 10
    s3_freq_cap: int = 3
    s3_move_min_freq: int = 2
    history_capacity: int = 1 << 20
    flags: int = 0
    rho_fp: Optional[Sequence[int]] = None  # exact fixed-point overrides
    beta_fp: Optional[Sequence[int]] = None

    def to_c(self, G: int) -> OrcParams:
        p = OrcParams()
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


class OracleCache:
    """One prefix-cache pool driven step by step on the host CPU."""

    def __init__(self, capacity_blocks: int, block_size: int, num_groups: int, policy: str, params: Params):
        self.N, self.bs, self.G = int(capacity_blocks), int(block_size), int(num_groups)
        self.policy = policy
        self.params = params
        self._p = params.to_c(self.G)
        self.C = self._p.num_contracts
        self._h = lib().orc_create(self.N, self.bs, self.G, POLICIES[policy], C.byref(self._p))
        if not self._h:
            raise ValueError("oracle rejected the parameters")

    def __del__(self):
        h = getattr(self, "_h", None)
        if h:
            lib().orc_destroy(h)
            self._h = None

    def step(self, now: int, groups, offsets, tokens, contracts=None, prefixes=None):
        g = np.ascontiguousarray(groups, dtype=np.int32)
        o = np.ascontiguousarray(offsets, dtype=np.int64)
        t = np.ascontiguousarray(tokens, dtype=np.int32)
        c = None if contracts is None else np.ascontiguousarray(contracts, dtype=np.int32)
        p = None if prefixes is None else np.ascontiguousarray(prefixes, dtype=np.uint64)
        R = len(g)
        cap = max(1, int(o[-1]) // self.bs if R else 1)
        res = {
            "hit_blocks": np.zeros(R, np.int32),
            "admitted_blocks": np.zeros(R, np.int32),
            "admitted_offsets": np.zeros(R + 1, np.int32),
            "admitted_ids": np.zeros(cap, np.int32),
            "evicted_ids": np.zeros(cap, np.int32),
            "invalidated_ids": np.zeros(cap, np.int32),
            "debt_raw": np.zeros(self.G, np.int64),
            "debt_norm": np.zeros(self.G, np.int64),
        }
        out = OrcOut()
        for k in ("hit_blocks", "admitted_blocks", "admitted_offsets", "admitted_ids",
                  "evicted_ids", "invalidated_ids", "debt_raw", "debt_norm"):
            setattr(out, k, _ptr(res[k]))
        st = lib().orc_step(self._h, int(now), R, _ptr(g), _ptr(o), _ptr(t), _ptr(c), _ptr(p), C.byref(out))
        res["status"] = int(st)
        if st != OK:
            return res
        res["admitted_ids"] = res["admitted_ids"][: out.n_admitted].copy()
        res["evicted_ids"] = res["evicted_ids"][: out.n_evicted].copy()
        res["invalidated_ids"] = res["invalidated_ids"][: out.n_invalidated].copy()
        return res

    def cached_prefix(self, groups, offsets, tokens) -> np.ndarray:
        g = np.ascontiguousarray(groups, dtype=np.int32)
        o = np.ascontiguousarray(offsets, dtype=np.int64)
        t = np.ascontiguousarray(tokens, dtype=np.int32)
        out = np.zeros(max(1, len(g)), np.int32)
        lib().orc_cached_prefix(self._h, len(g), _ptr(g), _ptr(o), _ptr(t), _ptr(out))
        return out[: len(g)]

    def clear_status(self):
        lib().orc_clear_status(self._h)

    def stats(self) -> np.ndarray:
        s = np.zeros((self.G, NUM_STATS), np.int64)
        lib().orc_stats(self._h, _ptr(s))
        return s

    def export(self) -> dict:
        N = self.N
        d = {
            "resident": np.zeros(N, np.uint8), "key": np.zeros(N, np.uint64),
            "group": np.zeros(N, np.int32), "contract": np.zeros(N, np.int32),
            "prefix": np.zeros(N, np.uint64), "klass": np.zeros(N, np.int32),
            "stamp": np.zeros(N, np.uint64), "acc": np.zeros(N, np.uint32),
            "freq": np.zeros(N, np.int32), "s3q": np.zeros(N, np.int32),
            "s3seq": np.zeros(N, np.uint64),
        }
        lib().orc_export_blocks(self._h, *[_ptr(d[k]) for k in (
            "resident", "key", "group", "contract", "prefix", "klass", "stamp", "acc", "freq", "s3q", "s3seq")])
        B = np.zeros(self.G * self.C, np.int64)
        tp, stp, s3c, ghc = (np.zeros(1, np.int64), np.zeros(1, np.uint64),
                             np.zeros(1, np.uint64), np.zeros(1, np.uint64))
        lib().orc_export_ledger(self._h, _ptr(B), _ptr(tp), _ptr(stp), _ptr(s3c), _ptr(ghc))
        d["B"] = B.reshape(self.G, self.C)
        d["t_prev"], d["step"], d["s3_ctr"], d["ghost_ctr"] = int(tp[0]), int(stp[0]), int(s3c[0]), int(ghc[0])
        nh = lib().orc_export_history(self._h, None, None, None, None)
        hg, hp = np.zeros(nh, np.int32), np.zeros(nh, np.uint64)
        hr, ha = np.zeros(nh, np.uint64), np.zeros(nh, np.uint8)
        lib().orc_export_history(self._h, _ptr(hg), _ptr(hp), _ptr(hr), _ptr(ha))
        d["history"] = (hg, hp, hr, ha)
        ng = lib().orc_export_ghost(self._h, None, None, None)
        gg, gk, gs = np.zeros(ng, np.int32), np.zeros(ng, np.uint64), np.zeros(ng, np.uint64)
        lib().orc_export_ghost(self._h, _ptr(gg), _ptr(gk), _ptr(gs))
        d["ghost"] = (gg, gk, gs)
        return d


# ---- building blocks, exposed for the pin tests ----------------------------
def splitmix64_stream(seed: int, n: int):
    st = C.c_uint64(seed & ((1 << 64) - 1))
    return [int(lib().orc_splitmix64_next(C.byref(st))) for _ in range(n)]


def mix64(z: int) -> int:
    return int(lib().orc_mix64(z & ((1 << 64) - 1)))


def nh(key_words, off: int, message, bs: int) -> int:
    K = np.ascontiguousarray(key_words, dtype=np.uint32)
    M = np.ascontiguousarray(message, dtype=np.int32)
    return int(lib().orc_nh(_ptr(K), off, _ptr(M), bs))


def chain_keys(seed: int, group: int, bs: int, tokens) -> np.ndarray:
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    out = np.zeros(max(1, len(t) // bs), np.uint64)
    n = lib().orc_chain_keys(seed & ((1 << 64) - 1), group, bs, _ptr(t), len(t), _ptr(out))
    return out[:n].copy()


def make_stamp(base: int, blocks_before: int, n: int, m: int) -> int:
    return int(lib().orc_make_stamp(base, blocks_before, n, m))


def alg2_loop(P, delta, eps, queues, m):
    """Literal Alg. 2 loop on abstract inputs; returns [(group, index_in_group), ...]."""
    G = len(P)
    P = np.ascontiguousarray(P, dtype=np.int64)
    delta = np.ascontiguousarray(delta, dtype=np.int64)
    qoff = np.zeros(G + 1, np.int64)
    for g in range(G):
        qoff[g + 1] = qoff[g] + len(queues[g])
    qkeys = np.ascontiguousarray(np.concatenate([np.asarray(q, np.uint64) for q in queues]) if G else [], np.uint64)
    og, oi = np.zeros(max(1, m), np.int32), np.zeros(max(1, m), np.int64)
    k = lib().orc_alg2_loop(G, _ptr(P), _ptr(delta), int(eps), _ptr(qoff), _ptr(qkeys), int(m), _ptr(og), _ptr(oi))
    return [(int(og[v]), int(oi[v])) for v in range(k)]
