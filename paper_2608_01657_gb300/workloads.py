"""Seeded synthetic request traces for the prefix-cache step.

This module only draws inputs: token ids, group ids and request boundaries.
It holds none of the cache's arithmetic, so both the CUDA library's tests and
the CPU oracle's tests can feed on it.  Every step is reproducible from
``(seed, step)``: per-step draws come from ``numpy.random.default_rng`` seeded
with a tuple that names the stream, so no step depends on how many numbers an
earlier step consumed (the conversation generators carry only which
conversation is active, not generator state).

The five traces stand in for the paper's workloads (Sec. V-A): one-touch
pollution, two-pass replay and a chat-shaped benign mix (a synthetic stand-in
for ShareGPT, which is not used), plus a 1,048,576-block scale trace.  Token
ids are int32, uniform in [0, 32000).
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field
from typing import Dict, Iterator, List, Optional, Sequence

import numpy as np

VOCAB = 32000
_TAGS = {"labels": 1, "hot": 2, "fresh": 3, "atk": 4, "sys": 5, "conv": 6, "emit": 7, "pick": 8, "fuzz": 9, "burst": 10}


def _rng(seed: int, tag: str, *ids: int) -> np.random.Generator:
    return np.random.default_rng([int(seed) & 0xFFFFFFFF, _TAGS[tag]] + [int(i) for i in ids])


def _tokens(rng: np.random.Generator, n: int) -> np.ndarray:
    return rng.integers(0, VOCAB, size=int(n), dtype=np.int32)


def _lognormal_len(rng: np.random.Generator, mu: float, sigma: float, lo: int, hi: int) -> int:
    return int(min(hi, max(lo, int(round(float(rng.lognormal(mu, sigma)))))))


def _zipf_probs(n: int, s: float) -> np.ndarray:
    w = 1.0 / np.arange(1, n + 1, dtype=np.float64) ** s
    return w / w.sum()


@dataclass
class Step:
    """One batch of requests: CSR token layout, one group id per request."""
    index: int
    now: int
    groups: np.ndarray          # int32 [R]
    offsets: np.ndarray         # int64 [R+1]
    tokens: np.ndarray          # int32 [T]
    contracts: Optional[np.ndarray] = None   # int32 [R] or None
    prefixes: Optional[np.ndarray] = None    # uint64 [R] or None

    @property
    def num_requests(self) -> int:
        return int(self.groups.shape[0])

    @property
    def num_tokens(self) -> int:
        return int(self.offsets[-1])


@dataclass
class WorkloadSpec:
    name: str
    num_groups: int
    capacity_blocks: int
    block_size: int
    requests_per_step: int
    total_requests: int
    rho: Sequence[float]            # refill per tick per contract, in blocks
    beta: Sequence[float]           # burst capacity per contract, in blocks
    contract_of_group: Optional[Sequence[int]] = None
    description: str = ""

    @property
    def num_steps(self) -> int:
        return -(-self.total_requests // self.requests_per_step)


def _pack(index: int, groups: List[int], pieces: List[List[np.ndarray]]) -> Step:
    lens = np.fromiter((sum(len(p) for p in ps) for ps in pieces), dtype=np.int64, count=len(pieces))
    offsets = np.zeros(len(pieces) + 1, np.int64)
    np.cumsum(lens, out=offsets[1:])
    flat = [p for ps in pieces for p in ps]
    tokens = np.concatenate(flat).astype(np.int32, copy=False) if flat else np.zeros(0, np.int32)
    return Step(index=index, now=index + 1, groups=np.asarray(groups, np.int32), offsets=offsets, tokens=tokens)


class _Fresh:
    """Fresh (never repeated) tokens for one step, carved from one draw."""

    def __init__(self, seed: int, step: int, total: int):
        self.buf = _tokens(_rng(seed, "fresh", step), total)
        self.pos = 0

    def take(self, n: int) -> np.ndarray:
        out = self.buf[self.pos:self.pos + n]
        self.pos += n
        return out


class _Chat:
    """Chat-shaped benign traffic for one group: 4 system prompts of U[256,1024]
    tokens, 8 active conversations of Geometric(0.3) turns (at most 8), turn
    lengths lognormal(ln 200, 1.0) clipped to [1, 4096]; request k of a
    conversation sends the system prompt followed by turns 1..k."""

    SLOTS = 8

    def __init__(self, seed: int, group: int):
        self.seed, self.group = seed, group
        self.sys = []
        for j in range(4):
            r = _rng(seed, "sys", group, j)
            self.sys.append(_tokens(r, int(r.integers(256, 1025))))
        self.next_conv = 0
        self.slots = [self._new_conv() for _ in range(self.SLOTS)]

    def _new_conv(self) -> dict:
        cid = self.next_conv
        self.next_conv += 1
        r = _rng(self.seed, "conv", self.group, cid)
        turns = min(8, int(r.geometric(0.3)))
        lens = [_lognormal_len(r, np.log(200.0), 1.0, 1, 4096) for _ in range(turns)]
        return {"sys": int(r.integers(0, 4)), "turns": [_tokens(r, n) for n in lens], "k": 0}

    def emit(self, slot: int) -> List[np.ndarray]:
        c = self.slots[slot]
        c["k"] += 1
        pieces = [self.sys[c["sys"]]] + c["turns"][: c["k"]]
        if c["k"] >= len(c["turns"]):
            self.slots[slot] = self._new_conv()
        return pieces


class Workload:
    """Base class: iterate ``Step`` objects in order from step 0."""

    spec: WorkloadSpec

    def __init__(self, spec: WorkloadSpec, seed: int):
        self.spec, self.seed = spec, int(seed)

    def steps(self, count: Optional[int] = None) -> Iterator[Step]:
        n = self.spec.num_steps if count is None else min(count, self.spec.num_steps)
        for s in range(n):
            yield self.make_step(s)

    def _range(self, s: int):
        R = self.spec.requests_per_step
        lo = s * R
        return lo, min(self.spec.total_requests, lo + R)

    def make_step(self, s: int) -> Step:  # pragma: no cover - abstract
        raise NotImplementedError


class OneTouch(Workload):
    """Victim group 0 reuses hot prefixes (plus a fresh suffix); attacker group 1
    sends only fresh prompts (one-touch pollution, Sec. V-A)."""

    def __init__(self, spec, seed, hot_len, n_hot, zipf_s, victim_suffix, atk_len, n_victim, n_attacker,
                 replay=False):
        super().__init__(spec, seed)
        self.hot = [_tokens(_rng(seed, "hot", 0, j), hot_len) for j in range(n_hot)]
        self.zipf = _zipf_probs(n_hot, zipf_s) if zipf_s is not None else None
        self.victim_suffix, self.atk_len, self.replay = victim_suffix, atk_len, replay
        labels = np.array([0] * n_victim + [1] * n_attacker, np.int32)
        _rng(seed, "labels").shuffle(labels)
        self.labels = labels
        # Per-group running index so that group order is preserved.
        self.rank = np.zeros_like(labels)
        for g in (0, 1):
            idx = np.nonzero(labels == g)[0]
            self.rank[idx] = np.arange(len(idx))
        self.n_attacker_unique = n_attacker // 2 if replay else n_attacker

    def _attacker(self, k: int) -> np.ndarray:
        k = k % self.n_attacker_unique if self.replay else k
        r = _rng(self.seed, "atk", k)
        n = self.atk_len(r)
        return _tokens(r, n)

    def make_step(self, s: int) -> Step:
        lo, hi = self._range(s)
        groups, pieces, fresh_need = [], [], 0
        plan = []
        for q in range(lo, hi):
            g = int(self.labels[q])
            groups.append(g)
            if g == 0:
                fresh_need += self.victim_suffix
            plan.append((g, int(self.rank[q])))
        fresh = _Fresh(self.seed, s, fresh_need)
        pick = _rng(self.seed, "pick", s)
        for g, k in plan:
            if g == 0:
                j = 0 if self.zipf is None else int(pick.choice(len(self.hot), p=self.zipf))
                pieces.append([self.hot[j], fresh.take(self.victim_suffix)])
            else:
                pieces.append([self._attacker(k)])
        return _pack(s, groups, pieces)


class BenignChat(Workload):
    """Chat-shaped benign mix over all groups (stand-in for the ShareGPT trace)."""

    def __init__(self, spec, seed):
        super().__init__(spec, seed)
        self.chats = [_Chat(seed, g) for g in range(spec.num_groups)]

    def make_step(self, s: int) -> Step:
        lo, hi = self._range(s)
        r = _rng(self.seed, "emit", s)
        gs = r.integers(0, self.spec.num_groups, size=hi - lo)
        slots = r.integers(0, _Chat.SLOTS, size=hi - lo)
        pieces = [self.chats[int(g)].emit(int(k)) for g, k in zip(gs, slots)]
        return _pack(s, [int(g) for g in gs], pieces)


class Scale(Workload):
    """64 groups: 0-7 victims (zipf(1.1) over 64 hot 4096-token prefixes + 128
    fresh tokens), 8-15 attackers (fresh lognormal(ln 4096, 0.7) prompts clipped
    to [256, 32768]), 16-63 benign chat; request groups uniform over 64."""

    def __init__(self, spec, seed, n_victim_groups=8, n_attacker_groups=8, n_hot=64, hot_len=4096):
        super().__init__(spec, seed)
        self.nv, self.na = n_victim_groups, n_attacker_groups
        self.n_hot, self.hot_len = n_hot, hot_len
        self.zipf = _zipf_probs(n_hot, 1.1)
        self._hot: Dict[tuple, np.ndarray] = {}
        self.chats = {g: _Chat(seed, g) for g in range(self.nv + self.na, spec.num_groups)}
        self.atk_count = 0

    def _hot_prefix(self, g: int, j: int) -> np.ndarray:
        key = (g, j)
        if key not in self._hot:
            self._hot[key] = _tokens(_rng(self.seed, "hot", g, j), self.hot_len)
        return self._hot[key]

    def make_step(self, s: int) -> Step:
        lo, hi = self._range(s)
        r = _rng(self.seed, "emit", s)
        gs = r.integers(0, self.spec.num_groups, size=hi - lo)
        pick = _rng(self.seed, "pick", s)
        atk_lens = []
        for g in gs:
            if self.nv <= g < self.nv + self.na:
                atk_lens.append(_lognormal_len(pick, np.log(4096.0), 0.7, 256, 32768))
        n_victims = int(np.sum(gs < self.nv))
        fresh = _Fresh(self.seed, s, 128 * n_victims + int(sum(atk_lens)))
        hot_choice = pick.choice(self.n_hot, size=n_victims, p=self.zipf)
        pieces, vi, ai = [], 0, 0
        for g in gs:
            g = int(g)
            if g < self.nv:
                pieces.append([self._hot_prefix(g, int(hot_choice[vi])), fresh.take(128)])
                vi += 1
            elif g < self.nv + self.na:
                pieces.append([fresh.take(atk_lens[ai])])
                ai += 1
            else:
                pieces.append(self.chats[g].emit(int(pick.integers(0, _Chat.SLOTS))))
        return _pack(s, [int(g) for g in gs], pieces)


class LowAndSlow(Workload):
    """Low-and-slow rotation (Sec. V-A): the victim (group 0) sends one
    request per step, cycling through four 1536-token hot prefixes (96
    blocks each) plus a 32-token fresh suffix; the attacker (group 1) spreads
    one-touch pressure over time, one fresh 1536-token prompt every third
    step.  A prefix's reuse distance is three other victim requests (294
    blocks with their suffixes)."""

    def __init__(self, spec, seed, n_hot=4, hot_len=1536, suffix=32, atk_len=1536, atk_every=3):
        super().__init__(spec, seed)
        self.hot = [_tokens(_rng(seed, "hot", 0, j), hot_len) for j in range(n_hot)]
        self.suffix, self.atk_len, self.atk_every = suffix, atk_len, atk_every

    def make_step(self, s: int) -> Step:
        fresh = _Fresh(self.seed, s, self.suffix + self.atk_len)
        groups = [0]
        pieces = [[self.hot[s % len(self.hot)], fresh.take(self.suffix)]]
        if s % self.atk_every == self.atk_every - 1:
            groups.append(1)
            pieces.append([fresh.take(self.atk_len)])
        return _pack(s, groups, pieces)


class DelayedReplay(Workload):
    """Delayed replay (the debt-gate ablation of Sec. V-D), one group per
    contract of Sec. V-A: victim (group 0, critical 64/256), attacker
    (group 1, best-effort 16/128), neutral (group 2, standard 40/192).

    * steps 0-2: the victim admits three 1536-token hot prefixes (96 blocks
      each); steps 3-5 replay them, so they are proven and promoted;
    * step 6 (tick 7): the attacker bursts two fresh 1536-token prompts,
      192 blocks against a 128-block bucket: 64 blocks of debt, cleared by
      refill at tick 7 + ceil(64 / 16) = 11;
    * ``wait`` empty steps, then the attacker replays both prompts (tick
      8 + wait): every one of the 192 blocks is replay-eligible, gated while
      debt is outstanding (wait 0 or 1, the half-clearance point), promoted
      from wait 3 on (the designed clearance time);
    * ``pressure`` steps of neutral pressure: the neutral group sends one
      fresh 1536-token prompt, then the victim sends hot prefix k % 3.
    The pool holds 511 blocks, so the attack fits without eviction and the
    pressure steps reclaim."""

    VICTIM, ATTACKER, NEUTRAL = 0, 1, 2
    HOT, LEN = 3, 1536
    BURST_STEP = 6

    def __init__(self, spec, seed, wait=0, pressure=4):
        super().__init__(spec, seed)
        self.hot = [_tokens(_rng(seed, "hot", 0, j), self.LEN) for j in range(self.HOT)]
        self.atk = [_tokens(_rng(seed, "burst", 1, j), self.LEN) for j in range(2)]
        self.wait, self.pressure = int(wait), int(pressure)
        self.replay_step = self.BURST_STEP + 1 + self.wait

    @property
    def num_steps(self) -> int:
        return self.replay_step + 1 + self.pressure

    def steps(self, count: Optional[int] = None) -> Iterator[Step]:
        n = self.num_steps if count is None else min(count, self.num_steps)
        for s in range(n):
            yield self.make_step(s)

    def make_step(self, s: int) -> Step:
        if s < 2 * self.HOT:
            return _pack(s, [self.VICTIM], [[self.hot[s % self.HOT]]])
        if s == self.BURST_STEP or s == self.replay_step:
            return _pack(s, [self.ATTACKER] * 2, [[a] for a in self.atk])
        if s < self.replay_step:
            return _pack(s, [], [])
        k = s - self.replay_step - 1
        fresh = _Fresh(self.seed, s, self.LEN)
        return _pack(s, [self.NEUTRAL, self.VICTIM], [[fresh.take(self.LEN)], [self.hot[k % self.HOT]]])


def _lognormal_2048(r):
    return _lognormal_len(r, np.log(2048.0), 0.5, 256, 8192)


CONFIGS = {
    0: WorkloadSpec("tiny one-touch pollution", 2, 256, 16, 16, 2000, rho=(48,), beta=(144,),
                    description="victim: fixed 512-token hot prefix + 64 fresh; attacker: 1024 fresh; 16 req/step"),
    1: WorkloadSpec("4096-block one-touch pollution", 2, 4096, 16, 64, 20000, rho=(384,), beta=(1152,),
                    description="victim: zipf(1.0) over 8 hot 2048-token prefixes + 128 fresh; attacker: "
                                "lognormal(ln 2048, 0.5) in [256, 8192] fresh; 64 req/step"),
    2: WorkloadSpec("two-pass replay", 2, 4096, 16, 64, 40000, rho=(384,), beta=(1152,),
                    description="victim as the 4096-block one-touch trace; attacker: 10000 fresh prompts, "
                                "then the same 10000 again in order; 64 req/step"),
    3: WorkloadSpec("benign chat-shaped mix", 16, 65536, 16, 256, 200000, rho=(512,), beta=(1536,),
                    description="4 system prompts U[256,1024] per group, multi-turn histories; 256 req/step"),
    4: WorkloadSpec("scale", 64, 1 << 20, 16, 4096, 2000000, rho=(2000,), beta=(6000,),
                    description="8 victim, 8 attacker, 48 benign groups; 4096 req/step"),
    5: WorkloadSpec("low-and-slow rotation", 2, 511, 16, 2, 600, rho=(64, 16), beta=(256, 128),
                    contract_of_group=(0, 1),
                    description="victim: 4 hot 1536-token prefixes in rotation + 32 fresh, one a step; "
                                "attacker: one fresh 1536-token prompt every third step; 511 usable blocks"),
    6: WorkloadSpec("delayed replay", 3, 511, 16, 2, 18, rho=(64, 40, 16), beta=(256, 192, 128),
                    contract_of_group=(0, 2, 1),
                    description="victim admits and replays 3 hot 1536-token prefixes; attacker bursts 192 "
                                "blocks into 64 blocks of debt, waits, replays them; then 4 steps of neutral "
                                "pressure (one fresh 1536-token prompt) with victim re-requests; 511 blocks"),
}


def make_workload(config: int, seed: int = 1, requests_per_step: Optional[int] = None,
                  total_requests: Optional[int] = None, wait: int = 0,
                  attacker_prompts: Optional[int] = None) -> Workload:
    """The seeded trace of one configuration (0..6).  ``requests_per_step``
    overrides the batch size (e.g. the discriminative 8-request variants);
    ``wait`` is the delayed-replay trace's number of empty steps between the
    attacker's burst and its replay; ``attacker_prompts`` shortens the
    two-pass replay trace (config 2) to that many fresh attacker prompts
    replayed once, with as many victim requests (the same 1:1 mix), so its
    second pass starts within a short run."""
    spec = CONFIGS[config]
    if config == 2 and attacker_prompts is not None:
        total_requests = 4 * int(attacker_prompts)
    if requests_per_step is not None or total_requests is not None:
        spec = dataclasses.replace(
            spec,
            requests_per_step=requests_per_step or spec.requests_per_step,
            total_requests=total_requests or spec.total_requests)
    if config == 0:
        return OneTouch(spec, seed, hot_len=512, n_hot=1, zipf_s=None, victim_suffix=64,
                        atk_len=lambda r: 1024, n_victim=1000, n_attacker=1000)
    if config == 1:
        return OneTouch(spec, seed, hot_len=2048, n_hot=8, zipf_s=1.0, victim_suffix=128,
                        atk_len=_lognormal_2048, n_victim=10000, n_attacker=10000)
    if config == 2:
        half = spec.total_requests // 2
        return OneTouch(spec, seed, hot_len=2048, n_hot=8, zipf_s=1.0, victim_suffix=128,
                        atk_len=_lognormal_2048, n_victim=half, n_attacker=half, replay=True)
    if config == 3:
        return BenignChat(spec, seed)
    if config == 4:
        return Scale(spec, seed)
    if config == 5:
        return LowAndSlow(spec, seed)
    if config == 6:
        return DelayedReplay(spec, seed, wait=wait)
    raise KeyError(config)


# ---------------------------------------------------------------------------
# Small adversarial traces for parity and invariant tests.
def fuzz_steps(seed: int, num_groups: int, requests_per_step: int, num_steps: int, block_size: int = 16,
               docs_per_group: int = 4, doc_blocks: int = 12, fresh_max_blocks: int = 3,
               ragged: bool = True, with_contracts: int = 0, with_prefixes: bool = False,
               now_stride: int = 1, empty_every: int = 0) -> List[Step]:
    """Requests that share prefixes at random depths (shared in-step prefixes,
    repeated documents, orphans once the pool is small), optionally with a
    ragged token tail, per-request contracts and explicit prefix ids."""
    docs = [[_tokens(_rng(seed, "hot", g, d), doc_blocks * block_size) for d in range(docs_per_group)]
            for g in range(num_groups)]
    out = []
    now = 0
    for s in range(num_steps):
        r = _rng(seed, "fuzz", s)
        now += int(r.integers(0, now_stride + 1)) if now_stride > 1 else now_stride
        R = 0 if (empty_every and s % empty_every == empty_every - 1) else requests_per_step
        groups, pieces, contracts, prefixes = [], [], [], []
        for _ in range(R):
            g = int(r.integers(0, num_groups))
            d = int(r.integers(0, docs_per_group))
            depth = int(r.integers(0, doc_blocks + 1))
            toks = [docs[g][d][: depth * block_size]]
            nf = int(r.integers(0, fresh_max_blocks + 1))
            if nf:
                toks.append(_tokens(r, nf * block_size))
            if ragged:
                toks.append(_tokens(r, int(r.integers(0, block_size))))
            groups.append(g)
            pieces.append(toks)
            contracts.append(int(r.integers(0, with_contracts)) if with_contracts else 0)
            prefixes.append(int(d) + 1 + 1000 * g)
        st = _pack(s, groups, pieces)
        st.now = now
        if with_contracts:
            st.contracts = np.asarray(contracts, np.int32)
        if with_prefixes:
            st.prefixes = np.asarray(prefixes, np.uint64)
        out.append(st)
    return out
