"""The low-and-slow rotation trace (Sec. V-A, Sec. V-B) on the oracle.

The victim cycles through four 96-block hot prefixes, one request a step
with a 2-block fresh suffix, so a prefix comes back after three other victim
requests: 294 blocks.  That fixes two results exactly, whatever the policy's
details:
* StaticQuota's victim partition holds Q = floor(511 / 2) = 255 < 294
  blocks, so recency inside it evicts every prefix before its next use: no
  victim prefix hit after warm-up (the paper reports 0.00%);
* without the attacker every shared policy keeps the whole rotation (294 +
  2-block suffixes < 511): every victim request hits its full prefix.
Under the slow attack the paper's ordering holds on this trace: PrefixShield
keeps the victim's prefixes while global recency loses part of them.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_01657_gb300 import workloads as W

WARM = 8  # steps before every prefix has been used once


def _victim_hits(policy, attack=True, nsteps=150):
    wl = W.make_workload(5, seed=3)
    sp = wl.spec
    orc = O.OracleCache(sp.capacity_blocks, sp.block_size, sp.num_groups, policy,
                        O.Params(rho=sp.rho, beta=sp.beta, contract_of_group=list(sp.contract_of_group)))
    hits = []
    for k, st in enumerate(wl.steps(nsteps)):
        g, o, t = st.groups, st.offsets, st.tokens
        if not attack:
            g, o, t = g[:1], o[:2], t[: o[1]]
        assert g[0] == 0
        r = orc.step(st.now, g, o, t)
        assert r["status"] == 0
        if k >= WARM:
            hits.append(min(96, int(r["hit_blocks"][0])))
    return np.array(hits)


def test_staticquota_partition_is_shorter_than_the_rotation():
    assert (_victim_hits("staticquota") == 0).all()
    assert (_victim_hits("staticquota", attack=False) == 0).all()


@pytest.mark.parametrize("policy", ["lru", "s3fifo", "prefixshield"])
def test_shared_pool_keeps_the_rotation_without_attack(policy):
    assert (_victim_hits(policy, attack=False) == 96).all()


def test_prefixshield_keeps_the_victim_under_slow_attack():
    ps, lru = _victim_hits("prefixshield"), _victim_hits("lru")
    assert (ps == 96).all()
    assert lru.mean() < 96
