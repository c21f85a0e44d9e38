"""Helpers shared by the test files (trace parsing, hand-built steps)."""
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def obj_tokens(name: str, bs: int = 16, blocks: int = 1) -> np.ndarray:
    """Deterministic, distinct token content for a named object."""
    base = 0
    for c in name:
        base = (base * 131 + ord(c)) % 1000003
    return np.array([(base * 7 + 13 * j) % 32000 for j in range(bs * blocks)], np.int32)


def make_step(prompts, groups=None, now=1):
    """prompts: list of int32 token arrays -> (groups, offsets, tokens, now)."""
    R = len(prompts)
    groups = np.zeros(R, np.int32) if groups is None else np.asarray(groups, np.int32)
    offs = np.zeros(R + 1, np.int64)
    for i, p in enumerate(prompts):
        offs[i + 1] = offs[i] + len(p)
    toks = np.concatenate(prompts).astype(np.int32) if R else np.zeros(0, np.int32)
    return groups, offs, toks, now


def parse_trace(fname):
    steps, final = [], {}
    for line in open(os.path.join(GOLDEN, fname)):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        if line.startswith("final"):
            k, v = line.split(":", 1)
            final[k.strip()] = v.split()
            continue
        parts = [p.strip() for p in line.split("|")]
        reqs = parts[1].split()
        hits = [int(x) for x in parts[2].split()]
        ev = [] if parts[3] == "-" else parts[3].split()
        steps.append((reqs, hits, ev))
    return steps, final


def params_line(fname):
    for line in open(os.path.join(GOLDEN, fname)):
        if line.startswith("# params:"):
            kv = {}
            for tok in line.split(":", 1)[1].split():
                if "=" in tok:
                    k, v = tok.split("=")
                    kv[k] = int(v)
            return kv
    return {}


# ---------------------------------------------------------------------------
# Invariant checker: given the state before and after one oracle step and the
# step's outputs, check what the paper fixes (I1, work conservation, fixed
# ownership, non-negative debt) and, for lru and prefixshield, that the victim
# set equals an independent closed form computed from the pre-step state.
def chain_keys_of(seed, step, bs):
    import oracle as O
    out = []
    for i in range(len(step[0])):
        g = int(step[0][i])
        toks = step[2][step[1][i]:step[1][i + 1]]
        out.append(O.chain_keys(seed, g, bs, toks))
    return out


def alg2_closed_form(P, delta, eps, queues, m):
    """Water-filling reading of Alg. 2: every eligible (group, j) item has the
    projected value P_g - j*delta_g (> eps); items are taken in order of value
    descending, ties by the candidate key; the rest come from the global
    fallback in key order.  Returns [(group, index)] in selection order."""
    items = []
    for g, q in enumerate(queues):
        j = 0
        while j < len(q) and P[g] - j * delta[g] > eps:
            items.append((-(P[g] - j * delta[g]), int(q[j]), g, j))
            j += 1
    items.sort()
    sel = [(g, j) for _, _, g, j in items[:m]]
    taken = {}
    for g, j in sel:
        taken[g] = max(taken.get(g, 0), j + 1)
    rest = sorted((int(q[j]), g, j) for g, q in enumerate(queues) for j in range(taken.get(g, 0), len(q)))
    sel += [(g, j) for _, g, j in rest[: m - len(sel)]]
    return sel


def check_step(oc, before, after, step_inputs, res, policy):
    import oracle as O
    N, bs = oc.N, oc.bs
    groups, offsets, tokens = step_inputs[0], step_inputs[1], step_inputs[2]
    R = len(groups)
    assert res["status"] == 0
    keys = chain_keys_of(oc.params.hash_seed, (groups, offsets, tokens), bs)
    n = np.array([len(k) for k in keys], np.int64)
    hit = res["hit_blocks"].astype(np.int64)
    adm = res["admitted_blocks"].astype(np.int64)
    assert np.all(hit >= 0) and np.all(adm >= 0) and np.all(hit + adm <= n)
    offs = res["admitted_offsets"]
    assert offs[0] == 0 and np.array_equal(np.diff(offs), adm)
    A, E, I = res["admitted_ids"], res["evicted_ids"], res["invalidated_ids"]
    assert len(A) == adm.sum()
    for arr in (A, E, I):
        assert np.all(np.diff(arr) > 0) and (len(arr) == 0 or (arr[0] >= 0 and arr[-1] < N))
    assert not set(E.tolist()) & set(I.tolist())
    # resident map before the step
    res_before = {(int(before["group"][b]), int(before["key"][b])): b for b in range(N) if before["resident"][b]}
    pinned = set()
    hres = np.zeros(R, np.int64)
    for i in range(R):
        g = int(groups[i])
        while hres[i] < n[i] and (g, int(keys[i][hres[i]])) in res_before:
            pinned.add(res_before[(g, int(keys[i][hres[i]]))])
            hres[i] += 1
    assert np.all(hres <= hit)
    assert not (set(E.tolist()) | set(I.tolist())) & pinned
    for b in list(E) + list(I):
        assert before["resident"][b]
    n_res_before = int(before["resident"].sum())
    free_after_inval = N - n_res_before + len(I)
    need = int(adm.sum())
    # work conservation: evict only what free blocks cannot cover
    assert len(E) == max(0, need - free_after_inval)
    free_ids = sorted(set(np.nonzero(before["resident"] == 0)[0].tolist()) | set(I.tolist()))
    want_alloc = sorted(free_ids[: min(need, len(free_ids))] + E.tolist())
    assert A.tolist() == want_alloc
    assert int(after["resident"].sum()) == n_res_before - len(E) - len(I) + need
    # ownership never changes while resident
    for b in range(N):
        if before["resident"][b] and after["resident"][b] and before["key"][b] == after["key"][b]:
            assert before["group"][b] == after["group"][b]
            assert before["contract"][b] == after["contract"][b]
            assert before["prefix"][b] == after["prefix"][b]
    # debt is never negative; normalization only shrinks it
    assert np.all(res["debt_raw"] >= 0) and np.all(res["debt_norm"] >= 0)
    assert np.all(res["debt_norm"] <= res["debt_raw"])
    # I1: the ledger moved by the refill and by exactly the admitted blocks
    unit = 1 << oc.params.fp_shift
    p = oc._p
    C = oc.C
    dt = step_inputs[3] - before["t_prev"]
    contracts = step_inputs[4] if len(step_inputs) > 4 and step_inputs[4] is not None else None
    charged = np.zeros((oc.G, C), np.int64)
    for i in range(R):
        c = int(contracts[i]) if contracts is not None else int(p.contract_of_group[int(groups[i])])
        charged[int(groups[i]), c] += adm[i]
    for g in range(oc.G):
        for c in range(C):
            refilled = min(p.beta_fp[c], int(before["B"][g, c]) + p.rho_fp[c] * dt)
            assert int(after["B"][g, c]) == refilled - charged[g, c] * unit
    # victim sets of lru and prefixshield from an independent closed form
    if len(E) and policy in ("lru", "prefixshield"):
        cand = [b for b in range(N) if before["resident"][b] and b not in pinned and b not in set(I.tolist())]
        if policy == "lru":
            want = sorted(sorted(cand, key=lambda b: int(before["stamp"][b]))[: len(E)])
        else:
            seg = not (oc.params.flags & O.FLAG_NO_SEGMENTATION)
            okey = lambda b: ((int(before["klass"][b]) if seg else 0) << 62) | int(before["stamp"][b])
            queues = [sorted((b for b in cand if int(before["group"][b]) == g), key=okey) for g in range(oc.G)]
            rmin = min(p.rho_fp[c] for c in range(C))
            delta = []
            for g in range(oc.G):
                rmax = max([p.rho_fp[c] for c in range(C) if after["B"][g, c] < 0] or [0])
                delta.append((unit * rmin) // rmax if rmax else 0)
            sel = alg2_closed_form([int(x) for x in res["debt_norm"]], delta, oc.params.epsilon_fp,
                                   [[okey(b) for b in q] for q in queues], len(E))
            want = sorted(queues[g][j] for g, j in sel)
        assert E.tolist() == want
    return hres


# ---------------------------------------------------------------------------
# GPU-vs-oracle comparison helpers.
OUT_KEYS = ("hit_blocks", "admitted_blocks", "admitted_offsets", "admitted_ids", "evicted_ids",
            "invalidated_ids", "debt_raw", "debt_norm")
BLOCK_KEYS = ("key", "group", "contract", "prefix", "klass", "stamp", "acc", "freq")


def compare_outputs(got, want, where=""):
    assert got["status"] == want["status"], f"{where}: status {got['status']} != {want['status']}"
    if want["status"] != 0:
        return
    for k in OUT_KEYS:
        a, b = np.asarray(got[k]), np.asarray(want[k])
        assert a.shape == b.shape and np.array_equal(a, b), (
            f"{where}: {k} differs" + (f" first at {int(np.nonzero(a != b)[0][0])}" if a.shape == b.shape else
                                       f" (len {a.shape} vs {b.shape})"))


def compare_state(got, want, where="", s3=False):
    assert np.array_equal(got["resident"], want["resident"]), f"{where}: residency differs"
    r = want["resident"].astype(bool)
    keys = BLOCK_KEYS + (("s3q", "s3seq") if s3 else ())
    for k in keys:
        a, b = got[k][r], want[k][r]
        if not np.array_equal(a, b):
            bad = np.nonzero(a != b)[0][0]
            raise AssertionError(f"{where}: block field {k} differs at resident #{bad}: {a[bad]} != {b[bad]}")
    assert np.array_equal(got["B"], want["B"]), f"{where}: balances differ"
    assert got["t_prev"] == want["t_prev"] and got["step"] == want["step"], f"{where}: clock/step differ"
    for a, b in zip(got["history"], want["history"]):
        assert np.array_equal(a, b), f"{where}: history differs"
    if s3:
        assert got["s3_ctr"] == want["s3_ctr"] and got["ghost_ctr"] == want["ghost_ctr"]
        for a, b in zip(got["ghost"], want["ghost"]):
            assert np.array_equal(a, b), f"{where}: ghost differs"
