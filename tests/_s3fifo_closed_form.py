"""The closed form of a batch of S3-FIFO evictions (Sec. V-A baseline; Yang et
al., SOSP 2023), as the CUDA library computes it, restated plainly so the CPU
tests can check it against the oracle's one-at-a-time loop.

Inputs: the small and main queues (live members, oldest first), each block's
frequency (already capped), the step's pinned blocks, the number m of
victims, the move threshold, the small queue's capacity and the sequence
counter before the step.  Returns None where the closed form does not apply
(the library then runs the sequential loop): the main queue would run empty
inside the step, or the cap is 16 or more.
"""


def s3_batch(S, M, f, pinned, m, cap, move_min, S_cap, ctr0):
    uS = [b for b in S if b not in pinned]
    K = len(uS)
    victim_pos = [j + 1 for j, b in enumerate(uS) if f[b] < move_min]  # 1-based
    T = len(victim_pos)
    # small phase: eviction t takes the small queue while the members popped
    # before it number at most D, and some unpinned member is left
    D = len(S) - S_cap
    nA = 0
    if D >= 0 and K >= 1 and m > 0:
        Dp = min(D, K - 1)
        nA = min(m, 1 + sum(1 for e in victim_pos if e <= Dp))
    cA = 0 if nA == 0 else (victim_pos[nA - 1] if nA <= T else K)
    consumed = uS[:cA]
    movers = [b for b in consumed if f[b] >= move_min]
    small_victims = [b for b in consumed if f[b] < move_min]
    MA = len(movers)
    seq, freq = {}, {}
    for r, b in enumerate(movers):
        seq[b] = ctr0 + 1 + r
    L = [b for b in M if b not in pinned] + movers
    mB = m - len(small_victims)
    if mB > len(L) or cap >= 16:
        return None
    victims = set(small_victims)
    visited = set()
    mid = []
    if mB > 0:
        fL = [f[b] for b in L]
        # the final round Rs: the first whose cumulative evictions reach mB
        cum, Rs = 0, 0
        for r in range(cap + 1):
            c = fL.count(r)
            if cum + c >= mB:
                Rs, k = r, mB - cum
                break
            cum += c
        P = [j for j, x in enumerate(fL) if x == Rs][k - 1]  # position of the last visit
        # reinsertions of the complete rounds before Rs - 1 and before Rs
        base = [0] * (Rs + 1)
        for r in range(1, Rs + 1):
            base[r] = base[r - 1] + sum(1 for x in fL if x >= r)
        g1, g2 = [], []
        ge = gt = 0
        for j, b in enumerate(L):
            x = fL[j]
            if x < Rs or (x == Rs and j <= P):
                victims.add(b)
                visited.add(b)
            elif j <= P:                      # reinserted in round Rs
                freq[b], seq[b] = x - Rs - 1, ctr0 + MA + base[Rs] + gt + 1
                g2.append(b)
                visited.add(b)
            elif Rs >= 1:                     # last reinserted in round Rs - 1
                freq[b], seq[b] = x - Rs, ctr0 + MA + base[Rs - 1] + ge + 1
                g1.append(b)
                visited.add(b)
            ge += x >= Rs
            gt += x > Rs
        ctr_end = ctr0 + MA + base[Rs] + sum(1 for x in fL[:P + 1] if x > Rs)
        mid = ([b for b in L[P + 1:] if b in set(movers)] if Rs == 0 else g1) + g2
    else:
        ctr_end = ctr0 + MA
        mid = list(movers)
    cons = set(consumed)
    new_small = [b for b in S if b in pinned or b not in cons]
    new_main = [b for b in M if b in pinned or b not in visited] + mid
    return dict(victims=victims, small_victims=small_victims, seq=seq, freq=freq, ctr_end=ctr_end,
                new_small=new_small, new_main=new_main)


def s3_loop(S, M, f, pinned, m, cap, move_min, S_cap, ctr0):
    """The published loop, one eviction at a time (queues as Python lists)."""
    f = dict(f)
    seq = {}
    US = [b for b in S if b not in pinned]
    UM = [b for b in M if b not in pinned]
    nS, ctr = len(S), ctr0
    victims, small_victims = [], []

    def evict_main():
        nonlocal ctr
        while True:
            b = UM.pop(0)
            if f[b] > 0:
                f[b] -= 1
                ctr += 1
                seq[b] = ctr
                UM.append(b)
            else:
                victims.append(b)
                return

    for _ in range(m):
        if not ((nS >= S_cap and US) or not UM):
            evict_main()
            continue
        done = False
        while US:
            b = US.pop(0)
            nS -= 1
            if f[b] >= move_min:
                ctr += 1
                seq[b] = ctr
                UM.append(b)
            else:
                victims.append(b)
                small_victims.append(b)
                done = True
                break
        if not done:
            evict_main()
    return set(victims), small_victims, seq, f, ctr
