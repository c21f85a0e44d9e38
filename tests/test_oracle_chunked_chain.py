"""Pin of the chunked evaluation of the block-key chain (reading R2), the
arithmetic the CUDA hashing kernel performs, against the oracle's
block-by-block chain.

The chain C_m = Kc C_{m-1} + D_m (mod 2^61 - 1) is evaluated on the GPU in
64-block chunks: within a chunk each half of 32 blocks is an inclusive scan of
the affine maps x -> Kc x + D by doubling (five rounds, multipliers
Kc^(2^q)); the chunk's total is Kc^(second half's blocks) times the first
half's total plus the second's; the value entering chunk k folds its
predecessors' totals in windows of 32 with powers of Kc^64; the second half
enters at Kc^32 times the chunk's entering value plus the first half's total.
Restated here with Python integers, it must give the oracle's keys for every
length, across half, chunk and window boundaries.
"""
import numpy as np
import pytest

import oracle as O

P61 = (1 << 61) - 1
M64 = (1 << 64) - 1


def _chunked_keys(seed, g, bs, tokens):
    stream = O.splitmix64_stream(seed, bs + 4)
    K = [w & 0xFFFFFFFF for w in stream[: bs + 2]]
    Kc = stream[bs + 2] % P61 or 1
    Kd = stream[bs + 3] % P61 or 1
    kc = [pow(Kc, j, P61) for j in range(33)]            # Kc^j, j = 0..32
    kc64 = [pow(Kc, 64 * t, P61) for t in range(33)]     # Kc^(64 t), t = 0..32
    n = len(tokens) // bs
    D = []
    for m in range(n):
        blk = tokens[m * bs:(m + 1) * bs]
        D.append((O.nh(K, 0, blk, bs) % P61 + Kd * (O.nh(K, 2, blk, bs) % P61)) % P61)
    seed_c = O.mix64(seed ^ (((g + 1) * 0x9E3779B97F4A7C15) & M64)) % P61

    def half_scan(m0, cnt):
        b = [D[m0 + l] if l < cnt else 0 for l in range(32)]
        for q in range(5):
            prev = list(b)
            for l in range(1 << q, 32):
                b[l] = (b[l] + kc[1 << q] * prev[l - (1 << q)]) % P61
        return b

    totals, C = [], [0] * n
    for k in range((n + 63) // 64):
        m0 = 64 * k
        nb = min(64, n - m0)
        nA, nB = min(32, nb), nb - min(32, nb)
        bA = half_scan(m0, nA)
        bB = half_scan(m0 + 32, nB) if nB else [0] * 32
        totA = bA[nA - 1]
        totals.append((kc[nB] * totA + bB[nB - 1]) % P61 if nB else totA)
        cin = seed_c
        for l0 in range(0, k, 32):
            w = min(32, k - l0)
            term = sum(kc64[w - 1 - lane] * totals[l0 + lane] for lane in range(w)) % P61
            cin = (kc64[w] * cin + term) % P61
        for l in range(nA):
            C[m0 + l] = (kc[l + 1] * cin + bA[l]) % P61
        cin_b = (kc[32] * cin + totA) % P61
        for l in range(nB):
            C[m0 + 32 + l] = (kc[l + 1] * cin_b + bB[l]) % P61
    keys = []
    for m, c in enumerate(C):
        x = O.mix64(c ^ (((m + 1) * 0xD1B54A32D192ED03) & M64))
        keys.append(1 if x in (0, M64) else x)
    return keys


@pytest.mark.parametrize("bs,lengths", [
    (16, (1, 31, 32, 33, 63, 64, 65, 96, 127, 128, 129, 2048, 2049, 2100)),
    (2, (1, 64, 65, 300)),
    (64, (1, 33, 64, 65, 130)),
])
def test_chunked_chain_equals_the_oracle(bs, lengths):
    rng = np.random.default_rng(bs)
    for nblk in lengths:
        t = rng.integers(0, 32000, nblk * bs + 5, dtype=np.int32)  # a ragged tail too
        for g in (0, 5):
            want = [int(x) for x in O.chain_keys(0x5EED, g, bs, t)]
            assert _chunked_keys(0x5EED, g, bs, t) == want, (bs, nblk, g)
