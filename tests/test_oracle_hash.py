"""Pins of the oracle's block-key function (chained full-block hashing).

The key function is this project's own definition, built from published parts
(SplitMix64 for the key schedule and the mixer, UMAC's NH with a Toeplitz-
shifted second key for the block digest).  Each part is pinned here against a
published value, a closed form, or a property that a plausible mistake breaks.
"""
import os

import numpy as np
import pytest

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
M64 = (1 << 64) - 1


def test_splitmix64_published_vector():
    lines = [l for l in open(os.path.join(GOLDEN, "splitmix64_seed1234567.txt")) if not l.startswith("#")]
    seed = int(lines[0].split()[1])
    want = [int(x) for x in lines[1:] if x.strip()]
    assert O.splitmix64_stream(seed, len(want)) == want


def test_mix64_is_the_splitmix_output_function():
    # splitmix64_next adds the golden gamma and applies the output function,
    # so mix64(s + gamma) must equal the next output from state s.
    gamma = 0x9E3779B97F4A7C15
    for s in (0, 1, 1234567, M64, 0xDEADBEEF12345678):
        assert O.mix64((s + gamma) & M64) == O.splitmix64_stream(s, 1)[0]
    assert O.mix64(0) == 0  # every step of the mixer maps 0 to 0


def _key(bs=16, seed=99):
    return [w & 0xFFFFFFFF for w in O.splitmix64_stream(seed, bs + 2)]


def _neg(k):  # int32 message word m with (m + k) mod 2^32 == 0
    v = (-k) & 0xFFFFFFFF
    return v - (1 << 32) if v >= (1 << 31) else v


def test_nh_zero_pairs():
    K = _key()
    # Zeroing the first word of every pair zeroes every product.
    M = [0] * 16
    for k in range(8):
        M[2 * k] = _neg(K[2 * k])
        M[2 * k + 1] = 12345 + k
    assert O.nh(K, 0, M, 16) == 0


def test_nh_single_pair_with_32bit_wrap():
    K = _key()
    M = [0] * 16
    for k in range(8):
        M[2 * k] = _neg(K[2 * k])
    # Pair 3 only: (m6 + K6) mod 2^32 = 5 and (m7 + K7) mod 2^32 = 7.
    M[6] = _neg(K[6]) + 5 if _neg(K[6]) + 5 < (1 << 31) else _neg(K[6]) + 5 - (1 << 32)
    M[7] = _neg(K[7]) + 7 if _neg(K[7]) + 7 < (1 << 31) else _neg(K[7]) + 7 - (1 << 32)
    assert O.nh(K, 0, M, 16) == 35


def test_nh_64bit_wrap():
    K = _key()
    M = [0] * 16
    for k in range(8):
        M[2 * k] = _neg(K[2 * k])
    # Two pairs with both factors 2^32 - 1: each product is 2^64 - 2^33 + 1,
    # their sum mod 2^64 is 2^64 - 2^34 + 2.
    for k in (1, 5):
        for j in (2 * k, 2 * k + 1):
            v = (0xFFFFFFFF - K[j]) & 0xFFFFFFFF
            M[j] = v - (1 << 32) if v >= (1 << 31) else v
    assert O.nh(K, 0, M, 16) == (1 << 64) - (1 << 34) + 2


def test_nh_toeplitz_shift_is_key_offset():
    K = _key()
    rng = np.random.default_rng(3)
    M = rng.integers(-2**31, 2**31, 16, dtype=np.int64).astype(np.int32)
    assert O.nh(K, 2, M, 16) == O.nh(K[2:] + [0, 0], 0, M, 16)


def test_nh_distinguishes_pair_order():
    # NH pairs words (0,1), (2,3), ...: swapping words across pairs changes
    # the digest, swapping within a pair does not.
    K = [0] * 18
    M = list(range(1, 17))
    base = O.nh(K, 0, M, 16)
    assert base == sum(M[2 * k] * M[2 * k + 1] for k in range(8))
    sw = M.copy(); sw[0], sw[1] = sw[1], sw[0]
    assert O.nh(K, 0, sw, 16) == base
    sw = M.copy(); sw[1], sw[2] = sw[2], sw[1]
    assert O.nh(K, 0, sw, 16) != base


@pytest.mark.parametrize("bs", [2, 4, 16, 32])
def test_chain_prefix_property_and_ragged_tail(bs):
    rng = np.random.default_rng(bs)
    t = rng.integers(0, 32000, 10 * bs + bs - 1, dtype=np.int32)  # ragged tail
    k = O.chain_keys(7, 3, bs, t)
    assert len(k) == 10
    for n in range(11):
        assert np.array_equal(O.chain_keys(7, 3, bs, t[: n * bs]), k[:n])
    # the tail tokens never matter
    t2 = t.copy(); t2[-1] += 1
    assert np.array_equal(O.chain_keys(7, 3, bs, t2), k)


def test_chain_change_propagates_forward_only():
    rng = np.random.default_rng(5)
    t = rng.integers(0, 32000, 12 * 16, dtype=np.int32)
    k = O.chain_keys(7, 0, 16, t)
    for j in (0, 5, 11):
        t2 = t.copy(); t2[j * 16 + 9] ^= 1
        k2 = O.chain_keys(7, 0, 16, t2)
        assert np.array_equal(k2[:j], k[:j])
        assert np.all(k2[j:] != k[j:])


def test_chain_namespaced_by_group_and_seed():
    t = np.arange(64, dtype=np.int32)
    a = O.chain_keys(7, 0, 16, t)
    assert np.all(O.chain_keys(7, 1, 16, t) != a)
    assert np.all(O.chain_keys(8, 0, 16, t) != a)


def test_chain_depth_is_part_of_the_key():
    # The same block content at two depths of one chain gives different keys,
    # and a repeated block gives a new key each time.
    blk = np.arange(16, dtype=np.int32)
    k = O.chain_keys(7, 0, 16, np.tile(blk, 6))
    assert len(set(int(x) for x in k)) == 6


def test_chain_keys_avoid_reserved_values():
    rng = np.random.default_rng(11)
    k = O.chain_keys(1, 0, 16, rng.integers(0, 32000, 4096 * 16, dtype=np.int32))
    assert not np.any(k == 0) and not np.any(k == np.uint64(M64))
    assert len(np.unique(k)) == len(k)


def test_stamps_order_step_request_then_reverse_position():
    """Stamps follow (step, request, deepest block first) and are dense: a step
    of requests with n = (3, 0, 2) full blocks from base 10 uses 10..14."""
    s = O.make_stamp
    n = [3, 0, 2]
    before = [0, 3, 3]
    got = {(i, m): s(10, before[i], n[i], m) for i in range(3) for m in range(n[i])}
    assert sorted(got.values()) == list(range(10, 15))
    # within a request the deeper block is released first, so it is older
    assert got[(0, 0)] > got[(0, 1)] > got[(0, 2)]
    # a later request is newer than every block of an earlier one
    assert min(got[(2, m)] for m in range(2)) > max(got[(0, m)] for m in range(3))
    # the next step starts after all of this step's stamps
    assert s(15, 0, 1, 0) > max(got.values())


P61 = (1 << 61) - 1


def _unmix64(z):
    """Inverse of the SplitMix64 output function (xorshifts and odd multipliers)."""
    def unxs(y, s):
        x = y
        k = s
        while k < 64:
            x = y ^ (x >> s)
            k += s
        return x & M64
    z = unxs(z & M64, 31)
    z = (z * pow(0x94D049BB133111EB, -1, 1 << 64)) & M64
    z = unxs(z, 27)
    z = (z * pow(0xBF58476D1CE4E5B9, -1, 1 << 64)) & M64
    return unxs(z, 30)


def test_unmix_inverts_mix():
    for z in (0, 1, 12345, M64, 0xDEADBEEFCAFEBABE):
        assert _unmix64(O.mix64(z)) == z


@pytest.mark.parametrize("bs,g", [(16, 0), (16, 5), (4, 2), (32, 1)])
def test_chain_is_the_affine_recurrence_mod_2p61m1(bs, g):
    """Recover C_m from each key and check C_m = Kc*C_{m-1} + D_m (mod p),
    C_{-1} = mix(seed ^ (g+1)*phi) mod p, D_m = NH0 + Kd*NH2 (mod p), with
    the key schedule taken from the pinned SplitMix64 stream."""
    seed = 0x1234ABCD
    rng = np.random.default_rng(bs + 7 * g)
    t = rng.integers(0, 32000, 9 * bs, dtype=np.int32)
    keys = [int(k) for k in O.chain_keys(seed, g, bs, t)]
    stream = O.splitmix64_stream(seed, bs + 4)
    K = [w & 0xFFFFFFFF for w in stream[: bs + 2]]
    Kc = stream[bs + 2] % P61 or 1
    Kd = stream[bs + 3] % P61 or 1
    C = O.mix64(seed ^ (((g + 1) * 0x9E3779B97F4A7C15) & M64)) % P61
    for m, key in enumerate(keys):
        Cm = _unmix64(key) ^ (((m + 1) * 0xD1B54A32D192ED03) & M64)
        blk = t[m * bs:(m + 1) * bs]
        D = (O.nh(K, 0, blk, bs) + Kd * (O.nh(K, 2, blk, bs) % P61)) % P61
        assert Cm == (Kc * C + D) % P61, m
        C = Cm
