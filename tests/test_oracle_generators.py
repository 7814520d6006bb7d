"""Pins for the oracle's counter-based generators.

The generators are not from the paper (it trains on data); they define the
synthetic workload.  They are pinned to published hash test vectors, to the
exact algebraic structure of the finalizers and to the moments of the
distributions they stand in for.
"""
import math
import os

import numpy as np
import pytest

GOLD = os.path.join(os.path.dirname(__file__), "golden", "hash_vectors.txt")


def _vectors(kind):
    out = []
    with open(GOLD) as f:
        for line in f:
            p = line.split()
            if p and p[0] == kind:
                out.append((int(p[1], 16), int(p[2], 16)))
    return out


@pytest.mark.parametrize("prec", ["f32", "f64"])
def test_splitmix64_published_vectors(prec, orc32, orc64):
    o = orc32 if prec == "f32" else orc64
    vs = _vectors("splitmix64")
    assert len(vs) == 3
    for state, out in vs:
        assert o.mix64(state) == out


def test_fmix32_published_vectors(orc32):
    vs = _vectors("fmix32")
    assert len(vs) == 3
    for seed, out in vs:
        assert orc32.fmix32(seed) == out


def _inv_xorshift(h, s):
    r = h
    for _ in range(32 // s + 1):
        r = h ^ (r >> s)
    return r & 0xFFFFFFFF


def test_fmix32_is_the_murmur_bijection(orc32):
    # Undo each step with the modular inverses of the two multipliers: if a
    # shift or a constant were wrong, the inverse would not recover the input.
    m1, m2 = 0x85EBCA6B, 0xC2B2AE35
    i1, i2 = pow(m1, -1, 2 ** 32), pow(m2, -1, 2 ** 32)
    rng = np.random.default_rng(1)
    for x in list(rng.integers(0, 2 ** 32, 300)) + [0, 1, 2 ** 32 - 1]:
        h = orc32.fmix32(int(x))
        h = _inv_xorshift(h, 16)
        h = (h * i2) & 0xFFFFFFFF
        h = _inv_xorshift(h, 13)
        h = (h * i1) & 0xFFFFFFFF
        h = _inv_xorshift(h, 16)
        assert h == int(x)


def test_hash_chain_composition(orc32):
    # hash(seed, tag, a, b) = mix64(mix64(mix64(mix64(seed)^tag)^a)^b)
    M = 2 ** 64
    for seed, tag, a, b in [(0, 1, 2, 3), (0x6A510C, 4, 7, 123456789), (M - 1, 7, 31, 0)]:
        s = orc32.mix64(seed)
        s = orc32.mix64(s ^ tag)
        s = orc32.mix64(s ^ a)
        assert orc32.hash(seed, tag, a, b) == orc32.mix64(s ^ b)


def test_hash_avalanche(orc32):
    # Each single-bit change of the counter flips about half the output bits.
    flips = []
    for k in range(64):
        a = orc32.hash(99, 4, 3, 1000)
        b = orc32.hash(99, 4, 3, 1000 ^ (1 << k))
        flips.append(bin(a ^ b).count("1"))
    assert 28 <= np.mean(flips) <= 36


def test_normal_standin_moments(orc64, orc32):
    # Irwin-Hall(4) of 24-bit uniforms, centred and scaled: mean 0, variance 1,
    # support [-2 sqrt3, 2 sqrt3], excess kurtosis -6/(5*4) = -0.3.
    n = 40000
    z = np.array([orc64.normal(5, 2, 3, k) for k in range(n)])
    assert abs(z.mean()) < 5 / math.sqrt(n)
    assert abs(z.var() - 1) < 0.03
    assert np.abs(z).max() <= 2 * math.sqrt(3)
    kurt = ((z - z.mean()) ** 4).mean() / z.var() ** 2 - 3
    assert abs(kurt + 0.3) < 0.08
    # f32 build: the same value rounded to float (one conversion + one product)
    z32 = np.array([orc32.normal(5, 2, 3, k) for k in range(2000)])
    assert np.all(np.abs(z32 - z[:2000]) <= 2.5e-7 * np.maximum(np.abs(z[:2000]), 1e-3))


def test_uniform_curvature_range(orc64):
    n = 20000
    h = np.array([orc64.uniform(9, 3, 0, k, 0.1, 0.9) for k in range(n)])
    assert h.min() >= 0.1 and h.max() < 1.0
    assert abs(h.mean() - 0.55) < 4 * 0.9 / math.sqrt(12 * n)
    assert abs(h.var() - 0.81 / 12) < 0.003


def test_noise_unit_variance_uniform(orc64):
    n = 40000
    xi = np.array([orc64.noise(11, 2, 5, k) for k in range(n)])
    s3 = math.sqrt(3)
    assert xi.min() >= -s3 and xi.max() < s3
    assert abs(xi.mean()) < 5 / math.sqrt(n)
    assert abs(xi.var() - 1) < 0.03
    # different steps / workers give (nearly) uncorrelated noise
    xi2 = np.array([orc64.noise(11, 2, 6, k) for k in range(n)])
    xi3 = np.array([orc64.noise(11, 3, 5, k) for k in range(n)])
    assert abs(np.corrcoef(xi, xi2)[0, 1]) < 0.03
    assert abs(np.corrcoef(xi, xi3)[0, 1]) < 0.03


def test_noise_grid_and_words_f32(orc64):
    # fp32 storage: xi = ((u >> 8) 2^-23 - 1) sqrt3 with u = fmix32 twice over
    # the element index k with the step key's halves: (xi / sqrt3 + 1) 2^23
    # is the integer u >> 8.
    seed, i, n = 29, 1, 3
    key = orc64.hash(seed, 4, i, n)
    lo, hi = key & 0xFFFFFFFF, key >> 32
    for k in [0, 1, 2, 3, 1001, 2 ** 26 + 5]:
        x = orc64.noise(seed, i, n, k)
        r = (x / math.sqrt(3) + 1) * 2 ** 23
        assert abs(r - round(r)) < 1e-6
        assert round(r) == orc64.fmix32(orc64.fmix32(k ^ lo) ^ hi) >> 8


def test_noise_grid_and_pair_words_bf16(orc32, orc64):
    # bf16 storage: every xi is q * (sqrt3 * 2^-15) for an integer q in [-2^15, 2^15),
    # rounded once in the build's precision (the f32 build scales fl32(sqrt3));
    # the two elements of a pair (2j, 2j+1) are the low and high halves of one
    # 32-bit word, fmix32 twice over j with the step key's halves (fmix32 and
    # hash are pinned above).
    s = math.sqrt(3) * 2.0 ** -15
    s32 = np.float32(np.float32(math.sqrt(3)) * np.float32(2.0 ** -15))
    seed, i, n = 17, 3, 9
    key = orc64.hash(seed, 4, i, n)
    lo, hi = key & 0xFFFFFFFF, key >> 32
    for j in [0, 1, 2, 1000, 2 ** 20 + 7, 2 ** 29 - 1]:
        q = []
        for k in (2 * j, 2 * j + 1):
            x = orc64.noise(seed, i, n, k, "bf16")
            r = round(x / s)
            assert abs(x - r * s) <= 1e-15 and -2 ** 15 <= r < 2 ** 15
            assert orc32.noise(seed, i, n, k, "bf16") == np.float32(np.float32(r) * s32)
            q.append(int(r))
        word = (q[0] + 2 ** 15) | ((q[1] + 2 ** 15) << 16)
        assert word == orc32.fmix32(orc32.fmix32(j ^ lo) ^ hi)


def test_noise_halves_uniform_and_uncorrelated_bf16(orc64):
    # bf16 storage: the 2^16-point grid is hit uniformly (chi-square over 64
    # bins), with unit variance, and the two halves of a word are uncorrelated.
    n = 2 ** 15
    xi = np.array([orc64.noise(23, 1, 4, k, "bf16") for k in range(2 * n)])
    assert xi.min() >= -math.sqrt(3) and xi.max() < math.sqrt(3)
    assert abs(xi.var() - 1) < 0.03
    cnt = np.histogram(xi, bins=64, range=(-math.sqrt(3), math.sqrt(3)))[0]
    exp = 2 * n / 64
    chi2 = ((cnt - exp) ** 2 / exp).sum()
    assert chi2 < 120          # 63 degrees of freedom: p < 1e-5 above 120
    assert abs(np.corrcoef(xi[0::2], xi[1::2])[0, 1]) < 0.03


def test_permutation_is_uniform(orc32):
    # every permutation of 4 elements appears with frequency 1/24
    from collections import Counter
    T = 24000
    cnt = Counter(tuple(orc32.permutation(3, t, 4)) for t in range(T))
    assert len(cnt) == 24
    exp = T / 24
    chi2 = sum((c - exp) ** 2 / exp for c in cnt.values())
    assert chi2 < 60  # 23 dof; p ~ 1e-4 at 53
    for t in range(50):
        p = orc32.permutation(3, t, 17)
        assert sorted(p.tolist()) == list(range(17))


def test_local_step_counts(orc32):
    H = orc32.draw_local_steps(0x6A510C, 32, 8)
    assert H.min() >= 1 and H.max() <= 8
    big = orc32.draw_local_steps(1, 8000, 8)
    cnt = np.bincount(big, minlength=9)[1:]
    assert cnt.min() > 850 and cnt.max() < 1150
