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
