"""The exact column sum of consensus-error terms (csrc/ce_sum.cuh) compiled for
the host and checked against exact rational arithmetic.

ce_add_group adds a group of fp32 terms to an fp64 sum: the terms within
2^26 of the group's largest, if normal, as their exact sum (one fp64
addition), every other term (below that window, subnormal, or any term of a
group holding an inf or a NaN) with an addition of its own.  Built here with
g++ and stand-ins for the four CUDA intrinsics it uses (bit casts and a
count of leading zeros), it must give, from a sum of 0, exactly
fl64(window sum) followed by the other terms in order, and the window sum
must be representable as a double."""
import os
import shutil
import struct
import subprocess
from fractions import Fraction

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "paper_2606_11081_gb300", "csrc", "ce_sum.cuh")

HARNESS = r"""
#include <cstdint>
#include <cstdio>
#include <cstring>
#define __device__
#define __forceinline__ inline
static inline uint32_t __float_as_uint(float f) { uint32_t u; std::memcpy(&u, &f, 4); return u; }
static inline int __clzll(long long x) { return x == 0 ? 64 : __builtin_clzll(static_cast<unsigned long long>(x)); }
static inline double __longlong_as_double(long long x) { double d; std::memcpy(&d, &x, 8); return d; }
#include "ce_sum.cuh"
int main() {
    unsigned a[8];
    while (std::scanf("%x %x %x %x %x %x %x %x", &a[0], &a[1], &a[2], &a[3], &a[4], &a[5], &a[6], &a[7]) == 8) {
        float e8[8];
        for (int k = 0; k < 8; ++k) std::memcpy(&e8[k], &a[k], 4);
        const float e4[4] = {e8[0], e8[1], e8[2], e8[3]};
        const float e2[2] = {e8[0], e8[1]};
        double s8 = 0.0, s4 = 0.0, s2 = 0.0;
        gasloc::ce_add_group<8>(e8, s8);
        gasloc::ce_add_group<4>(e4, s4);
        gasloc::ce_add_group<2>(e2, s2);
        unsigned long long b[3];
        std::memcpy(&b[0], &s8, 8);
        std::memcpy(&b[1], &s4, 8);
        std::memcpy(&b[2], &s2, 8);
        std::printf("%016llx %016llx %016llx\n", b[0], b[1], b[2]);
    }
    return 0;
}
"""


def f32_bits(v):
    return struct.unpack("<I", struct.pack("<f", float(v)))[0]


def expected(terms, group_min=4):
    """The helper's result from a sum of 0, in exact arithmetic."""
    acc = 0.0
    if len(terms) < group_min:       # small groups: one addition per term
        for v in terms:
            acc = acc + float(v)
        return acc
    ef = [(f32_bits(v) >> 23) & 0xFF for v in terms]
    emax = max(ef)
    if emax == 0xFF:
        for v in terms:
            acc = acc + float(v)
        return acc
    base = emax - 26
    window = Fraction(0)
    own = []
    for v, e in zip(terms, ef):
        if e == 0 or e < base:
            if float(v) != 0.0:
                own.append(float(v))
        else:
            window += Fraction(float(v))
    if window != 0:
        assert Fraction(float(window)) == window   # exact as a double
        acc = acc + float(window)
    for v in own:
        acc = acc + v
    return acc


def groups(n=12000, seed=7):
    rng = np.random.default_rng(seed)
    out = []
    for t in range(n):
        kind = t % 9
        if kind == 0:
            g = rng.standard_normal(8) ** 2
        elif kind == 1:
            g = rng.standard_normal(8) * 10.0 ** rng.integers(-30, 30, 8)
        elif kind == 2:
            g = np.where(rng.random(8) < 0.5, 0.0, rng.standard_normal(8))
        elif kind == 3:
            g = rng.standard_normal(8) * 10.0 ** rng.integers(-45, -36, 8)     # subnormal terms
        elif kind == 4:
            g = rng.standard_normal(8) * 3.0e38 / 8                           # near the fp32 top
        elif kind == 5:
            g = rng.standard_normal(8)
            g[rng.integers(0, 8)] = [np.inf, -np.inf, np.nan][t % 3]
        elif kind == 6:
            g = rng.standard_normal(8) * 2.0 ** rng.integers(-27, 1, 8)       # across the window's edge
        elif kind == 7:
            g = np.full(8, 2.0 ** 20) * (1 - 2 * (rng.random(8) < 0.5))       # cancellation to 0
        else:
            g = (1.0 + rng.integers(0, 1 << 23, 8) * 2.0 ** -23) * 2.0 ** 26  # full mantissas at the top
        out.append(np.asarray(g, dtype=np.float32))
    return out


@pytest.fixture(scope="module")
def harness(tmp_path_factory):
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("g++ not available")
    d = tmp_path_factory.mktemp("ce_sum")
    src = d / "harness.cpp"
    src.write_text(HARNESS)
    exe = d / "harness"
    subprocess.run([gxx, "-O2", "-std=c++17", "-ffp-contract=off", "-I", os.path.dirname(HEADER), str(src),
                    "-o", str(exe)], check=True)
    return str(exe)


def test_group_sums_are_exact(harness):
    gs = groups()
    inp = "\n".join(" ".join("%08x" % f32_bits(v) for v in g) for g in gs) + "\n"
    out = subprocess.run([harness], input=inp, capture_output=True, text=True, check=True).stdout.split()
    assert len(out) == 3 * len(gs)
    for i, g in enumerate(gs):
        for j, k in enumerate((8, 4, 2)):
            got = struct.unpack("<d", struct.pack("<Q", int(out[3 * i + j], 16)))[0]
            want = expected(g[:k])
            assert got == want or (np.isnan(got) and np.isnan(want)), (k, g[:k], got, want)


def test_group_sum_equals_the_exact_total_when_all_terms_fit(harness):
    # terms within one binade of each other, so all in the window: the result
    # is their exact sum (which a double holds)
    rng = np.random.default_rng(3)
    gs = [((0.5 + 0.5 * rng.random(8)) * 2.0 ** rng.integers(-20, 5)).astype(np.float32) for _ in range(500)]
    inp = "\n".join(" ".join("%08x" % f32_bits(v) for v in g) for g in gs) + "\n"
    out = subprocess.run([harness], input=inp, capture_output=True, text=True, check=True).stdout.split()
    for i, g in enumerate(gs):
        got = struct.unpack("<d", struct.pack("<Q", int(out[3 * i], 16)))[0]
        assert got == float(sum(Fraction(float(v)) for v in g))
