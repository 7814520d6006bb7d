// ce_sum.cuh -- a thread's running fp64 sum of consensus-error terms (one
// fp32 term per element, e = S2 - (S1/n) S1), taken a group of up to 8
// elements at a time.  Used by the kernels that hold a column of every
// worker in registers (4 elements per thread in the direct gossip kernel; the
// fused round's 2-element columns take the terms one at a time).  The other
// reductions add each term on its own: their arithmetic is issue-bound (bf16)
// or their rate is set by HBM, and the integer work below did not pay there.
//
// The terms of a group that are normal numbers within 2^26 of the group's
// largest are added exactly in a 64-bit integer whose unit is the window's
// lowest bit.  The integer stays below 2^53, so the group's sum is formed
// exactly as a double, with integer operations, and enters the fp64 sum with
// one addition.  A term below the window or subnormal is widened and added
// on its own, and so is every term of a group that holds an infinity or a
// NaN.  Either way each group adds its exact sum, so two reductions of the
// same terms (fused or standalone, flat or tensor list, a range or the
// whole) differ only in the order of their fp64 additions.  This GPU
// retires about one fp64 addition per SM per clock, so one per group rather
// than one per element keeps them off the critical path.
#pragma once
#include <cstdint>

namespace gasloc {

constexpr int kCeWindow = 26;   // exponent range of a group's exact sum: 8 terms of 24 + 26 bits < 2^53

// The double equal to s * 2^e2, for 0 < |s| < 2^53 and a normal result.
__device__ __forceinline__ double exact_scaled(long long s, int e2) {
    const unsigned long long neg = s < 0 ? 1ull : 0ull;
    const unsigned long long a = static_cast<unsigned long long>(s < 0 ? -s : s);
    const int lz = __clzll(static_cast<long long>(a));   // 11..63
    const unsigned long long frac = (a << (lz - 11)) & 0xFFFFFFFFFFFFFull;   // leading one at bit 52, dropped
    const unsigned long long ex = static_cast<unsigned long long>(63 - lz + e2 + 1023);
    return __longlong_as_double(static_cast<long long>((neg << 63) | (ex << 52) | frac));
}

// Adds the G terms (G <= 8; unused slots hold +0) to acc.
template <int G>
__device__ __forceinline__ void ce_add_group(const float (&e)[G], double &acc) {
    static_assert(G >= 1 && G <= 8, "at most 8 terms per group");
    if (G < 4) {   // too few terms for the integer work to pay: one at a time
#pragma unroll
        for (int k = 0; k < G; ++k) acc += static_cast<double>(e[k]);
        return;
    }
    uint32_t u[G];
    uint32_t emax = 0;
#pragma unroll
    for (int k = 0; k < G; ++k) {
        u[k] = __float_as_uint(e[k]);
        const uint32_t ef = (u[k] >> 23) & 0xffu;
        emax = ef > emax ? ef : emax;
    }
    // bit k: term k is added on its own, after the loop and behind one branch
    // (rarely taken), so that no fp64 instruction is issued on the common path
    uint32_t own = 0;
    long long s = 0;
    const int base = static_cast<int>(emax) - kCeWindow;   // biased exponent of the window's lowest bit's term
    if (emax == 0xffu) {   // an infinity or a NaN: every term on its own
        own = (1u << G) - 1u;
    } else {
#pragma unroll
        for (int k = 0; k < G; ++k) {
            const int ef = static_cast<int>((u[k] >> 23) & 0xffu);
            if (ef == 0 || ef < base) {   // zero, subnormal or below the window
                if (u[k] << 1) own |= 1u << k;
                continue;
            }
            // value = m * 2^(ef - 150) = (m << (ef - base)) * 2^(base - 150)
            const long long m = static_cast<long long>((u[k] & 0x7fffffu) | 0x800000u) << (ef - base);
            s += (u[k] >> 31) ? -m : m;
        }
    }
    if (s != 0) acc += exact_scaled(s, base - 150);
    if (own) {
#pragma unroll
        for (int k = 0; k < G; ++k)
            if ((own >> k) & 1u) acc += static_cast<double>(e[k]);
    }
}

}  // namespace gasloc
