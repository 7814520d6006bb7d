// step.cuh -- the per-worker scalars of a local step (Algorithm 1's inner
// AdamW with bias correction, App. B), computed on the device from the
// resident step counters so that no round needs host work.
#pragma once
#include <cstdint>

#include "internal.h"
#include "rng.cuh"

namespace gasloc {

// Scalars of worker i's local step number n, given p1 = beta1^n and
// p2 = beta2^n (n successive products from 1):
//   step = fl32(lr / (1 - p1)),  isb = fl32(1 / sqrt(1 - p2)),
//   noise key = hash(seed, 4, i, n),
// one IEEE double rounding per operation, as the host formulas.
__device__ __forceinline__ void write_step_scalars(StepTable *t, int i, int64_t n, double p1, double p2, double lr,
                                                   uint64_t seed) {
    const double bc1 = __dsub_rn(1.0, p1), bc2 = __dsub_rn(1.0, p2);
    t->step[i] = __double2float_rn(__ddiv_rn(lr, bc1));
    t->isb[i] = __double2float_rn(__ddiv_rn(1.0, __dsqrt_rn(bc2)));
    const uint64_t key = hash4(seed, kTagNoise, static_cast<uint64_t>(i), static_cast<uint64_t>(n));
    t->key_lo[i] = static_cast<uint32_t>(key);
    t->key_hi[i] = static_cast<uint32_t>(key >> 32);
}

}  // namespace gasloc
