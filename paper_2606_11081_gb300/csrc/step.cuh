// step.cuh -- the per-worker scalars of a local step (Algorithm 1's inner
// AdamW with bias correction, App. B), computed on the device from the
// resident step counters so that no round needs host work.
#pragma once
#include <cstdint>

#include "internal.h"
#include "rng.cuh"

namespace gasloc {

// Learning rate of local step n (the schedule's table for n <= steps, the
// held rate after; with no schedule steps = 0 and `after` is the constant lr).
__device__ __forceinline__ double lr_of_step(int64_t n, const double *sched, int64_t steps, double after) {
    return n <= steps ? sched[n - 1] : after;
}

// Scalars of worker i's local step number n with rate lr_n, given
// p1 = beta1^n and p2 = beta2^n (n successive products from 1):
//   step = fl32(lr_n / (1 - p1)),  isb = fl32(1 / sqrt(1 - p2)),
//   decay = fl32(1 - lr_n * wd),   noise key = hash(seed, 4, i, n),
// one IEEE double rounding per operation, as the host formulas.
__device__ __forceinline__ void write_step_scalars(StepTable *t, int i, int64_t n, double p1, double p2, double lr_n,
                                                   double wd, uint64_t seed) {
    const double bc1 = __dsub_rn(1.0, p1), bc2 = __dsub_rn(1.0, p2);
    t->step[i] = __double2float_rn(__ddiv_rn(lr_n, bc1));
    t->isb[i] = __double2float_rn(__ddiv_rn(1.0, __dsqrt_rn(bc2)));
    t->decay[i] = __double2float_rn(__dsub_rn(1.0, __dmul_rn(lr_n, wd)));
    const uint64_t key = hash4(seed, kTagNoise, static_cast<uint64_t>(i), static_cast<uint64_t>(n));
    t->key_lo[i] = static_cast<uint32_t>(key);
    t->key_hi[i] = static_cast<uint32_t>(key >> 32);
}

// Worker i has taken a local step: its counters advance (n, beta1^n,
// beta2^n) and its next step's scalars are written to the table.
__device__ __forceinline__ void advance_step(DevState *st, StepTable *t, int i, double beta1, double beta2,
                                             const double *lr_sched, int64_t lr_steps, double lr_after, double wd,
                                             uint64_t seed) {
    const int64_t n = st->nsteps[i] + 1;
    const double p1 = __dmul_rn(st->p1[i], beta1), p2 = __dmul_rn(st->p2[i], beta2);
    st->nsteps[i] = n;
    st->p1[i] = p1;
    st->p2[i] = p2;
    write_step_scalars(t, i, n + 1, __dmul_rn(p1, beta1), __dmul_rn(p2, beta2),
                       lr_of_step(n + 1, lr_sched, lr_steps, lr_after), wd, seed);
}

}  // namespace gasloc
