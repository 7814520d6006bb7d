// round.cu -- K_round: a round's last local step fused with its gossip round
// (Algorithm 1: the inner AdamW step that ends the round, then the
// communication step with the outer optimizer and the consensus error) in one
// kernel, for stores of few workers (n <= 4) with fp32 storage, where every
// worker takes that step.
//
// Every step of the round acts on each parameter index on its own (the
// synthetic gradient is diagonal, the mixing combines the workers' values at
// one index), so a thread that owns a column of V elements for all n workers
// can take each worker's step and then mix the new iterates in registers:
// the new y is stored (it is part of the replica state) but not read back, and
// the round is one pass over the store instead of two.  Per worker-element
// (GASLoC/Nesterov, the round's first step): x, m, v, c, b and the shared h
// read, y, m, v, x, b written -- 41 bytes against 49 for the two kernels.
//
// The arithmetic and its order are those of the local-step kernel
// (adamw_math.cuh) followed by those of the gossip kernels (mix.cuh), so a
// fused round is bit-identical to gasloc_local_steps + gasloc_gossip_round.
// Small stores only: at a few tiles per CTA both separate kernels are bound by
// their ramp and tail rather than by HBM, and one kernel pays those once.
//
// It is an opt-in variant (gasloc_fused_round).  The separate kernels make one
// HBM pass per local step, the last step's iterate written for the gossip
// kernel to read back, as where a trainer's gradient arrives between steps;
// that is the byte model gasloc_run and the benchmark's rounds keep.
//
// The step's per-worker scalars come from the step table; the last CTA to
// have read them (atomic ticket, nothing waits) advances every worker's step
// counters and writes their next step's scalars while the others work.  The
// last CTA to finish adds the CTAs' consensus-error partials in CTA order,
// stores the round's value and advances the round counter.
#include <cuda_runtime.h>

#include "adamw_math.cuh"
#include "check.cuh"
#include "f32x2.cuh"
#include "internal.h"
#include "mix.cuh"
#include "ptx.cuh"
#include "step.cuh"

namespace gasloc {

namespace {

constexpr int kV = kRoundColumn;                   // elements per consumer thread
constexpr int kTile = kRoundTile;                  // elements per tile
constexpr int kConsumers = kTile / kV;             // a column of kV elements each
constexpr int kThreads = kConsumers + 32;          // + the producer warp
constexpr int kStages = 2;
constexpr int kMinBlocks = 2;                      // CTAs per SM
static_assert(kConsumers % 32 == 0 && kConsumers * kV == kTile, "whole warps of consumers");
constexpr uint64_t kWaitNs = 2000000000ull;

// Rows of a tile in a stage: per worker (slot j * kPer + kind) the iterate
// (x on the worker's first step of the round, else y), m, v, c, then x where
// the iterate is y, the worker's own h under per-worker curvature and b where
// the outer update keeps one; after the workers' slots the tile's shared h.
template <int MODE, bool PER_WORKER_H, bool FROM_X>
struct Rows {
    static constexpr int kIt = 0, kM = 1, kVv = 2, kC = 3;
    static constexpr int kX = 4;
    static constexpr int kHw = kX + (FROM_X ? 0 : 1);
    static constexpr int kB = kHw + (PER_WORKER_H ? 1 : 0);
    static constexpr int kPer = kB + (ModeRows<MODE>::kHasB ? 1 : 0);
    static constexpr int kShared = kColumnWorkers * kPer;   // slot of the shared h row
    static constexpr int kSlots = kShared + (PER_WORKER_H ? 0 : 1);
    static constexpr size_t kStageBytes = static_cast<size_t>(kSlots) * kTile * sizeof(float);
    static constexpr size_t kBarOffset = kStages * kStageBytes;
    static constexpr size_t kDescOffset = kBarOffset + 2 * kStages * sizeof(uint64_t);
    static constexpr size_t kSmem = kDescOffset + kStages * 128;
};

// What the consumers need of a stage's tile, written by the producer beside
// its rows.
struct TileDesc {
    int64_t start, wstride, goff;   // tile start in the tensor, row stride, global index of element 0
    float *x, *y, *m, *v, *b;
    int32_t len, pad;
};
static_assert(sizeof(TileDesc) <= 128, "one 128-byte slot per stage");

// Barrier of the consumer warps only (the producer does not take part).
__device__ __forceinline__ void consumer_sync() {
    asm volatile("barrier.sync 1, %0;" ::"r"(kConsumers) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(ptx::smem_addr(bar)) : "memory");
}

template <int MODE, bool PER_WORKER_H, bool FROM_X>
__global__ void __launch_bounds__(kThreads, kMinBlocks) round_kernel(const RoundArgs a) {
    using R = ModeRows<MODE>;
    using RR = Rows<MODE, PER_WORKER_H, FROM_X>;
    using C = Col<kV>;
    using T = typename C::T;
    constexpr int NP = kV / 2;
    extern __shared__ __align__(128) unsigned char smem[];
    float *stages = reinterpret_cast<float *>(smem);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + RR::kBarOffset);
    uint64_t *empty = full + kStages;
    TileDesc *descs = reinterpret_cast<TileDesc *>(smem + RR::kDescOffset);
    __shared__ DenseRows dr;
    __shared__ float s_nstep[kColumnWorkers], s_isb[kColumnWorkers], s_dec[kColumnWorkers];
    __shared__ uint32_t s_klo[kColumnWorkers], s_khi[kColumnWorkers];
    __shared__ double red[kThreads / 32];
    __shared__ int last, last_copy;
    __shared__ int abort_flag;
    const int n = a.n_workers;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], kConsumers / 32);
        }
        ptx::fence_mbar_init();
        abort_flag = 0;
    }
    __syncthreads();   // the producer starts its copies at once; the consumers first read the round's tables
    const int64_t round = __ldcg(&a.state->round);   // advanced by the last CTA to finish, after every CTA read it
    const int64_t my_n = a.ntiles > blockIdx.x ? (a.ntiles - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
    const int lane = threadIdx.x & 31;
    auto slot = [&](int s, int k) { return stages + (static_cast<size_t>(s) * RR::kSlots + k) * kTile; };
    double ce_acc = 0.0;

    if (threadIdx.x >= kConsumers) {
        // ---------------------------------------------------------- producer ---
        const int nrows = n * RR::kPer;
        const int ncopies = nrows + (PER_WORKER_H ? 0 : 1);
        int64_t issued = 0;
        bool aborted = false;
        // tensor 0's descriptor read at once, beside the first tile's (a flat
        // store has no other)
        int32_t cur = 0;
        TensorDesc d = a.tens[0];
        for (int64_t it = 0; it < my_n; ++it) {
            const int s = static_cast<int>(it % kStages);
            if (it >= kStages) {
                const int64_t j = it - kStages;
                const bool ok = ptx::mbar_wait_bounded(&empty[s], static_cast<uint32_t>((j / kStages) & 1), kWaitNs);
                if (!__all_sync(0xffffffffu, ok)) {
                    aborted = true;
                    break;
                }
            }
            if (__any_sync(0xffffffffu, abort_flag != 0)) {
                aborted = true;
                break;
            }
            const Tile tl = a.tiles[blockIdx.x + it * gridDim.x];
            if (tl.tensor != cur) {
                d = a.tens[tl.tensor];
                cur = tl.tensor;
            }
            const int lenr = (tl.len + 3) & ~3;   // whole 16-byte pieces (the row padding is allocated)
            const uint32_t bytes = static_cast<uint32_t>(lenr) * sizeof(float);
            if (lane == 0) {
                // the descriptor's stores precede the arrive (release), the
                // consumers read it after their wait (acquire)
                TileDesc &u = descs[s];
                u.start = tl.start;
                u.wstride = d.wstride;
                u.goff = d.goff;
                u.x = static_cast<float *>(d.x);
                u.y = static_cast<float *>(d.y);
                u.m = static_cast<float *>(d.m);
                u.v = static_cast<float *>(d.v);
                u.b = static_cast<float *>(d.b);
                u.len = tl.len;
                ptx::mbar_arrive_expect_tx(&full[s], static_cast<uint32_t>(ncopies) * bytes);
            }
            __syncwarp();
            if (lane < ncopies && span_ok(0, lenr, kTile, a.err) && aligned16_ok(tl.start * 4, a.err)) {
                const float *src = nullptr;
                int k = RR::kShared;
                if (lane >= nrows) {   // the tile's shared curvature row
                    if (row_ok(0, 1, tl.start, lenr, d.wstride, a.err)) src = static_cast<const float *>(d.h) + tl.start;
                } else {
                    const int j = lane / RR::kPer, kind = lane % RR::kPer;
                    k = j * RR::kPer + kind;
                    if (row_ok(j, n, tl.start, lenr, d.wstride, a.err)) {
                        const int64_t o = j * d.wstride + tl.start;
                        const void *base = kind == RR::kIt ? (FROM_X ? d.x : d.y)
                                         : kind == RR::kM ? d.m
                                         : kind == RR::kVv ? d.v
                                         : kind == RR::kC ? d.c
                                         : (!FROM_X && kind == RR::kX) ? d.x
                                         : (PER_WORKER_H && kind == RR::kHw) ? d.h
                                                                              : d.b;
                        src = static_cast<const float *>(base) +
                              ((PER_WORKER_H && kind == RR::kHw) ? j * d.hstride + tl.start : o);
                    }
                }
                if (src) ptx::bulk_g2s(slot(s, k), src, bytes, &full[s]);
            }
            issued = it + 1;
        }
        if (aborted) {
            if (lane == 0) {
                abort_flag = 1;
                atomicCAS(a.err, static_cast<int32_t>(kDevOk), static_cast<int32_t>(kDevWaitTimeout));
            }
            // copies still in flight land before the CTA leaves (bounded)
            for (int64_t j = issued - kStages > 0 ? issued - kStages : 0; j < issued; ++j)
                ptx::mbar_wait_bounded(&full[j % kStages], static_cast<uint32_t>((j / kStages) & 1), kWaitNs);
            ce_acc = __longlong_as_double(0x7ff8000000000000ll);   // a NaN partial: the round failed
        }
    } else {
        // ------------------------------------------------------------ consumers ---
        dense_rows(a.topo, dr, n, a.err);
        if (threadIdx.x < n) {   // this step's scalars of worker i
            const int i = threadIdx.x;
            s_nstep[i] = -a.table->step[i];
            s_isb[i] = a.table->isb[i];
            s_dec[i] = a.sched ? a.table->decay[i] : a.decay;
            s_klo[i] = a.table->key_lo[i];
            s_khi[i] = a.table->key_hi[i];
        }
        consumer_sync();
        // The last CTA to have read the step's scalars (atomic ticket; nothing
        // waits) advances every worker's counters and writes the next step's
        // scalars, while the other CTAs already work on their tiles.
        if (threadIdx.x == 0) last_copy = atomicAdd(a.step_ticket, 1u) == gridDim.x - 1u;
        consumer_sync();
        if (last_copy && threadIdx.x < 32) {
            const int i = threadIdx.x;
            if (i < n)
                advance_step(a.state, a.table, i, a.beta1d, a.beta2d, a.lr_sched, a.lr_steps, a.lr_after, a.wd,
                             a.seed);
            if (i == 0) *a.step_ticket = 0u;
        }
        const Consts kc{x2::splat(a.beta1), x2::splat(a.beta2), x2::splat(a.omb1), x2::splat(a.omb2),
                        x2::splat(a.eps), x2::splat(a.sigma)};
        const OuterK ok2{x2::splat(-a.eta_out), x2::splat(a.mu), x2::splat(a.alpha), x2::splat(a.oma),
                         x2::splat(a.gamma), x2::splat(a.eta)};
        const float inv_n = static_cast<float>(1.0 / n);
        const int e0 = kV * threadIdx.x;
        for (int64_t it = 0; it < my_n; ++it) {
            const int s = static_cast<int>(it % kStages);
            bool ok = abort_flag == 0;
            if (ok && !ptx::mbar_wait_bounded(&full[s], static_cast<uint32_t>((it / kStages) & 1), kWaitNs)) {
                ok = false;
                abort_flag = 1;
                atomicCAS(a.err, static_cast<int32_t>(kDevOk), static_cast<int32_t>(kDevWaitTimeout));
            }
            const TileDesc u = descs[s];
            const bool active = ok && e0 < u.len;
            const int64_t off = u.start + e0;
            const int nvalid = u.len - e0 < kV ? u.len - e0 : kV;
            const uint32_t k0 = static_cast<uint32_t>(u.goff + off);   // global index of the column's first element
            auto row = [&](int k) { return *reinterpret_cast<const T *>(slot(s, k) + e0); };

            // the local step of every worker (its rows read from the stage);
            // the new y joins the column's rows
            T rows[R::kRows][kColumnWorkers];
            const T hs = PER_WORKER_H || !active ? C::zero() : row(RR::kShared);
#pragma unroll
            for (int j = 0; j < kColumnWorkers; ++j) {
                rows[0][j] = rows[1][j] = rows[R::kRows - 1][j] = C::zero();
                if (!active || j >= n) continue;
                const int base = j * RR::kPer;
                const T itj = row(base + RR::kIt);
                const T xj = FROM_X ? itj : row(base + RR::kX);
                const T h = PER_WORKER_H ? row(base + RR::kHw) : hs;
                const T mj = row(base + RR::kM), vj = row(base + RR::kVv), cj = row(base + RR::kC);
                const float2 nstep = x2::splat(s_nstep[j]), isb = x2::splat(s_isb[j]), dec = x2::splat(s_dec[j]);
                const uint32_t klo = s_klo[j], khi = s_khi[j];
                float2 yo[NP], mo[NP], vo[NP];
#pragma unroll
                for (int p = 0; p < NP; ++p)
                    yo[p] = adamw_pair(C::pair(itj, p), C::pair(mj, p), C::pair(vj, p), C::pair(cj, p), C::pair(h, p),
                                       noise_pair(k0 + 2 * p, klo, khi), nstep, isb, dec, kc, mo[p], vo[p]);
                const T yn = C::join(yo);
                if (row_ok(j, n, off, kV, u.wstride, a.err)) {
                    const int64_t o = j * u.wstride + off;
                    if (nvalid == kV) {
                        C::store(u.y + o, yn);
                        C::store(u.m + o, C::join(mo));
                        C::store(u.v + o, C::join(vo));
                    } else {
                        for (int l = 0; l < nvalid; ++l) {
                            const int p = l >> 1;
                            u.y[o + l] = (l & 1) ? yo[p].y : yo[p].x;
                            u.m[o + l] = (l & 1) ? mo[p].y : mo[p].x;
                            u.v[o + l] = (l & 1) ? vo[p].y : vo[p].x;
                        }
                    }
                }
                rows[0][j] = R::kMixX ? xj : yn;   // the mixed quantity: y (x in the DAdam modes)
                rows[1][j] = R::kMixX ? yn : xj;   // own x (own y in the DAdam modes)
                if (R::kHasB) rows[R::kRows - 1][j] = row(base + RR::kB);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[s]);   // every row of the stage is read
            if (active)
                column_update<MODE, kV>(rows, dr, n, ok2, round == 0, u.x, u.b, u.wstride, off, nvalid, inv_n,
                                        ce_acc, a.err);
        }
        if (abort_flag) ce_acc = __longlong_as_double(0x7ff8000000000000ll);
    }

    if (ce_partial_and_ticket(ce_acc, red, &last, a.partials, a.ticket) && threadIdx.x < 32) {
        const double sum = ce_sum_partials(a.partials);
        if (threadIdx.x == 0) {
            a.ce_ring[round % a.ce_ring_len] = sum / static_cast<double>(n);
            *a.ticket = 0u;
            a.state->round = round + 1;
        }
    }
}

template <int MODE>
const void *kernel_of(bool per_worker_h, bool from_x) {
    if (per_worker_h)
        return from_x ? reinterpret_cast<const void *>(round_kernel<MODE, true, true>)
                      : reinterpret_cast<const void *>(round_kernel<MODE, true, false>);
    return from_x ? reinterpret_cast<const void *>(round_kernel<MODE, false, true>)
                  : reinterpret_cast<const void *>(round_kernel<MODE, false, false>);
}

template <int MODE>
size_t smem_of(bool per_worker_h, bool from_x) {
    if (per_worker_h) return from_x ? Rows<MODE, true, true>::kSmem : Rows<MODE, true, false>::kSmem;
    return from_x ? Rows<MODE, false, true>::kSmem : Rows<MODE, false, false>::kSmem;
}

const void *round_kernel_ptr(int mode, bool per_worker_h, bool from_x) {
    switch (mode) {
    case kOutSgd: return kernel_of<kOutSgd>(per_worker_h, from_x);
    case kOutSgdm: return kernel_of<kOutSgdm>(per_worker_h, from_x);
    case kOutNesterov: return kernel_of<kOutNesterov>(per_worker_h, from_x);
    case kOutEq2: return kernel_of<kOutEq2>(per_worker_h, from_x);
    case kOutDadam: return kernel_of<kOutDadam>(per_worker_h, from_x);
    default: return kernel_of<kOutLocalDadam>(per_worker_h, from_x);
    }
}

size_t round_smem(int mode, bool per_worker_h, bool from_x) {
    switch (mode) {
    case kOutSgd: return smem_of<kOutSgd>(per_worker_h, from_x);
    case kOutSgdm: return smem_of<kOutSgdm>(per_worker_h, from_x);
    case kOutNesterov: return smem_of<kOutNesterov>(per_worker_h, from_x);
    case kOutEq2: return smem_of<kOutEq2>(per_worker_h, from_x);
    case kOutDadam: return smem_of<kOutDadam>(per_worker_h, from_x);
    default: return smem_of<kOutLocalDadam>(per_worker_h, from_x);
    }
}

}  // namespace

bool round_fits(int n, int storage) { return storage == kStoreF32 && n >= 1 && n <= kColumnWorkers; }

int round_blocks_per_sm(int mode, bool per_worker_h) {
    int lo = 0;
    for (int fx = 0; fx < 2; ++fx) {   // the smaller of the two variants' occupancies
        const void *f = round_kernel_ptr(mode, per_worker_h, fx != 0);
        const size_t smem = round_smem(mode, per_worker_h, fx != 0);
        int nb = 0;
        if (cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) !=
                cudaSuccess ||
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, f, kThreads, smem) != cudaSuccess)
            return 1;
        lo = fx == 0 ? nb : (nb < lo ? nb : lo);
    }
    return lo > 0 ? lo : 1;
}

cudaError_t launch_round(const RoundArgs &a, int grid, cudaStream_t s) {
    if (a.n_workers < 1 || a.n_workers > kColumnWorkers || a.mode < 0 || a.mode > kOutLocalDadam || grid < 1)
        return cudaErrorInvalidValue;
    void *args[] = {const_cast<RoundArgs *>(&a)};
    const bool pwh = a.per_worker_h != 0, fx = a.from_x != 0;
    const cudaError_t e = cudaLaunchKernel(round_kernel_ptr(a.mode, pwh, fx), dim3(static_cast<unsigned>(grid)),
                                           dim3(kThreads), args, round_smem(a.mode, pwh, fx), s);
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace gasloc
