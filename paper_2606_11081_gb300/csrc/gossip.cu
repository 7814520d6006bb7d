// gossip.cu -- K_gossip: one communication round of Algorithm 1 (or Eq. 2 /
// DAdam / Local-DAdam) for all workers, fused with the outer optimizer and the
// consensus-error reduction of the new replicas.
//
// Pipeline (persistent grid, one or two CTAs per SM, static round-robin over
// tiles):
//  * one producer warp moves ALL data with the TMA engine: each array of a
//    tile goes as 2-D tensor-map boxes of [n workers x 256 elements] -- every
//    worker's sent slice (y_j, or x_j if no worker took a local step) plus
//    the workers' own rows the update needs (x_i, b_i) -- into an S-stage
//    shared-memory ring whose "full" mbarrier counts the bytes (one 1-D bulk
//    copy per worker instead when only some workers took local steps); after
//    the consumers release a stage ("empty" mbarrier) it writes the updated
//    rows back with box stores before refilling the stage;
//  * 256 consumer threads never touch global memory in the loop: thread
//    (g, c) owns the 4-element column c of the tile for workers g, g+G, ...
//    (G = 1 or 2 for n <= 8, 2 for n <= 16, 4 for n <= 32), reads the
//    neighbours' rows from shared memory, applies the outer update in place
//    and accumulates the column's consensus-error terms.  Lanes are processed
//    in pairs with f32x2 instructions (each lane rounded as the scalar
//    operation would round it).
// Every neighbour slice is read from HBM once per round however many workers
// mix it: GASLoC/Nesterov moves 20 bytes per worker-element (y 4, x 4 + 4,
// b 4 + 4).  No block-wide barrier is taken inside the loop (a consumer-only
// named barrier per tile lets one thread per column reduce the consensus-error
// terms of all workers when G > 1).
//
// Arithmetic per element, one rounding per operation (the oracle's order):
//   acc_i = sum_{j in N_i ascending} fma(w_ij, s_j, acc)
//   Nesterov: D = x - acc; b = fma(mu, b, D); x = fma(-eta_out, fma(mu, b, D), x)
//   (SGD, SGDM, Eq. 2, DAdam, Local-DAdam: see outer_pair).
// Consensus error: per element e = S2 - (S1/n) S1 with S1 = sum_i (x_i - s),
// S2 = sum_i (x_i - s)^2 over ascending i, s = worker 0's new x; fp32 per
// element (the thread owning the column, or for G > 1 one thread per column
// after the tile's barrier), each element's term widened to fp64 on its own
// (the direct kernel below: a column's four terms as their exact sum,
// ce_sum.cuh), one partial per CTA, the last CTA (atomic ticket, nothing
// waits) adds the partials in CTA order.
//
// Waiting: every mbarrier wait is bounded (2 s).  A consumer that times out
// records kDevWaitTimeout and the CTA stops computing but keeps arriving on
// its barriers; the producer stops issuing, waits (bounded) for copies it has
// in flight and for its stores, and the CTA returns a NaN partial so that the
// ticket protocol completes.
#include <cuda_runtime.h>

#include <cstddef>
#include <type_traits>

#include "check.cuh"
#include "elem.cuh"
#include "f32x2.cuh"
#include "internal.h"
#include "mix.cuh"
#include "ptx.cuh"

namespace gasloc {

namespace {

constexpr int kConsumers = 256;                      // 8 warps
constexpr int kThreads = kConsumers + 32;            // + producer warp
constexpr int kMaxStages = 4;
constexpr size_t kOffFull = sizeof(Topo);            // 8320
constexpr size_t kOffEmpty = kOffFull + 8 * kMaxStages;
constexpr size_t kOffRed = kOffEmpty + 8 * kMaxStages;
constexpr size_t kOffFlags = kOffRed + 8 * (kThreads / 32);
constexpr size_t kOffStages = 8704;
static_assert(kOffFlags + 16 <= kOffStages, "smem layout");
static_assert(kOffStages % 128 == 0, "stage alignment");
__host__ __device__ constexpr size_t stage_offset(int) { return kOffStages; }
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr int kBox = 256;                            // elements per TMA box row (at most)
// Threads per column above 16 workers: 8, so that a tile is 128 elements
// (box rows of 128) and a stage of 32 workers' 3 rows is 48 KB, which leaves
// room for more stages per SM than 96 KB stages would.
constexpr int kGroupsMany = 8;

// Lanes at or past nvalid (>= 1) take keep's value.
__device__ __forceinline__ float4 keep_tail(float4 v, float4 keep, int nvalid) {
    if (nvalid < 2) v.y = keep.y;
    if (nvalid < 3) v.z = keep.z;
    if (nvalid < 4) v.w = keep.w;
    return v;
}

// Two consecutive elements from shared memory (8-byte aligned for fp32).
__device__ __forceinline__ float2 load2_smem(const float *p) { return *reinterpret_cast<const float2 *>(p); }
__device__ __forceinline__ float2 load2_smem(const bf16 *p) {
    const uint32_t u = *reinterpret_cast<const uint32_t *>(p);
    return make_float2(bf_lo(u), bf_hi(u));
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(ptx::smem_addr(bar)) : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_all() {
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// 2-D tensor copies through a tensor map in global memory: coordinates are
// {element, worker}; the element coordinate is a multiple of 4 (16 bytes).
__device__ __forceinline__ void tma_load_2d(void *dst_smem, const void *tmap, int32_t c0, int32_t c1,
                                            uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            ptx::smem_addr(dst_smem)),
        "l"(tmap), "r"(c0), "r"(c1), "r"(ptx::smem_addr(bar))
        : "memory");
}
__device__ __forceinline__ void tma_store_2d(const void *tmap, int32_t c0, int32_t c1, const void *src_smem) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(tmap), "r"(c0),
                 "r"(c1), "r"(ptx::smem_addr(src_smem))
                 : "memory");
}
// L2 policies of the TMA copies: 0 = no hint, 1 = evict first, 2 = evict
// last, 3 = evict normal (createpolicy, the whole line range).  Measured on
// the 8-worker GPT-2-small workload: evict-last loads and stores 0.987 of the
// copy peak, no hint 0.972, evict-first 0.963 (the 16- and 32-worker
// workloads: equal or slightly better with evict-last).
constexpr int kLoadPolicy = 2, kStorePolicy = 2;
template <int P>
__device__ __forceinline__ uint64_t l2_policy() {
    uint64_t pol = 0;
    if constexpr (P == 1)
        asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    else if constexpr (P == 2)
        asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    else if constexpr (P == 3)
        asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
template <int P>
__device__ __forceinline__ void tma_load_2d_p(void *dst_smem, const void *tmap, int32_t c0, int32_t c1, uint64_t *bar,
                                              uint64_t pol) {
    if constexpr (P == 0) {
        tma_load_2d(dst_smem, tmap, c0, c1, bar);
    } else {
        asm volatile(
            "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
            " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(ptx::smem_addr(dst_smem)),
            "l"(tmap), "r"(c0), "r"(c1), "r"(ptx::smem_addr(bar)), "l"(pol)
            : "memory");
    }
}
template <int P>
__device__ __forceinline__ void tma_store_2d_p(const void *tmap, int32_t c0, int32_t c1, const void *src_smem,
                                               uint64_t pol) {
    if constexpr (P == 0) {
        tma_store_2d(tmap, c0, c1, src_smem);
    } else {
        asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group.L2::cache_hint [%0, {%1, %2}], [%3], %4;" ::"l"(
                         tmap),
                     "r"(c0), "r"(c1), "r"(ptx::smem_addr(src_smem)), "l"(pol)
                     : "memory");
    }
}
__device__ __forceinline__ void tmap_acquire(const void *tmap) {
    asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(tmap) : "memory");
}

// Named barrier 1 over the 256 consumer threads (the producer warp never
// takes it).  The non-aligned form: threads of a warp may arrive separately.
__device__ __forceinline__ void consumer_barrier() {
    asm volatile("barrier.sync 1, %0;" ::"r"(kConsumers) : "memory");
}

// DENSE (bf16, one thread per column, n <= 8, not Eq. 2): the thread widens the n
// mixed rows of its column once and forms each worker's mix over the j < n
// of its neighbourhood in ascending order, with a dense weight row and a
// neighbour bitmask built from the round's table in the prologue.  The terms
// and their order are those of the neighbour lists, so the sums are the same
// bit for bit, and a non-finite row (a diverged replica) reaches only the
// workers that mix it.
constexpr int kDenseMax = 8;
constexpr int kDenseRow = 8;   // dense row i lives in tp->w[kDenseRow + i] and its neighbour mask in
                               // tp->nbr[kDenseRow + i][0] (rows >= n are free)

// NARROW: 128-element tiles and box rows (kGroupsMany threads per column,
// more than 16 workers); otherwise box rows of 256 elements.
template <int MODE, typename T, bool DENSE, bool NARROW>
__global__ void __launch_bounds__(kThreads, MODE == kOutEq2 ? 1 : 2) gossip_kernel(const GossipArgs a) {
    using R = ModeRows<MODE>;
    using E = Elem<T>;
    extern __shared__ __align__(128) unsigned char smem[];
    Topo *tp = reinterpret_cast<Topo *>(smem);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + kOffFull);
    uint64_t *empty = reinterpret_cast<uint64_t *>(smem + kOffEmpty);
    double *red = reinterpret_cast<double *>(smem + kOffRed);
    volatile int *flags = reinterpret_cast<volatile int *>(smem + kOffFlags);   // [0] abort, [1] last
    T *stages = reinterpret_cast<T *>(smem + stage_offset(a.groups));

    const int n = a.n_workers;
    const int TILE = a.tile;
    const int G = a.groups;
    const int cols = TILE / 4;
    const int S = a.stages;
    const size_t stage_elems = static_cast<size_t>(R::kRows) * n * TILE;
    constexpr int kVec = 16 / static_cast<int>(sizeof(T));   // elements per 16 bytes
    constexpr int bsh = NARROW ? 7 : 8;   // elements per box row (the tensor maps' box): 1 << bsh
    constexpr int BOX = 1 << bsh;
    const int NQ = TILE / BOX;   // sub-boxes per tile: kind k, sub-box q, worker j at ((k NQ + q) n + j) BOX
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    {   // neighbour table -> shared memory: rows 0..n-1 of nbr and w, and deg,
        // in 16-byte pieces (one or two per thread)
        static_assert(sizeof(Topo) % 16 == 0 && kMaxWorkers * 4 % 16 == 0, "Topo layout");
        constexpr int kRow = kMaxWorkers * 4 / 16;                         // pieces per row
        constexpr int kW = offsetof(Topo, w) / 16, kDeg = offsetof(Topo, deg) / 16;
        constexpr int kAll = sizeof(Topo) / 16;
        const int rows = n * kRow;
        const int4 *src = reinterpret_cast<const int4 *>(a.topo);
        int4 *dst = reinterpret_cast<int4 *>(tp);
        for (int q = threadIdx.x; q < 2 * rows + (kAll - kDeg); q += blockDim.x) {
            const int at = q < rows ? q : (q < 2 * rows ? kW + q - rows : kDeg + q - 2 * rows);
            dst[at] = src[at];
        }
    }
    if constexpr (DENSE) {   // dense weights and neighbour masks of the round, from the table in global memory
        const int t = threadIdx.x;
        if (t < kDenseMax * kDenseMax) {
            const int i = t / kDenseMax, j = t % kDenseMax;
            if (i < n && j < n) {
                float wij = 0.f;
                const int dg = a.topo->deg[i];
                for (int q = 0; q <= dg && q < kMaxWorkers; ++q)
                    if (a.topo->nbr[i][q] == j) wij = a.topo->w[i][q];
                tp->w[kDenseRow + i][j] = wij;
            }
        } else if (t < kDenseMax * kDenseMax + kDenseMax) {
            const int i = t - kDenseMax * kDenseMax;
            if (i < n) {
                uint32_t mask = 0;
                const int dg = a.topo->deg[i];
                for (int q = 0; q <= dg && q < kMaxWorkers; ++q) {
                    const int j = a.topo->nbr[i][q];
                    if (span_ok(j, j + 1, kDenseMax, a.err)) mask |= 1u << j;
                }
                tp->nbr[kDenseRow + i][0] = static_cast<int32_t>(mask);
            }
        }
    }
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], kConsumers / 32);
        }
        ptx::fence_mbar_init();
        flags[0] = 0;
        flags[1] = 0;
    }
    __syncthreads();

    const int64_t first = blockIdx.x, gstride = gridDim.x;
    const int64_t my_n = a.ntiles > first ? (a.ntiles - first + gstride - 1) / gstride : 0;
    double ce_acc = 0.0;
    // the round being executed; every CTA reads it before the last one to
    // finish advances it
    const int64_t round = __ldcg(&a.state->round);
    const bool first_round = round == 0;

    if (warp == kConsumers / 32) {
        // ------------------------------------------------------ producer ---
        // The whole warp moves the data.  Each array of a tile is loaded as
        // ceil(len / 256) 2-D boxes of [n workers x 256 elements] through the
        // tensor maps (one TMA operation for all workers; elements beyond the
        // tensor read as zero) and stored back the same way (writes beyond
        // the tensor are dropped).  Rows whose source differs between workers
        // (some workers took no local step this round) go as one 1-D bulk
        // copy per worker and sub-box instead.  Waits and abort decisions are
        // warp-uniform.
        const uint64_t ld_pol = l2_policy<kLoadPolicy>(), st_pol = l2_policy<kStorePolicy>();
        const uint32_t all_mask = n >= 32 ? 0xffffffffu : ((1u << n) - 1u);
        const bool all_fresh = (a.fresh_mask & all_mask) == all_mask;
        const bool none_fresh = (a.fresh_mask & all_mask) == 0u;
        const bool uniform = all_fresh || none_fresh;
        const int kvar = R::kMixX ? 1 : 0;   // the kind whose source depends on freshness
        auto blk = [&](T *st, int k, int q) { return st + static_cast<size_t>(k * NQ + q) * n * BOX; };
        auto tmap = [&](int tensor, int arr) {   // arr: 0 x, 1 y, 2 b
            return static_cast<const unsigned char *>(a.maps) + (static_cast<size_t>(tensor) * 3 + arr) * 128;
        };
        auto arr_of = [&](int k) {   // array a box of kind k is loaded from (uniform case)
            if (k == 2) return 2;
            if (k == kvar) return all_fresh ? 1 : 0;
            return 0;
        };
        int32_t fenced = -1;
        auto fence_maps = [&](int tensor) {   // maps written before launch: order them for the TMA proxy
            if (tensor == fenced) return;
            for (int arr = 0; arr < 3; ++arr) tmap_acquire(tmap(tensor, arr));
            fenced = tensor;
        };
        auto store_tile = [&](int64_t j) {   // box stores of tile j, spread over lanes
            const Tile tl = a.tiles[first + j * gstride];
            const int nq = (tl.len + BOX - 1) / BOX;
            T *st = stages + (j % S) * stage_elems;
            const int nops = (R::kHasB ? 2 : 1) * nq;
            fence_maps(tl.tensor);
            for (int o = lane; o < nops; o += 32) {
                const int k = 1 + o / nq, q = o % nq;
                const int arr = k == 1 ? 0 : 2;
                if (!aligned16_ok((tl.start + q * BOX) * static_cast<int64_t>(sizeof(T)), a.err)) continue;
                tma_store_2d_p<kStorePolicy>(tmap(tl.tensor, arr), static_cast<int32_t>(tl.start + q * BOX), 0,
                                             blk(st, k, q), st_pol);
            }
            bulk_commit();
        };
        auto wait_all_lanes = [&](uint64_t *bar, int64_t j) {
            const bool ok = ptx::mbar_wait_bounded(bar, static_cast<uint32_t>((j / S) & 1), kWaitLimitNs);
            return __all_sync(0xffffffffu, ok);
        };
        int64_t issued = 0;
        bool aborted = false;
        for (int64_t it = 0; it < my_n; ++it) {
            const int s = static_cast<int>(it % S);
            if (it >= S) {
                const int64_t j = it - S;
                if (!wait_all_lanes(&empty[s], j)) {
                    aborted = true;
                    break;
                }
                store_tile(j);
                bulk_wait_read_all();   // this lane's stores have read the stage
                __syncwarp();
            }
            if (__any_sync(0xffffffffu, flags[0] != 0)) {
                aborted = true;
                break;
            }
            const Tile tl = a.tiles[first + it * gstride];
            const TensorDesc &d = a.tens[tl.tensor];
            const int nq = (tl.len + BOX - 1) / BOX;
            const int lenr = (tl.len + kVec - 1) / kVec * kVec;   // whole 16-byte chunks
            T *st = stages + s * stage_elems;
            fence_maps(tl.tensor);
            // bytes this stage will receive
            uint32_t tx = 0;
            for (int k = 0; k < R::kRows; ++k) {
                if (k == kvar && !uniform) tx += static_cast<uint32_t>(n) * static_cast<uint32_t>(lenr) * sizeof(T);
                else tx += static_cast<uint32_t>(nq) * static_cast<uint32_t>(n * BOX * sizeof(T));
            }
            if (lane == 0) ptx::mbar_arrive_expect_tx(&full[s], tx);
            __syncwarp();
            const int nbox = R::kRows * nq;
            for (int o = lane; o < nbox; o += 32) {
                const int k = o / nq, q = o % nq;
                if (k == kvar && !uniform) continue;
                if (!aligned16_ok((tl.start + q * BOX) * static_cast<int64_t>(sizeof(T)), a.err)) continue;
                tma_load_2d_p<kLoadPolicy>(blk(st, k, q), tmap(tl.tensor, arr_of(k)),
                                           static_cast<int32_t>(tl.start + q * BOX), 0, &full[s], ld_pol);
            }
            if (!uniform) {   // per-worker source: y if the worker is fresh, else x
                for (int j = lane; j < n; j += 32) {
                    const bool fresh = (a.fresh_mask >> j) & 1u;
                    const T *src = static_cast<const T *>(fresh ? d.y : d.x) + j * d.wstride + tl.start;
                    for (int q = 0; q < nq; ++q) {
                        const int w = lenr - q * BOX < BOX ? lenr - q * BOX : BOX;
                        if (!row_ok(j, n, tl.start + q * BOX, w, d.wstride, a.err) ||
                            !aligned16_ok(static_cast<int64_t>(w) * sizeof(T), a.err))
                            continue;
                        ptx::bulk_g2s(blk(st, kvar, q) + static_cast<size_t>(j) * BOX, src + q * BOX,
                                      static_cast<uint32_t>(w * sizeof(T)), &full[s]);
                    }
                }
            }
            issued = it + 1;
        }
        if (!aborted) {
            for (int64_t j = my_n - S > 0 ? my_n - S : 0; j < my_n; ++j) {
                if (!wait_all_lanes(&empty[j % S], j)) {
                    aborted = true;
                    break;
                }
                store_tile(j);
            }
        }
        if (aborted) {
            if (lane == 0) {
                flags[0] = 1;
                atomicCAS(a.err, kDevOk, kDevWaitTimeout);
            }
            // copies still in flight land before the CTA leaves (bounded)
            for (int64_t j = issued - S > 0 ? issued - S : 0; j < issued; ++j)
                ptx::mbar_wait_bounded(&full[j % S], static_cast<uint32_t>((j / S) & 1), kWaitLimitNs);
        }
        bulk_wait_all();   // this lane's stores complete before the CTA leaves
        __syncwarp();
    } else {
        // ------------------------------------------------------ consumers ---
        const int g = threadIdx.x / cols;
        const int col = threadIdx.x % cols;
        const int e0 = 4 * col;
        const int qb = e0 >> bsh, rb = e0 & (BOX - 1);   // sub-box of the column, offset in it
        const float inv_n = static_cast<float>(1.0 / n);
        const OuterK ok2{x2::splat(-a.eta_out), x2::splat(a.mu), x2::splat(a.alpha), x2::splat(a.oma),
                         x2::splat(a.gamma), x2::splat(a.eta)};
        for (int64_t it = 0; it < my_n; ++it) {
            const int s = static_cast<int>(it % S);
            bool ok = !flags[0];
            if (ok && !ptx::mbar_wait_bounded(&full[s], static_cast<uint32_t>((it / S) & 1), kWaitLimitNs)) {
                ok = false;
                flags[0] = 1;
                atomicCAS(a.err, kDevOk, kDevWaitTimeout);
            }
            const int tlen = a.tiles[first + it * gstride].len;
            T *st = stages + s * stage_elems;
            // row of worker j, kind k, at this thread's column
            auto cp = [&](int k, int j) {
                return st + (static_cast<size_t>(k) * NQ + qb) * n * BOX + static_cast<size_t>(j) * BOX + rb;
            };
            float2 s1a = x2::splat(0.f), s1b = s1a, s2a = s1a, s2b = s1a;   // lanes 0-1, 2-3
            const bool active = ok && e0 < tlen;
            const int nvalid = tlen - e0 < 4 ? tlen - e0 : 4;
            float4 xr[8], br[8];                      // Eq. 2 results, written after a barrier
            int nr = 0;                               // Eq. 2 results held
            if (active) {
                float4 sh = make_float4(0.f, 0.f, 0.f, 0.f);   // G = 1: worker 0's new x (set at i = 0)
                float4 sall[DENSE ? kDenseMax : 1];           // DENSE: the column's mixed rows, widened once
                if constexpr (DENSE) {
#pragma unroll
                    for (int j = 0; j < kDenseMax; ++j)
                        if (j < n) sall[j] = E::load4_smem(cp(0, j));
                }
                for (int i = g; i < n; i += G) {
                    float2 acc01 = x2::splat(0.f), acc23 = acc01;
                    if constexpr (DENSE) {
                        const float *wr = &tp->w[kDenseRow + i][0];
                        const uint32_t nm = static_cast<uint32_t>(tp->nbr[kDenseRow + i][0]);
#pragma unroll
                        for (int j = 0; j < kDenseMax; ++j) {
                            if (j < n && ((nm >> j) & 1u)) {
                                const float2 w = x2::splat(wr[j]);
                                acc01 = x2::fma(w, x2::lo(sall[j]), acc01);
                                acc23 = x2::fma(w, x2::hi(sall[j]), acc23);
                            }
                        }
                    }
                    int dg = -1;   // DENSE: every neighbour was taken above
                    if constexpr (!DENSE) {
                        dg = tp->deg[i];
                        if (!span_ok(dg, dg + 1, kMaxWorkers, a.err)) dg = -1;
                    }
                    for (int q = 0; q <= dg; ++q) {
                        const int j = tp->nbr[i][q];
                        if (!span_ok(j, j + 1, n, a.err)) continue;
                        const float2 w = x2::splat(tp->w[i][q]);
                        const float4 sj = E::load4_smem(cp(0, j));
                        float2 s01 = x2::lo(sj), s23 = x2::hi(sj);
                        if (MODE == kOutEq2) {   // z_j = x_j + eta (y_j - x_j)
                            const float4 xj = E::load4_smem(cp(1, j));
                            s01 = x2::fma(ok2.eta, x2::sub(s01, x2::lo(xj)), x2::lo(xj));
                            s23 = x2::fma(ok2.eta, x2::sub(s23, x2::hi(xj)), x2::hi(xj));
                        }
                        acc01 = x2::fma(w, s01, acc01);
                        acc23 = x2::fma(w, s23, acc23);
                    }
                    T *p0 = cp(0, i);   // mixed row i
                    T *p1 = cp(1, i);   // own x (own y in the DAdam modes)
                    T *p2 = cp(2, i);   // own b
                    float4 xo, yo, zo = make_float4(0.f, 0.f, 0.f, 0.f), bo = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (R::kMixX) {
                        xo = E::load4_smem(p0);
                        yo = E::load4_smem(p1);
                    } else {
                        xo = E::load4_smem(p1);
                        yo = xo;
                    }
                    if (R::kHasB) bo = E::load4_smem(p2);
                    if (MODE == kOutEq2) {
                        const float4 y0 = E::load4_smem(p0);
                        zo = x2::join(x2::fma(ok2.eta, x2::sub(x2::lo(y0), x2::lo(xo)), x2::lo(xo)),
                                      x2::fma(ok2.eta, x2::sub(x2::hi(y0), x2::hi(xo)), x2::hi(xo)));
                    }
                    const float4 zp = (MODE == kOutEq2 && first_round) ? zo : bo;
                    float2 b01 = x2::lo(bo), b23 = x2::hi(bo);
                    // the consensus error is that of the replicas as stored
                    const float2 n01 = E::round2(outer_pair<MODE>(acc01, x2::lo(xo), x2::lo(yo), b01, x2::lo(zo),
                                                                  x2::lo(zp), ok2));
                    const float2 n23 = E::round2(outer_pair<MODE>(acc23, x2::hi(xo), x2::hi(yo), b23, x2::hi(zo),
                                                                  x2::hi(zp), ok2));
                    float4 xn4 = x2::join(n01, n23), bn4 = x2::join(b01, b23);
                    if (nvalid < 4) {   // padding keeps its value
                        xn4 = keep_tail(xn4, R::kMixX ? yo : xo, nvalid);
                        bn4 = keep_tail(bn4, bo, nvalid);
                    }
                    if (G == 1) {   // one thread sees every worker of the column
                        if (i == 0) sh = xn4;
                        ce_terms(x2::lo(xn4), x2::lo(sh), s1a, s2a);
                        ce_terms(x2::hi(xn4), x2::hi(sh), s1b, s2b);
                    }
                    if (MODE == kOutEq2) {
                        if (!span_ok(nr, nr + 1, 8, a.err)) break;
                        xr[nr] = xn4;
                        br[nr] = bn4;
                        ++nr;
                    } else {
                        E::store4_smem(p1, xn4);   // own row: read by this thread only
                        if (R::kHasB) E::store4_smem(p2, bn4);
                    }
                }
            }
            if (MODE == kOutEq2) {
                // Other threads read x_j to form z_j, so the new rows are written
                // only after every consumer has finished reading.  One barrier
                // site, reached by every consumer thread on every tile.
                consumer_barrier();
                if (active) {
                    int r = 0;
                    for (int i = g; i < n && r < nr; i += G, ++r) {
                        E::store4_smem(cp(1, i), xr[r]);
                        E::store4_smem(cp(2, i), br[r]);
                    }
                }
            }
            if (G > 1) {
                // Every group's new rows are in shared memory after this
                // barrier.  The column's G threads share its 4 elements
                // (4 / G each, or one each for the first 4 of G >= 4), and
                // each reduces its elements exactly as the G = 1 path does:
                // shift by worker 0's new x, ascending i.
                consumer_barrier();
                if (active && G == 2) {   // elements 2g, 2g + 1 as a pair
                    const int l0 = 2 * g;
                    if (l0 < nvalid) {
                        const float2 x0 = load2_smem(cp(1, 0) + l0);
                        float2 s1 = x2::splat(0.f), s2 = s1;
                        for (int i = 0; i < n; ++i) ce_terms(load2_smem(cp(1, i) + l0), x0, s1, s2);
                        ce_acc += static_cast<double>(__fmaf_rn(-__fmul_rn(s1.x, inv_n), s1.x, s2.x));
                        if (l0 + 1 < nvalid)
                            ce_acc += static_cast<double>(__fmaf_rn(-__fmul_rn(s1.y, inv_n), s1.y, s2.y));
                    }
                } else if (active && g < 4 && g < nvalid) {   // G >= 4: element g
                    const float x0 = E::load1(cp(1, 0) + g);
                    float s1 = 0.f, s2 = 0.f;
                    for (int i = 0; i < n; ++i) {
                        const float dv = __fsub_rn(E::load1(cp(1, i) + g), x0);
                        s1 = __fadd_rn(s1, dv);
                        s2 = __fmaf_rn(dv, dv, s2);
                    }
                    ce_acc += static_cast<double>(__fmaf_rn(-__fmul_rn(s1, inv_n), s1, s2));
                }
            } else if (active) {
                // consensus-error terms of the column: e = S2 - (S1 / n) S1 per element
                const float s1[4] = {s1a.x, s1a.y, s1b.x, s1b.y}, s2[4] = {s2a.x, s2a.y, s2b.x, s2b.y};
#pragma unroll
                for (int l = 0; l < 4; ++l)   // each element's term enters the fp64 sum on its own
                    if (l < nvalid) ce_acc += static_cast<double>(__fmaf_rn(-__fmul_rn(s1[l], inv_n), s1[l], s2[l]));
            }
            ptx::fence_proxy_async_smem();   // outputs visible to the bulk stores
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[s]);
        }
    }

    if (flags[0]) ce_acc = __longlong_as_double(0x7ff8000000000000ll);   // NaN partial
    // block reduction: warp shuffles, then warps in order
    for (int o = 16; o > 0; o >>= 1) ce_acc += __shfl_down_sync(0xffffffffu, ce_acc, o);
    if (lane == 0) red[warp] = ce_acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double s = 0.0;
        for (int w = 0; w < kThreads / 32; ++w) s += red[w];
        a.partials[blockIdx.x] = s;
        __threadfence();
        const unsigned t = atomicAdd(a.ticket, 1u);
        flags[1] = (t == gridDim.x - 1) ? 1 : 0;
    }
    __syncthreads();
    if (flags[1] && warp == 0) {
        __threadfence();
        double s = 0.0;
        for (unsigned b = lane; b < gridDim.x; b += 32) s += __ldcg(a.partials + b);
        for (int o = 16; o > 0; o >>= 1) s += __shfl_down_sync(0xffffffffu, s, o);
        if (lane == 0) {
            a.ce_ring[round % a.ce_ring_len] = s / static_cast<double>(n);
            *a.ticket = 0u;
            a.state->round = round + 1;
        }
    }
}

// ---------------------------------------------------------------------------
// Direct variant for few workers and small replicas (n <= kDirectMaxWorkers,
// fp32, a few 1024-element tiles per CTA).  With a replica store of about a
// hundred MB each CTA of the pipelined kernel above walks only 3-4 tiles, and
// every tile pays the whole chain of a stage: TMA load, consumers, release,
// box stores reading the stage, reload.  Here each thread loads its column of
// 4 elements for every worker and every row the update needs straight into
// registers (all loads of the tile issued before any arithmetic), forms every
// worker's update and stores x and b back: one memory round trip per tile.
// The arithmetic, its order and the consensus-error terms are those of the
// kernel above with one thread per column, so the results are bit-identical.
constexpr int kDirectMaxWorkers = kColumnWorkers;
constexpr int kDirectThreads = 256;   // a column of 4 elements each: 1024-element tiles

template <int MODE>
__global__ void __launch_bounds__(kDirectThreads, 2) gossip_direct_kernel(const GossipArgs a) {
    using R = ModeRows<MODE>;
    using E = Elem<float>;
    __shared__ DenseRows dr;
    __shared__ double red[kDirectThreads / 32];
    __shared__ int last;
    const int n = a.n_workers;
    dense_rows(a.topo, dr, n, a.err);
    __syncthreads();
    const int64_t round = __ldcg(&a.state->round);
    const OuterK ok2{x2::splat(-a.eta_out), x2::splat(a.mu), x2::splat(a.alpha), x2::splat(a.oma),
                     x2::splat(a.gamma), x2::splat(a.eta)};
    const float inv_n = static_cast<float>(1.0 / n);
    const uint32_t fresh = a.fresh_mask;
    double ce_acc = 0.0;
    const int e0 = 4 * threadIdx.x;
    // tensor 0's descriptor read at once, beside the first tile's (a flat
    // store has no other)
    int32_t cur = 0;
    TensorDesc d = a.tens[0];
    for (int64_t ti = blockIdx.x; ti < a.ntiles; ti += gridDim.x) {
        const Tile tl = a.tiles[ti];
        if (e0 >= tl.len) continue;
        if (tl.tensor != cur) {
            d = a.tens[tl.tensor];
            cur = tl.tensor;
        }
        const float *X = static_cast<const float *>(d.x), *Y = static_cast<const float *>(d.y);
        const float *B = static_cast<const float *>(d.b);
        const int64_t off = tl.start + e0;
        // all loads of the tile issued before any arithmetic
        float4 rows[R::kRows][kDirectMaxWorkers];
#pragma unroll
        for (int j = 0; j < kDirectMaxWorkers; ++j) {
            if (j >= n || !row_ok(j, n, off, 4, d.wstride, a.err)) {
#pragma unroll
                for (int k = 0; k < R::kRows; ++k) rows[k][j] = make_float4(0.f, 0.f, 0.f, 0.f);
                continue;
            }
            const int64_t o = j * d.wstride + off;
            const bool fr = (fresh >> j) & 1u;
            const float *k0 = R::kMixX ? X : (fr ? Y : X);
            const float *k1 = R::kMixX ? (fr ? Y : X) : X;
            rows[0][j] = E::load4<Cache::kL2>(k0 + o);
            rows[1][j] = E::load4<Cache::kL2>(k1 + o);
            if (R::kHasB) rows[R::kRows - 1][j] = E::load4<Cache::kL2>(B + o);
        }
        column_update<MODE, 4>(rows, dr, n, ok2, round == 0, static_cast<float *>(d.x), static_cast<float *>(d.b),
                               d.wstride, off, tl.len - e0 < 4 ? tl.len - e0 : 4, inv_n, ce_acc, a.err);
    }
    // one partial per CTA; the last CTA adds them in CTA order, stores the
    // round's value and advances the round counter
    if (ce_partial_and_ticket(ce_acc, red, &last, a.partials, a.ticket) && threadIdx.x < 32) {
        const double sum = ce_sum_partials(a.partials);
        if (threadIdx.x == 0) {
            a.ce_ring[round % a.ce_ring_len] = sum / static_cast<double>(n);
            *a.ticket = 0u;
            a.state->round = round + 1;
        }
    }
}

void *direct_kernel(int mode) {
    switch (mode) {
    case kOutSgd: return reinterpret_cast<void *>(gossip_direct_kernel<kOutSgd>);
    case kOutSgdm: return reinterpret_cast<void *>(gossip_direct_kernel<kOutSgdm>);
    case kOutNesterov: return reinterpret_cast<void *>(gossip_direct_kernel<kOutNesterov>);
    case kOutEq2: return reinterpret_cast<void *>(gossip_direct_kernel<kOutEq2>);
    case kOutDadam: return reinterpret_cast<void *>(gossip_direct_kernel<kOutDadam>);
    default: return reinterpret_cast<void *>(gossip_direct_kernel<kOutLocalDadam>);
    }
}

template <int MODE>
void *kernel_ptr(int storage, bool dense, bool narrow) {
    // dense mixing exists for bf16 only, and not for Eq. 2; narrow tiles only
    // without it (more than 16 workers)
    constexpr bool kCanDense = MODE != kOutEq2;
    if (narrow)
        return storage == kStoreBF16 ? reinterpret_cast<void *>(gossip_kernel<MODE, bf16, false, true>)
                                     : reinterpret_cast<void *>(gossip_kernel<MODE, float, false, true>);
    if (storage != kStoreBF16) return reinterpret_cast<void *>(gossip_kernel<MODE, float, false, false>);
    if (dense && kCanDense) return reinterpret_cast<void *>(gossip_kernel<MODE, bf16, kCanDense, false>);
    return reinterpret_cast<void *>(gossip_kernel<MODE, bf16, false, false>);
}

void *mode_kernel(int mode, int storage, bool dense, bool narrow) {
    switch (mode) {
    case kOutSgd: return kernel_ptr<kOutSgd>(storage, dense, narrow);
    case kOutSgdm: return kernel_ptr<kOutSgdm>(storage, dense, narrow);
    case kOutNesterov: return kernel_ptr<kOutNesterov>(storage, dense, narrow);
    case kOutEq2: return kernel_ptr<kOutEq2>(storage, false, narrow);
    case kOutDadam: return kernel_ptr<kOutDadam>(storage, dense, narrow);
    default: return kernel_ptr<kOutLocalDadam>(storage, dense, narrow);
    }
}

int mode_rows(int mode) { return (mode == kOutSgd || mode == kOutDadam) ? 2 : 3; }

}  // namespace

GossipShape gossip_shape(int n, int mode, int storage) {
    GossipShape sh{};
    // Threads per column (G).  Measured on the 8-worker exponential graph:
    // fp32 streams best with two (more warps per byte in flight, 97% of
    // the copy peak against 91% with one); bf16, whose tile is half the
    // bytes, is issue-bound and loses the extra consensus-error pass (65%
    // against 70%).  Up to 4 workers one thread per column (the 4-worker
    // ring: 0.51 of the copy peak against 0.48 with two, 0.36 with four).
    // From 9 to 16 workers two threads per column, above eight (kGroupsMany: 128-element tiles).
    sh.groups = n <= 4 ? 1 : (n <= 8 ? (storage == kStoreBF16 ? 1 : 2) : (n <= 16 ? 2 : kGroupsMany));
    // Dense mixing (every row of the column widened once, then w_ij * s_j
    // over all j with w_ij = 0 off the graph) for bf16 with one thread per
    // column: the 8-worker exponential graph's gossip went from 0.885 to 1.006
    // of the copy peak.  fp32 keeps the neighbour lists (the 4-worker ring
    // was 2% slower dense), and so does Eq. 2, whose mixed rows are formed
    // per neighbour.
    sh.dense = (storage == kStoreBF16 && sh.groups == 1 && n <= kDenseMax && mode != kOutEq2) ? 1 : 0;
    sh.tile = 4 * (kConsumers / sh.groups);
    sh.block = kThreads;
    const size_t esize = storage == kStoreBF16 ? 2 : 4;
    const size_t stage = static_cast<size_t>(mode_rows(mode)) * n * sh.tile * esize;
    const size_t off = stage_offset(sh.groups);
    // two CTAs per SM (twice the consumer warps) when two stages fit in half
    // of the SM's shared memory; otherwise one CTA with up to four stages
    const size_t half = (233472 - 2 * 1024) / 2;
    const int st2 = static_cast<int>((half - off) / stage);
    if (mode != kOutEq2 && half > off && st2 >= 2) {
        sh.stages = st2 > kMaxStages ? kMaxStages : st2;
    } else {
        const int st = static_cast<int>((232448 - off) / stage);
        sh.stages = st < 2 ? 2 : (st > kMaxStages ? kMaxStages : st);
    }
    sh.smem = off + sh.stages * stage;
    return sh;
}

cudaError_t gossip_set_smem(size_t smem) {
    for (int st = 0; st <= kStoreBF16; ++st)
        for (int m = 0; m <= kOutLocalDadam; ++m)
            for (int v = 0; v < 3; ++v) {   // neighbour lists, dense, narrow
                const cudaError_t e = cudaFuncSetAttribute(mode_kernel(m, st, v == 1, v == 2),
                                                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                           static_cast<int>(smem));
                if (e != cudaSuccess) return e;
            }
    return cudaSuccess;
}

int gossip_direct_blocks_per_sm(int mode) {
    int nb = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, reinterpret_cast<const void *>(direct_kernel(mode)),
                                                      kDirectThreads, 0) != cudaSuccess)
        return 1;
    return nb > 0 ? nb : 1;
}

bool gossip_direct_fits(int n, int storage) { return storage == kStoreF32 && n <= kDirectMaxWorkers; }

int gossip_blocks_per_sm(int mode, int storage, const GossipShape &sh) {
    int nb = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(
            &nb, reinterpret_cast<const void *>(mode_kernel(mode, storage, sh.dense != 0, sh.tile == 128)), kThreads,
            sh.smem) != cudaSuccess)
        return 1;
    return nb > 0 ? nb : 1;
}

cudaError_t launch_gossip(const GossipArgs &a, int grid, size_t smem, cudaStream_t s) {
    if (a.stages < 2 || a.stages > kMaxStages || a.groups < 1 || a.tile != 4 * (kConsumers / a.groups) ||
        (a.tile != 128 && a.tile % kBox != 0) || (a.tile == 128 && a.dense) || a.maps == nullptr)
        return cudaErrorInvalidValue;
    void *args[] = {const_cast<GossipArgs *>(&a)};
    if (a.direct) {   // a.tiles is then the 1024-element tile table
        if (a.storage != kStoreF32 || a.n_workers > kDirectMaxWorkers) return cudaErrorInvalidValue;
        const cudaError_t e = cudaLaunchKernel(direct_kernel(a.mode), dim3(static_cast<unsigned>(grid)),
                                               dim3(kDirectThreads), args, 0, s);
        return e != cudaSuccess ? e : cudaGetLastError();
    }
    void *kernel = mode_kernel(a.mode, a.storage, a.dense != 0, a.tile == 128);
    const cudaError_t e = cudaLaunchKernel(kernel, dim3(static_cast<unsigned>(grid)), dim3(kThreads), args, smem, s);
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace gasloc
