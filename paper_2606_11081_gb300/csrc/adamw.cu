// adamw.cu -- K_adamw: one inner AdamW step (Algorithm 1, inner loop; App. B
// settings) for every active worker, all replicas in one launch.
//
// Memory-bound streaming kernels: per active worker and element they read the
// iterate (x on the first step of a round, else y), m, v and the centre c and
// write y, m, v -- 28 bytes in fp32 storage, 14 in bf16 -- plus the shared
// curvature h per element (h is per worker in the heterogeneous workload).
// The synthetic gradient g = h (y - c) + sigma xi is formed in registers; xi
// comes from a 32-bit counter hash of the element index and the step key (of
// the index of the element pair with bf16 storage), so the gradient costs no
// memory traffic.  The step's per-worker scalars (bias corrections, noise
// keys) come from the step table; the launch's last CTA to copy it advances
// the step counters and writes the next step's scalars.
//
// fp32 storage (adamw_kernel): one thread owns a column of 4 consecutive
// elements of a tile and walks the active workers U at a time (U from 2 to 4,
// chosen per launch from the number of workers stepped and whether each has
// its own h: see Batch), issuing all of their loads before any arithmetic;
// CTAs claim their tiles from a global counter.
// bf16 storage (adamw_staged_kernel): a producer warp stages the rows in
// shared memory with bulk copies while 256 consumer threads compute (see
// there); with half the bytes per element the arithmetic sets the pace, and
// the consumers must not wait on their own loads.
//
// Per element: the arithmetic of adamw_math.cuh (in fp32, one IEEE rounding
// per operation); with bf16 storage the loads widen exactly and each stored
// value is rounded to bf16 (nearest, ties to even).
#include <cuda_runtime.h>

#include <type_traits>

#include "adamw_math.cuh"
#include "check.cuh"
#include "elem.cuh"
#include "f32x2.cuh"
#include "internal.h"
#include "ptx.cuh"
#include "rng.cuh"
#include "step.cuh"

namespace gasloc {

namespace {

constexpr int kBlock = 256;   // threads; a tile is 4 * kBlock elements

// Cache policies of the global accesses.  Caching in L2 (.cg) rather than
// marking the lines evict-first measured 4% faster on the 8-worker GPT-2-small
// workload (1.008 against 0.966 of the copy peak) and 2% on the 16-worker one.
constexpr Cache kLdIterate = Cache::kL2, kLdMoments = Cache::kL2, kLdCentre = Cache::kL2, kLdCurv = Cache::kL2;
constexpr Cache kSt = Cache::kL2;

// bf16 storage, 16 bits per element: element 2j takes the low half of
// word(j), element 2j + 1 the high half, and xi = q * (sqrt3 * 2^-15) with
// q = half - 2^15.  A byte permute puts a half h in the mantissa of 2^23 (the
// float 2^23 + h, exact); subtracting 2^23 + 2^15 leaves q exactly, and the
// product is the one rounding.  One hash serves two elements, which matters
// where the arithmetic, not the memory, sets the pace.  Columns start at even
// k unless a tensor starts at an odd global index; then the 4 elements span 3
// words.
__device__ __forceinline__ float biased_half(uint32_t w, bool high) {
    return __uint_as_float(__byte_perm(w, 0x4B000000u, high ? 0x7632u : 0x7610u));
}
__device__ __forceinline__ void noise4_pairs(uint32_t k, uint32_t klo, uint32_t khi, float2 &xi01, float2 &xi23) {
    const uint32_t j = k >> 1;
    const uint32_t w0 = noise_word(j, klo, khi), w1 = noise_word(j + 1u, klo, khi);
    float2 b01, b23;
    if ((k & 1u) == 0) {
        b01 = make_float2(biased_half(w0, false), biased_half(w0, true));
        b23 = make_float2(biased_half(w1, false), biased_half(w1, true));
    } else {
        const uint32_t w2 = noise_word(j + 2u, klo, khi);
        b01 = make_float2(biased_half(w0, true), biased_half(w1, false));
        b23 = make_float2(biased_half(w1, true), biased_half(w2, false));
    }
    const float2 bias = x2::splat(8421376.0f);   // 2^23 + 2^15
    const float2 scale = x2::splat(static_cast<float>(1.7320508075688772) * 0x1p-15f);
    xi01 = x2::mul(x2::sub(b01, bias), scale);
    xi23 = x2::mul(x2::sub(b23, bias), scale);
}

// SCHED: the learning rate follows a schedule, so the weight-decay factor
// differs between workers and comes from the step table; otherwise it is the
// launch-wide fl32(1 - lr * weight_decay).
template <int U, bool PER_WORKER_H, bool SCHED, typename T>
__global__ void __launch_bounds__(kBlock, 2) adamw_kernel(const AdamwArgs a) {
    static_assert(std::is_same<T, float>::value, "bf16 storage runs adamw_staged_kernel");
    using E = Elem<T>;
    const Consts kc{x2::splat(a.beta1), x2::splat(a.beta2), x2::splat(a.omb1), x2::splat(a.omb2),
                    x2::splat(a.eps), x2::splat(a.sigma)};
    // this step's per-worker scalars -> shared
    __shared__ StepTable tab;
    __shared__ int last_copy;
    for (int q = threadIdx.x; q < static_cast<int>(sizeof(StepTable) / 4); q += blockDim.x)
        reinterpret_cast<uint32_t *>(&tab)[q] = reinterpret_cast<const uint32_t *>(a.table)[q];
    __syncthreads();
    // The last CTA to have copied the scalars (atomic ticket; nothing waits)
    // advances the stepped workers' counters and writes the scalars of their
    // next step, while the other CTAs already work on their tiles.
    if (threadIdx.x == 0) last_copy = atomicAdd(a.ticket, 1u) == gridDim.x - 1u;
    __syncthreads();
    if (last_copy && threadIdx.x < 32) {
        const int i = threadIdx.x;
        if (i < a.n_workers && ((a.active_mask >> i) & 1u))
            advance_step(a.state, a.table, i, a.beta1d, a.beta2d, a.lr_sched, a.lr_steps, a.lr_after, a.wd, a.seed);
        if (i == 0) *a.ticket = 0u;
    }
    int32_t cur = -1;
    TensorDesc d{};
    // Tiles: blockIdx.x first, then claimed one at a time from a global
    // counter (claim k is tile gridDim.x + k), so that a CTA that drew slower
    // memory simply takes fewer (a static split left the slowest CTAs setting
    // the launch's end: the claimed tiles took the 8-, 16- and 32-worker
    // workloads from 1.001 / 0.987 / 1.006 to 1.024 / 1.000 / 1.015 of the
    // copy peak).  Thread 0 claims the next tile while the block works on this
    // one and publishes it after the tile's barrier, in one of two slots (a
    // slot is rewritten only after every thread has read it).
    __shared__ long long next_tile[2];
    int par = 0;
    for (int64_t ti = blockIdx.x; ti < a.ntiles; par ^= 1) {
        if (threadIdx.x == 0)
            next_tile[par] = static_cast<long long>(gridDim.x) + static_cast<long long>(atomicAdd(a.work, 1ull));
        const Tile tl = a.tiles[ti];
        const int e0 = 4 * threadIdx.x;
        if (e0 < tl.len) {
            if (tl.tensor != cur) {
                d = a.tens[tl.tensor];
                cur = tl.tensor;
            }
            const T *X = as<T>(static_cast<const void *>(d.x));
            const T *C = as<T>(static_cast<const void *>(d.c));
            const T *Hh = as<T>(static_cast<const void *>(d.h));
            T *Yw = as<T>(d.y), *Mw = as<T>(d.m), *Vw = as<T>(d.v);
            const int64_t off = tl.start + e0;
            const int nvalid = tl.len - e0 < 4 ? tl.len - e0 : 4;
            const uint32_t k0 = static_cast<uint32_t>(d.goff + off);   // global index of the column's first element
            float4 hs = make_float4(0.f, 0.f, 0.f, 0.f);
            if (!PER_WORKER_H && row_ok(0, 1, off, 4, d.wstride, a.err)) hs = E::template load4<kLdCurv>(Hh + off);

            for (int a0 = 0; a0 < a.n_active; a0 += U) {
                // every load of the batch is issued before any arithmetic; the
                // raw words stay packed until their worker is processed
                typename E::Raw Y[U], M[U], V[U], Cc[U], Hw[U];
                bool okr[U];   // worker row and column inside its buffers (checked build)
    #pragma unroll
                for (int u = 0; u < U; ++u) {
                    okr[u] = a0 + u < a.n_active && row_ok(a.worker[a0 + u], a.n_workers, off, 4, d.wstride, a.err);
                    if (okr[u]) {
                        const int i = a.worker[a0 + u];
                        const int64_t o = i * d.wstride + off;
                        const T *src = ((a.from_x_mask >> i) & 1u) ? X : Yw;
                        Y[u] = E::template load_raw<kLdIterate>(src + o);
                        M[u] = E::template load_raw<kLdMoments>(Mw + o);
                        V[u] = E::template load_raw<kLdMoments>(Vw + o);
                        Cc[u] = E::template load_raw<kLdCentre>(C + o);
                        if (PER_WORKER_H) Hw[u] = E::template load_raw<kLdCurv>(Hh + i * d.hstride + off);
                    }
                }
    #pragma unroll
                for (int u = 0; u < U; ++u) {
                    if (okr[u]) {
                        const int i = a.worker[a0 + u];
                        const float2 nstep = x2::splat(-tab.step[i]);
                        const float2 isb = x2::splat(tab.isb[i]);
                        const float2 dec = SCHED ? x2::splat(tab.decay[i]) : x2::splat(a.decay);
                        const uint32_t klo = tab.key_lo[i], khi = tab.key_hi[i];
                        const float4 h4 = PER_WORKER_H ? E::unpack(Hw[u]) : hs;
                        const float4 Yu = E::unpack(Y[u]), Mu = E::unpack(M[u]), Vu = E::unpack(V[u]),
                                     Cu = E::unpack(Cc[u]);
                        float2 m01, v01, m23, v23;
                        const float2 y01 = adamw_pair(x2::lo(Yu), x2::lo(Mu), x2::lo(Vu), x2::lo(Cu), x2::lo(h4),
                                                      noise_pair(k0, klo, khi), nstep, isb, dec, kc, m01, v01);
                        const float2 y23 = adamw_pair(x2::hi(Yu), x2::hi(Mu), x2::hi(Vu), x2::hi(Cu), x2::hi(h4),
                                                      noise_pair(k0 + 2, klo, khi), nstep, isb, dec, kc, m23, v23);
                        const float4 yo = x2::join(y01, y23), mo = x2::join(m01, m23), vo = x2::join(v01, v23);
                        const int64_t o = i * d.wstride + off;
                        if (nvalid == 4) {
                            E::template store4<kSt>(Yw + o, yo);
                            E::template store4<kSt>(Mw + o, mo);
                            E::template store4<kSt>(Vw + o, vo);
                        } else {
                            const float ya[4] = {yo.x, yo.y, yo.z, yo.w};
                            const float ma[4] = {mo.x, mo.y, mo.z, mo.w};
                            const float va[4] = {vo.x, vo.y, vo.z, vo.w};
                            for (int l = 0; l < nvalid; ++l) {
                                E::store1(Yw + o + l, ya[l]);
                                E::store1(Mw + o + l, ma[l]);
                                E::store1(Vw + o + l, va[l]);
                            }
                        }
                    }
                }
            }
        }
        __syncthreads();
        ti = next_tile[par];
    }
    // every block has made its last claim before it counts itself out; the
    // last one returns the counter to 0 for the next launch
    if (threadIdx.x == 0) {
        __threadfence();
        if (atomicAdd(a.work + 1, 1ull) == gridDim.x - 1ull) {
            atomicExch(a.work, 0ull);
            atomicExch(a.work + 1, 0ull);
        }
    }
}

// ---------------------------------------------------------------------------
// Staged variant, used with bf16 storage.  With half the bytes per element
// the arithmetic, not the memory, sets the pace, and a thread that waits on
// its own loads (as above) leaves no loads in flight while it computes.  Here
// a producer warp keeps the HBM busy: for each unit of work (a tile of 1024
// elements for a group of G workers) its lanes issue one 1-D bulk copy per
// row -- the iterate (y, or x on the worker's first step of the round), m, v,
// c, and h (the tile's shared row, or each worker's own) -- into a ring of
// kStages shared-memory stages, completing on the stage's `full` mbarrier.
// The 256 consumer threads (a column of 4 elements each) read their rows from
// shared memory, take the step exactly as above and store y, m, v straight to
// global memory, then release the stage on its `empty` mbarrier.  Every wait
// is bounded: on a timeout the CTA records kDevWaitTimeout, stops computing
// but keeps releasing stages, and the producer stops issuing and waits
// (bounded) for the copies it has in flight before it leaves.
constexpr int kStagedConsumers = 256;
constexpr int kStagedThreads = kStagedConsumers + 32;
constexpr int kStagedTile = 4 * kStagedConsumers;   // elements per tile (the host's tile size)
constexpr uint64_t kStagedWaitNs = 2000000000ull;

template <typename T, bool PER_WORKER_H>
struct StagedShape {
    // bf16, measured on the 8-worker GPT-2-small bf16 workload (fraction of
    // the copy peak): groups of 4 workers, 2 stages, 3 CTAs per SM 0.931; 3
    // stages and 2 CTAs 0.842; groups of 2 with 3 or 4 stages and 3 CTAs
    // 0.853 / 0.856; single workers, 4 stages, 4 CTAs 0.725.  fp32 (small
    // replica stores only), measured on the 4-worker 1 Mi ring: groups of 2
    // workers with 3 stages of 4 KB rows and 2 CTAs per SM 0.781; 2 stages
    // and 3 CTAs 0.769; single workers, 4 stages 0.727; groups of 4 with 2
    // stages (one CTA) 0.669; against 0.707 for the register-batched kernel.
    static constexpr bool kBf = std::is_same<T, bf16>::value;
    static constexpr int kGroup = kBf ? (PER_WORKER_H ? 3 : 4) : 2;   // workers per unit
    static constexpr int kStages = kBf ? 2 : 3;                   // ring depth
    static constexpr int kMinBlocks = kBf ? 3 : 2;                // CTAs per SM
    // Units claimed from a global counter (bf16: 0.962 -> 1.025 of the copy
    // peak on the 8-worker GPT-2-small bf16 workload, whose ~2,000 units per
    // CTA let slower CTAs fall behind a static split), or a static grid stride
    // (fp32 small stores: at a few units per CTA the claim's latency cost more,
    // 0.78 -> 0.72 on the 4-worker 1 Mi ring).
    static constexpr bool kDynamic = kBf;
    static constexpr int kArrs = PER_WORKER_H ? 5 : 4;            // rows per worker
    static constexpr int kSegs = kArrs * kGroup + (PER_WORKER_H ? 0 : 1);
    static constexpr size_t kStageBytes = static_cast<size_t>(kSegs) * kStagedTile * sizeof(T);
    static constexpr size_t kBarOffset = kStages * kStageBytes;
    static constexpr size_t kDescOffset = kBarOffset + 2 * kStages * sizeof(uint64_t);
    static constexpr size_t kSmem = kDescOffset + kStages * 64;
};

// What the consumers need of a unit's tile, written by the producer beside
// the stage's rows (so that the consumers make no global loads of their own).
struct UnitDesc {
    int64_t start, wstride, goff;   // tile start in the tensor, row stride, global index of element 0
    void *y, *m, *v;
    int32_t len;                    // elements of the tile; -1: no unit is left (the stage carries no rows)
    int32_t a0;                     // the unit's first worker slot (index into a.worker)
};
static_assert(sizeof(UnitDesc) <= 64, "one 64-byte slot per stage");

__device__ __forceinline__ void mbar_release(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(ptx::smem_addr(bar)) : "memory");
}

// Barrier of the staged kernel's consumer warps only (the producer does not take part).
__device__ __forceinline__ void staged_consumer_sync() {
    asm volatile("barrier.sync 1, %0;" ::"r"(kStagedConsumers) : "memory");
}

template <bool PER_WORKER_H, bool SCHED, typename T = bf16>
__global__ void __launch_bounds__(kStagedThreads, StagedShape<T, PER_WORKER_H>::kMinBlocks)
    adamw_staged_kernel(const AdamwArgs a) {
    using E = Elem<T>;
    using SS = StagedShape<T, PER_WORKER_H>;
    constexpr int kVec = 16 / static_cast<int>(sizeof(T));   // elements per 16-byte piece
    constexpr int G = SS::kGroup;
    constexpr int kStages = SS::kStages;
    extern __shared__ __align__(128) unsigned char smem[];
    T *stages = reinterpret_cast<T *>(smem);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + SS::kBarOffset);
    uint64_t *empty = full + kStages;
    UnitDesc *descs = reinterpret_cast<UnitDesc *>(smem + SS::kDescOffset);
    __shared__ StepTable tab;
    __shared__ int abort_flag;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], kStagedConsumers / 32);
        }
        ptx::fence_mbar_init();
        abort_flag = 0;
    }
    __syncthreads();   // the producer starts its copies at once; the consumers first copy the step's scalars

    // units of this CTA: its tiles (grid stride) x the groups of G active workers
    // units: the tiles x the groups of G active workers (unit u: tile
    // u / ngroups, group u % ngroups), claimed one at a time from a global
    // counter by the CTAs' producers where SS::kDynamic (a CTA that drew slower
    // memory simply claims fewer), else every group of tiles blockIdx.x,
    // blockIdx.x + gridDim.x, ... in turn
    const int ngroups = (a.n_active + G - 1) / G;
    const int64_t nunits = a.ntiles * ngroups;
    const int lane = threadIdx.x & 31;
    auto seg = [&](int s, int k) {   // row k of stage s
        return stages + (static_cast<size_t>(s) * SS::kSegs + k) * kStagedTile;
    };

    if (threadIdx.x >= kStagedConsumers) {
        // ---------------------------------------------------------- producer ---
        int64_t issued = 0;
        bool aborted = false;
        unsigned long long next = 0;   // the unit claimed for the next stage (lane 0's claim, broadcast)
        // tensor 0's descriptor read at once, beside the first tile's (a flat
        // store has no other)
        int32_t cur = 0;
        TensorDesc d = a.tens[0];
        if (SS::kDynamic) {
            if (lane == 0) next = atomicAdd(a.work, 1ull);
            next = __shfl_sync(0xffffffffu, next, 0);
        }
        for (int64_t it = 0;; ++it) {
            const int s = static_cast<int>(it % kStages);
            if (it >= kStages) {
                const int64_t j = it - kStages;
                const bool ok = ptx::mbar_wait_bounded(&empty[s], static_cast<uint32_t>((j / kStages) & 1),
                                                       kStagedWaitNs);
                if (!__all_sync(0xffffffffu, ok)) {
                    aborted = true;
                    break;
                }
            }
            if (__any_sync(0xffffffffu, abort_flag != 0)) {
                aborted = true;
                break;
            }
            const unsigned long long unit =
                SS::kDynamic ? next
                             : static_cast<unsigned long long>(blockIdx.x + (it / ngroups) * gridDim.x) * ngroups +
                                   static_cast<unsigned long long>(it % ngroups);
            if (unit >= static_cast<unsigned long long>(nunits)) {   // none left: tell the consumers
                if (lane == 0) {
                    descs[s].len = -1;
                    mbar_release(&full[s]);
                }
                issued = it + 1;
                break;
            }
            if (SS::kDynamic) {
                if (lane == 0) next = atomicAdd(a.work, 1ull);   // the next claim, in flight during this unit's copies
                next = __shfl_sync(0xffffffffu, next, 0);
            }
            const int64_t ti = static_cast<int64_t>(unit / ngroups);
            const int a0 = static_cast<int>(unit % ngroups) * G;
            const Tile tl = a.tiles[ti];
            if (tl.tensor != cur) {
                d = a.tens[tl.tensor];
                cur = tl.tensor;
            }
            const int nw = a.n_active - a0 < G ? a.n_active - a0 : G;
            const int lenr = (tl.len + kVec - 1) / kVec * kVec;   // whole 16-byte pieces (the row padding is allocated)
            const uint32_t bytes = static_cast<uint32_t>(lenr) * sizeof(T);
            const int nsegs = SS::kArrs * nw + (PER_WORKER_H ? 0 : 1);
            if (lane == 0) {
                // the descriptor's stores precede the arrive (release), the
                // consumers read it after their wait (acquire)
                UnitDesc &u = descs[s];
                u.start = tl.start;
                u.wstride = d.wstride;
                u.goff = d.goff;
                u.y = d.y;
                u.m = d.m;
                u.v = d.v;
                u.len = tl.len;
                u.a0 = a0;
                ptx::mbar_arrive_expect_tx(&full[s], static_cast<uint32_t>(nsegs) * bytes);
            }
            __syncwarp();
            if (lane < nsegs && span_ok(0, lenr, kStagedTile, a.err) &&
                aligned16_ok((tl.start) * static_cast<int64_t>(sizeof(T)), a.err)) {
                const T *src = nullptr;
                int k = lane;
                if (!PER_WORKER_H && lane == SS::kArrs * nw) {   // the tile's shared curvature row
                    if (row_ok(0, 1, tl.start, lenr, d.wstride, a.err)) src = as<T>(static_cast<const void *>(d.h)) + tl.start;
                    k = SS::kArrs * G;
                } else {
                    const int w = lane / SS::kArrs, arr = lane % SS::kArrs;
                    const int i = a.worker[a0 + w];
                    if (row_ok(i, a.n_workers, tl.start, lenr, d.wstride, a.err)) {
                        const int64_t o = i * d.wstride + tl.start;
                        const void *base = arr == 0 ? (((a.from_x_mask >> i) & 1u) ? d.x : d.y)
                                         : arr == 1 ? d.m : arr == 2 ? d.v : arr == 3 ? d.c : d.h;
                        src = as<T>(base) + (arr == 4 ? i * d.hstride + tl.start : o);
                    }
                }
                if (src) ptx::bulk_g2s(seg(s, k), src, bytes, &full[s]);
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
                ptx::mbar_wait_bounded(&full[j % kStages], static_cast<uint32_t>((j / kStages) & 1), kStagedWaitNs);
        }
        // every producer has made its last claim before it counts itself out;
        // the last one returns the counter to 0 for the next launch
        if (SS::kDynamic && lane == 0) {
            __threadfence();
            if (atomicAdd(a.work + 1, 1ull) == gridDim.x - 1ull) {
                atomicExch(a.work, 0ull);
                atomicExch(a.work + 1, 0ull);
            }
        }
        return;
    }

    // ------------------------------------------------------------ consumers ---
    for (int q = threadIdx.x; q < static_cast<int>(sizeof(StepTable) / 4); q += kStagedConsumers)
        reinterpret_cast<uint32_t *>(&tab)[q] = reinterpret_cast<const uint32_t *>(a.table)[q];
    staged_consumer_sync();
    // the last CTA to have copied the scalars advances the counters and
    // writes the next step's scalars (as in adamw_kernel); only warp 0 waits
    // for the ticket, the other warps go on to the first unit
    if (threadIdx.x < 32) {
        unsigned t = 0;
        if (lane == 0) t = atomicAdd(a.ticket, 1u);
        t = __shfl_sync(0xffffffffu, t, 0);
        if (t == gridDim.x - 1u) {
            const int i = lane;
            if (i < a.n_workers && ((a.active_mask >> i) & 1u))
                advance_step(a.state, a.table, i, a.beta1d, a.beta2d, a.lr_sched, a.lr_steps, a.lr_after, a.wd,
                             a.seed);
            if (i == 0) *a.ticket = 0u;
        }
    }
    const Consts kc{x2::splat(a.beta1), x2::splat(a.beta2), x2::splat(a.omb1), x2::splat(a.omb2),
                    x2::splat(a.eps), x2::splat(a.sigma)};
    const int e0 = 4 * threadIdx.x;
    for (int64_t it = 0;; ++it) {
        const int s = static_cast<int>(it % kStages);
        if (abort_flag != 0 ||
            !ptx::mbar_wait_bounded(&full[s], static_cast<uint32_t>((it / kStages) & 1), kStagedWaitNs)) {
            // a failed wait: stop here (the producer's waits are bounded too)
            abort_flag = 1;
            atomicCAS(a.err, static_cast<int32_t>(kDevOk), static_cast<int32_t>(kDevWaitTimeout));
            break;
        }
        const UnitDesc &u = descs[s];
        if (u.len < 0) break;   // no unit is left
        const int a0 = u.a0;
        if (e0 < u.len) {
            T *Yw = as<T>(u.y), *Mw = as<T>(u.m), *Vw = as<T>(u.v);
            const int64_t wstride = u.wstride;
            const int64_t off = u.start + e0;
            const int nvalid = u.len - e0 < 4 ? u.len - e0 : 4;
            const uint32_t k0 = static_cast<uint32_t>(u.goff + off);   // global index of the column's first element
            const int nw = a.n_active - a0 < G ? a.n_active - a0 : G;
            using Raw = typename E::Raw;   // 4 elements
            float4 hs = make_float4(0.f, 0.f, 0.f, 0.f);
            if (!PER_WORKER_H) hs = E::unpack(*reinterpret_cast<const Raw *>(seg(s, SS::kArrs * G) + e0));
#pragma unroll
            for (int w = 0; w < G; ++w) {
                if (w >= nw) break;
                const int i = a.worker[a0 + w];
                if (!row_ok(i, a.n_workers, off, 4, wstride, a.err)) continue;
                const Raw *rw = reinterpret_cast<const Raw *>(seg(s, SS::kArrs * w) + e0);
                constexpr int kSegStep = kStagedTile / 4;   // Raw words per row
                const float4 Yu = E::unpack(rw[0]), Mu = E::unpack(rw[kSegStep]), Vu = E::unpack(rw[2 * kSegStep]),
                             Cu = E::unpack(rw[3 * kSegStep]);
                const float4 h4 = PER_WORKER_H ? E::unpack(rw[4 * kSegStep]) : hs;
                const float2 nstep = x2::splat(-tab.step[i]);
                const float2 isb = x2::splat(tab.isb[i]);
                const float2 dec = SCHED ? x2::splat(tab.decay[i]) : x2::splat(a.decay);
                float2 m01, v01, m23, v23, xi01, xi23;
                if constexpr (SS::kBf) {   // 16-bit grid, one hash per element pair
                    noise4_pairs(k0, tab.key_lo[i], tab.key_hi[i], xi01, xi23);
                } else {                   // 24-bit grid, one hash per element
                    xi01 = noise_pair(k0, tab.key_lo[i], tab.key_hi[i]);
                    xi23 = noise_pair(k0 + 2, tab.key_lo[i], tab.key_hi[i]);
                }
                const float2 y01 = adamw_pair(x2::lo(Yu), x2::lo(Mu), x2::lo(Vu), x2::lo(Cu), x2::lo(h4), xi01, nstep,
                                              isb, dec, kc, m01, v01);
                const float2 y23 = adamw_pair(x2::hi(Yu), x2::hi(Mu), x2::hi(Vu), x2::hi(Cu), x2::hi(h4), xi23, nstep,
                                              isb, dec, kc, m23, v23);
                const float4 yo = x2::join(y01, y23), mo = x2::join(m01, m23), vo = x2::join(v01, v23);
                const int64_t o = i * wstride + off;
                if (nvalid == 4) {
                    E::template store4<kSt>(Yw + o, yo);
                    E::template store4<kSt>(Mw + o, mo);
                    E::template store4<kSt>(Vw + o, vo);
                } else {
                    const float ya[4] = {yo.x, yo.y, yo.z, yo.w};
                    const float ma[4] = {mo.x, mo.y, mo.z, mo.w};
                    const float va[4] = {vo.x, vo.y, vo.z, vo.w};
                    for (int l = 0; l < nvalid; ++l) {
                        E::store1(Yw + o + l, ya[l]);
                        E::store1(Mw + o + l, ma[l]);
                        E::store1(Vw + o + l, va[l]);
                    }
                }
            }
        }
        __syncwarp();
        if (lane == 0) mbar_release(&empty[s]);
    }
}

// Workers per load batch of adamw_kernel (16-byte loads of 4 or 5 rows per
// worker, all issued before the batch's arithmetic), chosen per launch from
// the number of workers it steps.  Measured on GB300 (fraction of the copy
// peak, whole launches at full size; every variant runs 2 CTAs of 256 threads
// per SM):
//   shared curvature:  8 workers  U = 4: 1.002, U = 3: 0.987, U = 2: 0.937
//                      16 workers U = 4: 0.957, U = 3: 0.987, U = 2: 0.937
//   own curvature:     32 / 26 / 22 / 17 / 16 / 11 workers U = 2: 1.001-1.007
//                      against U = 3: 0.964-0.980, U = 4: 0.84 (spills);
//                      7 / 3 workers U = 3: 1.02 / 1.03 against U = 2: 0.99 / 0.95.
template <typename T> struct Batch {
    static constexpr int kSharedFew = 4, kSharedMany = 3;       // shared h: <= 8 workers, more
    static constexpr int kOwnFew = 3, kOwnMany = 2;             // own h: <= 7 workers, more
    static constexpr int kSharedFewMax = 8, kOwnFewMax = 7;
};

template <int U, bool P, typename T>
int occupancy(int block) {
    int nb = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, adamw_kernel<U, P, false, T>, block, 0) != cudaSuccess)
        return 1;
    return nb > 0 ? nb : 1;
}

// CTAs per SM that every batch variant of the storage reaches (the grid is
// sized once per context)
template <typename T>
int blocks_per_sm(int block, bool per_worker_h) {
    using B = Batch<T>;
    const int a = per_worker_h ? occupancy<B::kOwnFew, true, T>(block) : occupancy<B::kSharedFew, false, T>(block);
    const int b = per_worker_h ? occupancy<B::kOwnMany, true, T>(block) : occupancy<B::kSharedMany, false, T>(block);
    return a < b ? a : b;
}

template <bool P, bool S, typename T>
const void *staged_ptr() {
    return reinterpret_cast<const void *>(adamw_staged_kernel<P, S, T>);
}

// Occupancy of the staged kernel with its shared memory (the attribute is set
// here, before the first launch).
template <typename T>
int staged_blocks_per_sm(bool per_worker_h) {
    const size_t smem = per_worker_h ? StagedShape<T, true>::kSmem : StagedShape<T, false>::kSmem;
    const void *k[2] = {per_worker_h ? staged_ptr<true, false, T>() : staged_ptr<false, false, T>(),
                        per_worker_h ? staged_ptr<true, true, T>() : staged_ptr<false, true, T>()};
    for (const void *f : k)
        if (cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) !=
            cudaSuccess)
            return 1;
    int nb = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, k[0], kStagedThreads, smem) != cudaSuccess) return 1;
    return nb > 0 ? nb : 1;
}

template <typename T>
void launch_staged(const AdamwArgs &a, int grid, cudaStream_t s) {
    const bool sched = a.lr_steps > 0;
    if (a.per_worker_h) {
        constexpr size_t m = StagedShape<T, true>::kSmem;
        if (sched)
            adamw_staged_kernel<true, true, T><<<grid, kStagedThreads, m, s>>>(a);
        else
            adamw_staged_kernel<true, false, T><<<grid, kStagedThreads, m, s>>>(a);
    } else {
        constexpr size_t m = StagedShape<T, false>::kSmem;
        if (sched)
            adamw_staged_kernel<false, true, T><<<grid, kStagedThreads, m, s>>>(a);
        else
            adamw_staged_kernel<false, false, T><<<grid, kStagedThreads, m, s>>>(a);
    }
}

template <typename T>
void launch(const AdamwArgs &a, int grid, cudaStream_t s) {
    using B = Batch<T>;
    const bool sched = a.lr_steps > 0;
    if (a.per_worker_h) {   // 5 loads per worker
        const bool few = a.n_active <= B::kOwnFewMax;
        if (few && sched) adamw_kernel<B::kOwnFew, true, true, T><<<grid, kBlock, 0, s>>>(a);
        else if (few) adamw_kernel<B::kOwnFew, true, false, T><<<grid, kBlock, 0, s>>>(a);
        else if (sched) adamw_kernel<B::kOwnMany, true, true, T><<<grid, kBlock, 0, s>>>(a);
        else adamw_kernel<B::kOwnMany, true, false, T><<<grid, kBlock, 0, s>>>(a);
    } else {                // 4 loads per worker and the tile's shared h
        const bool few = a.n_active <= B::kSharedFewMax;
        if (few && sched) adamw_kernel<B::kSharedFew, false, true, T><<<grid, kBlock, 0, s>>>(a);
        else if (few) adamw_kernel<B::kSharedFew, false, false, T><<<grid, kBlock, 0, s>>>(a);
        else if (sched) adamw_kernel<B::kSharedMany, false, true, T><<<grid, kBlock, 0, s>>>(a);
        else adamw_kernel<B::kSharedMany, false, false, T><<<grid, kBlock, 0, s>>>(a);
    }
}

}  // namespace

int adamw_blocks_per_sm(int block, bool per_worker_h, int storage) {
    return storage == kStoreBF16 ? staged_blocks_per_sm<bf16>(per_worker_h) : blocks_per_sm<float>(block, per_worker_h);
}

int adamw_staged_fp32_blocks_per_sm(bool per_worker_h) { return staged_blocks_per_sm<float>(per_worker_h); }

cudaError_t launch_adamw(const AdamwArgs &a, int grid, int block, cudaStream_t s) {
    (void)block;
    if (a.storage == kStoreBF16)
        launch_staged<bf16>(a, grid, s);
    else if (a.staged)
        launch_staged<float>(a, grid, s);
    else
        launch<float>(a, grid, s);
    return cudaGetLastError();
}

}  // namespace gasloc
