// gossip.cu -- K_gossip: one communication round of Algorithm 1 (or Eq. 2 /
// DAdam / Local-DAdam) for all workers, fused with the outer optimizer and the
// consensus-error reduction of the new replicas.
//
// Data movement.  A persistent CTA walks its tiles in a static round-robin.
// For each tile, one thread issues one 1-D bulk copy (TMA engine) per worker of
// that worker's sent slice (y_j, or x_j if it took no local step) into a
// shared-memory stage; S stages are in flight.  Every neighbour slice is
// therefore read from HBM exactly once per tile, however many workers mix it.
// The worker's own x_i and outer momentum b_i are streamed with 16-byte loads
// and stores.  GASLoC moves 20 bytes per worker-element: y (4, staged),
// x and b (8 read, 8 written).
//
// Compute.  Thread t owns the 16-byte column t of the tile for every worker:
//   acc_i = sum_{j in N_i, ascending} fma(w_ij, s_j, acc)
// then the outer update, then the column's consensus-error contribution
//   e_k = sum_i (x_ik - s)^2 - (sum_i (x_ik - s))^2 / n,  s = new x_0k,
// which equals sum_i (x_ik - xbar_k)^2 and needs no second pass.  Per-thread
// sums go to double, then warp shuffles, then one partial per CTA; the last
// CTA to finish (atomic ticket, no waiting) adds the partials in CTA order.
//
// Waiting.  Every wait on a stage barrier is bounded (2 s of wall time).  On
// a timeout the CTA records kDevWaitTimeout, waits (bounded) for its copies
// still in flight, contributes a NaN partial so that the ticket protocol
// completes, and returns.
#include <cuda_runtime.h>

#include "internal.h"
#include "ptx.cuh"

namespace gasloc {

namespace {

constexpr int kOutSgd = 0, kOutSgdm = 1, kOutNesterov = 2, kOutEq2 = 3, kOutDadam = 4,
              kOutLocalDadam = 5;
constexpr int kMaxStages = 4;
constexpr size_t kOffBars = sizeof(Topo);                       // 8320
constexpr size_t kOffRed = kOffBars + 8 * 8;                     // 8384
constexpr size_t kOffFlag = kOffRed + 32 * 8;                    // 8640
constexpr size_t kOffStages = 8704;                              // 128-byte aligned
static_assert(kOffFlag + 16 <= kOffStages, "smem layout");
static_assert(kOffStages % 128 == 0, "stage alignment");
constexpr uint64_t kWaitLimitNs = 2000000000ull;

template <int MODE>
struct ModeTraits {
    static constexpr bool kStageX = MODE == kOutEq2;                        // extra x rows
    static constexpr bool kMixX = MODE == kOutDadam || MODE == kOutLocalDadam;
    static constexpr bool kLoadX = MODE == kOutSgd || MODE == kOutSgdm || MODE == kOutNesterov;
    static constexpr bool kLoadB = MODE != kOutSgd && MODE != kOutDadam;
    static constexpr bool kWriteB = kLoadB;
    static constexpr bool kLoadY = kMixX;                                    // own y_i
};

__device__ __forceinline__ float lane_of(const float4 &v, int l) {
    return l == 0 ? v.x : (l == 1 ? v.y : (l == 2 ? v.z : v.w));
}

template <int MODE>
__device__ __forceinline__ float outer_update(float acc, float x, float y, float &b, float z,
                                              float zprev, const GossipArgs &a) {
    switch (MODE) {
    case kOutSgd: {
        const float D = __fsub_rn(x, acc);
        return __fmaf_rn(-a.eta_out, D, x);
    }
    case kOutSgdm: {
        const float D = __fsub_rn(x, acc);
        b = __fmaf_rn(a.mu, b, D);
        return __fmaf_rn(-a.eta_out, b, x);
    }
    case kOutNesterov: {
        const float D = __fsub_rn(x, acc);
        b = __fmaf_rn(a.mu, b, D);
        return __fmaf_rn(-a.eta_out, __fmaf_rn(a.mu, b, D), x);
    }
    case kOutEq2: {
        float xn = __fmaf_rn(a.alpha, acc, __fmul_rn(a.oma, z));
        xn = __fmaf_rn(a.gamma, __fsub_rn(z, zprev), xn);
        b = z;
        return xn;
    }
    case kOutDadam:
        return __fadd_rn(acc, __fsub_rn(y, x));
    default: {  // Local-DAdam
        const float D = __fsub_rn(x, acc);
        b = __fmaf_rn(a.mu, b, D);
        return __fmaf_rn(-a.eta_out, __fmaf_rn(a.mu, b, D), y);
    }
    }
}

template <int MODE>
__global__ void __launch_bounds__(256) gossip_kernel(const GossipArgs a) {
    using T = ModeTraits<MODE>;
    extern __shared__ __align__(128) unsigned char smem[];
    Topo *tp = reinterpret_cast<Topo *>(smem);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kOffBars);
    double *red = reinterpret_cast<double *>(smem + kOffRed);
    int *flag = reinterpret_cast<int *>(smem + kOffFlag);
    float *stages = reinterpret_cast<float *>(smem + kOffStages);

    const int n = a.n_workers;
    const int TILE = a.tile;
    const int S = a.stages;
    const int rows = T::kStageX ? 2 * n : n;
    const size_t stage_floats = static_cast<size_t>(rows) * TILE;

    {   // neighbour table -> shared memory
        const int *src = reinterpret_cast<const int *>(a.topo);
        int *dst = reinterpret_cast<int *>(tp);
        for (int q = threadIdx.x; q < static_cast<int>(sizeof(Topo) / 4); q += blockDim.x)
            dst[q] = src[q];
    }
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) ptx::mbar_init(&bars[s], 1);
        ptx::fence_mbar_init();
        *flag = 0;
    }
    __syncthreads();

    const int64_t first = blockIdx.x, gstride = gridDim.x;
    const int64_t my_n = a.ntiles > first ? (a.ntiles - first + gstride - 1) / gstride : 0;

    // Producer (thread 0): bulk-copy the sent rows of local tile `it`.
    auto issue = [&](int64_t it) {
        const Tile tl = a.tiles[first + it * gstride];
        const TensorDesc &d = a.tens[tl.tensor];
        const uint32_t bytes = static_cast<uint32_t>(((tl.len + 3) & ~3) * 4);
        uint64_t *bar = &bars[it % S];
        float *st = stages + (it % S) * stage_floats;
        ptx::mbar_arrive_expect_tx(bar, bytes * static_cast<uint32_t>(rows));
        for (int j = 0; j < n; ++j) {
            const float *base;
            if (T::kMixX) base = d.x;
            else base = ((a.fresh_mask >> j) & 1u) ? d.y : d.x;
            ptx::bulk_g2s(st + static_cast<size_t>(j) * TILE, base + j * d.wstride + tl.start, bytes,
                          bar);
        }
        if (T::kStageX)
            for (int j = 0; j < n; ++j)
                ptx::bulk_g2s(st + static_cast<size_t>(n + j) * TILE, d.x + j * d.wstride + tl.start,
                              bytes, bar);
    };
    if (threadIdx.x == 0)
        for (int64_t it = 0; it < my_n && it < S; ++it) issue(it);

    const float inv_n = static_cast<float>(1.0 / n);
    double ce_acc = 0.0;
    int32_t cur = -1;
    TensorDesc d{};
    bool aborted = false;
    int64_t it = 0;
    for (; it < my_n; ++it) {
        const int stage = static_cast<int>(it % S);
        const uint32_t parity = static_cast<uint32_t>((it / S) & 1);
        const bool ok = ptx::mbar_wait_bounded(&bars[stage], parity, kWaitLimitNs);
        if (__syncthreads_or(!ok)) {
            aborted = true;
            break;
        }
        const Tile tl = a.tiles[first + it * gstride];
        if (tl.tensor != cur) {
            d = a.tens[tl.tensor];
            cur = tl.tensor;
        }
        const int e0 = 4 * threadIdx.x;
        float *st = stages + stage * stage_floats;
        if (e0 < tl.len) {
            const int nvalid = tl.len - e0 < 4 ? tl.len - e0 : 4;
            const int64_t off = tl.start + e0;
            if (T::kStageX) {
                // z_j = fma(eta, y_j - x_j, x_j), in place over the sent rows
                for (int j = 0; j < n; ++j) {
                    float4 *yr = reinterpret_cast<float4 *>(st + static_cast<size_t>(j) * TILE + e0);
                    const float4 xr =
                        *reinterpret_cast<const float4 *>(st + static_cast<size_t>(n + j) * TILE + e0);
                    float4 z = *yr;
                    z.x = __fmaf_rn(a.eta, __fsub_rn(z.x, xr.x), xr.x);
                    z.y = __fmaf_rn(a.eta, __fsub_rn(z.y, xr.y), xr.y);
                    z.z = __fmaf_rn(a.eta, __fsub_rn(z.z, xr.z), xr.z);
                    z.w = __fmaf_rn(a.eta, __fsub_rn(z.w, xr.w), xr.w);
                    *yr = z;
                }
            }
            float s1[4] = {0.f, 0.f, 0.f, 0.f}, s2[4] = {0.f, 0.f, 0.f, 0.f}, sh[4] = {0.f, 0.f, 0.f, 0.f};
            constexpr int U = 4;
            for (int i0 = 0; i0 < n; i0 += U) {
                float4 X[U], B[U], Y[U];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int i = i0 + u;
                    if (i < n) {
                        const int64_t o = i * d.wstride + off;
                        if (T::kLoadX) X[u] = ptx::ld_stream(d.x + o);
                        if (T::kLoadB) B[u] = ptx::ld_stream(d.b + o);
                        if (T::kLoadY && ((a.fresh_mask >> i) & 1u)) Y[u] = ptx::ld_stream(d.y + o);
                    }
                }
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int i = i0 + u;
                    if (i >= n) continue;
                    // mix over N_i in ascending j
                    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
                    const int dg = tp->deg[i];
                    for (int q = 0; q <= dg; ++q) {
                        const int j = tp->nbr[i][q];
                        const float w = tp->w[i][q];
                        const float4 sj =
                            *reinterpret_cast<const float4 *>(st + static_cast<size_t>(j) * TILE + e0);
                        acc.x = __fmaf_rn(w, sj.x, acc.x);
                        acc.y = __fmaf_rn(w, sj.y, acc.y);
                        acc.z = __fmaf_rn(w, sj.z, acc.z);
                        acc.w = __fmaf_rn(w, sj.w, acc.w);
                    }
                    float4 xo;
                    if (T::kLoadX) {
                        xo = X[u];
                    } else if (T::kStageX) {
                        xo = *reinterpret_cast<const float4 *>(st + static_cast<size_t>(n + i) * TILE + e0);
                    } else {   // DAdam modes: the staged (mixed) rows are x
                        xo = *reinterpret_cast<const float4 *>(st + static_cast<size_t>(i) * TILE + e0);
                    }
                    float4 yo = xo;
                    if (T::kLoadY && ((a.fresh_mask >> i) & 1u)) yo = Y[u];
                    float4 zo = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (T::kStageX)
                        zo = *reinterpret_cast<const float4 *>(st + static_cast<size_t>(i) * TILE + e0);
                    float4 bo = T::kLoadB ? B[u] : make_float4(0.f, 0.f, 0.f, 0.f);
                    float4 zp = bo;
                    if (T::kStageX && a.first_round) zp = zo;
                    float4 xn;
                    xn.x = outer_update<MODE>(acc.x, xo.x, yo.x, bo.x, zo.x, zp.x, a);
                    xn.y = outer_update<MODE>(acc.y, xo.y, yo.y, bo.y, zo.y, zp.y, a);
                    xn.z = outer_update<MODE>(acc.z, xo.z, yo.z, bo.z, zo.z, zp.z, a);
                    xn.w = outer_update<MODE>(acc.w, xo.w, yo.w, bo.w, zo.w, zp.w, a);
                    const int64_t o = i * d.wstride + off;
                    if (nvalid == 4) {
                        ptx::st_stream(d.x + o, xn);
                        if (T::kWriteB) ptx::st_stream(d.b + o, bo);
                    } else {
                        for (int l = 0; l < nvalid; ++l) {
                            d.x[o + l] = lane_of(xn, l);
                            if (T::kWriteB) d.b[o + l] = lane_of(bo, l);
                        }
                    }
                    // consensus-error column sums, shifted by worker 0's new value
                    const float xa[4] = {xn.x, xn.y, xn.z, xn.w};
#pragma unroll
                    for (int l = 0; l < 4; ++l) {
                        if (i == 0) sh[l] = xa[l];
                        const float dv = __fsub_rn(xa[l], sh[l]);
                        s1[l] = __fadd_rn(s1[l], dv);
                        s2[l] = __fmaf_rn(dv, dv, s2[l]);
                    }
                }
            }
            float e = 0.f;
#pragma unroll
            for (int l = 0; l < 4; ++l)
                if (l < nvalid) e = __fadd_rn(e, __fmaf_rn(-__fmul_rn(s1[l], inv_n), s1[l], s2[l]));
            ce_acc += static_cast<double>(e);
        }
        __syncthreads();   // every thread is done with this stage
        if (threadIdx.x == 0 && it + S < my_n) {
            ptx::fence_proxy_async_smem();
            issue(it + S);
        }
    }

    if (aborted) {
        if (threadIdx.x == 0) {
            atomicCAS(a.err, kDevOk, kDevWaitTimeout);
            // drain the copies this CTA still has in flight (bounded)
            for (int64_t j = it; j < my_n && j < it + S; ++j)
                ptx::mbar_wait_bounded(&bars[j % S], static_cast<uint32_t>((j / S) & 1), kWaitLimitNs);
        }
        ce_acc = __longlong_as_double(0x7ff8000000000000ll);   // NaN partial
    }

    // block reduction: warp shuffles, then warps in order
    for (int o = 16; o > 0; o >>= 1) ce_acc += __shfl_down_sync(0xffffffffu, ce_acc, o);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) red[warp] = ce_acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double s = 0.0;
        for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) s += red[w];
        a.partials[blockIdx.x] = s;
        __threadfence();
        const unsigned t = atomicAdd(a.ticket, 1u);
        *flag = (t == gridDim.x - 1) ? 1 : 0;
    }
    __syncthreads();
    if (*flag && warp == 0) {
        __threadfence();
        double s = 0.0;
        for (unsigned b = lane; b < gridDim.x; b += 32) s += __ldcg(a.partials + b);
        for (int o = 16; o > 0; o >>= 1) s += __shfl_down_sync(0xffffffffu, s, o);
        if (lane == 0) {
            *a.ce_out = s / static_cast<double>(n);
            *a.ticket = 0u;
        }
    }
}

template <int MODE>
void *kernel_ptr() {
    return reinterpret_cast<void *>(gossip_kernel<MODE>);
}

void *mode_kernel(int mode) {
    switch (mode) {
    case kOutSgd: return kernel_ptr<kOutSgd>();
    case kOutSgdm: return kernel_ptr<kOutSgdm>();
    case kOutNesterov: return kernel_ptr<kOutNesterov>();
    case kOutEq2: return kernel_ptr<kOutEq2>();
    case kOutDadam: return kernel_ptr<kOutDadam>();
    default: return kernel_ptr<kOutLocalDadam>();
    }
}

}  // namespace

size_t gossip_smem_bytes(int n, int tile, int stages, int mode) {
    const int rows = mode == kOutEq2 ? 2 * n : n;
    return kOffStages + static_cast<size_t>(stages) * rows * tile * sizeof(float);
}

cudaError_t gossip_set_smem(size_t smem) {
    for (int m = 0; m <= kOutLocalDadam; ++m) {
        const cudaError_t e = cudaFuncSetAttribute(mode_kernel(m), cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

int gossip_blocks_per_sm(int block, size_t smem) {
    int nb = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, gossip_kernel<kOutNesterov>, block, smem) !=
        cudaSuccess)
        return 1;
    return nb > 0 ? nb : 1;
}

cudaError_t launch_gossip(const GossipArgs &a, int grid, int block, size_t smem, cudaStream_t s) {
    if (a.stages < 1 || a.stages > kMaxStages) return cudaErrorInvalidValue;
    switch (a.mode) {
    case kOutSgd: gossip_kernel<kOutSgd><<<grid, block, smem, s>>>(a); break;
    case kOutSgdm: gossip_kernel<kOutSgdm><<<grid, block, smem, s>>>(a); break;
    case kOutNesterov: gossip_kernel<kOutNesterov><<<grid, block, smem, s>>>(a); break;
    case kOutEq2: gossip_kernel<kOutEq2><<<grid, block, smem, s>>>(a); break;
    case kOutDadam: gossip_kernel<kOutDadam><<<grid, block, smem, s>>>(a); break;
    default: gossip_kernel<kOutLocalDadam><<<grid, block, smem, s>>>(a); break;
    }
    return cudaGetLastError();
}

}  // namespace gasloc
