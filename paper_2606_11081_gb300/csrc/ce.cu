// ce.cu -- K_ce: standalone consensus error of the current replicas,
//   CE = (1/n) sum_i sum_k (x_ik - xbar_k)^2   (||pi x||^2 / n),
// for states the gossip kernel has not already reduced (after a checkpoint
// load, a direct write of x, or before the first round).
//
// One thread owns a column of 4 elements and loads x_ik for all n workers (8
// loads in flight per batch; with bf16 storage the columns of two tiles are
// loaded together, so that a thread keeps as many bytes in flight as with
// fp32).  Per element the shifted one-pass form
// e_k = sum_i (x_ik - s)^2 - (sum_i (x_ik - s))^2 / n with s = x_0k, in fp32;
// each e_k is widened and added on its own, so the value of an element does
// not depend on the column it shares (nor on how a range is cut).
// Reduction: fp64 per thread, warp shuffles, one partial per CTA, the last
// CTA adds the partials in CTA order (atomic ticket; nothing waits).  Reads
// one element per worker-element (4 or 2 bytes).
#include <cuda_runtime.h>

#include "check.cuh"
#include "elem.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace gasloc {

namespace {

constexpr int kBlock = 256;

// TPI tiles per iteration: their loads are all issued before any arithmetic
// (bf16 takes two, so that a thread keeps as many bytes in flight as fp32).
template <typename T> struct CeShape { static constexpr int kTiles = 1; };
template <> struct CeShape<bf16> { static constexpr int kTiles = 2; };

template <typename T>
__global__ void __launch_bounds__(kBlock, 3) ce_kernel(const CeArgs a) {
    using E = Elem<T>;
    constexpr int TPI = CeShape<T>::kTiles;
    __shared__ double red[kBlock / 32];
    __shared__ int last;
    const int n = a.n_workers;
    const float inv_n = static_cast<float>(1.0 / n);
    const int e0 = 4 * threadIdx.x;
    double acc = 0.0;
    for (int64_t t0 = blockIdx.x; t0 < a.ntiles; t0 += static_cast<int64_t>(TPI) * gridDim.x) {
        const T *X[TPI];
        int64_t off[TPI], ws[TPI];   // column start; worker i's row starts at i * ws
        int nvalid[TPI];             // 0: this thread has no column in the tile
#pragma unroll
        for (int p = 0; p < TPI; ++p) {
            const int64_t ti = t0 + static_cast<int64_t>(p) * gridDim.x;
            nvalid[p] = 0;
            X[p] = nullptr;
            off[p] = ws[p] = 0;
            if (ti < a.ntiles) {
                const Tile tl = a.tiles[ti];
                if (e0 < tl.len) {
                    const TensorDesc &d = a.tens[tl.tensor];
                    X[p] = as<T>(static_cast<const void *>(d.x));
                    off[p] = tl.start + e0;
                    ws[p] = d.wstride;
                    nvalid[p] = tl.len - e0 < 4 ? tl.len - e0 : 4;
                }
            }
        }
        float s1[TPI][4], s2[TPI][4], sh[TPI][4];
#pragma unroll
        for (int p = 0; p < TPI; ++p)
#pragma unroll
            for (int l = 0; l < 4; ++l) s1[p][l] = s2[p][l] = sh[p][l] = 0.f;
        constexpr int U = 8;
        for (int i0 = 0; i0 < n; i0 += U) {
            typename E::Raw Xv[TPI][U];
#pragma unroll
            for (int p = 0; p < TPI; ++p)
#pragma unroll
                for (int u = 0; u < U; ++u)
                    if (nvalid[p] && i0 + u < n)
                        Xv[p][u] = row_ok(i0 + u, n, off[p], 4, ws[p], a.err)
                                       ? E::load_raw(X[p] + (i0 + u) * ws[p] + off[p])
                                       : typename E::Raw{};
#pragma unroll
            for (int p = 0; p < TPI; ++p) {
                if (!nvalid[p]) continue;
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    if (i0 + u >= n) continue;
                    const float4 xv = E::unpack(Xv[p][u]);
                    const float xa[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
                    for (int l = 0; l < 4; ++l) {
                        if (i0 + u == 0) sh[p][l] = xa[l];
                        const float dv = __fsub_rn(xa[l], sh[p][l]);
                        s1[p][l] = __fadd_rn(s1[p][l], dv);
                        s2[p][l] = __fmaf_rn(dv, dv, s2[p][l]);
                    }
                }
            }
        }
#pragma unroll
        for (int p = 0; p < TPI; ++p)
#pragma unroll
            for (int l = 0; l < 4; ++l)   // each element's term enters the fp64 sum on its own
                if (l < nvalid[p]) acc += static_cast<double>(__fmaf_rn(-__fmul_rn(s1[p][l], inv_n), s1[p][l], s2[p][l]));
    }
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_down_sync(0xffffffffu, acc, o);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) red[warp] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double s = 0.0;
        for (int w = 0; w < kBlock / 32; ++w) s += red[w];
        a.partials[blockIdx.x] = s;
        __threadfence();
        const unsigned t = atomicAdd(a.ticket, 1u);
        last = (t == gridDim.x - 1) ? 1 : 0;
    }
    __syncthreads();
    if (last && warp == 0) {
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

}  // namespace

int ce_blocks_per_sm(int block, int storage) {
    int nb = 0;
    const cudaError_t e = storage == kStoreBF16
                              ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, ce_kernel<bf16>, block, 0)
                              : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, ce_kernel<float>, block, 0);
    if (e != cudaSuccess) return 1;
    return nb > 0 ? nb : 1;
}

cudaError_t launch_ce(const CeArgs &a, int grid, int block, cudaStream_t s) {
    (void)block;
    if (a.storage == kStoreBF16)
        ce_kernel<bf16><<<grid, kBlock, 0, s>>>(a);
    else
        ce_kernel<float><<<grid, kBlock, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace gasloc
