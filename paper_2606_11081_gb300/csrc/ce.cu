// ce.cu -- K_ce: standalone consensus error of the current replicas,
//   CE = (1/n) sum_i sum_k (x_ik - xbar_k)^2   (||pi x||^2 / n),
// for states the gossip kernel has not already reduced (after a checkpoint
// load, a direct write of x, or before the first round).
//
// One thread owns a column of 4 elements and loads x_ik for all n workers (8
// loads in flight per batch).  Per element the shifted one-pass form
// e_k = sum_i (x_ik - s)^2 - (sum_i (x_ik - s))^2 / n with s = x_0k, in fp32.
// Reduction: fp64 per thread, warp shuffles, one partial per CTA, the last
// CTA adds the partials in CTA order (atomic ticket; nothing waits).  Reads
// one element per worker-element (4 or 2 bytes).
#include <cuda_runtime.h>

#include "elem.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace gasloc {

namespace {

constexpr int kBlock = 256;

template <typename T>
__global__ void __launch_bounds__(kBlock) ce_kernel(const CeArgs a) {
    using E = Elem<T>;
    __shared__ double red[kBlock / 32];
    __shared__ int last;
    const int n = a.n_workers;
    const float inv_n = static_cast<float>(1.0 / n);
    double acc = 0.0;
    int32_t cur = -1;
    TensorDesc d{};
    for (int64_t ti = blockIdx.x; ti < a.ntiles; ti += gridDim.x) {
        const Tile tl = a.tiles[ti];
        const int e0 = 4 * threadIdx.x;
        if (e0 >= tl.len) continue;
        if (tl.tensor != cur) {
            d = a.tens[tl.tensor];
            cur = tl.tensor;
        }
        const T *X = as<T>(static_cast<const void *>(d.x));
        const int64_t off = tl.start + e0;
        const int nvalid = tl.len - e0 < 4 ? tl.len - e0 : 4;
        float s1[4] = {0.f, 0.f, 0.f, 0.f}, s2[4] = {0.f, 0.f, 0.f, 0.f}, sh[4];
        constexpr int U = 8;
        for (int i0 = 0; i0 < n; i0 += U) {
            float4 Xv[U];
#pragma unroll
            for (int u = 0; u < U; ++u)
                if (i0 + u < n) Xv[u] = E::load4(X + (i0 + u) * d.wstride + off);
#pragma unroll
            for (int u = 0; u < U; ++u) {
                if (i0 + u >= n) continue;
                const float xa[4] = {Xv[u].x, Xv[u].y, Xv[u].z, Xv[u].w};
#pragma unroll
                for (int l = 0; l < 4; ++l) {
                    if (i0 + u == 0) sh[l] = xa[l];
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
        acc += static_cast<double>(e);
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
