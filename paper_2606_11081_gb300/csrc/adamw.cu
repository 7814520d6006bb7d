// adamw.cu -- K_adamw: one inner AdamW step (Algorithm 1, inner loop; App. B
// settings) for every active worker, all replicas in one launch.
//
// Memory-bound streaming kernel: per active worker and element it reads the
// iterate (x on the first step of a round, else y), m, v and the centre c and
// writes y, m, v -- 28 bytes -- plus 4 bytes of shared curvature h per element
// (h is per worker in the heterogeneous workload: 32 bytes per worker-element).
// One thread owns one 16-byte column of a tile and walks the active workers U
// at a time (U = 4, or 3 with per-worker h), issuing all of their 16-byte loads
// before any arithmetic so that 15-16 requests per thread stay in flight.  The synthetic gradient g = h (y - c) + sigma xi
// is formed in registers; xi comes from a 32-bit counter hash of the element
// index and the step key, so the gradient costs no memory traffic.
//
// Per element, one IEEE rounding per line (the order the oracle follows):
//   d = y - c;  t = h d;  g = fma(sigma, xi, t)
//   y = y * decay
//   m = fma(beta1, m, (1 - beta1) g)
//   v = fma(beta2, v, (1 - beta2) (g g))
//   den = fma(sqrt(v), isb, eps)
//   y = fma(-step, m / den, y)
#include <cuda_runtime.h>

#include "internal.h"
#include "ptx.cuh"
#include "rng.cuh"

namespace gasloc {

namespace {

constexpr int kBlock = 256;   // threads; a tile is 4 * kBlock elements

struct Consts {
    float decay, b1, b2, omb1, omb2, eps, sigma;
};

__device__ __forceinline__ float adamw_lane(float y, float m_in, float v_in, float c, float h,
                                            float xi, float step, float isb, const Consts &k,
                                            float &m_out, float &v_out) {
    const float d = __fsub_rn(y, c);
    const float t = __fmul_rn(h, d);
    const float g = __fmaf_rn(k.sigma, xi, t);
    y = __fmul_rn(y, k.decay);
    const float m = __fmaf_rn(k.b1, m_in, __fmul_rn(k.omb1, g));
    const float v = __fmaf_rn(k.b2, v_in, __fmul_rn(k.omb2, __fmul_rn(g, g)));
    const float den = __fmaf_rn(__fsqrt_rn(v), isb, k.eps);
    y = __fmaf_rn(-step, __fdiv_rn(m, den), y);
    m_out = m;
    v_out = v;
    return y;
}

// xi = ((u >> 8) * 2^-23 - 1) * sqrt3: uniform on [-sqrt3, sqrt3), unit variance.
__device__ __forceinline__ float noise_xi(uint32_t k, uint32_t klo, uint32_t khi) {
    const float sqrt3 = static_cast<float>(1.7320508075688772);
    const uint32_t u = noise_bits(k, klo, khi);
    const float a = __fmul_rn(__uint2float_rn(u >> 8), 0x1p-23f);
    return __fmul_rn(__fsub_rn(a, 1.0f), sqrt3);
}

template <int U, bool PER_WORKER_H>
__global__ void __launch_bounds__(kBlock, 2) adamw_kernel(const AdamwArgs a) {
    const Consts kc{a.decay, a.beta1, a.beta2, a.omb1, a.omb2, a.eps, a.sigma};
    // this step's per-worker scalars (written by the prep kernel) -> shared
    __shared__ StepTable tab;
    for (int q = threadIdx.x; q < static_cast<int>(sizeof(StepTable) / 4); q += blockDim.x)
        reinterpret_cast<uint32_t *>(&tab)[q] = reinterpret_cast<const uint32_t *>(a.table)[q];
    __syncthreads();
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
        const int64_t off = tl.start + e0;
        const int nvalid = tl.len - e0 < 4 ? tl.len - e0 : 4;
        const uint32_t k0 = static_cast<uint32_t>(d.goff + off);
        float4 hs = make_float4(0.f, 0.f, 0.f, 0.f);
        if (!PER_WORKER_H) hs = ptx::ld_stream(d.h + off);

        for (int a0 = 0; a0 < a.n_active; a0 += U) {
            float4 Y[U], M[U], V[U], C[U], Hh[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                if (a0 + u < a.n_active) {
                    const int i = a.worker[a0 + u];
                    const int64_t o = i * d.wstride + off;
                    const float *src = ((a.from_x_mask >> i) & 1u) ? d.x : d.y;
                    Y[u] = ptx::ld_stream(src + o);
                    M[u] = ptx::ld_stream(d.m + o);
                    V[u] = ptx::ld_stream(d.v + o);
                    C[u] = ptx::ld_stream(d.c + o);
                    if (PER_WORKER_H) Hh[u] = ptx::ld_stream(d.h + i * d.hstride + off);
                }
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                if (a0 + u < a.n_active) {
                    const int i = a.worker[a0 + u];
                    const float step = tab.step[i];
                    const float isb = tab.isb[i];
                    const uint32_t klo = tab.key_lo[i], khi = tab.key_hi[i];
                    const float4 h4 = PER_WORKER_H ? Hh[u] : hs;
                    float4 yo, mo, vo;
                    yo.x = adamw_lane(Y[u].x, M[u].x, V[u].x, C[u].x, h4.x, noise_xi(k0 + 0, klo, khi),
                                      step, isb, kc, mo.x, vo.x);
                    yo.y = adamw_lane(Y[u].y, M[u].y, V[u].y, C[u].y, h4.y, noise_xi(k0 + 1, klo, khi),
                                      step, isb, kc, mo.y, vo.y);
                    yo.z = adamw_lane(Y[u].z, M[u].z, V[u].z, C[u].z, h4.z, noise_xi(k0 + 2, klo, khi),
                                      step, isb, kc, mo.z, vo.z);
                    yo.w = adamw_lane(Y[u].w, M[u].w, V[u].w, C[u].w, h4.w, noise_xi(k0 + 3, klo, khi),
                                      step, isb, kc, mo.w, vo.w);
                    const int64_t o = i * d.wstride + off;
                    if (nvalid == 4) {
                        ptx::st_stream(d.y + o, yo);
                        ptx::st_stream(d.m + o, mo);
                        ptx::st_stream(d.v + o, vo);
                    } else {
                        const float ya[4] = {yo.x, yo.y, yo.z, yo.w};
                        const float ma[4] = {mo.x, mo.y, mo.z, mo.w};
                        const float va[4] = {vo.x, vo.y, vo.z, vo.w};
                        for (int l = 0; l < nvalid; ++l) {
                            d.y[o + l] = ya[l];
                            d.m[o + l] = ma[l];
                            d.v[o + l] = va[l];
                        }
                    }
                }
            }
        }
    }
}

}  // namespace

int adamw_blocks_per_sm(int block, bool per_worker_h) {
    int nb = 0;
    const cudaError_t e =
        per_worker_h ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, adamw_kernel<3, true>, block, 0)
                     : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, adamw_kernel<4, false>, block, 0);
    if (e != cudaSuccess) return 1;
    return nb > 0 ? nb : 1;
}

cudaError_t launch_adamw(const AdamwArgs &a, int grid, int block, cudaStream_t s) {
    (void)block;
    if (a.per_worker_h)
        adamw_kernel<3, true><<<grid, kBlock, 0, s>>>(a);   // 5 loads per worker
    else
        adamw_kernel<4, false><<<grid, kBlock, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace gasloc
