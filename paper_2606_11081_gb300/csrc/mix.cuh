// mix.cuh -- the per-element arithmetic of a gossip round (Algorithm 1's
// communication step, Eq. 2, DAdam, Local-DAdam) shared by the gossip kernels
// and the fused round kernel: the outer updates, the consensus-error terms,
// and the whole-column update used where a thread holds every worker's rows
// of its column in registers (at most kColumnWorkers workers).
//
// Per element, one rounding per operation (the oracle's order):
//   acc_i = sum_{j in N_i ascending} fma(w_ij, s_j, acc)
//   Nesterov: D = x - acc; b = fma(mu, b, D); x = fma(-eta_out, fma(mu, b, D), x)
//   (SGD, SGDM, Eq. 2, DAdam, Local-DAdam: see outer_pair)
// and the consensus-error term e = S2 - (S1/n) S1 with S1 = sum_i (x_i - s),
// S2 = sum_i (x_i - s)^2 over ascending i, s = worker 0's new x, in fp32.
// In the whole-column update a 4-element column's terms enter the thread's
// fp64 sum as their exact sum, a 2-element column's one at a time
// (ce_sum.cuh); elsewhere each term is widened and added on its own.
#pragma once
#include <cstdint>

#include "ce_sum.cuh"
#include "check.cuh"
#include "f32x2.cuh"
#include "internal.h"

namespace gasloc {

constexpr int kOutSgd = 0, kOutSgdm = 1, kOutNesterov = 2, kOutEq2 = 3, kOutDadam = 4,
              kOutLocalDadam = 5;

// Rows a worker contributes per column: kind 0 = the mixed quantity, kind 1 =
// own x (own y for the DAdam modes), kind 2 = own b.
template <int MODE>
struct ModeRows {
    static constexpr int kRows = (MODE == kOutSgd || MODE == kOutDadam) ? 2 : 3;
    static constexpr bool kMixX = MODE == kOutDadam || MODE == kOutLocalDadam;
    static constexpr bool kHasB = kRows == 3;
};

// Outer-step constants, each in both halves of a register pair.
struct OuterK {
    float2 neta_out, mu, alpha, oma, gamma, eta;
};

// Two lanes of the outer update (f32x2.cuh: each lane rounds as the scalar
// operation would).  acc = mixed value, x = own x, y = own y (DAdam modes),
// b = own b (updated), z / zprev = Eq. 2's z_t and z_{t-1}.
template <int MODE>
__device__ __forceinline__ float2 outer_pair(float2 acc, float2 x, float2 y, float2 &b, float2 z, float2 zprev,
                                             const OuterK &k) {
    switch (MODE) {
    case kOutSgd:
        return x2::fma(k.neta_out, x2::sub(x, acc), x);
    case kOutSgdm: {
        const float2 D = x2::sub(x, acc);
        b = x2::fma(k.mu, b, D);
        return x2::fma(k.neta_out, b, x);
    }
    case kOutNesterov: {
        const float2 D = x2::sub(x, acc);
        b = x2::fma(k.mu, b, D);
        return x2::fma(k.neta_out, x2::fma(k.mu, b, D), x);
    }
    case kOutEq2: {
        const float2 xn = x2::fma(k.alpha, acc, x2::mul(k.oma, z));
        b = z;
        return x2::fma(k.gamma, x2::sub(z, zprev), xn);
    }
    case kOutDadam:
        return x2::add(acc, x2::sub(y, x));
    default: {  // Local-DAdam
        const float2 D = x2::sub(x, acc);
        b = x2::fma(k.mu, b, D);
        return x2::fma(k.neta_out, x2::fma(k.mu, b, D), y);
    }
    }
}

// Consensus-error sums of two lanes: dv = x - shift, s1 += dv, s2 += dv dv.
__device__ __forceinline__ void ce_terms(float2 x, float2 shift, float2 &s1, float2 &s2) {
    const float2 dv = x2::sub(x, shift);
    s1 = x2::add(s1, dv);
    s2 = x2::fma(dv, dv, s2);
}

// ---------------------------------------------------------------------------
// Whole-column update for few workers.

constexpr int kColumnWorkers = 4;

// A column of V consecutive fp32 elements held in registers (V = 2 or 4),
// taken in lane pairs.
template <int V>
struct Col;
template <>
struct Col<2> {
    using T = float2;
    static __device__ __forceinline__ float2 pair(float2 v, int) { return v; }
    static __device__ __forceinline__ float2 join(const float2 (&p)[1]) { return p[0]; }
    static __device__ __forceinline__ float2 zero() { return make_float2(0.f, 0.f); }
    static __device__ __forceinline__ float2 load(const float *p) { return __ldcg(reinterpret_cast<const float2 *>(p)); }
    static __device__ __forceinline__ void store(float *p, float2 v) { __stcg(reinterpret_cast<float2 *>(p), v); }
};
template <>
struct Col<4> {
    using T = float4;
    static __device__ __forceinline__ float2 pair(float4 v, int p) { return p == 0 ? x2::lo(v) : x2::hi(v); }
    static __device__ __forceinline__ float4 join(const float2 (&p)[2]) { return x2::join(p[0], p[1]); }
    static __device__ __forceinline__ float4 zero() { return make_float4(0.f, 0.f, 0.f, 0.f); }
    static __device__ __forceinline__ float4 load(const float *p) { return __ldcg(reinterpret_cast<const float4 *>(p)); }
    static __device__ __forceinline__ void store(float *p, float4 v) { __stcg(reinterpret_cast<float4 *>(p), v); }
};

// The round's neighbour table for n <= kColumnWorkers workers in dense form:
// bit j of mask[i] is set iff j is in N_i (i itself included), with weight
// w[i][j] (0 elsewhere).  The table lists N_i once each, in ascending order,
// so mixing over j = 0..n-1 where the bit is set takes the terms of the list
// in its order: the same sums.  A thread holding every worker's rows in
// registers then indexes them statically, where following the list would
// select each neighbour's row out of the n with a chain of selects.
struct DenseRows {
    float w[kColumnWorkers][kColumnWorkers];
    uint32_t mask[kColumnWorkers];
};

// Row i built by thread i < n from the table in global memory (the caller
// synchronises before use).  The first kColumnWorkers entries of a row are
// read at once; entries past the degree are not used.
__device__ __forceinline__ void dense_rows(const Topo *src, DenseRows &dr, int n, int32_t *err) {
    const int i = threadIdx.x;
    if (i >= n || i >= kColumnWorkers) return;
    int32_t nb[kColumnWorkers];
    float wq[kColumnWorkers];
    const int dg = src->deg[i];
#pragma unroll
    for (int q = 0; q < kColumnWorkers; ++q) {
        nb[q] = src->nbr[i][q];
        wq[q] = src->w[i][q];
        dr.w[i][q] = 0.f;
    }
    uint32_t m = 0;
    if (span_ok(dg, dg + 1, kColumnWorkers, err)) {
#pragma unroll
        for (int q = 0; q < kColumnWorkers; ++q) {
            if (q > dg) break;
            const int j = nb[q];
            if (!span_ok(j, j + 1, n, err)) continue;
            m |= 1u << j;
            dr.w[i][j] = wq[q];
        }
    }
    dr.mask[i] = m;
}

// One column of V elements for every worker (n <= kColumnWorkers) from the
// rows held in registers (rows[kind][worker], kinds as ModeRows): the mixing
// over the round's neighbours (dense form), the outer update, the stores of x and b
// at X / B + worker * wstride + off (nvalid <= V elements), and the column's
// consensus-error terms added to ce_acc (ce_sum.cuh).
template <int MODE, int V>
__device__ __forceinline__ void column_update(const typename Col<V>::T (&rows)[ModeRows<MODE>::kRows][kColumnWorkers],
                                              const DenseRows &dr, int n, const OuterK &ok2, bool first_round, float *X,
                                              float *B, int64_t wstride, int64_t off, int nvalid, float inv_n,
                                              double &ce_acc, int32_t *err) {
    using R = ModeRows<MODE>;
    using C = Col<V>;
    using T = typename C::T;
    constexpr int NP = V / 2;
    float2 s1[NP], s2[NP], sh[NP];
#pragma unroll
    for (int p = 0; p < NP; ++p) s1[p] = s2[p] = sh[p] = x2::splat(0.f);
#pragma unroll
    for (int i = 0; i < kColumnWorkers; ++i) {
        if (i >= n) continue;
        float2 acc[NP];
#pragma unroll
        for (int p = 0; p < NP; ++p) acc[p] = x2::splat(0.f);
        const uint32_t mi = dr.mask[i];
#pragma unroll
        for (int j = 0; j < kColumnWorkers; ++j) {   // ascending j, as the neighbour list
            if (!((mi >> j) & 1u)) continue;
            const float2 w = x2::splat(dr.w[i][j]);
#pragma unroll
            for (int p = 0; p < NP; ++p) {
                float2 s = C::pair(rows[0][j], p);
                if (MODE == kOutEq2) {   // z_j = x_j + eta (y_j - x_j)
                    const float2 xp = C::pair(rows[1][j], p);
                    s = x2::fma(ok2.eta, x2::sub(s, xp), xp);
                }
                acc[p] = x2::fma(w, s, acc[p]);
            }
        }
        const T xo = R::kMixX ? rows[0][i] : rows[1][i];
        const T yo = R::kMixX ? rows[1][i] : xo;
        const T bo = R::kHasB ? rows[R::kRows - 1][i] : C::zero();
        float2 xn[NP], bn[NP];
#pragma unroll
        for (int p = 0; p < NP; ++p) {
            const float2 xp = C::pair(xo, p);
            float2 zo = x2::splat(0.f);
            if (MODE == kOutEq2) {
                const float2 y0 = C::pair(rows[0][i], p);
                zo = x2::fma(ok2.eta, x2::sub(y0, xp), xp);
            }
            float2 b = C::pair(bo, p);
            const float2 zprev = (MODE == kOutEq2 && first_round) ? zo : b;
            xn[p] = outer_pair<MODE>(acc[p], xp, C::pair(yo, p), b, zo, zprev, ok2);
            bn[p] = b;
        }
        if (i == 0) {
#pragma unroll
            for (int p = 0; p < NP; ++p) sh[p] = xn[p];
        }
#pragma unroll
        for (int p = 0; p < NP; ++p) ce_terms(xn[p], sh[p], s1[p], s2[p]);
        if (!row_ok(i, n, off, V, wstride, err)) continue;
        float *Xw = X + i * wstride + off;
        float *Bw = B + i * wstride + off;
        if (nvalid == V) {
            C::store(Xw, C::join(xn));
            if (R::kHasB) C::store(Bw, C::join(bn));
        } else {
            for (int l = 0; l < nvalid; ++l) {
                const float2 xp = xn[l >> 1], bp = bn[l >> 1];
                Xw[l] = (l & 1) ? xp.y : xp.x;
                if (R::kHasB) Bw[l] = (l & 1) ? bp.y : bp.x;
            }
        }
    }
    float e[V];   // the column's terms (0 past the tile's end)
#pragma unroll
    for (int l = 0; l < V; ++l) {
        const float a = (l & 1) ? s1[l >> 1].y : s1[l >> 1].x;
        const float q = (l & 1) ? s2[l >> 1].y : s2[l >> 1].x;
        e[l] = l < nvalid ? __fmaf_rn(-__fmul_rn(a, inv_n), a, q) : 0.f;
    }
    ce_add_group<V>(e, ce_acc);
}

// ---------------------------------------------------------------------------
// End of a round's kernel.

// The block's consensus-error partial (warp sums, then thread 0 adds the
// warps' sums in order) stored at partials[blockIdx.x], and the block's
// ticket.  Returns in every thread whether this block is the last one to
// finish (all others have stored their partials).  Every thread calls it.
__device__ __forceinline__ bool ce_partial_and_ticket(double ce_acc, double *red, int *last, double *partials,
                                                      unsigned int *ticket) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nwarps = (blockDim.x + 31) >> 5;
    for (int o = 16; o > 0; o >>= 1) ce_acc += __shfl_down_sync(0xffffffffu, ce_acc, o);
    if (lane == 0) red[warp] = ce_acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double sum = 0.0;
        for (int w = 0; w < nwarps; ++w) sum += red[w];
        partials[blockIdx.x] = sum;
        __threadfence();
        const unsigned t = atomicAdd(ticket, 1u);
        *last = (t == gridDim.x - 1) ? 1 : 0;
    }
    __syncthreads();
    return *last != 0;
}

// In the last block, warp 0: the partials added in block order (lane 0 gets
// the total).
__device__ __forceinline__ double ce_sum_partials(const double *partials) {
    const int lane = threadIdx.x & 31;
    __threadfence();
    double sum = 0.0;
    for (unsigned b = lane; b < gridDim.x; b += 32) sum += __ldcg(partials + b);
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_down_sync(0xffffffffu, sum, o);
    return sum;
}

}  // namespace gasloc
