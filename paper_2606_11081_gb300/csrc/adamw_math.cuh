// adamw_math.cuh -- the per-element arithmetic of one inner AdamW step
// (Algorithm 1, inner loop; App. B settings) on the synthetic quadratic, fp32
// storage: the gradient noise of an element and the step on a pair of
// elements.  Shared by the local-step kernels and the fused round kernel.
//
// Per element, in fp32 with one IEEE rounding per operation (the oracle's
// order; pairs of lanes share f32x2 instructions, which round each lane as
// the scalar operation does):
//   d = y - c;  t = h d;  g = fma(sigma, xi, t)
//   y = y * decay
//   m = fma(beta1, m, (1 - beta1) g)
//   v = fma(beta2, v, (1 - beta2) (g g))
//   den = fma(sqrt(v), isb, eps)
//   y = fma(-step, m / den, y)
#pragma once
#include <cstdint>

#include "f32x2.cuh"
#include "rng.cuh"

namespace gasloc {

// Per-step constants, each in both halves of a register pair.
struct Consts {
    float2 b1, b2, omb1, omb2, eps, sigma;
};

// Two lanes of the step; each paired operation rounds each lane exactly as
// the scalar operation does (f32x2.cuh), so the sequence is the one above.
__device__ __forceinline__ float2 adamw_pair(float2 y, float2 m_in, float2 v_in, float2 c, float2 h, float2 xi,
                                             float2 nstep, float2 isb, float2 decay, const Consts &k,
                                             float2 &m_out, float2 &v_out) {
    const float2 d = x2::sub(y, c);
    const float2 t = x2::mul(h, d);
    const float2 g = x2::fma(k.sigma, xi, t);
    y = x2::mul(y, decay);
    const float2 m = x2::fma(k.b1, m_in, x2::mul(k.omb1, g));
    const float2 v = x2::fma(k.b2, v_in, x2::mul(k.omb2, x2::mul(g, g)));
    const float2 den = x2::fma(make_float2(__fsqrt_rn(v.x), __fsqrt_rn(v.y)), isb, k.eps);
    y = x2::fma(nstep, make_float2(__fdiv_rn(m.x, den.x), __fdiv_rn(m.y, den.y)), y);
    m_out = m;
    v_out = v;
    return y;
}

// Gradient noise, uniform on [-sqrt3, sqrt3) with unit variance.
// fp32 storage, 24 bits per element: u = word(k) and
// xi = ((u >> 8) * 2^-23 - 1) * sqrt3.  (u >> 8) * 2^-23 - 1 equals
// ((u >> 8) - 2^23) * 2^-23 exactly and sqrt3 * 2^-23 is exact, so
// xi = fl(((u >> 8) - 2^23) * (sqrt3 * 2^-23)): the same real product rounded
// once, from one integer conversion.
__device__ __forceinline__ float noise_int(uint32_t k, uint32_t klo, uint32_t khi) {
    const uint32_t u = noise_word(k, klo, khi);
    return __int2float_rn(static_cast<int32_t>(u >> 8) - (1 << 23));
}
__device__ __forceinline__ float2 noise_pair(uint32_t k, uint32_t klo, uint32_t khi) {
    const float scale = static_cast<float>(1.7320508075688772) * 0x1p-23f;
    return x2::mul(make_float2(noise_int(k, klo, khi), noise_int(k + 1, klo, khi)), x2::splat(scale));
}

}  // namespace gasloc
