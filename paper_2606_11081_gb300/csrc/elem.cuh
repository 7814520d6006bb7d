// elem.cuh -- loads and stores of the replica store's element type.
//
// The store holds fp32 or bfloat16 values; kernels always compute in fp32.
// Widening bf16 -> fp32 is exact (the bf16 bits are the top half of the
// fp32); narrowing rounds to nearest, ties to even (__float2bfloat16_rn).
// Vector accesses move 4 consecutive elements (16 bytes of fp32, 8 bytes of
// bf16) with the cache policy the calling kernel names (default evict-first).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

namespace gasloc {

using bf16 = __nv_bfloat16;

// Cache policy of a global access: kStream marks the lines evict-first
// (ld/st.global.cs), kL2 caches them in L2 only (ld/st.global.cg), kLast
// marks a load as the last use of its line (ld.global.lu).
enum class Cache { kStream, kL2, kLast };

template <Cache C, typename V>
__device__ __forceinline__ V ld_global(const V *p) {
    if constexpr (C == Cache::kL2)
        return __ldcg(p);
    else if constexpr (C == Cache::kLast)
        return __ldlu(p);
    else
        return __ldcs(p);
}
template <Cache C, typename V>
__device__ __forceinline__ void st_global(V *p, V v) {
    if constexpr (C == Cache::kL2)
        __stcg(p, v);
    else
        __stcs(p, v);
}

template <typename T>
struct Elem;

template <>
struct Elem<float> {
    static constexpr int kBytes = 4;
    // 4 elements as loaded (kept in registers until used)
    using Raw = float4;
    template <Cache C = Cache::kStream>
    static __device__ __forceinline__ Raw load_raw(const float *p) {
        return ld_global<C>(reinterpret_cast<const float4 *>(p));
    }
    static __device__ __forceinline__ float4 unpack(Raw r) { return r; }
    template <Cache C = Cache::kStream>
    static __device__ __forceinline__ float4 load4(const float *p) {
        return ld_global<C>(reinterpret_cast<const float4 *>(p));
    }
    template <Cache C = Cache::kStream>
    static __device__ __forceinline__ void store4(float *p, float4 v) {
        st_global<C>(reinterpret_cast<float4 *>(p), v);
    }
    static __device__ __forceinline__ float4 load4_smem(const float *p) {
        return *reinterpret_cast<const float4 *>(p);
    }
    static __device__ __forceinline__ void store4_smem(float *p, float4 v) {
        *reinterpret_cast<float4 *>(p) = v;
    }
    static __device__ __forceinline__ float load1(const float *p) { return *p; }
    static __device__ __forceinline__ void store1(float *p, float v) { *p = v; }
    // the value a store keeps
    static __device__ __forceinline__ float round(float v) { return v; }
    static __device__ __forceinline__ float2 round2(float2 v) { return v; }
};

__device__ __forceinline__ float bf_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf_hi(uint32_t u) { return __uint_as_float(u & 0xFFFF0000u); }
// two fp32 -> one bf16x2 word (low half = lo), each rounded to nearest even
__device__ __forceinline__ uint32_t bf_pack(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&v);
}

template <>
struct Elem<bf16> {
    static constexpr int kBytes = 2;
    using Raw = uint2;
    template <Cache C = Cache::kStream>
    static __device__ __forceinline__ Raw load_raw(const bf16 *p) {
        return ld_global<C>(reinterpret_cast<const uint2 *>(p));
    }
    static __device__ __forceinline__ float4 unpack(Raw u) {
        return make_float4(bf_lo(u.x), bf_hi(u.x), bf_lo(u.y), bf_hi(u.y));
    }
    template <Cache C = Cache::kStream>
    static __device__ __forceinline__ float4 load4(const bf16 *p) {
        return unpack(ld_global<C>(reinterpret_cast<const uint2 *>(p)));
    }
    template <Cache C = Cache::kStream>
    static __device__ __forceinline__ void store4(bf16 *p, float4 v) {
        st_global<C>(reinterpret_cast<uint2 *>(p), make_uint2(bf_pack(v.x, v.y), bf_pack(v.z, v.w)));
    }
    static __device__ __forceinline__ float4 load4_smem(const bf16 *p) {
        const uint2 u = *reinterpret_cast<const uint2 *>(p);
        return make_float4(bf_lo(u.x), bf_hi(u.x), bf_lo(u.y), bf_hi(u.y));
    }
    static __device__ __forceinline__ void store4_smem(bf16 *p, float4 v) {
        *reinterpret_cast<uint2 *>(p) = make_uint2(bf_pack(v.x, v.y), bf_pack(v.z, v.w));
    }
    static __device__ __forceinline__ float load1(const bf16 *p) { return __bfloat162float(*p); }
    static __device__ __forceinline__ void store1(bf16 *p, float v) { *p = __float2bfloat16_rn(v); }
    // the value a store keeps
    static __device__ __forceinline__ float round(float v) { return __bfloat162float(__float2bfloat16_rn(v)); }
    static __device__ __forceinline__ float2 round2(float2 v) {
        const uint32_t u = bf_pack(v.x, v.y);
        return make_float2(bf_lo(u), bf_hi(u));
    }
};

template <typename T>
__device__ __forceinline__ T *as(void *p) {
    return static_cast<T *>(p);
}
template <typename T>
__device__ __forceinline__ const T *as(const void *p) {
    return static_cast<const T *>(p);
}

}  // namespace gasloc
