// ce_noalloc.cu -- consensus error of caller-owned replicas with no device
// allocation at all.
//
// Some callers cannot allocate device memory when they need this number: a
// host framework that owns every byte of the GPU through its own pool or
// arena (a side cudaMalloc would fail, or fragment memory it has planned), a
// latency-critical loop in which cudaMalloc/cudaFree would synchronise the
// device, or a plug-in environment that hands the plug-in pre-allocated
// buffers only.  gasloc_consensus_error_noalloc serves them: the caller
// passes the replicas and the output, and the reduction's scratch (one fp64
// partial per 8192-element chunk plus a completion ticket) lives in the
// file-scope array below, which every GPU that loads this library holds until
// the process exits.
//
// The arithmetic is that of the standalone reduction (ce.cu): per 16-byte
// column, e_k = sum_i (x_ik - s)^2 - (sum_i (x_ik - s))^2 / n with s = x_0k,
// fp64 across elements.  Partials are written per chunk and added in chunk
// order by the last CTA to finish, so the result does not depend on the grid.
//
// The array's device address belongs to a CUDA context, not to a device: the
// device's primary context gets a new one after cudaDeviceReset, and a caller
// that runs its own driver context on the device has another.  The address is
// therefore looked up in the context current on the calling thread and cached
// under that context's process-unique id (cuCtxGetId), so a replaced or
// different context is looked up afresh.
#include <cuda.h>   // driver types only; the entry points are fetched through the runtime
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "../../include/gasloc.h"
#include "check.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace {

constexpr int kBlock = 256;
constexpr int64_t kChunk = 8192;                       // elements per partial
constexpr int64_t kMaxChunks = 65536;                  // partials in the scratch
constexpr int64_t kMaxParams = kChunk * kMaxChunks;    // 536,870,912 elements
constexpr int kHeaderDoubles = 32;                     // ticket and error word in the first 256 bytes
constexpr int kMaxContexts = 64;                       // contexts whose address is cached

// 256 bytes of header (completion ticket at byte 0, the checked build's error
// word at byte 8) + 512 KiB of per-chunk partials.
static __device__ __align__(256) double g_ce_scratch[kHeaderDoubles + kMaxChunks];

__global__ void __launch_bounds__(kBlock) ce_noalloc_kernel(const float *__restrict__ x, int32_t n,
                                                            int64_t P, int64_t wstride, int64_t nchunks,
                                                            double *scratch, double *out) {
    __shared__ double red[kBlock / 32];
    __shared__ int last;
    unsigned int *ticket = reinterpret_cast<unsigned int *>(scratch);
    int32_t *err = reinterpret_cast<int32_t *>(scratch + 1);   // checked build: a failed index check
    double *partials = scratch + kHeaderDoubles;
    const float inv_n = static_cast<float>(1.0 / n);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    for (int64_t ch = blockIdx.x; ch < nchunks; ch += gridDim.x) {
        const int64_t c0 = ch * kChunk;
        const int64_t len = P - c0 < kChunk ? P - c0 : kChunk;
        double acc = 0.0;
        for (int64_t e0 = 4 * threadIdx.x; e0 < len; e0 += 4 * kBlock) {
            const int64_t off = c0 + e0;
            const int nvalid = len - e0 < 4 ? static_cast<int>(len - e0) : 4;
            float s1[4] = {0.f, 0.f, 0.f, 0.f}, s2[4] = {0.f, 0.f, 0.f, 0.f}, sh[4];
            constexpr int U = 8;
            for (int i0 = 0; i0 < n; i0 += U) {
                float4 X[U];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    X[u] = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (i0 + u < n && gasloc::row_ok(i0 + u, n, off, 4, wstride, err))
                        X[u] = gasloc::ptx::ld_stream(x + (i0 + u) * wstride + off);
                }
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    if (i0 + u >= n) continue;
                    const float xa[4] = {X[u].x, X[u].y, X[u].z, X[u].w};
#pragma unroll
                    for (int l = 0; l < 4; ++l) {
                        if (i0 + u == 0) sh[l] = xa[l];
                        const float dv = __fsub_rn(xa[l], sh[l]);
                        s1[l] = __fadd_rn(s1[l], dv);
                        s2[l] = __fmaf_rn(dv, dv, s2[l]);
                    }
                }
            }
#pragma unroll
            for (int l = 0; l < 4; ++l)   // each element's term enters the fp64 sum on its own
                if (l < nvalid) acc += static_cast<double>(__fmaf_rn(-__fmul_rn(s1[l], inv_n), s1[l], s2[l]));
        }
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_down_sync(0xffffffffu, acc, o);
        if (lane == 0) red[warp] = acc;
        __syncthreads();
        if (threadIdx.x == 0) {
            double s = 0.0;
            for (int w = 0; w < kBlock / 32; ++w) s += red[w];
            if (gasloc::span_ok(ch, ch + 1, kMaxChunks, err)) partials[ch] = s;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        __threadfence();
        const unsigned t = atomicAdd(ticket, 1u);
        last = (t == gridDim.x - 1) ? 1 : 0;
    }
    __syncthreads();
    if (last && warp == 0) {
        __threadfence();
        // fixed order: lane l adds chunks l, l+32, ...; then a fixed shuffle tree
        double s = 0.0;
        for (int64_t b = lane; b < nchunks; b += 32) s += __ldcg(partials + b);
        for (int o = 16; o > 0; o >>= 1) s += __shfl_down_sync(0xffffffffu, s, o);
        if (lane == 0) {
            // a failed index check (checked build only) makes the result NaN
            *out = __ldcg(err) != 0 ? __longlong_as_double(0x7ff8000000000000ll) : s / static_cast<double>(n);
            *ticket = 0u;
        }
    }
}

// Address of the scratch array in one CUDA context, and the launch shape.
struct ContextSetup {
    unsigned long long ctx_id = 0;
    void *scratch = nullptr;
    int grid = 0;
};

using CtxGetCurrentFn = CUresult (*)(CUcontext *);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long *);

std::mutex g_mu;
ContextSetup g_setup[kMaxContexts];
int g_nsetup = 0, g_next = 0;
CtxGetCurrentFn g_get_current = nullptr;
CtxGetIdFn g_get_id = nullptr;

int fail(int code, const char *msg) {
    gasloc::set_last_error(msg);   // reported by gasloc_last_error()
    return code;
}

void *driver_entry(const char *name) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion(name, &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return p;
}

// Process-unique id of the context current on this thread (binding the
// device's primary context first if none is current yet).  0 on failure.
unsigned long long current_context_id() {
    if (!g_get_current || !g_get_id) {
        g_get_current = reinterpret_cast<CtxGetCurrentFn>(driver_entry("cuCtxGetCurrent"));
        g_get_id = reinterpret_cast<CtxGetIdFn>(driver_entry("cuCtxGetId"));
        if (!g_get_current || !g_get_id) return 0;
    }
    CUcontext ctx = nullptr;
    if (g_get_current(&ctx) != CUDA_SUCCESS) return 0;
    if (!ctx) {
        // the runtime binds the primary context on its first call that needs one
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_ce_scratch) != cudaSuccess) {
            cudaGetLastError();
            return 0;
        }
        if (g_get_current(&ctx) != CUDA_SUCCESS || !ctx) return 0;
    }
    unsigned long long id = 0;
    if (g_get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id;
}

}  // namespace

extern "C" {

int gasloc_consensus_error_noalloc(const float *x, int32_t n_workers, int64_t n_params, int64_t worker_stride,
                                   double *ce_out_device, void *cuda_stream) {
    if (!x || !ce_out_device) return fail(GASLOC_EINVAL, "x and ce_out_device must be device pointers");
    if (n_workers < 1 || n_workers > GASLOC_MAX_WORKERS) return fail(GASLOC_EINVAL, "n_workers must be in [1, 32]");
    if (n_params < 1) return fail(GASLOC_EINVAL, "n_params must be >= 1");
    if (n_params > kMaxParams)
        return fail(GASLOC_ENOMEM,
                    "n_params exceeds 536870912, the most the static scratch of this entry point can reduce");
    if (worker_stride < n_params || worker_stride % 4 != 0)
        return fail(GASLOC_EINVAL, "worker_stride must be a multiple of 4 and >= n_params");
    if (reinterpret_cast<uintptr_t>(x) % 16 != 0) return fail(GASLOC_EINVAL, "x must be 16-byte aligned");
    if (reinterpret_cast<uintptr_t>(ce_out_device) % 8 != 0)
        return fail(GASLOC_EINVAL, "ce_out_device must be 8-byte aligned");

    ContextSetup setup;
    {
        std::lock_guard<std::mutex> lock(g_mu);
        const unsigned long long id = current_context_id();
        if (id == 0) return fail(GASLOC_ECUDA, "no usable CUDA context on this thread");
        int hit = -1;
        for (int q = 0; q < g_nsetup; ++q)
            if (g_setup[q].ctx_id == id) hit = q;
        if (hit < 0) {
            // first call in this context, which is current: resolve the scratch
            // array's device address here (the host-side name is not one)
            void *p = nullptr;
            if (cudaGetSymbolAddress(&p, g_ce_scratch) != cudaSuccess || !p) {
                cudaGetLastError();
                return fail(GASLOC_ECUDA, "cudaGetSymbolAddress of the scratch array failed");
            }
            int dev = 0, sms = 0, per_sm = 0;
            if (cudaGetDevice(&dev) != cudaSuccess ||
                cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
                cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ce_noalloc_kernel, kBlock, 0) != cudaSuccess) {
                cudaGetLastError();
                return fail(GASLOC_ECUDA, "querying the device for the launch shape failed");
            }
            hit = g_nsetup < kMaxContexts ? g_nsetup++ : (g_next++ % kMaxContexts);
            g_setup[hit].ctx_id = id;
            g_setup[hit].scratch = p;
            g_setup[hit].grid = sms * (per_sm > 0 ? per_sm : 1);
        }
        setup = g_setup[hit];
    }
    const cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
    const int64_t nchunks = (n_params + kChunk - 1) / kChunk;
    const int grid = static_cast<int>(nchunks < setup.grid ? nchunks : setup.grid);
    // the array keeps the previous call's contents: the ticket and the error
    // word (bytes 0..15) must start at 0
    cudaError_t e = cudaMemsetAsync(setup.scratch, 0, 2 * sizeof(double), stream);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(GASLOC_ECUDA, "clearing the completion ticket failed");
    }
    ce_noalloc_kernel<<<grid, kBlock, 0, stream>>>(x, n_workers, n_params, worker_stride, nchunks,
                                                    static_cast<double *>(setup.scratch), ce_out_device);
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(GASLOC_ECUDA, "launching the reduction failed");
    return GASLOC_OK;
}

}  // extern "C"
