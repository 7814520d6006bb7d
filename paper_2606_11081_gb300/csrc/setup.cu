// setup.cu -- one-time and cold-path kernels: replica initialisation, the
// per-round neighbour-table generator, the network average (output of
// Algorithm 1) and an index gather used for sampled checks.
#include <cuda_runtime.h>

#include "check.cuh"
#include "elem.cuh"
#include "internal.h"
#include "ptx.cuh"
#include "rng.cuh"
#include "step.cuh"

namespace gasloc {

namespace {

// Standard-normal stand-in: Irwin-Hall sum of four 24-bit uniforms,
// (s - 2^25) * fl32(sqrt3 * 2^-24): one rounding in the integer conversion,
// one in the product.
__device__ __forceinline__ float normal_std(uint64_t seed, uint64_t tag, uint64_t i, uint64_t k) {
    int32_t s = 0;
#pragma unroll
    for (uint64_t j = 0; j < 4; ++j) s += static_cast<int32_t>(top24(hash4(seed, tag, i, 4 * k + j)));
    const float scale = static_cast<float>(1.7320508075688772 * 5.9604644775390625e-08);
    return __fmul_rn(__int2float_rn(s - (1 << 25)), scale);
}

// h ~ U(0.1, 1): fma(0.9, r * 2^-24, 0.1).
__device__ __forceinline__ float curvature(uint64_t seed, uint64_t i, uint64_t k) {
    const float u = __fmul_rn(__uint2float_rn(top24(hash4(seed, kTagCurv, i, k))), 0x1p-24f);
    return __fmaf_rn(static_cast<float>(0.9), u, static_cast<float>(0.1));
}

// Initial state (stored values rounded to the element type).
template <typename T>
__global__ void init_kernel(const InitArgs a) {
    using E = Elem<T>;
    const float x0std = static_cast<float>(0.02);
    for (int64_t ti = blockIdx.x; ti < a.ntiles; ti += gridDim.x) {
        const Tile tl = a.tiles[ti];
        const TensorDesc d = a.tens[tl.tensor];
        T *X = as<T>(d.x), *Y = as<T>(d.y), *C = as<T>(d.c), *Hh = as<T>(d.h);
        for (int e = threadIdx.x; e < tl.len; e += blockDim.x) {
            const int64_t off = tl.start + e;
            const uint64_t k = static_cast<uint64_t>(d.goff + off);
            const float x0 = __fmul_rn(x0std, normal_std(a.seed, kTagX0, 0, k));
            for (int i = 0; i < a.n_workers; ++i) {
                if (!row_ok(i, a.n_workers, off, 1, d.wstride, a.err)) continue;
                const int64_t o = i * d.wstride + off;
                E::store1(X + o, x0);
                E::store1(Y + o, x0);
                E::store1(C + o, normal_std(a.seed, kTagCentre, static_cast<uint64_t>(i), k));
            }
            const int nh = a.per_worker_h ? a.n_workers : 1;
            for (int i = 0; i < nh; ++i)
                if (row_ok(i, nh, off, 1, a.per_worker_h ? d.hstride : d.wstride, a.err))
                    E::store1(Hh + i * d.hstride + off, curvature(a.seed, static_cast<uint64_t>(i), k));
        }
    }
}

// Neighbour table of round t, one warp.  Lane 0 draws the permutation
// (Fisher-Yates, Lemire multiply-shift); edges are bitmasks; each lane then
// applies edge activation to the edges it owns and builds its own row.
__global__ void topo_kernel(const TopoSpec spec, const int64_t round_arg, const int64_t *round_ptr, Topo *out) {
    const int64_t round = round_ptr ? *round_ptr : round_arg;
    __shared__ uint32_t adj[kMaxWorkers];
    __shared__ int32_t perm[kMaxWorkers];
    __shared__ int32_t deg[kMaxWorkers];
    const int n = spec.n;
    const int lane = threadIdx.x;
    if (lane < kMaxWorkers) adj[lane] = 0u;
    __syncwarp();
    if (lane == 0) {
        auto edge = [&](int a, int b) {
            if (a != b) { adj[a] |= 1u << b; adj[b] |= 1u << a; }
        };
        switch (spec.kind) {
        case kRing:
            for (int i = 0; i < n; ++i) edge(i, (i + 1) % n);
            break;
        case kComplete:
            for (int i = 0; i < n; ++i)
                for (int j = i + 1; j < n; ++j) edge(i, j);
            break;
        case kExp:
            for (int i = 0; i < n; ++i)
                for (int s = 1; s < n; s *= 2) edge(i, (i + s) % n);
            break;
        case kTorus:
            for (int r = 0; r < spec.rows; ++r)
                for (int c = 0; c < spec.cols; ++c) {
                    edge(r * spec.cols + c, ((r + 1) % spec.rows) * spec.cols + c);
                    edge(r * spec.cols + c, r * spec.cols + (c + 1) % spec.cols);
                }
            break;
        case kMatching:
        case kTwoPeer: {
            for (int q = 0; q < n; ++q) perm[q] = q;
            for (int q = n - 1; q >= 1; --q) {
                const uint64_t r = hash4(spec.seed, kTagPerm, static_cast<uint64_t>(round),
                                         static_cast<uint64_t>(q)) >> 32;
                const int j = static_cast<int>((r * static_cast<uint64_t>(q + 1)) >> 32);
                const int t = perm[q];
                perm[q] = perm[j];
                perm[j] = t;
            }
            if (spec.kind == kMatching) {
                for (int p = 0; p + 1 < n; p += 2) edge(perm[p], perm[p + 1]);
            } else {
                for (int q = 0; q < n; ++q) edge(perm[q], perm[(q + 1) % n]);
            }
            break;
        }
        default:
            break;
        }
    }
    __syncwarp();
    // edge activation: lane a decides the edges {a < b}
    uint32_t drop = 0u;
    if (spec.edge_thr < (1ull << 32) && lane < n) {
        const uint32_t mine = adj[lane];
        for (int b = lane + 1; b < n; ++b) {
            if (!((mine >> b) & 1u)) continue;
            const uint64_t r = hash4(spec.seed, kTagEdge, static_cast<uint64_t>(round),
                                     static_cast<uint64_t>(lane) * n + b) >> 32;
            if (!(r < spec.edge_thr)) drop |= 1u << b;
        }
    }
    __syncwarp();
    // apply the drops symmetrically: gather every lane's drop mask
    uint32_t row = lane < n ? adj[lane] : 0u;
    for (int a = 0; a < n; ++a) {
        const uint32_t da = __shfl_sync(0xffffffffu, drop, a);
        if (lane < n) {
            if (lane == a) row &= ~da;
            else if ((da >> lane) & 1u) row &= ~(1u << a);
        }
    }
    if (lane < n) deg[lane] = __popc(row);
    __syncwarp();
    if (lane < n) {
        const int di = deg[lane];
        int q = 0;
        double rest = 0.0;
        for (int j = 0; j < n; ++j) {
            if (j != lane && !((row >> j) & 1u)) continue;
            double w;
            if (spec.weights == 0) {            // uniform
                w = 1.0 / static_cast<double>(di + 1);
            } else if (spec.weights == 1) {     // Metropolis
                if (j == lane) {
                    w = 0.0;                     // filled below
                } else {
                    const int dm = di > deg[j] ? di : deg[j];
                    w = 1.0 / static_cast<double>(1 + dm);
                }
            } else {                             // lazy
                w = di == 0 ? 1.0 : (j == lane ? 0.5 : 0.5 / static_cast<double>(di));
            }
            out->nbr[lane][q] = j;
            out->w[lane][q] = __double2float_rn(w);
            ++q;
        }
        if (spec.weights == 1) {
            // self weight = 1 - sum of the others, summed in ascending j
            int qs = 0;
            for (int j = 0; j < n; ++j) {
                if (j == lane) continue;
                if (!((row >> j) & 1u)) continue;
                const int dm = di > deg[j] ? di : deg[j];
                rest += 1.0 / static_cast<double>(1 + dm);
            }
            for (int q2 = 0; q2 <= di; ++q2)
                if (out->nbr[lane][q2] == lane) qs = q2;
            out->w[lane][qs] = __double2float_rn(1.0 - rest);
        }
        for (; q < kMaxWorkers; ++q) {
            out->nbr[lane][q] = lane;
            out->w[lane][q] = 0.0f;
        }
        out->deg[lane] = di;
    }
}

// Scalars of every worker's next local step (step n_i + 1) from the
// device-resident counters, without advancing them (one warp; lane i =
// worker i).  Run after a start, a hyperparameter change or a checkpoint
// load; from then on every AdamW launch advances the counters of the workers
// it stepped and writes their next scalars itself.
__global__ void prep_kernel(const PrepArgs a) {
    const int i = threadIdx.x;
    if (i >= a.n_workers) return;
    const int64_t n = a.state->nsteps[i] + 1;
    write_step_scalars(a.table, i, n, __dmul_rn(a.state->p1[i], a.beta1), __dmul_rn(a.state->p2[i], a.beta2),
                       lr_of_step(n, a.lr_sched, a.lr_steps, a.lr_after), a.wd, a.seed);
}

// Loads of the average marked as the last use of their lines (ld.global.lu):
// measured 0.998 of the copy peak against 0.938 evict-first on the 8-worker
// GPT-2-small workload.
constexpr Cache kLdAverage = Cache::kLast;

// xbar = (1/n) sum_i x_i: per element an fp32 sum in ascending i, times
// fl32(1/n); fp32 out.  One thread owns a column of 4 elements of a tile and
// loads all n workers' values of it, 8 workers at a time (their loads issued
// together).  The output is stored as one 16-byte vector where its address
// allows (tensor offsets in a list layout can be odd), else element by element.
template <typename T>
__global__ void __launch_bounds__(256) average_kernel(const TensorDesc *tens, const Tile *tiles, int64_t ntiles,
                                                      int32_t n, float *dst, int64_t n_params, int32_t *err) {
    using E = Elem<T>;
    const float inv_n = static_cast<float>(1.0 / n);
    const int e0 = 4 * threadIdx.x;
    for (int64_t ti = blockIdx.x; ti < ntiles; ti += gridDim.x) {
        const Tile tl = tiles[ti];
        if (e0 >= tl.len) continue;
        const TensorDesc &d = tens[tl.tensor];
        const T *X = as<T>(static_cast<const void *>(d.x));
        const int64_t off = tl.start + e0;
        const int nvalid = tl.len - e0 < 4 ? tl.len - e0 : 4;
        float s[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        constexpr int U = 8;
        for (int i0 = 0; i0 < n; i0 += U) {
            typename E::Raw xv[U];
#pragma unroll
            for (int u = 0; u < U; ++u)
                if (i0 + u < n)
                    xv[u] = row_ok(i0 + u, n, off, 4, d.wstride, err)
                                ? E::template load_raw<kLdAverage>(X + (i0 + u) * d.wstride + off)
                                : typename E::Raw{};
#pragma unroll
            for (int u = 0; u < U; ++u) {
                if (i0 + u >= n) continue;
                const float4 v = E::unpack(xv[u]);
                s[0] = __fadd_rn(s[0], v.x);
                s[1] = __fadd_rn(s[1], v.y);
                s[2] = __fadd_rn(s[2], v.z);
                s[3] = __fadd_rn(s[3], v.w);
            }
        }
        if (!span_ok(d.loff + off, d.loff + off + nvalid, n_params, err)) continue;
        float *o = dst + d.loff + off;
        const float4 r = make_float4(__fmul_rn(s[0], inv_n), __fmul_rn(s[1], inv_n), __fmul_rn(s[2], inv_n),
                                     __fmul_rn(s[3], inv_n));
        if (nvalid == 4 && (reinterpret_cast<uintptr_t>(o) & 15u) == 0) {
            *reinterpret_cast<float4 *>(o) = r;
        } else {
            const float ra[4] = {r.x, r.y, r.z, r.w};
            for (int l = 0; l < nvalid; ++l) o[l] = ra[l];
        }
    }
}

template <typename T>
__global__ void gather_kernel(const TensorDesc *tens, int32_t ntens, int32_t which, int32_t worker,
                              const int64_t *idx, int64_t n, float *out, int32_t *err) {
    const int64_t q = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
    if (q >= n) return;
    const int64_t k = idx[q];
    // binary search for the tensor holding the context's element k
    int lo = 0, hi = ntens - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) / 2;
        if (tens[mid].loff <= k) lo = mid; else hi = mid - 1;
    }
    const TensorDesc d = tens[lo];
    const int64_t off = k - d.loff;
    if (k < 0 || off < 0 || off >= d.numel) {
        atomicCAS(err, kDevOk, kDevBadIndex);
        out[q] = 0.0f;
        return;
    }
    const void *base;
    int64_t stride = d.wstride;
    switch (which) {
    case 0: base = d.x; break;
    case 1: base = d.y; break;
    case 2: base = d.m; break;
    case 3: base = d.v; break;
    case 4: base = d.b; break;
    case 5: base = d.c; break;
    default: base = d.h; stride = d.hstride; break;
    }
    out[q] = Elem<T>::load1(static_cast<const T *>(base) + worker * stride + off);
}

// Host transfers of a bf16 store pass through an fp32 staging buffer on the
// device: narrowing rounds to nearest, ties to even; widening is exact.
__global__ void narrow_kernel(const float *src, bf16 *dst, int64_t n) {
    const int64_t step = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t k = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; k < n; k += step)
        dst[k] = __float2bfloat16_rn(src[k]);
}

__global__ void widen_kernel(const bf16 *src, float *dst, int64_t n) {
    const int64_t step = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t k = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; k < n; k += step)
        dst[k] = __bfloat162float(src[k]);
}

// Evaluates one row check that fails (row n of an n-row buffer) without
// touching memory: in the checked build it must record kDevBadIndex.
__global__ void check_selftest_kernel(int32_t *err) {
    if (threadIdx.x == 0) {
        const int64_t rows = 4, stride = 64;
        (void)row_ok(rows, rows, 0, 4, stride, err);
    }
}

// A wait on an mbarrier that nothing ever completes, through the bounded-wait
// routine the pipeline kernels use: it must give up after limit_ns, record
// kDevWaitTimeout and return.
__global__ void wait_selftest_kernel(uint64_t limit_ns, int32_t *err) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        ptx::mbar_init(&bar, 1);
        ptx::fence_mbar_init();
    }
    __syncthreads();
    const bool ok = ptx::mbar_wait_bounded(&bar, 0, limit_ns);
    if (!ok && threadIdx.x == 0) atomicCAS(err, kDevOk, kDevWaitTimeout);
}

}  // namespace

cudaError_t launch_wait_selftest(uint64_t limit_ns, int32_t *err, cudaStream_t s) {
    wait_selftest_kernel<<<1, 32, 0, s>>>(limit_ns, err);
    return cudaGetLastError();
}

cudaError_t launch_init(const InitArgs &a, int grid, cudaStream_t s) {
    if (a.storage == kStoreBF16)
        init_kernel<bf16><<<grid, 256, 0, s>>>(a);
    else
        init_kernel<float><<<grid, 256, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_topo(const TopoSpec &spec, int64_t round, const int64_t *round_ptr, Topo *out,
                        cudaStream_t s) {
    topo_kernel<<<1, 32, 0, s>>>(spec, round, round_ptr, out);
    return cudaGetLastError();
}

cudaError_t launch_prep(const PrepArgs &a, cudaStream_t s) {
    prep_kernel<<<1, 32, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_average(const TensorDesc *tens, const Tile *tiles, int64_t ntiles, int32_t n,
                           int32_t storage, float *dst, int64_t n_params, int32_t *err, int grid, cudaStream_t s) {
    if (storage == kStoreBF16)
        average_kernel<bf16><<<grid, 256, 0, s>>>(tens, tiles, ntiles, n, dst, n_params, err);
    else
        average_kernel<float><<<grid, 256, 0, s>>>(tens, tiles, ntiles, n, dst, n_params, err);
    return cudaGetLastError();
}

int checked_build() { return kChecked ? 1 : 0; }

cudaError_t launch_check_selftest(int32_t *err, cudaStream_t s) {
    check_selftest_kernel<<<1, 32, 0, s>>>(err);
    return cudaGetLastError();
}

cudaError_t launch_gather(const TensorDesc *tens, int32_t ntens, int32_t storage, int32_t which,
                          int32_t worker, const int64_t *idx, int64_t n, float *out, int32_t *err,
                          cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const unsigned grid = static_cast<unsigned>((n + 255) / 256);
    if (storage == kStoreBF16)
        gather_kernel<bf16><<<grid, 256, 0, s>>>(tens, ntens, which, worker, idx, n, out, err);
    else
        gather_kernel<float><<<grid, 256, 0, s>>>(tens, ntens, which, worker, idx, n, out, err);
    return cudaGetLastError();
}

cudaError_t launch_convert(const void *src, void *dst, int64_t n, bool narrow, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const int64_t want = (n + 255) / 256;
    const unsigned grid = static_cast<unsigned>(want < 152 * 16 ? want : 152 * 16);
    if (narrow)
        narrow_kernel<<<grid, 256, 0, s>>>(static_cast<const float *>(src), static_cast<bf16 *>(dst), n);
    else
        widen_kernel<<<grid, 256, 0, s>>>(static_cast<const bf16 *>(src), static_cast<float *>(dst), n);
    return cudaGetLastError();
}

uint64_t host_hash(uint64_t seed, uint64_t tag, uint64_t a, uint64_t b) {
    return hash4(seed, tag, a, b);
}

}  // namespace gasloc
