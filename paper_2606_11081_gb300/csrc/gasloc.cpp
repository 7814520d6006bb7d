// gasloc.cpp -- the C ABI of include/gasloc.h: argument checking, the
// structure-of-arrays replica store, per-step host scalars and kernel launches.
//
// Host arithmetic that the device results depend on (bias corrections, decay,
// the fp32 rounding of hyperparameters) is done in double and rounded once;
// this file is compiled with -ffp-contract=off so that no a*b+c is fused.
#include <cuda.h>   // tensor-map types only; the encoder is fetched through the runtime
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>   // header-only: ranges are no-ops unless a profiler is attached

#include "../../include/gasloc.h"
#include "internal.h"

using namespace gasloc;

namespace {

thread_local std::string g_err;

int fail(int code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return code;
}

int cuda_fail(cudaError_t e, const char *what) {
    return fail(GASLOC_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

constexpr int64_t kMaxParams = (int64_t(1) << 31) - 1;
constexpr int64_t kPadFloats = 64;
constexpr int kTileA = 1024;          // init / adamw / ce / average tiles (4 x 256 threads)
constexpr int kMaxLocalSteps = 1024;
constexpr int kCeRing = 4096;
// Rounds per replay of gasloc_run's longer graph (a single-round graph takes the rest).
constexpr int32_t kGraphBlock = 8;
constexpr int64_t kMaxScheduleSteps = int64_t(1) << 24;
constexpr int kDirectTilesPerCta = 8;   // the direct gossip variant up to this many 1024-element tiles per CTA
constexpr int kStagedTilesPerCta = 8;   // fp32 stores take the staged AdamW up to this many tiles per CTA
constexpr int64_t kRoundMaxElems = 8LL * kTileA;  // the fused round up to this many elements per CTA

int64_t round_up(int64_t v, int64_t m) { return (v + m - 1) / m * m; }

// Names the host-side span of an API call on profiler timelines.
struct NvtxRange {
    explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
};

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
        else
            cudaGetLastError();
    }
    return fn;
}

// 2-D map over one array of one tensor: [n workers][numel] elements with a
// row pitch of wstride elements, boxes of [n x box]; out-of-range elements
// read as zero and are not written.
bool make_map(CUtensorMap *m, void *base, int64_t numel, int64_t wstride, int32_t n, int storage, int box_elems) {
    EncodeTiledFn enc = encode_tiled();
    if (!enc) return false;
    const bool bf = storage == kStoreBF16;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(numel), static_cast<cuuint64_t>(n)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(wstride) * (bf ? 2 : 4)};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(box_elems), static_cast<cuuint32_t>(n)};
    const cuuint32_t estr[2] = {1, 1};
    return enc(m, bf ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims, strides, box,
               estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

void gasloc::set_last_error(const char *msg) { g_err = msg; }

struct gasloc_ctx {
    int32_t n = 0;
    int64_t P = 0;                   // parameters per replica this context holds (p_end - p_begin)
    int64_t P_global = 0;            // parameters per replica of the whole problem
    int64_t p_begin = 0, p_end = 0;  // the global indices [p_begin, p_end) this context holds
    std::vector<int64_t> layout;     // tensor sizes of the whole problem (gasloc_set_layout)
    TopoSpec spec{};
    uint64_t seed = 0;
    gasloc_hparams hp{};
    std::vector<int64_t> numels;
    gasloc_alloc_fn alloc = nullptr;   // numels: the context's pieces of those tensors (gasloc_start)
    gasloc_free_fn free_fn = nullptr;
    void *alloc_user = nullptr;
    cudaStream_t stream = nullptr;
    bool started = false;
    int sms = 0;

    // device store
    std::vector<TensorDesc> tens_h;
    std::vector<int64_t> goff;
    TensorDesc *tens_d = nullptr;
    Tile *tiles_a = nullptr;
    int64_t ntiles_a = 0;
    Tile *tiles_g = nullptr;
    int64_t ntiles_g = 0;
    int tile_g = 0;
    int grid_a = 0, grid_ce = 0;
    int grid_as = 0;                       // staged fp32 AdamW grid where it is used (0: not)
    int grid_gm[6] = {0, 0, 0, 0, 0, 0};   // gossip grid per outer mode
    int grid_gd[6] = {0, 0, 0, 0, 0, 0};   // direct gossip grid per outer mode (0: not used)
    Tile *tiles_r = nullptr;               // tiles of the fused round kernel (where it is used)
    int64_t ntiles_r = 0;
    int grid_r[6] = {0, 0, 0, 0, 0, 0};    // fused round grid per outer mode (0: not used)
    Topo *topo_d = nullptr, *topo_scratch = nullptr;
    void *maps_d = nullptr;   // [tensor][x, y, b] CUtensorMap
    double *partials = nullptr;
    unsigned int *ticket = nullptr;
    unsigned long long *work = nullptr;   // unit counter of the staged AdamW: [0] claimed, [1] producers done
    double *ce_d = nullptr;          // [0] standalone reduction result
    double *ce_ring = nullptr;       // consensus error of round t at [t % kCeRing]
    DevState *state_d = nullptr;     // device-resident step counters
    double *lr_sched_d = nullptr;    // lr of local steps 1..lr_steps (schedule of App. B)
    int64_t lr_sched_cap = 0, lr_steps = 0;
    double lr_after = 0.0;           // lr of every later step (the constant lr without a schedule)
    StepTable *table_d = nullptr;    // scalars of each worker's next local step
    float *avg_d = nullptr;          // n_params floats: the average on its way to host memory
    uint64_t table_gen = 0;          // gen at which table_d was last refreshed (0: never; gen starts at 1)
    cudaStream_t cap_stream = nullptr;
    cudaGraphExec_t graph = nullptr; // one round, captured by gasloc_run
    int32_t graph_H = 0;
    uint64_t graph_gen = 0, gen = 1; // configuration generation the graph was built for
    int64_t graph_launches = 0;      // kernels per replayed round
    cudaGraphExec_t graph_blk = nullptr;   // kGraphBlock consecutive rounds, for longer runs
    int32_t graph_blk_H = 0;
    uint64_t graph_blk_gen = 0;
    int64_t graph_blk_launches = 0;  // kernels per replay of the block
    int32_t *err_d = nullptr;
    void *pinned = nullptr;   // [ce double][err int32][Topo]
    std::vector<std::pair<void *, size_t>> allocs;

    // counters
    std::vector<int64_t> nsteps;
    std::vector<int32_t> Hi;
    bool has_Hi = false;
    uint32_t fresh_mask = 0;
    int64_t round = 0;
    bool ce_valid = false;
    bool topo_static = false, topo_ready = false;
    int64_t launches = 0;

    bool misaligned = false;   // an allocator hook returned a block off a 256-byte boundary
    void *dalloc(size_t bytes) {
        bytes = static_cast<size_t>(round_up(static_cast<int64_t>(bytes ? bytes : 1), 256));
        void *p = nullptr;
        if (alloc) {
            p = alloc(bytes, stream, alloc_user);
        } else if (cudaMalloc(&p, bytes) != cudaSuccess) {
            cudaGetLastError();
            p = nullptr;
        }
        if (p && (reinterpret_cast<uintptr_t>(p) & 255u) != 0) {
            // the bulk and tensor-map copies address rows at 16-byte
            // boundaries: hand the block back rather than fault on it
            if (free_fn) free_fn(p, stream, alloc_user);
            else if (!alloc) cudaFree(p);
            misaligned = true;
            return nullptr;
        }
        if (p) allocs.emplace_back(p, bytes);
        return p;
    }
    void dfree(void *p) {
        if (!p) return;
        for (size_t q = 0; q < allocs.size(); ++q)
            if (allocs[q].first == p) {
                allocs.erase(allocs.begin() + static_cast<long>(q));
                break;
            }
        if (free_fn) free_fn(p, stream, alloc_user);
        else cudaFree(p);
    }
    void release_all() {
        if (started || !allocs.empty()) cudaStreamSynchronize(stream);
        if (graph) cudaGraphExecDestroy(graph);
        graph = nullptr;
        if (graph_blk) cudaGraphExecDestroy(graph_blk);
        graph_blk = nullptr;
        if (cap_stream) cudaStreamDestroy(cap_stream);
        cap_stream = nullptr;
        for (auto &pr : allocs) {
            if (free_fn) free_fn(pr.first, stream, alloc_user);
            else cudaFree(pr.first);
        }
        allocs.clear();
        avg_d = nullptr;
        if (pinned) cudaFreeHost(pinned);
        pinned = nullptr;
    }
};

namespace {

double *pin_ce(gasloc_ctx *c) { return reinterpret_cast<double *>(c->pinned); }
int32_t *pin_err(gasloc_ctx *c) { return reinterpret_cast<int32_t *>(static_cast<char *>(c->pinned) + 8); }
Topo *pin_topo(gasloc_ctx *c) { return reinterpret_cast<Topo *>(static_cast<char *>(c->pinned) + 64); }

int parse_topology(const char *s, int32_t n, TopoSpec *spec) {
    if (!s) return fail(GASLOC_EINVAL, "topology is NULL");
    std::string t(s);
    spec->rows = spec->cols = 0;
    if (t == "none") spec->kind = kNone;
    else if (t == "ring") spec->kind = kRing;
    else if (t == "complete") spec->kind = kComplete;
    else if (t == "exp") spec->kind = kExp;
    else if (t == "matching") spec->kind = kMatching;
    else if (t == "2peer") spec->kind = kTwoPeer;
    else if (t.rfind("torus:", 0) == 0) {
        int r = 0, c = 0;
        char tail = 0;
        if (std::sscanf(t.c_str() + 6, "%dx%d%c", &r, &c, &tail) != 2 || r < 1 || c < 1)
            return fail(GASLOC_EINVAL, "bad torus spec '%s' (want torus:RxC)", s);
        if (static_cast<int64_t>(r) * c != n)
            return fail(GASLOC_EINVAL, "torus %dx%d does not have %d nodes", r, c, n);
        spec->kind = kTorus;
        spec->rows = r;
        spec->cols = c;
    } else {
        return fail(GASLOC_EINVAL, "unknown topology '%s'", s);
    }
    if ((spec->kind == kMatching || spec->kind == kTwoPeer) && n < 2)
        return fail(GASLOC_EINVAL, "randomized peer schemes need at least 2 workers");
    return GASLOC_OK;
}

int check_hparams(const gasloc_hparams *hp) {
    if (!(hp->lr >= 0.0) || !std::isfinite(hp->lr)) return fail(GASLOC_EINVAL, "lr must be >= 0");
    if (!(hp->beta1 >= 0.0 && hp->beta1 < 1.0) || !(hp->beta2 >= 0.0 && hp->beta2 < 1.0))
        return fail(GASLOC_EINVAL, "betas must be in [0, 1)");
    if (!(hp->eps > 0.0) || !std::isfinite(hp->eps)) return fail(GASLOC_EINVAL, "eps must be > 0");
    if (!(hp->weight_decay >= 0.0) || !std::isfinite(hp->weight_decay))
        return fail(GASLOC_EINVAL, "weight decay must be >= 0");
    if (!(hp->noise_sigma >= 0.0) || !std::isfinite(hp->noise_sigma))
        return fail(GASLOC_EINVAL, "noise sigma must be >= 0");
    if (!(hp->edge_prob >= 0.0 && hp->edge_prob <= 1.0)) return fail(GASLOC_EINVAL, "edge_prob must be in [0, 1]");
    if (!(hp->outer_lr >= 0.0) || !(hp->outer_momentum >= 0.0) || !(hp->eta >= 0.0) || !(hp->alpha >= 0.0) ||
        !(hp->gamma >= 0.0) || !std::isfinite(hp->outer_lr) || !std::isfinite(hp->outer_momentum) ||
        !std::isfinite(hp->eta) || !std::isfinite(hp->alpha) || !std::isfinite(hp->gamma))
        return fail(GASLOC_EINVAL, "outer hyperparameters must be finite and >= 0");
    if (hp->outer_mode < GASLOC_OUTER_SGD || hp->outer_mode > GASLOC_OUTER_LOCAL_DADAM)
        return fail(GASLOC_EINVAL, "unknown outer mode %d", hp->outer_mode);
    if (hp->weights < GASLOC_W_UNIFORM || hp->weights > GASLOC_W_LAZY)
        return fail(GASLOC_EINVAL, "unknown weight rule %d", hp->weights);
    if (hp->per_worker_h != 0 && hp->per_worker_h != 1) return fail(GASLOC_EINVAL, "per_worker_h must be 0 or 1");
    if (hp->storage != GASLOC_STORAGE_F32 && hp->storage != GASLOC_STORAGE_BF16)
        return fail(GASLOC_EINVAL, "unknown storage type %d", hp->storage);
    if (hp->lr_total_steps < 0 || hp->lr_total_steps > kMaxScheduleSteps)
        return fail(GASLOC_EINVAL, "lr_total_steps must be in [0, %lld]", (long long)kMaxScheduleSteps);
    auto frac = [](double v) { return v >= 0.0 && v <= 1.0; };
    if (!frac(hp->lr_warmup_frac) || !frac(hp->lr_warmup_start) || !frac(hp->lr_final_frac))
        return fail(GASLOC_EINVAL, "schedule fractions must be in [0, 1]");
    return GASLOC_OK;
}

void refresh_spec(gasloc_ctx *c) {
    c->spec.n = c->n;
    c->spec.seed = c->seed;
    c->spec.weights = c->hp.weights;
    const double thr = std::floor(c->hp.edge_prob * 4294967296.0);
    c->spec.edge_thr = static_cast<uint64_t>(thr);
    c->topo_static = (c->spec.kind != kMatching && c->spec.kind != kTwoPeer && c->spec.edge_thr >= (1ull << 32));
    c->topo_ready = false;
}

int check_started(const gasloc_ctx *c) {
    if (!c) return fail(GASLOC_EINVAL, "context is NULL");
    if (!c->started) return fail(GASLOC_ESTATE, "context not started (call gasloc_start)");
    return GASLOC_OK;
}

int sync_and_check(gasloc_ctx *c) {
    cudaError_t e = cudaMemcpyAsync(pin_err(c), c->err_d, sizeof(int32_t), cudaMemcpyDeviceToHost, c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "reading the device error flag");
    e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
    const int32_t err = *pin_err(c);
    if (err != kDevOk) {
        cudaMemsetAsync(c->err_d, 0, sizeof(int32_t), c->stream);
        cudaStreamSynchronize(c->stream);
        return fail(GASLOC_EDEVICE, "a kernel reported device error %d (%s)", err,
                    err == kDevWaitTimeout ? "bounded wait timed out" : "index out of range");
    }
    return GASLOC_OK;
}

// Writes the device step counters from the host mirrors (round, step counts)
// with beta^n formed as n successive products from 1 with the current betas,
// as the device forms them step by step.  Waits for the stream first.
int restore_step_counters(gasloc_ctx *c) {
    cudaError_t e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
    DevState ds{};
    ds.round = c->round;
    for (int32_t i = 0; i < kMaxWorkers; ++i) {
        double a = 1.0, b = 1.0;
        const int64_t ns = i < c->n ? c->nsteps[i] : 0;
        for (int64_t t = 0; t < ns; ++t) {
            a *= c->hp.beta1;
            b *= c->hp.beta2;
        }
        ds.nsteps[i] = ns;
        ds.p1[i] = a;
        ds.p2[i] = b;
    }
    if (cudaMemcpy(c->state_d, &ds, sizeof ds, cudaMemcpyHostToDevice) != cudaSuccess)
        return fail(GASLOC_ECUDA, "restoring the step counters failed");
    return GASLOC_OK;
}

// Learning rate of a worker's n-th local step under the schedule of App. B
// (see gasloc_hparams): warm-up from lr_warmup_start * lr over W =
// round(lr_warmup_frac * T) steps, then cosine decay to lr_final_frac * lr at
// step T, held after; T = 0: constant.  Double, one rounding per operation.
double sched_lr(const gasloc_hparams &hp, int64_t n) {
    const int64_t T = hp.lr_total_steps;
    if (T <= 0) return hp.lr;
    const int64_t W = static_cast<int64_t>(std::llround(hp.lr_warmup_frac * static_cast<double>(T)));
    if (n <= W) {
        const double s0 = hp.lr_warmup_start;
        return hp.lr * (s0 + (1.0 - s0) * (static_cast<double>(n - 1) / static_cast<double>(W)));
    }
    const int64_t span = T - W - 1;
    double q = span > 0 ? static_cast<double>(n - W - 1) / static_cast<double>(span) : 1.0;
    if (q > 1.0) q = 1.0;
    const double f = hp.lr_final_frac;
    const double pi = 3.14159265358979323846;
    return hp.lr * (f + (1.0 - f) * (0.5 * (1.0 + std::cos(pi * q))));
}

// Puts the rates of local steps 1..T of the current schedule on the device
// (the kernels index them by each worker's step count; later steps use
// lr_after).  Waits for the stream.
int upload_schedule(gasloc_ctx *c) {
    const int64_t T = c->hp.lr_total_steps;
    c->lr_after = sched_lr(c->hp, T + 1);
    c->lr_steps = 0;
    if (T == 0) return GASLOC_OK;
    cudaError_t e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
    if (T > c->lr_sched_cap) {
        c->dfree(c->lr_sched_d);
        c->lr_sched_d = static_cast<double *>(c->dalloc(static_cast<size_t>(T) * sizeof(double)));
        c->lr_sched_cap = c->lr_sched_d ? T : 0;
        if (!c->lr_sched_d) return fail(GASLOC_ENOMEM, "device allocation failed (lr schedule)");
    }
    std::vector<double> v(static_cast<size_t>(T));
    for (int64_t n = 1; n <= T; ++n) v[static_cast<size_t>(n - 1)] = sched_lr(c->hp, n);
    e = cudaMemcpy(c->lr_sched_d, v.data(), v.size() * sizeof(double), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "uploading the lr schedule");
    c->lr_steps = T;
    return GASLOC_OK;
}

int launch_checked(gasloc_ctx *c, cudaError_t e, const char *what) {
    if (e != cudaSuccess) return cuda_fail(e, what);
    ++c->launches;
    return GASLOC_OK;
}

int build_topology(gasloc_ctx *c, int64_t round, const int64_t *round_ptr, Topo *dst, cudaStream_t s) {
    return launch_checked(c, launch_topo(c->spec, round, round_ptr, dst, s), "topology kernel");
}

size_t esize_of(const gasloc_ctx *c) { return c->hp.storage == GASLOC_STORAGE_BF16 ? 2 : 4; }

// fp32 staging buffer on the device for host transfers of a bf16 store: the
// largest tensor, capped at 32 Mi elements (128 MiB).  The stream is
// synchronized before the buffer is released.
struct StagingBuffer {
    static constexpr int64_t kMaxElems = int64_t(1) << 25;
    gasloc_ctx *c;
    float *p = nullptr;
    int64_t elems = 0;
    explicit StagingBuffer(gasloc_ctx *ctx, bool want = true) : c(ctx) {
        if (!want) return;
        int64_t mx = 1;
        for (const TensorDesc &d : c->tens_h) mx = d.numel > mx ? d.numel : mx;
        elems = mx < kMaxElems ? mx : kMaxElems;
        p = static_cast<float *>(c->dalloc(static_cast<size_t>(elems) * 4));
    }
    ~StagingBuffer() {
        if (!p) return;
        cudaStreamSynchronize(c->stream);
        c->dfree(p);
    }
    StagingBuffer(const StagingBuffer &) = delete;
    StagingBuffer &operator=(const StagingBuffer &) = delete;
};

// Base address (bytes) of buffer `which` of a tensor; *stride in elements.
char *buffer_base(const TensorDesc &d, int which, int64_t *stride) {
    *stride = d.wstride;
    switch (which) {
    case GASLOC_BUF_X: return static_cast<char *>(d.x);
    case GASLOC_BUF_Y: return static_cast<char *>(d.y);
    case GASLOC_BUF_M: return static_cast<char *>(d.m);
    case GASLOC_BUF_V: return static_cast<char *>(d.v);
    case GASLOC_BUF_B: return static_cast<char *>(d.b);
    case GASLOC_BUF_C: return static_cast<char *>(d.c);
    case GASLOC_BUF_H: *stride = d.hstride; return static_cast<char *>(d.h);
    default: return nullptr;
    }
}

int check_which_worker(const gasloc_ctx *c, int32_t which, int32_t worker, bool allow_all) {
    if (which < GASLOC_BUF_X || which > GASLOC_BUF_H) return fail(GASLOC_EINVAL, "unknown buffer %d", which);
    const int32_t rows = (which == GASLOC_BUF_H && !c->hp.per_worker_h) ? 1 : c->n;
    if (worker == -1 && allow_all) return GASLOC_OK;
    if (worker < 0 || worker >= rows) return fail(GASLOC_EINVAL, "worker %d out of range", worker);
    return GASLOC_OK;
}

}  // namespace

// ------------------------------------------------------------------ API ----

extern "C" {

void gasloc_default_hparams(gasloc_hparams *hp) {
    if (!hp) return;
    std::memset(hp, 0, sizeof *hp);
    hp->lr = 3e-4;
    hp->beta1 = 0.9;
    hp->beta2 = 0.95;
    hp->eps = 1e-8;
    hp->weight_decay = 0.1;
    hp->noise_sigma = 0.01;
    hp->outer_lr = 0.7;
    hp->outer_momentum = 0.9;
    hp->eta = 1.0;
    hp->alpha = 1.0;
    hp->gamma = 0.0;
    hp->edge_prob = 1.0;
    hp->lr_total_steps = 0;
    hp->lr_warmup_frac = 0.1;
    hp->lr_warmup_start = 0.01;
    hp->lr_final_frac = 0.0;
    hp->outer_mode = GASLOC_OUTER_NESTEROV;
    hp->weights = GASLOC_W_UNIFORM;
    hp->per_worker_h = 0;
}

const char *gasloc_last_error(void) { return g_err.c_str(); }

int gasloc_init(int32_t n_workers, int64_t n_params, const char *topology, uint64_t seed, gasloc_ctx **out) {
    if (!out) return fail(GASLOC_EINVAL, "out is NULL");
    *out = nullptr;
    if (n_workers < 1 || n_workers > GASLOC_MAX_WORKERS)
        return fail(GASLOC_EINVAL, "n_workers must be in [1, %d], got %d", GASLOC_MAX_WORKERS, n_workers);
    if (n_params < 1 || n_params > kMaxParams)
        return fail(GASLOC_EINVAL, "n_params must be in [1, 2^31-1], got %lld", static_cast<long long>(n_params));
    TopoSpec spec{};
    int rc = parse_topology(topology, n_workers, &spec);
    if (rc) return rc;
    gasloc_ctx *c = new (std::nothrow) gasloc_ctx();
    if (!c) return fail(GASLOC_ENOMEM, "out of host memory");
    c->n = n_workers;
    c->P = n_params;
    c->P_global = n_params;
    c->p_begin = 0;
    c->p_end = n_params;
    c->layout.assign(1, n_params);
    c->spec = spec;
    c->seed = seed;
    gasloc_default_hparams(&c->hp);
    c->numels.assign(1, n_params);
    c->nsteps.assign(n_workers, 0);
    c->Hi.assign(n_workers, 0);
    refresh_spec(c);
    *out = c;
    return GASLOC_OK;
}

int gasloc_set_hparams(gasloc_ctx *c, const gasloc_hparams *hp) {
    if (!c || !hp) return fail(GASLOC_EINVAL, "NULL argument");
    int rc = check_hparams(hp);
    if (rc) return rc;
    if (c->started && (hp->per_worker_h != c->hp.per_worker_h || hp->storage != c->hp.storage))
        return fail(GASLOC_ESTATE, "per_worker_h and storage cannot change after gasloc_start");
    const bool new_betas = c->started && (hp->beta1 != c->hp.beta1 || hp->beta2 != c->hp.beta2);
    c->hp = *hp;
    c->gen += 1;
    refresh_spec(c);
    // bias corrections are 1 - beta^n with the current betas: re-form the
    // device products beta^n from the step counts
    if (c->started) {
        const int rc = upload_schedule(c);
        if (rc) return rc;
    }
    if (new_betas) return restore_step_counters(c);
    return GASLOC_OK;
}

int gasloc_get_hparams(const gasloc_ctx *c, gasloc_hparams *hp) {
    if (!c || !hp) return fail(GASLOC_EINVAL, "NULL argument");
    *hp = c->hp;
    return GASLOC_OK;
}

int gasloc_set_layout(gasloc_ctx *c, int32_t n_tensors, const int64_t *numels) {
    if (!c || !numels) return fail(GASLOC_EINVAL, "NULL argument");
    if (c->started) return fail(GASLOC_ESTATE, "layout cannot change after gasloc_start");
    if (n_tensors < 1 || n_tensors > (1 << 20)) return fail(GASLOC_EINVAL, "n_tensors out of range");
    int64_t tot = 0;
    for (int32_t t = 0; t < n_tensors; ++t) {
        if (numels[t] < 1) return fail(GASLOC_EINVAL, "tensor %d has %lld elements", t, (long long)numels[t]);
        tot += numels[t];
    }
    if (tot != c->P_global)
        return fail(GASLOC_EINVAL, "tensor sizes sum to %lld, not n_params %lld", (long long)tot,
                    (long long)c->P_global);
    c->layout.assign(numels, numels + n_tensors);
    return GASLOC_OK;
}

int gasloc_set_range(gasloc_ctx *c, int64_t p_begin, int64_t p_end) {
    if (!c) return fail(GASLOC_EINVAL, "context is NULL");
    if (c->started) return fail(GASLOC_ESTATE, "the range cannot change after gasloc_start");
    if (p_begin < 0 || p_end <= p_begin || p_end > c->P_global)
        return fail(GASLOC_EINVAL, "range [%lld, %lld) is not a non-empty part of [0, %lld)", (long long)p_begin,
                    (long long)p_end, (long long)c->P_global);
    c->p_begin = p_begin;
    c->p_end = p_end;
    c->P = p_end - p_begin;
    return GASLOC_OK;
}

int gasloc_get_range(const gasloc_ctx *c, int64_t *p_begin, int64_t *p_end, int64_t *n_params_global) {
    if (!c || !p_begin || !p_end || !n_params_global) return fail(GASLOC_EINVAL, "NULL argument");
    *p_begin = c->p_begin;
    *p_end = c->p_end;
    *n_params_global = c->P_global;
    return GASLOC_OK;
}

int gasloc_set_allocator(gasloc_ctx *c, gasloc_alloc_fn a, gasloc_free_fn f, void *user) {
    if (!c) return fail(GASLOC_EINVAL, "context is NULL");
    if (c->started) return fail(GASLOC_ESTATE, "allocator cannot change after gasloc_start");
    if ((a == nullptr) != (f == nullptr)) return fail(GASLOC_EINVAL, "give both alloc and free, or neither");
    c->alloc = a;
    c->free_fn = f;
    c->alloc_user = user;
    return GASLOC_OK;
}

int gasloc_set_stream(gasloc_ctx *c, void *s) {
    if (!c) return fail(GASLOC_EINVAL, "context is NULL");
    c->stream = static_cast<cudaStream_t>(s);
    return GASLOC_OK;
}

int gasloc_start(gasloc_ctx *c) {
    NvtxRange r("gasloc_start");
    if (!c) return fail(GASLOC_EINVAL, "context is NULL");
    if (c->started) return fail(GASLOC_ESTATE, "context already started");
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    e = cudaDeviceGetAttribute(&c->sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return cuda_fail(e, "multiprocessor count");

    const int32_t n = c->n;
    const int32_t nh = c->hp.per_worker_h ? n : 1;
    // the context's pieces of the problem's tensors: each tensor cut to
    // [p_begin, p_end), with the global index of its first element
    std::vector<int64_t> piece_goff;
    c->numels.clear();
    {
        int64_t off = 0;
        for (int64_t ne : c->layout) {
            const int64_t lo = std::max(off, c->p_begin), hi = std::min(off + ne, c->p_end);
            if (hi > lo) {
                c->numels.push_back(hi - lo);
                piece_goff.push_back(lo);
            }
            off += ne;
        }
    }
    // size check before any allocation
    int64_t need = 0;
    for (int64_t ne : c->numels) {
        const int64_t ws = round_up(ne, kPadFloats);
        need += (6LL * n + nh) * ws * static_cast<int64_t>(esize_of(c));
    }
    size_t fr = 0, tot = 0;
    if (cudaMemGetInfo(&fr, &tot) == cudaSuccess && static_cast<size_t>(need) > fr)
        return fail(GASLOC_ENOMEM, "replica store needs %lld bytes, %zu free", (long long)need, fr);

    // gossip launch shape (the tile depends on n only; stages and shared
    // memory on the mode's staged rows): size the attribute for the largest
    size_t smem_attr = 0;
    for (int st = 0; st < 2; ++st)
        for (int m = 0; m < 6; ++m) smem_attr = std::max(smem_attr, gossip_shape(n, m, st).smem);
    c->tile_g = gossip_shape(n, GASLOC_OUTER_NESTEROV, c->hp.storage).tile;
    e = gossip_set_smem(smem_attr);
    if (e != cudaSuccess) return cuda_fail(e, "gossip shared-memory attribute");

    auto oom = [&](const char *what) {
        c->release_all();
        c->tens_h.clear();
        if (c->misaligned)
            return fail(GASLOC_EINVAL, "the allocator returned a block that is not 256-byte aligned (%s)", what);
        return fail(GASLOC_ENOMEM, "device allocation failed (%s)", what);
    };

    // replica store
    c->tens_h.clear();
    c->goff.clear();
    for (size_t t = 0; t < c->numels.size(); ++t) {
        TensorDesc d{};
        d.numel = c->numels[t];
        d.wstride = round_up(d.numel, kPadFloats);
        d.hstride = c->hp.per_worker_h ? d.wstride : 0;
        d.goff = piece_goff[t];
        d.loff = piece_goff[t] - c->p_begin;
        void **arrs[6] = {&d.x, &d.y, &d.m, &d.v, &d.b, &d.c};
        for (void **a : arrs) {
            *a = c->dalloc(static_cast<size_t>(n) * d.wstride * esize_of(c));
            if (!*a) return oom("replica arrays");
        }
        d.h = c->dalloc(static_cast<size_t>(nh) * d.wstride * esize_of(c));
        if (!d.h) return oom("curvature");
        c->tens_h.push_back(d);
        c->goff.push_back(d.goff);
    }
    for (auto &pr : c->allocs) {
        e = cudaMemsetAsync(pr.first, 0, pr.second, c->stream);
        if (e != cudaSuccess) { c->release_all(); return cuda_fail(e, "zero fill"); }
    }

    // tile tables
    auto make_tiles = [&](int tile, std::vector<Tile> &v) {
        v.clear();
        for (size_t t = 0; t < c->numels.size(); ++t)
            for (int64_t s = 0; s < c->numels[t]; s += tile)
                v.push_back(Tile{static_cast<int32_t>(t), static_cast<int32_t>(std::min<int64_t>(tile, c->numels[t] - s)), s});
    };
    std::vector<Tile> ta, tg, tr;
    make_tiles(kTileA, ta);
    make_tiles(c->tile_g, tg);
    const bool fusable = round_fits(n, c->hp.storage);
    if (fusable) make_tiles(kRoundTile, tr);
    c->ntiles_a = static_cast<int64_t>(ta.size());
    c->ntiles_g = static_cast<int64_t>(tg.size());
    c->ntiles_r = static_cast<int64_t>(tr.size());

    c->tens_d = static_cast<TensorDesc *>(c->dalloc(sizeof(TensorDesc) * c->tens_h.size()));
    c->tiles_a = static_cast<Tile *>(c->dalloc(sizeof(Tile) * ta.size()));
    c->tiles_g = static_cast<Tile *>(c->dalloc(sizeof(Tile) * tg.size()));
    c->tiles_r = nullptr;
    if (fusable) {
        c->tiles_r = static_cast<Tile *>(c->dalloc(sizeof(Tile) * tr.size()));
        if (!c->tiles_r) return oom("tables");
    }
    std::vector<CUtensorMap> maps(c->tens_h.size() * 3);
    for (size_t t = 0; t < c->tens_h.size(); ++t) {
        const TensorDesc &d = c->tens_h[t];
        void *arrs[3] = {d.x, d.y, d.b};
        for (int k = 0; k < 3; ++k)
            if (!make_map(&maps[t * 3 + k], arrs[k], d.numel, d.wstride, n, c->hp.storage,
                          c->tile_g < 256 ? c->tile_g : 256)) {
                c->release_all();
                return fail(GASLOC_ECUDA, "cuTensorMapEncodeTiled failed for tensor %zu", t);
            }
    }
    c->maps_d = c->dalloc(sizeof(CUtensorMap) * maps.size());
    c->topo_d = static_cast<Topo *>(c->dalloc(sizeof(Topo)));
    c->topo_scratch = static_cast<Topo *>(c->dalloc(sizeof(Topo)));
    const int max_grid = c->sms * 32;
    c->partials = static_cast<double *>(c->dalloc(sizeof(double) * max_grid));
    c->ticket = static_cast<unsigned int *>(c->dalloc(sizeof(unsigned int) * 4));
    c->work = static_cast<unsigned long long *>(c->dalloc(sizeof(unsigned long long) * 4));
    c->ce_d = static_cast<double *>(c->dalloc(sizeof(double) * 2));
    c->ce_ring = static_cast<double *>(c->dalloc(sizeof(double) * kCeRing));
    c->state_d = static_cast<DevState *>(c->dalloc(sizeof(DevState)));
    c->table_d = static_cast<StepTable *>(c->dalloc(sizeof(StepTable)));
    c->err_d = static_cast<int32_t *>(c->dalloc(sizeof(int32_t) * 4));
    // allocated with the rest, so that reading the average back at the end of
    // a run costs the kernel and the copy only
    c->avg_d = static_cast<float *>(c->dalloc(static_cast<size_t>(c->P) * 4));
    if (!c->tens_d || !c->tiles_a || !c->tiles_g || !c->maps_d || !c->topo_d || !c->topo_scratch || !c->partials || !c->ticket ||
        !c->work ||
        !c->ce_d || !c->err_d || !c->ce_ring || !c->state_d || !c->table_d || !c->avg_d)
        return oom("tables");
    if (cudaMallocHost(&c->pinned, 64 + sizeof(Topo)) != cudaSuccess) {
        cudaGetLastError();
        c->pinned = nullptr;
        return oom("pinned host buffer");
    }
    DevState st0{};
    for (int i = 0; i < kMaxWorkers; ++i) st0.p1[i] = st0.p2[i] = 1.0;
    cudaError_t es[9];
    es[8] = fusable ? cudaMemcpyAsync(c->tiles_r, tr.data(), sizeof(Tile) * tr.size(), cudaMemcpyHostToDevice, c->stream)
                    : cudaSuccess;
    es[7] = cudaMemcpyAsync(c->state_d, &st0, sizeof st0, cudaMemcpyHostToDevice, c->stream);
    es[6] = cudaMemcpyAsync(c->maps_d, maps.data(), sizeof(CUtensorMap) * maps.size(), cudaMemcpyHostToDevice,
                            c->stream);
    es[0] = cudaMemcpyAsync(c->tens_d, c->tens_h.data(), sizeof(TensorDesc) * c->tens_h.size(), cudaMemcpyHostToDevice, c->stream);
    es[1] = cudaMemcpyAsync(c->tiles_a, ta.data(), sizeof(Tile) * ta.size(), cudaMemcpyHostToDevice, c->stream);
    es[2] = cudaMemcpyAsync(c->tiles_g, tg.data(), sizeof(Tile) * tg.size(), cudaMemcpyHostToDevice, c->stream);
    es[3] = cudaMemsetAsync(c->ticket, 0, sizeof(unsigned int) * 4, c->stream);
    if (es[3] == cudaSuccess) es[3] = cudaMemsetAsync(c->work, 0, sizeof(unsigned long long) * 4, c->stream);
    es[4] = cudaMemsetAsync(c->err_d, 0, sizeof(int32_t) * 4, c->stream);
    es[5] = cudaMemsetAsync(c->ce_d, 0, sizeof(double) * 2, c->stream);
    for (cudaError_t x : es)
        if (x != cudaSuccess) { c->release_all(); return cuda_fail(x, "table upload"); }
    // the host vectors are freed on return: make the uploads complete first
    e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) { c->release_all(); return cuda_fail(e, "table upload"); }

    c->grid_a = c->sms * adamw_blocks_per_sm(256, c->hp.per_worker_h != 0, c->hp.storage);
    // with fp32 storage and a small store (a few tiles per CTA) the staged
    // AdamW, whose producer warp loads the next unit while the consumers
    // compute, hides the load latency that is otherwise on every tile's path
    c->grid_as = 0;
    if (c->hp.storage == GASLOC_STORAGE_F32) {
        const int gs = c->sms * adamw_staged_fp32_blocks_per_sm(c->hp.per_worker_h != 0);
        if (c->ntiles_a <= static_cast<int64_t>(kStagedTilesPerCta) * gs) c->grid_as = gs;
    }
    for (int m = 0; m < 6; ++m) {
        const GossipShape sm = gossip_shape(n, m, c->hp.storage);
        c->grid_gm[m] = std::min(max_grid, c->sms * gossip_blocks_per_sm(m, c->hp.storage, sm));
    }
    c->grid_ce = std::min(max_grid, c->sms * ce_blocks_per_sm(256, c->hp.storage));
    // the direct gossip variant pays where each CTA of the pipelined one
    // would walk only a few tiles (few workers, a replica store of up to a few
    // hundred MB): one memory round trip per tile instead of a pipeline that
    // never fills
    for (int m = 0; m < 6; ++m) {
        c->grid_gd[m] = 0;
        if (!gossip_direct_fits(n, c->hp.storage)) continue;
        const int gd = std::min(max_grid, c->sms * gossip_direct_blocks_per_sm(m));
        if (c->ntiles_a <= static_cast<int64_t>(kDirectTilesPerCta) * gd) c->grid_gd[m] = gd;
    }
    // the fused round (gasloc_fused_round) for the same small stores
    for (int m = 0; m < 6; ++m) {
        c->grid_r[m] = 0;
        if (!fusable) continue;
        const int gr = std::min(max_grid, c->sms * round_blocks_per_sm(m, c->hp.per_worker_h != 0));
        if (c->P <= kRoundMaxElems * gr) c->grid_r[m] = gr;
    }

    int rc = upload_schedule(c);
    if (rc) { c->release_all(); return rc; }
    InitArgs ia{c->tens_d, c->tiles_a, c->ntiles_a, n, c->hp.per_worker_h, c->seed, c->hp.storage, c->err_d};
    rc = launch_checked(c, launch_init(ia, c->sms * 8, c->stream), "init kernel");
    if (rc) { c->release_all(); return rc; }
    c->started = true;
    c->round = 0;
    c->fresh_mask = 0;
    c->ce_valid = false;
    std::fill(c->nsteps.begin(), c->nsteps.end(), 0);
    refresh_spec(c);
    return GASLOC_OK;
}

int gasloc_set_local_steps(gasloc_ctx *c, const int32_t *H) {
    if (!c) return fail(GASLOC_EINVAL, "context is NULL");
    if (!H) {
        c->has_Hi = false;
        return GASLOC_OK;
    }
    for (int32_t i = 0; i < c->n; ++i)
        if (H[i] < 0 || H[i] > kMaxLocalSteps) return fail(GASLOC_EINVAL, "H_%d = %d out of [0, %d]", i, H[i], kMaxLocalSteps);
    c->Hi.assign(H, H + c->n);
    c->has_Hi = true;
    c->gen += 1;
    return GASLOC_OK;
}

int gasloc_draw_local_steps(gasloc_ctx *c, int32_t hmax) {
    if (!c) return fail(GASLOC_EINVAL, "context is NULL");
    if (hmax < 1 || hmax > kMaxLocalSteps) return fail(GASLOC_EINVAL, "hmax out of [1, %d]", kMaxLocalSteps);
    for (int32_t i = 0; i < c->n; ++i) {
        const uint64_t r = host_hash(c->seed, 7, static_cast<uint64_t>(i), 0) >> 32;
        c->Hi[i] = 1 + static_cast<int32_t>((r * static_cast<uint64_t>(hmax)) >> 32);
    }
    c->has_Hi = true;
    c->gen += 1;
    return GASLOC_OK;
}

int gasloc_get_local_steps(const gasloc_ctx *c, int32_t *H) {
    if (!c || !H) return fail(GASLOC_EINVAL, "NULL argument");
    if (!c->has_Hi) return fail(GASLOC_ESTATE, "no per-worker step counts set");
    std::copy(c->Hi.begin(), c->Hi.end(), H);
    return GASLOC_OK;
}

}  // extern "C"

namespace {

// Rewrites the step table from the device counters (every worker's next
// step) when the hyperparameters or the counters changed since it was last
// written by the device: after a start, gasloc_set_hparams or gasloc_load.
int refresh_step_table(gasloc_ctx *c, cudaStream_t s) {
    if (c->table_gen == c->gen) return GASLOC_OK;
    const gasloc_hparams &hp = c->hp;
    PrepArgs pa{c->state_d, c->table_d, c->n, hp.beta1, hp.beta2, hp.weight_decay, c->lr_sched_d, c->lr_steps,
                c->lr_after, c->seed};
    const int rc = launch_checked(c, launch_prep(pa, s), "step-scalar kernel");
    if (!rc) c->table_gen = c->gen;
    return rc;
}

// Enqueues the local steps of one call on stream s and advances the host
// mirrors (step counts, which workers are fresh).  Every step is one AdamW
// launch: it reads the step's scalars from the table, and its last CTA to
// read them advances the device counters and writes the next step's.
int enqueue_local_steps(gasloc_ctx *c, int32_t H, cudaStream_t s) {
    const gasloc_hparams &hp = c->hp;
    int rc0 = refresh_step_table(c, s);
    if (rc0) return rc0;
    int32_t hmax = H;
    if (H < 0) hmax = *std::max_element(c->Hi.begin(), c->Hi.end());
    AdamwArgs a{};
    a.tens = c->tens_d;
    a.tiles = c->tiles_a;
    a.ntiles = c->ntiles_a;
    a.n_workers = c->n;
    a.staged = c->grid_as > 0 ? 1 : 0;
    a.err = c->err_d;
    a.table = c->table_d;
    a.state = c->state_d;
    a.ticket = c->ticket + 1;   // slot 0: the gossip and consensus-error reductions
    a.work = c->work;
    a.lr_sched = c->lr_sched_d;
    a.lr_steps = c->lr_steps;
    a.lr_after = c->lr_after;
    a.wd = hp.weight_decay;
    a.decay = static_cast<float>(1.0 - hp.lr * hp.weight_decay);
    a.beta1d = hp.beta1;
    a.beta2d = hp.beta2;
    a.seed = c->seed;
    a.per_worker_h = hp.per_worker_h;
    a.storage = hp.storage;
    a.beta1 = static_cast<float>(hp.beta1);
    a.beta2 = static_cast<float>(hp.beta2);
    a.omb1 = static_cast<float>(1.0 - hp.beta1);
    a.omb2 = static_cast<float>(1.0 - hp.beta2);
    a.eps = static_cast<float>(hp.eps);
    a.sigma = static_cast<float>(hp.noise_sigma);
    for (int32_t st = 0; st < hmax; ++st) {
        int na = 0;
        uint32_t mask = 0;
        for (int32_t i = 0; i < c->n; ++i) {
            if (H < 0 && st >= c->Hi[i]) continue;
            a.worker[na++] = i;
            mask |= 1u << i;
        }
        if (na == 0) continue;
        a.active_mask = mask;
        a.n_active = na;
        a.from_x_mask = ~c->fresh_mask;
        const int rc = launch_checked(c, launch_adamw(a, a.staged ? c->grid_as : c->grid_a, 256, s), "adamw kernel");
        if (rc) return rc;
        for (int q = 0; q < na; ++q) c->nsteps[a.worker[q]] += 1;
        c->fresh_mask |= mask;
    }
    return GASLOC_OK;
}

// Enqueues one gossip round (the round's table where the graph is random,
// then the fused mixing / outer-update / consensus-error kernel) on stream s
// and advances the host mirrors.
int enqueue_gossip(gasloc_ctx *c, cudaStream_t s) {
    if (!c->topo_static || !c->topo_ready) {
        const int rc = build_topology(c, c->round, &c->state_d->round, c->topo_d, s);
        if (rc) return rc;
        c->topo_ready = c->topo_static;
    }
    const gasloc_hparams &hp = c->hp;
    GossipArgs a{};
    a.tens = c->tens_d;
    a.tiles = c->tiles_g;
    a.ntiles = c->ntiles_g;
    a.topo = c->topo_d;
    a.maps = c->maps_d;
    a.storage = hp.storage;
    a.n_workers = c->n;
    a.mode = hp.outer_mode;
    a.fresh_mask = c->fresh_mask;
    a.state = c->state_d;
    const GossipShape gs = gossip_shape(c->n, hp.outer_mode, hp.storage);
    const int grid_direct = c->grid_gd[hp.outer_mode];
    a.direct = grid_direct > 0 ? 1 : 0;
    if (a.direct) {
        a.tiles = c->tiles_a;
        a.ntiles = c->ntiles_a;
    }
    a.tile = gs.tile;
    a.groups = gs.groups;
    a.stages = gs.stages;
    a.dense = gs.dense;
    a.eta_out = static_cast<float>(hp.outer_lr);
    a.mu = static_cast<float>(hp.outer_momentum);
    a.eta = static_cast<float>(hp.eta);
    a.alpha = static_cast<float>(hp.alpha);
    a.oma = static_cast<float>(1.0 - hp.alpha);
    a.gamma = static_cast<float>(hp.gamma);
    a.partials = c->partials;
    a.ticket = c->ticket;
    a.ce_ring = c->ce_ring;
    a.ce_ring_len = kCeRing;
    a.err = c->err_d;
    const int rc = launch_checked(c, launch_gossip(a, a.direct ? grid_direct : c->grid_gm[hp.outer_mode], gs.smem, s),
                                  "gossip kernel");
    if (rc) return rc;
    c->round += 1;
    c->fresh_mask = 0;
    c->ce_valid = true;
    return GASLOC_OK;
}

// Enqueues one whole round for gasloc_fused_round: H local steps, then the
// gossip round.  Where the fused round kernel serves the store and every
// worker takes the round's last step from the same iterate (all from x, or
// all from y), the first H - 1 steps are AdamW launches and the last step
// runs fused with the gossip round; otherwise the round is enqueued as the
// two calls would enqueue it.  The results are the same either way.
int enqueue_round(gasloc_ctx *c, int32_t H, cudaStream_t s) {
    const gasloc_hparams &hp = c->hp;
    int32_t Hu = H;   // the workers' common step count (-1: they differ)
    if (H == GASLOC_PER_WORKER_STEPS) {
        Hu = c->Hi[0];
        for (int32_t i = 1; i < c->n; ++i)
            if (c->Hi[i] != Hu) Hu = -1;
    }
    const uint32_t all = c->n == 32 ? 0xffffffffu : (1u << c->n) - 1u;
    const int grid = c->grid_r[hp.outer_mode];
    const bool fuse = grid > 0 && Hu >= 1 && (Hu >= 2 || c->fresh_mask == 0 || c->fresh_mask == all);
    int rc;
    if (!fuse) {
        rc = H == 0 ? GASLOC_OK : enqueue_local_steps(c, H, s);
        return rc ? rc : enqueue_gossip(c, s);
    }
    if (Hu > 1) {
        rc = enqueue_local_steps(c, Hu - 1, s);
        if (rc) return rc;
    }
    rc = refresh_step_table(c, s);
    if (rc) return rc;
    if (!c->topo_static || !c->topo_ready) {
        rc = build_topology(c, c->round, &c->state_d->round, c->topo_d, s);
        if (rc) return rc;
        c->topo_ready = c->topo_static;
    }
    RoundArgs a{};
    a.tens = c->tens_d;
    a.tiles = c->tiles_r;
    a.ntiles = c->ntiles_r;
    a.table = c->table_d;
    a.state = c->state_d;
    a.topo = c->topo_d;
    a.beta1d = hp.beta1;
    a.beta2d = hp.beta2;
    a.wd = hp.weight_decay;
    a.lr_sched = c->lr_sched_d;
    a.lr_steps = c->lr_steps;
    a.lr_after = c->lr_after;
    a.seed = c->seed;
    a.n_workers = c->n;
    a.mode = hp.outer_mode;
    a.per_worker_h = hp.per_worker_h;
    a.from_x = c->fresh_mask == 0 ? 1 : 0;
    a.sched = c->lr_steps > 0 ? 1 : 0;
    a.decay = static_cast<float>(1.0 - hp.lr * hp.weight_decay);
    a.beta1 = static_cast<float>(hp.beta1);
    a.beta2 = static_cast<float>(hp.beta2);
    a.omb1 = static_cast<float>(1.0 - hp.beta1);
    a.omb2 = static_cast<float>(1.0 - hp.beta2);
    a.eps = static_cast<float>(hp.eps);
    a.sigma = static_cast<float>(hp.noise_sigma);
    a.eta_out = static_cast<float>(hp.outer_lr);
    a.mu = static_cast<float>(hp.outer_momentum);
    a.eta = static_cast<float>(hp.eta);
    a.alpha = static_cast<float>(hp.alpha);
    a.oma = static_cast<float>(1.0 - hp.alpha);
    a.gamma = static_cast<float>(hp.gamma);
    a.partials = c->partials;
    a.ticket = c->ticket;
    a.step_ticket = c->ticket + 1;   // the AdamW launches' slot
    a.ce_ring = c->ce_ring;
    a.ce_ring_len = kCeRing;
    a.err = c->err_d;
    rc = launch_checked(c, launch_round(a, grid, s), "round kernel");
    if (rc) return rc;
    for (int32_t i = 0; i < c->n; ++i) c->nsteps[i] += 1;
    c->round += 1;
    c->fresh_mask = 0;
    c->ce_valid = true;
    return GASLOC_OK;
}

int check_H(const gasloc_ctx *c, int32_t H) {
    if (H != GASLOC_PER_WORKER_STEPS && (H < 0 || H > kMaxLocalSteps))
        return fail(GASLOC_EINVAL, "H must be in [0, %d] or GASLOC_PER_WORKER_STEPS", kMaxLocalSteps);
    if (H == GASLOC_PER_WORKER_STEPS && !c->has_Hi) return fail(GASLOC_ESTATE, "per-worker steps requested but none set");
    return GASLOC_OK;
}

// Captures nr consecutive rounds (H local steps, then gossip) into an
// executable graph.  The step table is refreshed and a static neighbour
// table built outside the graph, so a replay holds AdamW, the round's table
// where it is drawn each round, and gossip.  Every kernel reads its round
// and step counters from device memory, so consecutive rounds in one graph
// are the rounds the calls would run.  The host mirrors are restored after
// the capture; the caller advances them once per replayed round.
int capture_rounds(gasloc_ctx *c, int32_t H, int32_t nr, cudaGraphExec_t *out, int64_t *launches_out) {
    if (*out) cudaGraphExecDestroy(*out);
    *out = nullptr;
    if (!c->cap_stream && cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking) != cudaSuccess) {
        cudaGetLastError();
        return fail(GASLOC_ECUDA, "creating the capture stream failed");
    }
    int rc = refresh_step_table(c, c->stream);
    if (rc) return rc;
    if (c->topo_static && !c->topo_ready) {
        rc = build_topology(c, c->round, nullptr, c->topo_d, c->stream);
        if (rc) return rc;
        c->topo_ready = true;
    }
    cudaError_t e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
    const std::vector<int64_t> nsteps0 = c->nsteps;
    const int64_t round0 = c->round, launches0 = c->launches;
    const bool ce0 = c->ce_valid;
    e = cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeThreadLocal);
    if (e != cudaSuccess) return cuda_fail(e, "begin capture");
    for (int32_t r = 0; r < nr && !rc; ++r) {
        rc = H == 0 ? GASLOC_OK : enqueue_local_steps(c, H, c->cap_stream);
        if (!rc) rc = enqueue_gossip(c, c->cap_stream);
    }
    cudaGraph_t g = nullptr;
    const cudaError_t e2 = cudaStreamEndCapture(c->cap_stream, &g);
    *launches_out = c->launches - launches0;
    c->nsteps = nsteps0;
    c->round = round0;
    c->launches = launches0;
    c->ce_valid = ce0;
    c->fresh_mask = 0;
    if (rc) {
        if (g) cudaGraphDestroy(g);
        return rc;
    }
    if (e2 != cudaSuccess) return cuda_fail(e2, "end capture");
    e = cudaGraphInstantiate(out, g, 0);
    cudaGraphDestroy(g);
    if (e != cudaSuccess) {
        *out = nullptr;
        return cuda_fail(e, "graph instantiate");
    }
    return GASLOC_OK;
}

}  // namespace

extern "C" {

int gasloc_local_steps(gasloc_ctx *c, int32_t H) {
    NvtxRange r("gasloc_local_steps");
    int rc = check_started(c);
    if (rc) return rc;
    rc = check_H(c, H);
    if (rc) return rc;
    if (H == 0) return GASLOC_OK;
    return enqueue_local_steps(c, H, c->stream);
}

int gasloc_gossip_round(gasloc_ctx *c) {
    NvtxRange r("gasloc_gossip_round");
    const int rc = check_started(c);
    if (rc) return rc;
    return enqueue_gossip(c, c->stream);
}

int gasloc_fused_round(gasloc_ctx *c, int32_t H) {
    NvtxRange r("gasloc_fused_round");
    int rc = check_started(c);
    if (rc) return rc;
    rc = check_H(c, H);
    if (rc) return rc;
    return enqueue_round(c, H, c->stream);
}

int gasloc_run(gasloc_ctx *c, int32_t rounds, int32_t H, double *ce_trace_host) {
    NvtxRange range("gasloc_run");
    int rc = check_started(c);
    if (rc) return rc;
    rc = check_H(c, H);
    if (rc) return rc;
    if (rounds < 0) return fail(GASLOC_EINVAL, "rounds must be >= 0");
    if (ce_trace_host && rounds > kCeRing) return fail(GASLOC_EINVAL, "a trace holds at most %d rounds", kCeRing);
    if (c->fresh_mask != 0) return fail(GASLOC_ESTATE, "gasloc_run starts at a round boundary (after a gossip round)");
    if (rounds == 0) return GASLOC_OK;
    const int64_t r0 = c->round;
    if (!c->graph || c->graph_gen != c->gen || c->graph_H != H) {
        rc = capture_rounds(c, H, 1, &c->graph, &c->graph_launches);
        if (rc) return rc;
        c->graph_gen = c->gen;
        c->graph_H = H;
    }
    if (rounds >= kGraphBlock && (!c->graph_blk || c->graph_blk_gen != c->gen || c->graph_blk_H != H)) {
        rc = capture_rounds(c, H, kGraphBlock, &c->graph_blk, &c->graph_blk_launches);
        if (rc) return rc;
        c->graph_blk_gen = c->gen;
        c->graph_blk_H = H;
    }
    // blocks of kGraphBlock rounds while that many are left, then single rounds
    for (int32_t r = 0; r < rounds;) {
        const bool blk = rounds - r >= kGraphBlock;
        const cudaError_t e = cudaGraphLaunch(blk ? c->graph_blk : c->graph, c->stream);
        if (e != cudaSuccess) return cuda_fail(e, "graph launch");
        const int32_t nr = blk ? kGraphBlock : 1;
        for (int32_t i = 0; i < c->n; ++i) c->nsteps[i] += static_cast<int64_t>(nr) * (H < 0 ? c->Hi[i] : H);
        c->round += nr;
        c->launches += blk ? c->graph_blk_launches : c->graph_launches;
        r += nr;
    }
    c->ce_valid = true;
    if (ce_trace_host) {
        for (int32_t r = 0; r < rounds; ++r) {
            const cudaError_t e = cudaMemcpyAsync(ce_trace_host + r, c->ce_ring + (r0 + r) % kCeRing, sizeof(double),
                                                  cudaMemcpyDeviceToHost, c->stream);
            if (e != cudaSuccess) return cuda_fail(e, "reading the consensus-error trace");
        }
        return sync_and_check(c);
    }
    return GASLOC_OK;
}

int gasloc_consensus_error(gasloc_ctx *c, double *out) {
    NvtxRange r("gasloc_consensus_error");
    int rc = check_started(c);
    if (rc) return rc;
    if (!out) return fail(GASLOC_EINVAL, "out is NULL");
    const double *src = c->ce_d;
    if (!c->ce_valid || c->round == 0) {
        CeArgs a{c->tens_d, c->tiles_a, c->ntiles_a, c->n, c->hp.storage, c->partials, c->ticket, c->ce_d, c->err_d};
        rc = launch_checked(c, launch_ce(a, c->grid_ce, 256, c->stream), "consensus-error kernel");
        if (rc) return rc;
    } else {
        src = c->ce_ring + (c->round - 1) % kCeRing;
    }
    cudaError_t e = cudaMemcpyAsync(pin_ce(c), src, sizeof(double), cudaMemcpyDeviceToHost, c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "reading the consensus error");
    rc = sync_and_check(c);
    if (rc) return rc;
    *out = *pin_ce(c);
    return GASLOC_OK;
}

int gasloc_consensus_error_async(gasloc_ctx *c, double *host_dst) {
    NvtxRange r("gasloc_consensus_error_async");
    int rc = check_started(c);
    if (rc) return rc;
    if (!host_dst) return fail(GASLOC_EINVAL, "dst is NULL");
    const double *src = c->ce_d;
    if (!c->ce_valid || c->round == 0) {
        CeArgs a{c->tens_d, c->tiles_a, c->ntiles_a, c->n, c->hp.storage, c->partials, c->ticket, c->ce_d, c->err_d};
        rc = launch_checked(c, launch_ce(a, c->grid_ce, 256, c->stream), "consensus-error kernel");
        if (rc) return rc;
    } else {
        src = c->ce_ring + (c->round - 1) % kCeRing;
    }
    // host or device memory: the copy's direction follows from the address
    cudaError_t e = cudaMemcpyAsync(host_dst, src, sizeof(double), cudaMemcpyDefault, c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "copying the consensus error");
    return GASLOC_OK;
}

int gasloc_synchronize(gasloc_ctx *c) {
    int rc = check_started(c);
    if (rc) return rc;
    return sync_and_check(c);
}

int gasloc_consensus_error_now(gasloc_ctx *c, double *out) {
    int rc = check_started(c);
    if (rc) return rc;
    c->ce_valid = false;
    return gasloc_consensus_error(c, out);
}

int gasloc_get_topology(gasloc_ctx *c, int64_t round, int32_t *nbr, float *w, int32_t *deg) {
    int rc = check_started(c);
    if (rc) return rc;
    if (!nbr || !w || !deg) return fail(GASLOC_EINVAL, "NULL output");
    if (round < 0) return fail(GASLOC_EINVAL, "round must be >= 0");
    rc = build_topology(c, round, nullptr, c->topo_scratch, c->stream);
    if (rc) return rc;
    cudaError_t e = cudaMemcpyAsync(pin_topo(c), c->topo_scratch, sizeof(Topo), cudaMemcpyDeviceToHost, c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "reading the topology");
    rc = sync_and_check(c);
    if (rc) return rc;
    const Topo *t = pin_topo(c);
    const int32_t n = c->n;
    for (int32_t i = 0; i < n; ++i) {
        deg[i] = t->deg[i];
        for (int32_t q = 0; q < n; ++q) {
            nbr[i * n + q] = q <= t->deg[i] ? t->nbr[i][q] : -1;
            w[i * n + q] = q <= t->deg[i] ? t->w[i][q] : 0.0f;
        }
    }
    return GASLOC_OK;
}

int gasloc_average(gasloc_ctx *c, float *dst) {
    int rc = check_started(c);
    if (rc) return rc;
    if (!dst) return fail(GASLOC_EINVAL, "dst is NULL");
    return launch_checked(c, launch_average(c->tens_d, c->tiles_a, c->ntiles_a, c->n, c->hp.storage, dst, c->P,
                                            c->err_d, c->sms * 8, c->stream),
                          "average kernel");
}

int gasloc_average_host(gasloc_ctx *c, float *dst) {
    int rc = check_started(c);
    if (rc) return rc;
    if (!dst) return fail(GASLOC_EINVAL, "dst is NULL");
    rc = gasloc_average(c, c->avg_d);
    if (!rc) {
        cudaError_t e = cudaMemcpyAsync(dst, c->avg_d, static_cast<size_t>(c->P) * 4, cudaMemcpyDeviceToHost, c->stream);
        if (e != cudaSuccess) rc = cuda_fail(e, "copying the average");
        else rc = sync_and_check(c);
    }
    cudaStreamSynchronize(c->stream);
    return rc;
}

int gasloc_buffer(gasloc_ctx *c, int32_t which, int32_t tensor, void **dptr, int64_t *worker_stride) {
    int rc = check_started(c);
    if (rc) return rc;
    if (!dptr) return fail(GASLOC_EINVAL, "dptr is NULL");
    if (tensor < 0 || tensor >= static_cast<int32_t>(c->tens_h.size())) return fail(GASLOC_EINVAL, "tensor out of range");
    int64_t stride = 0;
    char *p = buffer_base(c->tens_h[tensor], which, &stride);
    if (!p) return fail(GASLOC_EINVAL, "unknown buffer %d", which);
    *dptr = p;
    if (worker_stride) *worker_stride = stride;
    return GASLOC_OK;
}

int gasloc_read(gasloc_ctx *c, int32_t which, int32_t worker, float *host) {
    int rc = check_started(c);
    if (rc) return rc;
    if (!host) return fail(GASLOC_EINVAL, "host buffer is NULL");
    rc = check_which_worker(c, which, worker, false);
    if (rc) return rc;
    const size_t es = esize_of(c);
    if (es == 4) {
        for (const TensorDesc &d : c->tens_h) {
            int64_t stride = 0;
            const char *p = buffer_base(d, which, &stride) + static_cast<size_t>(worker * stride) * es;
            cudaError_t e = cudaMemcpyAsync(host + d.loff, p, static_cast<size_t>(d.numel) * 4,
                                            cudaMemcpyDeviceToHost, c->stream);
            if (e != cudaSuccess) return cuda_fail(e, "device-to-host copy");
        }
        return sync_and_check(c);
    }
    // bf16 store: widen on the device into an fp32 staging buffer, copy that
    StagingBuffer st(c);
    if (!st.p) return fail(GASLOC_ENOMEM, "device allocation failed (staging)");
    for (const TensorDesc &d : c->tens_h) {
        int64_t stride = 0;
        const char *p = buffer_base(d, which, &stride) + static_cast<size_t>(worker * stride) * es;
        for (int64_t k0 = 0; k0 < d.numel; k0 += st.elems) {
            const int64_t len = d.numel - k0 < st.elems ? d.numel - k0 : st.elems;
            rc = launch_checked(c, launch_convert(p + static_cast<size_t>(k0) * es, st.p, len, false, c->stream),
                                "widen kernel");
            if (rc) return rc;
            cudaError_t e = cudaMemcpyAsync(host + d.loff + k0, st.p, static_cast<size_t>(len) * 4,
                                            cudaMemcpyDeviceToHost, c->stream);
            if (e != cudaSuccess) return cuda_fail(e, "device-to-host copy");
        }
    }
    return sync_and_check(c);
}

int gasloc_write(gasloc_ctx *c, int32_t which, int32_t worker, const float *host) {
    int rc = check_started(c);
    if (rc) return rc;
    if (!host) return fail(GASLOC_EINVAL, "host buffer is NULL");
    rc = check_which_worker(c, which, worker, true);
    if (rc) return rc;
    const int32_t rows = (which == GASLOC_BUF_H && !c->hp.per_worker_h) ? 1 : c->n;
    const int32_t w0 = worker < 0 ? 0 : worker, w1 = worker < 0 ? rows : worker + 1;
    const size_t es = esize_of(c);
    // bf16 store: copy fp32 into a staging buffer, narrow it on the device
    StagingBuffer st(c, es == 2);
    if (es == 2 && !st.p) return fail(GASLOC_ENOMEM, "device allocation failed (staging)");
    for (const TensorDesc &d : c->tens_h) {
        int64_t stride = 0;
        char *p = buffer_base(d, which, &stride);
        const size_t bytes = static_cast<size_t>(d.numel) * es;
        char *row0 = p + static_cast<size_t>(w0 * stride) * es;
        cudaError_t e = cudaSuccess;
        if (es == 4) {
            e = cudaMemcpyAsync(row0, host + d.loff, bytes, cudaMemcpyHostToDevice, c->stream);
            if (e != cudaSuccess) return cuda_fail(e, "host-to-device copy");
        } else {
            for (int64_t k0 = 0; k0 < d.numel; k0 += st.elems) {
                const int64_t len = d.numel - k0 < st.elems ? d.numel - k0 : st.elems;
                e = cudaMemcpyAsync(st.p, host + d.loff + k0, static_cast<size_t>(len) * 4, cudaMemcpyHostToDevice,
                                    c->stream);
                if (e != cudaSuccess) return cuda_fail(e, "host-to-device copy");
                rc = launch_checked(c, launch_convert(st.p, row0 + static_cast<size_t>(k0) * es, len, true, c->stream),
                                    "narrow kernel");
                if (rc) return rc;
            }
        }
        for (int32_t i = w0 + 1; i < w1; ++i) {
            e = cudaMemcpyAsync(p + static_cast<size_t>(i * stride) * es, row0, bytes, cudaMemcpyDeviceToDevice,
                                c->stream);
            if (e != cudaSuccess) return cuda_fail(e, "device-to-device copy");
        }
    }
    if (which == GASLOC_BUF_X) c->ce_valid = false;
    return sync_and_check(c);
}

int gasloc_gather(gasloc_ctx *c, int32_t which, int32_t worker, int64_t n, const int64_t *idx, float *out) {
    int rc = check_started(c);
    if (rc) return rc;
    if (n < 0 || (n > 0 && (!idx || !out))) return fail(GASLOC_EINVAL, "bad gather arguments");
    rc = check_which_worker(c, which, worker, false);
    if (rc) return rc;
    for (int64_t q = 0; q < n; ++q)
        if (idx[q] < 0 || idx[q] >= c->P) return fail(GASLOC_EINVAL, "index %lld out of range", (long long)idx[q]);
    if (n == 0) return GASLOC_OK;
    int64_t *di = static_cast<int64_t *>(c->dalloc(static_cast<size_t>(n) * 8));
    float *dout = static_cast<float *>(c->dalloc(static_cast<size_t>(n) * 4));
    if (!di || !dout) {
        c->dfree(di);
        c->dfree(dout);
        return fail(GASLOC_ENOMEM, "device allocation failed (gather)");
    }
    cudaError_t e = cudaMemcpyAsync(di, idx, static_cast<size_t>(n) * 8, cudaMemcpyHostToDevice, c->stream);
    if (e == cudaSuccess) {
        rc = launch_checked(c, launch_gather(c->tens_d, static_cast<int32_t>(c->tens_h.size()), c->hp.storage, which,
                                             worker, di, n,
                                             dout, c->err_d, c->stream),
                            "gather kernel");
        if (!rc) {
            e = cudaMemcpyAsync(out, dout, static_cast<size_t>(n) * 4, cudaMemcpyDeviceToHost, c->stream);
            rc = e == cudaSuccess ? sync_and_check(c) : cuda_fail(e, "gather copy");
        }
    } else {
        rc = cuda_fail(e, "gather index upload");
    }
    cudaStreamSynchronize(c->stream);
    c->dfree(di);
    c->dfree(dout);
    return rc;
}

int gasloc_round(const gasloc_ctx *c, int64_t *round) {
    if (!c || !round) return fail(GASLOC_EINVAL, "NULL argument");
    *round = c->round;
    return GASLOC_OK;
}

int gasloc_steps_taken(const gasloc_ctx *c, int32_t worker, int64_t *steps) {
    if (!c || !steps) return fail(GASLOC_EINVAL, "NULL argument");
    if (worker < 0 || worker >= c->n) return fail(GASLOC_EINVAL, "worker out of range");
    *steps = c->nsteps[worker];
    return GASLOC_OK;
}

int gasloc_checked_build(void) { return checked_build(); }

int gasloc_selftest_index_check(gasloc_ctx *c) {
    int rc = check_started(c);
    if (rc) return rc;
    rc = launch_checked(c, launch_check_selftest(c->err_d, c->stream), "index-check self-test kernel");
    if (rc) return rc;
    return sync_and_check(c);
}

int gasloc_selftest_bounded_wait(gasloc_ctx *c, int64_t limit_ns) {
    int rc = check_started(c);
    if (rc) return rc;
    if (limit_ns < 1 || limit_ns > 2000000000LL) return fail(GASLOC_EINVAL, "limit_ns must be in [1, 2e9]");
    rc = launch_checked(c, launch_wait_selftest(static_cast<uint64_t>(limit_ns), c->err_d, c->stream),
                        "bounded-wait self-test kernel");
    if (rc) return rc;
    return sync_and_check(c);
}

int gasloc_launch_count(const gasloc_ctx *c, int64_t *count) {
    if (!c || !count) return fail(GASLOC_EINVAL, "NULL argument");
    *count = c->launches;
    return GASLOC_OK;
}

// Checkpoint file: header, counters, then every buffer's valid elements
// (tensor-major, then buffer, then worker).
namespace {
struct CkptHeader {
    char magic[8];
    int32_t version, n;
    int64_t P, n_tensors;
    uint64_t seed;
    int32_t kind, rows, cols, per_worker_h;
    int64_t round;
    uint32_t fresh_mask;
    int32_t has_Hi;
    int32_t storage;
    int32_t pad;
    int64_t p_begin, p_end;   // the range of the problem's parameters the checkpoint holds
};
}  // namespace

int gasloc_save(gasloc_ctx *c, const char *path) {
    int rc = check_started(c);
    if (rc) return rc;
    if (!path) return fail(GASLOC_EINVAL, "path is NULL");
    rc = sync_and_check(c);
    if (rc) return rc;
    FILE *f = std::fopen(path, "wb");
    if (!f) return fail(GASLOC_EIO, "cannot open '%s' for writing", path);
    CkptHeader h{};
    std::memcpy(h.magic, "GASLOCK4", 8);
    h.version = 4;
    h.n = c->n;
    h.P = c->P_global;
    h.p_begin = c->p_begin;
    h.p_end = c->p_end;
    h.n_tensors = static_cast<int64_t>(c->numels.size());
    h.seed = c->seed;
    h.kind = c->spec.kind;
    h.rows = c->spec.rows;
    h.cols = c->spec.cols;
    h.per_worker_h = c->hp.per_worker_h;
    h.round = c->round;
    h.fresh_mask = c->fresh_mask;
    h.has_Hi = c->has_Hi ? 1 : 0;
    h.storage = c->hp.storage;
    bool ok = std::fwrite(&h, sizeof h, 1, f) == 1;
    ok = ok && std::fwrite(c->numels.data(), 8, c->numels.size(), f) == c->numels.size();
    ok = ok && std::fwrite(&c->hp, sizeof c->hp, 1, f) == 1;
    ok = ok && std::fwrite(c->nsteps.data(), 8, c->n, f) == static_cast<size_t>(c->n);
    ok = ok && std::fwrite(c->Hi.data(), 4, c->n, f) == static_cast<size_t>(c->n);
    const size_t es = esize_of(c);
    std::vector<char> buf;
    for (const TensorDesc &d : c->tens_h) {
        buf.resize(static_cast<size_t>(d.numel) * es);
        for (int which = GASLOC_BUF_X; ok && which <= GASLOC_BUF_H; ++which) {
            const int32_t rows = (which == GASLOC_BUF_H && !c->hp.per_worker_h) ? 1 : c->n;
            int64_t stride = 0;
            const char *p = buffer_base(d, which, &stride);
            for (int32_t i = 0; ok && i < rows; ++i) {
                if (cudaMemcpy(buf.data(), p + static_cast<size_t>(i * stride) * es, buf.size(),
                               cudaMemcpyDeviceToHost) != cudaSuccess) {
                    std::fclose(f);
                    return fail(GASLOC_ECUDA, "checkpoint copy failed");
                }
                ok = std::fwrite(buf.data(), 1, buf.size(), f) == buf.size();
            }
        }
    }
    ok = (std::fclose(f) == 0) && ok;
    if (!ok) return fail(GASLOC_EIO, "short write to '%s'", path);
    return GASLOC_OK;
}

int gasloc_load(gasloc_ctx *c, const char *path) {
    int rc = check_started(c);
    if (rc) return rc;
    if (!path) return fail(GASLOC_EINVAL, "path is NULL");
    FILE *f = std::fopen(path, "rb");
    if (!f) return fail(GASLOC_EIO, "cannot open '%s'", path);
    CkptHeader h{};
    bool ok = std::fread(&h, sizeof h, 1, f) == 1 && std::memcmp(h.magic, "GASLOCK4", 8) == 0 && h.version == 4;
    if (!ok) { std::fclose(f); return fail(GASLOC_EIO, "'%s' is not a checkpoint", path); }
    if (h.n != c->n || h.P != c->P_global || h.p_begin != c->p_begin || h.p_end != c->p_end ||
        h.n_tensors != static_cast<int64_t>(c->numels.size()) || h.seed != c->seed ||
        h.kind != c->spec.kind || h.rows != c->spec.rows || h.cols != c->spec.cols ||
        h.per_worker_h != c->hp.per_worker_h || h.storage != c->hp.storage) {
        std::fclose(f);
        return fail(GASLOC_EINVAL, "checkpoint does not match this context");
    }
    std::vector<int64_t> numels(static_cast<size_t>(h.n_tensors));
    gasloc_hparams hp{};
    std::vector<int64_t> nsteps(c->n);
    std::vector<int32_t> Hi(c->n);
    ok = std::fread(numels.data(), 8, numels.size(), f) == numels.size() && numels == c->numels &&
         std::fread(&hp, sizeof hp, 1, f) == 1 &&
         std::fread(nsteps.data(), 8, nsteps.size(), f) == nsteps.size() &&
         std::fread(Hi.data(), 4, Hi.size(), f) == Hi.size();
    if (!ok) { std::fclose(f); return fail(GASLOC_EIO, "truncated checkpoint header"); }
    rc = sync_and_check(c);
    if (rc) { std::fclose(f); return rc; }
    const size_t es = esize_of(c);
    std::vector<char> buf;
    for (const TensorDesc &d : c->tens_h) {
        buf.resize(static_cast<size_t>(d.numel) * es);
        for (int which = GASLOC_BUF_X; ok && which <= GASLOC_BUF_H; ++which) {
            const int32_t rows = (which == GASLOC_BUF_H && !c->hp.per_worker_h) ? 1 : c->n;
            int64_t stride = 0;
            char *p = buffer_base(d, which, &stride);
            for (int32_t i = 0; ok && i < rows; ++i) {
                ok = std::fread(buf.data(), 1, buf.size(), f) == buf.size();
                if (ok && cudaMemcpy(p + static_cast<size_t>(i * stride) * es, buf.data(), buf.size(),
                                     cudaMemcpyHostToDevice) != cudaSuccess) {
                    std::fclose(f);
                    return fail(GASLOC_ECUDA, "checkpoint upload failed");
                }
            }
        }
    }
    std::fclose(f);
    if (!ok) return fail(GASLOC_EIO, "truncated checkpoint data");
    rc = check_hparams(&hp);
    if (rc) return rc;
    c->hp = hp;
    c->round = h.round;
    c->fresh_mask = h.fresh_mask;
    c->has_Hi = h.has_Hi != 0;
    c->Hi = Hi;
    c->nsteps = nsteps;
    rc = upload_schedule(c);   // the checkpoint's learning-rate schedule
    if (rc) return rc;
    rc = restore_step_counters(c);
    if (rc) return rc;
    c->gen += 1;
    c->ce_valid = false;
    refresh_spec(c);
    return GASLOC_OK;
}

void gasloc_destroy(gasloc_ctx *c) {
    if (!c) return;
    c->release_all();
    delete c;
}

}  // extern "C"
