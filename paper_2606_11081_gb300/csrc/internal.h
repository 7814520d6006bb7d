// internal.h -- structures shared by the C-ABI layer (gasloc.cpp) and the
// kernel translation units.  Not part of the public ABI.
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace gasloc {

constexpr int kMaxWorkers = 32;

// Element type of the replica store.
enum Storage : int32_t { kStoreF32 = 0, kStoreBF16 = 1 };

// One parameter tensor of the replica store.  Every array is one allocation
// of shape [n_workers][wstride] elements (fp32 or bf16; h: [1 or n][wstride]);
// wstride = numel rounded up to 64 elements so each worker slice is 128- or
// 256-byte aligned.  Padding is zero-filled at start and never written
// afterwards.  Kernels cast the pointers to their element type.
struct TensorDesc {
    void *x, *y, *m, *v, *b, *c, *h;
    int64_t numel;     // valid elements per worker
    int64_t wstride;   // floats between consecutive workers
    int64_t hstride;   // floats between workers in h (0 when shared)
    int64_t goff;      // global index of element 0 (concatenation order): keys the generators
    int64_t loff;      // index of element 0 in the context's own elements (goff minus the
                       // first global index the context holds): places host and output arrays
};

// A contiguous run of at most `tile` elements of one tensor.  start is a
// multiple of 4, so every tile begins on a 16-byte boundary.
struct Tile {
    int32_t tensor;
    int32_t len;
    int64_t start;
};

// Round-t neighbour table (row i: N_i ascending, deg[i] + 1 entries).
struct Topo {
    int32_t nbr[kMaxWorkers][kMaxWorkers];
    float w[kMaxWorkers][kMaxWorkers];
    int32_t deg[kMaxWorkers];
};

enum TopoKind : int32_t { kNone = 0, kRing = 1, kComplete = 2, kExp = 3, kTorus = 4,
                          kMatching = 5, kTwoPeer = 6 };

struct TopoSpec {
    int32_t kind, n, rows, cols, weights;
    int32_t pad;
    uint64_t seed;
    uint64_t edge_thr;   // edge kept iff hi32(hash) < edge_thr (2^32 = always)
};

// Device error codes (first one wins, written with atomicCAS).
enum DevError : int32_t { kDevOk = 0, kDevWaitTimeout = 1, kDevBadIndex = 2 };

// ---------------------------------------------------------------- kernels --

struct InitArgs {
    const TensorDesc *tens;
    const Tile *tiles;
    int64_t ntiles;
    int32_t n_workers;
    int32_t per_worker_h;
    uint64_t seed;
    int32_t storage;
    int32_t *err;          // device error word (checked build)
};

// Step counters of the replicas, resident on the device so that a round can
// be replayed from a CUDA graph: every per-step scalar is derived from here.
struct DevState {
    int64_t round;                    // completed gossip rounds
    int64_t nsteps[kMaxWorkers];      // local steps taken by each worker
    double p1[kMaxWorkers];           // beta1^n (n successive products from 1)
    double p2[kMaxWorkers];           // beta2^n
};

// Per-worker scalars of each worker's next local step (written by the prep
// kernel after a start, a hyperparameter change or a checkpoint load, and by
// every AdamW launch for the workers it stepped).
struct StepTable {
    float step[kMaxWorkers];          // fl32(lr_n / (1 - beta1^n)), lr_n the step's scheduled rate
    float isb[kMaxWorkers];           // fl32(1 / sqrt(1 - beta2^n))
    uint32_t key_lo[kMaxWorkers];     // noise key hash(seed, 4, i, n)
    uint32_t key_hi[kMaxWorkers];
    float decay[kMaxWorkers];         // fl32(1 - lr_n * weight_decay)
};

struct PrepArgs {
    const DevState *state;
    StepTable *table;
    int32_t n_workers;
    double beta1, beta2, wd;
    const double *lr_sched;               // lr of local steps 1..lr_steps
    int64_t lr_steps;
    double lr_after;                      // lr of later steps
    uint64_t seed;
};

struct AdamwArgs {
    const TensorDesc *tens;
    const Tile *tiles;
    int64_t ntiles;
    StepTable *table;                     // this step's scalars; the next step's on return
    DevState *state;                      // step counters, advanced for the active workers
    unsigned int *ticket;                 // CTAs that copied the table (returns to 0)
    uint32_t active_mask;                 // bit i: worker i takes this step
    double beta1d, beta2d, wd;            // for the next step's scalars
    const double *lr_sched;               // lr of local steps 1..lr_steps
    int64_t lr_steps;
    double lr_after;                      // lr of later steps
    uint64_t seed;
    int32_t n_active;
    int32_t per_worker_h;
    int32_t storage;
    uint32_t from_x_mask;                 // bit i: worker i starts from x
    int32_t worker[kMaxWorkers];
    float decay;                          // fl32(1 - lr * weight_decay) without a schedule
    float beta1, beta2, omb1, omb2, eps, sigma;
    int32_t n_workers;                    // rows of every per-worker array
    int32_t staged;                       // fp32: the staged kernel (small replica stores)
    unsigned long long *work;             // staged kernels: [0] units claimed, [1] producers done (return to 0)
    int32_t *err;                         // device error word (checked build)
};

struct GossipArgs {
    const TensorDesc *tens;
    const Tile *tiles;
    int64_t ntiles;
    const Topo *topo;
    const void *maps;      // per tensor: 2-D tensor maps of x, y, b (128 bytes each)
    int32_t storage;
    int32_t n_workers;
    int32_t mode;          // GASLOC_OUTER_*
    uint32_t fresh_mask;   // bit j: worker j took a local step this round
    DevState *state;       // round counter: t = 0 check, CE slot, advanced by the last CTA
    int32_t tile;          // elements per tile (4 x 256 / groups)
    int32_t groups;        // consumer threads per 16-byte column
    int32_t stages;
    int32_t dense;         // dense mixing variant (GossipShape::dense)
    int32_t direct;        // the direct variant (few workers, small replicas): tiles is the
                           // 1024-element tile table
    float eta_out, mu, eta, alpha, oma, gamma;
    double *partials;      // [gridDim] per-CTA consensus-error partials
    unsigned int *ticket;  // last-CTA-done counter (returns to 0)
    double *ce_ring;       // consensus error of round t goes to ce_ring[t % ring]
    int32_t ce_ring_len;
    int32_t *err;
};

// A round's last local step fused with its gossip round (round.cu): every
// worker takes the step; few workers, fp32 storage.
constexpr int kRoundColumn = 2;                  // elements per consumer thread of the fused round kernel
constexpr int kRoundTile = 512;                  // elements per tile of the fused round kernel
struct RoundArgs {
    const TensorDesc *tens;
    const Tile *tiles;                    // tiles of kRoundTile elements
    int64_t ntiles;
    StepTable *table;                     // this step's scalars; the next step's on return
    DevState *state;                      // step counters and round, advanced by the last CTA
    const Topo *topo;
    double beta1d, beta2d, wd;            // for the next step's scalars
    const double *lr_sched;               // lr of local steps 1..lr_steps
    int64_t lr_steps;
    double lr_after;                      // lr of later steps
    uint64_t seed;
    int32_t n_workers;
    int32_t mode;                         // GASLOC_OUTER_*
    int32_t per_worker_h;
    int32_t from_x;                       // every worker's step starts from x (its first of the round)
    int32_t sched;                        // the weight-decay factor comes from the step table
    float decay;                          // fl32(1 - lr * weight_decay) without a schedule
    float beta1, beta2, omb1, omb2, eps, sigma;
    float eta_out, mu, eta, alpha, oma, gamma;
    double *partials;                     // [gridDim] per-CTA consensus-error partials
    unsigned int *ticket;                 // last-CTA-done counter (returns to 0)
    unsigned int *step_ticket;            // CTAs that read the step's scalars (returns to 0)
    double *ce_ring;                      // consensus error of round t goes to ce_ring[t % ring]
    int32_t ce_ring_len;
    int32_t *err;                         // device error word (checked build)
};

struct CeArgs {
    const TensorDesc *tens;
    const Tile *tiles;
    int64_t ntiles;
    int32_t n_workers;
    int32_t storage;
    double *partials;
    unsigned int *ticket;
    double *ce_out;
    int32_t *err;          // device error word (checked build)
};

// Launchers (return cudaGetLastError()).
cudaError_t launch_init(const InitArgs &a, int grid, cudaStream_t s);
// round_ptr != nullptr: the round is read from device memory (graph replay).
cudaError_t launch_topo(const TopoSpec &spec, int64_t round, const int64_t *round_ptr, Topo *out,
                        cudaStream_t s);
cudaError_t launch_prep(const PrepArgs &a, cudaStream_t s);
cudaError_t launch_adamw(const AdamwArgs &a, int grid, int block, cudaStream_t s);
cudaError_t launch_gossip(const GossipArgs &a, int grid, size_t smem, cudaStream_t s);

// Launch shape of the gossip kernel for n workers and an outer mode.
struct GossipShape {
    int groups, tile, block, stages;
    int dense;   // one thread per column mixing with a dense weight row (n <= 8, not Eq. 2)
    size_t smem;
};
GossipShape gossip_shape(int n, int mode, int storage);
cudaError_t launch_ce(const CeArgs &a, int grid, int block, cudaStream_t s);
// The fused round kernel: whether it serves n workers with this storage, its
// CTAs per SM, and its launch.
bool round_fits(int n, int storage);
int round_blocks_per_sm(int mode, bool per_worker_h);
cudaError_t launch_round(const RoundArgs &a, int grid, cudaStream_t s);
cudaError_t launch_average(const TensorDesc *tens, const Tile *tiles, int64_t ntiles,
                           int32_t n_workers, int32_t storage, float *dst, int64_t n_params, int32_t *err,
                           int grid, cudaStream_t s);
// 1 if this library was built with the index checks, else 0; the self-test
// evaluates one failing row check (no memory access) on the device.
int checked_build();
cudaError_t launch_check_selftest(int32_t *err, cudaStream_t s);
cudaError_t launch_gather(const TensorDesc *tens, int32_t ntens, int32_t storage, int32_t which,
                          int32_t worker, const int64_t *idx, int64_t n, float *out, int32_t *err,
                          cudaStream_t s);

// fp32 -> bf16 (narrow, nearest even) or bf16 -> fp32 (widen) of n elements.
cudaError_t launch_convert(const void *src, void *dst, int64_t n, bool narrow, cudaStream_t s);
cudaError_t launch_wait_selftest(uint64_t limit_ns, int32_t *err, cudaStream_t s);

// Occupancy-derived persistent grid sizes.
int adamw_blocks_per_sm(int block, bool per_worker_h, int storage);
// CTAs per SM of the staged AdamW with fp32 storage (used for small stores).
int adamw_staged_fp32_blocks_per_sm(bool per_worker_h);
int gossip_blocks_per_sm(int mode, int storage, const GossipShape &shape);
// The direct gossip variant: whether it serves n workers with this storage,
// and its CTAs per SM.
bool gossip_direct_fits(int n, int storage);
int gossip_direct_blocks_per_sm(int mode);
int ce_blocks_per_sm(int block, int storage);
cudaError_t gossip_set_smem(size_t smem);

// Sets the thread-local message returned by gasloc_last_error().
void set_last_error(const char *msg);

// Host-side copy of the counter-based hash (same definition as the device).
uint64_t host_hash(uint64_t seed, uint64_t tag, uint64_t a, uint64_t b);

}  // namespace gasloc
