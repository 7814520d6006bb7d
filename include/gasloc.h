/*
 * gasloc.h -- C ABI of libgasloc, the GB300 (sm_103a) replica-update path of
 * GASLoC ("Unifying Local Communications and Local Updates for LLM
 * Pretraining", arXiv 2606.11081).
 *
 * The library simulates n workers whose fp32 replicas live together in one
 * GPU's memory as a structure of arrays and runs, per outer round t, the steps
 * of Algorithm 1:
 *   1. H_i inner AdamW steps per worker, x_i -> y_i (App. B optimisation
 *      settings), on the synthetic diagonal quadratic
 *      f_i(x) = 1/2 sum_k h_k (x_k - c_ik)^2 with gradient noise;
 *   2. one gossip round: each worker mixes the y_j of its round-t neighbourhood
 *      N_i (always containing i) with row-stochastic weights w_ij and applies
 *      the outer optimizer (Nesterov by default, App. B; SGDM, SGD; the
 *      accelerated-gossip update of Eq. 2; DAdam and Local-DAdam of App. C);
 *   3. the consensus error (1/n) sum_i ||x_i - xbar||^2 of the new replicas.
 *
 * Conventions (all entry points):
 *  - Every call returns a gasloc_status; on failure gasloc_last_error()
 *    returns a message (thread-local, valid until the next call on the thread).
 *  - Device memory is owned by the context.  It is obtained from the allocator
 *    registered with gasloc_set_allocator() (e.g. a framework's caching
 *    allocator) or, if none is registered, from cudaMalloc, and released by
 *    gasloc_destroy().
 *  - Work is enqueued asynchronously on the context's stream (default: the
 *    CUDA legacy default stream; see gasloc_set_stream).  Calls documented as
 *    "synchronising" wait for that stream before returning.
 *  - Parameters are fp32 on the device (bf16 with GASLOC_STORAGE_BF16, fp32
 *    arithmetic); the scalars of a step (bias corrections etc.) are computed
 *    in double from device-resident step counters and rounded once.
 *  - A context is not thread-safe.  Distinct contexts are independent.
 */
#ifndef GASLOC_H
#define GASLOC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct gasloc_ctx gasloc_ctx;

typedef enum {
    GASLOC_OK = 0,
    GASLOC_EINVAL = -1,   /* an argument is out of range or inconsistent   */
    GASLOC_ENOMEM = -2,   /* an allocation failed or a size limit was hit  */
    GASLOC_ECUDA = -3,    /* a CUDA runtime call or a launch failed        */
    GASLOC_ESTATE = -4,   /* call not valid in the context's current state */
    GASLOC_EDEVICE = -5,  /* a kernel set the device error flag            */
    GASLOC_EIO = -6       /* checkpoint file could not be read or written  */
} gasloc_status;

/* Outer update applied after mixing (Algorithm 1 "Optimizer^out"; Eq. 2; App. C). */
enum {
    GASLOC_OUTER_SGD = 0,          /* x -= eta_out * D                       */
    GASLOC_OUTER_SGDM = 1,         /* b = mu b + D; x -= eta_out * b          */
    GASLOC_OUTER_NESTEROV = 2,     /* b = mu b + D; x -= eta_out (D + mu b)   */
    GASLOC_OUTER_EQ2 = 3,          /* Eq. 2 on z = x + eta (y - x)            */
    GASLOC_OUTER_DADAM = 4,        /* x = sum_j w_ij x_j + (y - x)            */
    GASLOC_OUTER_LOCAL_DADAM = 5   /* Nesterov step of D = x - sum w x_j at y */
};

/* Mixing-weight rule applied to the round's graph. */
enum {
    GASLOC_W_UNIFORM = 0,          /* w_ij = 1/|N_i|  (Algorithm 1)           */
    GASLOC_W_METROPOLIS = 1,       /* w_ij = 1/(1+max(d_i,d_j)), w_ii = rest  */
    GASLOC_W_LAZY = 2              /* w_ii = 1/2, w_ij = 1/(2 d_i): W = I -
                                      Lambda^(k) of the k-Peer schemes        */
};

/* Buffers of the replica store (gasloc_buffer / gasloc_read / gasloc_write). */
enum {
    GASLOC_BUF_X = 0,   /* outer (anchor) parameters x_i                      */
    GASLOC_BUF_Y = 1,   /* inner iterate y_i                                  */
    GASLOC_BUF_M = 2,   /* AdamW first moment                                 */
    GASLOC_BUF_V = 3,   /* AdamW second moment                                */
    GASLOC_BUF_B = 4,   /* outer momentum (z_{t-1} in Eq. 2 mode)             */
    GASLOC_BUF_C = 5,   /* quadratic centre c_i                               */
    GASLOC_BUF_H = 6    /* curvature h (per worker if per_worker_h)           */
};

#define GASLOC_MAX_WORKERS 32
#define GASLOC_PER_WORKER_STEPS (-1)

typedef struct gasloc_hparams {
    /* inner AdamW (App. B): lr, (beta1, beta2), eps, weight decay */
    double lr, beta1, beta2, eps, weight_decay;
    /* sigma of the gradient noise sigma * xi, xi uniform with unit variance */
    double noise_sigma;
    /* outer optimizer: eta_out and mu (Nesterov/SGDM/Local-DAdam) */
    double outer_lr, outer_momentum;
    /* Eq. 1/2: eta (outer step on g = y - x), alpha (mixing), gamma (momentum) */
    double eta, alpha, gamma;
    /* probability that an edge of the base graph is active in a round */
    double edge_prob;
    int32_t outer_mode;     /* GASLOC_OUTER_* */
    int32_t weights;        /* GASLOC_W_*     */
    int32_t per_worker_h;   /* 1: one curvature vector per worker */
    int32_t storage;        /* GASLOC_STORAGE_F32 or GASLOC_STORAGE_BF16 */
    /* Learning-rate schedule of the inner AdamW (App. B), applied per worker
     * to its own local step count n: over lr_total_steps = T steps, a warm-up
     * of round(lr_warmup_frac * T) = W steps rising linearly from
     * lr_warmup_start * lr (n = 1) to lr (n = W + 1), then cosine decay
     *   lr * (f + (1 - f) (1 + cos(pi q)) / 2),  q = (n - W - 1) / (T - W - 1),
     * to f * lr = lr_final_frac * lr at n = T, held after.  The decoupled
     * weight decay scales with the step's rate.  T = 0: constant lr.
     * T <= 16,777,216; the fractions in [0, 1]. */
    int64_t lr_total_steps;
    double lr_warmup_frac, lr_warmup_start, lr_final_frac;
} gasloc_hparams;

/* Element type of the replica store (every array: x, y, m, v, b, c, h).  All
 * arithmetic is fp32; with bf16 storage each stored value is rounded to
 * bfloat16 (nearest, ties to even), which halves the bytes each step moves.
 * The host-facing calls (read, write, gather, average) always take fp32
 * arrays; gasloc_buffer exposes the raw elements. */
enum { GASLOC_STORAGE_F32 = 0, GASLOC_STORAGE_BF16 = 1 };

/* Device allocator hooks: alloc returns a device pointer (NULL on failure) of
 * at least `bytes` bytes, 256-byte aligned, usable on `stream`.  A block off
 * that boundary is handed back to free (the kernels' bulk copies need aligned
 * rows) and gasloc_start fails with GASLOC_EINVAL. */
typedef void *(*gasloc_alloc_fn)(size_t bytes, void *stream, void *user);
typedef void (*gasloc_free_fn)(void *ptr, void *stream, void *user);

/* Fills *hp with the defaults: AdamW lr 3e-4, betas (0.9, 0.95), eps 1e-8,
 * weight decay 0.1 (App. B); sigma 0.01; Nesterov with eta_out 0.7, mu 0.9;
 * eta = alpha = 1, gamma = 0; edge_prob 1; uniform weights; shared h;
 * constant lr (lr_total_steps 0; warm-up fraction 0.1 from 1% of the peak and
 * a final fraction of 0 when a schedule length is set, as App. B states). */
void gasloc_default_hparams(gasloc_hparams *hp);

/* Creates a context for n_workers (1..32) replicas of n_params (>= 1) fp32
 * parameters each, communicating over `topology`:
 *   "none", "ring", "complete", "exp" (peers at +-2^q), "torus:RxC" (R*C = n),
 *   "matching" (randomized 1-Peer, Sec. 3.2), "2peer" (randomized 2-Peer).
 * `seed` keys every random draw (initial point, centres, curvature, noise,
 * permutations, edge activation, H_i).  Nothing is allocated on the device
 * until gasloc_start().  Errors: EINVAL (n_workers, n_params, topology),
 * ENOMEM. */
int gasloc_init(int32_t n_workers, int64_t n_params, const char *topology, uint64_t seed,
                gasloc_ctx **out);

/* Sets the hyperparameters (copied); the next step uses them.  Before
 * gasloc_start any field may change; afterwards per_worker_h and storage may
 * not (ESTATE).  Bias corrections use the betas current at each step (1 -
 * beta^n, App. B's AdamW), so new betas on a started context re-form the
 * device products beta^n from the step counts (this waits for the stream).
 * EINVAL if lr < 0, beta not in [0,1), eps <= 0, edge_prob not in [0,1], an
 * unknown mode or weight rule, or eta/alpha/gamma/outer_lr negative. */
int gasloc_set_hparams(gasloc_ctx *ctx, const gasloc_hparams *hp);
int gasloc_get_hparams(const gasloc_ctx *ctx, gasloc_hparams *hp);

/* Declares that the n_params of each replica form a list of n_tensors
 * parameter tensors with the given element counts (sum = n_params), stored as
 * separate device allocations of shape [n_workers, numel].  Without this call
 * the replica is one flat tensor.  Element k of the concatenation is the
 * parameter index used by every generator.  Before gasloc_start only. */
int gasloc_set_layout(gasloc_ctx *ctx, int32_t n_tensors, const int64_t *numels);

/* Restricts the context to the parameters [p_begin, p_end) of every replica
 * (0 <= p_begin < p_end <= n_params), before gasloc_start.  Every step of
 * Algorithm 1 acts on each parameter index separately -- the gradient of the
 * synthetic quadratic is diagonal and the gossip mixes the workers' values at
 * one index -- so contexts holding disjoint ranges of the same problem (same
 * n_workers, n_params, topology, seed, hyperparameters and layout) evolve
 * exactly as the corresponding parts of one context holding all of it: every
 * generator is keyed on the global index, and every context builds the same
 * neighbour tables and H_i.  This is how the replicas are split over several
 * GPUs (one range per GPU), with no data exchanged between them.  After the
 * call the context holds n = p_end - p_begin parameters per replica: the
 * host arrays of gasloc_read / gasloc_write / gasloc_gather /
 * gasloc_average[_host] and the indices of gasloc_gather count from p_begin,
 * gasloc_buffer exposes the context's pieces of the tensors (a tensor list is
 * cut at the range's ends), and gasloc_consensus_error returns the range's
 * share (1/n_workers) sum_{k in range} sum_i (x_ik - xbar_k)^2, so that the
 * shares of a partition of [0, n_params) add up to the whole consensus error.
 * EINVAL for an empty or out-of-bounds range, ESTATE after gasloc_start. */
int gasloc_set_range(gasloc_ctx *ctx, int64_t p_begin, int64_t p_end);
/* The context's range and the problem's n_params (default: [0, n_params)). */
int gasloc_get_range(const gasloc_ctx *ctx, int64_t *p_begin, int64_t *p_end, int64_t *n_params_global);

/* Registers device allocator hooks (before gasloc_start only). */
int gasloc_set_allocator(gasloc_ctx *ctx, gasloc_alloc_fn alloc, gasloc_free_fn free_fn,
                         void *user);

/* Sets the cudaStream_t all later work is enqueued on. */
int gasloc_set_stream(gasloc_ctx *ctx, void *cuda_stream);

/* Allocates the replica store and initialises it on the device: identical
 * x_i = x_0 ~ N(0, 0.02^2) on every worker (Prop. 2 assumes equal initial
 * replicas), y_i = x_i, centres c_i ~ N(0,1), curvature h ~ U(0.1, 1), and
 * m = v = b = 0.  Besides the store (x, y, m, v, b, c per worker and h) it
 * allocates the round tables and one array of n_params floats for the
 * average's way to host memory.  Asynchronous.  ENOMEM if an allocation
 * fails, EINVAL if an allocator hook returns a misaligned block. */
int gasloc_start(gasloc_ctx *ctx);

/* Per-worker local step counts H_i (Sec. 3.2, heterogeneous local steps),
 * each in [0, 1024]; host array of n_workers entries, copied. */
int gasloc_set_local_steps(gasloc_ctx *ctx, const int32_t *H_i);
/* Draws H_i = 1 + floor(u_i * hmax) from the seed (u_i uniform), hmax >= 1. */
int gasloc_draw_local_steps(gasloc_ctx *ctx, int32_t hmax);
int gasloc_get_local_steps(const gasloc_ctx *ctx, int32_t *H_i);

/* Inner loop of Algorithm 1: H > 0 gives every worker H AdamW steps (H = 0:
 * none); H = GASLOC_PER_WORKER_STEPS gives worker i its H_i steps.  The first step
 * of a round starts from x_i; later ones from y_i.  Moments and step counters
 * persist across rounds.  Asynchronous.  ESTATE before gasloc_start. */
int gasloc_local_steps(gasloc_ctx *ctx, int32_t H);

/* Outer step of Algorithm 1 for round t: builds the round-t neighbour table
 * on the device, mixes each worker's sent quantity over N_i in ascending j,
 * applies the outer update and reduces the consensus error of the new x.
 * A worker that took no local step this round sends x_i.  Asynchronous. */
int gasloc_gossip_round(gasloc_ctx *ctx);

/* One complete outer round of Algorithm 1 -- H local steps (as
 * gasloc_local_steps: H > 0, GASLOC_PER_WORKER_STEPS or 0) followed by a
 * gossip round -- with the round's last local step fused into the gossip
 * kernel where the store allows: at most 4 workers with fp32 storage, up to
 * 8192 parameters per CTA of the GPU's grid (about 2.5 M on a 152-SM GPU),
 * every worker taking that step from the same iterate (all from x or all
 * from y).  The results are those of gasloc_local_steps(ctx, H) followed by
 * gasloc_gossip_round(ctx), bit for bit (the consensus error to the rounding
 * of its fp64 sum order); elsewhere the call enqueues exactly those two.  The
 * fused kernel reads the round's last iterate once instead of writing it for
 * the gossip kernel to read back: a variant outside the one-pass-per-step
 * byte model of the separate kernels, which gasloc_run and the benchmark's
 * rounds use.  Asynchronous; EINVAL for H outside [0, 1024] and not
 * GASLOC_PER_WORKER_STEPS, ESTATE for GASLOC_PER_WORKER_STEPS without H_i. */
int gasloc_fused_round(gasloc_ctx *ctx, int32_t H);

/* Runs `rounds` complete outer rounds -- H local steps (H > 0, or
 * GASLOC_PER_WORKER_STEPS for each worker's H_i, or 0) followed by a gossip
 * round -- exactly as that many gasloc_local_steps + gasloc_gossip_round
 * calls would, but replayed from CUDA graphs: one of 8 consecutive rounds
 * while at least 8 are left, one of a single round for the rest.  Each is
 * captured when first needed and reused until the hyperparameters, H or the
 * H_i change.  Every per-step scalar is derived on the device from device-resident
 * step counters, so the replayed rounds need no host work.  Must start at a
 * round boundary (ESTATE otherwise).  If ce_trace_host is not NULL it
 * receives the consensus error of each round (rounds <= 4096) and the call
 * synchronises; otherwise it is asynchronous. */
int gasloc_run(gasloc_ctx *ctx, int32_t rounds, int32_t H, double *ce_trace_host);

/* Consensus error CE = (1/n) sum_i sum_k (x_ik - xbar_k)^2 of the current
 * replicas (||pi x||^2 / n with pi = I - 11^T/n).  Returns the value the last
 * gossip round reduced when nothing changed x since, else reduces it now.
 * Synchronising; EDEVICE if a kernel reported an error since the last check. */
int gasloc_consensus_error(gasloc_ctx *ctx, double *out);
/* Same quantity, always reduced now from the current x by the standalone
 * reduction kernel (ignores the value the last gossip round produced). */
int gasloc_consensus_error_now(gasloc_ctx *ctx, double *out);

/* The quantity gasloc_consensus_error returns, copied to dst on the
 * context's stream without waiting for it: the per-round metric of a training
 * loop can be logged without draining the GPU's queue after every round.
 * dst is caller memory, host (page-locked memory keeps the copy asynchronous)
 * or device (e.g. the operand of an all-reduce that adds the shares of
 * contexts holding disjoint ranges, see gasloc_set_range).  *dst holds the
 * value once the stream has passed the copy, e.g. after gasloc_synchronize;
 * later rounds do not disturb a copy already enqueued. */
int gasloc_consensus_error_async(gasloc_ctx *ctx, double *dst);

/* Waits until every call enqueued on the context's stream has finished;
 * EDEVICE if a kernel reported an error (the flag is then cleared). */
int gasloc_synchronize(gasloc_ctx *ctx);

/* Consensus error of caller-owned replicas, for callers that cannot allocate
 * device memory at the point they need it: a framework that owns all device
 * memory through its own pool (a side cudaMalloc could fail or fragment it),
 * a latency-critical loop where cudaMalloc/cudaFree would synchronise the
 * device, or a plug-in that is handed pre-allocated buffers only.  The paper
 * has no counterpart; this is a service of the library.
 *   x: device pointer to fp32 values, n_workers rows of worker_stride floats
 *      each (row i is replica i; the caller owns all n_workers * worker_stride
 *      floats), 16-byte aligned, worker_stride a multiple of 4 and >=
 *      n_params.  The values must be fp32: the pointer gasloc_buffer returns
 *      for a context with a bf16 store is not valid input (its elements would
 *      be read as floats and the value would be wrong, with no error).
 *   ce_out_device: device pointer to one double that receives
 *      (1/n) sum_i ||x_i - xbar||^2 (same arithmetic as gasloc_consensus_error).
 *   cuda_stream: the stream the work is enqueued on (asynchronous).
 * Nothing is allocated: the reduction's scratch is a fixed 512 KiB + 256 B
 * array compiled into the library, held by every GPU that loads it until the
 * process exits.  n_params above 536,870,912 is rejected (GASLOC_ENOMEM).
 * The array's device address belongs to the CUDA context: the first call in
 * each context (the device's primary context, or a driver context the caller
 * created and made current) looks it up, with the launch shape, in the
 * context current on the calling thread and caches it under that context's
 * process-unique id; make that first call before any stream capture.  A
 * context that replaces another (after cudaDeviceReset or a primary-context
 * reset) has a new id, so the address is looked up again.  Every call reuses
 * the same array (its completion counter is cleared at the start of each
 * call): calls whose work overlaps on the GPU race, so serialise them (one
 * stream, or events).  In the index-checked build a failed check makes the
 * result NaN.  Errors: EINVAL (null or misaligned pointers, bad sizes), ENOMEM
 * (size limit), ECUDA. */
int gasloc_consensus_error_noalloc(const float *x, int32_t n_workers, int64_t n_params,
                                   int64_t worker_stride, double *ce_out_device, void *cuda_stream);

/* Neighbour table of round `round` as the device generates it: host arrays
 * nbr[n*n] (row i: N_i ascending, deg[i]+1 valid entries), w[n*n] (fp32) and
 * deg[n] (graph degree, self excluded).  Synchronising. */
int gasloc_get_topology(gasloc_ctx *ctx, int64_t round, int32_t *nbr, float *w, int32_t *deg);

/* Output of Algorithm 1: xbar = (1/n) sum_i x_i into dst (n_params fp32,
 * device memory; concatenation order).  Asynchronous. */
int gasloc_average(gasloc_ctx *ctx, float *dst_device);
/* Same into host memory (pinned or pageable), through a device buffer of
 * n_params floats that the context allocates in gasloc_start.
 * Synchronising. */
int gasloc_average_host(gasloc_ctx *ctx, float *dst_host);

/* Device pointer of buffer `which` for tensor `tensor`: worker i's slice
 * starts at *dptr + i * (*worker_stride) elements (fp32 or bf16 as the
 * storage type; worker_stride may be NULL; for GASLOC_BUF_H with a shared
 * curvature it is 0).  Valid until destroy. */
int gasloc_buffer(gasloc_ctx *ctx, int32_t which, int32_t tensor, void **dptr,
                  int64_t *worker_stride);

/* Copies buffer `which` of `worker` (flat, n_params fp32 values) to or from
 * host memory.  With bf16 storage the values pass through an fp32 staging
 * buffer on the device (the largest tensor, at most 32 Mi elements, taken
 * from the context's allocator for the call) and are widened exactly on read
 * or rounded to nearest even on write by a kernel; GASLOC_ENOMEM if the
 * staging buffer cannot be had.  In gasloc_write, worker = -1 writes every
 * worker (x_0 broadcast).  Synchronising. */
int gasloc_read(gasloc_ctx *ctx, int32_t which, int32_t worker, float *host_dst);
int gasloc_write(gasloc_ctx *ctx, int32_t which, int32_t worker, const float *host_src);

/* Gathers n elements (global indices idx[], host array) of buffer `which` of
 * `worker` into host out[].  Synchronising. */
int gasloc_gather(gasloc_ctx *ctx, int32_t which, int32_t worker, int64_t n,
                  const int64_t *idx, float *out);

/* Completed gossip rounds and local steps taken by a worker. */
int gasloc_round(const gasloc_ctx *ctx, int64_t *round);
int gasloc_steps_taken(const gasloc_ctx *ctx, int32_t worker, int64_t *steps);

/* Checkpoint: every buffer plus counters.  gasloc_load needs a started
 * context of the same shape, topology and seed.  Synchronising; EIO. */
int gasloc_save(gasloc_ctx *ctx, const char *path);
int gasloc_load(gasloc_ctx *ctx, const char *path);

/* Failure detection self-test.  Every wait the pipeline kernels make on an
 * mbarrier is bounded: on expiry the kernel records a device error, finishes
 * its in-flight copies and returns, and the next synchronising call reports
 * GASLOC_EDEVICE and clears the flag.  This call runs that exact wait routine
 * on a barrier nothing completes, with a limit of limit_ns (1 ns .. 2 s), so
 * the expected result is GASLOC_EDEVICE; the context stays usable afterwards.
 * (The paper argues that sparse exchanges tolerate failures that are skipped,
 * Sec. 3.2 "Fault tolerance"; detecting a stalled exchange is this library's
 * side of that.)  Synchronising. */
int gasloc_selftest_bounded_wait(gasloc_ctx *ctx, int64_t limit_ns);

/* Index checks, the stand-in for a memory sanitizer (none can be run on the
 * GPUs this library targets).  The same sources built with the checks
 * (build.build(checked=True) -> libgasloc_checked.so) test every worker row,
 * column range, neighbour index and TMA offset a kernel uses before the
 * access; a failed test skips the access and is reported as GASLOC_EDEVICE by
 * the next synchronising call.  Nothing traps.  The paper has no counterpart.
 * gasloc_checked_build returns 1 for the checked library, 0 for the normal one
 * (whose checks compile to nothing).  gasloc_selftest_index_check evaluates
 * one failing check on the device without touching memory: GASLOC_EDEVICE
 * from the checked library, GASLOC_OK from the normal one; the context stays
 * usable.  Synchronising. */
int gasloc_checked_build(void);
int gasloc_selftest_index_check(gasloc_ctx *ctx);

/* Launch counter of the library's kernels on this context (for accounting). */
int gasloc_launch_count(const gasloc_ctx *ctx, int64_t *count);

const char *gasloc_last_error(void);

/* Releases the context and all its device memory (waits for its stream). */
void gasloc_destroy(gasloc_ctx *ctx);

#ifdef __cplusplus
}
#endif
#endif /* GASLOC_H */
