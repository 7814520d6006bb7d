/*
 * oracle.h -- plain CPU oracle for the GASLoC replica-update path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library links, includes
 * or calls this code; only the test-suite, the smoke check and the CPU-baseline
 * leg of the benchmark load it.  It shares no header, helper or constant table
 * with the CUDA path.
 *
 * The oracle follows the method as the paper states it:
 *   - Algorithm 1 (GASLoC, general form): per worker, H_i inner optimizer steps
 *     from x_i to y_i; then each worker mixes the received y_j of its sampled
 *     neighbourhood N_i (which always contains i) and feeds the pseudo-gradient
 *     x_i - sum_j w_ij y_j to the outer optimizer.  The output is the network
 *     average of the x_i.
 *   - Eq. 1 / Eq. 2 (SGD form with the Laplacian, and its momentum version
 *     "accelerated gossip"): x <- z - alpha*Lambda*z + gamma*(z_t - z_{t-1}),
 *     z = x + eta*g, g = y - x.
 *   - Sec. 3.2 and App. B.1: randomized 1-Peer (random perfect matching from a
 *     uniform permutation) and 2-Peer (ring in the order of the permutation),
 *     redrawn every round.
 *   - App. B (optimisation): AdamW inner optimizer, Nesterov / SGDM / SGD outer
 *     optimizer.
 *   - App. C: DAdam and its delayed multi-step adaptation (Local-DAdam).
 *
 * Arithmetic is generic over REAL (compile with -DREAL=float or -DREAL=double).
 * The float build follows the per-element operation sequence written in the
 * comments of oracle.c one IEEE rounding at a time, because the first AdamW
 * step maps the gradient to its sign and so turns a last-bit difference into an
 * O(lr) one: the parity build takes that decision in the kernel's precision.
 * The double build is the same code in fp64 and is what the mathematical pins
 * check first.
 */
#ifndef GASLOC_ORACLE_H
#define GASLOC_ORACLE_H
#include <stdint.h>

enum { OC_TOPO_NONE = 0, OC_TOPO_RING = 1, OC_TOPO_COMPLETE = 2, OC_TOPO_EXP = 3,
       OC_TOPO_TORUS = 4, OC_TOPO_MATCHING = 5, OC_TOPO_TWOPEER = 6 };
enum { OC_W_UNIFORM = 0, OC_W_METROPOLIS = 1, OC_W_LAZY = 2 };
enum { OC_OUT_SGD = 0, OC_OUT_SGDM = 1, OC_OUT_NESTEROV = 2, OC_OUT_EQ2 = 3,
       OC_OUT_DADAM = 4, OC_OUT_LOCAL_DADAM = 5 };
enum { OC_BUF_X = 0, OC_BUF_Y = 1, OC_BUF_M = 2, OC_BUF_V = 3, OC_BUF_B = 4,
       OC_BUF_C = 5, OC_BUF_H = 6 };

typedef struct {
    int32_t  n_workers;       /* n in the paper */
    int32_t  topology;        /* OC_TOPO_* */
    int64_t  n_params;        /* d in the paper (per worker) */
    int32_t  torus_rows, torus_cols;
    int32_t  weights;         /* OC_W_* */
    int32_t  outer_mode;      /* OC_OUT_* */
    uint64_t seed;
    double   edge_prob;       /* per-round activation probability of each edge */
    double   lr, beta1, beta2, eps, weight_decay;   /* AdamW (inner) */
    double   noise_sigma;     /* sigma of the synthetic gradient noise */
    double   outer_lr, outer_momentum;              /* eta_out, mu */
    double   eta, alpha, gamma;                     /* Eq. 1 / Eq. 2 */
    int32_t  per_worker_h;    /* 1: curvature h_i per worker, 0: one h shared */
    int32_t  storage;         /* OC_STORE_F32, or OC_STORE_BF16: every stored
                                 value is rounded to bfloat16 (nearest, ties
                                 to even) */
    /* learning-rate schedule of App. B over a worker's local steps:
     * lr_total_steps T (0: constant lr), warm-up over a fraction of T from
     * lr_warmup_start * lr, then cosine decay to lr_final_frac * lr */
    int64_t  lr_total_steps;
    double   lr_warmup_frac, lr_warmup_start, lr_final_frac;
} oc_problem;

enum { OC_STORE_F32 = 0, OC_STORE_BF16 = 1 };

typedef struct oc_state oc_state;

#endif
