/*
 * oracle.c -- plain, slow CPU oracle for the GASLoC replica-update path.
 *
 * TEST INFRASTRUCTURE ONLY (see oracle.h).  Loops run round -> worker ->
 * element in the order the paper states the algorithm; the only parallelism is
 * an OpenMP split of the element loop, which cannot change any result because
 * every step is element-wise in the parameter index (the synthetic gradient is
 * diagonal and mixing happens across workers at one index).
 *
 * Build twice:  gcc -O2 -std=c11 -ffp-contract=off -fopenmp -DREAL=float  ...
 *               gcc -O2 -std=c11 -ffp-contract=off -fopenmp -DREAL=double ...
 * -ffp-contract=off keeps every a*b+c below as two roundings unless it is
 * written as fma().
 *
 * Random numbers.  Everything random in the method (initial point, quadratic
 * centres and curvatures, gradient noise, the per-round permutation of the
 * randomized k-Peer schemes, edge activation, per-worker step counts) is drawn
 * from counter-based hashes so that any element of any round can be
 * recomputed on its own:
 *   mix64  = the output function of SplitMix64 (Steele, Lea & Flood, OOPSLA
 *            2014): add the golden-ratio increment 0x9E3779B97F4A7C15, then
 *            z ^= z>>30, z *= 0xBF58476D1CE4E5B9, z ^= z>>27,
 *            z *= 0x94D049BB133111EB, z ^= z>>31.
 *   hash(seed, tag, a, b) = mix64(mix64(mix64(mix64(seed) ^ tag) ^ a) ^ b)
 *            tags: 1 x0, 2 centre c, 3 curvature h, 4 noise key, 5 round
 *            permutation, 6 edge activation, 7 local step counts H_i.
 *   fmix32 = the 32-bit finalizer of MurmurHash3 (Appleby, public domain):
 *            h ^= h>>16, h *= 0x85EBCA6B, h ^= h>>13, h *= 0xC2B2AE35,
 *            h ^= h>>16.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <tgmath.h>
#ifdef _OPENMP
#include <omp.h>
#endif
#include "oracle.h"

#ifndef REAL
#define REAL double
#endif

#define OC_MAXN 1024

/* ------------------------------------------------------------------------- */
/* Counter-based generators                                                  */
/* ------------------------------------------------------------------------- */

uint64_t oc_mix64(uint64_t z)
{
    z += 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

uint64_t oc_hash(uint64_t seed, uint64_t tag, uint64_t a, uint64_t b)
{
    uint64_t s = oc_mix64(seed);
    s = oc_mix64(s ^ tag);
    s = oc_mix64(s ^ a);
    return oc_mix64(s ^ b);
}

uint32_t oc_fmix32(uint32_t h)
{
    h ^= h >> 16;
    h *= 0x85EBCA6Bu;
    h ^= h >> 13;
    h *= 0xC2B2AE35u;
    h ^= h >> 16;
    return h;
}

static uint32_t hi32(uint64_t v) { return (uint32_t)(v >> 32); }
static uint32_t lo32(uint64_t v) { return (uint32_t)v; }

/* 24 high bits of a hash: an integer uniform on [0, 2^24). */
static uint32_t u24(uint64_t seed, uint64_t tag, uint64_t a, uint64_t b)
{
    return (uint32_t)(oc_hash(seed, tag, a, b) >> 40);
}

/* Standard-normal stand-in: Irwin-Hall sum of four 24-bit uniforms, centred
 * and scaled to unit variance:  z = (s - 2^25) * (sqrt(3) * 2^-24).
 * Exactly one rounding in the conversion of the integer and one in the
 * product (the scale constant is sqrt(3) rounded to double, times 2^-24,
 * rounded to REAL). */
static REAL normal01(uint64_t seed, uint64_t tag, uint64_t i, uint64_t k)
{
    int64_t s = 0;
    for (uint64_t j = 0; j < 4; ++j)
        s += (int64_t)u24(seed, tag, i, 4 * k + j);
    const REAL scale = (REAL)(1.7320508075688772 * 5.9604644775390625e-08);
    REAL zs = (REAL)(s - ((int64_t)1 << 25));
    return zs * scale;
}

/* Uniform on [lo, lo+span):  fma(span, r*2^-24, lo). */
static REAL uniform_lo_span(uint64_t seed, uint64_t tag, uint64_t i, uint64_t k,
                            REAL lo, REAL span)
{
    const REAL two_m24 = (REAL)5.9604644775390625e-08;
    REAL u = (REAL)u24(seed, tag, i, k) * two_m24;
    return fma(span, u, lo);
}

/* Gradient noise xi(i, n, k): uniform on [-sqrt3, sqrt3), unit variance.
 * K = hash(seed, 4, i, n) is the key of worker i's n-th (1-based) local step
 * and W(a) = fmix32(fmix32(a ^ lo32(K)) ^ hi32(K)), a taken modulo 2^32.
 *   fp32 storage, a grid of 2^24 points, one word per element:
 *     u = W(k),  xi = ((u >> 8) * 2^-23 - 1) * sqrt3.
 *   bf16 storage, a grid of 2^16 points, one word per pair of elements:
 *     element 2j takes the low 16 bits of W(j), element 2j+1 the high 16
 *     bits; with q = half - 2^15 (an integer in [-2^15, 2^15)),
 *     xi = q * (sqrt3 * 2^-15), one rounding (q and the power-of-two scaling
 *     of sqrt3 are exact).  A bf16 store keeps 8 significand bits, so the
 *     finer grid of the fp32 form would buy it nothing. */
static uint32_t noise_word(uint64_t key, uint64_t a)
{
    return oc_fmix32(oc_fmix32((uint32_t)a ^ lo32(key)) ^ hi32(key));
}

static REAL noise_xi(uint64_t key, uint64_t k, int storage)
{
    const REAL sqrt3 = (REAL)1.7320508075688772;
    if (storage == OC_STORE_BF16) {
        const REAL two_m15 = (REAL)3.0517578125e-05;
        const REAL scale = sqrt3 * two_m15;
        const uint32_t u = noise_word(key, k >> 1);
        const uint32_t half = (k & 1u) ? (u >> 16) : (u & 0xFFFFu);
        const REAL q = (REAL)((int32_t)half - 32768);
        return q * scale;
    }
    const REAL two_m23 = (REAL)1.1920928955078125e-07;
    const REAL one = (REAL)1;
    const uint32_t u = noise_word(key, k);
    const REAL a = (REAL)(u >> 8) * two_m23;
    return (a - one) * sqrt3;
}

/* ------------------------------------------------------------------------- */
/* bfloat16 storage                                                          */
/* ------------------------------------------------------------------------- */

/* Rounds a binary32 value to the nearest bfloat16 (the upper 16 bits of a
 * binary32), ties to even: add 0x7FFF plus the lowest kept bit, then clear
 * the low half.  Infinities pass through; NaNs stay NaN. */
static float bf16_round_f(float f)
{
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7F800000u) == 0x7F800000u) {
        if (u & 0x007FFFFFu) u |= 0x00400000u;    /* keep NaN quiet */
    } else {
        u += 0x7FFFu + ((u >> 16) & 1u);
    }
    u &= 0xFFFF0000u;
    memcpy(&f, &u, 4);
    return f;
}

double oc_bf16_round(double v) { return (double)bf16_round_f((float)v); }

/* The value a store keeps: unchanged in fp32 storage, rounded to bfloat16
 * in bf16 storage. */
static REAL stored(int storage, REAL v)
{
    return storage == OC_STORE_BF16 ? (REAL)bf16_round_f((float)v) : v;
}

/* Exported single-value generators (for the property tests). */
double oc_normal(uint64_t seed, uint64_t tag, uint64_t i, uint64_t k)
{ return (double)normal01(seed, tag, i, k); }
double oc_uniform(uint64_t seed, uint64_t tag, uint64_t i, uint64_t k, double lo, double span)
{ return (double)uniform_lo_span(seed, tag, i, k, (REAL)lo, (REAL)span); }
double oc_noise(uint64_t seed, uint64_t i, uint64_t n, uint64_t k, int32_t storage)
{ return (double)noise_xi(oc_hash(seed, 4, i, n), k, storage); }
int oc_real_size(void) { return (int)sizeof(REAL); }
int oc_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Uniform permutation of round t (Sec. 3.2: "we sample a permutation sigma
 * uniformly at random"): Fisher-Yates from the top, each draw mapped to
 * [0, q] by Lemire's multiply-shift j = (r * (q+1)) >> 32. */
void oc_permutation(uint64_t seed, int64_t t, int32_t n, int32_t *perm)
{
    for (int32_t q = 0; q < n; ++q) perm[q] = q;
    for (int32_t q = n - 1; q >= 1; --q) {
        uint64_t r = hi32(oc_hash(seed, 5, (uint64_t)t, (uint64_t)q));
        int32_t j = (int32_t)((r * (uint64_t)(q + 1)) >> 32);
        int32_t tmp = perm[q]; perm[q] = perm[j]; perm[j] = tmp;
    }
}

/* Per-worker local step counts H_i in {1, ..., hmax}, drawn once per run
 * (Sec. 3.2, "Robustness to heterogeneous bandwidth"). */
void oc_draw_local_steps(uint64_t seed, int32_t n, int32_t hmax, int32_t *H)
{
    for (int32_t i = 0; i < n; ++i) {
        uint64_t r = hi32(oc_hash(seed, 7, (uint64_t)i, 0));
        H[i] = 1 + (int32_t)((r * (uint64_t)hmax) >> 32);
    }
}

/* ------------------------------------------------------------------------- */
/* Communication graph and mixing weights of round t                         */
/* ------------------------------------------------------------------------- */

/* Adjacency (no self loops) of the round-t graph, before weights. */
static int build_adjacency(const oc_problem *pb, int64_t t, unsigned char *adj)
{
    const int32_t n = pb->n_workers;
    memset(adj, 0, (size_t)n * (size_t)n);
#define EDGE(a, b) do { int32_t a_ = (a), b_ = (b); \
        if (a_ != b_) { adj[a_ * n + b_] = 1; adj[b_ * n + a_] = 1; } } while (0)
    switch (pb->topology) {
    case OC_TOPO_NONE:
        break;
    case OC_TOPO_RING:
        for (int32_t i = 0; i < n; ++i) EDGE(i, (i + 1) % n);
        break;
    case OC_TOPO_COMPLETE:
        for (int32_t i = 0; i < n; ++i)
            for (int32_t j = i + 1; j < n; ++j) EDGE(i, j);
        break;
    case OC_TOPO_EXP:
        /* peers at +-2^q for every 2^q < n */
        for (int32_t i = 0; i < n; ++i)
            for (int64_t s = 1; s < n; s *= 2) EDGE(i, (int32_t)((i + s) % n));
        break;
    case OC_TOPO_TORUS: {
        const int32_t R = pb->torus_rows, C = pb->torus_cols;
        if (R < 1 || C < 1 || R * C != n) return -1;
        for (int32_t r = 0; r < R; ++r)
            for (int32_t c = 0; c < C; ++c) {
                EDGE(r * C + c, ((r + 1) % R) * C + c);
                EDGE(r * C + c, r * C + (c + 1) % C);
            }
        break;
    }
    case OC_TOPO_MATCHING:
    case OC_TOPO_TWOPEER: {
        int32_t perm[OC_MAXN];
        oc_permutation(pb->seed, t, n, perm);
        if (pb->topology == OC_TOPO_MATCHING) {
            /* pairs (sigma(2i-1), sigma(2i)); an odd last worker stays alone */
            for (int32_t p = 0; p + 1 < n; p += 2) EDGE(perm[p], perm[p + 1]);
        } else {
            /* cycle in the order of sigma, sigma(n+1) = sigma(1) */
            for (int32_t q = 0; q < n; ++q) EDGE(perm[q], perm[(q + 1) % n]);
        }
        break;
    }
    default:
        return -1;
    }
#undef EDGE
    if (pb->edge_prob < 1.0) {
        /* each undirected edge {a<b} stays active this round with prob. p */
        const uint64_t thr = (uint64_t)floor(pb->edge_prob * 4294967296.0);
        for (int32_t a = 0; a < n; ++a)
            for (int32_t b = a + 1; b < n; ++b) {
                if (!adj[a * n + b]) continue;
                uint64_t r = hi32(oc_hash(pb->seed, 6, (uint64_t)t,
                                          (uint64_t)a * (uint64_t)n + (uint64_t)b));
                if (!(r < thr)) { adj[a * n + b] = 0; adj[b * n + a] = 0; }
            }
    }
    return 0;
}

/* Neighbour table of round t: row i lists N_i = {i} U {j : (ij) in E_t} in
 * ascending order (nbr[i*n + q], q <= deg[i]) with its weights w_ij (double,
 * the exact rational rounded once).  Weights:
 *   uniform     w_ij = 1/|N_i|                       (Algorithm 1)
 *   metropolis  w_ij = 1/(1+max(d_i,d_j)), w_ii = 1 - sum_{j!=i} w_ij
 *   lazy        w_ii = 1/2, w_ij = 1/(2 d_i)  -- W = I - Lambda for the
 *               randomized 1-Peer and 2-Peer Laplacians of Sec. 3.2
 * A worker with no edge keeps w_ii = 1. */
int oc_topology(const oc_problem *pb, int64_t t, int32_t *nbr, double *w, int32_t *deg)
{
    const int32_t n = pb->n_workers;
    if (n < 1 || n > OC_MAXN) return -1;
    unsigned char *adj = (unsigned char *)malloc((size_t)n * (size_t)n);
    if (!adj) return -2;
    if (build_adjacency(pb, t, adj) != 0) { free(adj); return -1; }
    for (int32_t i = 0; i < n; ++i) {
        int32_t d = 0;
        for (int32_t j = 0; j < n; ++j) d += adj[i * n + j];
        deg[i] = d;
    }
    for (int32_t i = 0; i < n; ++i) {
        int32_t q = 0;
        for (int32_t j = 0; j < n; ++j) {
            if (j != i && !adj[i * n + j]) continue;
            nbr[i * n + q] = j;
            double wij;
            if (pb->weights == OC_W_UNIFORM) {
                wij = 1.0 / (double)(deg[i] + 1);
            } else if (pb->weights == OC_W_METROPOLIS) {
                if (j == i) {
                    double s = 0.0;
                    for (int32_t l = 0; l < n; ++l)
                        if (l != i && adj[i * n + l])
                            s += 1.0 / (double)(1 + (deg[i] > deg[l] ? deg[i] : deg[l]));
                    wij = 1.0 - s;
                } else {
                    wij = 1.0 / (double)(1 + (deg[i] > deg[j] ? deg[i] : deg[j]));
                }
            } else if (pb->weights == OC_W_LAZY) {
                if (deg[i] == 0) wij = 1.0;
                else wij = (j == i) ? 0.5 : 0.5 / (double)deg[i];
            } else {
                free(adj);
                return -1;
            }
            w[i * n + q] = wij;
            ++q;
        }
    }
    free(adj);
    return 0;
}

/* ------------------------------------------------------------------------- */
/* Replica state                                                             */
/* ------------------------------------------------------------------------- */

struct oc_state {
    oc_problem pb;
    int64_t nk;          /* number of parameter indices held */
    int64_t *kidx;       /* their global indices */
    REAL *x, *y, *m, *v, *b, *c, *h;   /* [N][nk]; h is [N or 1][nk] */
    int64_t *nsteps;     /* local steps taken by each worker so far */
    int32_t *fresh;      /* 1 if worker took >= 1 local step this round */
    int64_t round;       /* completed gossip rounds */
};

static void *xcalloc(size_t n, size_t sz) { return calloc(n ? n : 1, sz); }

void oc_destroy(oc_state *st)
{
    if (!st) return;
    free(st->kidx); free(st->x); free(st->y); free(st->m); free(st->v);
    free(st->b); free(st->c); free(st->h); free(st->nsteps); free(st->fresh);
    free(st);
}

/* Initial state: identical x_0 ~ N(0, 0.02^2) on every worker (Prop. 2 assumes
 * x_0^1 = ... = x_0^n), per-worker centres c_i ~ N(0,1), curvature
 * h ~ U(0.1, 1) (one per worker when per_worker_h), m = v = b = 0, y = x. */
oc_state *oc_create(const oc_problem *pb, const int64_t *kidx, int64_t nk)
{
    const int32_t n = pb->n_workers;
    if (n < 1 || n > OC_MAXN || nk < 0) return NULL;
    oc_state *st = (oc_state *)xcalloc(1, sizeof(oc_state));
    if (!st) return NULL;
    st->pb = *pb;
    st->nk = nk;
    const size_t tot = (size_t)n * (size_t)nk;
    const int32_t nh = pb->per_worker_h ? n : 1;
    st->kidx = (int64_t *)xcalloc((size_t)nk, sizeof(int64_t));
    st->x = (REAL *)xcalloc(tot, sizeof(REAL));
    st->y = (REAL *)xcalloc(tot, sizeof(REAL));
    st->m = (REAL *)xcalloc(tot, sizeof(REAL));
    st->v = (REAL *)xcalloc(tot, sizeof(REAL));
    st->b = (REAL *)xcalloc(tot, sizeof(REAL));
    st->c = (REAL *)xcalloc(tot, sizeof(REAL));
    st->h = (REAL *)xcalloc((size_t)nh * (size_t)nk, sizeof(REAL));
    st->nsteps = (int64_t *)xcalloc((size_t)n, sizeof(int64_t));
    st->fresh = (int32_t *)xcalloc((size_t)n, sizeof(int32_t));
    if (!st->kidx || !st->x || !st->y || !st->m || !st->v || !st->b || !st->c ||
        !st->h || !st->nsteps || !st->fresh) { oc_destroy(st); return NULL; }
    for (int64_t e = 0; e < nk; ++e) st->kidx[e] = kidx ? kidx[e] : e;

    const uint64_t seed = pb->seed;
    const int sto = pb->storage;
    const REAL x0std = (REAL)0.02, hlo = (REAL)0.1, hspan = (REAL)0.9;
    #pragma omp parallel for schedule(static)
    for (int64_t e = 0; e < nk; ++e) {
        const uint64_t k = (uint64_t)st->kidx[e];
        const REAL x0 = stored(sto, x0std * normal01(seed, 1, 0, k));
        for (int32_t i = 0; i < n; ++i) {
            const size_t o = (size_t)i * (size_t)nk + (size_t)e;
            st->x[o] = x0;
            st->y[o] = x0;
            st->c[o] = stored(sto, normal01(seed, 2, (uint64_t)i, k));
        }
        for (int32_t i = 0; i < nh; ++i)
            st->h[(size_t)i * (size_t)nk + (size_t)e] =
                stored(sto, uniform_lo_span(seed, 3, (uint64_t)i, k, hlo, hspan));
    }
    return st;
}

/* ------------------------------------------------------------------------- */
/* Inner loop: AdamW on the diagonal quadratic (Algorithm 1, inner loop)     */
/* ------------------------------------------------------------------------- */

/* One AdamW step (App. B: weight decay, (beta1, beta2)) of worker i on all its
 * held indices.  Gradient of f_i(x) = 1/2 sum_k h_k (x_k - c_ik)^2 plus noise:
 *   g = h*(y - c) + sigma*xi(i, n, k).
 * Host scalars of the n-th step (double, then rounded once to REAL):
 *   bc1 = 1 - beta1^n, bc2 = 1 - beta2^n (beta^n by n multiplications from 1),
 *   step = lr/bc1, isb = 1/sqrt(bc2), decay = 1 - lr*wd.
 * Per element, one rounding per line:
 *   d = y - c;  t = h*d;  g = fma(sigma, xi, t)
 *   y = y*decay
 *   m = fma(beta1, m, (1-beta1)*g)
 *   v = fma(beta2, v, (1-beta2)*(g*g))
 *   den = fma(sqrt(v), isb, eps)
 *   y = fma(-step, m/den, y)
 * The first step of a round starts from x_i (x_i^{(t,0)} = x_i^{(t)}). */
/* Learning rate of a worker's n-th local step (n >= 1).  App. B: a warm-up
 * over the first 10% of the schedule that starts at 1% of the peak rate, then
 * cosine decay.  Reading: with T = lr_total_steps and W = round(frac * T)
 * warm-up steps, the rate rises linearly from warmup_start * lr at n = 1
 * towards lr, reaches lr at n = W + 1, then follows
 *   lr * (f + (1 - f) * (1 + cos(pi * q)) / 2),  q = (n - W - 1) / (T - W - 1),
 * q clamped to [0, 1], so it is f * lr from n = T on.  T = 0: constant lr. */
double oc_sched_lr(const oc_problem *pb, int64_t n)
{
    const int64_t T = pb->lr_total_steps;
    if (T <= 0) return pb->lr;
    const int64_t W = (int64_t)llround(pb->lr_warmup_frac * (double)T);
    if (n <= W) {
        const double s0 = pb->lr_warmup_start;
        return pb->lr * (s0 + (1.0 - s0) * ((double)(n - 1) / (double)W));
    }
    const int64_t span = T - W - 1;
    double q = span > 0 ? (double)(n - W - 1) / (double)span : 1.0;
    if (q > 1.0) q = 1.0;
    const double f = pb->lr_final_frac;
    const double pi = 3.14159265358979323846;
    return pb->lr * (f + (1.0 - f) * (0.5 * (1.0 + cos(pi * q))));
}

static void adamw_step_worker(oc_state *st, int32_t i)
{
    const oc_problem *pb = &st->pb;
    const int64_t nk = st->nk;
    const int64_t n = st->nsteps[i] + 1;
    double p1 = 1.0, p2 = 1.0;
    for (int64_t s = 0; s < n; ++s) { p1 *= pb->beta1; p2 *= pb->beta2; }
    const double bc1 = 1.0 - p1, bc2 = 1.0 - p2;
    const double lr = oc_sched_lr(pb, n);
    const REAL step = (REAL)(lr / bc1);
    const REAL isb = (REAL)(1.0 / sqrt(bc2));
    const REAL decay = (REAL)(1.0 - lr * pb->weight_decay);
    const REAL b1 = (REAL)pb->beta1, b2 = (REAL)pb->beta2;
    const REAL omb1 = (REAL)(1.0 - pb->beta1), omb2 = (REAL)(1.0 - pb->beta2);
    const REAL eps = (REAL)pb->eps, sigma = (REAL)pb->noise_sigma;
    const uint64_t key = oc_hash(pb->seed, 4, (uint64_t)i, (uint64_t)n);
    const int first = !st->fresh[i];
    const int sto = pb->storage;
    REAL *x = st->x + (size_t)i * (size_t)nk;
    REAL *y = st->y + (size_t)i * (size_t)nk;
    REAL *m = st->m + (size_t)i * (size_t)nk;
    REAL *v = st->v + (size_t)i * (size_t)nk;
    const REAL *c = st->c + (size_t)i * (size_t)nk;
    const REAL *h = st->h + (pb->per_worker_h ? (size_t)i * (size_t)nk : 0);

    #pragma omp parallel for schedule(static)
    for (int64_t e = 0; e < nk; ++e) {
        REAL yy = first ? x[e] : y[e];
        const REAL xi = noise_xi(key, (uint64_t)st->kidx[e], sto);
        const REAL d = yy - c[e];
        const REAL t = h[e] * d;
        const REAL g = fma(sigma, xi, t);
        yy = yy * decay;
        const REAL mm = fma(b1, m[e], omb1 * g);
        const REAL vv = fma(b2, v[e], omb2 * (g * g));
        const REAL den = fma(sqrt(vv), isb, eps);
        yy = fma(-step, mm / den, yy);
        y[e] = stored(sto, yy); m[e] = stored(sto, mm); v[e] = stored(sto, vv);
    }
    st->nsteps[i] = n;
    st->fresh[i] = 1;
}

/* Replaces the hyperparameters of a running state (the inner AdamW and the
 * outer optimizer of Algorithm 1 / Eq. 2, and the mixing weights and edge
 * probability of the sampled neighbourhoods); sizes, graph, seed, curvature
 * layout and storage stay as created.  The next step uses the new values:
 * its bias corrections 1 - beta^n are formed from the current betas, as
 * every step's are. */
void oc_set_hparams(oc_state *st, const oc_problem *pb)
{
    oc_problem *q = &st->pb;
    q->weights = pb->weights;
    q->outer_mode = pb->outer_mode;
    q->edge_prob = pb->edge_prob;
    q->lr = pb->lr;
    q->beta1 = pb->beta1;
    q->beta2 = pb->beta2;
    q->eps = pb->eps;
    q->weight_decay = pb->weight_decay;
    q->noise_sigma = pb->noise_sigma;
    q->outer_lr = pb->outer_lr;
    q->outer_momentum = pb->outer_momentum;
    q->eta = pb->eta;
    q->alpha = pb->alpha;
    q->gamma = pb->gamma;
    q->lr_total_steps = pb->lr_total_steps;
    q->lr_warmup_frac = pb->lr_warmup_frac;
    q->lr_warmup_start = pb->lr_warmup_start;
    q->lr_final_frac = pb->lr_final_frac;
}

/* Runs a block of local steps.  H > 0: every worker takes H steps.  H <= 0:
 * worker i takes Hi[i] steps (heterogeneous H_i, Sec. 3.2). */
int oc_local_steps(oc_state *st, int32_t H, const int32_t *Hi)
{
    const int32_t n = st->pb.n_workers;
    for (int32_t i = 0; i < n; ++i) {
        const int32_t hi = H > 0 ? H : (Hi ? Hi[i] : 0);
        if (hi < 0) return -1;
        for (int32_t s = 0; s < hi; ++s) adamw_step_worker(st, i);
    }
    return 0;
}

/* ------------------------------------------------------------------------- */
/* Outer loop: gossip + outer optimizer (Algorithm 1; Eq. 1/2; App. C)       */
/* ------------------------------------------------------------------------- */

/* One communication round.  With y_j the worker's post-local iterate (x_j if
 * it took no local step this round):
 *   acc_i = sum_{j in N_i, ascending} w_ij * s_j   (acc = fma(w, s_j, acc))
 * where the mixed quantity s is y (GASLoC), z = fma(eta, y - x, x) (Eq. 1/2)
 * or x (DAdam, Local-DAdam).  Then, per mode:
 *   SGD       D = x - acc; x = fma(-eta_out, D, x)
 *   SGDM      D = x - acc; b = fma(mu, b, D); x = fma(-eta_out, b, x)
 *   NESTEROV  D = x - acc; b = fma(mu, b, D); x = fma(-eta_out, fma(mu, b, D), x)
 *   EQ2       x = fma(alpha, acc, (1-alpha)*z); x = fma(gamma, z - zprev, x);
 *             zprev (held in b) = z; zprev = z in the first round (t = 0)
 *   DADAM     x = acc + (y - x)
 *   LOCAL_DADAM  D = x - acc; b = fma(mu, b, D); x = fma(-eta_out, fma(mu, b, D), y)
 * The new state of all workers at an index is computed from the old one
 * before any of it is written. */
int oc_gossip_round(oc_state *st)
{
    const oc_problem *pb = &st->pb;
    const int32_t n = pb->n_workers;
    const int64_t nk = st->nk;
    int32_t *nbr = (int32_t *)malloc(sizeof(int32_t) * (size_t)n * (size_t)n);
    double *wd = (double *)malloc(sizeof(double) * (size_t)n * (size_t)n);
    int32_t *deg = (int32_t *)malloc(sizeof(int32_t) * (size_t)n);
    REAL *w = (REAL *)malloc(sizeof(REAL) * (size_t)n * (size_t)n);
    if (!nbr || !wd || !deg || !w) { free(nbr); free(wd); free(deg); free(w); return -2; }
    if (oc_topology(pb, st->round, nbr, wd, deg) != 0) {
        free(nbr); free(wd); free(deg); free(w); return -1;
    }
    for (int32_t q = 0; q < n * n; ++q) w[q] = (REAL)wd[q];

    const int mode = pb->outer_mode;
    const REAL eta_out = (REAL)pb->outer_lr, mu = (REAL)pb->outer_momentum;
    const REAL eta = (REAL)pb->eta, alpha = (REAL)pb->alpha, gamma = (REAL)pb->gamma;
    const REAL oma = (REAL)(1.0 - pb->alpha);
    const REAL zero = (REAL)0;
    const int first_round = st->round == 0;

    #pragma omp parallel for schedule(static)
    for (int64_t e = 0; e < nk; ++e) {
        REAL s[OC_MAXN], xn[OC_MAXN], bn[OC_MAXN];
        /* the quantity each worker sends */
        for (int32_t j = 0; j < n; ++j) {
            const size_t o = (size_t)j * (size_t)nk + (size_t)e;
            const REAL yj = st->fresh[j] ? st->y[o] : st->x[o];
            if (mode == OC_OUT_EQ2) s[j] = fma(eta, yj - st->x[o], st->x[o]);
            else if (mode == OC_OUT_DADAM || mode == OC_OUT_LOCAL_DADAM) s[j] = st->x[o];
            else s[j] = yj;
        }
        for (int32_t i = 0; i < n; ++i) {
            const size_t o = (size_t)i * (size_t)nk + (size_t)e;
            REAL acc = zero;
            for (int32_t q = 0; q <= deg[i]; ++q)
                acc = fma(w[i * n + q], s[nbr[i * n + q]], acc);
            const REAL x = st->x[o];
            const REAL yi = st->fresh[i] ? st->y[o] : x;
            REAL b = st->b[o];
            REAL xnew;
            switch (mode) {
            case OC_OUT_SGD: {
                const REAL D = x - acc;
                xnew = fma(-eta_out, D, x);
                break;
            }
            case OC_OUT_SGDM: {
                const REAL D = x - acc;
                b = fma(mu, b, D);
                xnew = fma(-eta_out, b, x);
                break;
            }
            case OC_OUT_NESTEROV: {
                const REAL D = x - acc;
                b = fma(mu, b, D);
                xnew = fma(-eta_out, fma(mu, b, D), x);
                break;
            }
            case OC_OUT_EQ2: {
                const REAL z = s[i];
                const REAL zprev = first_round ? z : b;
                xnew = fma(alpha, acc, oma * z);
                xnew = fma(gamma, z - zprev, xnew);
                b = z;
                break;
            }
            case OC_OUT_DADAM:
                xnew = acc + (yi - x);
                break;
            case OC_OUT_LOCAL_DADAM: {
                const REAL D = x - acc;
                b = fma(mu, b, D);
                xnew = fma(-eta_out, fma(mu, b, D), yi);
                break;
            }
            default:
                xnew = x;
                break;
            }
            xn[i] = xnew;
            bn[i] = b;
        }
        for (int32_t i = 0; i < n; ++i) {
            const size_t o = (size_t)i * (size_t)nk + (size_t)e;
            st->x[o] = stored(pb->storage, xn[i]);
            st->b[o] = stored(pb->storage, bn[i]);
        }
    }
    for (int32_t i = 0; i < n; ++i) st->fresh[i] = 0;
    st->round += 1;
    free(nbr); free(wd); free(deg); free(w);
    return 0;
}

/* Consensus error (Introduction; the projector pi of Sec. 3.1):
 *   CE = (1/n) sum_i ||x_i - xbar||^2 = ||pi x||^2 / n,  xbar = (1/n) sum_i x_i,
 * evaluated in double from the held values. */
double oc_consensus_error(const oc_state *st)
{
    const int32_t n = st->pb.n_workers;
    const int64_t nk = st->nk;
    double *ek = (double *)malloc(sizeof(double) * (size_t)(nk ? nk : 1));
    if (!ek) return -1.0;
    #pragma omp parallel for schedule(static)
    for (int64_t e = 0; e < nk; ++e) {
        double mean = 0.0;
        for (int32_t i = 0; i < n; ++i) mean += (double)st->x[(size_t)i * (size_t)nk + (size_t)e];
        mean /= (double)n;
        double acc = 0.0;
        for (int32_t i = 0; i < n; ++i) {
            const double d = (double)st->x[(size_t)i * (size_t)nk + (size_t)e] - mean;
            acc += d * d;
        }
        ek[e] = acc;
    }
    double tot = 0.0;
    for (int64_t e = 0; e < nk; ++e) tot += ek[e];
    free(ek);
    return tot / (double)n;
}

/* Network average, the output of Algorithm 1 (double). */
void oc_average(const oc_state *st, double *out)
{
    const int32_t n = st->pb.n_workers;
    const int64_t nk = st->nk;
    for (int64_t e = 0; e < nk; ++e) {
        double s = 0.0;
        for (int32_t i = 0; i < n; ++i) s += (double)st->x[(size_t)i * (size_t)nk + (size_t)e];
        out[e] = s / (double)n;
    }
}

/* ------------------------------------------------------------------------- */
/* Accessors                                                                 */
/* ------------------------------------------------------------------------- */

static REAL *buf_ptr(oc_state *st, int32_t which, int32_t worker)
{
    const int32_t n = st->pb.n_workers;
    if (worker < 0 || worker >= n) return NULL;
    const size_t off = (size_t)worker * (size_t)st->nk;
    switch (which) {
    case OC_BUF_X: return st->x + off;
    case OC_BUF_Y: return st->y + off;
    case OC_BUF_M: return st->m + off;
    case OC_BUF_V: return st->v + off;
    case OC_BUF_B: return st->b + off;
    case OC_BUF_C: return st->c + off;
    case OC_BUF_H: return st->h + (st->pb.per_worker_h ? off : 0);
    default: return NULL;
    }
}

int oc_get(oc_state *st, int32_t which, int32_t worker, double *out)
{
    REAL *p = buf_ptr(st, which, worker);
    if (!p) return -1;
    for (int64_t e = 0; e < st->nk; ++e) out[e] = (double)p[e];
    return 0;
}

/* Overwrites a buffer (values are rounded to REAL, then to the storage type). */
int oc_set(oc_state *st, int32_t which, int32_t worker, const double *in)
{
    REAL *p = buf_ptr(st, which, worker);
    if (!p) return -1;
    for (int64_t e = 0; e < st->nk; ++e) p[e] = stored(st->pb.storage, (REAL)in[e]);
    return 0;
}

int64_t oc_round(const oc_state *st) { return st->round; }
int64_t oc_steps_taken(const oc_state *st, int32_t worker)
{
    if (worker < 0 || worker >= st->pb.n_workers) return -1;
    return st->nsteps[worker];
}
