/*
 * relaysum_oracle.c -- plain, slow CPU oracle for one RelaySum/RelaySGD step.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may link, load or
 * call this file: only the tests, __graft_entry__.smoke() and the CPU-baseline
 * leg of bench.py use it.  It shares no code, header or table with the CUDA
 * library (paper_2110_04175_gb300/csrc); the only things the two agree on are
 * the public data layout (row-major [rows][len] arrays, directed edge 2u is
 * edges[u][0] -> edges[u][1] and 2u+1 is its reverse) and the published
 * definition of the Philox4x32-10 generator, which each side implements on
 * its own.
 *
 * Arithmetic is IEEE double throughout.  Every sum is a left fold in
 * ascending neighbour id; no blocking, fusion or reordering beyond that.
 *
 * What is computed (Vogels et al., "RelaySum for Decentralized Deep Learning
 * on Heterogeneous Data", Algorithm 1 "RelaySGD", Section 3):
 *
 *   x_i^{t+1/2}   = x_i^t - gamma * grad F_i(x_i^t; xi_i^t)          (Alg. 1, local step)
 *   m_{i->j}^{t}  = x_i^{t+1/2} + sum_{k in N(i)\j} m_{k->i}^{t-1}   (Alg. 1, relay message)
 *   c_{i->j}^{t}  = 1 + sum_{k in N(i)\j} c_{k->i}^{t-1}             (Alg. 1, counters)
 *   nbar_i^{t+1}  = 1 + sum_{j in N(i)} c_{j->i}^{t}                 (Alg. 1, models received)
 *   mode 0 (Alg. 1 rebuild):
 *     x_i^{t+1}   = (x_i^{t+1/2} + sum_{j in N(i)} m_{j->i}^{t}) / nbar_i^{t+1}
 *   mode 1 (robust rebuild, Section 4.4 "Robustness to unreliable communication"):
 *     x_i^{t+1}   = (x_i^{t+1/2} + sum_j m_{j->i}^{t} + (n - nbar_i^{t+1}) x_i^t) / n
 *
 * with m^{-1} = 0, c^{-1} = 0 and x_i^0 = x^0 for all i (Alg. 1, inputs).
 *
 * The local objective is the synthetic heterogeneous quadratic
 * f_i(x) = 1/2 ||x - mu_i||^2 with additive normal gradient noise (the
 * "random normal noise added to each gradient update" of Appendix
 * "Independence of heterogeneity"), so grad F_i(x; xi) = (x - mu_i) + sigma*xi.
 *
 * Random numbers: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel Random
 * Numbers: As Easy as 1, 2, 3", SC'11), key = (seed lo32, seed hi32),
 * counter = (coordinate quad q = c/4, row, step, stream).  Stream 0 is the
 * gradient noise of worker `row` at step `step`, stream 1 the Gaussian centre
 * `row`, stream 2 the shared initial model.  The four 32-bit words become
 * uniforms u = ((w >> 8) + 1) * 2^-24 in (0, 1]; Box-Muller turns words
 * (0, 1) into the normals of coordinates 4q, 4q+1 (cos, sin) and words (2, 3)
 * into those of 4q+2, 4q+3.
 *
 * parity pinned: every function here is checked against something other than
 * itself -- published Philox known-answer vectors, closed forms (counters,
 * subtree sums, fixed points, plain SGD and all-reduce special cases), an
 * exact-rational routing brute force on every tree of up to 6 nodes, the
 * paper's stacked-delay matrix form, torch.optim's SGD/Adam, and brute-force
 * restatements of Algorithms 5 and 6: tests/test_oracle_pins.py,
 * tests/test_bruteforce.py, tests/test_matrix_form.py and
 * tests/test_oracle_extensions.py.
 */
#define _USE_MATH_DEFINES
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifndef M_PI
#define M_PI 3.14159265358979323846
#endif

#define ORACLE_OK 0
#define ORACLE_EINVAL (-1)
#define ORACLE_ENOTTREE (-2)
#define ORACLE_ENOMEM (-3)

/* ---------------------------------------------------------------- Philox */

/* Philox4x32 constants from the SC'11 paper: the two round multipliers and
 * the two Weyl key increments (golden ratio and sqrt(3)-1). */
#define PHILOX_M0 0xD2511F53u
#define PHILOX_M1 0xCD9E8D57u
#define PHILOX_W0 0x9E3779B9u
#define PHILOX_W1 0xBB67AE85u

/* One Philox4x32-10 block: 10 rounds of the S-box/P-box network, the key
 * bumped by the Weyl increments between rounds. */
void oracle_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2],
                          uint32_t out[4]) {
    uint32_t c0 = ctr_in[0], c1 = ctr_in[1], c2 = ctr_in[2], c3 = ctr_in[3];
    uint32_t k0 = key_in[0], k1 = key_in[1];
    for (int round = 0; round < 10; ++round) {
        if (round > 0) {
            k0 += PHILOX_W0;
            k1 += PHILOX_W1;
        }
        uint64_t p0 = (uint64_t)PHILOX_M0 * (uint64_t)c0;
        uint64_t p1 = (uint64_t)PHILOX_M1 * (uint64_t)c2;
        uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        uint32_t n0 = hi1 ^ c1 ^ k0;
        uint32_t n1 = lo1;
        uint32_t n2 = hi0 ^ c3 ^ k1;
        uint32_t n3 = lo0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* 24 random bits -> uniform in (0, 1], exact in any binary format. */
double oracle_uniform(uint32_t w) {
    return (double)((w >> 8) + 1u) * (1.0 / 16777216.0);
}

/* The standard normal assigned to absolute coordinate c of (row, step,
 * stream) under `seed`: Box-Muller on the Philox block of quad c/4. */
double oracle_normal(uint64_t seed, int64_t c, uint32_t row, uint32_t step,
                     uint32_t stream) {
    uint32_t ctr[4] = {(uint32_t)(c / 4), row, step, stream};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t w[4];
    oracle_philox4x32_10(ctr, key, w);
    int r = (int)(c % 4);
    int pair = r / 2;
    double ua = oracle_uniform(w[2 * pair]);
    double ub = oracle_uniform(w[2 * pair + 1]);
    double radius = sqrt(-2.0 * log(ua));
    double angle = 2.0 * M_PI * ub;
    return (r % 2 == 0) ? radius * cos(angle) : radius * sin(angle);
}

/* ----------------------------------------------------------------- trees */

typedef struct {
    int n, E;
    int32_t *src, *dst;   /* directed edge e: src[e] -> dst[e]            */
    int32_t *nbr_off;     /* node i's neighbours: nbr[nbr_off[i] .. +deg) */
    int32_t *nbr;         /* ascending neighbour ids                      */
    int32_t *in_edge;     /* edge nbr[k] -> i, aligned with nbr           */
    int32_t *out_edge;    /* edge i -> nbr[k], aligned with nbr           */
} otree;

static void otree_free(otree *t) {
    free(t->src); free(t->dst); free(t->nbr_off); free(t->nbr);
    free(t->in_edge); free(t->out_edge);
    memset(t, 0, sizeof(*t));
}

static int cmp_i32(const void *a, const void *b) {
    int32_t x = *(const int32_t *)a, y = *(const int32_t *)b;
    return (x > y) - (x < y);
}

/* Builds the directed-edge view of an undirected tree given as n-1 pairs.
 * Rejects self loops, duplicate edges, out-of-range ids and disconnected
 * graphs (Section 3 "Setup": undirected graph without self loops; Alg. 1
 * needs a tree). */
static int otree_build(int n, const int32_t *edges, int n_edges, otree *t) {
    memset(t, 0, sizeof(*t));
    if (n < 1 || n_edges != n - 1) return ORACLE_ENOTTREE;
    int E = 2 * n_edges;
    t->n = n; t->E = E;
    t->src = malloc(sizeof(int32_t) * (E + 1));
    t->dst = malloc(sizeof(int32_t) * (E + 1));
    t->nbr_off = calloc((size_t)n + 1, sizeof(int32_t));
    t->nbr = malloc(sizeof(int32_t) * (E + 1));
    t->in_edge = malloc(sizeof(int32_t) * (E + 1));
    t->out_edge = malloc(sizeof(int32_t) * (E + 1));
    if (!t->src || !t->dst || !t->nbr_off || !t->nbr || !t->in_edge || !t->out_edge) {
        otree_free(t);
        return ORACLE_ENOMEM;
    }
    for (int u = 0; u < n_edges; ++u) {
        int a = edges[2 * u], b = edges[2 * u + 1];
        if (a < 0 || b < 0 || a >= n || b >= n || a == b) { otree_free(t); return ORACLE_ENOTTREE; }
        t->src[2 * u] = a; t->dst[2 * u] = b;
        t->src[2 * u + 1] = b; t->dst[2 * u + 1] = a;
    }
    /* neighbour lists sorted by id, with the matching edge numbers */
    for (int e = 0; e < E; ++e) t->nbr_off[t->src[e] + 1]++;
    for (int i = 0; i < n; ++i) t->nbr_off[i + 1] += t->nbr_off[i];
    int *fill = calloc((size_t)n, sizeof(int));
    if (!fill) { otree_free(t); return ORACLE_ENOMEM; }
    for (int e = 0; e < E; ++e) {
        int i = t->src[e];
        t->nbr[t->nbr_off[i] + fill[i]++] = t->dst[e];
    }
    free(fill);
    for (int i = 0; i < n; ++i) {
        int lo = t->nbr_off[i], hi = t->nbr_off[i + 1];
        qsort(t->nbr + lo, (size_t)(hi - lo), sizeof(int32_t), cmp_i32);
        for (int k = lo + 1; k < hi; ++k)
            if (t->nbr[k] == t->nbr[k - 1]) { otree_free(t); return ORACLE_ENOTTREE; }
        for (int k = lo; k < hi; ++k) {
            int j = t->nbr[k];
            for (int e = 0; e < E; ++e) {
                if (t->src[e] == j && t->dst[e] == i) t->in_edge[k] = e;
                if (t->src[e] == i && t->dst[e] == j) t->out_edge[k] = e;
            }
        }
    }
    /* connectivity: n-1 distinct edges and connected <=> tree */
    int *seen = calloc((size_t)n, sizeof(int));
    int *stack = malloc(sizeof(int) * (size_t)n);
    if (!seen || !stack) { free(seen); free(stack); otree_free(t); return ORACLE_ENOMEM; }
    int top = 0, reached = 1;
    seen[0] = 1; stack[top++] = 0;
    while (top > 0) {
        int i = stack[--top];
        for (int k = t->nbr_off[i]; k < t->nbr_off[i + 1]; ++k) {
            int j = t->nbr[k];
            if (!seen[j]) { seen[j] = 1; ++reached; stack[top++] = j; }
        }
    }
    free(seen); free(stack);
    if (reached != n) { otree_free(t); return ORACLE_ENOTTREE; }
    return ORACLE_OK;
}

/* ------------------------------------------------------ objective, init */

/* mu_i(c) = mu_scale * sum_k mix[i][k] * N_k(c), N_k the Gaussian centre k
 * (stream 1).  mu is [n][len] for absolute coordinates c0 .. c0+len-1. */
int oracle_fill_mu(int n, int K, const double *mix, double mu_scale,
                   uint64_t seed, int64_t c0, int64_t len, double *mu) {
    if (n < 1 || K < 0 || len < 0 || c0 < 0) return ORACLE_EINVAL;
    for (int i = 0; i < n; ++i)
        for (int64_t c = 0; c < len; ++c) {
            double s = 0.0;
            for (int k = 0; k < K; ++k)
                s += mix[(int64_t)i * K + k] * oracle_normal(seed, c0 + c, (uint32_t)k, 0u, 1u);
            mu[(int64_t)i * len + c] = mu_scale * s;
        }
    return ORACLE_OK;
}

/* out[c] = oracle_normal(seed, c0 + c, row, step, stream) for c < len: the
 * same numbers as one call per coordinate, for tests that need many. */
int oracle_fill_normals(uint64_t seed, int64_t c0, int64_t len, uint32_t row, uint32_t step,
                        uint32_t stream, double *out) {
    if (len < 0 || c0 < 0 || (len > 0 && !out)) return ORACLE_EINVAL;
    for (int64_t c = 0; c < len; ++c) out[c] = oracle_normal(seed, c0 + c, row, step, stream);
    return ORACLE_OK;
}

/* x_i^0 = x0_std * N(c) for every worker i: one shared draw (stream 2),
 * because Alg. 1 starts all workers from the same model. */
int oracle_fill_x0(int n, double x0_std, uint64_t seed, int64_t c0, int64_t len,
                   double *x) {
    if (n < 1 || len < 0 || c0 < 0) return ORACLE_EINVAL;
    for (int64_t c = 0; c < len; ++c) {
        double v = x0_std * oracle_normal(seed, c0 + c, 0u, 0u, 2u);
        for (int i = 0; i < n; ++i) x[(int64_t)i * len + c] = v;
    }
    return ORACLE_OK;
}

/* ------------------------------------------------------------ the steps */

/* Options beyond plain Algorithm 1.
 *
 * Local optimiser (replaces the local-step line of Alg. 1):
 *   opt 0  SGD:       x^{t+1/2} = x^t - lr g^t
 *   opt 1  Nesterov momentum (appendix "RelaySGD with momentum"), s1 = m,
 *          m^{-1} = 0:  m^t = beta1 m^{t-1} + g^t,
 *                       x^{t+1/2} = x^t - lr (g^t + beta1 m^t)
 *   opt 2  Adam (appendix "RelaySGD with Adam": PyTorch's standard Adam, all
 *          state local), s1 = m, s2 = v, both 0 at t = 0, k = t + 1:
 *          m = beta1 m + (1 - beta1) g,  v = beta2 v + (1 - beta2) g^2,
 *          x^{t+1/2} = x^t - (lr / (1 - beta1^k)) m / (sqrt(v) / sqrt(1 - beta2^k) + eps)
 * where g^t = (x^t - mu) + sigma xi^t.
 *
 * Lost messages (Section 4.4, Table 5): drop[(t - step0) * E + e] != 0 means
 * the message sent on directed edge e at step t never arrives: its receiver
 * sees m = 0 and c = 0, uses them in its rebuild and relays them onwards. */
typedef struct {
    int opt;
    double beta1, beta2, eps;
    const uint8_t *drop;  /* [steps][E] or NULL */
    int algo;             /* 0 RelaySGD (Alg. 1), 1 RelaySum/Grad (Alg. 6), 2 DME (Alg. 5) */
    int64_t *dme_count;   /* algo 2: s_i, [n], in/out */
} oracle_opts;

/* The two other algorithms of the appendix on the same relay mechanism:
 *
 *   RelaySum/Grad (Algorithm 6): the relayed value is the update
 *     u_i^t = x_i^{t+1/2} - x_i^t (= -lr g for SGD) and
 *     x_i^{t+1} = x_i^t + (u_i^t + sum_j m^t_{j->i}) / n      (no counters used)
 *
 *   RelaySum for distributed mean estimation (Algorithm 5): the relayed value
 *     is a sample dhat_i^t = mu_i + sigma xi_i^t; x holds the running sum y and
 *     y_i^{t+1} = y_i^t + dhat_i^t + sum_j m^t_{j->i},
 *     s_i^{t+1} = s_i^t + 1 + sum_j c^t_{j->i}   (dme_count),
 *   the estimate of worker i being y_i / s_i. */

int oracle_run_ext(int n, const int32_t *edges, int n_edges, int64_t c0, int64_t len,
                   double *x, const double *mu, double *msg, int32_t *counts, double *s1,
                   double *s2, double lr, double sigma, uint64_t seed, int64_t step0,
                   int64_t steps, int mode, const oracle_opts *opts, int32_t *nbar) {
    const int opt = opts ? opts->opt : 0;
    const int algo = opts ? opts->algo : 0;
    if (len < 0 || c0 < 0 || step0 < 0 || steps < 0 || (mode != 0 && mode != 1) || opt < 0 ||
        opt > 2 || algo < 0 || algo > 2)
        return ORACLE_EINVAL;
    if (algo == 2 && !opts->dme_count) return ORACLE_EINVAL;
    if ((opt >= 1 && !s1) || (opt == 2 && !s2)) return ORACLE_EINVAL;
    if (step0 + steps > 4294967296LL) return ORACLE_EINVAL;
    otree t;
    int rc = otree_build(n, edges, n_edges, &t);
    if (rc) return rc;
    int E = t.E;
    int32_t *c_new = malloc(sizeof(int32_t) * (E + 1));
    int32_t *nb = malloc(sizeof(int32_t) * (size_t)n);
    double *xh = malloc(sizeof(double) * (size_t)n * (size_t)(len > 0 ? len : 1));
    double *m_new = malloc(sizeof(double) * (size_t)(E + 1) * (size_t)(len > 0 ? len : 1));
    if (!c_new || !nb || !xh || !m_new) {
        free(c_new); free(nb); free(xh); free(m_new); otree_free(&t);
        return ORACLE_ENOMEM;
    }
    for (int64_t t_step = step0; t_step < step0 + steps; ++t_step) {
        const uint8_t *lost = (opts && opts->drop) ? opts->drop + (t_step - step0) * E : NULL;
        /* counters c^{t} from c^{t-1} */
        for (int e = 0; e < E; ++e) {
            int i = t.src[e], j = t.dst[e];
            int32_t s = 1;
            for (int k = t.nbr_off[i]; k < t.nbr_off[i + 1]; ++k)
                if (t.nbr[k] != j) s += counts[t.in_edge[k]];
            c_new[e] = (lost && lost[e]) ? 0 : s;
        }
        memcpy(counts, c_new, sizeof(int32_t) * (size_t)E);
        /* nbar^{t+1} from c^{t} */
        for (int i = 0; i < n; ++i) {
            int32_t s = 1;
            for (int k = t.nbr_off[i]; k < t.nbr_off[i + 1]; ++k) s += counts[t.in_edge[k]];
            nb[i] = s;
            if (algo == 2) opts->dme_count[i] += s;
        }
        /* local step (xh holds the relayed value: x^{t+1/2}, u or dhat) */
        const double k_adam = (double)(t_step + 1);
        for (int i = 0; i < n; ++i)
            for (int64_t c = 0; c < len; ++c) {
                const int64_t ic = (int64_t)i * len + c;
                double xv = x[ic];
                double xi = oracle_normal(seed, c0 + c, (uint32_t)i, (uint32_t)t_step, 0u);
                double g = (xv - mu[ic]) + sigma * xi;
                if (algo == 2) {
                    xh[ic] = mu[ic] + sigma * xi;  /* the sample dhat_i^t */
                    continue;
                }
                if (opt == 0) {
                    xh[ic] = xv - lr * g;
                } else if (opt == 1) {
                    s1[ic] = opts->beta1 * s1[ic] + g;
                    xh[ic] = xv - lr * (g + opts->beta1 * s1[ic]);
                } else {
                    const double b1 = opts->beta1, b2 = opts->beta2;
                    s1[ic] = b1 * s1[ic] + (1.0 - b1) * g;
                    s2[ic] = b2 * s2[ic] + (1.0 - b2) * g * g;
                    const double bc1 = 1.0 - pow(b1, k_adam), bc2 = 1.0 - pow(b2, k_adam);
                    const double denom = sqrt(s2[ic]) / sqrt(bc2) + opts->eps;
                    xh[ic] = xv - (lr / bc1) * s1[ic] / denom;
                }
                if (algo == 1) xh[ic] -= xv;  /* the update u = x^{t+1/2} - x^t */
            }
        /* relay messages m^{t} from x^{t+1/2} and m^{t-1} */
        for (int e = 0; e < E; ++e) {
            int i = t.src[e], j = t.dst[e];
            for (int64_t c = 0; c < len; ++c) {
                double s = xh[(int64_t)i * len + c];
                for (int k = t.nbr_off[i]; k < t.nbr_off[i + 1]; ++k)
                    if (t.nbr[k] != j) s += msg[(int64_t)t.in_edge[k] * len + c];
                m_new[(int64_t)e * len + c] = (lost && lost[e]) ? 0.0 : s;
            }
        }
        /* rebuild x^{t+1} */
        for (int i = 0; i < n; ++i)
            for (int64_t c = 0; c < len; ++c) {
                double s = xh[(int64_t)i * len + c];
                for (int k = t.nbr_off[i]; k < t.nbr_off[i + 1]; ++k)
                    s += m_new[(int64_t)t.in_edge[k] * len + c];
                if (algo == 1) {
                    x[(int64_t)i * len + c] += s / (double)n;
                } else if (algo == 2) {
                    x[(int64_t)i * len + c] += s;
                } else if (mode == 0) {
                    x[(int64_t)i * len + c] = s / (double)nb[i];
                } else {
                    double xold = x[(int64_t)i * len + c];
                    x[(int64_t)i * len + c] = (s + (double)(n - nb[i]) * xold) / (double)n;
                }
            }
        if (len > 0) memcpy(msg, m_new, sizeof(double) * (size_t)E * (size_t)len);
    }
    if (nbar) {
        /* nbar from the current counters (equals nb after the last step) */
        for (int i = 0; i < n; ++i) {
            int32_t s = 1;
            for (int k = t.nbr_off[i]; k < t.nbr_off[i + 1]; ++k) s += counts[t.in_edge[k]];
            nbar[i] = s;
        }
    }
    free(c_new); free(nb); free(xh); free(m_new); otree_free(&t);
    return ORACLE_OK;
}

/* Runs `steps` iterations t = step0 .. step0+steps-1 of Algorithm 1 on the
 * coordinate slice [c0, c0+len) of every worker.
 *
 *   x      [n][len]  in: x^{step0}            out: x^{step0+steps}
 *   mu     [n][len]  the quadratic centres mu_i
 *   msg    [E][len]  in: m^{step0-1}          out: m^{step0+steps-1}
 *   counts [E]       in: c^{step0-1}          out: c^{step0+steps-1}
 *   nbar   [n]       out: nbar^{step0+steps} (may be NULL)
 *
 * Coordinates never interact (every line of Alg. 1 is per coordinate) and
 * the noise is keyed by the absolute coordinate, so any slice reproduces
 * exactly the values of the full vector.  len == 0 runs the counters only. */
int oracle_run(int n, const int32_t *edges, int n_edges, int64_t c0, int64_t len,
               double *x, const double *mu, double *msg, int32_t *counts,
               double lr, double sigma, uint64_t seed, int64_t step0,
               int64_t steps, int mode, int32_t *nbar) {
    return oracle_run_ext(n, edges, n_edges, c0, len, x, mu, msg, counts, NULL, NULL, lr, sigma,
                          seed, step0, steps, mode, NULL, nbar);
}

/* Directed edge table of the oracle's own numbering, for cross-checks. */
int oracle_edges(int n, const int32_t *edges, int n_edges, int32_t *src, int32_t *dst) {
    otree t;
    int rc = otree_build(n, edges, n_edges, &t);
    if (rc) return rc;
    memcpy(src, t.src, sizeof(int32_t) * (size_t)t.E);
    memcpy(dst, t.dst, sizeof(int32_t) * (size_t)t.E);
    otree_free(&t);
    return ORACLE_OK;
}
