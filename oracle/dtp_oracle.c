/*
 * dtp_oracle.c -- TEST INFRASTRUCTURE: the reference oracle.
 *
 * A plain, slow, deliberately unoptimised CPU statement of what the
 * affinity-aware sharding hot path computes, written from
 * "Affinity-Aware Sharding for Delayed Tensor Parallelism" (arXiv 2609.13846):
 *
 *   oracle_affinity_fo     Sec. 3 "Affinity scores": the first-order damage
 *                          Delta_hk (the displayed equation for Delta) squared
 *                          and summed over tokens, in fp64.
 *   oracle_finalize        Sec. 3 "Affinity scores": the token mean E_t and the
 *                          ||w^d_k||^2 factor of S^{up,fo}.
 *   oracle_quantize        Sec. 3 "Objective": unit-mass normalisation, stated
 *                          as an exact fixed-point integer form (a positive
 *                          power-of-two scale, then floor).
 *   oracle_layout_score    Eq. (objective), up-edge term of one layer.
 *   oracle_neuron_step     Sec. 3 "Optimiser": the exact balanced linear
 *                          assignment of neurons given the head partition
 *                          (gain M_kl), lexicographically smallest optimum.
 *   oracle_head_step       Sec. 3 "Optimiser": exhaustive scoring of all
 *                          G!/((G/L)!)^L labelled balanced head partitions.
 *   oracle_search_layout   Sec. 3 "Optimiser": coordinate ascent from the
 *                          contiguous head assignment.
 *   oracle_hungarian_max   textbook Hungarian method (Kuhn 1955), used only
 *                          to cross-check the assignment step.
 *   oracle_down_*          Sec. 3 "Affinity scores", down edge: the write
 *                          alpha_k w^d_k of neuron k reaches KV group g of the
 *                          next layer through its pre-norm as (alpha_k/r') b_gk,
 *                          b_gk = W^qkv_g (gamma' . w^d_k); S_down = E_t[alpha_k^2
 *                          / r'^2] ||b_gk||^2.
 *   oracle_normalize_unit_mass, oracle_chain_search
 *                          Sec. 3 "Objective" (Eq. objective, both sums) and
 *                          "Optimiser" over all layers of a model.
 *   oracle_global_layout   Sec. 3 "Objective": the exact maximum of one layer's
 *                          up-edge J over all layouts (unlabelled partitions).
 *   oracle_head_writes     Sec. 3 "Affinity scores": head h's write into the
 *                          FFN input, p_h = gamma . (a_h W_o^(h)) / r.
 *   oracle_layout_order    Sec. 3 (sharding a permuted dense model): the
 *                          order that groups heads / neurons by device.
 *
 * Nothing here is shared with the CUDA library: no header, table or helper.
 * Only the tests, the smoke check and the benchmark's CPU-baseline leg load
 * this file's shared object; the product path never does.
 *
 * Conventions: row-major arrays; X [T,d], C [G,T,d], Wg/Wu [N,d] (nn.Linear
 * [out,in]); A [G,N]; h [G] and nu [N] hold device labels 0..D-1.
 * Status: 0 ok, -1 bad argument, -3 internal inconsistency.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_OK 0
#define OR_ERR_ARG (-1)
#define OR_ERR_INTERNAL (-3)
#define OR_DMAX 8
#define OR_GMAX 16
#define OR_FIXED_POINT_BITS 40

int oracle_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ------------------------------------------------------------------------ */
/* Affinity (Sec. 3 "Affinity scores")                                       */
/* ------------------------------------------------------------------------ */

static double dot(const double* a, const double* b, int n) {
    double s = 0.0;
    for (int i = 0; i < n; ++i) s += a[i] * b[i];
    return s;
}

/*
 * A[h,k] = sum_t Delta_{t,h,k}^2 with, for token t and neuron k,
 *   g = x_t . w^g_k,  u = x_t . w^u_k           (operating point)
 *   sigma = 1/(1+exp(-g)), silu = g*sigma, silu' = sigma*(1 + g*(1-sigma))
 *   Delta = silu'(g) * u * (p_h . w^g_k) + silu(g) * (p_h . w^u_k)
 * where p_h = C[h,t,:] is head h's piece of the normalised FFN input.
 * A is overwritten.  Threads split the neuron axis; each (h,k) entry is summed
 * over tokens in increasing t by one thread, so the result does not depend on
 * the thread count.
 */
void oracle_affinity_fo(const double* X, const double* C, const double* Wg, const double* Wu,
                        int64_t T, int d, int G, int N, double* A) {
    #pragma omp parallel for schedule(dynamic, 1)
    for (int k = 0; k < N; ++k) {
        const double* wg = Wg + (int64_t)k * d;
        const double* wu = Wu + (int64_t)k * d;
        /* column k of A belongs to this iteration alone; any number of heads */
        for (int h = 0; h < G; ++h) A[(int64_t)h * N + k] = 0.0;
        for (int64_t t = 0; t < T; ++t) {
            const double* x = X + t * d;
            double g = dot(x, wg, d);
            double u = dot(x, wu, d);
            double sigma = 1.0 / (1.0 + exp(-g));
            double silu = g * sigma;
            double dsilu = sigma * (1.0 + g * (1.0 - sigma));
            for (int h = 0; h < G; ++h) {
                const double* p = C + ((int64_t)h * T + t) * d;
                double pg = dot(p, wg, d);
                double pu = dot(p, wu, d);
                double delta = dsilu * u * pg + silu * pu;
                A[(int64_t)h * N + k] += delta * delta;
            }
        }
    }
}

/* The ADD score of Sec. 3 before the mean: A_add[h,k] = sum_t (p_h . w^g_k)^2 +
 * (p_h . w^u_k)^2, the squared additive contribution of head h's piece to
 * neuron k's two pre-activations (no operating point, no ||w^d_k||).
 * A_add is overwritten. */
void oracle_affinity_add(const double* C, const double* Wg, const double* Wu, int64_t T, int d, int G, int N,
                         double* A) {
    #pragma omp parallel for schedule(dynamic, 1)
    for (int k = 0; k < N; ++k) {
        const double* wg = Wg + (int64_t)k * d;
        const double* wu = Wu + (int64_t)k * d;
        for (int h = 0; h < G; ++h) {
            double acc = 0.0;
            for (int64_t t = 0; t < T; ++t) {
                const double* p = C + ((int64_t)h * T + t) * d;
                double pg = dot(p, wg, d);
                double pu = dot(p, wu, d);
                acc += pg * pg + pu * pu;
            }
            A[(int64_t)h * N + k] = acc;
        }
    }
}

/* A[h,k] *= wd_sqnorm[k] / T_total  (E_t mean and the ||w^d_k||^2 factor);
 * wd_sqnorm == NULL means the factor 1. */
void oracle_finalize(double* A, int G, int N, int64_t T_total, const double* wd_sqnorm) {
    for (int h = 0; h < G; ++h)
        for (int k = 0; k < N; ++k) {
            double f = wd_sqnorm ? wd_sqnorm[k] : 1.0;
            A[(int64_t)h * N + k] = A[(int64_t)h * N + k] * f / (double)T_total;
        }
}

/* ------------------------------------------------------------------------ */
/* Exact objective (Sec. 3 "Objective")                                      */
/* ------------------------------------------------------------------------ */

/*
 * Unit-mass normalisation divides a layer's matrix by its total mass, a
 * positive constant, so it moves no argmax inside the layer.  The exact form
 * used for the search: with e the binary exponent of max(A) (max(A) < 2^e),
 *   q[g,k] = floor(A[g,k] * 2^(40-e)),   0 <= q < 2^40.
 * All scores are then sums of int64 and do not depend on summation order.
 * *e_out receives e, or 0 when every entry is zero (then q = 0).
 */
int oracle_quantize(const float* A, int G, int N, int64_t* q, int* e_out) {
    float amax = 0.0f;
    for (int64_t i = 0; i < (int64_t)G * N; ++i) {
        float a = A[i];
        if (!(a >= 0.0f) || isinf(a)) return OR_ERR_ARG; /* negative, NaN or inf */
        if (a > amax) amax = a;
    }
    int e = 0;
    if (amax > 0.0f) frexp((double)amax, &e); /* amax = m * 2^e, 0.5 <= m < 1 */
    for (int64_t i = 0; i < (int64_t)G * N; ++i) {
        if (amax > 0.0f)
            q[i] = (int64_t)floor(ldexp((double)A[i], OR_FIXED_POINT_BITS - e));
        else
            q[i] = 0;
    }
    if (e_out) *e_out = e;
    return OR_OK;
}

/* Up-edge term of Eq. (objective) for one layer: the co-located mass
 * sum over (g,k) with h(g) == nu(k) of q[g,k]. */
int64_t oracle_layout_score(const int64_t* q, int G, int N, const int* h, const int* nu) {
    int64_t s = 0;
    for (int g = 0; g < G; ++g)
        for (int k = 0; k < N; ++k)
            if (h[g] == nu[k]) s += q[(int64_t)g * N + k];
    return s;
}

/* ------------------------------------------------------------------------ */
/* Neuron step: exact balanced assignment (Sec. 3 "Optimiser")               */
/* ------------------------------------------------------------------------ */

/* Gain of neuron k on device l: M[k,l] = sum over heads g with h(g) == l of q[g,k]. */
static void build_gain(const int64_t* q, int G, int N, int D, const int* h, int64_t* M) {
    memset(M, 0, sizeof(int64_t) * (size_t)N * D);
    for (int g = 0; g < G; ++g)
        for (int k = 0; k < N; ++k) M[(int64_t)k * D + h[g]] += q[(int64_t)g * N + k];
}

typedef struct { int64_t key; int k; } diff_item;

/* Sort order for D = 2: larger M_k0 - M_k1 first, then lower neuron index. */
static int diff_cmp(const void* pa, const void* pb) {
    const diff_item* a = (const diff_item*)pa;
    const diff_item* b = (const diff_item*)pb;
    if (a->key != b->key) return a->key > b->key ? -1 : 1;
    return a->k < b->k ? -1 : (a->k > b->k ? 1 : 0);
}

/*
 * D = 2 reduces to a sort: sum_k M[k,nu(k)] = sum_k M[k,1] + sum_{nu(k)=0} (M[k,0]-M[k,1]),
 * so device 0 takes the N/2 largest differences.  Among equal differences the
 * lower indices go to device 0, which is the lexicographically smallest
 * optimum.  The optimum is unique iff the N/2-th and (N/2+1)-th differences
 * differ.
 */
static void lap_sort_d2(const int64_t* M, int N, int* nu, int* unique) {
    diff_item* it = (diff_item*)malloc(sizeof(diff_item) * (size_t)N);
    for (int k = 0; k < N; ++k) {
        it[k].key = M[(int64_t)k * 2 + 0] - M[(int64_t)k * 2 + 1];
        it[k].k = k;
    }
    qsort(it, (size_t)N, sizeof(diff_item), diff_cmp);
    int cap = N / 2;
    for (int i = 0; i < N; ++i) nu[it[i].k] = (i < cap) ? 0 : 1;
    if (unique) *unique = (it[cap - 1].key != it[cap].key);
    free(it);
}

/* Exchange graph of an assignment: w[a][b] = max over neurons j on device a of
 * M[j,b] - M[j,a] (the gain of moving j from a to b), with its arg; only the
 * first `upto` neurons are considered. */
static void exchange_graph(const int64_t* M, int D, const int* nu, int upto,
                           int64_t w[OR_DMAX][OR_DMAX], int arg[OR_DMAX][OR_DMAX],
                           int has[OR_DMAX][OR_DMAX]) {
    for (int a = 0; a < D; ++a)
        for (int b = 0; b < D; ++b) has[a][b] = 0;
    for (int j = 0; j < upto; ++j) {
        int a = nu[j];
        if (a < 0) continue;
        for (int b = 0; b < D; ++b) {
            if (b == a) continue;
            int64_t v = M[(int64_t)j * D + b] - M[(int64_t)j * D + a];
            if (!has[a][b] || v > w[a][b]) { w[a][b] = v; arg[a][b] = j; has[a][b] = 1; }
        }
    }
}

/*
 * Successive shortest paths, one neuron at a time (any D).  Invariant: the
 * neurons 0..k-1 are assigned with at most N/D per device at maximum total
 * gain.  Inserting neuron k along the maximum-gain path
 *     k -> a1 -> a2 -> ... -> e        (e with spare capacity)
 * (k joins a1, the best mover of a1 goes to a2, ...) keeps the invariant; the
 * path is found by Bellman-Ford on the D device nodes of the exchange graph,
 * which has no positive cycle while the invariant holds.  After N insertions
 * every device holds exactly N/D neurons and the total gain is maximal.
 */
static int lap_ssp(const int64_t* M, int N, int D, int* nu) {
    int cap = N / D;
    int count[OR_DMAX] = {0};
    for (int k = 0; k < N; ++k) nu[k] = -1;
    int64_t w[OR_DMAX][OR_DMAX];
    int arg[OR_DMAX][OR_DMAX], has[OR_DMAX][OR_DMAX];
    for (int k = 0; k < N; ++k) {
        exchange_graph(M, D, nu, k, w, arg, has);
        int64_t dist[OR_DMAX];
        int pred[OR_DMAX];
        for (int a = 0; a < D; ++a) { dist[a] = M[(int64_t)k * D + a]; pred[a] = -1; }
        for (int round = 0; round < D - 1; ++round)
            for (int a = 0; a < D; ++a)
                for (int b = 0; b < D; ++b)
                    if (b != a && has[a][b] && dist[a] + w[a][b] > dist[b]) {
                        dist[b] = dist[a] + w[a][b];
                        pred[b] = a;
                    }
        int e = -1;
        for (int a = 0; a < D; ++a)
            if (count[a] < cap && (e < 0 || dist[a] > dist[e])) e = a;
        if (e < 0) return OR_ERR_INTERNAL;
        int path[OR_DMAX + 1], len = 0, v = e;
        while (v >= 0) {
            if (len > D) return OR_ERR_INTERNAL; /* a cycle would mean a positive cycle */
            path[len++] = v;
            v = pred[v];
        }
        /* path[len-1] is the device k joins; path[i] <- path[i+1] are the moves */
        for (int i = 0; i + 1 < len; ++i) nu[arg[path[i + 1]][path[i]]] = path[i];
        nu[k] = path[len - 1];
        count[e] += 1;
    }
    for (int a = 0; a < D; ++a)
        if (count[a] != cap) return OR_ERR_INTERNAL;
    return OR_OK;
}

/* Hall's condition for completing the assignment: every set S of devices can
 * take all remaining neurons whose tight devices lie inside S. */
static int hall_ok(const int64_t* cnt_mask, const int* rem, int D) {
    for (int S = 1; S < (1 << D); ++S) {
        int64_t need = 0, have = 0;
        for (int m = 1; m < (1 << D); ++m)
            if ((m & S) == m) need += cnt_mask[m];
        for (int l = 0; l < D; ++l)
            if (S & (1 << l)) have += rem[l];
        if (need > have) return 0;
    }
    return 1;
}

/*
 * Given one optimal assignment nu_opt, list every optimum and pick the
 * lexicographically smallest (ascending = 1) or largest (ascending = 0).
 * Linear-programming duality: device prices pi with
 *     pi_b - pi_a >= max_{j on a} (M[j,b] - M[j,a])
 * (longest paths in the exchange graph) are an optimal dual, and an
 * assignment is optimal iff it is balanced and puts every neuron k on a
 * device of its tight set T_k = argmax_l (M[k,l] - pi_l).  The greedy fixes
 * k = 0,1,... to the first tight device that still admits a balanced
 * completion (Hall's condition over device subsets).
 */
static int lap_extreme(const int64_t* M, int N, int D, const int* nu_opt, int ascending, int* nu) {
    int cap = N / D;
    int64_t w[OR_DMAX][OR_DMAX];
    int arg[OR_DMAX][OR_DMAX], has[OR_DMAX][OR_DMAX];
    exchange_graph(M, D, nu_opt, N, w, arg, has);
    int64_t pi[OR_DMAX];
    for (int a = 0; a < D; ++a) pi[a] = 0;
    for (int round = 0; round < D; ++round)
        for (int a = 0; a < D; ++a)
            for (int b = 0; b < D; ++b)
                if (b != a && has[a][b] && pi[a] + w[a][b] > pi[b]) pi[b] = pi[a] + w[a][b];
    /* a further improvement would mean a positive cycle, i.e. nu_opt not optimal */
    for (int a = 0; a < D; ++a)
        for (int b = 0; b < D; ++b)
            if (b != a && has[a][b] && pi[a] + w[a][b] > pi[b]) return OR_ERR_INTERNAL;

    int* tmask = (int*)malloc(sizeof(int) * (size_t)N);
    int64_t cnt_mask[1 << OR_DMAX];
    memset(cnt_mask, 0, sizeof(cnt_mask));
    for (int k = 0; k < N; ++k) {
        int64_t best = 0;
        for (int l = 0; l < D; ++l) {
            int64_t r = M[(int64_t)k * D + l] - pi[l];
            if (l == 0 || r > best) best = r;
        }
        int m = 0;
        for (int l = 0; l < D; ++l)
            if (M[(int64_t)k * D + l] - pi[l] == best) m |= 1 << l;
        if (!(m & (1 << nu_opt[k]))) { free(tmask); return OR_ERR_INTERNAL; }
        tmask[k] = m;
        cnt_mask[m] += 1;
    }
    int rem[OR_DMAX];
    for (int l = 0; l < D; ++l) rem[l] = cap;
    int status = OR_OK;
    for (int k = 0; k < N && status == OR_OK; ++k) {
        cnt_mask[tmask[k]] -= 1;
        int chosen = -1;
        for (int i = 0; i < D; ++i) {
            int l = ascending ? i : D - 1 - i;
            if (!(tmask[k] & (1 << l))) continue;
            rem[l] -= 1;
            if (hall_ok(cnt_mask, rem, D)) { chosen = l; break; }
            rem[l] += 1;
        }
        if (chosen < 0) status = OR_ERR_INTERNAL;
        else nu[k] = chosen;
    }
    free(tmask);
    return status;
}

/*
 * Neuron step.  nu = the lexicographically smallest balanced assignment
 * maximising sum_k M[k,nu(k)], M from q and the head partition h.  *unique is
 * set to 1 when that maximiser is the only one.  general != 0 forces the
 * successive-shortest-path solver for D = 2 as well (used to cross-check the
 * sort).
 */
/* Lexicographically smallest balanced assignment maximising sum_k M[k,nu(k)]
 * for a given gain matrix M [N][D]. */
static int neuron_step_from_gain(const int64_t* M, int N, int D, int* nu, int* unique, int general) {
    int status = OR_OK;
    if (D == 2 && !general) {
        lap_sort_d2(M, N, nu, unique);
    } else {
        int* opt = (int*)malloc(sizeof(int) * (size_t)N);
        int* hi = (int*)malloc(sizeof(int) * (size_t)N);
        status = lap_ssp(M, N, D, opt);
        if (status == OR_OK) status = lap_extreme(M, N, D, opt, 1, nu);
        if (status == OR_OK && unique) {
            status = lap_extreme(M, N, D, opt, 0, hi);
            *unique = (memcmp(nu, hi, sizeof(int) * (size_t)N) == 0);
        }
        free(opt);
        free(hi);
    }
    return status;
}

int oracle_neuron_step_ex(const int64_t* q, int G, int N, int D, const int* h, int* nu,
                          int* unique, int general) {
    if (D < 2 || D > OR_DMAX || N <= 0 || N % D || G <= 0 || G > OR_GMAX) return OR_ERR_ARG;
    int64_t* M = (int64_t*)malloc(sizeof(int64_t) * (size_t)N * D);
    build_gain(q, G, N, D, h, M);
    int status = neuron_step_from_gain(M, N, D, nu, unique, general);
    free(M);
    return status;
}

int oracle_neuron_step(const int64_t* q, int G, int N, int D, const int* h, int* nu, int* unique) {
    return oracle_neuron_step_ex(q, G, N, D, h, nu, unique, 0);
}

/* Total gain sum_k M[k,nu(k)] of an assignment (for tests). */
int64_t oracle_assignment_gain(const int64_t* q, int G, int N, int D, const int* h, const int* nu) {
    int64_t s = 0;
    for (int g = 0; g < G; ++g)
        for (int k = 0; k < N; ++k)
            if (h[g] == nu[k]) s += q[(int64_t)g * N + k];
    return s;
}

/* ------------------------------------------------------------------------ */
/* Head step: exhaustive labelled partitions (Sec. 3 "Optimiser")            */
/* ------------------------------------------------------------------------ */

typedef struct {
    int G, D, cap;
    const int64_t* B; /* [G][D] */
    int cur[OR_GMAX];
    int count[OR_DMAX];
    int best[OR_GMAX];
    int64_t best_score;
    int have_best;
    int64_t visited;
} part_walk;

/* Visits the labelled balanced partitions in lexicographic order of
 * (h(0), h(1), ...); a strictly larger score replaces the best, so among
 * equal scores the lexicographically smallest h is kept. */
static void part_rec(part_walk* s, int g, int64_t partial) {
    if (g == s->G) {
        s->visited += 1;
        if (!s->have_best || partial > s->best_score) {
            s->have_best = 1;
            s->best_score = partial;
            memcpy(s->best, s->cur, sizeof(int) * (size_t)s->G);
        }
        return;
    }
    for (int l = 0; l < s->D; ++l) {
        if (s->count[l] == s->cap) continue;
        s->count[l] += 1;
        s->cur[g] = l;
        part_rec(s, g + 1, partial + s->B[g * s->D + l]);
        s->count[l] -= 1;
    }
}

/* Number of labelled balanced partitions of G groups over D devices, counted
 * by walking them (no formula). */
int64_t oracle_count_partitions(int G, int D) {
    if (D <= 0 || G <= 0 || G % D || G > OR_GMAX || D > OR_DMAX) return -1;
    int64_t B[OR_GMAX * OR_DMAX];
    memset(B, 0, sizeof(B));
    part_walk s;
    memset(&s, 0, sizeof(s));
    s.G = G; s.D = D; s.cap = G / D; s.B = B;
    part_rec(&s, 0, 0);
    return s.visited;
}

/*
 * Head step.  With B[g,l] = sum over neurons k with nu(k) == l of q[g,k], the
 * co-located mass of a partition h is sum_g B[g,h(g)]; h = the best labelled
 * balanced partition, lexicographically smallest among ties.
 */
/* Best labelled balanced partition for column sums B [G][D] (lexicographically smallest among ties). */
static void head_step_from_sums(const int64_t* B, int G, int D, int* h, int64_t* score) {
    part_walk s;
    memset(&s, 0, sizeof(s));
    s.G = G; s.D = D; s.cap = G / D; s.B = B;
    part_rec(&s, 0, 0);
    memcpy(h, s.best, sizeof(int) * (size_t)G);
    if (score) *score = s.best_score;
}

int oracle_head_step(const int64_t* q, int G, int N, int D, const int* nu, int* h, int64_t* score) {
    if (D < 2 || D > OR_DMAX || G <= 0 || G % D || G > OR_GMAX || N <= 0) return OR_ERR_ARG;
    int64_t B[OR_GMAX * OR_DMAX];
    memset(B, 0, sizeof(B));
    for (int g = 0; g < G; ++g)
        for (int k = 0; k < N; ++k) B[g * D + nu[k]] += q[(int64_t)g * N + k];
    part_walk s;
    memset(&s, 0, sizeof(s));
    s.G = G; s.D = D; s.cap = G / D; s.B = B;
    part_rec(&s, 0, 0);
    memcpy(h, s.best, sizeof(int) * (size_t)G);
    if (score) *score = s.best_score;
    return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* Coordinate ascent (Sec. 3 "Optimiser")                                    */
/* ------------------------------------------------------------------------ */

/*
 * Start from the contiguous head assignment h(g) = floor(g*D/G).  One
 * iteration = neuron step, then head step.  Stop after `iters` iterations or
 * after the first iteration whose integer score does not strictly exceed the
 * previous one (the first iteration always counts).  Outputs the state after
 * the last iteration, its integer score, score / total mass, and the number
 * of iterations run.  *all_unique is 1 when every neuron step had a unique
 * optimum.
 */
int oracle_search_layout(const float* A, int G, int N, int D, int iters, int* h, int* nu,
                         int64_t* score_q, double* score, int* iters_done, int* all_unique) {
    if (D < 2 || D > OR_DMAX || G <= 0 || G % D || G > OR_GMAX || N <= 0 || N % D || iters < 1)
        return OR_ERR_ARG;
    int64_t* q = (int64_t*)malloc(sizeof(int64_t) * (size_t)G * N);
    int status = oracle_quantize(A, G, N, q, NULL);
    if (status != OR_OK) { free(q); return status; }
    int64_t total = 0;
    for (int64_t i = 0; i < (int64_t)G * N; ++i) total += q[i];
    for (int g = 0; g < G; ++g) h[g] = (g * D) / G;
    int64_t prev = -1, J = 0;
    int done = 0, uniq_all = 1;
    for (int it = 0; it < iters; ++it) {
        int uniq = 1;
        status = oracle_neuron_step(q, G, N, D, h, nu, &uniq);
        if (status != OR_OK) break;
        uniq_all &= uniq;
        status = oracle_head_step(q, G, N, D, nu, h, &J);
        if (status != OR_OK) break;
        done = it + 1;
        if (J <= prev) break;
        prev = J;
    }
    free(q);
    if (status != OR_OK) return status;
    *score_q = J;
    *score = total > 0 ? (double)J / (double)total : 0.0;
    *iters_done = done;
    if (all_unique) *all_unique = uniq_all;
    return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* Down edge (Sec. 3 "Affinity scores")                                      */
/* ------------------------------------------------------------------------ */

/* act2[k] = sum_t alpha_k(t)^2 / r'_t^2 with alpha_k = silu(g_k) u_k, neuron k's
 * activation on token t, and r'_t the rms of the residual entering the next
 * layer's pre-norm.  act2 is overwritten. */
void oracle_down_activation(const double* X, const double* Wg, const double* Wu, const double* rms_next,
                            int64_t T, int d, int N, double* act2) {
    #pragma omp parallel for schedule(dynamic, 1)
    for (int k = 0; k < N; ++k) {
        const double* wg = Wg + (int64_t)k * d;
        const double* wu = Wu + (int64_t)k * d;
        double acc = 0.0;
        for (int64_t t = 0; t < T; ++t) {
            const double* x = X + t * d;
            double g = dot(x, wg, d);
            double u = dot(x, wu, d);
            double alpha = g / (1.0 + exp(-g)) * u;
            double r = rms_next[t];
            acc += alpha * alpha / (r * r);
        }
        act2[k] = acc;
    }
}

/* bn[g,k] = || W^qkv_g (gamma' . w^d_k) ||^2 with W^qkv_g the R rows of the next
 * layer's q/k/v projections that belong to KV group g (Wqkv [G][R][d]), gamma'
 * the next pre-norm's gain [d] and w^d_k column k of W_down [d][N]. */
void oracle_down_weight_sqnorm(const double* Wqkv, const double* gamma, const double* Wdown, int G, int R, int d,
                               int N, double* bn) {
    #pragma omp parallel for schedule(dynamic, 1)
    for (int k = 0; k < N; ++k) {
        double* v = (double*)malloc(sizeof(double) * (size_t)d);
        for (int i = 0; i < d; ++i) v[i] = gamma[i] * Wdown[(int64_t)i * N + k];
        for (int g = 0; g < G; ++g) {
            double acc = 0.0;
            for (int r = 0; r < R; ++r) {
                double b = dot(Wqkv + ((int64_t)g * R + r) * d, v, d);
                acc += b * b;
            }
            bn[(int64_t)g * N + k] = acc;
        }
        free(v);
    }
}

/* S_down[g,k] = act2[k] / T_total * bn[g,k]: the mean over tokens times ||b_gk||^2.
 * Stored [G][N], the transpose of the paper's I x G orientation. */
void oracle_down_score(const double* act2, const double* bn, int G, int N, int64_t T_total, double* S) {
    for (int g = 0; g < G; ++g)
        for (int k = 0; k < N; ++k)
            S[(int64_t)g * N + k] = act2[k] / (double)T_total * bn[(int64_t)g * N + k];
}

/* ------------------------------------------------------------------------ */
/* Whole-model objective and optimiser (Sec. 3 "Objective", "Optimiser")     */
/* ------------------------------------------------------------------------ */

#define OR_NORM_BITS 43
#define OR_NORM_PRE_BITS 40

/*
 * Unit-mass normalisation (Sec. 3 "Objective": each matrix is normalised to
 * unit mass so every edge counts equally), in exact integers:
 *     q = floor(S * 2^(40-e)),  max(S) < 2^e          (q < 2^40)
 *     n = floor(q * 2^43 / sum(q))                     (sum(n) <= 2^43)
 * (the product q * 2^43 is formed in 128 bits), so n is the matrix's share of
 * its own mass in units of 2^-43; a neuron's gain, summed over one up and one
 * down matrix, stays below 2^44.  All-zero S gives n = 0.  Returns -1 for a
 * negative or non-finite entry.
 */
int oracle_normalize_unit_mass(const float* S, int64_t count, int64_t* n) {
    float smax = 0.0f;
    for (int64_t i = 0; i < count; ++i) {
        float a = S[i];
        if (!(a >= 0.0f) || isinf(a)) return OR_ERR_ARG;
        if (a > smax) smax = a;
    }
    if (smax == 0.0f) {
        for (int64_t i = 0; i < count; ++i) n[i] = 0;
        return OR_OK;
    }
    int e = 0;
    frexp((double)smax, &e);
    uint64_t total = 0;
    for (int64_t i = 0; i < count; ++i) {
        n[i] = (int64_t)floor(ldexp((double)S[i], OR_NORM_PRE_BITS - e));
        total += (uint64_t)n[i];
    }
    for (int64_t i = 0; i < count; ++i)
        n[i] = (int64_t)((((unsigned __int128)(uint64_t)n[i]) << OR_NORM_BITS) / total);
    return OR_OK;
}

/*
 * Coordinate ascent on J(h, nu) = sum_i up_i + sum_{i<L-1} down_i over L layers,
 *   up_i   = sum over (g,k) with h_i(g) == nu_i(k)     of nU_i[g,k]
 *   down_i = sum over (g,k) with nu_i(k) == h_{i+1}(g) of nD_i[g,k]
 * (nU, nD the unit-mass forms of S_up [L][G][N] and S_down [L-1][G][N]; S_down
 * stored group-major, the transpose of the paper's I x G).
 * One iteration: every layer's neuron step given all h (gain M_kl of Sec. 3),
 * then every layer's head step given all nu (column sums over nu_i for the up
 * edge and nu_{i-1} for the down edge).  Given the other block, each step
 * maximises J exactly, so J never decreases.  Start: contiguous heads and
 * neurons in every layer.  Stop after `iters` or the first iteration (after
 * the first) without a strict increase.  J_q is J in units of 2^-43.
 *
 * Ablations (Sec. 3 "Optimiser", Table 4): move_heads[i] == 0 keeps layer i's
 * heads contiguous, move_neurons[i] == 0 its neurons (NULL = every layer
 * moves); minimize != 0 minimises J instead (the anti-optimised layout) by
 * maximising -J with the same exact steps.
 */
int oracle_chain_search_ex(const float* S_up, const float* S_down, int L, int G, int N, int D, int iters,
                           const unsigned char* move_heads, const unsigned char* move_neurons, int minimize,
                           int* h, int* nu, int64_t* J_q, double* J, int* iters_done, int* all_unique) {
    if (L < 1 || D < 2 || D > OR_DMAX || G <= 0 || G % D || G > OR_GMAX || N <= 0 || N % D || iters < 1)
        return OR_ERR_ARG;
    const int64_t GN = (int64_t)G * N;
    const int64_t sign = minimize ? -1 : 1;
    int64_t* nU = (int64_t*)malloc(sizeof(int64_t) * (size_t)(L * GN));
    int64_t* nD = (int64_t*)malloc(sizeof(int64_t) * (size_t)((L > 1 ? L - 1 : 1) * GN));
    int64_t* M = (int64_t*)malloc(sizeof(int64_t) * (size_t)N * D);
    int status = OR_OK;
    for (int i = 0; i < L && status == OR_OK; ++i) status = oracle_normalize_unit_mass(S_up + i * GN, GN, nU + i * GN);
    for (int i = 0; i + 1 < L && status == OR_OK; ++i)
        status = oracle_normalize_unit_mass(S_down + i * GN, GN, nD + i * GN);
    for (int i = 0; i < L; ++i) {
        for (int g = 0; g < G; ++g) h[i * G + g] = (g * D) / G;
        for (int k = 0; k < N; ++k) nu[(int64_t)i * N + k] = (int)(((int64_t)k * D) / N);
    }
    int64_t prev = 0, total = 0;
    int done = 0, uniq_all = 1;
    for (int it = 0; it < iters && status == OR_OK; ++it) {
        for (int i = 0; i < L && status == OR_OK; ++i) {
            if (move_neurons && !move_neurons[i]) continue;
            /* M[k,l] = sign * (up gain from h_i + down gain from h_{i+1}) */
            memset(M, 0, sizeof(int64_t) * (size_t)N * D);
            for (int g = 0; g < G; ++g)
                for (int k = 0; k < N; ++k) {
                    M[(int64_t)k * D + h[i * G + g]] += sign * nU[i * GN + (int64_t)g * N + k];
                    if (i + 1 < L) M[(int64_t)k * D + h[(i + 1) * G + g]] += sign * nD[i * GN + (int64_t)g * N + k];
                }
            int uniq = 1;
            status = neuron_step_from_gain(M, N, D, nu + (int64_t)i * N, &uniq, 0);
            uniq_all &= uniq;
        }
        if (status != OR_OK) break;
        total = 0;
        for (int i = 0; i < L; ++i) {
            /* B[g,l] = sign * (up mass of g on device l under nu_i + down mass into g under nu_{i-1}) */
            int64_t B[OR_GMAX * OR_DMAX];
            memset(B, 0, sizeof(B));
            for (int g = 0; g < G; ++g)
                for (int k = 0; k < N; ++k) {
                    B[g * D + nu[(int64_t)i * N + k]] += sign * nU[i * GN + (int64_t)g * N + k];
                    if (i > 0) B[g * D + nu[(int64_t)(i - 1) * N + k]] += sign * nD[(i - 1) * GN + (int64_t)g * N + k];
                }
            int64_t sc = 0;
            if (move_heads && !move_heads[i]) {
                for (int g = 0; g < G; ++g) sc += B[g * D + h[i * G + g]];
            } else {
                head_step_from_sums(B, G, D, h + i * G, &sc);
            }
            total += sc;
        }
        done = it + 1;
        if (it > 0 && total <= prev) break;
        prev = total;
    }
    free(nU); free(nD); free(M);
    if (status != OR_OK) return status;
    *J_q = sign * total;
    *J = ldexp((double)(sign * total), -OR_NORM_BITS);
    *iters_done = done;
    if (all_unique) *all_unique = uniq_all;
    return OR_OK;
}

int oracle_chain_search(const float* S_up, const float* S_down, int L, int G, int N, int D, int iters, int* h,
                        int* nu, int64_t* J_q, double* J, int* iters_done, int* all_unique) {
    return oracle_chain_search_ex(S_up, S_down, L, G, N, D, iters, NULL, NULL, 0, h, nu, J_q, J, iters_done,
                                  all_unique);
}

/* J of a given layout (both sums of Eq. objective), in units of 2^-43. */
int64_t oracle_chain_score(const float* S_up, const float* S_down, int L, int G, int N, const int* h, const int* nu) {
    const int64_t GN = (int64_t)G * N;
    int64_t* n = (int64_t*)malloc(sizeof(int64_t) * (size_t)GN);
    int64_t J = 0;
    for (int i = 0; i < L; ++i) {
        if (oracle_normalize_unit_mass(S_up + i * GN, GN, n) != OR_OK) { J = -1; break; }
        for (int g = 0; g < G; ++g)
            for (int k = 0; k < N; ++k)
                if (h[i * G + g] == nu[(int64_t)i * N + k]) J += n[(int64_t)g * N + k];
        if (i + 1 < L) {
            if (oracle_normalize_unit_mass(S_down + i * GN, GN, n) != OR_OK) { J = -1; break; }
            for (int g = 0; g < G; ++g)
                for (int k = 0; k < N; ++k)
                    if (nu[(int64_t)i * N + k] == h[(i + 1) * G + g]) J += n[(int64_t)g * N + k];
        }
    }
    free(n);
    return J;
}

/*
 * Per-edge co-located mass of a layout, in units of 2^-43 of each edge's own
 * unit mass: edge[2i] = up_i, edge[2i+1] = down_i (i < L-1); 2L-1 entries.
 * up_i / 2^43 is the co-located fraction of layer i's up edge (0.25 expected
 * for a random layout at four devices).  Returns the number of invalid
 * matrices (0 on success).
 */
int oracle_chain_edge_scores(const float* S_up, const float* S_down, int L, int G, int N, const int* h, const int* nu,
                             int64_t* edge) {
    const int64_t GN = (int64_t)G * N;
    int64_t* n = (int64_t*)malloc(sizeof(int64_t) * (size_t)GN);
    int bad = 0;
    for (int i = 0; i < L; ++i) {
        int64_t e = 0;
        if (oracle_normalize_unit_mass(S_up + i * GN, GN, n) != OR_OK) ++bad;
        else
            for (int g = 0; g < G; ++g)
                for (int k = 0; k < N; ++k)
                    if (h[i * G + g] == nu[(int64_t)i * N + k]) e += n[(int64_t)g * N + k];
        edge[2 * i] = e;
        if (i + 1 < L) {
            e = 0;
            if (oracle_normalize_unit_mass(S_down + i * GN, GN, n) != OR_OK) ++bad;
            else
                for (int g = 0; g < G; ++g)
                    for (int k = 0; k < N; ++k)
                        if (nu[(int64_t)i * N + k] == h[(i + 1) * G + g]) e += n[(int64_t)g * N + k];
            edge[2 * i + 1] = e;
        }
    }
    free(n);
    return bad;
}

/* ------------------------------------------------------------------------ */
/* Global optimum of one layer's up-edge objective                           */
/* ------------------------------------------------------------------------ */

/*
 * J(h, nu) of one layer is unchanged when the device labels of h and nu are
 * permuted together, so its maximum is the best exact neuron step over the
 * UNLABELLED balanced head partitions: G!/((G/D)!^D D!) of them (35 for G=8,
 * D=2; 105 for D=4).  Each is visited once through its canonical labelling
 * (a restricted growth string: a device label first appears after all
 * smaller ones), generated recursively in lexicographic order; the first
 * partition with the largest exact neuron-step value wins, with that step's
 * lexicographically smallest nu.  This is the stronger reference the ascent
 * is measured against.
 */
typedef struct {
    const int64_t* q;
    int G, N, D, cap;
    int* cur;        /* [G] labels being built */
    int* cnt;        /* [D] heads per device so far */
    int64_t* M;      /* [N][D] */
    int* nu_tmp;     /* [N] */
    int64_t best;
    int* h_best;
    int* nu_best;
    int parts;
    int status;
} global_ctx;

static void global_rec(global_ctx* c, int k, int used) {
    if (c->status != OR_OK) return;
    if (k == c->G) {
        build_gain(c->q, c->G, c->N, c->D, c->cur, c->M);
        int uniq = 1;
        int st = neuron_step_from_gain(c->M, c->N, c->D, c->nu_tmp, &uniq, 0);
        if (st != OR_OK) { c->status = st; return; }
        int64_t v = 0;
        for (int i = 0; i < c->N; ++i) v += c->M[(int64_t)i * c->D + c->nu_tmp[i]];
        ++c->parts;
        if (v > c->best) {
            c->best = v;
            memcpy(c->h_best, c->cur, sizeof(int) * (size_t)c->G);
            memcpy(c->nu_best, c->nu_tmp, sizeof(int) * (size_t)c->N);
        }
        return;
    }
    /* label l: an existing device with room, or the next unused one */
    for (int l = 0; l <= used && l < c->D; ++l) {
        if (c->cnt[l] == c->cap) continue;
        c->cur[k] = l;
        ++c->cnt[l];
        global_rec(c, k + 1, l == used ? used + 1 : used);
        --c->cnt[l];
    }
}

int oracle_global_layout(const float* A, int G, int N, int D, int* h, int* nu, int64_t* score_q, double* score,
                         int* n_parts) {
    if (D < 2 || D > OR_DMAX || G <= 0 || G % D || G > OR_GMAX || N <= 0 || N % D) return OR_ERR_ARG;
    int64_t* q = (int64_t*)malloc(sizeof(int64_t) * (size_t)G * N);
    int status = oracle_quantize(A, G, N, q, NULL);
    if (status != OR_OK) { free(q); return status; }
    int cur[OR_GMAX], cnt[OR_DMAX];
    memset(cnt, 0, sizeof(cnt));
    global_ctx c = {q, G, N, D, G / D, cur, cnt, (int64_t*)malloc(sizeof(int64_t) * (size_t)N * D),
                    (int*)malloc(sizeof(int) * (size_t)N), -1, h, nu, 0, OR_OK};
    global_rec(&c, 0, 0);
    int64_t total = 0;
    for (int64_t i = 0; i < (int64_t)G * N; ++i) total += q[i];
    if (c.status == OR_OK) {
        *score_q = c.best;
        *score = total > 0 ? (double)c.best / (double)total : 0.0;
        *n_parts = c.parts;
    }
    free(c.M); free(c.nu_tmp); free(q);
    return c.status;
}

/* ------------------------------------------------------------------------ */
/* Diagnostics                                                               */
/* ------------------------------------------------------------------------ */

/*
 * Top-group share of a layer (Sec. 5, "Where the affinity concentrates"): for
 * each neuron the largest KV group's fraction of its up-edge affinity,
 * max_g A[g,k] / sum_g A[g,k], averaged over the neurons with a non-zero
 * column (0 when there is none).  1/G when the groups contribute equally.
 */
double oracle_top_group_share(const float* A, int G, int N) {
    double acc = 0.0;
    int n = 0;
    for (int k = 0; k < N; ++k) {
        double tot = 0.0, mx = 0.0;
        for (int g = 0; g < G; ++g) {
            const double a = A[(int64_t)g * N + k];
            tot += a;
            if (a > mx) mx = a;
        }
        if (tot > 0.0) { acc += mx / tot; ++n; }
    }
    return n ? acc / n : 0.0;
}

/* ------------------------------------------------------------------------ */
/* Producer and layout application                                           */
/* ------------------------------------------------------------------------ */

/*
 * Head writes into the FFN input (Sec. 3): attention head h's output a_h
 * (columns h*hd .. h*hd+hd-1 of attn [T, Hq*hd]) enters the residual as
 * a_h W_o^(h)T (the matching columns of W_o [d, Hq*hd]), and reaches the FFN
 * input through its pre-norm as gamma . (a_h W_o^(h)T) / r with r the rms of
 * the residual at that token (held fixed).  Row j of C sums the q_per_row
 * consecutive heads j*q_per_row ..; q_per_row = 1 gives one row per query
 * head, q_per_row = query heads per KV group gives the group's write.
 *   C [Hq/q_per_row, T, d] fp64, overwritten.
 */
void oracle_head_writes(const double* attn, const double* Wo, const double* gamma, const double* rms, int64_t T,
                        int d, int Hq, int hd, int q_per_row, double* C) {
    const int K = Hq * hd, rows = Hq / q_per_row, Kj = q_per_row * hd;
    #pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < T; ++t)
        for (int j = 0; j < rows; ++j)
            for (int i = 0; i < d; ++i) {
                double s = 0.0;
                for (int c = j * Kj; c < (j + 1) * Kj; ++c) s += attn[t * K + c] * Wo[(int64_t)i * K + c];
                C[((int64_t)j * T + t) * d + i] = gamma[i] * s / rms[t];
            }
}

/*
 * The order that groups items by device: order[p] = the item at position p
 * when items are listed device by device, each device's items in increasing
 * index.  For a balanced layout, positions p*D/n .. of the permuted model are
 * device floor(p D / n)'s contiguous shard.  Returns OR_ERR_ARG on a label
 * outside [0, D).
 */
int oracle_layout_order(const int* labels, int n, int D, int* order) {
    for (int k = 0; k < n; ++k)
        if (labels[k] < 0 || labels[k] >= D) return OR_ERR_ARG;
    int pos = 0;
    for (int l = 0; l < D; ++l)
        for (int k = 0; k < n; ++k)
            if (labels[k] == l) order[pos++] = k;
    return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* Textbook Hungarian method (cross-check only)                              */
/* ------------------------------------------------------------------------ */

/*
 * Maximum-weight perfect matching of an n x n integer matrix W (row-major) by
 * the O(n^3) Hungarian method with row/column potentials (Kuhn 1955; the
 * shortest-augmenting-path form).  Returns the optimal total; row_to_col
 * receives the matching.  Costs are the negated weights.
 */
int64_t oracle_hungarian_max(const int64_t* W, int n, int* row_to_col) {
    const int64_t INF = INT64_MAX / 4;
    int64_t* u = (int64_t*)calloc((size_t)n + 1, sizeof(int64_t));
    int64_t* v = (int64_t*)calloc((size_t)n + 1, sizeof(int64_t));
    int* p = (int*)calloc((size_t)n + 1, sizeof(int));   /* p[col] = row matched to col (1-based) */
    int* way = (int*)calloc((size_t)n + 1, sizeof(int));
    int64_t* minv = (int64_t*)malloc(sizeof(int64_t) * ((size_t)n + 1));
    char* used = (char*)malloc((size_t)n + 1);
    for (int i = 1; i <= n; ++i) {
        p[0] = i;
        int j0 = 0;
        for (int j = 0; j <= n; ++j) { minv[j] = INF; used[j] = 0; }
        do {
            used[j0] = 1;
            int i0 = p[j0], j1 = 0;
            int64_t delta = INF;
            for (int j = 1; j <= n; ++j) {
                if (used[j]) continue;
                int64_t cost = -W[(int64_t)(i0 - 1) * n + (j - 1)];
                int64_t cur = cost - u[i0] - v[j];
                if (cur < minv[j]) { minv[j] = cur; way[j] = j0; }
                if (minv[j] < delta) { delta = minv[j]; j1 = j; }
            }
            for (int j = 0; j <= n; ++j) {
                if (used[j]) { u[p[j]] += delta; v[j] -= delta; }
                else minv[j] -= delta;
            }
            j0 = j1;
        } while (p[j0] != 0);
        do {
            int j1 = way[j0];
            p[j0] = p[j1];
            j0 = j1;
        } while (j0);
    }
    int64_t total = 0;
    for (int j = 1; j <= n; ++j) {
        row_to_col[p[j] - 1] = j - 1;
        total += W[(int64_t)(p[j] - 1) * n + (j - 1)];
    }
    free(u); free(v); free(p); free(way); free(minv); free(used);
    return total;
}
