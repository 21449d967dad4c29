/*
 * PrefixPlace CPU oracle -- TEST INFRASTRUCTURE, NOT PART OF THE PRODUCT.
 *
 * A plain, slow, deliberately unoptimised restatement of the planner in
 * "PrefixPlace: Provable Prefix Key--Value Placement for LLM Serving under
 * Heterogeneous Compute and Transfer Costs" (arXiv 2608.01655).  Only the
 * test suite, the smoke check and the CPU-baseline leg of the benchmark may
 * load this library.  It shares no code, header, table or helper with the
 * CUDA library under paper_2608_01655_gb300/; neither includes the other.
 *
 * Everything is exact int64 arithmetic: costs are integer microseconds and
 * demand is an integer request count, so the paper's tolerance epsilon
 * (Section IV-C) is 0 and "strict improvement" is a plain ">".
 *
 * Notation follows the paper:
 *   Lambda_m(b)  demand of requester m on chunk b            (Section III-A)
 *   w_m(b)       recomputation cost  ("recompute" below)      (Section II-B)
 *   f_m(b)       fetch cost, requester-side                   (Eq. 1)
 *   f_{m<-h}(b)  fetch cost from holder h, source-dependent   (Section III-C)
 *   k_m          budget of worker m in slots
 * Chunks may occupy more than one slot ("weight"); the take branch of Eq. 9
 * then spends w_i slots and needs j >= w_i.  The paper's equal-sized chunks
 * are the special case weight == 1.
 *
 * Functions and the passage each one follows:
 *   or_preorder        Section IV-A: preorder b_1..b_n and next(i)
 *   or_objective       Lemma 1 / Eq. 4 (mode 0) and Eq. 6 (mode 1)
 *   or_marginal        Eq. 10 (mode 0) and Prop. 1 / Eq. 7 (mode 1)
 *   or_rooted_dp       Eq. 9, Theorem 1, Algorithm 1 procedure RootedDP
 *   or_standalone      standalone score (Section IV-C, Algorithm 1)
 *   or_default_orders  start orders (Section IV-C); permutations by SplitMix64
 *   or_safeguards      Algorithm 1's safeguard candidates (requester-side):
 *                      Independent, Popularity, LocalDedup (Sections IV-C, V-A)
 *   or_plan            Algorithm 1 procedure PrefixPlace (greedy, refinement,
 *                      starts, and the safeguard candidates when asked for)
 *   or_replan          epoch update with the amortisation rule (Section IV-D,
 *                      RQ5 of Section V)
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <pthread.h>

typedef struct {
    int32_t n;                 /* chunks */
    int32_t W;                 /* workers (the paper's M) */
    int32_t mode;              /* 0 requester-side f_m(b), 1 source-dependent f_{m<-h}(b) */
    const int32_t *parent;     /* [n]; -1 = child of the implicit no-cost dummy root */
    const int32_t *weight;     /* [n]; slots per chunk (>= 1) */
    const int64_t *demand;     /* [W][n]  Lambda_m(b) */
    const int64_t *recompute;  /* [W][n]  w_m(b) */
    const int64_t *transfer;   /* mode 0: [W][n] f_m(b);  mode 1: [W][W][n], f_{m<-h}(b) at [h][m][b] */
    const int32_t *budget;     /* [W]  k_m */
} or_inst;

static int64_t imax64(int64_t a, int64_t b) { return a > b ? a : b; }
static int64_t imin64(int64_t a, int64_t b) { return a < b ? a : b; }
static int64_t pos64(int64_t x) { return x > 0 ? x : 0; }          /* [x]_+ */

#define LAM(I, m, b) ((I)->demand[(size_t)(m) * (I)->n + (b)])
#define WCOST(I, m, b) ((I)->recompute[(size_t)(m) * (I)->n + (b)])
#define FREQ(I, m, b) ((I)->transfer[(size_t)(m) * (I)->n + (b)])
#define FPAIR(I, h, m, b) ((I)->transfer[((size_t)(h) * (I)->W + (m)) * (I)->n + (b)])
#define HOLDS(P, I, m, b) ((P)[(size_t)(m) * (I)->n + (b)] != 0)

/* ------------------------------------------------------------------------ */
/* Section IV-A: number the nodes in preorder and compute next(i).          */
/* Roots (parent -1) first, children visited in ascending node id.          */
/* order[i] = node at 0-based position i; next[i] = first position after    */
/* the subtree of order[i].  Returns 0, or -1 if parent[] is not a forest.   */
/* ------------------------------------------------------------------------ */
int or_preorder(int32_t n, const int32_t *parent, int32_t *order, int32_t *next)
{
    if (n < 0) return -1;
    if (n == 0) return 0;
    int32_t *nchild = calloc((size_t)n + 1, sizeof(int32_t));
    int32_t *first = calloc((size_t)n + 2, sizeof(int32_t));
    int32_t *kids = malloc(sizeof(int32_t) * (size_t)n);
    int32_t *fill = calloc((size_t)n + 1, sizeof(int32_t));
    int32_t *stack = malloc(sizeof(int32_t) * (size_t)n);
    int32_t *pos = malloc(sizeof(int32_t) * (size_t)n);
    int32_t *size = malloc(sizeof(int32_t) * (size_t)n);
    int rc = 0;
    /* slot n holds the children of the dummy root */
    for (int32_t v = 0; v < n; ++v) {
        int32_t p = parent[v];
        if (p < -1 || p >= n || p == v) { rc = -1; goto done; }
        nchild[p < 0 ? n : p]++;
    }
    for (int32_t u = 0; u <= n; ++u) first[u + 1] = first[u] + nchild[u];
    for (int32_t v = 0; v < n; ++v) {            /* ascending id -> sorted lists */
        int32_t u = parent[v] < 0 ? n : parent[v];
        kids[first[u] + fill[u]++] = v;
    }
    int32_t top = 0, cnt = 0;
    for (int32_t c = first[n + 1] - 1; c >= first[n]; --c) stack[top++] = kids[c];
    while (top > 0) {
        int32_t v = stack[--top];
        pos[v] = cnt;
        order[cnt++] = v;
        for (int32_t c = first[v + 1] - 1; c >= first[v]; --c) stack[top++] = kids[c];
    }
    if (cnt != n) { rc = -1; goto done; }        /* a cycle keeps nodes unreachable */
    for (int32_t v = 0; v < n; ++v) size[v] = 1;
    for (int32_t i = n - 1; i >= 0; --i) {
        int32_t v = order[i];
        if (parent[v] >= 0) size[parent[v]] += size[v];
    }
    for (int32_t i = 0; i < n; ++i) next[i] = i + size[order[i]];
done:
    free(nchild); free(first); free(kids); free(fill); free(stack); free(pos); free(size);
    return rc;
}

/* ------------------------------------------------------------------------ */
/* Eq. 2: a_m(b) = Lambda_m(b) * min{w_m(b), f_m(b)}                         */
/* Eq. 3: Delta(b) = sum_m Lambda_m(b) [w_m(b) - f_m(b)]_+                   */
/* Eq. 5: q_{m<-h}(b) = w_m(b) if h == m else [w_m(b) - f_{m<-h}(b)]_+       */
/* ------------------------------------------------------------------------ */
static int64_t eq2_local_value(const or_inst *I, int32_t m, int32_t b)
{
    return LAM(I, m, b) * imin64(WCOST(I, m, b), FREQ(I, m, b));
}

static int64_t eq3_coverage_value(const or_inst *I, int32_t b)
{
    int64_t s = 0;
    for (int32_t m = 0; m < I->W; ++m) s += LAM(I, m, b) * pos64(WCOST(I, m, b) - FREQ(I, m, b));
    return s;
}

static int64_t eq5_pair_saving(const or_inst *I, int32_t m, int32_t h, int32_t b)
{
    if (h == m) return WCOST(I, m, b);
    return pos64(WCOST(I, m, b) - FPAIR(I, h, m, b));
}

/* Lemma 1 / Eq. 4: F(T) = sum_m sum_{b in T_m} a_m(b) + sum_{b in U_m T_m} Delta(b). */
int64_t or_objective_F(const or_inst *I, const uint8_t *placement)
{
    int64_t total = 0;
    for (int32_t b = 0; b < I->n; ++b) {
        int covered = 0;
        for (int32_t m = 0; m < I->W; ++m)
            if (HOLDS(placement, I, m, b)) { total += eq2_local_value(I, m, b); covered = 1; }
        if (covered) total += eq3_coverage_value(I, b);
    }
    return total;
}

/* Eq. 6: F_pair(T) = sum_b sum_m Lambda_m(b) max_{h in H_b(T)} q_{m<-h}(b); max over {} = 0. */
int64_t or_objective_Fpair(const or_inst *I, const uint8_t *placement)
{
    int64_t total = 0;
    for (int32_t b = 0; b < I->n; ++b)
        for (int32_t m = 0; m < I->W; ++m) {
            int64_t best = 0;
            for (int32_t h = 0; h < I->W; ++h)
                if (HOLDS(placement, I, h, b)) best = imax64(best, eq5_pair_saving(I, m, h, b));
            total += LAM(I, m, b) * best;
        }
    return total;
}

int64_t or_objective(const or_inst *I, const uint8_t *placement)
{
    return I->mode == 0 ? or_objective_F(I, placement) : or_objective_Fpair(I, placement);
}

/* ------------------------------------------------------------------------ */
/* Worker h's exact node marginals against the other workers' placements.   */
/* mode 0, Eq. 10: p_h(b) = a_h(b) + 1{b not in U} Delta(b), U = U_{l!=h} T_l */
/* mode 1, Eq. 7:  p_h(b) = sum_m Lambda_m(b) [q_{m<-h}(b) - v_m^{(-h)}(b)]_+ */
/*   with v_m^{(-h)}(b) = max over current holders l != h of q_{m<-l}(b)     */
/*   (0 when there is none), recomputed here from w and f directly.          */
/* T_h itself is ignored, as Algorithm 1 empties it before the update.       */
/* ------------------------------------------------------------------------ */
void or_marginal(const or_inst *I, int32_t h, const uint8_t *placement, int64_t *profit)
{
    for (int32_t b = 0; b < I->n; ++b) {
        if (I->mode == 0) {
            int in_U = 0;
            for (int32_t l = 0; l < I->W; ++l)
                if (l != h && HOLDS(placement, I, l, b)) in_U = 1;
            profit[b] = eq2_local_value(I, h, b) + (in_U ? 0 : eq3_coverage_value(I, b));
        } else {
            int64_t s = 0;
            for (int32_t m = 0; m < I->W; ++m) {
                int64_t v = 0;
                for (int32_t l = 0; l < I->W; ++l)
                    if (l != h && HOLDS(placement, I, l, b)) v = imax64(v, eq5_pair_saving(I, m, l, b));
                s += LAM(I, m, b) * pos64(eq5_pair_saving(I, m, h, b) - v);
            }
            profit[b] = s;
        }
    }
}

/* ------------------------------------------------------------------------ */
/* RootedDP (Eq. 9, Theorem 1, Algorithm 1).  With 0-based positions         */
/* i = 0..n-1 and row n the boundary D[n][j] = 0:                            */
/*   D[i][0] = 0;  for j >= 1:                                               */
/*   D[i][j] = max{ D[next(i)][j],  p(b_i) + D[i+1][j - w_i] }               */
/* where the take branch needs j >= w_i (w_i == 1 is the paper's case).      */
/* The branch is recorded as "take" only when it is strictly larger, and    */
/* the backtrack starts at (0, k).  Returns D[0][k]; chosen[] is by node id. */
/*                                                                          */
/* variant 0: the whole (n+1) x (k+1) table of Eq. 9 and one decision per  */
/*            cell (Theorem 1's O(nk) time and memory).                     */
/* variant 1: the same recurrence; a row is freed after its last reader     */
/*            (min{i : next(i) = r or i + 1 = r}), decisions kept as bits.  */
/* variant -1: 0 when the table is at most 64 MiB, else 1.                  */
/* ------------------------------------------------------------------------ */
static int64_t rooted_dp_table(int32_t n, const int32_t *order, const int32_t *next,
                               const int32_t *weight, const int64_t *profit, int32_t k,
                               uint8_t *chosen)
{
    size_t K1 = (size_t)k + 1;
    int64_t *D = calloc(((size_t)n + 1) * K1, sizeof(int64_t));   /* row n stays 0 */
    uint8_t *take = calloc((size_t)n * K1 + 1, 1);
    for (int32_t i = n - 1; i >= 0; --i) {
        int32_t b = order[i];
        int32_t wi = weight[b];
        int64_t pi = profit[b];
        D[(size_t)i * K1 + 0] = 0;
        for (int32_t j = 1; j <= k; ++j) {
            int64_t s = D[(size_t)next[i] * K1 + j];                  /* skip b_i and its subtree */
            int64_t best = s;
            if (j >= wi) {
                int64_t t = pi + D[((size_t)i + 1) * K1 + (j - wi)];   /* take b_i */
                if (t > s) { best = t; take[(size_t)i * K1 + j] = 1; }
            }
            D[(size_t)i * K1 + j] = best;
        }
    }
    int64_t result = n > 0 ? D[k] : 0;
    int32_t i = 0, j = k;
    while (i < n) {                                                    /* backtrack */
        if (take[(size_t)i * K1 + j]) { chosen[order[i]] = 1; j -= weight[order[i]]; i += 1; }
        else i = next[i];
    }
    free(D); free(take);
    return result;
}

static int64_t rooted_dp_rows(int32_t n, const int32_t *order, const int32_t *next,
                              const int32_t *weight, const int64_t *profit, int32_t k,
                              uint8_t *chosen)
{
    size_t K1 = (size_t)k + 1;
    size_t words = (K1 + 63) / 64;
    int64_t **row = calloc((size_t)n + 1, sizeof(int64_t *));
    int32_t *last_use = malloc(sizeof(int32_t) * ((size_t)n + 1));
    uint64_t *take = calloc((size_t)n * words + 1, sizeof(uint64_t));
    for (int32_t r = 0; r <= n; ++r) last_use[r] = -1;
    for (int32_t i = n - 1; i >= 0; --i) {      /* smallest reader wins: it is processed last */
        last_use[i + 1] = i;
        last_use[next[i]] = i;
    }
    row[n] = calloc(K1, sizeof(int64_t));
    for (int32_t i = n - 1; i >= 0; --i) {
        int32_t b = order[i];
        int32_t wi = weight[b];
        int64_t pi = profit[b];
        int64_t *Di = calloc(K1, sizeof(int64_t));
        const int64_t *Dn = row[next[i]];
        const int64_t *D1 = row[i + 1];
        for (int32_t j = 1; j <= k; ++j) {
            int64_t s = Dn[j];
            int64_t best = s;
            if (j >= wi) {
                int64_t t = pi + D1[j - wi];
                if (t > s) { best = t; take[(size_t)i * words + j / 64] |= (uint64_t)1 << (j % 64); }
            }
            Di[j] = best;
        }
        row[i] = Di;
        if (last_use[i + 1] == i) { free(row[i + 1]); row[i + 1] = NULL; }
        if (next[i] != i + 1 && last_use[next[i]] == i) { free(row[next[i]]); row[next[i]] = NULL; }
    }
    int64_t result = n > 0 ? row[0][k] : 0;
    int32_t i = 0, j = k;
    while (i < n) {
        if ((take[(size_t)i * words + j / 64] >> (j % 64)) & 1) {
            chosen[order[i]] = 1; j -= weight[order[i]]; i += 1;
        } else i = next[i];
    }
    for (int32_t r = 0; r <= n; ++r) free(row[r]);
    free(row); free(last_use); free(take);
    return result;
}

int64_t or_rooted_dp_pre(int32_t n, const int32_t *order, const int32_t *next,
                         const int32_t *weight, const int64_t *profit, int32_t k,
                         uint8_t *chosen, int variant)
{
    memset(chosen, 0, (size_t)n);
    if (n == 0 || k <= 0) return 0;
    if (variant < 0)
        variant = (((size_t)n + 1) * ((size_t)k + 1) * sizeof(int64_t) <= ((size_t)64 << 20)) ? 0 : 1;
    return variant == 0 ? rooted_dp_table(n, order, next, weight, profit, k, chosen)
                        : rooted_dp_rows(n, order, next, weight, profit, k, chosen);
}

/* Returns D[1][k] (the optimum), or INT64_MIN if parent[] is not a forest. */
int64_t or_rooted_dp(int32_t n, const int32_t *parent, const int32_t *weight,
                     const int64_t *profit, int32_t k, uint8_t *chosen, int variant)
{
    int32_t *order = malloc(sizeof(int32_t) * ((size_t)n + 1));
    int32_t *next = malloc(sizeof(int32_t) * ((size_t)n + 1));
    int64_t r;
    if (or_preorder(n, parent, order, next) != 0) r = INT64_MIN;
    else r = or_rooted_dp_pre(n, order, next, weight, profit, k, chosen, variant);
    free(order); free(next);
    return r;
}

/* ------------------------------------------------------------------------ */
/* Standalone score of worker h: its exact single-worker optimum when no    */
/* other worker holds anything (U = {} in Eq. 10; no holders in Eq. 7).     */
/* ------------------------------------------------------------------------ */
int or_standalone(const or_inst *I, int64_t *score)
{
    int32_t n = I->n;
    int32_t *order = malloc(sizeof(int32_t) * ((size_t)n + 1));
    int32_t *next = malloc(sizeof(int32_t) * ((size_t)n + 1));
    if (or_preorder(n, I->parent, order, next) != 0) { free(order); free(next); return -1; }
    uint8_t *empty = calloc((size_t)I->W * n + 1, 1);
    int64_t *p = malloc(sizeof(int64_t) * ((size_t)n + 1));
    uint8_t *ch = malloc((size_t)n + 1);
    for (int32_t h = 0; h < I->W; ++h) {
        or_marginal(I, h, empty, p);
        score[h] = or_rooted_dp_pre(n, order, next, I->weight, p, I->budget[h], ch, -1);
    }
    free(order); free(next); free(empty); free(p); free(ch);
    return 0;
}

/* SplitMix64 (Steele, Lea and Flood, OOPSLA 2014): state += golden gamma,  */
/* then the variant-13 mix of the state.                                     */
static uint64_t splitmix64_next(uint64_t *state)
{
    uint64_t z = (*state += 0x9E3779B97F4A7C15ULL);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* The first `count` outputs of SplitMix64 from state `seed` (exposed so the */
/* tests can check the generator against its published outputs).             */
void or_splitmix64(uint64_t seed, int32_t count, uint64_t *out)
{
    uint64_t st = seed;
    for (int32_t i = 0; i < count; ++i) out[i] = splitmix64_next(&st);
}

/* Start orders (Section IV-C).  S == 1: identity.  Otherwise start 0 is     */
/* the standalone-score order (descending, ties to the lower worker id),     */
/* start 1 its reverse, and start s >= 2 the Fisher-Yates shuffle of the     */
/* identity driven by SplitMix64 seeded with s (j = next() mod (i + 1),      */
/* i = W-1 down to 1).                                                      */
int or_default_orders(const or_inst *I, int32_t S, int32_t *orders)
{
    int32_t W = I->W;
    for (int32_t s = 0; s < S; ++s)
        for (int32_t t = 0; t < W; ++t) orders[(size_t)s * W + t] = t;
    if (S <= 1) return 0;
    int64_t *score = malloc(sizeof(int64_t) * (size_t)W);
    if (or_standalone(I, score) != 0) { free(score); return -1; }
    int32_t *o = orders;
    for (int32_t a = 0; a < W; ++a)                  /* insertion sort: stable, plain */
        for (int32_t c = a; c > 0; --c) {
            int32_t x = o[c - 1], y = o[c];
            if (score[y] > score[x]) { o[c - 1] = y; o[c] = x; } else break;
        }
    for (int32_t t = 0; t < W; ++t) orders[(size_t)W + t] = o[W - 1 - t];
    for (int32_t s = 2; s < S; ++s) {
        int32_t *q = orders + (size_t)s * W;
        uint64_t st = (uint64_t)s;
        for (int32_t i = W - 1; i >= 1; --i) {
            int32_t j = (int32_t)(splitmix64_next(&st) % (uint64_t)(i + 1));
            int32_t tmp = q[i]; q[i] = q[j]; q[j] = tmp;
        }
    }
    free(score);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* One start of the planner (Section IV-C) for the worker sequence pi.       */
/* Every target begins empty.  Greedy pass (Theorem 3): the workers of pi,   */
/* one after another, each get the exact best prefix-complete target for    */
/* their marginals (Eq. 10 / Eq. 7) given what the workers before them      */
/* hold; the workers after them still hold nothing.  Refinement: at most R  */
/* passes over pi; in a pass each worker's target is solved again against   */
/* the others' current targets (its own is dropped first) and kept only if */
/* the objective, evaluated from scratch on the whole placement (Eq. 4 /    */
/* Eq. 6) right before and after, strictly grows; otherwise the old target  */
/* comes back.  A pass that kept no new target ends the start.              */
/* ------------------------------------------------------------------------ */
typedef struct {
    const or_inst *I;
    const int32_t *order, *next;
    const int32_t *pi;           /* [W] */
    int32_t R;
    uint8_t *T;                  /* [W][n] out */
    int64_t objective;           /* out */
    int32_t sweeps;              /* refinement sweeps run */
    int32_t accepted;            /* accepted refinement updates */
    int64_t cells;               /* DP cells evaluated, sum of n * k_h */
} or_start;

static void run_start(or_start *st)
{
    const or_inst *I = st->I;
    int32_t n = I->n, W = I->W;
    int64_t *p = malloc(sizeof(int64_t) * ((size_t)n + 1));
    uint8_t *Tnew = malloc((size_t)n + 1);
    uint8_t *Told = malloc((size_t)n + 1);
    memset(st->T, 0, (size_t)W * n);
    st->sweeps = 0; st->accepted = 0; st->cells = 0;
    for (int32_t t = 0; t < W; ++t) {                              /* WorkerGreedy */
        int32_t h = st->pi[t];
        or_marginal(I, h, st->T, p);
        or_rooted_dp_pre(n, st->order, st->next, I->weight, p, I->budget[h], Tnew, -1);
        st->cells += (int64_t)n * I->budget[h];
        memcpy(st->T + (size_t)h * n, Tnew, (size_t)n);
    }
    for (int32_t r = 0; r < st->R; ++r) {                          /* coordinate refinement */
        int improved = 0;
        st->sweeps++;
        for (int32_t t = 0; t < W; ++t) {
            int32_t h = st->pi[t];
            uint8_t *Th = st->T + (size_t)h * n;
            memcpy(Told, Th, (size_t)n);
            int64_t g_old = or_objective(I, st->T);
            memset(Th, 0, (size_t)n);
            or_marginal(I, h, st->T, p);
            or_rooted_dp_pre(n, st->order, st->next, I->weight, p, I->budget[h], Tnew, -1);
            st->cells += (int64_t)n * I->budget[h];
            memcpy(Th, Tnew, (size_t)n);
            int64_t g_new = or_objective(I, st->T);
            if (g_new > g_old) { improved = 1; st->accepted++; }
            else memcpy(Th, Told, (size_t)n);
        }
        if (!improved) break;
    }
    st->objective = or_objective(I, st->T);
    free(p); free(Tnew); free(Told);
}

/* ------------------------------------------------------------------------ */
/* Safeguard candidates (Algorithm 1, requester-side objective only; the    */
/* comparators of Section V-A).  Every worker's target is RootedDP(p, k_m)  */
/* with                                                                      */
/*   Independent  p(b) = Lambda_m(b) w_m(b): local demand weighted by       */
/*                recomputation cost, cross-worker reuse ignored;           */
/*   Popularity   p(b) = Lambda_m(b): local demand alone;                   */
/*   LocalDedup   workers in index order; a chunk that an earlier worker     */
/*                already holds is worth only the local value a_m(b) of     */
/*                Eq. 2, any other chunk Lambda_m(b) w_m(b) -- the worker's  */
/*                own saving from the first copy, not the requester-wide     */
/*                Delta(b) of Eq. 3.                                         */
/* placement: [3][W][n] out (Independent, Popularity, LocalDedup);           */
/* objective: [3] out, Eq. 4.  Returns 0; -1 if parent[] is not a forest;    */
/* -2 in the source-dependent mode (Algorithm 1 adds them only for the       */
/* requester-side objective).                                                */
/* ------------------------------------------------------------------------ */
int or_safeguards(const or_inst *I, uint8_t *placement, int64_t *objective)
{
    if (I->mode != 0) return -2;
    int32_t n = I->n, W = I->W;
    int32_t *order = malloc(sizeof(int32_t) * ((size_t)n + 1));
    int32_t *next = malloc(sizeof(int32_t) * ((size_t)n + 1));
    if (or_preorder(n, I->parent, order, next) != 0) { free(order); free(next); return -1; }
    int64_t *p = malloc(sizeof(int64_t) * ((size_t)n + 1));
    uint8_t *held = calloc((size_t)n + 1, 1);     /* LocalDedup: held by an earlier worker */
    memset(placement, 0, (size_t)3 * W * n);
    for (int32_t c = 0; c < 3; ++c) {
        uint8_t *X = placement + (size_t)c * W * n;
        for (int32_t m = 0; m < W; ++m) {
            for (int32_t b = 0; b < n; ++b) {
                if (c == 0) p[b] = LAM(I, m, b) * WCOST(I, m, b);
                else if (c == 1) p[b] = LAM(I, m, b);
                else p[b] = held[b] ? eq2_local_value(I, m, b) : LAM(I, m, b) * WCOST(I, m, b);
            }
            or_rooted_dp_pre(n, order, next, I->weight, p, I->budget[m], X + (size_t)m * n, -1);
            if (c == 2)
                for (int32_t b = 0; b < n; ++b) held[b] |= X[(size_t)m * n + b];
        }
        objective[c] = or_objective(I, X);
    }
    free(order); free(next); free(p); free(held);
    return 0;
}

typedef struct {
    or_start *starts;
    int32_t S;
    int32_t next_job;
    pthread_mutex_t lock;
} or_pool;

static void *pool_worker(void *arg)
{
    or_pool *pool = (or_pool *)arg;
    for (;;) {
        pthread_mutex_lock(&pool->lock);
        int32_t s = pool->next_job++;
        pthread_mutex_unlock(&pool->lock);
        if (s >= pool->S) return NULL;
        run_start(&pool->starts[s]);
    }
}

/* orders: [S][W] or NULL (then or_default_orders).  placement: [W][n] out, */
/* the best candidate's targets (highest objective, ties to the lowest      */
/* index).  With safeguards != 0 and the requester-side objective, the      */
/* Independent, Popularity and LocalDedup placements join the candidates as */
/* indices S, S+1, S+2 (Algorithm 1), and safeguard_obj [3] receives their  */
/* objectives (else it is left alone).  per_start_obj / sweeps / accepted:  */
/* [S] out or NULL.  Returns the best candidate index, or -1 on an invalid  */
/* tree.                                                                     */
int32_t or_plan(const or_inst *I, int32_t S, const int32_t *orders, int32_t R, int32_t n_threads,
                uint8_t *placement, int64_t *objective, int64_t *per_start_obj,
                int32_t *per_start_sweeps, int32_t *per_start_accepted, int64_t *cells_out,
                int safeguards, int64_t *safeguard_obj)
{
    int32_t n = I->n, W = I->W;
    int32_t *order = malloc(sizeof(int32_t) * ((size_t)n + 1));
    int32_t *next = malloc(sizeof(int32_t) * ((size_t)n + 1));
    if (or_preorder(n, I->parent, order, next) != 0) { free(order); free(next); return -1; }
    int32_t *ord = malloc(sizeof(int32_t) * (size_t)S * W + 1);
    if (orders) memcpy(ord, orders, sizeof(int32_t) * (size_t)S * W);
    else if (or_default_orders(I, S, ord) != 0) { free(order); free(next); free(ord); return -1; }
    or_start *st = calloc((size_t)S, sizeof(or_start));
    uint8_t *T = calloc((size_t)S * W * n + 1, 1);
    for (int32_t s = 0; s < S; ++s) {
        st[s].I = I; st[s].order = order; st[s].next = next;
        st[s].pi = ord + (size_t)s * W; st[s].R = R;
        st[s].T = T + (size_t)s * W * n;
    }
    if (n_threads < 1) n_threads = 1;
    if (n_threads > S) n_threads = S;
    or_pool pool = { st, S, 0, PTHREAD_MUTEX_INITIALIZER };
    pthread_t *th = malloc(sizeof(pthread_t) * (size_t)n_threads);
    for (int32_t t = 0; t < n_threads; ++t) pthread_create(&th[t], NULL, pool_worker, &pool);
    for (int32_t t = 0; t < n_threads; ++t) pthread_join(th[t], NULL);
    int32_t best = 0;
    int64_t cells = 0;
    for (int32_t s = 0; s < S; ++s) {
        if (st[s].objective > st[best].objective) best = s;
        if (per_start_obj) per_start_obj[s] = st[s].objective;
        if (per_start_sweeps) per_start_sweeps[s] = st[s].sweeps;
        if (per_start_accepted) per_start_accepted[s] = st[s].accepted;
        cells += st[s].cells;
    }
    if (!orders && S > 1)                      /* the standalone-score DPs of the default orders */
        for (int32_t m = 0; m < W; ++m) cells += (int64_t)n * I->budget[m];
    memcpy(placement, st[best].T, (size_t)W * n);
    *objective = st[best].objective;
    if (safeguards && I->mode == 0) {
        uint8_t *X = malloc((size_t)3 * W * n + 1);
        int64_t so[3];
        or_safeguards(I, X, so);
        for (int32_t c = 0; c < 3; ++c) {
            if (safeguard_obj) safeguard_obj[c] = so[c];
            if (so[c] > *objective) {
                *objective = so[c];
                best = S + c;
                memcpy(placement, X + (size_t)c * W * n, (size_t)W * n);
            }
        }
        for (int32_t c = 0; c < 3; ++c)        /* one DP per worker and candidate */
            for (int32_t m = 0; m < W; ++m) cells += (int64_t)n * I->budget[m];
        free(X);
    }
    if (cells_out) *cells_out = cells;
    free(th); free(st); free(T); free(order); free(next); free(ord);
    return best;
}

/* ------------------------------------------------------------------------ */
/* Epoch update (Section IV-D; the amortisation rule and break-even         */
/* requests of RQ5, Section V).  Under the refreshed instance I (new demand) */
/* the planner evaluates the incumbent T_old and a reoptimised target T_new  */
/* (or_plan with S starts and R sweeps).  Making T_new resident costs, for   */
/* every chunk b that worker m holds in T_new but not in T_old, what the     */
/* materialisation rule of Section III-A charges requester m for b under    */
/* the incumbent: the cheaper of recomputing and fetching from a worker that */
/* holds b in T_old, or recomputing when none does.  G is a saving per epoch */
/* of epoch_requests requests, so T_new is adopted iff                        */
/*   (G(T_new) - G(T_old)) * horizon_requests > cost * epoch_requests,        */
/* and break-even requests = ceil(cost * epoch_requests / (G_new - G_old))    */
/* (-1 without a gain; INT64_MAX when the ceiling does not fit in int64).  */
/* out5 = {G_old, G_new, cost, break_even, adopted};                          */
/* placement [W][n] out = the adopted target.  Returns 0, or -1 on an        */
/* invalid tree.                                                              */
/* ------------------------------------------------------------------------ */
int or_replan(const or_inst *I, const uint8_t *incumbent, int32_t S, const int32_t *orders, int32_t R,
              int64_t epoch_requests, int64_t horizon_requests, int32_t n_threads, int safeguards,
              uint8_t *placement, int64_t *out5)
{
    int32_t n = I->n, W = I->W;
    uint8_t *T = malloc((size_t)W * n + 1);
    int64_t g_new = 0;
    if (or_plan(I, S, orders, R, n_threads, T, &g_new, NULL, NULL, NULL, NULL, safeguards, NULL) < 0) {
        free(T);
        return -1;
    }
    int64_t g_old = or_objective(I, incumbent);
    int64_t cost = 0;
    for (int32_t m = 0; m < W; ++m)
        for (int32_t b = 0; b < n; ++b) {
            if (!HOLDS(T, I, m, b) || HOLDS(incumbent, I, m, b)) continue;
            int64_t c = WCOST(I, m, b);                 /* recompute */
            for (int32_t h = 0; h < W; ++h) {
                if (h == m || !HOLDS(incumbent, I, h, b)) continue;
                int64_t f = I->mode == 0 ? FREQ(I, m, b) : FPAIR(I, h, m, b);
                c = imin64(c, f);                       /* fetch from an incumbent holder */
            }
            cost += c;
        }
    int64_t gain = g_new - g_old;
    int64_t be = -1;
    if (gain > 0) {                     /* the ceiling, saturated at INT64_MAX */
        __int128 num = (__int128)cost * epoch_requests;
        __int128 q = (num + gain - 1) / gain;
        be = q > (__int128)INT64_MAX ? INT64_MAX : (int64_t)q;
    }
    int adopt = gain > 0 && (__int128)gain * horizon_requests > (__int128)cost * epoch_requests;
    memcpy(placement, adopt ? T : incumbent, (size_t)W * n);
    out5[0] = g_old; out5[1] = g_new; out5[2] = cost; out5[3] = be; out5[4] = adopt;
    free(T);
    return 0;
}

/* One step of Algorithm 1 for a single worker, exposed so that one update of */
/* a large plan can be checked on its own: marginals of h against placement  */
/* (T_h ignored), then RootedDP.  profit and chosen are by node id.           */
int64_t or_worker_update(const or_inst *I, int32_t h, const uint8_t *placement,
                         int64_t *profit, uint8_t *chosen)
{
    or_marginal(I, h, placement, profit);
    return or_rooted_dp(I->n, I->parent, I->weight, profit, I->budget[h], chosen, -1);
}
