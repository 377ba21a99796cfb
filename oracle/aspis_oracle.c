/*
 * aspis_oracle.c -- plain, slow, obviously-correct CPU oracle for the Aspis
 * parameter-server detection-and-aggregation step (Konstantinidis &
 * Ramamoorthy, "Aspis: Robust Detection for Distributed Learning").
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * execute this file.  Only the test suite, the smoke check and the CPU
 * baseline leg of the benchmark use it, to check the CUDA path and to time a
 * plain CPU implementation beside it.  It shares no code, header, table or
 * helper with the CUDA library.
 *
 * Every function follows one step of the paper, in the paper's order:
 *
 *   oracle_assign              Algorithm 2 (subset-based file assignment), Example 1
 *   oracle_file_agreement      per-file agreement alpha_i^{(j1,j2)} (Section 4, first display)
 *   oracle_pair_agreement      pair agreement count alpha^{(j1,j2)} (Section 4, second display)
 *   oracle_graph               edge rule of G: alpha == C(K-2,r-2) (Section 4, Algorithm 3)
 *   oracle_max_cliques_brute   all maximum cliques by enumerating every vertex subset (Algorithm 3)
 *   oracle_max_cliques_bk      the same by Bron-Kerbosch with pivoting (Tomita et al., cited in Section 4)
 *   oracle_max_cliques_wide    the same for up to 128 workers, also counting all maximal
 *                              cliques (the enumeration Table 5 times)
 *   oracle_select              Algorithm 1: Case 1 honest copy / Case 2 majority (Eq. 2)
 *   oracle_lower_median        coordinate-wise median of the chosen gradients (Algorithm 1, Case 2)
 *   oracle_mean                average of the chosen gradients (Algorithm 1, Case 1)
 *   oracle_sgd                 the model update with the aggregate (Section 2, Eq. 1;
 *                              Algorithm 1), with heavy-ball momentum (Appendix A.3)
 *   oracle_file_agreement_tol, oracle_select_tol, oracle_file_means
 *                              the variant for copies that are not bit-identical
 *                              (Section 5, after Algorithm 1: average the honest
 *                              copies, or the largest cluster of copies)
 *
 * Readings where the paper is silent (each also listed in the design notes):
 *   - file i <-> the i-th r-subset of workers in lexicographic order; Example 1
 *     fixes file 0 = {U1,...,Ur}.
 *   - "equal" gradients are bitwise-equal fp32 vectors (the paper guarantees
 *     honest copies are exactly equal), so +0 != -0 and equal NaN payloads are
 *     equal.
 *   - majority when no strict majority exists: the largest class of equal
 *     copies, ties to the class holding the lower slot.
 *   - median of an even count: the lower median, rank floor((n-1)/2), in the
 *     IEEE-754 totalOrder of the fp32 values; the output keeps the bits of
 *     the selected element.
 *   - Case 1 chooses the honest copy with the lowest slot; files with no
 *     honest worker are dropped.
 *   - the momentum of the experiments (0.9) is heavy-ball momentum without
 *     dampening, v <- mu*v + g, w <- w - eta*v, as in the paper's PyTorch
 *     framework; each of the two results is the exact value rounded once
 *     to fp32.
 *
 * Parity status: every function here is pinned by tests (closed-form counts,
 * Example 1, the Figure 3 graphs, Theorem 1, brute force, NetworkX clique
 * enumeration, sorting).  Two behaviours are readings rather than paper
 * facts: the plurality rule when no strict majority exists and the rounding
 * of the mean (checked against an exactly-rounded sum within a tolerance).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <pthread.h>

#define ORACLE_OK 0
#define ORACLE_EINVAL 1
#define ORACLE_ERANGE 2
#define ORACLE_EEMPTY 6

/* ---------------------------------------------------------------- helpers */

/* Binomial coefficient C(n,k) by the multiplicative formula; 0 when k<0 or k>n. */
int64_t oracle_binom(int64_t n, int64_t k)
{
    if (k < 0 || n < 0 || k > n) return 0;
    if (k > n - k) k = n - k;
    int64_t v = 1;
    for (int64_t i = 1; i <= k; ++i) v = v * (n - k + i) / i;
    return v;
}

/* Index of the unordered slot pair (s,t), s<t, among the C(r,2) pairs of one
 * file listed as (0,1),(0,2),...,(0,r-1),(1,2),...: the bit that holds
 * "copies s and t differ" in a per-file mismatch word. */
static int pair_bit(int r, int s, int t)
{
    int p = 0;
    for (int a = 0; a < r; ++a)
        for (int b = a + 1; b < r; ++b) {
            if (a == s && b == t) return p;
            ++p;
        }
    return -1;
}

/* ------------------------------------------------------------ Algorithm 2 */

/* Subset-based assignment.  File i is given to the workers of the i-th
 * r-subset S_i of {0,...,K-1} in lexicographic order (Example 1: S_0 is the
 * first r workers).  Outputs:
 *   file_workers[i*r + s]  worker of slot s of file i, ascending in s;
 *   worker_files[j*l + k]  k-th file of worker j, ascending in k;
 *   slot_of[j*l + k]       slot that worker j holds in that file.
 * Returns 0, or ORACLE_EINVAL for r<2, r>K (the paper requires r>1). */
int oracle_assign(int K, int r, uint8_t *file_workers, int32_t *worker_files,
                  uint8_t *slot_of)
{
    if (K < 2 || r < 2 || r > K || K > 255) return ORACLE_EINVAL;
    int64_t f = oracle_binom(K, r);
    int64_t l = oracle_binom(K - 1, r - 1);
    int S[256];
    for (int s = 0; s < r; ++s) S[s] = s;              /* S_0 = {0,...,r-1} */
    int32_t *fill = (int32_t *)calloc((size_t)K, sizeof(int32_t));
    if (!fill) return ORACLE_EINVAL;
    for (int64_t i = 0; i < f; ++i) {
        for (int s = 0; s < r; ++s) {
            int j = S[s];
            file_workers[i * r + s] = (uint8_t)j;
            worker_files[(int64_t)j * l + fill[j]] = (int32_t)i;
            slot_of[(int64_t)j * l + fill[j]] = (uint8_t)s;
            fill[j]++;
        }
        /* next r-subset in lexicographic order */
        int s = r - 1;
        while (s >= 0 && S[s] == K - r + s) --s;
        if (s < 0) break;
        S[s]++;
        for (int u = s + 1; u < r; ++u) S[u] = S[u - 1] + 1;
    }
    free(fill);
    return ORACLE_OK;
}

/* -------------------------------------------------- agreement alpha_i */

typedef struct {
    const float *copies;
    int64_t f0, f1, d, ld;
    int r;
    float tau;                 /* tolerant variant only */
    uint32_t *file_neq;
} agree_job;

static void *agree_worker(void *arg)
{
    agree_job *J = (agree_job *)arg;
    for (int64_t i = J->f0; i < J->f1; ++i) {
        uint32_t w = 0;
        for (int s = 0; s < J->r; ++s)
            for (int t = s + 1; t < J->r; ++t) {
                const float *a = J->copies + (i * J->r + s) * J->ld;
                const float *b = J->copies + (i * J->r + t) * J->ld;
                /* alpha_i^{(j_s,j_t)} = 1 iff the two returned vectors are equal;
                 * equality is of the fp32 bit patterns over the d coordinates */
                int equal = memcmp(a, b, (size_t)J->d * sizeof(float)) == 0;
                if (!equal) w |= 1u << pair_bit(J->r, s, t);
            }
        J->file_neq[i] = w;
    }
    return NULL;
}

/* Per-file agreement.  copies is [f][r][ld] fp32 (row (i,s) is the vector the
 * worker in slot s returned for file i; only the first d of ld are compared).
 * file_neq[i] bit pair_bit(s,t) is 1 iff alpha_i for that slot pair is 0. */
int oracle_file_agreement(const float *copies, int64_t f, int r, int64_t d,
                          int64_t ld, uint32_t *file_neq, int nthreads)
{
    if (r < 2 || r > 8 || d < 0 || ld < d || f < 0) return ORACLE_EINVAL;
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    pthread_t th[256];
    agree_job jobs[256];
    for (int t = 0; t < nthreads; ++t) {
        jobs[t].copies = copies;
        jobs[t].f0 = f * t / nthreads;
        jobs[t].f1 = f * (t + 1) / nthreads;
        jobs[t].d = d;
        jobs[t].ld = ld;
        jobs[t].r = r;
        jobs[t].file_neq = file_neq;
        pthread_create(&th[t], NULL, agree_worker, &jobs[t]);
    }
    for (int t = 0; t < nthreads; ++t) pthread_join(th[t], NULL);
    return ORACLE_OK;
}

/* ------------------------------------------------ pair count alpha^{(j1,j2)} */

/* alpha[j1*K + j2] = number of files shared by workers j1 and j2 on which
 * their copies agree: the sum of alpha_i over N(U_j1) ∩ N(U_j2).  The
 * diagonal is left 0. */
int oracle_pair_agreement(const uint32_t *file_neq, const uint8_t *file_workers,
                          int64_t f, int r, int K, int64_t *alpha)
{
    if (K < 2 || K > 255 || r < 2 || r > 8) return ORACLE_EINVAL;
    memset(alpha, 0, sizeof(int64_t) * (size_t)K * (size_t)K);
    for (int64_t i = 0; i < f; ++i)
        for (int s = 0; s < r; ++s)
            for (int t = s + 1; t < r; ++t) {
                int a = (file_neq[i] >> pair_bit(r, s, t)) & 1 ? 0 : 1;
                int j1 = file_workers[i * r + s], j2 = file_workers[i * r + t];
                alpha[(int64_t)j1 * K + j2] += a;
                alpha[(int64_t)j2 * K + j1] += a;
            }
    return ORACLE_OK;
}

/* -------------------------------------------------------------- graph G */

/* Edge (j1,j2) iff alpha^{(j1,j2)} equals C(K-2,r-2), i.e. the two workers
 * agree on every file they share (Algorithm 3, first loop).  adj[j] bit k is
 * the edge (j,k); no self loops; bits >= K are 0.  K <= 32. */
int oracle_graph(const int64_t *alpha, int K, int r, uint32_t *adj)
{
    if (K < 2 || K > 32 || r < 2) return ORACLE_EINVAL;
    int64_t shared = oracle_binom(K - 2, r - 2);
    for (int j1 = 0; j1 < K; ++j1) {
        uint32_t m = 0;
        for (int j2 = 0; j2 < K; ++j2)
            if (j2 != j1 && alpha[(int64_t)j1 * K + j2] == shared) m |= 1u << j2;
        adj[j1] = m;
    }
    return ORACLE_OK;
}

/* ------------------------------------------------- Algorithm 3: cliques */

static int popcount32(uint32_t x)
{
    int c = 0;
    while (x) { x &= x - 1; ++c; }
    return c;
}

static int is_clique(const uint32_t *adj, int K, uint32_t mask)
{
    for (int j = 0; j < K; ++j)
        if ((mask >> j) & 1)
            if (mask & ~(adj[j] | (1u << j))) return 0;
    return 1;
}

/* All maximum cliques by brute force over the 2^K vertex subsets (K <= 24):
 * omega = largest clique size, n_max = number of cliques of that size,
 * canon = the one with the smallest mask value. */
int oracle_max_cliques_brute(const uint32_t *adj, int K, int32_t *omega,
                             uint32_t *n_max, uint32_t *canon)
{
    if (K < 1 || K > 24) return ORACLE_ERANGE;
    int best = 0;
    uint32_t cnt = 0, first = 0;
    for (uint32_t mask = 1; mask < (1u << K); ++mask) {
        if (!is_clique(adj, K, mask)) continue;
        int sz = popcount32(mask);
        if (sz > best) { best = sz; cnt = 1; first = mask; }
        else if (sz == best) { ++cnt; if (mask < first) first = mask; }
    }
    *omega = best;
    *n_max = cnt;
    *canon = first;
    return ORACLE_OK;
}

/* Bron-Kerbosch enumeration of all maximal cliques with Tomita pivoting
 * (pivot = vertex of P∪X with most neighbours in P).  Every maximum clique is
 * maximal, so counting the maximal cliques of the largest size counts the
 * maximum cliques.  Plain recursion over bitmasks, K <= 32. */
typedef struct {
    const uint32_t *adj;
    int K;
    int best;
    uint32_t cnt, first;
    uint64_t calls;
} bk_state;

static void bk(bk_state *S, uint32_t R, uint32_t P, uint32_t X)
{
    S->calls++;
    if (P == 0 && X == 0) {               /* R is a maximal clique */
        int sz = popcount32(R);
        if (sz > S->best) { S->best = sz; S->cnt = 1; S->first = R; }
        else if (sz == S->best) { S->cnt++; if (R < S->first) S->first = R; }
        return;
    }
    uint32_t PX = P | X;
    int piv = -1, pbest = -1;
    for (int u = 0; u < S->K; ++u)
        if ((PX >> u) & 1) {
            int c = popcount32(P & S->adj[u]);
            if (c > pbest) { pbest = c; piv = u; }
        }
    uint32_t cand = P & ~S->adj[piv];
    for (int v = 0; v < S->K; ++v) {
        if (!((cand >> v) & 1)) continue;
        bk(S, R | (1u << v), P & S->adj[v], X & S->adj[v]);
        P &= ~(1u << v);
        X |= 1u << v;
    }
}

int oracle_max_cliques_bk(const uint32_t *adj, int K, int32_t *omega,
                          uint32_t *n_max, uint32_t *canon, uint64_t *calls)
{
    if (K < 1 || K > 32) return ORACLE_ERANGE;
    bk_state S;
    S.adj = adj;
    S.K = K;
    S.best = 0;
    S.cnt = 0;
    S.first = 0;
    S.calls = 0;
    uint32_t all = (K == 32) ? 0xffffffffu : ((1u << K) - 1u);
    bk(&S, 0, all, 0);
    *omega = S.best;
    *n_max = S.cnt;
    *canon = S.first;
    if (calls) *calls = S.calls;
    return ORACLE_OK;
}

/* ------------------------------- Algorithm 3 for up to 128 workers */

/* Vertex sets of up to 128 workers as four 32-bit words: worker k is bit
 * k % 32 of word k / 32.  A mask's value orders word 3 first. */
typedef struct {
    uint32_t w[4];
} vset;

static int vs_count(vset a)
{
    return popcount32(a.w[0]) + popcount32(a.w[1]) + popcount32(a.w[2]) + popcount32(a.w[3]);
}

static int vs_empty(vset a) { return (a.w[0] | a.w[1] | a.w[2] | a.w[3]) == 0; }

static int vs_has(vset a, int k) { return (int)((a.w[k >> 5] >> (k & 31)) & 1u); }

static vset vs_and(vset a, vset b)
{
    for (int i = 0; i < 4; ++i) a.w[i] &= b.w[i];
    return a;
}

static vset vs_andnot(vset a, vset b)
{
    for (int i = 0; i < 4; ++i) a.w[i] &= ~b.w[i];
    return a;
}

static vset vs_with(vset a, int k)
{
    a.w[k >> 5] |= 1u << (k & 31);
    return a;
}

static vset vs_without(vset a, int k)
{
    a.w[k >> 5] &= ~(1u << (k & 31));
    return a;
}

static int vs_less(vset a, vset b)
{
    for (int i = 3; i >= 0; --i)
        if (a.w[i] != b.w[i]) return a.w[i] < b.w[i];
    return 0;
}

typedef struct {
    vset adj[128];
    int K;
    int best;
    uint64_t cnt, maximal;
    vset first;
} bkw_state;

/* Bron-Kerbosch with Tomita pivoting, as oracle_max_cliques_bk, reporting
 * every maximal clique R (P and X empty). */
static void bkw(bkw_state *S, vset R, vset P, vset X)
{
    if (vs_empty(P) && vs_empty(X)) {
        int sz = vs_count(R);
        S->maximal++;
        if (sz > S->best) { S->best = sz; S->cnt = 1; S->first = R; }
        else if (sz == S->best) { S->cnt++; if (vs_less(R, S->first)) S->first = R; }
        return;
    }
    int piv = -1, pbest = -1;
    for (int u = 0; u < S->K; ++u)
        if (vs_has(P, u) || vs_has(X, u)) {
            int c = vs_count(vs_and(P, S->adj[u]));
            if (c > pbest) { pbest = c; piv = u; }
        }
    vset cand = vs_andnot(P, S->adj[piv]);
    for (int v = 0; v < S->K; ++v) {
        if (!vs_has(cand, v)) continue;
        bkw(S, vs_with(R, v), vs_and(P, S->adj[v]), vs_and(X, S->adj[v]));
        P = vs_without(P, v);
        X = vs_with(X, v);
    }
}

/* adj: [K][4] words, row j = neighbours of worker j.  An edge counts only
 * when both rows list it; self loops and bits >= K are ignored.  Outputs
 * omega, the number of maximum cliques, the maximum clique with the smallest
 * mask value (canon[4]) and the number of maximal cliques. */
int oracle_max_cliques_wide(const uint32_t *adj, int K, int32_t *omega, uint64_t *n_max,
                            uint32_t *canon, uint64_t *n_maximal)
{
    if (K < 1 || K > 128) return ORACLE_ERANGE;
    bkw_state *S = (bkw_state *)calloc(1, sizeof(bkw_state));
    if (!S) return ORACLE_EINVAL;
    S->K = K;
    for (int j = 0; j < K; ++j)
        for (int k = 0; k < K; ++k)
            if (k != j && ((adj[j * 4 + (k >> 5)] >> (k & 31)) & 1u) &&
                ((adj[k * 4 + (j >> 5)] >> (j & 31)) & 1u))
                S->adj[j] = vs_with(S->adj[j], k);
    vset all = {{0u, 0u, 0u, 0u}}, none = {{0u, 0u, 0u, 0u}};
    for (int k = 0; k < K; ++k) all = vs_with(all, k);
    bkw(S, none, all, none);
    *omega = S->best;
    *n_max = S->cnt;
    for (int i = 0; i < 4; ++i) canon[i] = S->first.w[i];
    *n_maximal = S->maximal;
    free(S);
    return ORACLE_OK;
}

/* ------------------------------------------------- Algorithm 1: selection */

/* Chooses, for each file, the copy that enters aggregation.
 *   success != 0 (Case 1): H = clique; the copy of the lowest slot whose
 *     worker is in H, or -1 (file dropped) when N(B_i) ∩ H is empty.
 *   success == 0 (Case 2): the majority m_i of Eq. 2: the copies split into
 *     classes of bitwise-equal vectors (copies s,t are equal iff their
 *     mismatch bit is 0); the largest class wins, ties to the class holding
 *     the lower slot; sel is that class's lowest slot.  No file is dropped.
 * Returns n_sel, the number of files with sel >= 0. */
int64_t oracle_select(const uint32_t *file_neq, const uint8_t *file_workers,
                      int64_t f, int r, uint32_t clique, int success, int8_t *sel)
{
    int64_t n_sel = 0;
    for (int64_t i = 0; i < f; ++i) {
        int pick = -1;
        if (success) {
            for (int s = 0; s < r; ++s)
                if ((clique >> file_workers[i * r + s]) & 1) { pick = s; break; }
        } else {
            int best = 0;
            for (int s = 0; s < r; ++s) {
                int size = 1;
                for (int t = 0; t < r; ++t) {
                    if (t == s) continue;
                    int a = s < t ? s : t, b = s < t ? t : s;
                    if (!((file_neq[i] >> pair_bit(r, a, b)) & 1)) ++size;
                }
                if (size > best) { best = size; pick = s; }
            }
        }
        sel[i] = (int8_t)pick;
        if (pick >= 0) ++n_sel;
    }
    return n_sel;
}

/* ---------------------------------------------- coordinate-wise median */

/* IEEE-754 totalOrder as an unsigned key: negatives reversed below
 * positives, -0 < +0, NaNs at the two ends by sign. */
static uint32_t order_key(uint32_t u)
{
    return (u >> 31) ? ~u : (u | 0x80000000u);
}

static uint32_t order_unkey(uint32_t k)
{
    return (k >> 31) ? (k & 0x7fffffffu) : ~k;
}

static int cmp_u32(const void *a, const void *b)
{
    uint32_t x = *(const uint32_t *)a, y = *(const uint32_t *)b;
    return (x > y) - (x < y);
}

typedef struct {
    const float *copies;
    int64_t f, ld, c0, c1;
    int r;
    const int8_t *sel;
    int64_t n_sel;
    int mode;
    float *out;
} agg_job;

static void *agg_worker(void *arg)
{
    agg_job *J = (agg_job *)arg;
    uint32_t *keys = (uint32_t *)malloc(sizeof(uint32_t) * (size_t)(J->n_sel > 0 ? J->n_sel : 1));
    for (int64_t c = J->c0; c < J->c1; ++c) {
        if (J->mode == 0) {
            /* gather the chosen value of every kept file at coordinate c */
            int64_t n = 0;
            for (int64_t i = 0; i < J->f; ++i) {
                if (J->sel[i] < 0) continue;
                uint32_t u;
                memcpy(&u, J->copies + (i * J->r + J->sel[i]) * J->ld + c, 4);
                keys[n++] = order_key(u);
            }
            qsort(keys, (size_t)n, sizeof(uint32_t), cmp_u32);
            uint32_t u = order_unkey(keys[(n - 1) / 2]);   /* lower median */
            memcpy(&J->out[c - J->c0], &u, 4);
        } else {
            /* mean: sum in double in file order, divide, round to fp32 */
            double acc = 0.0;
            for (int64_t i = 0; i < J->f; ++i) {
                if (J->sel[i] < 0) continue;
                acc += (double)J->copies[(i * J->r + J->sel[i]) * J->ld + c];
            }
            J->out[c - J->c0] = (float)(acc / (double)J->n_sel);
        }
    }
    free(keys);
    return NULL;
}

/* Coordinate-wise aggregation of the chosen copies over coordinates
 * [c0,c1): mode 0 = lower median (rank floor((n_sel-1)/2) in totalOrder,
 * output bit-identical to the chosen element), mode 1 = mean.
 * out has c1-c0 entries.  Returns ORACLE_EEMPTY when no file is kept. */
int oracle_aggregate(const float *copies, int64_t f, int r, int64_t ld,
                     const int8_t *sel, int mode, int64_t c0, int64_t c1,
                     float *out, int nthreads)
{
    if (c0 < 0 || c1 < c0 || c1 > ld || (mode != 0 && mode != 1)) return ORACLE_EINVAL;
    int64_t n_sel = 0;
    for (int64_t i = 0; i < f; ++i) n_sel += sel[i] >= 0;
    if (n_sel == 0) return ORACLE_EEMPTY;
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    pthread_t th[256];
    agg_job jobs[256];
    int64_t m = c1 - c0;
    for (int t = 0; t < nthreads; ++t) {
        jobs[t].copies = copies;
        jobs[t].f = f;
        jobs[t].ld = ld;
        jobs[t].r = r;
        jobs[t].sel = sel;
        jobs[t].n_sel = n_sel;
        jobs[t].mode = mode;
        jobs[t].c0 = c0 + m * t / nthreads;
        jobs[t].c1 = c0 + m * (t + 1) / nthreads;
        jobs[t].out = out + (jobs[t].c0 - c0);
        pthread_create(&th[t], NULL, agg_worker, &jobs[t]);
    }
    for (int t = 0; t < nthreads; ++t) pthread_join(th[t], NULL);
    return ORACLE_OK;
}

/* Lower median of each column of a dense [n][m] fp32 matrix (rows are the
 * chosen gradients of n files, gathered by the caller): out[c] is the
 * element of rank floor((n-1)/2) of column c in totalOrder, bit-identical. */
int oracle_lower_median(const float *vals, int64_t n, int64_t m, float *out)
{
    if (n <= 0) return ORACLE_EEMPTY;
    uint32_t *keys = (uint32_t *)malloc(sizeof(uint32_t) * (size_t)n);
    if (!keys) return ORACLE_EINVAL;
    for (int64_t c = 0; c < m; ++c) {
        for (int64_t i = 0; i < n; ++i) {
            uint32_t u;
            memcpy(&u, vals + i * m + c, 4);
            keys[i] = order_key(u);
        }
        qsort(keys, (size_t)n, sizeof(uint32_t), cmp_u32);
        uint32_t u = order_unkey(keys[(n - 1) / 2]);
        memcpy(&out[c], &u, 4);
    }
    free(keys);
    return ORACLE_OK;
}

/* Mean of each column of a dense [n][m] fp32 matrix: double sum in row order,
 * divided by n, rounded to fp32 (Algorithm 1, Case 1 update). */
int oracle_mean(const float *vals, int64_t n, int64_t m, float *out)
{
    if (n <= 0) return ORACLE_EEMPTY;
    for (int64_t c = 0; c < m; ++c) {
        double acc = 0.0;
        for (int64_t i = 0; i < n; ++i) acc += (double)vals[i * m + c];
        out[c] = (float)(acc / (double)n);
    }
    return ORACLE_OK;
}

/* One model update with the aggregated gradient g, over m coordinates.
 * Eq. 1 (Section 2) moves w against the batch gradient with step eta; the
 * PS of Algorithm 1 uses the aggregate of the chosen copies in its place.
 * The experiments add momentum 0.9 (Appendix A.3), read as heavy-ball
 * momentum:
 *     v[c] <- mu * v[c] + g[c]        then        w[c] <- w[c] - eta * v[c],
 * each the exact real value rounded once to fp32 (C99 fmaf is exactly
 * that).  mu == 0 is Eq. 1 itself, w[c] <- w[c] - eta * g[c], and v is not
 * touched (it may be NULL). */
int oracle_sgd(const float *g, float *w, float *v, int64_t m, float eta, float mu)
{
    if (m < 0 || (m > 0 && (!g || !w))) return ORACLE_EINVAL;
    if (mu != 0.0f && m > 0 && !v) return ORACLE_EINVAL;
    for (int64_t c = 0; c < m; ++c) {
        if (mu != 0.0f) {
            v[c] = fmaf(mu, v[c], g[c]);
            w[c] = fmaf(-eta, v[c], w[c]);
        } else {
            w[c] = fmaf(-eta, g[c], w[c]);
        }
    }
    return ORACLE_OK;
}

/* --------------------------------- copies that are not bit-identical */

/* Section 5 (after Algorithm 1) notes that honest copies differing by
 * floating-point effects can still be handled: in Case 1 the PS averages
 * the honest copies of a file, in Case 2 it clusters the copies and
 * averages the largest cluster.  Readings, which the paper leaves open:
 *   - copies a, b of a file are close iff |a[c] - b[c]| <= tau for every
 *     c < d, the difference and its magnitude in fp32 (never close where
 *     either value is NaN); the graph and clique steps use "close" for
 *     "equal";
 *   - clusters are the connected components of "close" among the r slots;
 *     the largest wins, ties to the one holding the lower slot;
 *   - the average of the chosen copies per coordinate is their arithmetic
 *     mean: summed in double in slot order, divided by their number, rounded
 *     once to fp32.  Identical copies give their common value exactly (also
 *     -0, infinities and NaNs). */

static void *agree_tol_worker(void *arg)
{
    agree_job *J = (agree_job *)arg;
    const float tau = J->tau;
    for (int64_t i = J->f0; i < J->f1; ++i) {
        uint32_t w = 0;
        for (int s = 0; s < J->r; ++s)
            for (int t = s + 1; t < J->r; ++t) {
                const float *a = J->copies + (i * J->r + s) * J->ld;
                const float *b = J->copies + (i * J->r + t) * J->ld;
                int close = 1;
                for (int64_t c = 0; c < J->d && close; ++c) {
                    float diff = a[c] - b[c];
                    if (!(fabsf(diff) <= tau)) close = 0;
                }
                if (!close) w |= 1u << pair_bit(J->r, s, t);
            }
        J->file_neq[i] = w;
    }
    return NULL;
}

/* file_neq[i] bit pair_bit(s,t) is 1 iff copies s and t of file i are not
 * close.  tau must be >= 0 (a NaN tau is rejected). */
int oracle_file_agreement_tol(const float *copies, int64_t f, int r, int64_t d, int64_t ld,
                              float tau, uint32_t *file_neq, int nthreads)
{
    if (r < 2 || r > 8 || d < 0 || ld < d || f < 0 || !(tau >= 0.0f)) return ORACLE_EINVAL;
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    pthread_t th[256];
    agree_job jobs[256];
    for (int t = 0; t < nthreads; ++t) {
        jobs[t].copies = copies;
        jobs[t].f0 = f * t / nthreads;
        jobs[t].f1 = f * (t + 1) / nthreads;
        jobs[t].d = d;
        jobs[t].ld = ld;
        jobs[t].r = r;
        jobs[t].tau = tau;
        jobs[t].file_neq = file_neq;
        pthread_create(&th[t], NULL, agree_tol_worker, &jobs[t]);
    }
    for (int t = 0; t < nthreads; ++t) pthread_join(th[t], NULL);
    return ORACLE_OK;
}

/* slot_mask[i] = the slots whose copies are averaged for file i (bit s =
 * slot s), 0 when the file is dropped.  Case 1 (success): the slots whose
 * worker is in the clique.  Case 2: the largest cluster.  Returns the
 * number of files kept. */
int64_t oracle_select_tol(const uint32_t *file_neq, const uint8_t *file_workers, int64_t f,
                          int r, uint32_t clique, int success, uint8_t *slot_mask)
{
    int64_t kept = 0;
    for (int64_t i = 0; i < f; ++i) {
        uint32_t m = 0;
        if (success) {
            for (int s = 0; s < r; ++s)
                if ((clique >> file_workers[i * r + s]) & 1u) m |= 1u << s;
        } else {
            int comp[8];
            for (int s = 0; s < r; ++s) comp[s] = s;
            /* union of close pairs, repeated until no label changes */
            for (int changed = 1; changed;) {
                changed = 0;
                for (int s = 0; s < r; ++s)
                    for (int t = s + 1; t < r; ++t)
                        if (!((file_neq[i] >> pair_bit(r, s, t)) & 1u) && comp[s] != comp[t]) {
                            int lo = comp[s] < comp[t] ? comp[s] : comp[t];
                            int hi = comp[s] < comp[t] ? comp[t] : comp[s];
                            for (int u = 0; u < r; ++u)
                                if (comp[u] == hi) comp[u] = lo;
                            changed = 1;
                        }
            }
            int best = -1, best_size = 0;
            for (int s = 0; s < r; ++s) {       /* labels are each component's lowest slot */
                if (comp[s] != s) continue;
                int size = 0;
                for (int u = 0; u < r; ++u) size += comp[u] == s;
                if (size > best_size) { best_size = size; best = s; }
            }
            for (int u = 0; u < r; ++u)
                if (comp[u] == best) m |= 1u << u;
        }
        slot_mask[i] = (uint8_t)m;
        if (m) ++kept;
    }
    return kept;
}

/* means[i*d + c] = the average of the copies in slot_mask[i]: their
 * arithmetic mean, summed in double in slot order, divided by their number
 * and rounded once to fp32 (Section 5's remark after Algorithm 1 says to
 * average them); files with an empty mask are left untouched.  Identical
 * copies give their common value exactly (k equal fp32 values sum exactly in
 * double). */
int oracle_file_means(const float *copies, int64_t f, int r, int64_t d, int64_t ld,
                      const uint8_t *slot_mask, float *means)
{
    if (r < 1 || r > 8 || d < 0 || ld < d || f < 0) return ORACLE_EINVAL;
    for (int64_t i = 0; i < f; ++i) {
        const uint32_t m = slot_mask[i];
        if (!m) continue;
        int k = 0;
        for (int s = 0; s < r; ++s)
            if ((m >> s) & 1u) ++k;
        for (int64_t c = 0; c < d; ++c) {
            /* the sum starts from the first chosen copy, not from +0, so a
             * sum of negative zeros stays -0 */
            double sum = 0.0;
            int first = 1;
            for (int s = 0; s < r; ++s) {
                if (!((m >> s) & 1u)) continue;
                const double x = (double)copies[(i * r + s) * ld + c];
                sum = first ? x : sum + x;
                first = 0;
            }
            means[i * d + c] = (float)(sum / (double)k);
        }
    }
    return ORACLE_OK;
}
