/*
 * twinkv_oracle.c -- reference oracle for the TwinKV redundancy audit and repair pass
 * (arXiv 2608.27128).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is a plain, slow, obviously-correct CPU
 * restatement of the paper's definitions, in fp64.  Only the test suite, the smoke
 * check of __graft_entry__ and the cpu_baseline leg of bench.py may load it.  The
 * CUDA library never links, includes or calls it, and it shares no code with the
 * CUDA library.
 *
 * What it computes, by paper passage:
 *   Sec. 3.2, Eq. 1      sim(i,j) = khat_i . khat_j with khat_i = k_i / ||k_i||_2,
 *                        evaluated as (k_i . k_j) / sqrt((k_i . k_i)(k_j . k_j)): the dot
 *                        products of bf16 keys are exact in double (16-bit products,
 *                        d <= 128 terms), so one rounding each remains for the product,
 *                        the square root and the quotient; the value is symmetric in
 *                        (i, j) and exactly 1 for positively scaled duplicates
 *   Sec. 3.2, twin rule  j is a twin candidate of i only if |i-j| > w (and j != i)
 *   Sec. 3.4, Eq. 4      b_i(S0) = max over j in S0, |i-j| > w, j != i of sim(i,j);
 *                        -1 when no such j exists
 *   (b_all)              the same maximum over every j (the twin relation of Sec. 3.2)
 *   Sec. 3.4, orphan     i not in S0 and b_i(S0) < tau
 *   Sec. 3.4, donor      j in S0, outside the sink/recent regions (Sec. 3.2, protected
 *                        regions), and b_j(S0) >= tau
 *   Sec. 3.4, repair     rank orphans by ascending b, donors by descending b,
 *                        m = min(|O|,|D|), evict the m most severe donors and admit
 *                        the m most severe orphans; |S1| = |S0|
 *   (dedup variant)      the repair with donors taken in severity order, where evicting
 *                        a donor keeps its twin (its b_i(S0) argmax) in place, so a
 *                        twin pair never loses both members
 *   Sec. 3.2, Eq. 2      r_i = number of j with |i-j| > w (j != i) and sim(i,j) > tau
 *   Sec. 3.2, Eq. 3      s_i = -r_i / n; the standalone policy keeps the K highest
 *                        scores, with the sink and recent regions given the maximum
 *                        score (always kept)
 *
 * Readings where the paper is silent (each one is listed in the design notes):
 *   - a key with zero norm has khat = 0, so its similarity with every key is 0;
 *   - equal similarities: the lower position j wins the argmax;
 *   - equal severities: the lower position comes first, for orphans and donors;
 *   - the k-th most severe donor is paired with the k-th most severe orphan;
 *   - b is computed once on S0; nothing is recomputed after a swap;
 *   - threshold comparisons use the threshold rounded to float, widened to double,
 *     so that a float implementation and this oracle compare against the same number;
 *   - keys are bf16 bit patterns; float32 keys are first rounded to bf16,
 *     round-to-nearest-even;
 *   - the dedup variant is this build's reading of the paper's remark that one member
 *     of a twin pair already holds a slot (Sec. 3.4): walking donors from the most
 *     severe, a donor is skipped when its twin was accepted for eviction earlier in
 *     the walk, or when it is the twin of an accepted donor (it now holds that
 *     donor's content); the walk stops after |O| accepted donors;
 *   - the standalone policy orders positions by (protected first, r ascending, i.e.
 *     s descending, then position ascending) and keeps the first K; a budget below
 *     the protected count keeps the lowest protected positions.
 *
 * Parity pins for every function here live in tests/test_oracle_pins.py and
 * tests/golden/ (closed forms, hand-derived worked examples, a float64 numpy matmul,
 * brute-force ranking and the paper's invariants).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ---- bf16 helpers (input decoding only) ---------------------------------------- */

/* bf16 is the upper half of an IEEE binary32: decoding is exact. */
static double bf16_to_double(uint16_t h)
{
    uint32_t bits = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

/* float32 -> bf16, round to nearest, ties to even (finite inputs). */
void twk_oracle_round_bf16(const float* in, uint16_t* out, long n)
{
    for (long t = 0; t < n; ++t) {
        uint32_t bits;
        memcpy(&bits, &in[t], sizeof bits);
        uint32_t lower = bits & 0xFFFFu;
        uint32_t upper = bits >> 16;
        if (lower > 0x8000u || (lower == 0x8000u && (upper & 1u)))
            upper += 1u;
        out[t] = (uint16_t)upper;
    }
}

/* ---- Eq. 1 ------------------------------------------------------------------------ */

/* k_i . k_j in double, terms in increasing t. */
static double dot_bf16(const uint16_t* a, const uint16_t* b, int d)
{
    double s = 0.0;
    for (int t = 0; t < d; ++t)
        s += bf16_to_double(a[t]) * bf16_to_double(b[t]);
    return s;
}

/* sim(i,j) of Eq. 1 from the dot product and the two squared norms; a zero key has
 * similarity 0 with every key. */
static double cosine(double dot_ij, double sq_i, double sq_j)
{
    if (sq_i == 0.0 || sq_j == 0.0)
        return 0.0;
    return dot_ij / sqrt(sq_i * sq_j);
}

/* sim(i, j) of Eq. 1 for keys i and j of one (layer, head) stored as bf16 rows of
 * length d.  Used by the comparator to score a candidate twin. */
double twk_oracle_sim(const uint16_t* key_i, const uint16_t* key_j, int d)
{
    return cosine(dot_bf16(key_i, key_j, d), dot_bf16(key_i, key_i, d),
                  dot_bf16(key_j, key_j, d));
}

/* ---- Eq. 4 and the best twin over all keys ------------------------------------- */

/*
 * For each unit u (one layer and KV head) and each requested row i, scan every
 * position j in increasing order and keep
 *   b_all / t_all : the largest sim(i,j) over j with |i-j| > w (j != i follows from
 *                   w >= 0) and its position (first maximum wins, so the lowest j);
 *   b_ret / t_ret : the same restricted to j with mask[j] != 0 (Eq. 4);
 *   b_all2/b_ret2 : the second-largest value of each scan (the largest value over
 *                   the eligible j other than the argmax), -INFINITY if there is none.
 * An empty candidate set gives b = -1 and t = -1 (Eq. 4).
 *
 * keys  : bf16 bits [U][N][d]
 * mask  : [U][N] (0 = evicted, non-zero = retained) or NULL (then b_ret/t_ret/b_ret2
 *         are not written)
 * rows  : list of nrows row positions evaluated in every unit, or NULL for all N rows
 * out   : [U][nrows]
 * Rows are independent; OpenMP (when compiled in) splits them across threads.
 */
void twk_oracle_audit(const uint16_t* keys, int U, int N, int d, const uint8_t* mask,
                      int window, const int32_t* rows, int nrows, double* b_all,
                      int32_t* t_all, double* b_all2, double* b_ret, int32_t* t_ret,
                      double* b_ret2)
{
    if (rows == NULL)
        nrows = N;
    double* sq = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
    for (int u = 0; u < U; ++u) {
        const uint16_t* K = keys + (long)u * N * d;
        const uint8_t* S0 = mask ? mask + (long)u * N : NULL;
        for (int i = 0; i < N; ++i)
            sq[i] = dot_bf16(&K[(long)i * d], &K[(long)i * d], d);
#pragma omp parallel for schedule(dynamic, 8)
        for (int r = 0; r < nrows; ++r) {
            int i = rows ? rows[r] : r;
            double best = -1.0, second = -INFINITY;
            int arg = -1;
            double rbest = -1.0, rsecond = -INFINITY;
            int rarg = -1;
            for (int j = 0; j < N; ++j) {
                int dist = (i > j) ? i - j : j - i;
                if (j == i || dist <= window)
                    continue;
                double s = cosine(dot_bf16(&K[(long)i * d], &K[(long)j * d], d), sq[i], sq[j]);
                if (arg < 0 || s > best) {
                    if (arg >= 0)
                        second = best;
                    best = s;
                    arg = j;
                } else if (s > second) {
                    second = s;
                }
                if (S0 && S0[j]) {
                    if (rarg < 0 || s > rbest) {
                        if (rarg >= 0)
                            rsecond = rbest;
                        rbest = s;
                        rarg = j;
                    } else if (s > rsecond) {
                        rsecond = s;
                    }
                }
            }
            long o = (long)u * nrows + r;
            b_all[o] = best;
            t_all[o] = arg;
            if (b_all2)
                b_all2[o] = second;
            if (S0) {
                b_ret[o] = rbest;
                t_ret[o] = rarg;
                if (b_ret2)
                    b_ret2[o] = rsecond;
            }
        }
    }
    free(sq);
}

/* ---- Sec. 3.4: orphans, donors, severity ranking and the swap ------------------ */

typedef struct {
    double b;
    int32_t pos;
} ranked;

/* orphans: ascending b, then ascending position */
static int cmp_orphan(const void* pa, const void* pb)
{
    const ranked* a = (const ranked*)pa;
    const ranked* b = (const ranked*)pb;
    if (a->b < b->b) return -1;
    if (a->b > b->b) return 1;
    return (a->pos > b->pos) - (a->pos < b->pos);
}

/* donors: descending b, then ascending position */
static int cmp_donor(const void* pa, const void* pb)
{
    const ranked* a = (const ranked*)pa;
    const ranked* b = (const ranked*)pb;
    if (a->b > b->b) return -1;
    if (a->b < b->b) return 1;
    return (a->pos > b->pos) - (a->pos < b->pos);
}

/*
 * One unit of the repair pass.  b[N] = b_i(S0) (Eq. 4), mask[N] = S0 (values 0/1),
 * tau = the threshold (already rounded to float and widened by the caller).
 * Protected: i < n_sink or i >= N - n_recent.
 * Writes out_mask[N] = S1, swaps[2k] = evicted donor, swaps[2k+1] = admitted orphan
 * for k < m, and the orphan/donor flags (either may be NULL).  Returns m.
 */
static int repair_unit(int N, const double* b, const uint8_t* mask, double tau, int n_sink,
                       int n_recent, uint8_t* out_mask, int32_t* swaps, uint8_t* is_orphan,
                       uint8_t* is_donor)
{
    ranked* orphans = (ranked*)malloc(sizeof(ranked) * (size_t)(N > 0 ? N : 1));
    ranked* donors = (ranked*)malloc(sizeof(ranked) * (size_t)(N > 0 ? N : 1));
    int n_orphans = 0, n_donors = 0;
    for (int i = 0; i < N; ++i) {
        int retained = mask[i] != 0;
        int protected_pos = (i < n_sink) || (i >= N - n_recent);
        int orphan = !retained && (b[i] < tau);
        int donor = retained && !protected_pos && (b[i] >= tau);
        if (orphan) {
            orphans[n_orphans].b = b[i];
            orphans[n_orphans].pos = i;
            ++n_orphans;
        }
        if (donor) {
            donors[n_donors].b = b[i];
            donors[n_donors].pos = i;
            ++n_donors;
        }
        if (is_orphan) is_orphan[i] = (uint8_t)orphan;
        if (is_donor) is_donor[i] = (uint8_t)donor;
    }
    qsort(orphans, (size_t)n_orphans, sizeof(ranked), cmp_orphan);
    qsort(donors, (size_t)n_donors, sizeof(ranked), cmp_donor);
    int m = n_orphans < n_donors ? n_orphans : n_donors;
    for (int i = 0; i < N; ++i)
        out_mask[i] = mask[i];
    for (int k = 0; k < m; ++k) {
        out_mask[donors[k].pos] = 0;
        out_mask[orphans[k].pos] = 1;
        swaps[2 * k] = donors[k].pos;
        swaps[2 * k + 1] = orphans[k].pos;
    }
    free(orphans);
    free(donors);
    return m;
}

/*
 * Repair over U units.  b[U][N] in double; budget[U] (or NULL = no check); the
 * per-unit swap list has room for N/2 pairs (m <= min(K, N-K) <= N/2), so
 * swaps is [U][N/2][2].  status[u]: 0 ok, 1 mask value outside {0,1}, 3 popcount of
 * the mask differs from budget[u]; a failed unit gets nswaps = -1 and S1 = S0.
 */
void twk_oracle_repair(int U, int N, const double* b, const uint8_t* mask,
                       const int32_t* budget, float threshold, int n_sink, int n_recent,
                       uint8_t* out_mask, int32_t* swaps, int32_t* nswaps, int32_t* status,
                       uint8_t* is_orphan, uint8_t* is_donor)
{
    double tau = (double)threshold;
    long cap = 2L * (N / 2);
    for (int u = 0; u < U; ++u) {
        const uint8_t* S0 = mask + (long)u * N;
        int bad_value = 0, count = 0;
        for (int i = 0; i < N; ++i) {
            if (S0[i] > 1) bad_value = 1;
            count += S0[i] != 0;
        }
        int st = 0;
        if (bad_value)
            st = 1;
        else if (budget && budget[u] != count)
            st = 3;
        status[u] = st;
        if (st != 0) {
            memcpy(out_mask + (long)u * N, S0, (size_t)N);
            nswaps[u] = -1;
            if (is_orphan) memset(is_orphan + (long)u * N, 0, (size_t)N);
            if (is_donor) memset(is_donor + (long)u * N, 0, (size_t)N);
            continue;
        }
        nswaps[u] = repair_unit(N, b + (long)u * N, S0, tau, n_sink, n_recent,
                                out_mask + (long)u * N, swaps + (long)u * cap,
                                is_orphan ? is_orphan + (long)u * N : NULL,
                                is_donor ? is_donor + (long)u * N : NULL);
    }
}

/* Selection-only entry: the same repair on float32 b values (for example, a GPU's own
 * b), widened exactly to double, so every comparison equals the float comparison. */
void twk_oracle_repair_f32(int U, int N, const float* b, const uint8_t* mask,
                           const int32_t* budget, float threshold, int n_sink, int n_recent,
                           uint8_t* out_mask, int32_t* swaps, int32_t* nswaps,
                           int32_t* status, uint8_t* is_orphan, uint8_t* is_donor)
{
    long n = (long)U * N;
    double* bd = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    for (long t = 0; t < n; ++t)
        bd[t] = (double)b[t];
    twk_oracle_repair(U, N, bd, mask, budget, threshold, n_sink, n_recent, out_mask, swaps,
                      nswaps, status, is_orphan, is_donor);
    free(bd);
}

/* ---- Sec. 3.2, Eq. 2-3: the standalone redundancy policy ----------------------- */

/*
 * Redundancy counts of Eq. 2.  For each unit u and requested row i:
 *   r[i]    = #{ j : |i-j| > w, j != i, sim(i,j) > tau }     (Eq. 2, strict)
 *   r_lo[i] = the same count with tau + band in place of tau
 *   r_hi[i] = the same count with tau - band in place of tau
 * so that r_lo <= r <= r_hi, and a count taken in lower precision lies in
 * [r_lo, r_hi] whenever its similarity errors stay below band.  tau is the
 * threshold rounded to float and widened.  rows as in twk_oracle_audit; r_lo and
 * r_hi may be NULL.  out: [U][nrows].
 */
void twk_oracle_count(const uint16_t* keys, int U, int N, int d, int window, float threshold,
                      double band, const int32_t* rows, int nrows, int32_t* r,
                      int32_t* r_lo, int32_t* r_hi)
{
    const double tau = (double)threshold;
    if (rows == NULL)
        nrows = N;
    double* sq = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
    for (int u = 0; u < U; ++u) {
        const uint16_t* K = keys + (long)u * N * d;
        for (int i = 0; i < N; ++i)
            sq[i] = dot_bf16(&K[(long)i * d], &K[(long)i * d], d);
#pragma omp parallel for schedule(dynamic, 8)
        for (int q = 0; q < nrows; ++q) {
            int i = rows ? rows[q] : q;
            int c = 0, c_lo = 0, c_hi = 0;
            for (int j = 0; j < N; ++j) {
                int dist = (i > j) ? i - j : j - i;
                if (j == i || dist <= window)
                    continue;
                double s = cosine(dot_bf16(&K[(long)i * d], &K[(long)j * d], d), sq[i], sq[j]);
                c += s > tau;
                c_lo += s > tau + band;
                c_hi += s > tau - band;
            }
            long o = (long)u * nrows + q;
            r[o] = c;
            if (r_lo) r_lo[o] = c_lo;
            if (r_hi) r_hi[o] = c_hi;
        }
    }
    free(sq);
}

typedef struct {
    int32_t prot;   /* 1 for a sink or recent position */
    int32_t r;
    int32_t pos;
} policy_rank;

/* Protected positions all carry the maximum score (Sec. 3.2), so they come first and
 * tie among themselves; unprotected ones follow by fewer twins (higher s = -r/n);
 * equal scores go by lower position. */
static int cmp_policy(const void* pa, const void* pb)
{
    const policy_rank* a = (const policy_rank*)pa;
    const policy_rank* b = (const policy_rank*)pb;
    if (a->prot != b->prot) return b->prot - a->prot;
    if (!a->prot && a->r != b->r) return (a->r > b->r) - (a->r < b->r);
    return (a->pos > b->pos) - (a->pos < b->pos);
}

/*
 * The standalone policy of Sec. 3.2: from the counts r[U][N] (Eq. 2), keep budget[u]
 * positions of each unit, ordered by (protected first, s = -r/N descending, position
 * ascending).  Protected: i < n_sink or i >= N - n_recent.  out_mask[U][N] gets 1 for
 * a kept position.  status[u]: 0 ok, 1 when budget[u] is outside [0, N] (then the
 * unit's mask is all 0).
 */
void twk_oracle_policy_select(int U, int N, const int32_t* r, int n_sink, int n_recent,
                              const int32_t* budget, uint8_t* out_mask, int32_t* status)
{
    policy_rank* e = (policy_rank*)malloc(sizeof(policy_rank) * (size_t)(N > 0 ? N : 1));
    for (int u = 0; u < U; ++u) {
        uint8_t* S = out_mask + (long)u * N;
        memset(S, 0, (size_t)N);
        const int K = budget[u];
        if (K < 0 || K > N) {
            status[u] = 1;
            continue;
        }
        status[u] = 0;
        for (int i = 0; i < N; ++i) {
            e[i].prot = (i < n_sink) || (i >= N - n_recent);
            e[i].r = r[(long)u * N + i];
            e[i].pos = i;
        }
        qsort(e, (size_t)N, sizeof(policy_rank), cmp_policy);
        for (int k = 0; k < K; ++k)
            S[e[k].pos] = 1;
    }
    free(e);
}

/* ---- Sec. 3.4 variant: the repair without evicting both members of a twin pair -- */

/*
 * Like twk_oracle_repair, with twin[U][N] = the argmax of b_i(S0) (Eq. 4) per
 * position.  Donors are walked in severity order (b descending, position ascending);
 * a donor is skipped when its twin has already been accepted for eviction in this
 * walk, or when it is itself the twin of an accepted donor; the walk stops once |O|
 * donors are accepted.  m = the number accepted; the m
 * most severe orphans are admitted, the k-th accepted donor paired with the k-th
 * orphan.  Status handling as in twk_oracle_repair.
 */
void twk_oracle_repair_dedup(int U, int N, const double* b, const int32_t* twin,
                             const uint8_t* mask, const int32_t* budget, float threshold,
                             int n_sink, int n_recent, uint8_t* out_mask, int32_t* swaps,
                             int32_t* nswaps, int32_t* status)
{
    const double tau = (double)threshold;
    const long cap = 2L * (N / 2);
    ranked* orphans = (ranked*)malloc(sizeof(ranked) * (size_t)(N > 0 ? N : 1));
    ranked* donors = (ranked*)malloc(sizeof(ranked) * (size_t)(N > 0 ? N : 1));
    uint8_t* evicted = (uint8_t*)malloc((size_t)(N > 0 ? N : 1));
    uint8_t* pinned = (uint8_t*)malloc((size_t)(N > 0 ? N : 1));
    for (int u = 0; u < U; ++u) {
        const uint8_t* S0 = mask + (long)u * N;
        const double* bu = b + (long)u * N;
        const int32_t* tw = twin + (long)u * N;
        uint8_t* S1 = out_mask + (long)u * N;
        int32_t* sw = swaps + (long)u * cap;
        int bad_value = 0, count = 0;
        for (int i = 0; i < N; ++i) {
            if (S0[i] > 1) bad_value = 1;
            count += S0[i] != 0;
        }
        int st = 0;
        if (bad_value)
            st = 1;
        else if (budget && budget[u] != count)
            st = 3;
        status[u] = st;
        memcpy(S1, S0, (size_t)N);
        if (st != 0) {
            nswaps[u] = -1;
            continue;
        }
        int n_o = 0, n_d = 0;
        for (int i = 0; i < N; ++i) {
            int retained = S0[i] != 0;
            int protected_pos = (i < n_sink) || (i >= N - n_recent);
            if (!retained && bu[i] < tau) {
                orphans[n_o].b = bu[i];
                orphans[n_o].pos = i;
                ++n_o;
            }
            if (retained && !protected_pos && bu[i] >= tau) {
                donors[n_d].b = bu[i];
                donors[n_d].pos = i;
                ++n_d;
            }
        }
        qsort(orphans, (size_t)n_o, sizeof(ranked), cmp_orphan);
        qsort(donors, (size_t)n_d, sizeof(ranked), cmp_donor);
        memset(evicted, 0, (size_t)N);
        memset(pinned, 0, (size_t)N);
        int m = 0;
        for (int k = 0; k < n_d && m < n_o; ++k) {
            int d = donors[k].pos;
            int t = tw[d];
            int has_twin = t >= 0 && t < N;
            if (pinned[d] || (has_twin && evicted[t]))
                continue;
            evicted[d] = 1;
            if (has_twin)
                pinned[t] = 1;
            sw[2 * m] = d;
            ++m;
        }
        for (int k = 0; k < m; ++k) {
            sw[2 * k + 1] = orphans[k].pos;
            S1[sw[2 * k]] = 0;
            S1[orphans[k].pos] = 1;
        }
        nswaps[u] = m;
    }
    free(orphans);
    free(donors);
    free(evicted);
    free(pinned);
}
