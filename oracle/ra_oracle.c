/*
 * ra_oracle.c -- the CPU oracle for Random Attention's decode hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, plain, single-threaded
 * statement of what the GPU library computes.  Only the tests, the smoke
 * check and the benchmark's CPU-baseline leg may load it; the product path
 * never does.  It shares no code, header, table or helper with the CUDA
 * library: everything below is written out from the paper (and, for the
 * counter-based generator, from its published definition).
 *
 * What it states:
 *   - Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers:
 *     as easy as 1, 2, 3", SC'11): the per-candidate random score.
 *   - Random Attention's selection (paper section 3): every evictable
 *     candidate gets an i.i.d. uniform score, the K best are kept
 *     (Eq. 1, section 2 "Periodic eviction with budget K and buffer r").
 *     Scores are 32-bit Philox words; "best" = smallest (key, ordinal),
 *     which draws a uniform K-subset exactly as a real-valued
 *     Uniform(0,1) top-K does.
 *   - The periodic trigger and the chronological compaction
 *     (section 2 and Appendix F "Engine details": every r steps, once the
 *     cache exceeds the budget plus the buffer; keep-sets sorted
 *     chronologically before the gather).
 *   - Decode attention o = sum_i softmax_i(q.k_i / sqrt(d)) v_i in fp64
 *     (section 2 "Notation"), grouped-query: a KV head's keep-set serves
 *     every query head of its group (Appendix F).
 *   - Order-free (hole-filling) compaction: keys drawn per position, the
 *     evicted slots refilled from the newest ones, the newest row kept in the
 *     last slot (attention is a sum over the cached set, so slot order
 *     carries nothing).
 *   - The scored comparator (section 2, "Baselines as choices of s"): the
 *     SnapKV score -- attention received from the last w queries, summed
 *     over the query heads of the group, max-pooled over neighbouring
 *     positions -- and a top-K by that score, with the prompt pinned.
 *
 * Parity status: every function here is pinned by the "not gpu" tests
 * (Philox against an independent Philox implementation, selection by brute
 * force and by the paper's closed-form survival law, attention by closed
 * forms and an independent library softmax, window scores by closed forms
 * and a brute-force softmax, pooling and top-K by hand-worked cases).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------- */
/* Philox4x32-10 (SC'11, section 3.3 of that paper).                          */
/* Round: two 32x32->64 multiplies by fixed multipliers, the high halves     */
/* xored with the other two words and the round key; the key is bumped by    */
/* two Weyl constants between rounds.                                        */
/* ------------------------------------------------------------------------- */
#define PHILOX_M4x32_0 0xD2511F53u
#define PHILOX_M4x32_1 0xCD9E8D57u
#define PHILOX_W32_0 0x9E3779B9u /* golden ratio */
#define PHILOX_W32_1 0xBB67AE85u /* sqrt(3) - 1 */

void ora_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    for (int round = 0; round < 10; ++round) {
        if (round > 0) {
            k0 += PHILOX_W32_0;
            k1 += PHILOX_W32_1;
        }
        uint64_t p0 = (uint64_t)PHILOX_M4x32_0 * (uint64_t)x0;
        uint64_t p1 = (uint64_t)PHILOX_M4x32_1 * (uint64_t)x2;
        uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        uint32_t y0 = hi1 ^ x1 ^ k0;
        uint32_t y1 = lo1;
        uint32_t y2 = hi0 ^ x3 ^ k1;
        uint32_t y3 = lo0;
        x0 = y0; x1 = y1; x2 = y2; x3 = y3;
    }
    out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/*
 * The random score of one candidate (section 3: s_i ~ Uniform(0,1), drawn
 * independently per KV head at every eviction).  The paper does not fix a
 * generator; this library's mapping is
 *     counter = (j, step, layer, head_id),  key = (seed_lo, seed_hi),
 *     score   = word 0 of Philox4x32-10,
 * with j the candidate's ordinal in slot order, step = number of generated
 * tokens appended when the eviction fires, and head_id = seq * kv_heads + h for
 * the batch a context starts with.  A request admitted into a slot later draws
 * its own stream: head_id = (a << 16) | (seq * kv_heads + h), a = the requests
 * the slot took before (the paper's per-request seed, Appendix H; ora_head_stream).
 */
uint32_t ora_head_stream(uint32_t admissions, uint32_t head) { return (admissions << 16) | head; }

uint32_t ora_random_key(uint64_t seed, uint32_t layer, uint32_t head_id, uint32_t step, uint32_t j)
{
    uint32_t ctr[4] = {j, step, layer, head_id};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t out[4];
    ora_philox4x32_10(ctr, key, out);
    return out[0];
}

/*
 * Scores of the policy variants the paper contrasts with Random Attention
 * (section 5 and Appendix D), all kept through the same Eq. 1 top-K:
 *   0 random   -- the method: an independent draw per KV head (see above);
 *   1 shared   -- the shared-draw control: one draw per (sequence, layer) that
 *                 every KV head uses (head_id = seq * kv_heads for all heads);
 *   2 recency  -- protected recency: the prompt plus the most recent window,
 *                 i.e. the K newest candidates (score N - 1 - j);
 *   3 block    -- history kept in contiguous blocks: every candidate of one
 *                 block of `block` consecutive positions shares one draw
 *                 (counter word 0 = position / block).
 * Ties of equal score go to the lower ordinal, as everywhere.
 */
uint32_t ora_policy_key(int policy, uint64_t seed, uint32_t layer, uint32_t seq, uint32_t kv_heads, uint32_t h,
                        uint32_t step, uint32_t j, uint32_t n_cand, int32_t position, int32_t block, uint32_t admissions)
{
    switch (policy) {
        case 1:
            return ora_random_key(seed, layer, ora_head_stream(admissions, seq * kv_heads), step, j);
        case 2:
            return n_cand - 1u - j;
        case 3:
            return ora_random_key(seed, layer, ora_head_stream(admissions, seq * kv_heads + h), step,
                                  (uint32_t)(position / block));
        default:
            return ora_random_key(seed, layer, ora_head_stream(admissions, seq * kv_heads + h), step, j);
    }
}

/* ------------------------------------------------------------------------- */
/* Selection: Eq. 1, S_t = top-K over the candidates of s_i.                 */
/* ------------------------------------------------------------------------- */
typedef struct {
    uint32_t key;
    int32_t ordinal;
} ora_cand;

static int ora_cmp_cand(const void* a, const void* b)
{
    const ora_cand* x = (const ora_cand*)a;
    const ora_cand* y = (const ora_cand*)b;
    if (x->key != y->key) return x->key < y->key ? -1 : 1;
    return x->ordinal < y->ordinal ? -1 : (x->ordinal > y->ordinal ? 1 : 0);
}

static int ora_cmp_i32(const void* a, const void* b)
{
    int32_t x = *(const int32_t*)a, y = *(const int32_t*)b;
    return x < y ? -1 : (x > y ? 1 : 0);
}

/*
 * Keep the K candidates with the smallest (key, ordinal), returned in
 * ascending ordinal order (Appendix F orders each keep-set by time before the
 * cache is compacted).  The plain definition: sort all, take K.
 * Returns 0, or -1 on bad arguments / allocation failure.
 */
int ora_select_keep(const uint32_t* keys, int n, int K, int32_t* keep_out)
{
    if (n < 0 || K < 0 || K > n) return -1;
    if (K == 0) return 0;
    ora_cand* c = (ora_cand*)malloc(sizeof(ora_cand) * (size_t)n);
    if (!c) return -1;
    for (int j = 0; j < n; ++j) {
        c[j].key = keys[j];
        c[j].ordinal = j;
    }
    qsort(c, (size_t)n, sizeof(ora_cand), ora_cmp_cand);
    for (int i = 0; i < K; ++i) keep_out[i] = c[i].ordinal;
    free(c);
    qsort(keep_out, (size_t)K, sizeof(int32_t), ora_cmp_i32);
    return 0;
}

/*
 * The periodic trigger (section 2: an eviction runs each time the r-token
 * buffer has filled; Appendix F: every r = 64 decode steps once the cache
 * holds more than K + r).  `c` counts the cached generated tokens, `g` the
 * generated tokens appended so far; the check runs after the step's append.
 * Fires iff g is a multiple of r and the candidates (everything but the
 * newest r) outnumber the budget.
 */
int ora_should_evict(int g, int c, int K, int r)
{
    return (r > 0) && (g > 0) && (g % r == 0) && (c - r > K);
}

/*
 * One eviction round for one (sequence, layer, KV head).
 *   gen[0..*c)  positions of the cached generated tokens, in slot order
 *               (ascending position); the prompt is not in this list -- it is
 *               never a candidate (section 3: the prompt is protected).
 * If the trigger fires: candidates are gen[0 .. c-r) (everything outside the
 * recent buffer), each gets its Philox score, the K smallest survive, and
 * gen becomes kept-candidates ++ the r buffer positions, in order.
 * evicted_out (may be NULL) receives the m evicted ordinals, ascending.
 * Returns m (0 when the trigger does not fire), or -1 on error.
 */
int ora_evict_head(int32_t* gen, int* c, int g, int K, int r, uint64_t seed, int layer,
                   int head_id, int32_t* evicted_out)
{
    int cc = *c;
    if (!ora_should_evict(g, cc, K, r)) return 0;
    int n = cc - r;
    uint32_t* keys = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)n);
    int32_t* keep = (int32_t*)malloc(sizeof(int32_t) * (size_t)(K > 0 ? K : 1));
    int32_t* next = (int32_t*)malloc(sizeof(int32_t) * (size_t)(K + r));
    if (!keys || !keep || !next) {
        free(keys); free(keep); free(next);
        return -1;
    }
    for (int j = 0; j < n; ++j)
        keys[j] = ora_random_key(seed, (uint32_t)layer, (uint32_t)head_id, (uint32_t)g, (uint32_t)j);
    if (ora_select_keep(keys, n, K, keep) != 0) {
        free(keys); free(keep); free(next);
        return -1;
    }
    int m = 0, ki = 0;
    for (int j = 0; j < n; ++j) {
        if (ki < K && keep[ki] == j) {
            next[ki] = gen[j];
            ++ki;
        } else {
            if (evicted_out) evicted_out[m] = j;
            ++m;
        }
    }
    for (int i = 0; i < r; ++i) next[K + i] = gen[n + i];
    memcpy(gen, next, sizeof(int32_t) * (size_t)(K + r));
    *c = K + r;
    free(keys); free(keep); free(next);
    return m;
}

/*
 * One eviction round under a policy variant (see ora_policy_key); same trigger,
 * candidates and compaction as ora_evict_head.
 */
int ora_evict_head_policy(int32_t* gen, int* c, int g, int K, int r, uint64_t seed, int layer, int seq,
                          int kv_heads, int h, int policy, int block, uint32_t admissions, int32_t* evicted_out)
{
    int cc = *c;
    if (!ora_should_evict(g, cc, K, r)) return 0;
    if (policy == 3 && block < 1) return -1;
    int n = cc - r;
    uint32_t* keys = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)n);
    int32_t* keep = (int32_t*)malloc(sizeof(int32_t) * (size_t)(K > 0 ? K : 1));
    int32_t* next = (int32_t*)malloc(sizeof(int32_t) * (size_t)(K + r));
    if (!keys || !keep || !next) {
        free(keys); free(keep); free(next);
        return -1;
    }
    for (int j = 0; j < n; ++j)
        keys[j] = ora_policy_key(policy, seed, (uint32_t)layer, (uint32_t)seq, (uint32_t)kv_heads, (uint32_t)h,
                                 (uint32_t)g, (uint32_t)j, (uint32_t)n, gen[j], block, admissions);
    if (ora_select_keep(keys, n, K, keep) != 0) {
        free(keys); free(keep); free(next);
        return -1;
    }
    int m = 0, ki = 0;
    for (int j = 0; j < n; ++j) {
        if (ki < K && keep[ki] == j) {
            next[ki] = gen[j];
            ++ki;
        } else {
            if (evicted_out) evicted_out[m] = j;
            ++m;
        }
    }
    for (int i = 0; i < r; ++i) next[K + i] = gen[n + i];
    memcpy(gen, next, sizeof(int32_t) * (size_t)(K + r));
    *c = K + r;
    free(keys); free(keep); free(next);
    return m;
}

/* ------------------------------------------------------------------------- */
/* Decode attention (section 2, "Notation"), fp64.                           */
/* ------------------------------------------------------------------------- */
static double ora_bf16_to_double(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/*
 * o_g = sum_i softmax_i(scale * q_g . k_i) v_i for each query head g of one
 * GQA group: q [G][d], k and v [n][d] (bf16 bit patterns), out [G][d].
 * scale <= 0 means 1/sqrt(d).  n == 0 leaves out at zero.
 */
void ora_attend(const uint16_t* q, const uint16_t* k, const uint16_t* v, int n, int G, int d,
                double scale, double* out)
{
    if (scale <= 0.0) scale = 1.0 / sqrt((double)d);
    double* s = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    for (int g = 0; g < G; ++g) {
        double* o = out + (size_t)g * d;
        for (int c = 0; c < d; ++c) o[c] = 0.0;
        if (n == 0 || !s) continue;
        double mx = -INFINITY;
        for (int i = 0; i < n; ++i) {
            double dot = 0.0;
            for (int c = 0; c < d; ++c)
                dot += ora_bf16_to_double(q[(size_t)g * d + c]) * ora_bf16_to_double(k[(size_t)i * d + c]);
            s[i] = scale * dot;
            if (s[i] > mx) mx = s[i];
        }
        double den = 0.0;
        for (int i = 0; i < n; ++i) {
            double w = exp(s[i] - mx);
            den += w;
            for (int c = 0; c < d; ++c) o[c] += w * ora_bf16_to_double(v[(size_t)i * d + c]);
        }
        for (int c = 0; c < d; ++c) o[c] /= den;
    }
    free(s);
}

/* ------------------------------------------------------------------------- */
/* Scored comparator (section 2, "Baselines as choices of s"): the SnapKV     */
/* score, the attention that the last w queries give each cached position,    */
/* max-pooled over neighbouring positions, then the K best kept.  The prompt  */
/* stays pinned and the buffer unscored, as in Random Attention, so the two   */
/* policies differ only in how candidates are ranked.                         */
/* ------------------------------------------------------------------------- */

/*
 * score[i] = sum over window queries u and query heads g of alpha_i(u, g), with
 *   alpha_i(u, g) = exp(scale * q_ug . k_i) / sum_{i': pos_i' <= qpos_u} exp(scale * q_ug . k_i')
 * when pos_i <= qpos_u (a decoding query sees no later position) and 0
 * otherwise.  q [n_q][G][d] and k [n_k][d] are bf16 bit patterns; q_pos [n_q]
 * and k_pos [n_k] are token positions; score [n_k] is fp64.  scale <= 0 means
 * 1/sqrt(d).  Every key, the prompt's included, takes part in the softmax;
 * the caller reads the entries of the candidates.
 */
void ora_window_scores(const uint16_t* q, const int32_t* q_pos, int n_q, int G, const uint16_t* k,
                       const int32_t* k_pos, int n_k, int d, double scale, double* score)
{
    if (scale <= 0.0) scale = 1.0 / sqrt((double)d);
    for (int i = 0; i < n_k; ++i) score[i] = 0.0;
    double* logit = (double*)malloc(sizeof(double) * (size_t)(n_k > 0 ? n_k : 1));
    if (!logit) return;
    for (int u = 0; u < n_q; ++u) {
        for (int g = 0; g < G; ++g) {
            const uint16_t* qr = q + ((size_t)u * G + g) * d;
            double mx = -INFINITY;
            for (int i = 0; i < n_k; ++i) {
                if (k_pos[i] > q_pos[u]) continue;
                double dot = 0.0;
                for (int c = 0; c < d; ++c)
                    dot += ora_bf16_to_double(qr[c]) * ora_bf16_to_double(k[(size_t)i * d + c]);
                logit[i] = scale * dot;
                if (logit[i] > mx) mx = logit[i];
            }
            if (mx == -INFINITY) continue; /* the query sees no key */
            double den = 0.0;
            for (int i = 0; i < n_k; ++i)
                if (k_pos[i] <= q_pos[u]) den += exp(logit[i] - mx);
            for (int i = 0; i < n_k; ++i)
                if (k_pos[i] <= q_pos[u]) score[i] += exp(logit[i] - mx) / den;
        }
    }
    free(logit);
}

/* out[i] = max of s[j] over |j - i| <= radius, 0 <= j < n (a window clipped at the ends). */
void ora_max_pool(const double* s, int n, int radius, double* out)
{
    for (int i = 0; i < n; ++i) {
        double m = s[i];
        for (int j = i - radius; j <= i + radius; ++j)
            if (j >= 0 && j < n && s[j] > m) m = s[j];
        out[i] = m;
    }
}

typedef struct {
    double s;
    int32_t i;
} ora_scored;

static int ora_cmp_scored(const void* a, const void* b)
{
    const ora_scored* x = (const ora_scored*)a;
    const ora_scored* y = (const ora_scored*)b;
    if (x->s != y->s) return x->s > y->s ? -1 : 1; /* larger score first */
    return (x->i > y->i) - (x->i < y->i);           /* then the earlier position */
}

/*
 * Top-K by score: the K largest of s[0..n), equal scores going to the lower
 * index.  keep_out receives the K indices in ascending (chronological) order.
 * Returns 0, or -1 on bad arguments.
 */
int ora_select_top(const double* s, int n, int K, int32_t* keep_out)
{
    if (n < 0 || K < 0 || K > n) return -1;
    ora_scored* a = (ora_scored*)malloc(sizeof(ora_scored) * (size_t)(n > 0 ? n : 1));
    if (!a) return -1;
    for (int i = 0; i < n; ++i) {
        a[i].s = s[i];
        a[i].i = i;
    }
    qsort(a, (size_t)n, sizeof(ora_scored), ora_cmp_scored);
    for (int i = 0; i < K; ++i) keep_out[i] = a[i].i;
    free(a);
    qsort(keep_out, (size_t)K, sizeof(int32_t), ora_cmp_i32);
    return 0;
}

/*
 * One scored eviction round of one head, the same cadence and compaction as
 * ora_evict_head but ranked by score: raw[0..n) holds the window score of each
 * candidate (n = c - r), pooled over +-radius neighbours; the K best survive.
 * Returns the number evicted (0 when the trigger does not fire), -1 on error.
 */
int ora_evict_head_scored(int32_t* gen, int* c, int g, int K, int r, const double* raw, int radius,
                          int32_t* evicted_out)
{
    const int cc = *c;
    if (!ora_should_evict(g, cc, K, r)) return 0;
    const int n = cc - r;
    double* pooled = (double*)malloc(sizeof(double) * (size_t)n);
    int32_t* keep = (int32_t*)malloc(sizeof(int32_t) * (size_t)(K > 0 ? K : 1));
    int32_t* next = (int32_t*)malloc(sizeof(int32_t) * (size_t)(K + r));
    if (!pooled || !keep || !next) {
        free(pooled); free(keep); free(next);
        return -1;
    }
    ora_max_pool(raw, n, radius, pooled);
    if (ora_select_top(pooled, n, K, keep) != 0) {
        free(pooled); free(keep); free(next);
        return -1;
    }
    int m = 0, ki = 0;
    for (int j = 0; j < n; ++j) {
        if (ki < K && keep[ki] == j) {
            next[ki++] = gen[j];
        } else {
            if (evicted_out) evicted_out[m] = j;
            ++m;
        }
    }
    for (int i = 0; i < r; ++i) next[K + i] = gen[n + i];
    memcpy(gen, next, sizeof(int32_t) * (size_t)(K + r));
    *c = K + r;
    free(pooled); free(keep); free(next);
    return m;
}

/* ------------------------------------------------------------------------- */
/* Order-free compaction.  Attention is a sum over the cached set (section 2, */
/* "Notation"), so the slots need no chronological order; the keep-set is a   */
/* random subset of positions -- in Appendix G's terms, a random permutation  */
/* of slot indices.  Keys are drawn per position, so the kept set does not    */
/* depend on the slot layout.                                                 */
/* ------------------------------------------------------------------------- */

/*
 * Policy score of the candidate at `position` when slots carry no order:
 *   0 random  -- Philox word 0 of counter (position, step, layer, seq * kv_heads + h);
 *   1 shared  -- the same with head id seq * kv_heads for every head;
 *   2 recency -- the newest positions score lowest: 0xFFFFFFFF - position;
 *   3 block   -- as ordered: counter word 0 = position / block.
 */
uint32_t ora_position_key(int policy, uint64_t seed, uint32_t layer, uint32_t seq, uint32_t kv_heads, uint32_t h,
                          uint32_t step, int32_t position, int32_t block, uint32_t admissions)
{
    switch (policy) {
        case 1:
            return ora_random_key(seed, layer, ora_head_stream(admissions, seq * kv_heads), step, (uint32_t)position);
        case 2:
            return 0xFFFFFFFFu - (uint32_t)position;
        case 3:
            return ora_random_key(seed, layer, ora_head_stream(admissions, seq * kv_heads + h), step,
                                  (uint32_t)(position / block));
        default:
            return ora_random_key(seed, layer, ora_head_stream(admissions, seq * kv_heads + h), step,
                                  (uint32_t)position);
    }
}

/*
 * One eviction round with hole-filling compaction.  Same trigger and the same
 * top-K (the K smallest (key, ordinal) among the n = c - r candidates, keys
 * by position).  The m = n - K evicted slots e_0 < ... < e_{m-1} are refilled
 * and the cache shrinks to c - m slots, the newest row (slot c - 1) ending in
 * the new last slot c - m - 1:
 *   - slot e_i takes the row of slot c - m + i, for i < m - 1;
 *   - if e_{m-1} is the new last slot, it takes the newest row; otherwise it
 *     takes the row of the new last slot, which then takes the newest row.
 * Every other slot keeps its row.  Defined for c <= K + 2r (the cache's
 * capacity), where m <= r and slots c - m .. c - 1 are all buffer slots.
 * Returns m (0 when the trigger does not fire) and the evicted ordinals, -1 on
 * error.
 */
int ora_evict_head_holefill(int32_t* gen, int* c, int g, int K, int r, uint64_t seed, int layer, int seq,
                            int kv_heads, int h, int policy, int block, uint32_t admissions, int32_t* evicted_out)
{
    const int cc = *c;
    if (!ora_should_evict(g, cc, K, r)) return 0;
    if (policy == 3 && block < 1) return -1;
    const int n = cc - r;
    if (n - K > r) return -1; /* the newest m slots must all be buffer slots: c <= K + 2r */
    uint32_t* keys = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)n);
    int32_t* keep = (int32_t*)malloc(sizeof(int32_t) * (size_t)(K > 0 ? K : 1));
    int32_t* ev = (int32_t*)malloc(sizeof(int32_t) * (size_t)n);
    if (!keys || !keep || !ev) {
        free(keys); free(keep); free(ev);
        return -1;
    }
    for (int j = 0; j < n; ++j)
        keys[j] = ora_position_key(policy, seed, (uint32_t)layer, (uint32_t)seq, (uint32_t)kv_heads, (uint32_t)h,
                                   (uint32_t)g, gen[j], block, admissions);
    if (ora_select_keep(keys, n, K, keep) != 0) {
        free(keys); free(keep); free(ev);
        return -1;
    }
    int m = 0, ki = 0;
    for (int j = 0; j < n; ++j) {
        if (ki < K && keep[ki] == j) ++ki;
        else ev[m++] = j;
    }
    const int last = cc - m - 1; /* the new last slot */
    for (int i = 0; i < m; ++i) {
        if (i < m - 1) {
            gen[ev[i]] = gen[cc - m + i];
        } else if (ev[i] == last) {
            gen[last] = gen[cc - 1];
        } else {
            gen[ev[i]] = gen[last];
            gen[last] = gen[cc - 1];
        }
        if (evicted_out) evicted_out[i] = ev[i];
    }
    *c = cc - m;
    free(keys); free(keep); free(ev);
    return m;
}
