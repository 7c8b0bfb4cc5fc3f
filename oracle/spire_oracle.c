/*
 * spire_oracle.c -- plain fp64 CPU oracle for the attention of one SPIRe
 * speculation round (Neelam et al., "SPIRe: Boosting LLM Inference Throughput
 * with Speculative Decoding", arXiv 2504.06419).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously correct
 * reference that the CUDA path is checked against.  Only the tests, the smoke
 * check and the benchmark's CPU-baseline leg may load it.  It shares no code,
 * header, table or helper with the CUDA library, and the CUDA library never
 * calls it.
 *
 * Everything is computed in double precision.  bf16 inputs are widened
 * exactly (a bf16 value is the top 16 bits of an IEEE binary32).  Softmax is
 * two-pass: first the maximum score, then exp-sum and the weighted sum of
 * values.  Keys are visited in increasing logical position.
 *
 * What each function follows:
 *   oracle_verify      -- the verification pass of a speculation round:
 *                         the target model runs on the k+1 block tokens in
 *                         parallel (Section 2, definition of t_verify next to
 *                         the Throughput Multiplier equation; Fig. 1 caption;
 *                         Table 1 caption), each block token attending
 *                         causally to the full KV cache (KV_target term of the
 *                         implementation-agnostic multiplier, Section 2).
 *   oracle_draft_*     -- the draft model's StreamingLLM attention mask:
 *                         attention sinks plus a sliding window, so the draft
 *                         KV cache has constant size (Section 3.1; Section 4,
 *                         items 2 and 3), over feedback-memory entries m_{<t}
 *                         (Section 3.3, the Feedback Transformer attention
 *                         equation and the per-layer memory equation).
 *   oracle_draft_slot  -- where logical memory position p lives in the
 *                         bounded cache (sinks fixed, window a ring).
 *   oracle_feedback_*  -- the draft step's memory vector and its K/V entry in
 *                         the bounded cache (Section 3.3).
 *   oracle_verify_tokens -- modified rejection sampling of a round's draft
 *                         tokens (Section 1; Section 6).
 *   oracle_magicdec    -- the MagicDec baseline's draft attention: sink +
 *                         window over the target's own paged cache, positions
 *                         inside the reduced cache (Section 3.1 footnote).
 *
 * Readings of points the paper leaves open:
 *   - scores are softmax_scale * <q, k>; the workloads pre-scale q, scale = 1;
 *   - verify ctx_lens[b] = L counts the cache entries including the k+1 block
 *     tokens; block row i (0..k) sees keys j < L - k + i;
 *   - GQA: query head h uses KV head h / (Hq / Hkv);
 *   - draft ctx_lens[b] = t is the number of memory entries m_0..m_{t-1};
 *     the visible set is V(t) = {p < min(n_sink, t)} u {max(0, t-window) <= p < t};
 *   - a sequence whose length breaks the rules (verify: L < k+1 or
 *     L > max_pages*page_size; draft: t < 1) or whose block table points
 *     outside the cache gets NaN in all of its output rows and the function
 *     returns a nonzero count of such sequences.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ---- exact bf16 -> double ---------------------------------------------- */
static double bf16_to_double(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* ---- one softmax-weighted average over an explicit key list -------------
 * keys[j] / vals[j] point at D bf16 values; n >= 1.  out[d] receives
 * sum_j p_j v_j[d] with p = softmax(scale * <q, k_j>), two passes. */
static void attend(const uint16_t *q, const uint16_t *const *keys,
                   const uint16_t *const *vals, int64_t n, int32_t D,
                   double scale, double *scores, double *out)
{
    double m = -INFINITY;
    for (int64_t j = 0; j < n; ++j) {
        double s = 0.0;
        for (int32_t d = 0; d < D; ++d)
            s += bf16_to_double(q[d]) * bf16_to_double(keys[j][d]);
        s *= scale;
        scores[j] = s;
        if (s > m)
            m = s;
    }
    double l = 0.0;
    for (int32_t d = 0; d < D; ++d)
        out[d] = 0.0;
    for (int64_t j = 0; j < n; ++j) {
        double p = exp(scores[j] - m);
        l += p;
        for (int32_t d = 0; d < D; ++d)
            out[d] += p * bf16_to_double(vals[j][d]);
    }
    for (int32_t d = 0; d < D; ++d)
        out[d] /= l;
}

/* ---- a tiny thread pool over independent (b, h) units ------------------- */
typedef void (*unit_fn)(void *ctx, int64_t unit, double *scores,
                        const uint16_t **keys, const uint16_t **vals);

typedef struct {
    unit_fn fn;
    void *ctx;
    int64_t n_units;
    int64_t max_keys;
    const uint8_t *unit_mask;
    int64_t next;
    pthread_mutex_t lock;
} pool_t;

static void *pool_worker(void *arg)
{
    pool_t *p = (pool_t *)arg;
    int64_t cap = p->max_keys > 0 ? p->max_keys : 1;
    double *scores = (double *)malloc(sizeof(double) * (size_t)cap);
    const uint16_t **keys = (const uint16_t **)malloc(sizeof(void *) * (size_t)cap);
    const uint16_t **vals = (const uint16_t **)malloc(sizeof(void *) * (size_t)cap);
    if (!scores || !keys || !vals) {
        free(scores); free((void *)keys); free((void *)vals);
        return (void *)1;
    }
    for (;;) {
        pthread_mutex_lock(&p->lock);
        int64_t u = p->next++;
        pthread_mutex_unlock(&p->lock);
        if (u >= p->n_units)
            break;
        if (p->unit_mask && !p->unit_mask[u])
            continue;
        p->fn(p->ctx, u, scores, keys, vals);
    }
    free(scores); free((void *)keys); free((void *)vals);
    return NULL;
}

static int run_pool(unit_fn fn, void *ctx, int64_t n_units, int64_t max_keys,
                    const uint8_t *unit_mask, int32_t n_threads)
{
    pool_t p = {fn, ctx, n_units, max_keys, unit_mask, 0, PTHREAD_MUTEX_INITIALIZER};
    if (n_threads < 1)
        n_threads = 1;
    if (n_threads > 1024)
        n_threads = 1024;
    pthread_t tids[1024];
    int started = 0, failed = 0;
    for (int i = 0; i < n_threads; ++i) {
        if (pthread_create(&tids[i], NULL, pool_worker, &p) != 0)
            break;
        ++started;
    }
    if (started == 0) {
        if (pool_worker(&p) != NULL)
            failed = 1;
    }
    for (int i = 0; i < started; ++i) {
        void *ret = NULL;
        pthread_join(tids[i], &ret);
        if (ret != NULL)
            failed = 1;
    }
    return failed ? -1 : 0;
}

/* ======================================================================== */
/* Verification attention                                                    */
/* ======================================================================== */
typedef struct {
    const uint16_t *q, *k_cache, *v_cache;
    const int32_t *block_table, *ctx_lens;
    int32_t B, k, Hq, Hkv, D, page_size, max_pages, num_pages;
    double scale;
    double *out;
    int32_t *bad;           /* per sequence: 1 if its lengths/pages break the rules */
} verify_ctx;

/* Index of key j of sequence b, KV head g, inside a [num_pages, Hkv, P, D]
 * cache, through the block table.  Returns NULL for a page id outside the
 * cache. */
static const uint16_t *paged_row(const verify_ctx *c, const uint16_t *cache,
                                 int32_t b, int32_t g, int64_t j)
{
    int64_t page = c->block_table[(int64_t)b * c->max_pages + j / c->page_size];
    if (page < 0 || page >= c->num_pages)
        return NULL;
    int64_t slot = j % c->page_size;
    return cache + (((page * c->Hkv + g) * c->page_size + slot) * c->D);
}

static void verify_unit(void *vctx, int64_t unit, double *scores,
                        const uint16_t **keys, const uint16_t **vals)
{
    verify_ctx *c = (verify_ctx *)vctx;
    int32_t b = (int32_t)(unit / c->Hq);
    int32_t h = (int32_t)(unit % c->Hq);
    int32_t group = c->Hq / c->Hkv;
    int32_t g = h / group;
    int64_t L = c->ctx_lens[b];
    int32_t rows = c->k + 1;
    int valid = L >= rows && L <= (int64_t)c->max_pages * c->page_size;
    for (int32_t i = 0; valid && i < rows; ++i) {
        int64_t n_i = L - c->k + i;            /* keys visible to block row i */
        for (int64_t j = 0; j < n_i; ++j) {
            keys[j] = paged_row(c, c->k_cache, b, g, j);
            vals[j] = paged_row(c, c->v_cache, b, g, j);
            if (!keys[j] || !vals[j]) {
                valid = 0;
                break;
            }
        }
        if (!valid)
            break;
        const uint16_t *qi = c->q + (((int64_t)b * rows + i) * c->Hq + h) * c->D;
        double *oi = c->out + (((int64_t)b * rows + i) * c->Hq + h) * c->D;
        attend(qi, keys, vals, n_i, c->D, c->scale, scores, oi);
    }
    if (!valid) {
        c->bad[b] = 1;
        for (int32_t i = 0; i < rows; ++i) {
            double *oi = c->out + (((int64_t)b * rows + i) * c->Hq + h) * c->D;
            for (int32_t d = 0; d < c->D; ++d)
                oi[d] = NAN;
        }
    }
}

/*
 * oracle_verify: out[b, i, h, :] for b < B, block row i <= k, query head h.
 *   q        bf16 bits [B, k+1, Hq, D]
 *   k_cache  bf16 bits [num_pages, Hkv, page_size, D]   (v_cache alike)
 *   block_table int32 [B, max_pages]; ctx_lens int32 [B]
 *   unit_mask  NULL, or uint8 [B*Hq]: compute only (b, h) with mask != 0
 *              (other outputs are left untouched)
 *   out        double [B, k+1, Hq, D]
 * Returns the number of sequences whose inputs break the rules (their rows
 * are NaN), or -1 on bad arguments / allocation failure.
 */
int64_t oracle_verify(const uint16_t *q, const uint16_t *k_cache,
                      const uint16_t *v_cache, const int32_t *block_table,
                      const int32_t *ctx_lens, int32_t B, int32_t k, int32_t Hq,
                      int32_t Hkv, int32_t D, int32_t page_size,
                      int32_t max_pages, int32_t num_pages, double scale,
                      const uint8_t *unit_mask, double *out, int32_t n_threads)
{
    if (B < 0 || k < 0 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || D < 1 ||
        page_size < 1 || max_pages < 0 || num_pages < 0)
        return -1;
    if (B == 0)
        return 0;
    int32_t *bad = (int32_t *)calloc((size_t)B, sizeof(int32_t));
    if (!bad)
        return -1;
    verify_ctx c = {q, k_cache, v_cache, block_table, ctx_lens, B, k, Hq, Hkv,
                    D, page_size, max_pages, num_pages, scale, out, bad};
    int64_t max_keys = (int64_t)max_pages * page_size;
    int rc = run_pool(verify_unit, &c, (int64_t)B * Hq, max_keys, unit_mask, n_threads);
    int64_t n_bad = 0;
    for (int32_t b = 0; b < B; ++b)
        n_bad += bad[b];
    free(bad);
    return rc ? -1 : n_bad;
}

/* ======================================================================== */
/* Draft static sparse attention                                             */
/* ======================================================================== */

/* Slot of logical memory position p in a cache of n_sink fixed slots followed
 * by a ring of `window` slots. */
int64_t oracle_draft_slot(int64_t p, int32_t n_sink, int32_t window)
{
    if (p < n_sink)
        return p;
    return n_sink + (p - n_sink) % window;
}

/* Membership of logical position p in V(t): the first n_sink entries and the
 * last `window` entries of m_0..m_{t-1}. */
static int visible(int64_t p, int64_t t, int32_t n_sink, int32_t window)
{
    if (p < 0 || p >= t)
        return 0;
    return p < n_sink || p >= t - window;
}

typedef struct {
    const uint16_t *q;
    const uint16_t *k_src, *v_src;   /* logical [B,Hkv,T,D] x2, or ring [B,2,Hkv,S,D] */
    int ring;
    const int32_t *ctx_lens;
    int32_t B, Hq, Hkv, D, n_sink, window;
    int64_t T;                        /* logical length capacity (logical form) */
    double scale;
    double *out;
    int32_t *bad;
} draft_ctx;

static void draft_unit(void *vctx, int64_t unit, double *scores,
                       const uint16_t **keys, const uint16_t **vals)
{
    draft_ctx *c = (draft_ctx *)vctx;
    int32_t b = (int32_t)(unit / c->Hq);
    int32_t h = (int32_t)(unit % c->Hq);
    int32_t g = h / (c->Hq / c->Hkv);
    int64_t t = c->ctx_lens[b];
    int64_t S = (int64_t)c->n_sink + c->window;
    double *o = c->out + ((int64_t)b * c->Hq + h) * c->D;
    int ok = t >= 1 && (c->ring || t <= c->T);
    int64_t n = 0;
    for (int64_t p = 0; ok && p < t; ++p) {
        if (!visible(p, t, c->n_sink, c->window))
            continue;
        if (c->ring) {
            int64_t s = oracle_draft_slot(p, c->n_sink, c->window);
            const uint16_t *base = c->k_src;  /* ring: k_src holds the whole [B,2,Hkv,S,D] */
            keys[n] = base + ((((int64_t)b * 2 + 0) * c->Hkv + g) * S + s) * c->D;
            vals[n] = base + ((((int64_t)b * 2 + 1) * c->Hkv + g) * S + s) * c->D;
        } else {
            keys[n] = c->k_src + (((int64_t)b * c->Hkv + g) * c->T + p) * c->D;
            vals[n] = c->v_src + (((int64_t)b * c->Hkv + g) * c->T + p) * c->D;
        }
        ++n;
    }
    if (!ok || n == 0) {
        c->bad[b] = 1;
        for (int32_t d = 0; d < c->D; ++d)
            o[d] = NAN;
        return;
    }
    attend(c->q + ((int64_t)b * c->Hq + h) * c->D, keys, vals, n, c->D,
           c->scale, scores, o);
}

static int64_t draft_common(draft_ctx *c, const uint8_t *unit_mask,
                            int32_t n_threads, int64_t max_keys)
{
    if (c->B < 0 || c->Hq < 1 || c->Hkv < 1 || c->Hq % c->Hkv != 0 ||
        c->D < 1 || c->n_sink < 0 || c->window < 1)
        return -1;
    if (c->B == 0)
        return 0;
    c->bad = (int32_t *)calloc((size_t)c->B, sizeof(int32_t));
    if (!c->bad)
        return -1;
    int rc = run_pool(draft_unit, c, (int64_t)c->B * c->Hq, max_keys, unit_mask, n_threads);
    int64_t n_bad = 0;
    for (int32_t b = 0; b < c->B; ++b)
        n_bad += c->bad[b];
    free(c->bad);
    return rc ? -1 : n_bad;
}

/*
 * oracle_draft_logical: the definition over a full-length logical memory.
 *   q       bf16 bits [B, Hq, D] (one draft query per sequence)
 *   k_log   bf16 bits [B, Hkv, T, D]: K of memory entries m_0..m_{T-1}
 *   v_log   bf16 bits [B, Hkv, T, D]
 *   ctx_lens int32 [B]: t, the number of memory entries the query may see
 *   out     double [B, Hq, D]
 */
int64_t oracle_draft_logical(const uint16_t *q, const uint16_t *k_log,
                             const uint16_t *v_log, const int32_t *ctx_lens,
                             int32_t B, int32_t Hq, int32_t Hkv, int32_t D,
                             int64_t T, int32_t n_sink, int32_t window,
                             double scale, const uint8_t *unit_mask,
                             double *out, int32_t n_threads)
{
    draft_ctx c = {q, k_log, v_log, 0, ctx_lens, B, Hq, Hkv, D, n_sink, window,
                   T, scale, out, NULL};
    return draft_common(&c, unit_mask, n_threads, T);
}

/*
 * oracle_draft_ring: the same visible set V(t), each entry read from its slot
 * of the bounded cache.
 *   kv   bf16 bits [B, 2, Hkv, n_sink + window, D]  (index 0 = K, 1 = V)
 */
int64_t oracle_draft_ring(const uint16_t *q, const uint16_t *kv,
                          const int32_t *ctx_lens, int32_t B, int32_t Hq,
                          int32_t Hkv, int32_t D, int32_t n_sink,
                          int32_t window, double scale,
                          const uint8_t *unit_mask, double *out,
                          int32_t n_threads)
{
    draft_ctx c = {q, kv, NULL, 1, ctx_lens, B, Hq, Hkv, D, n_sink, window,
                   0, scale, out, NULL};
    return draft_common(&c, unit_mask, n_threads, (int64_t)n_sink + window);
}

/*
 * oracle_ring_pack: write memory entries m_0..m_{t_b - 1} of a logical cache
 * into the bounded cache in order of increasing position, each to its slot
 * (a later entry overwrites an earlier one in the same ring slot).  Slots
 * never written are left untouched.
 */
int64_t oracle_ring_pack(const uint16_t *k_log, const uint16_t *v_log,
                         const int32_t *ctx_lens, int32_t B, int32_t Hkv,
                         int32_t D, int64_t T, int32_t n_sink, int32_t window,
                         uint16_t *kv)
{
    if (B < 0 || Hkv < 1 || D < 1 || n_sink < 0 || window < 1)
        return -1;
    int64_t S = (int64_t)n_sink + window;
    for (int32_t b = 0; b < B; ++b) {
        int64_t t = ctx_lens[b];
        if (t > T)
            return -1;
        for (int32_t g = 0; g < Hkv; ++g)
            for (int64_t p = 0; p < t; ++p) {
                int64_t s = oracle_draft_slot(p, n_sink, window);
                const uint16_t *ks = k_log + (((int64_t)b * Hkv + g) * T + p) * D;
                const uint16_t *vs = v_log + (((int64_t)b * Hkv + g) * T + p) * D;
                memcpy(kv + ((((int64_t)b * 2 + 0) * Hkv + g) * S + s) * D, ks, sizeof(uint16_t) * D);
                memcpy(kv + ((((int64_t)b * 2 + 1) * Hkv + g) * S + s) * D, vs, sizeof(uint16_t) * D);
            }
    }
    return 0;
}

/* ======================================================================== */
/* Feedback-memory append (the draft step's cache update)                    */
/* ======================================================================== */
/*
 * After the draft model has run token t, every draft layer i gets a new
 * memory vector: the softmax(w_i)-weighted average of the token's
 * activations x_t^0 (embedding) .. x_t^{n_layer} (Section 3.3, the per-layer
 * memory equation).  Layer i's attention reads keys and values of these
 * memory vectors, so the vector is projected by the layer's key and value
 * matrices and the result is stored in the bounded cache at the slot of
 * logical position p (Section 3.1: sinks plus a sliding window).
 *
 * Readings (the paper gives no formula beyond the memory equation):
 *   - keys and values are plain linear projections of m, no bias, no norm;
 *   - positional information uses the token's position in the original
 *     text (Section 3.1, footnote).  When rope_theta > 0 keys are rotated
 *     by that position with the half-split rotary form: for d < D/2 the
 *     pair (k[d], k[d + D/2]) is turned by the angle p * rope_theta^(-2d/D);
 *     values are never rotated;
 *   - the stored entry is rounded once, to nearest-even bf16.
 */

/* Round a double to the nearest bf16 (ties to even), returned as bits.
 * bf16 keeps 8 significant bits; the spacing of bf16 values in
 * [2^(e-1), 2^e) is 2^(e-8), and below 2^-126 it is fixed at 2^-133. */
static uint16_t double_to_bf16_bits(double v)
{
    if (isnan(v))
        return 0x7fc0;
    if (v == 0.0)
        return signbit(v) ? 0x8000 : 0x0000;
    int e;
    frexp(v, &e);                        /* |v| in [2^(e-1), 2^e) */
    int q = e - 8;
    if (q < -133)
        q = -133;
    double r = ldexp(nearbyint(ldexp(v, -q)), q);   /* exact scaling, RNE */
    float f = (float)r;                  /* exact: r has <= 8 significant bits */
    if (fabs(r) > 3.3895313892515355e38) /* beyond the largest finite bf16 */
        f = r > 0 ? INFINITY : -INFINITY;
    uint32_t u;
    memcpy(&u, &f, sizeof(u));
    return (uint16_t)(u >> 16);
}

uint16_t oracle_round_bf16(double v)
{
    return double_to_bf16_bits(v);
}

/*
 * oracle_feedback_mix: m[i, b, :] = sum_l exp(w[i, l]) x[l, b, :] /
 *                                   sum_l exp(w[i, l]).
 *   x  bf16 bits [n_act, B, d_model]  (n_act = n_layer + 1, x[0] = embedding)
 *   w  double [n_dl, n_act]
 *   m  double [n_dl, B, d_model]
 * The largest w of each layer is subtracted before exp (the same ratio).
 */
int64_t oracle_feedback_mix(const uint16_t *x, const double *w, int32_t n_act,
                            int32_t n_dl, int32_t B, int32_t d_model, double *m)
{
    if (n_act < 1 || n_dl < 1 || B < 0 || d_model < 1)
        return -1;
    double *a = (double *)malloc(sizeof(double) * (size_t)n_act);
    if (!a)
        return -1;
    for (int32_t i = 0; i < n_dl; ++i) {
        double wmax = w[(int64_t)i * n_act];
        for (int32_t l = 1; l < n_act; ++l)
            if (w[(int64_t)i * n_act + l] > wmax)
                wmax = w[(int64_t)i * n_act + l];
        double z = 0.0;
        for (int32_t l = 0; l < n_act; ++l) {
            a[l] = exp(w[(int64_t)i * n_act + l] - wmax);
            z += a[l];
        }
        for (int32_t b = 0; b < B; ++b)
            for (int32_t c = 0; c < d_model; ++c) {
                double s = 0.0;
                for (int32_t l = 0; l < n_act; ++l)
                    s += a[l] * bf16_to_double(x[((int64_t)l * B + b) * d_model + c]);
                m[((int64_t)i * B + b) * d_model + c] = s / z;
            }
    }
    free(a);
    return 0;
}

/*
 * oracle_feedback_append: the memory vectors of oracle_feedback_mix, then
 * for each draft layer i and sequence b
 *     K[g, d] = sum_c w_kv[i, g*D + d, c]          * m[i, b, c]
 *     V[g, d] = sum_c w_kv[i, Hkv*D + g*D + d, c]  * m[i, b, c]
 * rotated (K only, when rope_theta > 0) by position pos[b], rounded to bf16
 * and written to slot(pos[b]) of layer i's bounded cache.
 *   w_kv  bf16 bits [n_dl, 2*Hkv*D, d_model]
 *   pos   int32 [B]: logical position of the new entry (entries before it)
 *   kv    bf16 bits [n_dl, B, 2, Hkv, n_sink + window, D], updated in place;
 *         every other slot is left untouched
 * Returns the number of sequences with pos < 0 (nothing written for them),
 * or -1 on bad arguments.
 */
int64_t oracle_feedback_append(const uint16_t *x, const double *w,
                               const uint16_t *w_kv, const int32_t *pos,
                               int32_t n_act, int32_t n_dl, int32_t B,
                               int32_t d_model, int32_t Hkv, int32_t D,
                               int32_t n_sink, int32_t window,
                               double rope_theta, uint16_t *kv)
{
    if (n_act < 1 || n_dl < 1 || B < 0 || d_model < 1 || Hkv < 1 || D < 2 ||
        D % 2 != 0 || n_sink < 0 || window < 1 || rope_theta < 0.0)
        return -1;
    if (B == 0)
        return 0;
    int64_t S = (int64_t)n_sink + window;
    int64_t F = 2 * (int64_t)Hkv * D;          /* projected features per layer */
    double *m = (double *)malloc(sizeof(double) * (size_t)n_dl * B * d_model);
    double *y = (double *)malloc(sizeof(double) * (size_t)F);
    if (!m || !y) {
        free(m);
        free(y);
        return -1;
    }
    if (oracle_feedback_mix(x, w, n_act, n_dl, B, d_model, m) != 0) {
        free(m);
        free(y);
        return -1;
    }
    int64_t n_bad = 0;
    for (int32_t b = 0; b < B; ++b) {
        int64_t p = pos[b];
        if (p < 0) {
            ++n_bad;
            continue;
        }
        int64_t dst_slot = oracle_draft_slot(p, n_sink, window);
        for (int32_t i = 0; i < n_dl; ++i) {
            const double *mi = m + ((int64_t)i * B + b) * d_model;
            for (int64_t f = 0; f < F; ++f) {
                const uint16_t *row = w_kv + ((int64_t)i * F + f) * d_model;
                double acc = 0.0;
                for (int32_t c = 0; c < d_model; ++c)
                    acc += bf16_to_double(row[c]) * mi[c];
                y[f] = acc;
            }
            if (rope_theta > 0.0)
                for (int32_t g = 0; g < Hkv; ++g)
                    for (int32_t d = 0; d < D / 2; ++d) {
                        double ang = (double)p * pow(rope_theta, -2.0 * d / D);
                        double cs = cos(ang), sn = sin(ang);
                        double *k = y + (int64_t)g * D;
                        double a0 = k[d], a1 = k[d + D / 2];
                        k[d] = a0 * cs - a1 * sn;
                        k[d + D / 2] = a1 * cs + a0 * sn;
                    }
            for (int32_t kvi = 0; kvi < 2; ++kvi)
                for (int32_t g = 0; g < Hkv; ++g) {
                    uint16_t *dst = kv + (((((int64_t)i * B + b) * 2 + kvi) * Hkv + g) * S + dst_slot) * D;
                    const double *src = y + ((int64_t)kvi * Hkv + g) * D;
                    for (int32_t d = 0; d < D; ++d)
                        dst[d] = double_to_bf16_bits(src[d]);
                }
        }
    }
    free(m);
    free(y);
    return n_bad;
}

/* ======================================================================== */
/* Token verification (modified rejection sampling)                          */
/* ======================================================================== */
/*
 * The target accepts the draft tokens of a round one by one so that every
 * emitted token is a sample of the target's own distribution (Section 1:
 * modified rejection sampling; the token verification algorithm of the
 * paper's experiments, Section 6).  For sequence b with drafts x_1..x_k drawn
 * from the draft distributions q_1..q_k and target distributions p_1..p_{k+1}
 * from the verification pass:
 *   - draft i is accepted with probability min(1, p_i(x_i) / q_i(x_i)): with a
 *     uniform u_i in [0, 1), accepted iff u_i * q_i(x_i) < p_i(x_i);
 *   - at the first rejected i the round emits a token drawn from
 *     norm(max(0, p_i - q_i)) and stops; if all k are accepted it emits a
 *     bonus token drawn from p_{k+1}.
 * Readings: a draw from weights w is the exponential race
 * argmax_v w_v / E_v over w_v > 0 with E_v ~ Exp(1) given as input (ties to
 * the smallest v), which selects v with probability w_v / sum w; every
 * comparison, product, difference and quotient is taken in binary32, as the
 * kernel does, so both sides take the same integer decisions; if the
 * residual has no positive entry the draw uses p_i itself; a draft token
 * outside [0, V) counts as rejected, an E_v that is not > 0 is skipped, and
 * both are reported.
 */
static uint64_t race_key(float w, float e, int32_t v)
{
    /* larger key = better candidate: the score's bits (scores are >= 0, so
     * their bit patterns order like the values), then the smaller index */
    float s = w / e;
    uint32_t sb;
    memcpy(&sb, &s, sizeof(sb));
    return ((uint64_t)sb << 32) | (uint64_t)(~(uint32_t)v);
}

/* argmax_v w_v / e_v over w_v > 0, e_v > 0; returns -1 if no candidate. */
static int32_t race_draw(const float *p, const float *q, int use_residual,
                         const float *e, int32_t V, int32_t *bad_e)
{
    uint64_t best = 0;
    int32_t arg = -1;
    for (int32_t v = 0; v < V; ++v) {
        if (!(e[v] > 0.0f)) {
            *bad_e = 1;
            continue;
        }
        float w = use_residual ? p[v] - q[v] : p[v];
        if (!(w > 0.0f))
            continue;
        uint64_t key = race_key(w, e[v], v);
        if (key > best) {
            best = key;
            arg = v;
        }
    }
    return arg;
}

/*
 * oracle_verify_tokens:
 *   p       float [B, k+1, V]   target distributions p_1..p_{k+1}
 *   q       float [B, k, V]     draft distributions q_1..q_k
 *   x       int32 [B, k]        draft tokens x_1..x_k
 *   u       float [B, k]        acceptance uniforms
 *   e       float [B, V]        Exp(1) variates for the round's one draw
 *   out     int32 [B, k+1]      x_1..x_j, then the drawn token, then -1
 *   n_acc   int32 [B]           j, the number of accepted drafts
 * Returns the number of sequences with an invalid draft token, E value or an
 * empty distribution (their draw may be -1), or -1 on bad arguments.
 */
int64_t oracle_verify_tokens(const float *p, const float *q, const int32_t *x,
                             const float *u, const float *e, int32_t B,
                             int32_t k, int32_t V, int32_t *out,
                             int32_t *n_acc)
{
    if (B < 0 || k < 0 || V < 1)
        return -1;
    int64_t n_bad = 0;
    for (int32_t b = 0; b < B; ++b) {
        int32_t bad = 0;
        int32_t j = 0;
        for (; j < k; ++j) {
            int32_t t = x[(int64_t)b * k + j];
            if (t < 0 || t >= V) {
                bad = 1;
                break;
            }
            float pv = p[((int64_t)b * (k + 1) + j) * V + t];
            float qv = q[((int64_t)b * k + j) * V + t];
            float uq = u[(int64_t)b * k + j] * qv;
            if (!(uq < pv))
                break;
        }
        const float *pj = p + ((int64_t)b * (k + 1) + j) * V;
        const float *qj = j < k ? q + ((int64_t)b * k + j) * V : NULL;
        const float *eb = e + (int64_t)b * V;
        int32_t y = race_draw(pj, qj, j < k, eb, V, &bad);
        if (y < 0 && j < k)
            y = race_draw(pj, qj, 0, eb, V, &bad);
        if (y < 0)
            bad = 1;
        int32_t *o = out + (int64_t)b * (k + 1);
        for (int32_t i = 0; i < j; ++i)
            o[i] = x[(int64_t)b * k + i];
        o[j] = y;
        for (int32_t i = j + 1; i <= k; ++i)
            o[i] = -1;
        n_acc[b] = j;
        n_bad += bad;
    }
    return n_bad;
}

/* ======================================================================== */
/* MagicDec draft attention: StreamingLLM over the target's own paged cache  */
/* ======================================================================== */
/*
 * MagicDec drafts with the target model itself, attending to a sink +
 * sliding-window subset of the target's KV cache, and (as in StreamingLLM)
 * gives tokens their positions inside that reduced cache, not in the text
 * (Section 3.1 footnote; Section 4: sink 1, window 64).
 *
 * Readings: the target cache holds keys already turned by their original
 * position p (rotary, half-split pairs (d, d + D/2), angle p * theta^(-2d/D));
 * t = ctx_lens[b] entries are visible to the current token, its own included;
 * the visible positions are [0, s) and [w0, t) with s = min(n_sink, t) and
 * w0 = max(s, t - window); their cache indices are c = p for p < s and
 * c = s + (p - w0) otherwise, and the query's index is c_q = (number of
 * visible entries) - 1.  Each key is turned by (c - p) to sit at its cache
 * index and the (unrotated) query by c_q; both are rounded to bf16, as the
 * model's operands are; values are not rotated.  theta = 0: no rotation.
 * A length t < 1 or beyond the block table, or a page id outside the cache
 * among the visible entries, gives NaN rows and is counted.
 */
static void rotate_pairs(const uint16_t *src, double delta, int32_t D,
                         double theta, uint16_t *dst)
{
    for (int32_t d = 0; d < D / 2; ++d) {
        double a0 = bf16_to_double(src[d]), a1 = bf16_to_double(src[d + D / 2]);
        double r0 = a0, r1 = a1;
        if (theta > 0.0 && delta != 0.0) {
            double ang = delta * pow(theta, -2.0 * d / D);
            double cs = cos(ang), sn = sin(ang);
            r0 = a0 * cs - a1 * sn;
            r1 = a1 * cs + a0 * sn;
        }
        dst[d] = double_to_bf16_bits(r0);
        dst[d + D / 2] = double_to_bf16_bits(r1);
    }
}

int64_t oracle_magicdec(const uint16_t *q, const uint16_t *k_cache,
                        const uint16_t *v_cache, const int32_t *block_table,
                        const int32_t *ctx_lens, int32_t B, int32_t Hq,
                        int32_t Hkv, int32_t D, int32_t page_size,
                        int32_t max_pages, int32_t num_pages, int32_t n_sink,
                        int32_t window, double theta, double scale, double *out)
{
    if (B < 0 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || D < 2 || D % 2 != 0 ||
        page_size < 1 || n_sink < 0 || window < 1 || theta < 0.0)
        return -1;
    int64_t S = (int64_t)n_sink + window;
    uint16_t *kc = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)(S * D));
    uint16_t *qe = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)D);
    const uint16_t **keys = (const uint16_t **)malloc(sizeof(*keys) * (size_t)S);
    const uint16_t **vals = (const uint16_t **)malloc(sizeof(*vals) * (size_t)S);
    double *scores = (double *)malloc(sizeof(double) * (size_t)S);
    if (!kc || !qe || !keys || !vals || !scores) {
        free(kc); free(qe); free(keys); free(vals); free(scores);
        return -1;
    }
    int64_t n_bad = 0;
    for (int32_t b = 0; b < B; ++b) {
        int64_t t = ctx_lens[b];
        int ok = t >= 1 && t <= (int64_t)max_pages * page_size;
        int64_t s = ok ? (t < n_sink ? t : n_sink) : 0;
        int64_t w0 = ok ? (t - window > s ? t - window : s) : 0;
        int64_t n = s + (ok ? t - w0 : 0);
        for (int64_t c = 0; ok && c < n; ++c) {
            int64_t p = c < s ? c : w0 + (c - s);
            int64_t page = block_table[(int64_t)b * max_pages + p / page_size];
            if (page < 0 || page >= num_pages)
                ok = 0;
        }
        for (int32_t h = 0; h < Hq; ++h) {
            int32_t g = h / (Hq / Hkv);
            double *o = out + ((int64_t)b * Hq + h) * D;
            if (!ok) {
                for (int32_t d = 0; d < D; ++d)
                    o[d] = NAN;
                continue;
            }
            for (int64_t c = 0; c < n; ++c) {
                int64_t p = c < s ? c : w0 + (c - s);
                int64_t page = block_table[(int64_t)b * max_pages + p / page_size];
                int64_t row = ((page * Hkv + g) * page_size + p % page_size) * D;
                rotate_pairs(k_cache + row, (double)(c - p), D, theta, kc + c * D);
                keys[c] = kc + c * D;
                vals[c] = v_cache + row;
            }
            rotate_pairs(q + ((int64_t)b * Hq + h) * D, (double)(n - 1), D, theta, qe);
            attend(qe, keys, vals, n, D, scale, scores, o);
        }
        n_bad += !ok;
    }
    free(kc); free(qe); free(keys); free(vals); free(scores);
    return n_bad;
}
