/*
 * f2gen.c -- seeded synthetic workloads for the GF(2) encoder-learning path.
 *
 * This file only SYNTHESISES inputs.  It draws planted affine maps
 * y = A x XOR b over GF(2) (the model of Sec. 2.1, "encoding equation"),
 * field-structured feature bits, duplicate observations, injected
 * contradictions and span-structured queries.  It performs no Gaussian
 * elimination, no affine solve and no reduction of a query against a learned
 * basis: both the CPU oracle and the CUDA path consume what it writes.
 *
 * Bit conventions shared by every consumer:
 *   - a context's feature vector x has n bits, packed little-endian into
 *     W = ceil(n/32) uint32 words (bit j of x = bit j%32 of word j/32);
 *     bits at positions >= n are zero;
 *   - a 128-bit word y is four uint32 words, bit i of y = bit i%32 of word
 *     i/32 (the little-endian numbering of Appendix C);
 *   - column j of A is stored as one 128-bit word, so y = b XOR (XOR of the
 *     columns j with x_j = 1).
 *
 * Randomness: splitmix64 streams keyed by (seed, purpose, index), so every
 * context and every query has its own stream and the output does not depend
 * on the thread count.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------ RNG */

typedef struct {
    uint64_t s;
} rng_t;

static inline uint64_t mix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

static inline uint64_t rng_next(rng_t* r)
{
    r->s += 0x9E3779B97F4A7C15ULL;
    return mix64(r->s);
}

static inline uint64_t rng_below(rng_t* r, uint64_t m)
{
    return (uint64_t)(((unsigned __int128)rng_next(r) * m) >> 64);
}

static inline double rng_unit(rng_t* r)
{
    return (double)(rng_next(r) >> 11) * (1.0 / 9007199254740992.0);
}

static double rng_normal(rng_t* r)
{
    double u1 = 1.0 - rng_unit(r); /* (0, 1] */
    double u2 = rng_unit(r);
    return sqrt(-2.0 * log(u1)) * cos(6.283185307179586 * u2);
}

static rng_t rng_stream(uint64_t seed, uint64_t purpose, uint64_t index)
{
    rng_t r;
    r.s = mix64(seed ^ mix64(purpose * 0xD1B54A32D192ED03ULL + mix64(index + 0x632BE59BD9B4E019ULL)));
    return r;
}

/* --------------------------------------------------------------- params */

enum { LAYOUT_REGS_IMM16_ONEHOT = 0, LAYOUT_CYCLIC_FIELDS = 1, LAYOUT_UNIFORM_BITS = 2 };

typedef struct {
    int32_t num_ctx;
    int32_t layout;      /* LAYOUT_* */
    int32_t n_fixed;     /* > 0: every context has n = n_fixed feature bits */
    int32_t n_min;       /* otherwise n in [n_min, n_max] ... */
    int32_t n_max;
    int32_t pad0;
    double n_median;     /* ... lognormal(ln n_median, n_sigma) if n_sigma > 0, else uniform */
    double n_sigma;
    int64_t rows_fixed;  /* > 0: fresh rows = rows_fixed, duplicates = round(rows_fixed * dup_frac) */
    double rows_median;  /* otherwise total rows ~ lognormal(ln rows_median, rows_sigma) in [1, rows_max] */
    double rows_sigma;
    int64_t rows_max;
    double dup_frac;     /* share of duplicate observations */
    double density;      /* Bernoulli density of the planted A */
    int32_t n_contra;    /* contexts that receive one contradicting observation */
    int32_t n_two_stream;/* contexts whose fresh rows come from two variant streams */
    int64_t batch_rows;  /* > 0: batch-major row layout, batches of batch_rows rows per context */
} f2gen_params;

static int64_t round_pos(double v)
{
    return (int64_t)floor(v + 0.5);
}

/* Choose k distinct members of idx[0..m) uniformly (partial Fisher-Yates). */
static void choose_subset(rng_t* r, int32_t* idx, int64_t m, int64_t k)
{
    for (int64_t i = 0; i < k && i < m; ++i) {
        int64_t j = i + (int64_t)rng_below(r, (uint64_t)(m - i));
        int32_t t = idx[i];
        idx[i] = idx[j];
        idx[j] = t;
    }
}

/*
 * Per-context sizes.  Writes n_bits[c], fresh[c], dups[c], contra[c] (0/1)
 * and two_stream[c] (0/1).  Returns 0, or -1 on invalid parameters.
 */
int f2gen_plan(const f2gen_params* p, uint64_t seed, int32_t* n_bits, int64_t* fresh, int64_t* dups,
               uint8_t* contra, uint8_t* two_stream)
{
    const int32_t C = p->num_ctx;
    if (C <= 0) return -1;
    rng_t r = rng_stream(seed, 0, 0);
    for (int32_t c = 0; c < C; ++c) {
        int32_t n;
        if (p->n_fixed > 0) {
            n = p->n_fixed;
        } else if (p->n_sigma > 0) {
            n = (int32_t)round_pos(exp(log(p->n_median) + p->n_sigma * rng_normal(&r)));
            if (n < p->n_min) n = p->n_min;
            if (n > p->n_max) n = p->n_max;
        } else {
            n = p->n_min + (int32_t)rng_below(&r, (uint64_t)(p->n_max - p->n_min + 1));
        }
        n_bits[c] = n;
        int64_t u, d;
        if (p->rows_fixed > 0) {
            u = p->rows_fixed;
            d = round_pos((double)p->rows_fixed * p->dup_frac);
        } else {
            int64_t t = round_pos(exp(log(p->rows_median) + p->rows_sigma * rng_normal(&r)));
            if (t < 1) t = 1;
            if (t > p->rows_max) t = p->rows_max;
            u = round_pos((double)t * (1.0 - p->dup_frac));
            if (u < 1) u = 1;
            if (u > t) u = t;
            d = t - u;
        }
        fresh[c] = u;
        dups[c] = d;
        contra[c] = 0;
        two_stream[c] = 0;
    }
    int32_t* idx = (int32_t*)malloc(sizeof(int32_t) * (size_t)C);
    if (!idx) return -1;
    /* contradiction contexts: among contexts with a duplicate slot (or, without
       duplicates, at least two rows so that a row can copy an earlier one) */
    int64_t m = 0;
    for (int32_t c = 0; c < C; ++c)
        if (dups[c] > 0 || (p->dup_frac == 0.0 && fresh[c] >= 2)) idx[m++] = c;
    if (p->n_contra > m) {
        free(idx);
        return -1;
    }
    rng_t rc = rng_stream(seed, 0, 1);
    choose_subset(&rc, idx, m, p->n_contra);
    for (int32_t i = 0; i < p->n_contra; ++i) contra[idx[i]] = 1;
    for (int32_t c = 0; c < C; ++c) idx[c] = c;
    if (p->n_two_stream > C) {
        free(idx);
        return -1;
    }
    rng_t rt = rng_stream(seed, 0, 2);
    choose_subset(&rt, idx, C, p->n_two_stream);
    for (int32_t i = 0; i < p->n_two_stream; ++i) two_stream[idx[i]] = 1;
    free(idx);
    return 0;
}

/* ------------------------------------------------------- feature fields */

static inline void put_bits(uint32_t* xw, int n, int pos, int width, uint64_t v)
{
    for (int i = 0; i < width; ++i) {
        int b = pos + i;
        if (b >= n) return;
        if ((v >> i) & 1u) xw[b >> 5] |= 1u << (b & 31);
    }
}

/* Small-magnitude-heavy 32-bit immediate: bit length uniform in [1, 32],
   lower bits uniform (a log-uniform magnitude). */
static inline uint64_t draw_imm32(rng_t* r)
{
    int len = 1 + (int)rng_below(r, 32);
    uint64_t v = 1ull << (len - 1);
    if (len > 1) v |= rng_next(r) & ((1ull << (len - 1)) - 1);
    return v;
}

static void draw_x(rng_t* r, int layout, int n, uint32_t* xw, int W)
{
    memset(xw, 0, sizeof(uint32_t) * (size_t)W);
    if (layout == LAYOUT_UNIFORM_BITS) {
        for (int w = 0; w < W; ++w) xw[w] = (uint32_t)rng_next(r);
        if (n & 31) xw[W - 1] &= (1u << (n & 31)) - 1u;
        return;
    }
    int pos = 0, f = 0;
    while (pos < n) {
        int width;
        uint64_t v;
        if (layout == LAYOUT_REGS_IMM16_ONEHOT) {
            /* reg8, reg8, reg8, imm16, onehot8 (uniform values) */
            switch (f % 5) {
            case 0: case 1: case 2: width = 8; v = rng_below(r, 256); break;
            case 3: width = 16; v = rng_below(r, 65536); break;
            default: width = 8; v = 1ull << rng_below(r, 8); break;
            }
        } else {
            /* onehot8, reg8, pred4, imm32 (small-magnitude heavy) */
            switch (f % 4) {
            case 0: width = 8; v = 1ull << rng_below(r, 8); break;
            case 1: width = 8; v = rng_below(r, 256); break;
            case 2: width = 4; v = rng_below(r, 16); break;
            default: width = 32; v = draw_imm32(r); break;
            }
        }
        put_bits(xw, n, pos, width, v);
        pos += width;
        ++f;
    }
}

/* Bit offset of the first complete one-hot modifier group; -1 if none. */
int f2gen_onehot_offset(int32_t layout)
{
    if (layout == LAYOUT_REGS_IMM16_ONEHOT) return 40;
    if (layout == LAYOUT_CYCLIC_FIELDS) return 0;
    return -1;
}

/* ------------------------------------------------------------ fill pass */

typedef struct {
    const f2gen_params* p;
    uint64_t seed;
    const int32_t* n_bits;
    const int64_t* fresh;
    const int64_t* dups;
    const uint8_t* contra;
    const uint8_t* two_stream;
    const int64_t* row_off;
    const int64_t* x_off;
    uint32_t* x;
    uint32_t* y;
    uint32_t* A;
    const int64_t* a_off;
    uint32_t* b;
    int64_t* contra_pos;
    int32_t* contra_bit;
    int64_t next;
    pthread_mutex_t mu;
    int status;
} fill_job;

static inline int64_t dest_row(const fill_job* j, int32_t c, int64_t i)
{
    const int64_t br = j->p->batch_rows;
    if (br > 0) return (i / br) * ((int64_t)j->p->num_ctx * br) + (int64_t)c * br + (i % br);
    return j->row_off[c] + i;
}

static inline uint32_t* dest_x(const fill_job* j, int32_t c, int64_t i, int W)
{
    if (j->p->batch_rows > 0) return j->x + dest_row(j, c, i) * W;
    return j->x + j->x_off[c] + i * W;
}

static int fill_context(fill_job* j, int32_t c, uint8_t** kind_buf, int64_t* kind_cap,
                        int64_t** fresh_pos, int64_t* fresh_cap)
{
    const f2gen_params* p = j->p;
    const int n = j->n_bits[c];
    const int W = (n + 31) / 32;
    const int64_t U = j->fresh[c], D = j->dups[c], T = U + D;
    rng_t r = rng_stream(j->seed, 1, (uint64_t)c);
    rng_t rv[2] = {rng_stream(j->seed, 2, (uint64_t)c), rng_stream(j->seed, 3, (uint64_t)c)};

    /* planted map: columns of A, then b */
    uint32_t* Ac = j->A + j->a_off[c] * 4;
    const uint32_t thr = (uint32_t)fmin(4294967295.0, p->density * 4294967296.0);
    for (int col = 0; col < n; ++col) {
        for (int w = 0; w < 4; ++w) {
            uint32_t word = 0;
            if (p->density == 0.5) {
                word = (uint32_t)rng_next(&r);
            } else {
                for (int bit = 0; bit < 32; ++bit)
                    if ((uint32_t)rng_next(&r) < thr) word |= 1u << bit;
            }
            Ac[col * 4 + w] = word;
        }
    }
    uint32_t* bc = j->b + (int64_t)c * 4;
    for (int w = 0; w < 4; ++w) bc[w] = (uint32_t)rng_next(&r);

    /* slot kinds: 0 fresh, 1 duplicate; slot 0 is always fresh */
    if (T > *kind_cap) {
        free(*kind_buf);
        *kind_buf = (uint8_t*)malloc((size_t)T);
        if (!*kind_buf) return -1;
        *kind_cap = T;
    }
    if (U > *fresh_cap) {
        free(*fresh_pos);
        *fresh_pos = (int64_t*)malloc(sizeof(int64_t) * (size_t)U);
        if (!*fresh_pos) return -1;
        *fresh_cap = U;
    }
    uint8_t* kind = *kind_buf;
    int64_t* fpos = *fresh_pos;
    kind[0] = 0;
    for (int64_t i = 1; i < T; ++i) kind[i] = (i < U) ? 0 : 1;
    for (int64_t i = T - 1; i > 1; --i) { /* shuffle slots 1..T-1 */
        int64_t k = 1 + (int64_t)rng_below(&r, (uint64_t)i);
        uint8_t t = kind[i];
        kind[i] = kind[k];
        kind[k] = t;
    }

    /* contradiction position */
    int64_t cpos = -1;
    int cbit = -1;
    if (j->contra[c]) {
        if (D > 0) {
            int64_t m = (int64_t)rng_below(&r, (uint64_t)D);
            for (int64_t i = 0; i < T; ++i)
                if (kind[i] == 1 && m-- == 0) {
                    cpos = i;
                    break;
                }
        } else {
            int64_t br = p->batch_rows > 0 ? p->batch_rows : T;
            int64_t nb = T / br;
            int64_t bsel = nb > 0 ? (int64_t)rng_below(&r, (uint64_t)nb) : 0;
            cpos = bsel * br + (int64_t)rng_below(&r, (uint64_t)br);
            if (cpos <= 0) cpos = 1;
            if (cpos >= T) cpos = T - 1;
        }
        cbit = (int)rng_below(&r, 128);
    }
    j->contra_pos[c] = cpos;
    j->contra_bit[c] = cbit;

    int64_t nf = 0;
    for (int64_t i = 0; i < T; ++i) {
        uint32_t* xd = dest_x(j, c, i, W);
        uint32_t* yd = j->y + dest_row(j, c, i) * 4;
        if (kind[i] == 0 && i != cpos) {
            int v = j->two_stream[c] ? (int)rng_below(&r, 2) : 0;
            draw_x(&rv[v], p->layout, n, xd, W);
            uint32_t acc[4] = {bc[0], bc[1], bc[2], bc[3]};
            for (int col = 0; col < n; ++col)
                if ((xd[col >> 5] >> (col & 31)) & 1u)
                    for (int w = 0; w < 4; ++w) acc[w] ^= Ac[col * 4 + w];
            memcpy(yd, acc, sizeof acc);
            fpos[nf++] = i;
        } else {
            /* duplicate of a fresh row seen earlier (or, for an injected
               contradiction without duplicate slots, of any earlier row) */
            int64_t src;
            if (kind[i] == 1) {
                src = fpos[rng_below(&r, (uint64_t)nf)];
            } else {
                src = (int64_t)rng_below(&r, (uint64_t)i);
            }
            memcpy(xd, dest_x(j, c, src, W), sizeof(uint32_t) * (size_t)W);
            memcpy(yd, j->y + dest_row(j, c, src) * 4, sizeof(uint32_t) * 4);
            if (i == cpos) yd[cbit >> 5] ^= 1u << (cbit & 31);
        }
    }
    return 0;
}

static void* fill_worker(void* arg)
{
    fill_job* j = (fill_job*)arg;
    uint8_t* kind = NULL;
    int64_t kind_cap = 0;
    int64_t* fpos = NULL;
    int64_t fcap = 0;
    for (;;) {
        pthread_mutex_lock(&j->mu);
        int64_t c = j->next++;
        pthread_mutex_unlock(&j->mu);
        if (c >= j->p->num_ctx) break;
        if (fill_context(j, (int32_t)c, &kind, &kind_cap, &fpos, &fcap) != 0) {
            pthread_mutex_lock(&j->mu);
            j->status = -1;
            pthread_mutex_unlock(&j->mu);
            break;
        }
    }
    free(kind);
    free(fpos);
    return NULL;
}

/*
 * Fill rows.  CSR layout (batch_rows == 0): row i of context c goes to
 * y[row_off[c] + i] and x[x_off[c] + i*W_c].  Batch-major layout
 * (batch_rows > 0, all contexts with equal n and rows): row i of context c
 * goes to global row (i / B) * C * B + c * B + i % B, x at that row times W.
 * A gets column j of context c at 128-bit slot a_off[c] + j; b gets 128 bits
 * per context.  contra_pos[c] is the stream index of the injected
 * contradiction within context c (-1 if none), contra_bit[c] its flipped bit.
 */
int f2gen_fill(const f2gen_params* p, uint64_t seed, const int32_t* n_bits, const int64_t* fresh,
               const int64_t* dups, const uint8_t* contra, const uint8_t* two_stream,
               const int64_t* row_off, const int64_t* x_off, uint32_t* x, uint32_t* y, uint32_t* A,
               const int64_t* a_off, uint32_t* b, int64_t* contra_pos, int32_t* contra_bit,
               int32_t nthreads)
{
    fill_job j;
    memset(&j, 0, sizeof j);
    j.p = p;
    j.seed = seed;
    j.n_bits = n_bits;
    j.fresh = fresh;
    j.dups = dups;
    j.contra = contra;
    j.two_stream = two_stream;
    j.row_off = row_off;
    j.x_off = x_off;
    j.x = x;
    j.y = y;
    j.A = A;
    j.a_off = a_off;
    j.b = b;
    j.contra_pos = contra_pos;
    j.contra_bit = contra_bit;
    pthread_mutex_init(&j.mu, NULL);
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    pthread_t th[256];
    for (int t = 0; t < nthreads; ++t) pthread_create(&th[t], NULL, fill_worker, &j);
    for (int t = 0; t < nthreads; ++t) pthread_join(th[t], NULL);
    pthread_mutex_destroy(&j.mu);
    return j.status;
}

/* -------------------------------------------------------------- queries */

typedef struct {
    uint64_t seed;
    int32_t layout;
    int64_t Q;
    int32_t num_ctx;
    const int32_t* n_bits;
    const int64_t* rows;
    const int64_t* row_off;
    const int64_t* x_off;
    const uint32_t* x;
    const int64_t* contra_pos;
    int32_t ctx_mode;
    const double* zipf_cdf;
    const int32_t* rank_to_ctx;
    int64_t per_ctx;
    double out_frac;
    int32_t x_stride;
    int32_t* ctx_id;
    uint32_t* qx;
    uint8_t* expect_in;
    int64_t next;
    pthread_mutex_t mu;
} query_job;

#define QUERY_BLOCK 4096

static void make_query(query_job* j, int64_t q)
{
    rng_t r = rng_stream(j->seed, 7, (uint64_t)q);
    int32_t c;
    if (j->ctx_mode == 0) {
        c = (int32_t)(q / j->per_ctx);
    } else {
        double u = rng_unit(&r);
        int64_t lo = 0, hi = j->num_ctx - 1;
        while (lo < hi) {
            int64_t mid = (lo + hi) / 2;
            if (j->zipf_cdf[mid] > u) hi = mid;
            else lo = mid + 1;
        }
        c = j->rank_to_ctx[lo];
    }
    const int n = j->n_bits[c];
    const int W = (n + 31) / 32;
    uint32_t* out = j->qx + q * j->x_stride;
    memset(out, 0, sizeof(uint32_t) * (size_t)j->x_stride);
    const int k = 1 + 2 * (int)rng_below(&r, 3); /* 1, 3 or 5 training rows */
    const int64_t T = j->rows[c];
    for (int t = 0; t < k; ++t) {
        int64_t i;
        do {
            i = (int64_t)rng_below(&r, (uint64_t)T);
        } while (i == j->contra_pos[c] && T > 1);
        const uint32_t* src = j->x + j->x_off[c] + i * W;
        for (int w = 0; w < W; ++w) out[w] ^= src[w];
    }
    uint8_t in = 1;
    if (j->out_frac > 0 && rng_unit(&r) < j->out_frac) {
        int go = f2gen_onehot_offset(j->layout);
        int bit = go + (int)rng_below(&r, 8);
        out[bit >> 5] ^= 1u << (bit & 31);
        in = 0;
    }
    j->ctx_id[q] = c;
    j->expect_in[q] = in;
}

static void* query_worker(void* arg)
{
    query_job* j = (query_job*)arg;
    for (;;) {
        pthread_mutex_lock(&j->mu);
        int64_t blk = j->next++;
        pthread_mutex_unlock(&j->mu);
        int64_t q0 = blk * QUERY_BLOCK;
        if (q0 >= j->Q) break;
        int64_t q1 = q0 + QUERY_BLOCK < j->Q ? q0 + QUERY_BLOCK : j->Q;
        for (int64_t q = q0; q < q1; ++q) make_query(j, q);
    }
    return NULL;
}

/*
 * Queries over a generated training set (CSR layout).  ctx_mode 0: query q
 * belongs to context q / per_ctx; ctx_mode 1: context drawn Zipf(zipf_s) over
 * ranks, ranks mapped to contexts by a seeded permutation.  An in-span query
 * XORs the features of 1, 3 or 5 clean training rows (an odd count keeps the
 * affine constant).  With probability out_frac one bit of the first complete
 * one-hot modifier group is flipped: every training row has exactly one bit
 * set there, so any vector of the row span with constant 1 has odd parity on
 * that group and the flipped query lies outside the span.  expect_in[q] is 1
 * for the in-span construction, 0 for the flipped one.
 */
int f2gen_queries(uint64_t seed, int32_t layout, int64_t Q, int32_t num_ctx, const int32_t* n_bits,
                  const int64_t* rows, const int64_t* row_off, const int64_t* x_off, const uint32_t* x,
                  const int64_t* contra_pos, int32_t ctx_mode, double zipf_s, int64_t per_ctx,
                  double out_frac, int32_t x_stride, int32_t* ctx_id, uint32_t* qx, uint8_t* expect_in,
                  int32_t nthreads)
{
    if (out_frac > 0 && f2gen_onehot_offset(layout) < 0) return -1;
    if (ctx_mode == 0 && (per_ctx <= 0 || Q > per_ctx * (int64_t)num_ctx)) return -1;
    for (int32_t c = 0; c < num_ctx; ++c)
        if ((n_bits[c] + 31) / 32 > x_stride || rows[c] < 1) return -1;
    query_job j;
    memset(&j, 0, sizeof j);
    j.seed = seed;
    j.layout = layout;
    j.Q = Q;
    j.num_ctx = num_ctx;
    j.n_bits = n_bits;
    j.rows = rows;
    j.row_off = row_off;
    j.x_off = x_off;
    j.x = x;
    j.contra_pos = contra_pos;
    j.ctx_mode = ctx_mode;
    j.per_ctx = per_ctx;
    j.out_frac = out_frac;
    j.x_stride = x_stride;
    j.ctx_id = ctx_id;
    j.qx = qx;
    j.expect_in = expect_in;
    double* cdf = NULL;
    int32_t* perm = NULL;
    if (ctx_mode == 1) {
        cdf = (double*)malloc(sizeof(double) * (size_t)num_ctx);
        perm = (int32_t*)malloc(sizeof(int32_t) * (size_t)num_ctx);
        if (!cdf || !perm) {
            free(cdf);
            free(perm);
            return -1;
        }
        double s = 0;
        for (int32_t i = 0; i < num_ctx; ++i) {
            s += pow((double)(i + 1), -zipf_s);
            cdf[i] = s;
        }
        for (int32_t i = 0; i < num_ctx; ++i) cdf[i] /= s;
        cdf[num_ctx - 1] = 2.0;
        for (int32_t i = 0; i < num_ctx; ++i) perm[i] = i;
        rng_t rp = rng_stream(seed, 6, 0);
        for (int32_t i = num_ctx - 1; i > 0; --i) {
            int32_t k = (int32_t)rng_below(&rp, (uint64_t)i + 1);
            int32_t t = perm[i];
            perm[i] = perm[k];
            perm[k] = t;
        }
    }
    j.zipf_cdf = cdf;
    j.rank_to_ctx = perm;
    pthread_mutex_init(&j.mu, NULL);
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    pthread_t th[256];
    for (int t = 0; t < nthreads; ++t) pthread_create(&th[t], NULL, query_worker, &j);
    for (int t = 0; t < nthreads; ++t) pthread_join(th[t], NULL);
    pthread_mutex_destroy(&j.mu);
    free(cdf);
    free(perm);
    return 0;
}
