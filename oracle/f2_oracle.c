/*
 * f2_oracle.c -- plain CPU oracle for the GF(2) encoder-learning path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg load this file's library; the product path
 * never calls it.  It shares no code with the CUDA library.
 *
 * It restates the method of "Learning Exact NVIDIA SASS Encoders with F2
 * Linear Algebra" as literally as possible, one observation at a time:
 *
 *   - feature vector phi(x) = [1 || x], index 0 = affine constant, index 1+j =
 *     feature bit j (Sec. 2.1, parsed-value feature map; Table 6 indices);
 *   - augmented row [r | z] = [phi(x) | y] (Sec. 2.2, augmented row);
 *   - training, per row (Sec. 2.2 steps (1)-(5), Appendix B): (1) XOR-reduce
 *     against every stored pivot row, highest pivot first; (2) zero feature
 *     and zero output residual: redundant, discard; (3) zero feature but
 *     nonzero output residual: contradiction (reported, not inserted,
 *     learning continues); (4) otherwise the pivot is the highest set feature
 *     bit; (5) clear that pivot bit from every stored row, then store the row
 *     in pivot slot k.  The stored basis is therefore reduced (RREF);
 *   - affine solve: the map T(r_k) = z_k (Sec. 2.3, evidence map) extended
 *     by zero on non-pivot coordinates: W[k] = z_k for a pivot k, W[j] = 0
 *     otherwise; b = W[0] and column j of A is W[1+j];
 *   - encode (Sec. 2.3, Appendix B): reduce q = phi(x) with the stored rows,
 *     XOR z_k into a zero accumulator for every row used; a zero residual
 *     means q is in the span and the accumulator is the word; otherwise the
 *     query is rejected and the word is zero.
 *
 * Words: feature rows are uint64 arrays (bit k = bit k%64 of word k/64);
 * 128-bit outputs are two uint64.  Inputs and outputs use the library's
 * exchange format: uint32 words, 128-bit values as four uint32 (bit i = bit
 * i%32 of word i/32).  Feature bits at positions >= n are ignored.
 *
 * Nothing here is blocked, vectorised or reordered: each row is handled by a
 * full scan over the pivot slots.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define F2O_MAX_D 1025
#define F2O_MAX_NW ((F2O_MAX_D + 63) / 64)

typedef struct {
    int32_t n;           /* feature bits as supplied */
    int32_t d;           /* row width: n + 1 with the implicit constant, n in raw mode */
    int32_t nw;          /* uint64 words per feature row */
    int32_t rank;
    uint8_t contra;
    int64_t first_contra;
    uint64_t n_contra;
    int64_t rows_seen;
    uint8_t* occupied;   /* [d] */
    uint64_t* r;         /* [d][nw] */
    uint64_t* z;         /* [d][2] */
} f2o_ctx;

typedef struct {
    int32_t num_ctx;
    int32_t raw;         /* 1: rows are complete feature vectors, no constant added */
    f2o_ctx* ctx;
} f2o_state;

static inline int get_bit(const uint64_t* v, int k)
{
    return (int)((v[k >> 6] >> (k & 63)) & 1u);
}

static inline void set_bit(uint64_t* v, int k)
{
    v[k >> 6] |= 1ull << (k & 63);
}

static inline int is_zero(const uint64_t* v, int nw)
{
    for (int w = 0; w < nw; ++w)
        if (v[w]) return 0;
    return 1;
}

static inline int highest_bit(const uint64_t* v, int nw)
{
    for (int w = nw - 1; w >= 0; --w)
        if (v[w])
            for (int b = 63; b >= 0; --b)
                if ((v[w] >> b) & 1u) return w * 64 + b;
    return -1;
}

/* Returns NULL on invalid sizes (n outside [1, 1024] or d > 1025). */
f2o_state* f2o_create(int32_t num_ctx, const int32_t* n_bits, int32_t raw)
{
    if (num_ctx < 0) return NULL;
    f2o_state* s = (f2o_state*)calloc(1, sizeof(f2o_state));
    if (!s) return NULL;
    s->num_ctx = num_ctx;
    s->raw = raw ? 1 : 0;
    s->ctx = (f2o_ctx*)calloc((size_t)(num_ctx > 0 ? num_ctx : 1), sizeof(f2o_ctx));
    if (!s->ctx) {
        free(s);
        return NULL;
    }
    for (int32_t c = 0; c < num_ctx; ++c) {
        f2o_ctx* t = &s->ctx[c];
        t->n = n_bits[c];
        t->d = s->raw ? t->n : t->n + 1;
        if (t->n < 1 || t->n > 1024 || t->d > F2O_MAX_D) {
            for (int32_t k = 0; k < c; ++k) {
                free(s->ctx[k].occupied);
                free(s->ctx[k].r);
                free(s->ctx[k].z);
            }
            free(s->ctx);
            free(s);
            return NULL;
        }
        t->nw = (t->d + 63) / 64;
        t->first_contra = -1;
        t->occupied = (uint8_t*)calloc((size_t)t->d, 1);
        t->r = (uint64_t*)calloc((size_t)t->d * (size_t)t->nw, sizeof(uint64_t));
        t->z = (uint64_t*)calloc((size_t)t->d * 2, sizeof(uint64_t));
    }
    return s;
}

void f2o_destroy(f2o_state* s)
{
    if (!s) return;
    for (int32_t c = 0; c < s->num_ctx; ++c) {
        free(s->ctx[c].occupied);
        free(s->ctx[c].r);
        free(s->ctx[c].z);
    }
    free(s->ctx);
    free(s);
}

/* phi(x) = [1 || x] (or x itself in raw mode) as a feature row. */
static void form_row(const f2o_state* s, const f2o_ctx* t, const uint32_t* xw, uint64_t* q)
{
    memset(q, 0, sizeof(uint64_t) * (size_t)t->nw);
    const int shift = s->raw ? 0 : 1;
    if (!s->raw) set_bit(q, 0);
    for (int j = 0; j < t->n; ++j)
        if ((xw[j >> 5] >> (j & 31)) & 1u) set_bit(q, j + shift);
}

static void load_word128(const uint32_t* yw, uint64_t* z)
{
    z[0] = (uint64_t)yw[0] | ((uint64_t)yw[1] << 32);
    z[1] = (uint64_t)yw[2] | ((uint64_t)yw[3] << 32);
}

static void learn_row(const f2o_state* s, f2o_ctx* t, const uint32_t* xw, const uint32_t* yw)
{
    uint64_t q[F2O_MAX_NW];
    uint64_t z[2];
    form_row(s, t, xw, q);
    load_word128(yw, z);
    const int64_t idx = t->rows_seen++;

    /* (1) reduce against the stored pivots, highest first */
    for (int k = t->d - 1; k >= 0; --k) {
        if (t->occupied[k] && get_bit(q, k)) {
            const uint64_t* rk = t->r + (size_t)k * t->nw;
            for (int w = 0; w < t->nw; ++w) q[w] ^= rk[w];
            z[0] ^= t->z[2 * k];
            z[1] ^= t->z[2 * k + 1];
        }
    }
    if (is_zero(q, t->nw)) {
        if (z[0] == 0 && z[1] == 0) return; /* (2) redundant */
        /* (3) contradiction: same features, different encoding */
        t->contra = 1;
        if (t->first_contra < 0) t->first_contra = idx;
        t->n_contra++;
        return;
    }
    /* (4) pivot = highest set feature bit */
    const int k = highest_bit(q, t->nw);
    /* (5) clear the pivot bit from every stored row, then insert */
    for (int j = 0; j < t->d; ++j) {
        if (!t->occupied[j]) continue;
        uint64_t* rj = t->r + (size_t)j * t->nw;
        if (get_bit(rj, k)) {
            for (int w = 0; w < t->nw; ++w) rj[w] ^= q[w];
            t->z[2 * j] ^= z[0];
            t->z[2 * j + 1] ^= z[1];
        }
    }
    memcpy(t->r + (size_t)k * t->nw, q, sizeof(uint64_t) * (size_t)t->nw);
    t->z[2 * k] = z[0];
    t->z[2 * k + 1] = z[1];
    t->occupied[k] = 1;
    t->rank++;
}

/*
 * Stream the rows of contexts [c0, c1) in order.  Row i of context c:
 * y words at y + 4*(row_off[c] + i), feature words at
 * x + x_off[c] + i*ceil(n_c/32).  Different context ranges may run in
 * parallel threads.
 */
int f2o_learn(f2o_state* s, int32_t c0, int32_t c1, const int64_t* row_off, const int64_t* x_off,
              const uint32_t* x, const uint32_t* y)
{
    if (!s || c0 < 0 || c1 > s->num_ctx) return -1;
    for (int32_t c = c0; c < c1; ++c) {
        f2o_ctx* t = &s->ctx[c];
        const int W = (t->n + 31) / 32;
        const int64_t T = row_off[c + 1] - row_off[c];
        if (T < 0) return -1;
        for (int64_t i = 0; i < T; ++i)
            learn_row(s, t, x + x_off[c] + i * W, y + 4 * (row_off[c] + i));
    }
    return 0;
}

/* Canonical exchange layout (uint32 words, Wd = ceil(d/32)):
 *   rank[c], pivot words at pw_off[c] = sum_{c'<c} Wd_c',
 *   slot k of c at slot_off[c] = sum_{c'<c} d_c': x words at
 *   xw_off[c] + k*Wd_c (xw_off[c] = sum_{c'<c} d_c' * Wd_c'), z at 4*(slot_off[c]+k).
 * Empty slots are zero. */
int f2o_export(const f2o_state* s, int32_t* rank, uint32_t* pivot_mask, uint32_t* basis_x,
               uint32_t* basis_z, uint8_t* contra, int64_t* first_contra, uint64_t* n_contra,
               int64_t* rows_seen)
{
    int64_t slot = 0, xw = 0, pw = 0;
    for (int32_t c = 0; c < s->num_ctx; ++c) {
        const f2o_ctx* t = &s->ctx[c];
        const int Wd = (t->d + 31) / 32;
        rank[c] = t->rank;
        contra[c] = t->contra;
        first_contra[c] = t->first_contra;
        n_contra[c] = t->n_contra;
        rows_seen[c] = t->rows_seen;
        for (int w = 0; w < Wd; ++w) pivot_mask[pw + w] = 0;
        for (int k = 0; k < t->d; ++k) {
            uint32_t* bx = basis_x + xw + (int64_t)k * Wd;
            uint32_t* bz = basis_z + 4 * (slot + k);
            for (int w = 0; w < Wd; ++w) bx[w] = 0;
            for (int w = 0; w < 4; ++w) bz[w] = 0;
            if (!t->occupied[k]) continue;
            pivot_mask[pw + k / 32] |= 1u << (k % 32);
            const uint64_t* rk = t->r + (size_t)k * t->nw;
            for (int b = 0; b < t->d; ++b)
                if (get_bit(rk, b)) bx[b >> 5] |= 1u << (b & 31);
            for (int w = 0; w < 4; ++w)
                bz[w] = (uint32_t)(t->z[2 * k + w / 2] >> (32 * (w & 1)));
        }
        slot += t->d;
        xw += (int64_t)t->d * Wd;
        pw += Wd;
    }
    return 0;
}

/* Affine solve: W_out holds d_c 128-bit rows per context (at slot_off[c]):
 * W[k] = z_k for a pivot k, zero otherwise.  b = W[0], A[:, j] = W[1+j]. */
int f2o_solve(const f2o_state* s, uint32_t* W_out)
{
    int64_t slot = 0;
    for (int32_t c = 0; c < s->num_ctx; ++c) {
        const f2o_ctx* t = &s->ctx[c];
        for (int k = 0; k < t->d; ++k) {
            uint32_t* o = W_out + 4 * (slot + k);
            for (int w = 0; w < 4; ++w)
                o[w] = t->occupied[k] ? (uint32_t)(t->z[2 * k + w / 2] >> (32 * (w & 1))) : 0u;
        }
        slot += t->d;
    }
    return 0;
}

/* Encode queries [q0, q1): query q belongs to context ctx_id[q], its feature
 * words start at x + q*x_stride.  Writes the 128-bit word (zero when rejected)
 * and in_span = 1 (supported), 0 (rejected) or 0xFF (context id out of range). */
int f2o_encode(const f2o_state* s, int64_t q0, int64_t q1, const int32_t* ctx_id, const uint32_t* x,
               int32_t x_stride, uint32_t* y_out, uint8_t* in_span)
{
    uint64_t q[F2O_MAX_NW];
    for (int64_t i = q0; i < q1; ++i) {
        uint32_t* o = y_out + 4 * i;
        const int32_t c = ctx_id[i];
        if (c < 0 || c >= s->num_ctx) {
            for (int w = 0; w < 4; ++w) o[w] = 0;
            in_span[i] = 0xFF;
            continue;
        }
        const f2o_ctx* t = &s->ctx[c];
        form_row(s, t, x + i * (int64_t)x_stride, q);
        uint64_t acc[2] = {0, 0};
        for (int k = t->d - 1; k >= 0; --k) {
            if (t->occupied[k] && get_bit(q, k)) {
                const uint64_t* rk = t->r + (size_t)k * t->nw;
                for (int w = 0; w < t->nw; ++w) q[w] ^= rk[w];
                acc[0] ^= t->z[2 * k];
                acc[1] ^= t->z[2 * k + 1];
            }
        }
        const int ok = is_zero(q, t->nw);
        in_span[i] = (uint8_t)ok;
        for (int w = 0; w < 4; ++w) o[w] = ok ? (uint32_t)(acc[w / 2] >> (32 * (w & 1))) : 0u;
    }
    return 0;
}

/* Per-context summary without the basis: rank, contradiction flag, first
 * index, count and rows seen. */
int f2o_summary(const f2o_state* s, int32_t c, int32_t* rank, uint8_t* contra, int64_t* first,
                uint64_t* count, int64_t* rows_seen)
{
    if (!s || c < 0 || c >= s->num_ctx) return -1;
    const f2o_ctx* t = &s->ctx[c];
    *rank = t->rank;
    *contra = t->contra;
    *first = t->first_contra;
    *count = t->n_contra;
    *rows_seen = t->rows_seen;
    return 0;
}
