// Batched streaming Gaussian elimination over GF(2) (Sec. 2.2) on sm_103a.
//
// A call runs two passes over each context's rows (stream order = CSR order):
//
//  Pass 1 (dedup): the first occurrence of every distinct observation (x, y)
//  of a context is its representative; later equal rows are its duplicates.
//  A duplicate needs no elimination: its row equals an earlier row, so it
//  lies in the span when it arrives and is classified exactly as that earlier
//  row was -- redundant if the representative was consistent, a
//  contradiction if the representative was one (T never changes on the span).
//  Equality is decided by comparing the full rows (hash tables in shared
//  memory only propose the candidates), so the pass is exact.
//
//  Pass 2 (elimination) streams the representatives of each context, in
//  order, through a reduced basis B[k] = (r_k, z_k) held in shared memory:
//   1. reduce: each lane reduces its row against the basis as it stood at
//      the start of the round (the snapshot).  The basis is reduced (RREF,
//      the paper's step (5)), so the rows to XOR are exactly the pivots set
//      in the row itself; the warp walks the union of those pivots and every
//      lane XORs the broadcast row under its own bit;
//   2. classify: a zero feature residual means the row lies in the span of
//      the snapshot, and the map T fixed by the snapshot never changes
//      afterwards (contradicting rows are not inserted, insertions only
//      extend it), so the classification equals the one-row-at-a-time one:
//      zero word residual -> redundant, else contradiction (steps (2)-(3)).
//      A contradicting representative counts once for itself and once per
//      duplicate; its index is the first of them;
//   3. insert: the remaining rows (candidates) are eliminated among
//      themselves in stream order inside the warp (step (4)), then merged:
//      new rows go to their pivot slots and every older row is cleared at
//      the new pivot columns (step (5)).  The basis, including every z_k, is
//      the sequential algorithm's.
//
// Both passes give one warp to small contexts (many per CTA) and a whole CTA
// to large ones; contexts wider than 288 bits (d up to 1025) are eliminated
// by a separate wide kernel.  Single-block plan kernels validate the CSR
// batch and order the work longest-first.
#include <limits.h>
#include <string.h>

#include <mutex>

#include "f2_internal.cuh"

using namespace f2;

namespace {

// ---------------------------------------------------------------------------
// Check of a handed-off context (Sec. 2.2 steps (1)-(3) with the basis
// fixed).  Until a representative falls outside the span, the sequential
// algorithm leaves the basis as it is, so it classifies every such
// representative against this basis, and in any order: CTAs claim chunks
// of CHECK_CHUNK representatives, hold the basis in shared memory (a slot
// per pivot column) and reduce each representative by the pivot rows its
// own bits select (the warp walks the pivots set in any of its lanes).  A
// representative outside the span would extend the basis: the chunk
// records the first such one, and only representatives before the
// context's first are counted.  The last chunk of a context commits its
// counts; if some representative was outside the span, the context is
// listed for resume_kernel from that one on.
// ---------------------------------------------------------------------------
struct CheckArgs {
    const int64_t* row_off;
    const int64_t* x_off;
    const uint32_t* x;
    const uint4* y;
    const int32_t* rep_list;  // NULL: every row is its own representative
    const int32_t* rep_dup;
    const int32_t* rep_count;
    const int* snap_count;
    const int32_t* snap_list;
    const int32_t* snap_start;
    int* ctr;                 // [C] chunks claimed, [C] chunks done
    uint4* rec;               // two uint4 per chunk: (first outside, count lo, count hi, -), (first contradiction)
    int* resume_count;
    int32_t* resume_list;
    int32_t* resume_from;
};

struct LearnArgs {
    const int64_t* row_off;
    const int64_t* x_off;
    const uint32_t* x;
    const uint4* y;
    const int32_t* rep_list;   // representatives (row indices, per-context at row_off[c]); NULL = every row
    const int32_t* rep_dup;    // duplicates of each representative (NULL = none)
    const int32_t* rep_count;  // representatives per context (NULL = all rows)
    const int32_t* queue;
    int* counters;
    int warp_region_words;
    // contexts that reach full rank with rows left (not deduplicated): listed
    // here, the rest of their rows checked by verify_full_kernel
    int* late_count;
    int32_t* late_list;
    int32_t* late_start;
    unsigned long long* timing;  // per-context timestamps (F2_OPT_TIMING), NULL = off
    int tables;                  // reduce against a lookup table of the snapshot where it pays
    int small_region_words;      // shared memory of a warp-owned context of the small-width kernel
    int cta_region_words;        // shared memory of a CTA-owned context (the launch's dynamic size)
    // a CTA-owned context whose rank has not grown for HANDOFF_QUIET rounds,
    // with at least handoff_min representatives left, stops and is listed
    // here: check_snap_kernel checks the rest against its basis in parallel
    int handoff_min;             // 0 = never
    int* snap_count;
    int32_t* snap_list;
    int32_t* snap_start;         // its first representative left
    const int32_t* resume_from;  // resume_kernel: the first representative of each listed context
};

struct DedupArgs {
    const int64_t* row_off;
    const int64_t* x_off;
    const uint32_t* x;
    const uint4* y;
    int32_t* rep_list;
    int32_t* rep_dup;
    int32_t* rep_count;
    const int32_t* queue;
    int* counters;
    unsigned long long* timing;  // per-context timestamps (F2_OPT_TIMING), NULL = off
    int32_t* shard_reps;         // [DD_MAX_SHARDS * C]: representatives of each shard of a split context
    int32_t* shard_done;         // [C]: shards of a split context finished (the last one compacts)
};

// Per-context timestamps of a learn call (diagnostics, F2_OPT_TIMING):
// TIME_WORDS words per context -- %globaltimer at the start and end of its
// duplicate pass and of its elimination, then the SM ids that ran them.
constexpr int TIME_WORDS = 6;
__device__ __forceinline__ unsigned smid()
{
    unsigned r;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(r));
    return r;
}
__device__ __forceinline__ void time_mark(unsigned long long* timing, int c, int slot)
{
    if (timing) {
        timing[(size_t)TIME_WORDS * c + slot] = global_ns();
        timing[(size_t)TIME_WORDS * c + 4 + (slot >> 1)] = smid();
    }
}

// Shared-memory control area of an elimination group (32-bit words).
constexpr int CTL_P = 0;       // pivot mask, 48 words
constexpr int CTL_NPR = 48;    // pivots added during the current round, 48 words
constexpr int CTL_CAND = 96;   // per-warp candidate ballots, 32 words
constexpr int CTL_RANK = 160;  // rank
constexpr int CTL_CNT = 162;   // contradiction count (uint64, 8-byte aligned)
constexpr int CTL_FIRST = 164; // first contradiction index (int64)
constexpr int CTL_WORDS = 176; // size of the control area (16-byte multiple)

constexpr int FULL_THREADS = 1024;  // verify_full_kernel: one table shared by 32 warps
constexpr int FULL_CHUNK = 2048;   // rows of a full-rank context claimed at a time

// Pass 1: 16 warps per CTA, two CTAs per SM (64 registers a thread: the pass
// is bound by dependent per-row chains, so warps hide latency better than
// rows held in flight by one warp).  A warp-owned context (at most
// DD_WARP_MAX_ROWS rows) gets a table of next_pow2(2T) entries in a 6 KB
// region; a CTA-owned context a table of up to DD_CTA_E entries.  Entry =
// (fingerprint, row index) plus a duplicate counter: 12 bytes.
constexpr int DD_THREADS = 512;
constexpr int DD_WARPS = DD_THREADS / 32;
constexpr int DD_CTAS_PER_SM = 2;
constexpr int DD_WARP_MAX_ROWS = 256;           // warp-owned up to this many rows
constexpr int DD_QUAD_MAX_ROWS = 4096;          // 4-warp-owned up to this many rows
constexpr int DD_WARP_E = 512;
constexpr int DD_WARP_REGION = 3 * DD_WARP_E;   // words
constexpr int DD_QUAD_E = 4 * DD_WARP_E;
constexpr int DD_CTA_E = 8192;
constexpr int DD_SMEM = 4 * 3 * DD_CTA_E;       // bytes (also 16 warp regions)
constexpr int DD_K = 2;                         // rows per thread per round (feature rows of 1-2 words)
constexpr int DD_XW = NARROW_WD;                // widest feature row (words) of dedup_kernel<false>
constexpr int DD_XW_WIDE = 16;                  // widest of dedup_kernel<true> (one row in flight)
constexpr int DEDUP_PROBES = 8;                 // linear-probe limit
// A CTA-owned context with much more than its share of the call's rows is
// split into up to DD_MAX_SHARDS consecutive row ranges deduplicated by
// different CTAs (a queue item = context | shard << 24 | (shards - 1) << 28).
constexpr int DD_MAX_SHARDS = 8;
constexpr int SHARD_CTX_LIMIT = 1 << 24;
// Shards of at most this many rows (a shard's table of DD_CTA_E entries
// stays at most half full when half its rows repeat earlier ones).
#ifndef F2_DD_SHARD_ROWS
#define F2_DD_SHARD_ROWS 16384
#endif
constexpr int DD_SHARD_ROWS = F2_DD_SHARD_ROWS;
// A context of the 4-warp class with more than 1/DD_QUAD_SHARE of a shard
// share goes to a whole CTA (4 warps would finish it long after the SMs'
// median).
#ifndef F2_DD_QUAD_PROMOTE
#define F2_DD_QUAD_PROMOTE 1
#endif
constexpr int DD_QUAD_SHARE = 4;
// Neither applies below these sizes, where a CTA's fixed costs (its table,
// its barriers, the shards' compaction) outweigh what the split saves.
constexpr int DD_PROMOTE_MIN_ROWS = 1024;
constexpr int DD_SHARD_MIN_ROWS = 2048;
static_assert(DD_WARPS * DD_WARP_REGION * 4 <= DD_SMEM, "warp regions exceed the dedup shared memory");

__host__ __device__ __forceinline__ int elim_words(int d, int wd) { return CTL_WORDS + d * row_stride(wd); }

// Dispatch on a width 1..9 (feature words) to a template instantiation.
#define F2_SMALL_SWITCH(wd, CALL)    \
    switch (wd) {                    \
    case 1: CALL(1); break;          \
    case 2: CALL(2); break;          \
    case 3: CALL(3); break;          \
    default: break;                  \
    }

#define F2_BIG_SWITCH(wd, CALL)      \
    switch (wd) {                    \
    case 4: CALL(4); break;          \
    case 5: CALL(5); break;          \
    case 6: CALL(6); break;          \
    case 7: CALL(7); break;          \
    case 8: CALL(8); break;          \
    case 9: CALL(9); break;          \
    default: break;                  \
    }

#define F2_XWIDE_SWITCH(wd, CALL)    \
    switch (wd) {                    \
    case 10: CALL(10); break;        \
    case 11: CALL(11); break;        \
    case 12: CALL(12); break;        \
    case 13: CALL(13); break;        \
    case 14: CALL(14); break;        \
    case 15: CALL(15); break;        \
    case 16: CALL(16); break;        \
    default: break;                  \
    }

#define F2_NARROW_SWITCH(wd, CALL)   \
    switch (wd) {                    \
    case 1: CALL(1); break;          \
    case 2: CALL(2); break;          \
    case 3: CALL(3); break;          \
    case 4: CALL(4); break;          \
    case 5: CALL(5); break;          \
    case 6: CALL(6); break;          \
    case 7: CALL(7); break;          \
    case 8: CALL(8); break;          \
    case 9: CALL(9); break;          \
    default: break;                  \
    }


__device__ __forceinline__ bool nonzero4(const uint4& v) { return (v.x | v.y | v.z | v.w) != 0u; }

__device__ __forceinline__ void xor4(uint4& a, const uint4& b)
{
    a.x ^= b.x;
    a.y ^= b.y;
    a.z ^= b.z;
    a.w ^= b.w;
}

// Bit v set iff feature word v (< wd) still has a non-pivot column.  Words
// made only of pivot columns are never XOR-ed: the residual is zero there.
template <int WD>
__device__ __forceinline__ uint64_t mixed_words(const uint32_t (&P)[WD], int d, int wd)
{
    uint64_t m = 0;
#pragma unroll
    for (int v = 0; v < WD; ++v) {
        if (v < wd) {
            const uint32_t valid = (v < wd - 1 || (d & 31) == 0) ? 0xffffffffu : ((1u << (d & 31)) - 1u);
            if (P[v] != valid) m |= 1ull << v;
        }
    }
    return m;
}

// Feature words exactly as supplied (bits >= n cleared), and the word.
template <int WD>
__device__ __forceinline__ void load_raw(const uint32_t* __restrict__ xrow, const uint4* __restrict__ yrow,
                                         bool valid, int n, int xw, uint32_t (&xin)[WD], uint4& y)
{
#pragma unroll
    for (int v = 0; v < WD; ++v) {
        uint32_t t = 0;
        if (valid && v < xw) t = __ldg(xrow + v);
        if (v == xw - 1 && (n & 31)) t &= (1u << (n & 31)) - 1u;
        xin[v] = t;
    }
    y = valid ? __ldg(yrow) : make_uint4(0, 0, 0, 0);
}

// q = [1 || x] (index 0 = constant) or x itself for raw feature rows.
template <int WD>
__device__ __forceinline__ void make_q(const uint32_t (&xin)[WD], bool valid, uint32_t raw, uint32_t (&q)[WD])
{
    if (raw) {
#pragma unroll
        for (int v = 0; v < WD; ++v) q[v] = xin[v];
    } else {
        q[0] = (xin[0] << 1) | (valid ? 1u : 0u);
#pragma unroll
        for (int v = 1; v < WD; ++v) q[v] = (xin[v] << 1) | (xin[v - 1] >> 31);
    }
}

// 32-bit hash of an observation (feature words and word): FNV-1a over the
// words, then a murmur-style finalizer.
template <int WD>
__device__ __forceinline__ uint32_t hash_row(const uint32_t (&xin)[WD], const uint4& y)
{
    uint32_t h = 0x811C9DC5u;
#pragma unroll
    for (int v = 0; v < WD; ++v) h = (h ^ xin[v]) * 0x01000193u;
    h = (h ^ y.x) * 0x01000193u;
    h = (h ^ y.y) * 0x01000193u;
    h = (h ^ y.z) * 0x01000193u;
    h = (h ^ y.w) * 0x01000193u;
    h ^= h >> 16;
    h *= 0x85EBCA6Bu;
    h ^= h >> 13;
    h *= 0xC2B2AE35u;
    h ^= h >> 16;
    return h;
}

template <bool CTA>
__device__ __forceinline__ void group_sync()
{
    if (CTA) __syncthreads();
    else __syncwarp();
}

// ------------------------------------------------------------------ pass 1

__device__ __forceinline__ uint32_t fnv_step(uint32_t h, uint32_t w) { return (h ^ w) * 0x01000193u; }

__device__ __forceinline__ uint32_t fmix32(uint32_t h)
{
    h ^= h >> 16;
    h *= 0x85EBCA6Bu;
    h ^= h >> 13;
    h *= 0xC2B2AE35u;
    h ^= h >> 16;
    return h;
}

__device__ __forceinline__ uint32_t last_mask(int n) { return (n & 31) ? ((1u << (n & 31)) - 1u) : 0xffffffffu; }

// Full comparison of rows i and j of a context (feature bits < n and word).
__device__ __forceinline__ bool rows_equal(const uint32_t* __restrict__ xc, const uint4* __restrict__ yc, int xw, int n,
                                           int64_t i, const uint4& yi, int64_t j)
{
    const uint4 yj = __ldg(yc + j);
    if (yj.x != yi.x || yj.y != yi.y || yj.z != yi.z || yj.w != yi.w) return false;
    const uint32_t lm = last_mask(n);
    for (int v = 0; v < xw; ++v) {
        const uint32_t m = (v == xw - 1) ? lm : 0xffffffffu;
        if (((__ldg(xc + i * xw + v) ^ __ldg(xc + j * xw + v)) & m) != 0u) return false;
    }
    return true;
}

// Find the entry of row i's content starting at slot `slot`, inserting it
// if absent.  Returns the slot (whose index field ends as the smallest row
// index of that content), or -1 when the probe budget runs out (the row then
// counts as its own representative, which is always exact).
__device__ __noinline__ int dd_find_insert(uint2* tab, int E, uint32_t h, int64_t i, const uint4& yi,
                                           const uint32_t* __restrict__ xc, const uint4* __restrict__ yc, int xw,
                                           int n, uint32_t slot, int budget)
{
    const uint32_t fp = h | 1u;
    for (int p = 0; p < budget; ++p, slot = (slot + 1) & (uint32_t)(E - 1)) {
        uint2 e = tab[slot];
        if (e.x == 0u) {
            const unsigned long long want = ((unsigned long long)(uint32_t)i << 32) | fp;
            const unsigned long long old = atomicCAS(reinterpret_cast<unsigned long long*>(tab + slot), 0ull, want);
            if (old == 0ull) return (int)slot;
            e.x = (uint32_t)old;
            e.y = (uint32_t)(old >> 32);
        }
        if (e.x == fp && rows_equal(xc, yc, xw, n, i, yi, (int64_t)e.y)) {
            if ((uint32_t)i < e.y) atomicMin(&tab[slot].y, (uint32_t)i);
            return (int)slot;
        }
    }
    return -1;
}

// Group synchronisation for pass 1: a warp, a quad of 4 warps (named
// barrier 1 + quad index, 128 threads) or the whole CTA.
template <int G>
__device__ __forceinline__ void dd_sync()
{
    if (G == 1) __syncwarp();
    else if (G == DD_WARPS) __syncthreads();
    else asm volatile("bar.sync %0, %1;" ::"r"(1 + (int)(threadIdx.x >> 5) / G), "r"(32 * G) : "memory");
}

// One group of G warps finds the representatives of context c and writes
// them, in stream order, to rep_list[row_off[c] + k] with their duplicate
// counts in rep_dup; rep_count[c] = number of representatives.  Each thread
// takes DD_K rows a round (one for feature rows of 3 or more words).  Table slot: (fingerprint, smallest row index
// of that content) plus a duplicate counter; a full row comparison decides
// every match, so a row is a duplicate only if it equals an earlier row.
//
// Shard k of nsh takes the context's rows [lo, hi) = [T*k/nsh, T*(k+1)/nsh)
// and writes its representatives, numbered from lo, at
// rep_list[row_off[c] + lo + ...]; a row
// equal to a row of an earlier shard becomes its own representative there,
// which the elimination classifies exactly all the same (it lies in the span
// when it arrives).  The last shard to finish moves the shards' lists
// together, in stream order, and sets rep_count[c].  Returns whether the
// context is done (false in the shards that did not finish last).
//
// The queue item of the context a dedup CTA is on (context, shard, shard
// count); a CTA-owned pass reads it here, before and again after its rows, so
// that no register holds it through them.
__shared__ uint32_t dd_cta_item;

template <int G, int XW>
__device__ bool dedup_ctx(const StoreDev& s, const DedupArgs& a, int c, uint32_t* region, int E, int* wcnt)
{
    int shard = 0, nsh = 1;
    if constexpr (G == DD_WARPS) {
        const uint32_t qi = dd_cta_item;
        shard = (int)((qi >> 24) & 7u);
        nsh = (int)(qi >> 28) + 1;
    }
    constexpr int NT = 32 * G;
    const int lane = threadIdx.x & 31;
    const int gw = (G == 1) ? 0 : (int)((threadIdx.x >> 5) % G);  // warp within the group
    const int t = 32 * gw + lane;
    uint2* tab = reinterpret_cast<uint2*>(region);
    int* D = reinterpret_cast<int*>(region + 2 * E);
    const CtxDesc cd = s.desc[c];
    const int n = cd.n;
    const int Tc = (int)(a.row_off[c + 1] - a.row_off[c]);
    const int lo = (int)(((long long)Tc * shard) / nsh);
    const int64_t r0 = a.row_off[c] + lo;  // this shard's rows, and its part of rep_list / rep_dup
    const int T = (int)(((long long)Tc * (shard + 1)) / nsh) - lo;
    const uint32_t* xc = a.x + a.x_off[c] + (int64_t)lo * XW;
    const uint4* yc = a.y + r0;
    const uint32_t lm = last_mask(n);
    const uint32_t emask = (uint32_t)(E - 1);
    for (int e = t; e < E; e += NT) {
        tab[e] = make_uint2(0u, 0u);
        D[e] = 0;
    }
    dd_sync<G>();
    int nrep = 0;
    // the round's rows (no prefetch into registers: the other warps hide
    // the load latency)
    constexpr int K = (XW <= 2) ? DD_K : 1;
    for (int base = 0; base < T; base += NT * K) {
        int mine[K];
        uint32_t h[K];
        uint4 yv[K];
        uint32_t xv[K][XW];
#pragma unroll
        for (int j = 0; j < K; ++j) {
            const int i = base + j * NT + t;
            const bool ok = i < T;
            yv[j] = ok ? __ldg(yc + i) : make_uint4(0, 0, 0, 0);
#pragma unroll
            for (int v = 0; v < XW; ++v) {
                const uint32_t w = ok ? __ldg(xc + (int64_t)i * XW + v) : 0u;
                xv[j][v] = (v == XW - 1) ? (w & lm) : w;
            }
        }
#pragma unroll
        for (int j = 0; j < K; ++j) {
            uint32_t hh = 0x811C9DC5u;
#pragma unroll
            for (int v = 0; v < XW; ++v) hh = fnv_step(hh, xv[j][v]);
            h[j] = fmix32(fnv_step(fnv_step(fnv_step(fnv_step(hh, yv[j].x), yv[j].y), yv[j].z), yv[j].w));
        }
        // probe by fingerprint only (shared memory): the first slot holding
        // this fingerprint, or an empty slot that the row then claims
        uint2 ent[K];
        uint32_t cs[K];
#pragma unroll
        for (int j = 0; j < K; ++j) {
            const int i = base + j * NT + t;
            mine[j] = (i < T) ? -2 : -1;  // -2 = unresolved
            ent[j] = make_uint2(0u, 0u);
            cs[j] = 0u;
            if (i < T) {
                const uint32_t fp = h[j] | 1u;
                uint32_t slot = (h[j] >> 7) & emask;
                int p = 0;
                for (; p < DEDUP_PROBES; ++p, slot = (slot + 1) & emask) {
                    uint2 e = tab[slot];
                    if (e.x == 0u) {
                        const unsigned long long want = ((unsigned long long)(uint32_t)i << 32) | fp;
                        const unsigned long long old =
                            atomicCAS(reinterpret_cast<unsigned long long*>(tab + slot), 0ull, want);
                        if (old == 0ull) {
                            mine[j] = (int)slot;
                            break;
                        }
                        e.x = (uint32_t)old;
                        e.y = (uint32_t)(old >> 32);
                    }
                    if (e.x == fp) {
                        ent[j] = e;
                        cs[j] = slot;
                        break;
                    }
                }
                if (p == DEDUP_PROBES) mine[j] = -1;  // table region full: own representative
            }
        }
        // full comparison with the fingerprint matches: every load first
        bool need[K];
        uint4 yo[K];
        uint32_t xo[K][XW];
#pragma unroll
        for (int j = 0; j < K; ++j) {
            need[j] = mine[j] == -2;
            const int64_t o = need[j] ? (int64_t)ent[j].y : 0;
            yo[j] = need[j] ? __ldg(yc + o) : make_uint4(0, 0, 0, 0);
#pragma unroll
            for (int v = 0; v < XW; ++v) xo[j][v] = need[j] ? __ldg(xc + o * XW + v) : 0u;
        }
#pragma unroll
        for (int j = 0; j < K; ++j) {
            if (!need[j]) continue;
            bool e = yo[j].x == yv[j].x && yo[j].y == yv[j].y && yo[j].z == yv[j].z && yo[j].w == yv[j].w;
#pragma unroll
            for (int v = 0; v < XW; ++v) {
                const uint32_t w = (v == XW - 1) ? (xo[j][v] & lm) : xo[j][v];
                e = e && (w == xv[j][v]);
            }
            const int i = base + j * NT + t;
            if (e) {
                if ((uint32_t)i < ent[j].y) atomicMin(&tab[cs[j]].y, (uint32_t)i);
                mine[j] = (int)cs[j];
            } else {  // a different row with the same fingerprint: keep probing
                mine[j] = dd_find_insert(tab, E, h[j], i, yv[j], xc, yc, XW, n, (cs[j] + 1) & emask,
                                         DEDUP_PROBES - 1);
            }
        }
        dd_sync<G>();
        uint32_t bal[K];
#pragma unroll
        for (int j = 0; j < K; ++j) {
            const int i = base + j * NT + t;
            const bool valid = i < T;
            const int rep = (valid && mine[j] >= 0) ? (int)tab[mine[j]].y : i;
            const bool isrep = valid && rep == i;
            if (valid && !isrep) atomicAdd(D + mine[j], 1);
            bal[j] = __ballot_sync(FULL, isrep);
            if (G > 1 && lane == 0) wcnt[gw * K + j] = __popc(bal[j]);
        }
        if (G > 1) dd_sync<G>();
#pragma unroll
        for (int j = 0; j < K; ++j) {
            int before = 0, total = __popc(bal[j]);
            if (G > 1) {
                total = 0;
                for (int ww = 0; ww < G; ++ww) {
                    const int v = wcnt[ww * K + j];
                    if (ww < gw) before += v;
                    total += v;
                }
            }
            if ((bal[j] >> lane) & 1u) {
                const int pos = nrep + before + __popc(bal[j] & ((1u << lane) - 1u));
                a.rep_list[r0 + pos] = base + j * NT + t;  // within the shard (see below)
                a.rep_dup[r0 + pos] = mine[j];
            }
            nrep += total;
        }
        if (G > 1) dd_sync<G>();
    }
    dd_sync<G>();
    for (int k = t; k < nrep; k += NT) {
        const int slot = a.rep_dup[r0 + k];
        a.rep_dup[r0 + k] = (slot >= 0) ? D[slot] : 0;
    }
    if (t == 0) {
        // the call's work, for the elimination plan's thresholds
        atomicAdd(reinterpret_cast<unsigned long long*>(a.counters + CNT_WORK),
                  (unsigned long long)nrep * (unsigned long long)cd.d);
        atomicAdd(reinterpret_cast<unsigned long long*>(a.counters + CNT_REPS), (unsigned long long)nrep);
    }
    if constexpr (G == DD_WARPS) {
        const uint32_t qi = *reinterpret_cast<const volatile uint32_t*>(&dd_cta_item);
        shard = (int)((qi >> 24) & 7u);
        nsh = (int)(qi >> 28) + 1;
    }
    if (nsh == 1) {
        if (t == 0) a.rep_count[c] = nrep;
        dd_sync<G>();
        return true;
    }
    // a split context: publish this shard's count; the last shard to finish
    // moves the lists of shards 1.. down behind shard 0's (never upward: a
    // shard's list starts at or after its destination), chunk by chunk
    // through registers, renumbering their rows from the context's first
    __shared__ int s_last;
    __threadfence();  // this thread's list entries, before the count that publishes them
    dd_sync<G>();
    if (t == 0) {
        a.shard_reps[(size_t)DD_MAX_SHARDS * c + shard] = nrep;
        __threadfence();
        s_last = (atomicAdd(a.shard_done + c, 1) == nsh - 1);
    }
    dd_sync<G>();
    if (!s_last) return false;
    __threadfence();
    const int64_t cbase = a.row_off[c];
    const int Tall = (int)(a.row_off[c + 1] - cbase);
    int dst = 0;
    for (int k = 0; k < nsh; ++k) {
        const int src = (int)(((long long)Tall * k) / nsh);
        const int cnt = __ldcg(a.shard_reps + (size_t)DD_MAX_SHARDS * c + k);
        if (k > 0) {
            for (int b0 = 0; b0 < cnt; b0 += NT) {
                const int j = b0 + t;
                int32_t rl = 0, rd = 0;
                if (j < cnt) {
                    rl = __ldcg(a.rep_list + cbase + src + j) + src;
                    rd = __ldcg(a.rep_dup + cbase + src + j);
                }
                dd_sync<G>();
                if (j < cnt) {
                    a.rep_list[cbase + dst + j] = rl;
                    a.rep_dup[cbase + dst + j] = rd;
                }
                dd_sync<G>();
            }
        }
        dst += cnt;
    }
    if (t == 0) a.rep_count[c] = dst;
    dd_sync<G>();
    return true;
}

__device__ __forceinline__ int pow2_at_least(int v)
{
    int e = 64;
    while (e < v) e <<= 1;
    return e;
}

// Pass 1 kernel: CTA-owned contexts first, then quads, then warps.
template <bool WX>
__global__ void __launch_bounds__(DD_THREADS, DD_CTAS_PER_SM) dedup_kernel(StoreDev s, DedupArgs a)
{
    // WX: the contexts whose feature rows have DD_XW + 1 .. DD_XW_WIDE words
    constexpr int C_CTA = WX ? CLS_DDW_CTA : CLS_DD_CTA;
    constexpr int C_QUAD = WX ? CLS_DDW_QUAD : CLS_DD_QUAD;
    constexpr int C_WARP = WX ? CLS_DDW_WARP : CLS_DD_WARP;
    extern __shared__ __align__(16) uint32_t smem[];
    __shared__ int s_item[DD_WARPS];
    __shared__ int wcnt[DD_WARPS * DD_K];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    {
        const int n = a.counters[CNT_COUNT + C_CTA];
        const int b = a.counters[CNT_BEGIN + C_CTA];
        for (;;) {
            __syncthreads();
            if (threadIdx.x == 0) {
                const int it = atomicAdd(a.counters + CNT_HEAD + C_CTA, 1);
                s_item[0] = it;
                if (it < n) dd_cta_item = (uint32_t)a.queue[b + it];
            }
            __syncthreads();
            const int item = s_item[0];
            if (item >= n) break;
            const uint32_t qi = dd_cta_item;
            const int c = (int)(qi & (SHARD_CTX_LIMIT - 1));
            const int nsh = (int)(qi >> 28) + 1;
            const int T = (int)(a.row_off[c + 1] - a.row_off[c]);
            int E = pow2_at_least(2 * ((T + nsh - 1) / nsh));
            if (E > DD_CTA_E) E = DD_CTA_E;
            // a split context's pass: from its first shard's start to the end of the last one
            if (threadIdx.x == 0 && ((qi >> 24) & 7u) == 0) time_mark(a.timing, c, 0);
            bool done = true;
#define F2_DD_CTA(W) done = dedup_ctx<DD_WARPS, W>(s, a, c, smem, E, wcnt)
            if constexpr (WX) {
                F2_XWIDE_SWITCH(s.desc[c].xw, F2_DD_CTA)
            } else {
                F2_NARROW_SWITCH(s.desc[c].xw, F2_DD_CTA)
            }
#undef F2_DD_CTA
            if (threadIdx.x == 0 && done) time_mark(a.timing, c, 1);
        }
    }
    {
        const int q = warp / 4;
        const int n = a.counters[CNT_COUNT + C_QUAD];
        const int b = a.counters[CNT_BEGIN + C_QUAD];
        uint32_t* region = smem + q * 4 * DD_WARP_REGION;
        for (;;) {
            dd_sync<4>();
            if ((warp & 3) == 0 && lane == 0) s_item[q] = atomicAdd(a.counters + CNT_HEAD + C_QUAD, 1);
            dd_sync<4>();
            const int item = s_item[q];
            if (item >= n) break;
            const int c = a.queue[b + item];
            const int T = (int)(a.row_off[c + 1] - a.row_off[c]);
            int E = pow2_at_least(2 * T);
            if (E > DD_QUAD_E) E = DD_QUAD_E;
            if ((warp & 3) == 0 && lane == 0) time_mark(a.timing, c, 0);
#define F2_DD_QUAD(W) dedup_ctx<4, W>(s, a, c, region, E, wcnt + q * 4 * DD_K)
            if constexpr (WX) {
                F2_XWIDE_SWITCH(s.desc[c].xw, F2_DD_QUAD)
            } else {
                F2_NARROW_SWITCH(s.desc[c].xw, F2_DD_QUAD)
            }
#undef F2_DD_QUAD
            if ((warp & 3) == 0 && lane == 0) time_mark(a.timing, c, 1);
        }
    }
    {
        const int n = a.counters[CNT_COUNT + C_WARP];
        const int b = a.counters[CNT_BEGIN + C_WARP];
        uint32_t* region = smem + warp * DD_WARP_REGION;
        for (;;) {
            int item = 0;
            if (lane == 0) item = atomicAdd(a.counters + CNT_HEAD + C_WARP, 1);
            item = __shfl_sync(FULL, item, 0);
            if (item >= n) break;
            const int c = a.queue[b + item];
            const int T = (int)(a.row_off[c + 1] - a.row_off[c]);
            const int E = pow2_at_least(2 * T);
            if (lane == 0) time_mark(a.timing, c, 0);
#define F2_DD_WARP(W) dedup_ctx<1, W>(s, a, c, region, E, nullptr)
            if constexpr (WX) {
                F2_XWIDE_SWITCH(s.desc[c].xw, F2_DD_WARP)
            } else {
                F2_NARROW_SWITCH(s.desc[c].xw, F2_DD_WARP)
            }
#undef F2_DD_WARP
            if (lane == 0) time_mark(a.timing, c, 1);
        }
    }
}

// Step (1) against the snapshot S.  On return the residual is zero at every
// pivot column of words that are not "mixed"; the caller masks with ~P.
template <int WD>
__device__ __forceinline__ void reduce_snapshot(uint32_t (&xr)[WD], uint4& yr, const uint32_t* __restrict__ S,
                                                const uint32_t (&P)[WD], uint64_t mixed)
{
    constexpr int RS = row_stride(WD);
    // A stored row never changes another pivot bit of the lane's row, so the
    // bit that selects row b is the row's own bit b however the rows are
    // ordered: two pivots are taken per step, their loads issued together.
#pragma unroll
    for (int w = 0; w < WD; ++w) {
        uint32_t uw = __reduce_or_sync(FULL, xr[w] & P[w]);
        const bool xwork = (mixed & ((2ull << w) - 1ull)) != 0;
        const uint32_t sel = xr[w];
        while (uw) {
            const int b0 = __ffs(uw) - 1;
            uw &= uw - 1;
            const bool two = uw != 0u;
            const int b1 = two ? __ffs(uw) - 1 : b0;
            uw &= uw - 1;
            const uint32_t* row0 = S + (32 * w + b0) * RS;
            const uint32_t* row1 = S + (32 * w + b1) * RS;
            const uint32_t m0 = 0u - ((sel >> b0) & 1u);
            const uint32_t m1 = two ? 0u - ((sel >> b1) & 1u) : 0u;
            const uint4 z0 = *reinterpret_cast<const uint4*>(row0);
            const uint4 z1 = *reinterpret_cast<const uint4*>(row1);
            yr.x ^= (z0.x & m0) ^ (z1.x & m1);
            yr.y ^= (z0.y & m0) ^ (z1.y & m1);
            yr.z ^= (z0.z & m0) ^ (z1.z & m1);
            yr.w ^= (z0.w & m0) ^ (z1.w & m1);
            if (xwork) {
#pragma unroll
                for (int v4 = 0; v4 <= w / 4; ++v4) {
                    const uint4 xa = *reinterpret_cast<const uint4*>(row0 + 4 + 4 * v4);
                    const uint4 xb = *reinterpret_cast<const uint4*>(row1 + 4 + 4 * v4);
                    const uint32_t ea[4] = {xa.x, xa.y, xa.z, xa.w};
                    const uint32_t eb[4] = {xb.x, xb.y, xb.z, xb.w};
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int v = 4 * v4 + j;
                        if (v <= w && v < WD)
                            if ((mixed >> v) & 1ull) xr[v] ^= (ea[j] & m0) ^ (eb[j] & m1);
                    }
                }
            }
        }
    }
}

// Reduce a candidate (already zero at the snapshot's pivots) against rows
// inserted earlier in the same round (CTA mode).  Per lane.
template <int WD>
__device__ __forceinline__ void reduce_new(uint32_t (&xr)[WD], uint4& yr, const uint32_t* __restrict__ S,
                                           const uint32_t* __restrict__ NPR)
{
    constexpr int RS = row_stride(WD);
#pragma unroll
    for (int w = 0; w < WD; ++w) {
        uint32_t m = xr[w] & NPR[w];
        while (m) {
            const int b = __ffs(m) - 1;
            m &= m - 1;
            const uint32_t* row = S + (32 * w + b) * RS;
            xor4(yr, *reinterpret_cast<const uint4*>(row));
#pragma unroll
            for (int v = 0; v <= w; ++v) xr[v] ^= row[4 + v];
        }
    }
}

// Steps (4)-(5) for the candidate lanes of one warp, in lane (= stream)
// order.  Returns the number of rows inserted; NP receives their pivots.
// P (the pivots before this call) is not modified.
template <int WD>
__device__ int insert_block(uint32_t (&xr)[WD], uint4& yr, uint32_t cand, uint32_t* __restrict__ S,
                            const uint32_t (&P)[WD], int d, int lane, long long idx, long long& first,
                            unsigned long long& cnt, uint32_t (&NP)[WD], bool& contra_lane, uint32_t weight)
{
    constexpr int RS = row_stride(WD);
    int pk = -1;
    uint32_t newp = 0;
    while (cand) {
        const int i = __ffs(cand) - 1;
        cand &= cand - 1;
        int mine = -1;
#pragma unroll
        for (int v = 0; v < WD; ++v)
            if (xr[v]) mine = 32 * v + 31 - __clz(xr[v]);
        const int k = __shfl_sync(FULL, mine, i);
        if (k < 0) {  // reduced to zero by rows inserted earlier in this block
            if (lane == i && nonzero4(yr)) {
                cnt += weight;
                first = min(first, idx);
                contra_lane = true;
            }
            continue;
        }
        const int kw = k >> 5;
        const uint32_t kb = 1u << (k & 31);
        uint32_t sel = 0;
#pragma unroll
        for (int v = 0; v < WD; ++v)
            if (v == kw) sel = xr[v];
        const bool hit = (lane != i) && (sel & kb);
#pragma unroll
        for (int v = 0; v < WD; ++v) {
            const uint32_t t = __shfl_sync(FULL, xr[v], i);
            if (hit) xr[v] ^= t;
        }
        uint4 bz;
        bz.x = __shfl_sync(FULL, yr.x, i);
        bz.y = __shfl_sync(FULL, yr.y, i);
        bz.z = __shfl_sync(FULL, yr.z, i);
        bz.w = __shfl_sync(FULL, yr.w, i);
        if (hit) xor4(yr, bz);
        if (lane == i) pk = k;
        newp |= 1u << i;
    }
#pragma unroll
    for (int v = 0; v < WD; ++v) NP[v] = 0;
    if (!newp) return 0;
    if (pk >= 0) {
        uint32_t* row = S + pk * RS;
        *reinterpret_cast<uint4*>(row) = yr;
#pragma unroll
        for (int v = 0; v < RS - 4; ++v) row[4 + v] = (v < WD) ? xr[v] : 0u;
    }
#pragma unroll
    for (int v = 0; v < WD; ++v)
        NP[v] = __reduce_or_sync(FULL, (pk >= 0 && (pk >> 5) == v) ? (1u << (pk & 31)) : 0u);
    __syncwarp();
    // step (5): clear the new pivot columns from every previously stored row
    for (int j = lane; j < d; j += 32) {
        uint32_t pj = 0;
#pragma unroll
        for (int v = 0; v < WD; ++v)
            if (v == (j >> 5)) pj = P[v];
        if (!((pj >> (j & 31)) & 1u)) continue;
        uint32_t* rj = S + j * RS;
        uint32_t xj[WD];
        uint32_t hits = 0;
#pragma unroll
        for (int v = 0; v < WD; ++v) {
            xj[v] = rj[4 + v];
            hits |= xj[v] & NP[v];
        }
        if (!hits) continue;
        uint4 zj = *reinterpret_cast<const uint4*>(rj);
#pragma unroll
        for (int v = 0; v < WD; ++v) {
            uint32_t m = xj[v] & NP[v];
            while (m) {
                const int b = __ffs(m) - 1;
                m &= m - 1;
                const uint32_t* rk = S + (32 * v + b) * RS;
                xor4(zj, *reinterpret_cast<const uint4*>(rk));
#pragma unroll
                for (int u = 0; u <= v; ++u) xj[u] ^= rk[4 + u];
            }
        }
        *reinterpret_cast<uint4*>(rj) = zj;
#pragma unroll
        for (int v = 0; v < WD; ++v) rj[4 + v] = xj[v];
    }
    __syncwarp();
    return __popc(newp);
}

// The stored basis moves between global and shared memory by its pivot rows
// only: an empty slot is zero in the store and never read in shared memory
// (every read of S selects a pivot), and a slot that became a pivot stays one.
template <int WD>
__device__ void basis_to_smem(const StoreDev& s, const CtxDesc& cd, uint32_t* S, const uint32_t* Ps, int t, int nt)
{
    constexpr int RS = row_stride(WD);
    for (int k = t; k < cd.d; k += nt) {
        if (!((Ps[k >> 5] >> (k & 31)) & 1u)) continue;
        uint32_t* row = S + k * RS;
        *reinterpret_cast<uint4*>(row) = s.bz[cd.slot_off + k];
        const uint32_t* src = s.bx + cd.xw_off + (int64_t)k * cd.wd;
        for (int v = 0; v < RS - 4; ++v) row[4 + v] = (v < cd.wd) ? src[v] : 0u;
    }
}

template <int WD>
__device__ void basis_from_smem(const StoreDev& s, const CtxDesc& cd, const uint32_t* S, const uint32_t* Ps, int t,
                                int nt)
{
    constexpr int RS = row_stride(WD);
    for (int k = t; k < cd.d; k += nt) {
        if (!((Ps[k >> 5] >> (k & 31)) & 1u)) continue;
        const uint32_t* row = S + k * RS;
        s.bz[cd.slot_off + k] = *reinterpret_cast<const uint4*>(row);
        uint32_t* dst = s.bx + cd.xw_off + (int64_t)k * cd.wd;
        for (int v = 0; v < cd.wd; ++v) dst[v] = row[4 + v];
    }
}

__device__ __forceinline__ void warp_stats(long long& first, unsigned long long& cnt)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        first = min(first, __shfl_xor_sync(FULL, first, o));
        cnt += __shfl_xor_sync(FULL, cnt, o);
    }
}

__device__ __forceinline__ void commit_stats(const StoreDev& s, int c, long long first, unsigned long long cnt)
{
    if (cnt) {
        s.n_contra[c] += cnt;
        s.contra[c] = 1;
        if (s.first_contra[c] < 0) s.first_contra[c] = first;
    }
}

// ------------------------------------------------------------------ pass 2

// Set compressed residual bit tt (< 32 * TABLE_MAX_RW).
__device__ __forceinline__ void set_rbit(uint32_t (&er)[TABLE_MAX_RW], int tt)
{
#pragma unroll
    for (int u = 0; u < TABLE_MAX_RW; ++u)
        if ((tt >> 5) == u) er[u] |= 1u << (tt & 31);
}

constexpr int FL_WORDS = 64;  // free-coordinate list of a table: 128 uint16 entries

// The lookup table (layout in f2_internal.cuh) of the basis held in shared
// memory: pivot rows S (row stride row_stride(WD)), pivot mask P, rank; FL
// receives the non-pivot coordinates in increasing order (the meaning of the
// compressed residual bits).  All nt threads of the group take part.
template <int WD, bool CTA>
__device__ void build_table_smem(const uint32_t* __restrict__ S, const uint32_t (&P)[WD], int d, int wd, int rank,
                                 uint32_t* __restrict__ TB, uint16_t* __restrict__ FL, int t, int nt)
{
    constexpr int RS = row_stride(WD);
    const int np = (d + 3) >> 2, rw = (d - rank + 31) >> 5;
    uint32_t f[WD];  // non-pivot coordinates of each word
    int pre[WD];     // non-pivot coordinates in the words before
    {
        int acc = 0;
#pragma unroll
        for (int w = 0; w < WD; ++w) {
            const uint32_t valid = (w < wd) ? ((w == wd - 1 && (d & 31)) ? ((1u << (d & 31)) - 1u) : 0xffffffffu) : 0u;
            f[w] = ~P[w] & valid;
            pre[w] = acc;
            acc += __popc(f[w]);
        }
    }
    uint2* const Zl = reinterpret_cast<uint2*>(TB);
    uint2* const Zh = Zl + 16 * np;
    uint32_t* const R = TB + 64 * np;
    for (int j = t; j < 4 * np; j += nt) {
        uint4 z = make_uint4(0, 0, 0, 0);
        uint32_t er[TABLE_MAX_RW] = {0, 0, 0, 0};
        if (j < d) {
            const int w = j >> 5, b = j & 31;
            uint32_t fw = 0;
            int pw = 0;
#pragma unroll
            for (int u = 0; u < WD; ++u)
                if (u == w) {
                    fw = f[u];
                    pw = pre[u];
                }
            if ((fw >> b) & 1u) {  // a non-pivot coordinate: its unit vector
                const int tt = pw + __popc(fw & ((1u << b) - 1u));
                set_rbit(er, tt);
                FL[tt] = (uint16_t)j;
            } else {  // a pivot: z_j and r_j on the non-pivot coordinates
                const uint32_t* row = S + j * RS;
                z = *reinterpret_cast<const uint4*>(row);
#pragma unroll
                for (int u = 0; u < WD; ++u) {
                    if (u <= w) {
                        uint32_t bits = row[4 + u] & f[u];
                        while (bits) {
                            const int bb = __ffs(bits) - 1;
                            bits &= bits - 1u;
                            set_rbit(er, pre[u] + __popc(f[u] & ((1u << bb) - 1u)));
                        }
                    }
                }
            }
        }
        const int e = 16 * (j >> 2) + (1 << (j & 3));
        Zl[e] = make_uint2(z.x, z.y);
        Zh[e] = make_uint2(z.z, z.w);
#pragma unroll
        for (int u = 0; u < TABLE_MAX_RW; ++u)
            if (u < rw) R[u * 16 * np + e] = er[u];
        if ((j & 3) == 0) {
            const int e0 = 16 * (j >> 2);
            Zl[e0] = make_uint2(0, 0);
            Zh[e0] = make_uint2(0, 0);
#pragma unroll
            for (int u = 0; u < TABLE_MAX_RW; ++u)
                if (u < rw) R[u * 16 * np + e0] = 0u;
        }
    }
    group_sync<CTA>();
    // entries of two or more coordinates: XOR of their single entries
    for (int k = t; k < 16 * np; k += nt) {
        const int v = k & 15;
        if (__popc(v) < 2) continue;
        const int eb = k & ~15;
        uint2 lo = make_uint2(0, 0), hi = make_uint2(0, 0);
        uint32_t rr[TABLE_MAX_RW] = {0, 0, 0, 0};
#pragma unroll
        for (int bb = 0; bb < 4; ++bb) {
            if ((v >> bb) & 1) {
                const int es = eb + (1 << bb);
                const uint2 l = Zl[es], h = Zh[es];
                lo.x ^= l.x;
                lo.y ^= l.y;
                hi.x ^= h.x;
                hi.y ^= h.y;
#pragma unroll
                for (int u = 0; u < TABLE_MAX_RW; ++u)
                    if (u < rw) rr[u] ^= R[u * 16 * np + es];
            }
        }
        Zl[k] = lo;
        Zh[k] = hi;
#pragma unroll
        for (int u = 0; u < TABLE_MAX_RW; ++u)
            if (u < rw) R[u * 16 * np + k] = rr[u];
    }
    group_sync<CTA>();
}

// The full residual (feature words, zero at the pivots) from its compressed
// form: bit tt is the non-pivot coordinate FL[tt].
template <int WD>
__device__ __forceinline__ void decompress_residual(const uint32_t (&cr)[TABLE_MAX_RW], int rw,
                                                    const uint16_t* __restrict__ FL, uint32_t (&xr)[WD])
{
#pragma unroll
    for (int v = 0; v < WD; ++v) xr[v] = 0u;
#pragma unroll
    for (int u = 0; u < TABLE_MAX_RW; ++u) {
        uint32_t bits = (u < rw) ? cr[u] : 0u;
        while (bits) {
            const int bb = __ffs(bits) - 1;
            bits &= bits - 1u;
            const int coord = FL[32 * u + bb];
#pragma unroll
            for (int v = 0; v < WD; ++v)
                if ((coord >> 5) == v) xr[v] |= 1u << (coord & 31);
        }
    }
}

// Snapshot reduction by table: acc of the word parts into yr, the residual
// (zero at the pivots) into xr; returns whether it is nonzero.
template <int WD>
__device__ __forceinline__ bool reduce_by_table(uint32_t (&xr)[WD], uint4& yr, const uint32_t* __restrict__ TB,
                                                const uint16_t* __restrict__ FL, int np, int rw)
{
    uint32_t q[WD];
#pragma unroll
    for (int v = 0; v < WD; ++v) q[v] = xr[v];
    uint4 acc;
    uint32_t cr[TABLE_MAX_RW] = {0, 0, 0, 0};
    switch (rw) {
    case 0: {
        uint32_t r0[1];
        table_reduce<0, WD>(TB, np, q, acc, r0);
        break;
    }
    case 1: {
        uint32_t r1[1];
        table_reduce<1, WD>(TB, np, q, acc, r1);
        cr[0] = r1[0];
        break;
    }
    case 2: {
        uint32_t r2[2];
        table_reduce<2, WD>(TB, np, q, acc, r2);
        cr[0] = r2[0];
        cr[1] = r2[1];
        break;
    }
    case 3: {
        uint32_t r3[3];
        table_reduce<3, WD>(TB, np, q, acc, r3);
        cr[0] = r3[0];
        cr[1] = r3[1];
        cr[2] = r3[2];
        break;
    }
    default: {
        uint32_t r4[4];
        table_reduce<4, WD>(TB, np, q, acc, r4);
        cr[0] = r4[0];
        cr[1] = r4[1];
        cr[2] = r4[2];
        cr[3] = r4[3];
        break;
    }
    }
    yr.x ^= acc.x;
    yr.y ^= acc.y;
    yr.z ^= acc.z;
    yr.w ^= acc.w;
    const bool nz = (cr[0] | cr[1] | cr[2] | cr[3]) != 0u;
    if (nz) decompress_residual<WD>(cr, rw, FL, xr);
    else {
#pragma unroll
        for (int v = 0; v < WD; ++v) xr[v] = 0u;
    }
    return nz;
}

// Hand-off of saturated contexts (see LearnArgs): the quiet rounds before
// it, the widest basis the check can hold (shared memory words, a slot per
// coordinate) and its chunks of representatives; the row widths of the two
// instances of the wide kernel (the 10..17-word one takes part).
constexpr int HANDOFF_QUIET = 2;
constexpr int CHECK_BASIS_WORDS = 14336;  // 56 KB
constexpr int CHECK_CHUNK = 512;
constexpr int HANDOFF_CALL_FACTOR = 16;  // calls of fewer rows than this many hand-off minimums hand off none
constexpr int WIDE_WD = 33;    // widest row (d <= 1056)
constexpr int WIDE_M_WD = 17;  // rows of 10..17 words (d <= 544): half the registers, two CTAs per SM

// One group (a warp, or the whole CTA) streams the representatives of
// context c through its basis.
template <int WD, bool CTA>
__device__ void elim_ctx(const StoreDev& s, const LearnArgs& a, int c, uint32_t* region, int region_words)
{
    const int G = CTA ? (int)(blockDim.x >> 5) : 1;
    const int lane = threadIdx.x & 31;
    const int warp = CTA ? (int)(threadIdx.x >> 5) : 0;
    const int t = 32 * warp + lane;
    const int nt = 32 * G;
    const CtxDesc cd = s.desc[c];
    uint32_t* ctl = region;
    uint32_t* Ps = ctl + CTL_P;
    uint32_t* NPR = ctl + CTL_NPR;
    uint32_t* wc = ctl + CTL_CAND;
    int* rank_s = reinterpret_cast<int*>(ctl + CTL_RANK);
    unsigned long long* cnt_s = reinterpret_cast<unsigned long long*>(ctl + CTL_CNT);
    long long* first_s = reinterpret_cast<long long*>(ctl + CTL_FIRST);
    uint32_t* S = region + CTL_WORDS;
    const int rank0 = s.rank[c];
    if (t < 48) {
        Ps[t] = (t < cd.wd && rank0 != 0) ? s.pivot[cd.pw_off + t] : 0u;
        NPR[t] = 0u;
    }
    if (t == 0) {
        *rank_s = rank0;
        *cnt_s = 0ull;
        *first_s = LLONG_MAX;
    }
    group_sync<CTA>();
    if (rank0 != 0) {
        basis_to_smem<WD>(s, cd, S, Ps, t, nt);
        group_sync<CTA>();
    }
    uint32_t P[WD];
#pragma unroll
    for (int v = 0; v < WD; ++v) P[v] = Ps[v];
    uint64_t mixed = mixed_words<WD>(P, cd.d, cd.wd);
    // lookup table of the snapshot (rebuilt after a round that inserted):
    // after the basis rows, the free-coordinate list at the region's end
    constexpr int RS = row_stride(WD);
    uint32_t* const TB = S + cd.d * RS;
    uint16_t* const FL = reinterpret_cast<uint16_t*>(region + region_words - FL_WORDS);
    const int tab_cap = region_words - FL_WORDS - CTL_WORDS - cd.d * RS;
    const int np = (cd.d + 3) >> 2;
    bool dirty = true;
    const long long seen = s.rows_seen[c];
    const int64_t r0 = a.row_off[c];
    const int64_t T = a.row_off[c + 1] - r0;
    const int rc = a.rep_count ? a.rep_count[c] : -((int)T + 2);
    const bool deduped = rc >= 0;
    const int R = deduped ? rc : -(rc + 2);
    const int32_t* reps = deduped ? a.rep_list + r0 : nullptr;
    const int32_t* dups = deduped ? a.rep_dup + r0 : nullptr;
    const uint32_t* xc = a.x + a.x_off[c];
    const uint4* yc = a.y + r0;
    long long first = LLONG_MAX;
    unsigned long long cnt = 0;
    // prefetched round
    const int k0 = a.resume_from ? a.resume_from[c] : 0;  // the first representative of this launch
    int nk = k0 + t;
    bool nvalid = nk < R;
    int ni = nvalid ? (reps ? __ldg(reps + nk) : nk) : 0;
    uint32_t nw = (nvalid && dups) ? (uint32_t)__ldg(dups + nk) : 0u;
    uint32_t xn[WD];
    uint4 yn;
    load_raw<WD>(xc + (int64_t)ni * cd.xw, yc + ni, nvalid, cd.n, cd.xw, xn, yn);
    int stop_at = -1;
    int snap_at = -1;  // handed off from this representative on
    int quiet = 0;     // rounds in a row that inserted nothing
    int parity = 0;
    for (int base = k0; base < R; base += nt, parity ^= 1) {
        const bool valid = nvalid;
        const int i = ni;
        const uint32_t weight = 1u + nw;
        uint32_t xr[WD];
        make_q<WD>(xn, valid, s.raw, xr);
        uint4 yr = yn;
        nk += nt;
        nvalid = nk < R;
        ni = nvalid ? (reps ? __ldg(reps + nk) : nk) : 0;
        nw = (nvalid && dups) ? (uint32_t)__ldg(dups + nk) : 0u;
        load_raw<WD>(xc + (int64_t)ni * cd.xw, yc + ni, nvalid, cd.n, cd.xw, xn, yn);
        // step (1) against the snapshot: by lookup table where the table fits
        // and costs fewer instructions than walking the pivots (about d/4
        // lookups a row against about rank/2 two-pivot steps), else by walk
        int tmode = 0;  // 1 + residual words of the table, 0 = walk
        // (CTA-owned contexts only: their many rounds after the basis stops
        // growing repay the rebuilds; a warp-owned context has few rounds,
        // most of them inserting, and keeps the small shared-memory region
        // that lets more warps run)
        if constexpr (CTA && WD <= TABLE_MAX_WD) {
            if (a.tables) {
                const int rk = *rank_s;
                const int rw = (cd.d - rk + 31) >> 5;
                if (rw <= TABLE_MAX_RW && table_words(cd.d, rk) <= tab_cap && 4 * rk >= 5 * np) {
                    tmode = 1 + rw;
                    if (dirty) {
                        build_table_smem<WD, CTA>(S, P, cd.d, cd.wd, rk, TB, FL, t, nt);
                        dirty = false;
                    }
                }
            }
        }
        uint32_t nz = 0;
        if (tmode) {
            nz = reduce_by_table<WD>(xr, yr, TB, FL, np, tmode - 1) ? 1u : 0u;
        } else {
            reduce_snapshot<WD>(xr, yr, S, P, mixed);
#pragma unroll
            for (int v = 0; v < WD; ++v) {
                xr[v] &= ~P[v];
                nz |= xr[v];
            }
        }
        bool contra_lane = false;
        if (valid && !nz && nonzero4(yr)) {
            cnt += weight;
            first = min(first, seen + (long long)i);
            contra_lane = true;
        }
        const uint32_t cand = __ballot_sync(FULL, valid && nz != 0u);
        uint32_t wmask;
        if (CTA) {
            // two alternating ballot buffers: a round without candidates
            // ends without a barrier, so the next round's ballots must not
            // overwrite this round's before every warp has read them
            uint32_t* const wcp = wc + 16 * parity;
            if (lane == 0) wcp[warp] = cand;
            __syncthreads();
            wmask = 0;
            for (int ww = 0; ww < G; ++ww)
                if (wcp[ww]) wmask |= 1u << ww;
        } else {
            wmask = cand ? 1u : 0u;
        }
        if (wmask) {
            const int first_warp = __ffs(wmask) - 1;
            for (uint32_t wm = wmask; wm; wm &= wm - 1) {
                const int ww = __ffs(wm) - 1;
                if (warp == ww) {
                    if (CTA && ww != first_warp) reduce_new<WD>(xr, yr, S, NPR);
                    uint32_t NP[WD];
                    const int added = insert_block<WD>(xr, yr, cand, S, P, cd.d, lane, seen + (long long)i, first, cnt,
                                                       NP, contra_lane, weight);
                    if (lane == 0 && added) {
#pragma unroll
                        for (int v = 0; v < WD; ++v) {
                            Ps[v] = P[v] | NP[v];
                            NPR[v] |= NP[v];
                        }
                        *rank_s += added;
                    }
                }
                group_sync<CTA>();
#pragma unroll
                for (int v = 0; v < WD; ++v) P[v] = Ps[v];
            }
            mixed = mixed_words<WD>(P, cd.d, cd.wd);
            dirty = true;
            if (CTA) {
                if (t < 48) NPR[t] = 0u;
            }
            // (wide contexts) full rank with at least a chunk of rows left:
            // every later row is a check only (the rows are their own
            // representatives here)
            if constexpr (WD > NARROW_WD) {
                if (!deduped && a.late_list && R - (base + nt) >= FULL_CHUNK && *rank_s == cd.d) {
                    stop_at = base + nt;
                    break;
                }
            }
        }
        if constexpr (CTA && (WD <= NARROW_WD || WD == WIDE_M_WD)) {
            // every rank >= 1 saturated context with many representatives
            // left: hand the rest off to the parallel check (block-uniform)
            quiet = wmask ? 0 : quiet + 1;
            if (a.handoff_min > 0 && !a.resume_from && quiet >= HANDOFF_QUIET && R - (base + nt) >= a.handoff_min &&
                *rank_s < cd.d && cd.d * row_stride(WD) <= CHECK_BASIS_WORDS) {
                snap_at = base + nt;
                break;
            }
        }
        (void)contra_lane;
    }
    warp_stats(first, cnt);
    if (lane == 0 && cnt) {
        atomicAdd(cnt_s, cnt);
        atomicMin(first_s, first);
    }
    group_sync<CTA>();
    if (t < cd.wd) s.pivot[cd.pw_off + t] = Ps[t];
    basis_from_smem<WD>(s, cd, S, Ps, t, nt);
    if (t == 0) {
        s.rank[c] = *rank_s;
        commit_stats(s, c, *first_s, *cnt_s);
        if (snap_at >= 0) {  // rows_seen is advanced by check_snap_kernel (or resume_kernel)
            a.snap_start[c] = snap_at;
            a.snap_list[atomicAdd(a.snap_count, 1)] = c;
        } else if (stop_at < 0) {
            s.rows_seen[c] = seen + T;
        } else {  // rows_seen is advanced by verify_full_kernel
            a.late_start[c] = stop_at;
            a.late_list[atomicAdd(a.late_count, 1)] = c;
        }
    }
    group_sync<CTA>();
}

__device__ __forceinline__ int64_t check_slot(const CheckArgs& a, int c)
{
    return a.row_off[c] / CHECK_CHUNK + c;  // the context's first chunk record (chunks never overlap)
}

template <int WD>
__device__ void check_chunk(const StoreDev& s, const CheckArgs& a, int c, int kb, int ke, const uint32_t* S,
                            const uint32_t (&P)[WD], uint8_t* flags)
{
    const CtxDesc cd = s.desc[c];
    const int64_t r0 = a.row_off[c];
    const int32_t* reps = a.rep_list ? a.rep_list + r0 : nullptr;
    const uint32_t* xc = a.x + a.x_off[c];
    const uint4* yc = a.y + r0;
    const uint64_t mixed = mixed_words<WD>(P, cd.d, cd.wd);
    // every lane of a warp in each round: the pivot walk is warp-uniform
    for (int base = kb; base < ke; base += blockDim.x) {
        const int k = base + (int)threadIdx.x;
        const bool valid = k < ke;
        const int i = valid ? (reps ? __ldg(reps + k) : k) : 0;
        uint32_t xin[WD], q[WD];
        uint4 yr;
        load_raw<WD>(xc + (int64_t)i * cd.xw, yc + i, valid, cd.n, cd.xw, xin, yr);
        make_q<WD>(xin, valid, s.raw, q);
        reduce_snapshot<WD>(q, yr, S, P, mixed);
        uint32_t resid = 0;
#pragma unroll
        for (int w = 0; w < WD; ++w) resid |= q[w] & ~P[w];
        // 2: outside the span, 1: a contradiction, 0: redundant
        if (valid) flags[k - kb] = resid ? 2 : (nonzero4(yr) ? 1 : 0);
    }
}

// Shared memory of the check: the basis (a slot of row_stride words per
// column), the chunk's classes (CHECK_CHUNK bytes), then CHECK_CTL_WORDS of
// control (the pivot words, the claimed chunk, the chunk's sums).
constexpr int CHECK_CTL_WORDS = 64;
constexpr int CHECK_SMEM_BYTES = 4 * CHECK_BASIS_WORDS + CHECK_CHUNK + 4 * CHECK_CTL_WORDS;

__global__ void __launch_bounds__(256) check_snap_kernel(StoreDev s, CheckArgs a)
{
    extern __shared__ __align__(16) uint32_t smem[];
    uint32_t* const S = smem;
    uint8_t* const flags = reinterpret_cast<uint8_t*>(smem + CHECK_BASIS_WORDS);
    uint32_t* const ctl = smem + CHECK_BASIS_WORDS + CHECK_CHUNK / 4;
    uint32_t* const Ps = ctl;  // 48 pivot words
    int* const s_c = reinterpret_cast<int*>(ctl + 48);
    int* const s_k = s_c + 1;
    int* const s_first_out = s_c + 2;
    unsigned long long* const s_cnt = reinterpret_cast<unsigned long long*>(ctl + 52);
    long long* const s_first = reinterpret_cast<long long*>(ctl + 54);
    const int t = threadIdx.x;
    int q = 0, built = -1;
    for (;;) {
        if (t == 0) {  // the next chunk, contexts in list order
            int c = -1, k = 0;
            const int nq = *a.snap_count;
            for (; q < nq; ++q) {
                const int cq = a.snap_list[q];
                const int R = a.rep_list ? a.rep_count[cq] : (int)(a.row_off[cq + 1] - a.row_off[cq]);
                k = atomicAdd(a.ctr + cq, 1);
                if (a.snap_start[cq] + k * CHECK_CHUNK < R) {
                    c = cq;
                    break;
                }
            }
            *s_c = c;
            *s_k = k;
            *s_first_out = INT_MAX;
            *s_cnt = 0ull;
            *s_first = LLONG_MAX;
        }
        __syncthreads();
        const int c = *s_c;
        const int ck = *s_k;
        if (c < 0) break;
        const CtxDesc cd = s.desc[c];
        const int R = a.rep_list ? a.rep_count[c] : (int)(a.row_off[c + 1] - a.row_off[c]);
        const int st0 = a.snap_start[c];
        const int kb = st0 + ck * CHECK_CHUNK;
        const int ke = (kb + CHECK_CHUNK < R) ? kb + CHECK_CHUNK : R;
        if (built != c) {  // the basis into shared memory (pivot rows only)
            if (t < 48) Ps[t] = (t < cd.wd) ? s.pivot[cd.pw_off + t] : 0u;
            __syncthreads();
            // the stride of the instance that checks it (rows of 10..17 words: the 17-word one)
            const int rs = row_stride(cd.wd <= NARROW_WD ? cd.wd : WIDE_M_WD);
            for (int kk = t; kk < cd.d; kk += blockDim.x) {
                if (!((Ps[kk >> 5] >> (kk & 31)) & 1u)) continue;
                uint32_t* row = S + kk * rs;
                *reinterpret_cast<uint4*>(row) = s.bz[cd.slot_off + kk];
                const uint32_t* src = s.bx + cd.xw_off + (int64_t)kk * cd.wd;
                for (int v = 0; v < rs - 4; ++v) row[4 + v] = (v < cd.wd) ? src[v] : 0u;
            }
            built = c;
            __syncthreads();
        }
#define F2_CHECK(W)                                                   \
    {                                                                 \
        uint32_t P[W];                                                \
        for (int v = 0; v < W; ++v) P[v] = Ps[v];                     \
        check_chunk<W>(s, a, c, kb, ke, S, P, flags);                 \
    }
        switch (cd.wd) {
        case 1: F2_CHECK(1); break;
        case 2: F2_CHECK(2); break;
        case 3: F2_CHECK(3); break;
        case 4: F2_CHECK(4); break;
        case 5: F2_CHECK(5); break;
        case 6: F2_CHECK(6); break;
        case 7: F2_CHECK(7); break;
        case 8: F2_CHECK(8); break;
        case 9: F2_CHECK(9); break;
        default: F2_CHECK(WIDE_M_WD); break;
        }
#undef F2_CHECK
        __syncthreads();
        // the first representative outside the span, then the contradictions
        // before it (weights: the representative and its repeats)
        for (int j = t; j < ke - kb; j += blockDim.x)
            if (flags[j] == 2) atomicMin(s_first_out, kb + j);
        __syncthreads();
        const int fo = *s_first_out;
        unsigned long long cnt = 0;
        long long first = LLONG_MAX;
        for (int j = t; j < ke - kb && kb + j < fo; j += blockDim.x) {
            if (flags[j] != 1) continue;
            const int k = kb + j;
            const int i = a.rep_list ? __ldg(a.rep_list + a.row_off[c] + k) : k;
            cnt += 1u + (a.rep_dup ? (uint32_t)__ldg(a.rep_dup + a.row_off[c] + k) : 0u);
            first = min(first, (long long)i);
        }
        if (cnt) {
            atomicAdd(s_cnt, cnt);
            atomicMin(s_first, first);
        }
        __syncthreads();
        if (t == 0) {
            const int64_t slot = check_slot(a, c) + ck;
            const unsigned long long sc = *s_cnt;
            const long long sf = *s_first;
            a.rec[2 * slot] = make_uint4((uint32_t)fo, (uint32_t)sc, (uint32_t)(sc >> 32), 0u);
            a.rec[2 * slot + 1] = make_uint4((uint32_t)sf, (uint32_t)((unsigned long long)sf >> 32), 0u, 0u);
            __threadfence();
            const int nch = (R - st0 + CHECK_CHUNK - 1) / CHECK_CHUNK;
            if (atomicAdd(a.ctr + s.num_ctx + c, 1) == nch - 1) {  // the context's last chunk
                __threadfence();
                const int64_t s0 = check_slot(a, c);
                int f = INT_MAX;
                for (int k = 0; k < nch; ++k) f = min(f, (int)__ldcg(a.rec + 2 * (s0 + k)).x);
                unsigned long long tot = 0;
                long long fi = LLONG_MAX;
                for (int k = 0; k < nch; ++k) {
                    if (st0 + k * CHECK_CHUNK >= f) break;  // chunks past the first outside
                    const uint4 r = __ldcg(a.rec + 2 * (s0 + k));
                    const uint4 r2 = __ldcg(a.rec + 2 * (s0 + k) + 1);
                    tot += (unsigned long long)r.y | ((unsigned long long)r.z << 32);
                    fi = min(fi, (long long)((unsigned long long)r2.x | ((unsigned long long)r2.y << 32)));
                }
                const long long seen = s.rows_seen[c];
                if (tot) {
                    s.n_contra[c] += tot;
                    s.contra[c] = 1;
                    if (s.first_contra[c] < 0) s.first_contra[c] = seen + fi;
                }
                if (f == INT_MAX) {
                    s.rows_seen[c] = seen + (a.row_off[c + 1] - a.row_off[c]);
                } else {  // the rest from the first representative outside the span
                    a.resume_from[c] = f;
                    a.resume_list[atomicAdd(a.resume_count, 1)] = c;
                }
            }
        }
        __syncthreads();
    }
}

// Narrow elimination: CTA-owned contexts first (longest first), then
// warp-owned ones.  SMALL: the contexts of at most SMALL_WD words, with
// fixed 4 KB warp regions and a register budget for three CTAs per SM (80
// registers, no spills; four CTAs at 64 registers spill and ran 6% slower
// on the 78k-context, 81M-row learn); else
// the contexts of SMALL_WD + 1 .. NARROW_WD words.
static_assert(DEFAULT_SMALL_REGION_BYTES / 4 >= 32 * SMALL_WD * row_stride(SMALL_WD) + CTL_WORDS + FL_WORDS,
              "a warp region holds the basis of any small-width context");

//
// NW: warps of a CTA.  The 4..9-word kernel has an instance of four-warp CTAs
// (four per SM, the same warps per SM) for long calls: a CTA-owned context's
// insertions run one warp at a time while the group's other warps wait, so
// smaller groups waste less; in a short call the longest CTA-owned contexts
// bound the call and keep eight warps each.
template <bool SMALL, int NW = LEARN_WARPS>
__global__ void __launch_bounds__(NW * 32, SMALL ? 3 : 16 / NW) elim_narrow_kernel(StoreDev s, LearnArgs a)
{
    constexpr int C_CTA = SMALL ? CLS_CTA_S : CLS_CTA;
    constexpr int C_WARP = SMALL ? CLS_WARP_S : CLS_WARP;
    extern __shared__ __align__(16) uint32_t smem[];
    __shared__ int s_item;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_cta = a.counters[CNT_COUNT + C_CTA];
    const int b_cta = a.counters[CNT_BEGIN + C_CTA];
    for (;;) {
        __syncthreads();
        if (threadIdx.x == 0) s_item = atomicAdd(a.counters + CNT_HEAD + C_CTA, 1);
        __syncthreads();
        const int item = s_item;
        if (item >= n_cta) break;
        const int c = a.queue[b_cta + item];
        const int wd = s.desc[c].wd;
        if (threadIdx.x == 0) time_mark(a.timing, c, 2);
#define F2_CALL_CTA(W) elim_ctx<W, true>(s, a, c, smem, a.cta_region_words)
        if (SMALL) {
            F2_SMALL_SWITCH(wd, F2_CALL_CTA)
        } else {
            F2_BIG_SWITCH(wd, F2_CALL_CTA)
        }
#undef F2_CALL_CTA
        if (threadIdx.x == 0) time_mark(a.timing, c, 3);
    }
    const int n_w = a.counters[CNT_COUNT + C_WARP];
    const int b_w = a.counters[CNT_BEGIN + C_WARP];
    const int region_words = SMALL ? a.small_region_words : a.warp_region_words;
    uint32_t* region = smem + warp * region_words;
    for (;;) {
        int item = 0;
        if (lane == 0) item = atomicAdd(a.counters + CNT_HEAD + C_WARP, 1);
        item = __shfl_sync(FULL, item, 0);
        if (item >= n_w) break;
        const int c = a.queue[b_w + item];
        const int wd = s.desc[c].wd;
        if (lane == 0) time_mark(a.timing, c, 2);
#define F2_CALL_WARP(W) elim_ctx<W, false>(s, a, c, region, region_words)
        if (SMALL) {
            F2_SMALL_SWITCH(wd, F2_CALL_WARP)
        } else {
            F2_BIG_SWITCH(wd, F2_CALL_WARP)
        }
#undef F2_CALL_WARP
        if (lane == 0) time_mark(a.timing, c, 3);
    }
}


// Wide elimination: every context by a whole CTA, rows of up to WDT words.
template <int WDT, int CLS>
__global__ void __launch_bounds__(WIDE_WARPS * 32, WDT <= WIDE_M_WD ? 2 : 1) elim_wide_kernel(StoreDev s, LearnArgs a)
{
    extern __shared__ __align__(16) uint32_t smem[];
    __shared__ int s_item;
    const int n = a.counters[CNT_COUNT + CLS];
    const int b = a.counters[CNT_BEGIN + CLS];
    for (;;) {
        __syncthreads();
        if (threadIdx.x == 0) s_item = atomicAdd(a.counters + CNT_HEAD + CLS, 1);
        __syncthreads();
        const int item = s_item;
        if (item >= n) break;
        const int c = a.queue[b + item];
        if (threadIdx.x == 0) time_mark(a.timing, c, 2);
        elim_ctx<WDT, true>(s, a, c, smem, a.cta_region_words);
        if (threadIdx.x == 0) time_mark(a.timing, c, 3);
    }
}

// Validate the batch and order the work longest-first, in three kernels:
// per-context keys and a histogram (grid), the bucket offsets (one block),
// and the scatter into the queue (grid).  A key is (class, work bucket,
// width); within a class, buckets run from the most work to the least and,
// inside a bucket, widths in increasing order (so few template variants run
// at once).
//   mode 0 (dedup plan): every valid non-empty context with at most DD_XW
//     feature words goes to the warp, quad or CTA dedup queue by its row
//     count; rep_count[c] becomes 0 (filled by the dedup pass), -1 (invalid,
//     skipped) or -(T+2) (every row is its own representative);
//   mode 1 (elimination plan): contexts with rows to eliminate go to the
//     warp, CTA or wide elimination queue.
constexpr int PLAN_SUB = PLAN_BUCKETS * NARROW_WD;  // (bucket, width) keys per class
constexpr int PLAN_KEYS = NUM_CLASSES * PLAN_SUB;
static_assert(PLAN_KEYS <= PLAN_HIST_WORDS, "the plan histogram holds every key");

struct PlanArgs {
    const int64_t* row_off;
    const int64_t* x_off;
    int64_t total_rows;
    int64_t total_xw;
    int32_t* rep_count;
    int mode;
    int warp_region_words;
    int64_t heavy_rows;
    int64_t warp_work;
    int scale;     // mode 1: scale heavy_rows / warp_work to the totals of the duplicate pass
    int num_sms;
    long long shard_work;  // mode 0: rows x (xw + 4) of one shard share; 0 = no splitting
    int max_shards;        // mode 0: most shards of one context
    int shard_cap;         // mode 0: queue slots for shard items beyond one per context
    int32_t* queue;
    int32_t* keybuf;
    int* hist;     // PLAN_KEYS counts (zeroed before plan_key_kernel), then cursors
    int hist_zeroed;  // hist is zero already (else launch_plan clears it)
    int* counters;
};

// Ownership thresholds of the elimination plan, scaled to the call's work
// when the duplicate pass has measured it: a warp-owned context must not run
// (dependent round after round) much longer than the whole call.
struct PlanLimits {
    long long heavy_rows, warp_work;
};
__device__ __forceinline__ PlanLimits plan_limits(const PlanArgs& p)
{
    PlanLimits L{p.heavy_rows, p.warp_work};
    if (p.mode == 1 && p.scale) {
        const unsigned long long tw = *reinterpret_cast<const unsigned long long*>(p.counters + CNT_WORK);
        const unsigned long long tr = *reinterpret_cast<const unsigned long long*>(p.counters + CNT_REPS);
        const long long hr = (long long)(tr / ((unsigned long long)p.num_sms * HEAVY_REPS_DIV));
        const long long ww = (long long)(tw / ((unsigned long long)p.num_sms * WARP_WORK_DIV));
        L.heavy_rows = hr < HEAVY_ROWS_MIN ? HEAVY_ROWS_MIN : (hr > L.heavy_rows ? L.heavy_rows : hr);
        L.warp_work = ww < WARP_WORK_MIN ? WARP_WORK_MIN : (ww > L.warp_work ? L.warp_work : ww);
    }
    return L;
}

// Validates context c's part of the batch and returns its key (bits 0..15:
// class, work bucket and width; bits 16..18: shards - 1), or -1 when it has
// no work; nsh_out = its queue items.
__device__ __forceinline__ int plan_key_of(const StoreDev& s, const PlanArgs& p, const PlanLimits& L, int c,
                                           int& nsh_out)
{
    nsh_out = 0;
    const CtxDesc cd = s.desc[c];
    int64_t R;
    if (p.mode == 1 && p.rep_count) {
        R = p.rep_count[c];
        if (R <= -2) R = -(R + 2);
    } else {
        const int64_t a0 = p.row_off[c], a1 = p.row_off[c + 1];
        const int64_t rows = a1 - a0;
        const int64_t x0 = p.x_off[c];
        const bool ok = a0 >= 0 && rows >= 0 && rows < (1ll << 31) && a1 <= p.total_rows && x0 >= 0 &&
                        rows <= p.total_xw && x0 + rows * cd.xw <= p.total_xw;
        if (!ok) record_status(s.status, F2_ERR_ROWS);
        R = ok ? rows : -1;
        if (p.mode == 0 && p.rep_count) {
            // wide rows are not deduplicated; rows of a full-rank context
            // are checked one by one (verify_full_kernel)
            if (R > 0 && (cd.xw > DD_XW_WIDE || s.rank[c] == cd.d)) {
                p.rep_count[c] = (int32_t)(-(R + 2));
                R = 0;
            } else {
                p.rep_count[c] = (R > 0) ? 0 : (int32_t)R;
            }
        }
    }
    int key = -1;
    if (R > 0) {
        int cls;
        unsigned long long work;
        if (p.mode == 0) {
            cls = (R <= DD_WARP_MAX_ROWS) ? CLS_DD_WARP : (R <= DD_QUAD_MAX_ROWS ? CLS_DD_QUAD : CLS_DD_CTA);
            if (cd.xw > DD_XW) cls += CLS_DDW_CTA - CLS_DD_CTA;  // the 10..16-word instance
            work = (unsigned long long)R * (unsigned long long)(cd.xw + 4);
        } else {
            const bool heavy = elim_words(cd.d, cd.wd) > p.warp_region_words || R >= L.heavy_rows ||
                               R * cd.d > L.warp_work;
            if (s.rank[c] == cd.d) cls = CLS_FULL;
            else if (cd.wd > NARROW_WD) cls = (cd.wd <= WIDE_M_WD) ? CLS_WIDE_M : CLS_WIDE;
            else if (cd.wd <= SMALL_WD) cls = heavy ? CLS_CTA_S : CLS_WARP_S;
            else cls = heavy ? CLS_CTA : CLS_WARP;
            work = (unsigned long long)R * (unsigned long long)(cd.wd + 4) * (unsigned long long)cd.d;
        }
        int nsh = 1;
        if (p.mode == 0 && p.shard_work > 0) {
            if (F2_DD_QUAD_PROMOTE && (cls == CLS_DD_QUAD || cls == CLS_DDW_QUAD) && R >= DD_PROMOTE_MIN_ROWS &&
                (long long)work * DD_QUAD_SHARE > p.shard_work)
                cls += CLS_DD_CTA - CLS_DD_QUAD;
            if (cls == CLS_DD_CTA || cls == CLS_DDW_CTA) {
                long long k = (long long)work / p.shard_work;
                if (DD_SHARD_ROWS > 0 && (R + DD_SHARD_ROWS - 1) / DD_SHARD_ROWS > k)
                    k = (R + DD_SHARD_ROWS - 1) / DD_SHARD_ROWS;
                if (k > R / DD_SHARD_MIN_ROWS) k = R / DD_SHARD_MIN_ROWS;
                nsh = k < 1 ? 1 : (k > p.max_shards ? p.max_shards : (int)k);
                // the queue holds shard_cap extra items; past that, contexts stay whole
                if (nsh > 1 && atomicAdd(p.counters + CNT_SHARDS, nsh - 1) + (nsh - 1) > p.shard_cap) nsh = 1;
                work /= (unsigned long long)nsh;
            }
        }
        int bucket = 63 - __clzll(work);
        if (bucket >= PLAN_BUCKETS) bucket = PLAN_BUCKETS - 1;
        const int width = (p.mode == 0 ? cd.xw : cd.wd);
        const int sub = (PLAN_BUCKETS - 1 - bucket) * NARROW_WD + (width > NARROW_WD ? NARROW_WD : width) - 1;
        key = cls * PLAN_SUB + sub;
        key |= (nsh - 1) << 16;
        nsh_out = nsh;
    }
    return key;
}

__global__ void __launch_bounds__(256) plan_key_kernel(StoreDev s, PlanArgs p)
{
    __shared__ int hist[PLAN_KEYS];
    for (int i = threadIdx.x; i < PLAN_KEYS; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    const PlanLimits L = plan_limits(p);
    for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < s.num_ctx; c += gridDim.x * blockDim.x) {
        int nsh;
        const int kv = plan_key_of(s, p, L, c, nsh);
        if (kv >= 0) atomicAdd(&hist[kv & 0xFFFF], nsh);
        p.keybuf[c] = kv;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < PLAN_KEYS; i += blockDim.x)
        if (hist[i]) atomicAdd(p.hist + i, hist[i]);
}

// Exclusive scan of the key counts `hist` (global or shared) in key order by
// one block of 1024 threads; hist becomes the cursors and the class blocks of
// `counters` (first item, count, head) are set.
__device__ void plan_scan_block(int* hist, int* counters)
{
    constexpr int PER = (PLAN_KEYS + 1023) / 1024;
    __shared__ int wsum[32];
    __shared__ int s_total;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    int v[PER];
    int tot = 0;
#pragma unroll
    for (int j = 0; j < PER; ++j) {
        const int k = t * PER + j;
        v[j] = (k < PLAN_KEYS) ? hist[k] : 0;
        tot += v[j];
    }
    int inc = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(FULL, inc, o);
        if (lane >= o) inc += u;
    }
    if (lane == 31) wsum[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        int w = wsum[lane];
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int u = __shfl_up_sync(FULL, wi, o);
            if (lane >= o) wi += u;
        }
        wsum[lane] = wi - w;
        if (lane == 31) s_total = wi;
    }
    __syncthreads();
    int run = wsum[warp] + inc - tot;
#pragma unroll
    for (int j = 0; j < PER; ++j) {
        const int k = t * PER + j;
        if (k < PLAN_KEYS) hist[k] = run;  // becomes the cursor of key k
        run += v[j];
    }
    __syncthreads();
    // a class's items run from the cursor of its first key to that of the next class
    if (t < NUM_CLASSES) {
        const int b = hist[t * PLAN_SUB];
        const int e = (t + 1 < NUM_CLASSES) ? hist[(t + 1) * PLAN_SUB] : s_total;
        counters[CNT_BEGIN + t] = b;
        counters[CNT_HEAD + t] = 0;
        counters[CNT_COUNT + t] = e - b;
    }
}

__global__ void __launch_bounds__(1024) plan_scan_kernel(PlanArgs p) { plan_scan_block(p.hist, p.counters); }

// Queue item(s) of context c with key kv at the cursor of its key.
__device__ __forceinline__ void plan_place(const PlanArgs& p, int* cursor, int c, int kv)
{
    const int key = kv & 0xFFFF, nsh = (kv >> 16) + 1;
    if (nsh == 1) {
        p.queue[atomicAdd(cursor + key, 1)] = c;
    } else {  // one item per shard
        const int q0 = atomicAdd(cursor + key, nsh);
        for (int k = 0; k < nsh; ++k)
            p.queue[q0 + k] = (int32_t)((uint32_t)c | ((uint32_t)k << 24) | ((uint32_t)(nsh - 1) << 28));
    }
}

__global__ void __launch_bounds__(256) plan_scatter_kernel(StoreDev s, PlanArgs p)
{
    // the lanes of a warp with the same key take their slots with one atomic
    const int lane = threadIdx.x & 31;
    for (int b = blockIdx.x * blockDim.x; b < s.num_ctx; b += gridDim.x * blockDim.x) {
        const int c = b + (int)threadIdx.x;
        const int kv = (c < s.num_ctx) ? p.keybuf[c] : -1;
        const bool single = kv >= 0 && (kv >> 16) == 0;
        const int key = single ? kv : -1 - lane;  // a lane of its own unless a single item
        const unsigned peers = __match_any_sync(FULL, key);
        if (single) {
            const int leader = __ffs(peers) - 1;
            int q0 = 0;
            if (lane == leader) q0 = atomicAdd(p.hist + key, __popc(peers));
            q0 = __shfl_sync(peers, q0, leader);
            p.queue[q0 + __popc(peers & ((1u << lane) - 1u))] = c;
        } else if (kv >= 0) {
            plan_place(p, p.hist, c, kv);
        }
    }
}

// The three steps in one block, the histogram in shared memory, for stores
// of at most PLAN_SMALL_MAX contexts (one launch instead of a memset and
// three kernels: what a small batch waits for).
constexpr int PLAN_SMALL_MAX = 8192;
__global__ void __launch_bounds__(1024) plan_small_kernel(StoreDev s, PlanArgs p)
{
    __shared__ int hist[PLAN_KEYS];
    for (int i = threadIdx.x; i < PLAN_KEYS; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    const PlanLimits L = plan_limits(p);
    for (int c = threadIdx.x; c < s.num_ctx; c += blockDim.x) {
        int nsh;
        const int kv = plan_key_of(s, p, L, c, nsh);
        if (kv >= 0) atomicAdd(&hist[kv & 0xFFFF], nsh);
        p.keybuf[c] = kv;  // read back below by this same thread
    }
    __syncthreads();
    plan_scan_block(hist, p.counters);
    __syncthreads();
    for (int c = threadIdx.x; c < s.num_ctx; c += blockDim.x) {
        const int kv = p.keybuf[c];
        if (kv >= 0) plan_place(p, hist, c, kv);
    }
}

int launch_plan(const StoreDev& sd, const PlanArgs& pa, int num_sms, cudaStream_t cs)
{
    if (sd.num_ctx <= PLAN_SMALL_MAX) {
        plan_small_kernel<<<1, 1024, 0, cs>>>(sd, pa);
        return f2_cuda_status(cudaGetLastError());
    }
    if (!pa.hist_zeroed) {
        const cudaError_t e = cudaMemsetAsync(pa.hist, 0, sizeof(int) * PLAN_KEYS, cs);
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    int blocks = (sd.num_ctx + 255) / 256;
    if (blocks > num_sms * 2) blocks = num_sms * 2;
    if (blocks < 1) blocks = 1;
    plan_key_kernel<<<blocks, 256, 0, cs>>>(sd, pa);
    plan_scan_kernel<<<1, 1024, 0, cs>>>(pa);
    plan_scatter_kernel<<<blocks, 256, 0, cs>>>(sd, pa);
    return f2_cuda_status(cudaGetLastError());
}

inline bool is_aligned(const void* p, size_t al) { return ((uintptr_t)p % al) == 0; }

// ---------------------------------------------------------------------------
// Full-rank contexts.  When rank = d at the start of a call the reduced basis
// is the identity (every coordinate is a pivot and a reduced row has no other
// pivot bit), so every row lies in the span and T(q) = XOR of z_k over the set
// coordinates k of q.  A row is redundant if its word equals T(phi(x)) and a
// contradiction otherwise (Sec. 2.2 steps (2)-(3)); nothing is inserted, so
// the rows are independent.  CTAs claim chunks of FULL_CHUNK rows of a
// context, look T up in a 4-bit table of the z_k in shared memory (built when
// a CTA moves to a context: entry 16p + v = XOR of z_{4p+b} over the bits b
// of v), and the last chunk of a context commits the contradiction count,
// the first contradicting row and rows_seen.
// ---------------------------------------------------------------------------
constexpr int FULL_STAGE = FULL_THREADS;  // rows staged in shared memory at a time (one per thread)
// The table: low and high halves of the 16 entries of each group of four
// coordinates in two planes of 8-byte entries (a warp's lookups at one group
// fall in distinct banks), groups padded with zero entries to a multiple of
// eight (one 32-bit word of q = eight lookups, no bounds test), the high
// plane at a fixed distance from the low one and the base 1024-byte aligned,
// so that an entry's address is the word's base OR the nibble times eight,
// with the group and the plane in the loads' immediate offsets.
constexpr int FULL_NP_MAX = 8 * ((MAX_D + 31) / 32);      // 264 groups
constexpr int FULL_ZH_BYTES = FULL_NP_MAX * 16 * 8;        // 33,792: low plane, then the high plane
constexpr int FULL_TABLE_WORDS = 2 * FULL_ZH_BYTES / 4 + 256;  // both planes + alignment slack

struct FullArgs {
    const int64_t* row_off;
    const int64_t* x_off;
    const uint32_t* x;
    const uint4* y;
    const int32_t* queue;
    const int* counters;
    int* ctr;                         // [2C]: chunks claimed, chunks done
    const int* late_count;            // contexts listed by the elimination kernels
    const int32_t* late_list;
    const int32_t* late_start;        // their first row left
    unsigned long long* cnt;          // [C] contradicting rows of the call
    unsigned long long* first;        // [C] first contradicting row of the call (all ones: none)
    int table_words;                  // FULL_TABLE_WORDS
};

__global__ void __launch_bounds__(FULL_THREADS) verify_full_kernel(StoreDev s, FullArgs a)
{
    extern __shared__ uint4 full_smem[];
    // the table at the first 1024-byte boundary of the dynamic shared memory
    const uint32_t pad = ((1024u - (smem_addr(full_smem) & 1023u)) & 1023u) / 4u;
    uint32_t* const tabw = reinterpret_cast<uint32_t*>(full_smem) + pad;
    uint32_t* const stage = reinterpret_cast<uint32_t*>(full_smem) + a.table_words;
    __shared__ int s_q, s_k;
    __shared__ unsigned long long s_cnt, s_first;
    const int t = threadIdx.x, lane = t & 31;
    const int nfull = a.counters[CNT_COUNT + CLS_FULL];
    const int qb = a.counters[CNT_BEGIN + CLS_FULL];
    const int nq = nfull + *a.late_count;  // full at the start of the call, then full mid-call
    auto ctx_of = [&](int qq) { return qq < nfull ? a.queue[qb + qq] : a.late_list[qq - nfull]; };
    auto start_of = [&](int qq, int c) { return qq < nfull ? (int64_t)0 : (int64_t)a.late_start[c]; };
    int q = 0, built = -1;
    for (;;) {
        if (t == 0) {
            int k = 0;
            while (q < nq) {
                const int c = ctx_of(q);
                const int64_t T = a.row_off[c + 1] - a.row_off[c] - start_of(q, c);
                k = atomicAdd(a.ctr + c, 1);
                if ((int64_t)k * FULL_CHUNK < T) break;
                ++q;
            }
            s_q = q;
            s_k = k;
            s_cnt = 0ull;
            s_first = ~0ull;
        }
        __syncthreads();
        q = s_q;
        if (q >= nq) break;
        const int k = s_k;
        const int c = ctx_of(q);
        const int64_t i_first = start_of(q, c);
        const CtxDesc cd = s.desc[c];
        const int np = (cd.d + 3) >> 2;
        const int nw = (np + 7) >> 3;  // words of q, eight groups each
        uint2* Zl = reinterpret_cast<uint2*>(tabw);
        uint2* Zh = Zl + FULL_ZH_BYTES / 8;
        if (built != c) {
            for (int j = t; j < 4 * np; j += FULL_THREADS) {
                const uint4 z = (j < cd.d) ? __ldg(s.bz + cd.slot_off + j) : make_uint4(0, 0, 0, 0);
                const int e = (j >> 2) * 16 + (1 << (j & 3));
                Zl[e] = make_uint2(z.x, z.y);
                Zh[e] = make_uint2(z.z, z.w);
                if ((j & 3) == 0) {
                    Zl[e - 1] = make_uint2(0, 0);
                    Zh[e - 1] = make_uint2(0, 0);
                }
            }
            __syncthreads();
            for (int f = t; f < 16 * np; f += FULL_THREADS) {
                const int v = f & 15;
                if (__popc(v) < 2) continue;
                const int eb = f & ~15;
                uint2 lo = make_uint2(0, 0), hi = make_uint2(0, 0);
#pragma unroll
                for (int bb = 0; bb < 4; ++bb) {
                    if ((v >> bb) & 1) {
                        const uint2 l = Zl[eb + (1 << bb)], h = Zh[eb + (1 << bb)];
                        lo.x ^= l.x;
                        lo.y ^= l.y;
                        hi.x ^= h.x;
                        hi.y ^= h.y;
                    }
                }
                Zl[f] = lo;
                Zh[f] = hi;
            }
            for (int f = 16 * np + t; f < 128 * nw; f += FULL_THREADS) {  // padding groups
                Zl[f] = make_uint2(0, 0);
                Zh[f] = make_uint2(0, 0);
            }
            built = c;
        }
        const int64_t r0 = a.row_off[c];
        const int64_t T = a.row_off[c + 1] - r0;
        const int64_t i0 = i_first + (int64_t)k * FULL_CHUNK;
        const int64_t i1 = (i0 + FULL_CHUNK < T) ? i0 + FULL_CHUNK : T;
        const uint32_t* xc = a.x + a.x_off[c];
        const int xw = cd.xw;
        const int sst = xw | 1;  // odd staging stride: a row per lane reads distinct banks
        const uint32_t lm = (cd.n & 31) ? (1u << (cd.n & 31)) - 1u : 0xFFFFFFFFu;
        unsigned long long cnt = 0ull, first = ~0ull;
        for (int64_t b0 = i0; b0 < i1; b0 += FULL_STAGE) {
            const int nb = (int)((i1 - b0) < FULL_STAGE ? (i1 - b0) : FULL_STAGE);
            __syncthreads();  // the table is complete / the previous rows are consumed
            const uint32_t* src = xc + b0 * xw;  // the rows are contiguous
            {
                // word w = r * xw + v of the block, stepped by FULL_THREADS
                // without a division per word
                int r = t / xw, v = t - (t / xw) * xw;
                const int dr = FULL_THREADS / xw, dv = FULL_THREADS - dr * xw;
                for (int w = t; w < nb * xw; w += FULL_THREADS) {
                    stage[r * sst + v] = __ldg(src + w);
                    r += dr;
                    v += dv;
                    if (v >= xw) {
                        v -= xw;
                        ++r;
                    }
                }
            }
            __syncthreads();
            if (t < nb) {
                const int64_t i = b0 + t;
                const uint4 yi = __ldg(a.y + r0 + i);
                const uint32_t* xr = stage + t * sst;
                uint32_t a0 = 0, a1 = 0, a2 = 0, a3 = 0, prev = 0;
                const char* const zt = reinterpret_cast<const char*>(tabw);
                for (int w = 0; w < nw; ++w) {
                    uint32_t xv = (w < xw) ? xr[w] : 0u;
                    if (w == xw - 1) xv &= lm;
                    uint32_t qw;
                    if (s.raw) {
                        qw = xv;
                    } else {  // phi(x) = [1 || x]: the constant at index 0, x bit j at 1 + j
                        qw = (xv << 1) | (prev >> 31) | (w == 0 ? 1u : 0u);
                        prev = xv;
                    }
                    const char* const zb = zt + w * 1024;
                    // two lookups a step: entry byte offset = nibble * 8
#pragma unroll
                    for (int h = 0; h < 8; h += 2) {
                        const uint32_t oa = (h == 0) ? ((qw << 3) & 0x78u) : ((qw >> (4 * h - 3)) & 0x78u);
                        const uint32_t ob = (qw >> (4 * h + 1)) & 0x78u;
                        const uint2 la = *reinterpret_cast<const uint2*>(zb + oa + 128 * h);
                        const uint2 ha = *reinterpret_cast<const uint2*>(zb + oa + FULL_ZH_BYTES + 128 * h);
                        const uint2 lb = *reinterpret_cast<const uint2*>(zb + ob + 128 * (h + 1));
                        const uint2 hb = *reinterpret_cast<const uint2*>(zb + ob + FULL_ZH_BYTES + 128 * (h + 1));
                        a0 ^= la.x ^ lb.x;
                        a1 ^= la.y ^ lb.y;
                        a2 ^= ha.x ^ hb.x;
                        a3 ^= ha.y ^ hb.y;
                    }
                }
                if (a0 != yi.x || a1 != yi.y || a2 != yi.z || a3 != yi.w) {
                    ++cnt;
                    if ((unsigned long long)i < first) first = (unsigned long long)i;
                }
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            cnt += __shfl_xor_sync(FULL, cnt, o);
            const unsigned long long f2 = __shfl_xor_sync(FULL, first, o);
            first = f2 < first ? f2 : first;
        }
        if (lane == 0 && cnt) {
            atomicAdd(&s_cnt, cnt);
            atomicMin(&s_first, first);
        }
        __syncthreads();
        if (t == 0) {
            if (s_cnt) {
                atomicAdd(a.cnt + c, s_cnt);
                atomicMin(a.first + c, s_first);
            }
            __threadfence();
            const int nch = (int)((T - i_first + FULL_CHUNK - 1) / FULL_CHUNK);
            if (atomicAdd(a.ctr + s.num_ctx + c, 1) == nch - 1) {  // the context's last chunk
                __threadfence();
                const unsigned long long tot = atomicAdd(a.cnt + c, 0ull);
                const unsigned long long fi = atomicMin(a.first + c, ~0ull);
                const long long seen = s.rows_seen[c];
                if (tot) {
                    s.n_contra[c] += tot;
                    s.contra[c] = 1;
                    if (s.first_contra[c] < 0) s.first_contra[c] = seen + (long long)fi;
                }
                s.rows_seen[c] = seen + T;
            }
        }
        __syncthreads();
    }
}

// The contexts the check sent back: eliminated in stream order from their
// first representative outside the snapshot (no further hand-off), one CTA
// each.  Every width that can hand off has an instance here.
__global__ void __launch_bounds__(LEARN_WARPS * 32, 1) resume_kernel(StoreDev s, LearnArgs a, const int* resume_count,
                                                                     const int32_t* resume_list)
{
    extern __shared__ __align__(16) uint32_t smem[];
    __shared__ int s_item;
    const int n = *resume_count;
    for (;;) {
        __syncthreads();
        if (threadIdx.x == 0) s_item = atomicAdd(a.counters + CNT_HEAD + CLS_RESUME, 1);
        __syncthreads();
        const int item = s_item;
        if (item >= n) break;
        const int c = resume_list[item];
        const int wd = s.desc[c].wd;
#define F2_CALL_RESUME(W) elim_ctx<W, true>(s, a, c, smem, a.cta_region_words)
        switch (wd) {
        case 1: F2_CALL_RESUME(1); break;
        case 2: F2_CALL_RESUME(2); break;
        case 3: F2_CALL_RESUME(3); break;
        case 4: F2_CALL_RESUME(4); break;
        case 5: F2_CALL_RESUME(5); break;
        case 6: F2_CALL_RESUME(6); break;
        case 7: F2_CALL_RESUME(7); break;
        case 8: F2_CALL_RESUME(8); break;
        case 9: F2_CALL_RESUME(9); break;
        default: F2_CALL_RESUME(WIDE_M_WD); break;
        }
#undef F2_CALL_RESUME
    }
}

// Which elimination kernels a store needs, and their widest bases.

size_t narrow_smem(int max_narrow_words, int warp_region_words, int nw)
{
    const size_t cta = 4 * (size_t)max_narrow_words;
    const size_t warps = 4 * (size_t)nw * (size_t)warp_region_words;
    return cta > warps ? cta : warps;
}

// Calls of at least this many rows run the 4..9-word elimination in CTAs of
// four warps (see elim_narrow_kernel; F2_OPT_LONG_CALL_ROWS).
constexpr int64_t LONG_CALL_ROWS = DEFAULT_LONG_CALL_ROWS;

// A second stream for kernels that work on disjoint contexts: the first
// such kernel goes to `aux` (forked from the caller's stream), the others to
// the caller's stream, and join() makes the caller's stream wait for `aux`.
struct Fork {
    cudaStream_t cs, aux;
    cudaEvent_t ev_fork, ev_join;
    bool forked = false;
    cudaError_t e = cudaSuccess;
    cudaStream_t next(int kernels_left)
    {
        if (!aux || forked || kernels_left < 2) return cs;
        e = cudaEventRecord(ev_fork, cs);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(aux, ev_fork, 0);
        if (e != cudaSuccess) return cs;
        forked = true;
        return aux;
    }
    cudaError_t join()
    {
        if (!forked || e != cudaSuccess) return e;
        forked = false;
        e = cudaEventRecord(ev_join, aux);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, ev_join, 0);
        return e;
    }
};

// Enqueue pass 2 (plan + kernels) for one batch.
int launch_elimination(const StoreDev& sd, const LearnArgs& la, const int64_t* row_off, const int64_t* x_off,
                       int64_t total_rows, int64_t total_xw, int32_t* rep_count, int64_t heavy_rows,
                       int64_t warp_work, int32_t* queue, int32_t* keybuf, int* hist, int num_sms,
                       const Widths& wv, int* full_ctr, unsigned long long* full_cnt,
                       unsigned long long* full_first, cudaStream_t cs, Fork* fk = nullptr, int scale = 0,
                       bool prezeroed = false, int64_t long_rows = LONG_CALL_ROWS, const CheckArgs* check = nullptr)
{
    // prezeroed: the caller has cleared full_ctr's first 2C words and late
    // count, full_cnt, full_first (to -1) and hist
    // full_ctr: chunks claimed [C], chunks done [C], late start [C], late list [C], late count
    const int C = sd.num_ctx;
    LearnArgs lx = la;
    lx.late_start = full_ctr + 2 * C;
    lx.late_list = full_ctr + 3 * C;
    lx.late_count = full_ctr + 4 * C;
    if (!prezeroed) {
        cudaError_t e0 = cudaMemsetAsync(full_ctr, 0, sizeof(int) * 2 * (size_t)C, cs);
        if (e0 == cudaSuccess) e0 = cudaMemsetAsync(lx.late_count, 0, sizeof(int), cs);
        if (e0 == cudaSuccess) e0 = cudaMemsetAsync(full_cnt, 0, sizeof(unsigned long long) * (size_t)C, cs);
        if (e0 == cudaSuccess) e0 = cudaMemsetAsync(full_first, 0xff, sizeof(unsigned long long) * (size_t)C, cs);
        if (e0 != cudaSuccess) return f2_cuda_status(e0);
    }
    PlanArgs pa;
    pa.row_off = row_off;
    pa.x_off = x_off;
    pa.total_rows = total_rows;
    pa.total_xw = total_xw;
    pa.rep_count = rep_count;
    pa.mode = 1;
    pa.warp_region_words = la.warp_region_words;
    pa.heavy_rows = heavy_rows;
    pa.warp_work = warp_work;
    pa.scale = scale;
    pa.num_sms = num_sms;
    pa.shard_work = 0;
    pa.max_shards = 1;
    pa.shard_cap = 0;
    pa.queue = queue;
    pa.keybuf = keybuf;
    pa.hist = hist;
    pa.hist_zeroed = prezeroed;
    pa.counters = la.counters;
    int rc = launch_plan(sd, pa, num_sms, cs);
    if (rc != F2_OK) return rc;
    cudaError_t e;
    auto narrow = [&](auto kernel, size_t smem, cudaStream_t ks, int nw) -> int {
        cudaError_t er = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (er != cudaSuccess) return f2_cuda_status(er);
        int per_sm = 0;
        er = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, nw * 32, smem);
        if (er != cudaSuccess) return f2_cuda_status(er);
        if (per_sm < 1) per_sm = 1;
        LearnArgs lk = lx;
        lk.cta_region_words = (int)(smem / 4);
        kernel<<<num_sms * per_sm, nw * 32, smem, ks>>>(sd, lk);
        return f2_cuda_status(cudaGetLastError());
    };
    // the three width classes hold disjoint contexts: with a second stream
    // their kernels overlap (each fills the others' tails)
    Fork solo{cs, nullptr, nullptr, nullptr};
    Fork& f = fk ? *fk : solo;
    int left = (int)wv.has_narrow + (int)wv.has_wide + (int)wv.has_wide_m + (int)wv.has_small;
    auto wide = [&](auto kernel, int max_d, int wdt) -> int {
        const size_t smem = 4 * (size_t)elim_words(max_d, wdt);
        cudaError_t er = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (er != cudaSuccess) return f2_cuda_status(er);
        int per_sm = 0;
        er = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, WIDE_WARPS * 32, smem);
        if (er != cudaSuccess) return f2_cuda_status(er);
        if (per_sm < 1) per_sm = 1;
        const cudaStream_t ks = f.next(left--);
        if (f.e != cudaSuccess) return f2_cuda_status(f.e);
        LearnArgs lk = lx;
        lk.cta_region_words = (int)(smem / 4);
        kernel<<<num_sms * per_sm, WIDE_WARPS * 32, smem, ks>>>(sd, lk);
        return f2_cuda_status(cudaGetLastError());
    };
    if (wv.has_wide) {
        rc = wide(elim_wide_kernel<WIDE_WD, CLS_WIDE>, wv.max_wide_d, WIDE_WD);
        if (rc != F2_OK) return rc;
    }
    if (wv.has_wide_m) {
        rc = wide(elim_wide_kernel<WIDE_M_WD, CLS_WIDE_M>, wv.max_wide_m_d, WIDE_M_WD);
        if (rc != F2_OK) return rc;
    }
    const size_t small_words = (size_t)LEARN_WARPS * (size_t)la.small_region_words;
    const size_t small_smem = 4 * (small_words > (size_t)wv.max_small_words ? small_words : (size_t)wv.max_small_words);
    if (wv.has_narrow) {
        const cudaStream_t ks = f.next(left--);
        if (f.e != cudaSuccess) return f2_cuda_status(f.e);
        if (total_rows >= long_rows)
            rc = narrow(elim_narrow_kernel<false, 4>, narrow_smem(wv.max_narrow_words, la.warp_region_words, 4), ks, 4);
        else
            rc = narrow(elim_narrow_kernel<false>, narrow_smem(wv.max_narrow_words, la.warp_region_words, LEARN_WARPS),
                        ks, LEARN_WARPS);
        if (rc != F2_OK) return rc;
    }
    if (wv.has_small) {
        const cudaStream_t ks = f.next(left--);
        if (f.e != cudaSuccess) return f2_cuda_status(f.e);
        rc = narrow(elim_narrow_kernel<true>, small_smem, ks, LEARN_WARPS);
        if (rc != F2_OK) return rc;
    }
    e = f.join();
    if (e != cudaSuccess) return f2_cuda_status(e);
    if (check && la.handoff_min > 0) {
        // the handed-off contexts: their remaining representatives checked
        // in parallel, then any that met a representative outside the
        // span eliminated from there on
        const size_t csmem = CHECK_SMEM_BYTES;
        e = cudaFuncSetAttribute(check_snap_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)csmem);
        if (e != cudaSuccess) return f2_cuda_status(e);
        check_snap_kernel<<<num_sms * 2, 256, csmem, cs>>>(sd, *check);
        e = cudaGetLastError();
        if (e != cudaSuccess) return f2_cuda_status(e);
        int words = wv.max_small_words > wv.max_narrow_words ? wv.max_small_words : wv.max_narrow_words;
        if (wv.has_wide_m && elim_words(wv.max_wide_m_d, WIDE_M_WD) > words)
            words = elim_words(wv.max_wide_m_d, WIDE_M_WD);
        const size_t rsmem = 4 * (size_t)words;
        e = cudaFuncSetAttribute(resume_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)rsmem);
        if (e != cudaSuccess) return f2_cuda_status(e);
        LearnArgs lr = lx;
        lr.handoff_min = 0;
        lr.resume_from = check->resume_from;
        lr.cta_region_words = words;
        resume_kernel<<<num_sms, LEARN_WARPS * 32, rsmem, cs>>>(sd, lr, check->resume_count, check->resume_list);
        e = cudaGetLastError();
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    {  // full-rank contexts: at the start of the call (the plan decides on the
       // device which, if any) or reached during it (listed by the kernels above)
        FullArgs fa;
        fa.row_off = row_off;
        fa.x_off = x_off;
        fa.x = la.x;
        fa.y = la.y;
        fa.queue = queue;
        fa.counters = la.counters;
        fa.ctr = full_ctr;
        fa.late_count = lx.late_count;
        fa.late_list = lx.late_list;
        fa.late_start = lx.late_start;
        fa.cnt = full_cnt;
        fa.first = full_first;
        fa.table_words = FULL_TABLE_WORDS;
        const size_t smem = 4 * ((size_t)fa.table_words + (size_t)FULL_STAGE * (size_t)(wv.max_xw | 1));
        e = cudaFuncSetAttribute(verify_full_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return f2_cuda_status(e);
        int per_sm = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, verify_full_kernel, FULL_THREADS, smem);
        if (e != cudaSuccess) return f2_cuda_status(e);
        if (per_sm < 1) per_sm = 1;
        verify_full_kernel<<<num_sms * per_sm, FULL_THREADS, smem, cs>>>(sd, fa);
        e = cudaGetLastError();
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    return F2_OK;
}

Widths width_summary(const int32_t* n_bits, int32_t num_ctx, bool raw)
{
    Widths w;
    for (int32_t c = 0; c < num_ctx; ++c) {
        const int d = raw ? n_bits[c] : n_bits[c] + 1;
        const int wd = (d + 31) / 32;
        const int words = elim_words(d, wd);
        if (d > w.max_d) w.max_d = d;
        if ((n_bits[c] + 31) / 32 > w.max_xw) w.max_xw = (n_bits[c] + 31) / 32;
        if (wd <= SMALL_WD) {
            w.has_small = true;
            if (words > w.max_small_words) w.max_small_words = words;
        } else if (wd <= NARROW_WD) {
            w.has_narrow = true;
            if (words > w.max_narrow_words) w.max_narrow_words = words;
        } else if (wd <= WIDE_M_WD) {
            w.has_wide_m = true;
            if (d > w.max_wide_m_d) w.max_wide_m_d = d;
        } else {
            w.has_wide = true;
            if (d > w.max_wide_d) w.max_wide_d = d;
        }
    }
    return w;
}

}  // namespace

extern "C" int f2_learn_batched(f2_store* st, const int64_t* row_off, const uint32_t* x, const int64_t* x_off,
                                const uint32_t* y, int64_t total_rows, int64_t total_x_words,
                                f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_learn_batched");
    if (!st || total_rows < 0 || total_x_words < 0) return F2_ERR_INVALID_ARG;
    if (st->num_ctx == 0) return F2_OK;
    if (!row_off || !x_off || (!x && total_x_words) || (!y && total_rows)) return F2_ERR_INVALID_ARG;
    if (!is_aligned(row_off, 8) || !is_aligned(x_off, 8) || !is_aligned(x, 4) || !is_aligned(y, 16))
        return F2_ERR_ALIGN;
    cudaStream_t cs = (cudaStream_t)stream;
    cudaError_t e;
    const bool dedup = st->dedup && total_rows > 0;
    if (dedup && total_rows > st->rep_capacity) {  // per-row scratch of pass 1, grown stream-ordered
        if (st->rep_list) cudaFreeAsync(st->rep_list, cs);
        if (st->rep_dup) cudaFreeAsync(st->rep_dup, cs);
        st->rep_list = st->rep_dup = nullptr;
        st->rep_capacity = 0;
        e = f2_dev_alloc(st, (void**)&st->rep_list, sizeof(int32_t) * (size_t)total_rows, cs, true);
        if (e == cudaSuccess) e = f2_dev_alloc(st, (void**)&st->rep_dup, sizeof(int32_t) * (size_t)total_rows, cs, true);
        if (e != cudaSuccess) return F2_ERR_OOM;
        st->rep_capacity = total_rows;
    }
    // every scratch counter of the call, zeroed by one launch
    const size_t C = (size_t)st->num_ctx;
    if (st->handoff_min > 0) {  // the check's chunk records, grown stream-ordered
        const int64_t slots = total_rows / CHECK_CHUNK + (int64_t)C + 1;
        if (slots > st->check_rec_cap) {
            if (st->check_rec) cudaFreeAsync(st->check_rec, cs);
            st->check_rec = nullptr;
            st->check_rec_cap = 0;
            if (f2_dev_alloc(st, (void**)&st->check_rec, 2 * sizeof(uint4) * (size_t)slots, cs, true) != cudaSuccess)
                return F2_ERR_OOM;
            st->check_rec_cap = slots;
        }
    }
    F2FillList zl;
    if (st->timing_on) {  // diagnostics: per-context timestamps of this call
        const size_t bytes = sizeof(unsigned long long) * TIME_WORDS * C;
        if (!st->timing && f2_dev_alloc(st, (void**)&st->timing, bytes, cs, true) != cudaSuccess) return F2_ERR_OOM;
        zl.add(st->timing, bytes);
    }
    {  // hand-off: the two list counts and the chunk counters
        zl.add(st->hand, sizeof(int) * 2);
        zl.add(st->hand + 2 + 4 * C, sizeof(int) * 2 * C);
    }
    if (dedup) {  // the work totals and the shard items of the duplicate pass
        zl.add(st->counters + CNT_WORK, (CNT_WORDS - CNT_WORK) * sizeof(int));
        zl.add(st->shard_done, sizeof(int32_t) * C);
    }
    zl.add(st->full_ctr, sizeof(int) * 2 * C);        // full-rank chunks claimed and done
    zl.add(st->full_ctr + 4 * C, sizeof(int));        // late count
    zl.add(st->full_cnt, sizeof(unsigned long long) * C);
    zl.add(st->full_first, sizeof(unsigned long long) * C, 0xff);
    if (st->num_ctx > PLAN_SMALL_MAX)  // the histograms of the two plans (one block keeps its own)
        zl.add(st->plan_hist, sizeof(int) * 2 * PLAN_HIST_WORDS);
    e = f2_fill(zl, cs);
    if (e != cudaSuccess) return f2_cuda_status(e);
    const StoreDev sd = st->dev();
    {
        const int rc = f2_ensure_aux(st);
        if (rc != F2_OK) return rc;
    }
    Fork fk{cs, st->aux, st->ev_fork, st->ev_join};
    if (dedup) {
        PlanArgs pa;
        pa.row_off = row_off;
        pa.x_off = x_off;
        pa.total_rows = total_rows;
        pa.total_xw = total_x_words;
        pa.rep_count = st->rep_count;
        pa.mode = 0;
        pa.warp_region_words = 0;
        pa.heavy_rows = 0;
        pa.warp_work = 0;
        pa.scale = 0;
        pa.num_sms = st->num_sms;
        // a shard share: the call's rows x (feature words + 4) over four per SM
        pa.max_shards = st->dd_shards;
        pa.shard_cap = f2_shard_queue_extra(st->num_sms);
        pa.shard_work = (st->num_ctx < SHARD_CTX_LIMIT && st->dd_shards > 1)
                            ? (total_x_words + 4 * total_rows) / (4 * (long long)st->num_sms) + 1
                            : 0;
        pa.queue = st->queue;
        pa.keybuf = st->keybuf;
        pa.hist = st->plan_hist;
        pa.hist_zeroed = 1;
        pa.counters = st->counters;
        int rc = launch_plan(sd, pa, st->num_sms, cs);
        if (rc != F2_OK) return rc;
        DedupArgs da;
        da.row_off = row_off;
        da.x_off = x_off;
        da.x = x;
        da.y = reinterpret_cast<const uint4*>(y);
        da.rep_list = st->rep_list;
        da.rep_dup = st->rep_dup;
        da.rep_count = st->rep_count;
        da.queue = st->queue;
        da.counters = st->counters;
        da.timing = st->timing_on ? st->timing : nullptr;
        da.shard_reps = st->shard_reps;
        da.shard_done = st->shard_done;
        // the two instances hold disjoint contexts: side by side when both run
        const bool wide_rows = st->max_xw > DD_XW;  // some context has feature rows of 10..16 words
        e = cudaFuncSetAttribute(dedup_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, DD_SMEM);
        if (e != cudaSuccess) return f2_cuda_status(e);
        cudaStream_t ks = fk.next(wide_rows ? 2 : 1);
        if (fk.e != cudaSuccess) return f2_cuda_status(fk.e);
        dedup_kernel<false><<<DD_CTAS_PER_SM * st->num_sms, DD_THREADS, DD_SMEM, ks>>>(sd, da);
        e = cudaGetLastError();
        if (e != cudaSuccess) return f2_cuda_status(e);
        if (wide_rows) {
            e = cudaFuncSetAttribute(dedup_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, DD_SMEM);
            if (e != cudaSuccess) return f2_cuda_status(e);
            dedup_kernel<true><<<DD_CTAS_PER_SM * st->num_sms, DD_THREADS, DD_SMEM, fk.next(1)>>>(sd, da);
            e = cudaGetLastError();
            if (e != cudaSuccess) return f2_cuda_status(e);
        }
        e = fk.join();
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    LearnArgs la;
    la.row_off = row_off;
    la.x_off = x_off;
    la.x = x;
    la.y = reinterpret_cast<const uint4*>(y);
    la.rep_list = dedup ? st->rep_list : nullptr;
    la.rep_dup = dedup ? st->rep_dup : nullptr;
    la.rep_count = dedup ? st->rep_count : nullptr;
    la.queue = st->queue;
    la.counters = st->counters;
    la.timing = st->timing_on ? st->timing : nullptr;
    la.warp_region_words = (int)(st->warp_basis_bytes / 4);
    la.tables = st->elim_tables;
    la.small_region_words = (int)(st->small_basis_bytes / 4);
    la.cta_region_words = 0;  // set per launch
    // hand-off of saturated contexts, in calls long enough to have some
    la.handoff_min = (st->handoff_min > 0 && total_rows >= HANDOFF_CALL_FACTOR * st->handoff_min)
                         ? (int)st->handoff_min : 0;
    la.snap_count = st->hand;
    la.snap_list = st->hand + 2;
    la.snap_start = st->hand + 2 + C;
    la.resume_from = nullptr;
    if (!st->widths_ready) {  // fixed by the widths: computed once per store
        st->widths = width_summary(st->n_bits.data(), st->num_ctx, (st->flags & F2_FLAG_RAW_FEATURES) != 0);
        st->widths_ready = true;
    }
    const Widths& wv = st->widths;
    // Rows from which a context gets a whole CTA: unless set explicitly, it
    // scales with the batch -- in a short call a warp-owned context of a few
    // thousand rows, dependent round after round, would outlast everything
    // else, while in a long one warps keep the SMs fuller
    // else, and in a store of at most ALL_CTA_PER_SM contexts per SM, every
    // context gets one: none waits for a CTA, and a CTA takes eight warps'
    // rows per dependent round
    int64_t heavy = st->heavy_rows;
    const bool all_cta = !st->heavy_rows_set && st->num_ctx <= (int64_t)ALL_CTA_PER_SM * st->num_sms;
    if (all_cta) {
        heavy = 1;
    } else if (!st->heavy_rows_set && !dedup) {
        heavy = total_rows / HEAVY_ROWS_BATCH_DIV;
        if (heavy < HEAVY_ROWS_MIN) heavy = HEAVY_ROWS_MIN;
        if (heavy > st->heavy_rows) heavy = st->heavy_rows;
    }
    const int scale = dedup && !all_cta && !st->heavy_rows_set && !st->warp_work_set;
    CheckArgs ca;
    ca.row_off = row_off;
    ca.x_off = x_off;
    ca.x = x;
    ca.y = reinterpret_cast<const uint4*>(y);
    ca.rep_list = la.rep_list;
    ca.rep_dup = la.rep_dup;
    ca.rep_count = la.rep_count;
    ca.snap_count = la.snap_count;
    ca.snap_list = la.snap_list;
    ca.snap_start = la.snap_start;
    ca.resume_count = st->hand + 1;
    ca.resume_list = st->hand + 2 + 2 * C;
    ca.resume_from = st->hand + 2 + 3 * C;
    ca.ctr = st->hand + 2 + 4 * C;
    ca.rec = st->check_rec;
    return launch_elimination(sd, la, row_off, x_off, total_rows, total_x_words, dedup ? st->rep_count : nullptr,
                              heavy, st->warp_work, st->queue, st->keybuf, st->plan_hist + PLAN_HIST_WORDS,
                              st->num_sms, wv, st->full_ctr, st->full_cnt, st->full_first, cs, &fk, scale, true,
                              st->long_call_rows, &ca);
}

extern "C" int f2_learn_timing(const f2_store* st, uint64_t* out_host, f2_stream_t stream)
{
    if (!st || !out_host) return F2_ERR_INVALID_ARG;
    if (!st->timing) return F2_ERR_INVALID_ARG;  // no learn call since F2_OPT_TIMING was set
    cudaStream_t cs = (cudaStream_t)stream;
    cudaError_t e = cudaMemcpyAsync(out_host, st->timing, sizeof(uint64_t) * TIME_WORDS * (size_t)st->num_ctx,
                                    cudaMemcpyDeviceToHost, cs);
    if (e == cudaSuccess) e = cudaStreamSynchronize(cs);
    return f2_cuda_status(e);
}

// ---------------------------------------------------------------------------
// Allocation-free variant of f2_learn_batched (no counterpart in the paper;
// see f2_learn_batched_noalloc in f2gpu.h).  The scheduling scratch that a
// store would own lives in one file-scope device array of fixed capacity.

#include <mutex>

namespace {

struct NoallocScratch {
    CtxDesc desc[F2_NOALLOC_MAX_CTX];
    int32_t n_bits[F2_NOALLOC_MAX_CTX];
    int32_t queue[F2_NOALLOC_MAX_CTX];
    int32_t keybuf[F2_NOALLOC_MAX_CTX];
    int counters[CNT_WORDS];
    int plan_hist[PLAN_KEYS];
    int full_ctr[4 * F2_NOALLOC_MAX_CTX + 1];
    unsigned long long full_cnt[F2_NOALLOC_MAX_CTX];
    unsigned long long full_first[F2_NOALLOC_MAX_CTX];
};

// Device storage for the scratch; in host code this name is only a symbol
// handle, its device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_noalloc_scratch[sizeof(NoallocScratch)];

constexpr int NOALLOC_MAX_DEVICES = 64;
constexpr int NOALLOC_HEAVY_ROWS = DEFAULT_HEAVY_ROWS;
constexpr int NOALLOC_WARP_REGION_WORDS = DEFAULT_WARP_REGION_BYTES / 4;

struct NoallocDevice {
    NoallocScratch* scratch;
    int num_sms;
    bool ready;
};
NoallocDevice g_noalloc_dev[NOALLOC_MAX_DEVICES];
std::mutex g_noalloc_mu;

// Context descriptors and canonical offsets (exclusive prefix sums of d,
// d*wd and wd) for up to F2_NOALLOC_MAX_CTX contexts, one block.
__global__ void __launch_bounds__(1024) noalloc_desc_kernel(const int32_t* __restrict__ n_bits, int C, uint32_t raw,
                                                            CtxDesc* __restrict__ desc)
{
    constexpr int PER = (F2_NOALLOC_MAX_CTX + 1023) / 1024;
    __shared__ long long wsum[3][32];
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    long long a = 0, b = 0, c = 0;
    for (int i = 0; i < PER; ++i) {
        const int k = t * PER + i;
        if (k < C) {
            const int n = n_bits[k];
            const int d = raw ? n : n + 1;
            const int wd = (d + 31) / 32;
            a += d;
            b += (long long)d * wd;
            c += wd;
        }
    }
    long long ia = a, ib = b, ic = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long va = __shfl_up_sync(FULL, ia, o), vb = __shfl_up_sync(FULL, ib, o),
                        vc = __shfl_up_sync(FULL, ic, o);
        if (lane >= o) {
            ia += va;
            ib += vb;
            ic += vc;
        }
    }
    if (lane == 31) {
        wsum[0][warp] = ia;
        wsum[1][warp] = ib;
        wsum[2][warp] = ic;
    }
    __syncthreads();
    if (warp == 0) {
        long long sa = wsum[0][lane], sb = wsum[1][lane], sc = wsum[2][lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const long long va = __shfl_up_sync(FULL, sa, o), vb = __shfl_up_sync(FULL, sb, o),
                            vc = __shfl_up_sync(FULL, sc, o);
            if (lane >= o) {
                sa += va;
                sb += vb;
                sc += vc;
            }
        }
        wsum[0][lane] = sa - wsum[0][lane];
        wsum[1][lane] = sb - wsum[1][lane];
        wsum[2][lane] = sc - wsum[2][lane];
    }
    __syncthreads();
    long long ea = wsum[0][warp] + ia - a, eb = wsum[1][warp] + ib - b, ec = wsum[2][warp] + ic - c;
    for (int i = 0; i < PER; ++i) {
        const int k = t * PER + i;
        if (k < C) {
            CtxDesc cd;
            cd.n = n_bits[k];
            cd.d = raw ? cd.n : cd.n + 1;
            cd.wd = (cd.d + 31) / 32;
            cd.xw = (cd.n + 31) / 32;
            cd.slot_off = ea;
            cd.xw_off = eb;
            cd.pw_off = ec;
            cd.pad = 0;
            desc[k] = cd;
            ea += cd.d;
            eb += (long long)cd.d * cd.wd;
            ec += cd.wd;
        }
    }
}

// Host copy of the caller's widths: the device copy is made from here, so the
// caller's array is free again when the call returns (a copy from pageable
// memory is staged before cudaMemcpyAsync returns).  Guarded by g_noalloc_mu.
int32_t g_noalloc_nbits[F2_NOALLOC_MAX_CTX];

// Every kernel the allocation-free path can launch.  Loading a kernel's code
// (on its first launch, under lazy module loading) may allocate device
// memory, so the first call on a device loads all of them.
cudaError_t noalloc_load_kernels()
{
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, noalloc_desc_kernel);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, plan_key_kernel);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, plan_scan_kernel);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, plan_scatter_kernel);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, plan_small_kernel);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, elim_narrow_kernel<true>);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, elim_narrow_kernel<false>);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, elim_narrow_kernel<false, 4>);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, elim_wide_kernel<WIDE_WD, CLS_WIDE>);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, elim_wide_kernel<WIDE_M_WD, CLS_WIDE_M>);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, verify_full_kernel);
    return e;
}

// Once per device (with that device current): resolve the scratch address
// and load the kernels.
int noalloc_setup(NoallocDevice** out)
{
    int device = -1;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return f2_cuda_status(e);
    if (device < 0 || device >= NOALLOC_MAX_DEVICES) return F2_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    NoallocDevice& d = g_noalloc_dev[device];
    if (!d.ready) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || p == nullptr) return e != cudaSuccess ? f2_cuda_status(e) : F2_ERR_CUDA;
        int sms = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
        if (e == cudaSuccess) e = noalloc_load_kernels();
        if (e != cudaSuccess) return f2_cuda_status(e);
        d.scratch = static_cast<NoallocScratch*>(p);
        d.num_sms = sms;
        d.ready = true;
    }
    *out = &d;
    return F2_OK;
}

}  // namespace

extern "C" int f2_learn_batched_noalloc(int32_t num_ctx, const int32_t* n_bits_host, uint32_t flags,
                                        int32_t* rank_dev, uint32_t* pivot_mask_dev, uint32_t* basis_x_dev,
                                        uint32_t* basis_z_dev, uint8_t* contra_dev, int64_t* first_contra_dev,
                                        uint64_t* n_contra_dev, int64_t* rows_seen_dev, int32_t* status_dev,
                                        const int64_t* row_off_dev, const uint32_t* x_dev, const int64_t* x_off_dev,
                                        const uint32_t* y_dev, int64_t total_rows, int64_t total_x_words,
                                        f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_learn_batched_noalloc");
    if (num_ctx < 0 || num_ctx > F2_NOALLOC_MAX_CTX || (flags & ~F2_FLAG_RAW_FEATURES) || total_rows < 0 ||
        total_x_words < 0 || !status_dev)
        return F2_ERR_INVALID_ARG;
    if (num_ctx == 0)  // nothing to learn: only the status word is written
        return f2_cuda_status(cudaMemsetAsync(status_dev, 0, sizeof(int32_t), (cudaStream_t)stream));
    if (!n_bits_host || !rank_dev || !pivot_mask_dev || !basis_x_dev || !basis_z_dev || !contra_dev ||
        !first_contra_dev || !n_contra_dev || !rows_seen_dev || !row_off_dev || !x_off_dev ||
        (!x_dev && total_x_words) || (!y_dev && total_rows))
        return F2_ERR_INVALID_ARG;
    if (!is_aligned(row_off_dev, 8) || !is_aligned(x_off_dev, 8) || !is_aligned(x_dev, 4) || !is_aligned(y_dev, 16) ||
        !is_aligned(basis_z_dev, 16) || !is_aligned(first_contra_dev, 8) || !is_aligned(n_contra_dev, 8) ||
        !is_aligned(rows_seen_dev, 8) || !is_aligned(rank_dev, 4) || !is_aligned(pivot_mask_dev, 4) ||
        !is_aligned(basis_x_dev, 4) || !is_aligned(status_dev, 4))
        return F2_ERR_ALIGN;
    const bool raw = (flags & F2_FLAG_RAW_FEATURES) != 0;
    for (int32_t c = 0; c < num_ctx; ++c)
        if (n_bits_host[c] < 1 || n_bits_host[c] > MAX_N) return F2_ERR_NBITS;
    NoallocDevice* nd = nullptr;
    int rc = noalloc_setup(&nd);
    if (rc != F2_OK) return rc;
    NoallocScratch* sc = nd->scratch;
    cudaStream_t cs = (cudaStream_t)stream;

    cudaError_t e = cudaMemsetAsync(status_dev, 0, sizeof(int32_t), cs);
    if (e == cudaSuccess) {
        std::lock_guard<std::mutex> lock(g_noalloc_mu);
        memcpy(g_noalloc_nbits, n_bits_host, sizeof(int32_t) * (size_t)num_ctx);
        e = cudaMemcpyAsync(sc->n_bits, g_noalloc_nbits, sizeof(int32_t) * (size_t)num_ctx, cudaMemcpyHostToDevice,
                            cs);
    }
    if (e != cudaSuccess) return f2_cuda_status(e);
    noalloc_desc_kernel<<<1, 1024, 0, cs>>>(sc->n_bits, num_ctx, raw ? 1u : 0u, sc->desc);

    StoreDev sd;
    sd.desc = sc->desc;
    sd.rank = rank_dev;
    sd.contra = contra_dev;
    sd.first_contra = reinterpret_cast<long long*>(first_contra_dev);
    sd.n_contra = reinterpret_cast<unsigned long long*>(n_contra_dev);
    sd.rows_seen = reinterpret_cast<long long*>(rows_seen_dev);
    sd.pivot = pivot_mask_dev;
    sd.bx = basis_x_dev;
    sd.bz = reinterpret_cast<uint4*>(basis_z_dev);
    sd.status = status_dev;
    sd.num_ctx = num_ctx;
    sd.raw = raw ? 1u : 0u;
    LearnArgs la;
    la.row_off = row_off_dev;
    la.x_off = x_off_dev;
    la.x = x_dev;
    la.y = reinterpret_cast<const uint4*>(y_dev);
    la.rep_list = nullptr;  // every row is its own representative: no per-row scratch
    la.rep_dup = nullptr;
    la.rep_count = nullptr;
    la.queue = sc->queue;
    la.counters = sc->counters;
    la.timing = nullptr;
    la.tables = 1;
    la.small_region_words = DEFAULT_SMALL_REGION_BYTES / 4;
    la.cta_region_words = 0;
    la.handoff_min = 0;
    la.snap_count = nullptr;
    la.snap_list = nullptr;
    la.snap_start = nullptr;
    la.resume_from = nullptr;
    la.warp_region_words = NOALLOC_WARP_REGION_WORDS;
    const Widths wv = width_summary(n_bits_host, num_ctx, raw);
    return launch_elimination(sd, la, row_off_dev, x_off_dev, total_rows, total_x_words, nullptr, NOALLOC_HEAVY_ROWS,
                              DEFAULT_WARP_WORK, sc->queue, sc->keybuf, sc->plan_hist, nd->num_sms, wv, sc->full_ctr,
                              sc->full_cnt, sc->full_first, cs);
}
