// Internal definitions shared by the CUDA translation units of libf2gpu.so.
#pragma once

#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>
#include <stdint.h>

#include <vector>

#include "f2gpu.h"

namespace f2 {

struct HostIO;  // copy streams, events and staging of the host-input entry points

// An NVTX range over one API call (visible in Nsight timelines; costs a
// function-pointer check when no tool is attached).
struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange&) = delete;
    NvtxRange& operator=(const NvtxRange&) = delete;
};
#define F2_NVTX_RANGE(name) ::f2::NvtxRange f2_nvtx_range_(name)

constexpr unsigned FULL = 0xffffffffu;
constexpr int MAX_N = 1024;          // feature bits per context
constexpr int MAX_D = MAX_N + 1;     // row width with the affine constant
constexpr int NARROW_WD = 9;         // widest row (32-bit words) handled by the narrow kernels
constexpr int LEARN_WARPS = 8;       // warps per CTA of the narrow learn kernel
constexpr int WIDE_WARPS = 8;        // warps per CTA of the wide learn kernel
constexpr int PLAN_BUCKETS = 48;     // log2(work) buckets for longest-first ordering
constexpr int DEFAULT_WARP_REGION_BYTES = 12288;  // shared memory of one warp-owned context
constexpr int DEFAULT_SMALL_REGION_BYTES = 4096;  // the same in the small-width kernel (d <= 96)
constexpr int64_t DEFAULT_ENCODE_DIRECT_MAX = 65536;  // encode passes this small skip the grouping
constexpr int64_t DEFAULT_LONG_CALL_ROWS = int64_t(1) << 25;  // learn calls this long: 4-warp CTAs (4..9 words)
constexpr int64_t DEFAULT_HANDOFF_REPS = 0;  // representatives left for a saturated context to hand off (0: never)
constexpr int DEFAULT_HEAVY_ROWS = 4096;          // rows from which a context gets a whole CTA (at most)
constexpr int HEAVY_ROWS_MIN = 1024;              // ... and at least, when it scales with the batch:
constexpr int HEAVY_ROWS_BATCH_DIV = 20000;       // batch rows / this (no duplicate pass), or
constexpr int HEAVY_REPS_DIV = 20;                // representatives / (SMs x this) after the duplicate pass
constexpr int ALL_CTA_PER_SM = 2;                 // stores of at most this many contexts per SM: a CTA each
constexpr long long WARP_WORK_MIN = 32768;        // scaled warp work (rows x d) stays within
constexpr int WARP_WORK_DIV = 45;                 // [this, the option]: sum(rows x d) / (SMs x this)
constexpr long long DEFAULT_WARP_WORK = 131072;   // largest rows x d handled by one warp

// Scheduling counters written by the plan kernel, read by the learn kernels.
enum Counter {
    CNT_HEAD = 0,   // + class: next queue item of each class
    CNT_BEGIN = 16, // + class: first queue slot of each class
    CNT_COUNT = 32, // + class: number of contexts of each class
    CNT_WORK = 48,  // (uint64) sum over contexts of representatives x d, from the duplicate pass
    CNT_REPS = 50,  // (uint64) sum of the representatives
    CNT_SHARDS = 52,  // shard items beyond one per context claimed by the duplicate-pass plan
    CNT_WORDS = 54
};
// Work classes: elimination by a CTA / the wide kernel / a warp, dedup by a
// CTA / a quad of warps / a warp, elimination of the small-width contexts
// (wd <= SMALL_WD, their own kernel) by a CTA / a warp, and the contexts of
// full rank at the start of a call (rows checked independently).
enum Class {
    CLS_CTA = 0,
    CLS_WIDE = 1,
    CLS_WARP = 2,
    CLS_DD_CTA = 3,
    CLS_DD_QUAD = 4,
    CLS_DD_WARP = 5,
    CLS_CTA_S = 6,
    CLS_WARP_S = 7,
    CLS_FULL = 8,
    CLS_DDW_CTA = 9,   // dedup of feature rows of 10..16 words (their own kernel)
    CLS_DDW_QUAD = 10,
    CLS_DDW_WARP = 11,
    CLS_WIDE_M = 12,   // elimination of rows of 10..17 words (a narrower instance of the wide kernel)
    CLS_RESUME = 13,   // handed-off contexts sent back by the check (their queue head only)
    NUM_CLASSES = 14
};
static_assert(NUM_CLASSES <= CNT_BEGIN - CNT_HEAD, "counter blocks hold one entry per class");
constexpr int SMALL_WD = 3;
constexpr int PLAN_HIST_WORDS = 8192;  // key histogram of the plan kernels (>= number of keys)  // contexts of d <= 96 bits: fewer registers, twice the warps per SM

// Shared-memory and kernel selection of the elimination launches: the widest
// rows of each width class of a store.
struct Widths {
    int max_small_words = 0, max_narrow_words = 0, max_wide_m_d = 0, max_wide_d = 0;
    int max_d = 0, max_xw = 0;  // over every context (any may reach full rank)
    bool has_small = false, has_narrow = false, has_wide_m = false, has_wide = false;
};

// Per-context descriptor (device copy built at store creation).
struct CtxDesc {
    int32_t n;        // feature bits as supplied
    int32_t d;        // row width (n + 1, or n for raw feature rows)
    int32_t wd;       // 32-bit words of a feature row: ceil(d / 32)
    int32_t xw;       // 32-bit words of a supplied feature vector: ceil(n / 32)
    int64_t slot_off; // first 128-bit slot (basis z, solve output)
    int64_t xw_off;   // first basis feature word (d * wd words)
    int64_t pw_off;   // first pivot-mask word (wd words)
    int64_t pad;
};

// Device view of a store.
struct StoreDev {
    const CtxDesc* desc;
    int32_t* rank;
    uint8_t* contra;
    long long* first_contra;
    unsigned long long* n_contra;
    long long* rows_seen;
    uint32_t* pivot;
    uint32_t* bx;
    uint4* bz;
    int* status;
    int32_t num_ctx;
    uint32_t raw;
};

// Shared-memory row stride (32-bit words) of a basis slot: the 128-bit z
// first, then the wd feature words, padded to 16 bytes.
__host__ __device__ constexpr int row_stride(int wd) { return 4 * ((4 + wd + 3) / 4); }

// ---------------------------------------------------------------------------
// Lookup tables of a reduced basis (a Four-Russians table over 4-bit groups
// of coordinates), used by the encoder and by the elimination.  Reducing q
// against the reduced basis XORs, for every set coordinate j of q, the vector
// E_j:
//   j a pivot:     word part z_j, residual part r_j restricted to the
//                  non-pivot coordinates (r_j has no other pivot bit);
//   j not a pivot: word part 0, residual part the unit vector of j.
// Residuals live on the m = d - rank non-pivot coordinates only, so they are
// stored compressed (the t-th non-pivot coordinate in increasing order is
// bit t).  E is linear in q, so for each group p of four coordinates the
// table holds all 16 XOR combinations of E_{4p..4p+3}; a reduction then
// costs exactly ceil(d/4) lookups, and q lies in the span iff its compressed
// residual is zero (Sec. 2.3; Sec. 2.2 step (1)).
//
// Layout of a table with np = ceil(d/4) groups and rw = ceil(m/32) residual
// words (word offsets): low z half uint2[np*16] at 0, high z half at 32*np,
// residual word u uint32[np*16] at 64*np + 16*np*u; entry e = 16*p + v.  With
// eight-byte and four-byte planes the lookups of a warp at one position are
// free of bank conflicts (the 16 values of v fall in distinct banks).  A
// table is 16*np*(4 + rw) words, a multiple of 64 bytes.
// ---------------------------------------------------------------------------
constexpr int TABLE_MAX_WD = NARROW_WD;  // widest row with a table (d <= 288)
constexpr int TABLE_MAX_RW = 4;          // compressed residual words (m <= 128)

__host__ __device__ __forceinline__ int table_words(int d, int rank)
{
    const int np = (d + 3) >> 2, rw = (d - rank + 31) >> 5;
    return 16 * np * (4 + rw);
}

// acc = XOR of the word parts, r = compressed residual of q (consumed: its
// words are shifted out, eight coordinate groups per word).
template <int RW, int WD>
__device__ __forceinline__ void table_reduce(const uint32_t* tab, int np, uint32_t (&q)[WD], uint4& acc,
                                             uint32_t (&r)[RW > 0 ? RW : 1])
{
    // byte addressing: entry v of group h of a word sits at 8v (16v in the
    // residual planes: 4v) bytes from the word's plane bases, with the
    // group's offset an immediate; two lookups per step share three-input XORs
    const char* const base = reinterpret_cast<const char*>(tab);
    const int zh_off = np * 128;       // high plane, bytes from the low one
    const int r_off = np * 256;        // first residual plane
    const int r_stride = np * 64;      // between residual planes
    uint32_t a0 = 0, a1 = 0, a2 = 0, a3 = 0;
#pragma unroll
    for (int u = 0; u < (RW > 0 ? RW : 1); ++u) r[u] = 0;
    int left = np;
    int wo = 0;  // the word's byte offset in the low plane (1024 a word; 512 in a residual plane)
#pragma unroll 1
    for (; left >= 8; left -= 8, wo += 1024) {  // whole words of eight groups: no bounds test
        const uint32_t word = q[0];
#pragma unroll
        for (int v = 0; v < WD - 1; ++v) q[v] = q[v + 1];
        const char* const zl = base + wo;
        const char* const zh = zl + zh_off;
        const char* const rp = base + r_off + (wo >> 1);
#pragma unroll
        for (int h = 0; h < 8; h += 2) {
            const uint32_t oa = (h == 0) ? ((word << 3) & 0x78u) : ((word >> (4 * h - 3)) & 0x78u);
            const uint32_t ob = (word >> (4 * h + 1)) & 0x78u;
            const uint2 la = *reinterpret_cast<const uint2*>(zl + oa + 128 * h);
            const uint2 lb = *reinterpret_cast<const uint2*>(zl + ob + 128 * (h + 1));
            const uint2 ha = *reinterpret_cast<const uint2*>(zh + oa + 128 * h);
            const uint2 hb = *reinterpret_cast<const uint2*>(zh + ob + 128 * (h + 1));
            a0 ^= la.x ^ lb.x;
            a1 ^= la.y ^ lb.y;
            a2 ^= ha.x ^ hb.x;
            a3 ^= ha.y ^ hb.y;
#pragma unroll
            for (int u = 0; u < RW; ++u) {
                const char* ru = rp + u * r_stride;
                r[u] ^= *reinterpret_cast<const uint32_t*>(ru + (oa >> 1) + 64 * h) ^
                        *reinterpret_cast<const uint32_t*>(ru + (ob >> 1) + 64 * (h + 1));
            }
        }
    }
    if (left > 0) {  // the last word's groups
        const uint32_t word = q[0];
#pragma unroll
        for (int v = 0; v < WD - 1; ++v) q[v] = q[v + 1];
        const int g0 = np - left;  // its first group
        const uint2* Zl = reinterpret_cast<const uint2*>(tab) + 16 * g0;
        const uint2* Zh = Zl + np * 16;
        const uint32_t* R = tab + 64 * np + 16 * g0;
#pragma unroll
        for (int h = 0; h < 8; ++h) {
            if (h < left) {
                const int e = h * 16 + (int)((word >> (4 * h)) & 15u);
                const uint2 lo = Zl[e];
                const uint2 hi = Zh[e];
                a0 ^= lo.x;
                a1 ^= lo.y;
                a2 ^= hi.x;
                a3 ^= hi.y;
#pragma unroll
                for (int u = 0; u < RW; ++u) r[u] ^= R[u * (16 * np) + e];
            }
        }
    }
    acc = make_uint4(a0, a1, a2, a3);
}

__device__ __forceinline__ void record_status(int* status, int code)
{
    atomicCAS(status, 0, code);
}

// ---------------------------------------------------------------------------
// Asynchronous copies into shared memory (sm_90+ PTX): the 1-D bulk copy of
// the tensor-memory-access unit, completed on an mbarrier by transaction
// bytes, and the per-thread cp.async of 4/8/16 bytes.  Every wait is bounded
// by a %globaltimer deadline; a wait that runs out returns false and the
// caller records F2_ERR_TIMEOUT instead of hanging.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(unsigned long long* bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

// Make initialised mbarriers visible to the asynchronous proxy.
__device__ __forceinline__ void mbar_init_fence() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }

// Order this thread's earlier shared-memory accesses (generic proxy) before
// later asynchronous-proxy writes to the same memory.
__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ void mbar_arrive_expect_tx(unsigned long long* bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
}

// dst (shared) and src (global) 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_copy_g2s(void* dst, const void* src, uint32_t bytes, unsigned long long* bar)
{
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_addr(dst)),
                 "l"(src), "r"(bytes), "r"(smem_addr(bar))
                 : "memory");
}

// The same copy with an L2 cache-policy hint (a policy from l2_policy_*).
__device__ __forceinline__ void bulk_copy_g2s_hint(void* dst, const void* src, uint32_t bytes, unsigned long long* bar,
                                                   unsigned long long policy)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
            smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}

// L2 policy: keep the lines (evict last), for data read again soon.
__device__ __forceinline__ unsigned long long l2_policy_evict_last()
{
    unsigned long long p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}

__device__ __forceinline__ bool mbar_try_wait(unsigned long long* bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ unsigned long long global_ns()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

constexpr unsigned long long WAIT_LIMIT_NS = 200000000ull;  // 0.2 s: far above any copy's latency

// Wait for the phase of `bar` with the given parity to complete, at most
// WAIT_LIMIT_NS; false when the deadline passed first.
__device__ __forceinline__ bool mbar_wait_bounded(unsigned long long* bar, uint32_t parity)
{
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    while (!mbar_try_wait(bar, parity))
        if (global_ns() - t0 > WAIT_LIMIT_NS) return false;
    return true;
}

// Per-thread asynchronous copies (cp.async, L1-allocating for 4/8 bytes,
// L2-only for 16); completed by cp_async_wait_all.
__device__ __forceinline__ void cp_async4(void* dst, const void* src)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async16(void* dst, const void* src)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait_group()
{
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

}  // namespace f2

struct f2_store {
    int32_t num_ctx;
    uint32_t flags;
    int device;
    int num_sms;
    int32_t max_wd;
    int32_t max_xw;         // widest feature row (words) supplied
    int32_t max_d;
    int32_t n_wide;         // contexts with wd > NARROW_WD
    int64_t slots;
    int64_t basis_words;
    int64_t pivot_words;
    int64_t heavy_rows;
    int heavy_rows_set;     // F2_OPT_HEAVY_ROWS given explicitly (else it scales with the batch)
    int warp_work_set;      // F2_OPT_WARP_WORK given explicitly
    int64_t warp_basis_bytes;
    int64_t warp_work;
    int dedup;              // run the duplicate pass before elimination
    int elim_tables;        // snapshot reduction by lookup table where it pays
    int64_t small_basis_bytes;  // shared memory of a warp-owned context, small-width kernel
    int dd_shards;              // most CTAs one context's duplicate pass is split over
    int64_t enc_direct_max;     // encode passes of at most this many queries skip the grouping
    int64_t long_call_rows;     // learn calls of at least this many rows: 4-warp CTAs for 4..9-word contexts
    int64_t handoff_min;        // representatives left for a saturated context to hand off (0: never)
    int* hand;                  // hand-off lists: counts [2], snap list/start [2C], resume list/from [2C], chunk counters [2C]
    uint4* check_rec;           // the check's chunk records (2 x uint4 each), grown per call
    int64_t check_rec_cap;
    f2::Widths widths;      // width classes of the contexts (computed on first use)
    // second stream of the learn launches (kernels of independent width
    // classes run side by side), its fork and join events; created on first use
    mutable cudaStream_t aux;
    mutable cudaEvent_t ev_fork, ev_join;
    bool widths_ready;
    std::vector<int32_t> n_bits;
    std::vector<int64_t> slot_off, xw_off, pw_off;
    // device memory
    f2::CtxDesc* desc;
    int32_t* rank;
    uint8_t* contra;
    long long* first_contra;
    unsigned long long* n_contra;
    long long* rows_seen;
    uint32_t* pivot;
    uint32_t* bx;
    uint4* bz;
    int* status;
    // scheduling scratch of f2_learn_batched
    int32_t* queue;
    int32_t* keybuf;
    int* counters;
    int* plan_hist;         // key histogram / cursors of the plan kernels
    int32_t* rep_count;     // representatives per context (pass 1 output)
    int32_t* shard_reps;    // [8C]: representatives of each shard of a split context (pass 1)
    int32_t* shard_done;    // [C]: finished shards of a split context
    int32_t* rep_list;      // per-row scratch of pass 1 (capacity rep_capacity rows)
    int32_t* rep_dup;
    int64_t rep_capacity;
    // per-context scratch of the full-rank check: chunks claimed [C], chunks
    // done [C], first row left and list of the contexts that reached full rank
    // during a call [C each] and their count; contradiction count [C], first
    // contradicting row [C]
    int* full_ctr;
    unsigned long long* full_cnt;
    unsigned long long* full_first;
    // scratch of f2_encode_batched (grouping of the queries by context)
    mutable int32_t* enc_bins;              // bucket sizes / starts, tile sums, ticket
    mutable int64_t enc_bin_cap;
    mutable int32_t* enc_off;               // offset of each query inside its bucket
    mutable unsigned long long* enc_sorted; // (bucket << 32) | query, grouped
    mutable unsigned long long* enc_items;  // runs left to the per-warp kernel
    mutable int64_t enc_q_cap;
    mutable int enc_short_per_sm;           // resident CTAs of the per-warp encode kernel
    mutable int enc_runs_per_sm;            // resident CTAs of the table encode kernel
    int enc_table_min;                      // fewest queries of a context (per pass) that get a table
    int enc_chunk_shift;                    // log2 of the queries of one locality chunk
    int64_t enc_chunk_min;                  // fewest queries of a context (per pass) laid out chunk by chunk
    mutable uint8_t* enc_hot;               // per bucket: encoded with a table in this pass
    mutable long long* enc_tab_off;         // per bucket: word offset of its table in the pool
    mutable uint32_t* enc_pool;             // lookup tables of the contexts with many queries
    mutable int64_t enc_pool_words;
    mutable int64_t enc_meta_cap;           // buckets of enc_hot / enc_tab_off
    // test hook (F2_OPT_FAIL_ALLOC): device allocations left before one is
    // made to fail; -1 = off
    mutable int64_t fail_alloc_in;
    // diagnostics (F2_OPT_TIMING): per-context timestamps of the last learn call
    int timing_on;
    unsigned long long* timing;
    // host-input entry points (f2_learn_host, f2_encode_host)
    f2::HostIO* hio;
    int64_t host_chunk_bytes;               // bytes of rows (or queries) per copied chunk

    f2::StoreDev dev() const
    {
        f2::StoreDev s;
        s.desc = desc;
        s.rank = rank;
        s.contra = contra;
        s.first_contra = first_contra;
        s.n_contra = n_contra;
        s.rows_seen = rows_seen;
        s.pivot = pivot;
        s.bx = bx;
        s.bz = bz;
        s.status = status;
        s.num_ctx = num_ctx;
        s.raw = (flags & F2_FLAG_RAW_FEATURES) ? 1u : 0u;
        return s;
    }
};

constexpr int64_t DEFAULT_HOST_CHUNK_BYTES = int64_t(512) << 20;

// Host helpers (store.cu, encode.cu, host_io.cu).
void f2_host_io_free(f2_store* st);
int f2_cuda_status(cudaError_t e);
// Queue slots beyond one per context, for the shard items of split contexts.
inline int f2_shard_queue_extra(int num_sms) { return 16 * num_sms + 64; }

// Every device allocation made by a call on a store goes through here (the
// stream-ordered allocator with a stream, cudaMalloc without one), so the
// F2_OPT_FAIL_ALLOC hook can make it fail.
cudaError_t f2_dev_alloc(const f2_store* st, void** p, size_t bytes, cudaStream_t cs, bool stream_ordered);
// Byte fills of several device buffers in one kernel launch (what a call
// would otherwise spend one memset node on each); null or empty segments
// are skipped.
struct F2FillList {
    static constexpr int MAX = 12;
    void* p[MAX];
    unsigned long long bytes[MAX];
    unsigned int value[MAX];  // byte value
    int n = 0;
    bool overflow = false;  // more than MAX ranges: f2_fill refuses the list
    void add(void* ptr, size_t nbytes, unsigned int byte = 0)
    {
        if (!ptr || !nbytes) return;
        if (n == MAX) {
            overflow = true;
            return;
        }
        p[n] = ptr;
        bytes[n] = nbytes;
        value[n] = byte & 0xffu;
        ++n;
    }
};
cudaError_t f2_fill(const F2FillList& L, cudaStream_t cs);
int f2_ensure_aux(const f2_store* st);  // second stream and fork/join events, created on first use
int f2_encode_table_min_default();
int f2_encode_table_min_floor();
int f2_encode_chunk_shift_default();
long long f2_encode_chunk_min_default();
