// Batched encoding with a span check (Sec. 2.3, Appendix B) on sm_103a.
//
// q = phi(x) is reduced against its context's reduced basis; every stored row
// used also XORs its z_k into a zero accumulator.  Because the basis is
// reduced, the rows to use are exactly the pivots set in q itself.  A zero
// residual at the non-pivot columns proves q in the span and the accumulator
// is the word; otherwise the query is rejected and the word is zero.
//
// The queries are first grouped by context (pass 1 below); long runs of one
// context are then encoded with a lookup table of its basis in shared memory
// and the rest by a per-thread walk over the pivots set in q (pass 2).
#include "f2_internal.cuh"

using namespace f2;

namespace {

// q = phi(x) (or x itself for raw features) in WD words; words at and above
// cd.wd and bits at and above d are zero.
template <int WD>
__device__ __forceinline__ void load_q(const StoreDev& s, const CtxDesc& cd, const uint32_t* __restrict__ xq,
                                       uint32_t (&q)[WD])
{
    uint32_t xin[WD];
#pragma unroll
    for (int v = 0; v < WD; ++v) {
        uint32_t t = (v < cd.xw) ? __ldg(xq + v) : 0u;
        if (v == cd.xw - 1 && (cd.n & 31)) t &= (1u << (cd.n & 31)) - 1u;
        xin[v] = t;
    }
    if (s.raw) {
#pragma unroll
        for (int v = 0; v < WD; ++v) q[v] = xin[v];
    } else {
        q[0] = (xin[0] << 1) | 1u;
#pragma unroll
        for (int v = 1; v < WD; ++v) q[v] = (xin[v] << 1) | (xin[v - 1] >> 31);
    }
}

template <int WD>
__device__ __forceinline__ bool encode_one(const StoreDev& s, const CtxDesc& cd, const uint32_t* __restrict__ xq,
                                           uint4& acc)
{
    uint32_t q[WD];
    load_q<WD>(s, cd, xq, q);
    acc = make_uint4(0, 0, 0, 0);
    const uint32_t* __restrict__ P = s.pivot + cd.pw_off;
    const uint4* __restrict__ Z = s.bz + cd.slot_off;
    const uint32_t* __restrict__ X = s.bx + cd.xw_off;
#pragma unroll
    for (int w = 0; w < WD; ++w) {
        if (w < cd.wd) {
            const uint32_t pw = __ldg(P + w);
            uint32_t m = q[w] & pw;
            // up to four stored rows per step: their loads are independent, so
            // they are issued together before any XOR
            constexpr int U = (WD <= NARROW_WD) ? 4 : 1;
            while (m) {
                int k[U];
                bool use[U];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    use[u] = m != 0u;
                    k[u] = use[u] ? 32 * w + __ffs(m) - 1 : 0;
                    m &= m - 1;
                }
                uint4 z[U];
                uint32_t xv[U][WD];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    z[u] = use[u] ? __ldg(Z + k[u]) : make_uint4(0, 0, 0, 0);
                    const uint32_t* rk = X + (int64_t)k[u] * cd.wd;
#pragma unroll
                    for (int v = 0; v <= w; ++v) xv[u][v] = use[u] ? __ldg(rk + v) : 0u;
                }
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    acc.x ^= z[u].x;
                    acc.y ^= z[u].y;
                    acc.z ^= z[u].z;
                    acc.w ^= z[u].w;
#pragma unroll
                    for (int v = 0; v <= w; ++v) q[v] ^= xv[u][v];
                }
            }
        }
    }
    // rows of higher pivots change non-pivot bits of lower words, so the
    // residual is read only after every word has been processed
    uint32_t resid = 0;
#pragma unroll
    for (int w = 0; w < WD; ++w)
        if (w < cd.wd) resid |= q[w] & ~__ldg(P + w);
    return resid == 0;
}

// ---------------------------------------------------------------------------
// Pass 1: group the queries by context (a counting sort; the order inside a
// context's bucket is arbitrary, since every query's result depends only on
// the query).  Ids outside [0, num_ctx) go to the extra bucket num_ctx.
//
//   enc_count_kernel   a CTA aggregates ENC_TILE consecutive queries per
//                      context in a shared-memory hash table (one shared
//                      atomic per distinct context per warp), claims each
//                      context's share of its bucket with one global atomic,
//                      and writes every query's offset inside its bucket;
//   enc_scan_kernel    exclusive prefix of the bucket sizes: per tile of
//                      SCAN_TILE buckets, then the tile totals (by the last
//                      CTA to finish);
//   enc_scatter_kernel writes (bucket, query) to its bucket position.
// ---------------------------------------------------------------------------
constexpr int ENC_TILE = 2048;
constexpr int ENC_TILE_THREADS = 256;
constexpr int ENC_TILE_PER = ENC_TILE / ENC_TILE_THREADS;
constexpr int ENC_HT_BITS = 12;
constexpr int ENC_HT = 1 << ENC_HT_BITS;
static_assert(ENC_HT >= 2 * ENC_TILE, "hash table of a tile at most half full");
constexpr int SCAN_THREADS = 1024;
constexpr int SCAN_SHIFT = 12;
constexpr int SCAN_TILE = 1 << SCAN_SHIFT;  // 4 buckets per thread
constexpr int SCAT_THREADS = 256;
constexpr int SCAT_PER = 4;
constexpr int64_t ENC_SUB = int64_t(1) << 25;   // queries grouped per pass
constexpr int32_t EMPTY_KEY = -1;

__device__ __forceinline__ int32_t bucket_of(int32_t c, int32_t num_ctx)
{
    return (c < 0 || c >= num_ctx) ? num_ctx : c;
}

// Exclusive prefix sum over the CTA; total receives the sum of all v.
// ws needs THREADS/32 + 1 entries; the CTA may reuse ws after the call.
template <int THREADS, typename T>
__device__ __forceinline__ T block_exclusive_scan(T v, T* ws, T& total)
{
    constexpr int NW = THREADS / 32;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    T inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const T u = __shfl_up_sync(FULL, inc, o);
        if (lane >= o) inc += u;
    }
    if (lane == 31) ws[w] = inc;
    __syncthreads();
    if (w == 0) {
        const T sv = (lane < NW) ? ws[lane] : T(0);
        T si = sv;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const T u = __shfl_up_sync(FULL, si, o);
            if (lane >= o) si += u;
        }
        if (lane < NW) ws[lane] = si - sv;
        if (lane == NW - 1) ws[NW] = si;
    }
    __syncthreads();
    const T r = ws[w] + inc - v;
    total = ws[NW];
    __syncthreads();
    return r;
}

__global__ void __launch_bounds__(ENC_TILE_THREADS) enc_count_kernel(int32_t Q, const int32_t* __restrict__ ctx_id,
                                                                     int32_t num_ctx, int32_t* __restrict__ bins,
                                                                     int32_t* __restrict__ off)
{
    __shared__ int32_t key[ENC_HT];
    __shared__ int32_t cnt[ENC_HT];
    const int t = threadIdx.x, lane = t & 31;
    const int64_t base = (int64_t)blockIdx.x * ENC_TILE;
    int32_t bk[ENC_TILE_PER];
#pragma unroll
    for (int j = 0; j < ENC_TILE_PER; ++j) {  // all loads first
        const int64_t i = base + (int64_t)j * ENC_TILE_THREADS + t;
        bk[j] = (i < Q) ? bucket_of(__ldg(ctx_id + i), num_ctx) : EMPTY_KEY;
    }
    for (int h = t; h < ENC_HT; h += ENC_TILE_THREADS) {
        key[h] = EMPTY_KEY;
        cnt[h] = 0;
    }
    __syncthreads();
    const uint32_t below = (1u << lane) - 1u;
    int slot[ENC_TILE_PER], rank[ENC_TILE_PER];
#pragma unroll
    for (int j = 0; j < ENC_TILE_PER; ++j) {
        const int32_t b = bk[j];
        const uint32_t peers = __match_any_sync(FULL, b);
        const int leader = __ffs(peers) - 1;
        int sl = 0, r0 = 0;
        if (lane == leader && b != EMPTY_KEY) {
            // at most ENC_TILE distinct keys in ENC_HT slots: a free or
            // matching slot is always found within ENC_HT probes
            uint32_t h = ((uint32_t)b * 2654435761u) >> (32 - ENC_HT_BITS);
            for (int probe = 0; probe < ENC_HT; ++probe) {
                const int32_t prev = atomicCAS(&key[h], EMPTY_KEY, b);
                if (prev == EMPTY_KEY || prev == b) break;
                h = (h + 1) & (ENC_HT - 1);
            }
            sl = (int)h;
            r0 = atomicAdd(&cnt[h], __popc(peers));
        }
        slot[j] = __shfl_sync(FULL, sl, leader);
        rank[j] = __shfl_sync(FULL, r0, leader) + __popc(peers & below);
    }
    __syncthreads();
    // one global atomic per distinct context of the tile; all of a thread's
    // atomics are issued before any result is used
    constexpr int HPER = ENC_HT / ENC_TILE_THREADS;
    int got[HPER];
#pragma unroll
    for (int u = 0; u < HPER; ++u) {
        const int h = u * ENC_TILE_THREADS + t;
        const int32_t k = key[h];
        got[u] = (k != EMPTY_KEY) ? atomicAdd(bins + k, cnt[h]) : 0;
    }
    __syncthreads();
#pragma unroll
    for (int u = 0; u < HPER; ++u) cnt[u * ENC_TILE_THREADS + t] = got[u];
    __syncthreads();
#pragma unroll
    for (int j = 0; j < ENC_TILE_PER; ++j) {
        const int64_t i = base + (int64_t)j * ENC_TILE_THREADS + t;
        if (i < Q) off[i] = cnt[slot[j]] + rank[j];
    }
}

__global__ void __launch_bounds__(SCAN_THREADS) enc_scan_kernel(int32_t* __restrict__ bins, int32_t N,
                                                                int32_t* __restrict__ tsum,
                                                                int32_t* __restrict__ tpre,
                                                                int32_t* __restrict__ ticket)
{
    __shared__ int ws[SCAN_THREADS / 32 + 1];
    __shared__ int carry;
    __shared__ int last;
    const int t = threadIdx.x;
    const int T = gridDim.x;
    const int64_t b0 = (int64_t)blockIdx.x * SCAN_TILE + 4 * t;
    int v[4], sum = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        v[k] = (b0 + k < N) ? bins[b0 + k] : 0;
        sum += v[k];
    }
    int total;
    int run = block_exclusive_scan<SCAN_THREADS>(sum, ws, total);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        if (b0 + k < N) bins[b0 + k] = run;  // tile-local start
        run += v[k];
    }
    if (t == 0) {
        tsum[blockIdx.x] = total;
        __threadfence();
        last = (atomicAdd(ticket, 1) == T - 1);
        carry = 0;
    }
    __syncthreads();
    if (!last) return;
    __threadfence();
    for (int c0 = 0; c0 < T; c0 += SCAN_THREADS) {
        const int k = c0 + t;
        const int val = (k < T) ? __ldcg(tsum + k) : 0;
        int tot;
        const int e = block_exclusive_scan<SCAN_THREADS>(val, ws, tot);
        if (k < T) tpre[k] = carry + e;
        __syncthreads();
        if (t == 0) carry += tot;
        __syncthreads();
    }
}

__global__ void __launch_bounds__(SCAT_THREADS) enc_scatter_kernel(int32_t Q, const int32_t* __restrict__ ctx_id,
                                                                   int32_t num_ctx, const int32_t* __restrict__ bins,
                                                                   const int32_t* __restrict__ tpre,
                                                                   const int32_t* __restrict__ off,
                                                                   unsigned long long* __restrict__ sorted)
{
    const int64_t base = (int64_t)blockIdx.x * (SCAT_THREADS * SCAT_PER) + threadIdx.x;
    int32_t b[SCAT_PER], o[SCAT_PER];
#pragma unroll
    for (int j = 0; j < SCAT_PER; ++j) {  // every load of a step before any use
        const int64_t i = base + (int64_t)j * SCAT_THREADS;
        b[j] = (i < Q) ? bucket_of(__ldg(ctx_id + i), num_ctx) : -1;
        o[j] = (i < Q) ? __ldg(off + i) : 0;
    }
    int32_t p[SCAT_PER];
#pragma unroll
    for (int j = 0; j < SCAT_PER; ++j) {
        const int bb = b[j] < 0 ? 0 : b[j];
        p[j] = __ldg(bins + bb) + __ldg(tpre + (bb >> SCAN_SHIFT)) + o[j];
    }
#pragma unroll
    for (int j = 0; j < SCAT_PER; ++j) {
        const int64_t i = base + (int64_t)j * SCAT_THREADS;
        if (b[j] >= 0) sorted[p[j]] = ((unsigned long long)(uint32_t)b[j] << 32) | (uint32_t)i;
    }
}

// ---------------------------------------------------------------------------
// Pass 2: encode the grouped queries.
//
// enc_runs_kernel: a CTA takes RUN_SEG consecutive positions of the grouped
// order, i.e. a few runs of queries of one context each.  A run of at least
// table_min queries whose context fits the tables is encoded with a table of
// its basis (a Four-Russians table over 4-bit groups of coordinates).  The
// reduction of q against the reduced basis XORs, for every set coordinate j
// of q, the vector E_j:
//   j a pivot:     word part z_j, residual part r_j restricted to the
//                  non-pivot coordinates (r_j has no other pivot bit);
//   j not a pivot: word part 0, residual part the unit vector of j.
// Residuals live on the m = d - rank non-pivot coordinates only, so they are
// stored compressed (the t-th non-pivot coordinate in increasing order is
// bit t).  E is linear in q, so for each group p of four coordinates the
// table holds all 16 XOR combinations of E_{4p..4p+3}; a query then costs
// exactly ceil(d/4) lookups and is in the span iff its compressed residual is
// zero (Sec. 2.3: the word is T(q) = XOR of the z_k used; the query is
// rejected otherwise).  The other runs are cut into items of at most 32
// queries and appended to a list for enc_short_kernel.
//
// enc_short_kernel: a warp per item stages the context's basis rows in its
// shared-memory region with one round of loads, then every lane reduces its
// query against them in a warp-uniform walk over the pivots.
// ---------------------------------------------------------------------------
constexpr int RUN_THREADS = 512;  // two CTAs per SM: 32 warps (three CTAs of 256 gave 24)
constexpr int RUN_SEG = 2048;
constexpr int RUN_PER = RUN_SEG / RUN_THREADS;
constexpr int TAB_WD = NARROW_WD;             // widest context with a table (d <= 288)
constexpr int TAB_RW = 4;                     // compressed residual words (m <= 128)
constexpr int TAB_WORDS = 8192;               // one group of tables (32 KB); larger tables are not built
constexpr int MAX_TRUNS = 128;                // table runs of a segment: table_min >= RUN_SEG / MAX_TRUNS
constexpr int DEFAULT_TABLE_MIN = 32;
constexpr int ITEM_MAX = 32;                  // queries of a short item (one per lane)
constexpr int ITEM_POS_BITS = 25;             // item = position | (length - 1) << 25
static_assert(ENC_SUB <= (int64_t(1) << ITEM_POS_BITS), "item positions fit 25 bits");

struct RunSmem {
    uint4 table[TAB_WORDS / 4];
    unsigned long long ent[RUN_SEG];   // (bucket << 32) | query index
    uint32_t flat[RUN_SEG];            // table positions in order: position | table run << 16
    uint16_t starts[RUN_SEG + 1];      // run starts
    int16_t run_tr[RUN_SEG];           // table run of each run, -1 if none
    int32_t tr_ctx[MAX_TRUNS];
    int32_t tr_tab[MAX_TRUNS];         // word offset of the run's table in `table`
    int32_t tr_j0[MAX_TRUNS];          // first single-coordinate item of the run in its group
    int32_t tr_e0[MAX_TRUNS];          // first table entry of the run in its group
    int32_t tr_flat[MAX_TRUNS + 1];    // first flat index of the run
    long long tr_slot_off[MAX_TRUNS];  // the run's context: basis offsets
    long long tr_xw_off[MAX_TRUNS];
    long long tr_pw_off[MAX_TRUNS];
    int16_t tr_d[MAX_TRUNS];
    uint8_t tr_wd[MAX_TRUNS];
    int16_t tr_n[MAX_TRUNS];           // feature bits of the run's context
    uint8_t tr_np[MAX_TRUNS];
    uint8_t tr_rw[MAX_TRUNS];
    uint8_t tr_xw[MAX_TRUNS];
    int32_t g_first[MAX_TRUNS + 1];
    int32_t g_j[MAX_TRUNS];
    int32_t g_e[MAX_TRUNS];
    uint8_t g_xw[MAX_TRUNS];           // widest feature vector of the group's runs
    int32_t ws[RUN_THREADS / 32 + 1];
    int32_t n_groups;
    int32_t item_base;
};
static_assert(sizeof(RunSmem) + 1024 <= 233472 / 2, "two CTAs of enc_runs_kernel per SM");

__device__ __forceinline__ void encode_direct(const StoreDev& s, int32_t c, int64_t i, const uint32_t* __restrict__ x,
                                              int stride, uint4* __restrict__ y, uint8_t* __restrict__ in_span)
{
    uint4 acc = make_uint4(0, 0, 0, 0);
    uint8_t flag;
    if (c >= s.num_ctx) {
        record_status(s.status, F2_ERR_CTX_RANGE);
        flag = 0xFF;
    } else {
        const CtxDesc cd = s.desc[c];
        if (cd.xw > stride) {
            record_status(s.status, F2_ERR_STRIDE);
            flag = 0xFF;
        } else {
            const uint32_t* xq = x + i * stride;
            const bool ok = (cd.wd <= NARROW_WD) ? encode_one<NARROW_WD>(s, cd, xq, acc)
                                                 : encode_one<33>(s, cd, xq, acc);
            flag = ok ? 1 : 0;
            if (!ok) acc = make_uint4(0, 0, 0, 0);
        }
    }
    y[i] = acc;
    in_span[i] = flag;
}

// q = phi(x) from the raw feature words of a context with n bits.
template <int WD>
__device__ __forceinline__ void make_q(bool raw, int n, const uint32_t (&xr)[WD], uint32_t (&q)[WD])
{
    const int xw = (n + 31) >> 5;
    uint32_t xin[WD];
#pragma unroll
    for (int v = 0; v < WD; ++v) {
        uint32_t t = xr[v];
        if (v == xw - 1 && (n & 31)) t &= (1u << (n & 31)) - 1u;
        xin[v] = t;
    }
    if (raw) {
#pragma unroll
        for (int v = 0; v < WD; ++v) q[v] = xin[v];
    } else {
        q[0] = (xin[0] << 1) | 1u;
#pragma unroll
        for (int v = 1; v < WD; ++v) q[v] = (xin[v] << 1) | (xin[v - 1] >> 31);
    }
}

// The first xw (<= XW) feature words of a query, the rest zero.  With xvec
// (16-byte aligned rows: x aligned and the stride a multiple of 4 words)
// whole 16-byte pieces are loaded, which stay inside the row because xw <=
// stride; a random gather then costs one memory transaction per piece
// instead of one per word.
template <int XW>
__device__ __forceinline__ void load_x(const uint32_t* __restrict__ xq, int xw, bool xvec, uint32_t (&xo)[XW])
{
    if (xvec) {
#pragma unroll
        for (int v4 = 0; v4 * 4 < XW; ++v4) {
            uint4 p = make_uint4(0, 0, 0, 0);
            if (4 * v4 < xw) p = __ldg(reinterpret_cast<const uint4*>(xq) + v4);
            const uint32_t w[4] = {p.x, p.y, p.z, p.w};
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (4 * v4 + u < XW) xo[4 * v4 + u] = (4 * v4 + u < xw) ? w[u] : 0u;
        }
    } else {
#pragma unroll
        for (int v = 0; v < XW; ++v) xo[v] = (v < xw) ? __ldg(xq + v) : 0u;
    }
}

// E_j (see above) of context cd: word part z, compressed residual er.  The
// pivot words, z_j and r_j are loaded together (slots of non-pivots hold
// zeros), so a table costs one round of loads.
__device__ __forceinline__ void single_entry(const StoreDev& s, const CtxDesc& cd, int j, uint4& z,
                                             uint32_t (&er)[TAB_RW])
{
#pragma unroll
    for (int u = 0; u < TAB_RW; ++u) er[u] = 0;
    z = make_uint4(0, 0, 0, 0);
    if (j >= cd.d) return;
    const uint32_t* __restrict__ P = s.pivot + cd.pw_off;
    const uint32_t* __restrict__ row = s.bx + cd.xw_off + (int64_t)j * cd.wd;
    const int w = j >> 5, b = j & 31;
    uint32_t pv[TAB_WD], rv[TAB_WD];
#pragma unroll
    for (int u = 0; u < TAB_WD; ++u) {
        pv[u] = (u <= w) ? __ldg(P + u) : 0u;
        rv[u] = (u <= w) ? __ldg(row + u) : 0u;
    }
    const uint4 zj = __ldg(s.bz + cd.slot_off + j);
    auto set_bit = [&](int t) {
#pragma unroll
        for (int u = 0; u < TAB_RW; ++u)
            if ((t >> 5) == u) er[u] |= 1u << (t & 31);
    };
    int below = 0;  // non-pivot coordinates in the words before u (all full: u < w <= wd - 1)
    bool pivot = false;
#pragma unroll
    for (int u = 0; u < TAB_WD; ++u) {
        if (u == w) pivot = (pv[u] >> b) & 1u;
    }
    if (pivot) {
        z = zj;
#pragma unroll
        for (int u = 0; u < TAB_WD; ++u) {
            if (u <= w) {
                const uint32_t free_u = ~pv[u];
                uint32_t bits = rv[u] & free_u;  // r_j has no bit above j
                while (bits) {
                    const int bb = __ffs(bits) - 1;
                    set_bit(below + __popc(free_u & ((1u << bb) - 1u)));
                    bits &= bits - 1u;
                }
                below += __popc(free_u);
            }
        }
    } else {
#pragma unroll
        for (int u = 0; u < TAB_WD; ++u) {
            if (u < w) below += __popc(~pv[u]);
            if (u == w) set_bit(below + __popc(~pv[u] & ((1u << b) - 1u)));
        }
    }
}

// Table layout of one run with np groups and rw residual words (word
// offsets): low z half uint2[np*16] at 0, high z half at 32*np, residual word
// u uint32[np*16] at 64*np + 16*np*u; entry e = 16*p + v.  With eight-byte
// and four-byte planes the lookups of a warp at one position are free of bank
// conflicts (the 16 values of v fall in distinct banks).
template <int RW, int WD>
__device__ __forceinline__ bool table_query(const uint32_t* tab, int np, uint32_t (&q)[WD], uint4& acc)
{
    // one feature word (eight positions) per trip; q is consumed
    const uint2* Zl = reinterpret_cast<const uint2*>(tab);
    const uint2* Zh = Zl + np * 16;
    const uint32_t* R = tab + 64 * np;
    const int rstride = 16 * np;
    uint32_t a0 = 0, a1 = 0, a2 = 0, a3 = 0;
    uint32_t r[RW > 0 ? RW : 1];
#pragma unroll
    for (int u = 0; u < (RW > 0 ? RW : 1); ++u) r[u] = 0;
#pragma unroll 1
    for (int left = np; left > 0; left -= 8) {
        const uint32_t word = q[0];
#pragma unroll
        for (int v = 0; v < WD - 1; ++v) q[v] = q[v + 1];
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
                for (int u = 0; u < RW; ++u) r[u] ^= R[u * rstride + e];
            }
        }
        Zl += 128;
        Zh += 128;
        R += 128;
    }
    uint32_t res = 0;
#pragma unroll
    for (int u = 0; u < RW; ++u) res |= r[u];
    acc = make_uint4(a0, a1, a2, a3);
    return res == 0;
}

// largest i in [lo, hi] with a[i] <= f (a[lo] <= f)
__device__ __forceinline__ int find_item(const int32_t* a, int lo, int hi, int f)
{
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (a[mid] <= f)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

// Encode the queries at flat positions [fa, fb) of a segment with their
// runs' tables.  A query's feature words (at most XW) are fetched PF queries
// ahead of its lookups, so PF loads of each thread are in flight.
template <int WD, int XW, int PF>
__device__ __forceinline__ void query_group(const StoreDev& s, const RunSmem& sm, const uint32_t* table,
                                            const uint32_t* __restrict__ x, int stride, bool xvec,
                                            uint4* __restrict__ y, uint8_t* __restrict__ in_span, int fa, int fb)
{
    const int t = threadIdx.x;
    uint32_t xr[PF][XW];
    int64_t iq[PF];
    int trq[PF];
    auto fetch = [&](int kk, uint32_t (&xo)[XW], int64_t& i, int& tr) {
        tr = 0;
        i = 0;
        int xw = 0;
        if (kk < fb) {
            const uint32_t fv = sm.flat[kk];
            tr = (int)(fv >> 16);
            i = (int64_t)(uint32_t)sm.ent[fv & 0xFFFFu];
            xw = sm.tr_xw[tr];
        }
        load_x<XW>(x + i * stride, xw, xvec, xo);
    };
#pragma unroll
    for (int p = 0; p < PF; ++p) fetch(fa + t + p * RUN_THREADS, xr[p], iq[p], trq[p]);
    for (int k = fa + t; k < fb; k += RUN_THREADS) {
        uint32_t raw[WD];
#pragma unroll
        for (int v = 0; v < WD; ++v) raw[v] = (v < XW) ? xr[0][v] : 0u;
        const int tr = trq[0];
        const int64_t i = iq[0];
#pragma unroll
        for (int p = 0; p + 1 < PF; ++p) {
#pragma unroll
            for (int v = 0; v < XW; ++v) xr[p][v] = xr[p + 1][v];
            iq[p] = iq[p + 1];
            trq[p] = trq[p + 1];
        }
        fetch(k + PF * RUN_THREADS, xr[PF - 1], iq[PF - 1], trq[PF - 1]);
        uint32_t q[WD];
        make_q<WD>(s.raw != 0, sm.tr_n[tr], raw, q);
        const uint32_t* tab = table + sm.tr_tab[tr];
        const int np = sm.tr_np[tr];
        uint4 acc;
        bool ok;
        switch (sm.tr_rw[tr]) {
        case 0: ok = table_query<0, WD>(tab, np, q, acc); break;
        case 1: ok = table_query<1, WD>(tab, np, q, acc); break;
        case 2: ok = table_query<2, WD>(tab, np, q, acc); break;
        case 3: ok = table_query<3, WD>(tab, np, q, acc); break;
        default: ok = table_query<4, WD>(tab, np, q, acc); break;
        }
        y[i] = ok ? acc : make_uint4(0, 0, 0, 0);
        in_span[i] = ok ? 1 : 0;
    }
}

__global__ void __launch_bounds__(RUN_THREADS, 2) enc_runs_kernel(StoreDev s, int32_t n_total,
                                                                  const unsigned long long* __restrict__ sorted,
                                                                  const uint32_t* __restrict__ x, int stride,
                                                                  uint4* __restrict__ y,
                                                                  uint8_t* __restrict__ in_span, int table_min,
                                                                  unsigned long long* __restrict__ items,
                                                                  int32_t* __restrict__ n_items)
{
    extern __shared__ uint4 enc_smem[];
    RunSmem& sm = *reinterpret_cast<RunSmem*>(enc_smem);
    uint32_t* const table = reinterpret_cast<uint32_t*>(sm.table);
    const int t = threadIdx.x;
    const bool xvec = ((uintptr_t)x % 16) == 0 && (stride % 4) == 0;
    const int64_t seg0 = (int64_t)blockIdx.x * RUN_SEG;
    const int n = (int)((n_total - seg0) < RUN_SEG ? (n_total - seg0) : RUN_SEG);
    for (int k = t; k < n; k += RUN_THREADS) sm.ent[k] = __ldg(sorted + seg0 + k);
    __syncthreads();

    // runs: flag the first position of each run, number the runs
    const int k0 = t * RUN_PER;
    uint32_t first = 0;
    int nflag = 0;
    {
        uint32_t prev = (k0 > 0 && k0 <= n) ? (uint32_t)(sm.ent[k0 - 1] >> 32) : 0xFFFFFFFFu;
#pragma unroll
        for (int m = 0; m < RUN_PER; ++m) {
            const int k = k0 + m;
            if (k < n) {
                const uint32_t b = (uint32_t)(sm.ent[k] >> 32);
                if (k == 0 || b != prev) {
                    first |= 1u << m;
                    ++nflag;
                }
                prev = b;
            }
        }
    }
    int n_runs;
    const int r0 = block_exclusive_scan<RUN_THREADS>(nflag, sm.ws, n_runs);
    {
        int r = r0;
#pragma unroll
        for (int m = 0; m < RUN_PER; ++m)
            if ((first >> m) & 1u) sm.starts[r++] = (uint16_t)(k0 + m);
        if (t == 0) sm.starts[n_runs] = (uint16_t)n;
    }
    __syncthreads();

    // classify the runs, RUN_THREADS at a time: number the table runs (in
    // position order), count the items of the others
    int n_tr = 0, n_it = 0, my_base = 0;
    for (int c0 = 0; c0 < n_runs; c0 += RUN_THREADS) {
        const int rr = c0 + t;
        int nel = 0, nit = 0, len = 0;
        int32_t c = s.num_ctx;
        CtxDesc cd{};
        int32_t rk = 0;
        if (rr < n_runs) {
            len = (int)sm.starts[rr + 1] - (int)sm.starts[rr];
            c = (int32_t)(sm.ent[sm.starts[rr]] >> 32);
            if (c < s.num_ctx) {
                cd = s.desc[c];
                rk = s.rank[c];
            }
            const int np = (cd.d + 3) >> 2, rw = (cd.d - rk + 31) >> 5;
            const bool ok = len >= table_min && c < s.num_ctx && cd.wd <= TAB_WD && cd.xw <= stride &&
                            rw <= TAB_RW && 16 * np * (4 + rw) <= TAB_WORDS;
            nel = ok ? 1 : 0;
            nit = ok ? 0 : (len + ITEM_MAX - 1) / ITEM_MAX;
        }
        int tot;
        const int ex = block_exclusive_scan<RUN_THREADS>(nel | (nit << 16), sm.ws, tot);
        if (rr < n_runs) {
            if (nel) {
                const int tr = n_tr + (ex & 0xFFFF);
                sm.run_tr[rr] = (int16_t)tr;
                sm.tr_ctx[tr] = c;
                sm.tr_np[tr] = (uint8_t)((cd.d + 3) >> 2);
                sm.tr_rw[tr] = (uint8_t)((cd.d - rk + 31) >> 5);
                sm.tr_xw[tr] = (uint8_t)cd.xw;
                sm.tr_n[tr] = (int16_t)cd.n;
                sm.tr_d[tr] = (int16_t)cd.d;
                sm.tr_wd[tr] = (uint8_t)cd.wd;
                sm.tr_slot_off[tr] = cd.slot_off;
                sm.tr_xw_off[tr] = cd.xw_off;
                sm.tr_pw_off[tr] = cd.pw_off;
            } else {
                sm.run_tr[rr] = -1;
            }
        }
        n_tr += tot & 0xFFFF;
        n_it += tot >> 16;
    }
    // the item list slot is claimed now and used at the end, so the atomic's
    // latency overlaps the table work
    if (t == 0 && n_it) my_base = atomicAdd(n_items, n_it);
    __syncthreads();

    if (n_tr > 0) {  // block-uniform
        // table positions to `flat`, in order
        {
            int trs[RUN_PER];
            int nt = 0;
            int rid = r0 - 1;
#pragma unroll
            for (int m = 0; m < RUN_PER; ++m) {
                trs[m] = -1;
                if (k0 + m < n) {
                    if ((first >> m) & 1u) ++rid;
                    trs[m] = sm.run_tr[rid];
                    if (trs[m] >= 0) ++nt;
                }
            }
            int n_flat;
            int ft = block_exclusive_scan<RUN_THREADS>(nt, sm.ws, n_flat);
#pragma unroll
            for (int m = 0; m < RUN_PER; ++m) {
                if (trs[m] >= 0) {
                    if ((first >> m) & 1u) sm.tr_flat[trs[m]] = ft;
                    sm.flat[ft++] = (uint32_t)(k0 + m) | ((uint32_t)trs[m] << 16);
                }
            }
            if (t == 0) {
                sm.tr_flat[n_tr] = n_flat;
                // greedy groups of consecutive table runs that fit TAB_WORDS
                int g = 0, used = 0, j = 0, e = 0, gx = 0;
                sm.g_first[0] = 0;
                for (int tr = 0; tr < n_tr; ++tr) {
                    const int np = sm.tr_np[tr];
                    const int words = 16 * np * (4 + sm.tr_rw[tr]);
                    if (used + words > TAB_WORDS) {
                        sm.g_j[g] = j;
                        sm.g_e[g] = e;
                        sm.g_xw[g] = (uint8_t)gx;
                        sm.g_first[++g] = tr;
                        used = j = e = gx = 0;
                    }
                    gx = gx > sm.tr_xw[tr] ? gx : sm.tr_xw[tr];
                    sm.tr_tab[tr] = used;
                    sm.tr_j0[tr] = j;
                    sm.tr_e0[tr] = e;
                    used += words;
                    j += 4 * np;
                    e += 16 * np;
                }
                sm.g_j[g] = j;
                sm.g_e[g] = e;
                sm.g_xw[g] = (uint8_t)gx;
                sm.g_first[++g] = n_tr;
                sm.n_groups = g;
            }
        }
        __syncthreads();

        const int n_groups = sm.n_groups;
        for (int g = 0; g < n_groups; ++g) {
            const int ga = sm.g_first[g], gb = sm.g_first[g + 1] - 1;
            // single-coordinate entries E_j (v = 1, 2, 4, 8) and the zero entry
            for (int f = t; f < sm.g_j[g]; f += RUN_THREADS) {
                const int tr = find_item(sm.tr_j0, ga, gb, f);
                const int j = f - sm.tr_j0[tr];
                const int np = sm.tr_np[tr], rw = sm.tr_rw[tr];
                CtxDesc cd{};
                cd.d = sm.tr_d[tr];
                cd.wd = sm.tr_wd[tr];
                cd.slot_off = sm.tr_slot_off[tr];
                cd.xw_off = sm.tr_xw_off[tr];
                cd.pw_off = sm.tr_pw_off[tr];
                uint4 z;
                uint32_t er[TAB_RW];
                single_entry(s, cd, j, z, er);
                uint32_t* tab = table + sm.tr_tab[tr];
                uint2* Zl = reinterpret_cast<uint2*>(tab);
                uint2* Zh = Zl + np * 16;
                uint32_t* R = tab + 64 * np;
                const int e = (j >> 2) * 16 + (1 << (j & 3));
                Zl[e] = make_uint2(z.x, z.y);
                Zh[e] = make_uint2(z.z, z.w);
                for (int u = 0; u < rw; ++u) R[u * 16 * np + e] = er[u];
                if ((j & 3) == 0) {
                    const int e0 = (j >> 2) * 16;
                    Zl[e0] = make_uint2(0, 0);
                    Zh[e0] = make_uint2(0, 0);
                    for (int u = 0; u < rw; ++u) R[u * 16 * np + e0] = 0;
                }
            }
            __syncthreads();
            // entries of two or more coordinates: XOR of their single entries
            for (int f = t; f < sm.g_e[g]; f += RUN_THREADS) {
                const int v = f & 15;
                if (__popc(v) < 2) continue;
                const int tr = find_item(sm.tr_e0, ga, gb, f);
                const int e = f - sm.tr_e0[tr];
                const int np = sm.tr_np[tr], rw = sm.tr_rw[tr];
                uint32_t* tab = table + sm.tr_tab[tr];
                uint2* Zl = reinterpret_cast<uint2*>(tab);
                uint2* Zh = Zl + np * 16;
                uint32_t* R = tab + 64 * np;
                const int eb = e & ~15;
                uint2 lo = make_uint2(0, 0), hi = make_uint2(0, 0);
                uint32_t rr[TAB_RW] = {0, 0, 0, 0};
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
                        for (int u = 0; u < TAB_RW; ++u)
                            if (u < rw) rr[u] ^= R[u * 16 * np + es];
                    }
                }
                Zl[e] = lo;
                Zh[e] = hi;
#pragma unroll
                for (int u = 0; u < TAB_RW; ++u)
                    if (u < rw) R[u * 16 * np + e] = rr[u];
            }
            __syncthreads();
            // the queries of the group's runs
            const int fa = sm.tr_flat[ga], fb = sm.tr_flat[gb + 1];
            if (sm.g_xw[g] <= 4)
                query_group<5, 4, 3>(s, sm, table, x, stride, xvec, y, in_span, fa, fb);
            else
                query_group<TAB_WD, TAB_WD, 1>(s, sm, table, x, stride, xvec, y, in_span, fa, fb);
            __syncthreads();
        }
    }

    // items of the runs without a table, for enc_short_kernel (numbered in
    // run order again, RUN_THREADS runs at a time)
    if (t == 0) sm.item_base = my_base;
    __syncthreads();
    int it0 = sm.item_base;
    for (int c0 = 0; c0 < n_runs; c0 += RUN_THREADS) {
        const int rr = c0 + t;
        int a = 0, b = 0;
        uint32_t c = 0;
        if (rr < n_runs && sm.run_tr[rr] < 0) {
            a = sm.starts[rr];
            b = sm.starts[rr + 1];
            c = (uint32_t)(sm.ent[a] >> 32);
        }
        int tot;
        int it = it0 + block_exclusive_scan<RUN_THREADS>((b - a + ITEM_MAX - 1) / ITEM_MAX, sm.ws, tot);
        for (int p = a; p < b; p += ITEM_MAX) {
            const int len = (b - p) < ITEM_MAX ? (b - p) : ITEM_MAX;
            items[it++] = (unsigned long long)((uint32_t)(seg0 + p) | ((uint32_t)(len - 1) << ITEM_POS_BITS)) |
                          ((unsigned long long)c << 32);
        }
        it0 += tot;
    }
}

constexpr int SHORT_THREADS = 128;
constexpr int SHORT_WARPS = SHORT_THREADS / 32;
constexpr int SHORT_REGION = 2048;            // basis words staged per warp (8 KB)
constexpr int SHORT_MAX_D = 32 * TAB_WD;      // widest context staged (d <= 288)

struct ShortSmem {
    uint4 region[SHORT_WARPS][SHORT_REGION / 4];
    int16_t piv[SHORT_WARPS][SHORT_MAX_D];
    int32_t pbase[SHORT_WARPS][TAB_WD + 1];
};

__global__ void __launch_bounds__(SHORT_THREADS) enc_short_kernel(StoreDev s,
                                                                  const unsigned long long* __restrict__ sorted,
                                                                  const uint32_t* __restrict__ x, int stride,
                                                                  uint4* __restrict__ y,
                                                                  uint8_t* __restrict__ in_span,
                                                                  const unsigned long long* __restrict__ items,
                                                                  const int32_t* __restrict__ n_items)
{
    extern __shared__ uint4 short_smem[];
    ShortSmem& sm = *reinterpret_cast<ShortSmem*>(short_smem);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint32_t* const region = reinterpret_cast<uint32_t*>(sm.region[wid]);
    int16_t* const piv = sm.piv[wid];
    int32_t* const pbase = sm.pbase[wid];
    const int total = *n_items;
    const int nwarps = gridDim.x * SHORT_WARPS;
    const bool xvec = ((uintptr_t)x % 16) == 0 && (stride % 4) == 0;
    // An item is (position | (length - 1) << 25, context).  The loads of an
    // item that do not depend on its basis (the item, its queries' ids, the
    // context's descriptor and rank) are issued one item ahead.
    auto unpack = [&](unsigned long long it, int& pos, int& len, int32_t& c) {
        pos = (int)(it & ((1u << ITEM_POS_BITS) - 1u));
        len = (int)((it >> ITEM_POS_BITS) & 31u) + 1;
        c = (int32_t)(it >> 32);
    };
    int itx = blockIdx.x * SHORT_WARPS + wid;
    if (itx >= total) return;
    unsigned long long item = __ldg(items + itx);
    int pos, len;
    int32_t c;
    unpack(item, pos, len, c);
    unsigned long long en = __ldg(sorted + pos + (lane < len ? lane : 0));
    CtxDesc cd{};
    int rank = 0;
    if (c < s.num_ctx) {
        cd = s.desc[c];
        rank = s.rank[c];
    }
    while (true) {
        const int64_t i = (int64_t)(uint32_t)en;
        const int nxt = itx + nwarps;
        const unsigned long long item_n = (nxt < total) ? __ldg(items + nxt) : 0ull;
        const int rs = (4 + cd.wd + 3) & ~3;  // staged row stride, 16-byte aligned
        const bool staged = c < s.num_ctx && cd.wd <= TAB_WD && cd.xw <= stride && rank * rs <= SHORT_REGION;
        uint4 acc = make_uint4(0, 0, 0, 0);
        bool ok = false;
        if (staged) {
            // feature words and pivot words together
            uint32_t xr[TAB_WD];
            load_x<TAB_WD>(x + i * stride, lane < len ? cd.xw : 0, xvec, xr);
            const uint32_t pw = (lane < cd.wd) ? __ldg(s.pivot + cd.pw_off + lane) : 0u;
            // pivot list, word by word, and the staged rows [z_k | r_k]
            const int cnt = __popc(pw);
            int inc = cnt;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int u = __shfl_up_sync(FULL, inc, o);
                if (lane >= o) inc += u;
            }
            if (lane <= cd.wd) pbase[lane] = inc - cnt;
            {
                int idx = inc - cnt;
                uint32_t bits = pw;
                while (bits) {
                    piv[idx++] = (int16_t)(32 * lane + __ffs(bits) - 1);
                    bits &= bits - 1u;
                }
            }
            __syncwarp();
            {
                const int cols = 4 + cd.wd;
                const int per = 32 / cols;
                const int row_in = lane / cols, col = lane - row_in * cols;
                if (row_in < per) {
                    for (int idx = row_in; idx < rank; idx += per) {
                        const int k = piv[idx];
                        const uint32_t v =
                            (col < 4) ? __ldg(reinterpret_cast<const uint32_t*>(s.bz + cd.slot_off + k) + col)
                                      : __ldg(s.bx + cd.xw_off + (int64_t)k * cd.wd + (col - 4));
                        region[idx * rs + col] = v;
                    }
                }
            }
            __syncwarp();
            uint32_t q[TAB_WD];
            make_q<TAB_WD>(s.raw != 0, cd.n, xr, q);
            // every pivot k set in q: XOR row k (its bits lie in words <= k/32)
#pragma unroll
            for (int w = 0; w < TAB_WD; ++w) {
                if (w < cd.wd) {
                    const int e = pbase[w + 1];
                    for (int idx = pbase[w]; idx < e; ++idx) {
                        const int b = piv[idx] & 31;
                        const uint32_t use = 0u - ((q[w] >> b) & 1u);
                        const uint4* row = reinterpret_cast<const uint4*>(region + idx * rs);
                        const uint4 z = row[0];
                        acc.x ^= z.x & use;
                        acc.y ^= z.y & use;
                        acc.z ^= z.z & use;
                        acc.w ^= z.w & use;
#pragma unroll
                        for (int v4 = 0; v4 * 4 <= w; ++v4) {
                            const uint4 r = row[1 + v4];
                            if (4 * v4 + 0 <= w) q[4 * v4 + 0] ^= r.x & use;
                            if (4 * v4 + 1 <= w) q[4 * v4 + 1] ^= r.y & use;
                            if (4 * v4 + 2 <= w) q[4 * v4 + 2] ^= r.z & use;
                            if (4 * v4 + 3 <= w) q[4 * v4 + 3] ^= r.w & use;
                        }
                    }
                }
            }
            // every pivot bit is now clear; the query is in the span iff
            // nothing is left at the non-pivot coordinates
            uint32_t resid = 0;
#pragma unroll
            for (int v = 0; v < TAB_WD; ++v) resid |= q[v];
            ok = resid == 0;
        }
        // the next item's query ids, descriptor and rank
        int pos_n = 0, len_n = 1;
        int32_t c_n = s.num_ctx;
        unsigned long long en_n = 0;
        CtxDesc cd_n{};
        int rank_n = 0;
        if (nxt < total) {
            unpack(item_n, pos_n, len_n, c_n);
            en_n = __ldg(sorted + pos_n + (lane < len_n ? lane : 0));
            if (c_n < s.num_ctx) {
                cd_n = s.desc[c_n];
                rank_n = s.rank[c_n];
            }
        }
        if (lane < len) {
            if (staged) {
                y[i] = ok ? acc : make_uint4(0, 0, 0, 0);
                in_span[i] = ok ? 1 : 0;
            } else {  // bad ids, contexts wider than the stride or the region
                encode_direct(s, (int32_t)(en >> 32), i, x, stride, y, in_span);
            }
        }
        if (nxt >= total) break;
        __syncwarp();  // the region is rewritten by the next item
        itx = nxt;
        pos = pos_n;
        len = len_n;
        c = c_n;
        en = en_n;
        cd = cd_n;
        rank = rank_n;
    }
}

}  // namespace

extern "C" int f2_encode_batched(const f2_store* st, int64_t Q, const int32_t* ctx_id, const uint32_t* x,
                                 int32_t x_stride_words, uint32_t* y_out, uint8_t* in_span, f2_stream_t stream)
{
    if (!st || Q < 0 || x_stride_words < 1) return F2_ERR_INVALID_ARG;
    if (Q == 0) return F2_OK;
    if (!ctx_id || !x || !y_out || !in_span) return F2_ERR_INVALID_ARG;
    if (((uintptr_t)y_out % 16) != 0 || ((uintptr_t)x % 4) != 0 || ((uintptr_t)ctx_id % 4) != 0)
        return F2_ERR_ALIGN;
    cudaStream_t cs = (cudaStream_t)stream;
    const int64_t sub = Q < ENC_SUB ? Q : ENC_SUB;
    const int64_t N = (int64_t)st->num_ctx + 1;  // buckets (the last for bad ids)
    const int64_t T = (N + SCAN_TILE - 1) / SCAN_TILE;
    // bucket scratch (32-bit words): sizes / starts [N], tile sums and
    // prefixes [T], ticket, item count
    const int64_t bin_words = N + 2 * T + 2;
    cudaError_t e = cudaSuccess;
    // scratch, grown stream-ordered and kept by the store
    if (sub > st->enc_q_cap) {
        if (st->enc_off) cudaFreeAsync(st->enc_off, cs);
        if (st->enc_sorted) cudaFreeAsync(st->enc_sorted, cs);
        if (st->enc_items) cudaFreeAsync(st->enc_items, cs);
        st->enc_off = nullptr;
        st->enc_sorted = nullptr;
        st->enc_items = nullptr;
        st->enc_q_cap = 0;
        e = cudaMallocAsync((void**)&st->enc_off, sizeof(int32_t) * (size_t)sub, cs);
        if (e == cudaSuccess) e = cudaMallocAsync((void**)&st->enc_sorted, sizeof(unsigned long long) * (size_t)sub, cs);
        if (e == cudaSuccess) e = cudaMallocAsync((void**)&st->enc_items, sizeof(unsigned long long) * (size_t)sub, cs);
        if (e != cudaSuccess) return F2_ERR_OOM;
        st->enc_q_cap = sub;
    }
    if (bin_words > st->enc_bin_cap) {
        if (st->enc_bins) cudaFreeAsync(st->enc_bins, cs);
        st->enc_bins = nullptr;
        st->enc_bin_cap = 0;
        if (cudaMallocAsync((void**)&st->enc_bins, sizeof(int32_t) * (size_t)bin_words, cs) != cudaSuccess)
            return F2_ERR_OOM;
        st->enc_bin_cap = bin_words;
    }
    e = cudaFuncSetAttribute(enc_runs_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sizeof(RunSmem));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(enc_short_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)sizeof(ShortSmem));
    if (e != cudaSuccess) return f2_cuda_status(e);
    // enc_short_kernel deals its items round-robin to a grid of one resident wave
    if (st->enc_short_per_sm == 0) {
        int per = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, enc_short_kernel, SHORT_THREADS, sizeof(ShortSmem));
        if (e != cudaSuccess) return f2_cuda_status(e);
        st->enc_short_per_sm = per > 0 ? per : 1;
    }
    const int short_per_sm = st->enc_short_per_sm;
    int32_t* bins = st->enc_bins;
    int32_t* tsum = bins + N;
    int32_t* tpre = tsum + T;
    int32_t* ticket = tpre + T;
    int32_t* n_items = ticket + 1;
    unsigned long long* items = st->enc_items;
    const StoreDev sd = st->dev();
    for (int64_t q0 = 0; q0 < Q; q0 += sub) {
        const int32_t n = (int32_t)((Q - q0) < sub ? (Q - q0) : sub);
        const uint32_t* xq = x + q0 * x_stride_words;
        uint4* yq = reinterpret_cast<uint4*>(y_out) + q0;
        e = cudaMemsetAsync(bins, 0, sizeof(int32_t) * (size_t)N, cs);
        if (e == cudaSuccess) e = cudaMemsetAsync(ticket, 0, 2 * sizeof(int32_t), cs);
        if (e != cudaSuccess) return f2_cuda_status(e);
        enc_count_kernel<<<(n + ENC_TILE - 1) / ENC_TILE, ENC_TILE_THREADS, 0, cs>>>(n, ctx_id + q0, st->num_ctx,
                                                                                   bins, st->enc_off);
        enc_scan_kernel<<<(int)T, SCAN_THREADS, 0, cs>>>(bins, (int32_t)N, tsum, tpre, ticket);
        enc_scatter_kernel<<<(n + SCAT_THREADS * SCAT_PER - 1) / (SCAT_THREADS * SCAT_PER), SCAT_THREADS, 0, cs>>>(
            n, ctx_id + q0, st->num_ctx, bins, tpre, st->enc_off, st->enc_sorted);
        enc_runs_kernel<<<(n + RUN_SEG - 1) / RUN_SEG, RUN_THREADS, sizeof(RunSmem), cs>>>(
            sd, n, st->enc_sorted, xq, x_stride_words, yq, in_span + q0, st->enc_table_min, items, n_items);
        enc_short_kernel<<<st->num_sms * short_per_sm, SHORT_THREADS, sizeof(ShortSmem), cs>>>(
            sd, st->enc_sorted, xq, x_stride_words, yq, in_span + q0, items, n_items);
        e = cudaGetLastError();
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    return F2_OK;
}

namespace {

// Appendix C / D epilogue, one thread per query in query order (coalesced:
// the caller's control and state arrays are in query order too).
constexpr int SC_SHIFT = 105;   // scheduler control: bits 105..121 of the word
constexpr uint32_t SC_MASK = (1u << 17) - 1u;

__global__ void __launch_bounds__(256) epilogue_kernel(int64_t Q, int32_t num_ctx, const int32_t* __restrict__ ctx_id,
                                                       const uint8_t* __restrict__ in_span,
                                                       const uint32_t* __restrict__ sc,
                                                       const uint4* __restrict__ state,
                                                       const uint4* __restrict__ mask, uint4* __restrict__ y)
{
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < Q; q += (int64_t)gridDim.x * blockDim.x) {
        if (__ldg(in_span + q) != 1) continue;
        uint4 w = y[q];
        if (sc) {
            // bits 105..121 = bits 9..25 of word 3
            w.w ^= (__ldg(sc + q) & SC_MASK) << (SC_SHIFT - 96);
        }
        if (state && mask) {
            const int32_t c = __ldg(ctx_id + q);
            if (c >= 0 && c < num_ctx) {
                const uint4 m = __ldg(mask + c), h = __ldg(state + q);
                w.x = (w.x & ~m.x) | (h.x & m.x);
                w.y = (w.y & ~m.y) | (h.y & m.y);
                w.z = (w.z & ~m.z) | (h.z & m.z);
                w.w = (w.w & ~m.w) | (h.w & m.w);
            }
        }
        y[q] = w;
    }
}

}  // namespace

extern "C" int f2_encode_epilogue(const f2_store* st, int64_t Q, const int32_t* ctx_id, const uint8_t* in_span,
                                  const uint32_t* sc, const uint32_t* state, const uint32_t* opaque_mask,
                                  uint32_t* y, f2_stream_t stream)
{
    if (!st || Q < 0) return F2_ERR_INVALID_ARG;
    if (Q == 0) return F2_OK;
    if (!y || !in_span || !ctx_id) return F2_ERR_INVALID_ARG;
    if (((uintptr_t)y % 16) != 0 || ((uintptr_t)state % 16) != 0 || ((uintptr_t)opaque_mask % 16) != 0)
        return F2_ERR_ALIGN;
    int64_t blocks = (Q + 255) / 256;
    if (blocks > (int64_t)st->num_sms * 16) blocks = (int64_t)st->num_sms * 16;
    epilogue_kernel<<<(int)blocks, 256, 0, (cudaStream_t)stream>>>(
        Q, st->num_ctx, ctx_id, in_span, sc, reinterpret_cast<const uint4*>(state),
        reinterpret_cast<const uint4*>(opaque_mask), reinterpret_cast<uint4*>(y));
    return f2_cuda_status(cudaGetLastError());
}

int f2_encode_table_min_default() { return DEFAULT_TABLE_MIN; }
int f2_encode_table_min_floor() { return RUN_SEG / MAX_TRUNS; }
