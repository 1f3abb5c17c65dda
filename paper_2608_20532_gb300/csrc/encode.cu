// Batched encoding with a span check (Sec. 2.3, Appendix B) on sm_103a.
//
// q = phi(x) is reduced against its context's reduced basis; every stored row
// used also XORs its z_k into a zero accumulator.  Because the basis is
// reduced, the rows to use are exactly the pivots set in q itself.  A zero
// residual at the non-pivot coordinates proves q in the span and the accumulator
// is the word; otherwise the query is rejected and the word is zero.
//
// The queries are first grouped by context (pass 1 below); every context
// with many queries gets a lookup table of its basis, built once per pass in
// a pool, and its runs of queries are encoded from that table after a bulk
// asynchronous copy into shared memory; the other queries are encoded by a
// per-query walk over the pivot rows staged in shared memory (pass 2).
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
// Pass 1: group the queries (a counting sort; the order of the queries inside
// a bucket is arbitrary, since every query's result depends only on the
// query).  Ids outside [0, num_ctx) go to the extra bucket num_ctx.
//
// A bucket is (chunk, context), a chunk being 2^shift consecutive queries.
// The contexts that get a lookup table in this pass ("table contexts", at
// least table_min queries) are laid out chunk-major: the encoding of a chunk
// then reads and writes a window of the query arrays small enough to stay in
// L2, so the words and flags scattered back to query order merge into whole
// sectors there instead of costing a DRAM read-modify-write each.  Every
// other context keeps its queries of all chunks together (after the table
// contexts), so its basis is staged once.
//
//   enc_count_kernel   a CTA counts ENC_TILE queries (inside one chunk) per
//                      context in a shared-memory hash table, claims each
//                      context's share of its bucket with one global atomic,
//                      and writes every query's offset inside its bucket;
//   enc_table_kernel   per context: total over the chunks; a table context
//                      gets a slot in the store's table pool and its table
//                      is built there (one warp); writes the scan input (the
//                      chunk counts of table contexts, chunk-major, then the
//                      totals of the others) and, for the others, turns the
//                      chunk counts into their prefix over the chunks;
//   enc_scan_kernel    exclusive prefix of the scan input: per tile of
//                      SCAN_TILE entries, then the tile totals (by the last
//                      CTA to finish);
//   enc_scatter_kernel writes (context, query) to its grouped position.
// ---------------------------------------------------------------------------
constexpr int ENC_TILE = 2048;
constexpr int ENC_TILE_THREADS = 256;
constexpr int ENC_TILE_PER = ENC_TILE / ENC_TILE_THREADS;
constexpr int ENC_HT_BITS = 12;
constexpr int ENC_HT = 1 << ENC_HT_BITS;
static_assert(ENC_HT >= 2 * ENC_TILE, "hash table of a tile at most half full");
constexpr int SCAN_THREADS = 1024;
constexpr int SCAN_SHIFT = 12;
constexpr int SCAN_TILE = 1 << SCAN_SHIFT;  // 4 entries per thread
constexpr int SCAT_THREADS = 256;
constexpr int SCAT_PER = 4;
constexpr int64_t ENC_SUB = int64_t(1) << 25;   // queries grouped per pass
constexpr int ENC_MAX_CHUNKS = 64;              // chunks of a pass (the chunk grows with the pass)
constexpr int ENC_MIN_SHIFT = 11;               // a count tile lies inside one chunk
constexpr int DEFAULT_CHUNK_SHIFT = 20;
constexpr int32_t EMPTY_KEY = -1;
constexpr int TBL_THREADS = 256;
constexpr uint8_t HOT_TABLE = 1;    // the context's runs are encoded with its table
constexpr uint8_t HOT_CHUNKED = 2;  // the context's queries are laid out chunk by chunk
constexpr int64_t DEFAULT_CHUNK_MIN = 512;
constexpr int64_t POOL_MAX_WORDS = int64_t(1) << 28;  // table pool cap (1 GiB)
static_assert(ENC_TILE <= (1 << ENC_MIN_SHIFT), "count tiles never straddle a chunk");

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
                                                                     int32_t num_ctx, int shift, int32_t B,
                                                                     int32_t* __restrict__ cnt,
                                                                     int32_t* __restrict__ off)
{
    __shared__ int32_t key[ENC_HT];
    __shared__ int32_t hcnt[ENC_HT];
    const int t = threadIdx.x, lane = t & 31;
    const int64_t base = (int64_t)blockIdx.x * ENC_TILE;
    int32_t* const bins = cnt + (int64_t)(base >> shift) * B;  // the tile's chunk
    int32_t bk[ENC_TILE_PER];
#pragma unroll
    for (int j = 0; j < ENC_TILE_PER; ++j) {  // all loads first
        const int64_t i = base + (int64_t)j * ENC_TILE_THREADS + t;
        bk[j] = (i < Q) ? bucket_of(__ldg(ctx_id + i), num_ctx) : EMPTY_KEY;
    }
    for (int h = t; h < ENC_HT; h += ENC_TILE_THREADS) {
        key[h] = EMPTY_KEY;
        hcnt[h] = 0;
    }
    __syncthreads();
    const uint32_t below = (1u << lane) - 1u;
    uint32_t peers[ENC_TILE_PER];
    uint32_t slot[ENC_TILE_PER];
    int32_t prev[ENC_TILE_PER];
    bool lead[ENC_TILE_PER];
#pragma unroll
    for (int j = 0; j < ENC_TILE_PER; ++j) {
        peers[j] = __match_any_sync(FULL, bk[j]);
        lead[j] = lane == __ffs(peers[j]) - 1 && bk[j] != EMPTY_KEY;
        slot[j] = ((uint32_t)bk[j] * 2654435761u) >> (32 - ENC_HT_BITS);
    }
    // The first probe of every group is issued before any is resolved: at
    // most half of the table is used, so most groups are placed by it.
#pragma unroll
    for (int j = 0; j < ENC_TILE_PER; ++j) prev[j] = lead[j] ? atomicCAS(&key[slot[j]], EMPTY_KEY, bk[j]) : EMPTY_KEY;
#pragma unroll
    for (int j = 0; j < ENC_TILE_PER; ++j) {
        if (lead[j]) {
            // at most ENC_TILE distinct keys in ENC_HT slots: a free or
            // matching slot is always found within ENC_HT probes
            for (int probe = 1; probe < ENC_HT && prev[j] != EMPTY_KEY && prev[j] != bk[j]; ++probe) {
                slot[j] = (slot[j] + 1) & (ENC_HT - 1);
                prev[j] = atomicCAS(&key[slot[j]], EMPTY_KEY, bk[j]);
            }
        }
    }
    int r0[ENC_TILE_PER];
#pragma unroll
    for (int j = 0; j < ENC_TILE_PER; ++j) r0[j] = lead[j] ? atomicAdd(&hcnt[slot[j]], __popc(peers[j])) : 0;
    int rank[ENC_TILE_PER];
#pragma unroll
    for (int j = 0; j < ENC_TILE_PER; ++j) {
        const int leader = __ffs(peers[j]) - 1;
        slot[j] = __shfl_sync(FULL, slot[j], leader);
        rank[j] = __shfl_sync(FULL, r0[j], leader) + __popc(peers[j] & below);
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
        got[u] = (k != EMPTY_KEY) ? atomicAdd(bins + k, hcnt[h]) : 0;
    }
    __syncthreads();
#pragma unroll
    for (int u = 0; u < HPER; ++u) hcnt[u * ENC_TILE_THREADS + t] = got[u];
    __syncthreads();
#pragma unroll
    for (int j = 0; j < ENC_TILE_PER; ++j) {
        const int64_t i = base + (int64_t)j * ENC_TILE_THREADS + t;
        if (i < Q) off[i] = hcnt[slot[j]] + rank[j];
    }
}

// ---------------------------------------------------------------------------
// Lookup tables of the basis (layout and meaning in f2_internal.cuh), built
// once per pass for the contexts with many queries.
// ---------------------------------------------------------------------------
constexpr int TAB_WD = TABLE_MAX_WD;          // widest context with a table (d <= 288)
constexpr int TAB_RW = TABLE_MAX_RW;          // compressed residual words (m <= 128)
constexpr int TAB_WORDS = 6144;               // largest table (24 KB): one of two table buffers
constexpr int DEFAULT_TABLE_MIN = 64;

// E_j of context cd: word part z, compressed residual er.  The pivot words,
// z_j and r_j are loaded together (slots of non-pivots hold zeros), so an
// entry costs one round of loads.
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

// One warp writes block blk (coordinates 32*blk .. 32*blk + 31, i.e. eight
// groups) of the table of context c to `tab` (global memory).  Lane l
// computes E_j for j = 32*blk + l; the four lanes of a quad hold the four
// coordinates of one group and each writes four of its 16 entries (entry v
// = XOR of E_{4p+b} over the bits b of v).
__device__ void build_table(const StoreDev& s, int c, int blk, uint32_t* __restrict__ tab, int lane)
{
    const CtxDesc cd = s.desc[c];
    const int rank = s.rank[c];
    const int np = (cd.d + 3) >> 2, rw = (cd.d - rank + 31) >> 5;
    uint2* const Zl = reinterpret_cast<uint2*>(tab);
    uint2* const Zh = Zl + 16 * np;
    uint32_t* const R = tab + 64 * np;
    const int qb = lane & ~3, b = lane & 3;
    {
        const int j = 32 * blk + lane;
        uint4 z;
        uint32_t er[TAB_RW];
        single_entry(s, cd, j, z, er);
        uint4 zs[4];
        uint32_t es[4][TAB_RW];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            zs[k].x = __shfl_sync(FULL, z.x, qb + k);
            zs[k].y = __shfl_sync(FULL, z.y, qb + k);
            zs[k].z = __shfl_sync(FULL, z.z, qb + k);
            zs[k].w = __shfl_sync(FULL, z.w, qb + k);
#pragma unroll
            for (int u = 0; u < TAB_RW; ++u) es[k][u] = __shfl_sync(FULL, er[u], qb + k);
        }
        if (j < 4 * np) {
            // entries v = 4b .. 4b+3 of group p: 32 contiguous bytes per z
            // plane and 16 per residual plane, written as whole 16-byte stores
            const int p = j >> 2;
            uint4 a[4];
            uint32_t ra[4][TAB_RW];
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                const int v = 4 * b + m;
                a[m] = make_uint4(0, 0, 0, 0);
#pragma unroll
                for (int u = 0; u < TAB_RW; ++u) ra[m][u] = 0;
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    if ((v >> k) & 1) {
                        a[m].x ^= zs[k].x;
                        a[m].y ^= zs[k].y;
                        a[m].z ^= zs[k].z;
                        a[m].w ^= zs[k].w;
#pragma unroll
                        for (int u = 0; u < TAB_RW; ++u) ra[m][u] ^= es[k][u];
                    }
                }
            }
            const int e = 16 * p + 4 * b;
            uint4* zl = reinterpret_cast<uint4*>(Zl + e);
            uint4* zh = reinterpret_cast<uint4*>(Zh + e);
            zl[0] = make_uint4(a[0].x, a[0].y, a[1].x, a[1].y);
            zl[1] = make_uint4(a[2].x, a[2].y, a[3].x, a[3].y);
            zh[0] = make_uint4(a[0].z, a[0].w, a[1].z, a[1].w);
            zh[1] = make_uint4(a[2].z, a[2].w, a[3].z, a[3].w);
#pragma unroll
            for (int u = 0; u < TAB_RW; ++u)
                if (u < rw)
                    *reinterpret_cast<uint4*>(R + u * 16 * np + e) = make_uint4(ra[0][u], ra[1][u], ra[2][u], ra[3][u]);
        }
    }
}

// Per bucket b (a thread; consecutive buckets, so the chunk counts are read
// coalesced): its total over the chunks; table or not (a slot in the pool,
// claimed once per warp); the scan input; the table contexts are listed for
// enc_build_kernel.
__global__ void __launch_bounds__(TBL_THREADS) enc_table_kernel(StoreDev s, int32_t nch, int32_t B,
                                                                int32_t* __restrict__ cnt,
                                                                int32_t* __restrict__ scan_in,
                                                                uint8_t* __restrict__ hot,
                                                                long long* __restrict__ tab_off,
                                                                long long pool_words,
                                                                unsigned long long* __restrict__ pool_used,
                                                                int32_t* __restrict__ hot_list,
                                                                int32_t* __restrict__ n_hot, int table_min,
                                                                long long chunk_min, int stride)
{
    const int lane = threadIdx.x & 31;
    for (int c0 = (int)((blockIdx.x * (unsigned)TBL_THREADS + threadIdx.x) & ~31u); c0 < B;
         c0 += (int)(gridDim.x * (unsigned)TBL_THREADS)) {
        const int c = c0 + lane;
        int tot = 0, words = 0;
        if (c < B)
            for (int ch = 0; ch < nch; ++ch) tot += cnt[(int64_t)ch * B + c];
        if (c < s.num_ctx && tot >= table_min) {
            const CtxDesc cd = s.desc[c];
            const int rk = s.rank[c];
            const int w = table_words(cd.d, rk);
            const int rw = (cd.d - rk + 31) >> 5;
            if (cd.wd <= TAB_WD && cd.xw <= stride && rw <= TAB_RW && w <= TAB_WORDS) words = w;
        }
        // one pool claim and one list claim per warp
        int incl = words;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int u = __shfl_up_sync(FULL, incl, o);
            if (lane >= o) incl += u;
        }
        const int wsum = __shfl_sync(FULL, incl, 31);
        unsigned long long wbase = 0;
        if (lane == 31 && wsum) wbase = atomicAdd(pool_used, (unsigned long long)wsum);
        wbase = __shfl_sync(FULL, wbase, 31);
        const long long o = (long long)wbase + incl - words;
        const bool h = words > 0 && o + words <= pool_words;
        // the table's blocks of 32 coordinates are listed for enc_build_kernel
        const int nb = h ? (((s.desc[c].d + 3) >> 2) * 4 + 31) >> 5 : 0;
        int binc = nb;
#pragma unroll
        for (int o2 = 1; o2 < 32; o2 <<= 1) {
            const int u = __shfl_up_sync(FULL, binc, o2);
            if (lane >= o2) binc += u;
        }
        const int bsum = __shfl_sync(FULL, binc, 31);
        int lbase = 0;
        if (lane == 31 && bsum) lbase = atomicAdd(n_hot, bsum);
        lbase = __shfl_sync(FULL, lbase, 31);
        for (int k = 0; k < nb; ++k) hot_list[lbase + binc - nb + k] = (int32_t)(((uint32_t)c << 4) | (uint32_t)k);
        if (c < B) {
            const bool chunked = c < s.num_ctx && (long long)tot >= chunk_min;
            hot[c] = (h ? HOT_TABLE : 0) | (chunked ? HOT_CHUNKED : 0);
            tab_off[c] = h ? o : -1;
            if (chunked) {
                for (int ch = 0; ch < nch; ++ch) scan_in[(int64_t)ch * B + c] = cnt[(int64_t)ch * B + c];
                scan_in[(int64_t)nch * B + c] = 0;
            } else {
                int run = 0;
                for (int ch = 0; ch < nch; ++ch) {
                    const int v = cnt[(int64_t)ch * B + c];
                    scan_in[(int64_t)ch * B + c] = 0;
                    cnt[(int64_t)ch * B + c] = run;  // the bucket's queries before chunk ch
                    run += v;
                }
                scan_in[(int64_t)nch * B + c] = tot;
            }
        }
    }
}

// A warp per listed (table context, block of 32 coordinates) builds that
// part of the context's table in the pool.
__global__ void __launch_bounds__(TBL_THREADS) enc_build_kernel(StoreDev s, const int32_t* __restrict__ hot_list,
                                                                const int32_t* __restrict__ n_hot,
                                                                const long long* __restrict__ tab_off,
                                                                uint32_t* __restrict__ pool)
{
    const int lane = threadIdx.x & 31;
    const int nh = *n_hot;
    const int nw = (int)((gridDim.x * (unsigned)TBL_THREADS) >> 5);
    for (int k = (int)((blockIdx.x * (unsigned)TBL_THREADS + threadIdx.x) >> 5); k < nh; k += nw) {
        const uint32_t item = (uint32_t)__ldg(hot_list + k);
        const int c = (int)(item >> 4);
        build_table(s, c, (int)(item & 15u), pool + __ldg(tab_off + c), lane);
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

__device__ __forceinline__ int32_t scan_start(const int32_t* __restrict__ sta, const int32_t* __restrict__ tpre,
                                              int64_t k)
{
    return __ldg(sta + k) + __ldg(tpre + (k >> SCAN_SHIFT));
}

__global__ void __launch_bounds__(SCAT_THREADS) enc_scatter_kernel(int32_t Q, const int32_t* __restrict__ ctx_id,
                                                                   int32_t num_ctx, int shift, int32_t nch, int32_t B,
                                                                   const int32_t* __restrict__ cnt,
                                                                   const int32_t* __restrict__ sta,
                                                                   const int32_t* __restrict__ tpre,
                                                                   const uint8_t* __restrict__ hot,
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
        const int64_t i = base + (int64_t)j * SCAT_THREADS;
        const int bb = b[j] < 0 ? 0 : b[j];
        const int64_t ch = i >> shift;
        if (__ldg(hot + bb) & HOT_CHUNKED)
            p[j] = scan_start(sta, tpre, ch * B + bb) + o[j];
        else
            p[j] = scan_start(sta, tpre, (int64_t)nch * B + bb) + __ldg(cnt + ch * B + bb) + o[j];
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
// RUN_TABLE_MIN queries of a table context is encoded with its table: the
// CTA copies the tables of its runs from the pool into shared memory with
// bulk asynchronous copies (two buffers: the next group of tables is in
// flight while the queries of the current group are looked up).  The other
// runs are cut into items of at most 32 queries for enc_short_kernel.
//
// enc_short_kernel: a warp per item stages the context's pivot rows in its
// shared-memory region with asynchronous copies, then every lane reduces its
// query against them in a warp-uniform walk over the pivots.
// ---------------------------------------------------------------------------
constexpr int RUN_THREADS = 512;  // two CTAs per SM: 32 warps
constexpr int RUN_SEG = 2048;
constexpr int RUN_PER = RUN_SEG / RUN_THREADS;
constexpr int MAX_TRUNS = 128;                // table runs of a segment (the rest become items)
constexpr int RUN_TABLE_MIN = 4;              // shorter runs of a table context become items
constexpr int XS_WORDS = 4;                   // feature words of a table query staged in shared memory
constexpr int ITEM_MAX = 32;                  // queries of a short item (one per lane)
constexpr int ITEM_POS_BITS = 25;             // item = position | (length - 1) << 25
static_assert(ENC_SUB <= (int64_t(1) << ITEM_POS_BITS), "item positions fit 25 bits");

struct RunSmem {
    uint4 table[2][TAB_WORDS / 4];     // two table buffers
    uint4 xs[RUN_SEG];                 // first XS_WORDS feature words of each table query (flat order);
                                       // until they are staged, its first RUN_SEG words hold each run's context
    uint32_t idx[RUN_SEG];             // query index of each position
    uint32_t flat[RUN_SEG];            // table positions in order: position | table run << 16
    uint16_t starts[RUN_SEG + 1];      // run starts
    int16_t run_tr[RUN_SEG];           // table run of each run, -1 if none
    long long tr_src[MAX_TRUNS];       // word offset of the run's table in the pool
    int32_t tr_tab[MAX_TRUNS];         // word offset of the run's table in its buffer
    int32_t tr_words[MAX_TRUNS];
    int32_t tr_flat[MAX_TRUNS + 1];    // first flat index of the run
    int16_t tr_n[MAX_TRUNS];           // feature bits of the run's context
    uint8_t tr_np[MAX_TRUNS];
    uint8_t tr_rw[MAX_TRUNS];
    uint8_t tr_xw[MAX_TRUNS];
    int32_t g_first[MAX_TRUNS + 1];
    uint8_t g_xw[MAX_TRUNS];           // widest feature vector of the group's runs
    unsigned long long bar[2];         // completion of the copies into table[0] / table[1]
    int32_t ws[RUN_THREADS / 32 + 1];
    int32_t n_groups;
    int32_t item_base;
    int32_t failed;
};
static_assert(sizeof(RunSmem) + 1024 <= 233472 / 2, "two CTAs of enc_runs_kernel per SM");
static_assert(offsetof(RunSmem, table) % 16 == 0 && offsetof(RunSmem, xs) % 16 == 0 &&
                  offsetof(RunSmem, bar) % 8 == 0,
              "aligned buffers");

__device__ __forceinline__ void encode_direct(const StoreDev& s, int32_t c, int64_t i, const uint32_t* __restrict__ x,
                                              int stride, uint4* __restrict__ y, uint8_t* __restrict__ in_span)
{
    uint4 acc = make_uint4(0, 0, 0, 0);
    uint8_t flag;
    if ((uint32_t)c >= (uint32_t)s.num_ctx) {
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
            if (4 * v4 < xw) p = __ldcs(reinterpret_cast<const uint4*>(xq) + v4);
            const uint32_t w[4] = {p.x, p.y, p.z, p.w};
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (4 * v4 + u < XW) xo[4 * v4 + u] = (4 * v4 + u < xw) ? w[u] : 0u;
        }
    } else {
#pragma unroll
        for (int v = 0; v < XW; ++v) xo[v] = (v < xw) ? __ldcs(xq + v) : 0u;
    }
}

template <int RW, int WD>
__device__ __forceinline__ bool table_query(const uint32_t* tab, int np, uint32_t (&q)[WD], uint4& acc)
{
    uint32_t r[RW > 0 ? RW : 1];
    table_reduce<RW, WD>(tab, np, q, acc, r);
    uint32_t res = 0;
#pragma unroll
    for (int u = 0; u < RW; ++u) res |= r[u];
    return res == 0;
}

// Encode the queries at flat positions [fa, fb) of a segment with their
// runs' tables; the first XS_WORDS feature words of each are in sm.xs.
template <int WD>
__device__ __forceinline__ void query_group(const StoreDev& s, const RunSmem& sm, const uint32_t* table,
                                            const uint32_t* __restrict__ x, int stride, uint4* __restrict__ y,
                                            uint8_t* __restrict__ in_span, int fa, int fb)
{
    for (int f = fa + (int)threadIdx.x; f < fb; f += RUN_THREADS) {
        const uint32_t fv = sm.flat[f];
        const int tr = (int)(fv >> 16);
        const int64_t i = (int64_t)sm.idx[fv & 0xFFFFu];
        const int xw = sm.tr_xw[tr];
        const uint4 p = sm.xs[f];
        const uint32_t w4[4] = {p.x, p.y, p.z, p.w};
        uint32_t raw[WD];
#pragma unroll
        for (int v = 0; v < WD; ++v) {
            if (v < XS_WORDS) raw[v] = (v < xw) ? w4[v] : 0u;
            else raw[v] = (v < xw) ? __ldcs(x + i * stride + v) : 0u;
        }
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
                                                                  uint8_t* __restrict__ in_span,
                                                                  const uint8_t* __restrict__ hot,
                                                                  const long long* __restrict__ tab_off,
                                                                  const uint32_t* __restrict__ pool,
                                                                  unsigned long long* __restrict__ items,
                                                                  int32_t* __restrict__ n_items)
{
    extern __shared__ uint4 enc_smem[];
    RunSmem& sm = *reinterpret_cast<RunSmem*>(enc_smem);
    int32_t* const run_ctx = reinterpret_cast<int32_t*>(sm.xs);  // until the feature words are staged
    const int t = threadIdx.x;
    const bool xvec = ((uintptr_t)x % 16) == 0 && (stride % 4) == 0;
    const int64_t seg0 = (int64_t)blockIdx.x * RUN_SEG;
    const int n = (int)((n_total - seg0) < RUN_SEG ? (n_total - seg0) : RUN_SEG);
    if (t == 0) {
        mbar_init(&sm.bar[0], 1);
        mbar_init(&sm.bar[1], 1);
        mbar_init_fence();
        sm.failed = 0;
    }
    // this thread's positions: contexts in registers, query indices to smem
    const int k0 = t * RUN_PER;
    uint32_t cx[RUN_PER];
    uint32_t prev = 0xFFFFFFFFu;
    if (k0 > 0 && k0 <= n) prev = (uint32_t)(__ldcs(sorted + seg0 + k0 - 1) >> 32);
#pragma unroll
    for (int m = 0; m < RUN_PER; ++m) {
        const int k = k0 + m;
        cx[m] = 0xFFFFFFFFu;
        if (k < n) {
            const unsigned long long e = __ldcs(sorted + seg0 + k);
            cx[m] = (uint32_t)(e >> 32);
            sm.idx[k] = (uint32_t)e;
        }
    }
    // runs: flag the first position of each run, number the runs
    uint32_t first = 0;
    int nflag = 0;
#pragma unroll
    for (int m = 0; m < RUN_PER; ++m) {
        if (k0 + m < n) {
            if (k0 + m == 0 || cx[m] != prev) {
                first |= 1u << m;
                ++nflag;
            }
            prev = cx[m];
        }
    }
    int n_runs;
    const int r0 = block_exclusive_scan<RUN_THREADS>(nflag, sm.ws, n_runs);
    {
        int r = r0;
#pragma unroll
        for (int m = 0; m < RUN_PER; ++m)
            if ((first >> m) & 1u) {
                sm.starts[r] = (uint16_t)(k0 + m);
                run_ctx[r++] = (int32_t)cx[m];
            }
        if (t == 0) sm.starts[n_runs] = (uint16_t)n;
    }
    __syncthreads();

    // classify the runs, RUN_THREADS at a time: number the table runs (in
    // position order; those past MAX_TRUNS become items), count the items
    int n_tr = 0, n_it = 0, my_base = 0;
    for (int c0 = 0; c0 < n_runs; c0 += RUN_THREADS) {
        const int rr = c0 + t;
        int nel = 0, len = 0;
        int32_t c = s.num_ctx;
        if (rr < n_runs) {
            len = (int)sm.starts[rr + 1] - (int)sm.starts[rr];
            c = run_ctx[rr];
            nel = (c < s.num_ctx && len >= RUN_TABLE_MIN && (__ldg(hot + c) & HOT_TABLE)) ? 1 : 0;
        }
        int tot;
        const int ex = block_exclusive_scan<RUN_THREADS>(nel, sm.ws, tot);
        if (rr < n_runs) {
            const int tr = n_tr + ex;
            if (nel && tr < MAX_TRUNS) {
                const CtxDesc cd = s.desc[c];
                const int rk = s.rank[c];
                sm.run_tr[rr] = (int16_t)tr;
                sm.tr_np[tr] = (uint8_t)((cd.d + 3) >> 2);
                sm.tr_rw[tr] = (uint8_t)((cd.d - rk + 31) >> 5);
                sm.tr_xw[tr] = (uint8_t)cd.xw;
                sm.tr_n[tr] = (int16_t)cd.n;
                sm.tr_words[tr] = table_words(cd.d, rk);
                sm.tr_src[tr] = __ldg(tab_off + c);
            } else {
                sm.run_tr[rr] = -1;
                n_it += (len + ITEM_MAX - 1) / ITEM_MAX;  // this thread's items
            }
        }
        n_tr += tot;
    }
    if (n_tr > MAX_TRUNS) n_tr = MAX_TRUNS;
    {
        int tot_it;
        (void)block_exclusive_scan<RUN_THREADS>(n_it, sm.ws, tot_it);
        n_it = tot_it;
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
                // greedy groups of consecutive table runs that fit one buffer
                int g = 0, used = 0, gx = 0;
                sm.g_first[0] = 0;
                for (int tr = 0; tr < n_tr; ++tr) {
                    const int words = sm.tr_words[tr];
                    if (used + words > TAB_WORDS) {
                        sm.g_xw[g] = (uint8_t)gx;
                        sm.g_first[++g] = tr;
                        used = gx = 0;
                    }
                    gx = gx > sm.tr_xw[tr] ? gx : sm.tr_xw[tr];
                    sm.tr_tab[tr] = used;
                    used += words;
                }
                sm.g_xw[g] = (uint8_t)gx;
                sm.g_first[++g] = n_tr;
                sm.n_groups = g;
            }
        }
        __syncthreads();

        const int n_groups = sm.n_groups;
        // thread 0 copies the tables of group g into buffer g & 1
        auto issue = [&](int g) {
            const int ga = sm.g_first[g], gb = sm.g_first[g + 1];
            uint32_t bytes = 0;
            for (int tr = ga; tr < gb; ++tr) bytes += 4u * (uint32_t)sm.tr_words[tr];
            unsigned long long* bar = &sm.bar[g & 1];
            uint32_t* buf = reinterpret_cast<uint32_t*>(sm.table[g & 1]);
            const unsigned long long keep = l2_policy_evict_last();  // tables are read by many CTAs
            fence_proxy_async_smem();
            mbar_arrive_expect_tx(bar, bytes);
            for (int tr = ga; tr < gb; ++tr)
                bulk_copy_g2s_hint(buf + sm.tr_tab[tr], pool + sm.tr_src[tr], 4u * (uint32_t)sm.tr_words[tr], bar,
                                   keep);
        };
        if (t == 0) issue(0);
        // the first feature words of every table query, beside the copies
        {
            const int n_flat = sm.tr_flat[n_tr];
            uint32_t* xsw = reinterpret_cast<uint32_t*>(sm.xs);
            for (int f = t; f < n_flat; f += RUN_THREADS) {
                const uint32_t fv = sm.flat[f];
                const int64_t i = (int64_t)sm.idx[fv & 0xFFFFu];
                const uint32_t* src = x + i * stride;
                if (xvec) {
                    cp_async16(sm.xs + f, src);  // stride >= 4 words: inside the row
                } else {
                    const int xw = sm.tr_xw[fv >> 16];
                    for (int v = 0; v < XS_WORDS && v < xw; ++v) cp_async4(xsw + 4 * f + v, src + v);
                }
            }
            cp_async_commit();
        }
        int fail_g = -1;
        for (int g = 0; g < n_groups; ++g) {
            if (t == 0 && g + 1 < n_groups) issue(g + 1);
            if (g == 0) cp_async_wait_all();
            const bool ok = mbar_wait_bounded(&sm.bar[g & 1], (uint32_t)((g >> 1) & 1));
            if (!ok) sm.failed = 1;
            __syncthreads();
            if (sm.failed) {
                fail_g = g;
                break;
            }
            const uint32_t* table = reinterpret_cast<const uint32_t*>(sm.table[g & 1]);
            const int fa = sm.tr_flat[sm.g_first[g]], fb = sm.tr_flat[sm.g_first[g + 1]];
            if (sm.g_xw[g] <= 4)
                query_group<5>(s, sm, table, x, stride, y, in_span, fa, fb);
            else
                query_group<TAB_WD>(s, sm, table, x, stride, y, in_span, fa, fb);
            __syncthreads();
        }
        if (fail_g >= 0) {
            // a copy did not complete in time: record it, then let the copies
            // still in flight land before the CTA's shared memory is released
            if (t == 0) record_status(s.status, F2_ERR_TIMEOUT);
            for (int g = fail_g; g < n_groups && g <= fail_g + 1; ++g)
                (void)mbar_wait_bounded(&sm.bar[g & 1], (uint32_t)((g >> 1) & 1));
            return;
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
            c = (uint32_t)(__ldg(sorted + seg0 + a) >> 32);
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

// A warp per item (round robin over a grid of one resident wave).  The loads
// that do not depend on an item's basis (the item, its queries, the
// context's descriptor, rank and pivot words) run one item ahead; the basis
// rows themselves are fetched by asynchronous copies issued together, with
// the query's feature words and the next item's pivot words in flight
// beside them.
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
    // An item is (position | (length - 1) << 25, context).
    auto unpack = [&](unsigned long long it, int& pos, int& len, int32_t& c) {
        pos = (int)(it & ((1u << ITEM_POS_BITS) - 1u));
        len = (int)((it >> ITEM_POS_BITS) & 31u) + 1;
        c = (int32_t)(it >> 32);
    };
    int itx = blockIdx.x * SHORT_WARPS + wid;
    if (itx >= total) return;
    int pos, len;
    int32_t c;
    unpack(__ldg(items + itx), pos, len, c);
    unsigned long long en = __ldg(sorted + pos + (lane < len ? lane : 0));
    CtxDesc cd{};
    int rank = 0;
    if (c < s.num_ctx) {
        cd = s.desc[c];
        rank = s.rank[c];
    }
    uint32_t pw = (c < s.num_ctx && lane < cd.wd) ? __ldg(s.pivot + cd.pw_off + lane) : 0u;
    unsigned long long item_n = (itx + nwarps < total) ? __ldg(items + itx + nwarps) : 0ull;
    while (true) {
        const int nxt = itx + nwarps;
        // the next item's queries, descriptor and rank (its item word is in)
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
        const unsigned long long item_nn = (nxt + nwarps < total) ? __ldg(items + nxt + nwarps) : 0ull;

        const int64_t i = (int64_t)(uint32_t)en;
        const int rs = row_stride(cd.wd);  // staged row: [z_k | r_k], 16-byte aligned
        const bool staged = c < s.num_ctx && cd.wd <= TAB_WD && cd.xw <= stride && rank * rs <= SHORT_REGION;
        uint32_t xr[TAB_WD];
        if (staged) {
            // pivot list, word by word
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
            // the pivot rows: z_k by one 16-byte copy, r_k word by word
            for (int idx = lane; idx < rank; idx += 32)
                cp_async16(region + idx * rs, s.bz + cd.slot_off + piv[idx]);
            {
                const int wd = cd.wd;
                int idx = lane / wd, v = lane - (lane / wd) * wd;
                const int di = 32 / wd, dv = 32 - di * wd;
                for (int u = lane; u < rank * wd; u += 32) {
                    cp_async4(region + idx * rs + 4 + v, s.bx + cd.xw_off + (int64_t)piv[idx] * wd + v);
                    idx += di;
                    v += dv;
                    if (v >= wd) {
                        v -= wd;
                        ++idx;
                    }
                }
            }
            cp_async_commit();
            load_x<TAB_WD>(x + i * stride, lane < len ? cd.xw : 0, xvec, xr);
        }
        // the next item's pivot words, beside this item's copies
        const uint32_t pw_n =
            (nxt < total && c_n < s.num_ctx && lane < cd_n.wd) ? __ldg(s.pivot + cd_n.pw_off + lane) : 0u;
        uint4 acc = make_uint4(0, 0, 0, 0);
        bool ok = false;
        if (staged) {
            cp_async_wait_all();
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
        if (lane < len) {
            if (staged) {
                y[i] = ok ? acc : make_uint4(0, 0, 0, 0);
                in_span[i] = ok ? 1 : 0;
            } else {  // bad ids, contexts wider than the stride or the region
                encode_direct(s, (int32_t)(en >> 32), i, x, stride, y, in_span);
            }
        }
        if (nxt >= total) break;
        __syncwarp();  // the region and pivot list are rewritten by the next item
        itx = nxt;
        pos = pos_n;
        len = len_n;
        c = c_n;
        en = en_n;
        cd = cd_n;
        rank = rank_n;
        pw = pw_n;
        item_n = item_nn;
    }
}

// A small pass: every query on its own, its basis rows read from the store
// (L2), no grouping -- one launch where the grouped path takes eight, which
// is what a small batch waits for.
__global__ void __launch_bounds__(256) enc_direct_kernel(StoreDev s, int32_t n, const int32_t* __restrict__ ctx_id,
                                                         const uint32_t* __restrict__ x, int stride,
                                                         uint4* __restrict__ y, uint8_t* __restrict__ in_span)
{
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
        encode_direct(s, __ldg(ctx_id + i), i, x, stride, y, in_span);
}

}  // namespace

extern "C" int f2_encode_batched(const f2_store* st, int64_t Q, const int32_t* ctx_id, const uint32_t* x,
                                 int32_t x_stride_words, uint32_t* y_out, uint8_t* in_span, f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_encode_batched");
    if (!st || Q < 0 || x_stride_words < 1) return F2_ERR_INVALID_ARG;
    if (Q == 0) return F2_OK;
    if (!ctx_id || !x || !y_out || !in_span) return F2_ERR_INVALID_ARG;
    if (((uintptr_t)y_out % 16) != 0 || ((uintptr_t)x % 4) != 0 || ((uintptr_t)ctx_id % 4) != 0)
        return F2_ERR_ALIGN;
    cudaStream_t cs = (cudaStream_t)stream;
    if (Q <= st->enc_direct_max) {  // a small pass: no grouping, no scratch
        int blocks = (int)((Q + 255) / 256);
        if (blocks > 8 * st->num_sms) blocks = 8 * st->num_sms;
        enc_direct_kernel<<<blocks, 256, 0, cs>>>(st->dev(), (int32_t)Q, ctx_id, x, x_stride_words,
                                                 reinterpret_cast<uint4*>(y_out), in_span);
        return f2_cuda_status(cudaGetLastError());
    }
    const int64_t sub = Q < ENC_SUB ? Q : ENC_SUB;
    int shift = st->enc_chunk_shift;
    while ((sub >> shift) >= ENC_MAX_CHUNKS) ++shift;
    const int64_t nch_max = (sub + (int64_t(1) << shift) - 1) >> shift;
    const int64_t B = (int64_t)st->num_ctx + 1;  // buckets per chunk (the last for bad ids)
    // 32-bit scratch: chunk counts [nch*B], scan input / starts [(nch+1)*B],
    // scan tile sums and prefixes [T each], ticket, item count
    const int64_t scan_n = (nch_max + 1) * B;
    const int64_t T = (scan_n + SCAN_TILE - 1) / SCAN_TILE;
    // + the table-build work list [9B] and its count, an aligned 8-byte pool counter
    const int64_t bin_words = nch_max * B + scan_n + 2 * T + 2 + 9 * B + 1 + 4;
    const bool tables = st->enc_table_min <= sub && st->num_ctx < (1 << 27);  // work items pack (context, block)
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
        e = f2_dev_alloc(st, (void**)&st->enc_off, sizeof(int32_t) * (size_t)sub, cs, true);
        if (e == cudaSuccess)
            e = f2_dev_alloc(st, (void**)&st->enc_sorted, sizeof(unsigned long long) * (size_t)sub, cs, true);
        if (e == cudaSuccess)
            e = f2_dev_alloc(st, (void**)&st->enc_items, sizeof(unsigned long long) * (size_t)sub, cs, true);
        if (e != cudaSuccess) return F2_ERR_OOM;
        st->enc_q_cap = sub;
    }
    if (bin_words > st->enc_bin_cap) {
        if (st->enc_bins) cudaFreeAsync(st->enc_bins, cs);
        st->enc_bins = nullptr;
        st->enc_bin_cap = 0;
        if (f2_dev_alloc(st, (void**)&st->enc_bins, sizeof(int32_t) * (size_t)bin_words, cs, true) != cudaSuccess)
            return F2_ERR_OOM;
        st->enc_bin_cap = bin_words;
    }
    if (B > st->enc_meta_cap) {
        if (st->enc_hot) cudaFreeAsync(st->enc_hot, cs);
        if (st->enc_tab_off) cudaFreeAsync(st->enc_tab_off, cs);
        st->enc_hot = nullptr;
        st->enc_tab_off = nullptr;
        st->enc_meta_cap = 0;
        e = f2_dev_alloc(st, (void**)&st->enc_hot, (size_t)B, cs, true);
        if (e == cudaSuccess)
            e = f2_dev_alloc(st, (void**)&st->enc_tab_off, sizeof(long long) * (size_t)B, cs, true);
        if (e != cudaSuccess) return F2_ERR_OOM;
        st->enc_meta_cap = B;
    }
    if (tables && !st->enc_pool) {
        // room for the table of every context that can have one (a table
        // never outgrows its upper bound for rank 0), capped
        int64_t words = 0;
        for (int32_t c = 0; c < st->num_ctx; ++c) {
            const int d = (st->flags & F2_FLAG_RAW_FEATURES) ? st->n_bits[c] : st->n_bits[c] + 1;
            if ((d + 31) / 32 <= TAB_WD) {
                const int wmax = 16 * ((d + 3) / 4) * (4 + ((d + 31) / 32 < TAB_RW ? (d + 31) / 32 : TAB_RW));
                words += wmax < TAB_WORDS ? wmax : TAB_WORDS;
            }
        }
        if (words > POOL_MAX_WORDS) words = POOL_MAX_WORDS;
        if (words > 0) {
            if (f2_dev_alloc(st, (void**)&st->enc_pool, sizeof(uint32_t) * (size_t)words, cs, true) != cudaSuccess)
                return F2_ERR_OOM;
            st->enc_pool_words = words;
        }
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
    if (tables) {
        const int rc = f2_ensure_aux(st);
        if (rc != F2_OK) return rc;
    }
    int32_t* cnt = st->enc_bins;
    int32_t* sta = cnt + nch_max * B;
    int32_t* tsum = sta + scan_n;
    int32_t* tpre = tsum + T;
    int32_t* ticket = tpre + T;
    int32_t* n_items = ticket + 1;
    int32_t* hot_list = n_items + 1;
    int32_t* n_hot = hot_list + 9 * B;
    unsigned long long* pool_used = reinterpret_cast<unsigned long long*>(
        (reinterpret_cast<uintptr_t>(n_hot + 1) + 7) & ~uintptr_t(7));
    unsigned long long* items = st->enc_items;
    const StoreDev sd = st->dev();
    const int tbl_blocks = (int)((B + TBL_THREADS - 1) / TBL_THREADS);
    for (int64_t q0 = 0; q0 < Q; q0 += sub) {
        const int32_t n = (int32_t)((Q - q0) < sub ? (Q - q0) : sub);
        const int32_t nch = (int32_t)((n + (int64_t(1) << shift) - 1) >> shift);
        const int64_t sn = ((int64_t)nch + 1) * B;
        const int32_t Tn = (int32_t)((sn + SCAN_TILE - 1) / SCAN_TILE);
        const uint32_t* xq = x + q0 * x_stride_words;
        uint4* yq = reinterpret_cast<uint4*>(y_out) + q0;
        {  // the pass's counters, one launch
            F2FillList zl;
            zl.add(cnt, sizeof(int32_t) * (size_t)(nch * B));
            zl.add(ticket, 2 * sizeof(int32_t));
            zl.add(n_hot, sizeof(int32_t));
            zl.add(pool_used, sizeof(unsigned long long));
            e = f2_fill(zl, cs);
            if (e != cudaSuccess) return f2_cuda_status(e);
        }
        enc_count_kernel<<<(n + ENC_TILE - 1) / ENC_TILE, ENC_TILE_THREADS, 0, cs>>>(n, ctx_id + q0, st->num_ctx,
                                                                                   shift, (int32_t)B, cnt,
                                                                                   st->enc_off);
        enc_table_kernel<<<tbl_blocks, TBL_THREADS, 0, cs>>>(
            sd, nch, (int32_t)B, cnt, sta, st->enc_hot, st->enc_tab_off, tables ? (long long)st->enc_pool_words : 0,
            pool_used, hot_list, n_hot, tables ? st->enc_table_min : INT_MAX, (long long)st->enc_chunk_min,
            x_stride_words);
        // the tables are built on the second stream while the queries are
        // placed (scan, scatter) on the caller's
        if (tables) {
            e = cudaEventRecord(st->ev_fork, cs);
            if (e == cudaSuccess) e = cudaStreamWaitEvent(st->aux, st->ev_fork, 0);
            if (e != cudaSuccess) return f2_cuda_status(e);
            enc_build_kernel<<<st->num_sms * 8, TBL_THREADS, 0, st->aux>>>(sd, hot_list, n_hot, st->enc_tab_off,
                                                                          st->enc_pool);
            e = cudaEventRecord(st->ev_join, st->aux);
            if (e != cudaSuccess) return f2_cuda_status(e);
        }
        enc_scan_kernel<<<Tn, SCAN_THREADS, 0, cs>>>(sta, (int32_t)sn, tsum, tpre, ticket);
        enc_scatter_kernel<<<(n + SCAT_THREADS * SCAT_PER - 1) / (SCAT_THREADS * SCAT_PER), SCAT_THREADS, 0, cs>>>(
            n, ctx_id + q0, st->num_ctx, shift, nch, (int32_t)B, cnt, sta, tpre, st->enc_hot, st->enc_off,
            st->enc_sorted);
        if (tables) {
            e = cudaStreamWaitEvent(cs, st->ev_join, 0);
            if (e != cudaSuccess) return f2_cuda_status(e);
        }
        enc_runs_kernel<<<(n + RUN_SEG - 1) / RUN_SEG, RUN_THREADS, sizeof(RunSmem), cs>>>(
            sd, n, st->enc_sorted, xq, x_stride_words, yq, in_span + q0, st->enc_hot, st->enc_tab_off,
            st->enc_pool, items, n_items);
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
    F2_NVTX_RANGE("f2_encode_epilogue");
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
int f2_encode_table_min_floor() { return 1; }
int f2_encode_chunk_shift_default() { return DEFAULT_CHUNK_SHIFT; }
long long f2_encode_chunk_min_default() { return DEFAULT_CHUNK_MIN; }
