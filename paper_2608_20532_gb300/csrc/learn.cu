// Batched streaming Gaussian elimination over GF(2) (Sec. 2.2) on sm_103a.
//
// Every context owns a reduced basis B[k] = (r_k, z_k), kept in shared memory
// while its rows stream in.  A group of lanes processes the rows of one
// context in rounds of 32 rows per warp:
//
//  1. reduce: each lane reduces its row against the basis as it stood at the
//     start of the round (the snapshot).  The basis is reduced (RREF, the
//     paper's step (5)), so the rows to XOR are exactly the pivots set in the
//     row itself; the warp walks the union of those pivots and every lane
//     XORs the broadcast row under its own bit (shared-memory broadcast, no
//     bank conflicts);
//  2. classify: a zero feature residual means the row lies in the span of
//     the snapshot.  The map T fixed by the snapshot never changes afterwards
//     (rows that contradict it are not inserted, insertions only extend it),
//     so such a row is classified exactly as the one-row-at-a-time algorithm
//     would classify it: zero word residual -> redundant, else contradiction
//     (Sec. 2.2 steps (2)-(3));
//  3. insert: the remaining rows (candidates) are eliminated among themselves
//     in stream order inside the warp (lane order), which reproduces step (4)
//     for each of them, then merged: the new rows are stored at their pivot
//     slots and every older row is cleared at the new pivot columns (step
//     (5)).  The result is the same reduced basis, with the same z_k, as the
//     sequential algorithm's.
//
// Contexts with few rows and a small basis get one warp each (many per CTA);
// heavy contexts get a whole CTA whose warps reduce 256 rows per round and
// insert their candidates warp by warp in stream order.  Contexts wider than
// 288 bits (d up to 1025) run in a separate wide kernel, one CTA each.  A
// single-block plan kernel validates the CSR batch and orders contexts
// longest-first into one queue per class.
#include <limits.h>

#include "f2_internal.cuh"

using namespace f2;

namespace {

struct LearnArgs {
    const int64_t* row_off;
    const int64_t* x_off;
    const uint32_t* x;
    const uint4* y;
    const int32_t* queue;
    int* counters;
    int warp_region_words;
};

// Shared-memory control area of a CTA-mode context (32-bit words).
constexpr int CTL_P = 0;       // pivot mask, 48 words
constexpr int CTL_NPR = 48;    // pivots added during the current round, 48 words
constexpr int CTL_CAND = 96;   // candidate ballots, 2 x 32 words (round parity)
constexpr int CTL_RANK = 160;  // rank
constexpr int CTL_CNT = 162;   // contradiction count (uint64, 8-byte aligned)
constexpr int CTL_FIRST = 164; // first contradiction index (int64)
constexpr int CTL_WORDS = 176; // size of the control area (16-byte multiple)
constexpr int WARP_CTL = 16;   // control words in front of a warp-mode basis

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

// Load row i of a context into (q, y): q = [1 || x] (index 0 = constant),
// or x itself for raw feature rows.  Lanes past the end load zeros.
template <int WD>
__device__ __forceinline__ void load_row(const uint32_t* __restrict__ xrow, const uint4* __restrict__ yrow,
                                         bool valid, int n, int xw, uint32_t raw, uint32_t (&q)[WD],
                                         uint4& y)
{
    uint32_t xin[WD];
#pragma unroll
    for (int v = 0; v < WD; ++v) {
        uint32_t t = 0;
        if (valid && v < xw) t = __ldg(xrow + v);
        if (v == xw - 1 && (n & 31)) t &= (1u << (n & 31)) - 1u;
        xin[v] = t;
    }
    if (raw) {
#pragma unroll
        for (int v = 0; v < WD; ++v) q[v] = xin[v];
    } else {
        q[0] = (xin[0] << 1) | (valid ? 1u : 0u);
#pragma unroll
        for (int v = 1; v < WD; ++v) q[v] = (xin[v] << 1) | (xin[v - 1] >> 31);
    }
    y = valid ? __ldg(yrow) : make_uint4(0, 0, 0, 0);
}

// Step (1) against the snapshot S.  On return the residual is zero at every
// pivot column of words that are not "mixed"; the caller masks with ~P.
template <int WD>
__device__ __forceinline__ void reduce_snapshot(uint32_t (&xr)[WD], uint4& yr, const uint32_t* __restrict__ S,
                                                const uint32_t (&P)[WD], uint64_t mixed)
{
    constexpr int RS = row_stride(WD);
#pragma unroll
    for (int w = 0; w < WD; ++w) {
        uint32_t uw = __reduce_or_sync(FULL, xr[w] & P[w]);
        const bool xwork = (mixed & ((2ull << w) - 1ull)) != 0;
        while (uw) {
            const int b = __ffs(uw) - 1;
            uw &= uw - 1;
            const uint32_t* row = S + (32 * w + b) * RS;
            const uint32_t m = 0u - ((xr[w] >> b) & 1u);
            const uint4 z = *reinterpret_cast<const uint4*>(row);
            yr.x ^= z.x & m;
            yr.y ^= z.y & m;
            yr.z ^= z.z & m;
            yr.w ^= z.w & m;
            if (xwork) {
#pragma unroll
                for (int v4 = 0; v4 <= w / 4; ++v4) {
                    const uint4 xv = *reinterpret_cast<const uint4*>(row + 4 + 4 * v4);
                    const uint32_t e[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int v = 4 * v4 + j;
                        if (v <= w && v < WD)
                            if ((mixed >> v) & 1ull) xr[v] ^= e[j] & m;
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
                            unsigned long long& cnt, uint32_t (&NP)[WD])
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
                ++cnt;
                first = min(first, idx);
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

template <int WD>
__device__ void basis_to_smem(const StoreDev& s, const CtxDesc& cd, uint32_t* S, int t, int nt)
{
    constexpr int RS = row_stride(WD);
    for (int k = t; k < cd.d; k += nt) {
        *reinterpret_cast<uint4*>(S + k * RS) = s.bz[cd.slot_off + k];
        for (int v = cd.wd; v < RS - 4; ++v) S[k * RS + 4 + v] = 0;
    }
    const int words = cd.d * cd.wd;
    for (int idx = t; idx < words; idx += nt) {
        const int k = idx / cd.wd, v = idx - k * cd.wd;
        S[k * RS + 4 + v] = s.bx[cd.xw_off + idx];
    }
}

template <int WD>
__device__ void basis_from_smem(const StoreDev& s, const CtxDesc& cd, const uint32_t* S, int t, int nt)
{
    constexpr int RS = row_stride(WD);
    for (int k = t; k < cd.d; k += nt) s.bz[cd.slot_off + k] = *reinterpret_cast<const uint4*>(S + k * RS);
    const int words = cd.d * cd.wd;
    for (int idx = t; idx < words; idx += nt) {
        const int k = idx / cd.wd, v = idx - k * cd.wd;
        s.bx[cd.xw_off + idx] = S[k * RS + 4 + v];
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

// One warp owns context c.
template <int WD>
__device__ void learn_ctx_warp(const StoreDev& s, const LearnArgs& a, int c, uint32_t* region, int lane)
{
    const CtxDesc cd = s.desc[c];
    uint32_t* S = region + WARP_CTL;
    basis_to_smem<WD>(s, cd, S, lane, 32);
    uint32_t P[WD];
#pragma unroll
    for (int v = 0; v < WD; ++v) P[v] = (v < cd.wd) ? s.pivot[cd.pw_off + v] : 0u;
    __syncwarp();
    uint64_t mixed = mixed_words<WD>(P, cd.d, cd.wd);
    int rank = s.rank[c];
    const long long seen = s.rows_seen[c];
    const int64_t r0 = a.row_off[c];
    const int64_t T = a.row_off[c + 1] - r0;
    const uint32_t* xc = a.x + a.x_off[c];
    const uint4* yc = a.y + r0;
    long long first = LLONG_MAX;
    unsigned long long cnt = 0;
    for (int64_t base = 0; base < T; base += 32) {
        const int64_t i = base + lane;
        const bool valid = i < T;
        uint32_t xr[WD];
        uint4 yr;
        load_row<WD>(xc + (valid ? i : 0) * cd.xw, yc + (valid ? i : 0), valid, cd.n, cd.xw, s.raw, xr, yr);
        reduce_snapshot<WD>(xr, yr, S, P, mixed);
        uint32_t nz = 0;
#pragma unroll
        for (int v = 0; v < WD; ++v) {
            xr[v] &= ~P[v];
            nz |= xr[v];
        }
        if (valid && !nz && nonzero4(yr)) {
            ++cnt;
            first = min(first, seen + i);
        }
        const uint32_t cand = __ballot_sync(FULL, valid && nz != 0u);
        if (cand) {
            uint32_t NP[WD];
            rank += insert_block<WD>(xr, yr, cand, S, P, cd.d, lane, seen + i, first, cnt, NP);
#pragma unroll
            for (int v = 0; v < WD; ++v) P[v] |= NP[v];
            mixed = mixed_words<WD>(P, cd.d, cd.wd);
        }
    }
    __syncwarp();
#pragma unroll
    for (int v = 0; v < WD; ++v)
        if (lane == v && v < cd.wd) s.pivot[cd.pw_off + v] = P[v];
    basis_from_smem<WD>(s, cd, S, lane, 32);
    warp_stats(first, cnt);
    if (lane == 0) {
        s.rank[c] = rank;
        s.rows_seen[c] = seen + T;
        commit_stats(s, c, first, cnt);
    }
    __syncwarp();
}

// All warps of the CTA own context c.
template <int WD>
__device__ void learn_ctx_cta(const StoreDev& s, const LearnArgs& a, int c, uint32_t* smem)
{
    const int t = threadIdx.x, nt = blockDim.x;
    const int warp = t >> 5, lane = t & 31, nwarps = nt >> 5;
    const CtxDesc cd = s.desc[c];
    uint32_t* Ps = smem + CTL_P;
    uint32_t* NPR = smem + CTL_NPR;
    uint32_t* candw = smem + CTL_CAND;
    int* rank_s = reinterpret_cast<int*>(smem + CTL_RANK);
    unsigned long long* cnt_s = reinterpret_cast<unsigned long long*>(smem + CTL_CNT);
    long long* first_s = reinterpret_cast<long long*>(smem + CTL_FIRST);
    uint32_t* S = smem + CTL_WORDS;
    basis_to_smem<WD>(s, cd, S, t, nt);
    if (t < 48) {
        Ps[t] = (t < cd.wd) ? s.pivot[cd.pw_off + t] : 0u;
        NPR[t] = 0;
    }
    if (t == 0) {
        *rank_s = s.rank[c];
        *cnt_s = 0;
        *first_s = LLONG_MAX;
    }
    __syncthreads();
    uint32_t P[WD];
#pragma unroll
    for (int v = 0; v < WD; ++v) P[v] = Ps[v];
    uint64_t mixed = mixed_words<WD>(P, cd.d, cd.wd);
    const long long seen = s.rows_seen[c];
    const int64_t r0 = a.row_off[c];
    const int64_t T = a.row_off[c + 1] - r0;
    const uint32_t* xc = a.x + a.x_off[c];
    const uint4* yc = a.y + r0;
    long long first = LLONG_MAX;
    unsigned long long cnt = 0;
    int par = 0;
    for (int64_t base = 0; base < T; base += 32 * nwarps, par ^= 1) {
        const int64_t i = base + 32 * warp + lane;
        const bool valid = i < T;
        uint32_t xr[WD];
        uint4 yr;
        load_row<WD>(xc + (valid ? i : 0) * cd.xw, yc + (valid ? i : 0), valid, cd.n, cd.xw, s.raw, xr, yr);
        reduce_snapshot<WD>(xr, yr, S, P, mixed);
        uint32_t nz = 0;
#pragma unroll
        for (int v = 0; v < WD; ++v) {
            xr[v] &= ~P[v];
            nz |= xr[v];
        }
        if (valid && !nz && nonzero4(yr)) {
            ++cnt;
            first = min(first, seen + i);
        }
        const uint32_t cand = __ballot_sync(FULL, valid && nz != 0u);
        if (lane == 0) candw[32 * par + warp] = cand;
        __syncthreads();
        uint32_t wmask = 0;
        for (int ww = 0; ww < nwarps; ++ww)
            if (candw[32 * par + ww]) wmask |= 1u << ww;
        if (wmask) {
            const int first_warp = __ffs(wmask) - 1;
            for (uint32_t wm = wmask; wm; wm &= wm - 1) {
                const int ww = __ffs(wm) - 1;
                if (warp == ww) {
                    if (ww != first_warp) reduce_new<WD>(xr, yr, S, NPR);
                    uint32_t NP[WD];
                    const int added = insert_block<WD>(xr, yr, cand, S, P, cd.d, lane, seen + i, first, cnt, NP);
                    if (lane == 0 && added) {
#pragma unroll
                        for (int v = 0; v < WD; ++v) {
                            Ps[v] = P[v] | NP[v];
                            NPR[v] |= NP[v];
                        }
                        *rank_s += added;
                    }
                }
                __syncthreads();
#pragma unroll
                for (int v = 0; v < WD; ++v) P[v] = Ps[v];
            }
            mixed = mixed_words<WD>(P, cd.d, cd.wd);
            if (t < 48) NPR[t] = 0;
        }
    }
    warp_stats(first, cnt);
    if (lane == 0 && cnt) {
        atomicAdd(cnt_s, cnt);
        atomicMin(first_s, first);
    }
    __syncthreads();
    if (t < cd.wd) s.pivot[cd.pw_off + t] = Ps[t];
    basis_from_smem<WD>(s, cd, S, t, nt);
    if (t == 0) {
        s.rank[c] = *rank_s;
        s.rows_seen[c] = seen + T;
        commit_stats(s, c, *first_s, *cnt_s);
    }
    __syncthreads();
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

__global__ void __launch_bounds__(LEARN_WARPS * 32) learn_narrow_kernel(StoreDev s, LearnArgs a)
{
    extern __shared__ __align__(16) uint32_t smem[];
    __shared__ int s_item;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_cta = a.counters[CNT_COUNT + CLS_CTA];
    const int b_cta = a.counters[CNT_BEGIN + CLS_CTA];
    for (;;) {
        __syncthreads();
        if (threadIdx.x == 0) s_item = atomicAdd(a.counters + CNT_HEAD_CTA, 1);
        __syncthreads();
        const int item = s_item;
        if (item >= n_cta) break;
        const int c = a.queue[b_cta + item];
        const int wd = s.desc[c].wd;
#define F2_CALL_CTA(W) learn_ctx_cta<W>(s, a, c, smem)
        F2_NARROW_SWITCH(wd, F2_CALL_CTA)
#undef F2_CALL_CTA
    }
    const int n_w = a.counters[CNT_COUNT + CLS_WARP];
    const int b_w = a.counters[CNT_BEGIN + CLS_WARP];
    uint32_t* region = smem + warp * a.warp_region_words;
    for (;;) {
        int item = 0;
        if (lane == 0) item = atomicAdd(a.counters + CNT_HEAD_WARP, 1);
        item = __shfl_sync(FULL, item, 0);
        if (item >= n_w) break;
        const int c = a.queue[b_w + item];
        const int wd = s.desc[c].wd;
#define F2_CALL_WARP(W) learn_ctx_warp<W>(s, a, c, region, lane)
        F2_NARROW_SWITCH(wd, F2_CALL_WARP)
#undef F2_CALL_WARP
    }
}

constexpr int WIDE_WD = 33;

__global__ void __launch_bounds__(WIDE_WARPS * 32) learn_wide_kernel(StoreDev s, LearnArgs a)
{
    extern __shared__ __align__(16) uint32_t smem[];
    __shared__ int s_item;
    const int n = a.counters[CNT_COUNT + CLS_WIDE];
    const int b = a.counters[CNT_BEGIN + CLS_WIDE];
    for (;;) {
        __syncthreads();
        if (threadIdx.x == 0) s_item = atomicAdd(a.counters + CNT_HEAD_WIDE, 1);
        __syncthreads();
        const int item = s_item;
        if (item >= n) break;
        learn_ctx_cta<WIDE_WD>(s, a, a.queue[b + item], smem);
    }
}

// Validate the batch and build the longest-first queues (one block).
__global__ void __launch_bounds__(1024) plan_kernel(StoreDev s, const int64_t* __restrict__ row_off,
                                                    const int64_t* __restrict__ x_off, int64_t total_rows,
                                                    int64_t total_xw, int warp_region_words, int64_t heavy_rows,
                                                    int32_t* __restrict__ queue, int32_t* __restrict__ keybuf,
                                                    int* __restrict__ counters)
{
    __shared__ int hist[3][PLAN_BUCKETS];
    __shared__ int cursor[3][PLAN_BUCKETS];
    for (int i = threadIdx.x; i < 3 * PLAN_BUCKETS; i += blockDim.x) (&hist[0][0])[i] = 0;
    __syncthreads();
    for (int c = threadIdx.x; c < s.num_ctx; c += blockDim.x) {
        const CtxDesc cd = s.desc[c];
        const int64_t a0 = row_off[c], a1 = row_off[c + 1];
        const int64_t rows = a1 - a0;
        const int64_t x0 = x_off[c];
        const bool ok = a0 >= 0 && rows >= 0 && a1 <= total_rows && x0 >= 0 && rows <= total_xw &&
                        x0 + rows * cd.xw <= total_xw;
        int key = -1;
        if (!ok) {
            record_status(s.status, F2_ERR_ROWS);
        } else if (rows > 0) {
            const int basis_words = WARP_CTL + cd.d * row_stride(cd.wd);
            int cls;
            if (cd.wd > NARROW_WD) cls = CLS_WIDE;
            else if (basis_words > warp_region_words || rows >= heavy_rows) cls = CLS_CTA;
            else cls = CLS_WARP;
            const unsigned long long work = (unsigned long long)rows * (unsigned long long)(cd.wd + 4);
            int bucket = 63 - __clzll(work);
            if (bucket >= PLAN_BUCKETS) bucket = PLAN_BUCKETS - 1;
            key = cls * PLAN_BUCKETS + bucket;
            atomicAdd(&hist[cls][bucket], 1);
        }
        keybuf[c] = key;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int pos = 0;
        for (int cls = 0; cls < 3; ++cls) {
            counters[CNT_BEGIN + cls] = pos;
            for (int bk = PLAN_BUCKETS - 1; bk >= 0; --bk) {
                cursor[cls][bk] = pos;
                pos += hist[cls][bk];
            }
            counters[CNT_COUNT + cls] = pos - counters[CNT_BEGIN + cls];
        }
        counters[CNT_HEAD_CTA] = 0;
        counters[CNT_HEAD_WIDE] = 0;
        counters[CNT_HEAD_WARP] = 0;
    }
    __syncthreads();
    for (int c = threadIdx.x; c < s.num_ctx; c += blockDim.x) {
        const int key = keybuf[c];
        if (key >= 0) {
            const int p = atomicAdd(&cursor[key / PLAN_BUCKETS][key % PLAN_BUCKETS], 1);
            queue[p] = c;
        }
    }
}

inline bool is_aligned(const void* p, size_t al) { return ((uintptr_t)p % al) == 0; }

}  // namespace

extern "C" int f2_learn_batched(f2_store* st, const int64_t* row_off, const uint32_t* x, const int64_t* x_off,
                                const uint32_t* y, int64_t total_rows, int64_t total_x_words,
                                f2_stream_t stream)
{
    if (!st || total_rows < 0 || total_x_words < 0) return F2_ERR_INVALID_ARG;
    if (st->num_ctx == 0) return F2_OK;
    if (!row_off || !x_off || (!x && total_x_words) || (!y && total_rows)) return F2_ERR_INVALID_ARG;
    if (!is_aligned(row_off, 8) || !is_aligned(x_off, 8) || !is_aligned(x, 4) || !is_aligned(y, 16))
        return F2_ERR_ALIGN;
    cudaStream_t cs = (cudaStream_t)stream;
    const StoreDev sd = st->dev();
    const int warp_region_words = (int)(st->warp_basis_bytes / 4);
    plan_kernel<<<1, 1024, 0, cs>>>(sd, row_off, x_off, total_rows, total_x_words, warp_region_words,
                                    st->heavy_rows, st->queue, st->keybuf, st->counters);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return f2_cuda_status(e);

    LearnArgs la;
    la.row_off = row_off;
    la.x_off = x_off;
    la.x = x;
    la.y = reinterpret_cast<const uint4*>(y);
    la.queue = st->queue;
    la.counters = st->counters;
    la.warp_region_words = warp_region_words;

    // narrow kernel: CTA-mode contexts first (largest basis of any narrow
    // context), then the warp queue (LEARN_WARPS regions)
    int max_narrow_d = 0, max_narrow_wd = 1;
    for (int32_t c = 0; c < st->num_ctx; ++c) {
        const int d = (st->flags & F2_FLAG_RAW_FEATURES) ? st->n_bits[(size_t)c] : st->n_bits[(size_t)c] + 1;
        const int wd = (d + 31) / 32;
        if (wd <= NARROW_WD && d * row_stride(wd) > max_narrow_d * row_stride(max_narrow_wd)) {
            max_narrow_d = d;
            max_narrow_wd = wd;
        }
    }
    if (st->n_wide < st->num_ctx) {
        size_t cta_bytes = 4 * (size_t)(CTL_WORDS + max_narrow_d * row_stride(max_narrow_wd));
        size_t warp_bytes = 4 * (size_t)LEARN_WARPS * (size_t)warp_region_words;
        size_t smem = cta_bytes > warp_bytes ? cta_bytes : warp_bytes;
        e = cudaFuncSetAttribute(learn_narrow_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return f2_cuda_status(e);
        int per_sm = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, learn_narrow_kernel, LEARN_WARPS * 32, smem);
        if (e != cudaSuccess) return f2_cuda_status(e);
        if (per_sm < 1) per_sm = 1;
        learn_narrow_kernel<<<st->num_sms * per_sm, LEARN_WARPS * 32, smem, cs>>>(sd, la);
        e = cudaGetLastError();
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    if (st->n_wide > 0) {
        const size_t smem = 4 * (size_t)(CTL_WORDS + st->max_d * row_stride(WIDE_WD));
        e = cudaFuncSetAttribute(learn_wide_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return f2_cuda_status(e);
        int blocks = st->n_wide < st->num_sms ? st->n_wide : st->num_sms;
        learn_wide_kernel<<<blocks, WIDE_WARPS * 32, smem, cs>>>(sd, la);
        e = cudaGetLastError();
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    return F2_OK;
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
    int counters[16];
};

// Device storage for the scratch; in host code this name is only a symbol
// handle, its device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_noalloc_scratch[sizeof(NoallocScratch)];

constexpr int NOALLOC_MAX_DEVICES = 64;
constexpr int NOALLOC_NARROW_SMEM_DEFAULT = 4 * LEARN_WARPS * (8192 / 4);
constexpr int NOALLOC_HEAVY_ROWS = 4096;
constexpr int NOALLOC_WARP_REGION_WORDS = 8192 / 4;

struct NoallocDevice {
    NoallocScratch* scratch;
    int num_sms;
    bool ready;
};
NoallocDevice g_noalloc_dev[NOALLOC_MAX_DEVICES];
std::mutex g_noalloc_mu;

// Once per device (with that device current): resolve the scratch address.
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
        if (e != cudaSuccess) return f2_cuda_status(e);
        d.scratch = static_cast<NoallocScratch*>(p);
        d.num_sms = sms;
        d.ready = true;
    }
    *out = &d;
    return F2_OK;
}

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

}  // namespace

extern "C" int f2_learn_batched_noalloc(int32_t num_ctx, const int32_t* n_bits_host, uint32_t flags,
                                        int32_t* rank_dev, uint32_t* pivot_mask_dev, uint32_t* basis_x_dev,
                                        uint32_t* basis_z_dev, uint8_t* contra_dev, int64_t* first_contra_dev,
                                        uint64_t* n_contra_dev, int64_t* rows_seen_dev, int32_t* status_dev,
                                        const int64_t* row_off_dev, const uint32_t* x_dev, const int64_t* x_off_dev,
                                        const uint32_t* y_dev, int64_t total_rows, int64_t total_x_words,
                                        f2_stream_t stream)
{
    if (num_ctx < 0 || num_ctx > F2_NOALLOC_MAX_CTX || (flags & ~F2_FLAG_RAW_FEATURES) || total_rows < 0 ||
        total_x_words < 0 || !status_dev)
        return F2_ERR_INVALID_ARG;
    if (num_ctx == 0) return F2_OK;
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
    int max_narrow_bytes = 0, max_d = 0, n_wide = 0, n_narrow = 0;
    for (int32_t c = 0; c < num_ctx; ++c) {
        const int n = n_bits_host[c];
        if (n < 1 || n > MAX_N) return F2_ERR_NBITS;
        const int d = raw ? n : n + 1;
        const int wd = (d + 31) / 32;
        if (d > max_d) max_d = d;
        if (wd > NARROW_WD) {
            ++n_wide;
        } else {
            ++n_narrow;
            const int bytes = 4 * (CTL_WORDS + d * row_stride(wd));
            if (bytes > max_narrow_bytes) max_narrow_bytes = bytes;
        }
    }
    NoallocDevice* nd = nullptr;
    int rc = noalloc_setup(&nd);
    if (rc != F2_OK) return rc;
    NoallocScratch* sc = nd->scratch;
    cudaStream_t cs = (cudaStream_t)stream;

    cudaError_t e = cudaMemsetAsync(status_dev, 0, sizeof(int32_t), cs);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(sc->n_bits, n_bits_host, sizeof(int32_t) * (size_t)num_ctx, cudaMemcpyHostToDevice, cs);
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
    plan_kernel<<<1, 1024, 0, cs>>>(sd, row_off_dev, x_off_dev, total_rows, total_x_words, NOALLOC_WARP_REGION_WORDS,
                                    NOALLOC_HEAVY_ROWS, sc->queue, sc->keybuf, sc->counters);
    e = cudaGetLastError();
    if (e != cudaSuccess) return f2_cuda_status(e);

    LearnArgs la;
    la.row_off = row_off_dev;
    la.x_off = x_off_dev;
    la.x = x_dev;
    la.y = reinterpret_cast<const uint4*>(y_dev);
    la.queue = sc->queue;
    la.counters = sc->counters;
    la.warp_region_words = NOALLOC_WARP_REGION_WORDS;
    if (n_narrow) {
        const int smem = max_narrow_bytes > NOALLOC_NARROW_SMEM_DEFAULT ? max_narrow_bytes : NOALLOC_NARROW_SMEM_DEFAULT;
        e = cudaFuncSetAttribute(learn_narrow_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return f2_cuda_status(e);
        int per_sm = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, learn_narrow_kernel, LEARN_WARPS * 32, smem);
        if (e != cudaSuccess) return f2_cuda_status(e);
        if (per_sm < 1) per_sm = 1;
        learn_narrow_kernel<<<nd->num_sms * per_sm, LEARN_WARPS * 32, smem, cs>>>(sd, la);
        e = cudaGetLastError();
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    if (n_wide) {
        const int smem = 4 * (CTL_WORDS + max_d * row_stride(WIDE_WD));
        e = cudaFuncSetAttribute(learn_wide_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return f2_cuda_status(e);
        const int blocks = n_wide < nd->num_sms ? n_wide : nd->num_sms;
        learn_wide_kernel<<<blocks, WIDE_WARPS * 32, smem, cs>>>(sd, la);
        e = cudaGetLastError();
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    return F2_OK;
}
