// Batched encoding with a span check (Sec. 2.3, Appendix B) on sm_103a.
//
// One thread per query: q = phi(x) is reduced against its context's reduced
// basis; every stored row used also XORs its z_k into a zero accumulator.
// Because the basis is reduced, the rows to use are exactly the pivots set in
// q itself, walked word by word.  A zero residual at the non-pivot columns
// proves q in the span and the accumulator is the word; otherwise the query
// is rejected and the word is zero.
#include "f2_internal.cuh"

using namespace f2;

namespace {

template <int WD>
__device__ __forceinline__ bool encode_one(const StoreDev& s, const CtxDesc& cd, const uint32_t* __restrict__ xq,
                                           uint4& acc)
{
    uint32_t q[WD];
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

constexpr int ENC_THREADS = 256;
constexpr int ENC_CHUNK = 2048;    // queries grouped per CTA step
constexpr int ENC_BUCKETS = 256;   // context-hash buckets of a chunk

__device__ __forceinline__ void encode_query(const StoreDev& s, int64_t i, const int32_t* __restrict__ ctx_id,
                                             const uint32_t* __restrict__ x, int stride, uint4* __restrict__ y,
                                             uint8_t* __restrict__ in_span)
{
    const int c = __ldg(ctx_id + i);
    uint4 acc = make_uint4(0, 0, 0, 0);
    uint8_t flag;
    if (c < 0 || c >= s.num_ctx) {
        record_status(s.status, F2_ERR_CTX_RANGE);
        flag = 0xFF;
    } else {
        const CtxDesc cd = s.desc[c];
        const uint32_t* xq = x + i * stride;
        bool ok;
        if (cd.xw > stride) {
            record_status(s.status, F2_ERR_STRIDE);
            flag = 0xFF;
            ok = false;
        } else {
            ok = (cd.wd <= NARROW_WD) ? encode_one<NARROW_WD>(s, cd, xq, acc) : encode_one<33>(s, cd, xq, acc);
            flag = ok ? 1 : 0;
        }
        if (!ok) acc = make_uint4(0, 0, 0, 0);
    }
    y[i] = acc;
    in_span[i] = flag;
}

// Each CTA step takes ENC_CHUNK consecutive queries, partitions them in
// shared memory by a hash of their context id (a counting sort into
// ENC_BUCKETS buckets), and lets every thread encode the queries of the
// permuted order: a warp then mostly serves queries of one context, which
// share its basis rows in L1 and take similar paths.
__global__ void __launch_bounds__(ENC_THREADS, 3) encode_kernel(StoreDev s, int64_t Q, const int32_t* __restrict__ ctx_id,
                                                                const uint32_t* __restrict__ x, int stride,
                                                                uint4* __restrict__ y, uint8_t* __restrict__ in_span)
{
    __shared__ int hist[ENC_BUCKETS];
    __shared__ uint16_t perm[ENC_CHUNK];
    __shared__ uint8_t key[ENC_CHUNK];
    const int t = threadIdx.x;
    for (int64_t base = (int64_t)blockIdx.x * ENC_CHUNK; base < Q; base += (int64_t)gridDim.x * ENC_CHUNK) {
        const int n = (int)((Q - base) < ENC_CHUNK ? (Q - base) : ENC_CHUNK);
        hist[t] = 0;
        __syncthreads();
        for (int k = t; k < n; k += ENC_THREADS) {
            const uint32_t c = (uint32_t)__ldg(ctx_id + base + k);
            const uint8_t b = (uint8_t)((c * 2654435761u) >> 24);
            key[k] = b;
            atomicAdd(&hist[b], 1);
        }
        __syncthreads();
        if (t < 32) {  // exclusive scan of 256 bucket counts by one warp
            int v[ENC_BUCKETS / 32];
            int sum = 0;
#pragma unroll
            for (int j = 0; j < ENC_BUCKETS / 32; ++j) {
                v[j] = hist[t * (ENC_BUCKETS / 32) + j];
                sum += v[j];
            }
            int inc = sum;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int u = __shfl_up_sync(FULL, inc, o);
                if (t >= o) inc += u;
            }
            int run = inc - sum;
#pragma unroll
            for (int j = 0; j < ENC_BUCKETS / 32; ++j) {
                hist[t * (ENC_BUCKETS / 32) + j] = run;
                run += v[j];
            }
        }
        __syncthreads();
        for (int k = t; k < n; k += ENC_THREADS) perm[atomicAdd(&hist[key[k]], 1)] = (uint16_t)k;
        __syncthreads();
        for (int k = t; k < n; k += ENC_THREADS) encode_query(s, base + perm[k], ctx_id, x, stride, y, in_span);
        __syncthreads();
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
    int64_t blocks = (Q + ENC_CHUNK - 1) / ENC_CHUNK;
    const int64_t cap = (int64_t)st->num_sms * 3;
    if (blocks > cap) blocks = cap;
    encode_kernel<<<(int)blocks, ENC_THREADS, 0, (cudaStream_t)stream>>>(
        st->dev(), Q, ctx_id, x, x_stride_words, reinterpret_cast<uint4*>(y_out), in_span);
    return f2_cuda_status(cudaGetLastError());
}
