// Host-resident inputs: learning and encoding straight from host memory, the
// host<->device copies overlapped with the kernels.
//
// A learn call is cut into chunks of whole contexts (about chunk_bytes of
// rows each; contexts are independent, so chunk-wise learning gives the same
// state as one call).  A private copy stream moves chunks into a ring of
// LEARN_BUFS buffers while the caller's stream learns the ones before;
// events order each buffer's reuse; the chunk whose largest context is
// smallest goes
// last (what is left after the last copy is that chunk's learn, which its
// largest context bounds).  Encode calls are cut into chunks of queries with
// a third stage: the words of chunk j go back to the host on a second
// private stream while chunk j + 1 is encoded; the queries go in through a
// ring of ENC_IN buffers, so up to ENC_IN chunks are copied in ahead of the
// encoding (and of whatever the caller's stream runs before it).  Host
// arrays are read (and host outputs written) asynchronously: they must stay
// valid until the caller's stream has passed the call.
#include <algorithm>
#include <vector>

#include "f2_internal.cuh"

using namespace f2;

namespace f2 {

constexpr int ENC_IN = 4;      // query input buffers of f2_encode_host
constexpr int LEARN_BUFS = 2;  // chunk buffers of f2_learn_host (four measured no faster)

struct HostIO {
    int device = -1;
    cudaStream_t h2d = nullptr, d2h = nullptr;
    cudaEvent_t copied[LEARN_BUFS] = {}, freed[LEARN_BUFS] = {}, done[2] = {}, drained[2] = {}, last = nullptr;
    cudaEvent_t qcopied[ENC_IN] = {}, qused[ENC_IN] = {};
    // learn chunks: feature words, 128-bit words, CSR slices (a ring); the
    // rebased offsets of the current chunk (one buffer: rebased and used on
    // the caller's stream in order)
    uint32_t* x[LEARN_BUFS] = {};
    uint4* y[LEARN_BUFS] = {};
    int64_t* ro[LEARN_BUFS] = {};
    int64_t* xo[LEARN_BUFS] = {};
    int64_t x_cap = 0, y_cap = 0, c_cap = 0;
    int64_t* row_off = nullptr;
    int64_t* x_off = nullptr;
    int64_t full_cap = 0;
    // encode chunks: inputs in a ring, outputs double buffered
    int32_t* qc[ENC_IN] = {};
    uint32_t* qx[ENC_IN] = {};
    uint4* qy[2] = {};
    uint8_t* qs[2] = {};
    int64_t q_cap = 0, qx_cap = 0;
};

}  // namespace f2

namespace {

__global__ void __launch_bounds__(256) rebase_kernel(const int64_t* __restrict__ ro, const int64_t* __restrict__ xo,
                                                     int32_t c0, int32_t c1, int32_t C, int64_t xa,
                                                     int64_t* __restrict__ row_off, int64_t* __restrict__ x_off)
{
    // contexts outside [c0, c1) get no rows; offsets of the chunk's contexts
    // count from the chunk's first row and first feature word
    const int64_t r0 = ro[0];
    const int64_t rn = ro[c1 - c0] - r0;
    for (int c = blockIdx.x * blockDim.x + threadIdx.x; c <= C; c += gridDim.x * blockDim.x) {
        row_off[c] = (c <= c0) ? 0 : (c <= c1 ? ro[c - c0] - r0 : rn);
        if (c < C) {
            const bool in = c >= c0 && c < c1 && ro[c - c0 + 1] > ro[c - c0];
            x_off[c] = in ? xo[c - c0] - xa : 0;
        }
    }
}

cudaError_t sync_all(HostIO* h, cudaStream_t cs)
{
    cudaError_t e = cudaStreamSynchronize(cs);
    if (e == cudaSuccess && h->h2d) e = cudaStreamSynchronize(h->h2d);
    if (e == cudaSuccess && h->d2h) e = cudaStreamSynchronize(h->d2h);
    return e;
}

int host_io(f2_store* st, HostIO** out)
{
    if (!st->hio) {
        HostIO* h = new (std::nothrow) HostIO();
        if (!h) return F2_ERR_OOM;
        cudaError_t e = cudaGetDevice(&h->device);
        if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&h->h2d, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&h->d2h, cudaStreamNonBlocking);
        for (int b = 0; b < LEARN_BUFS && e == cudaSuccess; ++b) {
            e = cudaEventCreateWithFlags(&h->copied[b], cudaEventDisableTiming);
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->freed[b], cudaEventDisableTiming);
        }
        for (int b = 0; b < 2 && e == cudaSuccess; ++b) {
            e = cudaEventCreateWithFlags(&h->done[b], cudaEventDisableTiming);
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->drained[b], cudaEventDisableTiming);
        }
        for (int b = 0; b < ENC_IN && e == cudaSuccess; ++b) {
            e = cudaEventCreateWithFlags(&h->qcopied[b], cudaEventDisableTiming);
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->qused[b], cudaEventDisableTiming);
        }
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->last, cudaEventDisableTiming);
        st->hio = h;
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    *out = st->hio;
    return F2_OK;
}

// Grow a device buffer (contents are not kept); the caller has synchronized.
template <typename T>
cudaError_t grow(const f2_store* st, T*& p, int64_t& cap, int64_t need)
{
    if (need <= cap) return cudaSuccess;
    if (p) cudaFree(p);
    p = nullptr;
    cap = 0;
    const cudaError_t e = f2_dev_alloc(st, (void**)&p, sizeof(T) * (size_t)(need > 0 ? need : 1), nullptr, false);
    if (e == cudaSuccess) cap = need;
    return e;
}

struct Chunk {
    int32_t c0, c1;
    int64_t r0, r1, xa, xb;
    int64_t max_rows;  // rows of its largest context
};

}  // namespace

void f2_host_io_free(f2_store* st)
{
    HostIO* h = st->hio;
    if (!h) return;
    if (h->h2d) cudaStreamSynchronize(h->h2d);
    if (h->d2h) cudaStreamSynchronize(h->d2h);
    for (int b = 0; b < LEARN_BUFS; ++b) {
        void* bufs[] = {h->x[b], h->y[b], h->ro[b], h->xo[b]};
        for (void* p : bufs)
            if (p) cudaFree(p);
        cudaEvent_t evs[] = {h->copied[b], h->freed[b]};
        for (cudaEvent_t ev : evs)
            if (ev) cudaEventDestroy(ev);
    }
    for (int b = 0; b < 2; ++b) {
        void* bufs[] = {h->qy[b], h->qs[b]};
        for (void* p : bufs)
            if (p) cudaFree(p);
        cudaEvent_t evs[] = {h->done[b], h->drained[b]};
        for (cudaEvent_t ev : evs)
            if (ev) cudaEventDestroy(ev);
    }
    for (int b = 0; b < ENC_IN; ++b) {
        if (h->qc[b]) cudaFree(h->qc[b]);
        if (h->qx[b]) cudaFree(h->qx[b]);
        if (h->qcopied[b]) cudaEventDestroy(h->qcopied[b]);
        if (h->qused[b]) cudaEventDestroy(h->qused[b]);
    }
    if (h->last) cudaEventDestroy(h->last);
    if (h->row_off) cudaFree(h->row_off);
    if (h->x_off) cudaFree(h->x_off);
    if (h->h2d) cudaStreamDestroy(h->h2d);
    if (h->d2h) cudaStreamDestroy(h->d2h);
    delete h;
    st->hio = nullptr;
}

extern "C" int f2_learn_host(f2_store* st, const int64_t* row_off, const uint32_t* x, const int64_t* x_off,
                             const uint32_t* y, int64_t total_rows, int64_t total_x_words, f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_learn_host");
    if (!st || total_rows < 0 || total_x_words < 0) return F2_ERR_INVALID_ARG;
    const int32_t C = st->num_ctx;
    if (C == 0) return F2_OK;
    if (!row_off || !x_off || (!x && total_x_words) || (!y && total_rows)) return F2_ERR_INVALID_ARG;
    // validate the CSR batch on the host and cut it into chunks
    const int64_t target = st->host_chunk_bytes;
    std::vector<Chunk> chunks;
    Chunk cur{0, 0, row_off[0], row_off[0], INT64_MAX, 0, 0};
    int64_t bytes = 0;
    for (int32_t c = 0; c < C; ++c) {
        const int64_t a0 = row_off[c], a1 = row_off[c + 1], rows = a1 - a0;
        const int xw = (st->n_bits[c] + 31) / 32;
        if (a0 < 0 || rows < 0 || a1 > total_rows || x_off[c] < 0 ||
            (rows > 0 && x_off[c] + rows * xw > total_x_words))
            return F2_ERR_INVALID_ARG;
        if (rows > 0) {
            cur.xa = std::min(cur.xa, x_off[c]);
            cur.xb = std::max(cur.xb, x_off[c] + rows * xw);
            cur.max_rows = std::max(cur.max_rows, rows);
        }
        cur.c1 = c + 1;
        cur.r1 = a1;
        bytes += rows * (16 + 4 * (int64_t)xw);
        if (bytes >= target || c + 1 == C) {
            if (cur.r1 > cur.r0) {
                if (cur.xa == INT64_MAX) cur.xa = cur.xb = 0;
                chunks.push_back(cur);
            }
            cur = Chunk{c + 1, c + 1, a1, a1, INT64_MAX, 0, 0};
            bytes = 0;
        }
    }
    if (chunks.empty()) return F2_OK;
    // contexts are independent, so the chunks may go in any order: the one
    // with the smallest largest context last
    std::stable_sort(chunks.begin(), chunks.end(),
                     [](const Chunk& a, const Chunk& b) { return a.max_rows > b.max_rows; });
    HostIO* h = nullptr;
    int rc = host_io(st, &h);
    if (rc != F2_OK) return rc;
    cudaStream_t cs = (cudaStream_t)stream;
    int64_t need_x = 0, need_y = 0, need_c = 0;
    for (const Chunk& k : chunks) {
        need_x = std::max(need_x, k.xb - k.xa);
        need_y = std::max(need_y, k.r1 - k.r0);
        need_c = std::max<int64_t>(need_c, k.c1 - k.c0 + 1);
    }
    cudaError_t e = cudaSuccess;
    if (need_x > h->x_cap || need_y > h->y_cap || need_c > h->c_cap || C + 1 > h->full_cap) {
        e = sync_all(h, cs);
        for (int b = 0; b < LEARN_BUFS && e == cudaSuccess; ++b) {
            int64_t xc = h->x_cap, yc = h->y_cap, cc = h->c_cap, cc2 = h->c_cap;
            e = grow(st, h->x[b], xc, need_x);
            if (e == cudaSuccess) e = grow(st, h->y[b], yc, need_y);
            if (e == cudaSuccess) e = grow(st, h->ro[b], cc, need_c);
            if (e == cudaSuccess) e = grow(st, h->xo[b], cc2, need_c);
        }
        if (e == cudaSuccess) {
            h->x_cap = std::max(h->x_cap, need_x);
            h->y_cap = std::max(h->y_cap, need_y);
            h->c_cap = std::max(h->c_cap, need_c);
            int64_t fc = h->full_cap, fc2 = h->full_cap;
            e = grow(st, h->row_off, fc, (int64_t)C + 1);
            if (e == cudaSuccess) e = grow(st, h->x_off, fc2, (int64_t)C + 1);
            if (e == cudaSuccess) h->full_cap = std::max<int64_t>(h->full_cap, (int64_t)C + 1);
        }
        if (e != cudaSuccess) {
            // a buffer may have been freed: regrow every one on the next call
            h->x_cap = h->y_cap = h->c_cap = h->full_cap = 0;
            return f2_cuda_status(e);
        }
    }
    for (size_t j = 0; j < chunks.size(); ++j) {
        const Chunk& k = chunks[j];
        const int b = (int)(j % LEARN_BUFS);
        const int64_t nc = k.c1 - k.c0;
        // copy stream: this buffer is free once the learn LEARN_BUFS chunks back is done
        e = cudaStreamWaitEvent(h->h2d, h->freed[b], 0);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(h->ro[b], row_off + k.c0, sizeof(int64_t) * (size_t)(nc + 1),
                                cudaMemcpyHostToDevice, h->h2d);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(h->xo[b], x_off + k.c0, sizeof(int64_t) * (size_t)nc, cudaMemcpyHostToDevice,
                                h->h2d);
        if (e == cudaSuccess && k.xb > k.xa)
            e = cudaMemcpyAsync(h->x[b], x + k.xa, sizeof(uint32_t) * (size_t)(k.xb - k.xa), cudaMemcpyHostToDevice,
                                h->h2d);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(h->y[b], y + 4 * k.r0, sizeof(uint4) * (size_t)(k.r1 - k.r0),
                                cudaMemcpyHostToDevice, h->h2d);
        if (e == cudaSuccess) e = cudaEventRecord(h->copied[b], h->h2d);
        // caller's stream: learn the chunk, then release the half
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, h->copied[b], 0);
        if (e != cudaSuccess) return f2_cuda_status(e);
        int blocks = (C + 256) / 256;
        if (blocks > st->num_sms * 4) blocks = st->num_sms * 4;
        rebase_kernel<<<blocks, 256, 0, cs>>>(h->ro[b], h->xo[b], k.c0, k.c1, C, k.xa, h->row_off, h->x_off);
        e = cudaGetLastError();
        if (e != cudaSuccess) return f2_cuda_status(e);
        rc = f2_learn_batched(st, h->row_off, h->x[b], h->x_off, reinterpret_cast<const uint32_t*>(h->y[b]),
                              k.r1 - k.r0, k.xb - k.xa, stream);
        if (rc != F2_OK) return rc;
        e = cudaEventRecord(h->freed[b], cs);
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    return F2_OK;
}

extern "C" int f2_encode_host(const f2_store* cst, int64_t Q, const int32_t* ctx_id, const uint32_t* x,
                              int32_t x_stride_words, uint32_t* y_out, uint8_t* in_span, f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_encode_host");
    if (!cst || Q < 0 || x_stride_words < 1) return F2_ERR_INVALID_ARG;
    if (Q == 0) return F2_OK;
    if (!ctx_id || !x || !y_out || !in_span) return F2_ERR_INVALID_ARG;
    f2_store* st = const_cast<f2_store*>(cst);  // the copy machinery is scratch
    HostIO* h = nullptr;
    int rc = host_io(st, &h);
    if (rc != F2_OK) return rc;
    cudaStream_t cs = (cudaStream_t)stream;
    // at most chunk_bytes of queries per chunk, and at least four chunks when
    // there are enough queries, so that the words of a chunk go out while
    // the next ones are encoded
    const int64_t per_q = 4 + 4 * (int64_t)x_stride_words;
    int64_t qn = st->host_chunk_bytes / per_q;
    qn = std::min(qn, (Q + 3) / 4);
    if (qn < 65536) qn = 65536;
    if (qn > Q) qn = Q;
    cudaError_t e = cudaSuccess;
    if (qn > h->q_cap || qn * x_stride_words > h->qx_cap) {
        e = sync_all(h, cs);
        for (int b = 0; b < ENC_IN && e == cudaSuccess; ++b) {
            int64_t a = h->q_cap, ax = h->qx_cap;
            e = grow(st, h->qc[b], a, qn);
            if (e == cudaSuccess) e = grow(st, h->qx[b], ax, qn * x_stride_words);
        }
        for (int b = 0; b < 2 && e == cudaSuccess; ++b) {
            int64_t a2 = h->q_cap, a3 = h->q_cap;
            e = grow(st, h->qy[b], a2, qn);
            if (e == cudaSuccess) e = grow(st, h->qs[b], a3, qn);
        }
        if (e != cudaSuccess) {
            h->q_cap = h->qx_cap = 0;  // a buffer may have been freed: regrow every one next time
            return f2_cuda_status(e);
        }
        h->q_cap = std::max(h->q_cap, qn);
        h->qx_cap = std::max(h->qx_cap, qn * x_stride_words);
    }
    int j = 0;
    for (int64_t q0 = 0; q0 < Q; q0 += qn, ++j) {
        const int64_t n = std::min(qn, Q - q0);
        const int b = j & 1, bi = j % ENC_IN;
        // in: the input buffer is free once the encode ENC_IN chunks back is done
        e = cudaStreamWaitEvent(h->h2d, h->qused[bi], 0);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(h->qc[bi], ctx_id + q0, sizeof(int32_t) * (size_t)n, cudaMemcpyHostToDevice, h->h2d);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(h->qx[bi], x + q0 * x_stride_words, sizeof(uint32_t) * (size_t)(n * x_stride_words),
                                cudaMemcpyHostToDevice, h->h2d);
        if (e == cudaSuccess) e = cudaEventRecord(h->qcopied[bi], h->h2d);
        // encode: needs the inputs, and the half's outputs read out
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, h->qcopied[bi], 0);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, h->drained[b], 0);
        if (e != cudaSuccess) return f2_cuda_status(e);
        rc = f2_encode_batched(st, n, h->qc[bi], h->qx[bi], x_stride_words, reinterpret_cast<uint32_t*>(h->qy[b]),
                               h->qs[b], stream);
        if (rc != F2_OK) return rc;
        e = cudaEventRecord(h->qused[bi], cs);
        if (e == cudaSuccess) e = cudaEventRecord(h->done[b], cs);
        // out
        if (e == cudaSuccess) e = cudaStreamWaitEvent(h->d2h, h->done[b], 0);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(y_out + 4 * q0, h->qy[b], sizeof(uint4) * (size_t)n, cudaMemcpyDeviceToHost, h->d2h);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(in_span + q0, h->qs[b], (size_t)n, cudaMemcpyDeviceToHost, h->d2h);
        if (e == cudaSuccess) e = cudaEventRecord(h->drained[b], h->d2h);
        if (e != cudaSuccess) return f2_cuda_status(e);
    }
    // the caller's stream passes the call once the last words are on the host
    e = cudaEventRecord(h->last, h->d2h);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, h->last, 0);
    return f2_cuda_status(e);
}
