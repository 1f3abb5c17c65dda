// Store management, layout queries, checkpointing and the affine solve.
#include <stdlib.h>
#include <string.h>

#include <new>

#include "f2_internal.cuh"

using namespace f2;

int f2_cuda_status(cudaError_t e)
{
    if (e == cudaSuccess) return F2_OK;
    if (e == cudaErrorMemoryAllocation) return F2_ERR_OOM;
    return F2_ERR_CUDA;
}

static inline bool aligned(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

cudaError_t f2_dev_alloc(const f2_store* st, void** p, size_t bytes, cudaStream_t cs, bool stream_ordered)
{
    if (st->fail_alloc_in >= 0) {
        if (st->fail_alloc_in == 0) {  // the hooked allocation: fail once, then the hook is off
            st->fail_alloc_in = -1;
            *p = nullptr;
            return cudaErrorMemoryAllocation;
        }
        --st->fail_alloc_in;
    }
    return stream_ordered ? cudaMallocAsync(p, bytes, cs) : cudaMalloc(p, bytes);
}

namespace {

// Grid-stride byte fill of each segment: 16-byte stores between the
// segment's aligned head and tail, single bytes at both ends.
__global__ void __launch_bounds__(256) fill_kernel(F2FillList L)
{
    const size_t tid = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    const size_t nth = (size_t)gridDim.x * blockDim.x;
    for (int k = 0; k < L.n; ++k) {
        uint8_t* p = static_cast<uint8_t*>(L.p[k]);
        const size_t bytes = L.bytes[k];
        const uint8_t b = (uint8_t)L.value[k];
        const uint32_t w = 0x01010101u * b;
        size_t head = (16 - ((uintptr_t)p & 15)) & 15;
        if (head > bytes) head = bytes;
        const size_t n16 = (bytes - head) / 16;
        for (size_t i = tid; i < head; i += nth) p[i] = b;
        uint4* q = reinterpret_cast<uint4*>(p + head);
        for (size_t i = tid; i < n16; i += nth) q[i] = make_uint4(w, w, w, w);
        for (size_t i = head + 16 * n16 + tid; i < bytes; i += nth) p[i] = b;
    }
}

}  // namespace

cudaError_t f2_fill(const F2FillList& L, cudaStream_t cs)
{
    if (L.overflow) return cudaErrorInvalidValue;
    if (L.n == 0) return cudaSuccess;
    unsigned long long total = 0;
    for (int k = 0; k < L.n; ++k) total += L.bytes[k];
    // about 16 KB a block, at most 1024 blocks
    unsigned long long blocks = (total + 16383) / 16384;
    if (blocks > 1024) blocks = 1024;
    if (blocks < 1) blocks = 1;
    fill_kernel<<<(unsigned)blocks, 256, 0, cs>>>(L);
    return cudaGetLastError();
}

int f2_ensure_aux(const f2_store* st)
{
    if (st->aux) return F2_OK;
    int cur = -1;  // created on the store's device
    cudaError_t e = cudaGetDevice(&cur);
    if (e == cudaSuccess && cur != st->device) e = cudaSetDevice(st->device);
    // the second stream carries the kernel of the heaviest width class (the
    // wide or the 4..9-word elimination): at the highest priority its CTAs,
    // and so its longest contexts, are dispatched first
    int least = 0, greatest = 0;
    if (e == cudaSuccess) e = cudaDeviceGetStreamPriorityRange(&least, &greatest);
    if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&st->aux, cudaStreamNonBlocking, greatest);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&st->ev_fork, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&st->ev_join, cudaEventDisableTiming);
    if (cur >= 0 && cur != st->device) cudaSetDevice(cur);
    return f2_cuda_status(e);
}

extern "C" const char* f2_status_string(int status)
{
    switch (status) {
    case F2_OK: return "ok";
    case F2_ERR_INVALID_ARG: return "invalid argument";
    case F2_ERR_NBITS: return "feature width outside [1, 1024]";
    case F2_ERR_CTX_RANGE: return "context id out of range";
    case F2_ERR_ALIGN: return "pointer misaligned";
    case F2_ERR_OOM: return "out of memory";
    case F2_ERR_CUDA: return "CUDA runtime error";
    case F2_ERR_TIMEOUT: return "bounded device wait gave up";
    case F2_ERR_ROWS: return "CSR offsets decreasing or out of bounds";
    case F2_ERR_STRIDE: return "query stride narrower than the context's feature words";
    default: return "unknown status";
    }
}

static void free_store(f2_store* s)
{
    if (!s) return;
    f2_host_io_free(s);
    if (s->aux) cudaStreamDestroy(s->aux);
    if (s->ev_fork) cudaEventDestroy(s->ev_fork);
    if (s->ev_join) cudaEventDestroy(s->ev_join);
    void* ptrs[] = {s->desc,   s->rank,   s->contra,   s->first_contra, s->n_contra, s->rows_seen,
                    s->pivot,  s->bx,     s->bz,       s->status,       s->queue,    s->keybuf,
                    s->counters, s->plan_hist, s->rep_count, s->rep_list, s->rep_dup, s->shard_reps, s->shard_done,
                    s->hand, s->check_rec,
                    s->full_ctr, s->full_cnt, s->full_first,
                    s->enc_bins, s->enc_off, s->enc_sorted, s->enc_items, s->enc_hot, s->enc_tab_off,
                    s->enc_pool, s->timing};
    for (void* p : ptrs)
        if (p) cudaFree(p);
    delete s;
}

static cudaError_t zero_state(f2_store* s, cudaStream_t st)
{
    F2FillList L;  // one launch for the whole state
    L.add(s->rank, sizeof(int32_t) * (size_t)s->num_ctx);
    L.add(s->contra, (size_t)s->num_ctx);
    L.add(s->n_contra, sizeof(unsigned long long) * (size_t)s->num_ctx);
    L.add(s->rows_seen, sizeof(long long) * (size_t)s->num_ctx);
    L.add(s->pivot, sizeof(uint32_t) * (size_t)s->pivot_words);
    L.add(s->bx, sizeof(uint32_t) * (size_t)s->basis_words);
    L.add(s->bz, sizeof(uint4) * (size_t)s->slots);
    L.add(s->first_contra, sizeof(long long) * (size_t)s->num_ctx, 0xff);  // -1
    L.add(s->status, sizeof(int));
    return f2_fill(L, st);
}

extern "C" int f2_create(f2_store** out, int32_t num_ctx, const int32_t* n_bits_host, uint32_t flags,
                         f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_create");
    if (!out) return F2_ERR_INVALID_ARG;
    *out = nullptr;
    if (num_ctx < 0 || (num_ctx > 0 && !n_bits_host) || (flags & ~F2_FLAG_RAW_FEATURES))
        return F2_ERR_INVALID_ARG;
    for (int32_t c = 0; c < num_ctx; ++c)
        if (n_bits_host[c] < 1 || n_bits_host[c] > MAX_N) return F2_ERR_NBITS;
    f2_store* s = new (std::nothrow) f2_store();
    if (!s) return F2_ERR_OOM;
    s->num_ctx = num_ctx;
    s->flags = flags;
    s->heavy_rows = DEFAULT_HEAVY_ROWS;
    s->warp_basis_bytes = DEFAULT_WARP_REGION_BYTES;
    s->warp_work = DEFAULT_WARP_WORK;
    s->dedup = 1;
    s->elim_tables = 1;
    s->small_basis_bytes = DEFAULT_SMALL_REGION_BYTES;
    s->dd_shards = 4;
    s->enc_direct_max = DEFAULT_ENCODE_DIRECT_MAX;
    s->long_call_rows = DEFAULT_LONG_CALL_ROWS;
    s->handoff_min = DEFAULT_HANDOFF_REPS;
    s->enc_table_min = f2_encode_table_min_default();
    s->enc_chunk_shift = f2_encode_chunk_shift_default();
    s->enc_chunk_min = f2_encode_chunk_min_default();
    s->fail_alloc_in = -1;
    s->host_chunk_bytes = DEFAULT_HOST_CHUNK_BYTES;
    if (cudaGetDevice(&s->device) != cudaSuccess ||
        cudaDeviceGetAttribute(&s->num_sms, cudaDevAttrMultiProcessorCount, s->device) != cudaSuccess) {
        delete s;
        return F2_ERR_CUDA;
    }
    const bool raw = (flags & F2_FLAG_RAW_FEATURES) != 0;
    std::vector<CtxDesc> desc((size_t)num_ctx);
    s->n_bits.assign(n_bits_host, n_bits_host + num_ctx);
    s->slot_off.assign((size_t)num_ctx + 1, 0);
    s->xw_off.assign((size_t)num_ctx + 1, 0);
    s->pw_off.assign((size_t)num_ctx + 1, 0);
    for (int32_t c = 0; c < num_ctx; ++c) {
        CtxDesc& cd = desc[(size_t)c];
        cd.n = n_bits_host[c];
        cd.d = raw ? cd.n : cd.n + 1;
        cd.wd = (cd.d + 31) / 32;
        cd.xw = (cd.n + 31) / 32;
        cd.slot_off = s->slot_off[(size_t)c];
        cd.xw_off = s->xw_off[(size_t)c];
        cd.pw_off = s->pw_off[(size_t)c];
        cd.pad = 0;
        s->slot_off[(size_t)c + 1] = cd.slot_off + cd.d;
        s->xw_off[(size_t)c + 1] = cd.xw_off + (int64_t)cd.d * cd.wd;
        s->pw_off[(size_t)c + 1] = cd.pw_off + cd.wd;
        if (cd.wd > s->max_wd) s->max_wd = cd.wd;
        if (cd.xw > s->max_xw) s->max_xw = cd.xw;
        if (cd.d > s->max_d) s->max_d = cd.d;
        if (cd.wd > NARROW_WD) s->n_wide++;
    }
    s->slots = s->slot_off[(size_t)num_ctx];
    s->basis_words = s->xw_off[(size_t)num_ctx];
    s->pivot_words = s->pw_off[(size_t)num_ctx];

    cudaError_t e = cudaSuccess;
    auto alloc = [&](void** p, size_t bytes) {
        if (e == cudaSuccess) e = cudaMalloc(p, bytes ? bytes : 16);
    };
    const size_t C = (size_t)(num_ctx > 0 ? num_ctx : 1);
    alloc((void**)&s->desc, sizeof(CtxDesc) * C);
    alloc((void**)&s->rank, sizeof(int32_t) * C);
    alloc((void**)&s->contra, C);
    alloc((void**)&s->first_contra, sizeof(long long) * C);
    alloc((void**)&s->n_contra, sizeof(unsigned long long) * C);
    alloc((void**)&s->rows_seen, sizeof(long long) * C);
    alloc((void**)&s->pivot, sizeof(uint32_t) * (size_t)s->pivot_words);
    alloc((void**)&s->bx, sizeof(uint32_t) * (size_t)s->basis_words);
    alloc((void**)&s->bz, sizeof(uint4) * (size_t)s->slots);
    alloc((void**)&s->status, sizeof(int));
    // the queue also holds the shard items of split contexts
    alloc((void**)&s->queue, sizeof(int32_t) * (C + (size_t)f2_shard_queue_extra(s->num_sms)));
    alloc((void**)&s->keybuf, sizeof(int32_t) * C);
    alloc((void**)&s->counters, sizeof(int) * CNT_WORDS);
    alloc((void**)&s->rep_count, sizeof(int32_t) * C);
    alloc((void**)&s->shard_reps, sizeof(int32_t) * 8 * C);
    alloc((void**)&s->shard_done, sizeof(int32_t) * C);
    alloc((void**)&s->hand, sizeof(int) * (2 + 6 * C));
    alloc((void**)&s->plan_hist, sizeof(int) * 2 * PLAN_HIST_WORDS);  // the two plans of a learn call
    alloc((void**)&s->full_ctr, sizeof(int) * (4 * C + 1));
    alloc((void**)&s->full_cnt, sizeof(unsigned long long) * C);
    alloc((void**)&s->full_first, sizeof(unsigned long long) * C);
    cudaStream_t st = (cudaStream_t)stream;
    if (e == cudaSuccess && num_ctx)
        e = cudaMemcpyAsync(s->desc, desc.data(), sizeof(CtxDesc) * (size_t)num_ctx,
                            cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) e = zero_state(s, st);
    // the host vector `desc` must outlive the copy
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        int code = f2_cuda_status(e);
        free_store(s);
        return code;
    }
    *out = s;
    return F2_OK;
}

extern "C" void f2_destroy(f2_store* store)
{
    F2_NVTX_RANGE("f2_destroy");
    if (!store) return;
    cudaDeviceSynchronize();
    free_store(store);
}

extern "C" int f2_reset(f2_store* s, f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_reset");
    if (!s) return F2_ERR_INVALID_ARG;
    return f2_cuda_status(zero_state(s, (cudaStream_t)stream));
}

extern "C" int f2_layout(const f2_store* s, int64_t* slot_off, int64_t* xw_off, int64_t* pw_off)
{
    if (!s) return F2_ERR_INVALID_ARG;
    const size_t n = (size_t)s->num_ctx + 1;
    if (slot_off) memcpy(slot_off, s->slot_off.data(), n * sizeof(int64_t));
    if (xw_off) memcpy(xw_off, s->xw_off.data(), n * sizeof(int64_t));
    if (pw_off) memcpy(pw_off, s->pw_off.data(), n * sizeof(int64_t));
    return F2_OK;
}

extern "C" int f2_sizes(const f2_store* s, int32_t* num_ctx, int64_t* slots, int64_t* basis_words,
                        int64_t* pivot_words)
{
    if (!s) return F2_ERR_INVALID_ARG;
    if (num_ctx) *num_ctx = s->num_ctx;
    if (slots) *slots = s->slots;
    if (basis_words) *basis_words = s->basis_words;
    if (pivot_words) *pivot_words = s->pivot_words;
    return F2_OK;
}

extern "C" int f2_get_basis(const f2_store* s, int32_t* rank, uint32_t* pivot_mask, uint32_t* basis_x,
                            uint32_t* basis_z, uint8_t* contra, int64_t* first_contra, uint64_t* n_contra,
                            int64_t* rows_seen, f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_get_basis");
    if (!s) return F2_ERR_INVALID_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    const size_t C = (size_t)s->num_ctx;
    cudaError_t e = cudaSuccess;
    auto cp = [&](void* dst, const void* src, size_t bytes) {
        if (e == cudaSuccess && dst && bytes) e = cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, st);
    };
    cp(rank, s->rank, sizeof(int32_t) * C);
    cp(pivot_mask, s->pivot, sizeof(uint32_t) * (size_t)s->pivot_words);
    cp(basis_x, s->bx, sizeof(uint32_t) * (size_t)s->basis_words);
    cp(basis_z, s->bz, sizeof(uint4) * (size_t)s->slots);
    cp(contra, s->contra, C);
    cp(first_contra, s->first_contra, sizeof(int64_t) * C);
    cp(n_contra, s->n_contra, sizeof(uint64_t) * C);
    cp(rows_seen, s->rows_seen, sizeof(int64_t) * C);
    return f2_cuda_status(e);
}

// ------------------------------------------------------------ affine solve
//
// W[c][j] = z_j for a pivot j, 0 otherwise (the learned map T of Sec. 2.3
// extended by zero on the free coordinates).  One warp per context, lanes
// over slots: coalesced 16-byte stores.
__global__ void __launch_bounds__(256) solve_kernel(StoreDev s, uint4* __restrict__ W)
{
    const int lane = threadIdx.x & 31;
    const int warps = (gridDim.x * blockDim.x) >> 5;
    for (int c = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; c < s.num_ctx; c += warps) {
        const CtxDesc cd = s.desc[c];
        const uint32_t* P = s.pivot + cd.pw_off;
        for (int j = lane; j < cd.d; j += 32) {
            const bool piv = (__ldg(P + (j >> 5)) >> (j & 31)) & 1u;
            W[cd.slot_off + j] = piv ? __ldg(s.bz + cd.slot_off + j) : make_uint4(0, 0, 0, 0);
        }
    }
}

extern "C" int f2_solve_affine(const f2_store* s, uint32_t* W, f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_solve_affine");
    if (!s || (!W && s->slots)) return F2_ERR_INVALID_ARG;
    if (!aligned(W, 16)) return F2_ERR_ALIGN;
    if (s->num_ctx == 0) return F2_OK;
    const int threads = 256;
    int blocks = (int)((s->num_ctx + 7) / 8);
    const int cap = s->num_sms * 8;
    if (blocks > cap) blocks = cap;
    solve_kernel<<<blocks, threads, 0, (cudaStream_t)stream>>>(s->dev(), reinterpret_cast<uint4*>(W));
    return f2_cuda_status(cudaGetLastError());
}

extern "C" int f2_device_status(f2_store* s, int* status, f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_device_status");
    if (!s || !status) return F2_ERR_INVALID_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    int v = 0;
    cudaError_t e = cudaMemcpyAsync(&v, s->status, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e == cudaSuccess) e = cudaMemsetAsync(s->status, 0, sizeof(int), st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return f2_cuda_status(e);
    *status = v;
    return F2_OK;
}

// ------------------------------------------------------------ checkpoints

namespace {
struct CkptHeader {
    char magic[8];
    int32_t version;
    int32_t num_ctx;
    uint32_t flags;
    int32_t pad;
    int64_t slots, basis_words, pivot_words;
};

size_t ckpt_size(const f2_store* s)
{
    const size_t C = (size_t)s->num_ctx;
    return sizeof(CkptHeader) + C * sizeof(int32_t) /* n_bits */ + C * sizeof(int32_t) /* rank */ +
           C /* contra */ + C * 8 * 3 /* first, n_contra, rows_seen */ +
           (size_t)s->pivot_words * 4 + (size_t)s->basis_words * 4 + (size_t)s->slots * 16;
}
}  // namespace

extern "C" int f2_store_export(const f2_store* s, void* host_buf, size_t* size, f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_store_export");
    if (!s || !size) return F2_ERR_INVALID_ARG;
    const size_t need = ckpt_size(s);
    if (!host_buf) {
        *size = need;
        return F2_OK;
    }
    if (*size < need) return F2_ERR_INVALID_ARG;
    *size = need;
    cudaStream_t st = (cudaStream_t)stream;
    char* p = (char*)host_buf;
    CkptHeader h;
    memset(&h, 0, sizeof h);
    memcpy(h.magic, "F2GPUCK1", 8);
    h.version = 1;
    h.num_ctx = s->num_ctx;
    h.flags = s->flags;
    h.slots = s->slots;
    h.basis_words = s->basis_words;
    h.pivot_words = s->pivot_words;
    memcpy(p, &h, sizeof h);
    p += sizeof h;
    const size_t C = (size_t)s->num_ctx;
    memcpy(p, s->n_bits.data(), C * 4);
    p += C * 4;
    cudaError_t e = cudaSuccess;
    auto d2h = [&](const void* src, size_t bytes) {
        if (e == cudaSuccess && bytes) e = cudaMemcpyAsync(p, src, bytes, cudaMemcpyDeviceToHost, st);
        p += bytes;
    };
    d2h(s->rank, C * 4);
    d2h(s->contra, C);
    d2h(s->first_contra, C * 8);
    d2h(s->n_contra, C * 8);
    d2h(s->rows_seen, C * 8);
    d2h(s->pivot, (size_t)s->pivot_words * 4);
    d2h(s->bx, (size_t)s->basis_words * 4);
    d2h(s->bz, (size_t)s->slots * 16);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    return f2_cuda_status(e);
}

extern "C" int f2_store_import(f2_store* s, const void* host_buf, size_t size, f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_store_import");
    if (!s || !host_buf) return F2_ERR_INVALID_ARG;
    const size_t need = ckpt_size(s);
    if (size < need) return F2_ERR_INVALID_ARG;
    const char* p = (const char*)host_buf;
    CkptHeader h;
    memcpy(&h, p, sizeof h);
    if (memcmp(h.magic, "F2GPUCK1", 8) != 0 || h.version != 1 || h.num_ctx != s->num_ctx ||
        h.flags != s->flags || h.slots != s->slots || h.basis_words != s->basis_words ||
        h.pivot_words != s->pivot_words)
        return F2_ERR_INVALID_ARG;
    p += sizeof h;
    const size_t C = (size_t)s->num_ctx;
    if (memcmp(p, s->n_bits.data(), C * 4) != 0) return F2_ERR_INVALID_ARG;
    p += C * 4;
    cudaStream_t st = (cudaStream_t)stream;
    cudaError_t e = cudaSuccess;
    auto h2d = [&](void* dst, size_t bytes) {
        if (e == cudaSuccess && bytes) e = cudaMemcpyAsync(dst, p, bytes, cudaMemcpyHostToDevice, st);
        p += bytes;
    };
    h2d(s->rank, C * 4);
    h2d(s->contra, C);
    h2d(s->first_contra, C * 8);
    h2d(s->n_contra, C * 8);
    h2d(s->rows_seen, C * 8);
    h2d(s->pivot, (size_t)s->pivot_words * 4);
    h2d(s->bx, (size_t)s->basis_words * 4);
    h2d(s->bz, (size_t)s->slots * 16);
    // the caller's buffer must stay valid until the copies complete
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    return f2_cuda_status(e);
}

extern "C" int f2_set_option(f2_store* s, int option, int64_t value)
{
    if (!s) return F2_ERR_INVALID_ARG;
    switch (option) {
    case F2_OPT_HEAVY_ROWS:
        if (value < 1) return F2_ERR_INVALID_ARG;
        s->heavy_rows = value;
        s->heavy_rows_set = 1;
        return F2_OK;
    case F2_OPT_WARP_BASIS_BYTES:
        if (value < 0 || value > 24576) return F2_ERR_INVALID_ARG;
        s->warp_basis_bytes = (value / 16) * 16;
        return F2_OK;
    case F2_OPT_WARP_WORK:
        if (value < 0) return F2_ERR_INVALID_ARG;
        s->warp_work = value;
        s->warp_work_set = 1;
        return F2_OK;
    case F2_OPT_DEDUP:
        if (value != 0 && value != 1) return F2_ERR_INVALID_ARG;
        s->dedup = (int)value;
        return F2_OK;
    case F2_OPT_ENCODE_TABLE_MIN:
        if (value < f2_encode_table_min_floor() || value > (int64_t(1) << 30)) return F2_ERR_INVALID_ARG;
        s->enc_table_min = (int)value;
        return F2_OK;
    case F2_OPT_ENCODE_CHUNK_SHIFT:
        if (value < 11 || value > 25) return F2_ERR_INVALID_ARG;
        s->enc_chunk_shift = (int)value;
        return F2_OK;
    case F2_OPT_ENCODE_CHUNK_MIN:
        if (value < 1) return F2_ERR_INVALID_ARG;
        s->enc_chunk_min = value;
        return F2_OK;
    case F2_OPT_FAIL_ALLOC:
        if (value < -1) return F2_ERR_INVALID_ARG;
        s->fail_alloc_in = value;
        return F2_OK;
    case F2_OPT_ELIM_TABLES:
        if (value != 0 && value != 1) return F2_ERR_INVALID_ARG;
        s->elim_tables = (int)value;
        return F2_OK;
    case F2_OPT_SMALL_BASIS_BYTES:
        if (value < 4096 || value > 24576) return F2_ERR_INVALID_ARG;
        s->small_basis_bytes = (value / 16) * 16;
        return F2_OK;
    case F2_OPT_HANDOFF_REPS:
        if (value < 0 || value > (int64_t(1) << 30)) return F2_ERR_INVALID_ARG;
        s->handoff_min = value;
        return F2_OK;
    case F2_OPT_LONG_CALL_ROWS:
        if (value < 0) return F2_ERR_INVALID_ARG;
        s->long_call_rows = value;
        return F2_OK;
    case F2_OPT_ENCODE_DIRECT_MAX:
        if (value < 0 || value > (int64_t(1) << 30)) return F2_ERR_INVALID_ARG;
        s->enc_direct_max = value;
        return F2_OK;
    case F2_OPT_DEDUP_SHARDS:
        if (value < 1 || value > 8) return F2_ERR_INVALID_ARG;
        s->dd_shards = (int)value;
        return F2_OK;
    case F2_OPT_TIMING:
        if (value != 0 && value != 1) return F2_ERR_INVALID_ARG;
        s->timing_on = (int)value;
        return F2_OK;
    case F2_OPT_HOST_CHUNK_BYTES:
        if (value < (int64_t(1) << 16)) return F2_ERR_INVALID_ARG;
        s->host_chunk_bytes = value;
        return F2_OK;
    default:
        return F2_ERR_INVALID_ARG;
    }
}
