// Map pooling (Sec. 3): the exact-context bases of one (f, m) group -- or the
// shards of one context -- are combined and eliminated together; the group
// shares one map if the equations are consistent (and, as the caller
// decides, the output masks match), else its contexts keep separate maps.
//
// The merge is a learn call on a new store: each group is one context of
// raw feature rows (the members' phi-space basis rows, members in context
// order, pivots in increasing order), so the group's basis is the reduced
// echelon form of the union of the members' spans and its contradiction
// flag marks inconsistent equations.  The elimination kernels are reused.
#include <vector>

#include "f2_internal.cuh"

using namespace f2;

namespace {

// One warp per source context: lane over slots; the i-th pivot row of
// context c becomes row member_row[c] + i of the merge batch.
__global__ void __launch_bounds__(256) merge_gather_kernel(StoreDev s, const int64_t* __restrict__ member_row,
                                                           const int64_t* __restrict__ member_word,
                                                           uint32_t* __restrict__ x, uint4* __restrict__ y)
{
    const int lane = threadIdx.x & 31;
    const int warps = (gridDim.x * blockDim.x) >> 5;
    for (int c = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; c < s.num_ctx; c += warps) {
        const int64_t r0 = member_row[c];
        if (r0 < 0) continue;  // not merged
        const CtxDesc cd = s.desc[c];
        const uint32_t* P = s.pivot + cd.pw_off;
        int below = 0;  // pivots in the words before the current one
        for (int w = 0; w < cd.wd; ++w) {
            const uint32_t pw = __ldg(P + w);
            const int k = 32 * w + lane;
            if ((pw >> lane) & 1u) {
                const int i = below + __popc(pw & ((1u << lane) - 1u));
                y[r0 + i] = __ldg(s.bz + cd.slot_off + k);
                const uint32_t* src = s.bx + cd.xw_off + (int64_t)k * cd.wd;
                uint32_t* dst = x + member_word[c] + (int64_t)i * cd.wd;
                for (int v = 0; v < cd.wd; ++v) dst[v] = __ldg(src + v);
            }
            below += __popc(pw);
        }
    }
}

}  // namespace

extern "C" int f2_merge_bases(const f2_store* src, int32_t num_groups, const int32_t* group_of,
                              const uint32_t* out_mask, f2_store** out, uint8_t* mask_ok, f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_merge_bases");
    if (!out) return F2_ERR_INVALID_ARG;
    *out = nullptr;
    if (!src || num_groups < 0 || (src->num_ctx > 0 && !group_of)) return F2_ERR_INVALID_ARG;
    const int32_t C = src->num_ctx;
    const bool raw = (src->flags & F2_FLAG_RAW_FEATURES) != 0;
    // each group: members of one width d
    std::vector<int32_t> d_of(num_groups, 0);
    for (int32_t c = 0; c < C; ++c) {
        const int32_t g = group_of[c];
        if (g < -1 || g >= num_groups) return F2_ERR_CTX_RANGE;
        if (g < 0) continue;
        const int32_t d = raw ? src->n_bits[c] : src->n_bits[c] + 1;
        if (d_of[g] != 0 && d_of[g] != d) return F2_ERR_NBITS;
        d_of[g] = d;
    }
    for (int32_t g = 0; g < num_groups; ++g)
        if (d_of[g] == 0 || d_of[g] > MAX_N) return d_of[g] == 0 ? F2_ERR_INVALID_ARG : F2_ERR_NBITS;
    cudaStream_t cs = (cudaStream_t)stream;
    // the members' ranks fix the layout of the merge batch
    std::vector<int32_t> rank(C > 0 ? C : 1);
    cudaError_t e = cudaSuccess;
    if (C > 0) e = cudaMemcpyAsync(rank.data(), src->rank, sizeof(int32_t) * (size_t)C, cudaMemcpyDeviceToHost, cs);
    if (e == cudaSuccess) e = cudaStreamSynchronize(cs);
    if (e != cudaSuccess) return f2_cuda_status(e);
    std::vector<int64_t> g_rows(num_groups, 0);
    for (int32_t c = 0; c < C; ++c)
        if (group_of[c] >= 0) g_rows[group_of[c]] += rank[c];
    std::vector<int64_t> row_off(num_groups + 1, 0), x_off(num_groups > 0 ? num_groups : 1, 0);
    int64_t words = 0;
    for (int32_t g = 0; g < num_groups; ++g) {
        row_off[g + 1] = row_off[g] + g_rows[g];
        x_off[g] = words;
        words += g_rows[g] * ((d_of[g] + 31) / 32);
    }
    std::vector<int64_t> member_row(C > 0 ? C : 1, -1), member_word(C > 0 ? C : 1, 0);
    {
        std::vector<int64_t> next(row_off.begin(), row_off.end() - 1);
        for (int32_t c = 0; c < C; ++c) {
            const int32_t g = group_of[c];
            if (g < 0) continue;
            member_row[c] = next[g];
            member_word[c] = x_off[g] + (next[g] - row_off[g]) * ((d_of[g] + 31) / 32);
            next[g] += rank[c];
        }
    }
    const int64_t R = row_off[num_groups];
    int rc = f2_create(out, num_groups, d_of.data(), F2_FLAG_RAW_FEATURES, stream);
    if (rc != F2_OK) return rc;
    int64_t *d_row_off = nullptr, *d_x_off = nullptr, *d_member_row = nullptr, *d_member_word = nullptr;
    uint32_t* d_x = nullptr;
    uint4* d_y = nullptr;
    auto am = [&](void** p, size_t bytes) {
        if (e == cudaSuccess) e = f2_dev_alloc(src, p, bytes ? bytes : 16, cs, true);
    };
    am((void**)&d_row_off, sizeof(int64_t) * (size_t)(num_groups + 1));
    am((void**)&d_x_off, sizeof(int64_t) * x_off.size());
    am((void**)&d_member_row, sizeof(int64_t) * member_row.size());
    am((void**)&d_member_word, sizeof(int64_t) * member_word.size());
    am((void**)&d_x, sizeof(uint32_t) * (size_t)words);
    am((void**)&d_y, sizeof(uint4) * (size_t)R);
    auto up = [&](void* dst, const void* srcp, size_t bytes) {
        if (e == cudaSuccess && bytes) e = cudaMemcpyAsync(dst, srcp, bytes, cudaMemcpyHostToDevice, cs);
    };
    up(d_row_off, row_off.data(), sizeof(int64_t) * row_off.size());
    up(d_x_off, x_off.data(), sizeof(int64_t) * (size_t)num_groups);
    up(d_member_row, member_row.data(), sizeof(int64_t) * (size_t)C);
    up(d_member_word, member_word.data(), sizeof(int64_t) * (size_t)C);
    if (e == cudaSuccess && C > 0) {
        int blocks = (C + 7) / 8;
        if (blocks > src->num_sms * 16) blocks = src->num_sms * 16;
        merge_gather_kernel<<<blocks, 256, 0, cs>>>(src->dev(), d_member_row, d_member_word, d_x, d_y);
        e = cudaGetLastError();
    }
    if (e == cudaSuccess && num_groups > 0) {
        rc = f2_learn_batched(*out, d_row_off, d_x, d_x_off, reinterpret_cast<const uint32_t*>(d_y), R, words,
                              stream);
        if (rc != F2_OK) e = cudaErrorUnknown;
    }
    const void* tmp[] = {d_row_off, d_x_off, d_member_row, d_member_word, d_x, d_y};
    for (const void* p : tmp)
        if (p) cudaFreeAsync(const_cast<void*>(p), cs);
    // the host arrays above are read by the copies: wait before returning
    const cudaError_t es = cudaStreamSynchronize(cs);
    if (e == cudaSuccess) e = es;
    if (e != cudaSuccess || rc != F2_OK) {
        f2_destroy(*out);
        *out = nullptr;
        return rc != F2_OK ? rc : f2_cuda_status(e);
    }
    if (mask_ok) {
        // output masks (the learned bits of each context) must be equal for
        // a shared map; without masks every group passes
        std::vector<int32_t> first(num_groups, -1);
        for (int32_t g = 0; g < num_groups; ++g) mask_ok[g] = 1;
        for (int32_t c = 0; c < C && out_mask; ++c) {
            const int32_t g = group_of[c];
            if (g < 0) continue;
            if (first[g] < 0) {
                first[g] = c;
            } else {
                for (int v = 0; v < 4; ++v)
                    if (out_mask[4 * c + v] != out_mask[4 * first[g] + v]) mask_ok[g] = 0;
            }
        }
    }
    return F2_OK;
}
