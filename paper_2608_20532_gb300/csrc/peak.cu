// Integer-pipe throughput probe used to calibrate the ALU roofline: every
// thread runs eight independent chains of 3-input XOR (one LOP3 each).
#include "f2_internal.cuh"
#include "f2gpu_peak.h"

namespace {

__global__ void __launch_bounds__(256) lop3_peak_kernel(uint32_t* out, int iters, uint32_t seed)
{
    uint32_t a[8], b = seed ^ threadIdx.x, c = seed * 0x9e3779b9u + blockIdx.x;
#pragma unroll
    for (int j = 0; j < 8; ++j) a[j] = b * (j + 1) + c;
    for (int i = 0; i < iters; ++i) {
#pragma unroll
        for (int j = 0; j < 8; ++j) asm volatile("lop3.b32 %0, %0, %1, %2, 0x96;" : "+r"(a[j]) : "r"(b), "r"(c));
        b += 0x01000193u;  // keep the inputs live (IADD on the other integer pipe)
    }
    uint32_t r = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) r ^= a[j];
    if (r == 0x12345678u) out[blockIdx.x] = r;  // practically never taken; defeats dead-code removal
}

}  // namespace

extern "C" int f2_peak_lop3(uint32_t* out_dev, int32_t blocks, int32_t iters, int64_t* lop3_per_launch,
                            f2_stream_t stream)
{
    F2_NVTX_RANGE("f2_peak_lop3");
    if (!out_dev || blocks < 1 || iters < 1) return F2_ERR_INVALID_ARG;
    lop3_peak_kernel<<<blocks, 256, 0, (cudaStream_t)stream>>>(out_dev, iters, 0x2545F491u);
    if (lop3_per_launch) *lop3_per_launch = (int64_t)blocks * 256 * (int64_t)iters * 8;
    return f2_cuda_status(cudaGetLastError());
}
