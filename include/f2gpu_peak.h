/*
 * f2gpu_peak.h -- measurement aid of libf2gpu.so (no counterpart in the
 * paper): an integer-pipe throughput probe that calibrates the ALU roofline
 * against which the elimination and encode kernels are reported.
 */
#ifndef F2GPU_PEAK_H
#define F2GPU_PEAK_H

#include <stdint.h>

#include "f2gpu.h"

#ifdef __cplusplus
extern "C" {
#endif

/*
 * Launch `blocks` CTAs of 256 threads; every thread executes `iters` rounds of
 * eight independent 3-input XOR instructions (PTX lop3.b32).  *lop3_per_launch
 * (host, may be NULL) receives the number of LOP3 lane-operations the launch
 * executes; time the launch with CUDA events on `stream`.  out_dev (device,
 * `blocks` uint32) is written only to keep the work observable.
 * Errors: F2_ERR_INVALID_ARG (NULL out_dev, blocks < 1 or iters < 1), F2_ERR_CUDA.
 */
int f2_peak_lop3(uint32_t* out_dev, int32_t blocks, int32_t iters, int64_t* lop3_per_launch,
                 f2_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* F2GPU_PEAK_H */
