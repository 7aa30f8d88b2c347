/*
 * moeca_probe.h -- measurement helper of the MoECa library (no counterpart in
 * the paper).
 *
 * The fp32 debug path's expert FFN is plain FFMA work on the CUDA cores, so
 * its roofline is the device's fp32 FMA rate, which moeca_probe_ffma measures
 * on the device it runs on rather than taking a datasheet figure.
 *
 * moeca_probe_stream measures what a plain streaming kernel reaches at the
 * size and shape of the combine's traffic (Eq. 8: a token's rows read, one
 * row written): at tens of MB a launch's ramp and drain are a sizeable part
 * of its time, so the large-copy HBM peak is out of reach for any kernel of
 * that size, and this figure says how far.
 */
#ifndef MOECA_PROBE_H_
#define MOECA_PROBE_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Measure the fp32 FFMA throughput of CUDA device `device`: a kernel of
 * independent register FMA chains (8 per thread, no memory traffic in the
 * loop), 1024 threads per block, 2 blocks per SM, timed with CUDA events
 * after one warm-up launch.  *tflops receives 2 x FMAs / second / 1e12 and
 * *ms the timed launch's duration.  Allocates a 16-byte device buffer for
 * the kernel's result (so the chains are not optimised away) and frees it;
 * synchronises the device.  Returns 0, or -1 (NULL argument, bad device) /
 * -3 (a CUDA call failed). */
int32_t moeca_probe_ffma(int32_t device, int32_t iterations, double* tflops, double* ms);

/* Measure the streaming rate of CUDA device `device` at one shape: a kernel
 * reads `rows` rows of `row_bytes` bytes for each of `n_tokens` tokens (one
 * contiguous [n_tokens, rows, row_bytes] array), adds them as integers and
 * writes one row per token ([n_tokens, row_bytes]); one warp per token, every
 * row's 16-byte chunk of a lane loaded before use, up to four blocks of 8
 * warps per SM.  Before each launch a 512 MB buffer is read, so the launch
 * finds the L2 cache holding only clean lines of other data.  Two untimed
 * launches, then `reps` launches timed with CUDA events one by one; *us
 * receives the median duration in microseconds and *gbs the bytes read and
 * written per launch over it, in GB/s.  Allocates the three buffers (at most
 * 8 GB in all) and frees them; synchronises the device.  Constraints:
 * 1 <= rows <= 10, 16 <= row_bytes <= 65536 and a multiple of 16,
 * n_tokens >= 1, 1 <= reps <= 1000.  Returns 0, or -1 (a NULL pointer, bad
 * device, a constraint broken) / -3 (a CUDA call failed, allocation
 * included). */
int32_t moeca_probe_stream(int32_t device, int64_t n_tokens, int32_t rows, int32_t row_bytes, int32_t reps,
                           double* gbs, double* us);

#ifdef __cplusplus
}
#endif
#endif /* MOECA_PROBE_H_ */
