/*
 * moeca_probe.h -- measurement helper of the MoECa library (no counterpart in
 * the paper).
 *
 * The fp32 debug path's expert FFN is plain FFMA work on the CUDA cores, so
 * its roofline is the device's fp32 FMA rate, which this call measures on the
 * device it runs on rather than taking a datasheet figure.
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

#ifdef __cplusplus
}
#endif
#endif /* MOECA_PROBE_H_ */
