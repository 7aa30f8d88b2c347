// fp32 FMA-throughput probe (include/moeca_probe.h): the roofline of the fp32
// debug path's SIMT expert FFN.
#include <cuda_runtime.h>

#include "moeca_probe.h"

namespace {

constexpr int kChains = 8;
constexpr int kThreads = 1024;

__global__ void __launch_bounds__(kThreads) ffma_probe_kernel(float* out, int iters, float b, float c) {
  float a[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) a[j] = static_cast<float>(threadIdx.x) * 1e-3f + static_cast<float>(j);
#pragma unroll 4
  for (int it = 0; it < iters; ++it) {
#pragma unroll
    for (int j = 0; j < kChains; ++j) a[j] = fmaf(a[j], b, c);
  }
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < kChains; ++j) s += a[j];
  // Never true for these inputs; keeps every chain live.
  if (s == -1.2345e30f) out[0] = s;
}

}  // namespace

extern "C" int32_t moeca_probe_ffma(int32_t device, int32_t iterations, double* tflops, double* ms) {
  if (!tflops || !ms || iterations < 1) return -1;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev) {
    cudaGetLastError();
    return -1;
  }
  int n_sms = 0;
  float* buf = nullptr;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  float t = 0.f;
  const bool ok = cudaSetDevice(device) == cudaSuccess &&
                  cudaDeviceGetAttribute(&n_sms, cudaDevAttrMultiProcessorCount, device) == cudaSuccess &&
                  cudaMalloc(&buf, 16) == cudaSuccess && cudaEventCreate(&e0) == cudaSuccess &&
                  cudaEventCreate(&e1) == cudaSuccess;
  const dim3 grid(2 * n_sms), block(kThreads);
  bool ran = false;
  if (ok) {
    ffma_probe_kernel<<<grid, block>>>(buf, iterations, 0.99999f, 1e-6f);  // warm-up
    cudaEventRecord(e0);
    ffma_probe_kernel<<<grid, block>>>(buf, iterations, 0.99999f, 1e-6f);
    cudaEventRecord(e1);
    ran = cudaEventSynchronize(e1) == cudaSuccess && cudaGetLastError() == cudaSuccess &&
          cudaEventElapsedTime(&t, e0, e1) == cudaSuccess;
  }
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  if (buf) cudaFree(buf);
  if (!ok || !ran || t <= 0.f) {
    cudaGetLastError();
    return -3;
  }
  const double fmas = static_cast<double>(grid.x) * kThreads * kChains * static_cast<double>(iterations);
  *ms = t;
  *tflops = 2.0 * fmas / (t * 1e-3) / 1e12;
  return 0;
}
