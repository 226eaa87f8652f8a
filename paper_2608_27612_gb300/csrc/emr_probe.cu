// ALU throughput probes for the roofline denominators: FP32 FMA and the
// MUFU (special function unit) ex2, rcp and sin rates, each from 8
// independent dependency chains per thread at full occupancy.
#include <cuda_runtime.h>

#include "../../include/emr_probe.h"

namespace {

constexpr int kProbeThreads = 256;
constexpr int kUnroll = 16;

__device__ __forceinline__ float mufu_ex2(float x) {
  float r;
  asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
__device__ __forceinline__ float mufu_rcp(float x) {
  float r;
  asm volatile("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
__device__ __forceinline__ float mufu_sin(float x) {
  float r;
  asm volatile("sin.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

template <int OP>
__global__ void __launch_bounds__(kProbeThreads) probe_kernel(int iters, float* sink) {
  float a[8];
#pragma unroll
  for (int k = 0; k < 8; k++) a[k] = 0.25f + 1e-3f * float(threadIdx.x + k);
  for (int i = 0; i < iters; i++) {
#pragma unroll
    for (int u = 0; u < kUnroll; u++) {
#pragma unroll
      for (int k = 0; k < 8; k++) {
        if (OP == EMR_PROBE_FFMA) a[k] = fmaf(a[k], 0.999f, 0.0005f);
        if (OP == EMR_PROBE_EX2) a[k] = mufu_ex2(-a[k]);  // stays in [0.5, 1]
        if (OP == EMR_PROBE_RCP) a[k] = mufu_rcp(a[k] + 1.0f);  // stays in [0.5, 1]
        if (OP == EMR_PROBE_SIN) a[k] = mufu_sin(a[k]);
      }
    }
  }
  float s = 0.f;
#pragma unroll
  for (int k = 0; k < 8; k++) s += a[k];
  if (s == 1234.5678f) sink[blockIdx.x] = s;  // keeps the chains live
}

}  // namespace

extern "C" emr_status emr_probe_alu(int32_t op, int32_t blocks, int32_t iters, double* ops, float* ms, float* sink,
                                    void* stream) {
  if (op < EMR_PROBE_FFMA || op > EMR_PROBE_SIN || blocks <= 0 || iters <= 0 || !ops || !ms || !sink)
    return EMR_ERR_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaEvent_t e0, e1;
  if (cudaEventCreate(&e0) != cudaSuccess || cudaEventCreate(&e1) != cudaSuccess) return EMR_ERR_CUDA;
  cudaEventRecord(e0, st);
  switch (op) {
    case EMR_PROBE_FFMA: probe_kernel<EMR_PROBE_FFMA><<<blocks, kProbeThreads, 0, st>>>(iters, sink); break;
    case EMR_PROBE_EX2: probe_kernel<EMR_PROBE_EX2><<<blocks, kProbeThreads, 0, st>>>(iters, sink); break;
    case EMR_PROBE_RCP: probe_kernel<EMR_PROBE_RCP><<<blocks, kProbeThreads, 0, st>>>(iters, sink); break;
    default: probe_kernel<EMR_PROBE_SIN><<<blocks, kProbeThreads, 0, st>>>(iters, sink); break;
  }
  cudaEventRecord(e1, st);
  cudaError_t e = cudaEventSynchronize(e1);
  float t = 0.f;
  if (e == cudaSuccess) e = cudaEventElapsedTime(&t, e0, e1);
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  if (e != cudaSuccess) return EMR_ERR_CUDA;
  *ms = t;
  *ops = double(blocks) * kProbeThreads * double(iters) * kUnroll * 8;
  return EMR_OK;
}
