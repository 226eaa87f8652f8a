// Batched forward pass of assembled substrate networks (one CTA per network):
// every non-input node takes the sigmoid of the weighted sum of its sources'
// previous values, all nodes at once (synchronous update), for a fixed number
// of steps; input nodes hold the pattern. Patterns share the pass: node values
// are [node][pattern] in shared memory, two buffers.
#include <cuda_runtime.h>

#include "../../include/emr.h"

namespace {

constexpr int kAnnThreads = 256;

__global__ void __launch_bounds__(kAnnThreads) ann_forward_kernel(int32_t n_in, int32_t n_out,
                                                                  const int64_t* __restrict__ node_off,
                                                                  const int64_t* __restrict__ conn_off,
                                                                  const int32_t* __restrict__ conn_src,
                                                                  const int32_t* __restrict__ conn_dst,
                                                                  const float* __restrict__ conn_w, int32_t K,
                                                                  const float* __restrict__ patterns, int32_t steps,
                                                                  float* __restrict__ out) {
  extern __shared__ float sm[];
  const int64_t g = blockIdx.x;
  const int32_t N = n_in + n_out + int32_t(node_off[g + 1] - node_off[g]);
  const int64_t c0 = conn_off[g], c1 = conn_off[g + 1];
  float* cur = sm;
  float* nxt = sm + size_t(N) * K;
  int32_t* in_beg = reinterpret_cast<int32_t*>(sm + 2 * size_t(N) * K);  // [N + 1]: connections into node n
  // connections are sorted by destination: node n's are [in_beg[n], in_beg[n + 1])
  for (int32_t n = threadIdx.x; n <= N; n += blockDim.x) {
    int64_t lo = c0, hi = c1;  // first connection with dst >= n
    while (lo < hi) {
      const int64_t mid = (lo + hi) >> 1;
      if (conn_dst[mid] < n) lo = mid + 1; else hi = mid;
    }
    in_beg[n] = int32_t(lo - c0);
  }
  for (int32_t t = threadIdx.x; t < N * K; t += blockDim.x) {
    const int32_t n = t / K, k = t - n * K;
    cur[t] = n < n_in ? patterns[size_t(k) * n_in + n] : 0.f;
    nxt[t] = cur[t];
  }
  __syncthreads();
  for (int32_t step = 0; step < steps; step++) {
    for (int32_t t = threadIdx.x; t < (N - n_in) * K; t += blockDim.x) {
      const int32_t n = n_in + t / K, k = t % K;
      float z = 0.f;
      for (int32_t e = in_beg[n]; e < in_beg[n + 1]; e++)
        z = fmaf(conn_w[c0 + e], cur[size_t(conn_src[c0 + e]) * K + k], z);
      nxt[size_t(n) * K + k] = 1.f / (1.f + expf(-z));
    }
    __syncthreads();
    float* tmp = cur;
    cur = nxt;
    nxt = tmp;
  }
  for (int32_t t = threadIdx.x; t < K * n_out; t += blockDim.x) {
    const int32_t k = t / n_out, o = t - k * n_out;
    out[(size_t(g) * K + k) * n_out + o] = cur[size_t(n_in + o) * K + k];
  }
}

}  // namespace

extern "C" emr_status emr_ann_forward(int32_t P, int32_t n_in, int32_t n_out, int32_t max_hidden,
                                      const int64_t* node_off, const int64_t* conn_off, const int32_t* conn_src,
                                      const int32_t* conn_dst, const float* conn_w, int32_t K, const float* patterns,
                                      int32_t steps, float* out, void* stream) {
  if (P <= 0 || n_in <= 0 || n_out <= 0 || max_hidden < 0 || K <= 0 || steps < 0 || !node_off || !conn_off ||
      !patterns || !out)
    return EMR_ERR_ARG;
  const size_t N = size_t(n_in) + size_t(n_out) + size_t(max_hidden);
  const size_t smem = 2 * N * size_t(K) * 4 + (N + 1) * 4;
  int dev = 0, limit = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&limit, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
    return EMR_ERR_CUDA;
  if (smem > size_t(limit)) return EMR_ERR_RANGE;
  if (cudaFuncSetAttribute(ann_forward_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)) != cudaSuccess)
    return EMR_ERR_CUDA;
  ann_forward_kernel<<<unsigned(P), kAnnThreads, smem, static_cast<cudaStream_t>(stream)>>>(
      n_in, n_out, node_off, conn_off, conn_src, conn_dst, conn_w, K, patterns, steps, out);
  return cudaGetLastError() == cudaSuccess ? EMR_OK : EMR_ERR_CUDA;
}
