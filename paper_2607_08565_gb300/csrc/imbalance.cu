// Windowed load imbalance (Section 3.2, Figure 3(c)): each instance's load in
// a window is its average number of running requests there, and the window's
// imbalance is the maximum load over the mean across the instances. Both
// loads and their mean share the window length, so the kernels keep the
// running-request time S_i(w) in integer ticks and report max_i S_i(w), its
// lowest maximising instance and sum_i S_i(w); the imbalance is N max / sum.
//
//   k_imbalance_acc     thread per request: its running time cut at the
//                       window edges, added to S_{inst}(w) of each window it
//                       overlaps (atomicAdd on a [n_windows][N] grid).
//   k_imbalance_reduce  warp per window: lanes over the instances, maximum
//                       (lowest instance on ties) and sum by shuffles.

#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>

#include "smetric_impl.cuh"
#include "call_range.cuh"

using namespace smetric;

namespace {

constexpr unsigned kFullMask = 0xffffffffu;

__global__ void __launch_bounds__(256)
    k_imbalance_acc(const int32_t* __restrict__ inst, const int64_t* __restrict__ start,
                    const int64_t* __restrict__ end, int32_t n, int32_t N, int64_t T, int32_t n_windows,
                    unsigned long long* __restrict__ acc, int32_t* status) {
  const int64_t span = (int64_t)n_windows * T;
  for (int64_t r = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; r < n; r += (int64_t)gridDim.x * blockDim.x) {
    const int32_t i = inst[r];
    const int64_t s = start[r];
    int64_t e = end[r];
    if (i < 0 || i >= N || s < 0 || e < s) {
      latch_error(status, SMETRIC_ERR_INVALID_ARG);
      continue;
    }
    if (s >= span || e == s) continue;
    e = e < span ? e : span;
    // windows w with w T < e, from the one holding s; each overlap is positive
    for (int64_t w = s / T; w * T < e; ++w) {
      const int64_t lo = w * T, hi = lo + T;
      const int64_t a = s > lo ? s : lo, b = e < hi ? e : hi;
      atomicAdd(acc + w * N + i, (unsigned long long)(b - a));
    }
  }
}

__global__ void __launch_bounds__(256)
    k_imbalance_reduce(const unsigned long long* __restrict__ acc, int32_t N, int32_t n_windows,
                       int64_t* __restrict__ out_max, int32_t* __restrict__ out_argmax,
                       int64_t* __restrict__ out_sum) {
  const int lane = threadIdx.x & 31;
  const int64_t tw = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t w = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); w < n_windows; w += tw) {
    long long mx = -1, sm = 0;
    int am = 0;
    for (int i = lane; i < N; i += 32) {  // increasing i: strict > keeps the lowest
      const long long v = (long long)acc[w * N + i];
      sm += v;
      if (v > mx) {
        mx = v;
        am = i;
      }
    }
    for (int o = 16; o; o >>= 1) {
      const long long omx = __shfl_xor_sync(kFullMask, mx, o);
      const int oam = __shfl_xor_sync(kFullMask, am, o);
      sm += __shfl_xor_sync(kFullMask, sm, o);
      if (omx > mx || (omx == mx && oam < am)) {
        mx = omx;
        am = oam;
      }
    }
    if (lane == 0) {
      out_max[w] = mx;
      out_argmax[w] = am;
      out_sum[w] = sm;
    }
  }
}

}  // namespace

extern "C" {

int64_t smetric_imbalance_workspace_bytes(int32_t n_windows, int32_t num_instances) {
  if (n_windows < 0 || num_instances < 0) return 0;
  return (int64_t)sizeof(unsigned long long) * n_windows * num_instances;
}

int smetric_window_imbalance(smetric_index* idx, const int32_t* d_instance, const int64_t* d_start,
                             const int64_t* d_end, int32_t n_requests, int64_t window, int32_t n_windows,
                             void* d_workspace, int64_t workspace_bytes, int64_t* d_max, int32_t* d_argmax,
                             int64_t* d_sum, smetric_stream_t stream) {
  CallRange range("smetric_window_imbalance");
  int rc = check_device(idx);
  if (rc) return rc;
  const int32_t N = idx->cfg.num_instances;
  if (n_requests < 0 || n_requests > SMETRIC_IMBALANCE_MAX_REQUESTS || window < 1 ||
      window > SMETRIC_IMBALANCE_MAX_WINDOW || n_windows < 0 ||
      (int64_t)n_windows * N > SMETRIC_IMBALANCE_MAX_CELLS || (int64_t)n_windows > (1LL << 62) / window)
    return SMETRIC_ERR_INVALID_ARG;
  if (n_windows == 0) return SMETRIC_OK;
  const int64_t need = smetric_imbalance_workspace_bytes(n_windows, N);
  if (!d_max || !d_argmax || !d_sum || !d_workspace || workspace_bytes < need ||
      (reinterpret_cast<uintptr_t>(d_workspace) & 7) ||
      (n_requests > 0 && (!d_instance || !d_start || !d_end)))
    return SMETRIC_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  unsigned long long* acc = static_cast<unsigned long long*>(d_workspace);
  if (cudaMemsetAsync(acc, 0, (size_t)need, s) != cudaSuccess) return cuda_status(cudaErrorUnknown);
  if (n_requests > 0) {
    const int64_t want = ((int64_t)n_requests + 255) / 256;
    const unsigned grid = (unsigned)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)idx->num_sms * 8));
    k_imbalance_acc<<<grid, 256, 0, s>>>(d_instance, d_start, d_end, n_requests, N, window, n_windows, acc,
                                         idx->status);
    idx->launches += 1;
  }
  const int64_t want = ((int64_t)n_windows + 7) / 8;
  const unsigned grid = (unsigned)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)idx->num_sms * 8));
  k_imbalance_reduce<<<grid, 256, 0, s>>>(acc, N, n_windows, d_max, d_argmax, d_sum);
  idx->launches += 1;
  return cuda_status(cudaGetLastError());
}

}  // extern "C"
