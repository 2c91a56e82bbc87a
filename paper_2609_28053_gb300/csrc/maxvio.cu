// maxvio.cu -- the balance metric MaxVio (arXiv 2609.28053, Sec. 5 Metrics
// and App. E): MaxVio(B) = max_e [f_e(B) / fbar(B) - 1], fbar(B) = K |B| / E,
// in fp64, for the step's summed loads (Global) and for every microbatch
// (Local, the plain mean over the non-empty ones).
//
// One block.  Warps take microbatches for the largest load of each row, then
// one thread per microbatch does the fp64 division and subtraction (the
// expression is increasing in the load, so the maximum of the per-expert
// values is the value at the largest load).  Threads take experts for the
// summed loads.  Thread 0 averages the per-microbatch values in ascending
// microbatch order.
#include "eqb_device.cuh"

namespace eqb {

namespace {

constexpr int kThreads = 512;

__global__ void __launch_bounds__(kThreads) maxvio_kernel(const int32_t* __restrict__ loads,
                                                          const int64_t* __restrict__ off, int M, int E,
                                                          int K, double* out, double* per_mb) {
  // [M]: the largest load of each microbatch, then its value (NaN marks an
  // empty microbatch, which the mean skips; per_mb gets 0 for it)
  extern __shared__ double sv[];
  __shared__ long long wmax[kThreads / 32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;

  // Largest load of every microbatch (warps take microbatches).
  for (int l = wid; l < M; l += nw) {
    int m = 0;
    for (int e = lane; e < E; e += 32) m = max(m, loads[(int64_t)l * E + e]);
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) m = max(m, __shfl_xor_sync(kFull, m, s));
    if (lane == 0) sv[l] = (double)m;
  }
  __syncthreads();
  // The fp64 values, one thread per microbatch: fp64 throughput is low on
  // this part, so no lane repeats another's division.
  for (int l = threadIdx.x; l < M; l += blockDim.x) {
    const int64_t n = off[l + 1] - off[l];
    double v = 0.0;
    if (n > 0) {
      const double fbar = (double)K * (double)n / (double)E;
      v = sv[l] / fbar - 1.0;
    }
    sv[l] = n > 0 ? v : __longlong_as_double(0x7ff8000000000000LL);
    if (per_mb) per_mb[l] = v;
  }

  // Summed loads: eight rows in flight per thread (integer sums are exact
  // in any order).
  long long gm = 0;
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    long long f[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    int l = 0;
    for (; l + 8 <= M; l += 8) {
#pragma unroll
      for (int u = 0; u < 8; ++u) f[u] += loads[(int64_t)(l + u) * E + e];
    }
    for (; l < M; ++l) f[0] += loads[(int64_t)l * E + e];
    const long long t = ((f[0] + f[1]) + (f[2] + f[3])) + ((f[4] + f[5]) + (f[6] + f[7]));
    gm = t > gm ? t : gm;
  }
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) {
    const long long o = __shfl_xor_sync(kFull, gm, s);
    gm = o > gm ? o : gm;
  }
  if (lane == 0) wmax[wid] = gm;
  __syncthreads();

  if (threadIdx.x == 0) {
    long long fm = 0;
    for (int w = 0; w < nw; ++w) fm = wmax[w] > fm ? wmax[w] : fm;
    const int64_t T = off[M] - off[0];
    const double fbar = (double)K * (double)T / (double)E;
    out[0] = (double)fm / fbar - 1.0;
    // ascending microbatch order, from shared memory (a global load per
    // microbatch here would serialise M round trips)
    double sum = 0.0;
    int count = 0;
    for (int l = 0; l < M; ++l) {
      const double v = sv[l];
      if (v == v) {  // not the empty-microbatch mark
        sum += v;
        ++count;
      }
    }
    out[1] = count > 0 ? sum / (double)count : 0.0;
  }
}

}  // namespace

int launch_maxvio(const int32_t* loads, const int64_t* off, int M, int E, int K, double* out, double* per_mb,
                  cudaStream_t s) {
  const int smem = M * static_cast<int>(sizeof(double));
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(maxvio_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return kErrCuda;
  maxvio_kernel<<<1, kThreads, smem, s>>>(loads, off, M, E, K, out, per_mb);
  return cudaGetLastError() == cudaSuccess ? kOk : kErrCuda;
}

}  // namespace eqb
