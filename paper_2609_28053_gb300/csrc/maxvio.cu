// maxvio.cu -- the balance metric MaxVio (arXiv 2609.28053, Sec. 5 Metrics
// and App. E): MaxVio(B) = max_e [f_e(B) / fbar(B) - 1], fbar(B) = K |B| / E,
// in fp64, for the step's summed loads (Global) and for every microbatch
// (Local, the plain mean over the non-empty ones).
//
// One block.  Warps take microbatches: the largest load of the row, then one
// fp64 division and subtraction (the expression is increasing in the load,
// so the maximum of the per-expert values is the value at the largest load).
// Threads take experts for the summed loads.  Thread 0 averages the
// per-microbatch values in ascending microbatch order.
#include "eqb_device.cuh"

namespace eqb {

namespace {

constexpr int kThreads = 512;

__global__ void __launch_bounds__(kThreads) maxvio_kernel(const int32_t* __restrict__ loads,
                                                          const int64_t* __restrict__ off, int M, int E,
                                                          int K, double* out, double* per_mb) {
  extern __shared__ double sv[];  // [M] per-microbatch values
  __shared__ long long wmax[kThreads / 32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;

  for (int l = wid; l < M; l += nw) {
    const int64_t n = off[l + 1] - off[l];
    int m = 0;
    for (int e = lane; e < E; e += 32) m = max(m, loads[(int64_t)l * E + e]);
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) m = max(m, __shfl_xor_sync(kFull, m, s));
    double v = 0.0;
    if (n > 0) {
      const double fbar = (double)K * (double)n / (double)E;
      v = (double)m / fbar - 1.0;
    }
    if (lane == 0) {
      sv[l] = v;
      if (per_mb) per_mb[l] = v;
    }
  }

  long long gm = 0;
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    long long f = 0;
    for (int l = 0; l < M; ++l) f += loads[(int64_t)l * E + e];
    gm = f > gm ? f : gm;
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
    double sum = 0.0;
    int count = 0;
    for (int l = 0; l < M; ++l) {
      if (off[l + 1] > off[l]) {
        sum += sv[l];
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
