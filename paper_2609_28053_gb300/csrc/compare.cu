// compare.cu -- the two estimates of the global quantile that Sec. 2 of
// arXiv 2609.28053 contrasts with EQB, on the GPU:
//   rank-averaged QB       every data-parallel shard selects its own K/E
//                          quantile of the margins (exactly, with the same
//                          two radix passes as EQB, run over all shards at
//                          once with one histogram per shard), the shards'
//                          quantiles are averaged and centered as in Eq. (2);
//   fixed-resolution bins  256 equal-width bins of the margins summed over
//                          all tokens; the estimate is the upper edge of the
//                          first bin whose cumulative count reaches r,
//                          centered as in Eq. (2).
// Both finish with one small kernel that forms the fp64 estimates, sums them
// in ascending expert order for the mean and writes b_e = fp32(x_e - mean).
#include <cuda_runtime.h>
#include <stdint.h>

#include "eqb.h"
#include "eqb_device.cuh"

namespace eqb {

namespace {

// b_e = fp32(x_e - mean(x)), mean summed sequentially in ascending e.
__device__ void center_store(double* x, int E, float* b) {
  __shared__ double mean;
  __syncthreads();
  if (threadIdx.x == 0) {
    double acc = 0.0;
    for (int e = 0; e < E; ++e) acc += x[e];
    mean = acc / (double)E;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) b[e] = __double2float_rn(x[e] - mean);
}

// Average of the non-empty shards' quantiles (bf16 [P,E]) per expert,
// summed over the shards in ascending order, then centered.
__global__ void __launch_bounds__(256) shard_average_kernel(const uint16_t* q, const int64_t* off, int P, int E,
                                                            float* b) {
  __shared__ double x[kMaxE];
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    double acc = 0.0;
    int cnt = 0;
    for (int p = 0; p < P; ++p) {
      if (off[p + 1] > off[p]) {
        acc += (double)bf16_bits_to_f32(q[(int64_t)p * E + e]);
        ++cnt;
      }
    }
    x[e] = acc / (double)cnt;
  }
  center_store(x, E, b);
}

// Scratch of the rank average: per-shard histograms H and L [P,E,256],
// u [P,E], rho [P,E] int32 and the shard offsets [P+1] int64.
struct ShardWs {
  int32_t *H, *L;
  uint8_t* u;
  int32_t* rho;
  int64_t* off;
};
size_t carve_shards(void* base, int E, int P, ShardWs* w) {
  size_t o = 0;
  auto take = [&](size_t n) {
    uint8_t* p = base ? static_cast<uint8_t*>(base) + o : nullptr;
    o = (o + n + 255) / 256 * 256;
    return p;
  };
  const size_t PE = (size_t)P * (size_t)E;
  w->H = reinterpret_cast<int32_t*>(take(PE * 256 * 4));
  w->L = reinterpret_cast<int32_t*>(take(PE * 256 * 4));
  w->u = take(PE);
  w->rho = reinterpret_cast<int32_t*>(take(PE * 4));
  w->off = reinterpret_cast<int64_t*>(take(((size_t)P + 1) * 8));
  return o;
}

// Upper edge lo + (u_e + 1) w of the selected bin, then centered.
__global__ void __launch_bounds__(256) bin_edge_kernel(const uint8_t* u, int E, float lo, float w, float* b,
                                                       double* est) {
  __shared__ double x[kMaxE];
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    x[e] = (double)lo + (double)(u[e] + 1) * (double)w;
    if (est) est[e] = x[e];
  }
  center_store(x, E, b);
}

inline eqb_status st(int rc) { return static_cast<eqb_status>(rc); }
inline bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

eqb_status check_common(const eqb_bf16* z, const float* tau, int64_t T, int32_t E, int32_t K, float* b_out,
                        void* workspace, int32_t* err_flag) {
  if (T < 1 || E < 2 || K < 1 || K >= E) return EQB_ERR_INVALID_ARG;
  if (E > kMaxE || (E % 8) != 0) return EQB_ERR_UNSUPPORTED;
  if (T > (int64_t(1) << 31) - (int64_t(1) << 24)) return EQB_ERR_UNSUPPORTED;
  if (!z || !tau || !b_out || !workspace) return EQB_ERR_INVALID_ARG;
  if (!aligned(z, 16) || !aligned(tau, 4) || !aligned(b_out, 4) || !aligned(workspace, 256) ||
      !aligned(err_flag, 4))
    return EQB_ERR_INVALID_ARG;
  return EQB_OK;
}

}  // namespace

}  // namespace eqb

extern "C" {

size_t eqb_rank_averaged_workspace_bytes(int32_t E, int32_t P) {
  if (E < 1 || P < 1) return 0;
  eqb::ShardWs w;
  return eqb::carve_shards(nullptr, E, P, &w);
}

eqb_status eqb_rank_averaged_bias(const eqb_bf16* z, const float* tau, int64_t T, int32_t E, int32_t K,
                                  const int64_t* shard_offsets_host, int32_t P, eqb_bf16* q_shards,
                                  float* b_out, void* workspace, size_t workspace_bytes, int32_t* err_flag,
                                  void* stream) {
  eqb_status rs = eqb::check_common(z, tau, T, E, K, b_out, workspace, err_flag);
  if (rs != EQB_OK) return rs;
  if (P < 1 || P > 65535 || !shard_offsets_host || !q_shards || !eqb::aligned(q_shards, 2))
    return EQB_ERR_INVALID_ARG;
  if (shard_offsets_host[0] != 0 || shard_offsets_host[P] != T) return EQB_ERR_INVALID_ARG;
  for (int p = 0; p < P; ++p)
    if (shard_offsets_host[p + 1] < shard_offsets_host[p]) return EQB_ERR_INVALID_ARG;
  eqb::ShardWs w;
  if (eqb::carve_shards(workspace, E, P, &w) > workspace_bytes) return EQB_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const size_t hb = (size_t)P * (size_t)E * 256 * 4;
  if (cudaMemsetAsync(w.H, 0, hb, s) != cudaSuccess || cudaMemsetAsync(w.L, 0, hb, s) != cudaSuccess ||
      cudaMemcpyAsync(w.off, shard_offsets_host, ((size_t)P + 1) * 8, cudaMemcpyHostToDevice, s) != cudaSuccess)
    return EQB_ERR_CUDA;
  // Both radix passes over all tokens at once, each shard counted into its
  // own histogram, then one selection per (shard, expert).
  eqb::HistArgs h1{z, tau, T, E, nullptr, w.H, err_flag};
  h1.shard_off = w.off;
  h1.P = P;
  if (int rc = eqb::launch_hist(h1, 1, s)) return eqb::st(rc);
  if (int rc = eqb::launch_select_sharded(w.H, E, 1, w.off, P, K, w.u, w.rho, nullptr, err_flag, s))
    return eqb::st(rc);
  eqb::HistArgs h2{z, tau, T, E, w.u, w.L, nullptr};
  h2.shard_off = w.off;
  h2.P = P;
  if (int rc = eqb::launch_hist(h2, 2, s)) return eqb::st(rc);
  if (int rc = eqb::launch_select_sharded(w.L, E, 2, w.off, P, K, w.u, w.rho, q_shards, err_flag, s))
    return eqb::st(rc);
  eqb::shard_average_kernel<<<1, 256, 0, s>>>(q_shards, w.off, P, E, b_out);
  return cudaGetLastError() == cudaSuccess ? EQB_OK : EQB_ERR_CUDA;
}

eqb_status eqb_fixed_hist_bias(const eqb_bf16* z, const float* tau, int64_t T, int32_t E, int32_t K, float lo,
                               float width, float* b_out, double* estimate, void* workspace,
                               size_t workspace_bytes, int32_t* err_flag, void* stream) {
  eqb_status rs = eqb::check_common(z, tau, T, E, K, b_out, workspace, err_flag);
  if (rs != EQB_OK) return rs;
  if (!(width > 0.0f) || width == INFINITY || !(lo == lo) || lo == INFINITY || lo == -INFINITY)
    return EQB_ERR_INVALID_ARG;
  if (!eqb::aligned(estimate, 8)) return EQB_ERR_INVALID_ARG;
  eqb::StepWorkspace w;
  if (eqb::carve_workspace(workspace, E, &w) > workspace_bytes) return EQB_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(w.H, 0, (size_t)E * 1024, s) != cudaSuccess) return EQB_ERR_CUDA;
  eqb::HistArgs h{z, tau, T, E, nullptr, w.H, err_flag};
  h.lo = lo;
  h.inv_w = 1.0f / width;
  if (int rc = eqb::launch_hist(h, 3, s)) return eqb::st(rc);
  const int64_t r = eqb_target_rank(T, E, K);
  if (int rc = eqb::launch_select(w.H, E, 3, r, w.u, w.rho, nullptr, err_flag, s)) return eqb::st(rc);
  eqb::bin_edge_kernel<<<1, 256, 0, s>>>(w.u, E, lo, width, b_out, estimate);
  return cudaGetLastError() == cudaSuccess ? EQB_OK : EQB_ERR_CUDA;
}

}  // extern "C"
