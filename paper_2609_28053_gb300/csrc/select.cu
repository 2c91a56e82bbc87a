// select.cu -- Algorithm 1 steps 3, 5, 6 and the Eq. (2) centering
// (arXiv 2609.28053, Sec. 2 and App. C).
//
// One warp per expert scans its 256 bins: each lane owns 8 consecutive
// bins, a warp-wide inclusive prefix sum locates the lane whose range
// reaches the rank, and that lane walks its 8 bins.
//   pass 1: u_e = min{u : sum_{j<=u} H[e][j] >= r},  rho_e = r - sum_{j<u_e} H[e][j]
//   pass 2: v_e = min{v : sum_{j<=v} L[e][j] >= rho_e},
//           q_hat_e = kappa^{-1}((u_e << 8) | v_e)   (a zero returned as +0)
//   pass 3: pass 1 on a histogram of equal-width bins, whose edge bins hold
//           ordinary (clamped) margins rather than non-finite ones
//   pass 3: as pass 1 on a histogram of equal-width bins, where the edge bins
//           hold ordinary (clamped) values rather than non-finite margins
// The bias update reproduces the definition's fp64 sum in ascending expert
// order bit for bit (see bias_update_kernel), divides by E and subtracts.
#include "select_device.cuh"

namespace eqb {

namespace {

__global__ void __launch_bounds__(256) select_kernel(const int32_t* __restrict__ hist, int E, int pass,
                                                     int64_t r, uint8_t* __restrict__ u,
                                                     int32_t* __restrict__ rho,
                                                     uint16_t* __restrict__ q_hat, int32_t* err,
                                                     const int64_t* __restrict__ shard_off, int K) {
  griddep_wait();
  griddep_launch();
  const int lane = threadIdx.x & 31;
  const int e = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (e >= E) return;
  if (shard_off) {
    // shard blockIdx.y: its own histogram, outputs and rank ceil(n_p K / E)
    const int p = blockIdx.y;
    const int64_t n = shard_off[p + 1] - shard_off[p];
    hist += (int64_t)p * E * 256;
    u += (int64_t)p * E;
    rho += (int64_t)p * E;
    if (q_hat) q_hat += (int64_t)p * E;
    if (n <= 0) {
      if (lane == 0) {
        if (pass != 2) { u[e] = 0; rho[e] = 0; }
        else q_hat[e] = 0;
      }
      return;
    }
    r = (n * K + E - 1) / E;
  }
  const int32_t* h = hist + (int64_t)e * 256 + lane * 8;
  int64_t cnt[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) cnt[j] = h[j];
  const int64_t target = pass != 2 ? r : (int64_t)rho[e];
  const uint32_t u_e = pass == 2 ? u[e] : 0u;
  warp_select(cnt, e, pass, target, u_e, u, rho, q_hat, err, lane);
}

__global__ void bias_update_kernel(const uint16_t* __restrict__ q_hat, int E, float* __restrict__ b_next) {
  griddep_wait();
  block_bias_update<false>(q_hat, E, b_next, blockDim.x, [] { __syncthreads(); });
}

}  // namespace

int launch_select(const int32_t* hist, int E, int pass, int64_t r, uint8_t* u, int32_t* rho,
                  uint16_t* q_hat, int32_t* err, cudaStream_t s) {
  const int wpb = 8;
  const int64_t* none = nullptr;
  return launch_dependent(select_kernel, dim3((E + wpb - 1) / wpb), dim3(wpb * 32), 0, s, hist, E, pass, r, u, rho,
                          q_hat, err, none, 0) == cudaSuccess
             ? kOk
             : kErrCuda;
}

int launch_select_sharded(const int32_t* hist, int E, int pass, const int64_t* shard_off, int P, int K,
                          uint8_t* u, int32_t* rho, uint16_t* q_hat, int32_t* err, cudaStream_t s) {
  const int wpb = 8;
  dim3 grid((E + wpb - 1) / wpb, P);
  return launch_dependent(select_kernel, grid, dim3(wpb * 32), 0, s, hist, E, pass, (int64_t)0, u, rho, q_hat, err,
                          shard_off, K) == cudaSuccess
             ? kOk
             : kErrCuda;
}

int launch_bias_update(const uint16_t* q_hat, int E, float* b_next, cudaStream_t s) {
  return launch_dependent(bias_update_kernel, dim3(1), dim3(256), 0, s, q_hat, E, b_next) == cudaSuccess ? kOk
                                                                                                   : kErrCuda;
}

}  // namespace eqb
