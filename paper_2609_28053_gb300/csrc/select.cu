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
#include "eqb_device.cuh"

namespace eqb {

namespace {

constexpr int kSelectBiasMaxE = 1024;  // experts of one select_bias_kernel block

// One warp selects for expert e from its 256 counts, lane j holding bins
// 8j..8j+7 (cnt): pass 1 writes u[e] and rho[e] for the rank `target`, pass 2
// writes q_hat[e] (and *qs, when given) from u_e = u[e] and the rank target =
// rho[e], both read by the caller beside the counts.  Flags a count in
// high-byte bin 0x00 or 0xff (pass 1) and an unreachable rank.
__device__ __forceinline__ void warp_select(const int64_t (&cnt)[8], int e, int pass, int64_t target,
                                            uint32_t u_e, uint8_t* __restrict__ u, int32_t* __restrict__ rho,
                                            uint16_t* __restrict__ q_hat, int32_t* err, int lane,
                                            uint16_t* qs = nullptr) {
  int64_t local = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) local += cnt[j];
  int64_t incl = local;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int64_t o = __shfl_up_sync(kFull, incl, d);
    if (lane >= d) incl += o;
  }
  const int64_t excl = incl - local;
  const bool first = pass != 2;
  const unsigned hit = __ballot_sync(kFull, excl < target && target <= incl);
  if (pass == 1 && ((lane == 0 && cnt[0] != 0) || (lane == 31 && cnt[7] != 0)))
    raise_flag(err, kErrNonfinite);
  if (hit == 0u || target < 1) {
    if (lane == 0) {
      raise_flag(err, kErrRank);
      if (first) { u[e] = 255; rho[e] = 0; }
      else {
        q_hat[e] = 0x7fc0;  // NaN marks an unreachable rank
        if (qs) *qs = 0x7fc0;
      }
    }
    return;
  }
  if (lane == __ffs(hit) - 1) {
    int64_t below = excl;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (below + cnt[j] >= target) {
        const int bin = lane * 8 + j;
        if (first) {
          u[e] = static_cast<uint8_t>(bin);
          rho[e] = static_cast<int32_t>(target - below);
        } else {
          uint32_t q = kappa16_inv((u_e << 8) | static_cast<uint32_t>(bin));
          if (q == 0x8000u) q = 0u;
          q_hat[e] = static_cast<uint16_t>(q);
          if (qs) *qs = static_cast<uint16_t>(q);
        }
        break;
      }
      below += cnt[j];
    }
  }
}

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

// Exponent range of a non-zero bf16 pattern: [ulp exponent, leading-bit exponent].
__device__ __forceinline__ void bf16_exp_range(uint32_t x, int& lo, int& hi) {
  const int ex = (x >> 7) & 0xff;
  const uint32_t man = x & 0x7f;
  if (ex != 0) { lo = ex - 127 - 7; hi = ex - 127; }
  else { lo = -133; hi = -134 + (32 - __clz(man)); }  // subnormal
}

// b_next = q_hat - mean(q_hat), mean = (sum in ascending e, fp64) / E.
// If every non-zero q_hat lies within a window where all partial sums of up
// to E terms are exact in fp64 (leading-bit exponent - ulp exponent + 1 +
// ceil(log2 E) <= 52), any summation order gives the exact sum, so a warp
// tree reduction reproduces the sequential sum bit for bit.  Otherwise one
// thread sums in ascending order.
// The block computes b_next from q_hat (the threads of the block share the
// final subtraction; warp 0 forms the mean).  SHARED_Q: q_hat is the block's
// shared-memory copy; otherwise the global array, read through L2 (it may
// have been written earlier in the same kernel).
template <bool SHARED_Q>
__device__ __forceinline__ void block_bias_update(const uint16_t* q_hat, int E, float* __restrict__ b_next) {
  __shared__ double mean;
  auto q_at = [&](int e) -> uint32_t { return SHARED_Q ? q_hat[e] : __ldcg(q_hat + e); };

  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    double part = 0.0;
    int lo = 1 << 20, hi = -(1 << 20);
    for (int e = lane; e < E; e += 32) {
      const uint32_t x = q_at(e);
      if ((x & 0x7fffu) != 0u) {
        int l, h;
        bf16_exp_range(x, l, h);
        lo = min(lo, l);
        hi = max(hi, h);
      }
      part = __dadd_rn(part, (double)bf16_bits_to_f32(x));
    }
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
      lo = min(lo, __shfl_xor_sync(kFull, lo, d));
      hi = max(hi, __shfl_xor_sync(kFull, hi, d));
    }
    double sum;
    const int lg = 32 - __clz(E - 1);  // ceil(log2 E)
    if (hi - lo + 1 + lg <= 52 || hi < lo) {
#pragma unroll
      for (int d = 16; d > 0; d >>= 1) part = __dadd_rn(part, __shfl_xor_sync(kFull, part, d));
      sum = part;
    } else {
      sum = 0.0;
      if (lane == 0)
        for (int e = 0; e < E; ++e) sum = __dadd_rn(sum, (double)bf16_bits_to_f32(q_at(e)));
    }
    if (lane == 0) mean = __ddiv_rn(sum, (double)E);
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x)
    b_next[e] = __double2float_rn(__dsub_rn((double)bf16_bits_to_f32(q_at(e)), mean));
}


__global__ void bias_update_kernel(const uint16_t* __restrict__ q_hat, int E, float* __restrict__ b_next) {
  griddep_wait();
  block_bias_update<false>(q_hat, E, b_next);
}

// Algorithm 1 steps 5-6 and Eq. (2) in one block: the pass-2 selection of
// every expert (each warp loads the counts, rho and u of 4 experts before it
// scans them, so a batch costs one L2 round trip), then the bias update from
// the block's shared copy of q_hat.  Same results as select_kernel (pass 2)
// followed by bias_update_kernel.  E <= kSelectBiasMaxE.
__global__ void __launch_bounds__(1024) select_bias_kernel(const int32_t* __restrict__ hist, int E,
                                                           const uint8_t* __restrict__ u,
                                                           int32_t* __restrict__ rho,
                                                           uint16_t* __restrict__ q_hat, int32_t* err,
                                                           float* __restrict__ b_next) {
  constexpr int B = 4;
  __shared__ uint16_t qs[kSelectBiasMaxE];
  griddep_wait();
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
  for (int e0 = wid; e0 < E; e0 += nw * B) {
    int4 ca[B], cb[B];
    int32_t rk[B];
    uint32_t uk = 0u;  // u of the batch, one byte per expert
#pragma unroll
    for (int k = 0; k < B; ++k) {
      const int e = min(e0 + k * nw, E - 1);
      const int32_t* h = hist + (int64_t)e * 256 + lane * 8;
      ca[k] = __ldg(reinterpret_cast<const int4*>(h));
      cb[k] = __ldg(reinterpret_cast<const int4*>(h + 4));
      rk[k] = __ldcg(rho + e);
      uk |= static_cast<uint32_t>(__ldcg(u + e)) << (8 * k);
    }
#pragma unroll
    for (int k = 0; k < B; ++k) {
      const int e = e0 + k * nw;
      const int64_t cnt[8] = {ca[k].x, ca[k].y, ca[k].z, ca[k].w, cb[k].x, cb[k].y, cb[k].z, cb[k].w};
      if (e < E)
        warp_select(cnt, e, 2, (int64_t)rk[k], (uk >> (8 * k)) & 0xffu, const_cast<uint8_t*>(u), rho, q_hat, err,
                    lane, qs + e);
    }
  }
  __syncthreads();  // every q_hat is written
  block_bias_update<true>(qs, E, b_next);
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

int launch_select_bias(const int32_t* hist, int E, const uint8_t* u, int32_t* rho, uint16_t* q_hat, int32_t* err,
                       float* b_next, cudaStream_t s) {
  if (E > kSelectBiasMaxE) return kErrUnsupported;
  return launch_dependent(select_bias_kernel, dim3(1), dim3(1024), 0, s, hist, E, u, rho, q_hat, err, b_next) ==
                 cudaSuccess
             ? kOk
             : kErrCuda;
}

int launch_bias_update(const uint16_t* q_hat, int E, float* b_next, cudaStream_t s) {
  return launch_dependent(bias_update_kernel, dim3(1), dim3(256), 0, s, q_hat, E, b_next) == cudaSuccess ? kOk
                                                                                                   : kErrCuda;
}

}  // namespace eqb
