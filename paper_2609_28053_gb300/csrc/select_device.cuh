// select_device.cuh -- the per-expert selection of Algorithm 1 (steps 3 and
// 5-6) and the Eq. (2) centering (arXiv 2609.28053, Sec. 2 and App. C), as
// device functions shared by the selection kernels (select.cu) and by the
// histogram passes, whose last block to finish counting runs them in the
// one-call step (hist.cu).
#pragma once

#include "eqb_device.cuh"

namespace eqb {

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
// Threads [0, nthreads) of the block compute b_next from q_hat (they share
// the final subtraction; warp 0 forms the mean); sync() is their barrier.
// SHARED_Q: q_hat is the block's shared-memory copy; otherwise the global
// array, read through L2 (it may have been written earlier in the same
// kernel).
template <bool SHARED_Q, class Sync>
__device__ __forceinline__ void block_bias_update(const uint16_t* q_hat, int E, float* __restrict__ b_next,
                                                  int nthreads, Sync sync) {
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
  sync();
  for (int e = threadIdx.x; e < E; e += nthreads)
    b_next[e] = __double2float_rn(__dsub_rn((double)bf16_bits_to_f32(q_at(e)), mean));
}

}  // namespace eqb
