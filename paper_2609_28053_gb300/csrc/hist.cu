// hist.cu -- Algorithm 1's two margin-histogram passes (arXiv 2609.28053,
// Sec. 3 and App. C, steps 1 and 4).
//
// Both passes recompute every routing margin m = bf16_rne(tau_t - fp32(z))
// from z and tau instead of reading a stored margin array (Sec. 3: "the
// second pass simply rescans local margins").  The order-preserving key is
// k = kappa(m) (negative patterns complemented, others get the sign bit);
// pass 1 counts the high byte k >> 8, pass 2 counts the low byte k & 0xff of
// the margins whose high byte equals the selected u_e.
//
// Layout: the grid is (expert tiles) x (token ranges).  A CTA owns ET
// experts (ET = 64 when E allows) and keeps their ET x 256 int32 bins in
// shared memory (64 KiB), so three CTAs fit per SM.  Within a warp, ET/8
// lanes cover one token's ET experts with one 16-byte load each, so each
// load instruction of the warp reads whole contiguous row segments.  The
// bins of expert e_l are stored XOR-swizzled by (e_l >> 3): the lanes of one
// token hit distinct banks even when their margins share a bin.  At the end
// every CTA adds its non-zero bins into the global [E,256] histogram, which
// is how token partitions are summed in device memory.
#include "eqb_device.cuh"

namespace eqb {

namespace {

constexpr int kHistThreads = 512;
constexpr int kUnroll = 4;

template <int PASS, int LPT>
__global__ void __launch_bounds__(kHistThreads) hist_kernel(HistArgs a, int64_t tokens_per_cta) {
  extern __shared__ __align__(16) uint32_t bins[];
  constexpr int ET = LPT * 8;     // experts per CTA
  constexpr int TPS = 32 / LPT;   // tokens per warp step
  const int E = a.E;
  const int e0 = blockIdx.x * ET;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;
  const int c = lane % LPT;        // chunk of 8 experts inside the tile
  const int tok = lane / LPT;      // token slot inside the warp step

  for (int i = threadIdx.x; i < ET * 256; i += blockDim.x) bins[i] = 0;
  uint32_t uu[8];
  if (PASS == 2) {
#pragma unroll
    for (int j = 0; j < 8; ++j) uu[j] = a.u[e0 + c * 8 + j];
  }
  __syncthreads();

  const int64_t tb = (int64_t)blockIdx.y * tokens_per_cta;
  const int64_t te = min(tb + tokens_per_cta, a.T);
  uint32_t* my = bins + (c * 8) * 256;  // row of expert c*8 + 0
  const uint32_t sw = static_cast<uint32_t>(c);

  for (int64_t base = tb + (int64_t)wid * TPS; base < te; base += (int64_t)nw * TPS * kUnroll) {
    uint4 w[kUnroll];
    float tt[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t t = base + (int64_t)u * nw * TPS + tok;
      if (t < te) {
        w[u] = __ldcs(reinterpret_cast<const uint4*>(a.z + t * E + e0 + c * 8));
        tt[u] = __ldg(a.tau + t);
      } else {
        w[u] = make_uint4(0, 0, 0, 0);
        tt[u] = 0.f;
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t t = base + (int64_t)u * nw * TPS + tok;
      if (t >= te) continue;
      const float tv = tt[u];
      uint32_t m[4];
      m[0] = pack_bf16x2_rn(tv - bf16_lo(w[u].x), tv - bf16_hi(w[u].x));
      m[1] = pack_bf16x2_rn(tv - bf16_lo(w[u].y), tv - bf16_hi(w[u].y));
      m[2] = pack_bf16x2_rn(tv - bf16_lo(w[u].z), tv - bf16_hi(w[u].z));
      m[3] = pack_bf16x2_rn(tv - bf16_lo(w[u].w), tv - bf16_hi(w[u].w));
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const uint32_t x16 = (j & 1) ? (m[j >> 1] >> 16) : (m[j >> 1] & 0xffffu);
        const uint32_t k = kappa16(x16);
        if (PASS == 1) {
          atomicAdd(my + j * 256 + ((k >> 8) ^ sw), 1u);
        } else {
          if ((k >> 8) == uu[j]) atomicAdd(my + j * 256 + ((k & 0xffu) ^ sw), 1u);
        }
      }
    }
  }
  __syncthreads();

  for (int i = threadIdx.x; i < ET * 256; i += blockDim.x) {
    const uint32_t v = bins[i];
    if (v) {
      const int el = i >> 8;
      const int bin = (i & 255) ^ (el >> 3);
      atomicAdd(a.hist + (int64_t)(e0 + el) * 256 + bin, static_cast<int>(v));
      if (PASS == 1 && (bin == 0 || bin == 255)) raise_flag(a.err, kErrNonfinite);
    }
  }
}

template <int PASS, int LPT>
int launch_hist_t(const HistArgs& a, cudaStream_t s) {
  constexpr int ET = LPT * 8;
  DeviceInfo di;
  if (int rc = device_info(&di)) return rc;
  const int smem = ET * 256 * 4;
  const int nE = a.E / ET;
  int ctas_per_sm = (228 * 1024 - 1024) / (smem + 1024);
  if (ctas_per_sm > 4) ctas_per_sm = 4;
  if (ctas_per_sm < 1) ctas_per_sm = 1;
  int64_t nT = ((int64_t)di.sm_count * ctas_per_sm + nE - 1) / nE;
  // keep at least ~2048 tokens per CTA so the flush stays small
  const int64_t max_nT = (a.T + 2047) / 2048;
  if (nT > max_nT) nT = max_nT;
  if (nT < 1) nT = 1;
  const int64_t tpc = (a.T + nT - 1) / nT;
  auto kern = hist_kernel<PASS, LPT>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return kErrCuda;
  dim3 grid((unsigned)nE, (unsigned)nT);
  kern<<<grid, kHistThreads, smem, s>>>(a, tpc);
  return cudaGetLastError() == cudaSuccess ? kOk : kErrCuda;
}

template <int PASS>
int launch_hist_pass(const HistArgs& a, cudaStream_t s) {
  if (a.E % 64 == 0) return launch_hist_t<PASS, 8>(a, s);
  if (a.E % 32 == 0) return launch_hist_t<PASS, 4>(a, s);
  if (a.E % 16 == 0) return launch_hist_t<PASS, 2>(a, s);
  return launch_hist_t<PASS, 1>(a, s);
}

}  // namespace

int launch_hist(const HistArgs& a, int pass, cudaStream_t s) {
  return pass == 1 ? launch_hist_pass<1>(a, s) : launch_hist_pass<2>(a, s);
}

}  // namespace eqb
