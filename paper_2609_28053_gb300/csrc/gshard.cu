// gshard.cu -- the GShard auxiliary-loss gradient, the comparison injection
// beside LEI (arXiv 2609.28053, Sec. 2 and App. D, Eq. (gshard-grad)):
//   grad_s[t, j] += alpha / (n_l d_t) * (R_j - sum_e p_{t,e} R_e),
// with R_e = f_{l,e} / (K n_l) - 1/E for the token's microbatch l (n_l
// tokens), s = sigmoid(z), d_t = sum_e s_{t,e} and p = s / d_t.
//
// A stream like LEI (z read once, grad_s read and written once).  Each CTA
// takes a contiguous token range and, for every microbatch it meets, forms R
// (fp64, rounded to fp32) and alpha / n_l in shared memory.  LPT lanes share
// a token, 8 experts per lane and chunk (one 16-byte load of z, two of
// grad_s; CPL chunks per lane when E > 256); the score sum and the
// R-weighted sum are reduced over those lanes with shuffles, then each lane
// updates its gradients.
#include "eqb_device.cuh"

namespace eqb {

namespace {

constexpr int kGsThreads = 256;

template <int LPT, int CPL>
__global__ void __launch_bounds__(kGsThreads) gshard_kernel(GshardArgs a, int64_t tokens_per_cta) {
  constexpr int TPW = 32 / LPT;  // tokens per warp step
  __shared__ __align__(16) float Rs[kMaxE];
  __shared__ float cs;
  const int E = a.E, nch = E >> 3;
  const int64_t tb = (int64_t)blockIdx.x * tokens_per_cta;
  const int64_t te = min(tb + tokens_per_cta, a.T);
  if (tb >= te) return;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const int sub = lane & (LPT - 1), slot = lane / LPT;

  int64_t t = tb;
  while (t < te) {
    const int l = microbatch_of(a.off, a.M, t);
    const int64_t lo = __ldg(a.off + l), hi = __ldg(a.off + l + 1);
    const int64_t seg_end = (hi > t) ? min(te, hi) : te;
    __syncthreads();  // the previous segment is done with Rs and cs
    const int64_t n = hi - lo;
    for (int e = threadIdx.x; e < E; e += blockDim.x)
      Rs[e] = n > 0 ? __double2float_rn((double)__ldg(a.loads + (int64_t)l * E + e) / ((double)a.K * (double)n) -
                                        1.0 / (double)E)
                    : 0.f;
    if (threadIdx.x == 0) cs = n > 0 ? __double2float_rn((double)a.alpha / (double)n) : 0.f;
    __syncthreads();
    // this lane's chunks: sub, sub + LPT, ... (CPL of them, past nch unused)
    float r[CPL][8];
#pragma unroll
    for (int k = 0; k < CPL; ++k) {
      const int c = sub + k * LPT;
      if (c < nch) {
        const float4 r0 = reinterpret_cast<const float4*>(Rs)[2 * c];
        const float4 r1 = reinterpret_cast<const float4*>(Rs)[2 * c + 1];
        r[k][0] = r0.x; r[k][1] = r0.y; r[k][2] = r0.z; r[k][3] = r0.w;
        r[k][4] = r1.x; r[k][5] = r1.y; r[k][6] = r1.z; r[k][7] = r1.w;
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) r[k][i] = 0.f;
      }
    }
    const float c0 = cs;

    // Two tokens per lane per round, every load issued before any use, so
    // the z and grad loads of both overlap.
    const int64_t stride = (int64_t)nw * TPW;
    for (int64_t base = t + (int64_t)wid * TPW; base < seg_end; base += 2 * stride) {
      int64_t tok[2];
      bool ok[2];
      uint4 w[2][CPL];
      float4 g0[2][CPL], g1[2][CPL];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        tok[u] = base + u * stride + slot;
        ok[u] = tok[u] < seg_end;
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
          const int c = sub + k * LPT;
          if (ok[u] && c < nch) {
            w[u][k] = __ldcs(reinterpret_cast<const uint4*>(a.z + tok[u] * E) + c);
            const float4* gp = reinterpret_cast<const float4*>(a.g + tok[u] * E) + 2 * c;
            g0[u][k] = __ldcs(gp);
            g1[u][k] = __ldcs(gp + 1);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        float d = 0.f, num = 0.f;
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
          const int c = sub + k * LPT;
          if (ok[u] && c < nch) {
            const uint32_t zw[4] = {w[u][k].x, w[u][k].y, w[u][k].z, w[u][k].w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const float s0 = 1.0f / (1.0f + expf(-bf16_lo(zw[q])));
              const float s1 = 1.0f / (1.0f + expf(-bf16_hi(zw[q])));
              d = __fadd_rn(d, s0);
              num = __fadd_rn(num, __fmul_rn(s0, r[k][2 * q]));
              d = __fadd_rn(d, s1);
              num = __fadd_rn(num, __fmul_rn(s1, r[k][2 * q + 1]));
            }
          }
        }
#pragma unroll
        for (int m = 1; m < LPT; m <<= 1) {
          d = __fadd_rn(d, __shfl_xor_sync(kFull, d, m));
          num = __fadd_rn(num, __shfl_xor_sync(kFull, num, m));
        }
        if (!ok[u]) continue;
        const float mean = __fdiv_rn(num, d);
        const float coef = __fdiv_rn(c0, d);
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
          const int c = sub + k * LPT;
          if (c >= nch) continue;
          float4 x0 = g0[u][k], x1 = g1[u][k];
          x0.x = __fadd_rn(x0.x, __fmul_rn(coef, __fsub_rn(r[k][0], mean)));
          x0.y = __fadd_rn(x0.y, __fmul_rn(coef, __fsub_rn(r[k][1], mean)));
          x0.z = __fadd_rn(x0.z, __fmul_rn(coef, __fsub_rn(r[k][2], mean)));
          x0.w = __fadd_rn(x0.w, __fmul_rn(coef, __fsub_rn(r[k][3], mean)));
          x1.x = __fadd_rn(x1.x, __fmul_rn(coef, __fsub_rn(r[k][4], mean)));
          x1.y = __fadd_rn(x1.y, __fmul_rn(coef, __fsub_rn(r[k][5], mean)));
          x1.z = __fadd_rn(x1.z, __fmul_rn(coef, __fsub_rn(r[k][6], mean)));
          x1.w = __fadd_rn(x1.w, __fmul_rn(coef, __fsub_rn(r[k][7], mean)));
          float4* gp = reinterpret_cast<float4*>(a.g + tok[u] * E) + 2 * c;
          __stcs(gp, x0);
          __stcs(gp + 1, x1);
        }
      }
    }
    t = seg_end;
  }
}

template <int LPT, int CPL>
int launch_gs(const GshardArgs& a, cudaStream_t s) {
  DeviceInfo di;
  if (int rc = device_info(&di)) return rc;
  int64_t grid = (int64_t)di.sm_count * 8;
  const int64_t max_grid = (a.T + 255) / 256;  // at least 256 tokens per CTA
  if (grid > max_grid) grid = max_grid;
  if (grid < 1) grid = 1;
  const int64_t tpc = (a.T + grid - 1) / grid;
  gshard_kernel<LPT, CPL><<<(unsigned)grid, kGsThreads, 0, s>>>(a, tpc);
  return cudaGetLastError() == cudaSuccess ? kOk : kErrCuda;
}

}  // namespace

int launch_gshard(const GshardArgs& a, cudaStream_t s) {
  const int nch = a.E >> 3;
  if (nch <= 1) return launch_gs<1, 1>(a, s);
  if (nch <= 2) return launch_gs<2, 1>(a, s);
  if (nch <= 4) return launch_gs<4, 1>(a, s);
  if (nch <= 8) return launch_gs<8, 1>(a, s);
  if (nch <= 16) return launch_gs<16, 1>(a, s);
  if (nch <= 32) return launch_gs<32, 1>(a, s);
  if (nch <= 64) return launch_gs<32, 2>(a, s);
  if (nch <= 96) return launch_gs<32, 3>(a, s);
  if (nch <= 128) return launch_gs<32, 4>(a, s);
  return kErrUnsupported;
}

}  // namespace eqb
