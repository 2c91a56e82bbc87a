// lei.cu -- Load-Error Injection (arXiv 2609.28053, Sec. 4, Eq. (LEI) and
// Eq. (norm)).
//
// For microbatch l with n_l tokens and loads f_{l,e}:
//   rho_e = f_{l,e} / (K n_l / E) - 1,
//   sigma = tanh(xi) / xi with xi = max_e |rho_e| / c   (c > 0; 1 at xi = 0),
//   sigma = 1                                            (c <= 0, unnormalised),
//   grad_s[t, e] += eta * sigma * rho_e   for every t of the microbatch, every e.
//
// The path is a pure HBM stream (read and write grad_s once), so each CTA
// takes a contiguous token range, computes the E coefficients of each
// microbatch it meets (fp64, the threads striding over the experts, a block
// max for xi) into shared memory as fp32, and then streams its range with
// 16-byte loads and stores using evict-first cache hints.
//
// For the one-call step the coefficients are also formed once per microbatch
// into an [M,E] table (lei_coef_kernel), from which the histogram passes
// stream the injection beside their own work (hist.cu).
#include "eqb_device.cuh"

namespace eqb {

namespace {

constexpr int kLeiThreads = 256;
constexpr int kLeiUnroll = 4;

// Eq. (norm) coefficients eta * sigma * rho_e of one microbatch with n tokens
// and loads f (one row of [M,E]), computed by a whole block of kLeiThreads
// threads into out[0..E) (shared or global memory) and visible to the block
// on return.  fp64 throughput is low on this part, so each thread does only
// a multiply-add and a multiply per expert; the reciprocal of the target
// load and tanh are formed once.
__device__ void block_lei_coef(const int32_t* __restrict__ f, int64_t n, int E, int K, float eta, float c,
                               float* out) {
  __shared__ double red[kLeiThreads / 32];
  __shared__ double scal[2];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  __syncthreads();  // a previous call has finished reading scal and out
  if (threadIdx.x == 0) scal[0] = n > 0 ? (double)E / ((double)K * (double)n) : 0.0;  // 1 / fbar
  __syncthreads();
  const double inv_fbar = scal[0];
  // each thread holds the rho of experts threadIdx.x + k * kLeiThreads
  constexpr int kPer = kMaxE / kLeiThreads;
  double rho[kPer];
  double amax = 0.0;
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int e = threadIdx.x + k * kLeiThreads;
    rho[k] = (e < E && inv_fbar > 0.0) ? (double)__ldg(f + e) * inv_fbar - 1.0 : 0.0;
    amax = fmax(amax, fabs(rho[k]));
  }
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) amax = fmax(amax, __shfl_xor_sync(kFull, amax, d));
  if (lane == 0) red[wid] = amax;
  __syncthreads();
  if (threadIdx.x == 0) {
    double rmax = red[0];
    for (int w = 1; w < kLeiThreads / 32; ++w) rmax = fmax(rmax, red[w]);
    // sigma = tanh(xi) / xi in fp32: its relative error (a few ulp of fp32)
    // stays far inside the LEI tolerance, and it spares the serial fp64
    // division and tanh of this thread
    float sigma = 1.0f;
    if (c > 0.0f) {
      const float xi = __fdiv_rn(static_cast<float>(rmax), c);
      sigma = (xi == 0.0f) ? 1.0f : __fdiv_rn(tanhf(xi), xi);
    }
    scal[1] = (double)eta * (double)sigma;
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int e = threadIdx.x + k * kLeiThreads;
    if (e < E) out[e] = __double2float_rn(scal[1] * rho[k]);
  }
  __syncthreads();
}

__global__ void __launch_bounds__(kLeiThreads) lei_kernel(LeiArgs a, int64_t tokens_per_cta) {
  __shared__ __align__(16) float coef[kMaxE];
  griddep_wait();
  const int E = a.E, E4 = a.E >> 2;
  const int64_t tb = (int64_t)blockIdx.x * tokens_per_cta;
  const int64_t te = min(tb + tokens_per_cta, a.T);
  if (tb >= te) return;
  float4* g4 = reinterpret_cast<float4*>(a.g);
  const float4* c4 = reinterpret_cast<const float4*>(coef);

  int64_t t = tb;
  while (t < te) {
    const int l = microbatch_of(a.off, a.M, t + a.tbase);
    const int64_t lo = __ldg(a.off + l) - a.tbase, hi = __ldg(a.off + l + 1) - a.tbase;
    // Malformed offsets (off[M] < T) must not stall the loop: tokens past
    // the last boundary are treated as the last microbatch's.
    const int64_t seg_end = (hi > t) ? min(te, hi) : te;
    block_lei_coef(a.loads + (int64_t)l * E, hi - lo, E, a.K, a.eta, a.c, coef);

    // ---- stream grad_s[t .. seg_end) in float4 units
    const int64_t i0 = t * E4, i1 = seg_end * E4;
    const int S = blockDim.x;
    const int dcol = S % E4;
    int col = threadIdx.x % E4;
    int64_t i = i0 + threadIdx.x;
    for (; i + (int64_t)(kLeiUnroll - 1) * S < i1; i += (int64_t)kLeiUnroll * S) {
      float4 v[kLeiUnroll];
      int cc[kLeiUnroll];
#pragma unroll
      for (int u = 0; u < kLeiUnroll; ++u) {
        v[u] = __ldcs(g4 + i + (int64_t)u * S);
        cc[u] = col;
        col += dcol;
        if (col >= E4) col -= E4;
      }
#pragma unroll
      for (int u = 0; u < kLeiUnroll; ++u) {
        const float4 cf = c4[cc[u]];
        v[u].x = __fadd_rn(v[u].x, cf.x);
        v[u].y = __fadd_rn(v[u].y, cf.y);
        v[u].z = __fadd_rn(v[u].z, cf.z);
        v[u].w = __fadd_rn(v[u].w, cf.w);
        __stcs(g4 + i + (int64_t)u * S, v[u]);
      }
    }
    for (; i < i1; i += S) {
      float4 v = __ldcs(g4 + i);
      const float4 cf = c4[col];
      v.x = __fadd_rn(v.x, cf.x);
      v.y = __fadd_rn(v.y, cf.y);
      v.z = __fadd_rn(v.z, cf.z);
      v.w = __fadd_rn(v.w, cf.w);
      __stcs(g4 + i, v);
      col += dcol;
      if (col >= E4) col -= E4;
    }
    t = seg_end;
  }
}

// One block per microbatch: row l of the [M,E] coefficient table.
__global__ void __launch_bounds__(kLeiThreads) lei_coef_kernel(LeiArgs a, float* coef) {
  griddep_wait();
  griddep_launch();
  const int l = blockIdx.x;
  const int64_t n = __ldg(a.off + l + 1) - __ldg(a.off + l);
  block_lei_coef(a.loads + (int64_t)l * a.E, n, a.E, a.K, a.eta, a.c, coef + (int64_t)l * a.E);
}

}  // namespace

int launch_lei_coef(const LeiArgs& a, float* coef, cudaStream_t s) {
  if (a.M < 1) return kErrInvalidArg;
  return launch_dependent(lei_coef_kernel, dim3((unsigned)a.M), dim3(kLeiThreads), 0, s, a, coef) ==
                 cudaSuccess
             ? kOk
             : kErrCuda;
}

int launch_lei(const LeiArgs& a, cudaStream_t s) {
  DeviceInfo di;
  if (int rc = device_info(&di)) return rc;
  int64_t grid = (int64_t)di.sm_count * 8;
  // at least 256 tokens per CTA so the per-microbatch prologue stays small
  const int64_t max_grid = (a.T + 255) / 256;
  if (grid > max_grid) grid = max_grid;
  if (grid < 1) grid = 1;
  const int64_t tpc = (a.T + grid - 1) / grid;
  return launch_dependent(lei_kernel, dim3((unsigned)grid), dim3(kLeiThreads), 0, s, a, tpc) == cudaSuccess
             ? kOk
             : kErrCuda;
}

}  // namespace eqb
