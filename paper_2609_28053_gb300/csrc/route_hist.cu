// route_hist.cu -- routing and Algorithm 1's coarse pass in one pass over z
// (arXiv 2609.28053: Sec. 2 Eq. 1 and the QB paragraph; Algorithm 1 step 1,
// Sec. 3), for E = 128 and 256 with K + 1 <= 16.
//
// Each warp routes a 32-token tile staged in shared memory (route_row() of
// route_wide.cuh, thread per token: top-K set, cutoff tau_t, loads), then
// recounts the same staged tile for the coarse histogram H[e][h], h the high
// byte of kappa(m) for every margin m = bf16_rne(tau_t - fp32(z)), lane c
// taking the 8 experts of chunk c of each token.  z is read from DRAM once
// for both, where the separate kernels read it twice.
//
// Coarse bins: the window of 16-bit shared-memory counters of
// coarse_window.cuh (the 256 bins of all E experts would not leave room for
// the routing tiles).  Counters are added into H at least every 65,535
// tokens per block and at the end.
//
// On GB300 this kernel is slower than routing and the coarse pass as two
// kernels: both are bound by instruction issue (ALU pipe), not by DRAM, so
// saving the second read of z saves nothing while the counting competes with
// routing for the same ALU pipe at a third of the coarse pass's occupancy.
// The one-call step therefore uses the two kernels; this one is the
// one-read variant (eqb_route_hist_fused).
#include "coarse_window.cuh"
#include "route_wide.cuh"

namespace eqb {

namespace {

template <int E>
struct FusedLayout {
  using W = WideLayout<E>;
  static constexpr int RS = W::RS;
  static constexpr int TILE = W::TILE;
  static constexpr int ENT = W::ENT;
  static constexpr int WL = W::WL;
  static constexpr int WARP = W::WARP;          // tile, masks, load counters, mbarrier
  static constexpr int BINW = coarse_window_words(E);
  static constexpr int OFF_RD = 4 * E;
  static constexpr int OFF_RU = OFF_RD + 2 * E;
  static constexpr int OFF_BINS = OFF_RU + 2 * E;
  static constexpr int HEAD = (OFF_BINS + 4 * BINW + 15) & ~15;
};

// Warps per block: as many as shared memory holds, at most 16.
template <int E>
constexpr int fused_warps() {
  return (232448 - FusedLayout<E>::HEAD) / FusedLayout<E>::WARP < 16
             ? (232448 - FusedLayout<E>::HEAD) / FusedLayout<E>::WARP
             : 16;
}

template <int E, int KP1, int NW>
__global__ void __launch_bounds__(32 * NW, 1)
    route_hist_kernel(RouteArgs a, int32_t* __restrict__ hist, int64_t tiles_per_warp) {
  using L = FusedLayout<E>;
  constexpr int LPT = E / 8;     // lanes per token while counting
  constexpr int TPS = 32 / LPT;  // tokens per warp step while counting
  // counters gain at most one per token: add them into H at least this often
  constexpr int kFlushTiles = 65535 / (32 * NW);
  extern __shared__ __align__(16) uint8_t smem[];
  const int K = a.K;
  const int64_t T = a.T;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;

  float* bs = reinterpret_cast<float*>(smem);
  uint32_t* bdn = reinterpret_cast<uint32_t*>(smem + L::OFF_RD);
  uint32_t* bup = reinterpret_cast<uint32_t*>(smem + L::OFF_RU);
  uint32_t* bins = reinterpret_cast<uint32_t*>(smem + L::OFF_BINS);
  uint8_t* wreg = smem + L::HEAD + wid * L::WARP;
  uint8_t* tile = wreg;
  uint32_t* mw = reinterpret_cast<uint32_t*>(wreg + L::TILE);
  int* wl = reinterpret_cast<int*>(wreg + L::TILE + L::ENT);
  const uint32_t bar = saddr(wreg + L::TILE + L::ENT + L::WL);

  for (int i = threadIdx.x; i < L::BINW; i += blockDim.x) bins[i] = 0u;
  for (int e = lane; e < E; e += 32) wl[e] = 0;
  if (lane == 0) {
    bar_init(bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  griddep_wait();
  load_bias_tables<E>(a.b, bs, bdn, bup, a.err);
  __syncthreads();

  const uint4* bdn4 = reinterpret_cast<const uint4*>(bdn);
  const uint4* bup4 = reinterpret_cast<const uint4*>(bup);
  const uint8_t* rowp = tile + lane * L::RS;

  // ---- this lane's counters while counting: chunk cc of token slot ctok
  const int cc = lane % LPT, ctok = lane / LPT;
  uint32_t cbase[4], zbase;
  coarse_window_bases(saddr(bins), cc, cbase, zbase);

  // ---- the warp's contiguous tile range
  const int64_t ntiles = (T + 31) >> 5;
  const int64_t gw = (int64_t)blockIdx.x * NW + wid;
  const int64_t tb = min(gw * tiles_per_warp, ntiles);
  const int64_t te = min(tb + tiles_per_warp, ntiles);

  auto load_tile = [&](int64_t tl) {
    const int64_t t0 = tl << 5;
    const int rows = static_cast<int>(min((int64_t)32, T - t0));
    if (lane == 0) bar_expect_tx(bar, static_cast<uint32_t>(rows * E * 2));
    __syncwarp();
    if (lane < rows) {
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      bulk_copy(saddr(tile + lane * L::RS), a.z + (t0 + lane) * E, E * 2, bar);
    }
  };
  auto prefetch = [&](int64_t tl) {
    if (lane == 0 && tl < te) {
      const int64_t t0 = tl << 5;
      const uint32_t bytes = static_cast<uint32_t>(min((int64_t)32, T - t0) * E * 2);
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(a.z + t0 * E), "r"(bytes) : "memory");
    }
  };

  int cur_mb = -1;
  int64_t mb_lo = 0, mb_hi = 0;  // token range of cur_mb
  auto flush_loads = [&]() {
    __syncwarp();
    if (cur_mb >= 0) {
      for (int e = lane; e < E; e += 32) {
        const int v = wl[e];
        if (v) atomicAdd(a.loads + (int64_t)cur_mb * E + e, v);
        wl[e] = 0;
      }
    }
    __syncwarp();
  };

  bool alive = true;  // false once a copy ran out of time
  uint32_t phase = 0;
  if (tb < te) {
    load_tile(tb);
    prefetch(tb + 1);
  }
  // Every warp makes the same number of steps (tiles_per_warp), so the
  // block-wide flushes every kFlushTiles steps line up.
  for (int64_t k = 0; k < tiles_per_warp; ++k) {
    const int64_t tl = tb + k;
    if (tl < te && alive) {
      if (!__all_sync(kFull, bar_wait_bounded(bar, phase, kRouteWaitLimit))) {
        // The copy did not complete in time: report it, give the copy one
        // more bounded wait, and stop routing (the barriers below still run).
        raise_flag(a.err, kErrCuda);
        bar_wait_bounded(bar, phase, kRouteWaitLimit);
        alive = false;
      }
    }
    if (tl < te && alive) {
      phase ^= 1u;
      const int64_t t = (tl << 5) + lane;
      const bool valid = t < T;

      float v[KP1];
      int id[KP1];
      route_row<E, KP1>(rowp, bs, bdn4, bup4, mw, lane, valid, a.err, v, id);
      const float tau_t = list_tau<KP1>(v, K);

      // ---- coarse histogram of the tile's margins from the staged copy
#pragma unroll 2
      for (int j0 = 0; j0 < 32; j0 += TPS) {
        const int j = j0 + ctok;
        const float tv = __shfl_sync(kFull, tau_t, j);
        if ((tl << 5) + j < T)
          coarse_window_count<false>(lds128(tile + j * L::RS + 16 * cc), tv, cbase, zbase, cc, hist, a.err);
      }
      __syncwarp();  // every lane is done with the tile
      if (tl + 1 < te) {
        load_tile(tl + 1);
        prefetch(tl + 2);
      }

      // ---- outputs
      if (valid) {
        a.tau[t] = tau_t;
        if (!isfinite(tau_t)) raise_flag(a.err, kErrNonfinite);
        if (a.idx) {
          int32_t* out = a.idx + t * K;
#pragma unroll
          for (int j = 0; j < KP1; ++j)
            if (j < K) out[j] = id[j];
        }
      }
      if (a.loads) {
        const int64_t t0 = tl << 5;
        const int64_t t_last = min(t0 + 31, T - 1);
        if (!(t0 >= mb_lo && t_last < mb_hi)) {
          // the tile leaves the current microbatch: per-lane lookup
          const int l = valid ? microbatch_of(a.off, a.M, t) : -1;
          const int l0 = __shfl_sync(kFull, l, 0);
          if (l0 != cur_mb) {
            flush_loads();
            cur_mb = l0;
            mb_lo = __ldg(a.off + l0);
            mb_hi = __ldg(a.off + l0 + 1);
          }
          if (valid) {
#pragma unroll
            for (int j = 0; j < KP1; ++j) {
              if (j < K) {
                if (l == cur_mb) atomicAdd(wl + id[j], 1);
                else atomicAdd(a.loads + (int64_t)l * E + id[j], 1);
              }
            }
          }
        } else if (valid) {
#pragma unroll
          for (int j = 0; j < KP1; ++j)
            if (j < K) atomicAdd(wl + id[j], 1);
        }
      }
    }
    if ((k + 1) % kFlushTiles == 0 && k + 1 < tiles_per_warp) {
      __syncthreads();
      coarse_window_flush(bins, L::BINW, hist, threadIdx.x, blockDim.x);
      __syncthreads();
    }
  }
  if (a.loads) flush_loads();
  __syncthreads();
  coarse_window_flush(bins, L::BINW, hist, threadIdx.x, blockDim.x);
}

template <int E, int KP1>
int launch_fused_t(const RouteArgs& a, int32_t* hist, cudaStream_t s) {
  using L = FusedLayout<E>;
  constexpr int NW = fused_warps<E>();
  DeviceInfo di;
  if (int rc = device_info(&di)) return rc;
  const int smem = L::HEAD + NW * L::WARP;
  if (smem > di.max_smem_optin) return kErrUnsupported;
  const int64_t ntiles = (a.T + 31) / 32;
  int64_t grid = di.sm_count;
  const int64_t max_grid = (ntiles + NW - 1) / NW;
  if (grid > max_grid) grid = max_grid;
  const int64_t tpw = (ntiles + grid * NW - 1) / (grid * NW);
  auto kern = route_hist_kernel<E, KP1, NW>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return kErrCuda;
  return launch_dependent(kern, dim3((unsigned)grid), dim3(NW * 32), smem, s, a, hist, tpw) == cudaSuccess
             ? kOk
             : kErrCuda;
}

template <int E>
int launch_fused_e(const RouteArgs& a, int32_t* hist, cudaStream_t s) {
  const int kp1 = a.K + 1;
  if (kp1 <= 2) return launch_fused_t<E, 2>(a, hist, s);
  if (kp1 <= 3) return launch_fused_t<E, 3>(a, hist, s);
  if (kp1 <= 4) return launch_fused_t<E, 4>(a, hist, s);
  if (kp1 <= 7) return launch_fused_t<E, 7>(a, hist, s);
  if (kp1 <= 8) return launch_fused_t<E, 8>(a, hist, s);
  if (kp1 <= 9) return launch_fused_t<E, 9>(a, hist, s);
  if (kp1 <= 16) return launch_fused_t<E, 16>(a, hist, s);
  return kErrUnsupported;
}

}  // namespace

bool route_hist_supported(int E, int K) { return (E == 128 || E == 256) && K + 1 <= 16; }

int launch_route_hist(const RouteArgs& a, int32_t* hist, cudaStream_t s) {
  if (a.tbase != 0 || !hist || a.T < 1) return kErrInvalidArg;
  if (a.E == 256) return launch_fused_e<256>(a, hist, s);
  if (a.E == 128) return launch_fused_e<128>(a, hist, s);
  return kErrUnsupported;
}

}  // namespace eqb
