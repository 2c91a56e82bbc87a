// route_wide.cu -- top-K routing, cutoff tau_t and per-microbatch loads
// (Sec. 2, Eq. 1 and the QB paragraph of arXiv 2609.28053) for the wide rows
// E = 128, 256, 384 and 512 with K + 1 <= 16, the row width fixed at compile
// time.
//
// One thread owns one token; a warp owns a tile of 32 consecutive tokens,
// which each lane brings into shared memory with one bulk copy of its row
// (completion on a per-warp mbarrier) while the next tile is prefetched into
// L2.  Rows are padded to a stride of 4 (mod 8) words so the 32 lanes reading
// the same 16-byte chunk of their own rows hit distinct banks.  The per-token
// work (bound from packed chunk maxima, candidate masks, exact insertion of
// the candidates) is route_row() in route_wide.cuh.
// Loads are counted in per-warp shared counters for the warp's current
// microbatch and flushed when it changes.
#include "route_wide.cuh"

namespace eqb {

namespace {

// Warps per block: as many as shared memory holds (12 at E = 256), at most 16.
template <int E>
constexpr int wide_max_warps() {
  return (232448 - WideLayout<E>::HEAD) / WideLayout<E>::WARP < 16
             ? (232448 - WideLayout<E>::HEAD) / WideLayout<E>::WARP
             : 16;
}

template <int E, int KP1>
__global__ void __launch_bounds__(32 * wide_max_warps<E>(), 1)
    route_wide_kernel(RouteArgs a, int64_t tiles_per_warp) {
  using L = WideLayout<E>;
  extern __shared__ __align__(16) uint8_t smem[];
  const int K = a.K;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;

  float* bs = reinterpret_cast<float*>(smem);
  uint32_t* bdn = reinterpret_cast<uint32_t*>(smem + 4 * E);  // RD(b) packed pairs
  uint32_t* bup = bdn + E / 2;                                 // RU(b) packed pairs
  uint8_t* wreg = smem + L::HEAD + wid * L::WARP;
  uint8_t* tile = wreg;
  uint32_t* mw = reinterpret_cast<uint32_t*>(wreg + L::TILE);  // [NCH/4][32 lanes]
  int* wl = reinterpret_cast<int*>(wreg + L::TILE + L::ENT);
  const uint32_t bar = saddr(wreg + L::TILE + L::ENT + L::WL);

  griddep_wait();
  load_bias_tables<E>(a.b, bs, bdn, bup, a.err);
  for (int e = lane; e < E; e += 32) wl[e] = 0;
  if (lane == 0) {
    bar_init(bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  __syncthreads();

  const int64_t ntiles = (a.T + 31) >> 5;
  const int64_t gw = (int64_t)blockIdx.x * nw + wid;
  const int64_t tb = gw * tiles_per_warp;
  const int64_t te = min(tb + tiles_per_warp, ntiles);
  if (tb >= te) return;
  const uint4* bdn4 = reinterpret_cast<const uint4*>(bdn);
  const uint4* bup4 = reinterpret_cast<const uint4*>(bup);
  const uint8_t* rowp = tile + lane * L::RS;

  // Lane r copies row r of the tile (rows past T are left as they are: their
  // results are never stored).
  auto load_tile = [&](int64_t tl) {
    const int64_t t0 = tl << 5;
    const int rows = static_cast<int>(min((int64_t)32, a.T - t0));
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
      const uint32_t bytes = static_cast<uint32_t>(min((int64_t)32, a.T - t0) * E * 2);
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

  uint32_t phase = 0;
  load_tile(tb);
  prefetch(tb + 1);
  for (int64_t tl = tb; tl < te; ++tl) {
    if (!__all_sync(kFull, bar_wait_bounded(bar, phase, kRouteWaitLimit))) {
      // The copy did not complete in time: report it, give the copies in
      // flight one more bounded wait, and stop.
      raise_flag(a.err, kErrCuda);
      bar_wait_bounded(bar, phase, kRouteWaitLimit);
      return;
    }
    phase ^= 1u;

    const int64_t t = (tl << 5) + lane;
    const bool valid = t < a.T;

    float v[KP1];
    int id[KP1];
    route_row<E, KP1>(rowp, bs, bdn4, bup4, mw, lane, valid, a.err, v, id);
    __syncwarp();  // every lane is done with the tile

    if (tl + 1 < te) {
      load_tile(tl + 1);
      prefetch(tl + 2);
    }

    // ---- outputs
    if (valid) {
      const float tau_t = list_tau<KP1>(v, K);
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
      const int64_t t_last = min(t0 + 31, a.T - 1) + a.tbase;
      if (!(t0 + a.tbase >= mb_lo && t_last < mb_hi)) {
        // the tile leaves the current microbatch: per-lane lookup
        const int l = valid ? microbatch_of(a.off, a.M, t + a.tbase) : -1;
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
  if (a.loads) flush_loads();
}

template <int E, int KP1>
int launch_wide_t(const RouteArgs& a, cudaStream_t s) {
  using L = WideLayout<E>;
  DeviceInfo di;
  if (int rc = device_info(&di)) return rc;
  int nw = (di.max_smem_optin - L::HEAD) / L::WARP;
  if (nw > wide_max_warps<E>()) nw = wide_max_warps<E>();
  if (nw < 1) return kErrUnsupported;
  const int smem = L::HEAD + nw * L::WARP;
  int ctas_per_sm = (228 * 1024 - 1024) / (smem + 1024);
  if (ctas_per_sm < 1) ctas_per_sm = 1;
  if (ctas_per_sm > 4) ctas_per_sm = 4;
  const int64_t ntiles = (a.T + 31) / 32;
  int64_t grid = (int64_t)di.sm_count * ctas_per_sm;
  const int64_t max_grid = (ntiles + nw - 1) / nw;
  if (grid > max_grid) grid = max_grid;
  const int64_t total_warps = grid * nw;
  const int64_t tpw = (ntiles + total_warps - 1) / total_warps;
  auto kern = route_wide_kernel<E, KP1>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return kErrCuda;
  return launch_dependent(kern, dim3((unsigned)grid), dim3(nw * 32), smem, s, a, tpw) == cudaSuccess ? kOk
                                                                                         : kErrCuda;
}

template <int E>
int launch_wide_e(const RouteArgs& a, cudaStream_t s) {
  const int kp1 = a.K + 1;
  if (kp1 <= 2) return launch_wide_t<E, 2>(a, s);
  if (kp1 <= 3) return launch_wide_t<E, 3>(a, s);
  if (kp1 <= 4) return launch_wide_t<E, 4>(a, s);
  if (kp1 <= 7) return launch_wide_t<E, 7>(a, s);
  if (kp1 <= 8) return launch_wide_t<E, 8>(a, s);
  if (kp1 <= 9) return launch_wide_t<E, 9>(a, s);
  if (kp1 <= 16) return launch_wide_t<E, 16>(a, s);
  return kErrUnsupported;
}

}  // namespace

bool route_wide_supported(int E, int K) {
  return (E == 128 || E == 256 || E == 384 || E == 512) && K + 1 <= 16;
}

int launch_route_wide(const RouteArgs& a, cudaStream_t s) {
  if (a.E == 256) return launch_wide_e<256>(a, s);
  if (a.E == 128) return launch_wide_e<128>(a, s);
  if (a.E == 512) return launch_wide_e<512>(a, s);
  if (a.E == 384) return launch_wide_e<384>(a, s);
  return kErrUnsupported;
}

}  // namespace eqb
