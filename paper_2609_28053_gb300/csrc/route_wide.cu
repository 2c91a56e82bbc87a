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
// work is the three phases of route.cu with every loop over the row unrolled:
//   A. packed bf16x2 maxima of L_e = bf16(z_e + RD(b_e)) per 8-expert chunk,
//      the chunks c and c + NCH/2 sharing one word.  Sorting the words
//      (bf16x2 max/min network) sorts both half-rows' chunk maxima at once,
//      and the KP1-th largest of all chunk maxima is
//      min_{i<KP1} max(A[i], B[KP1-1-i]) for the two sorted lists A, B.
//      KP1 >= K+1 chunks each hold an element with L at or above it, so,
//      moved down two bf16 steps, it is <= tau_t; two more steps give the
//      filter threshold.
//   B. per-chunk masks of U_e = bf16(z_e + RU(b_e)) >= threshold, every one
//      of the experts with s_e >= tau_t among them, kept in shared memory,
//      with the set of non-zero mask words (32 experts each).
//   C. the listed experts, in ascending index, are inserted into a sorted
//      (K+1)-list by their exact fp32 score s_e = fp32(z_e) + b_e; a new
//      element goes after equal scores, so ties keep the lower index first.
// Loads are counted in per-warp shared counters for the warp's current
// microbatch and flushed when it changes.
#include "eqb_device.cuh"

namespace eqb {

namespace {

constexpr uint32_t kWaitLimit = 1u << 20;  // polls of at most ~1 us: about a second

// Bounded wait for the phase of parity `parity`.
__device__ __forceinline__ bool bar_wait(uint32_t bar, uint32_t parity) {
  return bar_wait_bounded(bar, parity, kWaitLimit);
}

// One contiguous global -> shared copy by the bulk-copy engine.
__device__ __forceinline__ void bulk_copy(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}
__device__ __forceinline__ uint32_t lds_u16(const void* p) {
  return *reinterpret_cast<const uint16_t*>(p);
}

// (max of the even experts, max of the odd experts) of one chunk of L.
__device__ __forceinline__ uint32_t chunk_max(const uint4& w, const uint4& bd) {
  return hmax2_nan_bf16(hmax2_nan_bf16(hadd2_bf16(w.x, bd.x), hadd2_bf16(w.y, bd.y)),
                        hmax2_nan_bf16(hadd2_bf16(w.z, bd.z), hadd2_bf16(w.w, bd.w)));
}

__host__ __device__ constexpr int wide_row_stride(int E) { return 4 * (E / 2 + ((4 - E / 2) & 7)); }

template <int E>
struct WideLayout {
  static constexpr int NCH = E / 8;              // 16-byte chunks per row
  static constexpr int RS = wide_row_stride(E);  // staged row stride, bytes
  static constexpr int TILE = 32 * RS;
  static constexpr int ENT = 32 * (NCH / 4) * 4;  // chunk masks, four per word, per lane
  static constexpr int WL = 4 * E;               // load counters
  static constexpr int WARP = (TILE + ENT + WL + 8 + 15) & ~15;  // + the mbarrier
  static constexpr int HEAD = 4 * E + 2 * (2 * E);               // b, RD(b), RU(b)
};

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
  constexpr int NCH = L::NCH, NH = NCH / 2;
  constexpr int NP = NH <= 8 ? 8 : NH <= 16 ? 16 : 32;  // sorted length (a power of two)
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
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    const float v = a.b[e];
    bs[e] = v;
    if (!isfinite(v)) raise_flag(a.err, kErrNonfinite);
  }
  for (int q = threadIdx.x; q < E / 2; q += blockDim.x) {
    const float b0 = a.b[2 * q], b1 = a.b[2 * q + 1];
    bdn[q] = bf16_round_down(b0) | (bf16_round_down(b1) << 16);
    bup[q] = bf16_round_up(b0) | (bf16_round_up(b1) << 16);
  }
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
    if (!__all_sync(kFull, bar_wait(bar, phase))) {
      // The copy did not complete in time: report it, give the copies in
      // flight one more bounded wait, and stop.
      raise_flag(a.err, kErrCuda);
      bar_wait(bar, phase);
      return;
    }
    phase ^= 1u;

    const int64_t t = (tl << 5) + lane;
    const bool valid = t < a.T;

    // ---- A: chunk maxima of L, chunks c and c + NH in one word (words past
    // NH, when NH is not a power of two, hold -inf in both halves)
    uint32_t cm[NP];
#pragma unroll
    for (int c = NH; c < NP; ++c) cm[c] = 0xff80ff80u;
#pragma unroll
    for (int c = 0; c < NH; ++c) {
      // At E > 256 the unrolled loads would not fit in registers if all were
      // hoisted: let at most eight pairs of chunks be in flight.
      if (NH > 16 && c > 0 && (c & 7) == 0) asm volatile("" ::: "memory");
      const uint32_t qa = chunk_max(lds128(rowp + 16 * c), bdn4[c]);
      const uint32_t qb = chunk_max(lds128(rowp + 16 * (c + NH)), bdn4[c + NH]);
      cm[c] = hmax2_nan_bf16(prmt(qa, qb, 0x5410u), prmt(qa, qb, 0x7632u));
    }
    uint32_t anynan = cm[0];
#pragma unroll
    for (int c = 1; c < NH; ++c) anynan = hmax2_nan_bf16(anynan, cm[c]);
    if (valid && ((anynan & 0x7fffu) > 0x7f80u || (anynan >> 16 & 0x7fffu) > 0x7f80u))
      raise_flag(a.err, kErrNonfinite);
    sort_desc_bf16x2<NP>(cm);
    float theta = INFINITY;
#pragma unroll
    for (int i = 0; i < KP1; ++i) {
      const int j = KP1 - 1 - i;
      const float x = i < NP ? bf16_lo(cm[i < NP ? i : 0]) : -INFINITY;
      const float y = j < NP ? bf16_hi(cm[j < NP ? j : 0]) : -INFINITY;
      theta = fminf(theta, fmaxf(x, y));
    }
    // Near zero, flushing of subnormal bf16 sums could move L by up to
    // 2^-126; lowering theta below that range keeps the bound safe.
    if (fabsf(theta) < 0x1p-124f) theta = -0x1p-124f;
    const uint32_t thf = bf16_steps_down(__float_as_uint(theta) >> 16, 4u);
    const uint32_t thf2 = thf | (thf << 16);

    // ---- B: per-chunk masks of U >= threshold, stored four to a word (bit
    // 8u + j of word k is expert 32k + 8u + j), and the set of non-zero words
    uint32_t hits = 0u;
#pragma unroll
    for (int k = 0; k < NCH / 4; ++k) {
      uint32_t word = 0u;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int c = 4 * k + u;
        const uint4 w = lds128(rowp + 16 * c);
        const uint4 bu = bup4[c];
        const uint32_t r0 = hge2_bf16(hadd2_bf16(w.x, bu.x), thf2);
        const uint32_t r1 = hge2_bf16(hadd2_bf16(w.y, bu.y), thf2);
        const uint32_t r2 = hge2_bf16(hadd2_bf16(w.z, bu.z), thf2);
        const uint32_t r3 = hge2_bf16(hadd2_bf16(w.w, bu.w), thf2);
        // element 2q -> bit 2q (low half of r_q), element 2q+1 -> bit 16+2q
        const uint32_t y = (r0 & 0x00010001u) | (r1 & 0x00040004u) | (r2 & 0x00100010u) | (r3 & 0x00400040u);
        word |= ((y | (y >> 15)) & 0xffu) << (8 * u);
      }
      mw[(k << 5) | lane] = word;
      hits |= (word != 0u ? 1u : 0u) << k;
    }

    // ---- C: exact top-(K+1) of the experts with a hit, in ascending index,
    // one per lane per step, taken from the mask words 32 experts at a time;
    // the next candidate's z and b are read one step ahead.  Refills are
    // branch-free, and a lane that is done inserts -inf, which leaves its
    // list unchanged.
    float v[KP1];
    int id[KP1];
#pragma unroll
    for (int j = 0; j < KP1; ++j) { v[j] = -INFINITY; id[j] = 0; }
    int wb = 0;  // first expert of the current mask word
    uint32_t m = 0u;
    auto fetch = [&]() -> int {
      const bool need = m == 0u && hits != 0u;
      const int k = __ffs(hits) - 1;
      const uint32_t word = mw[((need ? k : 0) << 5) | lane];
      m = need ? word : m;
      wb = need ? k << 5 : wb;
      hits = need ? hits & (hits - 1u) : hits;
      const int e = m != 0u ? wb + __ffs(m) - 1 : -1;
      m &= m - 1u;
      return e;
    };
    int e0 = fetch();
    uint32_t z0 = lds_u16(rowp + 2 * max(e0, 0));
    float b0 = bs[max(e0, 0)];
    while (__any_sync(kFull, e0 >= 0)) {
      const int e1 = fetch();
      const uint32_t z1 = lds_u16(rowp + 2 * max(e1, 0));
      const float b1 = bs[max(e1, 0)];
      insert_sorted<KP1>(v, id, e0 >= 0 ? bf16_bits_to_f32(z0) + b0 : -INFINITY, e0);
      e0 = e1;
      z0 = z1;
      b0 = b1;
    }
    __syncwarp();  // every lane is done with the tile

    if (tl + 1 < te) {
      load_tile(tl + 1);
      prefetch(tl + 2);
    }

    // ---- outputs
    if (valid) {
      float tau_t = v[0];
#pragma unroll
      for (int j = 1; j < KP1; ++j) tau_t = (j == K) ? v[j] : tau_t;
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
