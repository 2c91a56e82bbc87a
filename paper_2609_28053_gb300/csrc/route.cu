// route.cu -- top-K routing, cutoff tau_t and per-microbatch loads
// (Sec. 2, Eq. 1 and the QB paragraph of arXiv 2609.28053).
//
// One thread owns one token.  A warp stages a tile of 32 consecutive token
// rows of z (one contiguous block of 32 * E bf16) in shared memory with
// coalesced 16-byte cp.async copies; for wide rows the next tile is
// prefetched into L2, for narrow rows it is double-buffered.  Rows are padded
// to a stride of 4 (mod 8) words, so the 32 lanes reading the same 16-byte
// column chunk of their own rows hit 32 distinct banks and the per-expert
// constants they need are broadcasts.
//
// Exact scores are s_e = fp32(z_e) + b_e (fp32, round to nearest even).  The
// exact work is confined to a small candidate set found with packed bf16x2
// arithmetic (two experts per instruction):
//   A. lower bound: L_e = bf16(z_e + RD(b_e)) never exceeds the bf16
//      rounding of s_e, so the (K+1)st largest of G group maxima of L, moved
//      down one bf16 step, is <= tau_t (K+1 groups each hold an element at
//      or above it).  Two steps down is the filter threshold.
//   B. filter: U_e = bf16(z_e + RU(b_e)) >= threshold keeps every e with
//      s_e >= tau_t (and a few more).  Per 8-expert chunk the passing experts
//      form an 8-bit mask; chunks with a non-zero mask are listed per lane.
//   C. exact selection: the listed experts, in ascending index, are inserted
//      into a sorted (K+1)-list by their exact fp32 score; a new element goes
//      after equal scores, so ties keep the lower expert index first.  Any
//      number of candidates (ties) is handled exactly.
// Loads are counted in per-warp shared counters for the warp's current
// microbatch and flushed to global memory when it changes; each warp owns a
// contiguous range of tiles, so flushes are rare.
#include "eqb_device.cuh"

namespace eqb {

namespace {


__host__ __device__ inline int row_stride_bytes(int E) {
  int w = E / 2;                     // 32-bit words per row
  return 4 * (w + ((4 - w) & 7));    // stride == 4 (mod 8) words
}

__host__ __device__ inline int align16(int x) { return (x + 15) & ~15; }

__host__ __device__ inline int head_bytes(int E) { return align16(4 * E) + 2 * align16(2 * E); }

__host__ __device__ inline int warp_region_bytes(int E, int nbuf) {
  return align16(nbuf * 32 * row_stride_bytes(E) + (E / 8) * 32 * 2 + 4 * E);  // tile, chunk lists, loads
}

template <int KP1, int G>
__global__ void __launch_bounds__(512) route_kernel(RouteArgs a, int64_t tiles_per_warp, int nbuf) {
  extern __shared__ __align__(16) uint8_t smem[];
  const int E = a.E, K = a.K;
  const int nch = E >> 3;
  const int rs = row_stride_bytes(E);
  const int tile_bytes = 32 * rs;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;

  float* bs = reinterpret_cast<float*>(smem);
  uint32_t* bdn = reinterpret_cast<uint32_t*>(smem + align16(4 * E));   // RD(b) packed pairs
  uint32_t* bup = bdn + align16(2 * E) / 4;                              // RU(b) packed pairs
  uint8_t* wreg = smem + head_bytes(E) + wid * warp_region_bytes(E, nbuf);
  uint8_t* tiles = wreg;
  uint16_t* ent = reinterpret_cast<uint16_t*>(wreg + nbuf * tile_bytes);
  int* wl = reinterpret_cast<int*>(wreg + nbuf * tile_bytes + nch * 32 * 2);

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
  __syncthreads();

  const int64_t ntiles = (a.T + 31) >> 5;
  const int64_t gw = (int64_t)blockIdx.x * nw + wid;
  const int64_t tb = gw * tiles_per_warp;
  const int64_t te = min(tb + tiles_per_warp, ntiles);
  if (tb >= te) return;
  const uint4* bdn4 = reinterpret_cast<const uint4*>(bdn);
  const uint4* bup4 = reinterpret_cast<const uint4*>(bup);

  // cp.async copies of one tile: row r, chunks lane, lane + 32, ...
  auto issue = [&](int64_t tile, int buf) {
    uint8_t* dst = tiles + buf * tile_bytes;
    const int64_t t0 = tile << 5;
    for (int c = lane; c < nch; c += 32) {
#pragma unroll 4
      for (int r = 0; r < 32; ++r) {
        const bool ok = t0 + r < a.T;
        const uint16_t* src = ok ? a.z + (t0 + r) * E + c * 8 : a.z;
        cp_async16(dst + r * rs + c * 16, src, ok ? 16 : 0);
      }
    }
  };
  // Bring the given tile into L2 ahead of its cp.async copies.
  auto prefetch = [&](int64_t tile) {
    if (lane == 0 && tile < te) {
      const int64_t t0 = tile << 5;
      const int64_t rows = min((int64_t)32, a.T - t0);
      const uint32_t bytes = static_cast<uint32_t>(rows * E * 2);
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(a.z + t0 * E), "r"(bytes)
                   : "memory");
    }
  };

  int cur_mb = -1;
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

  int buf = 0;
  if (nbuf == 2) {
    issue(tb, 0);
    cp_async_commit();
  }
  for (int64_t tile = tb; tile < te; ++tile) {
    if (nbuf == 2) {
      if (tile + 1 < te) issue(tile + 1, buf ^ 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      issue(tile, 0);
      cp_async_commit();
      prefetch(tile + 1);
      cp_async_wait<0>();
    }
    __syncwarp();

    const uint8_t* rowp = tiles + buf * tile_bytes + lane * rs;
    const int64_t t = (tile << 5) + lane;
    const bool valid = t < a.T;

    // ---- A: packed bf16 group maxima of the lower bounds L
    constexpr int U = G / 8;
    uint32_t gm2[G / 2];
#pragma unroll
    for (int g = 0; g < G / 2; ++g) gm2[g] = 0xff80ff80u;  // -inf, -inf
    for (int c0 = 0; c0 < nch; c0 += U) {
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int c = c0 + u;
        if (c < nch) {
          const uint4 w = lds128(rowp + c * 16);
          const uint4 bd = bdn4[c];
          gm2[u * 4 + 0] = hmax2_nan_bf16(gm2[u * 4 + 0], hadd2_bf16(w.x, bd.x));
          gm2[u * 4 + 1] = hmax2_nan_bf16(gm2[u * 4 + 1], hadd2_bf16(w.y, bd.y));
          gm2[u * 4 + 2] = hmax2_nan_bf16(gm2[u * 4 + 2], hadd2_bf16(w.z, bd.z));
          gm2[u * 4 + 3] = hmax2_nan_bf16(gm2[u * 4 + 3], hadd2_bf16(w.w, bd.w));
        }
      }
    }
    float gm[G];
    bool has_nan = false;
#pragma unroll
    for (int g = 0; g < G / 2; ++g) {
      gm[2 * g] = bf16_lo(gm2[g]);
      gm[2 * g + 1] = bf16_hi(gm2[g]);
      has_nan |= (gm[2 * g] != gm[2 * g]) || (gm[2 * g + 1] != gm[2 * g + 1]);
    }
    if (has_nan && valid) raise_flag(a.err, kErrNonfinite);
    sort_desc<G>(gm);
    float theta = gm[0];
#pragma unroll
    for (int g = 1; g < G; ++g) theta = (g == K) ? gm[g] : theta;
    // Near zero, flushing of subnormal bf16 sums could move L by up to
    // 2^-126; lowering theta below that range keeps the bound safe.
    if (fabsf(theta) < 0x1p-124f) theta = -0x1p-124f;
    // Filter threshold: one bf16 step below theta is enough.  KP1 experts have
    // L_e >= theta, and L_e = RN_bf16(z + RD(b)) <= RN_bf16(s_e) (RN is monotone,
    // RD(b) <= b, s_e the exact sum), so their exact sums are >= theta - half a
    // bf16 step and their fp32 scores >= pred(theta): tau >= pred(theta).  An
    // expert with fp32 score >= tau has an exact sum within half an fp32 step
    // of it or above, so U_e = RN_bf16(z + RU(b)) >= RN_bf16(s_e) >= pred(theta).
    // Two steps keep one step of margin (near zero theta was moved below the
    // range where subnormal flushing could matter).
    const uint32_t thf = bf16_steps_down(__float_as_uint(theta) >> 16, 2u);
    const uint32_t thf2 = thf | (thf << 16);

    // ---- B: per-chunk masks of U >= threshold, chunks with a hit listed
    int cnt = 0;
#pragma unroll 2
    for (int c = 0; c < nch; ++c) {
      const uint4 w = lds128(rowp + c * 16);
      const uint4 bu = bup4[c];
      const uint32_t r0 = hge2_bf16(hadd2_bf16(w.x, bu.x), thf2);
      const uint32_t r1 = hge2_bf16(hadd2_bf16(w.y, bu.y), thf2);
      const uint32_t r2 = hge2_bf16(hadd2_bf16(w.z, bu.z), thf2);
      const uint32_t r3 = hge2_bf16(hadd2_bf16(w.w, bu.w), thf2);
      // element 2q -> bit 2q (low half of r_q), element 2q+1 -> bit 16+2q
      uint32_t y = r0 & 0x00010001u;
      y |= r1 & 0x00040004u;
      y |= r2 & 0x00100010u;
      y |= r3 & 0x00400040u;
      const uint32_t mask = (y | (y >> 15)) & 0xffu;
      if (mask) {
        ent[(cnt << 5) | lane] = static_cast<uint16_t>((c << 8) | mask);
        ++cnt;
      }
    }

    // ---- C: exact top-(K+1) of the listed candidates
    float v[KP1];
    int id[KP1];
#pragma unroll
    for (int j = 0; j < KP1; ++j) { v[j] = -INFINITY; id[j] = 0; }
    // One candidate per lane per iteration: a lane whose current chunk mask
    // is used up loads its next entry, so the warp runs for the largest
    // candidate count of its lanes.  The next candidate's z and b are read
    // one iteration ahead, off the insertion's critical path.
    int ei = 0, cbase = 0;
    uint32_t m = 0u;
    auto next = [&](int& e_out) -> bool {
      if (m == 0u && ei < cnt) {
        const uint32_t en = ent[(ei << 5) | lane];
        cbase = static_cast<int>(en >> 8) * 8;
        m = en & 0xffu;
        ++ei;
      }
      if (m == 0u) return false;
      e_out = cbase + __ffs(m) - 1;
      m &= m - 1u;
      return true;
    };
    int e_cur = 0;
    bool have = next(e_cur);
    uint32_t zc = have ? *reinterpret_cast<const uint16_t*>(rowp + 2 * e_cur) : 0u;
    float bc = have ? bs[e_cur] : 0.f;
    while (__any_sync(kFull, have)) {
      int e_nxt = 0;
      const bool have_nxt = next(e_nxt);
      uint32_t zn = 0u;
      float bn = 0.f;
      if (have_nxt) {
        zn = *reinterpret_cast<const uint16_t*>(rowp + 2 * e_nxt);
        bn = bs[e_nxt];
      }
      if (have) insert_sorted<KP1>(v, id, bf16_bits_to_f32(zc) + bc, e_cur);
      have = have_nxt;
      e_cur = e_nxt;
      zc = zn;
      bc = bn;
    }
    __syncwarp();

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
      const int l = valid ? microbatch_of(a.off, a.M, t + a.tbase) : -1;
      const int l0 = __shfl_sync(kFull, l, 0);
      if (l0 != cur_mb) {
        flush_loads();
        cur_mb = l0;
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
    }
    __syncwarp();
    if (nbuf == 2) buf ^= 1;
  }
  if (a.loads) flush_loads();
}

template <int KP1>
int launch_route_kp1(const RouteArgs& a, cudaStream_t s) {
  constexpr int G = KP1 <= 16 ? 16 : 32;
  DeviceInfo di;
  if (int rc = device_info(&di)) return rc;
  const int head = head_bytes(a.E);
  // Wide rows: one tile buffer per warp (more resident warps) with an L2
  // prefetch of the next tile; narrow rows: double buffering.
  const int nbuf = a.E >= 128 ? 1 : 2;
  const int wbytes = warp_region_bytes(a.E, nbuf);
  int nw = (di.max_smem_optin - head) / wbytes;
  if (nw > 16) nw = 16;
  if (nw < 1) return kErrUnsupported;
  const int smem = head + nw * wbytes;
  int ctas_per_sm = (228 * 1024 - 1024) / (smem + 1024);
  if (ctas_per_sm < 1) ctas_per_sm = 1;
  if (ctas_per_sm > 4) ctas_per_sm = 4;
  const int64_t ntiles = (a.T + 31) / 32;
  int64_t grid = (int64_t)di.sm_count * ctas_per_sm;
  const int64_t max_grid = (ntiles + nw - 1) / nw;
  if (grid > max_grid) grid = max_grid;
  const int64_t total_warps = grid * nw;
  const int64_t tpw = (ntiles + total_warps - 1) / total_warps;
  auto kern = route_kernel<KP1, G>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return kErrCuda;
  return launch_dependent(kern, dim3((unsigned)grid), dim3(nw * 32), smem, s, a, tpw, nbuf) == cudaSuccess
             ? kOk
             : kErrCuda;
}

}  // namespace

int launch_route(const RouteArgs& a, cudaStream_t s) {
  if (route_wide_supported(a.E, a.K)) return launch_route_wide(a, s);
  const int kp1 = a.K + 1;
  if (kp1 <= 2) return launch_route_kp1<2>(a, s);
  if (kp1 <= 3) return launch_route_kp1<3>(a, s);
  if (kp1 <= 4) return launch_route_kp1<4>(a, s);
  if (kp1 <= 7) return launch_route_kp1<7>(a, s);
  if (kp1 <= 8) return launch_route_kp1<8>(a, s);
  if (kp1 <= 9) return launch_route_kp1<9>(a, s);
  if (kp1 <= 16) return launch_route_kp1<16>(a, s);
  if (kp1 <= 32) return launch_route_kp1<32>(a, s);
  return kErrUnsupported;
}

}  // namespace eqb
