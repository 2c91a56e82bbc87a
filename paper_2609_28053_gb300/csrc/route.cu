// route.cu -- top-K routing, cutoff tau_t and per-microbatch loads
// (Sec. 2, Eq. 1 and the QB paragraph of arXiv 2609.28053).
//
// One thread owns one token.  A warp stages a tile of 32 consecutive token
// rows of z (32 * E bf16, one contiguous block of global memory) in shared
// memory with coalesced 16-byte cp.async copies, double-buffered so the next
// tile streams in while the current one is processed.  Rows are padded to a
// stride of 4 (mod 8) words, so the 32 lanes reading the same 16-byte column
// chunk of their own rows hit 32 distinct banks, and the bias chunk they all
// need is a broadcast.
//
// Per token (s_e = fp32(z_e) + b_e, fp32 round-to-nearest-even):
//   A. group maxima: element j of chunk c goes to group (c mod G/8)*8 + j;
//      theta = the (K+1)st largest of the G group maxima.  K+1 distinct
//      groups each hold an element >= theta, so theta <= tau_t.
//   B. candidates: every e with s_e >= theta (a superset of the top-(K+1)
//      set, ties included) is appended, in ascending e, to a per-lane list.
//   C. exact selection: stable insertion of the candidates into a sorted
//      (K+1)-list (a new candidate goes after equal scores, displaced
//      entries shift down), so equal scores keep the lower index first.  A lane whose list overflows (many ties
//      at theta) falls back to K+1 exact scans of its row.
// Loads are counted in per-warp shared counters for the warp's current
// microbatch and flushed to global memory when the microbatch changes; each
// warp owns a contiguous range of tiles, so flushes are rare.
#include "eqb_device.cuh"

namespace eqb {

namespace {

constexpr int kCap = 32;   // candidate slots per token (power of two)
constexpr int kNbuf = 2;   // tile buffers per warp

__host__ __device__ inline int row_stride_bytes(int E) {
  int w = E / 2;                 // 32-bit words per row
  return 4 * (w + ((4 - w) & 7));  // stride == 4 (mod 8) words
}

__host__ __device__ inline int align16(int x) { return (x + 15) & ~15; }

__host__ __device__ inline int warp_region_bytes(int E) {
  return align16(kNbuf * 32 * row_stride_bytes(E) + kCap * 32 + 4 * E);
}

template <int N>
__device__ __forceinline__ void sort_desc(float (&a)[N]) {
#pragma unroll
  for (int k = 2; k <= N; k <<= 1) {
#pragma unroll
    for (int j = k >> 1; j > 0; j >>= 1) {
#pragma unroll
      for (int i = 0; i < N; ++i) {
        const int l = i ^ j;
        if (l > i) {
          const float x = a[i], y = a[l];
          const float hi = fmaxf(x, y), lo = fminf(x, y);
          if ((i & k) == 0) { a[i] = hi; a[l] = lo; } else { a[i] = lo; a[l] = hi; }
        }
      }
    }
  }
}

// Insert (s, e) into the descending list (v, id).  Candidates arrive in
// ascending e, so a new element goes after equal scores (strict compare);
// once it has been placed, every later slot shifts down unconditionally.
template <int KP1>
__device__ __forceinline__ void insert_sorted(float (&v)[KP1], int (&id)[KP1], float s, int e) {
  bool moved = false;
#pragma unroll
  for (int j = 0; j < KP1; ++j) {
    const bool gt = moved || s > v[j];
    moved = gt;
    const float tv = v[j];
    const int ti = id[j];
    v[j] = gt ? s : tv;
    id[j] = gt ? e : ti;
    s = gt ? tv : s;
    e = gt ? ti : e;
  }
}

template <int KP1, int G>
__global__ void __launch_bounds__(512) route_kernel(RouteArgs a, int64_t tiles_per_warp) {
  extern __shared__ __align__(16) uint8_t smem[];
  const int E = a.E, K = a.K;
  const int nch = E >> 3;
  const int rs = row_stride_bytes(E);
  const int tile_bytes = 32 * rs;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;

  float* bs = reinterpret_cast<float*>(smem);
  const float4* bs4 = reinterpret_cast<const float4*>(smem);
  uint8_t* wreg = smem + align16(4 * E) + wid * warp_region_bytes(E);
  uint8_t* tiles = wreg;
  uint8_t* cand = wreg + kNbuf * tile_bytes;
  int* wl = reinterpret_cast<int*>(cand + kCap * 32);

  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    const float v = a.b[e];
    bs[e] = v;
    if (!isfinite(v)) raise_flag(a.err, kErrNonfinite);
  }
  for (int e = lane; e < E; e += 32) wl[e] = 0;
  __syncthreads();

  const int64_t ntiles = (a.T + 31) >> 5;
  const int64_t gw = (int64_t)blockIdx.x * nw + wid;
  const int64_t tb = gw * tiles_per_warp;
  const int64_t te = min(tb + tiles_per_warp, ntiles);
  if (tb >= te) return;

  // Issue the cp.async copies of one tile: row r, chunk `lane`.
  auto issue = [&](int64_t tile, int buf) {
    uint8_t* dst = tiles + buf * tile_bytes;
    const int64_t t0 = tile << 5;
    if (lane < nch) {
#pragma unroll 4
      for (int r = 0; r < 32; ++r) {
        const bool ok = t0 + r < a.T;
        const uint16_t* src = ok ? a.z + (t0 + r) * E + lane * 8 : a.z;
        cp_async16(dst + r * rs + lane * 16, src, ok ? 16 : 0);
      }
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

  issue(tb, 0);
  cp_async_commit();
  int buf = 0;
  for (int64_t tile = tb; tile < te; ++tile) {
    if (tile + 1 < te) issue(tile + 1, buf ^ 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncwarp();

    const uint8_t* rowp = tiles + buf * tile_bytes + lane * rs;
    const int64_t t = (tile << 5) + lane;
    const bool valid = t < a.T;

    // ---- A: group maxima and the lower bound theta <= tau_t
    constexpr int U = G / 8;
    float gm[G];
#pragma unroll
    for (int g = 0; g < G; ++g) gm[g] = -INFINITY;
    for (int c0 = 0; c0 < nch; c0 += U) {
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int c = c0 + u;
        if (c < nch) {
          const uint4 w = lds128(rowp + c * 16);
          const float4 b0 = bs4[2 * c], b1 = bs4[2 * c + 1];
          gm[u * 8 + 0] = fmax_nan(gm[u * 8 + 0], bf16_lo(w.x) + b0.x);
          gm[u * 8 + 1] = fmax_nan(gm[u * 8 + 1], bf16_hi(w.x) + b0.y);
          gm[u * 8 + 2] = fmax_nan(gm[u * 8 + 2], bf16_lo(w.y) + b0.z);
          gm[u * 8 + 3] = fmax_nan(gm[u * 8 + 3], bf16_hi(w.y) + b0.w);
          gm[u * 8 + 4] = fmax_nan(gm[u * 8 + 4], bf16_lo(w.z) + b1.x);
          gm[u * 8 + 5] = fmax_nan(gm[u * 8 + 5], bf16_hi(w.z) + b1.y);
          gm[u * 8 + 6] = fmax_nan(gm[u * 8 + 6], bf16_lo(w.w) + b1.z);
          gm[u * 8 + 7] = fmax_nan(gm[u * 8 + 7], bf16_hi(w.w) + b1.w);
        }
      }
    }
    bool has_nan = false;
#pragma unroll
    for (int g = 0; g < G; ++g) has_nan |= (gm[g] != gm[g]);
    if (has_nan && valid) raise_flag(a.err, kErrNonfinite);
    sort_desc<G>(gm);
    float theta = gm[0];
#pragma unroll
    for (int g = 1; g < G; ++g) theta = (g == K) ? gm[g] : theta;

    // ---- B: candidates s_e >= theta, ascending e
    int cnt = 0;
    for (int c = 0; c < nch; ++c) {
      const uint4 w = lds128(rowp + c * 16);
      const float4 b0 = bs4[2 * c], b1 = bs4[2 * c + 1];
      float s[8];
      s[0] = bf16_lo(w.x) + b0.x; s[1] = bf16_hi(w.x) + b0.y;
      s[2] = bf16_lo(w.y) + b0.z; s[3] = bf16_hi(w.y) + b0.w;
      s[4] = bf16_lo(w.z) + b1.x; s[5] = bf16_hi(w.z) + b1.y;
      s[6] = bf16_lo(w.w) + b1.z; s[7] = bf16_hi(w.w) + b1.w;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (s[j] >= theta) {
          cand[((cnt & (kCap - 1)) << 5) | lane] = static_cast<uint8_t>(c * 8 + j);
          ++cnt;
        }
      }
    }

    // ---- C: exact top-(K+1) among the candidates
    float v[KP1];
    int id[KP1];
#pragma unroll
    for (int j = 0; j < KP1; ++j) { v[j] = -INFINITY; id[j] = 0; }
    const int n = min(__reduce_max_sync(kFull, cnt), kCap);
    for (int i = 0; i < n; ++i) {
      if (i < cnt) {
        const int e = cand[(i << 5) | lane];
        const float s = bf16_bits_to_f32(*reinterpret_cast<const uint16_t*>(rowp + 2 * e)) + bs[e];
        insert_sorted<KP1>(v, id, s, e);
      }
    }
    const bool overflow = cnt > kCap;
    if (__any_sync(kFull, overflow)) {
      if (overflow) {
        // Exact fallback: K+1 scans, each taking the next element in the
        // order (score descending, index ascending).
        float pv = INFINITY;
        int pi = -1;
#pragma unroll 1
        for (int k = 0; k < KP1; ++k) {
          if (k <= K) {
            float bv = -INFINITY;
            int bi = 0;  // stays a valid index even if nothing qualifies (NaN rows)
            bool found = false;
            for (int e = 0; e < E; ++e) {
              const float s = bf16_bits_to_f32(*reinterpret_cast<const uint16_t*>(rowp + 2 * e)) + bs[e];
              const bool after = (s < pv) || (s == pv && e > pi);
              if (after && (!found || s > bv)) { bv = s; bi = e; found = true; }
            }
#pragma unroll
            for (int j = 0; j < KP1; ++j)
              if (j == k) { v[j] = bv; id[j] = bi; }
            pv = bv;
            pi = bi;
          }
        }
      }
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
      const int l = valid ? microbatch_of(a.off, a.M, t) : -1;
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
    buf ^= 1;
  }
  if (a.loads) flush_loads();
}

template <int KP1>
int launch_route_kp1(const RouteArgs& a, cudaStream_t s) {
  constexpr int G = KP1 <= 16 ? 16 : 32;
  DeviceInfo di;
  if (int rc = device_info(&di)) return rc;
  const int head = align16(4 * a.E);
  const int wbytes = warp_region_bytes(a.E);
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
  kern<<<(unsigned)grid, nw * 32, smem, s>>>(a, tpw);
  return cudaGetLastError() == cudaSuccess ? kOk : kErrCuda;
}

}  // namespace

int launch_route(const RouteArgs& a, cudaStream_t s) {
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
