// route_wide.cuh -- the per-token part of wide-row routing (Sec. 2, Eq. 1
// and the QB paragraph of arXiv 2609.28053), shared by the routing kernel
// (route_wide.cu) and the routing + coarse-histogram kernel (route_hist.cu).
//
// One thread owns one token whose row of z sits in shared memory (rows of a
// 32-token tile padded to a stride of 4 (mod 8) words, so the 32 lanes
// reading the same 16-byte chunk of their own rows hit distinct banks).  The
// row width E is a compile-time constant, so every loop over the row unrolls:
//   A. packed bf16x2 maxima of L_e = bf16(z_e + RD(b_e)) per 8-expert chunk,
//      the chunks c and c + NCH/2 sharing one word.  Sorting the words
//      (bf16x2 max/min network) sorts both half-rows' chunk maxima at once,
//      and the KP1-th largest of all chunk maxima is
//      min_{i<KP1} max(A[i], B[KP1-1-i]) for the two sorted lists A, B.
//      KP1 >= K+1 chunks each hold an element with L at or above it, so one
//      bf16 step below it is <= tau_t and bounds every expert that can be
//      selected; two steps below it is the filter threshold.
//   B. per-chunk masks of U_e = bf16(z_e + RU(b_e)) >= threshold, every one
//      of the experts with s_e >= tau_t among them, kept in shared memory,
//      with the set of non-zero mask words (32 experts each).
//   C. the listed experts, in ascending index, are inserted into a sorted
//      (K+1)-list by their exact fp32 score s_e = fp32(z_e) + b_e; a new
//      element goes after equal scores, so ties keep the lower index first.
#pragma once

#include "eqb_device.cuh"

namespace eqb {

// Polls of at most ~1 us each before a bulk-copy wait gives up: about a second.
constexpr uint32_t kRouteWaitLimit = 1u << 20;

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

// The block's copy of the bias: b as fp32, and RD(b), RU(b) as packed bf16
// pairs (the bounds of phases A and B).  A non-finite b raises the flag.
template <int E>
__device__ __forceinline__ void load_bias_tables(const float* __restrict__ b, float* bs, uint32_t* bdn, uint32_t* bup,
                                                 int32_t* err) {
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    const float v = b[e];
    bs[e] = v;
    if (!isfinite(v)) raise_flag(err, kErrNonfinite);
  }
  for (int q = threadIdx.x; q < E / 2; q += blockDim.x) {
    const float b0 = b[2 * q], b1 = b[2 * q + 1];
    bdn[q] = bf16_round_down(b0) | (bf16_round_down(b1) << 16);
    bup[q] = bf16_round_up(b0) | (bf16_round_up(b1) << 16);
  }
}

// Phases A-C for the token whose row starts at rowp: on return v[0..KP1)
// holds the top-(K+1) scores in descending order (ties: lower index first)
// and id[] their experts, so tau_t = v[K].  mw is the warp's mask-word area
// ([NCH/4][32 lanes] words).  Every lane of the warp must call it (phase C
// is a warp-wide loop); `valid` only gates the non-finite check.
template <int E, int KP1>
__device__ __forceinline__ void route_row(const uint8_t* rowp, const float* bs, const uint4* bdn4, const uint4* bup4,
                                          uint32_t* mw, int lane, bool valid, int32_t* err, float (&v)[KP1],
                                          int (&id)[KP1]) {
  constexpr int NCH = E / 8, NH = NCH / 2;
  constexpr int NP = NH <= 8 ? 8 : NH <= 16 ? 16 : 32;  // sorted length (a power of two)

  // ---- A: chunk maxima of L, chunks c and c + NH in one word (words past
  // NH, when NH is not a power of two, hold -inf in both halves)
  uint32_t cm[NP];
#pragma unroll
  for (int c = NH; c < NP; ++c) cm[c] = 0xff80ff80u;
#pragma unroll
  for (int c = 0; c < NH; ++c) {
    // From E = 256 on the unrolled loads do not fit in registers if all are
    // hoisted (at E = 256 the 168 registers of a 12-warp block spilled):
    // let at most eight pairs of chunks be in flight.
    if (NH > 8 && c > 0 && (c & 7) == 0) asm volatile("" ::: "memory");
    const uint32_t qa = chunk_max(lds128(rowp + 16 * c), bdn4[c]);
    const uint32_t qb = chunk_max(lds128(rowp + 16 * (c + NH)), bdn4[c + NH]);
    cm[c] = hmax2_nan_bf16(prmt(qa, qb, 0x5410u), prmt(qa, qb, 0x7632u));
  }
  uint32_t anynan = cm[0];
#pragma unroll
  for (int c = 1; c < NH; ++c) anynan = hmax2_nan_bf16(anynan, cm[c]);
  if (valid && ((anynan & 0x7fffu) > 0x7f80u || (anynan >> 16 & 0x7fffu) > 0x7f80u)) raise_flag(err, kErrNonfinite);
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
}

// tau_t = v[K] of the sorted list (K < KP1 chosen at run time).
template <int KP1>
__device__ __forceinline__ float list_tau(const float (&v)[KP1], int K) {
  float tau_t = v[0];
#pragma unroll
  for (int j = 1; j < KP1; ++j) tau_t = (j == K) ? v[j] : tau_t;
  return tau_t;
}

}  // namespace eqb
