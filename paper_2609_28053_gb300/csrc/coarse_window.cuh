// coarse_window.cuh -- Algorithm 1's coarse histogram (arXiv 2609.28053,
// step 1, Sec. 3) counted in a window of shared-memory bins, for kernels
// whose shared memory is mostly taken by other work (the one-read routing
// kernel, the router projection's epilogue).
//
// The block keeps 16-bit counters (two experts per word) only for the bins
// that hold practically every margin: |m| in [2^-15, 2^17), both signs (32 of
// the 256 high bytes), and high byte 0 (+0, subnormal and the smallest
// normal positive margins: the cutoff expert's own margin whenever its bias
// is 0).  A margin outside is added straight to the global histogram.  In
// terms of the internal key hk = kappa(m) >> 8 ^ 0x80, sl = (hk - 56) mod 256
// lies in [0, 16) for m >= 0 and in [128, 144) for m < 0 inside the window,
// and the counter of pair row r and sl is word 289 (r >> 3) + 16 pos(r) + sl
// with pos(r) = ((r & 3) << 1) | ((r >> 2) & 1): the two 16-word segments of
// a row are 128 words apart, eight rows fill 256 words, the (r >> 3) skew
// puts equal bins of the lanes of a warp in distinct banks, and the high-
// byte-0 counters of the eight rows follow in the 33 spare words.
//
// Lane c of a counting warp takes the 8 experts 8c..8c+7 (one 16-byte chunk)
// of a token: pair rows 4c..4c+3.  A counter gains at most one per token, so
// the block's counters must be added into H at least every 65,535 tokens.
#pragma once

#include "eqb_device.cuh"

namespace eqb {

constexpr uint32_t kWinBias = 0x00c800c8u;  // -56 mod 256 in both 16-bit lanes
constexpr int kWinLo = 56;

// Shared-memory words of the window bins of E experts.
__host__ __device__ constexpr int coarse_window_words(int E) { return (E / 16) * 289; }

// The counter addresses of lane chunk cc: the four pair rows, and the
// high-byte-0 counters of those rows (zbase + 4p).
__device__ __forceinline__ void coarse_window_bases(uint32_t bins_saddr, int cc, uint32_t (&cbase)[4],
                                                    uint32_t& zbase) {
#pragma unroll
  for (int p = 0; p < 4; ++p)
    cbase[p] = bins_saddr + 4u * static_cast<uint32_t>(289 * (cc >> 1) + 16 * ((p << 1) | (cc & 1)));
  zbase = bins_saddr + 4u * static_cast<uint32_t>(289 * (cc >> 1) + 256 + 4 * (cc & 1));
}

// A pair with a margin outside the window and not of high byte 0: the rare
// case.
__device__ __forceinline__ void coarse_window_outside_body(uint32_t y, uint32_t k, uint32_t crow, uint32_t zword,
                                                           int e0, int32_t* hist, int32_t* err) {
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const uint32_t sh = (y >> (16 * h)) & 0xffu;
    const uint32_t hk = (k >> (8 + 16 * h)) & 0xffu;  // internal high byte
    const uint32_t inc = h ? 0x10000u : 1u;
    if ((sh & 0x70u) == 0u) {
      red_shared_add(crow + 4u * (sh & 0x8fu), inc);
    } else if (hk == 0u) {
      red_shared_add(zword, inc);
    } else {
      const uint32_t hb = hk ^ 0x80u;  // true high byte
      atomicAdd(hist + (int64_t)(e0 + h) * 256 + hb, 1);
      if (hb == 0u || hb == 255u) raise_flag(err, kErrNonfinite);
    }
  }
}

// The same out of line, for kernels whose other work keeps the memory system
// busy (the router projection's x stream): there an instruction fetch that
// misses the cache costs far more than the call, so the counting loop is kept
// small.
static __device__ __noinline__ void coarse_window_outside(uint32_t y, uint32_t k, uint32_t crow, uint32_t zword,
                                                          int e0, int32_t* hist, int32_t* err) {
  coarse_window_outside_body(y, k, crow, zword, e0, hist, err);
}

// Count the margins bf16_rne(tv - fp32(z)) of one token's chunk cc (8
// experts, 4 packed words w4) into the window (high byte 0 included), or
// into hist ([E,256], global) outside it.  Margins of magnitude >= 2^127 or
// non-finite raise EQB_ERR_NONFINITE.  OUTLINE: the high-byte-0 counters on
// the common path and everything else outside the window as a call (small
// code); otherwise both inline (fewer registers).
template <bool OUTLINE>
__device__ __forceinline__ void coarse_window_count(const uint4& w4, float tv, const uint32_t (&cbase)[4],
                                                    uint32_t zbase, int cc, int32_t* hist, int32_t* err) {
  const uint32_t zw[4] = {w4.x, w4.y, w4.z, w4.w};
  const uint64_t tt = f32x2_splat(tv);
#pragma unroll
  for (int p = 0; p < 4; ++p) {
    const uint32_t m = margins_bf16x2(tt, zw[p]);
    const uint32_t k = kappa2_internal(m);
    const uint32_t y = prmt(k, 0u, 0x4341u) + kWinBias;  // (hk - 56) per 16-bit lane (+ a carry bit)
    if constexpr (OUTLINE) {
      // high byte 0 (y_h == 0xc8) counted here too: with b = 0 every token
      // has one such margin, the cutoff expert's own
      const uint32_t y0 = y & 0xffffu, y1 = y >> 16;
      const bool w0 = (y0 & 0x70u) == 0u, w1 = (y1 & 0x70u) == 0u;
      if ((w0 || y0 == 0xc8u) && (w1 || y1 == 0xc8u)) {
        const uint32_t a0 = w0 ? cbase[p] + 4u * (y0 & 0x8fu) : zbase + 4u * p;
        const uint32_t a1 = w1 ? cbase[p] + 4u * (y1 & 0x8fu) : zbase + 4u * p;
        if (a0 == a1) {
          red_shared_add(a0, 0x10001u);
        } else {
          red_shared_add(a0, 1u);
          red_shared_add(a1, 0x10000u);
        }
      } else {
        coarse_window_outside(y, k, cbase[p], zbase + 4u * p, cc * 8 + 2 * p, hist, err);
      }
    } else {
      if ((y & 0x00700070u) == 0u) {
        const uint32_t s0 = y & 0x8fu, s1 = (y >> 16) & 0x8fu;
        if (s0 == s1) {
          red_shared_add(cbase[p] + 4u * s0, 0x10001u);
        } else {
          red_shared_add(cbase[p] + 4u * s0, 1u);
          red_shared_add(cbase[p] + 4u * s1, 0x10000u);
        }
      } else {
        coarse_window_outside_body(y, k, cbase[p], zbase + 4u * p, cc * 8 + 2 * p, hist, err);
      }
    }
  }
}

// Add the non-zero window counters into hist and clear them; thread tid of
// nthreads takes words tid, tid + nthreads, ...
__device__ __forceinline__ void coarse_window_flush(uint32_t* bins, int words, int32_t* hist, int tid, int nthreads) {
  for (int w = tid; w < words; w += nthreads) {
    const uint32_t v = bins[w];
    if (!v) continue;
    bins[w] = 0u;
    const int blk = w / 289, o = w - 289 * blk;
    int e, hb;
    if (o < 256) {
      const int pos = (o & 127) >> 4, sl = (o & 15) | (o & 128);
      e = 2 * (8 * blk + (((pos & 1) << 2) | (pos >> 1)));
      hb = ((sl + kWinLo) & 0xff) ^ 0x80;
    } else {
      e = 2 * (8 * blk + (o - 256));  // the row's high-byte-0 counter
      hb = 0x80;
    }
    if (v & 0xffffu) atomicAdd(hist + (int64_t)e * 256 + hb, static_cast<int>(v & 0xffffu));
    if (v >> 16) atomicAdd(hist + (int64_t)(e + 1) * 256 + hb, static_cast<int>(v >> 16));
  }
}

}  // namespace eqb
