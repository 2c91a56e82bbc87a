// hist.cu -- Algorithm 1's two margin-histogram passes (arXiv 2609.28053,
// Sec. 3 and App. C, steps 1 and 4).
//
// Both passes recompute every routing margin m = bf16_rne(tau_t - fp32(z))
// from z and tau instead of reading a stored margin array (Sec. 3: the second
// pass rescans the local margins).  Keys are kappa(m) (negative patterns
// complemented, others with the sign bit set).  Pass 1 counts the high byte of
// every key; pass 2 counts the low byte of the keys whose high byte is u_e.
// Pass 3 is the fixed-resolution histogram that Sec. 2 compares against:
// 256 equal bins, j = floor((m - lo) * inv_w) clamped to [0, 255].
//
// Work per element is kept to a handful of instructions by working on packed
// pairs: one 32-bit word of z holds two experts, their two fp32 differences
// are one packed f32x2 subtraction, rounded with one cvt.rn.bf16x2, and one
// PRMT (sign replicate) plus one LOP3 give both internal keys (kappa ^ 0x8000, so the stored high byte is the
// true one ^ 0x80 and is translated back at the flush).
//
// Bins: a CTA owns ET experts (all E when E <= 256 is a power of two) and
// keeps their 256 bins as 16-bit counters, two experts per 32-bit word: the
// experts of one z word share a word, the even one in the low half, so the
// increment is a constant.  ET * 512 bytes: 128 KiB for E = 256.  The ET/8
// lanes covering one token each own 8 experts; lane c's rows start c words
// past a 1 KiB boundary so equal bins of the 32 lanes fall in 32 banks.  A
// counter gains at most one per token, so the CTA flushes (adds its non-zero
// counters into the global int32 [E,256] histogram) at least every 65,535
// tokens; the flush is also how token partitions are summed in device memory.
// Each lane keeps eight 16-byte loads in flight (eight tokens per round),
// which covers the DRAM latency without L2 prefetches.
//
// Fused with Load-Error Injection (the one-call step): the passes are bound
// by issue, not by DRAM, while LEI (Sec. 4) is a pure DRAM stream that needs
// only the loads.  A fused block gives a quarter of its warps to streaming
// grad_s[t, e] += coef[mb(t), e] over its slice of a token range from the
// start, the other warps count, and each counting warp joins the stream when
// its counting is done; the stream is cut into chunks of about 8 KiB of
// grad_s handed out by a shared counter, so no warp idles while the block
// has work.  Each pass carries half of the step's tokens, which turns both
// passes into DRAM-bound ones.
#include "select_device.cuh"

namespace eqb {

namespace {

constexpr int kUnroll = 8;  // 16-byte loads in flight per lane (64 registers at 1024 threads)
constexpr int64_t kFlushTokens = 65535;
// The injection share of a fused block (see above): chunks of about 8 KiB of
// grad_s from this block's slice of [ls.t0, ls.t1), taken through the shared
// counter *next.  Every element gets one fp32 addition (round to nearest) of
// its microbatch's coefficient, as in lei.cu.
__device__ __forceinline__ void stream_lei(const LeiStream& ls, int E, int* next) {
  int64_t q0, q1;
  lei_block_slice(ls.t0, ls.t1, (int64_t)blockIdx.y * gridDim.x + blockIdx.x, (int64_t)gridDim.x * gridDim.y, &q0,
                  &q1);
  int64_t mlo = 1, mhi = 0;  // token range of microbatch ml (none yet)
  int ml = 0;
  while (lei_warp_next_chunk(ls, E, q0, q1, next, mlo, mhi, ml)) {
  }
}

// Algorithm 1's selection in the pass's last block to finish counting (see
// HistArgs::done), by its nw counting warps (warp wid, lane) with barrier
// sync(): pass 1 selects u, rho for every expert at rank a.r; pass 2 selects
// q_hat from u, rho into global memory and a shared copy qs, then forms
// b_next (Eq. 2).  Each warp loads the counts of three experts at a time
// (four spill registers of the counting loop); the counts were added by
// every block's atomics and are read from L2.
template <int PASS, class Sync>
__device__ void last_block_select(const HistArgs& a, int nw, int wid, int lane, uint16_t* qs, Sync sync) {
  constexpr int B = 3;
  const int E = a.E;
  for (int e0 = wid; e0 < E; e0 += nw * B) {
    int4 ca[B], cb[B];
    int32_t rk[B];
    uint32_t uk[B];
#pragma unroll
    for (int k = 0; k < B; ++k) {
      const int e = min(e0 + k * nw, E - 1);
      const int4* h = reinterpret_cast<const int4*>(a.hist + (int64_t)e * 256 + lane * 8);
      ca[k] = __ldcg(h);
      cb[k] = __ldcg(h + 1);
      rk[k] = PASS == 2 ? __ldcg(a.rho + e) : 0;
      uk[k] = PASS == 2 ? __ldcg(a.sel_u + e) : 0u;
    }
#pragma unroll
    for (int k = 0; k < B; ++k) {
      const int e = e0 + k * nw;
      if (e >= E) break;
      const int64_t cnt[8] = {ca[k].x, ca[k].y, ca[k].z, ca[k].w, cb[k].x, cb[k].y, cb[k].z, cb[k].w};
      if (PASS == 1)
        warp_select(cnt, e, 1, a.r, 0u, a.sel_u, a.rho, nullptr, a.sel_err, lane);
      else
        warp_select(cnt, e, 2, (int64_t)rk[k], uk[k], a.sel_u, a.rho, a.q_hat, a.sel_err, lane, qs + e);
    }
  }
  if (PASS == 2) {
    sync();  // every q_hat is in qs
    block_bias_update<true>(qs, E, a.b_next, nw * 32, sync);
  }
}

template <int LPT>
struct HistLayout {
  static constexpr int ET = LPT * 8;            // experts per CTA
  static constexpr int TPS = 32 / LPT;          // tokens per warp step
  static constexpr int kRows = ET / 2;          // one row per expert pair
  static constexpr int kWords = kRows * 256 + LPT;
  __host__ __device__ static int row_word(int row) { return row * 256 + (row >> 2); }
};

template <int PASS, int LPT, bool LEI>
__global__ void __launch_bounds__(1024) hist_kernel(HistArgs a, int64_t tokens_per_cta, LeiStream ls) {
  using Lay = HistLayout<LPT>;
  extern __shared__ __align__(16) uint32_t bins[];
  __shared__ int lei_next;  // next injection chunk of this block (fused only)
  const int E = a.E;
  const int e0 = blockIdx.x * Lay::ET;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nw = LEI ? (blockDim.x >> 5) - (blockDim.x >> 7) : (blockDim.x >> 5);  // counting warps
  const int nt = nw * 32;
  const int c = lane % LPT;     // 8-expert chunk of the tile owned by this lane
  const int tok = lane / LPT;   // token slot inside the warp step
  // Barrier of the counting warps (all warps unless fused).
  auto sync_counting = [&]() {
    if (LEI) asm volatile("bar.sync 1, %0;" ::"r"(nt) : "memory");
    else __syncthreads();
  };

  for (int i = threadIdx.x; i < Lay::kWords; i += blockDim.x) bins[i] = 0u;
  if (LEI && threadIdx.x == 0) lei_next = 0;
  // Shared address of this lane's first pair row; pair p adds p * 1 KiB.
  const uint32_t base = static_cast<uint32_t>(__cvta_generic_to_shared(bins)) +
                        4u * static_cast<uint32_t>(Lay::row_word(4 * c));
  uint32_t sel[4] = {0, 0, 0, 0};
  // internal high bytes (u ^ 0x80) of the selected bins, placed where the
  // internal keys carry them: bits 8-15 (even expert) and 24-31 (odd).
  auto load_sel = [&](const uint8_t* ub) {
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const uint32_t ue = ub[e0 + c * 8 + 2 * p] ^ 0x80u;
      const uint32_t uo = ub[e0 + c * 8 + 2 * p + 1] ^ 0x80u;
      sel[p] = (ue << 8) | (uo << 24);
    }
  };
  griddep_wait();  // the bins were zeroed above; global reads start here
  if (PASS == 2 && !a.shard_off) load_sel(a.u);
  __syncthreads();
  if (LEI && wid >= nw) {
    stream_lei(ls, E, &lei_next);
    return;
  }

  // Token indices fit in 32 bits (T < 2^31 is checked on the host).
  const int tb = static_cast<int>(min((int64_t)blockIdx.y * tokens_per_cta, a.T));
  const int te = static_cast<int>(min((int64_t)tb + tokens_per_cta, a.T));
  const int step = nw * Lay::TPS;  // tokens per warp round
  const size_t zstride = static_cast<size_t>(step) * E;
  const uint16_t* zlane = a.z + e0 + c * 8;

  auto process = [&](const uint4& w4, float tv) {
    const uint32_t zw[4] = {w4.x, w4.y, w4.z, w4.w};
    const uint64_t tt = f32x2_splat(tv);
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const uint32_t m = margins_bf16x2(tt, zw[p]);
      const uint32_t k = kappa2_internal(m);
      const uint32_t row = base + 1024u * p;
      if (PASS == 1) {
        const uint32_t he = prmt(k, 0u, 0x4441u), ho = k >> 24;  // internal high bytes
        const bool same = he == ho;
        red_shared_add(row + 4u * he, same ? 0x10001u : 1u);
        if (!same) red_shared_add(row + 4u * ho, 0x10000u);
      } else if (PASS == 3) {
        // equal-width bins: j = floor((m - lo) * inv_w), clamped to [0, 255]
        const uint32_t he = static_cast<uint32_t>(min(max(__float2int_rd(__fmul_rn(__fsub_rn(bf16_lo(m), a.lo), a.inv_w)), 0), 255));
        const uint32_t ho = static_cast<uint32_t>(min(max(__float2int_rd(__fmul_rn(__fsub_rn(bf16_hi(m), a.lo), a.inv_w)), 0), 255));
        const bool same = he == ho;
        red_shared_add(row + 4u * he, same ? 0x10001u : 1u);
        if (!same) red_shared_add(row + 4u * ho, 0x10000u);
      } else {
        const uint32_t d = (k ^ sel[p]) & 0xff00ff00u;
        if ((d & 0x0000ff00u) == 0u) red_shared_add(row + 4u * (k & 0xffu), 1u);
        if ((d & 0xff000000u) == 0u) red_shared_add(row + 4u * prmt(k, 0u, 0x4442u), 0x10000u);
      }
    }
  };

  for (int cb = tb; cb < te;) {
    int ce = static_cast<int>(min((int64_t)cb + kFlushTokens, (int64_t)te));
    int64_t hbase = 0;  // this chunk's histogram (shards: one per shard)
    if (a.shard_off) {
      const int sp = microbatch_of(a.shard_off, a.P, cb);
      const int64_t send = __ldg(a.shard_off + sp + 1);
      if (send > cb && send < ce) ce = static_cast<int>(send);  // chunks end at shard boundaries
      hbase = (int64_t)sp * E * 256;
      if (PASS == 2) load_sel(a.u + (int64_t)sp * E);
    }
    int t = cb + wid * Lay::TPS + tok;
    const uint16_t* zp = zlane + static_cast<size_t>(t) * E;
    // full rounds of kUnroll tokens per lane, no guards
    for (; t + (kUnroll - 1) * step < ce; t += kUnroll * step, zp += kUnroll * zstride) {
      uint4 w[kUnroll];
      float tt[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        w[u] = __ldcs(reinterpret_cast<const uint4*>(zp + u * zstride));
        tt[u] = __ldg(a.tau + t + u * step);
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) process(w[u], tt[u]);
    }
    for (; t < ce; t += step, zp += zstride) process(__ldcs(reinterpret_cast<const uint4*>(zp)), __ldg(a.tau + t));
    sync_counting();
    // Flush: add every non-zero 16-bit counter to the global histogram.
    for (int i = threadIdx.x; i < Lay::kRows * 256; i += nt) {
      const int row = i >> 8, slot = i & 255;
      const int wi = Lay::row_word(row) + slot;
      const uint32_t v = bins[wi];
      if (v) {
        bins[wi] = 0u;
        const int bin = (PASS == 1) ? (slot ^ 0x80) : slot;  // pass 1 stores internal keys
        const int ee = e0 + 2 * row;
        if (v & 0xffffu) atomicAdd(a.hist + hbase + (int64_t)ee * 256 + bin, static_cast<int>(v & 0xffffu));
        if (v >> 16) atomicAdd(a.hist + hbase + (int64_t)(ee + 1) * 256 + bin, static_cast<int>(v >> 16));
        if (PASS == 1 && (bin == 0 || bin == 255)) raise_flag(a.err, kErrNonfinite);
      }
    }
    sync_counting();
    cb = ce;
  }
  if (PASS != 3 && a.done && !a.shard_off) {
    // The last block to get here selects.  After the barrier above (every
    // flush of this block issued), one thread's fence releases the block's
    // flushes before its count; the last block's fence after its count
    // orders the other blocks' flushes before its reads.
    __shared__ int sel_last;
    if (threadIdx.x == 0) {
      __threadfence();
      const bool last = atomicAdd(a.done, 1) == (int)(gridDim.x * gridDim.y) - 1;
      if (last) __threadfence();
      sel_last = last;
    }
    sync_counting();
    if (sel_last) {
      // the bins are clear and no longer used: they hold the q_hat copy
      last_block_select<PASS>(a, nw, wid, lane, reinterpret_cast<uint16_t*>(bins), sync_counting);
    }
  }
  if (LEI) stream_lei(ls, E, &lei_next);
}

template <int PASS, int LPT, bool LEI>
int launch_hist_t(const HistArgs& a, const LeiStream& ls, cudaStream_t s) {
  using Lay = HistLayout<LPT>;
  DeviceInfo di;
  if (int rc = device_info(&di)) return rc;
  const int smem = Lay::kWords * 4;
  const int nE = a.E / Lay::ET;
  int ctas_per_sm = (228 * 1024 - 1024) / (smem + 1024);
  if (ctas_per_sm < 1) ctas_per_sm = 1;
  // One 1024-thread block per SM whenever the bins are large: the same
  // threads per SM as several smaller blocks, but a third of the zeroing and
  // flushing of the block-local counters (E = 64, 128: 10-20% faster).
  if (smem >= 32 * 1024) ctas_per_sm = 1;
  const int threads = ctas_per_sm == 1 ? 1024 : 512;
  if (ctas_per_sm > 2048 / threads) ctas_per_sm = 2048 / threads;
  int64_t nT = ((int64_t)di.sm_count * ctas_per_sm + nE - 1) / nE;
  const int64_t max_nT = (a.T + 2047) / 2048;  // keep >= ~2K tokens per CTA
  if (nT > max_nT) nT = max_nT;
  if (nT < 1) nT = 1;
  const int64_t tpc = (a.T + nT - 1) / nT;
  auto kern = hist_kernel<PASS, LPT, LEI>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return kErrCuda;
  dim3 grid((unsigned)nE, (unsigned)nT);
  return launch_dependent(kern, grid, dim3(threads), smem, s, a, tpc, ls) == cudaSuccess ? kOk : kErrCuda;
}

template <int PASS, bool LEI>
int launch_hist_pass(const HistArgs& a, const LeiStream& ls, cudaStream_t s) {
  if (a.E % 256 == 0) return launch_hist_t<PASS, 32, LEI>(a, ls, s);
  if (a.E % 128 == 0) return launch_hist_t<PASS, 16, LEI>(a, ls, s);
  if (a.E % 64 == 0) return launch_hist_t<PASS, 8, LEI>(a, ls, s);
  if (a.E % 32 == 0) return launch_hist_t<PASS, 4, LEI>(a, ls, s);
  if (a.E % 16 == 0) return launch_hist_t<PASS, 2, LEI>(a, ls, s);
  return launch_hist_t<PASS, 1, LEI>(a, ls, s);
}

}  // namespace

int launch_hist(const HistArgs& a, int pass, cudaStream_t s) {
  const LeiStream none;
  if (pass == 3) return launch_hist_pass<3, false>(a, none, s);
  return pass == 1 ? launch_hist_pass<1, false>(a, none, s) : launch_hist_pass<2, false>(a, none, s);
}

int launch_hist_lei(const HistArgs& a, int pass, const LeiStream& ls, cudaStream_t s) {
  if (!ls.g || !ls.coef || !ls.off || ls.M < 1 || ls.t0 < 0 || ls.t1 < ls.t0) return kErrInvalidArg;
  return pass == 1 ? launch_hist_pass<1, true>(a, ls, s) : launch_hist_pass<2, true>(a, ls, s);
}

}  // namespace eqb
