// router_gemm.cu -- router logits z_t = W_r x_t (arXiv 2609.28053, Sec. 2,
// Eq. 1), z = bf16_rne(x W_r^T) with fp32 accumulation on the tensor cores.
//
// A persistent kernel, one CTA per SM, 6 warps with fixed roles:
//   warp 0      TMA producer: 128-row x 64-column bf16 tiles of x and the
//               matching [E x 64] tile of W_r, 128-byte swizzled, into a ring
//               of shared-memory stages guarded by mbarriers (full/empty);
//   warp 1      owns the tensor memory (TMEM) and issues tcgen05.mma
//               (M=128, N=E, K=16, bf16 inputs, fp32 accumulate) from one
//               thread; tcgen05.commit frees each stage and, at the end of a
//               tile, signals the accumulator as full;
//   warps 2..5  epilogue: tcgen05.ld of the accumulator (warp w reads TMEM
//               lanes 32*(w%4) ..+31 = its 32 rows), round to bf16, store z;
//               with routing (E = 64, 128) each lane also routes its token
//               from the accumulator, and with the coarse histogram the warp
//               then recounts its 32 stored rows (read back from L2, lane c
//               taking experts 8c..8c+7 of a token) into the window bins of
//               coarse_window.cuh (Algorithm 1 step 1), so the coarse pass
//               does not read z again.
// Two accumulators (2 x E fp32 columns of TMEM) alternate, so the epilogue
// of one tile overlaps the MMAs of the next.
//
// Every wait is bounded: a wait that runs out sets a shared abort flag that
// makes all roles leave their loops, the MMA thread drains its outstanding
// tensor-core work through one more commit, TMEM is freed, and the kernel
// reports EQB_ERR_CUDA through the error word.
#include <cuda.h>

#include "coarse_window.cuh"
#include "eqb_device.cuh"

namespace eqb {

namespace {

constexpr int kBM = 128;  // rows of x per tile (UMMA M)
constexpr int kBK = 64;   // bf16 columns per stage: one 128-byte swizzle atom
constexpr uint32_t kSpinLimit = 1u << 20;  // polls of at most ~1 us: about a second

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(1000u)
      : "memory");
  return ok != 0;
}
// Bounded wait for the phase of parity `parity`; false if it timed out or
// another role aborted.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  for (uint32_t i = 0; i < kSpinLimit; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 63u && *abort_flag) return false;
  }
  *abort_flag = 1;
  return false;
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int c0,
                                            int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1)
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// UMMA shared-memory descriptor of a K-major tile stored as 128-byte swizzled
// rows (8-row atoms of 1 KiB): start address >> 4 (bits 0-13), leading byte
// offset 16 B (unused for this layout), stride byte offset 1 KiB between
// 8-row groups (bits 32-45), descriptor version 1 (bit 46), swizzle mode
// 128B (value 2 in bits 61-63).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(16u >> 4) << 16;
  d |= static_cast<uint64_t>(1024u >> 4) << 32;
  d |= static_cast<uint64_t>(1u) << 46;
  d |= static_cast<uint64_t>(2u) << 61;
  return d;
}

// Instruction descriptor, kind::f16: fp32 accumulator (bits 4-5 = 1), A and
// B bf16 (bits 7-9 = 1, 10-12 = 1), both K-major, N >> 3 in bits 17-22,
// M >> 4 in bits 24-28.
__host__ __device__ constexpr uint32_t umma_idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((static_cast<uint32_t>(N) >> 3) << 17) |
         ((static_cast<uint32_t>(M) >> 4) << 24);
}

__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

constexpr uint32_t kTmemCols = 512;  // the whole TMEM of the SM: one CTA per SM

struct GemmArgs {
  uint16_t* z;
  int T, d, N, S;
  int32_t* err;
  // routing from the accumulator (EC > 0): as in eqb_route_topk
  const float* b;
  int K;
  const int64_t* off;
  int M;
  int32_t* idx;
  float* tau;
  int32_t* loads;
  int32_t* hist;  // the coarse histogram [E,256] (+=), HIST kernels only
};

// Routing state of one token: the running top-(K+1) of s = fp32(z) + b.
template <int KP1>
struct TopState {
  float v[KP1];
  int id[KP1];
  bool nan;
};

// Insert the 32 experts c0 .. c0+31 of one token, given as 16 packed bf16
// words (the rounded logits), in index order: exact stable insertion, so
// ties keep the lower index first.
template <int KP1>
__device__ __forceinline__ void route_chunk(TopState<KP1>& st, const uint32_t (&p)[16], int c0,
                                            const float* bsm) {
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const float zf = (i & 1) ? bf16_hi(p[i >> 1]) : bf16_lo(p[i >> 1]);
    const float sc = zf + bsm[c0 + i];
    st.nan |= (sc != sc);
    insert_sorted<KP1>(st.v, st.id, sc, c0 + i);
  }
}

// The cutoff tau_t = v[K] of a routed token.
template <int KP1>
__device__ __forceinline__ float top_tau(const TopState<KP1>& st, int K) {
  float tau_t = st.v[0];
#pragma unroll
  for (int j = 1; j < KP1; ++j) tau_t = (j == K) ? st.v[j] : tau_t;
  return tau_t;
}

// tau and the top-K list of one routed token.
template <int EC, int KP1>
__device__ __forceinline__ void route_outputs(const TopState<KP1>& st, int row, const GemmArgs& a) {
  const int K = a.K;
  const float tau_t = top_tau<KP1>(st, K);
  a.tau[row] = tau_t;
  if (st.nan || !isfinite(tau_t)) raise_flag(a.err, kErrNonfinite);
  if (a.idx) {
#pragma unroll
    for (int j = 0; j < KP1; ++j)
      if (j < K) a.idx[static_cast<int64_t>(row) * K + j] = st.id[j];
  }
}

// Per-warp expert counts of the microbatch `cur` not yet added to loads: EC
// 16-bit counters packed in pairs (expert e in the half e & 1 of word e / 2).
// A warp adds at most 32 to a counter per tile and flushes before 2047 tiles
// have passed, so no half overflows.
template <int EC>
struct WarpLoads {
  uint32_t* cnt;  // EC / 2 shared words of this warp
  int cur;        // microbatch being counted, -1 before the first
  int tiles;      // tiles counted since the last flush
};

template <int EC>
__device__ __forceinline__ void flush_loads(WarpLoads<EC>& wl, const GemmArgs& a, int lane) {
  __syncwarp();  // every lane's shared-memory adds are visible
  if (wl.cur >= 0) {
#pragma unroll
    for (int w = lane; w < EC / 2; w += 32) {
      const uint32_t c = wl.cnt[w];
      if (c) {
        wl.cnt[w] = 0;
        int32_t* dst = a.loads + static_cast<int64_t>(wl.cur) * EC + 2 * w;
        if (c & 0xffffu) atomicAdd(dst, static_cast<int>(c & 0xffffu));
        if (c >> 16) atomicAdd(dst + 1, static_cast<int>(c >> 16));
      }
    }
  }
  __syncwarp();
  wl.tiles = 0;
}

// Count the top-K experts of this lane's token (if valid) into its
// microbatch.  Tokens of the microbatch the warp is counting go to shared
// memory; a tile that starts another microbatch flushes first, and the few
// tokens of a tile that straddles a boundary go straight to global memory.
// Called by all 32 lanes.
template <int EC, int KP1>
__device__ __forceinline__ void count_loads(WarpLoads<EC>& wl, const TopState<KP1>& st, bool valid, int row,
                                            const GemmArgs& a, int lane) {
  const int l = valid ? microbatch_of(a.off, a.M, row) : -1;
  const bool same = !valid || l == wl.cur;
  if (!__all_sync(0xffffffffu, same) || wl.tiles >= 2047) {
    flush_loads<EC>(wl, a, lane);
    const uint32_t vm = __ballot_sync(0xffffffffu, valid);
    if (vm) wl.cur = __shfl_sync(0xffffffffu, l, __ffs(vm) - 1);
  }
  ++wl.tiles;
  if (!valid) return;
  const int K = a.K;
  if (l == wl.cur) {
#pragma unroll
    for (int j = 0; j < KP1; ++j)
      if (j < K) red_shared_add(smem_u32(wl.cnt + (st.id[j] >> 1)), 1u << ((st.id[j] & 1) * 16));
  } else {
#pragma unroll
    for (int j = 0; j < KP1; ++j)
      if (j < K) atomicAdd(a.loads + static_cast<int64_t>(l) * EC + st.id[j], 1);
  }
}

// EC = 0: the plain GEMM for any supported N.  EC > 0: N = EC and the
// epilogue also routes each token (K + 1 <= KP1).  HIST: the epilogue also
// counts the coarse histogram into a.hist (launched only when no block
// counts more than 65,535 tokens, so the 16-bit window counters are added
// into H once, at the end).
template <int EC, int KP1, bool HIST>
__global__ void __launch_bounds__(192, 1)
    router_gemm_kernel(const __grid_constant__ CUtensorMap tmx, const __grid_constant__ CUtensorMap tmw,
                       GemmArgs a) {
  uint16_t* __restrict__ z = a.z;
  const int T = a.T, d = a.d, N = a.N, S = a.S;
  int32_t* err = a.err;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;  // 1 KiB alignment for the swizzle atoms
  uint8_t* sm = smem_raw + (base - raw);
  const uint32_t a_bytes = kBM * kBK * 2;
  const uint32_t b_bytes = static_cast<uint32_t>(N) * kBK * 2;
  const uint32_t stage_bytes = a_bytes + b_bytes;
  const uint32_t bars = base + static_cast<uint32_t>(S) * stage_bytes;  // 8-byte mbarriers
  auto full = [&](int s) { return bars + 8u * s; };
  auto empty = [&](int s) { return bars + 8u * (S + s); };
  auto accf = [&](int b) { return bars + 8u * (2 * S + b); };
  auto acce = [&](int b) { return bars + 8u * (2 * S + 2 + b); };
  const uint32_t drain = bars + 8u * (2 * S + 4);
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(sm + static_cast<size_t>(S) * stage_bytes +
                                                      8u * (2 * S + 5));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  // routing only: b (EC floats), then 4 warps x EC/2 packed load counters
  float* bsm = reinterpret_cast<float*>(tmem_holder + 4);
  uint32_t* lcnt = reinterpret_cast<uint32_t*>(bsm + EC);
  uint32_t* bins = lcnt + 2 * EC;  // coarse window counters (HIST)
  constexpr int kBinWords = HIST ? coarse_window_words(EC) : 0;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (EC > 0) {
    for (int e = threadIdx.x; e < EC; e += blockDim.x) {
      const float bv = a.b[e];
      bsm[e] = bv;
      if (!isfinite(bv)) raise_flag(err, kErrNonfinite);
    }
    for (int w = threadIdx.x; w < 2 * EC; w += blockDim.x) lcnt[w] = 0;
    for (int w = threadIdx.x; w < kBinWords; w += blockDim.x) bins[w] = 0u;
  }
  const int ntiles = (T + kBM - 1) / kBM;
  const int KB = d / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full(s), 1);
      mbar_init(empty(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf(b), 1);
      mbar_init(acce(b), 128);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_holder)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmx)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmw)) : "memory");
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x) {
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(empty(stage), phase ^ 1u, abort_flag)) { ok = false; break; }
          const uint32_t dst = base + static_cast<uint32_t>(stage) * stage_bytes;
          mbar_expect_tx(full(stage), stage_bytes);
          tma_load_2d(dst, &tmx, full(stage), kb * kBK, tile * kBM);
          tma_load_2d(dst + a_bytes, &tmw, full(stage), kb * kBK, 0);
          if (++stage == S) { stage = 0; phase ^= 1u; }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_bf16(kBM, N);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      int it = 0;
      for (int tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x, ++it) {
        const int buf = it & 1;
        const uint32_t use = static_cast<uint32_t>(it >> 1);
        if (!mbar_wait(acce(buf), (use & 1u) ^ 1u, abort_flag)) break;
        tc_fence_after();
        const uint32_t dt = tmem + static_cast<uint32_t>(buf * N);
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(full(stage), phase, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sa = base + static_cast<uint32_t>(stage) * stage_bytes;
          const uint64_t ad = sw128_desc(sa), bd = sw128_desc(sa + a_bytes);
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk)  // K = 16 per MMA: +32 bytes in the atom
            umma_bf16(dt, ad + 2u * kk, bd + 2u * kk, idesc, (kb | kk) != 0 ? 1u : 0u);
          umma_commit(empty(stage));
          if (++stage == S) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        umma_commit(accf(buf));
      }
      // Drain: all MMAs issued above complete before TMEM is released.
      umma_commit(drain);
      for (uint32_t i = 0; i < kSpinLimit; ++i)
        if (mbar_try_wait(drain, 0u)) break;
    }
  } else {
    const int q = warp & 3;  // TMEM lane quarter accessible to this warp
    const uint32_t lane_base = static_cast<uint32_t>(q * 32) << 16;
    WarpLoads<EC> wl{lcnt + (warp - 2) * (EC / 2), -1, 0};
    // coarse counting: lane cc of token slot ctok takes experts 8cc..8cc+7
    constexpr int LPT = EC > 0 ? EC / 8 : 1, TPS = 32 / LPT;
    const int cc = lane % LPT, ctok = lane / LPT;
    uint32_t cbase[4], zbase = 0;
    if constexpr (HIST) coarse_window_bases(smem_u32(bins), cc, cbase, zbase);
    int it = 0;
    for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++it) {
      const int buf = it & 1;
      const uint32_t use = static_cast<uint32_t>(it >> 1);
      // the warp leaves together (the loop body has warp-wide operations)
      if (!__all_sync(0xffffffffu, mbar_wait(accf(buf), use & 1u, abort_flag))) break;
      tc_fence_after();
      const int row = tile * kBM + q * 32 + lane;
      if constexpr (EC == 0) {
        for (int c = 0; c < N; c += 32) {
          uint32_t r[32];
          tmem_ld32(tmem + lane_base + static_cast<uint32_t>(buf * N + c), r);
          if (row < T) {
            uint4* dst = reinterpret_cast<uint4*>(z + static_cast<size_t>(row) * N + c);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              if (c + 8 * v >= N) break;  // N is a multiple of 16, not always of 32
              uint4 o;
              o.x = pack_bf16x2_rn(__uint_as_float(r[8 * v + 0]), __uint_as_float(r[8 * v + 1]));
              o.y = pack_bf16x2_rn(__uint_as_float(r[8 * v + 2]), __uint_as_float(r[8 * v + 3]));
              o.z = pack_bf16x2_rn(__uint_as_float(r[8 * v + 4]), __uint_as_float(r[8 * v + 5]));
              o.w = pack_bf16x2_rn(__uint_as_float(r[8 * v + 6]), __uint_as_float(r[8 * v + 7]));
              dst[v] = o;
            }
          }
        }
        tc_fence_before();
        mbar_arrive(acce(buf));
      } else {
        // 32 columns at a time: round to bf16, store z, insert into the
        // token's running top-(K+1).  The accumulator stays in TMEM until the
        // whole row is read; routing a tile takes far less time than the MMAs
        // of the next one, which use the other accumulator meanwhile.
        TopState<KP1> st;
#pragma unroll
        for (int j = 0; j < KP1; ++j) { st.v[j] = -INFINITY; st.id[j] = 0; }
        st.nan = false;
#pragma unroll 1
        for (int c = 0; c < EC; c += 32) {
          uint32_t r[32], p[16];
          tmem_ld32(tmem + lane_base + static_cast<uint32_t>(buf * EC + c), r);
#pragma unroll
          for (int i = 0; i < 16; ++i) p[i] = pack_bf16x2_rn(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1]));
          if (row < T) {
            uint4* dst = reinterpret_cast<uint4*>(z + static_cast<size_t>(row) * EC + c);
#pragma unroll
            for (int v = 0; v < 4; ++v) dst[v] = make_uint4(p[4 * v], p[4 * v + 1], p[4 * v + 2], p[4 * v + 3]);
          }
          route_chunk<KP1>(st, p, c, bsm);
        }
        tc_fence_before();
        mbar_arrive(acce(buf));
        if (row < T) route_outputs<EC, KP1>(st, row, a);
        if (a.loads) count_loads<EC, KP1>(wl, st, row < T, row, a, lane);
        if constexpr (HIST) {
          // the coarse histogram of the warp's 32 rows, read back from L2
          // (every lane's z stores of this tile are ordered before the loads)
          // Four rows a batch, their loads issued before the batch's counts
          // (the shared-memory adds are ordered against memory); the loop
          // over batches stays rolled to keep the epilogue's code small.
          __syncwarp();
          const float tau_t = top_tau<KP1>(st, a.K);
          const int row0 = tile * kBM + q * 32;
          constexpr int NJ = 32 / TPS, NB = 4;
#pragma unroll 1
          for (int i0 = 0; i0 < NJ; i0 += NB) {
            uint4 w4[NB];
#pragma unroll
            for (int i = 0; i < NB; ++i) {
              const int j = (i0 + i) * TPS + ctok;
              w4[i] = row0 + j < T
                          ? __ldcg(reinterpret_cast<const uint4*>(z + static_cast<size_t>(row0 + j) * EC + 8 * cc))
                          : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int i = 0; i < NB; ++i) {
              const int j = (i0 + i) * TPS + ctok;
              const float tv = __shfl_sync(0xffffffffu, tau_t, j);
              if (row0 + j < T) coarse_window_count<true>(w4[i], tv, cbase, zbase, cc, a.hist, err);
            }
          }
        }
      }
    }
    if constexpr (EC > 0) {
      if (a.loads) flush_loads<EC>(wl, a, lane);
    }
  }
  tc_fence_before();
  __syncthreads();
  if constexpr (HIST) coarse_window_flush(bins, kBinWords, a.hist, threadIdx.x, blockDim.x);
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols)
                 : "memory");
  }
  if (threadIdx.x == 0 && *abort_flag) raise_flag(err, kErrCuda);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                                  CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 2-D bf16 tensor map over a row-major [rows, cols] matrix, box [box_rows, 64]
// (64 bf16 = one 128-byte swizzle atom per row).
bool make_map(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

namespace {

template <int EC, int KP1, bool HIST>
int launch_gemm(const uint16_t* x, const uint16_t* W, GemmArgs a, cudaStream_t s) {
  DeviceInfo di;
  if (int rc = device_info(&di)) return rc;
  CUtensorMap tmx, tmw;
  if (!make_map(&tmx, x, static_cast<uint64_t>(a.T), static_cast<uint64_t>(a.d), kBM)) return kErrCuda;
  if (!make_map(&tmw, W, static_cast<uint64_t>(a.N), static_cast<uint64_t>(a.d), static_cast<uint32_t>(a.N)))
    return kErrCuda;
  const int stage_bytes = (kBM + a.N) * kBK * 2;
  // alignment slack, 2S+5 mbarriers (S <= 8), TMEM address + abort flag, b,
  // the epilogue warps' load counters
  const int extra = 1024 + 8 * (2 * 8 + 5) + 16 + 4 * EC + 8 * EC + (HIST ? 4 * coarse_window_words(EC) : 0);
  int S = (di.max_smem_optin - extra) / stage_bytes;
  if (S > 8) S = 8;
  if (S < 2) return kErrUnsupported;
  a.S = S;
  const int smem = S * stage_bytes + extra;
  const int ntiles = (a.T + kBM - 1) / kBM;
  const int grid = ntiles < di.sm_count ? ntiles : di.sm_count;
  if (cudaFuncSetAttribute(router_gemm_kernel<EC, KP1, HIST>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
      cudaSuccess)
    return kErrCuda;
  router_gemm_kernel<EC, KP1, HIST><<<grid, 192, smem, s>>>(tmx, tmw, a);
  return cudaGetLastError() == cudaSuccess ? kOk : kErrCuda;
}

}  // namespace

int launch_router_gemm(const uint16_t* x, const uint16_t* W, int64_t T, int d, int E, uint16_t* z,
                       int32_t* err, cudaStream_t s) {
  GemmArgs a{z, static_cast<int>(T), d, E, 0, err, nullptr, 0, nullptr, 0, nullptr, nullptr, nullptr, nullptr};
  return launch_gemm<0, 1, false>(x, W, a, s);
}

namespace {

template <int EC, bool HIST>
int launch_route_ec(const uint16_t* x, const uint16_t* W, const GemmArgs& a, cudaStream_t s) {
  return a.K + 1 <= 3 ? launch_gemm<EC, 3, HIST>(x, W, a, s) : launch_gemm<EC, 9, HIST>(x, W, a, s);
}

}  // namespace

int launch_router_route(const uint16_t* x, const uint16_t* W, int64_t T, int d, int E, int K, const float* b,
                        const int64_t* off, int M, uint16_t* z, int32_t* idx, float* tau, int32_t* loads,
                        int32_t* hist, int32_t* err, cudaStream_t s) {
  GemmArgs a{z, static_cast<int>(T), d, E, 0, err, b, K, off, M, idx, tau, loads, hist};
  if (E != 64 && E != 128) return kErrUnsupported;
  bool in_epilogue = false;
  if (hist) {
    // the epilogue's 16-bit window counters are added into H once, at the
    // end: only while no block counts more than 65,535 tokens
    DeviceInfo di;
    if (int rc = device_info(&di)) return rc;
    const int64_t ntiles = (T + kBM - 1) / kBM;
    const int64_t grid = ntiles < di.sm_count ? ntiles : di.sm_count;
    in_epilogue = (ntiles + grid - 1) / grid * kBM <= 65535;
  }
  int rc;
  if (E == 64) rc = in_epilogue ? launch_route_ec<64, true>(x, W, a, s) : launch_route_ec<64, false>(x, W, a, s);
  else rc = in_epilogue ? launch_route_ec<128, true>(x, W, a, s) : launch_route_ec<128, false>(x, W, a, s);
  if (rc || !hist || in_epilogue) return rc;
  // larger T: the coarse pass as its own kernel over the z just written
  HistArgs h{z, tau, T, E, nullptr, hist, err};
  return launch_hist(h, 1, s);
}

}  // namespace eqb
