// eqb_device.cuh -- device helpers shared by the EQB / LEI kernels.
//
// bf16 values are handled as raw 16-bit patterns packed two per 32-bit
// word (lower half = lower expert index).  All fp32 arithmetic is IEEE
// round-to-nearest-even without flush-to-zero (the library is built without
// fast-math and with -fmad=false), so scores and margins are reproducible
// bit for bit.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "eqb_internal.h"

namespace eqb {

constexpr unsigned kFull = 0xffffffffu;

// Programmatic dependent launch.  The step's kernels are launched as
// dependents of the previous kernel in the stream, so a kernel's launch and
// its block-local set-up overlap the previous kernel's drain; each kernel
// calls griddep_wait() before it touches global memory (it returns once the
// previous grid has completed and its writes are visible; a no-op for a grid
// not launched as a dependent).  The implicit trigger at completion saves
// 17 us on the global step against plain launches.  Only the short kernels
// that precede a histogram pass (the LEI coefficient table, a selection)
// trigger their successor early, at their start: the pass's blocks take the
// SMs those leave idle and zero their bins meanwhile (1-3 us per step on
// every workload).  Early triggers in every kernel cost 60 us on the global
// step.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Let the next kernel in the stream launch now (it still waits, in
// griddep_wait, for this grid to complete).
__device__ __forceinline__ void griddep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Launch `kern` as a programmatic dependent of the previous work in `s`.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_dependent(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                    cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr.val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

// bf16 in the low / high half of a packed word -> fp32 (exact).
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ float bf16_bits_to_f32(uint32_t x16) { return __uint_as_float(x16 << 16); }

// Two fp32 values -> packed bf16x2, round to nearest even (lo -> low half).
__device__ __forceinline__ uint32_t pack_bf16x2_rn(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// (t - lo, t - hi) for the two bf16 values of a packed word, as one packed
// fp32 subtraction (round to nearest even, subnormals kept), rounded to a
// bf16 pair: the margins of two experts.  tt holds t in both halves.
__device__ __forceinline__ uint64_t f32x2_splat(float t) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %1};" : "=l"(r) : "f"(t));
  return r;
}
__device__ __forceinline__ uint32_t margins_bf16x2(uint64_t tt, uint32_t zw) {
  uint64_t zz, dd;
  asm("mov.b64 %0, {%1, %2};" : "=l"(zz) : "f"(__uint_as_float(zw << 16)), "f"(__uint_as_float(zw & 0xffff0000u)));
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(dd) : "l"(tt), "l"(zz));
  float lo, hi;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(dd));
  return pack_bf16x2_rn(lo, hi);
}

// fp32 max that propagates NaN (used where a NaN must stay visible).
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}

// Order-preserving 16-bit key of a bf16 pattern (Algorithm 1's kappa):
// negative patterns are complemented, non-negative ones get the sign bit.
__device__ __forceinline__ uint32_t kappa16(uint32_t x16) {
  return (x16 & 0x8000u) ? (~x16 & 0xffffu) : (x16 | 0x8000u);
}

__device__ __forceinline__ uint32_t kappa16_inv(uint32_t k16) {
  return (k16 & 0x8000u) ? (k16 & 0x7fffu) : (~k16 & 0xffffu);
}

// 16-byte shared-memory load.
__device__ __forceinline__ uint4 lds128(const void* p) { return *reinterpret_cast<const uint4*>(p); }

// Ampere-style asynchronous 16-byte global->shared copy (L2 only).  With
// src_bytes = 0 nothing is read and the destination is zero-filled.
__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gmem_src, int src_bytes) {
  uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(smem_dst));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d), "l"(gmem_src),
               "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

// Microbatch of token t: the largest l with off[l] <= t (empty microbatches
// are skipped automatically).  Requires 0 <= t < off[M].
__device__ __forceinline__ int microbatch_of(const int64_t* __restrict__ off, int M, int64_t t) {
  int lo = 0, hi = M - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (__ldg(off + mid) <= t) lo = mid; else hi = mid - 1;
  }
  return lo;
}

__device__ __forceinline__ void raise_flag(int32_t* err, int code) {
  if (err) atomicCAS(err, 0, code);
}

}  // namespace eqb

namespace eqb {

// ---- packed bf16x2 helpers (two bf16 values per 32-bit word)

__device__ __forceinline__ uint32_t hadd2_bf16(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("add.rn.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

__device__ __forceinline__ uint32_t hmax2_nan_bf16(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// max / min per half (a NaN half loses to a number).
__device__ __forceinline__ uint32_t hmax2_bf16(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
__device__ __forceinline__ uint32_t hmin2_bf16(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("min.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Per half: 0xffff where a >= b, else 0 (NaN compares false).
__device__ __forceinline__ uint32_t hge2_bf16(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("set.ge.u32.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Byte permute with the PTX default mode (a selector nibble with bit 3 set
// replicates the sign bit of the selected byte).
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
  uint32_t r;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
  return r;
}

// Internal keys of two packed bf16 patterns: kappa(x) ^ 0x8000 per half,
// i.e. x ^ 0x7fff for negative x, x otherwise.  The internal high byte is the
// true high byte ^ 0x80; the low byte is the true low byte.
__device__ __forceinline__ uint32_t kappa2_internal(uint32_t m) {
  const uint32_t sm = prmt(m, 0u, 0xBB99u);  // 0xffff per negative half
  return m ^ (sm & 0x7fff7fffu);
}

// bf16 pattern of fp32 x rounded toward -inf / +inf (exact values kept).
__device__ __forceinline__ uint32_t bf16_round_down(float x) {
  const uint32_t u = __float_as_uint(x);
  const uint32_t hi = u >> 16;
  if ((u & 0xffffu) == 0u) return hi;
  return (u & 0x80000000u) ? hi + 1u : hi;
}
__device__ __forceinline__ uint32_t bf16_round_up(float x) {
  const uint32_t u = __float_as_uint(x);
  const uint32_t hi = u >> 16;
  if ((u & 0xffffu) == 0u) return hi;
  return (u & 0x80000000u) ? hi : hi + 1u;
}

__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

__device__ __forceinline__ void red_shared_add(uint32_t saddr, uint32_t v) {
  asm volatile("red.shared.add.u32 [%0], %1;" ::"r"(saddr), "r"(v));
}


// Insert (s, e) into the descending list (v, id).  Candidates arrive in
// ascending e, so the new element goes after equal scores: its slot is
// p = #{j : v[j] >= s}; slots below p keep their entry, slot p takes the new
// one, slots above p take their predecessor's.  Every slot is computed from
// the old list, so there is no serial dependency between slots.
template <int KP1>
__device__ __forceinline__ void insert_sorted(float (&v)[KP1], int (&id)[KP1], float s, int e) {
  bool ge[KP1];
#pragma unroll
  for (int j = 0; j < KP1; ++j) ge[j] = v[j] >= s;
#pragma unroll
  for (int j = KP1 - 1; j >= 1; --j) {
    v[j] = ge[j] ? v[j] : (ge[j - 1] ? s : v[j - 1]);
    id[j] = ge[j] ? id[j] : (ge[j - 1] ? e : id[j - 1]);
  }
  v[0] = ge[0] ? v[0] : s;
  id[0] = ge[0] ? id[0] : e;
}

// Bitonic sort of N (a power of two) floats, descending.
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

// Bitonic sort, descending, of two independent N-element sequences packed
// as bf16 pairs: the low halves of a[0..N-1] form one, the high halves the
// other.  N is a power of two.
template <int N>
__device__ __forceinline__ void sort_desc_bf16x2(uint32_t (&a)[N]) {
#pragma unroll
  for (int k = 2; k <= N; k <<= 1) {
#pragma unroll
    for (int j = k >> 1; j > 0; j >>= 1) {
#pragma unroll
      for (int i = 0; i < N; ++i) {
        const int l = i ^ j;
        if (l > i) {
          const uint32_t hi = hmax2_bf16(a[i], a[l]), lo = hmin2_bf16(a[i], a[l]);
          if ((i & k) == 0) { a[i] = hi; a[l] = lo; } else { a[i] = lo; a[l] = hi; }
        }
      }
    }
  }
}

// bf16 pattern `steps` representable values below x (toward -inf), clamped
// at -inf.  Works on the order-preserving key.
__device__ __forceinline__ uint32_t bf16_steps_down(uint32_t x, uint32_t steps) {
  const uint32_t k = kappa16(x);
  const uint32_t kmin = 0x0080u + steps;  // key of -max_finite is 0x0080
  return k >= kmin ? kappa16_inv(k - steps) : 0xff80u;
}

// ---- shared-memory mbarriers (CTA scope)

__device__ __forceinline__ uint32_t saddr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void bar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void bar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
// One poll: true once the phase of parity `parity` has completed; otherwise
// the thread is suspended for at most about a microsecond (the time hint).
__device__ __forceinline__ bool bar_try_wait(uint32_t bar, uint32_t parity) {
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
// Wait for the phase of parity `parity`, giving up after `limit` polls:
// false means the phase did not complete (the caller reports an error and
// returns; no wait in this library is unbounded).
__device__ __forceinline__ bool bar_wait_bounded(uint32_t bar, uint32_t parity, uint32_t limit) {
  for (uint32_t i = 0; i < limit; ++i)
    if (bar_try_wait(bar, parity)) return true;
  return false;
}

// ---- Load-Error Injection streamed by one warp (Sec. 4, Eq. LEI), used by
// the histogram passes that carry LEI beside their counting.

// Token slice [q0, q1) of block `cta` out of `nct` blocks over [t0, t1).
__device__ __forceinline__ void lei_block_slice(int64_t t0, int64_t t1, int64_t cta, int64_t nct, int64_t* q0,
                                                int64_t* q1) {
  const int64_t n = t1 - t0;
  const int64_t per = (n + nct - 1) / nct;
  *q0 = t0 + min(cta * per, n);
  *q1 = t0 + min(cta * per + per, n);
}

// One warp adds coef[mb(t), e] to grad_s[t, e] for the tokens [ta, tb), in
// fp32 round to nearest, with evict-first 16-byte loads and stores and
// U loads in flight per lane.  (mlo, mhi, ml) caches the token range of
// the last microbatch looked up (start with mlo > mhi).  Tokens past the
// last boundary (malformed offsets) are the last microbatch's.
template <int U = 8>
__device__ __forceinline__ void lei_warp_tokens(const LeiStream& ls, int E, int64_t ta, int64_t tb, int64_t& mlo,
                                                int64_t& mhi, int& ml) {
  const int lane = threadIdx.x & 31;
  const int E4 = E >> 2;
  const int dcol = 32 % E4;
  float4* g4 = reinterpret_cast<float4*>(ls.g);
  const float4* c4 = reinterpret_cast<const float4*>(ls.coef);
  while (ta < tb) {
    if (ta < mlo || ta >= mhi) {
      ml = microbatch_of(ls.off, ls.M, ta);
      mlo = __ldg(ls.off + ml);
      mhi = __ldg(ls.off + ml + 1);
    }
    const int64_t se = mhi > ta ? min(tb, mhi) : tb;
    const float4* crow = c4 + (int64_t)ml * E4;
    int64_t i = ta * E4 + lane;
    const int64_t i1 = se * E4;
    int col = static_cast<int>(i % E4);
    for (; i + 32 * (U - 1) < i1; i += 32 * U) {
      float4 v[U];
      int cc[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        v[u] = __ldcs(g4 + i + 32 * u);
        cc[u] = col;
        col += dcol;
        if (col >= E4) col -= E4;
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const float4 cf = __ldg(crow + cc[u]);
        v[u].x = __fadd_rn(v[u].x, cf.x);
        v[u].y = __fadd_rn(v[u].y, cf.y);
        v[u].z = __fadd_rn(v[u].z, cf.z);
        v[u].w = __fadd_rn(v[u].w, cf.w);
        __stcs(g4 + i + 32 * u, v[u]);
      }
    }
    for (; i < i1; i += 32) {
      float4 v = __ldcs(g4 + i);
      const float4 cf = __ldg(crow + col);
      v.x = __fadd_rn(v.x, cf.x);
      v.y = __fadd_rn(v.y, cf.y);
      v.z = __fadd_rn(v.z, cf.z);
      v.w = __fadd_rn(v.w, cf.w);
      __stcs(g4 + i, v);
      col += dcol;
      if (col >= E4) col -= E4;
    }
    ta = se;
  }
}

// Tokens per chunk of a block's LEI slice: about 8 KiB of grad_s.
__device__ __forceinline__ int lei_chunk_tokens(int E) { return max(1, 2048 / E); }

// One warp takes the next chunk of [q0, q1) through the block's shared
// counter *next and streams it (U loads in flight per lane); false when the
// slice is used up.
template <int U = 8>
__device__ __forceinline__ bool lei_warp_next_chunk(const LeiStream& ls, int E, int64_t q0, int64_t q1, int* next,
                                                    int64_t& mlo, int64_t& mhi, int& ml) {
  int c = 0;
  if ((threadIdx.x & 31) == 0) c = atomicAdd(next, 1);
  c = __shfl_sync(kFull, c, 0);
  const int ch = lei_chunk_tokens(E);
  const int64_t ta = q0 + (int64_t)c * ch;
  if (ta >= q1) return false;
  lei_warp_tokens<U>(ls, E, ta, min(ta + ch, q1), mlo, mhi, ml);
  return true;
}
}  // namespace eqb
