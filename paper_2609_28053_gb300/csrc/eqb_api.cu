// eqb_api.cu -- the exported C ABI of libeqb.so (declared in include/eqb.h):
// host-side argument validation, then one launch per call on the caller's
// stream.  Invalid calls return before touching the GPU.
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "eqb.h"
#include "eqb_internal.h"

namespace eqb {

namespace {
constexpr int kMaxDevices = 64;
std::atomic<int> g_info_ready[kMaxDevices];
DeviceInfo g_info[kMaxDevices];
}  // namespace

int device_info(DeviceInfo* out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return kErrCuda;
  if (dev < 0 || dev >= kMaxDevices) return kErrUnsupported;
  if (g_info_ready[dev].load(std::memory_order_acquire)) {
    *out = g_info[dev];
    return kOk;
  }
  DeviceInfo di;
  if (cudaDeviceGetAttribute(&di.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return kErrCuda;
  if (cudaDeviceGetAttribute(&di.max_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
      cudaSuccess)
    return kErrCuda;
  g_info[dev] = di;
  g_info_ready[dev].store(1, std::memory_order_release);
  *out = di;
  return kOk;
}

}  // namespace eqb

namespace {

inline bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Sizes the library supports (the paper allows 1 <= K < E).
inline eqb_status check_shape(int64_t T, int32_t E, int32_t K, bool need_k) {
  if (T < 0 || E < 2) return EQB_ERR_INVALID_ARG;
  if (need_k && (K < 1 || K >= E)) return EQB_ERR_INVALID_ARG;
  if (E > eqb::kMaxE || (E % 8) != 0) return EQB_ERR_UNSUPPORTED;
  if (need_k && K + 1 > 32) return EQB_ERR_UNSUPPORTED;
  // 32-bit token loop indices need headroom above T.
  if (T > (int64_t(1) << 31) - (int64_t(1) << 24)) return EQB_ERR_UNSUPPORTED;
  return EQB_OK;
}

inline cudaStream_t as_stream(void* s) { return reinterpret_cast<cudaStream_t>(s); }

inline eqb_status to_status(int rc) { return static_cast<eqb_status>(rc); }

}  // namespace

extern "C" {

const char* eqb_status_string(int status) {
  switch (status) {
    case EQB_OK: return "EQB_OK";
    case EQB_ERR_INVALID_ARG: return "EQB_ERR_INVALID_ARG";
    case EQB_ERR_UNSUPPORTED: return "EQB_ERR_UNSUPPORTED";
    case EQB_ERR_CUDA: return "EQB_ERR_CUDA";
    case EQB_ERR_NONFINITE: return "EQB_ERR_NONFINITE";
    case EQB_ERR_RANK: return "EQB_ERR_RANK";
    default: return "EQB_ERR_UNKNOWN";
  }
}

int eqb_version(void) { return 100; }

int64_t eqb_target_rank(int64_t T, int32_t E, int32_t K) {
  if (T < 0 || E < 1 || K < 1) return -1;
  if (T > (INT64_MAX / 2) / (K > 0 ? K : 1)) return -1;
  return (T * (int64_t)K + E - 1) / E;
}

eqb_status eqb_route_topk(const eqb_bf16* z, const float* b, int64_t T, int32_t E, int32_t K,
                          const int64_t* mb_offsets, int32_t M, int32_t* topk_idx, float* tau,
                          int32_t* loads, int32_t* hist_hi, int32_t* err_flag, void* stream) {
  eqb_status st = check_shape(T, E, K, true);
  if (st != EQB_OK) return st;
  if (!z || !b || !tau) return EQB_ERR_INVALID_ARG;
  if (loads && (!mb_offsets || M < 1)) return EQB_ERR_INVALID_ARG;
  if (!aligned(z, 16) || !aligned(b, 4) || !aligned(tau, 4) || !aligned(topk_idx, 4) ||
      !aligned(loads, 4) || !aligned(hist_hi, 4) || !aligned(mb_offsets, 8) || !aligned(err_flag, 4))
    return EQB_ERR_INVALID_ARG;
  if (T == 0) return EQB_OK;
  eqb::RouteArgs a{z, b, T, E, K, mb_offsets, M, 0, topk_idx, tau, loads, err_flag};
  int rc = eqb::launch_route(a, as_stream(stream));
  if (rc != 0 || !hist_hi) return to_status(rc);
  eqb::HistArgs h{z, tau, T, E, nullptr, hist_hi, err_flag};
  return to_status(eqb::launch_hist(h, 1, as_stream(stream)));
}

eqb_status eqb_route_hist_fused(const eqb_bf16* z, const float* b, int64_t T, int32_t E, int32_t K,
                                const int64_t* mb_offsets, int32_t M, int32_t* topk_idx, float* tau,
                                int32_t* loads, int32_t* hist_hi, int32_t* err_flag, void* stream) {
  eqb_status st = check_shape(T, E, K, true);
  if (st != EQB_OK) return st;
  if (!eqb::route_hist_supported(E, K)) return EQB_ERR_UNSUPPORTED;
  if (!z || !b || !tau || !hist_hi) return EQB_ERR_INVALID_ARG;
  if (loads && (!mb_offsets || M < 1)) return EQB_ERR_INVALID_ARG;
  if (!aligned(z, 16) || !aligned(b, 4) || !aligned(tau, 4) || !aligned(topk_idx, 4) ||
      !aligned(loads, 4) || !aligned(hist_hi, 4) || !aligned(mb_offsets, 8) || !aligned(err_flag, 4))
    return EQB_ERR_INVALID_ARG;
  if (T == 0) return EQB_OK;
  eqb::RouteArgs a{z, b, T, E, K, mb_offsets, M, 0, topk_idx, tau, loads, err_flag};
  return to_status(eqb::launch_route_hist(a, hist_hi, as_stream(stream)));
}

eqb_status eqb_margin_hist_pass1(const eqb_bf16* z, const float* tau, int64_t T, int32_t E,
                                 int32_t* hist_hi, int32_t* err_flag, void* stream) {
  eqb_status st = check_shape(T, E, 1, false);
  if (st != EQB_OK) return st;
  if (!z || !tau || !hist_hi) return EQB_ERR_INVALID_ARG;
  if (!aligned(z, 16) || !aligned(tau, 4) || !aligned(hist_hi, 4) || !aligned(err_flag, 4))
    return EQB_ERR_INVALID_ARG;
  if (T == 0) return EQB_OK;
  eqb::HistArgs h{z, tau, T, E, nullptr, hist_hi, err_flag};
  return to_status(eqb::launch_hist(h, 1, as_stream(stream)));
}

eqb_status eqb_margin_hist_pass2(const eqb_bf16* z, const float* tau, int64_t T, int32_t E,
                                 const uint8_t* u, int32_t* hist_lo, void* stream) {
  eqb_status st = check_shape(T, E, 1, false);
  if (st != EQB_OK) return st;
  if (!z || !tau || !u || !hist_lo) return EQB_ERR_INVALID_ARG;
  if (!aligned(z, 16) || !aligned(tau, 4) || !aligned(hist_lo, 4)) return EQB_ERR_INVALID_ARG;
  if (T == 0) return EQB_OK;
  eqb::HistArgs h{z, tau, T, E, u, hist_lo, nullptr};
  return to_status(eqb::launch_hist(h, 2, as_stream(stream)));
}

eqb_status eqb_select_quantile(const int32_t* hist, int32_t E, int32_t pass, int64_t r, uint8_t* u,
                               int32_t* rho, eqb_bf16* q_hat, int32_t* err_flag, void* stream) {
  eqb_status st = check_shape(0, E, 1, false);
  if (st != EQB_OK) return st;
  if (!hist || !u || !rho) return EQB_ERR_INVALID_ARG;
  if (pass != 1 && pass != 2) return EQB_ERR_INVALID_ARG;
  if (pass == 1 && r < 1) return EQB_ERR_INVALID_ARG;
  if (pass == 2 && !q_hat) return EQB_ERR_INVALID_ARG;
  if (!aligned(hist, 4) || !aligned(rho, 4) || !aligned(q_hat, 2) || !aligned(err_flag, 4))
    return EQB_ERR_INVALID_ARG;
  return to_status(eqb::launch_select(hist, E, pass, r, u, rho, q_hat, err_flag, as_stream(stream)));
}

eqb_status eqb_bias_update(const eqb_bf16* q_hat, int32_t E, float* b_next, void* stream) {
  if (E < 1) return EQB_ERR_INVALID_ARG;
  if (E > eqb::kMaxE) return EQB_ERR_UNSUPPORTED;
  if (!q_hat || !b_next || !aligned(q_hat, 2) || !aligned(b_next, 4)) return EQB_ERR_INVALID_ARG;
  return to_status(eqb::launch_bias_update(q_hat, E, b_next, as_stream(stream)));
}

eqb_status lei_inject_grad(float* grad_s, const int32_t* loads, const int64_t* mb_offsets, int32_t M,
                           int64_t T, int32_t E, int32_t K, float eta, float c, void* stream) {
  eqb_status st = check_shape(T, E, K, true);
  if (st != EQB_OK) return st;
  if (!grad_s || !loads || !mb_offsets || M < 1) return EQB_ERR_INVALID_ARG;
  if (!(eta == eta) || !(c == c)) return EQB_ERR_INVALID_ARG;
  if (!aligned(grad_s, 16) || !aligned(loads, 4) || !aligned(mb_offsets, 8)) return EQB_ERR_INVALID_ARG;
  if (T == 0) return EQB_OK;
  eqb::LeiArgs a{grad_s, loads, mb_offsets, M, 0, T, E, K, eta, c};
  return to_status(eqb::launch_lei(a, as_stream(stream)));
}

eqb_status lei_coefficients(const int32_t* loads, const int64_t* mb_offsets, int32_t M, int32_t E, int32_t K,
                            float eta, float c, float* coef, void* stream) {
  eqb_status st = check_shape(0, E, K, true);
  if (st != EQB_OK) return st;
  if (!loads || !mb_offsets || !coef || M < 1) return EQB_ERR_INVALID_ARG;
  if (!(eta == eta) || !(c == c)) return EQB_ERR_INVALID_ARG;
  if (!aligned(loads, 4) || !aligned(mb_offsets, 8) || !aligned(coef, 16)) return EQB_ERR_INVALID_ARG;
  eqb::LeiArgs a{nullptr, loads, mb_offsets, M, 0, 0, E, K, eta, c};
  return to_status(eqb::launch_lei_coef(a, coef, as_stream(stream)));
}

eqb_status eqb_margin_hist_lei(const eqb_bf16* z, const float* tau, int64_t T, int32_t E, int32_t pass,
                               const uint8_t* u, int32_t* hist, int32_t* err_flag, float* grad_s,
                               const float* coef, const int64_t* mb_offsets, int32_t M, int64_t lei_t0,
                               int64_t lei_t1, void* stream) {
  eqb_status st = check_shape(T, E, 1, false);
  if (st != EQB_OK) return st;
  if (pass != 1 && pass != 2) return EQB_ERR_INVALID_ARG;
  if (!z || !tau || !hist || (pass == 2 && !u) || !grad_s || !coef || !mb_offsets || M < 1)
    return EQB_ERR_INVALID_ARG;
  if (lei_t0 < 0 || lei_t1 < lei_t0 || lei_t1 > T) return EQB_ERR_INVALID_ARG;
  if (!aligned(z, 16) || !aligned(tau, 4) || !aligned(hist, 4) || !aligned(err_flag, 4) ||
      !aligned(grad_s, 16) || !aligned(coef, 16) || !aligned(mb_offsets, 8))
    return EQB_ERR_INVALID_ARG;
  if (T == 0) return EQB_OK;
  eqb::HistArgs h{z, tau, T, E, pass == 2 ? u : nullptr, hist, pass == 1 ? err_flag : nullptr};
  eqb::LeiStream ls{grad_s, coef, mb_offsets, M, lei_t0, lei_t1};
  return to_status(eqb::launch_hist_lei(h, pass, ls, as_stream(stream)));
}

eqb_status eqb_router_logits(const eqb_bf16* x, const eqb_bf16* W_r, int64_t T, int32_t d, int32_t E,
                             eqb_bf16* z, int32_t* err_flag, void* stream) {
  if (T < 0 || d < 1 || E < 1) return EQB_ERR_INVALID_ARG;
  if ((d % 64) != 0 || (E % 16) != 0 || E > 256) return EQB_ERR_UNSUPPORTED;
  if (T > (int64_t(1) << 31) - (int64_t(1) << 24)) return EQB_ERR_UNSUPPORTED;
  if (!x || !W_r || !z) return EQB_ERR_INVALID_ARG;
  if (!aligned(x, 16) || !aligned(W_r, 16) || !aligned(z, 16) || !aligned(err_flag, 4))
    return EQB_ERR_INVALID_ARG;
  if (T == 0) return EQB_OK;
  return to_status(eqb::launch_router_gemm(x, W_r, T, d, E, z, err_flag, as_stream(stream)));
}

eqb_status eqb_router_route(const eqb_bf16* x, const eqb_bf16* W_r, int64_t T, int32_t d, int32_t E,
                            int32_t K, const float* b, const int64_t* mb_offsets, int32_t M, eqb_bf16* z,
                            int32_t* topk_idx, float* tau, int32_t* loads, int32_t* hist_hi, int32_t* err_flag,
                            void* stream) {
  if (T < 0 || d < 1 || E < 2 || K < 1 || K >= E) return EQB_ERR_INVALID_ARG;
  if ((d % 64) != 0 || (E != 64 && E != 128) || K > 8) return EQB_ERR_UNSUPPORTED;
  if (T > (int64_t(1) << 31) - (int64_t(1) << 24)) return EQB_ERR_UNSUPPORTED;
  if (!x || !W_r || !z || !b || !tau) return EQB_ERR_INVALID_ARG;
  if (loads && (!mb_offsets || M < 1)) return EQB_ERR_INVALID_ARG;
  if (!aligned(x, 16) || !aligned(W_r, 16) || !aligned(z, 16) || !aligned(b, 4) || !aligned(tau, 4) ||
      !aligned(topk_idx, 4) || !aligned(loads, 4) || !aligned(hist_hi, 4) || !aligned(mb_offsets, 8) ||
      !aligned(err_flag, 4))
    return EQB_ERR_INVALID_ARG;
  if (T == 0) return EQB_OK;
  return to_status(eqb::launch_router_route(x, W_r, T, d, E, K, b, mb_offsets, M, z, topk_idx, tau, loads,
                                            hist_hi, err_flag, as_stream(stream)));
}

eqb_status eqb_maxvio(const int32_t* loads, const int64_t* mb_offsets, int32_t M, int32_t E, int32_t K,
                      double* maxvio, double* per_mb, void* stream) {
  if (M < 1 || E < 1 || K < 1) return EQB_ERR_INVALID_ARG;
  if (M > 16384) return EQB_ERR_UNSUPPORTED;
  if (!loads || !mb_offsets || !maxvio) return EQB_ERR_INVALID_ARG;
  if (!aligned(loads, 4) || !aligned(mb_offsets, 8) || !aligned(maxvio, 8) || !aligned(per_mb, 8))
    return EQB_ERR_INVALID_ARG;
  return to_status(eqb::launch_maxvio(loads, mb_offsets, M, E, K, maxvio, per_mb, as_stream(stream)));
}

eqb_status gshard_inject_grad(float* grad_s, const eqb_bf16* z, const int32_t* loads, const int64_t* mb_offsets,
                              int32_t M, int64_t T, int32_t E, int32_t K, float alpha, void* stream) {
  if (T < 0 || E < 1 || K < 1 || M < 1) return EQB_ERR_INVALID_ARG;
  if ((E % 8) != 0 || E > eqb::kMaxE) return EQB_ERR_UNSUPPORTED;
  if (T > (int64_t(1) << 31) - (int64_t(1) << 24)) return EQB_ERR_UNSUPPORTED;
  if (!(alpha == alpha) || alpha == INFINITY || alpha == -INFINITY) return EQB_ERR_INVALID_ARG;
  if (!grad_s || !z || !loads || !mb_offsets) return EQB_ERR_INVALID_ARG;
  if (!aligned(grad_s, 16) || !aligned(z, 16) || !aligned(loads, 4) || !aligned(mb_offsets, 8))
    return EQB_ERR_INVALID_ARG;
  if (T == 0) return EQB_OK;
  eqb::GshardArgs a{grad_s, z, loads, mb_offsets, M, T, E, K, alpha};
  return to_status(eqb::launch_gshard(a, as_stream(stream)));
}

}  // extern "C"
