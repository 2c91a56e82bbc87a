// step.cu -- one call for a layer's whole routing-balance step (the host-side
// order of launches; every step runs in the library's kernels).
//
// Order of work, as in the paper: routing (Sec. 2), Algorithm 1's coarse
// pass, selection, fine pass, selection and the Eq. (2) bias update, and
// Load-Error Injection (Sec. 4, Eqs. LEI and norm).  LEI needs only the
// loads, so when its [M,E] coefficient table fits the workspace the
// coefficients are formed right after routing and the two histogram passes
// stream the injection, half of the tokens each; otherwise it runs last.
// All on one stream.
// eqb_router_layer_step starts one step earlier, at the router projection
// (Eq. 1), and routes from the projection's accumulators where it can; that
// kernel also counts the coarse histogram, so the fine pass alone reads z
// again and carries all of LEI.
#include <cuda_runtime.h>
#include <stdint.h>

#include "eqb.h"
#include "eqb_internal.h"

namespace eqb {

size_t carve_workspace(void* base, int E, StepWorkspace* w) {
  size_t off = 0;
  auto take = [&](size_t n) {
    uint8_t* p = base ? static_cast<uint8_t*>(base) + off : nullptr;
    off += carve_round(n);
    return p;
  };
  w->H = reinterpret_cast<int32_t*>(take(static_cast<size_t>(E) * 256 * 4));
  w->L = reinterpret_cast<int32_t*>(take(static_cast<size_t>(E) * 256 * 4));
  w->done = reinterpret_cast<int32_t*>(take(8));
  w->u = take(static_cast<size_t>(E));
  w->rho = reinterpret_cast<int32_t*>(take(static_cast<size_t>(E) * 4));
  w->q = reinterpret_cast<uint16_t*>(take(static_cast<size_t>(E) * 2));
  w->coef = reinterpret_cast<float*>(take(static_cast<size_t>(kLeiCoefCap) * 4));
  return off;
}

}  // namespace eqb

namespace {

using Workspace = eqb::StepWorkspace;
inline size_t carve(void* base, int E, Workspace* w) { return eqb::carve_workspace(base, E, w); }

inline bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }
inline eqb_status st(int rc) { return static_cast<eqb_status>(rc); }

}  // namespace

extern "C" {

size_t eqb_layer_workspace_bytes(int32_t E) {
  if (E < 1) return 0;
  Workspace w;
  return carve(nullptr, E, &w);
}

}  // extern "C"

namespace {

// Checks shared by both step entry points; carves the workspace into w.
eqb_status check_step(const eqb_bf16* z, const float* b, int64_t T, int32_t E, int32_t K,
                      const int64_t* mb_offsets, const int64_t* mb_offsets_host, int32_t M,
                      int32_t* topk_idx, float* tau, int32_t* loads, float* b_next, float* grad_s,
                      float eta, float c, void* workspace, size_t workspace_bytes, int32_t* err_flag,
                      Workspace* w) {
  if (T < 1 || E < 2 || K < 1 || K >= E || M < 1) return EQB_ERR_INVALID_ARG;
  if (E > eqb::kMaxE || (E % 8) != 0 || K + 1 > 32) return EQB_ERR_UNSUPPORTED;
  if (T > (int64_t(1) << 31) - (int64_t(1) << 24)) return EQB_ERR_UNSUPPORTED;
  if (!z || !b || !mb_offsets || !tau || !loads || !b_next || !workspace) return EQB_ERR_INVALID_ARG;
  if (grad_s && (!(eta == eta) || !(c == c))) return EQB_ERR_INVALID_ARG;
  if (!aligned(z, 16) || !aligned(b, 4) || !aligned(mb_offsets, 8) || !aligned(topk_idx, 4) ||
      !aligned(tau, 4) || !aligned(loads, 4) || !aligned(b_next, 4) || !aligned(grad_s, 16) ||
      !aligned(workspace, 256) || !aligned(err_flag, 4))
    return EQB_ERR_INVALID_ARG;
  if (workspace_bytes < carve(workspace, E, w)) return EQB_ERR_INVALID_ARG;
  if (mb_offsets_host) {
    if (mb_offsets_host[0] != 0 || mb_offsets_host[M] != T) return EQB_ERR_INVALID_ARG;
    for (int l = 0; l < M; ++l)
      if (mb_offsets_host[l + 1] < mb_offsets_host[l]) return EQB_ERR_INVALID_ARG;
  }
  return EQB_OK;
}

eqb_status clear(const Workspace& w, int32_t* loads, int32_t E, int32_t M, cudaStream_t s) {
  // H, L and the block counters are adjacent in the workspace (H and L each
  // E*1 KiB, a multiple of the 256-byte carve alignment): one memset clears
  // them.
  if (cudaMemsetAsync(w.H, 0, 2 * eqb::carve_round(static_cast<size_t>(E) * 1024) + eqb::carve_round(8), s) !=
          cudaSuccess ||
      cudaMemsetAsync(loads, 0, static_cast<size_t>(M) * E * 4, s) != cudaSuccess)
    return EQB_ERR_CUDA;
  return EQB_OK;
}

// The two histogram passes of the step, each with its selection run by the
// pass's last block to finish counting (so neither selection is a launch of
// its own, and each overlaps the other blocks' LEI streaming): pass 1 counts
// H and selects u, rho at rank r; pass 2 counts L from u and selects q_hat,
// then b_next (Eq. 2).
eqb::HistArgs pass1_args(const Workspace& w, const eqb_bf16* z, const float* tau, int64_t T, int32_t E, int64_t r,
                         int32_t* err_flag) {
  eqb::HistArgs h{z, tau, T, E, nullptr, w.H, err_flag};
  h.done = w.done;
  h.r = r;
  h.sel_u = w.u;
  h.rho = w.rho;
  h.sel_err = err_flag;
  return h;
}
eqb::HistArgs pass2_args(const Workspace& w, const eqb_bf16* z, const float* tau, int64_t T, int32_t E,
                         float* b_next, int32_t* err_flag) {
  eqb::HistArgs h{z, tau, T, E, w.u, w.L, nullptr};
  h.done = w.done + 1;
  h.sel_u = w.u;
  h.rho = w.rho;
  h.q_hat = w.q;
  h.b_next = b_next;
  h.sel_err = err_flag;
  return h;
}

// Everything after routing: Algorithm 1's two passes with their selections,
// the Eq. (2) bias update and LEI.  When the [M,E] coefficient table fits the
// workspace, the coefficients are formed once and each histogram pass
// streams the injection of half of the tokens beside its counting (the
// passes are issue-bound, the injection DRAM-bound); the results are the
// same bits as the separate LEI launch.
eqb_status after_routing(const Workspace& w, const eqb_bf16* z, int64_t T, int32_t E, int32_t K,
                         const int64_t* mb_offsets, int32_t M, int64_t r, const float* tau,
                         const int32_t* loads, float* b_next, float* grad_s, float eta, float c,
                         int32_t* err_flag, cudaStream_t s) {
  const eqb::HistArgs h1 = pass1_args(w, z, tau, T, E, r, err_flag);
  const eqb::HistArgs h2 = pass2_args(w, z, tau, T, E, b_next, err_flag);
  if (grad_s && static_cast<int64_t>(M) * E <= eqb::kLeiCoefCap) {
    eqb::LeiArgs la{grad_s, loads, mb_offsets, M, 0, T, E, K, eta, c};
    if (int rc = eqb::launch_lei_coef(la, w.coef, s)) return st(rc);
    const int64_t th = T / 2;
    eqb::LeiStream l1{grad_s, w.coef, mb_offsets, M, 0, th};
    eqb::LeiStream l2{grad_s, w.coef, mb_offsets, M, th, T};
    if (int rc = eqb::launch_hist_lei(h1, 1, l1, s)) return st(rc);
    if (int rc = eqb::launch_hist_lei(h2, 2, l2, s)) return st(rc);
    return EQB_OK;
  }
  if (int rc = eqb::launch_hist(h1, 1, s)) return st(rc);
  if (int rc = eqb::launch_hist(h2, 2, s)) return st(rc);
  if (grad_s) {
    eqb::LeiArgs la{grad_s, loads, mb_offsets, M, 0, T, E, K, eta, c};
    if (int rc = eqb::launch_lei(la, s)) return st(rc);
  }
  return EQB_OK;
}

// Everything after routing when the coarse histogram H was already counted
// (the router projection's epilogue): selection, the fine pass with its
// selection and the bias update, with LEI streamed entirely by the fine pass
// when the [M,E] coefficient table fits the workspace, else run last.
eqb_status after_coarse(const Workspace& w, const eqb_bf16* z, int64_t T, int32_t E, int32_t K,
                        const int64_t* mb_offsets, int32_t M, int64_t r, const float* tau, const int32_t* loads,
                        float* b_next, float* grad_s, float eta, float c, int32_t* err_flag, cudaStream_t s) {
  const bool lei = grad_s && static_cast<int64_t>(M) * E <= eqb::kLeiCoefCap;
  if (lei) {
    eqb::LeiArgs la{grad_s, loads, mb_offsets, M, 0, T, E, K, eta, c};
    if (int rc = eqb::launch_lei_coef(la, w.coef, s)) return st(rc);
  }
  if (int rc = eqb::launch_select(w.H, E, 1, r, w.u, w.rho, nullptr, err_flag, s)) return st(rc);
  const eqb::HistArgs h2 = pass2_args(w, z, tau, T, E, b_next, err_flag);
  if (lei) {
    eqb::LeiStream l2{grad_s, w.coef, mb_offsets, M, 0, T};
    if (int rc = eqb::launch_hist_lei(h2, 2, l2, s)) return st(rc);
  } else {
    if (int rc = eqb::launch_hist(h2, 2, s)) return st(rc);
    if (grad_s) {
      eqb::LeiArgs la{grad_s, loads, mb_offsets, M, 0, T, E, K, eta, c};
      if (int rc = eqb::launch_lei(la, s)) return st(rc);
    }
  }
  return EQB_OK;
}

}  // namespace

extern "C" {

eqb_status eqb_layer_step(const eqb_bf16* z, const float* b, int64_t T, int32_t E, int32_t K,
                          const int64_t* mb_offsets, const int64_t* mb_offsets_host, int32_t M,
                          int64_t r, int32_t* topk_idx, float* tau, int32_t* loads, float* b_next,
                          float* grad_s, float eta, float c, void* workspace, size_t workspace_bytes,
                          int32_t* err_flag, void* stream) {
  Workspace w;
  eqb_status rs = check_step(z, b, T, E, K, mb_offsets, mb_offsets_host, M, topk_idx, tau, loads, b_next,
                             grad_s, eta, c, workspace, workspace_bytes, err_flag, &w);
  if (rs != EQB_OK) return rs;
  if (r <= 0) r = eqb_target_rank(T, E, K);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if ((rs = clear(w, loads, E, M, s)) != EQB_OK) return rs;
  eqb::RouteArgs ra{z, b, T, E, K, mb_offsets, M, 0, topk_idx, tau, loads, err_flag};
  if (int rc = eqb::launch_route(ra, s)) return st(rc);
  return after_routing(w, z, T, E, K, mb_offsets, M, r, tau, loads, b_next, grad_s, eta, c, err_flag, s);
}

eqb_status eqb_router_layer_step(const eqb_bf16* x, const eqb_bf16* W_r, int64_t T, int32_t d, int32_t E,
                                 int32_t K, const float* b, const int64_t* mb_offsets,
                                 const int64_t* mb_offsets_host, int32_t M, int64_t r, eqb_bf16* z,
                                 int32_t* topk_idx, float* tau, int32_t* loads, float* b_next,
                                 float* grad_s, float eta, float c, void* workspace,
                                 size_t workspace_bytes, int32_t* err_flag, void* stream) {
  if (!x || !W_r || d < 1) return EQB_ERR_INVALID_ARG;
  if ((d % 64) != 0 || (E % 16) != 0) return EQB_ERR_UNSUPPORTED;
  if (!aligned(x, 16) || !aligned(W_r, 16)) return EQB_ERR_INVALID_ARG;
  Workspace w;
  eqb_status rs = check_step(z, b, T, E, K, mb_offsets, mb_offsets_host, M, topk_idx, tau, loads, b_next,
                             grad_s, eta, c, workspace, workspace_bytes, err_flag, &w);
  if (rs != EQB_OK) return rs;
  if (r <= 0) r = eqb_target_rank(T, E, K);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if ((rs = clear(w, loads, E, M, s)) != EQB_OK) return rs;
  if ((E == 64 || E == 128) && K <= 8) {
    // projection, routing and the coarse histogram in one kernel
    if (int rc = eqb::launch_router_route(x, W_r, T, d, E, K, b, mb_offsets, M, z, topk_idx, tau, loads, w.H,
                                          err_flag, s))
      return st(rc);
    return after_coarse(w, z, T, E, K, mb_offsets, M, r, tau, loads, b_next, grad_s, eta, c, err_flag, s);
  } else {
    if (int rc = eqb::launch_router_gemm(x, W_r, T, d, E, z, err_flag, s)) return st(rc);
    eqb::RouteArgs ra{z, b, T, E, K, mb_offsets, M, 0, topk_idx, tau, loads, err_flag};
    if (int rc = eqb::launch_route(ra, s)) return st(rc);
  }
  return after_routing(w, z, T, E, K, mb_offsets, M, r, tau, loads, b_next, grad_s, eta, c, err_flag, s);
}

}  // extern "C"
