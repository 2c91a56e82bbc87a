// step_noalloc.cu -- eqb_layer_step with a workspace compiled into the
// library, for callers that cannot allocate device memory themselves.
//
// Who needs it: code hosted inside a framework or server that owns all of
// the device memory through its own pool (an allocation behind the pool's
// back can fail or throw off its accounting), and code that must not stall
// on, or fail at, an allocation in the middle of its work.  Such callers
// still provide the inputs and outputs; only the step's scratch (the two
// [E,256] histograms, u, rho and q_hat) lives here.
//
// The scratch is one file-scope device array sized for the largest supported
// E (256 experts): eqb_layer_workspace_bytes(256) = 788,480 bytes (the two
// [256,256] histograms, two block counters, u, rho, q_hat and the
// 65,536-float LEI coefficient table).  Every GPU that loads this library
// holds it until the process exits.  Host code cannot use the array's name as a
// device address, so the first call on each device, with that device
// current, looks the address up once with cudaGetSymbolAddress; make that
// first call before any stream capture.  All calls on a device share the
// array and it keeps the previous call's contents: the step clears the
// histograms itself before counting, and calls that overlap on the GPU (on
// different streams, or from different threads) race on it.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "eqb.h"
#include "eqb_internal.h"

namespace {

// eqb_layer_workspace_bytes(256): the carve of step.cu measures exactly this.
constexpr size_t kStaticWorkspaceBytes = eqb::step_workspace_bytes(256);
static __device__ __align__(256) unsigned char g_step_scratch[kStaticWorkspaceBytes];

constexpr int kMaxDevices = 64;
void* g_scratch_ptr[kMaxDevices] = {};
std::mutex g_scratch_mu;

// Device address of the scratch array on the current device (looked up once
// per device); NULL on failure.
void* scratch_on_current_device() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_step_scratch) != cudaSuccess) return nullptr;
    g_scratch_ptr[dev] = p;
  }
  return g_scratch_ptr[dev];
}

}  // namespace

extern "C" eqb_status eqb_layer_step_noalloc(const eqb_bf16* z, const float* b, int64_t T, int32_t E,
                                             int32_t K, const int64_t* mb_offsets,
                                             const int64_t* mb_offsets_host, int32_t M, int64_t r,
                                             int32_t* topk_idx, float* tau, int32_t* loads,
                                             float* b_next, float* grad_s, float eta, float c,
                                             int32_t* err_flag, void* stream) {
  if (E < 2 || E > 256) return E < 2 ? EQB_ERR_INVALID_ARG : EQB_ERR_UNSUPPORTED;
  const size_t need = eqb_layer_workspace_bytes(E);
  if (need == 0 || need > kStaticWorkspaceBytes) return EQB_ERR_UNSUPPORTED;
  // The workspace entry point validates the remaining arguments before any
  // work is queued; the scratch address is only needed once they pass.
  if (T < 1 || K < 1 || K >= E || M < 1 || !z || !b || !mb_offsets || !tau || !loads || !b_next)
    return EQB_ERR_INVALID_ARG;
  void* ws = scratch_on_current_device();
  if (!ws) return EQB_ERR_CUDA;
  return eqb_layer_step(z, b, T, E, K, mb_offsets, mb_offsets_host, M, r, topk_idx, tau, loads, b_next,
                        grad_s, eta, c, ws, kStaticWorkspaceBytes, err_flag, stream);
}
