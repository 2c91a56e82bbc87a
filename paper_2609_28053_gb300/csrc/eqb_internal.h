// eqb_internal.h -- launch-side declarations shared by the .cu files of
// libeqb.so (not part of the public ABI; see include/eqb.h for that).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace eqb {

// Status codes mirrored from eqb.h for device code.
enum : int {
  kOk = 0,
  kErrInvalidArg = 1,
  kErrUnsupported = 2,
  kErrCuda = 3,
  kErrNonfinite = 4,
  kErrRank = 5,
};

struct DeviceInfo {
  int sm_count;
  int max_smem_optin;  // bytes of dynamic shared memory a block may opt into
};

// Cached per-device attributes (queried once per device).
int device_info(DeviceInfo* out);

// Load-Error Injection streamed by a histogram pass beside its own work:
// grad_s[t, e] += coef[mb(t), e] for the tokens [t0, t1), from the [M,E]
// coefficient table of launch_lei_coef.  Token numbers are absolute.
struct LeiStream {
  float* g = nullptr;  // nullptr: no injection
  const float* coef = nullptr;
  const int64_t* off = nullptr;
  int M = 0;
  int64_t t0 = 0, t1 = 0;
};

struct RouteArgs {
  const uint16_t* z;
  const float* b;
  int64_t T;
  int E, K;
  const int64_t* off;  // microbatch boundaries, absolute token numbers
  int M;
  int64_t tbase;       // absolute number of token 0 of this call
  int32_t* idx;
  float* tau;
  int32_t* loads;
  int32_t* err;
};

// Largest expert count of the routing, EQB, LEI, GShard and MaxVio paths
// (per-expert state of the per-microbatch kernels lives in shared memory).
constexpr int kMaxE = 1024;

struct HistArgs {
  const uint16_t* z;
  const float* tau;
  int64_t T;
  int E;
  const uint8_t* u;  // pass 2 only
  int32_t* hist;
  int32_t* err;
  float lo = 0.f, inv_w = 0.f;  // pass 3 (equal-width bins) only
  // Optional token shards (device int64 [P+1]): shard p's counts go to
  // hist + p*E*256, and pass 2 takes shard p's selected bins from u + p*E.
  const int64_t* shard_off = nullptr;
  int P = 0;
  // Algorithm 1's selection run by the pass's last block to finish counting
  // (the one-call step; no shards): *done counts the blocks that finished
  // (zero before the pass).  Pass 1 selects u, rho at rank r; pass 2 selects
  // q_hat from u, rho and forms b_next (Eq. 2).  Selection flags go to
  // sel_err.
  int32_t* done = nullptr;
  int64_t r = 0;
  uint8_t* sel_u = nullptr;
  int32_t* rho = nullptr;
  uint16_t* q_hat = nullptr;
  float* b_next = nullptr;
  int32_t* sel_err = nullptr;
};

struct LeiArgs {
  float* g;
  const int32_t* loads;
  const int64_t* off;  // microbatch boundaries, absolute token numbers
  int M;
  int64_t tbase;       // absolute number of token 0 of this call
  int64_t T;
  int E, K;
  float eta, c;
};

struct GshardArgs {
  float* g;
  const uint16_t* z;
  const int32_t* loads;
  const int64_t* off;
  int M;
  int64_t T;
  int E, K;
  float alpha;
};

// Capacity (floats) of the step's LEI coefficient table: the fused step
// (injection streamed by the histogram passes) runs when M * E fits.
constexpr int64_t kLeiCoefCap = 65536;

// The step's scratch, carved from one caller-provided buffer (256-byte
// aligned pieces): the two [E,256] histograms and the passes' two block
// counters (adjacent, cleared together before every step), u, rho, q_hat and
// the [M,E] LEI coefficient table.
struct StepWorkspace {
  int32_t* H;
  int32_t* L;
  int32_t* done;  // [2]: blocks of pass 1 and of pass 2 done counting
  uint8_t* u;
  int32_t* rho;
  uint16_t* q;
  float* coef;
};
constexpr size_t carve_round(size_t n) { return (n + 255) / 256 * 256; }
constexpr size_t step_workspace_bytes(int E) {
  return 2 * carve_round(static_cast<size_t>(E) * 1024) + carve_round(8) + carve_round(static_cast<size_t>(E)) +
         carve_round(4 * static_cast<size_t>(E)) + carve_round(2 * static_cast<size_t>(E)) +
         carve_round(4 * static_cast<size_t>(kLeiCoefCap));
}
// Carves `base` (or, with base == nullptr, only measures); returns the bytes
// used, step_workspace_bytes(E) by construction.
size_t carve_workspace(void* base, int E, StepWorkspace* w);

int launch_route(const RouteArgs& a, cudaStream_t s);
bool route_wide_supported(int E, int K);
int launch_route_wide(const RouteArgs& a, cudaStream_t s);
// Routing and the coarse histogram (hist, [E,256] +=) in one pass over z
// (route_hist.cu; E = 128 or 256, K + 1 <= 16).
bool route_hist_supported(int E, int K);
int launch_route_hist(const RouteArgs& a, int32_t* hist, cudaStream_t s);
int launch_hist(const HistArgs& a, int pass, cudaStream_t s);
// A histogram pass (1 or 2) with the injection `ls` streamed beside it.
int launch_hist_lei(const HistArgs& a, int pass, const LeiStream& ls, cudaStream_t s);
int launch_select(const int32_t* hist, int E, int pass, int64_t r, uint8_t* u, int32_t* rho,
                  uint16_t* q_hat, int32_t* err, cudaStream_t s);
// One selection per token shard (device int64 [P+1]): shard p reads
// hist + p*E*256 and writes u, rho, q_hat + p*E at its own rank
// ceil(n_p K / E); an empty shard gets u = rho = 0 and q_hat = +0.
int launch_select_sharded(const int32_t* hist, int E, int pass, const int64_t* shard_off, int P, int K,
                          uint8_t* u, int32_t* rho, uint16_t* q_hat, int32_t* err, cudaStream_t s);
int launch_bias_update(const uint16_t* q_hat, int E, float* b_next, cudaStream_t s);
int launch_lei(const LeiArgs& a, cudaStream_t s);
// The [M,E] fp32 table of Eq. (norm) coefficients, row l for microbatch l
// (bit-identical to the coefficients launch_lei forms).
int launch_lei_coef(const LeiArgs& a, float* coef, cudaStream_t s);
int launch_router_gemm(const uint16_t* x, const uint16_t* W, int64_t T, int d, int E, uint16_t* z,
                       int32_t* err, cudaStream_t s);
int launch_gshard(const GshardArgs& a, cudaStream_t s);
int launch_maxvio(const int32_t* loads, const int64_t* off, int M, int E, int K, double* out, double* per_mb,
                  cudaStream_t s);
// The router projection routing each token from its accumulators (E = 64 or
// 128, K <= 8); with hist (nullable) also the coarse histogram ([E,256] +=),
// counted in the epilogue when no block routes more than 65,535 tokens, else
// by the coarse pass over z after it.
int launch_router_route(const uint16_t* x, const uint16_t* W, int64_t T, int d, int E, int K, const float* b,
                        const int64_t* off, int M, uint16_t* z, int32_t* idx, float* tau, int32_t* loads,
                        int32_t* hist, int32_t* err, cudaStream_t s);

}  // namespace eqb
