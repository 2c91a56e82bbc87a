/*
 * eqb.h -- C ABI of libeqb.so: the per-layer MoE routing-balance path of
 * Exact Quantile Balancing (EQB) and Load-Error Injection (LEI),
 * arXiv 2609.28053, on one NVIDIA GB300 (sm_103a).
 *
 * Notation follows the paper: T tokens, E routed experts, K experts per
 * token, router logits z[T,E], expert bias b[E], cutoff tau_t = the (K+1)st
 * largest entry of z_t + b, expert loads f_e, target rank r = TK/E.
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Pointers named as device buffers are CUDA device (or managed) pointers
 *    that the caller allocates and owns.  Unless a function says otherwise,
 *    the library allocates no device memory and keeps no state between calls.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Every call only enqueues work on it and returns without
 *    synchronising; results are valid once the stream has reached them.
 *  - Row-major layouts with the expert index fastest: z[t*E + e].
 *  - bf16 values travel as their raw 16-bit patterns (eqb_bf16).
 *  - Outputs documented as "+=" are accumulated into; the caller zeroes them
 *    first.  This is what lets token partitions (the data-parallel ranks of
 *    Algorithm 1, here slices of one batch) be summed in device memory, and
 *    lets a multi-GPU caller insert its own all-reduce between passes.
 *  - Return value: an eqb_status.  Arguments are validated on the host
 *    before anything is launched; an invalid call launches nothing.
 *    EQB_ERR_CUDA reports a launch failure (cudaGetLastError after launch).
 *  - Errors found by the device (non-finite data, an unreachable rank) are
 *    written to the optional device word `err_flag` (int32, nullable) as the
 *    eqb_status code; the caller zeroes it before the call and reads it after
 *    synchronising.  Outputs of a call that flagged an error are unspecified.
 *  - Microbatches (the paper's local batches B_l, Sec. 2) are contiguous
 *    token ranges given by device int64 offsets[M+1]: offsets[0] = 0,
 *    offsets[M] = T, non-decreasing (empty microbatches are allowed).
 *    The library reads them on the device; they are not checked on the host.
 *  - Supported sizes: 1 <= K, K + 1 <= 32, K < E, E a multiple of 8 with
 *    E <= 1024, T <= 2^31 - 2^24.  T = 0 is a valid no-op for the streaming
 *    calls.
 *  - Device buffers of bf16 logits must be 16-byte aligned; fp32 gradient
 *    buffers 16-byte aligned.  Misaligned pointers give EQB_ERR_INVALID_ARG.
 */
#ifndef EQB_H
#define EQB_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t eqb_bf16; /* raw bf16 bit pattern */

typedef enum eqb_status {
  EQB_OK = 0,
  EQB_ERR_INVALID_ARG = 1, /* host-side validation failed; nothing launched */
  EQB_ERR_UNSUPPORTED = 2, /* valid by the paper, outside the sizes the library supports */
  EQB_ERR_CUDA = 3,        /* a CUDA launch or runtime call failed */
  EQB_ERR_NONFINITE = 4,   /* device flag: non-finite z, b or score, or a
                              margin of magnitude >= 2^127 */
  EQB_ERR_RANK = 5         /* device flag: a histogram holds fewer than r
                              margins for some expert */
} eqb_status;

/* Human-readable name of a status code (static string). */
const char *eqb_status_string(int status);

/* Library version as MAJOR*10000 + MINOR*100 + PATCH. */
int eqb_version(void);

/* Target rank r = ceil(T*K / E) (Sec. 3: r = TK/E, assumed integral by the
 * paper; rounded up otherwise, the inverse-CDF quantile).  Returns -1 for
 * invalid arguments.  Host only. */
int64_t eqb_target_rank(int64_t T, int32_t E, int32_t K);

/* Routing and the coarse EQB pass.  Sec. 2 (Eq. 1 and the QB paragraph),
 * Algorithm 1 step 1.
 *
 * For each token t: s_e = fp32(z_{t,e}) + b_e (fp32, round to nearest
 * even); the top-K set of s (ties to the lower expert index), written to
 * topk_idx[t, 0..K-1] in descending score order; tau[t] = the (K+1)st
 * largest s (fp32).  loads[l, e] += number of tokens of microbatch l whose
 * top-K set contains e.
 *
 * hist_hi (nullable): when given, also accumulates Algorithm 1's coarse
 * histogram: for every (t, e), the margin m = bf16_rne(tau_t - fp32(z_{t,e}))
 * is encoded by the order-preserving key kappa(m) (bf16 pattern x ->
 * x & 0x8000 ? ~x : x | 0x8000, 16 bits) and hist_hi[e, kappa(m) >> 8] += 1.
 *
 *   z         device bf16 [T,E], 16-byte aligned          (in)
 *   b         device fp32 [E]                              (in)
 *   mb_offsets device int64 [M+1] (nullable iff loads is NULL)
 *   topk_idx  device int32 [T,K]   (nullable)              (out)
 *   tau       device fp32 [T]                              (out)
 *   loads     device int32 [M,E] += (nullable)             (in/out)
 *   hist_hi   device int32 [E,256] += (nullable)           (in/out)
 *   err_flag  device int32 (nullable): EQB_ERR_NONFINITE for a non-finite
 *             b_e or NaN score, or (with hist_hi) a non-finite margin.
 *
 * With hist_hi the coarse pass runs as a second kernel over z (on GB300 the
 * two kernels are faster than the one-read eqb_route_hist_fused).
 */
eqb_status eqb_route_topk(const eqb_bf16 *z, const float *b, int64_t T, int32_t E,
                          int32_t K, const int64_t *mb_offsets, int32_t M,
                          int32_t *topk_idx, float *tau, int32_t *loads,
                          int32_t *hist_hi, int32_t *err_flag, void *stream);

/* Routing and the coarse pass in one pass over z (Sec. 2 Eq. 1 and the QB
 * paragraph; Algorithm 1 step 1): the results of eqb_route_topk with hist_hi,
 * from one kernel that routes each 32-token tile staged in shared memory and
 * then counts the same staged tile, so z is read from DRAM once instead of
 * twice.  E = 128 or 256 and K + 1 <= 16, else EQB_ERR_UNSUPPORTED.
 * Arguments as in eqb_route_topk; hist_hi is required.  Bit-identical
 * outputs; slower than the two kernels on GB300, where both are bound by
 * instruction issue rather than by DRAM. */
eqb_status eqb_route_hist_fused(const eqb_bf16 *z, const float *b, int64_t T, int32_t E,
                                int32_t K, const int64_t *mb_offsets, int32_t M,
                                int32_t *topk_idx, float *tau, int32_t *loads,
                                int32_t *hist_hi, int32_t *err_flag, void *stream);

/* Coarse pass on its own (Algorithm 1 step 1): recomputes the margins from z
 * and tau and accumulates hist_hi[e, kappa(m) >> 8] += 1 over T tokens.
 * Margins of magnitude >= 2^127 or non-finite set EQB_ERR_NONFINITE: kappa
 * gives them the high bytes 0x00 and 0xff, which the method's domain
 * (|m| < 2^127) leaves out. */
eqb_status eqb_margin_hist_pass1(const eqb_bf16 *z, const float *tau, int64_t T,
                                 int32_t E, int32_t *hist_hi, int32_t *err_flag,
                                 void *stream);

/* Fine pass (Algorithm 1 step 4; Sec. 3 "the second pass simply rescans
 * local margins whose high byte matches the selected bin"): recomputes
 * every margin from z and tau and, where kappa(m) >> 8 == u[e], accumulates
 * hist_lo[e, kappa(m) & 0xff] += 1.  No margin array is materialised.
 *   u        device uint8 [E] (from eqb_select_quantile pass 1)
 *   hist_lo  device int32 [E,256] += */
eqb_status eqb_margin_hist_pass2(const eqb_bf16 *z, const float *tau, int64_t T,
                                 int32_t E, const uint8_t *u, int32_t *hist_lo,
                                 void *stream);

/* Selection on a summed histogram (Algorithm 1 steps 3, 5 and 6).
 *   pass 1: reads hist = H [E,256]; writes u[e] = min{u : sum_{j<=u} H[e,j]
 *           >= r} and rho[e] = r - sum_{j<u_e} H[e,j].  r is the global
 *           target rank (eqb_target_rank of the whole batch).  Sets
 *           EQB_ERR_NONFINITE if a margin landed in high byte 0x00 or 0xff
 *           (magnitude >= 2^127 or non-finite) and EQB_ERR_RANK if H[e,:]
 *           sums to less than r.
 *   pass 2: reads hist = L [E,256], u and rho; writes v_e = min{v :
 *           sum_{j<=v} L[e,j] >= rho_e} and q_hat[e] = kappa^{-1}((u_e << 8)
 *           | v_e), the exact r-th smallest margin (a zero as +0).
 *   q_hat is ignored in pass 1; r is ignored in pass 2. */
eqb_status eqb_select_quantile(const int32_t *hist, int32_t E, int32_t pass,
                               int64_t r, uint8_t *u, int32_t *rho, eqb_bf16 *q_hat,
                               int32_t *err_flag, void *stream);

/* Bias update of Eq. (2): b_next[e] = (float)((double)q_hat[e] - mean) with
 * mean = (sum over e = 0..E-1 in ascending order, in fp64) / E.  The fixed
 * order makes the result bit-reproducible.  b_next is used for routing in
 * the next optimizer step. */
eqb_status eqb_bias_update(const eqb_bf16 *q_hat, int32_t E, float *b_next,
                           void *stream);

/* Load-Error Injection, Sec. 4 Eq. (LEI) with the normalisation Eq. (norm).
 * For each microbatch l with n_l tokens (empty ones are skipped):
 *   rho_e = f_{l,e} / (K n_l / E) - 1;
 *   c > 0:  xi = max_e |rho_e| / c,  sigma = tanh(xi) / xi (1 at xi = 0);
 *   c <= 0: sigma = 1 (unnormalised LEI);
 *   grad_s[t, e] += eta * sigma * rho_e for every t in the microbatch and
 *   every expert e.  rho and the product eta * sigma * rho are formed in
 *   fp64 (sigma in fp32, within a few fp32 ulps of tanh(xi) / xi), rounded
 *   to fp32, and added in fp32.
 *   grad_s  device fp32 [T,E], 16-byte aligned, updated in place
 *   loads   device int32 [M,E] (the local loads from eqb_route_topk) */
eqb_status lei_inject_grad(float *grad_s, const int32_t *loads,
                           const int64_t *mb_offsets, int32_t M, int64_t T,
                           int32_t E, int32_t K, float eta, float c, void *stream);

/* The Load-Error Injection coefficients (Sec. 4, Eqs. LEI and norm) as a
 * table: coef[l, e] = (float)(eta * sigma_l * rho_{l,e}), rho and sigma of
 * microbatch l as in lei_inject_grad, by the same arithmetic (so the same
 * bits as the coefficient lei_inject_grad adds).  An empty microbatch
 * gets a row of zeros.
 *   loads  device int32 [M,E]                          (in)
 *   coef   device fp32 [M,E], 16-byte aligned          (out) */
eqb_status lei_coefficients(const int32_t *loads, const int64_t *mb_offsets,
                            int32_t M, int32_t E, int32_t K, float eta, float c,
                            float *coef, void *stream);

/* A histogram pass of Algorithm 1 with part of Load-Error Injection streamed
 * beside it, in one kernel: pass 1 is eqb_margin_hist_pass1 (hist = hist_hi,
 * err_flag used, u ignored), pass 2 is eqb_margin_hist_pass2 (hist =
 * hist_lo, u required, err_flag ignored), and for the tokens t in
 * [lei_t0, lei_t1) every grad_s[t, e] += coef[l(t), e] in fp32, l(t) the
 * microbatch of t (Sec. 4, Eq. LEI).  The counting is issue-bound and the
 * injection DRAM-bound, so the two share the GPU better than back to back.
 * Results are bit-identical to the separate calls; the one-call step runs
 * pass 1 with the first half of the tokens and pass 2 with the rest.
 *   grad_s  device fp32 [T,E], 16-byte aligned, updated in place on [lei_t0, lei_t1)
 *   coef    device fp32 [M,E] from lei_coefficients, 16-byte aligned
 *   0 <= lei_t0 <= lei_t1 <= T, else EQB_ERR_INVALID_ARG. */
eqb_status eqb_margin_hist_lei(const eqb_bf16 *z, const float *tau, int64_t T,
                               int32_t E, int32_t pass, const uint8_t *u,
                               int32_t *hist, int32_t *err_flag, float *grad_s,
                               const float *coef, const int64_t *mb_offsets,
                               int32_t M, int64_t lei_t0, int64_t lei_t1,
                               void *stream);

/* Bytes of device workspace eqb_layer_step needs for E experts (the two
 * [E,256] histograms, two block counters, u, rho, q_hat and a 65,536-float
 * LEI coefficient table, each 256-byte aligned; 788,480 bytes for
 * E = 256). */
size_t eqb_layer_workspace_bytes(int32_t E);

/* One layer's whole routing-balance step in one call, in the paper's order:
 * routing (Sec. 2), Algorithm 1's coarse pass, selection, fine pass,
 * selection, the Eq. (2) bias update, then Load-Error Injection (Sec. 4,
 * Eqs. LEI and norm) on grad_s when grad_s is given.  Results are identical
 * to the individual calls above.  When M * E <= 65,536 the LEI coefficients
 * are formed right after routing (lei_coefficients) and the injection is
 * streamed by the two histogram passes, half of the tokens each
 * (eqb_margin_hist_lei); otherwise LEI runs last (lei_inject_grad).  Each
 * histogram pass's selection (eqb_select_quantile; after the fine pass also
 * eqb_bias_update) runs in the pass's own last block to finish counting,
 * while the other blocks are still streaming LEI.
 *   z, b, mb_offsets, M, topk_idx (nullable), tau, eta, c: as in
 *             eqb_route_topk / lei_inject_grad;
 *   mb_offsets_host host copy of mb_offsets (nullable; validated when given)
 *   r         global target rank; r <= 0 means eqb_target_rank(T, E, K)
 *   loads     device int32 [M,E], overwritten (zeroed by the call)
 *   b_next    device fp32 [E] (out): the bias for the next step
 *   grad_s    device fp32 [T,E] updated in place, or NULL (no LEI)
 *   workspace device buffer of at least eqb_layer_workspace_bytes(E) bytes,
 *             256-byte aligned, owned by the caller; its contents on return
 *             are the step's histograms and selections
 * Histograms are local to the call, so this entry point is for a single
 * process; a multi-GPU caller all-reduces between the per-pass calls. */
eqb_status eqb_layer_step(const eqb_bf16 *z, const float *b, int64_t T, int32_t E, int32_t K,
                          const int64_t *mb_offsets, const int64_t *mb_offsets_host, int32_t M,
                          int64_t r, int32_t *topk_idx, float *tau, int32_t *loads, float *b_next,
                          float *grad_s, float eta, float c, void *workspace,
                          size_t workspace_bytes, int32_t *err_flag, void *stream);

/* eqb_layer_step for callers that cannot allocate device memory (no
 * counterpart in the paper; a library convenience).  Plugins hosted by a
 * framework or server that owns all device memory through its own pool, and
 * code that must not stall on or fail at an allocation, can call this
 * instead: it takes the same inputs and outputs but no workspace, and uses a
 * scratch array compiled into the library.
 *   - The scratch is eqb_layer_workspace_bytes(256) = 788,480 bytes: the
 *     step's two histograms, block counters, u, rho, q_hat and the
 *     65,536-float LEI coefficient table, enough for E <= 256; E > 256 returns
 *     EQB_ERR_UNSUPPORTED.  Every GPU that loads the library keeps
 *     this array until the process exits.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current; make it before any
 *     stream capture.  It allocates nothing.  The address is kept for the
 *     life of the process: after cudaDeviceReset on that device it is stale,
 *     and calls must not be made there again.
 *   - All calls on a device share the array, which keeps the previous
 *     call's contents (the step zeroes the histograms before counting);
 *     calls that overlap on the GPU race on it.
 * Arguments and results are those of eqb_layer_step. */
eqb_status eqb_layer_step_noalloc(const eqb_bf16 *z, const float *b, int64_t T, int32_t E,
                                  int32_t K, const int64_t *mb_offsets,
                                  const int64_t *mb_offsets_host, int32_t M, int64_t r,
                                  int32_t *topk_idx, float *tau, int32_t *loads, float *b_next,
                                  float *grad_s, float eta, float c, int32_t *err_flag,
                                  void *stream);

/* Router logits, Sec. 2 (Eq. 1: z_t = W_r x_t):
 *   z[t, e] = bf16_rne(sum_k x[t, k] * W_r[e, k]),
 * bf16 inputs, fp32 accumulation on the tensor cores (tcgen05, accumulators
 * in tensor memory).  The accumulation order is the hardware's, so an entry
 * can differ from the exactly rounded value by one bf16 ulp plus the fp32
 * accumulation error.
 *   x        device bf16 [T, d] row-major, 16-byte aligned     (in)
 *   W_r      device bf16 [E, d] row-major, 16-byte aligned     (in)
 *   z        device bf16 [T, E] row-major, 16-byte aligned     (out)
 *   err_flag device int32 (nullable): EQB_ERR_CUDA if the kernel's pipeline
 *            stalled and it gave up waiting (no result is then valid).
 * Supported: d a positive multiple of 64, E a multiple of 16 with
 * 16 <= E <= 256, 0 <= T <= 2^31 - 2^24.  Uses all tensor memory of each SM
 * it runs on, one block per SM. */
eqb_status eqb_router_logits(const eqb_bf16 *x, const eqb_bf16 *W_r, int64_t T, int32_t d,
                             int32_t E, eqb_bf16 *z, int32_t *err_flag, void *stream);

/* GShard auxiliary-loss gradient: the comparison injection beside LEI
 * (Sec. 2, the loss alpha sum_e F_e P^G_e with F stop-gradient; App. D,
 * Eq. (gshard-grad)).  For every token t of microbatch l (n_l tokens):
 *   s_e = sigmoid(fp32(z_{t,e})),  d_t = sum_e s_e,  p_e = s_e / d_t,
 *   R_e = f_{l,e} / (K n_l) - 1/E,
 *   grad_s[t, j] += alpha / (n_l d_t) * (R_j - sum_e p_e R_e).
 * R and alpha / n_l are formed in fp64 and rounded to fp32; the rest is fp32
 * (expf, sums over the token's experts, no fused multiply-add).
 *   grad_s     device fp32 [T,E], 16-byte aligned (in/out)
 *   z          device bf16 [T,E], 16-byte aligned (in): the unbiased logits
 *   loads      device int32 [M,E] (in), mb_offsets device int64 [M+1] (in):
 *              as in lei_inject_grad
 * Supported: E a multiple of 8, E <= 1024, 0 <= T <= 2^31 - 2^24. */
eqb_status gshard_inject_grad(float *grad_s, const eqb_bf16 *z, const int32_t *loads,
                              const int64_t *mb_offsets, int32_t M, int64_t T, int32_t E,
                              int32_t K, float alpha, void *stream);

/* The two estimates of the global quantile that Sec. 2 compares EQB with.
 * Both take the margins m = bf16_rne(tau_t - fp32(z_{t,e})) of
 * eqb_margin_hist_pass1 (so tau comes from eqb_route_topk), end with the
 * Eq. (2) centering b_e = fp32(x_e - mean(x)) (fp64, mean summed in ascending
 * expert order), and use a caller-provided workspace (256-byte aligned).
 * Supported: E a multiple of 8, E <= 1024, T >= 1.
 *
 * Rank-averaged QB: every shard p (token range [offsets[p], offsets[p+1]))
 * selects its own K/E quantile exactly (the r_p-th smallest margin,
 * r_p = ceil(n_p K / E), by the same two radix passes as EQB); x_e is the
 * mean over the non-empty shards of those quantiles (fp64, summed in
 * ascending shard order).  Its workspace is
 * eqb_rank_averaged_workspace_bytes(E, P) bytes (per-shard histograms).
 *   shard_offsets_host  host int64 [P+1], 0 = first <= ... <= last = T,
 *                       1 <= P <= 65535
 *   q_shards            device bf16 [P,E] (out): row p holds shard p's
 *                       quantiles (+0 for an empty shard)
 *   err_flag            as in eqb_select_quantile
 * The result depends on how the tokens are sharded; EQB's does not. */
size_t eqb_rank_averaged_workspace_bytes(int32_t E, int32_t P);
eqb_status eqb_rank_averaged_bias(const eqb_bf16 *z, const float *tau, int64_t T, int32_t E,
                                  int32_t K, const int64_t *shard_offsets_host, int32_t P,
                                  eqb_bf16 *q_shards, float *b_out, void *workspace,
                                  size_t workspace_bytes, int32_t *err_flag, void *stream);

/* Fixed-resolution histogram: 256 equal-width bins over all tokens, margin m
 * in bin j = floor(fp32(fp32(m - lo) * fp32(1 / width))) clamped to
 * [0, 255]; x_e = lo + (j_e + 1) * width (fp64), the upper edge of the first
 * bin whose cumulative count reaches r = ceil(T K / E).  Its resolution is
 * the bin width, the limitation EQB removes.  Its workspace is
 * eqb_layer_workspace_bytes(E) bytes.
 *   lo, width   finite, width > 0
 *   estimate    device double [E] (out, nullable): x before centering */
eqb_status eqb_fixed_hist_bias(const eqb_bf16 *z, const float *tau, int64_t T, int32_t E,
                               int32_t K, float lo, float width, float *b_out, double *estimate,
                               void *workspace, size_t workspace_bytes, int32_t *err_flag,
                               void *stream);

/* Balance metric MaxVio, Sec. 5 (Metrics) and App. E (balance metrics):
 *   MaxVio(B) = max_e [ f_e(B) / fbar(B) - 1 ],   fbar(B) = K |B| / E,
 * in fp64 (fbar formed as (K * |B|) / E, then one division and one
 * subtraction).
 *   maxvio[0]  Global MaxVio: the loads summed over the M microbatches,
 *              |B| = offsets[M] - offsets[0].
 *   maxvio[1]  Local MaxVio: the plain mean, summed in ascending order, of
 *              the per-microbatch values over the non-empty microbatches (an
 *              empty one has no fbar); 0 if every microbatch is empty.
 *   loads      device int32 [M,E] (in): per-microbatch loads, as written by
 *              eqb_route_topk or eqb_layer_step
 *   mb_offsets device int64 [M+1] (in): as in eqb_route_topk
 *   maxvio     device double [2] (out), 8-byte aligned
 *   per_mb     device double [M] (out, nullable): each microbatch's MaxVio,
 *              0 for an empty one
 * The paper reports the maximum over layers and a mean over steps; a caller
 * takes those across calls.  Supported: 1 <= M <= 16384. */
eqb_status eqb_maxvio(const int32_t *loads, const int64_t *mb_offsets, int32_t M, int32_t E,
                      int32_t K, double *maxvio, double *per_mb, void *stream);

/* Router logits, routing and the coarse pass in one kernel: eqb_router_logits
 * followed by eqb_route_topk, with each token routed straight from the
 * tensor-memory accumulator of its row, so z is written once and not read
 * back for routing.  The paper computes the same steps one after the other
 * (Sec. 2, Eq. 1, then top-K of s = z + b, then Algorithm 1 step 1); fusing
 * them is a property of this library.
 *   x, W_r, z   as in eqb_router_logits; z is still written (the fine pass
 *               and LEI read it)
 *   b, K, mb_offsets, M, topk_idx, tau, loads, hist_hi, err_flag
 *               as in eqb_route_topk: topk_idx [T,K] (nullable), tau [T],
 *               loads [M,E] += (nullable; then mb_offsets may be NULL),
 *               hist_hi [E,256] += (nullable): the coarse histogram, counted
 *               in the same kernel from the rows it just stored (read back
 *               from L2) when no block of the kernel routes more than 65,535
 *               tokens (T <= 65,408 x the SM count: 511 tiles of 128 rows per
 *               block), else by the coarse pass over z after it
 * Results equal those of the calls made one after the other on the same
 * inputs, bit for bit.  err_flag: EQB_ERR_NONFINITE as in eqb_route_topk,
 * EQB_ERR_CUDA as in eqb_router_logits.
 * Supported: E in {64, 128}, 1 <= K <= 8, K < E, d a positive multiple of
 * 64, 0 <= T <= 2^31 - 2^24; other shapes return EQB_ERR_UNSUPPORTED (make
 * the two calls instead). */
eqb_status eqb_router_route(const eqb_bf16 *x, const eqb_bf16 *W_r, int64_t T, int32_t d,
                            int32_t E, int32_t K, const float *b, const int64_t *mb_offsets,
                            int32_t M, eqb_bf16 *z, int32_t *topk_idx, float *tau,
                            int32_t *loads, int32_t *hist_hi, int32_t *err_flag, void *stream);

/* The routing-balance step of one layer from the router input: the router
 * projection z = bf16(x W_r^T) (Sec. 2, Eq. 1) followed by everything
 * eqb_layer_step does.  For E in {64, 128} and K <= 8 the projection, the
 * routing and the coarse histogram run as one kernel (eqb_router_route with
 * hist_hi), and the fine pass then streams all of LEI (when M * E <=
 * 65,536); otherwise eqb_router_logits then eqb_route_topk and the schedule
 * of eqb_layer_step.  The other steps are those of
 * eqb_layer_step, and so are the arguments from b on; z is an output here
 * (device bf16 [T,E], 16-byte aligned).
 *   x, W_r, d   as in eqb_router_logits.
 * Returns EQB_ERR_UNSUPPORTED for d not a multiple of 64 or E not a
 * multiple of 16, beside eqb_layer_step's own conditions. */
eqb_status eqb_router_layer_step(const eqb_bf16 *x, const eqb_bf16 *W_r, int64_t T, int32_t d,
                                 int32_t E, int32_t K, const float *b,
                                 const int64_t *mb_offsets, const int64_t *mb_offsets_host,
                                 int32_t M, int64_t r, eqb_bf16 *z, int32_t *topk_idx,
                                 float *tau, int32_t *loads, float *b_next, float *grad_s,
                                 float eta, float c, void *workspace, size_t workspace_bytes,
                                 int32_t *err_flag, void *stream);

/* Self-test of failure detection (no GPU fault involved): every wait in the
 * library's kernels is a bounded poll of a shared-memory mbarrier, and a
 * kernel whose pipeline stalls gives up, writes EQB_ERR_CUDA to its error
 * word and returns, leaving the context usable.  This call runs one block
 * that polls, `polls` times, a barrier that nothing completes, and reports
 * the stall the same way.  The paper has no counterpart.
 *   err_flag  device int32 (out): EQB_ERR_CUDA once the wait gives up
 *   polls     1 .. 2^24 */
eqb_status eqb_selftest_stalled_wait(int32_t *err_flag, int32_t polls, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* EQB_H */
