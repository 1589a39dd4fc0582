/*
 * specdiff.h - C ABI of the GB300 (sm_103a) verification step of speculative
 * diffusion sampling ("Accelerating Speculative Diffusions via Block
 * Verification").
 *
 * One verification call takes, for B independent chains, a window of L drafted
 * Gaussian transition steps in dimension d:
 *   x_draft   [B, L, d]  yhat_{k+1} .. yhat_{k+L}   drafted states
 *   mu_target [B, L, d]  m^q_{k}   .. m^q_{k+L-1}  target means  (Eq. target-distribution)
 *   mu_draft  [B, L, d]  m^p_{k}   .. m^p_{k+L-1}  draft means   (Eq. draft-distribution)
 *   sigma     [B, L]     sigma_{k} .. sigma_{k+L-1} shared std of both kernels
 * and returns, per chain, the accepted length tau-1 and the state emitted at
 * step k+tau (residual draw, bonus step or last accepted draft).
 *
 * Conventions for every entry point:
 *   - Array pointers are DEVICE pointers owned by the caller unless stated
 *     otherwise; nothing is retained after the call returns.  All arrays are
 *     dense row-major (C order) with the shapes given.
 *   - Arguments are validated on the host before anything is launched; a
 *     rejected call returns a negative SDV_E* code and launches nothing.
 *   - Work is enqueued asynchronously on `stream` (a cudaStream_t; NULL = the
 *     legacy default stream).  No call allocates device memory or traps on the
 *     device, and none synchronises except sdv_sampler_run and sdv_sampler_end,
 *     which read the number of rounds back.  A launch failure returns SDV_ECUDA;
 *     sdv_last_cuda_error() then gives the cudaError_t.
 *   - Results are a pure function of (inputs, seed, options): reductions use a
 *     fixed order and no floating-point atomics.
 *   - Random numbers come from Philox4x32-10 (Salmon et al., SC'11) keyed by
 *     the 64-bit seed, with counter (chain b, index, stream id, sub):
 *       coin eta_j of chain b, step j (0-based) : (b, j, 0, 0) word 0
 *       residual uniform w of chain b          : (b, 0, 1, 0) word 0
 *       residual Gaussian G, element i         : (b, i/4, 2, 0) words -> Box-Muller pairs
 *       bonus-step Gaussian                    : (b, i/4, 3, 0)
 *     uniform(x) = (x + 1/2) 2^-32;  Box-Muller on (w0,w1) and (w2,w3).
 *   - Arithmetic is fp32 (bf16 inputs are widened exactly); outputs y_out use
 *     the input dtype.
 */
#ifndef SPECDIFF_H
#define SPECDIFF_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- return codes ---------------------------------------------------- */
#define SDV_OK            0
#define SDV_EINVAL       (-1)  /* bad size, mode, dtype, option or NULL pointer */
#define SDV_EALIGN       (-2)  /* a pointer is not aligned to its element size  */
#define SDV_ECUDA        (-3)  /* a kernel launch failed (see sdv_last_cuda_error) */
#define SDV_ENOWORKSPACE (-4)  /* workspace NULL or smaller than required       */

/* ---- enums ----------------------------------------------------------- */
#define SDV_MODE_SAMPLE 0      /* Algorithm token-verification (sample verification) */
#define SDV_MODE_BLOCK  1      /* Algorithm block-verification                     */

#define SDV_F32  0             /* float32 x / means / y_out */
#define SDV_BF16 1             /* bfloat16 x / means / y_out (fp32 arithmetic) */

#define SDV_RESIDUAL_DECOMPOSITION 0  /* Algorithm decomposition-res + u-sample */
#define SDV_RESIDUAL_REFLECTION    1  /* Algorithm reflect-res (sample verification only) */

/* per-chain status bits (status_out) */
#define SDV_STATUS_ZERO_DELTA     1u  /* |Delta_tau| = 0 at the residual: y = m^q + sigma G      */
#define SDV_STATUS_NONFINITE      2u  /* a log ratio, |Delta| or sigma in the window is not finite */
#define SDV_STATUS_USAMPLE_RANGE  4u  /* U-sampler found no bracket (U clamped)                  */

#define SDV_MAX_L 64           /* largest supported window */

typedef void *sdv_stream_t;    /* cudaStream_t */

/* Library identification and error text. */
const char *sdv_version(void);
const char *sdv_strerror(int code);
/* cudaError_t of the last SDV_ECUDA returned on this host thread (0 if none). */
int sdv_last_cuda_error(void);

/*
 * Bytes of device workspace sdv_verify / sdv_verify_ex / sdv_log_ratios /
 * sdv_verify_pipelined need for (B, L, d, dtype); 0 for invalid sizes.  The caller
 * allocates it (any 256-byte aligned device buffer, its contents arbitrary) and may
 * reuse it across calls of any sizes on one stream.
 */
size_t sdv_workspace_bytes(int B, int L, int64_t d, int dtype);

/*
 * sdv_verify - the whole verification step (log ratios, acceptance rule,
 * residual draw), Algorithms token-/block-verification, decomposition-res and
 * u-sample, in the log form of App. "Density ratio calculations":
 *   Delta_j = (m^p - m^q)/sigma, Z_j = (yhat - m^p)/sigma,
 *   ell_j = log N(Z+Delta)/N(Z) = -Z^T Delta - |Delta|^2/2.
 * sample: tau = first j with eta_j >= min{1, e^ell_j}, else L+1.
 * block:  log alpha_j = min{0, log alpha_{j-1} + ell_j};
 *         h_j = v_j/(v_j + 1 - alpha_j) (j < L), h_L = alpha_L,
 *         v_j = alpha_j Phi(log alpha_j/D_{j+1} + D_{j+1}/2) - Phi(log alpha_j/D_{j+1} - D_{j+1}/2);
 *         tau = 1 + max{j : eta_j < h_j}, the max being 0 when no coin succeeds.
 * residual (tau <= L): y = m^q_tau + sigma_tau (U e + G - e e^T G),
 *         e = Delta_tau/|Delta_tau|, U = Psi_alpha^{-1}(w), alpha = alpha_{tau-1}
 *         (1 in sample mode), Psi_alpha of Eq. u-cdf.
 * full accept (tau = L+1): y = x_draft[b, L-1].
 *
 *   x_draft, mu_target, mu_draft : [B, L, d] of `dtype`
 *   sigma          : fp32, element (b, j) at sigma[b*sigma_stride_b + j];
 *                    sigma_stride_b = 0 shares one row [L] across chains
 *   B >= 1, 1 <= L <= SDV_MAX_L, d >= 1
 *   seed           : Philox key; mode: SDV_MODE_*
 *   accepted_len   : [B] int32 out, tau - 1 in [0, L]
 *   y_out          : [B, d] out, `dtype`
 *   log_ratio_out  : [B, L] fp32 out or NULL: ell_j (0 past the window)
 *   delta_norm_out : [B, L] fp32 out or NULL: |Delta_j|
 *   status_out     : [B] uint32 out or NULL: SDV_STATUS_* bits
 *   workspace      : >= sdv_workspace_bytes(B, L, d, dtype) bytes of device memory
 * Inputs must not alias outputs.
 */
int sdv_verify(const void *x_draft, const void *mu_target, const void *mu_draft,
               const float *sigma, int64_t sigma_stride_b,
               int B, int L, int64_t d, int dtype,
               uint64_t seed, int mode,
               int32_t *accepted_len, void *y_out,
               float *log_ratio_out, float *delta_norm_out, uint32_t *status_out,
               void *workspace, size_t workspace_bytes, sdv_stream_t stream);

/*
 * sdv_verify_ex - sdv_verify plus the options the end-to-end sampler needs
 * (Algorithm full-block-verification):
 *   L_eff          : [B] int32 or NULL: window length gamma_k of each chain,
 *                    0 <= L_eff[b] <= L; steps j >= L_eff[b] are never read.
 *                    0 marks an inactive chain: accepted_len = 0, its y_out row
 *                    and status are not written.
 *   mu_target_bonus: [B, d] `dtype` or NULL: m^q_{k+gamma_k}; when given, a
 *                    full accept emits the bonus step y = m^q_bonus + sigma_bonus G_bonus
 *   sigma_bonus    : [B] fp32 (required with mu_target_bonus)
 *   residual_kind  : SDV_RESIDUAL_DECOMPOSITION or SDV_RESIDUAL_REFLECTION
 *                    (reflection needs mode == SDV_MODE_SAMPLE)
 *   omega          : temperature (App. Temperature): the acceptance rule uses
 *                    ell/omega^2, block h_j and alpha_res take the tempered
 *                    alpha; omega = 1 is the exact method
 *   chain_aux_out  : [B, 4] fp32 out or NULL: (U, log alpha_res, |Delta_tau|,
 *                    sigma_tau); NaN where not applicable
 */
int sdv_verify_ex(const void *x_draft, const void *mu_target, const void *mu_draft,
                  const float *sigma, int64_t sigma_stride_b,
                  int B, int L, int64_t d, int dtype,
                  uint64_t seed, int mode,
                  const int32_t *L_eff,
                  const void *mu_target_bonus, const float *sigma_bonus,
                  int residual_kind, float omega,
                  int32_t *accepted_len, void *y_out,
                  float *log_ratio_out, float *delta_norm_out, uint32_t *status_out,
                  float *chain_aux_out,
                  void *workspace, size_t workspace_bytes, sdv_stream_t stream);

/*
 * sdv_verify_pipelined - sdv_verify_ex for a stream of independent calls: the
 * call may start streaming its window before the previous kernel on `stream` has
 * finished, so that the latency-bound end of one call (the last chains' acceptance
 * rule, U-draw and residual) overlaps the next call's read of its window.  The
 * verification itself is the same (Algorithms token-/block-verification,
 * decomposition-res, u-sample): log ratios, accepted lengths and status equal
 * sdv_verify_ex's bit for bit; U and y agree within the library's accuracy (rows of
 * up to 4096 elements finish in a 64-thread CTA with the one-warp U-sampler).
 * Precondition (the caller's promise; nothing checks it): the window (x_draft,
 * mu_target, mu_draft, sigma, L_eff, mu_target_bonus, sigma_bonus) is not written by
 * earlier work on `stream` that may still be running: the previous kernel, and the
 * earlier calls of a run of pipelined calls (the window is read while they finish).
 * The workspace needs no preparation: its two sets of tile partials are used
 * alternately by consecutive calls, each partial stored with a tag of its call; a
 * stream overwrites a slot only after the call that wrote it has read it (else it
 * waits for the previous kernel), and the finishing kernel waits for the whole stream
 * of its call when it reads a partial without its call's tag.
 * Outputs are written only after the previous call on `stream` has written its own,
 * so consecutive calls may share output buffers.  Rows longer than 16384 elements
 * add two residual kernels, which overlap the next call's stream too.  Same
 * arguments, return codes and ownership as sdv_verify_ex; the workspace must not be
 * shared with calls on other streams.
 */
int sdv_verify_pipelined(const void *x_draft, const void *mu_target, const void *mu_draft,
                         const float *sigma, int64_t sigma_stride_b,
                         int B, int L, int64_t d, int dtype,
                         uint64_t seed, int mode,
                         const int32_t *L_eff,
                         const void *mu_target_bonus, const float *sigma_bonus,
                         int residual_kind, float omega,
                         int32_t *accepted_len, void *y_out,
                         float *log_ratio_out, float *delta_norm_out, uint32_t *status_out,
                         float *chain_aux_out,
                         void *workspace, size_t workspace_bytes, sdv_stream_t stream);

/*
 * sdv_verify_noalloc - sdv_verify without a workspace argument, for callers that
 * cannot allocate device memory.  (The paper has no counterpart; this is a
 * deployment option of this library.)  Such callers include plug-ins loaded into a
 * host program that owns every device allocation through its own allocator, and
 * real-time loops where cudaMalloc's implicit synchronisation and possible failure
 * are not allowed.  They still pass their inputs and outputs; the scratch comes from
 * a static device array of SDV_NOALLOC_SCRATCH_BYTES inside this library, which every
 * GPU that loads the library holds until the process exits.
 *   - Same arguments, semantics and results as sdv_verify.
 *   - Returns SDV_ENOWORKSPACE, launching nothing, when
 *     sdv_workspace_bytes(B, L, d, dtype) > SDV_NOALLOC_SCRATCH_BYTES.
 *   - Calls no cudaMalloc / cudaFree or any other allocating routine.
 *   - Every call looks up the array's device address (cudaGetSymbolAddress) with
 *     the caller's device current, so the address stays valid across a
 *     cudaDeviceReset.  The first call on a device may also load the library's
 *     device code there; make that first call before any stream capture on the
 *     device.
 *   - Every call on a device shares the one array, which keeps the previous call's
 *     contents: the counters that must start at zero are cleared by each call on its
 *     own stream, but calls that overlap on the GPU (other streams, other host
 *     threads, same device) race on the array.  Serialise them, e.g. on one stream.
 */
#define SDV_NOALLOC_SCRATCH_BYTES (1u << 22)
int sdv_verify_noalloc(const void *x_draft, const void *mu_target, const void *mu_draft,
                       const float *sigma, int64_t sigma_stride_b,
                       int B, int L, int64_t d, int dtype,
                       uint64_t seed, int mode,
                       int32_t *accepted_len, void *y_out,
                       float *log_ratio_out, float *delta_norm_out, uint32_t *status_out,
                       sdv_stream_t stream);

/*
 * sdv_log_ratios - only the fused reduction over d (App. "Density ratio
 * calculations"): ell_j = -Z_j^T Delta_j - |Delta_j|^2/2 and |Delta_j| for
 * every (b, j) with j < L_eff[b] (all j if L_eff is NULL; 0 elsewhere).
 * Shapes and dtype as in sdv_verify; log_ratio_out and delta_norm_out are
 * [B, L] fp32 and required.
 */
int sdv_log_ratios(const void *x_draft, const void *mu_target, const void *mu_draft,
                   const float *sigma, int64_t sigma_stride_b,
                   int B, int L, int64_t d, int dtype, const int32_t *L_eff,
                   float *log_ratio_out, float *delta_norm_out,
                   void *workspace, size_t workspace_bytes, sdv_stream_t stream);

/*
 * sdv_accept_scan - only the acceptance rule over the window
 * (Algorithms token-/block-verification and their temperature variants),
 * from given log ratios and norms:
 *   log_ratio, delta_norm : [B, L] fp32 (ell_j, |Delta_j|); L_eff as above
 *   tau_out               : [B] int32 out, tau in [1, L_eff+1] (0 if inactive)
 *   log_alpha_res_out     : [B] fp32 out or NULL, log alpha_{tau-1} (0 in sample mode)
 * Coins eta_j are drawn from `seed` exactly as in sdv_verify.
 */
int sdv_accept_scan(const float *log_ratio, const float *delta_norm,
                    int B, int L, const int32_t *L_eff, uint64_t seed, int mode, float omega,
                    int32_t *tau_out, float *log_alpha_res_out, sdv_stream_t stream);

/*
 * sdv_usample - only the residual's 1-D draw, U = Psi_alpha^{-1}(w)
 * (Proposition decomposition, Eq. u-cdf, Algorithm u-sample), for n
 * independent items:
 *   delta_norm [n] fp32 (> 0), log_alpha [n] fp32 (<= 0),
 *   w_bits [n] uint32: the 32-bit Philox word, w = (w_bits + 1/2) 2^-32,
 *   U_out [n] fp32 out, status_out [n] uint32 out or NULL.
 */
int sdv_usample(const float *delta_norm, const float *log_alpha, const uint32_t *w_bits,
                int n, float *U_out, uint32_t *status_out, sdv_stream_t stream);

/*
 * sdv_philox - raw Philox4x32-10 blocks: out[i][0..3] for counter ctr[i][0..3]
 * and key (seed lo, seed hi); ctr and out are [n][4] uint32 device arrays.
 */
int sdv_philox(const uint32_t *ctr, uint64_t seed, int n, uint32_t *out, sdv_stream_t stream);

/*
 * sdv_normals - the Gaussian noise the kernels draw: out[b][i] for chain b,
 * element i on Philox stream `stream_id` and sub-counter `sub`
 * (counter (b, i/4, stream_id, sub), Box-Muller), fp32 [B, d] out.
 */
int sdv_normals(uint64_t seed, int B, int64_t d, int stream_id, uint32_t sub,
                float *out, sdv_stream_t stream);

/*
 * sdv_special - the special functions the acceptance rule and the U-sampler build on,
 * evaluated by the kernels' own device code at n points z (fp32 device arrays):
 *   which = 0: erfcx(z) = exp(z^2) erfc(z) (the library's own approximation)
 *   which = 1: log Phi(z)
 *   which = 2: g'(z) = lambda(z) + z, lambda = phi/Phi (inverse Mills ratio)
 * (App. "Density ratio calculations": the CDF differences of h_j and Eq. u-cdf are
 * evaluated from these in log space.)  out[i] for z[i]; SDV_EINVAL for another which.
 */
int sdv_special(int which, const float *z, int n, float *out, sdv_stream_t stream);

/* ---- end-to-end sampler on an analytic Gaussian-mixture target --------------
 *
 * Model (Eq. forward-process, backward-process, target-distribution): a
 * variance-preserving forward SDE with beta(t) = beta_min + (beta_max - beta_min) t,
 * f_t = -beta/2, g_t = sqrt(beta), abar_t = exp(-int_0^t beta); data distribution
 * sum_c w_c N(mu_c, comp_var I) (means [C, d], log_weights [C], C <= SDV_MAX_COMPONENTS),
 * so q_t = sum_c w_c N(sqrt(abar_t) mu_c, (abar_t comp_var + 1 - abar_t) I) with an exact
 * score.  K generative steps, t_k = k/K, delta = 1/K, churn eps > 0:
 *   m^q_k(y) = y + delta [beta/2 y + (1 + eps^2)/2 beta s_{1-t_k}(y)],
 *   sigma_k = sqrt(delta) eps sqrt(beta), beta and s at forward time max(1 - t_k, t_floor).
 * The Free drafter (Sec. "Self-Speculative Drafter") uses the same drift with the score
 * kept from the previous round's parallel verification; the Frozen drafter
 * (Eq. frozen-draft-drift) recomputes it at each round's start state.
 * Random numbers: Y_0 from Philox stream 5 (seed), draft noise stream 4 with sub-counter =
 * draft step (round seed), plain-chain noise stream 6 with sub-counter = k (seed); round r
 * is keyed by the (r+1)-th SplitMix64 output of a stream started at `seed`.
 */
#define SDV_MAX_COMPONENTS 16
#define SDV_DRAFTER_FREE   0
#define SDV_DRAFTER_FROZEN 1

/*
 * sdv_gmm_target - the target call (the "target model" of Eq. target-distribution):
 * for n state rows `states` [n, d] fp32 at generative steps k [n] (int32, 0 <= k <= K),
 * writes m^q_k(state) to mq_out [n, d] and the score to score_out [n, d] (either may be
 * NULL, not both).
 */
int sdv_gmm_target(const float *states, const int32_t *k, int n, int64_t d,
                   const float *means, const float *log_weights, int C, float comp_var,
                   int K, float churn, float beta_min, float beta_max, float t_floor,
                   float *mq_out, float *score_out, sdv_stream_t stream);

/*
 * sdv_free_draft - the drafter: for chain b, gamma_b = L_eff[b] elementwise steps from
 * y [B, d] starting at step k[b] with the cached score `score` [B, d]:
 *   mu_draft[b, i] = m^p_{k+i}, x_draft[b, i] = yhat_{k+i+1} = m^p + sigma_{k+i} G_i,
 *   sigma[b, i] = sigma_{k+i}, for i < gamma_b (other rows untouched).  G_i: stream 4,
 * sub-counter i, key `seed`.  x_draft and mu_draft are [B, L, d]; sigma is [B, L].
 */
int sdv_free_draft(const float *y, const float *score, const int32_t *k, const int32_t *L_eff,
                   int B, int L, int64_t d, int K, float churn, float beta_min, float beta_max,
                   float t_floor, uint64_t seed, float *x_draft, float *mu_draft, float *sigma,
                   sdv_stream_t stream);

/* Bytes of device workspace sdv_sampler_run needs for (B, L, d); 0 for invalid sizes. */
size_t sdv_sampler_workspace_bytes(int B, int L, int64_t d);

/*
 * sdv_sampler_run - speculative sampling of B chains (Alg. full-block-verification with
 * the chosen drafter and verification mode) until every chain has reached step K or
 * `max_rounds` rounds have run.  One round: gamma_k = min(L, K - k) draft steps, the
 * parallel target call at yhat_k .. yhat_{k+gamma_k}, sdv_verify_ex (residual or bonus
 * step), then k <- min(k + tau, K); a window that reaches K takes no bonus step.
 * The rounds run as one CUDA graph launched on `stream`: a while node whose body is
 * one round (draft, target call, verification, update), the round counter and seed
 * held in the workspace and the loop ended on the device once no chain is active or
 * max_rounds rounds ran.  Unlike the other entry points this call synchronises (it
 * waits for the graph to read back the number of rounds), so it cannot itself be
 * captured into a graph.
 *   y_out [B, d] fp32 out: the chains' states (Y_K when finished)
 *   k_out [B], chain_rounds_out [B], tau_sum_out [B] int32 out or NULL: step reached,
 *     rounds taken part in, sum of tau over those rounds
 *   rounds_out: host int32 out, rounds run
 */
int sdv_sampler_run(int B, int L, int64_t d, const float *means, const float *log_weights, int C,
                    float comp_var, int K, float churn, float beta_min, float beta_max,
                    float t_floor, uint64_t seed, int mode, int drafter, int max_rounds,
                    float *y_out, int32_t *k_out, int32_t *chain_rounds_out,
                    int32_t *tau_sum_out, int32_t *rounds_out, void *workspace,
                    size_t workspace_bytes, sdv_stream_t stream);

/*
 * Host-driven rounds: the same sampler as sdv_sampler_run, one call per round.
 * sdv_sampler_begin draws Y_0 and makes the initial target call (the chains'
 * bookkeeping and round state live in the workspace); each sdv_sampler_round
 * enqueues one round (the same kernels, in the same order, as one iteration of
 * sdv_sampler_run's graph, so that begin + R rounds + end gives the same results
 * as sdv_sampler_run with max_rounds = R while a chain is active; a round with no
 * active chain only advances the round counter); sdv_sampler_end synchronises
 * `stream` and returns the same outputs as sdv_sampler_run.  Every round must pass
 * the arguments given to begin (and one mode and drafter throughout).  All three
 * return SDV_EINVAL / SDV_ENOWORKSPACE / SDV_EALIGN for bad arguments as
 * sdv_sampler_run does, before launching anything.
 */
int sdv_sampler_begin(int B, int L, int64_t d, const float *means, const float *log_weights, int C,
                      float comp_var, int K, float churn, float beta_min, float beta_max,
                      float t_floor, uint64_t seed, void *workspace, size_t workspace_bytes,
                      sdv_stream_t stream);
int sdv_sampler_round(int B, int L, int64_t d, const float *means, const float *log_weights, int C,
                      float comp_var, int K, float churn, float beta_min, float beta_max,
                      float t_floor, uint64_t seed, int mode, int drafter, void *workspace,
                      size_t workspace_bytes, sdv_stream_t stream);
int sdv_sampler_end(int B, int L, int64_t d, void *workspace, size_t workspace_bytes, float *y_out,
                    int32_t *k_out, int32_t *chain_rounds_out, int32_t *tau_sum_out,
                    int32_t *rounds_out, sdv_stream_t stream);

/*
 * sdv_em_sample - the plain (non-speculative) Euler-Maruyama chain, Y_{k+1} =
 * m^q_k(Y_k) + sigma_k G_k for k = 0 .. K-1 from Y_0 (stream 5), G_k from stream 6 with
 * sub-counter k; y_out [B, d] fp32 out.  K kernel launches on `stream`.
 */
int sdv_em_sample(int B, int64_t d, const float *means, const float *log_weights, int C,
                  float comp_var, int K, float churn, float beta_min, float beta_max,
                  float t_floor, uint64_t seed, float *y_out, sdv_stream_t stream);

/*
 * Profiling aid (not part of the method): when enabled, sdv_verify /
 * sdv_verify_ex calls made on this host thread record CUDA events on their
 * stream into a ring of `slots` entries (one call in `every`, see
 * sdv_timing_stride; every call by default): before the first kernel of the
 * call, after it (the fused verify kernel; with B >= 512 chains the streaming
 * kernel of the many-chain path), and after the kernels that follow it (the
 * many-chain finishing kernel, and the separate residual kernels used for rows
 * longer than 4096 elements).  Calls made by sdv_sampler_run / sdv_sampler_round
 * are not recorded.  The records are ordinary stream work, so they are captured into
 * a CUDA graph like the kernels (an event record costs a few microseconds of
 * graph time, hence the stride).  The events are created here (host objects; no
 * device memory).  slots = 0 disables timing and destroys the events.
 */
int sdv_timing_enable(int slots);

/*
 * Records events for one call in `every` (every >= 1; the default 1 records
 * every call) while timing is enabled.  SDV_EINVAL for every < 1.
 */
int sdv_timing_stride(int every);

/*
 * Waits for the events of the last `n_calls` recorded calls (1 <= n_calls <=
 * slots) and writes their summed phase times in milliseconds:
 * ms3[0] the first kernel (the fused verify kernel: log-ratio pass, acceptance,
 * U-draw and, for rows up to 4096 elements, the residual write; or, with B >= 512,
 * the many-chain streaming kernel), ms3[1] the kernels after it (the many-chain
 * finishing kernel and the long-row residual kernels; the time of the event
 * records alone when there are none), ms3[2] reserved (0).  SDV_EINVAL if timing
 * is off or fewer calls were recorded.
 */
int sdv_timing_read(int n_calls, float *ms3);

#ifdef __cplusplus
}
#endif

#endif /* SPECDIFF_H */
