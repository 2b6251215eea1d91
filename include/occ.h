/*
 * occ.h -- C ABI of the GB300 (sm_103a) library for the decoupled off-policy
 * correction of "Missing Old Logits in Asynchronous Agentic RL" (arXiv 2605.12070).
 *
 * The library computes, on one GPU and with hand-written CUDA kernels:
 *   - per-token log-probabilities of the sampled tokens under a policy's
 *     logits (the factors of the ratios of Eq. 1);
 *   - the decoupled PPO loss: the discrepancy ratio r_d = pi_old / mu_old is
 *     masked to a band (Eq. 4), the staleness ratio r_s = pi_theta / pi_old
 *     goes through the advantage-sign-dependent PPO clip (Eqs. 2-3), the loss
 *     is reduced to a token mean, and the gradient with respect to the logits
 *     is written in the same pass;
 *   - the revised PPO-EWMA update of the proximal parameters that stand in
 *     for missing old logits (Eq. 5, App. B), with the auto-reset of Sec. 5.2.
 *
 * Conventions shared by every entry point:
 *   - Every pointer argument is caller-owned DEVICE memory unless marked
 *     "host".  No entry point of the path allocates or frees memory (the
 *     host-buffer helpers occ_host_alloc / occ_host_free exist for that).
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = the legacy
 *     default stream).  A returned OCC_OK means the work was enqueued.
 *     Kernels launch on the current device, which must hold every device
 *     pointer of the call and the stream.
 *   - Arguments are validated on the host before anything is launched; an
 *     invalid call returns an error status, launches nothing and records a
 *     message readable with occ_last_error() (per host thread).
 *   - Data-dependent problems found on the device (a token id outside
 *     [0, V)) never trap: the token is dropped and a bit is set in
 *     occ_loss_stats.err.
 *   - Logits are row-major [T, V] with a row stride `ld` >= V elements.
 *     Rows whose start is 16-byte aligned (base address and ld * element size
 *     multiples of 16) use the vectorised kernels.  Rows off that boundary
 *     run the same kernels peeled (scalar loads up to the boundary, then
 *     16-byte loads) when every other row array of the call (old logits,
 *     dlogits) has the same element size and sits at the same byte offsets
 *     (base addresses and row strides congruent modulo 16 bytes) and
 *     V >= 128 (bf16) / 64 (f32); any other layout runs on a scalar-load
 *     kernel.  All three meet the same accuracy bounds; occ_last_kernel()
 *     names the one a call took.
 *   - Rows of the vector kernels (aligned or peeled) of
 *     occ_decoupled_loss_fwd_bwd and occ_decoupled_loss_fused (the fused call
 *     without entropy or KL outputs) keep part of each
 *     current-logits row in tensor memory: rows over 112 KB hold 128 KB there
 *     (512-thread CTAs allocating 256 columns each, two per SM), rows of 64
 *     to 112 KB hold 64 KB (256 threads, 128 columns, four per SM), rows of up
 *     to 64 KB hold 32 KB (128-thread CTAs, 64 columns, eight per SM), when
 *     the row is long enough for the blocks to lie in whole rounds of the row
 *     walk.  Such a kernel holds all 512 tensor-memory columns of the SMs it
 *     runs on until it ends (tcgen05.alloc); a kernel of another stream that
 *     allocates tensor memory on the same SM waits for it.  The results are
 *     bit for bit those of the plain kernel (OCC_OPT_FUSED_TMEM /
 *     OCC_OPT_K2_TMEM = 0).
 */
#ifndef OCC_H_
#define OCC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define OCC_VERSION 1

typedef enum {
  OCC_OK = 0,
  OCC_ERR_INVALID_ARG = 1, /* null pointer, negative size, ld < V, bad threshold, overlap */
  OCC_ERR_UNSUPPORTED = 2, /* dtype or size the library does not handle             */
  OCC_ERR_MISALIGNED = 3,  /* a scalar array not aligned to its element size         */
  OCC_ERR_CUDA = 4,        /* a CUDA runtime call or launch failed                   */
  OCC_ERR_WORKSPACE = 5    /* workspace missing or smaller than occ_loss_workspace_bytes */
} occ_status;

typedef enum { OCC_F32 = 0, OCC_BF16 = 1 } occ_dtype;

/* Bits of occ_loss_stats.err (device-detected data problems). */
#define OCC_DATA_ERR_BAD_ID 1 /* some token id was outside [0, V); those tokens were dropped */

/* Bits of the per-token flags written by occ_decoupled_loss_fwd_bwd. */
#define OCC_FLAG_IN_BAND 1 /* r_d inside [rd_lo, rd_hi]                        (Eq. 4) */
#define OCC_FLAG_CLIPPED 2 /* PPO clip rejects the token, i.e. MIS_ppo = 0      (Eq. 3) */
#define OCC_FLAG_ACTIVE 4  /* valid, in band and not clipped: carries gradient          */
#define OCC_FLAG_VALID 8   /* loss mask set and id in range                             */

/* Loss options (HOST struct, read during the call). */
typedef struct {
  double rd_lo, rd_hi;      /* inclusive band on r_d, e.g. [1/c, c] (Eq. 4); 0 <= rd_lo <= rd_hi */
  double eps_low, eps_high; /* clip interval [1 - eps_low, 1 + eps_high] on r_s (Eq. 3, App. A);
                               0 <= eps_low <= 1, eps_high >= 0                                */
  double grad_scale;        /* upstream d(objective)/d(loss); multiplies dlogits only (1 = plain) */
  int64_t denom;            /* > 0: token-mean denominator N given by the caller;
                               <= 0: N = number of valid tokens, counted on the device        */
  int32_t rd_weight;        /* 1: token weight M(r_d) r_d (Table 5, "PPO-EWMA & train_infer");
                               0: weight M(r_d) only (Table 5, "decoupled PPO & train_infer")  */
  int32_t dlogits_f32;      /* 1: write float32 dlogits even for bf16 logits                   */
  int32_t proxy;            /* source of log pi_old (Table 1 proxies, App. A):
                               OCC_PROXY_NONE: the logp_old argument (pi_old, pi_prox of Eq. 5 or
                                 pi_async computed from their own logits);
                               OCC_PROXY_LOGLINEAR: log pi_prox = alpha log mu_old +
                                 (1 - alpha) log pi_theta, per token;
                               OCC_PROXY_ARITHMETIC: pi_prox = alpha mu_old + (1 - alpha) pi_theta
                                 ("linear_prox"), per token.
                               A proxy is a constant in the gradient (not differentiated). */
  int32_t reserved;
  double alpha;             /* behaviour-policy weight of the proxy, in [0, 1]              */
} occ_loss_params;

#define OCC_PROXY_NONE 0
#define OCC_PROXY_LOGLINEAR 1
#define OCC_PROXY_ARITHMETIC 2

/* Loss results (DEVICE struct, fully written by every successful call). */
typedef struct {
  double loss_sum;   /* sum_t loss_t                                             */
  double loss;       /* loss_sum / N, 0 when N = 0 (token mean)                  */
  int64_t n_valid;   /* tokens with mask set and id in range                     */
  int64_t n_rd_out;  /* valid tokens with r_d outside the band                   */
  int64_t n_clipped; /* valid tokens rejected by the PPO clip                    */
  int64_t n_active;  /* valid, in band, not clipped; rho = n_active / n_valid    */
  int64_t denom;     /* the N that was used                                      */
  int32_t err;       /* OCC_DATA_ERR_* bits                                      */
  int32_t reserved;
} occ_loss_stats;

/* PPO-EWMA state (DEVICE struct, caller-owned; save it with theta_prox to resume). */
typedef struct {
  double w;         /* cumulative weight w^(t-1) of App. B: 0 for an empty history,
                       1/(1-beta) for the stationary (plain EWMA) regime            */
  double coef_a;    /* coefficients of the last update: theta_prox <- a theta_prox + b theta */
  double coef_b;
  int32_t streak;   /* consecutive updates whose rho was below tau               */
  int32_t n_resets; /* resets performed so far                                   */
  int32_t last_reset; /* 1 if the last update was a reset                        */
  int32_t reserved;
} occ_ewma_state;

/*
 * occ_token_logprob -- log pi(y_t) for every row of a logits matrix.
 *
 * Computes lse[t] = log sum_v exp(logits[t, v]) with a single streaming pass
 * over the vocabulary, and logp[t] = logits[t, ids[t]] - lse[t].  These are
 * the per-token factors of the ratios of Eq. 1 (used for pi_old, or for the
 * proxy pi_prox of Eq. 5 / pi_async of Table 1).
 *
 *   logits   [T, ld] row-major, dtype dt (bf16 or f32); only columns [0, V) are read
 *   T, V, ld T >= 0 rows, 1 <= V <= 2^31 - 1 columns (ids are int32; a larger
 *            V is OCC_ERR_UNSUPPORTED), row stride ld >= V (elements)
 *   ids      [T] int32 sampled token ids
 *   logp_out [T] float32 (written); NaN where ids[t] is outside [0, V)
 *   lse_out  [T] float32 or NULL
 * Accumulation is float32 per element; the row epilogue works in float-float
 * (unevaluated sums of two floats, about 48 significant bits).
 */
occ_status occ_token_logprob(const void* logits, occ_dtype dt, int64_t T, int64_t V, int64_t ld,
                             const int32_t* ids, float* logp_out, float* lse_out, void* stream);

/* Bytes of device workspace occ_decoupled_loss_fwd_bwd needs for T tokens. */
size_t occ_loss_workspace_bytes(int64_t T, int64_t V);

/*
 * occ_decoupled_loss_fwd_bwd -- the decoupled PPO loss and its logits gradient.
 *
 * For every token t (Sec. 3.2, Eqs. 1-4; Table 5 for the role of r_d):
 *   m_t      = loss_mask[t] != 0 and 0 <= ids[t] < V  (valid)
 *   logp_t   = log softmax(logits[t])[ids[t]]
 *   r_d      = exp(logp_old[t] - logp_mu[t]),   M_d = 1{rd_lo <= r_d <= rd_hi}
 *   r_s      = exp(logp_t - logp_old[t])
 *   MIS_ppo  = A_t >= 0 ? r_s <= 1 + eps_high : r_s >= 1 - eps_low
 *   w_d      = rd_weight ? r_d : 1
 *   loss_t   = -m_t M_d w_d min(r_s A_t, clip(r_s, 1 - eps_low, 1 + eps_high) A_t)
 *   loss     = sum_t loss_t / N,  N = sum_t m_t (or params->denom)
 *   dlogits[t, v] = g_t (1[v = ids[t]] - softmax(logits[t])_v),
 *   g_t      = -grad_scale m_t M_d MIS_ppo w_d r_s A_t / N
 * Threshold decisions are taken in log-ratio space in float-float arithmetic
 * (about 48 significant bits; the proxies of Table 1 are formed in float64).
 *
 *   logits     [T, ld] bf16 or f32 (dt); read once
 *   ids        [T] int32;  logp_old, logp_mu, adv: [T] float32 (logp_old may be NULL when
 *              p->proxy != OCC_PROXY_NONE: log pi_old is then built from logp_mu and logp_t)
 *   loss_mask  [T] uint8 or NULL (= all ones)
 *   p          HOST pointer to the options
 *   logp_out   [T] float32 or NULL: logp_t for valid tokens, 0 for dropped ones
 *   flags_out  [T] uint8 or NULL: OCC_FLAG_* bits (0 for dropped tokens)
 *   dlogits    [T, ld_grad] or NULL (forward only); dtype = dt, or f32 when
 *              p->dlogits_f32; may be exactly `logits` (in place, same ld and dtype)
 *              but must not overlap it otherwise.  Rows of dropped tokens are zero.
 *   stats      DEVICE occ_loss_stats, fully overwritten
 *   workspace  DEVICE scratch of at least occ_loss_workspace_bytes(T, V) bytes,
 *              16-byte aligned; contents need not be initialised
 * Tokens with m_t = 0 are not read from `logits` at all.  The result is
 * deterministic (no floating-point atomics).
 */
occ_status occ_decoupled_loss_fwd_bwd(const void* logits, occ_dtype dt, int64_t T, int64_t V,
                                      int64_t ld, const int32_t* ids, const float* logp_old,
                                      const float* logp_mu, const float* adv,
                                      const uint8_t* loss_mask, const occ_loss_params* p,
                                      float* logp_out, uint8_t* flags_out, void* dlogits,
                                      int64_t ld_grad, occ_loss_stats* stats, void* workspace,
                                      size_t ws_bytes, void* stream);

/*
 * occ_decoupled_loss_fused -- occ_token_logprob on the old logits and
 * occ_decoupled_loss_fwd_bwd on the current logits in one launch.
 *
 * Each token's old row (pi_old, or the proxy pi_prox of Eq. 5 / pi_async of
 * Table 1) and current row are streamed by the same CTA, so log pi_old(y_t)
 * never leaves the kernel and enters the r_d / r_s decisions (Eqs. 1-4) in
 * float-float; the old row of a dropped token (mask 0 or bad id) is not read.
 * Results equal the two-call sequence up to that float32 rounding of log pi_old.
 * Optionally, in the same pass and with no extra memory traffic, per-token
 * diagnostics of the proximal reference's lag (Sec. 5.2, App. E):
 *   entropy_out[t] = H(pi_theta(.|t)) = lse - sum_v p_v z_v
 *   kl_out[t]      = KL(pi_old(.|t) || pi_theta(.|t))
 * (both 0 for dropped tokens).
 *
 *   logits_old   [T, ld_old], same dtype as logits, ld_old >= V
 *   logp_old_out [T] float32 or NULL: log pi_old(y_t) of valid tokens (0 for dropped,
 *                NaN for a bad id)
 *   entropy_out, kl_out [T] float32 or NULL
 * Every other argument is as in occ_decoupled_loss_fwd_bwd (the same workspace size);
 * dlogits must not overlap logits_old.
 */
occ_status occ_decoupled_loss_fused(const void* logits, const void* logits_old, occ_dtype dt,
                                    int64_t T, int64_t V, int64_t ld, int64_t ld_old,
                                    const int32_t* ids, const float* logp_mu, const float* adv,
                                    const uint8_t* loss_mask, const occ_loss_params* p,
                                    float* logp_out, float* logp_old_out, uint8_t* flags_out,
                                    float* entropy_out, float* kl_out, void* dlogits,
                                    int64_t ld_grad, occ_loss_stats* stats, void* workspace,
                                    size_t ws_bytes, void* stream);

/*
 * occ_decoupled_loss_fwd_bwd_noalloc -- occ_decoupled_loss_fwd_bwd without a
 * caller-supplied workspace.  (The paper has no counterpart: this is an
 * interface convenience.)
 *
 * For callers that cannot allocate device memory themselves -- for instance a
 * plain C plugin running inside a framework whose caching allocator owns all
 * of the GPU's memory, or a loop that must not call cudaMalloc/cudaFree
 * because those can synchronize the device.  Arguments, results and
 * validation are those of occ_decoupled_loss_fwd_bwd minus (workspace,
 * ws_bytes).  Neither the caller nor the library allocates anything: the
 * scratch is a fixed 4 MiB array in the library's device globals, which
 * every GPU that loads the library holds until the process exits.
 *   - T may be at most OCC_NOALLOC_MAX_TOKENS; larger batches are rejected
 *     with OCC_ERR_UNSUPPORTED before anything is launched.
 *   - The size limit is checked right after p != NULL and T >= 0, before
 *     the other arguments.
 *   - The library uses the scratch array of the CURRENT device, so that
 *     device must hold the logits and every other pointer and the stream;
 *     logits on another device are rejected with OCC_ERR_INVALID_ARG.
 *   - The first call on a device (with that device current) looks up the
 *     array's device address; make that first call before any stream capture.
 *     If the lookup fails, the call returns OCC_ERR_CUDA and the next call
 *     on that device tries again.
 *   - All calls share the one array: calls that may overlap on the GPU (other
 *     streams, other host threads) race with each other.  Serialise them.
 *     Every call writes all the scratch it later reads, so nothing left over
 *     from an earlier call affects the result.
 */
#define OCC_NOALLOC_MAX_TOKENS 786432
occ_status occ_decoupled_loss_fwd_bwd_noalloc(const void* logits, occ_dtype dt, int64_t T,
                                              int64_t V, int64_t ld, const int32_t* ids,
                                              const float* logp_old, const float* logp_mu,
                                              const float* adv, const uint8_t* loss_mask,
                                              const occ_loss_params* p, float* logp_out,
                                              uint8_t* flags_out, void* dlogits, int64_t ld_grad,
                                              occ_loss_stats* stats, void* stream);

/*
 * occ_ewma_update -- revised PPO-EWMA step on flat float32 parameters.
 *
 * App. B recursion: w <- 1 + beta w, theta_prox <- a theta_prox + b theta with
 * a = beta w_prev / w, b = 1 / w (a + b = 1; the closed form is Eq. 5).
 * Auto-reset (Sec. 5.2): when `stats` is given and has n_valid > 0, rho =
 * n_active / n_valid; a step with rho < tau extends `streak`, any other step
 * clears it; when streak reaches `min_streak` (1 = the paper's rule), or when
 * force_reset != 0, theta_prox <- theta exactly, w <- 1, streak <- 0.
 * The decision is taken on the device; the host never waits.
 *
 *   theta_prox [n] float32, updated in place;  theta [n] float32
 *   n          >= 0 elements (64-bit)
 *   beta       in [0, 1)
 *   st         DEVICE occ_ewma_state, read and updated
 *   stats      DEVICE occ_loss_stats of the latest loss step, or NULL (no auto-reset)
 *   tau        reset threshold on rho;  min_streak >= 1
 */
occ_status occ_ewma_update(float* theta_prox, const float* theta, int64_t n, double beta,
                           occ_ewma_state* st, const occ_loss_stats* stats, double tau,
                           int32_t min_streak, int32_t force_reset, void* stream);

/*
 * occ_ewma_update_bf16 -- occ_ewma_update with the proximal parameters stored
 * in bf16 (2 bytes per parameter, the footprint of the paper's host-side EWMA
 * copy, Table 3a).
 *
 * Same coefficients, reset rule and state as occ_ewma_update.  Each parameter
 * is updated in float32 from its bf16 value, v = tp + b (theta - tp), and
 * rounded back to bf16: to nearest-even when sr_seed == 0, else
 * stochastically -- 16 random bits are added below the bf16 unit in the last
 * place before truncation, so an EWMA step smaller than half a bf16 ulp is
 * kept in expectation.  Parameter i takes 16-bit lane (i mod 4), least
 * significant first, of the (i / 4)-th output of the SplitMix64 generator
 * started at sr_seed.  Pass a different seed per step.
 *
 *   theta_prox [n] bf16, updated in place;  theta [n] float32 or bf16 (theta_dt)
 */
occ_status occ_ewma_update_bf16(void* theta_prox, const void* theta, occ_dtype theta_dt,
                                int64_t n, double beta, occ_ewma_state* st,
                                const occ_loss_stats* stats, double tau, int32_t min_streak,
                                int32_t force_reset, uint64_t sr_seed, void* stream);

/*
 * occ_ewma_update_host -- the PPO-EWMA step with the proximal parameters kept
 * in PINNED HOST memory (where the paper keeps its EWMA copy, Table 3a),
 * streamed through the GPU.
 *
 * theta_prox_host (float32 or bf16, prox_dt) is copied in chunks into two
 * slots of the caller's device `staging` buffer, updated there (the
 * occ_ewma_update / occ_ewma_update_bf16 arithmetic; theta [n] is on the
 * device) and copied back, alternating stream0 and stream1 so that copies in
 * both directions overlap the updates.  The coefficient step runs once, on
 * stream0; the call's work is complete when stream0 reaches the point of the
 * call (stream1 is joined back into stream0).  A float32 buffer needs float32
 * theta.  staging_bytes sets the chunk size (two slots; at least 2 x 16 bytes
 * of elements); theta_prox_host and staging are 16-byte aligned.  Returns
 * OCC_ERR_INVALID_ARG if theta_prox_host is not page-locked.
 */
occ_status occ_ewma_update_host(void* theta_prox_host, occ_dtype prox_dt, const void* theta,
                                occ_dtype theta_dt, int64_t n, double beta, occ_ewma_state* st,
                                const occ_loss_stats* stats, double tau, int32_t min_streak,
                                int32_t force_reset, uint64_t sr_seed, void* staging,
                                size_t staging_bytes, void* stream0, void* stream1);

/* Sets a DEVICE occ_ewma_state to {w = w0, streak = 0, n_resets = 0}: w0 = 0 for an
 * empty history, 1/(1-beta) to start in the stationary regime. */
occ_status occ_ewma_state_init(occ_ewma_state* st, double w0, void* stream);

/*
 * occ_host_alloc / occ_host_free -- a PINNED HOST buffer for the inputs of an
 * end-to-end step.  This is host plumbing: the paper has no counterpart.
 *
 * occ_host_alloc maps `bytes` (rounded up to the host's transparent-huge-page
 * size; a buffer smaller than one huge page is rounded to the base page and
 * gets base pages) of anonymous memory starting on that boundary, advises the
 * kernel to back it with huge pages and page-locks it with cudaHostRegister.
 * The buffer is an ordinary page-locked buffer for cudaMemcpyAsync and for
 * occ_ewma_update_host; huge pages only cut the host link's address
 * translation when copies stream through tens of GB.  If the kernel declines
 * huge pages the buffer is backed by base pages and works the same, slower.
 * Contents are zero.  *out receives the pointer, or NULL on failure.
 * Returns OCC_ERR_INVALID_ARG for bytes == 0 or a failed mmap and
 * OCC_ERR_CUDA if the memory cannot be registered (no device, or no
 * page-lockable memory left); nothing stays mapped after a failure.
 *
 * occ_host_free unregisters and unmaps a buffer from occ_host_alloc; `bytes`
 * is the size passed to occ_host_alloc.  The caller must make sure no copy
 * from or to it is still in flight.  NULL is a no-op.
 */
occ_status occ_host_alloc(size_t bytes, void** out);
occ_status occ_host_free(void* ptr, size_t bytes);

/*
 * occ_set_option / occ_get_option -- launch-shape overrides.  (The paper has
 * no counterpart: these are measurement plumbing.)
 *
 * Every call picks its kernel's launch shape by itself; an option overrides
 * that choice for measurements (sweeps of CTA sizes, shared-memory heads and
 * loads in flight).  Every shape meets the same accuracy bounds.
 * The library reads no environment variable: an option changes only when a
 * caller sets it.  Options are process-wide and read when a call is launched;
 * set them between calls.  A value of -1 restores the automatic choice.
 * occ_set_option returns OCC_ERR_INVALID_ARG for an unknown option or a value
 * outside the listed ones; occ_get_option returns -1 for an unknown option.
 */
typedef enum {
  OCC_OPT_K1_WARP = 0,         /* 1: one warp per occ_token_logprob row; 0: CTAs      */
  OCC_OPT_K1_THREADS = 1,      /* threads per occ_token_logprob CTA: 128, 256, 512   */
  OCC_OPT_K2_THREADS = 2,      /* threads per occ_decoupled_loss_fwd_bwd CTA: 128, 256, 512 */
  OCC_OPT_K2_HEAD_BYTES = 3,   /* its shared-memory head, bytes (0 = re-read all from L2) */
  OCC_OPT_K2_UNROLL = 4,       /* vectors in flight per thread of its 512-thread kernel: 4, 6, 8 */
  OCC_OPT_FUSED_THREADS = 5,   /* threads per occ_decoupled_loss_fused CTA: 128, 256, 512 */
  OCC_OPT_FUSED_HEAD_BYTES = 6, /* its shared-memory head, bytes                       */
  OCC_OPT_FUSED_TMEM = 7,      /* 0: no tensor-memory row cache for long rows; 1: allowed */
  OCC_OPT_K2_TMEM = 8,         /* the same for occ_decoupled_loss_fwd_bwd              */
  OCC_OPT_COUNT_ = 9
} occ_option;
occ_status occ_set_option(occ_option opt, int64_t value);
int64_t occ_get_option(occ_option opt);

/* Static description of a status code. */
const char* occ_status_string(occ_status s);

/* Message of the last failed call on this host thread ("" if none). */
const char* occ_last_error(void);

/* The row kernel that the last call on this host thread launched, as a static
 * string: "k1_logprob_warp", "k1_logprob_warp/peel", "k1_logprob_vec",
 * "k1_logprob_vec/peel", "k1_logprob_scalar",
 * "k2_loss_l2", "k2_loss_l2/peel", "k2_loss_l2/tmem", "k2_loss_l2/peel/tmem",
 * "k2_loss_stream", "k2_fused_l2", "k2_fused_l2/peel", "k2_fused_l2/tmem",
 * "k2_fused_l2/peel/tmem", "k2_fused_stream", "k3_ewma_vec", "k3_ewma_scalar",
 * "k3_ewma_bf16"; "" when the call launched none (e.g. T = 0 or an invalid
 * argument).  "/peel" marks the vector kernel run on rows that start off a
 * 16-byte boundary, "/tmem" its tensor-memory tier.  Never freed; valid until
 * the next call on the thread. */
const char* occ_last_kernel(void);

/* OCC_VERSION of the built library. */
int occ_version(void);

#ifdef __cplusplus
}
#endif

#endif /* OCC_H_ */
