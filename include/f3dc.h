/*
 * f3dc.h -- C-ABI of libf3dc.so, the GB300 (sm_103a) Fast3Dcache cached
 * denoising step.
 *
 * Method: Fast3Dcache (arXiv 2511.22533).  One sampler step of a
 * TRELLIS-style sparse-structure flow transformer:
 *   1. cache budget c_t from the three-phase rule and the Predictive
 *      Caching Scheduler Constraint (PCSC)           -- Sec. 4.2, Sec. 4.3,
 *                                                        Algorithm 1 step 1
 *   2. Spatiotemporal Stability Criterion (SSC) score and selection of the
 *      c_t most stable tokens                         -- Sec. 4.1-4.2 (V_i,
 *                                                        Eq. ICE, Eq. ssc,
 *                                                        Eq. normalize),
 *                                                        Algorithm 1 SSC
 *   3. the flow transformer on the active tokens only -- Sec. 4.2 (token
 *                                                        compaction), Supp.
 *                                                        Sec. F (block)
 *   4. cache merge and rectified-flow Euler update    -- Algorithm 1 step 3,
 *                                                        Sec. 3.1
 *   5. dynamic-voxel count at the anchor step         -- Sec. 4.1 Eq. 1
 *
 * Conventions for every call:
 *   - Every call returns an f3dc_status; nothing aborts or throws across the
 *     ABI.  f3dc_last_error() returns text for the last failure.
 *   - "device" pointers are CUDA device pointers on the handle's device;
 *     "host" pointers are ordinary host memory.  The library never takes
 *     ownership of caller memory.
 *   - Latent grids are token-major fp32 [B, N, C] with token index
 *     i = (d * D + h) * D + w on a cubic D^3 grid; C must be 8.
 *   - Velocities are bf16 (raw 16-bit words) [B, N, C], same token order.
 *   - Calls that take a `stream` (a cudaStream_t, NULL = legacy default
 *     stream) are asynchronous on it unless stated otherwise.
 *   - A handle is thread-compatible, not thread-safe: one thread at a time.
 *   - Argument errors are reported before any launch (F3DC_ERR_INVALID_ARG);
 *     launch / runtime errors give F3DC_ERR_CUDA; kernels that detect an
 *     inconsistency (an out-of-range index, a bounded wait that ran out)
 *     record it in a device status word read by f3dc_device_status().
 */
#ifndef F3DC_H
#define F3DC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum f3dc_status {
    F3DC_OK = 0,
    F3DC_ERR_INVALID_ARG = 1,
    F3DC_ERR_CUDA = 2,
    F3DC_ERR_OOM = 3,
    F3DC_ERR_UNSUPPORTED = 4,
    F3DC_ERR_TIMEOUT = 5,
    F3DC_ERR_NONFINITE = 6,
    F3DC_ERR_DEVICE = 7
} f3dc_status;

/* Device status word bits (f3dc_device_status). */
#define F3DC_DEV_TIMEOUT 1u     /* a bounded wait inside a kernel ran out */
#define F3DC_DEV_BAD_INDEX 2u   /* an index or count outside its range */
#define F3DC_DEV_BAD_PLAN 4u    /* selection produced a count != N - quota */

/* tau refresh readings (Sec. 4.3 Phase 2; Algorithm 1 SSC).
 * PERIOD:  at most tau-1 consecutive cached steps, then a forced full step
 *          (a full refresh every tau steps).
 * LITERAL: a forced full step once tau consecutive steps were cached. */
#define F3DC_REFRESH_PERIOD 0
#define F3DC_REFRESH_LITERAL 1

typedef struct f3dc_config {
    int32_t grid;        /* cubic latent grid side D; N = D^3 tokens (N % 32 == 0) */
    int32_t channels;    /* latent channels C; must be 8 */
    int32_t width;       /* transformer width W (multiple of 128, <= 2048) */
    int32_t blocks;      /* transformer blocks L */
    int32_t heads;       /* attention heads H; W / H must be 32 or 64 */
    int32_t mlp_ratio;   /* MLP hidden = mlp_ratio * W; must be 4 */
    int32_t cond_tokens; /* condition tokens N_c */
    int32_t cond_dim;    /* condition dim D_c (multiple of 64) */
    int32_t steps;       /* Euler steps T */
    int32_t max_batch;   /* largest B any call will use */
    int32_t gamma_up;    /* decoder sub-voxels per latent token (Sec. 4.2 gamma_up) */
    int32_t tau;         /* refresh interval tau; <= 0 disables */
    int32_t f_corr;      /* Phase-3 correction period; <= 0 disables */
    int32_t refresh_mode;/* F3DC_REFRESH_PERIOD or F3DC_REFRESH_LITERAL */
    double eta;          /* time-shift factor (Supp. Sec. D), TRELLIS default 3 */
    double rho_a;        /* anchor fraction, k_a = ceil(T rho_a) */
    double mu;           /* PCSC log-linear slope */
    double omega;        /* SSC weight of the acceleration term */
    double xi;           /* Phase-3 cached fraction */
    double rho_cfg_off;  /* Phase-3 start, k_off = ceil(T rho_cfg_off) */
    double cfg_strength; /* classifier-free guidance strength s (Supp. Sec. D): the steps
                          * whose start time t_k >= cfg_t_lo use v = v_u + s (v_c - v_u),
                          * v_u predicted for the all-zero condition on the same active
                          * tokens; 0 disables guidance.  With s > 0, max_batch <= 32
                          * (a guided step runs 2 B samples) */
    double cfg_t_lo;     /* lower end of the CFG interval [cfg_t_lo, 1]; TRELLIS 0.5 */
    int32_t ssc_accel;   /* SSC acceleration term: 0 the first difference |v(t-1) - v(t-2)|
                          * (Sec. 4.1), 1 the second difference
                          * |(v(t-1) - v(t-2)) - (v(t-2) - v(t-3))| over the ring's three slots */
    int32_t decoder;     /* grid decoder O(S) of Eq. 1 at the anchor step: 0 the linear
                          * stand-in (dec_w), 1 the convolutional stand-in (dc*_w: 3x3x3
                          * convolutions C->16 at D^3, 2x up, 16->8, 2x up, 8->1 at (4D)^3,
                          * ReLU between; needs gamma_up = 64) */
} f3dc_config;

/* Weights: one bf16 device blob in layout version 2 -- every tensor
 * row-major ([out, in] for linear layers), concatenated in this order, each
 * starting at a multiple of 64 elements (W = width, C = channels,
 * Dc = cond_dim, Wm = 4 W, G = gamma_up):
 *   in_w [W,C], in_b [W], t_w1 [W,256], t_b1 [W], t_w2 [W,W], t_b2 [W],
 *   for each block: mod_w [6W,W], mod_b [6W], qkv_w [3W,W], qkv_b [3W],
 *     qn_g [W], kn_g [W], o_w [W,W], o_b [W], ln2_g [W], ln2_b [W],
 *     cq_w [W,W], cq_b [W], ckv_w [2W,Dc], ckv_b [2W], co_w [W,W], co_b [W],
 *     fc1_w [Wm,W], fc1_b [Wm], fc2_w [W,Wm], fc2_b [W],
 *   fmod_w [2W,W], fmod_b [2W], out_w [C,W], out_b [C], dec_w [C,G],
 *   dc1_w [16, C*27], dc1_b [16], dc2_w [8, 16*27], dc2_b [8], dc3_w [1, 8*27],
 *   dc3_b [1] (the convolutional stand-in decoder, 3x3x3 taps k = 9 (dz+1) +
 *   3 (dy+1) + (dx+1) innermost).
 * f3dc_create copies what it needs into library-owned memory; the caller
 * may free the blob when f3dc_create returns. */
typedef struct f3dc_weights {
    int32_t layout_version; /* must be 2 */
    const void *blob;       /* device pointer, bf16 */
    size_t blob_elems;      /* must equal f3dc_weights_elems(cfg) */
} f3dc_weights;

typedef struct f3dc_handle f3dc_handle;

/* Fills *cfg with the TRELLIS-L-shaped defaults: 16^3 x 8 latent, W 1024,
 * 24 blocks, 16 heads, 1374 x 1024 condition, T 25, and the paper's
 * default hyperparameters (Supp. "More Ablation Study": mu -0.07, omega
 * 0.7, tau 3, xi 0.7, f_corr 3, rho_a 0.2, rho_CFG-OFF 0.75) with eta 3
 * (Supp. Sec. D) and gamma_up 64.  Host only. */
f3dc_status f3dc_config_default(f3dc_config *cfg);

/* Number of bf16 elements of a layout-v2 weight blob for cfg.  Host only;
 * returns 0 for an invalid cfg. */
size_t f3dc_weights_elems(const f3dc_config *cfg);

/* Shifted time schedule (Supp. Sec. D): t_out[k-1] = t_k for k = 1..T+1,
 * t_k = eta t_l / (1 + (eta-1) t_l), t_l = 1 - (k-1)/T, computed in fp64 and
 * rounded to fp32.  t_out: host [T+1].  Host only. */
f3dc_status f3dc_time_schedule(const f3dc_config *cfg, float *t_out);

/* Cache budget for 1-based step k (Algorithm 1 step 1 with PCSC, Sec. 4.2):
 * Phase 1 (k <= ceil(T rho_a)): 0; Phase 2: floor(N - sigma exp(mu (k -
 * k_a)) / gamma_up) clamped to [0, N]; Phase 3 (k >= ceil(T rho_cfg_off)):
 * floor(N xi), or 0 on every f_corr-th step.  If consec_inout is not NULL
 * the tau refresh rule is applied on top and *consec_inout (consecutive
 * cached steps so far, start at 0) is updated.  quota_out receives the
 * number of tokens to CACHE; phase_out (nullable) receives 1, 2 or 3.
 * sigma: dynamic voxels measured at the anchor step (Eq. 1).  Host only,
 * pure; never touches a GPU. */
f3dc_status f3dc_pcsc_quota(const f3dc_config *cfg, double sigma, int32_t k,
                            int32_t *consec_inout, int32_t *quota_out, int32_t *phase_out);

/* Creates a handle on the current CUDA device: validates cfg, copies and
 * repacks the weights, allocates every work buffer for up to max_batch
 * samples and builds the TMA descriptors.  `stream` orders the copies.
 * Synchronizes the stream before returning. */
f3dc_status f3dc_create(const f3dc_config *cfg, const f3dc_weights *w, void *stream,
                        f3dc_handle **out);

/* Frees everything the handle owns (synchronizes the device). NULL is OK. */
f3dc_status f3dc_destroy(f3dc_handle *h);

/* Text of the last error on this handle (or of the last failed
 * f3dc_create / host-only call when h is NULL).  Valid until the next call. */
const char *f3dc_last_error(const f3dc_handle *h);

/* Reads and clears the device status word (F3DC_DEV_* bits); synchronizes
 * the handle's last stream.  *status_out = 0 means no kernel reported a
 * problem. */
f3dc_status f3dc_device_status(f3dc_handle *h, uint32_t *status_out);

/* SSC selection (Sec. 4.1-4.2 Eq. ssc / Eq. normalize, Algorithm 1 SSC):
 * for each sample b, V_i = ||v_prev1_i||_2, A_i = ||v_prev1_i - v_prev2_i||_2
 * (fp32, channels summed in order, one rounding per op), per-sample min-max
 * normalisation (NaN skipped; degenerate range -> 0), C_i = omega nA + (1 -
 * omega) nV, then the quota_dev[b] lowest (C_i, i) are cached (NaN scores
 * are never cached) and the rest are active.
 *   v_prev1, v_prev2: device bf16 [B, N, C]  -- v^(k-1), v^(k-2)
 *   quota_dev:        device int32 [B], clamped to [0, N]
 *   active_idx_out:   device int32 [B, N]; sample b's active tokens in
 *                     ascending order at offset b*N (n_active_out[b] valid)
 *   n_active_out:     device int32 [B] (= N - clamp(quota))
 *   cached_mask_out:  device uint8 [B, N] (1 = cached), nullable
 * Asynchronous on `stream`. */
f3dc_status f3dc_ssc_select(f3dc_handle *h, const void *v_prev1, const void *v_prev2, int32_t B,
                            const int32_t *quota_dev, int32_t *active_idx_out,
                            int32_t *n_active_out, uint8_t *cached_mask_out, void *stream);

/* Projects the cross-attention keys / values of every block from the
 * condition tokens (step-invariant, done once per sampler run).
 *   cond: device bf16 [B, N_c, D_c].  Asynchronous on `stream`. */
f3dc_status f3dc_set_cond(f3dc_handle *h, const void *cond, int32_t B, void *stream);

/* One cached denoising step k (1-based) in place (Algorithm 1, steps 2-3):
 * SSC selection under quota_dev, the flow transformer at t_k on the active
 * tokens (condition from the last f3dc_set_cond; with cfg_strength > 0 and
 * t_k >= cfg_t_lo also for the zero condition, guided velocity), cache
 * merge, Euler update S <- S - (t_k - t_{k+1}) v_t.
 *   S_inout: device fp32 [B, N, C]
 *   v_ring:  device bf16 [3, B, N, C] velocity history; slot k % 3 receives
 *            v_t, slots (k-1) % 3 and (k-2) % 3 hold v^(k-1), v^(k-2), and
 *            slot k % 3 still holds v^(k-3) when the selection reads it
 *            (ssc_accel = 1).  Zero it before step 1 (Algorithm 1
 *            initialises v_cache to 0).
 *   quota_dev: device int32 [B] tokens to cache (apply tau beforehand).
 *   dyn_voxels_dev: nullable device int64 [B]; when given, the step also
 *            counts the dynamic voxels (Eq. 1) between the grids decoded
 *            (cfg.decoder) before and after the update and ADDS them there.
 * Asynchronous on `stream`. */
f3dc_status f3dc_step(f3dc_handle *h, int32_t k, int32_t B, float *S_inout, void *v_ring,
                      const int32_t *quota_dev, int64_t *dyn_voxels_dev, void *stream);

/* Algorithm 1 end to end for B samples: f3dc_set_cond, zeroed history, for
 * k = 1..T the three-phase budget (PCSC forecast calibrated with the
 * dynamic voxels measured at the anchor step k_a) with the tau rule, then
 * f3dc_step.
 *   S_inout: device fp32 [B, N, C]: noise in, S_0 out
 *   cond:    device bf16 [B, N_c, D_c]
 *   sigma_override: host double [B], nullable; replaces the measured sigma
 *            in the forecast (the measured value is still reported)
 *   quota_schedule: host int32 [T, B], nullable; replaces the three-phase
 *            rule (tau still applies)
 *   quota_log: host int32 [T, B], nullable; effective cache quota per step
 *   sigma_out: host double [B], nullable; measured dynamic voxels at k_a
 * Synchronizes the stream at the anchor step when the forecast needs the
 * measured sigma, and at the end when quota_log or sigma_out is given. */
f3dc_status f3dc_sample(f3dc_handle *h, float *S_inout, const void *cond, int32_t B,
                        const double *sigma_override, const int32_t *quota_schedule,
                        int32_t *quota_log, double *sigma_out, void *stream);

/* The dynamic-voxel curve of Sec. 4.1 (Eq. 1 at every step of a sampler
 * run without caching -- the curve of the paper's Fig. 2 that the PCSC
 * slope is fitted to), with the handle's decoder.
 *   S_inout: device fp32 [B, N, C]: noise in, S_0 out
 *   cond:    device bf16 [B, N_c, D_c]
 *   curve_out: host int64 [T, B]: dS_k between the grids before and after
 *            step k (1-based) at index (k - 1) B + b
 * Runs the T steps with quota 0 and synchronizes the stream at the end. */
f3dc_status f3dc_dynamic_voxel_curve(f3dc_handle *h, float *S_inout, const void *cond, int32_t B,
                                     int64_t *curve_out, void *stream);

/* Data-driven PCSC slope (Supp. "Data-driven Parameter Selection"): for each
 * of n curves ([n, T] host doubles, dS of 1-based step k at index k - 1), a
 * RANSAC line fit of ln dS_k against k over steps k_lo..k_hi (the paper uses
 * 8..18), every pair of points a hypothesis (deterministic), the most
 * inliers (|residual| <= tol in ln units; ties: smaller inlier sum of
 * squares, then the earlier pair) refitted by least squares over its
 * inliers; steps with dS_k = 0 carry no point; a curve is kept iff it has
 * >= 3 points and inliers >= min_frac of them; *mu_out = the median of the
 * kept slopes (mean of the middle two for an even count; NaN if none).
 * slopes_out, kept_out: host [n], nullable.  Host only, pure. */
f3dc_status f3dc_fit_mu(const double *curves, int32_t n, int32_t T, int32_t k_lo, int32_t k_hi, double tol,
                        double min_frac, double *mu_out, double *slopes_out, int32_t *kept_out);

/* ---------------------------------------------------------------------- */
/* Measurement support.                                                    */
/* ---------------------------------------------------------------------- */

/* Per-kernel-family totals collected while profiling is on. */
typedef struct f3dc_kernel_stats {
    char name[24];     /* kernel family, e.g. "gemm", "attn_self", "ssc_select" */
    int64_t launches;  /* launches recorded */
    double total_ms;   /* summed CUDA-event durations on the launching stream */
    double flops;      /* algorithmic floating-point work of those launches */
    double bytes;      /* algorithmic DRAM bytes of those launches */
} f3dc_kernel_stats;

/* Turns per-launch timing on (enable != 0) or off, clearing the totals.
 * While on, every kernel launch is bracketed by CUDA events on its stream
 * and each f3dc_step synchronizes its stream once at the end to read them;
 * the algorithmic work of a launch is derived from the step's active-token
 * counts (GEMM 2 M N K with M the active tokens; attention 4 W sum a_b^2 and
 * 4 W M N_c; row kernels their read + write bytes). */
f3dc_status f3dc_profile(f3dc_handle *h, int32_t enable);

/* Copies up to `capacity` family totals into out (host) and sets *count.
 * Synchronizes the handle's last stream. */
f3dc_status f3dc_profile_read(f3dc_handle *h, f3dc_kernel_stats *out, int32_t capacity, int32_t *count);

/* f3dc_sample runs each run of consecutive steps that needs no host
 * decision in between as one CUDA graph (captured on first use per batch
 * size, latent buffer and step range, replayed afterwards; every step reads
 * its quota and row plan from device memory).  enable = 0 launches every
 * kernel directly instead.  Default: enabled.  Graphs are not used while
 * profiling is on. */
f3dc_status f3dc_set_graphs(f3dc_handle *h, int32_t enable);

/* Number of kernels this handle has launched since it was created (a graph
 * replay counts every kernel it contains). */
f3dc_status f3dc_launch_count(const f3dc_handle *h, int64_t *count);

/* ---------------------------------------------------------------------- */
/* Diagnostic entry points (kernel-level parity checks).                   */
/* ---------------------------------------------------------------------- */

/* The flow transformer alone (Sec. 4.2 active-subset forward, Supp. Sec. F
 * block) at time t for given active sets, using the condition of the last
 * f3dc_set_cond.
 *   S: device fp32 [B, N, C];  active_idx: device int32 [B, N] (sample b's
 *   list at offset b*N);  n_active: device int32 [B];
 *   v_out: device fp32 [B, N, C]; row j < n_active[b] of sample b receives
 *   the velocity of token active_idx[b*N + j] (other rows untouched).
 * Asynchronous on `stream`. */
f3dc_status f3dc_forward(f3dc_handle *h, float t, int32_t B, const float *S,
                         const int32_t *active_idx, const int32_t *n_active, float *v_out,
                         void *stream);

/* Epilogues of the tensor-core GEMM. */
#define F3DC_EPI_BIAS 0   /* out bf16 = acc + bias */
#define F3DC_EPI_GELU 1   /* out bf16 = gelu_tanh(acc + bias) */
#define F3DC_EPI_RESID 2  /* out fp32 += gate * (acc + bias), gate nullable (1) */

/* out[m, n] = epi(sum_k A[m, k] B[n, k]) -- the tcgen05 GEMM of the
 * transformer (nn.Linear convention: B is [N, K] row-major).  When the output
 * tiles (128 rows x 64/128/256 columns) would leave at least half of the SMs
 * idle and K >= 2048, the K range is split over several CTAs whose fp32
 * partials go to a split-K workspace that this call allocates once per device
 * and keeps for the life of the process; results do not depend on the split
 * (partials are summed in a fixed order), and calls on one device must not
 * overlap.  A bounded wait inside the kernel that runs out (F3DC_DEV_TIMEOUT;
 * the output is then incomplete) is recorded in the device status word that
 * f3dc_gemm_status reads.
 *   A: device bf16 [M, K] row-major; B: device bf16 [N, K] row-major;
 *   bias: device bf16 [N], nullable; gate: device fp32 [N], nullable;
 *   out: device bf16 [M, N] (BIAS, GELU) or fp32 [M, N] (RESID).
 *   K % 64 == 0, N % 64 == 0; any M >= 1.  Pointers 16-byte aligned.
 * Asynchronous on `stream`. */
f3dc_status f3dc_gemm(const void *A, const void *B, const void *bias, const float *gate,
                      void *out, int32_t M, int32_t N, int32_t K, int32_t epilogue, void *stream);

/* f3dc_gemm for callers that must not allocate device memory.  The paper has
 * no counterpart: this is a library service.  Code running while a CUDA graph
 * is captured in global mode cannot call cudaMalloc, some frameworks own all
 * device memory through their own pool and forbid side allocations, and
 * latency-critical loops must not enter the driver's allocator; f3dc_gemm,
 * which allocates its split-K workspace on first use per device, serves none
 * of them.  This call makes f3dc_gemm's launch decisions (the CTA-pair kernel
 * for 256-wide tiles without a split, otherwise the single-CTA kernel with
 * the same split rule and summation order), so its output equals f3dc_gemm's
 * bit for bit, with the same arguments and errors; but it takes the split-K
 * workspace from a fixed 20 MiB array (plus 4 KiB of counters) compiled into
 * libf3dc; every GPU that loads the library holds that array until the
 * process exits.  It calls no allocation routine.
 *   - The first call on a device resolves the array's device address (with
 *     that device current); make that first call before any stream capture.
 *   - A problem whose split-K partials would exceed 20 MiB is rejected with
 *     F3DC_ERR_INVALID_ARG and a message giving both sizes; on a GB300 (152
 *     SMs) every shape fits, since a split never uses more partial tiles than
 *     the device has SMs.
 *   - All calls share the array and it keeps the previous call's contents:
 *     a call that splits K clears the arrival counters on `stream` before its
 *     launch, and calls whose executions overlap on the GPU (different
 *     streams, or different host threads without ordering) race on it.
 *   - A bounded wait that runs out is recorded like f3dc_gemm's (read it with
 *     f3dc_gemm_status).
 * Failures are described by f3dc_last_error(NULL).  Asynchronous on `stream`. */
f3dc_status f3dc_gemm_noalloc(const void *A, const void *B, const void *bias, const float *gate, void *out,
                              int32_t M, int32_t N, int32_t K, int32_t epilogue, void *stream);

/* Reads and clears the current device's status word of the standalone
 * kernel calls (f3dc_gemm, f3dc_gemm_noalloc, f3dc_attention): F3DC_DEV_*
 * bits recorded by their kernels since the last read, e.g. F3DC_DEV_TIMEOUT
 * when a bounded wait ran out and part of the output was left unwritten.
 * Synchronizes the device first.
 * The word is a static device variable of the library: this call allocates
 * nothing.  Failures are described by f3dc_last_error(NULL). */
f3dc_status f3dc_gemm_status(uint32_t *status_out);

/* ---------------------------------------------------------------------- */
/* Fault injection (tests of the failure paths).                           */
/* ---------------------------------------------------------------------- */

/* Process-wide, host-side fault injection for tests; off by default.  Nothing
 * here faults, traps or hangs a GPU.  Not thread-safe: set it while no other
 * thread calls the library.
 *   fail_alloc_at: f3dc_create's device allocation number fail_alloc_at
 *     (counted from 0 in each call) is reported as failed without being
 *     attempted, so f3dc_create frees what it holds and returns F3DC_ERR_OOM;
 *     -1 turns it off.
 *   gemm_missing_arrivals, gemm_wait_ns: the split-K arrival wait of f3dc_gemm
 *     expects this many arrivals beyond the splits that exist (arrivals no CTA
 *     makes) and gives up after gemm_wait_ns nanoseconds (0: the default 1 s);
 *     the kernel then records F3DC_DEV_TIMEOUT (read with f3dc_gemm_status),
 *     leaves the waiting tiles unwritten and returns.  0 turns it off.
 *   attn_missing_kv: 1 makes f3dc_attention's first CTA skip the load of the
 *     last key tile of its first item, so the waits on that tile run out
 *     (after 1 s); the kernel records F3DC_DEV_TIMEOUT (read with
 *     f3dc_gemm_status), leaves that CTA's items unwritten and returns.  0
 *     turns it off. */
typedef struct f3dc_fault_injection {
    int32_t fail_alloc_at;
    int32_t gemm_missing_arrivals;
    int64_t gemm_wait_ns;
    int32_t attn_missing_kv;
} f3dc_fault_injection;

/* Sets the fault injection (NULL: all off).  Host only. */
f3dc_status f3dc_set_fault_injection(const f3dc_fault_injection *fi);

/* Single-sequence multi-head attention softmax(q k^T / sqrt(dh)) v with the
 * tensor-core flash kernel.
 *   q: device bf16 [nq, ldq] (head h at columns h*dh); k, v: device bf16
 *   [nk, ldkv] likewise; out: device bf16 [nq, H*dh].  dh = 32 or 64;
 *   ldq, ldkv multiples of 8.  Asynchronous on `stream`. */
f3dc_status f3dc_attention(const void *q, int32_t ldq, const void *k, const void *v, int32_t ldkv,
                           void *out, int32_t nq, int32_t nk, int32_t heads, int32_t dh,
                           void *stream);

#ifdef __cplusplus
}
#endif
#endif /* F3DC_H */
