/*
 * wdc.h -- C ABI of libwdc.so: the WorldDynCache cached denoising rollout on
 * one NVIDIA GB300 (sm_103a).
 *
 * The method (arxiv 2608.01845, "WorldDynCache: Risk-Controlled Latent Dynamics
 * Approximation for Diffusion World Models") replaces some exact transitions
 *     z_{t-1} = Psi_t(z_t, F_theta(z_t, t, c))                       (Eq. 1)
 * of a diffusion world model's rollout by a surrogate
 *     z_hat_{t-1} = G_t(z_t, H_t)                                   (Eq. 1-5)
 * whenever a calibrated, accumulated transition risk allows it (Eq. 6-10).
 *
 * Conventions for every entry point:
 *  - Errors are reported by return code only; nothing aborts or throws across
 *    the ABI.  Argument errors are detected before any launch.  After an error
 *    wdc_last_error(ctx) holds a one-line description.
 *  - Pointers named "device" must point to memory of the context's device;
 *    latents are fp32, contiguous [C, F, H, W] (flat N = C*F*H*W elements) and
 *    16-byte aligned.  The caller owns every pointer it passes; the context
 *    owns its weights, bank latents, workspace and controller state.
 *  - Work is enqueued on the given stream (a cudaStream_t; NULL = the legacy
 *    default stream).  Calls that must return a decision to the host
 *    (wdc_surrogate_step, wdc_rollout) synchronise that stream.
 *  - Step index convention: step k = 0..T-1 maps z_k to z_{k+1}; the paper's
 *    t counts down (t = T - k).  Noise levels sigma_k = 1 - k/T (optionally
 *    time-shifted), model timestep 1000*sigma_k, phase q_k = sigma_k.
 *  - A context is not thread-safe; use one per host thread.
 */
#ifndef WDC_H
#define WDC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum wdc_status {
    WDC_OK = 0,
    WDC_ERR_INVALID_ARG = 1,   /* bad pointer, size, alignment or config        */
    WDC_ERR_CUDA = 2,          /* a CUDA runtime/driver call failed              */
    WDC_ERR_UNSUPPORTED = 3,   /* valid request this library does not implement    */
    WDC_ERR_TIMEOUT = 4,       /* a bounded device-side wait gave up             */
    WDC_ERR_NONFINITE = 5,     /* reserved: non-finite data where it is an error */
    WDC_ERR_STATE = 6,         /* call out of order for the context's state      */
    WDC_ERR_OOM = 7            /* device allocation failed                       */
} wdc_status;

enum { WDC_F32 = 0, WDC_BF16 = 1 };

#define WDC_MAX_BANK 8          /* largest supported bank capacity K           */
#define WDC_MAX_BATCH 16        /* most latents one batched forward may hold   */
#define WDC_SUMMARY_DIM 256     /* the fixed summary s(.) (section "Kernelized Nonlinear Observation") */
#define WDC_SKETCH 120          /* buckets of each latent block of s(.)        */

typedef struct wdc_ctx wdc_ctx;
typedef void* wdc_stream;       /* a cudaStream_t */

/* The denoiser F_theta: an adaLN DiT over video-latent tokens.  The paper
 * takes F_theta from the backbone (Introduction, Eq. 1); layer layout:
 *   x = [Linear(cond tokens); Linear(patchify(z)) + sinusoidal position]
 *   per block: x += g1*(Wo Attn(LN(x)(1+s1)+b1) + bo);
 *              x += g2*(W2 GELU_tanh(W1(LN(x)(1+s2)+b2) + b1') + b2')
 *   v = unpatchify(Wf(LN(x_video)(1+sf)+bf) + bf')
 * layers == 0 creates a context without a denoiser (controller and fused step
 * kernels only); then the latent shape [in_ch, frames, height, width] is
 * arbitrary. */
typedef struct wdc_dit_config {
    int layers, hidden, heads, head_dim, mlp, temb_dim, freq_dim;
    int in_ch, frames, height, width, patch;
    int cond_tokens, cond_dim;
    int dual_stream;            /* 1: separate block weights for condition tokens */
    int dtype;                  /* WDC_F32 (fp32 parity mode) or WDC_BF16          */
    int max_batch;              /* latents one batched forward may hold, counting
                                   both halves of a guided pair (0 or 1: single;
                                   at most WDC_MAX_BATCH); activation buffers
                                   are sized for it */
} wdc_dit_config;

/* Flow-matching Euler schedule: sigma_k = 1 - k/T, shifted by
 * s*sigma/(1+(s-1)*sigma) when shift != 1. */
typedef struct wdc_schedule {
    int T;
    double shift;
} wdc_schedule;

/* Constants of Eq. 3-10.  The paper defers their values to supplementary
 * material; wdc_default_cache_params() fills the readings this library uses. */
typedef struct wdc_cache_params {
    int bank_capacity;          /* FIFO capacity K of the bank, 1..WDC_MAX_BANK  */
    int min_support;            /* |N_t| needed for adequate support             */
    double sim_min, q_gap_max;  /* compatibility (Eq. 3 text)                    */
    double gamma_q, tau_in;     /* retrieval score and temperature (Eq. 3)       */
    double tau_obs;             /* observation temperature tau (Eq. 5)           */
    double alpha_min, alpha_max;/* clip of the scheduler scaling (Eq. 4)         */
    double eps, eps_nu;         /* Eq. 4/7/8 epsilon; RMS-normalisation epsilon  */
    uint32_t sketch_seed;       /* seed of the summary's sign hash               */
    double w_z, w_age, w_phase, w_cam, w_depth;   /* proxy weights (Eq. 6)       */
    double eta_init, eta_min, eta_max, beta_d;    /* calibration (Eq. 8)         */
    double a_cam, a_depth, a_phase;               /* impact weight (Eq. 9)       */
    double lambda_, tau_risk;                     /* decay and threshold (Eq. 9-10) */
    int max_age;                /* pre-decision anchor age limit (Eq. 10 text)   */
    int n_init_exact, n_final_exact;              /* mandatory-exact phases      */
    int flags;                  /* WDC_ABL_* ablation bits, WDC_OBS_RESIDUAL     */
    int period;                 /* WDC_ABL_PERIODIC: exact step every `period`   */
    double ridge;               /* WDC_ABL_LINEAR_OBS: relative ridge            */
} wdc_cache_params;

/* Ablation variants (section "Ablation Study", Tables 3 and 4), bits of
 * wdc_cache_params.flags.  The paper names them and defers their definitions
 * to supplementary material; these are this library's readings.  Any
 * combination is accepted (WDC_ABL_SECANT makes WDC_ABL_LINEAR_OBS and
 * WDC_ABL_NO_SUPPORT moot: the secant uses no retrieval or observation).
 *   PERIODIC      Eq. 10's risk test replaced by a fixed period: Surrogate iff
 *                 Available_t and age_t + 1 < period (Available_t kept).
 *   SECANT        native latent secant candidate z_hat = z_t + alpha_t
 *                 (z_a - z_a,in): the latest exact displacement scaled by
 *                 Eq. 4's alpha; its support term holds whenever the bank is
 *                 non-empty.  The context keeps that displacement (one more
 *                 latent-sized buffer, written by the exact-step pass).
 *   INSTANT_RISK  instantaneous risk: lambda = 0 in Eq. 9 (R_cand = Delta_t).
 *   NO_IMPACT     w/o impact weighting: w_t = 1 in Eq. 9.
 *   NO_CALIB      w/o counterfactual calibration: eta_d stays eta_init (d_cf
 *                 is still measured and reported).
 *   NO_SUPPORT    w/o support constraint: retrieval over the whole bank (no
 *                 compatibility filter); the support term always holds.
 *   LINEAR_OBS    linear observation: Eq. 5's softmax weights replaced by the
 *                 ridge least-squares coefficients beta of s(phi_hat) on the
 *                 records' output summaries, (G + rho I) beta = S_out s_hat,
 *                 G_ij = s_out_i . s_out_j, rho = ridge * trace(G) / n_bank;
 *                 z_hat = sum_i beta_i z_out_i.
 *   NO_COND       condition descriptors left out of the lift (Eq. 2): the
 *                 camera / depth entries of every summary are zero; the
 *                 controller (Eq. 6, 9) still uses them. */
#define WDC_ABL_PERIODIC     0x01
#define WDC_ABL_SECANT       0x02
#define WDC_ABL_INSTANT_RISK 0x04
#define WDC_ABL_NO_IMPACT    0x08
#define WDC_ABL_NO_CALIB     0x10
#define WDC_ABL_NO_SUPPORT   0x20
#define WDC_ABL_LINEAR_OBS   0x40
#define WDC_ABL_NO_COND      0x80
#define WDC_ABL_ALL          0xFF

/* Reading flag (also in wdc_cache_params.flags), not an ablation:
 *   OBS_RESIDUAL  residual reading of Eq. 5's observation: the kernel weights
 *                 blend the records' exact latent displacements instead of
 *                 their outputs, z_hat = z_t + sum_i kappa_i (z_out_i - z_in_i).
 *                 Eq. 5 as printed (the default) is a convex combination of
 *                 stored exact outputs and so cannot move the latent past the
 *                 bank; this reading can.  The context keeps one displacement
 *                 buffer per bank slot (written by the exact-step pass); like
 *                 the secant's, they are not part of wdc_state_host and
 *                 wdc_state_set clears them. */
#define WDC_OBS_RESIDUAL     0x100

/* Model condition c of one step.  tokens: [cond_tokens, cond_dim] fp32, device
 * or host memory (NULL only when layers == 0).  cam/depth: the camera/motion
 * and depth/geometry descriptors of the lift (Eq. 2); zero when missing. */
typedef struct wdc_cond {
    const float* tokens;
    double cam[4];
    double depth[4];
} wdc_cond;

/* Per-step record filled by the step calls (host memory). */
typedef struct wdc_step_info {
    int k;
    int decision;               /* 1 Surrogate, 0 Exact (Eq. 10)                 */
    int finite, supported, n_compat, n_bank, age;
    double q, alpha, p, d_hat, w, delta, R_cand, R, eta, d_cf, d_z, r;
    double kappa[WDC_MAX_BANK], pi[WDC_MAX_BANK];
} wdc_step_info;

/* One bank record's small fields (section "Local Lifted Evolution"): the
 * summaries of the lifted input and output and their increment, the phases,
 * the relative RMS increment r of the transition and its descriptors. */
typedef struct wdc_record_host {
    double s_in[WDC_SUMMARY_DIM], s_out[WDC_SUMMARY_DIM], s_dphi[WDC_SUMMARY_DIM];
    double q_in, q_out, r;
    double cam[4], depth[4];
} wdc_record_host;

/* Host view of the controller and memory state.  In wdc_state_set the
 * "derived" fields are ignored and recomputed on the device from the latents. */
typedef struct wdc_state_host {
    int n_bank;                 /* records rec[0..n_bank-1], oldest first        */
    int age;                    /* surrogate steps since the latest exact step   */
    double R, eta;              /* stored risk and calibration gain              */
    double q_a_in, q_a_out;     /* latest exact interval                         */
    double cam_a[4], depth_a[4];/* descriptors of the latest exact step          */
    wdc_record_host rec[WDC_MAX_BANK];
    /* derived (read back only) */
    double cur_sketch[WDC_SKETCH], cur_sumsq, cur_sumsq_anchor;
    double anchor_sketch[WDC_SKETCH], anchor_sumsq;
    double s_phi[WDC_SUMMARY_DIM];
    int cand_supported, cand_finite;
    double cand_p;
} wdc_state_host;

/* Parameter tensors of the denoiser (wdc_set_tensor).  Shapes, [out, in] for
 * Linear weights; D hidden, E temb_dim, M mlp, P = in_ch*patch*patch, Fd freq_dim. */
enum wdc_tensor_id {
    WDC_T_PATCH_W = 0,  /* [D, P]    */  WDC_T_PATCH_B = 1,  /* [D]   */
    WDC_T_COND_W = 2,   /* [D, Dc]   */  WDC_T_COND_B = 3,   /* [D]   */
    WDC_T_T1_W = 4,     /* [E, Fd]   */  WDC_T_T1_B = 5,     /* [E]   */
    WDC_T_T2_W = 6,     /* [E, E]    */  WDC_T_T2_B = 7,     /* [E]   */
    WDC_T_FMOD_W = 8,   /* [2D, E]   */  WDC_T_FMOD_B = 9,   /* [2D]  */
    WDC_T_FINAL_W = 10, /* [P, D]    */  WDC_T_FINAL_B = 11, /* [P]   */
    /* per (layer, stream) */
    WDC_T_MOD_W = 12,   /* [6D, E]   */  WDC_T_MOD_B = 13,   /* [6D]  */
    WDC_T_QKV_W = 14,   /* [3D, D]   */  WDC_T_QKV_B = 15,   /* [3D]  */
    WDC_T_O_W = 16,     /* [D, D]    */  WDC_T_O_B = 17,     /* [D]   */
    WDC_T_FC1_W = 18,   /* [M, D]    */  WDC_T_FC1_B = 19,   /* [M]   */
    WDC_T_FC2_W = 20,   /* [D, M]    */  WDC_T_FC2_B = 21,   /* [D]   */
    WDC_T_COUNT = 22
};

/* ------------------------------------------------------------------ lifetime */
const char* wdc_status_string(wdc_status s);
/* Fills the parameter readings used by default (see wdc_cache_params). */
wdc_status wdc_default_cache_params(wdc_cache_params* out);
/* Creates a context on CUDA device `device`: validates the configs, allocates
 * the weights (when layers > 0), the K bank latents, two candidate buffers,
 * the velocity buffer, the DiT workspace and the device controller state.
 * WDC_ERR_OOM if device memory is short. */
wdc_status wdc_create(const wdc_dit_config* cfg, const wdc_schedule* sched,
                      const wdc_cache_params* params, int device, wdc_ctx** out);
void wdc_destroy(wdc_ctx* ctx);
/* Replaces the constants of Eq. 3-10 (validated as in wdc_create).  The bank
 * capacity must stay the same (WDC_ERR_INVALID_ARG otherwise); the state is
 * kept, so call it between rollouts. */
wdc_status wdc_set_cache_params(wdc_ctx* ctx, const wdc_cache_params* params);
const char* wdc_last_error(const wdc_ctx* ctx);
size_t wdc_latent_numel(const wdc_ctx* ctx);
/* Number of kernels this context has launched so far (all streams). */
unsigned long long wdc_launch_count(const wdc_ctx* ctx);
/* Synchronises the device and returns (then clears) the bits the kernels have
 * set in the context's error word: 1 = a bounded device-side wait timed out,
 * 4 = the two CTAs of a tensor-core pair saw different tensor-memory bases,
 * 8 = a bf16 model's QKV projection produced a value of V beyond fp16's range
 * (|v| > 65504), which was saturated to +-65504 when V^T was stored for the
 * attention (NaN is kept). */
wdc_status wdc_device_errors(wdc_ctx* ctx, unsigned* bits);
/* Self-test of the bounded device-side waits (the paper has no counterpart):
 * one CTA waits on an mbarrier that nothing completes, through the same
 * bounded wait the tensor-core kernels use, with a limit of `limit_ns`
 * (1 us .. 1 s).  When the limit passes the wait gives up, sets bit 1 in the
 * context's error word and raises the CTA's abort flag, which releases the
 * CTA's other waiting thread; the kernel then returns normally.  Lets a test
 * check the timeout path and that the context stays usable afterwards,
 * without faulting or hanging the GPU.  Asynchronous on `stream`. */
wdc_status wdc_selftest_wait_timeout(wdc_ctx* ctx, unsigned long long limit_ns, wdc_stream stream);

/* ------------------------------------------------------------------ weights */
/* Copies one parameter tensor (host fp32, `count` elements, shape as listed in
 * wdc_tensor_id) into the model, converting to the model dtype (bf16:
 * round-to-nearest-even).  layer/stream are ignored for global tensors. */
wdc_status wdc_set_tensor(wdc_ctx* ctx, int tensor_id, int layer, int stream,
                          const float* host, size_t count);
/* Reads one parameter tensor back into `host` (fp32, `count` elements, the
 * wdc_set_tensor layout); bf16 values are widened exactly.  Synchronous.  Lets
 * a checker evaluate the model the device actually holds (e.g. after
 * wdc_init_weights).  WDC_ERR_INVALID_ARG on a size mismatch or bad id. */
wdc_status wdc_get_tensor(wdc_ctx* ctx, int tensor_id, int layer, int stream,
                          float* host, size_t count);
/* Initialises every matrix N(0, std^2) and every bias to 0 on the device from
 * a counter-based Philox4x32-10 stream (Salmon et al., SC'11) keyed by seed. */
wdc_status wdc_init_weights(wdc_ctx* ctx, unsigned long long seed, float std);

/* ------------------------------------------------------------------ F_theta */
/* v = F_theta(z_t, t, c) (Eq. 1): z_t device fp32 latent, t the model timestep,
 * cond_tokens device fp32 [cond_tokens, cond_dim], v device fp32 latent-shaped
 * output.  Asynchronous. */
wdc_status wdc_dit_forward(wdc_ctx* ctx, const float* z_t, float t, const float* cond_tokens,
                           float* v, wdc_stream stream);
/* Batched F_theta (the paper runs one trajectory at a time and is silent on
 * batching and on classifier-free guidance; both are serving extensions that
 * do not change what one sample computes).  B latents z_t[b] (device fp32,
 * 16-byte aligned) at the same model timestep t, each with its own condition
 * tokens cond_tokens[b] (device fp32 [cond_tokens, cond_dim]; the array may
 * be NULL when the model has no condition tokens).  One forward holds all of
 * them: every GEMM and row-wise kernel runs once over all samples' tokens,
 * the attention once over all samples' heads (each sample attends to its own
 * tokens only).  Writes v[b] (device fp32, 16-byte aligned, latent-shaped).
 *   cfg == 0: v[b] = F(z_t[b], t, c_b); needs B <= max_batch.
 *   cfg == 1: guided velocity v[b] = F(z, t, 0) + guidance (F(z, t, c_b) -
 *             F(z, t, 0)), where 0 is the all-zero token set (the null
 *             condition); the 2B forwards share one batch, so 2B <= max_batch.
 * A sample's velocity is bitwise the same as that of wdc_dit_forward on it
 * alone.  Host arrays z_t, cond_tokens and v hold B pointers each.  Errors:
 * WDC_ERR_INVALID_ARG for B < 1, B (2B) > max_batch or a null / unaligned
 * pointer.  Asynchronous. */
wdc_status wdc_dit_forward_batch(wdc_ctx* ctx, int B, const float* const* z_t, float t,
                                 const float* const* cond_tokens, int cfg, float guidance,
                                 float* const* v, wdc_stream stream);
/* One DiT block in place on the token sequence x (device, model dtype,
 * [cond_tokens + video_tokens, hidden]) with modulation mod6 (device fp32,
 * [streams][6][hidden] = shift1, scale1, gate1, shift2, scale2, gate2). */
wdc_status wdc_dit_block_forward(wdc_ctx* ctx, int layer, void* x, const float* mod6,
                                 wdc_stream stream);
/* Timestep conditioning: writes [layers][streams][6][hidden] block modulations
 * followed by the final layer's [2][hidden] into mod_out (device fp32). */
wdc_status wdc_dit_modulation(wdc_ctx* ctx, float t, float* mod_out, wdc_stream stream);

/* The schedule's T + 1 noise levels sigma_0..sigma_T (fp64, as the context
 * computes them: sigma_k = 1 - k/T, time-shifted when shift != 1) into the
 * host array out[T + 1].  Step k runs the denoiser at model timestep
 * (float)(1000 sigma_k) and its phase is q_k = sigma_k (section
 * "Condition-Aware Lifted State": the normalised timestep stands in for the
 * scheduler phase). */
wdc_status wdc_schedule_sigmas(const wdc_ctx* ctx, double* out);

/* ------------------------------------------------------------------ diagnostics
 * Device reductions for the synthetic diagnostics of section "Motivation and
 * Observations" (Fig. 2) and section "Transition Risk Controller" (Fig. 3a):
 * for latents a, b and c (device fp32, N elements each, 16-byte aligned; c may
 * be NULL, read as zero) writes to the host array out[5]
 *   out[0] = sum (a - c)^2,  out[1] = sum (b - c)^2,  out[2] = sum (a - c)(b - c),
 *   out[3] = sum (a - b)^2,  out[4] = sum b^2
 * (fp32 arithmetic, deterministic fixed-order reductions), from which the
 * downstream impact ||a - b|| / ||b|| and the direction error between the
 * increments a - c and b - c follow.  Synchronises the stream. */
wdc_status wdc_latent_pair_stats(wdc_ctx* ctx, const float* a, const float* b, const float* c, double* out,
                                 wdc_stream stream);
/* Pearson and Spearman (average ranks) correlations of two host samples x, y
 * of n >= 2 values (Fig. 3a: predicted versus counterfactual defect); NaN
 * when a sample is constant.  Host code, no context or device needed. */
wdc_status wdc_correlations(const double* x, const double* y, int n, double* pearson, double* spearman);

/* ------------------------------------------------------------------ Psi_t */
/* z_next = Psi_k(z_t, v) = z_t + (sigma_{k+1} - sigma_k) v (Eq. 1, flow-matching
 * Euler), elementwise fp32 (one fused multiply-add).  z_next may equal z_t. */
wdc_status wdc_scheduler_step(wdc_ctx* ctx, int k, const float* z_t, const float* v,
                              float* z_next, wdc_stream stream);

/* ------------------------------------------------------------------ cache state */
/* Starts a rollout from z_T (device): empties the bank, R = 0,
 * eta = eta_init, age = 0, anchor z_a := a copy of z_T, and computes the
 * current latent's statistics. */
wdc_status wdc_state_reset(wdc_ctx* ctx, const float* z_T, wdc_stream stream);
/* Reads the controller/memory state back (synchronises the stream). */
wdc_status wdc_state_get(wdc_ctx* ctx, wdc_state_host* out, wdc_stream stream);
/* Installs a state: the small fields from `in`, bank latents copied from
 * z_out[0..in->n_bank-1] (device), the anchor = the newest record's latent
 * (or a copy of z_cur when the bank is empty), and recomputes the derived
 * statistics from z_cur (device) and the anchor.  For tests and resume.  The
 * exact-step displacements kept for WDC_ABL_SECANT / WDC_OBS_RESIDUAL are not
 * part of this state: they are cleared to zero (those candidates equal z_t
 * until exact steps refill them). */
wdc_status wdc_state_set(wdc_ctx* ctx, const wdc_state_host* in, const float* const* z_out,
                         const float* z_cur, wdc_stream stream);

/* ------------------------------------------------------------------ steps */
/* Surrogate candidate and decision of step k (Eq. 2-6, 9, 10) in one fused,
 * HBM-bound pass: lifts the current state (its statistics are held by the
 * context), retrieves and evolves in summary space, and when supported writes
 * z_hat = sum_i kappa_i z_out_i (Eq. 5) to `z_hat` (device, N floats) while
 * reducing the statistics the next step needs; then decides.  On Surrogate the
 * state advances (R <- R_cand, age += 1) and z_hat becomes the current latent
 * (keep the buffer alive until the next step).  On Exact the caller runs
 * F_theta and wdc_risk_update.  Synchronises the stream; `info` (host) gets
 * the step record. */
wdc_status wdc_surrogate_step(wdc_ctx* ctx, int k, const wdc_cond* c, float* z_hat,
                              wdc_step_info* info, wdc_stream stream);
/* Exact branch of step k (Eq. 1, 7, 8; section "Reliability Decision"): one
 * fused pass writes z_exact = Psi_k(z_t, v) straight into the bank's FIFO slot,
 * reduces the counterfactual defect against z_cf (the candidate of the same
 * step, or NULL), calibrates eta_d when that candidate was supported and
 * finite, decays R <- lambda R and inserts the record lifted with the
 * pre-insertion anchor and history.  *z_next receives the device address of
 * z_exact (owned by the context, valid until that slot is recycled).
 * `info` may be NULL; when given, the stream is synchronised and it is
 * completed with d_cf, R, eta and r. */
wdc_status wdc_risk_update(wdc_ctx* ctx, int k, const wdc_cond* c, const float* z_t,
                           const float* v, const float* z_cf, const float** z_next,
                           wdc_step_info* info, wdc_stream stream);

/* ------------------------------------------------------------------ rollouts */
/* The cached rollout (section "Inference and Complexity"): T steps from z_T,
 * each a wdc_surrogate_step and, on Exact, wdc_dit_forward + wdc_risk_update.
 * z_T and z_out may be device or host pointers (host ones are staged through
 * the context's buffers).  conds: n_cond == 1 (used for every step) or T
 * entries; their tokens may be device or host memory (host tokens are copied
 * into a staging buffer the context keeps, grown on the first call that needs
 * more; the call allocates device memory then).  decisions (host int[T]) and trace (host wdc_step_info[T]) may be
 * NULL.  Synchronises the stream once per step. */
wdc_status wdc_rollout(wdc_ctx* ctx, const float* z_T, const wdc_cond* conds, int n_cond,
                       float* z_out, int* decisions, wdc_step_info* trace, wdc_stream stream);
/* The cached rollout of wdc_rollout with device-side control flow (the
 * paper has no counterpart; it changes where the per-step bookkeeping runs,
 * not what is computed): one CUDA graph with a WHILE node over the T steps,
 * a SWITCH node on the bank size selecting the fused skip pass, and IF nodes
 * on the decision, which the skip pass's last CTA sets on the device; so there
 * is no host synchronisation between steps.  Same decisions and latents as
 * wdc_rollout with one condition `cond` for every step.  z_T / z_out and the
 * condition tokens may be host or device memory.  The graph is built on the
 * first call (and again when the pass mode flags WDC_ABL_SECANT /
 * WDC_OBS_RESIDUAL change); the event profiler must be off.  Afterwards the
 * context's step-API state is that of the rollout's end. */
wdc_status wdc_rollout_graph(wdc_ctx* ctx, const float* z_T, const wdc_cond* cond, float* z_out,
                             int* decisions, wdc_step_info* trace, wdc_stream stream);
/* B independent cached rollouts advanced in lockstep (the paper's method per
 * sample; batching itself has no counterpart in the paper).  ctxs[b] holds
 * sample b's cache state and controller parameters; ctxs[0] also owns the
 * denoiser that every sample's exact steps run through (its max_batch must
 * cover the largest exact batch: B, or 2B with cfg), the others may be
 * created with layers == 0.  All contexts must be distinct, on one device,
 * with the same latent size and schedule.  At step k every sample's skip pass
 * runs and decides (one stream synchronisation for all), then the samples
 * that decided Exact share one batched forward (wdc_dit_forward_batch, with
 * cfg / guidance as there) and each runs its anchor pass.  z_T[b] and z_out[b]
 * may be device or host pointers; conds holds B * n_cond entries (sample-major,
 * n_cond 1 or T) whose tokens must be device pointers when the model has
 * condition tokens.  decisions (host int[B*T]) and trace (host
 * wdc_step_info[B*T]), sample-major, may be NULL.  Each sample's decisions,
 * trace and final latent equal those of wdc_rollout on that sample alone
 * (with cfg, of the guided velocity).  Argument errors are reported on
 * ctxs[0]; an error inside one sample's step pass on that sample's context. */
wdc_status wdc_rollout_batch(wdc_ctx* const* ctxs, int B, const float* const* z_T,
                             const wdc_cond* conds, int n_cond, int cfg, float guidance,
                             float* const* z_out, int* decisions, wdc_step_info* trace,
                             wdc_stream stream);
/* The uncached rollout: wdc_dit_forward + wdc_scheduler_step at every step. */
wdc_status wdc_native_rollout(wdc_ctx* ctx, const float* z_T, const wdc_cond* conds, int n_cond,
                              float* z_out, wdc_stream stream);

/* ------------------------------------------------------------------ profiling
 * Per-kernel-class timing for roofline reporting: when enabled, every launch
 * of the library is bracketed by two CUDA events recorded on its launch
 * stream.  wdc_profile_read synchronises the device and returns, per class,
 * the summed event time (ms) and the number of timed launches since the last
 * enable or read (which clears them).  Every launch of the library is on the
 * caller's stream (a dual-stream model's condition rows share their GEMM
 * launches with the video rows), so the per-class times do not overlap.
 * Disabled by default; costs two cudaEventRecord calls per launch when on.
 * Not a method step (no counterpart in the paper). */
enum wdc_kernel_class {
    WDC_K_GEMM = 0,    /* tcgen05 / SIMT GEMMs of the denoiser            */
    WDC_K_ATTN = 1,    /* attention                                      */
    WDC_K_NORM = 2,    /* LayerNorm + modulation                         */
    WDC_K_SKIP = 3,    /* fused skip pass (wdc_surrogate_step)           */
    WDC_K_ANCHOR = 4,  /* fused anchor pass (wdc_risk_update)            */
    WDC_K_OTHER = 5,   /* timestep MLP, patchify, Psi, statistics, init  */
    WDC_K_COUNT = 6
};
wdc_status wdc_profile_enable(wdc_ctx* ctx, int on);
wdc_status wdc_profile_read(wdc_ctx* ctx, double* ms, unsigned long long* launches);

/* ------------------------------------------------------------------ operators
 * The denoiser's hot kernels, exposed for parity tests and roofline timing.   */
/* C = epilogue(A W^T): A [M, K], W [N, K] (model dtype, device, row-major);
 * bias [N] fp32 or NULL; gelu != 0 applies GELU_tanh; when res != NULL
 * C = res + gate * (.) with gate [N] fp32 (NULL = 1) and res/C [M, N] in the
 * model dtype (res may equal C).  A bf16 model runs every GEMM on the tcgen05
 * kernel, which needs N % 32 == 0 and K % 8 == 0: other shapes return
 * WDC_ERR_UNSUPPORTED (the fp32 parity mode takes any shape). */
wdc_status wdc_op_gemm(wdc_ctx* ctx, const void* A, const void* W, const float* bias, void* C,
                       int M, int N, int K, int gelu, const void* res, const float* gate,
                       wdc_stream stream);
/* O = softmax(Q K^T / sqrt(d)) V per head, non-causal: q, k [heads, L, d],
 * vt [heads, d, ldv] (V transposed, row stride ldv), o [L, heads*d]; device
 * memory, 16-byte aligned.  q, k and o are in the model dtype; vt is fp32
 * for an fp32 model (ldv = L) and fp16 for a bf16 model (the QKV projection
 * stores V that way so that the PV product takes the probabilities in fp16),
 * with ldv = L rounded up to a multiple of 8 so that every V^T row starts on
 * a 16-byte boundary; the padding columns are never read.  Any L >= 1; d 64
 * or 128.  A bf16 model may split the last (head, query block) units of the
 * launch over the key range and merge them with a second kernel through a
 * workspace the context owns, so two attention calls of one context must
 * not run concurrently on different streams. */
wdc_status wdc_op_attention(wdc_ctx* ctx, const void* q, const void* k, const void* vt, void* o,
                            int heads, int L, int d, wdc_stream stream);

/* ------------------------------------------------------------------ allocation-free variant
 * wdc_observe_noalloc: the streaming half of the skip pass -- the kernelised
 * observation z_hat = sum_i kappa_i z_out_i over K latents together with the
 * statistics the next lift needs -- for callers that cannot call cudaMalloc
 * (code running under another framework's memory manager or inside a
 * pre-sized arena, processes that must not allocate device memory after set-up).
 * The paper has no counterpart: it is a deployment variant of the same kernel.
 *
 * It allocates nothing and needs no wdc_ctx.  Its scratch (per-CTA partial sums
 * and a completion counter, 256 CTAs x 248 floats + 256 bytes = 254 KB) is a
 * file-scope __device__ array that every GPU loading libwdc.so holds until the
 * process exits.  The first call on a device, with that device current, looks
 * up the array's device address (cudaGetSymbolAddress) and caches it; make that
 * first call before any stream capture.  The cached address belongs to the
 * device's primary context as it was at that first call: after a
 * cudaDeviceReset (or anything else that destroys and re-creates the primary
 * context) restart the process before calling this entry point again.  Each
 * call clears the counter on `stream` before its kernel.  All calls on a
 * device share the scratch, so
 * calls that overlap on the GPU (different streams, no ordering) race; order
 * them on one stream.
 *
 *   z_out      host array of K device pointers (fp32 latents, n elements,
 *              16-byte aligned), 1 <= K <= WDC_MAX_BANK
 *   kappa      host array of K weights (used in fp32, as the skip pass does)
 *   z_a        device fp32 latent (the anchor) for sum (z_hat - z_a)^2
 *   z_hat      device fp32 output, n elements (must not alias the inputs)
 *   stats      device output, 123 doubles: [0..119] raw signed bucket sums
 *              sum_{bucket(i)=b} sign(i) z_hat_i (the summary sketch before its
 *              sqrt(120/n) scale), [120] sum z_hat^2, [121] sum (z_hat - z_a)^2,
 *              [122] count of non-finite z_hat elements
 *   n          elements, 1 <= n < 2^31 (the sign hash indexes 32 bits)
 *   sketch_seed  seed of the sign hash (wdc_cache_params.sketch_seed)
 * Returns WDC_ERR_INVALID_ARG for sizes or pointers outside these limits,
 * WDC_ERR_CUDA if the symbol lookup or the launch fails.  Asynchronous. */
wdc_status wdc_observe_noalloc(const float* const* z_out, int K, const double* kappa, const float* z_a,
                               float* z_hat, double* stats, size_t n, uint32_t sketch_seed, wdc_stream stream);

#ifdef __cplusplus
}
#endif
#endif /* WDC_H */
