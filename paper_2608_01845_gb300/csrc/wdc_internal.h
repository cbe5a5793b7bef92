// Internal declarations shared by the libwdc translation units.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cstdint>
#include <cstddef>
#include <string>
#include <vector>

#include "../../include/wdc.h"

namespace wdc {

constexpr int kSketch = WDC_SKETCH;          // 120 buckets per latent block
constexpr int kRun = 128;                    // elements per sketch run
constexpr int kSummary = WDC_SUMMARY_DIM;    // 256
constexpr int kMaxBank = WDC_MAX_BANK;
constexpr int kOffDz = kSketch;              // offsets inside a summary vector
constexpr int kOffCam = 2 * kSketch;
constexpr int kOffDepth = kOffCam + 4;
constexpr int kOffQ = kOffDepth + 4;
constexpr int kOffH = kOffQ + 1;

// Error bits written by kernels into the context's device error word.
enum : unsigned { kErrTimeout = 1u, kErrBounds = 2u, kErrTmem = 4u, kErrVSaturated = 8u };

// ---------------------------------------------------------------- device state
// Device state is fp32 throughout.  On GB300 an fp64 operation has a
// dependent latency of about 65 cycles (fp32: 5) and a conversion between the
// two about as much, so the step kernels' scalar chains (lift, retrieval,
// controller) run in fp32; the host converts at the API boundary, and
// differences of schedule values (q_{k+1} - q_k, a record's interval) are
// formed in fp64 on the host and rounded once.

// One bank record (section "Local Lifted Evolution").
struct DevRecord {
    alignas(16) float s_in[kSummary];
    alignas(16) float s_out[kSummary];
    alignas(16) float s_dphi[kSummary];
    float n_in, n_out;            // Euclidean norms of s_in and s_out
    float q_in, q_out, dq, r;     // dq = q_out - q_in (rounded from fp64)
    float cam[4], depth[4];
};

// Per-step output mirrored to the host (widened into wdc_step_info there).
struct StepOut {
    int decision, finite, supported, n_compat;
    float q, alpha, p, d_hat, w, delta, R_cand, R, eta, d_cf, d_z, r;
    float kappa[kMaxBank], pi[kMaxBank];
};

// Schedule values of step k, from the fp64 schedule, rounded once.
struct StepScalars {
    float q_k, q_next;            // phases q_k = sigma_k, q_{k+1}
    float dq;                     // sigma_{k+1} - sigma_k (also Psi's step)
    float t_model;                // 1000 sigma_k
};

// Continuous controller/memory state (discrete state -- bank ring, age -- is
// owned by the host and passed per launch).
struct DevState {
    float R, eta;
    float q_a_in, q_a_out, q_a_dq;  // latest exact interval and its length
    float cam_a[4], depth_a[4];
    DevRecord rec[kMaxBank];                       // indexed by ring slot
    alignas(16) float cur_S[kSketch];              // raw signed bucket sums over the current latent
    float cur_sumsq, cur_sumsq_anchor;             // sum z^2, sum (z - z_a)^2
    alignas(16) float anchor_S[kSketch];
    float anchor_sumsq;
    alignas(16) float s_phi[kSummary];             // summary of the current state (this step)
    int cand_k, cand_supported, cand_finite;
    float cand_p;
    alignas(16) float cand_S[kSketch];
    float cand_sumsq, cand_sumsq_anchor;
    StepOut out;
    // discrete state of the graph rollout (device-resident mirror of the
    // host's ring head, bank size and age)
    int g_k, g_n_bank, g_head, g_age;
    float g_t_model;                   // 1000 * sigma_k for the denoiser's timestep path
};

struct ParamsDev {
    int K, min_support, max_age, n_init_exact, n_final_exact;
    unsigned seed;
    float sim_min, q_gap_max, gamma_q, tau_in, tau_obs, alpha_min, alpha_max, eps, eps_nu;
    float w_z, w_age, w_phase, w_cam, w_depth, eta_min, eta_max, beta_d;
    float a_cam, a_depth, a_phase, lam, tau_risk;    // lam = 0 under WDC_ABL_INSTANT_RISK
    int flags, period;                               // WDC_ABL_* bits; periodic placement
    float ridge;                                     // linear observation
};

enum StreamMode { kModeStats = 0, kModeSkip = 1, kModeAnchor = 2, kModeObserve = 3, kModeSecant = 4, kModeResidual = 5 };

// Launch arguments of the fused latent-pass kernels (passed by value).
struct PassArgs {
    long long n;
    int nsrc;                          // skip: records in age order (oldest first)
    const float* src[kMaxBank];        // skip: bank latents by age; anchor/stats: src[0] = z_k;
                                       // secant: src[0] = z_k, src[1] = z_a - z_a,in;
                                       // residual: the records' displacements by age
    int slot[kMaxBank];                // ring slot of each record, by age
    const float* anchor;               // z_a
    const float* zcur;                 // residual: z_k
    const float* v;                    // anchor: velocity
    const float* zcf;                  // anchor: counterfactual candidate or nullptr
    float* out;                        // skip: z_hat; anchor: z_exact (bank slot)
    float* out2;                       // anchor: z_exact - z_k (the slot's displacement) or nullptr
    int k, T, age, ins_slot;
    StepScalars sk;                    // q_k, q_{k+1}, sigma_{k+1} - sigma_k, model timestep
    float cam[4], depth[4];
    ParamsDev prm;
    DevState* st;
    float* partials;                   // [kPartials][gridDim.x] (value-major)
    unsigned* counter;
    unsigned* err;
    float kappa[kMaxBank];             // observe: caller-given weights
    double* stats_out;                 // observe: caller-given statistics output
    // graph rollout (device-side control flow)
    int graph;                         // skip tail sets the branch conditions below
    unsigned long long h_exact, h_accept;   // cudaGraphConditionalHandle values
    float* out3;                       // anchor: z_exact also into the graph's current latent
};

// ---------------------------------------------------------------- context
struct GraphRollout;

struct Ctx {
    wdc_dit_config cfg{};
    wdc_schedule sched{};
    wdc_cache_params prm{};
    int device = 0;
    int num_sms = 0;
    size_t n = 0;                      // latent numel
    std::vector<double> sigma;         // T+1 noise levels (host, fp64)
    std::vector<StepScalars> stepf;    // [T] per-step fp32 schedule values
    std::string last_error;
    unsigned long long launches = 0;

    // memory
    DevState* st = nullptr;
    float* partials = nullptr;
    unsigned* counter = nullptr;
    unsigned* err = nullptr;
    double* pstat = nullptr;           // wdc_latent_pair_stats output (5 doubles)
    StepOut* out_host = nullptr;       // pinned
    DevState* st_host = nullptr;       // pinned staging of the device state (reset / get / set)
    float* bank[kMaxBank] = {};
    float* z_init = nullptr;           // anchor before the first exact step
    float* cand[2] = {};               // rollout candidate buffers
    float* vbuf = nullptr;
    float* zstage = nullptr;           // host-pointer staging for rollouts
    float* cond_stage = nullptr;       // host condition tokens staged for rollouts (grown on demand)
    size_t cond_stage_bytes = 0;
    float* disp[kMaxBank] = {};        // secant / residual reading: z_out - z_in per bank slot
    const float* cur_latent = nullptr; // current latent of the step API (read by secant / residual)

    // host mirror of the discrete state
    int n_bank = 0, head = 0, age = 0;
    int last_surrogate_k = -1;
    int anchor_is_init = 1;

    // denoiser
    struct DiT* dit = nullptr;
    // split-key attention partials of a sample's last round (bf16 models):
    // per sample of the batch, unnormalised O rows [num_sms x 256][128] and
    // (base, row sum) pairs
    float* attn_part = nullptr;
    float* attn_ml = nullptr;
    int attn_part_samples = 0;

    // graph rollout (device-side control flow), built on first use
    GraphRollout* grollout = nullptr;

    // optional per-class event timing (wdc_profile_enable)
    bool prof = false;
    std::vector<cudaEvent_t> ev[WDC_K_COUNT];      // begin/end pairs
    size_t ev_used[WDC_K_COUNT] = {};
    unsigned long long cls_launches[WDC_K_COUNT] = {};
};

// Brackets one launch for the optional profiler and counts it.
struct LaunchScope {
    Ctx* c;
    int cls;
    cudaStream_t s;
    cudaEvent_t end = nullptr;
    LaunchScope(Ctx* c_, int cls_, cudaStream_t s_);
    ~LaunchScope();
};

// ---------------------------------------------------------------- helpers
#define WDC_CUDA_TRY(ctx, call)                                                   \
    do {                                                                          \
        cudaError_t e__ = (call);                                                 \
        if (e__ != cudaSuccess) {                                                 \
            (ctx)->last_error = std::string(#call) + ": " + cudaGetErrorString(e__); \
            return e__ == cudaErrorMemoryAllocation ? WDC_ERR_OOM : WDC_ERR_CUDA; \
        }                                                                         \
    } while (0)

wdc_status fail(Ctx* c, wdc_status s, const std::string& msg);
void fill_info(const StepOut& o, int k, int n_bank, int age, wdc_step_info* info);

// graph_rollout.cu
wdc_status graph_rollout(Ctx* c, const float* z_T, bool z_dev, const wdc_cond* cd, const float* tokens_dev,
                         float* z_out, bool out_dev, int* decisions, wdc_step_info* trace, cudaStream_t s);
void graph_rollout_destroy(Ctx* c);

// step_kernels.cu
constexpr int kPartials = 2 * kSketch + 8;     // per-block partial sums
int pass_grid(const Ctx* c);
wdc_status launch_pass(Ctx* c, int mode, const PassArgs& a, cudaStream_t s);
wdc_status launch_pass_ptr(Ctx* c, int mode, int K, const PassArgs* pa, cudaStream_t s);
ParamsDev to_dev_params(const wdc_cache_params& p);
// wdc_latent_pair_stats: five sums over three latents into out_dev (device, 5 doubles)
wdc_status launch_pair_stats(Ctx* c, const float* a, const float* b, const float* cz, double* out_dev,
                             cudaStream_t s);

// dit.cu
wdc_status dit_create(Ctx* c);
void dit_destroy(Ctx* c);
wdc_status dit_set_tensor(Ctx* c, int id, int layer, int stream, const float* host, size_t count);
wdc_status dit_get_tensor(Ctx* c, int id, int layer, int stream, float* host, size_t count);
wdc_status dit_init_weights(Ctx* c, unsigned long long seed, float std);
wdc_status dit_forward(Ctx* c, const float* z, float t, const float* cond, float* v, cudaStream_t s);
// B latents at one timestep through one batched forward; cfg doubles the
// batch with null-condition twins and writes the guided velocity.
wdc_status dit_forward_guided(Ctx* c, int B, const float* const* z, float t, const float* const* cond, int cfg,
                              float guidance, float* const* v, cudaStream_t s);
void dit_set_timestep_source(Ctx* c, const float* t_src);   // null: the t argument of dit_forward
wdc_status dit_block(Ctx* c, int layer, void* x, const float* mod6, cudaStream_t s);
wdc_status dit_modulation(Ctx* c, float t, float* mod_out, cudaStream_t s);
wdc_status op_gemm(Ctx* c, const void* A, const void* W, const float* bias, void* C, int M, int N, int K,
                   int gelu, const void* res, const float* gate, cudaStream_t s);
wdc_status op_attention(Ctx* c, const void* q, const void* k, const void* vt, void* o, int heads, int L,
                        int d, cudaStream_t s);

}  // namespace wdc
