// C ABI of libwdc.so (declared in include/wdc.h): context lifetime, weights,
// the controller/memory state, the two step calls and the rollouts.
//
// Host-side control flow of the cached rollout (section "Inference and
// Complexity"): per step, one fused skip pass decides on the device; the host
// reads the 1-KB step record (one stream synchronisation) and, on Exact, runs
// the denoiser and the fused anchor pass.  The host mirrors only the discrete
// state (bank ring, anchor age); every continuous quantity of Eq. 2-10 lives
// in device memory and is updated by the kernels' tails.
#include "wdc_internal.h"
#include "ptx.cuh"

#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>

using namespace wdc;

namespace wdc {
wdc_status fail(Ctx* c, wdc_status s, const std::string& msg) {
    if (c) c->last_error = msg;
    return s;
}

void fill_info(const StepOut& o, int k, int n_bank, int age, wdc_step_info* info) {
    if (!info) return;
    info->k = k;
    info->decision = o.decision;
    info->finite = o.finite;
    info->supported = o.supported;
    info->n_compat = o.n_compat;
    info->n_bank = n_bank;
    info->age = age;
    info->q = o.q; info->alpha = o.alpha; info->p = o.p; info->d_hat = o.d_hat; info->w = o.w;
    info->delta = o.delta; info->R_cand = o.R_cand; info->R = o.R; info->eta = o.eta;
    info->d_cf = o.d_cf; info->d_z = o.d_z; info->r = o.r;
    for (int i = 0; i < WDC_MAX_BANK; ++i) { info->kappa[i] = o.kappa[i]; info->pi[i] = o.pi[i]; }
}


static cudaEvent_t next_event(Ctx* c, int cls) {
    auto& v = c->ev[cls];
    if (c->ev_used[cls] == v.size()) {
        cudaEvent_t e;
        if (cudaEventCreate(&e) != cudaSuccess) { cudaGetLastError(); return nullptr; }
        v.push_back(e);
    }
    return v[c->ev_used[cls]++];
}

LaunchScope::LaunchScope(Ctx* c_, int cls_, cudaStream_t s_) : c(c_), cls(cls_), s(s_) {
    c->launches++;
    if (c->prof) {
        // reserve both events of the pair up front so begin/end never misalign
        cudaEvent_t b = next_event(c, cls);
        cudaEvent_t e = b ? next_event(c, cls) : nullptr;
        if (b && e) {
            cudaEventRecord(b, s);
            end = e;
            c->cls_launches[cls]++;
        } else if (b) {
            c->ev_used[cls]--;
        }
    }
}
LaunchScope::~LaunchScope() {
    if (end) cudaEventRecord(end, s);
}
}  // namespace wdc

namespace {

__global__ void psi_kernel(const float* __restrict__ z, const float* __restrict__ v, float* __restrict__ out,
                           long long n, float dsig) {
    const long long i4 = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const long long base = i4 * 4;
    if (base + 3 < n) {
        const float4 a = *reinterpret_cast<const float4*>(z + base);
        const float4 b = *reinterpret_cast<const float4*>(v + base);
        float4 r;
        r.x = fmaf(dsig, b.x, a.x); r.y = fmaf(dsig, b.y, a.y);
        r.z = fmaf(dsig, b.z, a.z); r.w = fmaf(dsig, b.w, a.w);
        *reinterpret_cast<float4*>(out + base) = r;
    } else {
        for (long long i = base; i < n; ++i) out[i] = fmaf(dsig, v[i], z[i]);
    }
}

// Bounded-wait self-test: an mbarrier that nothing completes (see
// wdc_selftest_wait_timeout).  Thread 0 gives up after limit_ns; thread 32
// is released by the abort flag that thread 0 raises.
__global__ void wait_probe_kernel(unsigned* err, unsigned long long limit_ns) {
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        abort_flag = 0;
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) mbar_wait(&bar, 0, &abort_flag, err, limit_ns);
    if (threadIdx.x == 32) mbar_wait(&bar, 0, &abort_flag, err, 2 * limit_ns + 1000000ull);
    __syncthreads();
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

bool is_device_ptr(const void* p) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

wdc_status check_cfg(Ctx* c, const wdc_dit_config& g) {
    if (g.in_ch <= 0 || g.frames <= 0 || g.height <= 0 || g.width <= 0)
        return fail(c, WDC_ERR_INVALID_ARG, "latent shape must be positive");
    if (g.layers < 0) return fail(c, WDC_ERR_INVALID_ARG, "layers must be >= 0");
    if (g.max_batch < 0 || g.max_batch > WDC_MAX_BATCH) return fail(c, WDC_ERR_INVALID_ARG, "max_batch must be 0..16");
    if (g.layers == 0) return WDC_OK;
    if (g.dtype != WDC_F32 && g.dtype != WDC_BF16) return fail(c, WDC_ERR_INVALID_ARG, "dtype must be WDC_F32 or WDC_BF16");
    if (g.head_dim != 64 && g.head_dim != 128) return fail(c, WDC_ERR_UNSUPPORTED, "head_dim must be 64 or 128");
    if (g.heads <= 0 || g.hidden != g.heads * g.head_dim) return fail(c, WDC_ERR_INVALID_ARG, "hidden != heads*head_dim");
    if (g.patch <= 0 || g.height % g.patch || g.width % g.patch) return fail(c, WDC_ERR_INVALID_ARG, "patch must divide height and width");
    if (g.in_ch * g.patch * g.patch > 1024) return fail(c, WDC_ERR_UNSUPPORTED, "patch feature size > 1024");
    if (g.mlp <= 0 || g.mlp % 64 || g.hidden % 64 || g.hidden > 4096) return fail(c, WDC_ERR_UNSUPPORTED, "hidden/mlp must be multiples of 64, hidden <= 4096");
    if (g.temb_dim <= 0 || g.freq_dim <= 0 || g.freq_dim % 2) return fail(c, WDC_ERR_INVALID_ARG, "bad temb/freq dims");
    if (g.cond_tokens < 0 || (g.cond_tokens > 0 && g.cond_dim <= 0)) return fail(c, WDC_ERR_INVALID_ARG, "bad condition tokens");
    if (g.dual_stream && g.cond_tokens == 0) return fail(c, WDC_ERR_INVALID_ARG, "dual_stream needs condition tokens");
    return WDC_OK;
}

wdc_status check_params(Ctx* c, const wdc_cache_params& p) {
    if (p.bank_capacity < 1 || p.bank_capacity > WDC_MAX_BANK) return fail(c, WDC_ERR_INVALID_ARG, "bank_capacity must be 1..8");
    if (!(p.tau_in > 0) || !(p.tau_obs > 0)) return fail(c, WDC_ERR_INVALID_ARG, "temperatures must be > 0");
    if (!(p.alpha_min <= p.alpha_max)) return fail(c, WDC_ERR_INVALID_ARG, "alpha_min > alpha_max");
    if (!(p.eta_min <= p.eta_max) || !(p.eta_min >= 0)) return fail(c, WDC_ERR_INVALID_ARG, "bad eta bounds");
    if (!(p.beta_d >= 0 && p.beta_d <= 1)) return fail(c, WDC_ERR_INVALID_ARG, "beta_d must be in [0,1]");
    if (!(p.lambda_ >= 0)) return fail(c, WDC_ERR_INVALID_ARG, "lambda must be >= 0");
    if (p.min_support < 0 || p.max_age < 0 || p.n_init_exact < 0 || p.n_final_exact < 0)
        return fail(c, WDC_ERR_INVALID_ARG, "negative integer parameter");
    if (p.flags & ~(WDC_ABL_ALL | WDC_OBS_RESIDUAL)) return fail(c, WDC_ERR_INVALID_ARG, "unknown flag");
    if ((p.flags & WDC_ABL_PERIODIC) && p.period < 1) return fail(c, WDC_ERR_INVALID_ARG, "period must be >= 1");
    if ((p.flags & WDC_ABL_LINEAR_OBS) && !(p.ridge >= 0 && p.ridge < 1e300))
        return fail(c, WDC_ERR_INVALID_ARG, "ridge must be finite and >= 0");
    return WDC_OK;
}


int slot_of(const Ctx* c, int age_idx) { return (c->head + age_idx) % c->prm.bank_capacity; }
int newest_slot(const Ctx* c) { return slot_of(c, c->n_bank - 1); }

const float* anchor_ptr(const Ctx* c) { return c->n_bank > 0 ? c->bank[newest_slot(c)] : c->z_init; }

PassArgs base_args(Ctx* c, int k) {
    PassArgs a;
    std::memset(&a, 0, sizeof(a));
    a.n = (long long)c->n;
    a.k = k;
    a.T = c->sched.T;
    a.age = c->age;
    a.sk = c->stepf[k];
    a.prm = to_dev_params(c->prm);
    a.st = c->st;
    a.partials = c->partials;
    a.counter = c->counter;
    a.err = c->err;
    return a;
}

void set_cond(PassArgs& a, const wdc_cond* cd) {
    for (int j = 0; j < 4; ++j) {
        a.cam[j] = cd ? (float)cd->cam[j] : 0.f;
        a.depth[j] = cd ? (float)cd->depth[j] : 0.f;
    }
}

// Skip pass + async copy of the step record into `dst` (pinned); no sync.
bool needs_disp(const Ctx* c) { return c->prm.flags & (WDC_ABL_SECANT | WDC_OBS_RESIDUAL); }

// z_cur (the current latent) is read only by the secant and the residual reading.
wdc_status enqueue_skip(Ctx* c, int k, const wdc_cond* cd, const float* z_cur, float* z_hat, StepOut* dst,
                        cudaStream_t s) {
    PassArgs a = base_args(c, k);
    set_cond(a, cd);
    a.nsrc = c->n_bank;
    for (int i = 0; i < c->n_bank; ++i) a.slot[i] = slot_of(c, i);
    int mode = kModeSkip;
    if (needs_disp(c) && (!z_cur || !c->disp[0]))
        return fail(c, WDC_ERR_STATE, "this candidate needs the current latent and the displacement buffers");
    if (c->prm.flags & WDC_ABL_SECANT) {
        mode = kModeSecant;
        a.src[0] = z_cur;
        a.src[1] = c->disp[c->n_bank > 0 ? newest_slot(c) : 0];
    } else if (c->prm.flags & WDC_OBS_RESIDUAL) {
        mode = kModeResidual;
        a.zcur = z_cur;
        for (int i = 0; i < c->n_bank; ++i) a.src[i] = c->disp[a.slot[i]];
    } else {
        for (int i = 0; i < c->n_bank; ++i) a.src[i] = c->bank[a.slot[i]];
    }
    a.anchor = anchor_ptr(c);
    a.out = z_hat;
    wdc_status st = launch_pass(c, mode, a, s);
    if (st) return st;
    WDC_CUDA_TRY(c, cudaMemcpyAsync(dst, &c->st->out, sizeof(StepOut), cudaMemcpyDeviceToHost, s));
    return WDC_OK;
}

wdc_status enqueue_anchor(Ctx* c, int k, const wdc_cond* cd, const float* z_t, const float* v, const float* z_cf,
                          const float** z_next, StepOut* dst, cudaStream_t s) {
    const int K = c->prm.bank_capacity;
    const int ins = c->n_bank < K ? slot_of(c, c->n_bank) : c->head;
    PassArgs a = base_args(c, k);
    set_cond(a, cd);
    a.src[0] = z_t;
    a.v = v;
    a.zcf = z_cf;
    a.anchor = anchor_ptr(c);
    a.out = c->bank[ins];
    a.out2 = needs_disp(c) ? c->disp[ins] : nullptr;
    a.ins_slot = ins;
    wdc_status st = launch_pass(c, kModeAnchor, a, s);
    if (st) return st;
    if (dst) WDC_CUDA_TRY(c, cudaMemcpyAsync(dst, &c->st->out, sizeof(StepOut), cudaMemcpyDeviceToHost, s));
    if (c->n_bank < K) c->n_bank++;
    else c->head = (c->head + 1) % K;
    c->age = 0;
    c->anchor_is_init = 0;
    c->last_surrogate_k = -1;
    if (z_next) *z_next = c->bank[ins];
    c->cur_latent = c->bank[ins];
    return WDC_OK;
}

// Per-slot exact-step displacements for the secant and the residual reading
// (allocated on first use, zeroed).
wdc_status ensure_disp(Ctx* c) {
    if (!needs_disp(c) || c->disp[0]) return WDC_OK;
    for (int i = 0; i < c->prm.bank_capacity; ++i) {
        WDC_CUDA_TRY(c, cudaMalloc((void**)&c->disp[i], c->n * sizeof(float)));
        WDC_CUDA_TRY(c, cudaMemset(c->disp[i], 0, c->n * sizeof(float)));
    }
    return WDC_OK;
}

wdc_status clear_disp(Ctx* c, cudaStream_t s) {
    for (int i = 0; i < kMaxBank; ++i)
        if (c->disp[i]) WDC_CUDA_TRY(c, cudaMemsetAsync(c->disp[i], 0, c->n * sizeof(float), s));
    return WDC_OK;
}

wdc_status stats_pass(Ctx* c, const float* z_cur, cudaStream_t s) {
    PassArgs a = base_args(c, 0);
    a.src[0] = z_cur;
    a.anchor = anchor_ptr(c);
    return launch_pass(c, kModeStats, a, s);
}

wdc_status sync(Ctx* c, cudaStream_t s) {
    WDC_CUDA_TRY(c, cudaStreamSynchronize(s));
    return WDC_OK;
}

}  // namespace

extern "C" {

const char* wdc_status_string(wdc_status s) {
    switch (s) {
        case WDC_OK: return "ok";
        case WDC_ERR_INVALID_ARG: return "invalid argument";
        case WDC_ERR_CUDA: return "CUDA error";
        case WDC_ERR_UNSUPPORTED: return "unsupported";
        case WDC_ERR_TIMEOUT: return "device wait timed out";
        case WDC_ERR_NONFINITE: return "non-finite value";
        case WDC_ERR_STATE: return "call out of order";
        case WDC_ERR_OOM: return "out of device memory";
    }
    return "unknown status";
}

wdc_status wdc_default_cache_params(wdc_cache_params* p) {
    if (!p) return WDC_ERR_INVALID_ARG;
    std::memset(p, 0, sizeof(*p));
    p->bank_capacity = 4; p->min_support = 1;
    p->sim_min = 0.0; p->q_gap_max = 0.25; p->gamma_q = 10.0; p->tau_in = 0.1; p->tau_obs = 0.05;
    p->alpha_min = 0.5; p->alpha_max = 2.0; p->eps = 1e-8; p->eps_nu = 1e-12; p->sketch_seed = 0x2545F491u;
    p->w_z = 1.0; p->w_age = 0.05; p->w_phase = 1.0; p->w_cam = 0.5; p->w_depth = 0.5;
    p->eta_init = 1.0; p->eta_min = 0.1; p->eta_max = 10.0; p->beta_d = 0.8;
    p->a_cam = 0.5; p->a_depth = 0.5; p->a_phase = 1.0; p->lambda_ = 0.9; p->tau_risk = 0.5;
    p->max_age = 6; p->n_init_exact = 1; p->n_final_exact = 0; p->flags = 0;
    p->period = 8; p->ridge = 1e-6;
    return WDC_OK;
}

wdc_status wdc_create(const wdc_dit_config* cfg, const wdc_schedule* sched, const wdc_cache_params* params,
                      int device, wdc_ctx** out) {
    if (!out) return WDC_ERR_INVALID_ARG;
    *out = nullptr;
    if (!cfg || !sched || !params) return WDC_ERR_INVALID_ARG;
    Ctx* c = new (std::nothrow) Ctx();
    if (!c) return WDC_ERR_OOM;
    wdc_status st;
    auto bail = [&](wdc_status s) {
        wdc_destroy(reinterpret_cast<wdc_ctx*>(c));
        return s;
    };
    c->cfg = *cfg;
    c->sched = *sched;
    c->prm = *params;
    c->device = device;
    if ((st = check_cfg(c, c->cfg))) return bail(st);
    if ((st = check_params(c, c->prm))) return bail(st);
    if (sched->T < 1 || !(sched->shift > 0)) return bail(WDC_ERR_INVALID_ARG);
    if (cudaSetDevice(device) != cudaSuccess) { cudaGetLastError(); return bail(WDC_ERR_CUDA); }
    if (cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess) return bail(WDC_ERR_CUDA);
    c->n = (size_t)cfg->in_ch * cfg->frames * cfg->height * cfg->width;
    if (c->n >= (1ull << 31)) return bail(WDC_ERR_UNSUPPORTED);
    c->sigma.resize(sched->T + 1);
    for (int k = 0; k <= sched->T; ++k) {
        double s = 1.0 - (double)k / (double)sched->T;
        if (sched->shift != 1.0) s = sched->shift * s / (1.0 + (sched->shift - 1.0) * s);
        c->sigma[k] = s;
    }
    c->stepf.resize(sched->T);
    for (int k = 0; k < sched->T; ++k) {
        StepScalars& f = c->stepf[k];
        f.q_k = (float)c->sigma[k];
        f.q_next = (float)c->sigma[k + 1];
        f.dq = (float)(c->sigma[k + 1] - c->sigma[k]);
        f.t_model = (float)(1000.0 * c->sigma[k]);
    }
    const size_t lat = c->n * sizeof(float);
    auto dm = [&](void** p, size_t b) -> bool {
        if (cudaMalloc(p, b) != cudaSuccess) { cudaGetLastError(); return false; }
        cudaMemset(*p, 0, b);
        return true;
    };
    if (!dm((void**)&c->st, sizeof(DevState))) return bail(WDC_ERR_OOM);
    if (!dm((void**)&c->partials, (size_t)c->num_sms * kPartials * sizeof(float))) return bail(WDC_ERR_OOM);
    if (!dm((void**)&c->counter, 64)) return bail(WDC_ERR_OOM);
    if (!dm((void**)&c->err, 64)) return bail(WDC_ERR_OOM);
    if (!dm((void**)&c->pstat, 64)) return bail(WDC_ERR_OOM);
    for (int i = 0; i < c->prm.bank_capacity; ++i)
        if (!dm((void**)&c->bank[i], lat)) return bail(WDC_ERR_OOM);
    if (!dm((void**)&c->z_init, lat)) return bail(WDC_ERR_OOM);
    if (!dm((void**)&c->cand[0], lat) || !dm((void**)&c->cand[1], lat)) return bail(WDC_ERR_OOM);
    if (!dm((void**)&c->vbuf, lat)) return bail(WDC_ERR_OOM);
    if (cudaMallocHost((void**)&c->out_host, sizeof(StepOut) * (sched->T + 2)) != cudaSuccess) return bail(WDC_ERR_OOM);
    if (cudaMallocHost((void**)&c->st_host, sizeof(DevState)) != cudaSuccess) return bail(WDC_ERR_OOM);
    if ((st = ensure_disp(c))) return bail(st);
    if (cfg->layers > 0) {
        if ((st = dit_create(c))) return bail(st);
    }
    *out = reinterpret_cast<wdc_ctx*>(c);
    return WDC_OK;
}

void wdc_destroy(wdc_ctx* h) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return;
    graph_rollout_destroy(c);
    cudaSetDevice(c->device);
    dit_destroy(c);
    cudaFree(c->st);
    cudaFree(c->partials);
    cudaFree(c->counter);
    cudaFree(c->err);
    cudaFree(c->pstat);
    for (int i = 0; i < kMaxBank; ++i) cudaFree(c->bank[i]);
    cudaFree(c->z_init);
    cudaFree(c->cand[0]);
    cudaFree(c->cand[1]);
    cudaFree(c->vbuf);
    cudaFree(c->zstage);
    cudaFree(c->cond_stage);
    for (int i = 0; i < kMaxBank; ++i) cudaFree(c->disp[i]);
    if (c->out_host) cudaFreeHost(c->out_host);
    if (c->st_host) cudaFreeHost(c->st_host);
    for (int k = 0; k < WDC_K_COUNT; ++k)
        for (cudaEvent_t e : c->ev[k]) cudaEventDestroy(e);
    delete c;
}

wdc_status wdc_selftest_wait_timeout(wdc_ctx* h, unsigned long long limit_ns, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (limit_ns < 1000ull || limit_ns > 1000000000ull) return fail(c, WDC_ERR_INVALID_ARG, "limit_ns must be 1e3..1e9");
    cudaSetDevice(c->device);
    LaunchScope ls(c, WDC_K_OTHER, (cudaStream_t)stream);
    wait_probe_kernel<<<1, 64, 0, (cudaStream_t)stream>>>(c->err, limit_ns);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("wait self-test: ") + cudaGetErrorString(e));
    return WDC_OK;
}

wdc_status wdc_set_cache_params(wdc_ctx* h, const wdc_cache_params* params) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c || !params) return WDC_ERR_INVALID_ARG;
    wdc_status st = check_params(c, *params);
    if (st) return st;
    if (params->bank_capacity != c->prm.bank_capacity)
        return fail(c, WDC_ERR_INVALID_ARG, "bank_capacity cannot change after wdc_create");
    c->prm = *params;
    cudaSetDevice(c->device);
    return ensure_disp(c);
}

const char* wdc_last_error(const wdc_ctx* h) {
    const Ctx* c = reinterpret_cast<const Ctx*>(h);
    return c ? c->last_error.c_str() : "null context";
}

size_t wdc_latent_numel(const wdc_ctx* h) {
    const Ctx* c = reinterpret_cast<const Ctx*>(h);
    return c ? c->n : 0;
}

wdc_status wdc_device_errors(wdc_ctx* h, unsigned* bits) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c || !bits) return WDC_ERR_INVALID_ARG;
    cudaSetDevice(c->device);
    WDC_CUDA_TRY(c, cudaDeviceSynchronize());
    WDC_CUDA_TRY(c, cudaMemcpy(bits, c->err, sizeof(unsigned), cudaMemcpyDeviceToHost));
    WDC_CUDA_TRY(c, cudaMemset(c->err, 0, sizeof(unsigned)));
    return WDC_OK;
}

wdc_status wdc_profile_enable(wdc_ctx* h, int on) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    cudaSetDevice(c->device);
    WDC_CUDA_TRY(c, cudaDeviceSynchronize());
    c->prof = on != 0;
    for (int k = 0; k < WDC_K_COUNT; ++k) { c->ev_used[k] = 0; c->cls_launches[k] = 0; }
    return WDC_OK;
}

wdc_status wdc_profile_read(wdc_ctx* h, double* ms, unsigned long long* launches) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c || !ms || !launches) return WDC_ERR_INVALID_ARG;
    cudaSetDevice(c->device);
    WDC_CUDA_TRY(c, cudaDeviceSynchronize());
    for (int k = 0; k < WDC_K_COUNT; ++k) {
        double tot = 0.0;
        for (size_t i = 0; i + 1 < c->ev_used[k]; i += 2) {
            float t = 0.f;
            if (cudaEventElapsedTime(&t, c->ev[k][i], c->ev[k][i + 1]) == cudaSuccess) tot += t;
            else cudaGetLastError();
        }
        ms[k] = tot;
        launches[k] = c->cls_launches[k];
        c->ev_used[k] = 0;
        c->cls_launches[k] = 0;
    }
    return WDC_OK;
}

unsigned long long wdc_launch_count(const wdc_ctx* h) {
    const Ctx* c = reinterpret_cast<const Ctx*>(h);
    return c ? c->launches : 0;
}

wdc_status wdc_set_tensor(wdc_ctx* h, int tensor_id, int layer, int stream, const float* host, size_t count) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    cudaSetDevice(c->device);
    return dit_set_tensor(c, tensor_id, layer, stream, host, count);
}

wdc_status wdc_get_tensor(wdc_ctx* h, int tensor_id, int layer, int stream, float* host, size_t count) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    cudaSetDevice(c->device);
    return dit_get_tensor(c, tensor_id, layer, stream, host, count);
}

wdc_status wdc_init_weights(wdc_ctx* h, unsigned long long seed, float std) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    cudaSetDevice(c->device);
    return dit_init_weights(c, seed, std);
}

wdc_status wdc_dit_forward(wdc_ctx* h, const float* z_t, float t, const float* cond_tokens, float* v, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (z_t && !aligned16(z_t)) return fail(c, WDC_ERR_INVALID_ARG, "z_t must be 16-byte aligned");
    cudaSetDevice(c->device);
    return dit_forward(c, z_t, t, cond_tokens, v, (cudaStream_t)stream);
}

wdc_status wdc_dit_forward_batch(wdc_ctx* h, int B, const float* const* z_t, float t, const float* const* cond_tokens,
                                 int cfg, float guidance, float* const* v, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (B < 1 || B > WDC_MAX_BATCH) return fail(c, WDC_ERR_INVALID_ARG, "B must be 1..16");
    cudaSetDevice(c->device);
    return dit_forward_guided(c, B, z_t, t, cond_tokens, cfg ? 1 : 0, guidance, v, (cudaStream_t)stream);
}

wdc_status wdc_dit_block_forward(wdc_ctx* h, int layer, void* x, const float* mod6, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    cudaSetDevice(c->device);
    return dit_block(c, layer, x, mod6, (cudaStream_t)stream);
}

wdc_status wdc_dit_modulation(wdc_ctx* h, float t, float* mod_out, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (!mod_out) return fail(c, WDC_ERR_INVALID_ARG, "null mod_out");
    cudaSetDevice(c->device);
    return dit_modulation(c, t, mod_out, (cudaStream_t)stream);
}

wdc_status wdc_schedule_sigmas(const wdc_ctx* h, double* out) {
    const Ctx* c = reinterpret_cast<const Ctx*>(h);
    if (!c || !out) return WDC_ERR_INVALID_ARG;
    for (size_t k = 0; k < c->sigma.size(); ++k) out[k] = c->sigma[k];
    return WDC_OK;
}

wdc_status wdc_latent_pair_stats(wdc_ctx* h, const float* a, const float* b, const float* cz, double* out,
                                 wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (!a || !b || !out) return fail(c, WDC_ERR_INVALID_ARG, "null pointer");
    if (!aligned16(a) || !aligned16(b) || (cz && !aligned16(cz)))
        return fail(c, WDC_ERR_INVALID_ARG, "latents must be 16-byte aligned device pointers");
    cudaSetDevice(c->device);
    cudaStream_t s = (cudaStream_t)stream;
    wdc_status st = launch_pair_stats(c, a, b, cz, c->pstat, s);
    if (st) return st;
    WDC_CUDA_TRY(c, cudaMemcpyAsync(out, c->pstat, 5 * sizeof(double), cudaMemcpyDeviceToHost, s));
    WDC_CUDA_TRY(c, cudaStreamSynchronize(s));
    return WDC_OK;
}

// Average ranks (ties share the mean of their positions), 0-based.
static void average_ranks(const double* x, int n, std::vector<double>& r) {
    std::vector<int> idx(n);
    for (int i = 0; i < n; ++i) idx[i] = i;
    std::stable_sort(idx.begin(), idx.end(), [&](int p, int q) { return x[p] < x[q]; });
    r.assign(n, 0.0);
    for (int i = 0; i < n;) {
        int j = i;
        while (j + 1 < n && x[idx[j + 1]] == x[idx[i]]) ++j;
        const double avg = 0.5 * (i + j);
        for (int m = i; m <= j; ++m) r[idx[m]] = avg;
        i = j + 1;
    }
}

static double pearson(const double* x, const double* y, int n) {
    double mx = 0, my = 0;
    for (int i = 0; i < n; ++i) { mx += x[i]; my += y[i]; }
    mx /= n;
    my /= n;
    double sxy = 0, sxx = 0, syy = 0;
    for (int i = 0; i < n; ++i) {
        const double dx = x[i] - mx, dy = y[i] - my;
        sxy += dx * dy;
        sxx += dx * dx;
        syy += dy * dy;
    }
    return (sxx > 0 && syy > 0) ? sxy / std::sqrt(sxx * syy) : NAN;
}

wdc_status wdc_correlations(const double* x, const double* y, int n, double* pearson_out, double* spearman_out) {
    if (!x || !y || !pearson_out || !spearman_out || n < 2) return WDC_ERR_INVALID_ARG;
    *pearson_out = pearson(x, y, n);
    std::vector<double> rx, ry;
    average_ranks(x, n, rx);
    average_ranks(y, n, ry);
    *spearman_out = pearson(rx.data(), ry.data(), n);
    return WDC_OK;
}

wdc_status wdc_scheduler_step(wdc_ctx* h, int k, const float* z_t, const float* v, float* z_next, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (k < 0 || k >= c->sched.T) return fail(c, WDC_ERR_INVALID_ARG, "k out of range");
    if (!z_t || !v || !z_next) return fail(c, WDC_ERR_INVALID_ARG, "null pointer");
    if (!aligned16(z_t) || !aligned16(v) || !aligned16(z_next)) return fail(c, WDC_ERR_INVALID_ARG, "latents must be 16-byte aligned");
    cudaSetDevice(c->device);
    const long long n = (long long)c->n;
    const unsigned grid = (unsigned)(((n + 3) / 4 + 255) / 256);
    {
        LaunchScope ls(c, WDC_K_OTHER, (cudaStream_t)stream);
        psi_kernel<<<grid, 256, 0, (cudaStream_t)stream>>>(z_t, v, z_next, n, c->stepf[k].dq);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("scheduler_step: ") + cudaGetErrorString(e));
    return WDC_OK;
}

wdc_status wdc_state_reset(wdc_ctx* h, const float* z_T, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (!z_T || !aligned16(z_T)) return fail(c, WDC_ERR_INVALID_ARG, "z_T must be a 16-byte aligned device pointer");
    cudaSetDevice(c->device);
    cudaStream_t s = (cudaStream_t)stream;
    WDC_CUDA_TRY(c, cudaMemcpyAsync(c->z_init, z_T, c->n * sizeof(float), cudaMemcpyDeviceToDevice, s));
    c->n_bank = 0;
    c->head = 0;
    c->age = 0;
    c->anchor_is_init = 1;
    c->last_surrogate_k = -1;
    c->cur_latent = c->z_init;
    wdc_status cs = clear_disp(c, s);
    if (cs) return cs;
    DevState* hs = c->st_host;           // pinned staging owned by the context
    std::memset(hs, 0, sizeof(DevState));
    hs->R = 0.f;
    hs->eta = (float)c->prm.eta_init;
    hs->q_a_in = hs->q_a_out = (float)c->sigma[0];
    hs->q_a_dq = 0.f;
    hs->cand_k = -1;
    cudaError_t e = cudaMemcpyAsync(c->st, hs, sizeof(DevState), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("state_reset: ") + cudaGetErrorString(e));
    return stats_pass(c, c->z_init, s);
}

wdc_status wdc_state_get(wdc_ctx* h, wdc_state_host* out, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c || !out) return WDC_ERR_INVALID_ARG;
    cudaSetDevice(c->device);
    DevState* hs = c->st_host;           // pinned staging owned by the context
    cudaError_t e = cudaMemcpyAsync(hs, c->st, sizeof(DevState), cudaMemcpyDeviceToHost, (cudaStream_t)stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) {
        return fail(c, WDC_ERR_CUDA, std::string("state_get: ") + cudaGetErrorString(e));
    }
    std::memset(out, 0, sizeof(*out));
    out->n_bank = c->n_bank;
    out->age = c->age;
    out->R = hs->R;
    out->eta = hs->eta;
    out->q_a_in = hs->q_a_in;
    out->q_a_out = hs->q_a_out;
    for (int j = 0; j < 4; ++j) { out->cam_a[j] = hs->cam_a[j]; out->depth_a[j] = hs->depth_a[j]; }
    for (int i = 0; i < c->n_bank; ++i) {
        const DevRecord& r = hs->rec[slot_of(c, i)];
        wdc_record_host& o = out->rec[i];
        for (int j = 0; j < kSummary; ++j) {
            o.s_in[j] = r.s_in[j];
            o.s_out[j] = r.s_out[j];
            o.s_dphi[j] = r.s_dphi[j];
        }
        o.q_in = r.q_in; o.q_out = r.q_out; o.r = r.r;
        for (int j = 0; j < 4; ++j) { o.cam[j] = r.cam[j]; o.depth[j] = r.depth[j]; }
    }
    for (int j = 0; j < kSketch; ++j) {
        out->cur_sketch[j] = hs->cur_S[j];
        out->anchor_sketch[j] = hs->anchor_S[j];
    }
    out->cur_sumsq = hs->cur_sumsq;
    out->cur_sumsq_anchor = hs->cur_sumsq_anchor;
    out->anchor_sumsq = hs->anchor_sumsq;
    for (int j = 0; j < kSummary; ++j) out->s_phi[j] = hs->s_phi[j];
    out->cand_supported = hs->cand_supported;
    out->cand_finite = hs->cand_finite;
    out->cand_p = hs->cand_p;
    return WDC_OK;
}

wdc_status wdc_state_set(wdc_ctx* h, const wdc_state_host* in, const float* const* z_out, const float* z_cur,
                         wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c || !in) return WDC_ERR_INVALID_ARG;
    if (in->n_bank < 0 || in->n_bank > c->prm.bank_capacity) return fail(c, WDC_ERR_INVALID_ARG, "n_bank out of range");
    if (in->age < 0) return fail(c, WDC_ERR_INVALID_ARG, "negative age");
    if (!z_cur || !aligned16(z_cur)) return fail(c, WDC_ERR_INVALID_ARG, "z_cur must be a 16-byte aligned device pointer");
    if (in->n_bank > 0 && !z_out) return fail(c, WDC_ERR_INVALID_ARG, "z_out required for a non-empty bank");
    for (int i = 0; i < in->n_bank; ++i)
        if (!z_out[i] || !aligned16(z_out[i])) return fail(c, WDC_ERR_INVALID_ARG, "bank latents must be 16-byte aligned device pointers");
    cudaSetDevice(c->device);
    cudaStream_t s = (cudaStream_t)stream;
    DevState* hs = c->st_host;           // pinned staging owned by the context
    std::memset(hs, 0, sizeof(DevState));
    hs->R = (float)in->R;
    hs->eta = (float)in->eta;
    hs->q_a_in = (float)in->q_a_in;
    hs->q_a_out = (float)in->q_a_out;
    hs->q_a_dq = (float)(in->q_a_out - in->q_a_in);
    for (int j = 0; j < 4; ++j) { hs->cam_a[j] = (float)in->cam_a[j]; hs->depth_a[j] = (float)in->depth_a[j]; }
    hs->cand_k = -1;
    for (int i = 0; i < in->n_bank; ++i) {
        DevRecord& r = hs->rec[i];
        const wdc_record_host& o = in->rec[i];
        double a = 0, b = 0;
        for (int j = 0; j < kSummary; ++j) {
            r.s_in[j] = (float)o.s_in[j];
            r.s_out[j] = (float)o.s_out[j];
            r.s_dphi[j] = (float)o.s_dphi[j];
            a += (double)r.s_in[j] * r.s_in[j];
            b += (double)r.s_out[j] * r.s_out[j];
        }
        r.n_in = (float)std::sqrt(a);
        r.n_out = (float)std::sqrt(b);
        r.q_in = (float)o.q_in;
        r.q_out = (float)o.q_out;
        r.dq = (float)(o.q_out - o.q_in);
        r.r = (float)o.r;
        for (int j = 0; j < 4; ++j) { r.cam[j] = (float)o.cam[j]; r.depth[j] = (float)o.depth[j]; }
    }
    cudaError_t e = cudaMemcpyAsync(c->st, hs, sizeof(DevState), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("state_set: ") + cudaGetErrorString(e));
    c->head = 0;
    c->n_bank = in->n_bank;
    c->age = in->age;
    c->last_surrogate_k = -1;
    c->cur_latent = z_cur;
    if (wdc_status cs = clear_disp(c, s)) return cs;
    for (int i = 0; i < in->n_bank; ++i)
        WDC_CUDA_TRY(c, cudaMemcpyAsync(c->bank[i], z_out[i], c->n * sizeof(float), cudaMemcpyDeviceToDevice, s));
    if (in->n_bank == 0) {
        WDC_CUDA_TRY(c, cudaMemcpyAsync(c->z_init, z_cur, c->n * sizeof(float), cudaMemcpyDeviceToDevice, s));
        c->anchor_is_init = 1;
    } else {
        c->anchor_is_init = 0;
    }
    return stats_pass(c, z_cur, s);
}

wdc_status wdc_surrogate_step(wdc_ctx* h, int k, const wdc_cond* cd, float* z_hat, wdc_step_info* info,
                              wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (k < 0 || k >= c->sched.T) return fail(c, WDC_ERR_INVALID_ARG, "k out of range");
    if (!z_hat || !aligned16(z_hat)) return fail(c, WDC_ERR_INVALID_ARG, "z_hat must be a 16-byte aligned device pointer");
    for (int i = 0; i < c->prm.bank_capacity; ++i)
        if (z_hat == c->bank[i]) return fail(c, WDC_ERR_INVALID_ARG, "z_hat must not be a bank buffer");
    cudaSetDevice(c->device);
    cudaStream_t s = (cudaStream_t)stream;
    const int age_before = c->age, nb = c->n_bank;
    wdc_status st = enqueue_skip(c, k, cd, c->cur_latent, z_hat, &c->out_host[0], s);
    if (st) return st;
    if ((st = sync(c, s))) return st;
    const StepOut& o = c->out_host[0];
    if (o.decision) {
        c->age++;
        c->cur_latent = z_hat;
    }
    c->last_surrogate_k = k;
    fill_info(o, k, nb, age_before, info);
    return WDC_OK;
}

wdc_status wdc_risk_update(wdc_ctx* h, int k, const wdc_cond* cd, const float* z_t, const float* v,
                           const float* z_cf, const float** z_next, wdc_step_info* info, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (k < 0 || k >= c->sched.T) return fail(c, WDC_ERR_INVALID_ARG, "k out of range");
    if (c->last_surrogate_k != k) return fail(c, WDC_ERR_STATE, "wdc_risk_update(k) must follow wdc_surrogate_step(k)");
    if (!z_t || !v || !aligned16(z_t) || !aligned16(v) || (z_cf && !aligned16(z_cf)))
        return fail(c, WDC_ERR_INVALID_ARG, "latents must be 16-byte aligned device pointers");
    cudaSetDevice(c->device);
    cudaStream_t s = (cudaStream_t)stream;
    const int nb = c->n_bank, age_before = c->age;
    wdc_status st = enqueue_anchor(c, k, cd, z_t, v, z_cf, z_next, info ? &c->out_host[1] : nullptr, s);
    if (st) return st;
    if (info) {
        if ((st = sync(c, s))) return st;
        const StepOut& o = c->out_host[1];
        info->d_cf = o.d_cf;
        info->R = o.R;
        info->eta = o.eta;
        info->r = o.r;
        info->n_bank = nb;
        info->age = age_before;
    }
    return WDC_OK;
}

static wdc_status rollout_impl(Ctx* c, const float* z_T, const wdc_cond* conds, int n_cond, float* z_out,
                               int* decisions, wdc_step_info* trace, cudaStream_t s, bool cached) {
    const int T = c->sched.T;
    if (!z_T || !z_out || !conds) return fail(c, WDC_ERR_INVALID_ARG, "null pointer");
    if (n_cond != 1 && n_cond != T) return fail(c, WDC_ERR_INVALID_ARG, "n_cond must be 1 or T");
    if (!c->dit) return fail(c, WDC_ERR_UNSUPPORTED, "rollout needs a denoiser (layers > 0)");
    const size_t bytes = c->n * sizeof(float);
    const bool in_dev = is_device_ptr(z_T), out_dev = is_device_ptr(z_out);
    if (in_dev && !aligned16(z_T)) return fail(c, WDC_ERR_INVALID_ARG, "z_T must be 16-byte aligned");
    // condition tokens: device pointers are used directly, host ones staged
    const size_t cond_elems = (size_t)c->cfg.cond_tokens * c->cfg.cond_dim;
    std::vector<const float*> tok(n_cond, nullptr);
    for (int i = 0; i < n_cond; ++i) {
        if (cond_elems == 0) continue;
        if (!conds[i].tokens) return fail(c, WDC_ERR_INVALID_ARG, "condition tokens required");
        if (is_device_ptr(conds[i].tokens)) { tok[i] = conds[i].tokens; continue; }
        // host tokens go through the context's staging buffer, kept between
        // calls and grown when a call needs more
        const size_t need = cond_elems * sizeof(float) * n_cond;
        if (c->cond_stage_bytes < need) {
            WDC_CUDA_TRY(c, cudaStreamSynchronize(s));   // a failed earlier call may still read the old one
            cudaFree(c->cond_stage);
            c->cond_stage = nullptr;
            c->cond_stage_bytes = 0;
            if (cudaMalloc((void**)&c->cond_stage, need) != cudaSuccess) {
                cudaGetLastError();
                c->cond_stage = nullptr;
                return fail(c, WDC_ERR_OOM, "condition staging");
            }
            c->cond_stage_bytes = need;
        }
        WDC_CUDA_TRY(c, cudaMemcpyAsync(c->cond_stage + cond_elems * i, conds[i].tokens, cond_elems * sizeof(float),
                                        cudaMemcpyHostToDevice, s));
        tok[i] = c->cond_stage + cond_elems * i;
    }

    WDC_CUDA_TRY(c, cudaMemcpyAsync(c->cand[0], z_T, bytes, in_dev ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, s));
    float* cur = c->cand[0];
    int cur_cand = 0;
    wdc_status st;
    if (!cached) {
        for (int k = 0; k < T; ++k) {
            const int ci = n_cond == 1 ? 0 : k;
            if ((st = dit_forward(c, cur, (float)(1000.0 * c->sigma[k]), tok[ci], c->vbuf, s))) return st;
            if ((st = wdc_scheduler_step(reinterpret_cast<wdc_ctx*>(c), k, cur, c->vbuf, cur, s))) return st;
        }
    } else {
        if ((st = wdc_state_reset(reinterpret_cast<wdc_ctx*>(c), cur, s))) return st;
        for (int k = 0; k < T; ++k) {
            const int ci = n_cond == 1 ? 0 : k;
            const wdc_cond* cd = &conds[ci];
            float* zh = c->cand[cur_cand == 0 ? 1 : 0];
            const int nb = c->n_bank, age_before = c->age;
            if ((st = enqueue_skip(c, k, cd, cur, zh, &c->out_host[k], s))) return st;
            if ((st = sync(c, s))) return st;
            const int dec = c->out_host[k].decision;
            c->last_surrogate_k = k;
            if (decisions) decisions[k] = dec;
            if (trace) fill_info(c->out_host[k], k, nb, age_before, &trace[k]);
            if (dec) {
                c->age++;
                cur = zh;
                cur_cand = cur_cand == 0 ? 1 : 0;
            } else {
                const bool cf = c->out_host[k].supported && c->out_host[k].finite;
                if ((st = dit_forward(c, cur, (float)(1000.0 * c->sigma[k]), tok[ci], c->vbuf, s))) return st;
                const float* zn = nullptr;
                if ((st = enqueue_anchor(c, k, cd, cur, c->vbuf, cf ? zh : nullptr, &zn, &c->out_host[T], s))) return st;
                if (trace) {
                    if ((st = sync(c, s))) return st;
                    trace[k].d_cf = c->out_host[T].d_cf;
                    trace[k].R = c->out_host[T].R;
                    trace[k].eta = c->out_host[T].eta;
                    trace[k].r = c->out_host[T].r;
                }
                cur = const_cast<float*>(zn);
                cur_cand = -1;
            }
        }
    }
    WDC_CUDA_TRY(c, cudaMemcpyAsync(z_out, cur, bytes, out_dev ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost, s));
    return sync(c, s);
}

wdc_status wdc_rollout(wdc_ctx* h, const float* z_T, const wdc_cond* conds, int n_cond, float* z_out, int* decisions,
                       wdc_step_info* trace, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    cudaSetDevice(c->device);
    return rollout_impl(c, z_T, conds, n_cond, z_out, decisions, trace, (cudaStream_t)stream, true);
}

wdc_status wdc_rollout_graph(wdc_ctx* h, const float* z_T, const wdc_cond* cond, float* z_out, int* decisions,
                             wdc_step_info* trace, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (!z_T || !z_out || !cond) return fail(c, WDC_ERR_INVALID_ARG, "null pointer");
    if (!c->dit) return fail(c, WDC_ERR_UNSUPPORTED, "rollout needs a denoiser (layers > 0)");
    const size_t cond_elems = (size_t)c->cfg.cond_tokens * c->cfg.cond_dim;
    if (cond_elems && !cond->tokens) return fail(c, WDC_ERR_INVALID_ARG, "condition tokens required");
    cudaSetDevice(c->device);
    const bool in_dev = is_device_ptr(z_T), out_dev = is_device_ptr(z_out);
    const bool tok_dev = cond_elems && is_device_ptr(cond->tokens);
    return graph_rollout(c, z_T, in_dev, cond, tok_dev ? cond->tokens : nullptr, z_out, out_dev, decisions, trace,
                         (cudaStream_t)stream);
}

wdc_status wdc_rollout_batch(wdc_ctx* const* hs, int B, const float* const* z_T, const wdc_cond* conds, int n_cond,
                             int cfg, float guidance, float* const* z_out, int* decisions, wdc_step_info* trace,
                             wdc_stream stream) {
    if (!hs || !hs[0]) return WDC_ERR_INVALID_ARG;
    Ctx* c0 = reinterpret_cast<Ctx*>(hs[0]);
    cudaSetDevice(c0->device);
    cudaStream_t s = (cudaStream_t)stream;
    const int T = c0->sched.T;
    if (B < 1 || B > WDC_MAX_BATCH) return fail(c0, WDC_ERR_INVALID_ARG, "B must be 1..16");
    if (!c0->dit) return fail(c0, WDC_ERR_UNSUPPORTED, "ctxs[0] must own a denoiser (layers > 0)");
    const int max_batch = c0->cfg.max_batch > 1 ? c0->cfg.max_batch : 1;
    if ((cfg ? 2 * B : B) > max_batch) return fail(c0, WDC_ERR_INVALID_ARG, "batch larger than ctxs[0]'s max_batch");
    if (!z_T || !z_out || !conds) return fail(c0, WDC_ERR_INVALID_ARG, "null pointer array");
    if (n_cond != 1 && n_cond != T) return fail(c0, WDC_ERR_INVALID_ARG, "n_cond must be 1 or T");
    const size_t cond_elems = (size_t)c0->cfg.cond_tokens * c0->cfg.cond_dim;
    std::vector<Ctx*> cs(B);
    for (int b = 0; b < B; ++b) {
        Ctx* cb = reinterpret_cast<Ctx*>(hs[b]);
        if (!cb) return fail(c0, WDC_ERR_INVALID_ARG, "null context");
        for (int a = 0; a < b; ++a)
            if (cs[a] == cb) return fail(c0, WDC_ERR_INVALID_ARG, "every sample needs its own context");
        if (cb->device != c0->device || cb->n != c0->n || cb->sched.T != T || cb->sigma != c0->sigma)
            return fail(c0, WDC_ERR_INVALID_ARG, "contexts differ in device, latent size or schedule");
        if (!z_T[b] || !z_out[b]) return fail(c0, WDC_ERR_INVALID_ARG, "null latent");
        for (int i = 0; i < n_cond && cond_elems; ++i)
            if (!conds[b * n_cond + i].tokens || !is_device_ptr(conds[b * n_cond + i].tokens))
                return fail(c0, WDC_ERR_INVALID_ARG, "condition tokens must be device pointers");
        cs[b] = cb;
    }
    const size_t bytes = c0->n * sizeof(float);
    std::vector<float*> cur(B);
    std::vector<int> cur_cand(B, 0);
    wdc_status st;
    for (int b = 0; b < B; ++b) {
        Ctx* cb = cs[b];
        const bool in_dev = is_device_ptr(z_T[b]);
        if (in_dev && !aligned16(z_T[b])) return fail(c0, WDC_ERR_INVALID_ARG, "z_T must be 16-byte aligned");
        WDC_CUDA_TRY(c0, cudaMemcpyAsync(cb->cand[0], z_T[b], bytes, in_dev ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, s));
        cur[b] = cb->cand[0];
        if ((st = wdc_state_reset(reinterpret_cast<wdc_ctx*>(cb), cur[b], s))) return st;
    }
    std::vector<int> ex;
    std::vector<float*> zh(B);
    std::vector<const float*> zs, toks;
    std::vector<float*> vs;
    for (int k = 0; k < T; ++k) {
        const int ci = n_cond == 1 ? 0 : k;
        std::vector<int> nb(B), age(B);
        for (int b = 0; b < B; ++b) {
            Ctx* cb = cs[b];
            zh[b] = cb->cand[cur_cand[b] == 0 ? 1 : 0];
            nb[b] = cb->n_bank;
            age[b] = cb->age;
            if ((st = enqueue_skip(cb, k, &conds[b * n_cond + ci], cur[b], zh[b], &cb->out_host[k], s))) return st;
        }
        if ((st = sync(c0, s))) return st;
        ex.clear(); zs.clear(); toks.clear(); vs.clear();
        for (int b = 0; b < B; ++b) {
            Ctx* cb = cs[b];
            const StepOut& o = cb->out_host[k];
            cb->last_surrogate_k = k;
            if (decisions) decisions[b * T + k] = o.decision;
            if (trace) fill_info(o, k, nb[b], age[b], &trace[b * T + k]);
            if (o.decision) {
                cb->age++;
                cur[b] = zh[b];
                cur_cand[b] = cur_cand[b] == 0 ? 1 : 0;
            } else {
                ex.push_back(b);
                zs.push_back(cur[b]);
                toks.push_back(cond_elems ? conds[b * n_cond + ci].tokens : nullptr);
                vs.push_back(cb->vbuf);
            }
        }
        if (ex.empty()) continue;
        if ((st = dit_forward_guided(c0, (int)ex.size(), zs.data(), (float)(1000.0 * c0->sigma[k]), toks.data(), cfg ? 1 : 0,
                                     guidance, vs.data(), s)))
            return st;
        for (int b : ex) {
            Ctx* cb = cs[b];
            const StepOut& o = cb->out_host[k];
            const bool cf = o.supported && o.finite;
            const float* zn = nullptr;
            if ((st = enqueue_anchor(cb, k, &conds[b * n_cond + ci], cur[b], cb->vbuf, cf ? zh[b] : nullptr, &zn,
                                     &cb->out_host[T], s)))
                return st;
            cur[b] = const_cast<float*>(zn);
            cur_cand[b] = -1;
        }
        if (trace) {
            if ((st = sync(c0, s))) return st;
            for (int b : ex) {
                const StepOut& o = cs[b]->out_host[T];
                wdc_step_info& ti = trace[b * T + k];
                ti.d_cf = o.d_cf;
                ti.R = o.R;
                ti.eta = o.eta;
                ti.r = o.r;
            }
        }
    }
    for (int b = 0; b < B; ++b) {
        const bool out_dev = is_device_ptr(z_out[b]);
        WDC_CUDA_TRY(c0, cudaMemcpyAsync(z_out[b], cur[b], bytes, out_dev ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost, s));
    }
    return sync(c0, s);
}

wdc_status wdc_native_rollout(wdc_ctx* h, const float* z_T, const wdc_cond* conds, int n_cond, float* z_out,
                              wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    cudaSetDevice(c->device);
    return rollout_impl(c, z_T, conds, n_cond, z_out, nullptr, nullptr, (cudaStream_t)stream, false);
}

wdc_status wdc_op_gemm(wdc_ctx* h, const void* A, const void* W, const float* bias, void* C, int M, int N, int K,
                       int gelu, const void* res, const float* gate, wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (c->cfg.layers == 0) return fail(c, WDC_ERR_UNSUPPORTED, "operators need a model dtype (layers > 0)");
    cudaSetDevice(c->device);
    return op_gemm(c, A, W, bias, C, M, N, K, gelu, res, gate, (cudaStream_t)stream);
}

wdc_status wdc_op_attention(wdc_ctx* h, const void* q, const void* k, const void* vt, void* o, int heads, int L, int d,
                            wdc_stream stream) {
    Ctx* c = reinterpret_cast<Ctx*>(h);
    if (!c) return WDC_ERR_INVALID_ARG;
    if (c->cfg.layers == 0) return fail(c, WDC_ERR_UNSUPPORTED, "operators need a model dtype (layers > 0)");
    cudaSetDevice(c->device);
    return op_attention(c, q, k, vt, o, heads, L, d, (cudaStream_t)stream);
}

}  // extern "C"
