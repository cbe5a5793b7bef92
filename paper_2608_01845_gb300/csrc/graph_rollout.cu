// Cached rollout with device-side control flow (no per-step host sync).
//
// The whole rollout is one CUDA graph:
//
//   WHILE (k < T) {
//     plan_kernel        reads the device-resident discrete state (step k,
//                        bank size, ring head, age) and writes the launch
//                        arguments of this step's skip pass and anchor pass
//                        into device memory; sets the SWITCH value
//     SWITCH (bank size) the fused skip pass specialised for that many
//                        records (arguments read from device memory); its
//                        last CTA decides (Eq. 10) and sets the two IFs
//     IF (exact)         the denoiser forward on the current latent
//                        (timestep read from device memory) and the fused
//                        anchor pass, which also writes z_exact into the
//                        current-latent buffer
//     IF (surrogate)     copy of the candidate into the current-latent buffer
//     update_kernel      step record, decision, bank size / head / age, k + 1
//   }
//
// The kernels, their arithmetic and their order are those of the host-driven
// rollout (wdc_rollout), so the two give the same decisions and latents; only
// the places the per-step bookkeeping lives in differ.
#include "wdc_internal.h"

#include <cstring>

namespace wdc {

namespace {

struct PlanArgs {
    PassArgs tmpl;                   // constant fields of both passes
    const float* bank[kMaxBank];
    float* disp[kMaxBank];
    const float* z_init;
    float* cand;
    float* zcur;
    float* vbuf;
    const StepScalars* stepf;        // [T]
    int K, mode, needs_disp;
    PassArgs* skip;                  // outputs
    PassArgs* anchor;
    int* pre;                        // [T][2]: bank size, age at the start of step k
    unsigned long long h_switch;
};

__global__ void plan_kernel(const PlanArgs* __restrict__ pp) {
    if (threadIdx.x != 0) return;
    const PlanArgs& p = *pp;
    DevState* st = p.tmpl.st;
    const int k = st->g_k, nb = st->g_n_bank, head = st->g_head, age = st->g_age, K = p.K;
    if (k < 0 || k >= p.tmpl.T || nb < 0 || nb > K || head < 0 || head >= K) {
        // out of range (never in a well-formed rollout): run no pass this step
        atomicOr(p.tmpl.err, kErrBounds);
        cudaGraphSetConditional((cudaGraphConditionalHandle)p.h_switch, 0xffffffffu);
        cudaGraphSetConditional((cudaGraphConditionalHandle)p.tmpl.h_exact, 0u);
        cudaGraphSetConditional((cudaGraphConditionalHandle)p.tmpl.h_accept, 0u);
        return;
    }
    auto slot_of = [&](int i) { return (head + i) % K; };
    const float* anchor = nb > 0 ? p.bank[slot_of(nb - 1)] : p.z_init;

    PassArgs a = p.tmpl;
    a.k = k;
    a.age = age;
    a.sk = p.stepf[k];
    a.nsrc = nb;
    for (int i = 0; i < nb; ++i) a.slot[i] = slot_of(i);
    if (p.mode == kModeSecant) {
        a.src[0] = p.zcur;
        a.src[1] = p.disp[nb > 0 ? slot_of(nb - 1) : 0];
    } else if (p.mode == kModeResidual) {
        a.zcur = p.zcur;
        for (int i = 0; i < nb; ++i) a.src[i] = p.disp[slot_of(i)];
    } else {
        for (int i = 0; i < nb; ++i) a.src[i] = p.bank[slot_of(i)];
    }
    a.anchor = anchor;
    a.out = p.cand;
    *p.skip = a;

    PassArgs b = p.tmpl;
    b.graph = 0;
    b.k = k;
    b.age = age;
    b.sk = p.stepf[k];
    b.nsrc = 0;
    const int ins = nb < K ? slot_of(nb) : head;
    b.src[0] = p.zcur;
    b.v = p.vbuf;
    b.zcf = p.cand;          // the anchor tail uses it only if this step's candidate was supported and finite
    b.anchor = anchor;
    b.out = const_cast<float*>(p.bank[ins]);
    b.out2 = p.needs_disp ? p.disp[ins] : nullptr;
    b.out3 = p.zcur;
    b.ins_slot = ins;
    *p.anchor = b;

    st->g_t_model = p.stepf[k].t_model;
    p.pre[2 * k] = nb;
    p.pre[2 * k + 1] = age;
    cudaGraphSetConditional((cudaGraphConditionalHandle)p.h_switch,
                            p.mode == kModeSecant ? 0u : (unsigned)nb);
}

struct UpdateArgs {
    DevState* st;
    StepOut* trace;                  // [T]
    int* dec;                        // [T]
    int K, T;
    unsigned long long h_loop;
};

__global__ void update_kernel(const __grid_constant__ UpdateArgs u) {
    if (threadIdx.x != 0) return;
    DevState* st = u.st;
    const int k = st->g_k;
    if (k < 0 || k >= u.T) {             // never in a well-formed rollout: stop the loop
        cudaGraphSetConditional((cudaGraphConditionalHandle)u.h_loop, 0u);
        return;
    }
    const int d = st->out.decision;
    u.trace[k] = st->out;
    u.dec[k] = d;
    if (d) {
        st->g_age += 1;
    } else {
        if (st->g_n_bank < u.K) st->g_n_bank += 1;
        else st->g_head = (st->g_head + 1) % u.K;
        st->g_age = 0;
    }
    st->g_k = k + 1;
    cudaGraphSetConditional((cudaGraphConditionalHandle)u.h_loop, k + 1 < u.T ? 1u : 0u);
}

#define WDC_G(call)                                                                                \
    do {                                                                                           \
        cudaError_t e__ = (call);                                                                  \
        if (e__ != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string(#call) + ": " + cudaGetErrorString(e__)); \
    } while (0)

wdc_status add_conditional(Ctx* c, cudaGraph_t g, cudaGraphNode_t* node, const cudaGraphNode_t* dep, int ndep,
                           cudaGraphConditionalHandle h, cudaGraphConditionalNodeType type, unsigned size,
                           cudaGraph_t** bodies) {
    // zero-initialised storage (the struct's union has no default constructor)
    alignas(cudaGraphNodeParams) unsigned char raw[sizeof(cudaGraphNodeParams)] = {};
    cudaGraphNodeParams* np = reinterpret_cast<cudaGraphNodeParams*>(raw);
    np->type = cudaGraphNodeTypeConditional;
    np->conditional.handle = h;
    np->conditional.type = type;
    np->conditional.size = size;
    WDC_G(cudaGraphAddNode(node, g, dep, nullptr, ndep, np));
    *bodies = np->conditional.phGraph_out;
    return WDC_OK;
}

}  // namespace

// Graph resources of a context (built on first use, rebuilt when the pass
// mode changes).
struct GraphRollout {
    int mode = -1, K = 0, T = 0;
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    cudaStream_t cap = nullptr;
    float* zcur = nullptr;
    float* cond = nullptr;           // [cond_tokens, cond_dim] fp32 copy of this rollout's tokens
    StepScalars* stepf = nullptr;
    PassArgs* args = nullptr;        // [2]: skip, anchor
    PlanArgs* plan = nullptr;
    StepOut* trace = nullptr;
    int* dec = nullptr;
    int* pre = nullptr;
    unsigned long long h_switch = 0, h_exact = 0, h_accept = 0;
    ~GraphRollout() {
        if (exec) cudaGraphExecDestroy(exec);
        if (graph) cudaGraphDestroy(graph);
        if (cap) cudaStreamDestroy(cap);
        cudaFree(zcur);
        cudaFree(cond);
        cudaFree(stepf);
        cudaFree(args);
        cudaFree(plan);
        cudaFree(trace);
        cudaFree(dec);
        cudaFree(pre);
    }
};

void graph_rollout_destroy(Ctx* c) {
    delete c->grollout;
    c->grollout = nullptr;
}

static int pass_mode_of(const Ctx* c) {
    if (c->prm.flags & WDC_ABL_SECANT) return kModeSecant;
    if (c->prm.flags & WDC_OBS_RESIDUAL) return kModeResidual;
    return kModeSkip;
}

static wdc_status build_graph(Ctx* c, GraphRollout* G) {
    const int K = c->prm.bank_capacity, T = c->sched.T;
    const int mode = pass_mode_of(c);
    if (G->exec) { cudaGraphExecDestroy(G->exec); G->exec = nullptr; }
    if (G->graph) { cudaGraphDestroy(G->graph); G->graph = nullptr; }
    cudaGraph_t g;
    WDC_G(cudaGraphCreate(&g, 0));
    G->graph = g;
    cudaGraphConditionalHandle h_loop, h_switch, h_exact, h_accept;
    WDC_G(cudaGraphConditionalHandleCreate(&h_loop, g, 1, cudaGraphCondAssignDefault));
    cudaGraphNode_t loop;
    cudaGraph_t* lb;
    wdc_status st;
    if ((st = add_conditional(c, g, &loop, nullptr, 0, h_loop, cudaGraphCondTypeWhile, 1, &lb))) return st;
    cudaGraph_t body = lb[0];
    WDC_G(cudaGraphConditionalHandleCreate(&h_switch, body, 0, 0));
    WDC_G(cudaGraphConditionalHandleCreate(&h_exact, body, 0, 0));
    WDC_G(cudaGraphConditionalHandleCreate(&h_accept, body, 0, 0));

    // plan
    cudaGraphNode_t n_plan, n_switch, n_exact, n_accept, n_update;
    {
        void* params[] = {&G->plan};
        cudaKernelNodeParams kp;
        std::memset(&kp, 0, sizeof(kp));
        kp.func = (void*)plan_kernel;
        kp.gridDim = dim3(1);
        kp.blockDim = dim3(32);
        kp.kernelParams = params;
        WDC_G(cudaGraphAddKernelNode(&n_plan, body, nullptr, 0, &kp));
    }
    // SWITCH on the bank size: the skip pass specialised for it
    cudaGraph_t* sb;
    const unsigned nsw = mode == kModeSecant ? 1u : (unsigned)(K + 1);
    if ((st = add_conditional(c, body, &n_switch, &n_plan, 1, h_switch, cudaGraphCondTypeSwitch, nsw, &sb))) return st;
    for (unsigned i = 0; i < nsw; ++i) {
        WDC_G(cudaStreamBeginCaptureToGraph(G->cap, sb[i], nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
        wdc_status ls = launch_pass_ptr(c, mode, (int)i, &G->args[0], G->cap);
        cudaGraph_t got;
        cudaError_t e = cudaStreamEndCapture(G->cap, &got);
        if (ls) return ls;
        if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("skip-pass capture: ") + cudaGetErrorString(e));
    }
    // IF exact: forward + anchor pass
    cudaGraph_t* eb;
    if ((st = add_conditional(c, body, &n_exact, &n_switch, 1, h_exact, cudaGraphCondTypeIf, 1, &eb))) return st;
    {
        WDC_G(cudaStreamBeginCaptureToGraph(G->cap, eb[0], nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
        dit_set_timestep_source(c, &c->st->g_t_model);
        wdc_status fs = dit_forward(c, G->zcur, 0.0f, G->cond, c->vbuf, G->cap);
        dit_set_timestep_source(c, nullptr);
        wdc_status as = fs ? fs : launch_pass_ptr(c, kModeAnchor, 0, &G->args[1], G->cap);
        cudaGraph_t got;
        cudaError_t e = cudaStreamEndCapture(G->cap, &got);
        if (fs) return fs;
        if (as) return as;
        if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("forward capture: ") + cudaGetErrorString(e));
    }
    // IF surrogate: the candidate becomes the current latent
    cudaGraph_t* ab;
    if ((st = add_conditional(c, body, &n_accept, &n_exact, 1, h_accept, cudaGraphCondTypeIf, 1, &ab))) return st;
    {
        cudaGraphNode_t cp;
        WDC_G(cudaGraphAddMemcpyNode1D(&cp, ab[0], nullptr, 0, G->zcur, c->cand[0], c->n * sizeof(float),
                                       cudaMemcpyDeviceToDevice));
    }
    // update
    {
        UpdateArgs u;
        u.st = c->st;
        u.trace = G->trace;
        u.dec = G->dec;
        u.K = K;
        u.T = T;
        u.h_loop = (unsigned long long)h_loop;
        void* params[] = {&u};
        cudaKernelNodeParams kp;
        std::memset(&kp, 0, sizeof(kp));
        kp.func = (void*)update_kernel;
        kp.gridDim = dim3(1);
        kp.blockDim = dim3(32);
        kp.kernelParams = params;
        WDC_G(cudaGraphAddKernelNode(&n_update, body, &n_accept, 1, &kp));
    }
    WDC_G(cudaGraphInstantiate(&G->exec, g, 0));
    G->mode = mode;
    G->K = K;
    G->T = T;
    // the handles go into the per-rollout plan template
    G->h_switch = (unsigned long long)h_switch;
    G->h_exact = (unsigned long long)h_exact;
    G->h_accept = (unsigned long long)h_accept;
    return WDC_OK;
}

wdc_status graph_rollout(Ctx* c, const float* z_T, bool z_dev, const wdc_cond* cd, const float* tokens_dev,
                         float* z_out, bool out_dev, int* decisions, wdc_step_info* trace, cudaStream_t s) {
    const int T = c->sched.T, K = c->prm.bank_capacity;
    const size_t bytes = c->n * sizeof(float);
    if (c->prof) return fail(c, WDC_ERR_UNSUPPORTED, "the graph rollout does not run with the event profiler on");
    if (!c->grollout) {
        GraphRollout* G = new (std::nothrow) GraphRollout();
        if (!G) return WDC_ERR_OOM;
        c->grollout = G;
        WDC_G(cudaStreamCreateWithFlags(&G->cap, cudaStreamNonBlocking));
        WDC_G(cudaMalloc((void**)&G->zcur, bytes));
        const size_t ce = (size_t)c->cfg.cond_tokens * c->cfg.cond_dim;
        WDC_G(cudaMalloc((void**)&G->cond, (ce ? ce : 1) * sizeof(float)));
        WDC_G(cudaMalloc((void**)&G->stepf, T * sizeof(StepScalars)));
        WDC_G(cudaMemcpy(G->stepf, c->stepf.data(), T * sizeof(StepScalars), cudaMemcpyHostToDevice));
        WDC_G(cudaMalloc((void**)&G->args, 2 * sizeof(PassArgs)));
        WDC_G(cudaMalloc((void**)&G->plan, sizeof(PlanArgs)));
        WDC_G(cudaMalloc((void**)&G->trace, T * sizeof(StepOut)));
        WDC_G(cudaMalloc((void**)&G->dec, T * sizeof(int)));
        WDC_G(cudaMalloc((void**)&G->pre, 2 * T * sizeof(int)));
    }
    GraphRollout* G = c->grollout;
    wdc_status st;
    if (!G->exec || G->mode != pass_mode_of(c)) {
        WDC_G(cudaDeviceSynchronize());
        if ((st = build_graph(c, G))) return st;
    }
    // inputs into the graph's fixed buffers
    WDC_G(cudaMemcpyAsync(G->zcur, z_T, bytes, z_dev ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, s));
    const size_t ce = (size_t)c->cfg.cond_tokens * c->cfg.cond_dim;
    if (ce) WDC_G(cudaMemcpyAsync(G->cond, tokens_dev ? tokens_dev : cd->tokens, ce * sizeof(float),
                                  tokens_dev ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, s));
    // this rollout's constants (parameters and descriptors may change between rollouts)
    PlanArgs p;
    std::memset(&p, 0, sizeof(p));
    p.tmpl.n = (long long)c->n;
    p.tmpl.T = T;
    p.tmpl.prm = to_dev_params(c->prm);
    p.tmpl.st = c->st;
    p.tmpl.partials = c->partials;
    p.tmpl.counter = c->counter;
    p.tmpl.err = c->err;
    for (int j = 0; j < 4; ++j) {
        p.tmpl.cam[j] = cd ? cd->cam[j] : 0.0;
        p.tmpl.depth[j] = cd ? cd->depth[j] : 0.0;
    }
    p.tmpl.graph = 1;
    p.tmpl.h_exact = G->h_exact;
    p.tmpl.h_accept = G->h_accept;
    for (int i = 0; i < K; ++i) {
        p.bank[i] = c->bank[i];
        p.disp[i] = c->disp[i];
    }
    p.z_init = c->z_init;
    p.cand = c->cand[0];
    p.zcur = G->zcur;
    p.vbuf = c->vbuf;
    p.stepf = G->stepf;
    p.K = K;
    p.mode = G->mode;
    p.needs_disp = (c->prm.flags & (WDC_ABL_SECANT | WDC_OBS_RESIDUAL)) ? 1 : 0;
    p.skip = &G->args[0];
    p.anchor = &G->args[1];
    p.pre = G->pre;
    p.h_switch = G->h_switch;
    WDC_G(cudaMemcpyAsync(G->plan, &p, sizeof(p), cudaMemcpyHostToDevice, s));
    WDC_G(cudaStreamSynchronize(s));     // the staging struct above is pageable host memory
    // state reset on the current latent, then the discrete state at zero
    if ((st = wdc_state_reset(reinterpret_cast<wdc_ctx*>(c), G->zcur, (wdc_stream)s))) return st;
    WDC_G(cudaMemsetAsync(&c->st->g_k, 0, 4 * sizeof(int), s));
    WDC_G(cudaGraphLaunch(G->exec, s));
    WDC_G(cudaMemcpyAsync(z_out, G->zcur, bytes, out_dev ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost, s));
    std::vector<StepOut> tr(T);
    std::vector<int> dec(T), pre(2 * T);
    int ring[4];
    WDC_G(cudaMemcpyAsync(tr.data(), G->trace, T * sizeof(StepOut), cudaMemcpyDeviceToHost, s));
    WDC_G(cudaMemcpyAsync(dec.data(), G->dec, T * sizeof(int), cudaMemcpyDeviceToHost, s));
    WDC_G(cudaMemcpyAsync(pre.data(), G->pre, 2 * T * sizeof(int), cudaMemcpyDeviceToHost, s));
    WDC_G(cudaMemcpyAsync(ring, &c->st->g_k, 4 * sizeof(int), cudaMemcpyDeviceToHost, s));
    WDC_G(cudaStreamSynchronize(s));
    for (int k = 0; k < T; ++k) {
        if (decisions) decisions[k] = dec[k];
        if (trace) fill_info(tr[k], k, pre[2 * k], pre[2 * k + 1], &trace[k]);
    }
    // the host mirror follows the device state, so the step API can continue
    c->n_bank = ring[1];
    c->head = ring[2];
    c->age = ring[3];
    c->anchor_is_init = c->n_bank == 0;
    c->last_surrogate_k = -1;
    c->cur_latent = G->zcur;
    return WDC_OK;
}

}  // namespace wdc
