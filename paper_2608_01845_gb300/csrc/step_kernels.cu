// Fused, HBM-bound latent passes of the cached rollout.
//
//  * skip pass   (wdc_surrogate_step): per-CTA scalar head = lift summary
//    (Eq. 2), transition retrieval (Eq. 3), scheduler scaling and lifted
//    evolution in summary space (Eq. 4), observation weights (Eq. 5); then one
//    streaming pass z_hat = sum_i kappa_i z_out_i (Eq. 5) that also reduces the
//    statistics the next step's lift needs; the last CTA runs the controller
//    tail: proxy (Eq. 6), risk (Eq. 9), Available and the decision (Eq. 10).
//  * anchor pass (wdc_risk_update): z_exact = Psi(z_k, v) (Eq. 1) written into
//    the bank slot, counterfactual-defect sums (Eq. 7) and the new record's
//    statistics in the same pass; the last CTA calibrates eta_d (Eq. 8),
//    decays R and inserts the record (section "Reliability Decision").
//  * stats pass  (state reset/set): statistics of the current latent and the
//    anchor.
//  * variants of the skip pass's stream: the native latent secant (ablation,
//    z_hat = z_k + alpha (z_a - z_a,in)) and the residual reading of Eq. 5
//    (z_hat = z_k + sum_i kappa_i (z_out_i - z_in_i)); the anchor pass then
//    also stores the slot's displacement z_exact - z_k.
//
// Summary statistics: because the summary's latent blocks are a linear sketch
// S of RMS-normalised vectors, S(nu(z)) = S(z)/(rms(z)+eps_nu) and
// S(nu(z - z_a)) = (S(z) - S(z_a))/(rms(z - z_a)+eps_nu); a pass therefore
// reduces raw signed bucket sums and sums of squares, never a normalised copy.
// The sketch assigns element i to bucket floor(i/128) mod 120 with sign bit 31
// of lowbias32(i ^ seed) (C. Wellons' integer hash), so one warp handles one
// 128-element run = one bucket with 128-bit loads.
//
// Reductions are deterministic: per-warp bucket rows in shared memory, fixed-
// order block combination in fp64, per-block partials, and a last-block-done
// final reduction in fixed order.  No kernel here waits on another CTA.
#include "wdc_internal.h"

#include <cmath>
#include <cstddef>
#include <cstring>
#include <mutex>

namespace wdc {

namespace {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;

__device__ __forceinline__ uint32_t lowbias32(uint32_t x) {
    x ^= x >> 16;
    x *= 0x7feb352du;
    x ^= x >> 15;
    x *= 0x846ca68bu;
    x ^= x >> 16;
    return x;
}

// sign(i) * x: flips the sign bit of x when bit 31 of the hash is set.
__device__ __forceinline__ float signed_term(uint32_t idx, uint32_t seed, float x) {
    uint32_t h = lowbias32(idx ^ seed) & 0x80000000u;
    return __int_as_float(__float_as_int(x) ^ (int)h);
}

// Butterfly sum over the 32 lanes (a fixed-order tree: every lane ends with
// the same value).
// Bulk prefetch of `bytes` (a multiple of 16, 16-byte aligned) into L2.
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
// Runs per warp whose bank reads are prefetched while warp 0 forms the head.
constexpr int kPrefetchRuns = 4;

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Compensated (Kahan) accumulation s += x, c = running compensation.
__device__ __forceinline__ void kahan_add(float& s, float& c, float x) {
    const float y = x - c;
    const float t = s + y;
    c = (t - s) - y;
    s = t;
}

// Sum NV values over the first 256 threads (8 warps) in fixed order; result in
// out[0..NV) (shared).  Every thread of the block must call it.
template <int NV>
__device__ __forceinline__ void reduce256(float (&v)[NV], float* scratch, float* out) {
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
#pragma unroll
    for (int j = 0; j < NV; ++j) v[j] = warp_sum_f(v[j]);
    if (lane == 0 && w < 8) {
#pragma unroll
        for (int j = 0; j < NV; ++j) scratch[w * NV + j] = v[j];
    }
    __syncthreads();
    if (t < NV) {
        const float* s = scratch + t;
        out[t] = ((s[0] + s[NV]) + (s[2 * NV] + s[3 * NV])) + ((s[4 * NV] + s[5 * NV]) + (s[6 * NV] + s[7 * NV]));
    }
    __syncthreads();
}

// fp64 variant of reduce256 (the linear observation's ill-conditioned ridge
// system only).
template <int NV>
__device__ __forceinline__ void reduce256d(double (&v)[NV], double* scratch, double* out) {
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
#pragma unroll
    for (int j = 0; j < NV; ++j)
#pragma unroll
        for (int o = 16; o; o >>= 1) v[j] += __shfl_xor_sync(0xffffffffu, v[j], o);
    if (lane == 0 && w < 8) {
#pragma unroll
        for (int j = 0; j < NV; ++j) scratch[w * NV + j] = v[j];
    }
    __syncthreads();
    if (t < NV) {
        double acc = 0.0;
        for (int q = 0; q < 8; ++q) acc += scratch[q * NV + t];
        out[t] = acc;
    }
    __syncthreads();
}

// The part of the device state a pass reads, copied into shared memory by all
// threads at the start in one batch of independent loads; the head and the
// tails then work from shared memory.  (Read in place, the head and the
// controller tail were chains of dependent L2 round trips -- the state may sit
// in the other die's half of L2 -- that cost about 10 us per launch.)
struct alignas(16) StateIn {
    float cur_S[kSketch], anchor_S[kSketch];
    float s_phi[kSummary];                 // anchor pass: the pre-insertion summary
    float n_in[kMaxBank], n_out[kMaxBank]; // records by age (oldest first)
    float q_in[kMaxBank], dq[kMaxBank], r[kMaxBank];
    float cur_sumsq, cur_sumsq_anchor, anchor_sumsq, R, eta, q_a_out, q_a_dq, cand_p;
    float cam_a[4], depth_a[4];
    int cand_k, cand_supported, cand_finite;
};
// The records' summaries by age; shares storage with the stream's bucket
// rows, which are used only after the head.
struct alignas(16) RecSummaries {
    float s_in[kMaxBank][kSummary], s_out[kMaxBank][kSummary], s_dphi[kMaxBank][kSummary];
};

struct HeadShared {
    float phi[kSummary];
    float hat[kSummary];
    float scratch[8 * (kMaxBank + 1)];
    float red[kMaxBank + 1];
    double dscratch[8 * kMaxBank];          // linear observation: fp64 reduction scratch
    double gram[kMaxBank + 1][kMaxBank];    // linear observation: the records' Gram matrix, then S_out s_hat
    float sim_in[kMaxBank], sim_out[kMaxBank], pi[kMaxBank], kappa[kMaxBank];
    float alpha;
    int compat[kMaxBank];
    int n_compat, supported;
};

// Linear observation (ablation): kappa <- beta, the ridge least-squares
// coefficients of s(phi_hat) on the records' output summaries,
// (G + rho I) beta = S_out s_hat with G_ij = s_out_i . s_out_j and
// rho = ridge * trace(G) / K, solved by Cholesky in fp64 (G + rho I is
// positive definite for rho > 0).  The system is ill-conditioned at a small
// ridge, so G and S_out s_hat are reduced in fp64 here.
template <int K>
__device__ __noinline__ void linear_readout(const PassArgs& a, const RecSummaries& rs, HeadShared& hs) {
    if constexpr (K > 0) {
        const int t = threadIdx.x;
        // one row of G per reduction (keeps K values per thread); row K = S_out s_hat
        for (int i = 0; i <= K; ++i) {
            double v[K];
            const double si = (t < kSummary) ? (i < K ? (double)rs.s_out[i][t] : (double)hs.hat[t]) : 0.0;
#pragma unroll
            for (int j = 0; j < K; ++j) v[j] = (t < kSummary) ? si * (double)rs.s_out[j][t] : 0.0;
            reduce256d<K>(v, hs.dscratch, hs.gram[i]);
        }
        double b[K];
        if (t == 0) {
#pragma unroll
            for (int i = 0; i < K; ++i) b[i] = hs.gram[K][i];
        }
        if (t == 0) {
            double A[K][K];
            double tr = 0.0;
            for (int i = 0; i < K; ++i) {
                for (int j = 0; j < K; ++j) A[i][j] = 0.5 * (hs.gram[i][j] + hs.gram[j][i]);
                tr += A[i][i];
            }
            if (tr == 0.0) {
#pragma unroll
                for (int i = 0; i < K; ++i) hs.kappa[i] = 0.f;
            } else {
                const double rho = (double)a.prm.ridge * tr / K;
#pragma unroll
                for (int i = 0; i < K; ++i) A[i][i] += rho;
                // Cholesky A = L L^T (L in the lower triangle of A)
                for (int j = 0; j < K; ++j) {
                    double d = A[j][j];
                    for (int m = 0; m < j; ++m) d -= A[j][m] * A[j][m];
                    d = sqrt(d);
                    A[j][j] = d;
                    for (int i = j + 1; i < K; ++i) {
                        double x = A[i][j];
                        for (int m = 0; m < j; ++m) x -= A[i][m] * A[j][m];
                        A[i][j] = x / d;
                    }
                }
                double y[K], beta[K];
                for (int i = 0; i < K; ++i) {
                    double x = b[i];
                    for (int m = 0; m < i; ++m) x -= A[i][m] * y[m];
                    y[i] = x / A[i][i];
                }
                for (int i = K - 1; i >= 0; --i) {
                    double x = y[i];
                    for (int m = i + 1; m < K; ++m) x -= A[m][i] * beta[m];
                    beta[i] = x / A[i][i];
                }
                for (int i = 0; i < K; ++i) hs.kappa[i] = (float)beta[i];
            }
        }
        __syncthreads();
    }
}

// Skip-pass head, Eq. 2-5 scalar part, in fp32, run by one warp of every CTA
// (so no CTA waits for another): lane l owns the summary entries l, l+32, ...,
// every dot product is a lane-local sum followed by a butterfly, and every
// lane then holds the totals, so each lane evaluates the small softmaxes of
// Eq. 3 and 5 itself and no block barrier is needed.  (Spread over 256
// threads with block reductions, the same head took ~9k cycles, most of it in
// barriers.)  The head and the controller tails are one chain of dependent
// scalar steps per launch, so they use the fast division and exponential
// intrinsics (a few ulp; the tolerances are 1e-5).  Writes hs.phi, hs.hat,
// hs.alpha and, for K > 0, hs.sim_in/sim_out/compat/pi/kappa/n_compat/
// supported; the caller synchronises the block afterwards.
template <int K>
__device__ void skip_head_warp(const PassArgs& a, const StateIn& S, const RecSummaries& rs, HeadShared& hs) {
    constexpr int J = kSummary / 32;                  // entries per lane
    const int lane = threadIdx.x & 31;
    const float N = (float)a.n;
    const float sc = sqrtf(__fdividef((float)kSketch, N));
    const float eps_nu = a.prm.eps_nu;
    const bool no_cond = a.prm.flags & WDC_ABL_NO_COND;
    const float inv_cur = __fdividef(sc, sqrtf(__fdividef(S.cur_sumsq, N)) + eps_nu);
    const float inv_dz = __fdividef(sc, sqrtf(__fdividef(S.cur_sumsq_anchor, N)) + eps_nu);
    // s(phi_k): current-state summary (Eq. 2 through the linear sketch)
    float ph[J];
#pragma unroll
    for (int j = 0; j < J; ++j) {
        const int t = lane + 32 * j;
        float val;
        if (t < kSketch) {
            val = S.cur_S[t] * inv_cur;
        } else if (t < 2 * kSketch) {
            const int b = t - kSketch;
            val = (S.cur_S[b] - S.anchor_S[b]) * inv_dz;
        } else if (t < kOffDepth) {
            val = no_cond ? 0.f : a.cam[t - kOffCam];
        } else if (t < kOffQ) {
            val = no_cond ? 0.f : a.depth[t - kOffDepth];
        } else if (t == kOffQ) {
            val = a.sk.q_k;
        } else {
            // h(H): [r_1..3, T*(q_in - q_out)_1..3, n_bank/K], newest record first
            const int h = t - kOffH;
            val = 0.f;
            if (h < 3) {
                if (h < a.nsrc) val = S.r[a.nsrc - 1 - h];
            } else if (h < 6) {
                if (h - 3 < a.nsrc) val = -(float)a.T * S.dq[a.nsrc - 1 - (h - 3)];
            } else {
                val = __fdividef((float)a.nsrc, (float)a.prm.K);
            }
        }
        ph[j] = val;
        hs.phi[t] = val;
    }
    // Eq. 4: alpha = clip(|q_{t-1}-q_t| / (|q_{a-1}-q_a| + eps), alpha_min, alpha_max)
    const float alpha =
        fminf(fmaxf(__fdividef(fabsf(a.sk.dq), fabsf(S.q_a_dq) + a.prm.eps), a.prm.alpha_min), a.prm.alpha_max);
    if (lane == 0) hs.alpha = alpha;
    if constexpr (K > 0) {
        // Eq. 3: similarities with the records' lifted inputs
        float d[K + 1];
#pragma unroll
        for (int i = 0; i <= K; ++i) d[i] = 0.f;
#pragma unroll
        for (int j = 0; j < J; ++j) {
            const int t = lane + 32 * j;
#pragma unroll
            for (int i = 0; i < K; ++i) d[i] = fmaf(ph[j], rs.s_in[i][t], d[i]);
            d[K] = fmaf(ph[j], ph[j], d[K]);
        }
#pragma unroll
        for (int i = 0; i <= K; ++i) d[i] = warp_sum_f(d[i]);
        const float nphi = sqrtf(d[K]);
        const bool filter = !(a.prm.flags & WDC_ABL_NO_SUPPORT);   // w/o support: N_t = whole bank
        const float gq = a.prm.gamma_q, inv_tin = __fdividef(1.0f, a.prm.tau_in);
        int nc = 0;
        float mx = -INFINITY, ell[K], pi[K], sim[K];
        bool compat[K];
#pragma unroll
        for (int i = 0; i < K; ++i) {
            sim[i] = (nphi == 0.f || S.n_in[i] == 0.f) ? 0.f : __fdividef(d[i], nphi * S.n_in[i]);
            const float dq = a.sk.q_k - S.q_in[i];
            compat[i] = !filter || ((sim[i] >= a.prm.sim_min) && (fabsf(dq) <= a.prm.q_gap_max));
            ell[i] = (sim[i] - gq * dq * dq) * inv_tin;
            if (compat[i]) { ++nc; mx = fmaxf(mx, ell[i]); }
        }
        float tot = 0.f;
#pragma unroll
        for (int i = 0; i < K; ++i) {
            pi[i] = compat[i] ? __expf(ell[i] - mx) : 0.f;
            tot += pi[i];
        }
        const float inv_tot = nc > 0 ? __fdividef(1.0f, tot) : 0.f;
#pragma unroll
        for (int i = 0; i < K; ++i) pi[i] *= inv_tot;
        // Eq. 4 in summary space, then Eq. 5 similarities with the lifted outputs
        float e[K + 1];
#pragma unroll
        for (int i = 0; i <= K; ++i) e[i] = 0.f;
#pragma unroll
        for (int j = 0; j < J; ++j) {
            const int t = lane + 32 * j;
            float acc = 0.f;
#pragma unroll
            for (int i = 0; i < K; ++i)
                if (pi[i] != 0.f) acc = fmaf(pi[i], rs.s_dphi[i][t], acc);
            const float hv = fmaf(alpha, acc, ph[j]);
            hs.hat[t] = hv;
#pragma unroll
            for (int i = 0; i < K; ++i) e[i] = fmaf(hv, rs.s_out[i][t], e[i]);
            e[K] = fmaf(hv, hv, e[K]);
        }
#pragma unroll
        for (int i = 0; i <= K; ++i) e[i] = warp_sum_f(e[i]);
        const float nh = sqrtf(e[K]);
        const float inv_tau = __fdividef(1.0f, a.prm.tau_obs);
        float so[K];
        float mo = -INFINITY;
#pragma unroll
        for (int i = 0; i < K; ++i) {
            so[i] = (nh == 0.f || S.n_out[i] == 0.f) ? 0.f : __fdividef(e[i], nh * S.n_out[i]);
            e[i] = so[i] * inv_tau;
            mo = fmaxf(mo, e[i]);
        }
        float to = 0.f;
#pragma unroll
        for (int i = 0; i < K; ++i) { e[i] = __expf(e[i] - mo); to += e[i]; }
        const float inv = __fdividef(1.0f, to);
        if (lane == 0) {
#pragma unroll
            for (int i = 0; i < K; ++i) {
                hs.sim_in[i] = sim[i];
                hs.compat[i] = compat[i];
                hs.pi[i] = pi[i];
                hs.sim_out[i] = so[i];
                hs.kappa[i] = e[i] * inv;
            }
            hs.n_compat = nc;
            hs.supported = filter ? (nc >= a.prm.min_support) : 1;
        }
    }
}

// Per-block scalar slots: the stream's five sums and the non-finite count.
constexpr int kScalars = 6;
// Most blocks one pass launch may have (the final reduction's register tile).
constexpr int kMaxPassBlocks = 256;

// 16-byte aligned: load_state stores float4 values into the snapshot arrays.
struct alignas(16) PassShared {
    union {
        float wb[2][kWarps][kSketch]; // per-warp bucket rows (2 sketches for the stats pass)
        RecSummaries rs;              // the head's record summaries (before the stream)
    };
    float blk[kWarps][kScalars];
    float fin[kPartials];
    StateIn S;
    int last;
};

static_assert(alignof(PassShared) >= 16 && alignof(StateIn) >= 16 && alignof(RecSummaries) >= 16,
              "float4 snapshot stores need 16-byte aligned shared arrays");
static_assert(offsetof(PassShared, S) % 16 == 0 && offsetof(PassShared, rs) == 0, "snapshot offsets");
static_assert(sizeof(PassArgs) % 8 == 0 && alignof(PassArgs) <= 16, "the argument copy moves whole words");
static_assert(offsetof(StateIn, cur_S) % 16 == 0 && offsetof(StateIn, anchor_S) % 16 == 0 &&
              offsetof(StateIn, s_phi) % 16 == 0, "snapshot vector offsets");
static_assert((kSummary * sizeof(float)) % 16 == 0, "summary rows stay 16-byte aligned");
static_assert(offsetof(DevRecord, s_in) % 16 == 0 && offsetof(DevRecord, s_out) % 16 == 0 &&
              offsetof(DevRecord, s_dphi) % 16 == 0 && sizeof(DevRecord) % 16 == 0, "record layout");
static_assert(offsetof(DevState, rec) % 16 == 0 && offsetof(DevState, cur_S) % 16 == 0 &&
              offsetof(DevState, anchor_S) % 16 == 0 && offsetof(DevState, s_phi) % 16 == 0, "state layout");

// Copies what this mode reads of the device state into shared memory (one
// batch of independent loads spread over the block's threads).
template <int MODE>
__device__ __forceinline__ void load_state(const PassArgs& a, PassShared& ps) {
    const DevState* st = a.st;
    const int t = threadIdx.x;
    StateIn& S = ps.S;
    const bool head = MODE == kModeSkip || MODE == kModeResidual || MODE == kModeSecant;
    if (MODE == kModeSkip || MODE == kModeResidual) {
        // summaries of the nsrc records by age: 3 arrays x 64 float4 each
        for (int idx = t; idx < a.nsrc * 192; idx += kThreads) {
            const int i = idx / 192, rem = idx - i * 192, which = rem >> 6, c = rem & 63;
            const DevRecord& R = st->rec[a.slot[i]];
            const float* src = which == 0 ? R.s_in : (which == 1 ? R.s_out : R.s_dphi);
            float* dst = which == 0 ? ps.rs.s_in[i] : (which == 1 ? ps.rs.s_out[i] : ps.rs.s_dphi[i]);
            reinterpret_cast<float4*>(dst)[c] = __ldcg(reinterpret_cast<const float4*>(src) + c);
        }
    }
    if (head || MODE == kModeAnchor) {
        const int u = t - 384;                   // threads 384.. take the vectors and scalars
        if (u >= 0 && u < 30) reinterpret_cast<float4*>(S.cur_S)[u] = __ldcg(reinterpret_cast<const float4*>(st->cur_S) + u);
        else if (u >= 32 && u < 62)
            reinterpret_cast<float4*>(S.anchor_S)[u - 32] = __ldcg(reinterpret_cast<const float4*>(st->anchor_S) + (u - 32));
        else if (MODE == kModeAnchor && u >= 64 && u < 128)
            reinterpret_cast<float4*>(S.s_phi)[u - 64] = __ldcg(reinterpret_cast<const float4*>(st->s_phi) + (u - 64));
        else if (u >= 128 && u < 128 + kMaxBank) {
            const int i = u - 128;
            if (i < a.nsrc) {
                const DevRecord& R = st->rec[a.slot[i]];
                S.n_in[i] = __ldcg(&R.n_in);
                S.n_out[i] = __ldcg(&R.n_out);
                S.q_in[i] = __ldcg(&R.q_in);
                S.dq[i] = __ldcg(&R.dq);
                S.r[i] = __ldcg(&R.r);
            }
        } else if (u >= 160 && u < 168) {
            const int j = u - 160;
            if (j < 4) S.cam_a[j] = __ldcg(&st->cam_a[j]);
            else S.depth_a[j - 4] = __ldcg(&st->depth_a[j - 4]);
        } else if (u == 168) S.cur_sumsq = __ldcg(&st->cur_sumsq);
        else if (u == 169) S.cur_sumsq_anchor = __ldcg(&st->cur_sumsq_anchor);
        else if (u == 170) S.anchor_sumsq = __ldcg(&st->anchor_sumsq);
        else if (u == 171) S.R = __ldcg(&st->R);
        else if (u == 172) S.eta = __ldcg(&st->eta);
        else if (u == 173) S.q_a_dq = __ldcg(&st->q_a_dq);
        else if (u == 174) S.q_a_out = __ldcg(&st->q_a_out);
        else if (u == 175) S.cand_p = __ldcg(&st->cand_p);
        else if (u == 176) S.cand_k = __ldcg(&st->cand_k);
        else if (u == 177) S.cand_supported = __ldcg(&st->cand_supported);
        else if (u == 178) S.cand_finite = __ldcg(&st->cand_finite);
    }
}

// Sum over the 32 warps' rows of one bucket, in a fixed pairwise order.
__device__ __forceinline__ float sum_warp_rows(const float (&rows)[kWarps][kSketch], int b) {
    float x[kWarps];
#pragma unroll
    for (int w = 0; w < kWarps; ++w) x[w] = rows[w][b];
#pragma unroll
    for (int h = kWarps / 2; h; h >>= 1)
#pragma unroll
        for (int w = 0; w < h; ++w) x[w] += x[w + h];
    return x[0];
}

template <int MODE, int K>
__device__ __forceinline__ void pass_body(const PassArgs& a_in) {
    __shared__ HeadShared hs;
    __shared__ PassShared ps;
    // The launch arguments, copied into shared memory by all threads at once:
    // read in place, every newly touched line of the ~0.6 KB argument block
    // is a miss of its own, and the head's and the controller tail's scalar
    // chains walk many of them one after another (several microseconds per
    // launch, measured).
    __shared__ __align__(16) uint32_t s_args[(sizeof(PassArgs) + 3) / 4];
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    for (int i = t; i < (int)((sizeof(PassArgs) + 3) / 4); i += kThreads)
        s_args[i] = reinterpret_cast<const uint32_t*>(&a_in)[i];
    __syncthreads();
    const PassArgs& a = *reinterpret_cast<const PassArgs*>(s_args);
    const uint32_t seed = a.prm.seed;
    const long long n = a.n;
    const long long nruns = (n + kRun - 1) / kRun;
    const long long full = n / kRun;

    load_state<MODE>(a, ps);
    __syncthreads();

    bool do_stream = true;
    float kap[K > 0 ? K : 1];
    float alpha_f = 0.f;
    if constexpr ((MODE == kModeSkip || MODE == kModeResidual || MODE == kModeObserve) && K > 0) {
        // while warp 0 forms the head, the other warps start the HBM reads of
        // their first runs (into L2): lane i < K takes bank record i, lane K
        // the anchor (observe / residual) or the current latent (residual)
        if (warp != 0 && lane <= K) {
            const float* src = lane < K ? a.src[lane] : (MODE == kModeSkip ? nullptr : a.anchor);
            const long long gw = (long long)blockIdx.x * kWarps + warp;
            const long long stride = (long long)gridDim.x * kWarps;
            if (src) {
                for (int it = 0; it < kPrefetchRuns; ++it) {
                    const long long r = gw + it * stride;
                    if (r >= full) break;
                    prefetch_l2(src + r * kRun, kRun * 4);
                }
            }
        }
    }
    if (MODE == kModeSkip || MODE == kModeResidual) {
        if (warp == 0) skip_head_warp<K>(a, ps.S, ps.rs, hs);
        __syncthreads();
        if (a.prm.flags & WDC_ABL_LINEAR_OBS) linear_readout<K>(a, ps.rs, hs);
        do_stream = (K > 0) && hs.supported;
#pragma unroll
        for (int i = 0; i < K; ++i) kap[i] = hs.kappa[i];
    } else if (MODE == kModeSecant) {
        if (warp == 0) skip_head_warp<0>(a, ps.S, ps.rs, hs);   // lift summary and alpha only: no retrieval
        __syncthreads();
        do_stream = a.nsrc > 0;
        alpha_f = hs.alpha;
    } else if (MODE == kModeObserve) {
#pragma unroll
        for (int i = 0; i < K; ++i) kap[i] = a.kappa[i];
    }
    // the bucket rows share storage with the record summaries the head read
    for (int i = t; i < 2 * kWarps * kSketch; i += kThreads) (&ps.wb[0][0][0])[i] = 0.f;
    __syncthreads();

    // per-thread accumulators: plain fp32 over up to 16 runs (64 terms), then
    // a compensated fp32 outer sum
    float acc[5] = {0, 0, 0, 0, 0}, cmp[5] = {0, 0, 0, 0, 0};
    float fac[5] = {0, 0, 0, 0, 0};
    int nonfinite = 0;
    int since = 0;
    const float dsig = a.sk.dq;

    if (do_stream) {
        const long long gw = (long long)blockIdx.x * kWarps + warp;
        const long long stride = (long long)gridDim.x * kWarps;
        long long r = gw;
        if constexpr ((MODE == kModeSkip || MODE == kModeObserve) && K > 0) {
            // two full runs per iteration: both runs' loads are in flight
            // together (a bank of two records alone keeps too few bytes in
            // flight per SM to cover the HBM latency)
            auto stats = [&](const float4& zh, const float4& za, long long base, long long rr) {
                const float ov[4] = {zh.x, zh.y, zh.z, zh.w};
                const float av[4] = {za.x, za.y, za.z, za.w};
                float sg = 0.f;
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float d = ov[e] - av[e];
                    sg += signed_term((uint32_t)(base + e), seed, ov[e]);
                    fac[0] = fmaf(ov[e], ov[e], fac[0]);
                    fac[1] = fmaf(d, d, fac[1]);
                    nonfinite += isfinite(ov[e]) ? 0 : 1;
                }
                sg = warp_sum_f(sg);
                if (lane == 0) ps.wb[0][warp][(int)(rr % kSketch)] += sg;
            };
            for (; r + stride < full; r += 2 * stride) {
                const long long b0 = r * kRun + lane * 4, b1 = (r + stride) * kRun + lane * 4;
                float4 x0[K], x1[K], za0, za1;
#pragma unroll
                for (int i = 0; i < K; ++i) {
                    x0[i] = __ldg(reinterpret_cast<const float4*>(a.src[i] + b0));
                    x1[i] = __ldg(reinterpret_cast<const float4*>(a.src[i] + b1));
                }
                if constexpr (MODE == kModeObserve) {
                    za0 = __ldg(reinterpret_cast<const float4*>(a.anchor + b0));
                    za1 = __ldg(reinterpret_cast<const float4*>(a.anchor + b1));
                } else {
                    za0 = x0[K - 1];             // the anchor is the newest record
                    za1 = x1[K - 1];
                }
                float4 z0, z1;
                z0.x = kap[0] * x0[0].x; z0.y = kap[0] * x0[0].y; z0.z = kap[0] * x0[0].z; z0.w = kap[0] * x0[0].w;
                z1.x = kap[0] * x1[0].x; z1.y = kap[0] * x1[0].y; z1.z = kap[0] * x1[0].z; z1.w = kap[0] * x1[0].w;
#pragma unroll
                for (int i = 1; i < K; ++i) {
                    z0.x = fmaf(kap[i], x0[i].x, z0.x); z0.y = fmaf(kap[i], x0[i].y, z0.y);
                    z0.z = fmaf(kap[i], x0[i].z, z0.z); z0.w = fmaf(kap[i], x0[i].w, z0.w);
                    z1.x = fmaf(kap[i], x1[i].x, z1.x); z1.y = fmaf(kap[i], x1[i].y, z1.y);
                    z1.z = fmaf(kap[i], x1[i].z, z1.z); z1.w = fmaf(kap[i], x1[i].w, z1.w);
                }
                *reinterpret_cast<float4*>(a.out + b0) = z0;
                *reinterpret_cast<float4*>(a.out + b1) = z1;
                stats(z0, za0, b0, r);
                stats(z1, za1, b1, r + stride);
                since += 2;
                if (since >= 16) {
#pragma unroll
                    for (int j = 0; j < 5; ++j) { kahan_add(acc[j], cmp[j], fac[j]); fac[j] = 0.f; }
                    since = 0;
                }
            }
        }
        for (; r < nruns; r += stride) {
            const long long base = r * kRun + lane * 4;
            float o[4], sa[4], sb[4];   // o: primary value, sa/sb: stats-pass anchor
            bool valid[4];
            if (r < full) {
#pragma unroll
                for (int e = 0; e < 4; ++e) valid[e] = true;
                if constexpr (MODE == kModeSkip && K > 0) {
                    float4 x[K];
#pragma unroll
                    for (int i = 0; i < K; ++i) x[i] = __ldg(reinterpret_cast<const float4*>(a.src[i] + base));
                    float4 zh;
                    zh.x = kap[0] * x[0].x; zh.y = kap[0] * x[0].y; zh.z = kap[0] * x[0].z; zh.w = kap[0] * x[0].w;
#pragma unroll
                    for (int i = 1; i < K; ++i) {
                        zh.x = fmaf(kap[i], x[i].x, zh.x); zh.y = fmaf(kap[i], x[i].y, zh.y);
                        zh.z = fmaf(kap[i], x[i].z, zh.z); zh.w = fmaf(kap[i], x[i].w, zh.w);
                    }
                    *reinterpret_cast<float4*>(a.out + base) = zh;
                    o[0] = zh.x; o[1] = zh.y; o[2] = zh.z; o[3] = zh.w;
                    sa[0] = x[K - 1].x; sa[1] = x[K - 1].y; sa[2] = x[K - 1].z; sa[3] = x[K - 1].w;
                } else if constexpr (MODE == kModeObserve && K > 0) {
                    float4 x[K];
#pragma unroll
                    for (int i = 0; i < K; ++i) x[i] = __ldg(reinterpret_cast<const float4*>(a.src[i] + base));
                    const float4 za = __ldg(reinterpret_cast<const float4*>(a.anchor + base));
                    float4 zh;
                    zh.x = kap[0] * x[0].x; zh.y = kap[0] * x[0].y; zh.z = kap[0] * x[0].z; zh.w = kap[0] * x[0].w;
#pragma unroll
                    for (int i = 1; i < K; ++i) {
                        zh.x = fmaf(kap[i], x[i].x, zh.x); zh.y = fmaf(kap[i], x[i].y, zh.y);
                        zh.z = fmaf(kap[i], x[i].z, zh.z); zh.w = fmaf(kap[i], x[i].w, zh.w);
                    }
                    *reinterpret_cast<float4*>(a.out + base) = zh;
                    o[0] = zh.x; o[1] = zh.y; o[2] = zh.z; o[3] = zh.w;
                    sa[0] = za.x; sa[1] = za.y; sa[2] = za.z; sa[3] = za.w;
                } else if constexpr (MODE == kModeResidual && K > 0) {
                    // residual reading: z_hat = z_k + sum_i kappa_i (z_out_i - z_in_i)
                    float4 zh = __ldg(reinterpret_cast<const float4*>(a.zcur + base));
                    const float4 za = __ldg(reinterpret_cast<const float4*>(a.anchor + base));
#pragma unroll
                    for (int i = 0; i < K; ++i) {
                        const float4 d = __ldg(reinterpret_cast<const float4*>(a.src[i] + base));
                        zh.x = fmaf(kap[i], d.x, zh.x); zh.y = fmaf(kap[i], d.y, zh.y);
                        zh.z = fmaf(kap[i], d.z, zh.z); zh.w = fmaf(kap[i], d.w, zh.w);
                    }
                    *reinterpret_cast<float4*>(a.out + base) = zh;
                    o[0] = zh.x; o[1] = zh.y; o[2] = zh.z; o[3] = zh.w;
                    sa[0] = za.x; sa[1] = za.y; sa[2] = za.z; sa[3] = za.w;
                } else if constexpr (MODE == kModeSecant) {
                    // native latent secant: z_hat = z_k + alpha (z_a - z_a,in)
                    const float4 z = __ldg(reinterpret_cast<const float4*>(a.src[0] + base));
                    const float4 dz = __ldg(reinterpret_cast<const float4*>(a.src[1] + base));
                    const float4 za = __ldg(reinterpret_cast<const float4*>(a.anchor + base));
                    float4 zh;
                    zh.x = fmaf(alpha_f, dz.x, z.x); zh.y = fmaf(alpha_f, dz.y, z.y);
                    zh.z = fmaf(alpha_f, dz.z, z.z); zh.w = fmaf(alpha_f, dz.w, z.w);
                    *reinterpret_cast<float4*>(a.out + base) = zh;
                    o[0] = zh.x; o[1] = zh.y; o[2] = zh.z; o[3] = zh.w;
                    sa[0] = za.x; sa[1] = za.y; sa[2] = za.z; sa[3] = za.w;
                } else if constexpr (MODE == kModeAnchor) {
                    // plain loads: z_k / z_a may alias the slot written below (bank capacity 1)
                    const float4 z = *reinterpret_cast<const float4*>(a.src[0] + base);
                    const float4 v = *reinterpret_cast<const float4*>(a.v + base);
                    const float4 za = *reinterpret_cast<const float4*>(a.anchor + base);
                    float4 ze;
                    ze.x = fmaf(dsig, v.x, z.x); ze.y = fmaf(dsig, v.y, z.y);
                    ze.z = fmaf(dsig, v.z, z.z); ze.w = fmaf(dsig, v.w, z.w);
                    *reinterpret_cast<float4*>(a.out + base) = ze;
                    if (a.out3) *reinterpret_cast<float4*>(a.out3 + base) = ze;
                    if (a.out2) {
                        float4 dz;
                        dz.x = ze.x - z.x; dz.y = ze.y - z.y; dz.z = ze.z - z.z; dz.w = ze.w - z.w;
                        *reinterpret_cast<float4*>(a.out2 + base) = dz;
                    }
                    o[0] = ze.x; o[1] = ze.y; o[2] = ze.z; o[3] = ze.w;
                    sa[0] = za.x; sa[1] = za.y; sa[2] = za.z; sa[3] = za.w;
                    sb[0] = z.x; sb[1] = z.y; sb[2] = z.z; sb[3] = z.w;
                    if (a.zcf) {
                        const float4 c = *reinterpret_cast<const float4*>(a.zcf + base);
                        fac[0] += (fabsf(ze.x - c.x) + fabsf(ze.y - c.y)) + (fabsf(ze.z - c.z) + fabsf(ze.w - c.w));
                    }
                } else if constexpr (MODE == kModeStats) {
                    const float4 z = __ldg(reinterpret_cast<const float4*>(a.src[0] + base));
                    const float4 za = __ldg(reinterpret_cast<const float4*>(a.anchor + base));
                    o[0] = z.x; o[1] = z.y; o[2] = z.z; o[3] = z.w;
                    sa[0] = za.x; sa[1] = za.y; sa[2] = za.z; sa[3] = za.w;
                }
            } else {
                // ragged last run: scalar, bounds-checked
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const long long idx = base + e;
                    valid[e] = idx < n;
                    o[e] = 0.f; sa[e] = 0.f; sb[e] = 0.f;
                    if (!valid[e]) continue;
                    if constexpr (MODE == kModeSkip && K > 0) {
                        float zh = kap[0] * a.src[0][idx];
#pragma unroll
                        for (int i = 1; i < K; ++i) zh = fmaf(kap[i], a.src[i][idx], zh);
                        a.out[idx] = zh;
                        o[e] = zh;
                        sa[e] = a.src[K - 1][idx];
                    } else if constexpr (MODE == kModeObserve && K > 0) {
                        float zh = kap[0] * a.src[0][idx];
#pragma unroll
                        for (int i = 1; i < K; ++i) zh = fmaf(kap[i], a.src[i][idx], zh);
                        a.out[idx] = zh;
                        o[e] = zh;
                        sa[e] = a.anchor[idx];
                    } else if constexpr (MODE == kModeResidual && K > 0) {
                        float zh = a.zcur[idx];
#pragma unroll
                        for (int i = 0; i < K; ++i) zh = fmaf(kap[i], a.src[i][idx], zh);
                        a.out[idx] = zh;
                        o[e] = zh;
                        sa[e] = a.anchor[idx];
                    } else if constexpr (MODE == kModeSecant) {
                        const float zh = fmaf(alpha_f, a.src[1][idx], a.src[0][idx]);
                        a.out[idx] = zh;
                        o[e] = zh;
                        sa[e] = a.anchor[idx];
                    } else if constexpr (MODE == kModeAnchor) {
                        // read z_k and z_a before the store: they may alias the slot
                        const float z = a.src[0][idx];
                        const float za = a.anchor[idx];
                        const float ze = fmaf(dsig, a.v[idx], z);
                        a.out[idx] = ze;
                        if (a.out3) a.out3[idx] = ze;
                        if (a.out2) a.out2[idx] = ze - z;
                        o[e] = ze;
                        sa[e] = za;
                        sb[e] = z;
                        if (a.zcf) fac[0] += fabsf(ze - a.zcf[idx]);
                    } else if constexpr (MODE == kModeStats) {
                        o[e] = a.src[0][idx];
                        sa[e] = a.anchor[idx];
                    }
                }
            }
            // statistics of the primary value
            float sg = 0.f, sg2 = 0.f;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                if (!valid[e]) continue;
                const float x = o[e];
                const float d = x - sa[e];
                const uint32_t idx = (uint32_t)(base + e);
                sg += signed_term(idx, seed, x);
                if (MODE == kModeSkip || MODE == kModeObserve || MODE == kModeSecant || MODE == kModeResidual) {
                    fac[0] = fmaf(x, x, fac[0]);
                    fac[1] = fmaf(d, d, fac[1]);
                    nonfinite += isfinite(x) ? 0 : 1;
                } else if (MODE == kModeAnchor) {
                    fac[1] += fabsf(x);
                    fac[2] = fmaf(x, x, fac[2]);
                    fac[3] = fmaf(d, d, fac[3]);
                    const float dz = x - sb[e];
                    fac[4] = fmaf(dz, dz, fac[4]);
                } else {
                    fac[0] = fmaf(x, x, fac[0]);
                    fac[1] = fmaf(d, d, fac[1]);
                    fac[2] = fmaf(sa[e], sa[e], fac[2]);
                    sg2 += signed_term(idx, seed, sa[e]);
                }
            }
            sg = warp_sum_f(sg);
            const int bucket = (int)(r % kSketch);
            if (lane == 0) ps.wb[0][warp][bucket] += sg;
            if (MODE == kModeStats) {
                sg2 = warp_sum_f(sg2);
                if (lane == 0) ps.wb[1][warp][bucket] += sg2;
            }
            if (++since >= 16) {
#pragma unroll
                for (int j = 0; j < 5; ++j) { kahan_add(acc[j], cmp[j], fac[j]); fac[j] = 0.f; }
                since = 0;
            }
        }
    }
    float sum[kScalars];
#pragma unroll
    for (int j = 0; j < 5; ++j) {
        kahan_add(acc[j], cmp[j], fac[j]);
        sum[j] = acc[j] - cmp[j];
    }
    sum[5] = (float)nonfinite;

    // block combination (fixed order): warp trees, then a tree over the warps
#pragma unroll
    for (int j = 0; j < kScalars; ++j) sum[j] = warp_sum_f(sum[j]);
    if (lane == 0) {
#pragma unroll
        for (int j = 0; j < kScalars; ++j) ps.blk[warp][j] = sum[j];
    }
    __syncthreads();
    // partials are value-major, [kPartials][gridDim.x], so the last block
    // reads each value's per-block entries with coalesced loads
    const int G = gridDim.x;
    float* part = a.partials + blockIdx.x;
    const int nsk = (MODE == kModeStats) ? 2 : 1;       // sketches reduced by this mode
    if (t < nsk * kSketch) {
        part[(size_t)t * G] = sum_warp_rows(ps.wb[t / kSketch], t % kSketch);
    } else if (warp == kWarps - 1) {
        // the last warp: one lane per warp row, a butterfly per scalar
#pragma unroll
        for (int j = 0; j < kScalars; ++j) {
            const float v = warp_sum_f(ps.blk[lane][j]);
            if (lane == 0) part[(size_t)(2 * kSketch + j) * G] = v;
        }
    }
    __threadfence();
    __syncthreads();
    if (t == 0) {
        const unsigned prev = atomicAdd(a.counter, 1u);
        ps.last = (prev == gridDim.x - 1);
    }
    __syncthreads();
    if (!ps.last) return;
    __threadfence();

    // final reduction over the blocks, fixed order: each warp takes values
    // w, w + 32, ...; lane l sums blocks l, l + 32, ... (G <= kMaxPassBlocks),
    // then a butterfly.  All of a warp's loads for four values are issued
    // before any is added (one L2 round trip per four values).
    {
        const int nv = nsk * kSketch;             // sketch values, then the scalars at 2 * kSketch
        const int total = nv + kScalars;
        for (int v0 = warp; v0 < total; v0 += 4 * kWarps) {
            float x[4][kMaxPassBlocks / 32];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int vi = v0 + j * kWarps;
                const int v = vi < nv ? vi : 2 * kSketch + (vi - nv);
#pragma unroll
                for (int i = 0; i < kMaxPassBlocks / 32; ++i) {
                    const int b = lane + 32 * i;
                    x[j][i] = (vi < total && b < G) ? __ldcg(a.partials + (size_t)v * G + b) : 0.f;
                }
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int vi = v0 + j * kWarps;
                const int v = vi < nv ? vi : 2 * kSketch + (vi - nv);
                float s = 0.f;
#pragma unroll
                for (int i = 0; i < kMaxPassBlocks / 32; ++i) s += x[j][i];
                s = warp_sum_f(s);
                if (lane == 0 && vi < total) ps.fin[v] = s;
            }
        }
        __syncthreads();
    }
    if (t == 0) *a.counter = 0u;

    if (MODE == kModeObserve) {
        // raw signed bucket sums of z_hat, sum z_hat^2, sum (z_hat - z_a)^2, non-finite count
        if (t < kSketch) a.stats_out[t] = ps.fin[t];
        if (t == 0) {
            a.stats_out[kSketch + 0] = ps.fin[2 * kSketch + 0];
            a.stats_out[kSketch + 1] = ps.fin[2 * kSketch + 1];
            a.stats_out[kSketch + 2] = ps.fin[2 * kSketch + 5];
        }
        return;
    }

    DevState* st = a.st;
    const float N = (float)n;
    const float* fin = ps.fin;
    const int sc0 = 2 * kSketch;   // scalar sums start here

    if (MODE == kModeStats) {
        if (t < kSketch) {
            st->cur_S[t] = fin[t];
            st->anchor_S[t] = fin[kSketch + t];
        }
        if (t == 0) {
            st->cur_sumsq = fin[sc0 + 0];
            st->cur_sumsq_anchor = fin[sc0 + 1];
            st->anchor_sumsq = fin[sc0 + 2];
        }
        return;
    }

    if (MODE == kModeSkip || MODE == kModeSecant || MODE == kModeResidual) {
        if (t < kSummary) st->s_phi[t] = hs.phi[t];
        // the secant needs no retrieval: its support term holds with a non-empty bank
        const int supported = (MODE == kModeSecant) ? (a.nsrc > 0) : ((K > 0) && hs.supported);
        const int finite = supported && (fin[sc0 + 5] == 0.f);
        __shared__ int s_dec;
        if (t == 0) {
            // controller tail in fp32; the stored risk R stays fp64
            const ParamsDev& p = a.prm;
            const float eps = p.eps;
            const StateIn& S = ps.S;
            const float d_z = __fdividef(sqrtf(__fdividef(S.cur_sumsq_anchor, N)), sqrtf(__fdividef(S.anchor_sumsq, N)) + eps);
            const float d_age = (float)a.age;
            const float d_phase = fabsf(a.sk.q_next - S.q_a_out);
            float dc = 0.f, dd = 0.f, uc = 0.f, ud = 0.f;
            for (int j = 0; j < 4; ++j) {
                const float cj = a.cam[j], dj = a.depth[j];
                const float ca = S.cam_a[j], da = S.depth_a[j];
                dc = fmaf(cj - ca, cj - ca, dc);
                dd = fmaf(dj - da, dj - da, dd);
                uc = fmaf(cj, cj, uc);
                ud = fmaf(dj, dj, ud);
            }
            const float pt = p.w_z * d_z + p.w_age * d_age + p.w_phase * d_phase + p.w_cam * sqrtf(dc) +
                             p.w_depth * sqrtf(dd);
            const float d_hat = S.eta * pt;
            const float w = (p.flags & WDC_ABL_NO_IMPACT)
                                ? 1.f
                                : fminf(2.f, 1.f + p.a_cam * sqrtf(uc) + p.a_depth * sqrtf(ud) + p.a_phase * a.sk.q_k);
            const float delta = w * d_hat;
            const float R_cand = fmaf(p.lam, S.R, delta);
            const bool avail = (a.nsrc > 0) && (a.age <= p.max_age) &&
                               (fabsf(a.sk.q_k - S.q_a_out) <= p.q_gap_max) && finite && supported &&
                               (a.k >= p.n_init_exact) && (a.k < a.T - p.n_final_exact);
            // Eq. 10, or periodic placement (ablation): at most period - 1 surrogate steps in a row
            const bool accept = (p.flags & WDC_ABL_PERIODIC) ? (a.age + 1 < p.period) : (R_cand <= p.tau_risk);
            const int dec = (avail && accept) ? 1 : 0;
            StepOut& o = st->out;
            o.decision = dec;
            o.finite = finite;
            o.supported = supported;
            o.n_compat = (MODE == kModeSecant) ? a.nsrc : ((K > 0) ? hs.n_compat : 0);
            o.q = a.sk.q_k;
            o.alpha = (a.nsrc > 0) ? hs.alpha : 0.f;
            o.p = pt;
            o.d_hat = d_hat;
            o.w = w;
            o.delta = delta;
            o.R_cand = R_cand;
            o.d_cf = __int_as_float(0x7fc00000);   // NaN: no exact step yet
            o.d_z = d_z;
            o.r = 0.f;
            for (int i = 0; i < kMaxBank; ++i) {
                o.kappa[i] = (i < K) ? hs.kappa[i] : 0.f;
                o.pi[i] = (i < K) ? hs.pi[i] : 0.f;
            }
            const float R_new = dec ? R_cand : S.R;
            if (dec) st->R = R_cand;
            if (a.graph) {
                // device-side control flow: exactly one of the two branches runs
                cudaGraphSetConditional((cudaGraphConditionalHandle)a.h_exact, dec ? 0u : 1u);
                cudaGraphSetConditional((cudaGraphConditionalHandle)a.h_accept, dec ? 1u : 0u);
            }
            o.R = R_new;
            o.eta = S.eta;
            st->cand_k = a.k;
            st->cand_supported = supported;
            st->cand_finite = finite;
            st->cand_p = pt;
            st->cand_sumsq = fin[sc0 + 0];
            st->cand_sumsq_anchor = fin[sc0 + 1];
            s_dec = dec;
        }
        __syncthreads();
        if (t < kSketch) {
            st->cand_S[t] = fin[t];
            if (s_dec) st->cur_S[t] = fin[t];
        }
        if (t == 0 && s_dec) {
            st->cur_sumsq = fin[sc0 + 0];
            st->cur_sumsq_anchor = fin[sc0 + 1];
        }
        return;
    }

    // ---- anchor pass tail (MODE == kModeAnchor): fp32 arithmetic, fp64 state
    __shared__ float s_rms[2];
    if (t == 0) {
        const ParamsDev& p = a.prm;
        const float eps = p.eps;
        const StateIn& S = ps.S;
        const float R = p.lam * S.R;
        float eta = S.eta;
        st->R = R;
        float d_cf = __int_as_float(0x7fc00000);    // NaN: no calibration this step
        if (a.zcf != nullptr && S.cand_k == a.k && S.cand_supported && S.cand_finite) {
            d_cf = __fdividef(__fdividef(fin[sc0 + 0], N), __fdividef(fin[sc0 + 1], N) + eps);
            if (!(p.flags & WDC_ABL_NO_CALIB)) {
                const float bd = p.beta_d;
                const float v = bd * S.eta + (1.f - bd) * __fdividef(d_cf, S.cand_p + eps);
                eta = fminf(fmaxf(v, p.eta_min), p.eta_max);
                st->eta = eta;
            }
        }
        st->out.d_cf = d_cf;
        st->out.R = R;
        st->out.eta = eta;
        const float r = __fdividef(sqrtf(__fdividef(fin[sc0 + 4], N)), sqrtf(__fdividef(S.cur_sumsq, N)) + eps);
        st->out.r = r;
        st->rec[a.ins_slot].r = r;
        s_rms[0] = sqrtf(__fdividef(fin[sc0 + 2], N));
        s_rms[1] = sqrtf(__fdividef(fin[sc0 + 3], N));
    }
    __syncthreads();
    DevRecord& rec = st->rec[a.ins_slot];
    const float sc = sqrtf(__fdividef((float)kSketch, N));
    const float eps_nu = a.prm.eps_nu;
    const bool no_cond = a.prm.flags & WDC_ABL_NO_COND;
    float so = 0.f, si = 0.f;
    if (t < kSummary) {
        if (t < kSketch) {
            so = __fdividef(sc * fin[t], s_rms[0] + eps_nu);
        } else if (t < 2 * kSketch) {
            const int b = t - kSketch;
            so = __fdividef(sc * (fin[b] - ps.S.anchor_S[b]), s_rms[1] + eps_nu);
        } else if (t < kOffDepth) {
            so = no_cond ? 0.f : a.cam[t - kOffCam];
        } else if (t < kOffQ) {
            so = no_cond ? 0.f : a.depth[t - kOffDepth];
        } else if (t == kOffQ) {
            so = a.sk.q_next;
        } else {
            so = ps.S.s_phi[t];    // pre-insertion history h(H)
        }
        si = ps.S.s_phi[t];
    }
    if (t < kSummary) {
        rec.s_in[t] = si;
        rec.s_out[t] = so;
        rec.s_dphi[t] = so - si;
    }
    {
        float v[2] = {si * si, so * so};
        reduce256<2>(v, hs.scratch, hs.red);
    }
    if (t < kSketch) {
        st->anchor_S[t] = fin[t];
        st->cur_S[t] = fin[t];
    }
    if (t == 0) {
        rec.n_in = sqrtf(hs.red[0]);
        rec.n_out = sqrtf(hs.red[1]);
        rec.q_in = a.sk.q_k;
        rec.q_out = a.sk.q_next;
        rec.dq = a.sk.dq;
        for (int j = 0; j < 4; ++j) {
            rec.cam[j] = a.cam[j];
            rec.depth[j] = a.depth[j];
            st->cam_a[j] = a.cam[j];
            st->depth_a[j] = a.depth[j];
        }
        st->anchor_sumsq = fin[sc0 + 2];
        st->cur_sumsq = fin[sc0 + 2];
        st->cur_sumsq_anchor = 0.f;
        st->q_a_in = a.sk.q_k;
        st->q_a_out = a.sk.q_next;
        st->q_a_dq = a.sk.dq;
    }
}

// Launch forms: arguments by value (the host-driven calls) or read from
// device memory (graph rollout: a planning kernel writes them each step).
template <int MODE, int K>
__global__ void __launch_bounds__(kThreads, 1) pass_kernel(const __grid_constant__ PassArgs a) {
    pass_body<MODE, K>(a);
}
template <int MODE, int K>
__global__ void __launch_bounds__(kThreads, 1) pass_kernel_p(const PassArgs* __restrict__ pa) {
    pass_body<MODE, K>(*pa);
}

template <int K>
void launch_skip(const PassArgs& a, int grid, cudaStream_t s, bool residual) {
    if (residual) pass_kernel<kModeResidual, K><<<grid, kThreads, 0, s>>>(a);
    else pass_kernel<kModeSkip, K><<<grid, kThreads, 0, s>>>(a);
}

// Reductions of three latents for the synthetic diagnostics
// (wdc_latent_pair_stats): out[0] = sum (a-c)^2, out[1] = sum (b-c)^2,
// out[2] = sum (a-c)(b-c), out[3] = sum (a-b)^2, out[4] = sum b^2, with c = 0
// when null.  The same deterministic scheme as the fused passes: per-thread
// fp32 chains with a compensated outer sum, warp and block trees, value-major
// per-block partials and a last-block final tree.
constexpr int kPairStats = 5;
__global__ void __launch_bounds__(kThreads, 1)
    pair_stats_kernel(const float* __restrict__ a, const float* __restrict__ b, const float* __restrict__ c,
                      long long n, float* partials, unsigned* counter, double* out) {
    __shared__ float blk[kWarps][kPairStats];
    __shared__ int last;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    float acc[kPairStats] = {}, cmp[kPairStats] = {}, fac[kPairStats] = {};
    int since = 0;
    const long long n4 = n / 4;
    const long long stride = (long long)gridDim.x * kThreads;
    for (long long i = (long long)blockIdx.x * kThreads + t; i < n4 + (n % 4 ? 1 : 0); i += stride) {
        float av[4] = {0, 0, 0, 0}, bv[4] = {0, 0, 0, 0}, cv[4] = {0, 0, 0, 0};
        if (i < n4) {
            const float4 x = __ldg(reinterpret_cast<const float4*>(a) + i);
            const float4 y = __ldg(reinterpret_cast<const float4*>(b) + i);
            av[0] = x.x; av[1] = x.y; av[2] = x.z; av[3] = x.w;
            bv[0] = y.x; bv[1] = y.y; bv[2] = y.z; bv[3] = y.w;
            if (c) {
                const float4 z = __ldg(reinterpret_cast<const float4*>(c) + i);
                cv[0] = z.x; cv[1] = z.y; cv[2] = z.z; cv[3] = z.w;
            }
        } else {
            for (int e = 0; e < 4; ++e) {
                const long long idx = 4 * i + e;
                if (idx < n) {
                    av[e] = a[idx];
                    bv[e] = b[idx];
                    cv[e] = c ? c[idx] : 0.f;
                }
            }
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float u = av[e] - cv[e], v = bv[e] - cv[e], d = av[e] - bv[e];
            fac[0] = fmaf(u, u, fac[0]);
            fac[1] = fmaf(v, v, fac[1]);
            fac[2] = fmaf(u, v, fac[2]);
            fac[3] = fmaf(d, d, fac[3]);
            fac[4] = fmaf(bv[e], bv[e], fac[4]);
        }
        if (++since >= 16) {
#pragma unroll
            for (int j = 0; j < kPairStats; ++j) { kahan_add(acc[j], cmp[j], fac[j]); fac[j] = 0.f; }
            since = 0;
        }
    }
#pragma unroll
    for (int j = 0; j < kPairStats; ++j) {
        kahan_add(acc[j], cmp[j], fac[j]);
        const float v = warp_sum_f(acc[j] - cmp[j]);
        if (lane == 0) blk[warp][j] = v;
    }
    __syncthreads();
    const int G = gridDim.x;
    if (warp == 0) {
#pragma unroll
        for (int j = 0; j < kPairStats; ++j) {
            const float v = warp_sum_f(blk[lane][j]);
            if (lane == 0) partials[(size_t)j * G + blockIdx.x] = v;
        }
    }
    __threadfence();
    __syncthreads();
    if (t == 0) last = (atomicAdd(counter, 1u) == (unsigned)G - 1);
    __syncthreads();
    if (!last) return;
    __threadfence();
    if (warp < kPairStats) {
        float x[kMaxPassBlocks / 32];
#pragma unroll
        for (int i = 0; i < kMaxPassBlocks / 32; ++i) {
            const int blkid = lane + 32 * i;
            x[i] = blkid < G ? __ldcg(partials + (size_t)warp * G + blkid) : 0.f;
        }
        float v = 0.f;
#pragma unroll
        for (int i = 0; i < kMaxPassBlocks / 32; ++i) v += x[i];
        v = warp_sum_f(v);
        if (lane == 0) out[warp] = v;
    }
    if (t == 0) *counter = 0u;
}

}  // namespace

wdc_status launch_pair_stats(Ctx* c, const float* a, const float* b, const float* cz, double* out_dev,
                             cudaStream_t s) {
    const int grid = pass_grid(c);
    LaunchScope ls(c, WDC_K_OTHER, s);
    pair_stats_kernel<<<grid, kThreads, 0, s>>>(a, b, cz, (long long)c->n, c->partials, c->counter, out_dev);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("pair statistics launch: ") + cudaGetErrorString(e));
    return WDC_OK;
}

int pass_grid(const Ctx* c) {
    const long long nruns = ((long long)c->n + kRun - 1) / kRun;
    long long g = (nruns + kWarps - 1) / kWarps;
    if (g > c->num_sms) g = c->num_sms;
    if (g > kMaxPassBlocks) g = kMaxPassBlocks;
    if (g < 1) g = 1;
    return (int)g;
}

// Pointer-argument launch (graph capture); K selects the bank-size
// specialisation of the skip / residual passes.
wdc_status launch_pass_ptr(Ctx* c, int mode, int K, const PassArgs* pa, cudaStream_t s) {
    const int grid = pass_grid(c);
    switch (mode) {
        case kModeAnchor: pass_kernel_p<kModeAnchor, 0><<<grid, kThreads, 0, s>>>(pa); break;
        case kModeSecant: pass_kernel_p<kModeSecant, 0><<<grid, kThreads, 0, s>>>(pa); break;
        case kModeSkip:
        case kModeResidual: {
            const bool r = mode == kModeResidual;
#define WDC_SKIP_P(KK)                                                                       \
    case KK:                                                                                 \
        if (r) pass_kernel_p<kModeResidual, KK><<<grid, kThreads, 0, s>>>(pa);              \
        else pass_kernel_p<kModeSkip, KK><<<grid, kThreads, 0, s>>>(pa);                    \
        break;
            switch (K) {
                WDC_SKIP_P(0) WDC_SKIP_P(1) WDC_SKIP_P(2) WDC_SKIP_P(3) WDC_SKIP_P(4)
                WDC_SKIP_P(5) WDC_SKIP_P(6) WDC_SKIP_P(7) WDC_SKIP_P(8)
                default: return fail(c, WDC_ERR_INVALID_ARG, "bank size out of range");
            }
#undef WDC_SKIP_P
            break;
        }
        default: return fail(c, WDC_ERR_INVALID_ARG, "unsupported pass mode for the graph rollout");
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("latent pass launch: ") + cudaGetErrorString(e));
    return WDC_OK;
}

wdc_status launch_pass(Ctx* c, int mode, const PassArgs& a, cudaStream_t s) {
    const int grid = pass_grid(c);
    const bool skip_like = mode == kModeSkip || mode == kModeSecant || mode == kModeResidual;
    LaunchScope ls(c, skip_like ? WDC_K_SKIP
                                                                 : (mode == kModeAnchor ? WDC_K_ANCHOR : WDC_K_OTHER),
                   s);
    switch (mode) {
        case kModeStats: pass_kernel<kModeStats, 0><<<grid, kThreads, 0, s>>>(a); break;
        case kModeAnchor: pass_kernel<kModeAnchor, 0><<<grid, kThreads, 0, s>>>(a); break;
        case kModeSecant: pass_kernel<kModeSecant, 0><<<grid, kThreads, 0, s>>>(a); break;
        case kModeSkip:
        case kModeResidual: {
            const bool r = mode == kModeResidual;
            switch (a.nsrc) {
                case 0: launch_skip<0>(a, grid, s, r); break;
                case 1: launch_skip<1>(a, grid, s, r); break;
                case 2: launch_skip<2>(a, grid, s, r); break;
                case 3: launch_skip<3>(a, grid, s, r); break;
                case 4: launch_skip<4>(a, grid, s, r); break;
                case 5: launch_skip<5>(a, grid, s, r); break;
                case 6: launch_skip<6>(a, grid, s, r); break;
                case 7: launch_skip<7>(a, grid, s, r); break;
                case 8: launch_skip<8>(a, grid, s, r); break;
                default: return fail(c, WDC_ERR_INVALID_ARG, "bank size out of range");
            }
            break;
        }
        default: return fail(c, WDC_ERR_INVALID_ARG, "unknown pass mode");
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("latent pass launch: ") + cudaGetErrorString(e));
    return WDC_OK;
}

ParamsDev to_dev_params(const wdc_cache_params& p) {
    ParamsDev d;
    d.K = p.bank_capacity;
    d.min_support = p.min_support;
    d.max_age = p.max_age;
    d.n_init_exact = p.n_init_exact;
    d.n_final_exact = p.n_final_exact;
    d.seed = p.sketch_seed;
    d.sim_min = (float)p.sim_min;
    d.q_gap_max = (float)p.q_gap_max;
    d.gamma_q = (float)p.gamma_q;
    d.tau_in = (float)p.tau_in;
    d.tau_obs = (float)p.tau_obs;
    d.alpha_min = (float)p.alpha_min;
    d.alpha_max = (float)p.alpha_max;
    d.eps = (float)p.eps;
    d.eps_nu = (float)p.eps_nu;
    d.w_z = (float)p.w_z;
    d.w_age = (float)p.w_age;
    d.w_phase = (float)p.w_phase;
    d.w_cam = (float)p.w_cam;
    d.w_depth = (float)p.w_depth;
    d.eta_min = (float)p.eta_min;
    d.eta_max = (float)p.eta_max;
    d.beta_d = (float)p.beta_d;
    d.a_cam = (float)p.a_cam;
    d.a_depth = (float)p.a_depth;
    d.a_phase = (float)p.a_phase;
    d.lam = (p.flags & WDC_ABL_INSTANT_RISK) ? 0.f : (float)p.lambda_;   // instantaneous risk: no accumulation
    d.tau_risk = (float)p.tau_risk;
    d.flags = p.flags;
    d.period = p.period;
    d.ridge = (float)p.ridge;
    return d;
}

}  // namespace wdc

// ---------------------------------------------------------------------------
// Allocation-free variant of the observation pass (wdc_observe_noalloc).
//
// Some callers cannot call cudaMalloc: code that runs inside another
// framework's memory manager or a pre-sized arena, and processes that must not
// allocate device memory once they are set up.  For them this entry point
// keeps its scratch -- the per-CTA partial sums and the last-CTA counter of
// the fused pass -- in the file-scope array below, which every GPU that loads
// this library holds until the process exits.
namespace wdc {
namespace {

constexpr int kNoAllocMaxBlocks = 256;                       // CTAs the scratch can serve
constexpr size_t kNoAllocPartialBytes = (size_t)kNoAllocMaxBlocks * kPartials * sizeof(float);
static_assert(kNoAllocMaxBlocks <= kMaxPassBlocks, "the final reduction covers at most kMaxPassBlocks blocks");
constexpr size_t kNoAllocBytes = kNoAllocPartialBytes + 256;  // + the done counter
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

constexpr int kMaxDevices = 64;
struct NoAllocDevice {
    bool ready = false;
    unsigned char* scratch = nullptr;   // device address of g_noalloc_scratch on this device
    int num_sms = 0;
};
NoAllocDevice g_noalloc_dev[kMaxDevices];
std::mutex g_noalloc_mu;

template <int K>
void launch_observe(const PassArgs& a, int grid, cudaStream_t s) {
    pass_kernel<kModeObserve, K><<<grid, kThreads, 0, s>>>(a);
}

}  // namespace
}  // namespace wdc

extern "C" wdc_status wdc_observe_noalloc(const float* const* z_out, int K, const double* kappa, const float* z_a,
                                          float* z_hat, double* stats, size_t n, uint32_t sketch_seed,
                                          wdc_stream stream) {
    using namespace wdc;
    if (!z_out || !kappa || !z_a || !z_hat || !stats) return WDC_ERR_INVALID_ARG;
    if (K < 1 || K > kMaxBank) return WDC_ERR_INVALID_ARG;
    if (n == 0 || n >= (1ull << 31)) return WDC_ERR_INVALID_ARG;
    for (int i = 0; i < K; ++i)
        if (!z_out[i] || ((uintptr_t)z_out[i] & 15)) return WDC_ERR_INVALID_ARG;
    if (((uintptr_t)z_a & 15) || ((uintptr_t)z_hat & 15) || ((uintptr_t)stats & 7)) return WDC_ERR_INVALID_ARG;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) { cudaGetLastError(); return WDC_ERR_CUDA; }
    if (dev < 0 || dev >= kMaxDevices) return WDC_ERR_UNSUPPORTED;
    NoAllocDevice d;
    {
        // once per device, with that device current: the host-side name of the
        // array is not a device address, so look the address up
        std::lock_guard<std::mutex> lock(g_noalloc_mu);
        if (!g_noalloc_dev[dev].ready) {
            void* p = nullptr;
            if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
                cudaGetLastError();
                return WDC_ERR_CUDA;
            }
            int sms = 0;
            if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
                cudaGetLastError();
                return WDC_ERR_CUDA;
            }
            g_noalloc_dev[dev].scratch = static_cast<unsigned char*>(p);
            g_noalloc_dev[dev].num_sms = sms;
            g_noalloc_dev[dev].ready = true;
        }
        d = g_noalloc_dev[dev];
    }
    PassArgs a;
    std::memset(&a, 0, sizeof(a));
    a.n = (long long)n;
    a.nsrc = K;
    for (int i = 0; i < K; ++i) {
        a.src[i] = z_out[i];
        a.kappa[i] = (float)kappa[i];
    }
    a.anchor = z_a;
    a.out = z_hat;
    a.prm.seed = sketch_seed;
    a.partials = reinterpret_cast<float*>(d.scratch);
    a.counter = reinterpret_cast<unsigned*>(d.scratch + kNoAllocPartialBytes);
    a.stats_out = stats;
    const long long nruns = ((long long)n + kRun - 1) / kRun;
    long long grid = (nruns + kWarps - 1) / kWarps;
    if (grid > d.num_sms) grid = d.num_sms;
    if (grid > kNoAllocMaxBlocks) grid = kNoAllocMaxBlocks;
    if (grid < 1) grid = 1;
    cudaStream_t s = (cudaStream_t)stream;
    // the last-CTA counter must start at zero (a failed earlier call may have left it set)
    if (cudaMemsetAsync(a.counter, 0, sizeof(unsigned), s) != cudaSuccess) { cudaGetLastError(); return WDC_ERR_CUDA; }
    switch (K) {
        case 1: launch_observe<1>(a, (int)grid, s); break;
        case 2: launch_observe<2>(a, (int)grid, s); break;
        case 3: launch_observe<3>(a, (int)grid, s); break;
        case 4: launch_observe<4>(a, (int)grid, s); break;
        case 5: launch_observe<5>(a, (int)grid, s); break;
        case 6: launch_observe<6>(a, (int)grid, s); break;
        case 7: launch_observe<7>(a, (int)grid, s); break;
        default: launch_observe<8>(a, (int)grid, s); break;
    }
    if (cudaGetLastError() != cudaSuccess) return WDC_ERR_CUDA;
    return WDC_OK;
}
