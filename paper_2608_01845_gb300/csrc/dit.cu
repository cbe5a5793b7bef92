// The exact denoiser F_theta (Eq. 1): an adaLN-modulated DiT over video-latent
// tokens, and its orchestration on one GPU.
//
// Layer layout (the paper takes F_theta from its backbone; this is the DiT
// reading shared with the CPU oracle):
//   x = [Linear(cond tokens); Linear(patchify(z)) + sinusoidal position]
//   per block: x += gate1 * (W_o Attn(LN(x)(1+scale1)+shift1) + b_o)
//              x += gate2 * (W_2 GELU_tanh(W_1 (LN(x)(1+scale2)+shift2) + b_1) + b_2)
//   v = unpatchify(W_f (LN(x_video)(1+scale_f)+shift_f) + b_f)
//   modulations = W_mod SiLU(temb), temb = W_t2 SiLU(W_t1 f(t) + b_t1) + b_t2.
//
// fp32 mode (parity) runs every kernel in fp32 SIMT form.  bf16 mode keeps
// activations and weights in bf16 with fp32 accumulation; its GEMMs and
// attention are the tcgen05/TMEM kernels of gemm_tc.cu and attn_tc.cu.
#include "dit_kernels.cuh"

#include <cmath>
#include <cstring>
#include <type_traits>
#include <vector>

namespace wdc {

// tcgen05 paths (gemm_tc.cu, attn_tc.cu); return false when the shape is not
// supported so the caller can report it.
bool tc_gemm_supported(int M, int N, int K);
wdc_status tc_gemm(Ctx* c, const void* A, const void* W, int M, int N, int K, const Epi& e, cudaStream_t s);
wdc_status tc_gemm_grouped(Ctx* c, const void* A0, const void* W0, int M0, const Epi& e0, const void* A1,
                           const void* W1, int M1, const Epi& e1, int N, int K, cudaStream_t s);
bool tc_attention_supported(int L, int d);
wdc_status tc_attention(Ctx* c, const void* q, const void* k, const void* vt, int ldv, void* o, int H, int L, int d,
                        int Hs, int Lc, cudaStream_t s);

struct Lin {
    void* w = nullptr;
    float* b = nullptr;
    int out = 0, in = 0;
};

struct DiT {
    int dtype = WDC_F32;
    size_t esz = 4;
    int S = 1;                            // weight streams (2 with dual_stream)
    int D = 0, H = 0, d = 0, M = 0, E = 0, Fd = 0, P = 0, Lc = 0, Lv = 0, L = 0, Dc = 0, layers = 0;
    int ldv = 0;                          // V^T row stride: L, rounded up to 8 tokens in bf16 (16-byte TMA rows)
    int B = 1;                            // most samples one forward holds (activation buffers sized for it)
    Lin patch, cond, t1, t2, fin;
    void* modW = nullptr;                 // [(layers*S*6 + 2) * D, E]
    float* modB = nullptr;
    size_t mod_rows = 0;
    std::vector<Lin> qkv, o, fc1, fc2;    // index layer * S + stream
    // activations / workspace
    void *x = nullptr, *h = nullptr, *q = nullptr, *k = nullptr, *vt = nullptr, *ao = nullptr, *m = nullptr;
    void *tok = nullptr, *condx = nullptr, *pe = nullptr;
    float *feat = nullptr, *h1 = nullptr, *temb = nullptr, *mods = nullptr;
    float* vb = nullptr;                  // [B, latent] velocities of a batched forward (B > 1)
    std::vector<void*> allocs;
    // set while a graph rollout captures the forward: the timestep comes from
    // device memory at replay time
    const float* t_src = nullptr;
};

namespace {

// ---------------------------------------------------------------- small kernels
// t_src (device, or null): the timestep is read there instead (graph rollout).
__global__ void features_kernel(float t, const float* t_src, int half, float* out) {
    const int j = threadIdx.x + blockIdx.x * blockDim.x;
    if (j >= half) return;
    if (t_src) t = *t_src;
    const double w = exp(-log(10000.0) * (double)j / (double)half);
    const double a = (double)t * w;
    out[j] = (float)cos(a);
    out[half + j] = (float)sin(a);
}

// y[r] = act(W[r,:] . x + b[r]); one warp per row.  act: 0 none, 1 SiLU.
template <typename T>
__global__ void gemv_kernel(const T* __restrict__ W, const float* __restrict__ x, const float* __restrict__ b,
                            float* __restrict__ y, int rows, int cols, int act) {
    const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
    if (warp >= rows) return;
    const T* w = W + (size_t)warp * cols;
    float s = 0.f;
    for (int c = lane; c < cols; c += 32) s = fmaf(ld_act<T>(w + c), x[c], s);
#pragma unroll
    for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) {
        float v = s + (b ? b[warp] : 0.f);
        if (act == 1) v = v / (1.0f + expf(-v));
        y[warp] = v;
    }
}

// h[r] = LN(x[r]) * (1 + scale) + shift, one warp per row, rows [r0, r1).
template <typename T, int VPT>
__global__ void ln_mod_kernel(const T* __restrict__ x, T* __restrict__ h, int r0, int r1, int D,
                              const float* __restrict__ shift, const float* __restrict__ scale, int h_row_off) {
    const int row = r0 + ((blockIdx.x * blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
    if (row >= r1) return;
    const T* xr = x + (size_t)row * D;
    float v[VPT];
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < VPT; ++i) {
        const int c = lane + 32 * i;
        v[i] = (c < D) ? ld_act<T>(xr + c) : 0.f;
        s += v[i];
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const float mean = s / (float)D;
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < VPT; ++i) {
        const int c = lane + 32 * i;
        const float dlt = (c < D) ? v[i] - mean : 0.f;
        q += dlt * dlt;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
    const float rstd = 1.0f / sqrtf(q / (float)D + 1e-6f);
    T* hr = h + (size_t)(row - h_row_off) * D;
#pragma unroll
    for (int i = 0; i < VPT; ++i) {
        const int c = lane + 32 * i;
        if (c < D) hr[c] = to_act<T>(fmaf((v[i] - mean) * rstd, 1.0f + scale[c], shift[c]));
    }
}

// bf16 variant for D = 256 NV, a persistent streaming kernel: one block of 8
// warps per SM, each warp walks rows r0 + warp_id, r0 + warp_id + 8 * grid,
// ...  Lane l owns the 8-element vectors l, l+32, ... of a row (a warp moves
// 512 contiguous bytes per access).  Rows arrive through a per-warp ring of
// kLnRing row buffers in shared memory filled by cp.async (16 bytes per lane
// per vector): while a warp normalises row i, rows i+1 .. i+kLnRing-1 are in
// flight, so an SM keeps 8 * kLnRing rows (144 KB at D = 3072) of loads
// outstanding.  Each lane copies and reads only its own vectors, so its own
// cp.async.wait_group is all the ordering it needs.  The block stages
// (1 + scale) and shift in shared memory once.
constexpr int kLnRing = 3;
constexpr int kLnWarps = 8;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(smem)),
                 "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

template <int NV>
__global__ void __launch_bounds__(kLnWarps * 32, 1)
    ln_mod_stream_kernel(const __nv_bfloat16* __restrict__ x, __nv_bfloat16* __restrict__ h, int r0, int r1, int D,
                         const float* __restrict__ shift, const float* __restrict__ scale, int h_row_off) {
    __shared__ float4 s_sc[NV * 64], s_sh[NV * 64];        // 256 NV floats each
    extern __shared__ uint4 ring[];                        // [warp][kLnRing][NV * 32]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int stride = gridDim.x * kLnWarps;
    uint4* my = ring + (size_t)warp * kLnRing * NV * 32;
    auto issue = [&](int slot, int row) {
        if (row < r1) {
            const uint4* src = reinterpret_cast<const uint4*>(x + (size_t)row * D);
#pragma unroll
            for (int i = 0; i < NV; ++i) cp_async16(my + (slot * NV + i) * 32 + lane, src + i * 32 + lane);
        }
        cp_async_commit();                                 // one group per row, empty past the end
    };
    const int row0 = r0 + blockIdx.x * kLnWarps + warp;
#pragma unroll
    for (int j = 0; j < kLnRing - 1; ++j) issue(j, row0 + j * stride);
    for (int i = threadIdx.x; i < NV * 64; i += blockDim.x) {
        float4 a = __ldg(reinterpret_cast<const float4*>(scale) + i);
        a.x += 1.0f; a.y += 1.0f; a.z += 1.0f; a.w += 1.0f;
        s_sc[i] = a;
        s_sh[i] = __ldg(reinterpret_cast<const float4*>(shift) + i);
    }
    __syncthreads();
    int slot = 0;
    for (int row = row0; row < r1; row += stride) {
        issue((slot + kLnRing - 1) % kLnRing, row + (kLnRing - 1) * stride);
        cp_async_wait<kLnRing - 1>();                      // this lane's copies of `row` have landed
        const uint4* buf = my + slot * NV * 32;
        float v[NV][8];
        float sm = 0.f;
#pragma unroll
        for (int i = 0; i < NV; ++i) {
            const uint4 u = buf[i * 32 + lane];
            const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[q]));
                v[i][2 * q] = f.x;
                v[i][2 * q + 1] = f.y;
                sm += f.x + f.y;
            }
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) sm += __shfl_xor_sync(0xffffffffu, sm, o);
        const float mean = sm / (float)D;
        float q2 = 0.f;
#pragma unroll
        for (int i = 0; i < NV; ++i)
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const float dlt = v[i][e] - mean;
                q2 += dlt * dlt;
            }
#pragma unroll
        for (int o = 16; o; o >>= 1) q2 += __shfl_xor_sync(0xffffffffu, q2, o);
        const float rstd = 1.0f / sqrtf(q2 / (float)D + 1e-6f);
        uint4* hr = reinterpret_cast<uint4*>(h + (size_t)(row - h_row_off) * D);
#pragma unroll
        for (int i = 0; i < NV; ++i) {
            const int c4 = (i * 32 + lane) * 2;               // float4 index of column (i*32+lane)*8
            const float4 sc0 = s_sc[c4], sc1 = s_sc[c4 + 1];
            const float4 sh0 = s_sh[c4], sh1 = s_sh[c4 + 1];
            const float sc[8] = {sc0.x, sc0.y, sc0.z, sc0.w, sc1.x, sc1.y, sc1.z, sc1.w};
            const float sh[8] = {sh0.x, sh0.y, sh0.z, sh0.w, sh1.x, sh1.y, sh1.z, sh1.w};
            uint32_t w[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float a = fmaf((v[i][2 * q] - mean) * rstd, sc[2 * q], sh[2 * q]);
                const float b = fmaf((v[i][2 * q + 1] - mean) * rstd, sc[2 * q + 1], sh[2 * q + 1]);
                __nv_bfloat162 hb = __floats2bfloat162_rn(a, b);
                w[q] = *reinterpret_cast<uint32_t*>(&hb);
            }
            hr[i * 32 + lane] = make_uint4(w[0], w[1], w[2], w[3]);
        }
        slot = slot + 1 == kLnRing ? 0 : slot + 1;
    }
    cp_async_wait<0>();                                    // no copy left in flight at exit
}

// Per-sample device pointers of a batch, passed by value.
struct BatchPtrs {
    const float* p[WDC_MAX_BATCH];
};

// tok[b][(f, h', w'), (c, ph, pw)] = z_b[c, f, h'*p+ph, w'*p+pw]
template <typename T>
__global__ void patchify_kernel(BatchPtrs z, int nb, T* __restrict__ tok, int C, int F, int Hh, int Ww, int p) {
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const int P = C * p * p, hp = Hh / p, wp = Ww / p;
    const long long per = (long long)F * hp * wp * P;
    if (i >= per * nb) return;
    const int b = (int)(i / per);
    const long long ii = i - b * per;
    const int col = (int)(ii % P);
    const long long m = ii / P;
    const int f = (int)(m / (hp * wp)), rem = (int)(m % (hp * wp)), h2 = rem / wp, w2 = rem % wp;
    const int c = col / (p * p), r2 = col % (p * p), ph = r2 / p, pw = r2 % p;
    tok[i] = to_act<T>(z.p[b][(((size_t)c * F + f) * Hh + h2 * p + ph) * Ww + w2 * p + pw]);
}

// dst[b][i] = src_b[i] in the model dtype; a null src_b is the all-zero set.
template <typename T>
__global__ void convert_kernel(BatchPtrs src, int nb, T* __restrict__ dst, long long per) {
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= per * nb) return;
    const int b = (int)(i / per);
    const float* sp = src.p[b];
    dst[i] = to_act<T>(sp ? sp[i - b * per] : 0.0f);
}

// Guided velocity (cfg) or plain scatter of a batched forward's [nb, n]
// velocities into the callers' buffers: cfg: rows (2b, 2b+1) = (conditional,
// null-condition) forwards of sample b, v_b = v_u + g (v_c - v_u).
__global__ void guide_kernel(const float* __restrict__ vb, long long n, int B, int cfg, float g, BatchPtrs dst) {
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n * B) return;
    const int b = (int)(i / n);
    const long long j = i - b * n;
    float v;
    if (cfg) {
        const float vc = vb[(2 * b) * n + j], vu = vb[(2 * b + 1) * n + j];
        v = fmaf(g, vc - vu, vu);
    } else {
        v = vb[i];
    }
    const_cast<float*>(dst.p[b])[j] = v;
}

template <typename T>
__global__ void posemb_kernel(T* __restrict__ pe, int n, int D) {
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (long long)n * D) return;
    const int row = (int)(i / D), col = (int)(i % D), j = col / 2;
    const double w = pow(10000.0, -2.0 * (double)j / (double)D);
    const double a = (double)row * w;
    pe[i] = to_act<T>((float)((col & 1) ? cos(a) : sin(a)));
}

// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) + Box-Muller.
__device__ __forceinline__ void philox(uint32_t c[4], uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t hi0 = __umulhi(0xD2511F53u, c[0]), lo0 = 0xD2511F53u * c[0];
        const uint32_t hi1 = __umulhi(0xCD9E8D57u, c[2]), lo1 = 0xCD9E8D57u * c[2];
        const uint32_t n0 = hi1 ^ c[1] ^ k0, n2 = hi0 ^ c[3] ^ k1;
        c[0] = n0; c[1] = lo1; c[2] = n2; c[3] = lo0;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
}

template <typename T>
__global__ void normal_init_kernel(T* __restrict__ dst, long long n, unsigned long long seed, uint32_t stream_id,
                                   float std) {
    const long long i4 = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i4 * 4 >= n) return;
    uint32_t c[4] = {(uint32_t)i4, (uint32_t)(i4 >> 32), stream_id, 0x57444331u};
    philox(c, (uint32_t)seed, (uint32_t)(seed >> 32));
    const float u0 = ((float)c[0] + 0.5f) * 2.3283064365386963e-10f;
    const float u1 = ((float)c[1] + 0.5f) * 2.3283064365386963e-10f;
    const float u2 = ((float)c[2] + 0.5f) * 2.3283064365386963e-10f;
    const float u3 = ((float)c[3] + 0.5f) * 2.3283064365386963e-10f;
    const float r0 = sqrtf(-2.0f * logf(u0)), r1 = sqrtf(-2.0f * logf(u2));
    float s0, c0, s1, c1;
    sincospif(2.0f * u1, &s0, &c0);
    sincospif(2.0f * u3, &s1, &c1);
    const float v[4] = {r0 * c0, r0 * s0, r1 * c1, r1 * s1};
#pragma unroll
    for (int j = 0; j < 4; ++j)
        if (i4 * 4 + j < n) dst[i4 * 4 + j] = to_act<T>(std * v[j]);
}

// ---------------------------------------------------------------- SIMT GEMM
// C = epilogue(A W^T), A [M, K], W [N, K]; 64x64 tiles, 4x4 per thread,
// sequential-k fp32 accumulation.
template <typename T>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const T* __restrict__ A, const T* __restrict__ W, int M,
                                                         int N, int K, const Epi e) {
    __shared__ float As[16][68];
    __shared__ float Ws[16][68];
    const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
    const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    for (int k0 = 0; k0 < K; k0 += 16) {
        for (int i = threadIdx.x; i < 1024; i += 256) {
            const int r = i / 16, kk = i % 16, gk = k0 + kk;
            const int gm = m0 + r, gn = n0 + r;
            As[kk][r] = (gm < M && gk < K) ? ld_act<T>(A + (size_t)gm * K + gk) : 0.f;
            Ws[kk][r] = (gn < N && gk < K) ? ld_act<T>(W + (size_t)gn * K + gk) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Ws[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int m = m0 + ty * 4 + i, n = n0 + tx * 4 + j;
            if (m < M && n < N) epi_apply<T>(e, m, n, acc[i][j]);
        }
}

// ---------------------------------------------------------------- SIMT attention
// One thread per query row, online softmax over key tiles staged in shared memory.
template <typename T, typename TV, int HD>
__global__ void __launch_bounds__(128) attn_simt_kernel(const T* __restrict__ q, const T* __restrict__ k,
                                                         const TV* __restrict__ vt, int ldv, T* __restrict__ o, int Hs,
                                                         int nb, int Lc, int L, float scale) {
    constexpr int KT = HD <= 64 ? 64 : 32;
    __shared__ float Ks[KT][HD + 1];
    __shared__ float Vs[KT][HD + 1];
    const int h = blockIdx.y;
    const int qi = blockIdx.x * 128 + threadIdx.x;
    float qr[HD], acc[HD];
#pragma unroll
    for (int dd = 0; dd < HD; ++dd) {
        qr[dd] = (qi < L) ? ld_act<T>(q + ((size_t)h * L + qi) * HD + dd) : 0.f;
        acc[dd] = 0.f;
    }
    float mx = -INFINITY, l = 0.f;
    for (int j0 = 0; j0 < L; j0 += KT) {
        for (int i = threadIdx.x; i < KT * HD; i += 128) {
            const int jj = i / HD, dd = i % HD;
            Ks[jj][dd] = (j0 + jj < L) ? ld_act<T>(k + ((size_t)h * L + j0 + jj) * HD + dd) : 0.f;
            const int dv = i / KT, jv = i % KT;
            Vs[jv][dv] = (j0 + jv < L) ? ld_act<TV>(vt + ((size_t)h * HD + dv) * ldv + j0 + jv) : 0.f;
        }
        __syncthreads();
        const int nk = min(KT, L - j0);
        for (int jj = 0; jj < nk; ++jj) {
            float s = 0.f;
#pragma unroll
            for (int dd = 0; dd < HD; ++dd) s = fmaf(qr[dd], Ks[jj][dd], s);
            s *= scale;
            if (s > mx) {
                const float corr = expf(mx - s);
                l *= corr;
#pragma unroll
                for (int dd = 0; dd < HD; ++dd) acc[dd] *= corr;
                mx = s;
            }
            const float pj = expf(s - mx);
            l += pj;
#pragma unroll
            for (int dd = 0; dd < HD; ++dd) acc[dd] = fmaf(pj, Vs[jj][dd], acc[dd]);
        }
        __syncthreads();
    }
    if (qi < L) {
        const float inv = 1.0f / l;
        const int b = h / Hs, hs = h - b * Hs;
        const size_t orow = (size_t)batch_row(b, qi, nb, Lc, L);
#pragma unroll
        for (int dd = 0; dd < HD; ++dd) o[orow * Hs * HD + hs * HD + dd] = to_act<T>(acc[dd] * inv);
    }
}

inline unsigned blocks_for(long long n, int per) { return (unsigned)((n + per - 1) / per); }

template <typename T>
void launch_ln_mod(const void* x, void* h, int r0, int r1, int D, const float* shift, const float* scale,
                   int h_row_off, int num_sms, cudaStream_t s) {
    const int rows = r1 - r0;
    if (rows <= 0) return;
    const unsigned grid = blocks_for((long long)rows * 32, 256);
    const T* xp = reinterpret_cast<const T*>(x);
    T* hp = reinterpret_cast<T*>(h);
    if constexpr (std::is_same<T, __nv_bfloat16>::value) {
        const bool vec_ok = D % 256 == 0 && ((uintptr_t)x & 15) == 0 && ((uintptr_t)h & 15) == 0 &&
                            ((uintptr_t)shift & 15) == 0 && ((uintptr_t)scale & 15) == 0;
        if (vec_ok && D == 3072) {
            constexpr size_t ring_bytes = (size_t)kLnWarps * kLnRing * 12 * 32 * sizeof(uint4);
            static bool attr = false;
            if (!attr) {
                cudaFuncSetAttribute(ln_mod_stream_kernel<12>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)ring_bytes);
                attr = true;
            }
            const int blocks = (rows + kLnWarps - 1) / kLnWarps;
            const unsigned g = (unsigned)(blocks < num_sms ? blocks : num_sms);
            ln_mod_stream_kernel<12><<<g, kLnWarps * 32, ring_bytes, s>>>(xp, hp, r0, r1, D, shift, scale, h_row_off);
            return;
        }
    }
    if (D <= 256) ln_mod_kernel<T, 8><<<grid, 256, 0, s>>>(xp, hp, r0, r1, D, shift, scale, h_row_off);
    else if (D <= 1024) ln_mod_kernel<T, 32><<<grid, 256, 0, s>>>(xp, hp, r0, r1, D, shift, scale, h_row_off);
    else ln_mod_kernel<T, 128><<<grid, 256, 0, s>>>(xp, hp, r0, r1, D, shift, scale, h_row_off);
}

}  // namespace

// ---------------------------------------------------------------- dispatch
// bf16 runs on the tcgen05 kernels only: a shape outside their limits is an
// error, not a silent SIMT run.  The SIMT kernels serve the fp32 parity mode.
static wdc_status gemm(Ctx* c, const void* A, const void* W, int M, int N, int K, const Epi& e, cudaStream_t s) {
    if (M <= 0 || N <= 0) return WDC_OK;
    if (c->cfg.dtype == WDC_BF16) {
        if (!tc_gemm_supported(M, N, K))
            return fail(c, WDC_ERR_UNSUPPORTED, "bf16 GEMM " + std::to_string(M) + "x" + std::to_string(N) + "x" +
                                                    std::to_string(K) + ": the tcgen05 GEMM needs N % 32 == 0 and K % 8 == 0");
        LaunchScope ls(c, WDC_K_GEMM, s);
        return tc_gemm(c, A, W, M, N, K, e, s);
    }
    LaunchScope ls(c, WDC_K_GEMM, s);
    dim3 grid(blocks_for(N, 64), blocks_for(M, 64));
    gemm_simt_kernel<float><<<grid, 256, 0, s>>>(reinterpret_cast<const float*>(A),
                                                 reinterpret_cast<const float*>(W), M, N, K, e);
    return WDC_OK;
}

// H heads in all = nb samples x Hs heads; sample b's output rows follow the
// batch's stream-major token layout (Lc condition tokens per sample).
// Two GEMMs with the same N and K (the dual-stream block's video rows and
// condition rows, each with its own weights and epilogue): one grouped
// tcgen05 launch in bf16, two SIMT launches in the fp32 parity mode.
static wdc_status gemm2(Ctx* c, const void* A0, const void* W0, int M0, const Epi& e0, const void* A1,
                        const void* W1, int M1, const Epi& e1, int N, int K, cudaStream_t s) {
    if (c->cfg.dtype != WDC_BF16) {
        wdc_status st = gemm(c, A0, W0, M0, N, K, e0, s);
        return st ? st : gemm(c, A1, W1, M1, N, K, e1, s);
    }
    if (!tc_gemm_supported(M0 > 0 ? M0 : 1, N, K))
        return fail(c, WDC_ERR_UNSUPPORTED, "bf16 GEMM N=" + std::to_string(N) + " K=" + std::to_string(K) +
                                                ": the tcgen05 GEMM needs N % 32 == 0 and K % 8 == 0");
    LaunchScope ls(c, WDC_K_GEMM, s);
    return tc_gemm_grouped(c, A0, W0, M0, e0, A1, W1, M1, e1, N, K, s);
}

// V^T rows have stride ldv (>= L).  bf16 runs on the tcgen05 kernel only;
// the SIMT kernel serves the fp32 parity mode.
static wdc_status attention(Ctx* c, const void* q, const void* k, const void* vt, int ldv, void* o, int H, int L,
                            int d, int Hs, int Lc, cudaStream_t s) {
    if (c->cfg.dtype == WDC_BF16) {
        if (!tc_attention_supported(L, d))
            return fail(c, WDC_ERR_UNSUPPORTED, "bf16 attention needs head_dim 64 or 128 and L > 0");
        return tc_attention(c, q, k, vt, ldv, o, H, L, d, Hs, Lc, s);     // times its own launches
    }
    LaunchScope ls(c, WDC_K_ATTN, s);
    dim3 grid(blocks_for(L, 128), H);
    const float scale = 1.0f / sqrtf((float)d);
    const int nb = H / Hs;
    using T = float;
    if (d == 64)
        attn_simt_kernel<T, T, 64><<<grid, 128, 0, s>>>((const T*)q, (const T*)k, (const T*)vt, ldv, (T*)o, Hs, nb, Lc, L, scale);
    else
        attn_simt_kernel<T, T, 128><<<grid, 128, 0, s>>>((const T*)q, (const T*)k, (const T*)vt, ldv, (T*)o, Hs, nb, Lc, L, scale);
    return WDC_OK;
}

static void ln_mod(Ctx* c, const void* x, void* h, int r0, int r1, const float* shift, const float* scale,
                   int h_row_off, cudaStream_t s) {
    if (r1 <= r0) return;
    LaunchScope ls(c, WDC_K_NORM, s);
    if (c->cfg.dtype == WDC_BF16)
        launch_ln_mod<__nv_bfloat16>(x, h, r0, r1, c->cfg.hidden, shift, scale, h_row_off, c->num_sms, s);
    else
        launch_ln_mod<float>(x, h, r0, r1, c->cfg.hidden, shift, scale, h_row_off, c->num_sms, s);
}

// ---------------------------------------------------------------- lifetime
static wdc_status dalloc(Ctx* c, void** p, size_t bytes) {
    DiT* t = c->dit;
    cudaError_t e = cudaMalloc(p, bytes ? bytes : 16);
    if (e != cudaSuccess) return fail(c, WDC_ERR_OOM, std::string("cudaMalloc: ") + cudaGetErrorString(e));
    t->allocs.push_back(*p);
    cudaMemset(*p, 0, bytes ? bytes : 16);
    return WDC_OK;
}

static wdc_status alloc_lin(Ctx* c, Lin& l, int out, int in) {
    l.out = out;
    l.in = in;
    wdc_status s = dalloc(c, &l.w, (size_t)out * in * c->dit->esz);
    if (s) return s;
    return dalloc(c, (void**)&l.b, (size_t)out * sizeof(float));
}

wdc_status dit_create(Ctx* c) {
    const wdc_dit_config& g = c->cfg;
    DiT* t = new DiT();
    c->dit = t;
    t->dtype = g.dtype;
    t->esz = g.dtype == WDC_BF16 ? 2 : 4;
    t->S = g.dual_stream ? 2 : 1;
    t->D = g.hidden;
    t->H = g.heads;
    t->d = g.head_dim;
    t->M = g.mlp;
    t->E = g.temb_dim;
    t->Fd = g.freq_dim;
    t->P = g.in_ch * g.patch * g.patch;
    t->Lc = g.cond_tokens;
    t->Lv = g.frames * (g.height / g.patch) * (g.width / g.patch);
    t->L = t->Lc + t->Lv;
    t->ldv = t->dtype == WDC_BF16 ? (t->L + 7) / 8 * 8 : t->L;
    t->Dc = g.cond_dim;
    t->layers = g.layers;
    t->B = g.max_batch > 1 ? g.max_batch : 1;
    wdc_status s;
    if ((s = alloc_lin(c, t->patch, t->D, t->P))) return s;
    if ((s = alloc_lin(c, t->cond, t->D, t->Dc > 0 ? t->Dc : 1))) return s;
    if ((s = alloc_lin(c, t->t1, t->E, t->Fd))) return s;
    if ((s = alloc_lin(c, t->t2, t->E, t->E))) return s;
    if ((s = alloc_lin(c, t->fin, t->P, t->D))) return s;
    t->mod_rows = ((size_t)t->layers * t->S * 6 + 2) * t->D;
    if ((s = dalloc(c, &t->modW, t->mod_rows * t->E * t->esz))) return s;
    if ((s = dalloc(c, (void**)&t->modB, t->mod_rows * sizeof(float)))) return s;
    const int n = t->layers * t->S;
    t->qkv.resize(n);
    t->o.resize(n);
    t->fc1.resize(n);
    t->fc2.resize(n);
    for (int i = 0; i < n; ++i) {
        if ((s = alloc_lin(c, t->qkv[i], 3 * t->D, t->D))) return s;
        if ((s = alloc_lin(c, t->o[i], t->D, t->D))) return s;
        if ((s = alloc_lin(c, t->fc1[i], t->M, t->D))) return s;
        if ((s = alloc_lin(c, t->fc2[i], t->D, t->M))) return s;
    }
    const size_t LD = (size_t)t->B * t->L * t->D * t->esz;
    if ((s = dalloc(c, &t->x, LD))) return s;
    if ((s = dalloc(c, &t->h, LD))) return s;
    if ((s = dalloc(c, &t->q, LD))) return s;
    if ((s = dalloc(c, &t->k, LD))) return s;
    if ((s = dalloc(c, &t->vt, (size_t)t->B * t->ldv * t->D * t->esz))) return s;
    if ((s = dalloc(c, &t->ao, LD))) return s;
    if ((s = dalloc(c, &t->m, (size_t)t->B * t->L * t->M * t->esz))) return s;
    if ((s = dalloc(c, &t->tok, (size_t)t->B * t->Lv * t->P * t->esz))) return s;
    if ((s = dalloc(c, &t->condx, (size_t)t->B * (t->Lc > 0 ? t->Lc : 1) * (t->Dc > 0 ? t->Dc : 1) * t->esz))) return s;
    if (t->B > 1 && (s = dalloc(c, (void**)&t->vb, (size_t)t->B * c->n * sizeof(float)))) return s;
    if ((s = dalloc(c, &t->pe, (size_t)t->Lv * t->D * t->esz))) return s;
    if ((s = dalloc(c, (void**)&t->feat, (size_t)t->Fd * sizeof(float)))) return s;
    if ((s = dalloc(c, (void**)&t->h1, (size_t)t->E * sizeof(float)))) return s;
    if ((s = dalloc(c, (void**)&t->temb, (size_t)t->E * sizeof(float)))) return s;
    if ((s = dalloc(c, (void**)&t->mods, t->mod_rows * sizeof(float)))) return s;
    if (t->dtype == WDC_BF16) {
        const size_t rows = (size_t)t->B * c->num_sms * 256;
        if ((s = dalloc(c, (void**)&c->attn_part, rows * 128 * sizeof(float)))) return s;
        if ((s = dalloc(c, (void**)&c->attn_ml, rows * 2 * sizeof(float)))) return s;
        c->attn_part_samples = t->B;
    }
    const long long npe = (long long)t->Lv * t->D;
    LaunchScope ls(c, WDC_K_OTHER, 0);
    if (t->dtype == WDC_BF16)
        posemb_kernel<__nv_bfloat16><<<blocks_for(npe, 256), 256>>>((__nv_bfloat16*)t->pe, t->Lv, t->D);
    else
        posemb_kernel<float><<<blocks_for(npe, 256), 256>>>((float*)t->pe, t->Lv, t->D);
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("DiT init: ") + cudaGetErrorString(e));
    return WDC_OK;
}

void dit_destroy(Ctx* c) {
    if (!c->dit) return;
    for (void* p : c->dit->allocs) cudaFree(p);
    delete c->dit;
    c->dit = nullptr;
    c->attn_part = nullptr;
    c->attn_ml = nullptr;
    c->attn_part_samples = 0;
}

static uint16_t f32_to_bf16_bits(float f) {
    uint32_t u;
    std::memcpy(&u, &f, 4);
    if ((u & 0x7f800000u) == 0x7f800000u) return (uint16_t)((u >> 16) | ((u & 0xffff) ? 0x40 : 0));
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

static wdc_status upload(Ctx* c, void* dst, const float* host, size_t count, bool model_dtype) {
    if (!model_dtype || c->dit->dtype == WDC_F32) {
        WDC_CUDA_TRY(c, cudaMemcpy(dst, host, count * sizeof(float), cudaMemcpyHostToDevice));
        return WDC_OK;
    }
    std::vector<uint16_t> tmp(count);
    for (size_t i = 0; i < count; ++i) tmp[i] = f32_to_bf16_bits(host[i]);
    WDC_CUDA_TRY(c, cudaMemcpy(dst, tmp.data(), count * 2, cudaMemcpyHostToDevice));
    return WDC_OK;
}

// Device location of parameter tensor `id`: pointer, element count and
// whether it is stored in the model dtype (matrices) or fp32 (biases).
struct TensorLoc {
    void* p = nullptr;
    size_t count = 0;
    bool model_dtype = false;
};

static wdc_status locate_tensor(Ctx* c, int id, int layer, int stream, TensorLoc& loc) {
    DiT* t = c->dit;
    if (!t) return fail(c, WDC_ERR_UNSUPPORTED, "context has no denoiser (layers == 0)");
    const bool per_layer = id >= WDC_T_MOD_W;
    if (per_layer && (layer < 0 || layer >= t->layers || stream < 0 || stream >= t->S))
        return fail(c, WDC_ERR_INVALID_ARG, "layer/stream out of range");
    const int li = layer * t->S + stream;
    Lin* lin = nullptr;
    const bool bias = (id % 2) == 1;
    switch (id) {
        case WDC_T_PATCH_W: case WDC_T_PATCH_B: lin = &t->patch; break;
        case WDC_T_COND_W: case WDC_T_COND_B: lin = &t->cond; break;
        case WDC_T_T1_W: case WDC_T_T1_B: lin = &t->t1; break;
        case WDC_T_T2_W: case WDC_T_T2_B: lin = &t->t2; break;
        case WDC_T_FINAL_W: case WDC_T_FINAL_B: lin = &t->fin; break;
        case WDC_T_QKV_W: case WDC_T_QKV_B: lin = &t->qkv[li]; break;
        case WDC_T_O_W: case WDC_T_O_B: lin = &t->o[li]; break;
        case WDC_T_FC1_W: case WDC_T_FC1_B: lin = &t->fc1[li]; break;
        case WDC_T_FC2_W: case WDC_T_FC2_B: lin = &t->fc2[li]; break;
        case WDC_T_MOD_W: case WDC_T_MOD_B: case WDC_T_FMOD_W: case WDC_T_FMOD_B: {
            const bool blk = id == WDC_T_MOD_W || id == WDC_T_MOD_B;
            const size_t row0 = blk ? (size_t)li * 6 * t->D : (size_t)t->layers * t->S * 6 * t->D;
            const size_t rows = blk ? 6 * (size_t)t->D : 2 * (size_t)t->D;
            if (bias) {
                loc.p = t->modB + row0;
                loc.count = rows;
            } else {
                loc.p = (char*)t->modW + row0 * t->E * t->esz;
                loc.count = rows * t->E;
                loc.model_dtype = true;
            }
            return WDC_OK;
        }
        default: return fail(c, WDC_ERR_INVALID_ARG, "unknown tensor id");
    }
    if (bias) {
        loc.p = lin->b;
        loc.count = (size_t)lin->out;
    } else {
        loc.p = lin->w;
        loc.count = (size_t)lin->out * lin->in;
        loc.model_dtype = true;
    }
    return WDC_OK;
}

wdc_status dit_set_tensor(Ctx* c, int id, int layer, int stream, const float* host, size_t count) {
    if (c->dit && !host) return fail(c, WDC_ERR_INVALID_ARG, "null host pointer");
    TensorLoc loc;
    wdc_status st = locate_tensor(c, id, layer, stream, loc);
    if (st) return st;
    if (count != loc.count) return fail(c, WDC_ERR_INVALID_ARG, "tensor size mismatch");
    return upload(c, loc.p, host, count, loc.model_dtype);
}

// Reads a parameter back to host fp32 (bf16 values widen exactly).
wdc_status dit_get_tensor(Ctx* c, int id, int layer, int stream, float* host, size_t count) {
    if (c->dit && !host) return fail(c, WDC_ERR_INVALID_ARG, "null host pointer");
    TensorLoc loc;
    wdc_status st = locate_tensor(c, id, layer, stream, loc);
    if (st) return st;
    if (count != loc.count) return fail(c, WDC_ERR_INVALID_ARG, "tensor size mismatch");
    if (!loc.model_dtype || c->dit->dtype == WDC_F32) {
        WDC_CUDA_TRY(c, cudaMemcpy(host, loc.p, count * sizeof(float), cudaMemcpyDeviceToHost));
        return WDC_OK;
    }
    std::vector<uint16_t> tmp(count);
    WDC_CUDA_TRY(c, cudaMemcpy(tmp.data(), loc.p, count * 2, cudaMemcpyDeviceToHost));
    for (size_t i = 0; i < count; ++i) {
        const uint32_t u = (uint32_t)tmp[i] << 16;
        std::memcpy(&host[i], &u, 4);
    }
    return WDC_OK;
}

static void init_normal(Ctx* c, void* dst, size_t n, unsigned long long seed, uint32_t sid, float std) {
    const unsigned grid = blocks_for((long long)(n + 3) / 4, 256);
    LaunchScope ls(c, WDC_K_OTHER, 0);
    if (c->dit->dtype == WDC_BF16)
        normal_init_kernel<__nv_bfloat16><<<grid, 256>>>((__nv_bfloat16*)dst, (long long)n, seed, sid, std);
    else
        normal_init_kernel<float><<<grid, 256>>>((float*)dst, (long long)n, seed, sid, std);
}

wdc_status dit_init_weights(Ctx* c, unsigned long long seed, float std) {
    DiT* t = c->dit;
    if (!t) return fail(c, WDC_ERR_UNSUPPORTED, "context has no denoiser (layers == 0)");
    uint32_t sid = 1;
    auto lin = [&](Lin& l) {
        init_normal(c, l.w, (size_t)l.out * l.in, seed, sid++, std);
        cudaMemset(l.b, 0, (size_t)l.out * sizeof(float));
    };
    lin(t->patch); lin(t->cond); lin(t->t1); lin(t->t2); lin(t->fin);
    init_normal(c, t->modW, t->mod_rows * t->E, seed, sid++, std);
    cudaMemset(t->modB, 0, t->mod_rows * sizeof(float));
    for (size_t i = 0; i < t->qkv.size(); ++i) { lin(t->qkv[i]); lin(t->o[i]); lin(t->fc1[i]); lin(t->fc2[i]); }
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("init_weights: ") + cudaGetErrorString(e));
    return WDC_OK;
}

// ---------------------------------------------------------------- forward
wdc_status dit_modulation(Ctx* c, float t_model, float* mod_out, cudaStream_t s) {
    DiT* t = c->dit;
    if (!t) return fail(c, WDC_ERR_UNSUPPORTED, "context has no denoiser (layers == 0)");
    float* dst = mod_out ? mod_out : t->mods;
    const int half = t->Fd / 2;
    {
        LaunchScope ls(c, WDC_K_OTHER, s);
        features_kernel<<<blocks_for(half, 128), 128, 0, s>>>(t_model, t->t_src, half, t->feat);
    }
    auto gv = [&](const void* W, const float* x, const float* b, float* y, int rows, int cols, int act) {
        const unsigned grid = blocks_for((long long)rows * 32, 256);
        LaunchScope ls(c, WDC_K_OTHER, s);
        if (t->dtype == WDC_BF16)
            gemv_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>((const __nv_bfloat16*)W, x, b, y, rows, cols, act);
        else
            gemv_kernel<float><<<grid, 256, 0, s>>>((const float*)W, x, b, y, rows, cols, act);
    };
    gv(t->t1.w, t->feat, t->t1.b, t->h1, t->E, t->Fd, 1);
    gv(t->t2.w, t->h1, t->t2.b, t->temb, t->E, t->E, 1);   // SiLU(temb)
    gv(t->modW, t->temb, t->modB, dst, (int)t->mod_rows, t->E, 0);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("modulation: ") + cudaGetErrorString(e));
    return WDC_OK;
}

// One block on x (device, [nb*L, D], stream-major batch rows) with mod
// (device fp32, [S][6][D]).
static wdc_status run_block(Ctx* c, int layer, void* x, const float* mod, int nb, cudaStream_t s) {
    DiT* t = c->dit;
    const int D = t->D;
    const size_t es = t->esz;
    // stream s rows: s = 0 video [nb*Lc, nb*L), s = 1 cond [0, nb*Lc); single stream: all rows
    int r0[2], r1[2];
    if (t->S == 2) { r0[0] = nb * t->Lc; r1[0] = nb * t->L; r0[1] = 0; r1[1] = nb * t->Lc; }
    else { r0[0] = 0; r1[0] = nb * t->L; }
    wdc_status st;
    // Each GEMM of the block is one launch: with dual-stream weights the
    // video rows and the condition rows (each with its stream's weights and
    // modulation) are the two problems of one grouped launch, so the
    // condition rows' tiles fill the SMs the video tiles leave idle in their
    // last wave.  The LayerNorms run per row range.
    const int S = t->S;
    const float* m6[2] = {mod, mod + (size_t)(S - 1) * 6 * D};
    auto rows_of = [&](int sidx) { return r1[sidx] - r0[sidx]; };
    auto at_row = [&](void* base, int sidx, int width) { return (char*)base + (size_t)r0[sidx] * width * es; };
    auto lin_gemm = [&](const std::vector<Lin>& W, const void* A, int width, int N, Epi* e) -> wdc_status {
        const Lin& w0 = W[layer * S];
        if (S == 1) return gemm(c, at_row(const_cast<void*>(A), 0, width), w0.w, rows_of(0), N, width, e[0], s);
        const Lin& w1 = W[layer * S + 1];
        return gemm2(c, at_row(const_cast<void*>(A), 0, width), w0.w, rows_of(0), e[0],
                     at_row(const_cast<void*>(A), 1, width), w1.w, rows_of(1), e[1], N, width, s);
    };
    for (int sidx = 0; sidx < S; ++sidx) ln_mod(c, x, t->h, r0[sidx], r1[sidx], m6[sidx] + 0 * D, m6[sidx] + 1 * D, 0, s);
    {
        Epi e[2];
        for (int sidx = 0; sidx < S; ++sidx) {
            e[sidx] = Epi{};
            e[sidx].mode = kEpiQKV; e[sidx].bias = t->qkv[layer * S + sidx].b;
            e[sidx].q = t->q; e[sidx].k = t->k; e[sidx].vt = t->vt;
            e[sidx].L = t->L; e[sidx].H = t->H; e[sidx].d = t->d; e[sidx].D = D; e[sidx].row_off = r0[sidx];
            e[sidx].nb = nb; e[sidx].Lc = t->Lc; e[sidx].ldv = t->ldv;
            e[sidx].err = c->err;
        }
        if ((st = lin_gemm(t->qkv, t->h, D, 3 * D, e))) return st;
    }
    if ((st = attention(c, t->q, t->k, t->vt, t->ldv, t->ao, nb * t->H, t->L, t->d, t->H, t->Lc, s))) return st;
    {
        Epi e[2];
        for (int sidx = 0; sidx < S; ++sidx) {
            char* xr = at_row(x, sidx, D);
            e[sidx] = Epi{};
            e[sidx].mode = kEpiResid; e[sidx].bias = t->o[layer * S + sidx].b; e[sidx].out = xr; e[sidx].res = xr;
            e[sidx].ldo = D; e[sidx].gate = m6[sidx] + 2 * D;
        }
        if ((st = lin_gemm(t->o, t->ao, D, D, e))) return st;
    }
    for (int sidx = 0; sidx < S; ++sidx) ln_mod(c, x, t->h, r0[sidx], r1[sidx], m6[sidx] + 3 * D, m6[sidx] + 4 * D, 0, s);
    {
        Epi e[2];
        for (int sidx = 0; sidx < S; ++sidx) {
            e[sidx] = Epi{};
            e[sidx].mode = kEpiStore; e[sidx].bias = t->fc1[layer * S + sidx].b; e[sidx].gelu = 1;
            e[sidx].out = at_row(t->m, sidx, t->M); e[sidx].ldo = t->M;
        }
        if ((st = lin_gemm(t->fc1, t->h, D, t->M, e))) return st;
    }
    {
        Epi e[2];
        for (int sidx = 0; sidx < S; ++sidx) {
            char* xr = at_row(x, sidx, D);
            e[sidx] = Epi{};
            e[sidx].mode = kEpiResid; e[sidx].bias = t->fc2[layer * S + sidx].b; e[sidx].out = xr; e[sidx].res = xr;
            e[sidx].ldo = D; e[sidx].gate = m6[sidx] + 5 * D;
        }
        if ((st = lin_gemm(t->fc2, t->m, t->M, D, e))) return st;
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("block: ") + cudaGetErrorString(e));
    return WDC_OK;
}

void dit_set_timestep_source(Ctx* c, const float* t_src) {
    if (c->dit) c->dit->t_src = t_src;
}

wdc_status dit_block(Ctx* c, int layer, void* x, const float* mod6, cudaStream_t s) {
    if (!c->dit) return fail(c, WDC_ERR_UNSUPPORTED, "context has no denoiser (layers == 0)");
    if (layer < 0 || layer >= c->dit->layers) return fail(c, WDC_ERR_INVALID_ARG, "layer out of range");
    if (!x || !mod6) return fail(c, WDC_ERR_INVALID_ARG, "null pointer");
    return run_block(c, layer, x, mod6, 1, s);
}

// nb samples at one timestep: z[b] (device fp32 latents), cond[b] (device
// fp32 condition tokens, null = the all-zero set); velocities into v
// ([nb, latent], device fp32).
wdc_status dit_forward_batch(Ctx* c, int nb, const float* const* z, float t_model, const float* const* cond,
                             float* v, cudaStream_t s) {
    DiT* t = c->dit;
    if (!t) return fail(c, WDC_ERR_UNSUPPORTED, "context has no denoiser (layers == 0)");
    if (nb < 1 || nb > t->B) return fail(c, WDC_ERR_INVALID_ARG, "batch larger than the context's max_batch");
    if (!z || !v) return fail(c, WDC_ERR_INVALID_ARG, "null pointer");
    BatchPtrs zp{}, cp{};
    for (int b = 0; b < nb; ++b) {
        if (!z[b]) return fail(c, WDC_ERR_INVALID_ARG, "null latent");
        zp.p[b] = z[b];
        cp.p[b] = cond ? cond[b] : nullptr;
    }
    wdc_status st;
    if ((st = dit_modulation(c, t_model, nullptr, s))) return st;
    const int D = t->D;
    const size_t es = t->esz;
    const wdc_dit_config& g = c->cfg;
    // embed: condition tokens (rows [0, nb*Lc)), then patches + position
    // (rows [nb*Lc, nb*L))
    if (t->Lc > 0) {
        const long long per = (long long)t->Lc * t->Dc;
        {
            LaunchScope ls(c, WDC_K_OTHER, s);
            if (t->dtype == WDC_BF16)
                convert_kernel<__nv_bfloat16><<<blocks_for(per * nb, 256), 256, 0, s>>>(cp, nb, (__nv_bfloat16*)t->condx, per);
            else
                convert_kernel<float><<<blocks_for(per * nb, 256), 256, 0, s>>>(cp, nb, (float*)t->condx, per);
        }
        Epi e{};
        e.mode = kEpiStore; e.bias = t->cond.b; e.out = t->x; e.ldo = D;
        if ((st = gemm(c, t->condx, t->cond.w, nb * t->Lc, D, t->Dc, e, s))) return st;
    }
    {
        const long long nt = (long long)t->Lv * t->P * nb;
        {
            LaunchScope ls(c, WDC_K_OTHER, s);
            if (t->dtype == WDC_BF16)
                patchify_kernel<__nv_bfloat16><<<blocks_for(nt, 256), 256, 0, s>>>(zp, nb, (__nv_bfloat16*)t->tok, g.in_ch, g.frames, g.height, g.width, g.patch);
            else
                patchify_kernel<float><<<blocks_for(nt, 256), 256, 0, s>>>(zp, nb, (float*)t->tok, g.in_ch, g.frames, g.height, g.width, g.patch);
        }
        Epi e{};
        char* xv = (char*)t->x + (size_t)nb * t->Lc * D * es;
        e.mode = kEpiResid; e.bias = t->patch.b; e.out = xv; e.res = t->pe; e.res_rows = t->Lv; e.ldo = D; e.gate = nullptr;
        if ((st = gemm(c, t->tok, t->patch.w, nb * t->Lv, D, t->P, e, s))) return st;
    }
    for (int l = 0; l < t->layers; ++l)
        if ((st = run_block(c, l, t->x, t->mods + (size_t)l * t->S * 6 * D, nb, s))) return st;
    // final layer on the video tokens, unpatchified into v (fp32)
    const float* fm = t->mods + (size_t)t->layers * t->S * 6 * D;
    ln_mod(c, t->x, t->h, nb * t->Lc, nb * t->L, fm, fm + D, nb * t->Lc, s);
    Epi e{};
    e.mode = kEpiUnpatch; e.bias = t->fin.b; e.v = v; e.C = g.in_ch; e.F = g.frames; e.Hh = g.height; e.Ww = g.width; e.p = g.patch;
    if ((st = gemm(c, t->h, t->fin.w, nb * t->Lv, t->P, D, e, s))) return st;
    cudaError_t ce = cudaGetLastError();
    if (ce != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("forward: ") + cudaGetErrorString(ce));
    return WDC_OK;
}

wdc_status dit_forward(Ctx* c, const float* z, float t_model, const float* cond, float* v, cudaStream_t s) {
    if (!c->dit) return fail(c, WDC_ERR_UNSUPPORTED, "context has no denoiser (layers == 0)");
    if (!z || !v || (c->dit->Lc > 0 && !cond)) return fail(c, WDC_ERR_INVALID_ARG, "null pointer");
    return dit_forward_batch(c, 1, &z, t_model, &cond, v, s);
}

// Batched, optionally guided forward into the callers' velocity buffers
// (the ABI's wdc_dit_forward_batch): z, cond, v hold B entries; cfg doubles
// the batch as (conditional, null condition) pairs.
wdc_status dit_forward_guided(Ctx* c, int B, const float* const* z, float t_model, const float* const* cond, int cfg,
                              float guidance, float* const* v, cudaStream_t s) {
    DiT* t = c->dit;
    if (!t) return fail(c, WDC_ERR_UNSUPPORTED, "context has no denoiser (layers == 0)");
    const int nb = cfg ? 2 * B : B;
    if (B < 1 || nb > t->B) return fail(c, WDC_ERR_INVALID_ARG, "batch larger than the context's max_batch");
    if (!z || !v || (t->Lc > 0 && !cond)) return fail(c, WDC_ERR_INVALID_ARG, "null pointer array");
    BatchPtrs out{};
    const float* zz[WDC_MAX_BATCH];
    const float* cc[WDC_MAX_BATCH];
    for (int b = 0; b < B; ++b) {
        if (!z[b] || !v[b] || (t->Lc > 0 && !cond[b])) return fail(c, WDC_ERR_INVALID_ARG, "null pointer");
        if (((uintptr_t)z[b] | (uintptr_t)v[b]) & 15) return fail(c, WDC_ERR_INVALID_ARG, "latents must be 16-byte aligned");
        out.p[b] = v[b];
        const int i = cfg ? 2 * b : b;
        zz[i] = z[b];
        cc[i] = t->Lc > 0 ? cond[b] : nullptr;
        if (cfg) {
            zz[i + 1] = z[b];
            cc[i + 1] = nullptr;
        }
    }
    if (nb == 1) return dit_forward_batch(c, 1, zz, t_model, cc, v[0], s);
    wdc_status st = dit_forward_batch(c, nb, zz, t_model, cc, t->vb, s);
    if (st) return st;
    const long long n = (long long)c->n;
    {
        LaunchScope ls(c, WDC_K_OTHER, s);
        guide_kernel<<<blocks_for(n * B, 256), 256, 0, s>>>(t->vb, n, B, cfg, guidance, out);
    }
    cudaError_t ce = cudaGetLastError();
    if (ce != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("guidance: ") + cudaGetErrorString(ce));
    return WDC_OK;
}

// ---------------------------------------------------------------- operators
wdc_status op_gemm(Ctx* c, const void* A, const void* W, const float* bias, void* C, int M, int N, int K, int gelu,
                   const void* res, const float* gate, cudaStream_t s) {
    if (!A || !W || !C || M <= 0 || N <= 0 || K <= 0) return fail(c, WDC_ERR_INVALID_ARG, "bad gemm arguments");
    Epi e{};
    e.mode = res ? kEpiResid : kEpiStore; e.bias = bias; e.gelu = gelu; e.out = C; e.ldo = N; e.res = res; e.gate = gate;
    wdc_status st = gemm(c, A, W, M, N, K, e, s);
    if (st) return st;
    cudaError_t ce = cudaGetLastError();
    if (ce != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("gemm: ") + cudaGetErrorString(ce));
    return WDC_OK;
}

wdc_status op_attention(Ctx* c, const void* q, const void* k, const void* vt, void* o, int H, int L, int d,
                        cudaStream_t s) {
    if (!q || !k || !vt || !o || H <= 0 || L <= 0 || (d != 64 && d != 128))
        return fail(c, WDC_ERR_INVALID_ARG, "bad attention arguments");
    const int ldv = c->cfg.dtype == WDC_BF16 ? (L + 7) / 8 * 8 : L;
    wdc_status st = attention(c, q, k, vt, ldv, o, H, L, d, H, 0, s);
    if (st) return st;
    cudaError_t ce = cudaGetLastError();
    if (ce != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("attention: ") + cudaGetErrorString(ce));
    return WDC_OK;
}

}  // namespace wdc
