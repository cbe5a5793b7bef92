// Shared device pieces of the DiT denoiser: element access for fp32/bf16
// activations and the fused GEMM epilogues used by both the SIMT and the
// tcgen05 GEMM kernels.
#pragma once

#include "wdc_internal.h"

#include <cuda_fp16.h>

namespace wdc {

template <typename T> __device__ __forceinline__ float ld_act(const T* p);
template <> __device__ __forceinline__ float ld_act<float>(const float* p) { return *p; }
template <> __device__ __forceinline__ float ld_act<__nv_bfloat16>(const __nv_bfloat16* p) { return __bfloat162float(*p); }
template <> __device__ __forceinline__ float ld_act<__half>(const __half* p) { return __half2float(*p); }

// V^T of the bf16 model is stored in fp16 (10-bit mantissa) so that the
// attention's PV product can take P in fp16.  A value beyond fp16's range
// (|v| > 65504, infinities included) is saturated to +-65504 and `sat` is
// set, so that the caller can report it; NaN stays NaN.
__device__ __forceinline__ __half to_vt_half(float v, bool& sat) {
    const bool big = fabsf(v) > 65504.0f;
    sat |= big;
    return __float2half_rn(big ? copysignf(65504.0f, v) : v);
}

template <typename T> __device__ __forceinline__ T to_act(float v);
template <> __device__ __forceinline__ float to_act<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 to_act<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

// GELU, tanh form: 0.5 x (1 + tanh(u)) with u = sqrt(2/pi) (x + 0.044715 x^3).
// Written as x * sigmoid(2u) = x / (1 + 2^(-2u log2 e)) -- the same function
// (1 + tanh(u) = 2 / (1 + e^(-2u))) -- with the hardware exp2 and a
// reciprocal: no cancellation for negative x, far fewer instructions than tanhf.
__device__ __forceinline__ float gelu_tanh_f(float x) {
    const float k0 = 0.7978845608028654f;   // sqrt(2/pi)
    const float k1 = 0.044715f;
    const float m2log2e = -2.0f * 1.4426950408889634f;
    const float u = k0 * fmaf(k1 * x * x, x, x);
    float e;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(u * m2log2e));
    return __fdividef(x, 1.0f + e);
}

enum EpiMode { kEpiStore = 0, kEpiResid = 1, kEpiQKV = 2, kEpiUnpatch = 3 };

// Token rows of a batch of nb samples (L tokens each, the first Lc of them
// condition tokens) are laid out stream-major: rows [0, nb*Lc) hold the
// condition tokens of samples 0..nb-1, rows [nb*Lc, nb*L) their video tokens.
// Row-wise kernels and the GEMMs see one [nb*L, D] matrix; the dual-stream
// row blocks stay contiguous.  nb == 1 is the single-sample sequence.
__host__ __device__ __forceinline__ void batch_token(int row, int nb, int Lc, int L, int& b, int& tok) {
    if (nb <= 1) { b = 0; tok = row; return; }
    const int cond_rows = nb * Lc;
    if (row < cond_rows) {
        b = row / Lc;
        tok = row - b * Lc;
    } else {
        const int j = row - cond_rows, Lv = L - Lc;
        b = j / Lv;
        tok = Lc + (j - b * Lv);
    }
}
__host__ __device__ __forceinline__ int batch_row(int b, int tok, int nb, int Lc, int L) {
    return tok < Lc ? b * Lc + tok : nb * Lc + b * (L - Lc) + (tok - Lc);
}

// Epilogue of C = A W^T on one output element (row m of this GEMM, column n).
struct Epi {
    int mode;
    const float* bias;        // [N] or null
    int gelu;
    void* out;                // kEpiStore / kEpiResid: [M, ldo]
    int ldo;
    const void* res;          // kEpiResid: [M, ldo] (may equal out)
    const float* gate;        // kEpiResid: [N] or null (= 1)
    int res_rows;             // kEpiResid: > 0 reads residual row m % res_rows
    // kEpiQKV: q, k [nb*H, L, d], vt [nb*H, d, ldv] (ldv >= L: the V^T row
    // stride); (sample, token) of batch row row_off + m (batch_token); head
    // of sample b = b*H + h
    void* q; void* k; void* vt;
    int L, H, d, D, row_off, nb, Lc, ldv;
    unsigned* err;            // kEpiQKV: receives kErrVSaturated (may be null)
    // kEpiUnpatch: v fp32 [nb][C, F, Hh, Ww]; row m = (sample, f, h', w'),
    // column = (c, ph, pw)
    float* v;
    int C, F, Hh, Ww, p;
};

template <typename T>
__device__ __forceinline__ void epi_apply(const Epi& e, int m, int n, float acc) {
    float x = acc + (e.bias ? e.bias[n] : 0.0f);
    if (e.gelu) x = gelu_tanh_f(x);
    switch (e.mode) {
        case kEpiStore:
            reinterpret_cast<T*>(e.out)[(size_t)m * e.ldo + n] = to_act<T>(x);
            break;
        case kEpiResid: {
            const size_t idx = (size_t)m * e.ldo + n;
            const size_t ridx = (size_t)(e.res_rows > 0 ? m % e.res_rows : m) * e.ldo + n;
            const float r = ld_act<T>(reinterpret_cast<const T*>(e.res) + ridx);
            const float g = e.gate ? e.gate[n] : 1.0f;
            reinterpret_cast<T*>(e.out)[idx] = to_act<T>(fmaf(g, x, r));
            break;
        }
        case kEpiQKV: {
            const int which = n / e.D, c = n % e.D, dd = c % e.d;
            int b, tok;
            batch_token(e.row_off + m, e.nb, e.Lc, e.L, b, tok);
            const size_t h = (size_t)b * e.H + c / e.d;
            if (which == 0)
                reinterpret_cast<T*>(e.q)[(h * e.L + tok) * e.d + dd] = to_act<T>(x);
            else if (which == 1)
                reinterpret_cast<T*>(e.k)[(h * e.L + tok) * e.d + dd] = to_act<T>(x);
            else if constexpr (sizeof(T) == 2) {
                bool sat = false;
                reinterpret_cast<__half*>(e.vt)[(h * e.d + dd) * e.ldv + tok] = to_vt_half(x, sat);
                if (sat && e.err) atomicOr(e.err, kErrVSaturated);
            }
            else
                reinterpret_cast<T*>(e.vt)[(h * e.d + dd) * e.ldv + tok] = to_act<T>(x);
            break;
        }
        case kEpiUnpatch: {
            const int hp = e.Hh / e.p, wp = e.Ww / e.p, Lv = e.F * hp * wp;
            const int b = m / Lv, mm = m - b * Lv;
            const int f = mm / (hp * wp), rem = mm % (hp * wp), h2 = rem / wp, w2 = rem % wp;
            const int c = n / (e.p * e.p), r2 = n % (e.p * e.p), ph = r2 / e.p, pw = r2 % e.p;
            e.v[(size_t)b * e.C * e.F * e.Hh * e.Ww +
                (((size_t)c * e.F + f) * e.Hh + h2 * e.p + ph) * e.Ww + w2 * e.p + pw] = x;
            break;
        }
    }
}

}  // namespace wdc
