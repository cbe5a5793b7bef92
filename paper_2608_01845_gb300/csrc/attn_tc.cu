// Non-causal softmax attention on the tcgen05 tensor cores (sm_103a):
// O = softmax(Q K^T / sqrt(d)) V per head, joint over all L tokens (the DiT's
// full spatio-temporal attention).  Q, K [H, L, d] bf16, V^T [H, d, L] fp16,
// O [L, H*d] bf16; S = Q K^T in fp32, P in fp16, fp32 accumulation of O;
// d = 64 or 128.
//
// One CTA per (head, 256 query rows), 12 warps in three warpgroups:
//   warpgroup 0 (control, registers lowered to 40 per thread)
//     warp 0    TMA producer: the two 128-row Q tiles once, then K / V^T
//               tiles of BK keys into a shared-memory ring (128-byte swizzle);
//     warps 1, 2 MMA issuers, one thread per query tile t:
//               S(t) = Q(t) K^T into TMEM (BK fp32 columns) and
//               O(t) += P(t) V into TMEM;
//   warpgroups 1, 2 (softmax of query tile 0, 1; registers raised to 232)
//               one thread per query row = TMEM lane: exp2 numerators, row
//               sums, O rescaling in TMEM when the exponent base moves, final
//               1/l normalisation and the bf16 store.
// The exponent base of a row only moves when a tile could produce a numerator
// above 2^8: each tile is first exponentiated against the running base with
// no max pass (no max -> exp dependency); only when its row sum exceeds 2^8
// -- the only way a numerator can -- does the row take the tile max, move the
// base and recompute (O and l share the base, so the result is unchanged).
// The first tile sets the base from its own max.  S stays in registers until
// that check, hence the register split.
// P (fp16 pairs) is written to tensor memory and read as the TMEM A operand
// of the PV MMA (shared memory is left to Q, K and V).  The numerators are
// formed in packed fp16: x = s * scale - base in fp32 (fma.f32x2), one
// conversion to f16x2 and one ex2.approx.f16x2 per pair, which is already
// the P word; row sums accumulate per 16 pairs in f16x2 and in fp32 beyond.
// In fp16, x keeps 11 significant bits (error <= 2^-9 absolute for
// |x| < 8, below the rounding of P itself where P matters) and P keeps 11
// (bf16 would keep 8).
// TMEM, per query tile t: S (BK columns), P (BK / 2) and O (d) side by side
// -- d = 64 with BK = 128 keys per step, d = 128 with BK = 64, 256 and 224
// columns a tile.  P has its own columns, so S(t) may be overwritten as soon
// as the softmax has loaded it: each issuer runs
//     S(t, j), PV(t, j-1)
// and the MMA of S(t, j+1) overlaps the softmax of step j instead of
// waiting behind PV(t, j).
// Grid: one CTA per (head, 256-query) unit, one CTA per SM.  The units of a
// sample's last, partial round are split over the key range instead: each
// part runs the same pipeline over its steps and writes its unnormalised O,
// exponent base and row sum to a workspace of the context, and
// attn_combine_kernel merges the parts, so the round's CTAs fill the SMs.
// Keys past L are masked (TMA zero-fills out-of-range K / V^T).  Every
// mbarrier wait is bounded.
#include "dit_kernels.cuh"
#include "ptx.cuh"

#include <cuda_fp16.h>

namespace wdc {

namespace {

constexpr int BQ = 128;        // query rows per tile (two tiles per CTA)
// Register split: launch allocation 168 per thread (65536 / 384 rounded
// down to a multiple of 8); the control warpgroup hands registers to the two
// softmax warpgroups: 128 * 40 + 256 * 232 = 384 * 168.
constexpr uint32_t kRegsLaunch = 168;

template <int D>
struct AttnCfg {
    static constexpr int BK = D == 64 ? 128 : 64;           // keys per step
    static constexpr int THREADS = 384;                     // 3 warpgroups
    static constexpr int ISSUERS = 2;                       // one MMA thread per query tile
    static constexpr int ATOMS = D / 64;                    // 128-byte atoms along d
    static constexpr uint32_t Q_TILE = BQ * D * 2;          // one query tile
    static constexpr uint32_t K_TILE = BK * D * 2;
    static constexpr uint32_t V_TILE = D * BK * 2;
    static constexpr uint32_t STAGE = K_TILE + V_TILE;      // 32 KB for both head sizes
    static constexpr int STAGES = D == 64 ? 3 : 5;
    static constexpr uint32_t SMEM = 2 * Q_TILE + STAGES * STAGE + 1024 + 256;
    static constexpr uint32_t TMEM_COLS = 512;
    static constexpr uint32_t REGS_CONTROL = 40;
    static constexpr uint32_t REGS_SOFTMAX = 232;
    static_assert(128 * REGS_CONTROL + 256 * REGS_SOFTMAX <= 384 * kRegsLaunch, "register split exceeds the launch");
    static_assert(2 * (BK + BK / 2 + D) <= (int)TMEM_COLS, "S, P and O of two tiles exceed tensor memory");
    static_assert(SMEM <= 227 * 1024, "shared memory per CTA");
    // TMEM column of S, P and O of query tile t
    __device__ static constexpr uint32_t s_col(int t) { return (uint32_t)(BK + BK / 2 + D) * t; }
    __device__ static constexpr uint32_t p_col(int t) { return s_col(t) + BK; }
    __device__ static constexpr uint32_t o_col(int t) { return s_col(t) + BK + BK / 2; }
};


struct AttnArgs {
    int H, L, n_kv, q_blocks;
    int Hs, nb, Lc;           // heads per sample, samples, condition tokens (output row mapping)
    float scale_log2;
    __nv_bfloat16* o;
    unsigned* err;
    // per sample: units_s = Hs * q_blocks units (head, 256-query block);
    // those from n_full on are split over the key range into `split` CTAs
    // each, which write unnormalised partials.  The split depends on the
    // sample's own grid only, so a sample's attention is the same bits in a
    // batched launch as alone.
    int units_s, n_full, split;
    float* part_o;            // [part slot][256 rows][d]
    float* part_ml;           // [part slot][256 rows][base, row sum]
};

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Three-input maximum (one instruction for two comparisons).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

__device__ __forceinline__ uint32_t pack2(float a, float b) {
    __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&h);
}

// Two f32 values as one paired-fp32 operand (lo = a, hi = b).
__device__ __forceinline__ uint64_t pair(float a, float b) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
    return r;
}

// Two softmax numerators: x pair (fma.f32x2) -> f16x2 -> ex2.approx.f16x2
// (one SFU instruction for both) = the P word; the pair is added into an
// f16x2 partial sum.
__device__ __forceinline__ uint32_t exp2_pair_h(float s0, float s1, uint64_t scale2, uint64_t nm2, uint32_t& acc) {
    uint32_t p;
    asm("{\n .reg .b64 x;\n .reg .f32 a, b;\n .reg .b32 h;\n"
        " mov.b64 x, {%2, %3};\n"
        " fma.rn.f32x2 x, x, %4, %5;\n"
        " mov.b64 {a, b}, x;\n"
        " cvt.rn.f16x2.f32 h, b, a;\n"
        " ex2.approx.f16x2 %0, h;\n"
        " add.rn.f16x2 %1, %1, %0;\n}"
        : "=r"(p), "+r"(acc)
        : "f"(s0), "f"(s1), "l"(scale2), "l"(nm2));
    return p;
}

__device__ __forceinline__ float half2_sum(uint32_t v) {
    __half2 h = *reinterpret_cast<__half2*>(&v);
    return __low2float(h) + __high2float(h);
}


// BATCH: heads of several samples, output rows through the batch's
// stream-major token layout; otherwise row = token, head = h (one sample).
template <int D, bool BATCH>
__global__ void __launch_bounds__(AttnCfg<D>::THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tk,
                   const __grid_constant__ CUtensorMap tv, const __grid_constant__ AttnArgs g) {
    using C = AttnCfg<D>;
    constexpr int BKV = C::BK;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sq = smem;                                       // [2 tiles][ATOMS][128 x 128 B]
    uint8_t* skv = smem + 2 * C::Q_TILE;                      // [STAGES][K | V^T]
    uint64_t* bars = reinterpret_cast<uint64_t*>(skv + C::STAGES * C::STAGE);
    uint64_t* q_full = bars;
    uint64_t* kv_full = q_full + 1;
    uint64_t* kv_empty = kv_full + C::STAGES;
    uint64_t* s_full = kv_empty + C::STAGES;                  // [2]
    uint64_t* s_free = s_full + 2;                            // [2]
    uint64_t* p_full = s_free + 2;                            // [2]
    uint64_t* p_free = p_full + 2;                            // [2]
    uint64_t* o_final = p_free + 2;                           // [2]
    uint64_t* mma_done = o_final + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // unit (head, 256-query block) of this CTA: per sample, n_full whole
    // units, then the key-range parts of the sample's last units (keys of
    // steps j0 .. j0 + nj - 1)
    const int n_split_s = g.units_s - g.n_full;
    const int per_sample = g.n_full + n_split_s * g.split;
    const int smp = blockIdx.x / per_sample, rem = blockIdx.x - smp * per_sample;
    const bool is_part = rem >= g.n_full;
    const int pidx = rem - g.n_full;                          // part CTA within the sample
    const int unit = smp * g.units_s + (is_part ? g.n_full + pidx / g.split : rem);
    const int part = is_part ? pidx % g.split : 0;
    const int pslot = smp * n_split_s * g.split + pidx;       // workspace slot of a part CTA
    const int h = unit / g.q_blocks;
    const int q0 = (unit % g.q_blocks) * (2 * BQ);
    const int n_kv = g.n_kv;
    const int j0 = is_part ? part * n_kv / g.split : 0;
    const int nj = (is_part ? (part + 1) * n_kv / g.split : n_kv) - j0;

    if (threadIdx.x == 0) {
        mbar_init(q_full, 1);
        for (int s = 0; s < C::STAGES; ++s) {
            mbar_init(&kv_full[s], 1);
            mbar_init(&kv_empty[s], C::ISSUERS);   // one commit per MMA issuer
        }
        for (int w = 0; w < 2; ++w) {
            mbar_init(&s_full[w], 1);
            mbar_init(&s_free[w], 4);
            mbar_init(&p_full[w], 4);
            mbar_init(&p_free[w], 1);
            mbar_init(&o_final[w], 1);
        }
        mbar_init(mma_done, C::ISSUERS);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tmap(&tq);
        prefetch_tmap(&tk);
        prefetch_tmap(&tv);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, C::TMEM_COLS);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const int wg = warp >> 2;

    if (wg == 0) {
      setmaxnreg_dec<C::REGS_CONTROL>();
      if (warp == 0) {
        if (lane == 0) {
            // Q: two tiles x ATOMS boxes of [128 rows x 64 d]
            mbar_arrive_expect_tx(q_full, 2 * C::Q_TILE);
            for (int t = 0; t < 2; ++t)
                for (int a = 0; a < C::ATOMS; ++a)
                    tma_load_3d(sq + t * C::Q_TILE + a * (BQ * 128), &tq, q_full, 64 * a, q0 + t * BQ, h);
            int stage = 0;
            uint32_t phase = 0;
            bool armed[C::STAGES];
            uint32_t armed_phase[C::STAGES];
            for (int s = 0; s < C::STAGES; ++s) armed[s] = false;
            for (int j = j0; j < j0 + nj; ++j) {
                if (!mbar_wait(&kv_empty[stage], phase ^ 1u, abort_flag, g.err)) break;
                mbar_arrive_expect_tx(&kv_full[stage], C::STAGE);
                uint8_t* sk = skv + stage * C::STAGE;
                uint8_t* sv = sk + C::K_TILE;
                for (int a = 0; a < C::ATOMS; ++a) tma_load_3d(sk + a * (BKV * 128), &tk, &kv_full[stage], 64 * a, j * BKV, h);
                for (int a = 0; a < BKV / 64; ++a) tma_load_3d(sv + a * (D * 128), &tv, &kv_full[stage], j * BKV + 64 * a, 0, h);
                armed[stage] = true;
                armed_phase[stage] = phase;
                if (++stage == C::STAGES) { stage = 0; phase ^= 1u; }
            }
            {
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(q_full, 0) && globaltimer() - t0 < kWaitLimitNs) {
                }
            }
            for (int s = 0; s < C::STAGES; ++s) {
                if (!armed[s]) continue;
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(&kv_full[s], armed_phase[s]) && globaltimer() - t0 < kWaitLimitNs) {
                }
            }
        }
      } else if (warp == 1 || warp == 2) {
        if (lane == 0) {
            constexpr uint32_t idesc_s = idesc_bf16(BQ, BKV);
            constexpr uint32_t idesc_o = idesc_f16(BQ, D);       // P (fp16, TMEM) x V (fp16, shared memory)
            const uint32_t sq0 = smem_u32(sq);
            bool ok = mbar_wait(q_full, 0, abort_flag, g.err);
            int stage = 0, prev = 0;
            uint32_t phase = 0;
            // S(t) = Q(t) K^T into TMEM (BK fp32 columns)
            auto issue_s = [&](int t, int st) {
                const uint32_t kb = smem_u32(skv + st * C::STAGE);
                const uint32_t qb = sq0 + t * C::Q_TILE;
#pragma unroll
                for (int ks = 0; ks < D / 16; ++ks) {
                    const uint32_t off = (ks >> 2) * (BQ * 128) + (ks & 3) * 32;
                    const uint32_t koff = (ks >> 2) * (BKV * 128) + (ks & 3) * 32;
                    tc_mma(tmem + C::s_col(t), sdesc_sw128(qb + off), sdesc_sw128(kb + koff), idesc_s, ks != 0);
                }
            };
            // O(t) (+)= P(t) V, A = P in TMEM (16 bf16 = 8 columns per K step)
            auto issue_pv = [&](int t, int st, bool acc) {
                const uint32_t vb = smem_u32(skv + st * C::STAGE + C::K_TILE);
#pragma unroll
                for (int ks = 0; ks < BKV / 16; ++ks) {
                    const uint32_t voff = (ks >> 2) * (D * 128) + (ks & 3) * 32;
                    tc_mma_ts(tmem + C::o_col(t), tmem + C::p_col(t) + ks * 8, sdesc_sw128(vb + voff), idesc_o,
                              (acc || ks != 0) ? 1u : 0u);
                }
            };
            // this thread issues the MMAs of query tile t only; the other
            // tile has its own issuer, so neither waits behind the other's
            // softmax
            const int t = warp - 1;
            for (int j = 0; j < nj && ok; ++j) {
                if (!mbar_wait(&kv_full[stage], phase, abort_flag, g.err)) { ok = false; break; }
                tc_fence_after();
                if (j > 0) {
                    if (!mbar_wait(&s_free[t], (j - 1) & 1, abort_flag, g.err)) { ok = false; break; }
                    tc_fence_after();
                }
                issue_s(t, stage);
                tc_commit(&s_full[t]);
                if (j > 0) {
                    if (!mbar_wait(&p_full[t], (j - 1) & 1, abort_flag, g.err)) { ok = false; break; }
                    tc_fence_after();
                    issue_pv(t, prev, j > 1);
                    tc_commit(&p_free[t]);
                    tc_commit(&kv_empty[prev]);
                }
                prev = stage;
                if (++stage == C::STAGES) { stage = 0; phase ^= 1u; }
            }
            if (ok && mbar_wait(&p_full[t], (nj - 1) & 1, abort_flag, g.err)) {
                tc_fence_after();
                issue_pv(t, prev, nj > 1);
                tc_commit(&kv_empty[prev]);
                tc_commit(&o_final[t]);
            }
            tc_commit(mma_done);
            const unsigned long long t0 = globaltimer();
            while (!mbar_try_wait(mma_done, 0) && globaltimer() - t0 < kWaitLimitNs) {
            }
        }
      }
    } else {
        setmaxnreg_inc<C::REGS_SOFTMAX>();
        // softmax warpgroups: t = query tile, quarter = TMEM lane quarter
        const int t = wg - 1;
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;                 // row within the tile = TMEM lane
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        const uint32_t s_addr = tmem + lane_base + C::s_col(t);
        const uint32_t p_addr = tmem + lane_base + C::p_col(t);
        const uint32_t o_addr = tmem + lane_base + C::o_col(t);
        const int last_valid = g.L - (n_kv - 1) * BKV;       // keys in the last tile
        const int mask_step = (j0 + nj == n_kv && last_valid < BKV) ? nj - 1 : -1;   // this CTA's ragged step
        float m_run = -INFINITY, l_run = 0.f;
        const uint64_t scale2 = pair(g.scale_log2, g.scale_log2);
        bool ok = true;
        for (int j = 0; j < nj; ++j) {                  // j counts this CTA's steps
            if (!mbar_wait(&s_full[t], j & 1, abort_flag, g.err)) { ok = false; break; }
            tc_fence_after();
            float s[BKV];
#pragma unroll
            for (int c = 0; c < BKV / 32; ++c) tmem_ld32(s_addr + c * 32, *reinterpret_cast<uint32_t(*)[32]>(&s[c * 32]));
            tmem_ld_wait();
            // S(t) is in registers: the MMA may compute S(t, j+1) now
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&s_free[t]);
            if (j == mask_step) {
#pragma unroll
                for (int c = 0; c < BKV; ++c)
                    if (c >= last_valid) s[c] = -INFINITY;
            }
            auto tile_max = [&]() {
                // 8 independent partial maxima (short dependency chains)
                float m8[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) m8[i] = fmaxf(s[i], s[8 + i]);
#pragma unroll
                for (int c = 16; c < BKV; c += 16)
#pragma unroll
                    for (int i = 0; i < 8; ++i) m8[i] = fmax3(m8[i], s[c + i], s[c + 8 + i]);
                return fmax3(fmax3(m8[0], m8[1], m8[2]), fmax3(m8[3], m8[4], m8[5]), fmaxf(m8[6], m8[7]));
            };
            // numerators 2^(s * scale - base) into p (fp16 pairs); returns their sum
            uint32_t p[BKV / 2];
            auto numerators = [&](float base) {
                uint32_t sum4[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) sum4[i] = 0u;
                const uint64_t nm2 = pair(-base, -base);
#pragma unroll
                for (int c = 0; c < BKV; c += 2) p[c / 2] = exp2_pair_h(s[c], s[c + 1], scale2, nm2, sum4[(c / 2) & 3]);
                return (half2_sum(sum4[0]) + half2_sum(sum4[1])) + (half2_sum(sum4[2]) + half2_sum(sum4[3]));
            };
            float base = (j == 0) ? tile_max() * g.scale_log2 : m_run;
            float sum;
            // A numerator above 2^8 implies a row sum above 2^8 (so does a
            // non-finite one): only then take the tile max, move the base and
            // recompute, as a second pass of the same code.
#pragma unroll 1
            for (int pass = 0;; ++pass) {
                sum = numerators(base);
                const bool redo = pass == 0 && !(sum <= 256.0f);
                if (!__any_sync(0xffffffffu, redo)) break;
                if (redo) base = fmaxf(base, tile_max() * g.scale_log2);
            }
            const bool moved = base != m_run;
            const float corr = ex2(m_run - base);     // 1 when the base stays; 0 before the first tile
            l_run = l_run * corr + sum;
            m_run = base;
            // PV(t, j-1) must be done before P(t) is overwritten and O(t) rescaled
            if (j > 0) {
                if (!mbar_wait(&p_free[t], (j - 1) & 1, abort_flag, g.err)) { ok = false; break; }
                tc_fence_after();
            }
            if (j > 0 && __any_sync(0xffffffffu, moved)) {
                // PV(t, j-1) is complete: rescale O in place
#pragma unroll
                for (int c = 0; c < D; c += 32) {
                    uint32_t o[32];
                    tmem_ld32(o_addr + c, o);
                    tmem_ld_wait();
                    uint32_t lo[16], hi[16];
#pragma unroll
                    for (int q = 0; q < 16; ++q) {
                        lo[q] = __float_as_uint(__uint_as_float(o[q]) * corr);
                        hi[q] = __float_as_uint(__uint_as_float(o[16 + q]) * corr);
                    }
                    tmem_st16(o_addr + c, lo);
                    tmem_st16(o_addr + c + 16, hi);
                }
            }
            // P (BK / 2 columns of fp16 pairs)
#pragma unroll
            for (int c = 0; c < BKV / 2; c += 16) tmem_st16(p_addr + c, *reinterpret_cast<uint32_t(*)[16]>(&p[c]));
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&p_full[t]);
        }
        if (ok && is_part && mbar_wait(&o_final[t], 0, abort_flag, g.err)) {
            // a part of a split unit: unnormalised O with its base and row
            // sum, merged by the combine kernel
            tc_fence_after();
            const size_t prow = (size_t)pslot * (2 * BQ) + t * BQ + row;
            float4* dst = reinterpret_cast<float4*>(g.part_o + prow * D);
#pragma unroll
            for (int c = 0; c < D; c += 32) {
                uint32_t o[32];
                tmem_ld32(o_addr + c, o);
                tmem_ld_wait();
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    dst[c / 4 + q] = make_float4(__uint_as_float(o[4 * q]), __uint_as_float(o[4 * q + 1]),
                                                 __uint_as_float(o[4 * q + 2]), __uint_as_float(o[4 * q + 3]));
            }
            reinterpret_cast<float2*>(g.part_ml)[prow] = make_float2(m_run, l_run);
        } else if (ok && mbar_wait(&o_final[t], 0, abort_flag, g.err)) {
            tc_fence_after();
            const int tok = q0 + t * BQ + row;
            const float inv = 1.0f / l_run;
#pragma unroll
            for (int c = 0; c < D; c += 32) {
                uint32_t o[32];
                tmem_ld32(o_addr + c, o);
                tmem_ld_wait();
                if (tok < g.L) {
                    // head h = (sample, head within the sample); O row of
                    // (sample, token) in the batch's stream-major token rows
                    size_t orow = (size_t)tok;
                    int hs = h;
                    if constexpr (BATCH) {
                        const int b = h / g.Hs;
                        hs = h - b * g.Hs;
                        orow = (size_t)batch_row(b, tok, g.nb, g.Lc, g.L);
                    }
                    uint4* dst = reinterpret_cast<uint4*>(g.o + orow * g.Hs * D + (size_t)hs * D + c);
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        uint4 w;
                        w.x = pack2(__uint_as_float(o[8 * q + 0]) * inv, __uint_as_float(o[8 * q + 1]) * inv);
                        w.y = pack2(__uint_as_float(o[8 * q + 2]) * inv, __uint_as_float(o[8 * q + 3]) * inv);
                        w.z = pack2(__uint_as_float(o[8 * q + 4]) * inv, __uint_as_float(o[8 * q + 5]) * inv);
                        w.w = pack2(__uint_as_float(o[8 * q + 6]) * inv, __uint_as_float(o[8 * q + 7]) * inv);
                        dst[q] = w;
                    }
                }
            }
        }
        tc_fence_before();
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::TMEM_COLS);
    }
}

// Merges the key-range parts of each split unit: one warp per query row,
// lane l owning columns l, l + 32, ...: O = sum_p 2^(m_p - m) O_p / l with
// m = max_p m_p and l = sum_p 2^(m_p - m) l_p (bases in the log2 domain of
// the numerators).
template <int D, bool BATCH>
__global__ void __launch_bounds__(256) attn_combine_kernel(const AttnArgs g, int n_split_units) {
    const int w = (int)((blockIdx.x * 256u + threadIdx.x) >> 5), lane = threadIdx.x & 31;
    if (w >= n_split_units * 2 * BQ) return;
    const int ug = w / (2 * BQ), r = w - ug * (2 * BQ);      // split unit over all samples, row
    const int n_split_s = g.units_s - g.n_full;
    const int smp = ug / n_split_s, u = ug - smp * n_split_s;
    const int unit = smp * g.units_s + g.n_full + u;
    const int h = unit / g.q_blocks;
    const int tok = (unit % g.q_blocks) * (2 * BQ) + r;
    if (tok >= g.L) return;
    const float2* ml = reinterpret_cast<const float2*>(g.part_ml);
    const size_t slot0 = (size_t)ug * g.split;                // = smp * n_split_s * split + u * split
    float m = -INFINITY;
    for (int p = 0; p < g.split; ++p) m = fmaxf(m, ml[(slot0 + p) * (2 * BQ) + r].x);
    float l = 0.f, acc[D / 32];
#pragma unroll
    for (int i = 0; i < D / 32; ++i) acc[i] = 0.f;
    for (int p = 0; p < g.split; ++p) {
        const size_t prow = (slot0 + p) * (2 * BQ) + r;
        const float2 mp = ml[prow];
        const float f = ex2(mp.x - m);
        l = fmaf(mp.y, f, l);
        const float* po = g.part_o + prow * D;
#pragma unroll
        for (int i = 0; i < D / 32; ++i) acc[i] = fmaf(f, po[lane + 32 * i], acc[i]);
    }
    size_t orow = (size_t)tok;
    int hs = h;
    if constexpr (BATCH) {
        const int b = h / g.Hs;
        hs = h - b * g.Hs;
        orow = (size_t)batch_row(b, tok, g.nb, g.Lc, g.L);
    }
    const float inv = 1.0f / l;
    __nv_bfloat16* dst = g.o + orow * g.Hs * D + (size_t)hs * D;
#pragma unroll
    for (int i = 0; i < D / 32; ++i) dst[lane + 32 * i] = __float2bfloat16_rn(acc[i] * inv);
}

// Units of a sample's last, partial round are split over the key range so
// that its CTAs fill the SMs: r = units mod SMs leftover units, each in
// min(8, SMs / r, steps) parts (none when the grid is whole rounds).
int attn_split(int units, int num_sms, int n_kv, int& n_full) {
    n_full = units;
    const int r = units % num_sms;
    if (r == 0) return 1;
    int split = num_sms / r;
    if (split > 8) split = 8;
    if (split > n_kv) split = n_kv;
    if (split < 2) return 1;
    n_full = units - r;
    return split;
}

template <int D, bool BATCH>
wdc_status launch(Ctx* c, const void* q, const void* k, const void* vt, int ldv, void* o, int H, int L, int Hs,
                  int Lc, cudaStream_t s) {
    using Cf = AttnCfg<D>;
    constexpr int BKV = Cf::BK;
    static bool attr = false;
    static bool regs_ok = false;
    if (!attr) {
        cudaFuncSetAttribute(attn_tc_kernel<D, BATCH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cf::SMEM);
        // the warpgroups' register requests must fit the launch allocation,
        // or setmaxnreg.inc would wait forever: refuse to launch otherwise
        cudaFuncAttributes fa;
        regs_ok = cudaFuncGetAttributes(&fa, attn_tc_kernel<D, BATCH>) == cudaSuccess &&
                  fa.maxThreadsPerBlock >= Cf::THREADS &&
                  (uint32_t)fa.numRegs * Cf::THREADS >= 128 * Cf::REGS_CONTROL + 256 * Cf::REGS_SOFTMAX;
        cudaGetLastError();
        attr = true;
    }
    if (!regs_ok) return fail(c, WDC_ERR_UNSUPPORTED, "attention kernel's register allocation is below its warpgroup split");
    CUtensorMap tq, tk, tv;
    std::string why;
    const uint64_t row = (uint64_t)D * 2, head = (uint64_t)L * D * 2;
    if (!encode_tmap_3d(&tq, q, D, L, H, row, head, 64, BQ, 1, &why) ||
        !encode_tmap_3d(&tk, k, D, L, H, row, head, 64, BKV, 1, &why) ||
        !encode_tmap_3d(&tv, vt, L, D, H, (uint64_t)ldv * 2, (uint64_t)ldv * D * 2, 64, D, 1, &why, true))
        return fail(c, WDC_ERR_CUDA, why);
    AttnArgs g;
    g.H = H;
    g.L = L;
    g.Hs = Hs;
    g.nb = H / Hs;
    g.Lc = Lc;
    g.n_kv = (L + BKV - 1) / BKV;
    g.q_blocks = (L + 2 * BQ - 1) / (2 * BQ);
    g.scale_log2 = 1.4426950408889634f / sqrtf((float)D);
    g.o = reinterpret_cast<__nv_bfloat16*>(o);
    g.err = c->err;
    g.units_s = Hs * g.q_blocks;
    g.split = attn_split(g.units_s, c->num_sms, g.n_kv, g.n_full);
    // the workspace holds num_sms part CTAs per sample of the model's batch
    if (!c->attn_part || g.nb > c->attn_part_samples) g.split = 1;
    if (g.split == 1) g.n_full = g.units_s;
    g.part_o = c->attn_part;
    g.part_ml = c->attn_ml;
    const int n_split = g.nb * (g.units_s - g.n_full);       // split units over all samples
    {
        LaunchScope ls(c, WDC_K_ATTN, s);
        attn_tc_kernel<D, BATCH><<<g.nb * (g.n_full + (g.units_s - g.n_full) * g.split), Cf::THREADS, Cf::SMEM, s>>>(
            tq, tk, tv, g);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("tcgen05 attention launch: ") + cudaGetErrorString(e));
    }
    if (n_split > 0) {
        LaunchScope ls(c, WDC_K_OTHER, s);
        const int threads = n_split * 2 * BQ * 32;
        attn_combine_kernel<D, BATCH><<<(threads + 255) / 256, 256, 0, s>>>(g, n_split);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("attention combine launch: ") + cudaGetErrorString(e));
    }
    return WDC_OK;
}

}  // namespace

// Any L: V^T rows are padded to ldv (a multiple of 8 tokens, so every TMA row
// starts on a 16-byte boundary); keys past L are zero-filled by TMA and masked.
bool tc_attention_supported(int L, int d) { return L > 0 && (d == 64 || d == 128); }

wdc_status tc_attention(Ctx* c, const void* q, const void* k, const void* vt, int ldv, void* o, int H, int L, int d,
                        int Hs, int Lc, cudaStream_t s) {
    if (((uintptr_t)q | (uintptr_t)k | (uintptr_t)vt | (uintptr_t)o) & 15)
        return fail(c, WDC_ERR_INVALID_ARG, "attention operands must be 16-byte aligned");
    if (ldv < L || ldv % 8) return fail(c, WDC_ERR_INVALID_ARG, "V^T row stride must be >= L and a multiple of 8");
    if (Hs <= 0 || H % Hs || Lc < 0 || Lc >= L) return fail(c, WDC_ERR_INVALID_ARG, "bad attention batch layout");
    if (Hs == H)
        return d == 64 ? launch<64, false>(c, q, k, vt, ldv, o, H, L, Hs, Lc, s)
                       : launch<128, false>(c, q, k, vt, ldv, o, H, L, Hs, Lc, s);
    return d == 64 ? launch<64, true>(c, q, k, vt, ldv, o, H, L, Hs, Lc, s)
                   : launch<128, true>(c, q, k, vt, ldv, o, H, L, Hs, Lc, s);
}

}  // namespace wdc
