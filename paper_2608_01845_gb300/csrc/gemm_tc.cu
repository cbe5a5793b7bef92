// Dense bf16 GEMM on the 5th-generation tensor cores (tcgen05, sm_103a) with
// the DiT's fused epilogues: C = epilogue(A W^T), A [M, K], W [N, K] bf16,
// fp32 accumulation in tensor memory.
//
// Persistent kernel, one CTA per SM, 6 warps:
//   warp 0      TMA producer: A (128 x 64) and W (256 x 64) tiles into a
//               4-stage shared-memory ring (128-byte swizzle), one mbarrier
//               pair per stage;
//   warp 1      MMA issuer: one thread issues tcgen05.mma 128x256x16 into one
//               of two TMEM accumulators (2 x 256 columns), commits the smem
//               stage back to the producer and the accumulator to the
//               epilogue;
//   warps 2-5   epilogue: tcgen05.ld 32 columns at a time (each warp owns its
//               32-lane TMEM quarter = 32 rows), bias / GELU / gated residual /
//               QKV scatter / unpatchify, 16-byte global stores; then release
//               the accumulator so the next tile's MMAs overlap this epilogue.
// Tiles are visited N-fastest inside groups of N tiles sized so a group's
// slab of W stays in L2 (about 40 MB), so W is read from DRAM about once and
// A once per group.
// Tails: TMA zero-fills rows past M / N and columns past K; the epilogue
// masks rows >= M.  Every mbarrier wait is bounded.
#include "dit_kernels.cuh"
#include "ptx.cuh"

#include <cudaTypedefs.h>

#include <mutex>

namespace wdc {

namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int kGemmThreads = 192;
constexpr uint32_t A_BYTES = BM * BK * 2;
constexpr uint32_t B_BYTES = BN * BK * 2;
constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
constexpr uint32_t TMEM_COLS = 2 * BN;
constexpr uint32_t IDESC = idesc_bf16(BM, BN);
constexpr size_t SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + 256;

struct GemmArgs {
    int M, N, K;
    int m_tiles, n_tiles, k_blocks;
    int group_n;            // pair kernel: N tiles per raster group
    Epi e;
    unsigned* err;
    // pair kernel, grouped launch: a second problem with the same N and K
    // (its own A, W, M and epilogue) whose tiles follow the first problem's
    int nprob;              // 1 or 2
    int M1, m_pairs1;
    Epi e1;
};

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
    __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ float2 unpack_bf16(uint32_t u) {
    __nv_bfloat162 h = *reinterpret_cast<__nv_bfloat162*>(&u);
    return __bfloat1622float2(h);
}

// Epilogue of 32 consecutive columns col0..col0+31 of one row.
__device__ __forceinline__ void epilogue_chunk(const Epi& e, int m, int col0, const uint32_t (&r)[32]) {
    float v[32];
    if (e.bias) {
        const float4* b4 = reinterpret_cast<const float4*>(e.bias + col0);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const float4 b = __ldg(b4 + j);
            v[4 * j + 0] = __uint_as_float(r[4 * j + 0]) + b.x;
            v[4 * j + 1] = __uint_as_float(r[4 * j + 1]) + b.y;
            v[4 * j + 2] = __uint_as_float(r[4 * j + 2]) + b.z;
            v[4 * j + 3] = __uint_as_float(r[4 * j + 3]) + b.w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
    }
    if (e.gelu) {
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = gelu_tanh_f(v[j]);
    }
    if (e.mode == kEpiStore || e.mode == kEpiResid) {
        __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(e.out) + (size_t)m * e.ldo + col0;
        uint4* o4 = reinterpret_cast<uint4*>(out);
        if (e.mode == kEpiResid) {
            const int rm = e.res_rows > 0 ? m % e.res_rows : m;
            const uint4* r4 = reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(e.res) +
                                                             (size_t)rm * e.ldo + col0);
            float g[32];
            if (e.gate) {
                const float4* g4 = reinterpret_cast<const float4*>(e.gate + col0);
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const float4 t = __ldg(g4 + j);
                    g[4 * j] = t.x; g[4 * j + 1] = t.y; g[4 * j + 2] = t.z; g[4 * j + 3] = t.w;
                }
            } else {
#pragma unroll
                for (int j = 0; j < 32; ++j) g[j] = 1.0f;
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint4 rr = r4[q];
                const uint32_t w[4] = {rr.x, rr.y, rr.z, rr.w};
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                    const float2 f = unpack_bf16(w[t]);
                    const int j = 8 * q + 2 * t;
                    v[j] = fmaf(g[j], v[j], f.x);
                    v[j + 1] = fmaf(g[j + 1], v[j + 1], f.y);
                }
            }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint4 w;
            w.x = pack_bf16(v[8 * q + 0], v[8 * q + 1]);
            w.y = pack_bf16(v[8 * q + 2], v[8 * q + 3]);
            w.z = pack_bf16(v[8 * q + 4], v[8 * q + 5]);
            w.w = pack_bf16(v[8 * q + 6], v[8 * q + 7]);
            o4[q] = w;
        }
        return;
    }
    if (e.mode == kEpiQKV) {
        const int which = col0 / e.D, c = col0 % e.D, dd0 = c % e.d;
        int b, tok;
        batch_token(e.row_off + m, e.nb, e.Lc, e.L, b, tok);
        const size_t h = (size_t)b * e.H + c / e.d;
        if (which < 2) {
            __nv_bfloat16* base = reinterpret_cast<__nv_bfloat16*>(which == 0 ? e.q : e.k) +
                                  (h * e.L + tok) * e.d + dd0;
            uint4* o4 = reinterpret_cast<uint4*>(base);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                uint4 w;
                w.x = pack_bf16(v[8 * q + 0], v[8 * q + 1]);
                w.y = pack_bf16(v[8 * q + 2], v[8 * q + 3]);
                w.z = pack_bf16(v[8 * q + 4], v[8 * q + 5]);
                w.w = pack_bf16(v[8 * q + 6], v[8 * q + 7]);
                o4[q] = w;
            }
        } else {
            __half* base = reinterpret_cast<__half*>(e.vt) + (h * e.d + dd0) * e.ldv + tok;
            bool sat = false;
#pragma unroll
            for (int j = 0; j < 32; ++j) base[(size_t)j * e.ldv] = to_vt_half(v[j], sat);
            if (sat && e.err) atomicOr(e.err, kErrVSaturated);
        }
        return;
    }
    // kEpiUnpatch: fp32 scatter into the latent
    Epi e2 = e;
    e2.bias = nullptr;
    e2.gelu = 0;
#pragma unroll 4
    for (int j = 0; j < 32; ++j) epi_apply<__nv_bfloat16>(e2, m, col0 + j, v[j]);
}

__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ GemmArgs g) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
    uint64_t* empty = full + STAGES;
    uint64_t* tfull = empty + STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* mma_done = tempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], 4);
        }
        mbar_init(mma_done, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tmap(&tmA);
        prefetch_tmap(&tmB);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, TMEM_COLS);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const int num_tiles = g.m_tiles * g.n_tiles;

    if (warp == 0) {
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t armed_phase[STAGES];
            bool armed[STAGES];
            for (int s = 0; s < STAGES; ++s) armed[s] = false;
            bool ok = true;
            for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
                const int m_blk = tile / g.n_tiles, n_blk = tile % g.n_tiles;
                for (int kb = 0; kb < g.k_blocks; ++kb) {
                    if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, g.err)) { ok = false; break; }
                    mbar_arrive_expect_tx(&full[stage], STAGE_BYTES);
                    uint8_t* sa = smem + stage * STAGE_BYTES;
                    tma_load_2d(sa, &tmA, &full[stage], kb * BK, m_blk * BM);
                    tma_load_2d(sa + A_BYTES, &tmB, &full[stage], kb * BK, n_blk * BN);
                    armed[stage] = true;
                    armed_phase[stage] = phase;
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
            }
            // drain: every issued copy has landed before the CTA may exit
            for (int s = 0; s < STAGES; ++s) {
                if (!armed[s]) continue;
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(&full[s], armed_phase[s]) && globaltimer() - t0 < kWaitLimitNs) {
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
                if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, g.err)) break;
                tc_fence_after();
                const uint32_t d = tmem_base + (uint32_t)(acc * BN);
                for (int kb = 0; kb < g.k_blocks; ++kb) {
                    if (!mbar_wait(&full[stage], phase, abort_flag, g.err)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(smem + stage * STAGE_BYTES);
                    const uint32_t b0 = a0 + A_BYTES;
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k)
                        tc_mma(d, sdesc_sw128(a0 + k * 32), sdesc_sw128(b0 + k * 32), IDESC, (kb | k) != 0);
                    tc_commit(&empty[stage]);
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
                tc_commit(&tfull[acc]);
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1u;
            }
            // all MMAs issued by this thread have completed before TMEM is freed
            tc_commit(mma_done);
            const unsigned long long t0 = globaltimer();
            while (!mbar_try_wait(mma_done, 0) && globaltimer() - t0 < kWaitLimitNs) {
            }
        }
    } else {
        const int lg = warp & 3;   // TMEM lane quarter this warp may access
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
            const int m_blk = tile / g.n_tiles, n_blk = tile % g.n_tiles;
            if (!mbar_wait(&tfull[acc], acc_phase, abort_flag, g.err)) break;
            tc_fence_after();
            const int m = m_blk * BM + lg * 32 + lane;
            const uint32_t taddr = tmem_base + ((uint32_t)(lg * 32) << 16) + (uint32_t)(acc * BN);
            for (int c0 = 0; c0 < BN; c0 += 32) {
                const int col0 = n_blk * BN + c0;
                if (col0 >= g.N) break;
                uint32_t r[32];
                tmem_ld32(taddr + c0, r);
                tmem_ld_wait();
                if (m < g.M) epilogue_chunk(g.e, m, col0, r);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[acc]);
            acc ^= 1;
            if (acc == 0) acc_phase ^= 1u;
        }
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, TMEM_COLS);
    }
}

// ---------------------------------------------------------------------------
// CTA-pair variant (clusters of 2, tcgen05 .cta_group::2): each pair computes a
// 256 x 256 tile with 256 x 256 x 16 MMAs issued by the even CTA; each CTA
// holds its 128 rows of A and its 128-row half of the W tile (32 KB per stage,
// 6 stages), so twice the MMA work is buffered per shared-memory byte.  Both
// CTAs' tile copies complete on the even CTA's mbarrier (the pair form of the
// tensor copy), which the even CTA arms with both CTAs' bytes; the even CTA's
// commits release both CTAs' stages and accumulators.  The
// pair allocation is collective (both CTAs receive the same TMEM base; the
// leader's base is used for every access and a mismatch is reported), and two
// 256-column accumulators let a tile's epilogue overlap the next tile's MMAs.
constexpr int STAGES2 = 7;
constexpr uint32_t A2_BYTES = 128 * BK * 2;
constexpr uint32_t B2_BYTES = 128 * BK * 2;                  // half of the 256-row W tile
constexpr uint32_t STAGE2_BYTES = A2_BYTES + B2_BYTES;
constexpr uint32_t TMEM2_COLS = 512;
constexpr uint32_t IDESC2 = idesc_bf16(256, 256);
constexpr size_t SMEM2_BYTES = STAGES2 * STAGE2_BYTES + 1024 + 512;

// Pair-kernel raster: the N tiles are split into groups of group_n; inside a
// group the tiles run N-fastest over every 256-row M block.  A group's slab
// of W (group_n * 256 rows * K) stays in L2 while A streams through once per
// group, so W is read from DRAM about once and A once per group.
__device__ __forceinline__ void pair_tile(const GemmArgs& g, int m_pairs, int tile, int& m_blk, int& n_blk) {
    const int per_group = m_pairs * g.group_n;
    const int grp = tile / per_group, r = tile - grp * per_group;
    const int n_first = grp * g.group_n;
    const int width = min(g.group_n, g.n_tiles - n_first);
    m_blk = r / width;
    n_blk = n_first + (r - m_blk * width);
}

// Tile `tile` of a (possibly grouped) pair launch: problem index, 256-row M
// block and N block.  The first problem's tiles use the raster groups, the
// second problem's follow in plain N-fastest order, so they fill the pairs
// the first problem leaves idle in its last wave.
__device__ __forceinline__ int grouped_tile(const GemmArgs& g, int m_pairs0, int tiles0, int tile, int& m_blk,
                                            int& n_blk) {
    if (tile < tiles0) {
        pair_tile(g, m_pairs0, tile, m_blk, n_blk);
        return 0;
    }
    const int r = tile - tiles0;
    m_blk = r / g.n_tiles;
    n_blk = r - m_blk * g.n_tiles;
    return 1;
}

__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmA1, const __grid_constant__ CUtensorMap tmB1,
                    const __grid_constant__ GemmArgs g) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES2 * STAGE2_BYTES);   // even CTA: both halves landed
    uint64_t* empty = full + STAGES2;
    uint64_t* tfull = empty + STAGES2;         // [2]
    uint64_t* tempty = tfull + 2;              // [2] even CTA: both CTAs' epilogues are done
    uint64_t* mma_done = tempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const int cluster_id = blockIdx.x >> 1, n_clusters = gridDim.x >> 1;
    const int m_pairs = (g.m_tiles + 1) >> 1;  // 256-row tiles (m_tiles counts 128-row tiles)
    const int tiles0 = m_pairs * g.n_tiles;
    const int num_tiles = tiles0 + (g.nprob > 1 ? g.m_pairs1 * g.n_tiles : 0);
    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES2; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], 8);          // 4 epilogue warps in each CTA
        }
        mbar_init(mma_done, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tmap(&tmA);
        prefetch_tmap(&tmB);
        if (g.nprob > 1) {
            prefetch_tmap(&tmA1);
            prefetch_tmap(&tmB1);
        }
    }
    if (warp == 1) {
        tmem_alloc2(tmem_slot, TMEM2_COLS);
        tmem_relinquish2();
    }
    __syncthreads();
    cluster_sync_all();
    tc_fence_after();
    const uint32_t own_base = *tmem_slot;
    const uint32_t tmem = rank == 0 ? own_base : ld_shared_cluster_u32(mapa_shared(smem_u32(tmem_slot), 0));
    if (threadIdx.x == 0 && tmem != own_base) atomicOr(g.err, kErrTmem);
    const uint32_t leader_tempty0 = mapa_shared(smem_u32(&tempty[0]), 0);
    const uint32_t leader_tempty1 = mapa_shared(smem_u32(&tempty[1]), 0);

    if (warp == 0) {
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t armed_phase[STAGES2];
            bool armed[STAGES2];
            for (int s = 0; s < STAGES2; ++s) armed[s] = false;
            bool ok = true;
            for (int tile = cluster_id; tile < num_tiles && ok; tile += n_clusters) {
                int mb, nb;
                const int prob = grouped_tile(g, m_pairs, tiles0, tile, mb, nb);
                const CUtensorMap* mA = prob ? &tmA1 : &tmA;
                const CUtensorMap* mB = prob ? &tmB1 : &tmB;
                const int m0 = mb * 256 + (int)rank * 128;
                const int n0 = nb * BN + (int)rank * 128;
                for (int kb = 0; kb < g.k_blocks; ++kb) {
                    if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, g.err)) { ok = false; break; }
                    if (rank == 0) mbar_arrive_expect_tx(&full[stage], 2 * STAGE2_BYTES);
                    const uint32_t fb = mapa_shared(smem_u32(&full[stage]), 0);
                    uint8_t* sa = smem + stage * STAGE2_BYTES;
                    tma_load_2d_pair(sa, mA, fb, kb * BK, m0);
                    tma_load_2d_pair(sa + A2_BYTES, mB, fb, kb * BK, n0);
                    armed[stage] = true;
                    armed_phase[stage] = phase;
                    if (++stage == STAGES2) { stage = 0; phase ^= 1u; }
                }
            }
            // drain: every copy of the pair has landed (even CTA's full) and the
            // MMAs have released every stage (both CTAs' empty)
            for (int s = 0; s < STAGES2; ++s) {
                if (!armed[s]) continue;
                if (rank == 0) {
                    const unsigned long long t0 = globaltimer();
                    while (!mbar_try_wait(&full[s], armed_phase[s]) && globaltimer() - t0 < kWaitLimitNs) {
                    }
                }
                const unsigned long long t1 = globaltimer();
                while (!mbar_try_wait(&empty[s], armed_phase[s]) && globaltimer() - t1 < kWaitLimitNs) {
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0 && rank == 0) {
            // MMA issuer for the pair
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            for (int tile = cluster_id; tile < num_tiles && ok; tile += n_clusters) {
                if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, g.err)) break;
                tc_fence_after();
                const uint32_t d = tmem + (uint32_t)(acc * BN);
                for (int kb = 0; kb < g.k_blocks; ++kb) {
                    if (!mbar_wait(&full[stage], phase, abort_flag, g.err)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(smem + stage * STAGE2_BYTES);
                    const uint32_t b0 = a0 + A2_BYTES;
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k)
                        tc_mma2(d, sdesc_sw128(a0 + k * 32), sdesc_sw128(b0 + k * 32), IDESC2, (kb | k) != 0);
                    tc_commit2_mc(&empty[stage], (uint16_t)0x3);
                    if (++stage == STAGES2) { stage = 0; phase ^= 1u; }
                }
                tc_commit2_mc(&tfull[acc], (uint16_t)0x3);
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1u;
            }
            tc_commit2_mc(mma_done, (uint16_t)0x1);
            const unsigned long long t0 = globaltimer();
            while (!mbar_try_wait(mma_done, 0) && globaltimer() - t0 < kWaitLimitNs) {
            }
        }
    } else {
        const int lg = warp & 3;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int tile = cluster_id; tile < num_tiles; tile += n_clusters) {
            int mb, n_blk;
            const int prob = grouped_tile(g, m_pairs, tiles0, tile, mb, n_blk);
            const int Mp = prob ? g.M1 : g.M;
            const int mrow = mb * 256 + (int)rank * 128;
            if (!mbar_wait(&tfull[acc], acc_phase, abort_flag, g.err)) break;
            tc_fence_after();
            const int m = mrow + lg * 32 + lane;
            const uint32_t taddr = tmem + ((uint32_t)(lg * 32) << 16) + (uint32_t)(acc * BN);
            for (int c0 = 0; c0 < BN; c0 += 32) {
                const int col0 = n_blk * BN + c0;
                if (col0 >= g.N) break;
                uint32_t r[32];
                tmem_ld32(taddr + c0, r);
                tmem_ld_wait();
                if (m < Mp) {
                    // two direct calls (each reads its epilogue from the
                    // kernel parameters; a selected reference would copy it)
                    if (prob) epilogue_chunk(g.e1, m, col0, r);
                    else epilogue_chunk(g.e, m, col0, r);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if (rank == 0) mbar_arrive(&tempty[acc]);
                else mbar_arrive_remote(acc == 0 ? leader_tempty0 : leader_tempty1);
            }
            acc ^= 1;
            if (acc == 0) acc_phase ^= 1u;
        }
    }
    __syncthreads();
    cluster_sync_all();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc2(own_base, TMEM2_COLS);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
        else
            cudaGetLastError();
    });
    return fn;
}

}  // namespace

bool encode_tmap_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                    uint32_t box_inner, uint32_t box_outer, std::string* why) {
    auto fn = get_encode();
    if (!fn) { if (why) *why = "cuTensorMapEncodeTiled unavailable"; return false; }
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t es[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) { if (why) *why = "cuTensorMapEncodeTiled failed: " + std::to_string((int)r); return false; }
    return true;
}

bool encode_tmap_3d(CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t s1_bytes,
                    uint64_t s2_bytes, uint32_t b0, uint32_t b1, uint32_t b2, std::string* why, bool f16) {
    auto fn = get_encode();
    if (!fn) { if (why) *why = "cuTensorMapEncodeTiled unavailable"; return false; }
    cuuint64_t dims[3] = {d0, d1, d2};
    cuuint64_t strides[2] = {s1_bytes, s2_bytes};
    cuuint32_t box[3] = {b0, b1, b2};
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = fn(map, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3,
                    const_cast<void*>(base), dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) { if (why) *why = "cuTensorMapEncodeTiled failed: " + std::to_string((int)r); return false; }
    return true;
}

bool tc_gemm_supported(int M, int N, int K) { return M > 0 && N > 0 && K > 0 && N % 32 == 0 && K % 8 == 0; }

namespace {

wdc_status check_operands(Ctx* c, const void* A, const void* W, const Epi& e) {
    if (((uintptr_t)A & 15) || ((uintptr_t)W & 15)) return fail(c, WDC_ERR_INVALID_ARG, "GEMM operands must be 16-byte aligned");
    if ((e.mode == kEpiStore || e.mode == kEpiResid) &&
        (e.ldo % 8 || ((uintptr_t)e.out & 15) || (e.res && ((uintptr_t)e.res & 15))))
        return fail(c, WDC_ERR_INVALID_ARG, "GEMM output must be 16-byte aligned with ldo % 8 == 0");
    if (e.bias && ((uintptr_t)e.bias & 15)) return fail(c, WDC_ERR_INVALID_ARG, "bias must be 16-byte aligned");
    if (e.gate && ((uintptr_t)e.gate & 15)) return fail(c, WDC_ERR_INVALID_ARG, "gate must be 16-byte aligned");
    if (e.mode == kEpiQKV && (e.D % 32 || e.d % 32)) return fail(c, WDC_ERR_UNSUPPORTED, "QKV epilogue needs d % 32 == 0");
    return WDC_OK;
}

void set_attrs() {
    static bool attr_set = false;
    if (!attr_set) {
        cudaFuncSetAttribute(gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES);
        cudaFuncSetAttribute(gemm_tc2_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM2_BYTES);
        attr_set = true;
    }
}

GemmArgs make_args(Ctx* c, int M, int N, int K, const Epi& e) {
    GemmArgs g{};
    g.M = M;
    g.N = N;
    g.K = K;
    g.m_tiles = (M + BM - 1) / BM;
    g.n_tiles = (N + BN - 1) / BN;
    g.k_blocks = (K + BK - 1) / BK;
    // raster groups: a W slab of at most ~40 MB per group (L2 is 126 MB,
    // shared with the streamed A and the output), as few groups as that
    // allows.  For deep K (> 4096) a 256-row slab of A is itself large
    // and re-reading A per group costs more than it saves (measured on the
    // 17776 x 3072 x 12288 MLP-down GEMM): plain N-fastest order there.
    g.group_n = g.n_tiles;
    if (K <= 4096) {
        const double slab_per_tile = 256.0 * K * 2.0;
        int gn = (int)(40.0e6 / slab_per_tile);
        gn = gn < 1 ? 1 : (gn > g.n_tiles ? g.n_tiles : gn);
        const int groups = (g.n_tiles + gn - 1) / gn;
        g.group_n = (g.n_tiles + groups - 1) / groups;  // balance the groups
    }
    g.e = e;
    g.err = c->err;
    g.nprob = 1;
    return g;
}

// Pair-kernel launch: a persistent grid of as many CTA pairs as can be
// resident, capped by the tile count.
wdc_status launch_pair(Ctx* c, const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& ta1,
                       const CUtensorMap& tb1, const GemmArgs& g, cudaStream_t s) {
    const int tiles = ((g.m_tiles + 1) / 2) * g.n_tiles + (g.nprob > 1 ? g.m_pairs1 * g.n_tiles : 0);
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(kGemmThreads, 1, 1);
    cfg.dynamicSmemBytes = SMEM2_BYTES;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    static int max_clusters = 0;
    if (max_clusters == 0) {
        cfg.gridDim = dim3(c->num_sms, 1, 1);
        if (cudaOccupancyMaxActiveClusters(&max_clusters, gemm_tc2_kernel, &cfg) != cudaSuccess || max_clusters < 1) {
            cudaGetLastError();
            max_clusters = c->num_sms / 2;
        }
    }
    int clusters = max_clusters < c->num_sms / 2 ? max_clusters : c->num_sms / 2;
    if (tiles < clusters) clusters = tiles;
    cfg.gridDim = dim3(2 * clusters, 1, 1);
    cudaLaunchKernelEx(&cfg, gemm_tc2_kernel, ta, tb, ta1, tb1, g);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("tcgen05 GEMM launch: ") + cudaGetErrorString(err));
    return WDC_OK;
}

}  // namespace

wdc_status tc_gemm(Ctx* c, const void* A, const void* W, int M, int N, int K, const Epi& e, cudaStream_t s) {
    wdc_status st = check_operands(c, A, W, e);
    if (st) return st;
    set_attrs();
    const bool pair = M >= 256 && c->num_sms >= 2;
    CUtensorMap ta, tb;
    std::string why;
    if (!encode_tmap_2d(&ta, A, (uint64_t)K, (uint64_t)M, (uint64_t)K * 2, BK, BM, &why) ||
        !encode_tmap_2d(&tb, W, (uint64_t)K, (uint64_t)N, (uint64_t)K * 2, BK, pair ? BN / 2 : BN, &why))
        return fail(c, WDC_ERR_CUDA, why);
    const GemmArgs g = make_args(c, M, N, K, e);
    if (pair) return launch_pair(c, ta, tb, ta, tb, g, s);
    const int tiles = g.m_tiles * g.n_tiles;
    const int grid = tiles < c->num_sms ? tiles : c->num_sms;
    gemm_tc_kernel<<<grid, kGemmThreads, SMEM_BYTES, s>>>(ta, tb, g);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return fail(c, WDC_ERR_CUDA, std::string("tcgen05 GEMM launch: ") + cudaGetErrorString(err));
    return WDC_OK;
}

// Two GEMMs with the same N and K in one launch of the pair kernel (the
// dual-stream blocks' video rows and condition rows): problem 1's tiles
// follow problem 0's, filling the pairs problem 0 leaves idle in its last
// wave.  When problem 0 is too short for the pair kernel the two run as two
// launches on the stream.
wdc_status tc_gemm_grouped(Ctx* c, const void* A0, const void* W0, int M0, const Epi& e0, const void* A1,
                           const void* W1, int M1, const Epi& e1, int N, int K, cudaStream_t s) {
    if (M1 <= 0) return tc_gemm(c, A0, W0, M0, N, K, e0, s);
    if (M0 <= 0) return tc_gemm(c, A1, W1, M1, N, K, e1, s);
    if (M0 < 256 || c->num_sms < 2) {
        wdc_status st = tc_gemm(c, A0, W0, M0, N, K, e0, s);
        return st ? st : tc_gemm(c, A1, W1, M1, N, K, e1, s);
    }
    wdc_status st = check_operands(c, A0, W0, e0);
    if (!st) st = check_operands(c, A1, W1, e1);
    if (st) return st;
    set_attrs();
    CUtensorMap ta, tb, ta1, tb1;
    std::string why;
    if (!encode_tmap_2d(&ta, A0, (uint64_t)K, (uint64_t)M0, (uint64_t)K * 2, BK, BM, &why) ||
        !encode_tmap_2d(&tb, W0, (uint64_t)K, (uint64_t)N, (uint64_t)K * 2, BK, BN / 2, &why) ||
        !encode_tmap_2d(&ta1, A1, (uint64_t)K, (uint64_t)M1, (uint64_t)K * 2, BK, BM, &why) ||
        !encode_tmap_2d(&tb1, W1, (uint64_t)K, (uint64_t)N, (uint64_t)K * 2, BK, BN / 2, &why))
        return fail(c, WDC_ERR_CUDA, why);
    GemmArgs g = make_args(c, M0, N, K, e0);
    g.nprob = 2;
    g.M1 = M1;
    g.m_pairs1 = (M1 + 255) / 256;
    g.e1 = e1;
    return launch_pair(c, ta, tb, ta1, tb1, g, s);
}

}  // namespace wdc
