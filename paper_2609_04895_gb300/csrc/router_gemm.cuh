// Router heads on the 5th-generation tensor cores (sm_103a).
//
// For one layer l the three heads are one GEMM (Sec. 2, 3.2, 3.3):
//   Z_l[rows, H*N] = H_l[rows, d] . W_cat,l[H*N, d]^T,   rows = (stream, token)
// bf16 operands staged by TMA into 128-byte-swizzled shared memory, fp32
// accumulators in TMEM (tcgen05.mma issued by one thread), then a per-row
// softmax of every head read back with tcgen05.ld.  A tile is 128 rows =
// SB streams x TB tokens of one layer.  The kernel is persistent: one CTA
// per SM walks tiles in layer-major order so that the CTAs running together
// share one layer's weights in L2.
//
// Warp roles (192 threads): warp 0 = TMA producer, warp 1 = TMEM allocator
// and MMA issuer, warps 2..5 = epilogue (warp w reads TMEM lanes
// 32*(w%4) .. +31, i.e. tile rows of that lane quarter).
#pragma once

#include "crc_device.cuh"

namespace crc {

constexpr int pow2ceil_i(int x) {
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}
constexpr int imax(int a, int b) { return a > b ? a : b; }
constexpr int imin(int a, int b) { return a < b ? a : b; }

template <int NH, int H>
struct RouterCfg {
    static constexpr int BM = 128;                       // tile rows (TMEM lanes)
    static constexpr int BK = 64;                        // 64 bf16 = one 128-byte swizzle row
    static constexpr int NCOL = NH * H;                  // accumulator columns
    static constexpr int NMMA = NCOL <= 256 ? 1 : 2;     // MMAs per K step (N <= 256 each)
    static constexpr int NCH = NCOL / NMMA;              // columns per MMA
    static constexpr int ACC_COLS = pow2ceil_i(imax(32, NCOL));
    static constexpr int NACC = (2 * ACC_COLS <= 512) ? 2 : 1;   // TMEM double buffering
    static constexpr int TMEM_COLS = ACC_COLS * NACC;
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = NCOL * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    // Epilogue staging for TMA stores: per epilogue warp two 32 x 32 fp32
    // tiles (128-byte rows, 128-byte swizzle), used when a head is >= 32 wide.
    static constexpr bool TMA_STORE = NH >= 32;
    static constexpr int STAGING_BYTES = TMA_STORE ? 4 * 2 * 4096 : 0;
    static constexpr int STAGES =
        imin(8, (232448 - 1024 - 256 - STAGING_BYTES) / STAGE_BYTES);
    static constexpr int B_BOX_ROWS = NMMA == 1 ? NCOL : NCH;   // TMA box rows <= 256
    static constexpr int B_BOXES = NCOL / B_BOX_ROWS;
    static constexpr uint32_t IDESC = idesc_bf16_f32(BM, NCH);
    static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + STAGING_BYTES + 256;
    static constexpr int THREADS = 192;

    static_assert(NH % 16 == 0 && NH >= 16 && NH <= 128, "experts per head");
    static_assert(NCH % 16 == 0 && NCH >= 16 && NCH <= 256, "MMA N");
    static_assert(TMEM_COLS <= 512, "TMEM columns");
    static_assert(STAGES >= 2, "pipeline depth");
    static_assert((A_BYTES % 1024) == 0 && (B_BYTES % 1024) == 0, "swizzle atom alignment");
};

struct RouterArgs {
    float* scores;       // [B][Ts][L][3][NH]
    uint32_t* err;       // latched device error
    int B, L, d;
    int t_begin;         // token coordinate of the first token of this call
    int T_ext;           // tokens in this call
    int SB, TB;          // a tile is SB streams x TB tokens
    int n_sb, n_tb;
    int num_tiles;       // L * n_sb * n_tb
    int kblocks;         // ceil(d / 64)
};

// ---------------------------------------------------------------------------
// Softmax arithmetic, shared by the router and the fused epilogues so that
// both produce the same bits.  exp(z - m) = 2^(z*log2(e) - m*log2(e)): one
// FMA per score and the SFU base-2 exponential (approximate, subnormal
// results flushed to zero).  Scores go in pairs (2j, 2j+1) through packed
// f32x2 instructions, each lane rounded like its scalar form.  The head sum
// is (sum over the first half of the experts) + (sum over the second half),
// each half's sum the total of two running partial sums (even and odd
// positions, in order); then p = e * (1 / sum), the reciprocal rounded to
// nearest.  (Halves let two CTAs that hold one half each agree on the sum.)
// ---------------------------------------------------------------------------
constexpr float kLog2E = 1.4426950408889634f;

__device__ __forceinline__ uint64_t f2pack(float a, float b) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
    return r;
}
__device__ __forceinline__ void f2unpack(uint64_t v, float& a, float& b) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}
__device__ __forceinline__ uint64_t f2fma(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}
__device__ __forceinline__ uint64_t f2add(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t f2mul(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ float ex2_sfu(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

// Running maximum over W scores (W even).
template <int W>
__device__ __forceinline__ float max_of(const float* z, float m) {
#pragma unroll
    for (int i = 0; i < W; i += 2) m = fmax3(m, z[i], z[i + 1]);
    return m;
}

// exp(z - m) of a head, in place, chunk after chunk, with its running sum.
struct HeadExp {
    uint64_t sum, k, b;
    __device__ __forceinline__ void init(float m) {
        const float nb = -__fmul_rn(m, kLog2E);
        k = f2pack(kLog2E, kLog2E);
        b = f2pack(nb, nb);
        sum = f2pack(0.f, 0.f);
    }
    template <int W>
    __device__ __forceinline__ void exp_in_place(float* z) {
#pragma unroll
        for (int i = 0; i < W; i += 2) {
            float u, v;
            f2unpack(f2fma(f2pack(z[i], z[i + 1]), k, b), u, v);
            z[i] = ex2_sfu(u);
            z[i + 1] = ex2_sfu(v);
            sum = f2add(sum, f2pack(z[i], z[i + 1]));
        }
    }
    // this accumulator's sum (one half of a head)
    __device__ __forceinline__ float part() const {
        float u, v;
        f2unpack(sum, u, v);
        return __fadd_rn(u, v);
    }
};

// 1 / (first-half sum + second-half sum): a head's normaliser.
__device__ __forceinline__ float head_inv(float s0, float s1) { return __frcp_rn(__fadd_rn(s0, s1)); }

// z <- z * r (probabilities from exps), W even.
template <int W>
__device__ __forceinline__ void scale_in_place(float* z, float r) {
    const uint64_t rr = f2pack(r, r);
#pragma unroll
    for (int i = 0; i < W; i += 2) f2unpack(f2mul(f2pack(z[i], z[i + 1]), rr), z[i], z[i + 1]);
}

// From the native and Temporal exps: z <- p^R = e^R * r^R and
// y <- s^T = p^R + e^T * r^T, product and sum rounded separately as when the
// scan adds the stored p^R and p^T.  Scalar on purpose: a packed multiply
// followed by a packed add may be fused into one packed FMA by the assembler,
// which rounds once.
template <int W>
__device__ __forceinline__ void retention_in_place(float* z, float* y, float rR, float rT) {
#pragma unroll
    for (int i = 0; i < W; ++i) {
        z[i] = __fmul_rn(z[i], rR);
        y[i] = __fadd_rn(z[i], __fmul_rn(y[i], rT));
    }
}

// Softmax of one head held in registers, in place.
template <int NH>
__device__ __forceinline__ void head_softmax(float (&z)[NH]) {
    const float m = max_of<NH>(z, -INFINITY);
    HeadExp h0, h1;
    h0.init(m);
    h1.init(m);
    h0.exp_in_place<NH / 2>(z);
    h1.exp_in_place<NH / 2>(z + NH / 2);
    scale_in_place<NH>(z, head_inv(h0.part(), h1.part()));
}

template <int NH, int H>
__global__ void __launch_bounds__(192, 1)
    router_heads_kernel(const __grid_constant__ CUtensorMap tmap_h,
                        const __grid_constant__ CUtensorMap tmap_w,
                        const __grid_constant__ CUtensorMap tmap_s, RouterArgs a) {
    using Cfg = RouterCfg<NH, H>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* tiles = smem;
    uint8_t* staging = smem + Cfg::STAGES * Cfg::STAGE_BYTES;          // 1024-aligned
    uint64_t* full_bar =
        reinterpret_cast<uint64_t*>(staging + Cfg::STAGING_BYTES);
    uint64_t* empty_bar = full_bar + Cfg::STAGES;
    uint64_t* tfull_bar = empty_bar + Cfg::STAGES;
    uint64_t* tempty_bar = tfull_bar + Cfg::NACC;
    uint64_t* drain_bar = tempty_bar + Cfg::NACC;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < Cfg::STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int s = 0; s < Cfg::NACC; ++s) {
            mbar_init(&tfull_bar[s], 1);
            mbar_init(&tempty_bar[s], 4);
        }
        mbar_init(drain_bar, 1);
        fence_mbar_init();
        tma_prefetch_desc(&tmap_h);
        tma_prefetch_desc(&tmap_w);
        if (Cfg::TMA_STORE) tma_prefetch_desc(&tmap_s);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const int tiles_per_layer = a.n_sb * a.n_tb;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA
        if (lane == 0) {
            const uint64_t pol_h = l2_evict_first_policy();   // streamed once
            const uint64_t pol_w = l2_evict_last_policy();    // reused by every tile
            int stage = 0;
            uint32_t phase = 0;
            int issued = 0, failed = 0;
            for (int tile = blockIdx.x; tile < a.num_tiles && !failed; tile += gridDim.x) {
                const int l = tile / tiles_per_layer;
                const int r = tile % tiles_per_layer;
                const int sb = r / a.n_tb, tb = r % a.n_tb;
                for (int kb = 0; kb < a.kblocks; ++kb) {
                    if (!mbar_wait(&empty_bar[stage], phase ^ 1)) {
                        latch_error(a.err, CRC_ETIMEOUT);
                        failed = 1;
                        break;
                    }
                    uint8_t* sa = tiles + stage * Cfg::STAGE_BYTES;
                    uint8_t* sb_ = sa + Cfg::A_BYTES;
                    mbar_arrive_expect_tx(&full_bar[stage], Cfg::STAGE_BYTES);
                    tma_load_4d(sa, &tmap_h, &full_bar[stage], kb * Cfg::BK, l,
                                a.t_begin + tb * a.TB, sb * a.SB, pol_h);
#pragma unroll
                    for (int c = 0; c < Cfg::B_BOXES; ++c)
                        tma_load_3d(sb_ + c * Cfg::B_BOX_ROWS * 128, &tmap_w, &full_bar[stage],
                                    kb * Cfg::BK, c * Cfg::B_BOX_ROWS, l, pol_w);
                    ++issued;
                    if (++stage == Cfg::STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
            }
            // Never leave with copies in flight: wait for every issued stage to land.
            int s = stage;
            uint32_t ph = phase;
            for (int k = 0; k < imin(issued, Cfg::STAGES); ++k) {
                if (--s < 0) {
                    s = Cfg::STAGES - 1;
                    ph ^= 1;
                }
                if (!mbar_wait(&full_bar[s], ph)) latch_error(a.err, CRC_ETIMEOUT);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA
        if (lane == 0) {
            int stage = 0, acc = 0;
            uint32_t phase = 0, acc_phase = 0;
            int failed = 0;
            for (int tile = blockIdx.x; tile < a.num_tiles && !failed; tile += gridDim.x) {
                if (!mbar_wait(&tempty_bar[acc], acc_phase ^ 1)) {
                    latch_error(a.err, CRC_ETIMEOUT);
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * Cfg::ACC_COLS);
                for (int kb = 0; kb < a.kblocks; ++kb) {
                    if (!mbar_wait(&full_bar[stage], phase)) {
                        latch_error(a.err, CRC_ETIMEOUT);
                        failed = 1;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(tiles + stage * Cfg::STAGE_BYTES);
                    const uint32_t sb_ = sa + Cfg::A_BYTES;
#pragma unroll
                    for (int kk = 0; kk < Cfg::BK / 16; ++kk) {
                        const uint64_t adesc = sw128_kmajor_desc(sa + kk * 32);
#pragma unroll
                        for (int c = 0; c < Cfg::NMMA; ++c) {
                            const uint64_t bdesc =
                                sw128_kmajor_desc(sb_ + c * Cfg::NCH * 128 + kk * 32);
                            umma_bf16(d_tmem + c * Cfg::NCH, adesc, bdesc, Cfg::IDESC,
                                      (kb | kk) != 0);
                        }
                    }
                    umma_commit(&empty_bar[stage]);   // frees the stage when these MMAs finish
                    if (++stage == Cfg::STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
                if (failed) break;
                umma_commit(&tfull_bar[acc]);          // accumulator ready for the epilogue
                if (Cfg::NACC == 2) {
                    acc ^= 1;
                    if (acc == 0) acc_phase ^= 1;
                } else {
                    acc_phase ^= 1;
                }
            }
            // All issued MMAs must be complete before TMEM is released.
            umma_commit(drain_bar);
            if (!mbar_wait(drain_bar, 0)) latch_error(a.err, CRC_ETIMEOUT);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        uint8_t* my_stage = staging + (warp - 2) * 2 * 4096;
        int buf = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int tile = blockIdx.x; tile < a.num_tiles; tile += gridDim.x) {
            if (!mbar_wait(&tfull_bar[acc], acc_phase)) {
                latch_error(a.err, CRC_ETIMEOUT);
                break;
            }
            tc_fence_after();
            const int l = tile / tiles_per_layer;
            const int r = tile % tiles_per_layer;
            const int sb = r / a.n_tb, tb = r % a.n_tb;
            const uint32_t tbase =
                tmem_base + (uint32_t)(acc * Cfg::ACC_COLS) + ((uint32_t)(quarter * 32) << 16);
#pragma unroll 1
            for (int h = 0; h < H; ++h) {
                float z[NH];
                if constexpr (NH >= 32) {
#pragma unroll
                    for (int c = 0; c < NH / 32; ++c)
                        tmem_ld32(tbase + (uint32_t)(h * NH + c * 32), z + 32 * c);
                } else {
                    tmem_ld16f(tbase + (uint32_t)(h * NH), z);
                }
                tmem_ld_wait();
#pragma unroll
                for (int c = 0; c < NH / 16; ++c) pin16(z + 16 * c);
                if (h == H - 1) {             // accumulator fully read: hand it back early
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&tempty_bar[acc]);
                }
                head_softmax<NH>(z);
                if constexpr (Cfg::TMA_STORE) {
                    // this warp's 32 rows: streams str0.., tokens tok0.. of the scores box
                    const int row0 = quarter * 32;
                    const int str0 = sb * a.SB + row0 / a.TB;
                    const int tok0 = tb * a.TB + row0 % a.TB;
#pragma unroll
                    for (int c = 0; c < NH / 32; ++c) {
                        uint8_t* sbuf = my_stage + buf * 4096;
                        buf ^= 1;
                        if (lane == 0) bulk_wait_read<1>();   // the store that used sbuf is done
                        __syncwarp();
                        float4* dst = reinterpret_cast<float4*>(sbuf + lane * 128);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            dst[j ^ (lane & 7)] = make_float4(z[32 * c + 4 * j], z[32 * c + 4 * j + 1],
                                                              z[32 * c + 4 * j + 2],
                                                              z[32 * c + 4 * j + 3]);
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_5d(&tmap_s, sbuf, c * 32, h, l, tok0, str0);
                            bulk_commit();
                        }
                    }
                } else {
                    const int b = sb * a.SB + row / a.TB;
                    const int t = tb * a.TB + row % a.TB;
                    if (b < a.B && t < a.T_ext) {
                        float4* o = reinterpret_cast<float4*>(
                            a.scores + (((size_t)b * a.T_ext + t) * a.L + l) * (size_t)(3 * NH) +
                            h * NH);
#pragma unroll
                        for (int i = 0; i < NH / 4; ++i)
                            o[i] = make_float4(z[4 * i], z[4 * i + 1], z[4 * i + 2], z[4 * i + 3]);
                    }
                }
            }
            if (Cfg::NACC == 2) {
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1;
            } else {
                acc_phase ^= 1;
            }
        }
        if (Cfg::TMA_STORE && lane == 0) bulk_wait<0>();   // every store has landed
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
    }
}

}  // namespace crc
