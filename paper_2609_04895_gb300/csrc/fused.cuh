// Fused route-and-cache: the router heads on the tensor cores and the cache
// scan run in ONE persistent kernel: the router probabilities are never
// written out as scores; each tile's record (Top-K set, s^T, p^S: 1.04 KB per
// decision for N = 128) passes through a ring of three token blocks of tiles
// in the workspace, read once by the scan warps (from L2 when the scan keeps
// up, else written back to DRAM and read from there).
//
// Per CTA (one per SM, cooperative launch so that all CTAs are resident), 12 warps
// (14 when R > 4):
//   warp 0      TMA producer  (hidden tile + [3N x 64] weight slab per stage)
//   warp 1      TMEM owner, tcgen05.mma issuer
//   warps 2..5  epilogue: per tile row (thread = row) the three softmaxes,
//               s^T = p^R + p^T, the Top-K set of p^R (sorting networks on
//               the values, then an exact threshold-and-ties pass) and p^S; the
//               row's record (Top-K mask, s^T, p^S) goes to a ring slot with
//               coalesced stores, then the tile is published
//   warps 6..   scan warps: take items (chain, block of TB tokens) in token
//               order from a global counter, wait for the tiles they read and
//               for the chain's previous block, run Algorithm 2 / 1 on each
//               token (scan_apply), store the chain state and release the
//               tiles they read
// Tile k covers rows = SB streams x TB tokens of one layer, in the order
// (token block, layer, stream group).  Ring slot = k % RING; a slot is
// rewritten only after every reader of its previous tile is done (monotonic
// reader counters, uniform target 3*SB per tile: the epilogue adds phantom
// counts for readers a tile does not have).  RING holds three token blocks of
// tiles: an item of block tb reads tiles of blocks tb and tb-1 only, so the
// producer of block tb+3 waits only on items whose inputs already exist.
// Every wait is bounded; on expiry the kernel latches CRC_ETIMEOUT, raises an
// abort flag that every other wait also watches, and unwinds.
#pragma once

#include "cache_scan.cuh"
#include "router_gemm.cuh"

namespace crc {

struct FusedArgs {
    uint8_t* state;
    int B, L, N, K, C, R, T;
    int SB, TB, n_bg, n_tb;
    int tiles_per_tb, num_tiles, ring, kblocks;
    int n_items;
    uint32_t* ctl;          // [0] next item, [1] abort flag
    uint32_t* tile_done;    // [ring] epilogue warps that published the slot (4 per tile)
    uint32_t* readers;      // [ring] finished readers (+ phantom counts), 3*SB per tile
    uint32_t* prog;         // [B*L] token blocks finished per chain
    uint8_t* ring_base;
    size_t slot_bytes;
    // optional per-access trace of the call ([B][T][L] bytes, [B][T][L][NW]
    // bitmasks), each null when not wanted
    uint8_t* tr_miss;
    uint8_t* tr_pro;
    uint32_t* tr_mid;
    uint32_t* tr_after;
    uint32_t* tr_sel;
};

// Ring slot layout for tile rows r in [0,128): Top-K mask words [NW][128] u32,
// then s^T and p^S as [N/4][128] float4 (chunk-major: a warp's store of one
// chunk for its 32 rows is 512 contiguous bytes).
template <int NH>
struct RingLayout {
    static constexpr int NW = (NH + 31) / 32;
    static constexpr size_t SEL = 0;
    static constexpr size_t ST = (size_t)NW * 128 * 4;
    static constexpr size_t PS = ST + (size_t)NH * 128 * 4;
    static constexpr size_t bytes(bool has_s) { return has_s ? PS + (size_t)NH * 128 * 4 : PS; }
};

__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Single-thread bounded wait for *p >= target.  False on timeout or abort.
__device__ __forceinline__ bool wait_geq(const uint32_t* p, uint32_t target, uint32_t* abort_flag,
                                         uint32_t* err, uint64_t limit_ns = kWaitLimitNs) {
    if (ld_acquire_u32(p) >= target) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
#pragma unroll 1
        for (int i = 0; i < 32; ++i) {
            __nanosleep(64);
            if (ld_acquire_u32(p) >= target) return true;
        }
        if (ld_acquire_u32(abort_flag)) return false;
        if (globaltimer_ns() - t0 > limit_ns) {
            latch_error(err, CRC_ETIMEOUT);
            atomicExch(abort_flag, 1u);
            return false;
        }
    }
}

// Loads of data another CTA may have written during this kernel go to L2
// (ld.global.cg): the per-SM L1 is not coherent.
template <int V>
__device__ __forceinline__ Vec<V> ldcg_vec(const float* p, bool ok) {
    Vec<V> r;
    if (!ok) {
#pragma unroll
        for (int i = 0; i < V; ++i) r.v[i] = 0.f;
        return r;
    }
    if constexpr (V == 4) {
        const float4 x = __ldcg(reinterpret_cast<const float4*>(p));
        r.v[0] = x.x; r.v[1] = x.y; r.v[2] = x.z; r.v[3] = x.w;
    } else if constexpr (V == 2) {
        const float2 x = __ldcg(reinterpret_cast<const float2*>(p));
        r.v[0] = x.x; r.v[1] = x.y;
    } else if constexpr (V == 8) {
        const float4 x = __ldcg(reinterpret_cast<const float4*>(p));
        const float4 y = __ldcg(reinterpret_cast<const float4*>(p) + 1);
        r.v[0] = x.x; r.v[1] = x.y; r.v[2] = x.z; r.v[3] = x.w;
        r.v[4] = y.x; r.v[5] = y.y; r.v[6] = y.z; r.v[7] = y.w;
    } else {
        r.v[0] = __ldcg(p);
    }
    return r;
}

template <int V>
__device__ __forceinline__ uint32_t lane_bits_cg(const uint32_t* words, int lane, int N) {
    const int e0 = lane * V;
    if (e0 >= N) return 0u;
    return (__ldcg(words + (e0 >> 5)) >> (e0 & 31)) & ((1u << V) - 1u);
}

template <int CW>
__device__ __forceinline__ void tmem_cols(uint32_t taddr, float* z) {
    if constexpr (CW == 32) {
        tmem_ld32(taddr, z);
    } else {
        tmem_ld16f(taddr, z);
    }
}
template <int CW>
__device__ __forceinline__ void tmem_put(uint32_t taddr, const float* z) {
    if constexpr (CW == 32) {
        tmem_st32(taddr, z);
    } else {
        tmem_st16(taddr, z);
    }
}
template <int CW>
__device__ __forceinline__ void pin_cols(float* z) {
#pragma unroll
    for (int c = 0; c < CW / 16; ++c) pin16(z + 16 * c);
}

// V experts of lane `lane` from a chunk-major [N/4][128] float4 array, row r.
template <int V>
__device__ __forceinline__ void ring_vec(const uint8_t* base, int lane, int r, float (&out)[V]) {
    if constexpr (V == 4) {
        const float4 f = __ldcg(reinterpret_cast<const float4*>(base) + (size_t)lane * 128 + r);
        out[0] = f.x; out[1] = f.y; out[2] = f.z; out[3] = f.w;
    } else if constexpr (V == 8) {
        const float4 f = __ldcg(reinterpret_cast<const float4*>(base) + (size_t)(2 * lane) * 128 + r);
        const float4 g =
            __ldcg(reinterpret_cast<const float4*>(base) + (size_t)(2 * lane + 1) * 128 + r);
        out[0] = f.x; out[1] = f.y; out[2] = f.z; out[3] = f.w;
        out[4] = g.x; out[5] = g.y; out[6] = g.z; out[7] = g.w;
    } else if constexpr (V == 2) {
        const float2 f = __ldcg(reinterpret_cast<const float2*>(
            base + ((size_t)(lane >> 1) * 128 + r) * 16 + (lane & 1) * 8));
        out[0] = f.x; out[1] = f.y;
    } else {
        out[0] = __ldcg(reinterpret_cast<const float*>(
            base + ((size_t)(lane >> 2) * 128 + r) * 16 + (lane & 3) * 4));
    }
}

// The scan role of the fused kernels (one warp per item): items (chain,
// block of TB tokens) come from a global counter in token order; each waits
// (bounded) for the chain's previous block and for the tiles it reads (a tile
// is complete when `publishers` epilogue warps have published it), runs
// Algorithm 2 / 1 on each token (scan_apply) and releases the tiles through
// the monotonic reader counters.
template <int NH, int V, bool ALL_VALID, bool TRACED>
__device__ __forceinline__ void fused_scan_role(const FusedArgs& a, uint32_t* err,
                                                uint32_t* abort_flag, int64_t t0g,
                                                uint32_t parity, int lane, uint32_t publishers) {
    using RL = RingLayout<NH>;
    StateLayout lay = state_layout(a.B, a.L, a.N);
    ChainState* chains = reinterpret_cast<ChainState*>(a.state + lay.chains);
    float* retention = reinterpret_cast<float*>(a.state + lay.retention);
    float* carry = reinterpret_cast<float*>(a.state + lay.carry);
    const int N = a.N, L = a.L;
    uint32_t valid = 0u;
#pragma unroll
    for (int v = 0; v < V; ++v)
        if (lane * V + v < N) valid |= 1u << v;
    const bool has = valid != 0u;
    const bool want_s = a.R > 0;
    const uint32_t e0 = (uint32_t)lane * V;
    const int NW = (N + 31) >> 5;
    const bool traced = TRACED && (a.tr_miss || a.tr_pro || a.tr_mid || a.tr_after || a.tr_sel);
    while (true) {
        uint32_t item = 0u;
        if (lane == 0) item = atomicAdd(&a.ctl[0], 1u);
        item = __shfl_sync(kFull, item, 0);
        if (item >= (uint32_t)a.n_items) break;
        const int tb = (int)(item / (uint32_t)(L * a.B));
        const int rem = (int)(item % (uint32_t)(L * a.B));
        const int l = rem / a.B, b = rem % a.B;
        const int bg = b / a.SB, sbi = b % a.SB;
        const int chain = b * L + l;
        const int k_own = (tb * L + l) * a.n_bg + bg;
        const int k_ps = (tb * L + (l > 0 ? l - 1 : L - 1)) * a.n_bg + bg;
        const int k_prev = (l == 0 && tb > 0) ? ((tb - 1) * L + L - 1) * a.n_bg + bg : -1;
        const bool read_ps = want_s && (l > 0 || a.TB >= 2);
        // debug builds: the item's stream, layer, block, tiles and rows exist
        if (!CRC_IN_BOUNDS(b < a.B && l < L && tb < a.n_tb && k_own < a.num_tiles &&
                               k_ps < a.num_tiles && k_prev < a.num_tiles &&
                               sbi * a.TB + a.TB <= 128 && parity < 2u,
                           err))
            break;
        // wait for the chain's previous block and the tiles this item reads
        bool ok = true;
        if (lane == 0) {
            ok = wait_geq(&a.prog[chain], (uint32_t)tb, abort_flag, err);
            auto ready = [&](int k) {
                return wait_geq(&a.tile_done[k % a.ring], publishers * (uint32_t)(k / a.ring + 1),
                                abort_flag, err);
            };
            ok = ok && ready(k_own);
            if (read_ps) ok = ok && ready(k_ps);
            if (want_s && k_prev >= 0) ok = ok && ready(k_prev);
        }
        ok = __shfl_sync(kFull, ok, 0);
        if (!ok) break;

        ChainState& cs = chains[chain];
        ChainRegs<V> cr;
        cr.cache = lane_bits_cg<V>(cs.bits, lane, N);
        cr.count = (int)__reduce_add_sync(kFull, (uint32_t)__popc(cr.cache));
        {
            Vec<V> x = ldcg_vec<V>(retention + (size_t)chain * N + e0, has);
#pragma unroll
            for (int v = 0; v < V; ++v) cr.aT[v] = x.v[v];
        }
        cr.hits = cr.misses = cr.pro = 0u;
        const uint8_t* own = a.ring_base + (size_t)(k_own % a.ring) * a.slot_bytes;
        const uint8_t* psl = a.ring_base + (size_t)(k_ps % a.ring) * a.slot_bytes;
        const uint8_t* prv =
            k_prev >= 0 ? a.ring_base + (size_t)(k_prev % a.ring) * a.slot_bytes : nullptr;
        const float* carry_in = carry + ((size_t)parity * a.B + b) * N + e0;
        const int steps = imin(a.TB, a.T - tb * a.TB);
        const int last_row = sbi * a.TB + steps - 1;
        // inputs of step tbi: s^T, the Top-K bits and p^S of the predecessor
        // the first step of this block with a causal predecessor (refinement)
        const int refine_from =
            (int)(t0g + (int64_t)tb * a.TB >= 1 ? 0 : 1 - (t0g + (int64_t)tb * a.TB));
        // the Top-K word is fetched whole and its bits taken at use, so the
        // load stays in flight across the step instead of stalling the fetch
        auto fetch = [&](int tbi, float (&sT)[V], float (&pS)[V], uint32_t& selw) {
            const int r = sbi * a.TB + tbi;
#pragma unroll
            for (int v = 0; v < V; ++v) sT[v] = pS[v] = 0.f;
            selw = 0u;
            if (!has) return;
            ring_vec<V>(own + RL::ST, lane, r, sT);
            selw = __ldcg(reinterpret_cast<const uint32_t*>(own + RL::SEL) +
                          (size_t)(e0 >> 5) * 128 + r);
            if (want_s && tbi >= refine_from) {
                if (l > 0) {
                    ring_vec<V>(psl + RL::PS, lane, r, pS);
                } else if (tbi > 0) {
                    ring_vec<V>(psl + RL::PS, lane, r - 1, pS);
                } else if (prv) {
                    ring_vec<V>(prv + RL::PS, lane, sbi * a.TB + a.TB - 1, pS);
                } else {
                    Vec<V> x = ldcg_vec<V>(carry_in, true);
#pragma unroll
                    for (int v = 0; v < V; ++v) pS[v] = x.v[v];
                }
            }
        };
        // Pull the next 128-byte lines of this lane's chunks into L2 ahead of
        // use (rows r .. r+7 of a chunk share one line; sel words 32 rows).
        auto prefetch_rows = [&](int tbi) {
            if (!has || tbi >= steps) return;
            const int r = sbi * a.TB + tbi;
            const int ch = (int)(e0 >> 2);
            asm volatile("prefetch.global.L2 [%0];" ::"l"(own + RL::ST +
                                                           ((size_t)ch * 128 + r) * 16));
            if (want_s)
                asm volatile("prefetch.global.L2 [%0];" ::"l"(psl + RL::PS +
                                                               ((size_t)ch * 128 + r) * 16));
            if ((tbi & 31) == 0)
                asm volatile("prefetch.global.L2 [%0];" ::"l"(
                    own + RL::SEL + ((size_t)(e0 >> 5) * 128 + r) * 4));
        };
        prefetch_rows(8);
        prefetch_rows(16);
        float cT[V], cS[V];
        uint32_t csel;
        fetch(0, cT, cS, csel);
        for (int tbi = 0; tbi < steps; ++tbi) {
            float nT[V], nS[V];
            uint32_t nsel = 0u;
            if (tbi + 1 < steps) fetch(tbi + 1, nT, nS, nsel);
            if ((tbi & 7) == 0) prefetch_rows(tbi + 24);
            const bool refine = want_s && tbi >= refine_from;
            const uint32_t sel = (csel >> (e0 & 31)) & ((1u << V) - 1u);
            int nD;
            if (traced && CRC_IN_BOUNDS(tb * a.TB + tbi < a.T, err)) {
                // the refinement on its own, so the cache between the phases is seen
                const size_t unit = ((size_t)b * a.T + tb * a.TB + tbi) * L + l;
                const int pro = refine ? scan_refine<V, ALL_VALID>(cr, cS, valid, lane, a.C, a.R)
                                       : 0;
                if (a.tr_mid) store_cache_words<V>(cr.cache, lane, N, a.tr_mid + unit * NW);
                scan_apply<V, ALL_VALID>(cr, cT, cS, false, valid, lane, a.K, a.C, a.R, sel,
                                         &nD);
                cr.pro += (uint32_t)pro;
                if (a.tr_after) store_cache_words<V>(cr.cache, lane, N, a.tr_after + unit * NW);
                if (a.tr_sel && has && (e0 & 31u) == 0u) a.tr_sel[unit * NW + (e0 >> 5)] = csel;
                if (lane == 0) {
                    if (a.tr_miss) a.tr_miss[unit] = (uint8_t)nD;
                    if (a.tr_pro) a.tr_pro[unit] = (uint8_t)pro;
                }
            } else {
                scan_apply<V, ALL_VALID>(cr, cT, cS, refine, valid, lane, a.K, a.C, a.R, sel,
                                         &nD);
            }
            // debug builds: every expert the step made resident lies in this
            // lane's range and the cache holds at most C experts
            (void)CRC_IN_BOUNDS((cr.cache & ~valid) == 0u && cr.count <= a.C, err);
#pragma unroll
            for (int v = 0; v < V; ++v) {
                cT[v] = nT[v];
                cS[v] = nS[v];
            }
            csel = nsel;
        }
        // the last layer hands p^S of the call's last token to layer 0 of the next call
        if (l == L - 1 && want_s && tb * a.TB + a.TB >= a.T && steps > 0 && has) {
            float pl[V];
            ring_vec<V>(own + RL::PS, lane, last_row, pl);   // has: lane owns experts
            float* dst = carry + ((size_t)(parity ^ 1u) * a.B + b) * N + e0;
#pragma unroll
            for (int v = 0; v < V; ++v)
                if (lane * V + v < N) dst[v] = pl[v];
        }
        // store the chain
        for (int w = 0; w < NW; ++w) {
            const uint32_t contrib = (has && (e0 >> 5) == (uint32_t)w) ? (cr.cache << (e0 & 31)) : 0u;
            const uint32_t wd = __reduce_or_sync(kFull, contrib);
            if (lane == 0) cs.bits[w] = wd;
        }
        if (has) {
#pragma unroll
            for (int v = 0; v < V; ++v)
                if (lane * V + v < N) retention[(size_t)chain * N + e0 + v] = cr.aT[v];
        }
        if (lane == 0) {
            cs.hits = __ldcg(&cs.hits) + cr.hits;
            cs.misses = __ldcg(&cs.misses) + cr.misses;
            cs.proactive = __ldcg(&cs.proactive) + cr.pro;
        }
        // release the tiles and the chain
        __threadfence();
        __syncwarp();
        if (lane == 0) {
            atomicAdd(&a.readers[k_own % a.ring], 1u);
            if (want_s) {
                if (l > 0 || a.TB >= 2) atomicAdd(&a.readers[k_ps % a.ring], 1u);
                if (k_prev >= 0) atomicAdd(&a.readers[k_prev % a.ring], 1u);
            }
            atomicExch(&a.prog[chain], (uint32_t)(tb + 1));
        }
    }
}

// PAIR: the GEMM runs on CTA pairs (tcgen05.mma.cta_group::2, M = 256): each
// CTA of a pair loads its own 128-row hidden tile and half of the weight rows
// of every MMA (96 of 192), so a stage carries 37.5 % fewer bytes per flop;
// the even CTA issues the MMAs into both CTAs' TMEM.
template <int NH, int H, bool PAIR = false>
struct FusedCfg {
    using RC = RouterCfg<NH, H>;
    static constexpr int GEMM_WARPS = 6;
    // Scan warps per CTA, chosen at launch from the refinement budget.  Six
    // keep up with the GEMM when R <= 4; more of them only take issue slots
    // from the epilogue (Qwen3-30B shape: 6 -> 4.20 ms, 7 -> 4.24, 8 -> 4.29,
    // 10 -> 4.35; 5 and 4 fall behind the tiles, 4.36 and 4.96).  With R = 8
    // a step has up to twice the refinement rounds and six fall behind (one
    // 128-token chunk of the Qwen3-235B shape: 15.9 ms with 6, 15.25 with 8,
    // 15.17 with 10; with R = 2: 14.7-15.0 with 6 or 8).  The kernel's roles
    // do not depend on the count: every warp past the GEMM warps scans.
    static constexpr int SCAN_WARPS = 6;
    static constexpr int SCAN_WARPS_WIDE = 8;
    static constexpr int THREADS = 32 * (GEMM_WARPS + SCAN_WARPS);
    static constexpr int MAX_THREADS = 32 * (GEMM_WARPS + SCAN_WARPS_WIDE);
    static int threads_for(int R) {
        return 32 * (GEMM_WARPS + (R > 4 ? SCAN_WARPS_WIDE : SCAN_WARPS));
    }
    static constexpr int B_ROWS = PAIR ? RC::NCOL / 2 : RC::NCOL;        // weight rows per CTA
    static constexpr int B_BOX_ROWS = PAIR ? RC::NCH / 2 : RC::B_BOX_ROWS;
    static constexpr int B_BOXES = B_ROWS / B_BOX_ROWS;
    static constexpr int STAGE_BYTES = RC::A_BYTES + B_ROWS * RC::BK * 2;
    static constexpr uint32_t IDESC = PAIR ? idesc_bf16_f32(2 * RC::BM, RC::NCH) : RC::IDESC;
    // PAIR: the Temporal head's exps are parked in shared memory (fp32,
    // [NH/4][128 rows] float4) and p^R's in the spare TMEM columns, so the
    // accumulator goes back to the MMA after two passes over those heads
    static constexpr bool PARK_T = PAIR && RC::NACC == 1;
    static constexpr int PARK_T_BYTES = PARK_T ? RC::BM * NH * 4 : 0;
    static constexpr int STAGES = imin(8, (232448 - 1024 - 256 - PARK_T_BYTES) / STAGE_BYTES);
    static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + PARK_T_BYTES + 256;
    static constexpr int CW = NH < 32 ? NH : 32;     // TMEM columns per load
    static constexpr int NCHK = NH / CW;
    static_assert(STAGES >= 2, "pipeline depth");
    static_assert(!PAIR || B_BOXES == RC::NMMA, "CTA pairs: one weight box per MMA half");
    static_assert((STAGE_BYTES % 1024) == 0 && ((B_BOX_ROWS * 128) % 1024) == 0,
                  "swizzle atom alignment");
};

// TRACED: compiled with the scan role's trace writes (any trace array given).
template <int NH, int H, int V, bool ALL_VALID, int KP, bool PAIR = false, bool TRACED = false>
__global__ void __launch_bounds__(512, 1)
    fused_route_cache_kernel(const __grid_constant__ CUtensorMap tmap_h,
                             const __grid_constant__ CUtensorMap tmap_w, FusedArgs a) {
    using Cfg = FusedCfg<NH, H, PAIR>;
    using RC = typename Cfg::RC;
    using RL = RingLayout<NH>;
    constexpr int CW = Cfg::CW;
    constexpr int NCHK = Cfg::NCHK;
    // exps of chunk c in place, into the accumulator of the head half it covers
    auto chunk_exp = [](int c, float* v, HeadExp& e0, HeadExp& e1) {
        if constexpr (NCHK >= 2) {
            if (c < NCHK / 2)
                e0.exp_in_place<CW>(v);
            else
                e1.exp_in_place<CW>(v);
        } else {                                        // one chunk holds both halves
            e0.exp_in_place<CW / 2>(v);
            e1.exp_in_place<CW / 2>(v + CW / 2);
        }
    };

    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* tiles = smem;
    float4* tpark = reinterpret_cast<float4*>(smem + Cfg::STAGES * Cfg::STAGE_BYTES);
    uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem + Cfg::STAGES * Cfg::STAGE_BYTES +
                                                     Cfg::PARK_T_BYTES);
    uint64_t* empty_bar = full_bar + Cfg::STAGES;
    uint64_t* tfull_bar = empty_bar + Cfg::STAGES;
    uint64_t* tempty_bar = tfull_bar + RC::NACC;
    uint64_t* drain_bar = tempty_bar + RC::NACC;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    // PAIR: rank 0 issues the MMAs for both CTAs; the tile loops below step by
    // gridDim.x from blockIdx.x, so the two CTAs of a pair hold the adjacent
    // tiles 2j and 2j + 1 (same token block and layer: the launch makes the
    // stream count even) at every iteration.
    const uint32_t rank = PAIR ? cluster_ctarank() : 0u;
    const bool leader = rank == 0u;

    StateHeader* hdr = reinterpret_cast<StateHeader*>(a.state);
    uint32_t* err = &hdr->error;
    uint32_t* abort_flag = a.ctl + 1;
    const bool hdr_ok = hdr->magic == kStateMagic && hdr->L == a.L && hdr->N == a.N &&
                        hdr->K == a.K && hdr->C == a.C && hdr->R == a.R && hdr->B == a.B &&
                        hdr->policy == 0u;
    const int64_t t0g = hdr->t_next;
    const uint32_t parity = hdr->parity;

    if (threadIdx.x == 0) {
        for (int s = 0; s < Cfg::STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int s = 0; s < RC::NACC; ++s) {
            mbar_init(&tfull_bar[s], 1);
            mbar_init(&tempty_bar[s], PAIR ? 8 : 4);       // both CTAs' epilogue warps
        }
        mbar_init(drain_bar, 1);
        fence_mbar_init();
        tma_prefetch_desc(&tmap_h);
        tma_prefetch_desc(&tmap_w);
    }
    if (warp == 1) {
        if constexpr (PAIR) {
            tmem_alloc_pair(tmem_slot, RC::TMEM_COLS);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(tmem_slot, RC::TMEM_COLS);
            tmem_relinquish();
        }
    }
    tc_fence_before();
    __syncthreads();
    if constexpr (PAIR) cluster_sync();             // the peer's barriers exist before any remote use
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const int num_tiles = hdr_ok ? a.num_tiles : 0;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA
        if (lane == 0) {
            const uint64_t pol_h = l2_evict_first_policy();
            const uint64_t pol_w = l2_evict_last_policy();
            int stage = 0, issued = 0, failed = 0;
            uint32_t phase = 0;
            // PAIR: both CTAs' loads of a stage complete on the even CTA's full
            // barrier, which expects the bytes of both
            const uint32_t lead_full = PAIR ? cluster_map(&full_bar[0], 0u) : 0u;
            for (int k = blockIdx.x; k < num_tiles && !failed; k += gridDim.x) {
                const int tb = k / a.tiles_per_tb;
                const int rem = k % a.tiles_per_tb;
                const int l = rem / a.n_bg, bg = rem % a.n_bg;
                for (int kb = 0; kb < a.kblocks; ++kb) {
                    const bool freed = PAIR ? mbar_wait_cluster(&empty_bar[stage], phase ^ 1)
                                            : mbar_wait(&empty_bar[stage], phase ^ 1);
                    if (!freed || ld_acquire_u32(abort_flag)) {
                        if (!ld_acquire_u32(abort_flag)) {
                            latch_error(err, CRC_ETIMEOUT);
                            atomicExch(abort_flag, 1u);
                        }
                        failed = 1;
                        break;
                    }
                    uint8_t* sa = tiles + stage * Cfg::STAGE_BYTES;
                    uint8_t* sw = sa + RC::A_BYTES;
                    if constexpr (PAIR) {
                        if (leader) mbar_arrive_expect_tx(&full_bar[stage], 2 * Cfg::STAGE_BYTES);
                        const uint32_t fb = lead_full + (uint32_t)(stage * 8);
                        tma_load_4d_pair(sa, &tmap_h, fb, kb * RC::BK, l, tb * a.TB, bg * a.SB,
                                         pol_h);
                        // rows [c*NCH + rank*NCH/2, +NCH/2) of MMA c's weight block
#pragma unroll
                        for (int c = 0; c < Cfg::B_BOXES; ++c)
                            tma_load_3d_pair(sw + c * Cfg::B_BOX_ROWS * 128, &tmap_w, fb,
                                             kb * RC::BK, c * RC::NCH + (int)rank * Cfg::B_BOX_ROWS,
                                             l, pol_w);
                    } else {
                        mbar_arrive_expect_tx(&full_bar[stage], Cfg::STAGE_BYTES);
                        tma_load_4d(sa, &tmap_h, &full_bar[stage], kb * RC::BK, l, tb * a.TB,
                                    bg * a.SB, pol_h);
#pragma unroll
                        for (int c = 0; c < Cfg::B_BOXES; ++c)
                            tma_load_3d(sw + c * Cfg::B_BOX_ROWS * 128, &tmap_w, &full_bar[stage],
                                        kb * RC::BK, c * Cfg::B_BOX_ROWS, l, pol_w);
                    }
                    ++issued;
                    if (++stage == Cfg::STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
            }
            int s = stage;
            uint32_t ph = phase;
            // (PAIR: only the even CTA's barriers see the loads; the odd CTA
            // stays until its loads landed through the final cluster barrier)
            for (int k = 0; k < ((PAIR && !leader) ? 0 : imin(issued, Cfg::STAGES)); ++k) {
                if (--s < 0) {
                    s = Cfg::STAGES - 1;
                    ph ^= 1;
                }
                if (!mbar_wait(&full_bar[s], ph)) latch_error(err, CRC_ETIMEOUT);
            }
        }
    } else if (warp == 1 && PAIR && !leader) {
        // the odd CTA's MMA warp only takes part in the TMEM allocation
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA
        if (lane == 0) {
            int stage = 0, acc = 0, failed = 0;
            uint32_t phase = 0, acc_phase = 0;
            for (int k = blockIdx.x; k < num_tiles && !failed; k += gridDim.x) {
                const bool acc_free = PAIR ? mbar_wait_cluster(&tempty_bar[acc], acc_phase ^ 1)
                                           : mbar_wait(&tempty_bar[acc], acc_phase ^ 1);
                if (!acc_free) {
                    latch_error(err, CRC_ETIMEOUT);
                    atomicExch(abort_flag, 1u);
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * RC::ACC_COLS);
                for (int kb = 0; kb < a.kblocks; ++kb) {
                    const bool landed = PAIR ? mbar_wait_cluster(&full_bar[stage], phase)
                                             : mbar_wait(&full_bar[stage], phase);
                    if (!landed) {
                        latch_error(err, CRC_ETIMEOUT);
                        atomicExch(abort_flag, 1u);
                        failed = 1;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(tiles + stage * Cfg::STAGE_BYTES);
                    const uint32_t sw = sa + RC::A_BYTES;
#pragma unroll
                    for (int kk = 0; kk < RC::BK / 16; ++kk) {
                        const uint64_t adesc = sw128_kmajor_desc(sa + kk * 32);
#pragma unroll
                        for (int c = 0; c < RC::NMMA; ++c) {
                            const uint64_t bdesc =
                                sw128_kmajor_desc(sw + c * Cfg::B_BOX_ROWS * 128 + kk * 32);
                            if constexpr (PAIR)
                                umma_bf16_pair(d_tmem + c * RC::NCH, adesc, bdesc, Cfg::IDESC,
                                               (kb | kk) != 0);
                            else
                                umma_bf16(d_tmem + c * RC::NCH, adesc, bdesc, Cfg::IDESC,
                                          (kb | kk) != 0);
                        }
                    }
                    if constexpr (PAIR)
                        umma_commit_pair(&empty_bar[stage]);
                    else
                        umma_commit(&empty_bar[stage]);
                    if (++stage == Cfg::STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
                if (failed) break;
                if constexpr (PAIR)
                    umma_commit_pair(&tfull_bar[acc]);
                else
                    umma_commit(&tfull_bar[acc]);
                if (RC::NACC == 2) {
                    acc ^= 1;
                    if (acc == 0) acc_phase ^= 1;
                } else {
                    acc_phase ^= 1;
                }
            }
            if constexpr (PAIR)
                umma_commit_pair_local(drain_bar);
            else
                umma_commit(drain_bar);
            if (!mbar_wait(drain_bar, 0)) latch_error(err, CRC_ETIMEOUT);
        }
    } else if (warp < Cfg::GEMM_WARPS) {
        // ------------------------------------------------------------ epilogue
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const uint32_t target_per_tile = 3u * (uint32_t)a.SB;
        int acc = 0;
        uint32_t acc_phase = 0;
        // PAIR: the accumulator is released to the even CTA's MMA issuer
        const uint32_t tempty_peer = PAIR ? cluster_map(&tempty_bar[0], 0u) : 0u;
        auto release_acc = [&](int which) {
            if constexpr (PAIR) {
                if (!leader) {
                    mbar_arrive_remote(tempty_peer + (uint32_t)(which * 8));
                    return;
                }
            }
            mbar_arrive(&tempty_bar[which]);
        };
        for (int k = blockIdx.x; k < num_tiles; k += gridDim.x) {
            const bool filled = PAIR ? mbar_wait_cluster(&tfull_bar[acc], acc_phase)
                                     : mbar_wait(&tfull_bar[acc], acc_phase);
            if (!filled) {
                latch_error(err, CRC_ETIMEOUT);
                atomicExch(abort_flag, 1u);
                break;
            }
            tc_fence_after();
            const int tb = k / a.tiles_per_tb;
            const int rem = k % a.tiles_per_tb;
            const int l = rem / a.n_bg, bg = rem % a.n_bg;
            const int slot = k % a.ring;
            const uint32_t gen = (uint32_t)(k / a.ring);
            // the slot's previous tile must be fully read
            bool ok = CRC_IN_BOUNDS(slot < a.ring && l < a.L && bg < a.n_bg && tb < a.n_tb, err);
            if (lane == 0 && gen > 0 && ok)
                ok = wait_geq(&a.readers[slot], target_per_tile * gen, abort_flag, err);
            ok = __shfl_sync(kFull, ok, 0);
            uint8_t* slot_p = a.ring_base + (size_t)slot * a.slot_bytes;
            float4* sT_p = reinterpret_cast<float4*>(slot_p + RL::ST);
            float4* pS_p = reinterpret_cast<float4*>(slot_p + RL::PS);
            uint32_t* sel_p = reinterpret_cast<uint32_t*>(slot_p + RL::SEL);
            const uint32_t tbase =
                tmem_base + (uint32_t)(acc * RC::ACC_COLS) + ((uint32_t)(quarter * 32) << 16);
            float z[CW], y[CW];

            // Spatio head: p^S
            if constexpr (H == 3) {
                float m = -INFINITY;
#pragma unroll 1
                for (int c = 0; c < NCHK; ++c) {
                    tmem_cols<CW>(tbase + (uint32_t)(2 * NH + c * CW), z);
                    tmem_ld_wait();
                    pin_cols<CW>(z);
                    m = max_of<CW>(z, m);
                }
                // each exp(z - max) is computed once and parked in the
                // accumulator's own TMEM columns for the normalising pass
                HeadExp x0, x1;
                x0.init(m);
                x1.init(m);
#pragma unroll 1
                for (int c = 0; c < NCHK; ++c) {
                    tmem_cols<CW>(tbase + (uint32_t)(2 * NH + c * CW), z);
                    tmem_ld_wait();
                    pin_cols<CW>(z);
                    chunk_exp(c, z, x0, x1);
                    tmem_put<CW>(tbase + (uint32_t)(2 * NH + c * CW), z);
                }
                tmem_st_wait();
                const float r = head_inv(x0.part(), x1.part());
#pragma unroll 1
                for (int c = 0; c < NCHK; ++c) {
                    tmem_cols<CW>(tbase + (uint32_t)(2 * NH + c * CW), z);
                    tmem_ld_wait();
                    pin_cols<CW>(z);
                    scale_in_place<CW>(z, r);
                    if (ok) {
#pragma unroll
                        for (int q = 0; q < CW / 4; ++q)
                            pS_p[(size_t)(c * CW / 4 + q) * 128 + row] =
                                make_float4(z[4 * q], z[4 * q + 1], z[4 * q + 2], z[4 * q + 3]);
                    }
                }
            }

            // native and Temporal heads: s^T and the Top-K set of p^R
            // With a single accumulator, p^R is parked in the spare TMEM columns
            // [NCOL, NCOL + NH) so the accumulator can be handed back to the MMA
            // before the Top-K selection runs.  PARK_T: the max pass also parks
            // the raw logits (native in those columns, Temporal in shared
            // memory) and the accumulator goes back at once; the exps are
            // taken from the parked copies, the same values in the same order.
            constexpr bool PARK = RC::NACC == 1 && RC::NCOL + NH <= RC::ACC_COLS;
            const uint32_t pbase = tbase + (uint32_t)RC::NCOL;
            auto park_t = [&](int c) {
#pragma unroll
                for (int q = 0; q < CW / 4; ++q)
                    tpark[(c * CW / 4 + q) * 128 + row] =
                        make_float4(y[4 * q], y[4 * q + 1], y[4 * q + 2], y[4 * q + 3]);
            };
            auto unpark_t = [&](int c) {
#pragma unroll
                for (int q = 0; q < CW / 4; ++q) {
                    const float4 f = tpark[(c * CW / 4 + q) * 128 + row];
                    y[4 * q] = f.x;
                    y[4 * q + 1] = f.y;
                    y[4 * q + 2] = f.z;
                    y[4 * q + 3] = f.w;
                }
            };
            float mR = -INFINITY, mT = -INFINITY;
#pragma unroll 1
            for (int c = 0; c < NCHK; ++c) {
                tmem_cols<CW>(tbase + (uint32_t)(c * CW), z);
                tmem_cols<CW>(tbase + (uint32_t)(NH + c * CW), y);
                tmem_ld_wait();
                pin_cols<CW>(z);
                pin_cols<CW>(y);
                mR = max_of<CW>(z, mR);
                mT = max_of<CW>(y, mT);
                if constexpr (Cfg::PARK_T) {
                    tmem_put<CW>(pbase + (uint32_t)(c * CW), z);
                    park_t(c);
                }
            }
            if constexpr (Cfg::PARK_T) {
                tmem_st_wait();
                tc_fence_before();                        // accumulator columns fully read
                __syncwarp();
                if (lane == 0) release_acc(acc);
            }
            HeadExp r0, r1, t0, t1;
            r0.init(mR);
            r1.init(mR);
            t0.init(mT);
            t1.init(mT);
#pragma unroll 1
            for (int c = 0; c < NCHK; ++c) {
                if constexpr (Cfg::PARK_T) {
                    tmem_cols<CW>(pbase + (uint32_t)(c * CW), z);
                    unpark_t(c);
                    tmem_ld_wait();
                    pin_cols<CW>(z);
                } else {
                    tmem_cols<CW>(tbase + (uint32_t)(c * CW), z);
                    tmem_cols<CW>(tbase + (uint32_t)(NH + c * CW), y);
                    tmem_ld_wait();
                    pin_cols<CW>(z);
                    pin_cols<CW>(y);
                }
                chunk_exp(c, z, r0, r1);
                chunk_exp(c, y, t0, t1);
                if constexpr (Cfg::PARK_T) {
                    tmem_put<CW>(pbase + (uint32_t)(c * CW), z);
                    park_t(c);
                } else {
                    tmem_put<CW>(tbase + (uint32_t)(c * CW), z);
                    tmem_put<CW>(tbase + (uint32_t)(NH + c * CW), y);
                }
            }
            tmem_st_wait();
            const float rR = head_inv(r0.part(), r1.part()), rT = head_inv(t0.part(), t1.part());
            TopKAcc<KP> topk;
            topk.init();
            if constexpr (Cfg::PARK_T) {
#pragma unroll 1
                for (int c = 0; c < NCHK; ++c) {
                    tmem_cols<CW>(pbase + (uint32_t)(c * CW), z);
                    unpark_t(c);
                    tmem_ld_wait();
                    pin_cols<CW>(z);
                    retention_in_place<CW>(z, y, rR, rT);         // z = p^R, y = s^T
                    if (ok) {
#pragma unroll
                        for (int q = 0; q < CW / 4; ++q)
                            sT_p[(size_t)(c * CW / 4 + q) * 128 + row] =
                                make_float4(y[4 * q], y[4 * q + 1], y[4 * q + 2], y[4 * q + 3]);
                    }
                    tmem_put<CW>(pbase + (uint32_t)(c * CW), z);
#pragma unroll
                    for (int g = 0; g < CW; g += 16) topk.add16(z + g);
                }
                tmem_st_wait();
            }
#pragma unroll 1
            for (int c = 0; c < (Cfg::PARK_T ? 0 : NCHK); ++c) {
                tmem_cols<CW>(tbase + (uint32_t)(c * CW), z);
                tmem_cols<CW>(tbase + (uint32_t)(NH + c * CW), y);
                tmem_ld_wait();
                pin_cols<CW>(z);
                pin_cols<CW>(y);
                retention_in_place<CW>(z, y, rR, rT);             // z = p^R, y = s^T
                if (ok) {
#pragma unroll
                    for (int q = 0; q < CW / 4; ++q)
                        sT_p[(size_t)(c * CW / 4 + q) * 128 + row] =
                            make_float4(y[4 * q], y[4 * q + 1], y[4 * q + 2], y[4 * q + 3]);
                }
                if constexpr (PARK) {
                    tmem_put<CW>(pbase + (uint32_t)(c * CW), z);
                } else {
#pragma unroll
                    for (int g = 0; g < CW; g += 16) topk.add16(z + g);
                }
            }
            if constexpr (PARK && !Cfg::PARK_T) {
                tmem_st_wait();
                tc_fence_before();                        // accumulator columns fully read
                __syncwarp();
                if (lane == 0) release_acc(acc);
#pragma unroll 1
                for (int c = 0; c < NCHK; ++c) {
                    tmem_cols<CW>(pbase + (uint32_t)(c * CW), z);
                    tmem_ld_wait();
                    pin_cols<CW>(z);
#pragma unroll
                    for (int g = 0; g < CW; g += 16) topk.add16(z + g);
                }
            }
            const float th = topk.theta(a.K);
            int need = topk.need(a.K, th);
            uint32_t word = 0u;
#pragma unroll 1
            for (int c = 0; c < NCHK; ++c) {
                if constexpr (PARK) {
                    tmem_cols<CW>(pbase + (uint32_t)(c * CW), z);
                    tmem_ld_wait();
                    pin_cols<CW>(z);
                } else {
                    tmem_cols<CW>(tbase + (uint32_t)(c * CW), z);
                    tmem_ld_wait();
                    pin_cols<CW>(z);
                    if (c == NCHK - 1) {                  // accumulator fully read
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) release_acc(acc);
                    }
                    scale_in_place<CW>(z, rR);                    // p^R
                }
#pragma unroll
                for (int q = 0; q < CW / 4; ++q) {
                    const float4 f = make_float4(z[4 * q], z[4 * q + 1], z[4 * q + 2], z[4 * q + 3]);
                    word |= take4(f, th, need) << ((c * CW + 4 * q) & 31);
                }
                if (((c + 1) * CW) % 32 == 0 || c == NCHK - 1) {
                    if (ok) sel_p[(size_t)((c * CW) >> 5) * 128 + row] = word;
                    word = 0u;
                }
            }
            // publish this warp's 32 rows
            __threadfence();
            __syncwarp();
            if (lane == 0 && ok) {
                atomicAdd(&a.tile_done[slot], 1u);
                if (quarter == 0) {
                    // phantom readers: 3*SB per tile minus the readers this tile has
                    const int nsb = imin(a.SB, a.B - bg * a.SB);
                    int readers = nsb;
                    if (a.R > 0) {
                        if (l < a.L - 1) {
                            readers += nsb;
                        } else {
                            if (a.TB >= 2) readers += nsb;
                            if (tb + 1 < a.n_tb) readers += nsb;
                        }
                    }
                    atomicAdd(&a.readers[slot], target_per_tile - (uint32_t)readers);
                }
            }
            if (RC::NACC == 2) {
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1;
            } else {
                acc_phase ^= 1;
            }
            if (!ok) break;
        }
    } else if (hdr_ok) {
        fused_scan_role<NH, V, ALL_VALID, TRACED>(a, err, abort_flag, t0g, parity, lane, 4u);
    }
    tc_fence_before();
    __syncthreads();
    // PAIR: neither CTA leaves (or frees TMEM) while the other may still
    // arrive on its barriers or have MMAs write its TMEM
    if constexpr (PAIR) cluster_sync();
    if (warp == 1) {
        tc_fence_after();
        if constexpr (PAIR)
            tmem_dealloc_pair(tmem_base, RC::TMEM_COLS);
        else
            tmem_dealloc(tmem_base, RC::TMEM_COLS);
    }
    // the last CTA to finish advances the token counter and flips the carry slot
    if (threadIdx.x == 0) {
        if (!hdr_ok && blockIdx.x == 0) latch_error(err, CRC_ESTATE);
        __threadfence();
        const uint32_t prev = atomicAdd(&hdr->done, 1u);
        if (prev == gridDim.x - 1) {
            __threadfence();
            if (hdr_ok && !ld_acquire_u32(abort_flag)) {
                hdr->t_next = t0g + a.T;
                hdr->parity = parity ^ 1u;
            }
            hdr->done = 0u;
            __threadfence();
        }
    }
}

}  // namespace crc
