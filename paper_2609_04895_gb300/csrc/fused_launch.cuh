// Host side of the fused route-and-cache kernel: tile plan, workspace layout,
// tensor maps and the cooperative launch (all CTAs resident at once, which the
// kernel's producer / consumer waits rely on).
#pragma once

#include <algorithm>
#include <cstdlib>

#include "crc_internal.h"
#include "fused.cuh"

namespace crc {

inline bool plain_cluster_launch() {
    static const bool on = [] {
        const char* v = std::getenv("CRC_PLAIN_CLUSTER_LAUNCH");
        return v && v[0] == '1' && v[1] == '\0';
    }();
    return on;
}

struct FusedPlan {
    int SB, TB, n_bg, n_tb, tiles_per_tb, num_tiles, ring, n_items;
    size_t slot_bytes, ctl_bytes, total;
};

// Tile = SB streams x TB tokens of one layer, TB as long as the call allows
// (128 tokens of one stream when T >= 128).  Tiles go in the order (token
// block, layer, stream group), so a layer's weights are fetched once per
// token block; the ring holds three token blocks of records.  T = 0 gives the
// largest layout.
inline FusedPlan fused_plan(const crc_problem& p, int T) {
    FusedPlan f;
    int tb = 128;
    if (T > 0)
        while (tb > 1 && tb / 2 >= T) tb >>= 1;
    f.TB = tb;
    f.SB = 128 / tb;
    f.n_bg = (p.B + f.SB - 1) / f.SB;
    f.tiles_per_tb = p.L * f.n_bg;
    f.n_tb = (T + f.TB - 1) / f.TB;
    f.num_tiles = f.n_tb * f.tiles_per_tb;
    f.ring = 3 * f.tiles_per_tb;
    if (T > 0) f.ring = std::min(f.ring, f.num_tiles);
    f.n_items = f.n_tb * p.L * p.B;
    const int NW = (p.N + 31) / 32;
    f.slot_bytes = (size_t)128 * 4 * (NW + p.N * (p.R > 0 ? 2 : 1));
    const size_t ctl = 256 + (size_t)4 * 3 * f.tiles_per_tb * 2 + (size_t)4 * p.B * p.L;
    f.ctl_bytes = (ctl + 255) & ~(size_t)255;
    f.total = f.ctl_bytes + (size_t)3 * f.tiles_per_tb * f.slot_bytes;
    return f;
}

// PAIR launches clusters of two CTAs (the GEMM on CTA pairs), cooperatively so
// that every CTA is resident; a device that refuses that launch gets the
// single-CTA kernel from then on (CRC_EUNSUPPORTED).
template <int NH, int H, int V, bool ALL_VALID, int KP, bool PAIR, bool TRACED>
int launch_fused_t(const crc_problem& p, const uint16_t* hidden, const uint16_t* w_cat, int T,
                   void* state, void* workspace, const crc_trace* trace,
                      cudaStream_t stream) {
    using Cfg = FusedCfg<NH, H, PAIR>;
    using RC = typename Cfg::RC;
    const FusedPlan f = fused_plan(p, T);
    if (PAIR && (f.SB != 1 || f.n_bg % 2 != 0)) return CRC_EUNSUPPORTED;
    auto kern = fused_route_cache_kernel<NH, H, V, ALL_VALID, KP, PAIR, TRACED>;
    // -1: not set up yet in this process; 0: refused; else the grid
    static int grid = -1;
    if (grid == 0) return CRC_EUNSUPPORTED;
    if (grid < 0) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 Cfg::SMEM_BYTES) != cudaSuccess) {
            (void)cudaGetLastError();
            grid = 0;
            return CRC_EUNSUPPORTED;
        }
        if (PAIR) {
            cudaLaunchAttribute at[1];
            at[0].id = cudaLaunchAttributeClusterDimension;
            at[0].val.clusterDim.x = 2;
            at[0].val.clusterDim.y = 1;
            at[0].val.clusterDim.z = 1;
            cudaLaunchConfig_t c = {};
            c.gridDim = dim3((unsigned)(sm_count() / 2 * 2));
            c.blockDim = dim3(Cfg::MAX_THREADS);
            c.dynamicSmemBytes = Cfg::SMEM_BYTES;
            c.attrs = at;
            c.numAttrs = 1;
            int ncl = 0;
            if (cudaOccupancyMaxActiveClusters(&ncl, (const void*)kern, &c) != cudaSuccess ||
                ncl < 1) {
                (void)cudaGetLastError();
                grid = 0;
                return CRC_EUNSUPPORTED;
            }
            grid = std::min(2 * ncl, sm_count() / 2 * 2);
        } else {
            int per_sm = 0;
            if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, Cfg::MAX_THREADS,
                                                              Cfg::SMEM_BYTES) != cudaSuccess ||
                per_sm < 1) {
                (void)cudaGetLastError();
                grid = 0;
                return CRC_EUNSUPPORTED;
            }
            grid = sm_count();
        }
    }
    CUtensorMap mh, mw;
    if (!make_hidden_map(&mh, hidden, p.B, T, p.L, p.d, f.TB, f.SB)) return CRC_ECUDA;
    if (!make_weight_map(&mw, w_cat, p.L, 3 * NH, p.d, Cfg::B_BOX_ROWS)) return CRC_ECUDA;
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    if (cudaMemsetAsync(ws, 0, f.ctl_bytes, stream) != cudaSuccess) return CRC_ECUDA;
    FusedArgs a;
    a.state = static_cast<uint8_t*>(state);
    a.B = p.B;
    a.L = p.L;
    a.N = p.N;
    a.K = p.K;
    a.C = p.C;
    a.R = p.R;
    a.T = T;
    a.SB = f.SB;
    a.TB = f.TB;
    a.n_bg = f.n_bg;
    a.n_tb = f.n_tb;
    a.tiles_per_tb = f.tiles_per_tb;
    a.num_tiles = f.num_tiles;
    a.ring = f.ring;
    a.kblocks = (p.d + RC::BK - 1) / RC::BK;
    a.n_items = f.n_items;
    a.ctl = reinterpret_cast<uint32_t*>(ws);
    a.tile_done = reinterpret_cast<uint32_t*>(ws + 256);
    a.readers = a.tile_done + f.ring;
    a.prog = a.readers + f.ring;
    a.ring_base = ws + f.ctl_bytes;
    a.slot_bytes = f.slot_bytes;
    a.tr_miss = trace ? trace->misses_dev : nullptr;
    a.tr_pro = trace ? trace->proactive_dev : nullptr;
    a.tr_mid = trace ? trace->cache_mid_dev : nullptr;
    a.tr_after = trace ? trace->cache_after_dev : nullptr;
    a.tr_sel = trace ? trace->topk_set_dev : nullptr;
    void* args[] = {(void*)&mh, (void*)&mw, (void*)&a};
    const int threads = Cfg::threads_for(p.R);
    cudaError_t e;
    if (PAIR) {
        cudaLaunchAttribute at[2];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = 2;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        at[1].id = cudaLaunchAttributeCooperative;
        at[1].val.cooperative = 1;
        cudaLaunchConfig_t c = {};
        c.gridDim = dim3((unsigned)grid);
        c.blockDim = dim3(threads);
        c.dynamicSmemBytes = Cfg::SMEM_BYTES;
        c.stream = stream;
        c.attrs = at;
        // CRC_PLAIN_CLUSTER_LAUNCH=1 drops the cooperative attribute so that a
        // kernel profiler, which cannot replay a cooperative cluster launch,
        // can run the same kernel; the grid still fits the GPU at once (the
        // occupancy query above), and were it ever not co-resident, the bounded
        // waits would end the call with CRC_ETIMEOUT
        c.numAttrs = plain_cluster_launch() ? 1 : 2;
        {
            ProfScope prof(CRC_KERNEL_FUSED, stream);
            e = cudaLaunchKernelExC(&c, (const void*)kern, args);
        }
        if (e != cudaSuccess) {
            (void)cudaGetLastError();
            grid = 0;
            return CRC_EUNSUPPORTED;
        }
    } else {
        ProfScope prof(CRC_KERNEL_FUSED, stream);
        e = cudaLaunchCooperativeKernel((const void*)kern, grid, threads, args,
                                        Cfg::SMEM_BYTES, stream);
    }
    note_launch();
    return e == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

// The GEMM on CTA pairs (N = 128: three heads, or two in update-only mode)
// when the tiles pair up; CRC_EUNSUPPORTED sends the call to one CTA per tile.
template <int NH, int H, int V, bool ALL_VALID, bool TRACED>
int launch_fused_pair(const crc_problem& p, const uint16_t* hidden, const uint16_t* w_cat, int T,
                      void* state, void* workspace, const crc_trace* trace,
                      cudaStream_t stream) {
    if constexpr (NH != 128) {
        return CRC_EUNSUPPORTED;
    } else {
        if (p.K <= 2)
            return launch_fused_t<NH, H, V, ALL_VALID, 2, true, TRACED>(p, hidden, w_cat, T,
                                                                        state, workspace, trace,
                                                                        stream);
        if (p.K <= 4)
            return launch_fused_t<NH, H, V, ALL_VALID, 4, true, TRACED>(p, hidden, w_cat, T,
                                                                        state, workspace, trace,
                                                                        stream);
        if (p.K <= 8)
            return launch_fused_t<NH, H, V, ALL_VALID, 8, true, TRACED>(p, hidden, w_cat, T,
                                                                        state, workspace, trace,
                                                                        stream);
        return CRC_EUNSUPPORTED;
    }
}

// Dispatch on heads (R > 0 needs the Spatio head) and the Top-K network width.
template <int NH, int V, bool ALL_VALID, bool TRACED>
int launch_fused_mode(const crc_problem& p, const uint16_t* hidden, const uint16_t* w_cat,
                       int T, void* state, void* workspace, const crc_trace* trace,
                       cudaStream_t stream) {
#define CRC_FUSED_KP(HV)                                                                      \
    {                                                                                         \
        const int rc = launch_fused_pair<NH, HV, V, ALL_VALID, TRACED>(p, hidden, w_cat, T,   \
                                                                       state, workspace,      \
                                                                       trace, stream);        \
        if (rc != CRC_EUNSUPPORTED) return rc;                                                \
    }                                                                                         \
    if (p.K <= 2)                                                                             \
        return launch_fused_t<NH, HV, V, ALL_VALID, 2, false, TRACED>(                        \
            p, hidden, w_cat, T, state, workspace, trace, stream);                            \
    if (p.K <= 4)                                                                             \
        return launch_fused_t<NH, HV, V, ALL_VALID, 4, false, TRACED>(                        \
            p, hidden, w_cat, T, state, workspace, trace, stream);                            \
    if (p.K <= 8)                                                                             \
        return launch_fused_t<NH, HV, V, ALL_VALID, 8, false, TRACED>(                        \
            p, hidden, w_cat, T, state, workspace, trace, stream);                            \
    return CRC_EUNSUPPORTED;
    if (p.R > 0) {
        CRC_FUSED_KP(3)
    } else {
        CRC_FUSED_KP(2)
    }
#undef CRC_FUSED_KP
}

// The kernel without trace writes unless the call asks for a trace array.
template <int NH, int V, bool ALL_VALID>
int launch_fused_for_n(const crc_problem& p, const uint16_t* hidden, const uint16_t* w_cat,
                       int T, void* state, void* workspace, const crc_trace* trace,
                       cudaStream_t stream) {
    const bool traced = trace && (trace->misses_dev || trace->proactive_dev ||
                                  trace->cache_mid_dev || trace->cache_after_dev ||
                                  trace->topk_set_dev);
    return traced ? launch_fused_mode<NH, V, ALL_VALID, true>(p, hidden, w_cat, T, state,
                                                              workspace, trace, stream)
                  : launch_fused_mode<NH, V, ALL_VALID, false>(p, hidden, w_cat, T, state,
                                                               workspace, nullptr, stream);
}

}  // namespace crc
