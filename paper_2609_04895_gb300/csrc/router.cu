// Host launcher of the router-heads kernel: tensor maps, tile plan, dispatch.
#include <cudaTypedefs.h>

#include <mutex>

#include "crc_internal.h"
#include "router_gemm.cuh"

namespace crc {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// hidden [B][T_total][L][d] bf16 viewed as a 4-D tensor (d, L, T, B); a box is
// 64 hidden elements (one 128-byte swizzle row) x 1 layer x TB tokens x SB streams.
bool make_hidden_map(CUtensorMap* m, const uint16_t* hidden, int B, int T_total, int L, int d,
                     int TB, int SB) {
    auto enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[4] = {(cuuint64_t)d, (cuuint64_t)L, (cuuint64_t)T_total, (cuuint64_t)B};
    cuuint64_t strides[3] = {(cuuint64_t)d * 2, (cuuint64_t)L * d * 2,
                             (cuuint64_t)T_total * L * d * 2};
    cuuint32_t box[4] = {64, 1, (cuuint32_t)TB, (cuuint32_t)SB};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<uint16_t*>(hidden), dims,
               strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// W_cat [L][3N][d] bf16 viewed as (d, 3N, L); a box is 64 x rows x 1 layer.
bool make_weight_map(CUtensorMap* m, const uint16_t* w, int L, int N3, int d, int rows) {
    auto enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)N3, (cuuint64_t)L};
    cuuint64_t strides[2] = {(cuuint64_t)d * 2, (cuuint64_t)N3 * d * 2};
    cuuint32_t box[3] = {64, (cuuint32_t)rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<uint16_t*>(w), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// scores [B][T_ext][L][3][NH] fp32 viewed as (NH, 3, L, T, B); a store box is
// 32 scores x 1 head x 1 layer x TBq tokens x SBq streams (32 rows, 128-byte rows).
bool make_scores_map(CUtensorMap* m, float* scores, int B, int T_ext, int L, int NH, int TBq,
                     int SBq) {
    auto enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[5] = {(cuuint64_t)NH, 3, (cuuint64_t)L, (cuuint64_t)T_ext, (cuuint64_t)B};
    cuuint64_t strides[4] = {(cuuint64_t)NH * 4, (cuuint64_t)3 * NH * 4,
                             (cuuint64_t)L * 3 * NH * 4, (cuuint64_t)T_ext * L * 3 * NH * 4};
    cuuint32_t box[5] = {32, 1, 1, (cuuint32_t)TBq, (cuuint32_t)SBq};
    cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 5, scores, dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {

template <int NH, int H>
int launch_router_t(const crc_problem& p, const uint16_t* hidden, int T_total, int t_begin,
                    int T_ext, const uint16_t* w_cat, float* scores, uint32_t* err,
                    cudaStream_t stream) {
    using Cfg = RouterCfg<NH, H>;
    int TB = 1;
    while (TB < T_ext && TB < Cfg::BM) TB <<= 1;
    const int SB = Cfg::BM / TB;
    CUtensorMap mh, mw;
    if (!make_hidden_map(&mh, hidden, p.B, T_total, p.L, p.d, TB, SB)) return CRC_ECUDA;
    if (!make_weight_map(&mw, w_cat, p.L, 3 * NH, p.d, Cfg::B_BOX_ROWS)) return CRC_ECUDA;
    CUtensorMap ms = mh;   // unused when a head is narrower than one 32-score store box
    if (Cfg::TMA_STORE) {
        const int TBq = TB < 32 ? TB : 32;
        if (!make_scores_map(&ms, scores, p.B, T_ext, p.L, NH, TBq, 32 / TBq)) return CRC_ECUDA;
    }
    RouterArgs a;
    a.scores = scores;
    a.err = err;
    a.B = p.B;
    a.L = p.L;
    a.d = p.d;
    a.t_begin = t_begin;
    a.T_ext = T_ext;
    a.SB = SB;
    a.TB = TB;
    a.n_sb = (p.B + SB - 1) / SB;
    a.n_tb = (T_ext + TB - 1) / TB;
    a.num_tiles = p.L * a.n_sb * a.n_tb;
    a.kblocks = (p.d + Cfg::BK - 1) / Cfg::BK;
    static bool attr_set = false;   // per instantiation
    if (!attr_set) {
        if (cudaFuncSetAttribute(router_heads_kernel<NH, H>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 Cfg::SMEM_BYTES) != cudaSuccess)
            return CRC_ECUDA;
        attr_set = true;
    }
    const int grid = a.num_tiles < sm_count() ? a.num_tiles : sm_count();
    {
        ProfScope prof(CRC_KERNEL_ROUTER, stream);
        router_heads_kernel<NH, H><<<grid, Cfg::THREADS, Cfg::SMEM_BYTES, stream>>>(mh, mw, ms, a);
    }
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

}  // namespace

int launch_router(const crc_problem& p, const uint16_t* hidden, int T_total, int t_begin,
                  int T_ext, const uint16_t* w_cat, int heads, float* scores,
                  uint32_t* err_word, cudaStream_t stream) {
    if (T_ext <= 0) return CRC_OK;
#define CRC_ROUTER_CASE(NHV)                                                                \
    case NHV:                                                                               \
        return heads == 3 ? launch_router_t<NHV, 3>(p, hidden, T_total, t_begin, T_ext,     \
                                                    w_cat, scores, err_word, stream)        \
                          : launch_router_t<NHV, 2>(p, hidden, T_total, t_begin, T_ext,     \
                                                    w_cat, scores, err_word, stream);
    switch (p.N) {
        CRC_ROUTER_CASE(16)
        CRC_ROUTER_CASE(32)
        CRC_ROUTER_CASE(64)
        CRC_ROUTER_CASE(128)
        default:
            return CRC_EUNSUPPORTED;
    }
#undef CRC_ROUTER_CASE
}

}  // namespace crc
