// Seeded synthetic inputs on the device (not part of the method).
//
// Definition (identical bits to the host generator):
//  * Philox4x32-10 (Salmon et al., SC'11): multipliers 0xD2511F53 (word 0)
//    and 0xCD9E8D57 (word 2), round output (hi1^c1^k0, lo1, hi0^c3^k1, lo0),
//    key bumped by 0x9E3779B9 / 0xBB67AE85 between rounds.
//  * one call -> 8 x 16-bit integers -> two Irwin-Hall(4) unit variates:
//    fp32(u0+u1+u2+u3 - 131070) * fp32(sqrt(3 / (65536^2 - 1))).
//  * hidden: AR(1) over layers g = rho_l*g + s_l*eps, then AR(1) over tokens
//    h = rho_t*h_prev + s_t*g, each product and sum a separate round-to-
//    nearest fp32 operation; stored as bf16 (round to nearest even).
//    Counters (pair j, layer l, token t, stream b | attempt << 16), key
//    (seed, 0x48494444).
//  * weights: bf16(eps * fp32(1/sqrt(d))), counters (j, expert, head, layer),
//    key (seed, 0x57474854).
#include <cuda_bf16.h>

#include "crc_internal.h"

namespace crc {
namespace {

constexpr uint32_t kTagHidden = 0x48494444u;
constexpr uint32_t kTagWeight = 0x57474854u;

__device__ __forceinline__ void philox4x32_10(uint32_t (&c)[4], uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        if (r) {
            k0 += 0x9E3779B9u;
            k1 += 0xBB67AE85u;
        }
        const uint32_t hi0 = __umulhi(0xD2511F53u, c[0]), lo0 = 0xD2511F53u * c[0];
        const uint32_t hi1 = __umulhi(0xCD9E8D57u, c[2]), lo1 = 0xCD9E8D57u * c[2];
        const uint32_t n0 = hi1 ^ c[1] ^ k0;
        const uint32_t n2 = hi0 ^ c[3] ^ k1;
        c[0] = n0;
        c[1] = lo1;
        c[2] = n2;
        c[3] = lo0;
    }
}

__device__ __forceinline__ float irwin_hall4(uint32_t wa, uint32_t wb) {
    const int s = (int)(wa & 0xFFFFu) + (int)(wa >> 16) + (int)(wb & 0xFFFFu) + (int)(wb >> 16);
    return __fmul_rn((float)(s - 131070), __uint_as_float(0x37DDB3D7u));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
    const uint32_t lo = __bfloat16_as_ushort(__float2bfloat16_rn(a));
    const uint32_t hi = __bfloat16_as_ushort(__float2bfloat16_rn(b));
    return lo | (hi << 16);
}

struct HiddenArgs {
    int B, T, L, d, t0;
    uint32_t seed;
    float rt, st, rl, sl;
    const uint8_t* attempts;   // [B][T][L] or null
    uint32_t* out;             // bf16 pairs [B][T][L][d/2]
    float2* carry;             // [B][L][d/2]
};

// One block per (stream, 128 element pairs); the token recurrence's carry
// h_{t-1, l} for every layer lives in shared memory ([L][128] float2).
constexpr int kSynthPairs = 128;

__global__ void __launch_bounds__(kSynthPairs) synth_hidden_kernel(HiddenArgs a) {
    extern __shared__ float2 carry_s[];
    const int pairs = a.d >> 1;
    const int blocks_per_stream = (pairs + kSynthPairs - 1) / kSynthPairs;
    const int b = blockIdx.x / blocks_per_stream;
    const int j = (blockIdx.x % blocks_per_stream) * kSynthPairs + threadIdx.x;
    const bool live = j < pairs;
    if (live && a.t0 > 0)
        for (int l = 0; l < a.L; ++l)
            carry_s[l * kSynthPairs + threadIdx.x] = a.carry[((size_t)b * a.L + l) * pairs + j];
    if (!live) return;
    for (int t = 0; t < a.T; ++t) {
        const uint32_t tg = (uint32_t)(a.t0 + t);
        float g0 = 0.f, g1 = 0.f;
        for (int l = 0; l < a.L; ++l) {
            const uint32_t att = a.attempts ? a.attempts[((size_t)b * a.T + t) * a.L + l] : 0u;
            uint32_t c[4] = {(uint32_t)j, (uint32_t)l, tg, (uint32_t)b | (att << 16)};
            philox4x32_10(c, a.seed, kTagHidden);
            const float e0 = irwin_hall4(c[0], c[1]);
            const float e1 = irwin_hall4(c[2], c[3]);
            if (l == 0) {
                g0 = e0;
                g1 = e1;
            } else {
                g0 = __fadd_rn(__fmul_rn(a.rl, g0), __fmul_rn(a.sl, e0));
                g1 = __fadd_rn(__fmul_rn(a.rl, g1), __fmul_rn(a.sl, e1));
            }
            float2& cs = carry_s[l * kSynthPairs + threadIdx.x];
            float h0 = g0, h1 = g1;
            if (tg > 0) {
                h0 = __fadd_rn(__fmul_rn(a.rt, cs.x), __fmul_rn(a.st, g0));
                h1 = __fadd_rn(__fmul_rn(a.rt, cs.y), __fmul_rn(a.st, g1));
            }
            cs = make_float2(h0, h1);
            a.out[(((size_t)b * a.T + t) * a.L + l) * pairs + j] = pack_bf16x2(h0, h1);
        }
    }
    for (int l = 0; l < a.L; ++l)
        a.carry[((size_t)b * a.L + l) * pairs + j] = carry_s[l * kSynthPairs + threadIdx.x];
}

struct WeightArgs {
    int L, N, d, copy_init;
    uint32_t seed;
    float scale;
    uint32_t* out;   // bf16 pairs [L][3N][d/2]
};

__global__ void synth_weights_kernel(WeightArgs a) {
    const int pairs = a.d >> 1;
    const size_t total = (size_t)a.L * 3 * a.N * pairs;
    const size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= total) return;
    const int j = (int)(idx % pairs);
    const int rowi = (int)((idx / pairs) % (3 * a.N));
    const int l = (int)(idx / ((size_t)pairs * 3 * a.N));
    int h = rowi / a.N;
    const int e = rowi % a.N;
    int ls = l;
    if (a.copy_init && h > 0) {          // W^T_l = W^R_l, W^S_l = W^R_{l+1 mod L}
        ls = (h == 1) ? l : (l + 1) % a.L;
        h = 0;
    }
    uint32_t c[4] = {(uint32_t)j, (uint32_t)e, (uint32_t)h, (uint32_t)ls};
    philox4x32_10(c, a.seed, kTagWeight);
    const float e0 = __fmul_rn(irwin_hall4(c[0], c[1]), a.scale);
    const float e1 = __fmul_rn(irwin_hall4(c[2], c[3]), a.scale);
    a.out[idx] = pack_bf16x2(e0, e1);
}

}  // namespace

int launch_synth_hidden(int B, int T, int L, int d, int t0, uint32_t seed, double rho_t,
                        double rho_l, const uint8_t* attempts, uint16_t* out, float* carry,
                        cudaStream_t stream) {
    HiddenArgs a;
    a.B = B;
    a.T = T;
    a.L = L;
    a.d = d;
    a.t0 = t0;
    a.seed = seed;
    a.rt = (float)rho_t;
    a.st = (float)sqrt(1.0 - rho_t * rho_t);
    a.rl = (float)rho_l;
    a.sl = (float)sqrt(1.0 - rho_l * rho_l);
    a.attempts = attempts;
    a.out = reinterpret_cast<uint32_t*>(out);
    a.carry = reinterpret_cast<float2*>(carry);
    const int blocks = B * ((d / 2 + kSynthPairs - 1) / kSynthPairs);
    const size_t smem = (size_t)L * kSynthPairs * sizeof(float2);
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(synth_hidden_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem) != cudaSuccess)
        return CRC_EUNSUPPORTED;
    {
        ProfScope prof(CRC_KERNEL_SYNTH, stream);
        synth_hidden_kernel<<<blocks, kSynthPairs, smem, stream>>>(a);
    }
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

int launch_synth_weights(int L, int N, int d, uint32_t seed, int copy_init, uint16_t* out,
                         cudaStream_t stream) {
    WeightArgs a;
    a.L = L;
    a.N = N;
    a.d = d;
    a.copy_init = copy_init;
    a.seed = seed;
    a.scale = (float)(1.0 / sqrt((double)d));
    a.out = reinterpret_cast<uint32_t*>(out);
    const int threads = 256;
    const size_t n = (size_t)L * 3 * N * (d / 2);
    {
        ProfScope prof(CRC_KERNEL_SYNTH, stream);
        synth_weights_kernel<<<(unsigned)((n + threads - 1) / threads), threads, 0, stream>>>(a);
    }
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

}  // namespace crc
