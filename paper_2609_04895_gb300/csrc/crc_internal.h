// Host-side internals shared by the translation units of the library.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/crc.h"

namespace crc {

// Count of kernels launched by the library (reported by crc_launch_count).
void note_launch();

// Brackets one kernel launch with CUDA events on its stream while
// crc_profile_begin() .. crc_profile_end() is active; otherwise a no-op.
struct ProfScope {
    ProfScope(int kind, cudaStream_t stream);
    ~ProfScope();
    int slot;
    cudaStream_t stream;
};

// Library-wide device error word for calls without a state.
uint32_t* device_error_word();

// Streaming multiprocessors of the current device.
int sm_count();

// Router heads over tokens [t_begin, t_begin + T_ext) of hidden [B][T_total][L][d];
// scores [B][T_ext][L][3][N].
int launch_router(const crc_problem& p, const uint16_t* hidden, int T_total, int t_begin,
                  int T_ext, const uint16_t* w_cat, int heads, float* scores,
                  uint32_t* err_word, cudaStream_t stream);

// Cache scan over T tokens of scores [B][T][L][3][N]; trace arrays are
// [B][trace_T][L][..] and this call writes tokens trace_t0 .. trace_t0 + T - 1.
int launch_scan(const crc_problem& p, const float* scores, int T, void* state,
                const crc_trace* trace, int trace_T, int trace_t0, cudaStream_t stream);

// Tensor maps (router.cu): hidden [B][T_total][L][d] as (d, L, T, B) with a
// 64 x 1 x TB x SB box; W_cat [L][3N][d] as (d, 3N, L) with a 64 x rows x 1 box.
bool make_hidden_map(CUtensorMap* m, const uint16_t* hidden, int B, int T_total, int L, int d,
                     int TB, int SB);
bool make_weight_map(CUtensorMap* m, const uint16_t* w, int L, int N3, int d, int rows);

// Fused route-and-cache (fused_*.cu): workspace bytes that enable it for this
// problem, and the launch (CRC_EUNSUPPORTED when the problem is outside it).
size_t fused_workspace_bytes(const crc_problem& p);
int launch_fused(const crc_problem& p, const uint16_t* hidden, const uint16_t* w_cat, int T,
                 void* state, void* workspace, size_t workspace_bytes, const crc_trace* trace,
                 cudaStream_t stream);
int launch_fused_n16(const crc_problem& p, const uint16_t* hidden, const uint16_t* w_cat, int T,
                     void* state, void* workspace, const crc_trace* trace,
                     cudaStream_t stream);
int launch_fused_n32(const crc_problem& p, const uint16_t* hidden, const uint16_t* w_cat, int T,
                     void* state, void* workspace, const crc_trace* trace,
                     cudaStream_t stream);
int launch_fused_n64(const crc_problem& p, const uint16_t* hidden, const uint16_t* w_cat, int T,
                     void* state, void* workspace, const crc_trace* trace,
                     cudaStream_t stream);
// Cache scan under a comparison policy (policy_scan.cuh).
int launch_policy_scan(const crc_problem& p, const float* scores, int T, void* state,
                       const crc_trace* trace, int trace_T, int trace_t0, int policy,
                       int lambda2, cudaStream_t stream);
int launch_fused_n128(const crc_problem& p, const uint16_t* hidden, const uint16_t* w_cat, int T,
                      void* state, void* workspace, const crc_trace* trace,
                     cudaStream_t stream);

// Soft Top-B coverage losses (loss.cu): the work split over token chunks and
// the launch; workspace = per-task sums, 16 bytes per task.
struct LossPlan {
    int nchunks, chunk;
};
LossPlan loss_plan(int B, int L, int T);
// Per-task partial sums the loss kernels may write (the workspace of
// crc_cache_loss): the plan's tasks, or for N <= 32, whose chunks are sized
// at launch, B * L tasks per 32 tokens.
long long loss_task_slots(int B, int L, int T, int N);
int launch_cache_loss(const crc_problem& p, const float* probs, int T, int heads, int top_b,
                      double tau, double w_T, double w_ST, float* loss, double* means,
                      float* grad, void* workspace, cudaStream_t stream);

int launch_state_init(const crc_problem& p, void* state, size_t bytes, cudaStream_t stream);

int launch_synth_hidden(int B, int T, int L, int d, int t0, uint32_t seed, double rho_t,
                        double rho_l, const uint8_t* attempts, uint16_t* out, float* carry,
                        cudaStream_t stream);
int launch_synth_weights(int L, int N, int d, uint32_t seed, int copy_init, uint16_t* out,
                         cudaStream_t stream);

}  // namespace crc
