// Host-side declarations shared by the kernel files and the C-ABI layer.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

namespace sas {

using bf16 = __nv_bfloat16;

// Builds a 3-D TMA descriptor over a dense bf16 tensor [outer][rows][inner]
// with a (box_inner x box_rows x 1) box and 128-byte swizzle.  box_inner must
// be 64 (one 128-byte swizzle span).  Out-of-range rows read as zero.
// Returns 0 on success, else a CUresult.
int make_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows, uint64_t outer,
                      uint32_t box_inner, uint32_t box_rows);

struct KernelEnv {
    cudaStream_t stream;
    int* status;        // device status word
    long long limit;    // bounded-wait budget in SM cycles
};

// ---- tcgen05 GEMM:  C[b] = epi(A[b] @ B[b % b_mod]^T (+ bias)), bf16 out (the MLP).
// A: [batches][M][K], B: [nb][N][K], C: [batches][M][ldc] (row stride ldc).
// N must be a multiple of bn (64, 128 or 256), K a multiple of 64.
struct GemmProblem {
    const void* A;
    const void* B;
    void* C;
    const void* bias;    // bf16 [N] or nullptr
    int M, N, K;
    int batches, b_mod;
    long long c_batch_stride;
    int ldc;
    int gelu;            // 1: exact-erf GELU epilogue
    int bn;              // 64, 128 or 256
    int max_ctas;        // persistent grid size cap (0: one per SM)
};
cudaError_t launch_gemm(const GemmProblem& p, const KernelEnv& env, const char** err);

// ---- a1: block summaries and key projection
// Kt[bh][m][:] = bf16(Wk[h] @ mean(K[bh][64m : 64m+64][:])) for m < F = N / 64.
cudaError_t launch_pool(const void* K, const void* Wk, void* Kt, int BH, int H, int N, int d, int d_sel,
                        const KernelEnv& env);

// ---- a2-a4: selection.  Per query row: the log-sum-exp of its C_i causal
// scores, the Top-K blocks (ascending, -1 padded) with their log-gates, and
// per 128-row tile the sorted union of kept blocks below the tile's diagonal.
struct SelectArgs {
    int BH, H, N, C, T, topk, d_sel;
    int gate_act;                   // 0 softmax (log g = s - LSE), 1 sigmoid, 2 logit (log g = s)
    float score_scale;              // 1/sqrt(d_sel) for projected scores, 1 for given scores
    const float* scores;            // SCORES_GIVEN: [BH][N][C]
    const void* Q;                  // MEANPOOL_PROJ: queries bf16 [BH][N][d]
    const void* Wq;                 // MEANPOOL_PROJ: query projection bf16 [H][d_sel][d]
    const void* Kt;                 // MEANPOOL_PROJ: projected block summaries bf16 [BH][F][d_sel]
    int d;
    int F;
    int32_t* sel_idx;               // [BH][N][topk]
    float* sel_logg;                // [BH][N][topk]
    int32_t* union_idx;             // [BH][T][C]
    int32_t* union_cnt;             // [BH][T]
};
cudaError_t launch_select(const SelectArgs& a, const KernelEnv& env, const char** err);

// ---- a5: fused gated block-sparse attention forward.
struct AttnArgs {
    const void* Q;
    const void* K;
    const void* V;
    void* O;
    float* LSE;                 // may be null
    const int32_t* union_idx;
    const int32_t* union_cnt;
    const int32_t* sel_idx;
    const float* sel_logg;
    int BH, N, d, C, T, topk, mode;
    int gate_pos;               // 0 inner (+ log g in the logits), 1 outer (g scales P after the softmax)
    float sm_scale;
    int* sched;                 // 16 zeroed bytes owned by the caller, left zeroed after each launch
};
cudaError_t launch_attn(const AttnArgs& a, const KernelEnv& env, const char** err);

// ---- failure-path self test (bounded wait on a barrier nothing completes)
cudaError_t launch_wait_selftest(int* status, long long limit, cudaStream_t stream);

}  // namespace sas
