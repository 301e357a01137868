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

// Raises `func`'s dynamic shared-memory limit to at least `bytes` on the
// current device.  The attribute belongs to the device, so it is recorded per
// (kernel, device): the first launch on each device sets it, later ones find
// the record and call nothing (so a launch inside a stream capture that was
// preceded by one outside it sets nothing).  Thread-safe.
// max_carveout also asks for the largest shared-memory carveout (L1 shrinks to
// what is left), for kernels that need it to fit several CTAs on an SM.
cudaError_t ensure_smem_attr(const void* func, size_t bytes, bool max_carveout = false);
// Multiprocessor count of the current device (cached per device, thread-safe).
int device_sm_count();

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
// Packed sequences (tiles non-null, F = N / 64 + max_seqs slots): block m of
// sequence s goes to slot floor(cu[s] / 64) + s + m (the tile table's entries
// carry the sequence index s).
cudaError_t launch_pool(const void* K, const void* Wk, void* Kt, int BH, int H, int N, int d, int d_sel,
                        const KernelEnv& env, int F = -1, const int4* tiles = nullptr, const int* ntiles = nullptr,
                        int T = 0);

// ---- a2-a4: selection.  Per query row: the log-sum-exp of its C_i causal
// scores, the Top-K blocks (ascending, -1 padded) with their log-gates, and
// per 128-row tile the sorted union of kept blocks below the tile's diagonal.
struct SelectArgs {
    int BH, H, N, C, T, topk, d_sel;   // BH, H: selection groups (KV heads) x batch, KV heads
    int G;                          // query heads per group (MEANPOOL_PROJ: the gate query reads all G)
    int gate_act;                   // 0 softmax (log g = s - LSE), 1 sigmoid, 2 logit (log g = s)
    float score_scale;              // 1/sqrt(d_sel) for projected scores, 1 for given scores
    const float* scores;            // SCORES_GIVEN: [BH][N][C]
    const void* Q;                  // MEANPOOL_PROJ: queries bf16 [BH][N][d]
    const void* Wq;                 // MEANPOOL_PROJ: gate-query projection bf16 [H][d_sel][G d]
    const void* Kt;                 // MEANPOOL_PROJ: projected block summaries bf16 [BH][F][d_sel]
    int d;
    int F;
    int32_t* sel_idx;               // [BH][N][topk]
    float* sel_logg;                // [BH][N][topk]
    int32_t* union_idx;             // [BH][T][C]
    int32_t* union_cnt;             // [BH][T]
    // packed sequences (given scores only): T tile slots, the first *ntiles
    // used; tiles[g] = {first row, tile index within the sequence, sequence
    // length, 0}; N is then the token capacity of each head.  Null otherwise.
    const int4* tiles;
    const int* ntiles;
    // full training scope: no Top-K; each row's log-sum-exp of its scores into
    // full_lse [BH][N] and, with the learned selector, its scores into
    // full_table [BH][N][C] (entries m < C_i).  Null in the sparse scope.
    float* full_lse;
    float* full_table;
    // full*: a noise table [BH][N][C] added to the scores before the gate and
    // the Top-K (null otherwise)
    const float* noise;
};
cudaError_t launch_select(const SelectArgs& a, const KernelEnv& env, const char** err);
// Builds the tile table of packed sequences cu[0..S] (device offsets) with
// sequences of at most max_len tokens within Ncap rows; bad offsets set the
// status word to SAS_ERR_INVALID_ARG and leave *ntiles = 0.  Slots are
// ordered by local tile index, longest sequences first: local tile t of the
// sequence of rank r sits at slot tile_off[t] + r (tile_off: ceil(max_len /
// 128) + 1 ints).
cudaError_t launch_varlen_tiles(const int32_t* cu, int S, int Ncap, int max_len, int4* tiles, int* ntiles,
                                int* tile_off, const KernelEnv& env);

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
    int BH, N, d, C, T, topk, mode;    // BH: query heads x batch
    int G;                      // query heads per KV group (1 without GQA): K, V, lists of group bh / G
    const int4* tiles;          // packed sequences: as in SelectArgs (null otherwise)
    const int* ntiles;
    int gate_pos;               // 0 inner (+ log g in the logits), 1 outer (g scales P after the softmax)
    float sm_scale;
    int* sched;                 // 16 zeroed bytes owned by the caller, left zeroed after each launch
    // full training scope: every historical block of a row kept with
    // log g_m = full_table[row][m] - full_lse[row] (tables per KV group); null otherwise
    const float* full_table;
    const float* full_lse;
    // head-packed GQA tiles (seg_rows = 128 / G tokens of each of the G heads;
    // 0: tiles of 128 rows of one head): segment unions [BH/G][nseg][cap]
    // (cap = min(C, seg_rows topk)) and their counts; nseg = ceil(N / seg_rows),
    // or with packed sequences G per tile slot (nseg = T G, part k of slot g at g G + k)
    int seg_rows;
    int nseg;
    const int32_t* seg_union_idx;
    const int32_t* seg_union_cnt;
};
cudaError_t launch_attn(const AttnArgs& a, const KernelEnv& env, const char** err);
// Segment unions for head-packed tiles: per (KV group, segment of seg_rows
// tokens) the sorted union of the tokens' kept blocks (from the kept lists).
cudaError_t launch_seg_unions(const int32_t* sel_idx, int BHkv, int N, int C, int topk, int seg_rows, int nseg,
                              int32_t* seg_union_idx, int32_t* seg_union_cnt, const KernelEnv& env,
                              const int4* tiles = nullptr, const int* ntiles = nullptr);

// ---- decode step (Alg. 2, per-group selection over a paged cache).
struct DecodeArgs {
    int B, Hq, Hkv, G, d, d_sel, topk, max_blocks, num_pages;
    int dense;
    float sm_scale;
    const void* q;              // bf16 [B][Hq][d]
    const void* k_new;          // bf16 [B][Hkv][d] or null
    const void* v_new;
    void* K_cache;              // bf16 [P][Hkv][64][d]
    void* V_cache;
    const int32_t* block_table; // [B][max_blocks]
    const int32_t* seq_lens;    // [B]
    const void* Wq;             // bf16 [Hkv][d_sel][G*d]
    const void* Wk;             // bf16 [Hkv][d_sel][d]
    void* Ksum;                 // bf16 [B][Hkv][max_blocks][d_sel]
    void* O;                    // bf16 [B][Hq][d]
    float* LSE;                 // [B][Hq] or null
    int32_t* sel_idx;           // [B][Hkv][topk] or null
    // workspace
    void* qt;                   // bf16 [B*Hkv][d_sel] gate queries
    uint32_t* cand_key;         // [B*Hkv][nsplit_s][max(topk,1)] per-CTA Top-K candidates (order keys)
    int32_t* cand_idx;          // [B*Hkv][nsplit_s][max(topk,1)] their blocks (-1: empty slot)
    int32_t* list;              // [B*Hkv][64] kept blocks, ascending
    int32_t* list_n;            // [B*Hkv]
    float* part;                // [B*Hkv][nsplit_a][G][d + 2] split-attention partials
    int* cnt_sel;               // [B*Hkv] arrival counters, zero between launches
    int* cnt_attn;              // [B*Hkv]
    int nsplit_s;               // score CTAs per group (kDecScoreChunk blocks each)
    int nsplit_a, bpc, nst;     // attention CTAs per group, list entries per CTA, ring stages
};
constexpr int kDecScoreChunk = 256;
// Attention split for a group list of at most max_len entries.
void decode_attn_split(int max_len, int d, int* nsplit, int* bpc, int* nst);
// Dynamic shared memory the score and attention kernels need.
size_t decode_score_smem(int nsplit, int topk, int d_sel);
size_t decode_attn_smem(int d, int G, int nst, int bpc);
// Sets the kernels' shared-memory limits for these arguments (before any capture).
cudaError_t decode_prepare(const DecodeArgs& a);
cudaError_t launch_decode_prep(const DecodeArgs& a, const KernelEnv& env);
cudaError_t launch_decode_score(const DecodeArgs& a, const KernelEnv& env);
cudaError_t launch_decode_attn(const DecodeArgs& a, const KernelEnv& env);
cudaError_t launch_decode_summarize(const DecodeArgs& a, const KernelEnv& env);

// ---- backward of the training forward (Alg. 4), d = 128, inner softmax gates.
struct AttnBwdArgs {
    const void* Q;
    const void* K;
    const void* V;
    const void* O;
    const void* dO;
    const float* LSE;
    const int32_t* union_idx;   // the forward's per-tile block lists
    const int32_t* union_cnt;
    const int32_t* sel_idx;     // the forward's kept lists and log-gates
    const float* sel_logg;
    const float* scores;        // given scores (for ds) or null
    void* dQ;
    void* dK;
    void* dV;
    float* dlogg;               // [BH / G][N][topk] (per KV group: the G heads' sum)
    float* ds;                  // [BH / G][N][C] or null
    float* dlogg_heads;         // G > 1: [BH][N][topk] per query head, summed into dlogg
    // workspace
    float* delta;               // [BH][N]
    int32_t* inv_cnt;           // [BH*T]
    int32_t* inv_off;           // [BH*T + 1]
    int32_t* inv_cursor;        // [BH*T]
    int32_t* inv_tiles;         // entries of the inverted lists
    int32_t* inv_pos;           // their block positions
    int32_t* slot_off;          // [BH*T + 1] first offset slot of each tile
    float* offs;                // [slots][128] per-row offsets written by pass 1
    // packed sequences: the forward's tile table (as in SelectArgs) and its
    // per-local-tile first slots; null for [B, H, N, d] batches
    const int4* tiles;
    const int* ntiles;
    const int* tile_off;
    // head-packed tiles (as in AttnArgs; seg_rows = 0: tiles of one head):
    // segments of seg_rows tokens x G heads, their unions with row stride seg_cap
    int seg_rows, nseg, seg_cap;
    const int32_t* seg_union_idx;
    const int32_t* seg_union_cnt;
    int N, C, T, BH, topk, mode, d;
    int G;                      // query heads per KV group: K, V, the lists and the gate gradients are per group
    float sm_scale;
    // pass 1 and the gate gradients only (no pass 2; dQ and offs may be null): the
    // gate pass of the hard Top-K gate under the straight-through estimator
    bool gate_only;
    int act;                    // gate activation (sas_gate_act) of the score gradient
    int pos;                    // gate position (sas_gate_pos): 1 = outer, o = softmax(z) (g . V)
};
extern const int kBwdMaxTiles;   // query tiles per head the backward supports (head-packed: segments + G)
cudaError_t launch_bwd_slots(const AttnBwdArgs& a, const KernelEnv& env, long long* total);
cudaError_t launch_attn_bwd(const AttnBwdArgs& a, const KernelEnv& env, const char** err);
// Kept lists that hold every historical block of each row (idx[m] = m, lg[m] =
// s_m - lse of the row, [BHkv][N][C]) and tile unions of every block below the
// tile's diagonal ([BHkv][T][C], counts [BHkv][T]); s and lse per KV group.
cudaError_t launch_bwd_dense_lists(const float* s, const float* lse, int BHkv, int N, int C, int T, int32_t* idx,
                                   float* lg, int32_t* uidx, int32_t* ucnt, const KernelEnv& env);
// Each row's log-sum-exp over its C_i = floor(i / 64) scores ([rows][C] fp32,
// rows = heads x N), 0 for C_i = 0.
cudaError_t launch_row_lse(const float* scores, int N, int C, long long rows, float* out, const KernelEnv& env);

// ---- failure-path self test (bounded wait on a barrier nothing completes)
cudaError_t launch_wait_selftest(int* status, long long limit, cudaStream_t stream);

}  // namespace sas
