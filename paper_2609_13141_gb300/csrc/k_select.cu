// a2-a4: selector scores, causal log-gates and exact Top-K block selection.
//
// For query row i (block c_i = floor(i/64), C_i = c_i historical blocks):
//   LSE_i      = log sum_{m < C_i} exp(s_im)                  (Eq. normalized_log_gate)
//   I_i        = the K largest s_im, ties to the lower index   (Eq. selected_context)
//   sel_idx_i  = I_i in ascending order, -1 padded
//   sel_logg_i = s_im - LSE_i for m in I_i                      (log g of the kept blocks)
// and for each 128-row tile t the sorted union of kept blocks below the tile's
// two diagonal blocks (m < 2t): the list of historical key blocks the
// attention kernel visits for that tile (Alg. 3 skips the others).
//
// Selection compares the fp32 scores directly (Alg. 2 selects on s; the
// order is the same as on g because log g = s - LSE), so the Top-K decision
// never depends on how LSE was rounded.
//
// One CTA owns one (batch*head, 128-row tile); one thread owns one row and
// keeps its running max/sum and its Top-K candidates (a column of a shared
// array, so the 32 rows of a warp never share a bank).  Candidates arrive in
// ascending block order, so a later candidate with an equal score is worse
// and only a strictly larger score evicts the current worst entry.
//
// Two score sources:
//   * scores given: 32x32 score sub-tiles are staged through shared memory
//     with coalesced 128-byte row loads;
//   * learned selector: s = Qt Kt^T / sqrt(d_sel) is computed on the tensor
//     cores -- TMA brings the tile's 128 projected queries once and 64-block
//     chunks of projected block summaries in a double-buffered ring, one
//     thread issues tcgen05.mma (M=128, N=64) into two TMEM buffers, and the
//     row threads read their scores back with tcgen05.ld.
#include <math_constants.h>

#include "internal.h"
#include "ptx.cuh"

namespace sas {
namespace {

constexpr int kRows = 128;
constexpr float kLog2e = 1.4426950408889634f;

struct SelParams {
    int N, C, T, F, topk;
    float score_scale;
    const float* scores;
    int32_t* sel_idx;
    float* sel_logg;
    int32_t* union_idx;
    int32_t* union_cnt;
    int* status;
    long long limit;
};

// Per-row selection state.  ts/tm point at this row's column of the shared
// candidate arrays (element e of the column at offset e * kRows).
struct RowSel {
    float mx, sum;
    float* ts;
    int* tm;
    int K, cnt;
    float worst_s;
    int worst_m, worst_pos;
};

__device__ __forceinline__ void rescan_worst(RowSel& r) {
    float ws = CUDART_INF_F;
    int wm = -1, wp = 0;
    for (int e = 0; e < r.K; ++e) {
        const float s = r.ts[e * kRows];
        const int m = r.tm[e * kRows];
        if (s < ws || (s == ws && m > wm)) { ws = s; wm = m; wp = e; }
    }
    r.worst_s = ws;
    r.worst_m = wm;
    r.worst_pos = wp;
}

__device__ __forceinline__ void topk_push(RowSel& r, float s, int m) {
    if (r.cnt < r.K) {
        r.ts[r.cnt * kRows] = s;
        r.tm[r.cnt * kRows] = m;
        if (++r.cnt == r.K) rescan_worst(r);
    } else if (s > r.worst_s) {
        r.ts[r.worst_pos * kRows] = s;
        r.tm[r.worst_pos * kRows] = m;
        rescan_worst(r);
    }
}

// Consumes 32 scores of blocks m0 .. m0+31; entries at or past C_i are ignored.
__device__ __forceinline__ void row_consume32(RowSel& r, const float (&v)[32], int m0, int Ci) {
    const int lim = Ci - m0;
    if (lim <= 0) return;
    float cm = -CUDART_INF_F;
#pragma unroll
    for (int j = 0; j < 32; ++j)
        if (j < lim) cm = fmaxf(cm, v[j]);
    const float nm = fmaxf(r.mx, cm);
    float acc = 0.f;
#pragma unroll
    for (int j = 0; j < 32; ++j)
        if (j < lim) acc += fast_exp2((v[j] - nm) * kLog2e);
    r.sum = r.sum * fast_exp2((r.mx - nm) * kLog2e) + acc;
    r.mx = nm;
    if (r.K > 0) {
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (j < lim) topk_push(r, v[j], m0 + j);
    }
}

// Sorts the kept blocks by index, writes sel_idx / sel_logg for row i and
// marks kept blocks below `diag` (= 2t) in the tile's union bitmap.
__device__ __forceinline__ void row_finish(RowSel& r, const SelParams& p, long long row_off, int Ci, int diag,
                                           uint32_t* bitmap) {
    const int n = r.cnt;
    const float lse = Ci > 0 ? r.mx + logf(r.sum) : 0.f;
    for (int a = 1; a < n; ++a) {
        const int km = r.tm[a * kRows];
        const float ks = r.ts[a * kRows];
        int b = a - 1;
        while (b >= 0 && r.tm[b * kRows] > km) {
            r.tm[(b + 1) * kRows] = r.tm[b * kRows];
            r.ts[(b + 1) * kRows] = r.ts[b * kRows];
            --b;
        }
        r.tm[(b + 1) * kRows] = km;
        r.ts[(b + 1) * kRows] = ks;
    }
    int32_t* oi = p.sel_idx + row_off * p.topk;
    float* ol = p.sel_logg + row_off * p.topk;
    for (int e = 0; e < p.topk; ++e) {
        if (e < n) {
            const int m = r.tm[e * kRows];
            oi[e] = m;
            ol[e] = r.ts[e * kRows] - lse;
            if (m < diag) atomicOr(&bitmap[m >> 5], 1u << (m & 31));
        } else {
            oi[e] = -1;
            ol[e] = 0.f;
        }
    }
}

// One warp turns the tile bitmap (blocks < diag) into a sorted list.
__device__ __forceinline__ void compact_union(const uint32_t* bitmap, int diag, int32_t* out, int32_t* out_cnt) {
    const int lane = threadIdx.x & 31;
    const int nwords = (diag + 31) >> 5;
    int base = 0;
    for (int w0 = 0; w0 < nwords; w0 += 32) {
        const int w = w0 + lane;
        uint32_t bits = w < nwords ? bitmap[w] : 0u;
        const int cnt = __popc(bits);
        int incl = cnt;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += v;
        }
        int pos = base + incl - cnt;
        while (bits) {
            const int b = __ffs(bits) - 1;
            bits &= bits - 1;
            out[pos++] = w * 32 + b;
        }
        base += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) *out_cnt = base;
}

// ------------------------------------------------------------ scores given

__global__ void __launch_bounds__(128) select_given_kernel(SelParams p) {
    extern __shared__ __align__(16) uint8_t dsm[];
    __shared__ float stage[4][32][33];

    const int t = p.T - 1 - static_cast<int>(blockIdx.x);
    const int bh = blockIdx.y;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int r = threadIdx.x;
    const int i = t * kRows + r;
    const bool valid = i < p.N;
    const int Ci = valid ? (i >> 6) : 0;
    const int diag = 2 * t;

    float* ts = reinterpret_cast<float*>(dsm);
    int* tm = reinterpret_cast<int*>(ts + p.topk * kRows);
    uint32_t* bitmap = reinterpret_cast<uint32_t*>(tm + p.topk * kRows);
    const int nwords = (p.C + 31) >> 5;
    for (int w = threadIdx.x; w < nwords; w += blockDim.x) bitmap[w] = 0u;
    __syncthreads();

    RowSel rs{-CUDART_INF_F, 0.f, ts + r, tm + r, p.topk, 0, 0.f, 0, 0};

    const int row0 = t * kRows + warp * 32;
    const int last = min(row0 + 31, p.N - 1);
    const int Cw = row0 < p.N ? (last >> 6) : 0;   // largest C_i among the warp's rows
    const float* sbase = p.scores + static_cast<long long>(bh) * p.N * p.C;
    for (int m0 = 0; m0 < Cw; m0 += 32) {
        const int m = m0 + lane;
#pragma unroll 4
        for (int rho = 0; rho < 32; ++rho) {
            const int row = row0 + rho;
            float v = 0.f;
            if (row < p.N && m < p.C) v = __ldg(sbase + static_cast<long long>(row) * p.C + m);
            stage[warp][lane][rho] = v;
        }
        __syncwarp();
        float v[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = stage[warp][j][lane] * p.score_scale;
        __syncwarp();
        row_consume32(rs, v, m0, Ci);
    }
    if (valid) row_finish(rs, p, static_cast<long long>(bh) * p.N + i, Ci, diag, bitmap);
    __syncthreads();
    if (warp == 0)
        compact_union(bitmap, diag, p.union_idx + (static_cast<long long>(bh) * p.T + t) * p.C,
                      p.union_cnt + static_cast<long long>(bh) * p.T + t);
}

// --------------------------------------------------------- learned selector

template <int DS>
struct SelProjCfg {
    static constexpr int Q_BYTES = kRows * DS * 2;
    static constexpr int KC_BYTES = 64 * DS * 2;   // 64 blocks per chunk
    static constexpr int TILE_BYTES = Q_BYTES + 2 * KC_BYTES;
    static constexpr uint32_t IDESC = idesc_bf16(kRows, 64, 0, 0);
};

template <int DS>
__global__ void __launch_bounds__(192, 1)
select_proj_kernel(const __grid_constant__ CUtensorMap mapQt, const __grid_constant__ CUtensorMap mapKt, SelParams p) {
    using Cfg = SelProjCfg<DS>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    __shared__ uint64_t q_full, kc_full[2], kc_empty[2], s_full[2], s_free[2], drain_bar;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag;

    const uint32_t warp = warp_id(), lane = lane_id();
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + ((1024u - (raw & 1023u)) & 1023u);
    uint8_t* q_s = smem;
    uint8_t* kc_s = smem + Cfg::Q_BYTES;
    float* ts = reinterpret_cast<float*>(smem + Cfg::TILE_BYTES);
    int* tm = reinterpret_cast<int*>(ts + p.topk * kRows);
    uint32_t* bitmap = reinterpret_cast<uint32_t*>(tm + p.topk * kRows);

    const int t = p.T - 1 - static_cast<int>(blockIdx.x);
    const int bh = blockIdx.y;
    const int diag = 2 * t;
    const int nb = min(2 * t + 1, p.F);          // blocks scored for this tile
    const int nchunks = (nb + 63) >> 6;

    const int nwords = (p.C + 31) >> 5;
    for (int w = threadIdx.x; w < nwords; w += blockDim.x) bitmap[w] = 0u;
    if (threadIdx.x == 0) {
        mbar_init(&q_full, 1);
        for (int b = 0; b < 2; ++b) {
            mbar_init(&kc_full[b], 1);
            mbar_init(&kc_empty[b], 1);
            mbar_init(&s_full[b], 1);
            mbar_init(&s_free[b], 128);
        }
        mbar_init(&drain_bar, 1);
        abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc(&tmem_base_sh, 128);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = tmem_base_sh;
    const WaitCtl wc{&abort_flag, p.status, p.limit};

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer
        if (nchunks > 0) {
            tma_prefetch_desc(&mapQt);
            tma_prefetch_desc(&mapKt);
            mbar_arrive_expect_tx(&q_full, Cfg::Q_BYTES);
#pragma unroll
            for (int a = 0; a < DS / 64; ++a)
                tma_load_3d(q_s + a * (kRows * 128), &mapQt, &q_full, a * 64, t * kRows, bh);
            int issued = 0;
            bool ok = true;
            for (int c = 0; c < nchunks; ++c) {
                const int b = c & 1;
                if (!mbar_wait(&kc_empty[b], ((c >> 1) & 1) ^ 1u, wc)) { ok = false; break; }
                mbar_arrive_expect_tx(&kc_full[b], Cfg::KC_BYTES);
#pragma unroll
                for (int a = 0; a < DS / 64; ++a)
                    tma_load_3d(kc_s + b * Cfg::KC_BYTES + a * (64 * 128), &mapKt, &kc_full[b], a * 64, c * 64, bh);
                ++issued;
            }
            if (!ok) {
                mbar_wait_drain(&q_full, 0, p.limit, p.status);
                for (int q = issued - 1; q >= 0 && q >= issued - 2; --q)
                    mbar_wait_drain(&kc_full[q & 1], (q >> 1) & 1, p.limit, p.status);
            }
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer: S[c&1] = Qt (128 x DS) * Kt_chunk (64 x DS)^T
        if (nchunks > 0 && mbar_wait(&q_full, 0, wc)) {
            const uint32_t q_addr = smem_u32(q_s);
            for (int c = 0; c < nchunks; ++c) {
                const int b = c & 1;
                const uint32_t ph = (c >> 1) & 1;
                if (!mbar_wait(&kc_full[b], ph, wc)) break;
                if (!mbar_wait(&s_free[b], ph ^ 1u, wc)) break;
                tc_fence_after();
                const uint32_t k_addr = smem_u32(kc_s + b * Cfg::KC_BYTES);
#pragma unroll
                for (int k = 0; k < DS / 16; ++k) {
                    const uint32_t off_q = (k >> 2) * (kRows * 128) + (k & 3) * 32;
                    const uint32_t off_k = (k >> 2) * (64 * 128) + (k & 3) * 32;
                    umma_bf16(tmem_base + b * 64, smem_desc_sw128(q_addr + off_q, 16, 1024),
                              smem_desc_sw128(k_addr + off_k, 16, 1024), Cfg::IDESC, k > 0);
                }
                umma_commit(&s_full[b]);
                umma_commit(&kc_empty[b]);
            }
        }
        umma_commit(&drain_bar);
        mbar_wait_drain(&drain_bar, 0, p.limit, p.status);
    } else if (warp >= 2) {
        // ---------------- row threads
        const int q = warp & 3;
        const int r = q * 32 + lane;
        const int i = t * kRows + r;
        const bool valid = i < p.N;
        const int Ci = valid ? (i >> 6) : 0;
        RowSel rs{-CUDART_INF_F, 0.f, ts + r, tm + r, p.topk, 0, 0.f, 0, 0};
        const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
        for (int c = 0; c < nchunks; ++c) {
            const int b = c & 1;
            if (!mbar_wait_warp(&s_full[b], (c >> 1) & 1, wc)) break;
            tc_fence_after();
            uint32_t u0[32], u1[32];
            tmem_ld32(lane_addr + b * 64, u0);
            tmem_ld32(lane_addr + b * 64 + 32, u1);
            tmem_wait_ld();
            tc_fence_before();
            mbar_arrive(&s_free[b]);
            float v[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(u0[j]) * p.score_scale;
            row_consume32(rs, v, c * 64, Ci);
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(u1[j]) * p.score_scale;
            row_consume32(rs, v, c * 64 + 32, Ci);
        }
        if (valid && !abort_flag) row_finish(rs, p, static_cast<long long>(bh) * p.N + i, Ci, diag, bitmap);
        named_bar_sync(1, 128);
        if (warp == 2)
            compact_union(bitmap, diag, p.union_idx + (static_cast<long long>(bh) * p.T + t) * p.C,
                          p.union_cnt + static_cast<long long>(bh) * p.T + t);
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, 128);
    }
}

template <int DS>
cudaError_t launch_proj(const SelectArgs& a, const SelParams& p, size_t extra, const KernelEnv& env,
                        const char** err) {
    using Cfg = SelProjCfg<DS>;
    const size_t smem = 1024 + Cfg::TILE_BYTES + extra;
    if (smem > 227 * 1024) { *err = "selection: top-K too large for shared memory"; return cudaErrorInvalidValue; }
    cudaError_t e = cudaFuncSetAttribute(select_proj_kernel<DS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) { *err = "cudaFuncSetAttribute(select)"; return e; }
    CUtensorMap mq, mk;
    if (make_tmap_bf16_3d(&mq, a.Qt, DS, a.N, a.BH, 64, kRows) != 0) { *err = "tensor map Qt"; return cudaErrorInvalidValue; }
    if (make_tmap_bf16_3d(&mk, a.Kt, DS, a.F > 0 ? a.F : 1, a.BH, 64, 64) != 0) { *err = "tensor map Kt"; return cudaErrorInvalidValue; }
    dim3 grid(a.T, a.BH);
    select_proj_kernel<DS><<<grid, 192, smem, env.stream>>>(mq, mk, p);
    e = cudaGetLastError();
    if (e != cudaSuccess) *err = "select launch";
    return e;
}

}  // namespace

cudaError_t launch_select(const SelectArgs& a, const KernelEnv& env, const char** err) {
    SelParams p;
    p.N = a.N; p.C = a.C; p.T = a.T; p.F = a.F; p.topk = a.topk;
    p.score_scale = a.score_scale;
    p.scores = a.scores;
    p.sel_idx = a.sel_idx; p.sel_logg = a.sel_logg;
    p.union_idx = a.union_idx; p.union_cnt = a.union_cnt;
    p.status = env.status; p.limit = env.limit;
    const size_t extra = static_cast<size_t>(a.topk) * kRows * 8 + static_cast<size_t>((a.C + 31) / 32) * 4;
    if (a.scores != nullptr) {
        if (extra > 180 * 1024) { *err = "selection: top-K too large for shared memory"; return cudaErrorInvalidValue; }
        cudaError_t e = cudaFuncSetAttribute(select_given_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(extra));
        if (e != cudaSuccess) { *err = "cudaFuncSetAttribute(select_given)"; return e; }
        dim3 grid(a.T, a.BH);
        select_given_kernel<<<grid, 128, extra, env.stream>>>(p);
        e = cudaGetLastError();
        if (e != cudaSuccess) *err = "select launch";
        return e;
    }
    if (a.d_sel == 128) return launch_proj<128>(a, p, extra, env, err);
    if (a.d_sel == 64) return launch_proj<64>(a, p, extra, env, err);
    *err = "selection: unsupported d_sel";
    return cudaErrorInvalidValue;
}

}  // namespace sas
