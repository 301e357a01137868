// a2-a4: selector scores, causal log-gates and exact Top-K block selection.
//
// For query row i (block c_i = floor(i/64), C_i = c_i historical blocks):
//   LSE_i      = log sum_{m < C_i} exp(s_im)                  (Eq. normalized_log_gate)
//   I_i        = the K largest s_im, ties to the lower index   (Eq. selected_context)
//   sel_idx_i  = I_i in ascending order, -1 padded
//   sel_logg_i = s_im - LSE_i for m in I_i                      (log g of the kept blocks)
// (with the ablation activations of Sec. 4.2 instead: log sigmoid(s_im), or s_im itself)
// and for each 128-row tile t the sorted union of kept blocks below the tile's
// two diagonal blocks (m < 2t): the list of historical key blocks the
// attention kernel visits for that tile (Alg. 3 skips the others).
//
// Selection compares the fp32 scores directly (Alg. 2 selects on s; the
// order is the same as on g because log g = s - LSE), so the Top-K decision
// never depends on how LSE was rounded.
//
// One CTA owns one (batch*head, 128-row tile); one thread owns one row and
// keeps its running max/sum and its Top-K candidates (registers for K <= 32,
// a shared-memory column otherwise) with replace-the-worst updates.  Under
// GQA the "head" is a KV group: its G query heads share the selection
// (Sec. 5.3).  Packed sequences: a tile table (varlen_tiles_kernel) gives each
// CTA its tile's first row, tile index within its sequence and sequence
// length, so blocks and causality restart at every sequence.
//
// Two score sources:
//   * scores given: 32x32 score sub-tiles are staged through shared memory
//     with coalesced 128-byte row loads;
//   * learned selector: on the tensor cores, one thread first projects the
//     tile's 128 queries (q~ = Q Wq^T into TMEM; under GQA q~ = Wq_g [q_0; ...;
//     q_{G-1}], accumulated over G rounds of one head each); the row threads round q~
//     to bf16 in TMEM, where it is the A operand of the score product; then
//     s = q~ Kt^T / sqrt(d_sel) runs chunk by chunk (M=128, N=64) over
//     64-block chunks of projected summaries in a double-buffered TMA ring,
//     and the row threads read their scores back with tcgen05.ld.
#include <math_constants.h>

#include "internal.h"
#include "ptx.cuh"

namespace sas {
namespace {

constexpr int kRows = 128;
constexpr float kLog2e = 1.4426950408889634f;

struct SelParams {
    int BH, N, C, T, F, topk;
    int gate_act;                 // 0 softmax, 1 sigmoid, 2 logit (see staged_gate)
    float score_scale;
    const float* scores;
    int32_t* sel_idx;
    float* sel_logg;
    int32_t* union_idx;
    int32_t* union_cnt;
    const int4* tiles;            // packed sequences: {first row, local tile, sequence length} per tile slot
    const int* ntiles;            // their number (device); both null for [B, H, N] inputs
    int* status;
    long long limit;
    float* full_lse;              // full training scope (see SelectArgs)
    float* full_table;
    const float* noise;           // full*: added to every score before gate and Top-K
};

// Where a CTA's 128-row tile lies: its union-list slot, its tile index within
// its sequence, the sequence's first row in the head's token axis and the
// sequence length.  [B, H, N] inputs: one sequence of N rows per head.
struct TileGeo {
    int slot, t, base, n;
    int seq;   // the sequence's index (packed sequences; 0 otherwise)
};

// One CTA per (head, 128-row tile) on a 1-D grid: the tile index falls with
// the block index and the head varies fastest, so the tiles with the longest
// histories of every head are dispatched first and the light ones fill the tail.
__device__ __forceinline__ int tile_of_block(int T, int BH) { return T - 1 - static_cast<int>(blockIdx.x / BH); }
__device__ __forceinline__ int head_of_block(int BH) { return static_cast<int>(blockIdx.x % BH); }
// Packed sequences: the tile table is already ordered longest history first.
__device__ __forceinline__ TileGeo tile_geo(const SelParams& p) {
    if (p.tiles == nullptr) {
        const int t = tile_of_block(p.T, p.BH);
        return {t, t, 0, p.N, 0};
    }
    const int g = static_cast<int>(blockIdx.x / p.BH);
    const int4 v = __ldg(p.tiles + g);
    return {g, v.y, v.x, v.z, v.w};
}

// Online log-sum-exp of a row's scores.
struct RowLse {
    float mx, sum;
};

__device__ __forceinline__ void lse_update(RowLse& l, const float (&v)[32], int lim) {
    float cm = -CUDART_INF_F;
#pragma unroll
    for (int j = 0; j < 32; ++j)
        if (j < lim) cm = fmaxf(cm, v[j]);
    const float nm = fmaxf(l.mx, cm);
    float acc = 0.f;
#pragma unroll
    for (int j = 0; j < 32; ++j)
        if (j < lim) acc += fast_exp2((v[j] - nm) * kLog2e);
    l.sum = l.sum * fast_exp2((l.mx - nm) * kLog2e) + acc;
    l.mx = nm;
}

// ---- Top-K for K <= 32: the kept (score, block) pairs live in registers.
// Slot e holds block e while the row's first K blocks stream in, so a row
// with C_i <= K never reorders anything.  Later blocks replace the current
// worst entry (lowest score; among equal scores the highest block) when
// strictly better: a later block with an equal score ranks below every kept
// one because ties go to the lower block.  The work grows with the number of
// replacements (about K ln(C_i / K) for scores in random order), not with C_i.
// Block indices are kept as floats (exact: the C ABI caps N at 2^30 tokens, so
// blocks stay below 2^24); the worst entry is found with two shallow reduction
// trees (minimum score, then the highest block among the slots at that score)
// instead of a serial scan, and replaced by its block index, which is unique.
struct RegTopK {
    float s[32];
    float mf[32];   // block index; slots at or past K hold +inf / kEmptyBlock
    float ws;       // worst kept score
    float wmf;      // its block
    bool replaced;
};

constexpr float kEmptyBlock = 1073741824.f;   // 2^30: above every block index, sorts last

__device__ __forceinline__ void reg_init(RegTopK& t) {
    t.replaced = false;
    t.ws = -CUDART_INF_F;
    t.wmf = 0.f;
}

__device__ __forceinline__ void reg_rescan(RegTopK& t) {
    // minimum score: 3-input min tree (slots past K hold +inf and never win)
    float a[11];
#pragma unroll
    for (int g = 0; g < 10; ++g) a[g] = min3f(t.s[3 * g], t.s[3 * g + 1], t.s[3 * g + 2]);
    a[10] = fminf(t.s[30], t.s[31]);
    const float b0 = min3f(a[0], a[1], a[2]), b1 = min3f(a[3], a[4], a[5]);
    const float b2 = min3f(a[6], a[7], a[8]), b3 = fminf(a[9], a[10]);
    const float ws = fminf(min3f(b0, b1, b2), b3);
    // the highest block among the slots holding that score
    float c[11];
#pragma unroll
    for (int g = 0; g < 10; ++g)
        c[g] = max3f(t.s[3 * g] == ws ? t.mf[3 * g] : -1.f, t.s[3 * g + 1] == ws ? t.mf[3 * g + 1] : -1.f,
                     t.s[3 * g + 2] == ws ? t.mf[3 * g + 2] : -1.f);
    c[10] = fmaxf(t.s[30] == ws ? t.mf[30] : -1.f, t.s[31] == ws ? t.mf[31] : -1.f);
    const float d0 = max3f(c[0], c[1], c[2]), d1 = max3f(c[3], c[4], c[5]);
    const float d2 = max3f(c[6], c[7], c[8]), d3 = fmaxf(c[9], c[10]);
    t.ws = ws;
    t.wmf = fmaxf(max3f(d0, d1, d2), d3);
}

__device__ __forceinline__ void reg_offer(RegTopK& t, float x, int idx) {
    if (x > t.ws) {
        const float xf = static_cast<float>(idx);
#pragma unroll
        for (int e = 0; e < 32; ++e) {
            const bool hit = t.mf[e] == t.wmf;
            t.s[e] = hit ? x : t.s[e];
            t.mf[e] = hit ? xf : t.mf[e];
        }
        t.replaced = true;
        reg_rescan(t);
    }
}

// Positions j (within a 32-block chunk) whose score beats `thr`; j < lim only.
__device__ __forceinline__ uint32_t beats_mask(const float (&v)[32], int lo, int lim, float thr) {
    uint32_t mask = 0;
#pragma unroll
    for (int j = 0; j < 32; ++j)
        if (j >= lo && j < lim && v[j] > thr) mask |= 1u << j;
    return mask;
}

// Consumes the scores of blocks 32c .. 32c+31 (entries at or past C_i ignored).
// v holds them in registers; col[j * stride] holds the same values in shared
// memory, read only for the few positions that can enter the Top-K.
__device__ __forceinline__ void reg_consume(RegTopK& t, RowLse& l, const float (&v)[32], const float* col,
                                            int stride, int c, int Ci, int K) {
    const int lim = Ci - 32 * c;
    if (lim <= 0) return;
    lse_update(l, v, lim);
    if (K == 0) return;
    int lo = 0;
    if (c == 0) {
        const int nf = min(K, lim);
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            // unused slots carry the largest block index so that sorting sinks them
            t.s[j] = j < nf ? v[j] : CUDART_INF_F;
            t.mf[j] = j < nf ? static_cast<float>(j) : kEmptyBlock;
        }
        if (Ci <= K) return;
        reg_rescan(t);
        lo = K;
    }
    // The threshold only rises while the chunk is consumed, so this mask is a
    // superset of the entries that will actually replace one.
    uint32_t mask = beats_mask(v, lo, lim, t.ws);
    while (mask) {
        const int j = __ffs(mask) - 1;
        mask &= mask - 1;
        reg_offer(t, col[j * stride], 32 * c + j);
    }
}

// Sorts the kept entries by block index (bitonic network; empty slots carry
// the largest index and sink to the end).
__device__ __forceinline__ void reg_sort_by_block(RegTopK& t) {
#pragma unroll
    for (int k = 2; k <= 32; k <<= 1) {
#pragma unroll
        for (int j = k >> 1; j > 0; j >>= 1) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                const int l = i ^ j;
                if (l > i) {
                    const bool up = (i & k) == 0;
                    const bool sw = up ? (t.mf[i] > t.mf[l]) : (t.mf[i] < t.mf[l]);
                    const float si = t.s[i], sl = t.s[l];
                    const float mi = t.mf[i], ml = t.mf[l];
                    t.s[i] = sw ? sl : si;
                    t.s[l] = sw ? si : sl;
                    t.mf[i] = sw ? ml : mi;
                    t.mf[l] = sw ? mi : ml;
                }
            }
        }
    }
}

// ---- Top-K for 32 < K <= 128: the kept pairs live in a shared-memory column
// of this row (element e at offset e * kRows, so a warp's rows use distinct
// banks), with the same fill / replace rule.
struct SmemTopK {
    float* s;
    int* m;
    float ws;
    int wm, wpos;
    bool replaced;
};

__device__ __forceinline__ void smem_rescan(SmemTopK& t, int K) {
    float ws = CUDART_INF_F;
    int wm = -1, wp = 0;
#pragma unroll 8
    for (int e = 0; e < K; ++e) {
        const float se = t.s[e * kRows];
        const int me = t.m[e * kRows];
        if (se < ws || (se == ws && me > wm)) {
            ws = se;
            wm = me;
            wp = e;
        }
    }
    t.ws = ws;
    t.wm = wm;
    t.wpos = wp;
}

__device__ __forceinline__ void smem_consume(SmemTopK& t, RowLse& l, const float (&v)[32], const float* col,
                                             int stride, int c, int Ci, int K) {
    const int lim = Ci - 32 * c;
    if (lim <= 0) return;
    lse_update(l, v, lim);
    const int m0 = 32 * c;
    // fill: the row's first K blocks take slots 0 .. K-1 in order (at most
    // the 32 blocks of this chunk)
    const int nfill = min(min(lim, 32), K - m0);
    for (int j = 0; j < nfill; ++j) {
        t.s[(m0 + j) * kRows] = col[j * stride];
        t.m[(m0 + j) * kRows] = m0 + j;
    }
    if (Ci <= K || m0 + 32 <= K - 1) return;
    int lo = 0;
    if (m0 < K) {
        smem_rescan(t, K);
        lo = K - m0;
    }
    uint32_t mask = beats_mask(v, lo, lim, t.ws);
    while (mask) {
        const int j = __ffs(mask) - 1;
        mask &= mask - 1;
        const float x = col[j * stride];
        if (x > t.ws) {
            t.s[t.wpos * kRows] = x;
            t.m[t.wpos * kRows] = m0 + j;
            t.replaced = true;
            smem_rescan(t, K);
        }
    }
}

__device__ __forceinline__ void smem_sort_by_block(SmemTopK& t, int n) {
    for (int a = 1; a < n; ++a) {
        const int km = t.m[a * kRows];
        const float ks = t.s[a * kRows];
        int b = a - 1;
        while (b >= 0 && t.m[b * kRows] > km) {
            t.m[(b + 1) * kRows] = t.m[b * kRows];
            t.s[(b + 1) * kRows] = t.s[b * kRows];
            --b;
        }
        t.m[(b + 1) * kRows] = km;
        t.s[(b + 1) * kRows] = ks;
    }
}

// log g of a kept block from its score (Eq. general_gate with the activation of
// Sec. 4.2): softmax s - LSE; logit s; sigmoid log(1/(1+e^-s)).  The row pass
// stages s - LSE (softmax) or s (the others); copy_out turns a staged s into
// log sigmoid(s), off the per-row path.
__device__ __forceinline__ float staged_gate(float s, float lse, int act) {
    return act == 0 ? s - lse : s;
}

__device__ __forceinline__ float log_sigmoid(float s) {
    return -(fmaxf(-s, 0.f) + log1pf(expf(-fabsf(s))));
}

// Output staging: each row's K entries are written to shared memory and then
// copied to global memory with coalesced stores.  Entry e of row r sits at
// r * stride + e * es: row-major with a row stride of K + 1 words (scores
// given) or entry-major (learned selector); either way a warp's rows hit
// distinct banks.
struct Staging {
    int32_t* idx;
    float* lg;
    int stride;
    int es;
};

__device__ __forceinline__ void stage_entry(const Staging& st, int r, int e, int m, float lg) {
    st.idx[r * st.stride + e * st.es] = m;
    st.lg[r * st.stride + e * st.es] = lg;
}

// Copies the staged rows (the tile's first `rows`, from row `row0` of the
// head's token axis) to sel_idx / sel_logg.  Consecutive threads take
// consecutive entries of a row, so stores coalesce.
__device__ __forceinline__ void copy_out(const Staging& st, const SelParams& p, int bh, long long row0, int rows,
                                         int tid, int nthreads) {
    const int K = p.topk;
    if (K == 0) return;
    const long long base = (static_cast<long long>(bh) * p.N + row0) * K;
    int r = tid / K, e = tid - r * K;
    const int dr = nthreads / K, de = nthreads - dr * K;
    const bool sigm = p.gate_act == 1;
    for (int q = tid; q < rows * K; q += nthreads) {
        const int m = st.idx[r * st.stride + e * st.es];
        const float lg = st.lg[r * st.stride + e * st.es];
        p.sel_idx[base + q] = m;
        p.sel_logg[base + q] = (sigm && m >= 0) ? log_sigmoid(lg) : lg;
        r += dr;
        e += de;
        if (e >= K) {
            e -= K;
            ++r;
        }
    }
}

// Finishes one row: log-gates, ascending order, staging, tile-union bits.
template <class TK>
__device__ __forceinline__ void row_emit(TK& t, const RowLse& l, const Staging& st, int r, int Ci, int K, int diag,
                                         uint32_t* bitmap, int act);

template <>
__device__ __forceinline__ void row_emit<RegTopK>(RegTopK& t, const RowLse& l, const Staging& st, int r, int Ci,
                                                  int K, int diag, uint32_t* bitmap, int act) {
    const int n = min(K, Ci);
    const float lse = Ci > 0 ? l.mx + logf(l.sum) : 0.f;
    if (t.replaced) reg_sort_by_block(t);
#pragma unroll
    for (int e = 0; e < 32; ++e) {
        if (e < K) {
            const bool kept = e < n;
            const int m = static_cast<int>(t.mf[e]);
            stage_entry(st, r, e, kept ? m : -1, kept ? staged_gate(t.s[e], lse, act) : 0.f);
            if (kept && static_cast<unsigned>(m) < static_cast<unsigned>(diag))
                atomicOr(&bitmap[m >> 5], 1u << (m & 31));
        }
    }
}

template <>
__device__ __forceinline__ void row_emit<SmemTopK>(SmemTopK& t, const RowLse& l, const Staging& st, int r, int Ci,
                                                   int K, int diag, uint32_t* bitmap, int act) {
    const int n = min(K, Ci);
    const float lse = Ci > 0 ? l.mx + logf(l.sum) : 0.f;
    if (t.replaced) smem_sort_by_block(t, n);
    for (int e = 0; e < K; ++e) {
        if (e < n) {
            const int m = t.m[e * kRows];
            stage_entry(st, r, e, m, staged_gate(t.s[e * kRows], lse, act));
            if (static_cast<unsigned>(m) < static_cast<unsigned>(diag)) atomicOr(&bitmap[m >> 5], 1u << (m & 31));
        } else {
            stage_entry(st, r, e, -1, 0.f);
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

// One warp turns a byte map of the tile's kept blocks (< diag) into a sorted list.
__device__ __forceinline__ void compact_union_bytes(const uint8_t* map, int diag, int32_t* out, int32_t* out_cnt) {
    const int lane = threadIdx.x & 31;
    int base = 0;
    for (int m0 = 0; m0 < diag; m0 += 32) {
        const int m = m0 + lane;
        const bool set = m < diag && map[m] != 0;
        const uint32_t bal = __ballot_sync(0xffffffffu, set);
        if (set) out[base + __popc(bal & ((1u << lane) - 1u))] = m;
        base += __popc(bal);
    }
    if (lane == 0) *out_cnt = base;
}

// Shared-memory plan of the per-row state and outputs (bytes).
__host__ __device__ constexpr size_t smem_topk_bytes(int K) { return K > 32 ? size_t(K) * kRows * 8 : 0; }
__host__ __device__ constexpr size_t staging_bytes(int K) { return size_t(kRows) * (K + 1) * 8; }
__host__ __device__ constexpr size_t bitmap_bytes(int C) { return size_t((C + 31) / 32) * 4; }

// ------------------------------------------------------------ scores given

template <bool REG, bool NOISE>
__global__ void __launch_bounds__(128, 3) select_given_kernel(SelParams p) {
    extern __shared__ __align__(16) uint8_t dsm[];
    __shared__ float stage[4][32][33];

    if (p.tiles != nullptr && static_cast<int>(blockIdx.x / p.BH) >= __ldg(p.ntiles)) return;   // spare slot
    const TileGeo geo = tile_geo(p);
    const int t = geo.t;
    const int bh = head_of_block(p.BH);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int r = threadIdx.x;
    const int i = t * kRows + r;            // row within its sequence
    const bool valid = i < geo.n;
    const int Ci = valid ? (i >> 6) : 0;
    const int diag = 2 * t;
    const int K = p.topk;

    uint8_t* ptr = dsm;
    SmemTopK stk{};
    if constexpr (!REG) {
        stk.s = reinterpret_cast<float*>(ptr) + r;
        stk.m = reinterpret_cast<int*>(ptr + size_t(K) * kRows * 4) + r;
        stk.ws = -CUDART_INF_F;
        ptr += smem_topk_bytes(K);
    }
    const Staging st{reinterpret_cast<int32_t*>(ptr), reinterpret_cast<float*>(ptr + size_t(kRows) * (K + 1) * 4),
                     K + 1, 1};
    ptr += staging_bytes(K);
    uint32_t* bitmap = reinterpret_cast<uint32_t*>(ptr);
    const int nwords = (p.C + 31) >> 5;
    for (int w = threadIdx.x; w < nwords; w += blockDim.x) bitmap[w] = 0u;
    __syncthreads();

    RegTopK rtk;
    reg_init(rtk);
    RowLse lse{-CUDART_INF_F, 0.f};

    const int row0 = t * kRows + warp * 32;
    const int last = min(row0 + 31, geo.n - 1);
    const int Cw = row0 < geo.n ? (last >> 6) : 0;   // largest C_i among the warp's rows
    const float* sbase = p.scores + (static_cast<long long>(bh) * p.N + geo.base) * p.C;
    const float* nbase = NOISE ? p.noise + (static_cast<long long>(bh) * p.N + geo.base) * p.C : nullptr;
    for (int c = 0; 32 * c < Cw; ++c) {
        const int m = 32 * c + lane;
        // block m of the warp's 32 rows: all loads issued before the first is used
        float w[32];
#pragma unroll
        for (int rho = 0; rho < 32; ++rho) {
            const int row = row0 + rho;
            w[rho] = (row < geo.n && m < p.C) ? __ldg(sbase + static_cast<long long>(row) * p.C + m) : 0.f;
        }
        if constexpr (NOISE) {
#pragma unroll
            for (int rho = 0; rho < 32; ++rho) {
                const int row = row0 + rho;
                if (row < geo.n && m < p.C)   // full*: s~ = s + eps in fp32
                    w[rho] = __fadd_rn(w[rho], __ldg(nbase + static_cast<long long>(row) * p.C + m));
            }
        }
#pragma unroll
        for (int rho = 0; rho < 32; ++rho) stage[warp][lane][rho] = w[rho];
        __syncwarp();
        float v[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            v[j] = stage[warp][j][lane] * p.score_scale;
            stage[warp][j][lane] = v[j];
        }
        const float* col = &stage[warp][0][lane];
        if constexpr (REG) reg_consume(rtk, lse, v, col, 33, c, Ci, K);
        else smem_consume(stk, lse, v, col, 33, c, Ci, K);
        __syncwarp();
    }
    if (valid) {
        if constexpr (REG) row_emit(rtk, lse, st, r, Ci, K, diag, bitmap, p.gate_act);
        else row_emit(stk, lse, st, r, Ci, K, diag, bitmap, p.gate_act);
    }
    __syncthreads();
    copy_out(st, p, bh, static_cast<long long>(geo.base) + t * kRows, min(kRows, geo.n - t * kRows), threadIdx.x,
             128);
    if (warp == 0)
        compact_union(bitmap, diag, p.union_idx + (static_cast<long long>(bh) * p.T + geo.slot) * p.C,
                      p.union_cnt + static_cast<long long>(bh) * p.T + geo.slot);
}

// --------------------------------------------------------- learned selector

// The learned-selector kernel keeps the projected queries q~ in TMEM, rounded
// to bf16, as the A operand of the score products; its shared-memory plan is
// under SelProjCfg.  A CTA needs 128 TMEM columns and (K <= 36) about 72 KB of
// shared memory, so three CTAs (twelve row warps) share an SM.
//
// Top-K without per-row replacement.  Replacing the worst kept entry whenever a
// better score arrives diverges across the 32 rows of a warp (each row
// replaces at different times, so the warp pays for every row's replacements),
// so the score chunks are streamed several times instead, with uniform work
// per score (the score products are cheap to re-issue):
//   pass A: the row's log-sum-exp, maximum, minimum and the first two moments
//           of its scores;
//   pass B: a histogram of the scores above a low threshold lo in kBins bins
//           of width (hi - lo) / (kBins - 1), the last one open above (lo and
//           hi placed from the moments where about K + 5 sqrt(K) and K -
//           5 sqrt(K) scores of a normal sample lie above them); it locates
//           the bin holding the K-th largest score;
//   pass C: every score in that bin or above is appended to the row's list in
//           block order; afterwards the best R = K - (number above the bin)
//           of the boundary bin's scores, by (score descending, block
//           ascending), stay and the list is compacted in place;
//   pass D: only if some row of the tile could not use A-C (its scores are
//           too concentrated for the bins: equal scores, a crowded boundary bin):
//           that row runs replace-the-worst over all its scores.
// Every pass places a score in its bin with the same rounded operations (no
// contraction), so the passes agree on every score.
constexpr int kBins = 44;                           // histogram bins per row (pass B)
constexpr int kBoundaryMax = 12;                    // boundary-bin scores a row's list holds beyond K
constexpr size_t kHistBytes = size_t(kBins) * kRows * 4;
// Bin arithmetic: v = 2^23 + (u - lo) / w, rounded to an integer by the add
// itself (the float spacing at 2^23 is 1), holds the bin in the low bits of
// its representation, so the bin's shared-memory word follows from the bits
// of v with one integer multiply-add.
constexpr float kBinMagic = 8388608.f;
constexpr uint32_t kBinMagicBits = 0x4B000000u;
constexpr float kBinTop = kBinMagic + float(kBins - 1);

constexpr int kChunk = 32;                          // blocks per score chunk (one TMEM buffer, one MMA)
constexpr int kRing = 3;                            // summary-chunk stages in shared memory
constexpr int kListSmall = kBins;                   // list capacity when K + kBoundaryMax fits the histogram words
constexpr int kListBig = 64 + kBoundaryMax;         // list capacity for larger K
// Row stride (words) of the lists and histograms: row-major with an odd stride,
// so that a warp's 32 rows fall in 32 different banks and a row's entries are
// consecutive words (the copy-out reads them in order).
__host__ __device__ constexpr int list_stride(int cap) { return (cap + 1) | 1; }

// Shared-memory plan (bytes from the 1024-aligned base):
//   [0, LIST): the rows' list blocks (row r at word r * STRIDE); before that
//              the histograms (bin b of row r at word r * STRIDE + b), and
//              during the projection a 64-column half of the Q tile;
//   [LIST, 2 LIST): the rows' list products;
//   ring: the summary-chunk stages, during the projection a 64-column slice of Wq;
//   then the tile's union map (one byte per block).
template <int D, int DS, bool BIGK>
struct SelProjCfg {
    static constexpr int CAP = BIGK ? kListBig : kListSmall;   // list entries per row
    static constexpr int STRIDE = list_stride(CAP);            // words between rows (odd)
    static constexpr int LIST_BYTES = STRIDE * kRows * 4;      // one of the two list arrays
    static constexpr int QH_BYTES = kRows * 64 * 2;            // a 64-column half of the Q tile
    static constexpr int WQH_BYTES = DS * 64 * 2;              // a 64-column slice of Wq
    static constexpr int KC_BYTES = kChunk * DS * 2;           // one chunk of projected summaries
    static constexpr int RING_BYTES = kRing * KC_BYTES > WQH_BYTES ? kRing * KC_BYTES : WQH_BYTES;
    static constexpr int OFF_LG = LIST_BYTES;
    static constexpr int OFF_RING = 2 * LIST_BYTES;
    static constexpr int OFF_BITMAP = OFF_RING + RING_BYTES;
    static constexpr uint32_t IDESC_PROJ = idesc_bf16(kRows, DS, 0, 0);
    static constexpr uint32_t IDESC_S = idesc_bf16(kRows, kChunk, 0, 0);
    // TMEM (128 columns): q~ in fp32 at 0 .. DS-1 during the projection, then in
    // bf16 at 0 .. DS/2-1; the two score buffers at 64 and 96
    static constexpr int TMEM_S = 64;
    static_assert(STRIDE >= kBins && LIST_BYTES >= QH_BYTES, "histogram / Q half exceed the list");
    static_assert(DS <= 128 && D % 64 == 0 && DS % 64 == 0, "projection shape");
};

constexpr int kPassA = 0, kPassB = 1, kPassC = 2, kPassD = 3;
constexpr int kPassW = 4;   // full training scope: write every score to the table
constexpr int kRowAll = 0, kRowNormal = 1, kRowFail = 2;   // C_i <= K: keep all; thresholds; fallback

template <int D, int DS, bool BIGK>
__host__ __device__ constexpr size_t proj_smem_bytes(int C) {
    return size_t(SelProjCfg<D, DS, BIGK>::OFF_BITMAP) + ((C + 15) & ~15);
}

// Selection works on the raw products u = q~ . K~ (the scores are s = u / sqrt(d_sel),
// an order-preserving scale): thresholds, bins and ties are all on u, and s is
// formed only for the log-sum-exp and the emitted log-gates.
//
// The bin value of a product at or above lo (monotone in u; the top bin takes
// everything from about hi up).  Passes B and C form it with the packed
// operations, which round exactly like these scalar ones.
__device__ __forceinline__ float bin_v(float u, float neg_lo, float inv_w) {
    return fminf(__fmaf_rn(__fadd_rn(u, neg_lo), inv_w, kBinMagic), kBinTop);
}

// The per-row state carried across the passes.
struct RowSel {
    RowLse l;                   // pass A: running max of u, sum of exp(s - s_max)
    float v0;                   // pass A: shift (the row's first product)
    uint64_t s1, s2;            // pass A: packed sums of (u - v0) and (u - v0)^2
    float mn;                   // pass A: minimum
    float lo, inv_w;            // histogram origin and inverse bin width (lo = -inf: keep all, +inf: fallback)
    int mode;                   // kRowAll / kRowNormal / kRowFail
    float tb;                   // after B: bin value of the boundary bin (pass C takes v >= tb)
    int hi_bin, nabove;         // after B: first bin kept whole, products above the boundary bin
    int pos;                    // pass C / D: entries in the row's list
    float ws;                   // pass D: worst kept product, its slot
    int wpos;
};

// Shared-memory addresses of one row's list and histogram.
constexpr uint32_t kListStep = 4;   // bytes between a row's list entries
struct RowAddr {
    uint32_t list;              // the row's list entry 0 (int32 block; its fp32 product OFF_LG bytes on); entry e at + e * kListStep
    uint32_t hist_off;          // the row's histogram word of bin b at hist_off + bits(v) * 4 (mod 2^32)
};

// Pass D state of a row: entries staged, worst kept product and its slot.
struct FallbackState {
    int pos;
    float ws;
    int wpos;
};

// Pass D, one product: the row's first K' products fill its list, a later one
// replaces the worst kept entry (lowest product; among equal ones the highest
// block, which ranks last because ties go to the lower block) when strictly
// larger.  Kept out of line: the fallback is rare, and its loops inlined at every
// one of the 32 unrolled positions would crowd the hot passes out of the
// instruction cache.  Entry e of the row at idx[e * es], sc[e * es].
__device__ __noinline__ FallbackState fallback_offer(FallbackState f, float u, int m, int32_t* idx, float* sc,
                                                     int Kp, int es) {
    if (f.pos < Kp) {
        idx[f.pos * es] = m;
        sc[f.pos * es] = u;
        ++f.pos;
        if (f.pos < Kp) return f;
    } else if (u > f.ws) {
        idx[f.wpos * es] = m;
        sc[f.wpos * es] = u;
    } else {
        return f;
    }
    float ws = CUDART_INF_F;
    int wm = -1, wp = 0;
    for (int e = 0; e < Kp; ++e) {
        const float se = sc[e * es];
        const int me = idx[e * es];
        if (se < ws || (se == ws && me > wm)) {
            ws = se;
            wm = me;
            wp = e;
        }
    }
    f.ws = ws;
    f.wpos = wp;
    return f;
}

// Sorts a row's first n list entries by block index (insertion sort: rare
// fallback rows).
__device__ __forceinline__ void staged_sort_by_block(const Staging& st, int r, int n) {
    int32_t* idx = st.idx + r * st.stride;
    float* sc = st.lg + r * st.stride;
    const int es = st.es;
    for (int a = 1; a < n; ++a) {
        const int km = idx[a * es];
        const float ks = sc[a * es];
        int b = a - 1;
        while (b >= 0 && idx[b * es] > km) {
            idx[(b + 1) * es] = idx[b * es];
            sc[(b + 1) * es] = sc[b * es];
            --b;
        }
        idx[(b + 1) * es] = km;
        sc[(b + 1) * es] = ks;
    }
}

// One half-chunk (32 products of blocks m0 .. m0 + 31) of pass `kind` for one
// row.  FULL: all 32 are within the row's history (the common case, no
// per-entry range test); otherwise entries j >= lim = C_i - m0 are ignored.
// Passes B and C always run FULL: the caller turns the products past the
// history into NaN, which no comparison takes.
// c = scale * log2(e) (exp of s - s_max as exp2 of u c - u_max c).
template <bool FULL, uint32_t OFF_LG>
__device__ __forceinline__ void row_pass(RowSel& rs, int kind, const float* u, int m0, int lim, int Kp,
                                         const RowAddr& ra, const Staging& st, int r, float c) {
    if (kind == kPassA) {
        if (m0 == 0) rs.v0 = u[0];
        float cm = -CUDART_INF_F, mn = rs.mn;
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
            const bool in0 = FULL || j < lim, in1 = FULL || j + 1 < lim;
            cm = max3f(cm, in0 ? u[j] : -CUDART_INF_F, in1 ? u[j + 1] : -CUDART_INF_F);
            mn = min3f(mn, in0 ? u[j] : CUDART_INF_F, in1 ? u[j + 1] : CUDART_INF_F);
        }
        const float nm = fmaxf(rs.l.mx, cm);
        const float noff = -nm * c;
        const uint64_t c2 = f32x2(c, c), off2 = f32x2(noff, noff);
        const uint64_t nv0 = f32x2(-rs.v0, -rs.v0);
        uint64_t acc[2] = {0, 0};
        uint64_t s1 = rs.s1, s2 = rs.s2;
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
            const bool in0 = FULL || j < lim, in1 = FULL || j + 1 < lim;
            float a0, a1;
            f32x2_split(fma_f32x2(f32x2(u[j], u[j + 1]), c2, off2), a0, a1);
            const float e0 = in0 ? fast_exp2(a0) : 0.f, e1 = in1 ? fast_exp2(a1) : 0.f;
            acc[(j >> 1) & 1] = add_f32x2(acc[(j >> 1) & 1], f32x2(e0, e1));
            uint64_t x = add_f32x2(f32x2(u[j], u[j + 1]), nv0);
            if (!FULL) {
                float x0, x1;
                f32x2_split(x, x0, x1);
                x = f32x2(in0 ? x0 : 0.f, in1 ? x1 : 0.f);
            }
            s1 = add_f32x2(s1, x);
            s2 = fma_f32x2(x, x, s2);
        }
        float q0, q1, q2, q3;
        f32x2_split(acc[0], q0, q1);
        f32x2_split(acc[1], q2, q3);
        const float scale_old = rs.l.mx == -CUDART_INF_F ? 0.f : fast_exp2((rs.l.mx - nm) * c);
        rs.l.sum = rs.l.sum * scale_old + ((q0 + q1) + (q2 + q3));
        rs.l.mx = nm;
        rs.s1 = s1;
        rs.s2 = s2;
        rs.mn = mn;
    } else if (kind == kPassB) {
        const uint64_t nlo2 = f32x2(-rs.lo, -rs.lo), iw2 = f32x2(rs.inv_w, rs.inv_w);
        const uint64_t mg2 = f32x2(kBinMagic, kBinMagic);
        const float lo = rs.lo;
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
            float v0, v1;
            f32x2_split(fma_f32x2(add_f32x2(f32x2(u[j], u[j + 1]), nlo2), iw2, mg2), v0, v1);
            red_shared_inc_if_ge(u[j], lo, ra.hist_off + __float_as_uint(fminf(v0, kBinTop)) * 4u);
            red_shared_inc_if_ge(u[j + 1], lo, ra.hist_off + __float_as_uint(fminf(v1, kBinTop)) * 4u);
        }
    } else if (kind == kPassC) {
        // v >= tb needs no clamp (tb <= kBinTop) and no test of u >= lo: a product
        // below lo has v <= 2^23 < tb, as the boundary bin is at least bin 1
        // (bin 0 sends the row to the fallback), and for rows that keep every
        // score tb = -inf and v = +inf
        const uint64_t nlo2 = f32x2(-rs.lo, -rs.lo), iw2 = f32x2(rs.inv_w, rs.inv_w);
        const uint64_t mg2 = f32x2(kBinMagic, kBinMagic);
        const float tb = rs.tb;
        uint32_t addr = ra.list + static_cast<uint32_t>(rs.pos) * kListStep;
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
            float v0, v1;
            f32x2_split(fma_f32x2(add_f32x2(f32x2(u[j], u[j + 1]), nlo2), iw2, mg2), v0, v1);
            st_shared_split_if_ge<OFF_LG>(u[j], v0, tb, addr, static_cast<uint32_t>(m0 + j), kListStep);
            st_shared_split_if_ge<OFF_LG>(u[j + 1], v1, tb, addr, static_cast<uint32_t>(m0 + j + 1), kListStep);
        }
        rs.pos = static_cast<int>((addr - ra.list) / kListStep);
    } else {   // kPassD: replace-the-worst for the rows the bins could not resolve
        if (rs.mode != kRowFail) return;
        FallbackState f{rs.pos, rs.ws, rs.wpos};
        int32_t* idx = st.idx + r * st.stride;
        float* sc = st.lg + r * st.stride;
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (FULL || j < lim) f = fallback_offer(f, u[j], m0 + j, idx, sc, Kp, st.es);
        rs.pos = f.pos;
        rs.ws = f.ws;
        rs.wpos = f.wpos;
    }
}

__device__ __forceinline__ void row_set_all(RowSel& rs) {
    rs.mode = kRowAll;
    rs.lo = -CUDART_INF_F;
    rs.inv_w = 1.f;
    rs.tb = -CUDART_INF_F;   // pass C takes every score of the history
    rs.hi_bin = 0;
}
__device__ __forceinline__ void row_set_fail(RowSel& rs) {
    rs.mode = kRowFail;
    rs.lo = CUDART_INF_F;   // passes B and C take nothing from this row
    rs.tb = CUDART_INF_F;
    rs.hi_bin = kBins;
}

// After pass A: the histogram range of a row with more than K blocks.
__device__ __forceinline__ void row_after_a(RowSel& rs, int Ci, int K) {
    if (Ci <= K) {
        row_set_all(rs);
        return;
    }
    const float n = static_cast<float>(Ci);
    float a0, a1, b0, b1;
    f32x2_split(rs.s1, a0, a1);
    f32x2_split(rs.s2, b0, b1);
    const float mean = (a0 + a1) / n;
    const float var = fmaxf(fmaf(-mean, mean, (b0 + b1) / n), 0.f);
    const float sd = sqrtf(var);
    // a normal sample has a fraction P(Z > z) above mean + sd z; lo leaves about
    // K + 5 sqrt(K) products above it, hi about K - 5 sqrt(K) (at least half a one)
    const float kf = static_cast<float>(K), dk = 5.f * sqrtf(kf);
    const float p_lo = (kf + dk) / n, p_hi = fmaxf(kf - dk, 0.5f) / n;
    float lo = rs.mn, hi = rs.l.mx;
    if (p_lo < 1.f) lo = fmaxf(rs.mn, rs.v0 + mean + sd * 1.41421356f * erfinvf(1.f - 2.f * p_lo));
    if (p_hi < 1.f) hi = fminf(rs.l.mx, rs.v0 + mean + sd * 1.41421356f * erfinvf(1.f - 2.f * p_hi));
    const float span = hi - lo;
    const float inv_w = static_cast<float>(kBins - 1) / span;
    if (span > 0.f && isfinite(inv_w)) {
        rs.mode = kRowNormal;
        rs.lo = lo;
        rs.inv_w = inv_w;
        rs.tb = CUDART_INF_F;   // nothing is listed before pass B has placed the K-th product
        rs.hi_bin = kBins;
    } else {
        row_set_fail(rs);
    }
}

// After pass B: the bin holding the K-th largest product (scanning from the top).
// hist: the row's counters (bin b at hist[b]).
__device__ __forceinline__ void row_after_b(RowSel& rs, const uint32_t* hist, int Kp) {
    if (rs.mode != kRowNormal) return;
    int cum = 0, bstar = -1, nabove = 0, nb = 0;
#pragma unroll
    for (int b = kBins - 1; b >= 0; --b) {
        const int cb = static_cast<int>(hist[b]);
        if (bstar < 0 && cum + cb >= Kp) {
            bstar = b;
            nabove = cum;
            nb = cb;
        }
        cum += cb;
    }
    if (bstar <= 0) {
        // fewer than K' products above lo (the estimate was too high), or the
        // K-th in the lowest bin, which pass C cannot tell from just below lo
        row_set_fail(rs);
        return;
    }
    const bool take_all = nabove + nb == Kp;
    if (!take_all && nb > kBoundaryMax) {
        row_set_fail(rs);
        return;
    }
    rs.tb = kBinMagic + static_cast<float>(bstar);
    rs.hi_bin = take_all ? bstar : bstar + 1;
    rs.nabove = nabove;
}

// After pass C: the list holds, in block order, the nabove products above the
// boundary bin and (unless the bin is taken whole) the boundary bin's products.
// The best R = K' - nabove of the latter, by (product descending, block
// ascending), stay; the list is compacted in place.
__device__ __forceinline__ void row_after_c(RowSel& rs, const Staging& st, int r, int Kp) {
    if (rs.mode != kRowNormal || rs.pos <= Kp) return;
    int32_t* idx = st.idx + r * st.stride;
    float* sc = st.lg + r * st.stride;
    const int es = st.es;
    const int n = rs.pos;   // <= K' - 1 + kBoundaryMax < 128
    const int R = Kp - rs.nabove;
    const float nlo = -rs.lo, iw = rs.inv_w;
    const float tk = kBinMagic + static_cast<float>(rs.hi_bin);   // bins kept whole
    // bit a of (bl, bh): entry a is in the boundary bin; likewise the kept ones
    uint64_t bl = 0, bh = 0;
    for (int a = 0; a < n; ++a) {
        if (bin_v(sc[a * es], nlo, iw) < tk) {
            if (a < 64) bl |= 1ull << a;
            else bh |= 1ull << (a - 64);
        }
    }
    uint64_t kl = 0, kh = 0;
    for (int hx = 0; hx < 2; ++hx) {
        for (uint64_t mx = hx ? bh : bl; mx != 0; mx &= mx - 1) {
            const int x = hx * 64 + __ffsll(static_cast<long long>(mx)) - 1;
            const float ux = sc[x * es];
            int rank = 0;
            for (int hy = 0; hy < 2; ++hy)
                for (uint64_t my = hy ? bh : bl; my != 0; my &= my - 1) {
                    const int y = hy * 64 + __ffsll(static_cast<long long>(my)) - 1;
                    const float uy = sc[y * es];
                    rank += (uy > ux || (uy == ux && y < x)) ? 1 : 0;   // y < x: lower block
                }
            if (rank < R) {
                if (hx) kh |= 1ull << (x - 64);
                else kl |= 1ull << x;
            }
        }
    }
    int out = 0;
    for (int a = 0; a < n; ++a) {
        const uint64_t bw = a < 64 ? bl : bh, kw = a < 64 ? kl : kh;
        const int sh = a & 63;
        if (!((bw >> sh) & 1ull) || ((kw >> sh) & 1ull)) {
            idx[out * es] = idx[a * es];
            sc[out * es] = sc[a * es];
            ++out;
        }
    }
    rs.pos = out;
}

// Registers: three CTAs of 192 threads share an SM for K <= 36 (two above).  An
// SM sub-partition holds 16K registers and takes up to five of those 18 warps,
// so a thread may have 96.
template <int D, int DS, bool BIGK>
__global__ void __maxnreg__(BIGK ? 168 : 96)
select_proj_kernel(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapWq,
                   const __grid_constant__ CUtensorMap mapKt, SelParams p, int H, int G) {
    // H: KV heads (selection groups), G: query heads per group.  The gate query of
    // group bh is q~ = Wq[bh % H] [q_{bh G}; ...; q_{bh G + G - 1}]: rounds that
    // each stage a 64-column half of one head's Q tile and the matching columns
    // of Wq and accumulate.
    using Cfg = SelProjCfg<D, DS, BIGK>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    if (p.tiles != nullptr && static_cast<int>(blockIdx.x / p.BH) >= __ldg(p.ntiles)) return;   // spare slot
    __shared__ uint64_t in_full, in_empty, proj_done, qt_ready, kc_full[kRing], kc_empty[kRing], s_full[2], s_free[2],
        drain_bar, plan_bar;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag, fail_flag;

    const uint32_t warp = warp_id(), lane = lane_id();
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + ((1024u - (raw & 1023u)) & 1023u);
    const int K = p.topk;
    uint8_t* qh_s = smem;                                  // Q half (projection), then histograms / list blocks
    uint8_t* ring = smem + Cfg::OFF_RING;                  // Wq slice (projection), then summary chunks
    uint32_t* hist = reinterpret_cast<uint32_t*>(smem);
    // list entry e of row r: block at word e * kRows + r, product OFF_LG bytes on
    const Staging st{reinterpret_cast<int32_t*>(smem), reinterpret_cast<float*>(smem + Cfg::OFF_LG), Cfg::STRIDE, 1};
    uint8_t* umap = smem + Cfg::OFF_BITMAP;   // union map: byte m set when some row keeps block m

    // the tile: its index within its sequence, the sequence's first row and
    // length, and the summary slot of the sequence's block 0 (packed sequences:
    // floor(cu[s] / 64) + s, see the block-summary pass)
    const TileGeo geo = tile_geo(p);
    const int t = geo.t;
    const int seq_n = geo.n;
    const int kt0 = p.tiles == nullptr ? 0 : geo.base / 64 + geo.seq;
    const int bh = head_of_block(p.BH);
    const int diag = 2 * t;
    // full training scope: no Top-K, the scores and their log-sum-exp are written out
    const bool full = p.full_lse != nullptr;
    // full*: noise added to the scores before the gate and the Top-K
    const bool noisy = p.noise != nullptr;
    const int nb = min(2 * t + 1, seq_n / 64);  // blocks scored for this tile (full blocks of its sequence)
    const int nchunks = (K > 0 || full) ? (nb + kChunk - 1) / kChunk : 0;
    // the most blocks any row of the tile has: a histogram pass only when it exceeds K
    const int last_row = min(seq_n, (t + 1) * kRows) - 1;
    const int tile_ci = last_row >= t * kRows ? (last_row >> 6) : 0;
    const bool pass_b = !full && tile_ci > K;
    // passes over the chunks, in order; D runs only if a row fails (decided after B)
    const int npre = nchunks > 0 ? (full || !pass_b ? 2 : 3) : 0;   // A, [B], C  or  A, W
    // a history of at most two chunks stays in the two TMEM score buffers: its
    // products are computed once and every pass reads them again
    const bool resident = nchunks <= 2;
    const int rounds_total = G * (D / 64);   // projection rounds

    for (int w = threadIdx.x; w < ((p.C + 15) >> 2); w += blockDim.x) reinterpret_cast<uint32_t*>(umap)[w] = 0u;
    if (threadIdx.x == 0) {
        mbar_init(&in_full, 1);
        mbar_init(&in_empty, 1);
        mbar_init(&proj_done, 1);
        mbar_init(&qt_ready, 4);
        for (int s = 0; s < kRing; ++s) {
            mbar_init(&kc_full[s], 1);
            mbar_init(&kc_empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&s_full[b], 1);
            mbar_init(&s_free[b], 4);   // one arrive per row warp
        }
        mbar_init(&drain_bar, 1);
        mbar_init(&plan_bar, 4);   // one arrive per row warp once its rows know their mode (after pass B)
        abort_flag = 0;
        fail_flag = 0;
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
            tma_prefetch_desc(&mapQ);
            tma_prefetch_desc(&mapWq);
            tma_prefetch_desc(&mapKt);
            bool ok = true;
            int rounds = 0;
            for (int rd = 0; rd < rounds_total; ++rd) {
                // round rd: columns 64 a .. 64 a + 63 of query head bh G + hq and the
                // matching columns hq D + 64 a .. of Wq
                const int hq = rd / (D / 64), a = rd % (D / 64);
                if (rd > 0 && !mbar_wait(&in_empty, (rd - 1) & 1, wc)) { ok = false; break; }
                mbar_arrive_expect_tx(&in_full, Cfg::QH_BYTES + Cfg::WQH_BYTES);
                tma_load_3d(qh_s, &mapQ, &in_full, a * 64, geo.base + t * kRows, bh * G + hq);
                tma_load_3d(ring, &mapWq, &in_full, hq * D + a * 64, 0, bh % H);
                ++rounds;
            }
            int issued = 0;
            if (ok) ok = mbar_wait(&proj_done, 0, wc);   // the ring is free once the projection ran
            const int npass = resident ? 1 : npre;
            for (int ps = 0; ok && ps < npass + 1; ++ps) {
                if (resident && ps == npass) break;
                if (ps == npass) {
                    // after the pre-planned passes: pass D if a row failed
                    if (!pass_b) break;
                    if (!mbar_wait(&plan_bar, 0, wc)) { ok = false; break; }
                    if (!*reinterpret_cast<volatile int*>(&fail_flag)) break;
                }
                for (int c = 0; ok && c < nchunks; ++c) {
                    const int gc = issued;
                    const int s = gc % kRing;
                    if (!mbar_wait(&kc_empty[s], ((gc / kRing) & 1) ^ 1u, wc)) { ok = false; break; }
                    mbar_arrive_expect_tx(&kc_full[s], Cfg::KC_BYTES);
#pragma unroll
                    for (int a = 0; a < DS / 64; ++a)
                        tma_load_3d(ring + s * Cfg::KC_BYTES + a * (kChunk * 128), &mapKt, &kc_full[s], a * 64,
                                    kt0 + c * kChunk, bh);
                    ++issued;
                }
            }
            if (!ok) {
                if (rounds > 0) mbar_wait_drain(&in_full, (rounds - 1) & 1, p.limit, p.status);
                for (int q = issued - 1; q >= 0 && q >= issued - kRing; --q)
                    mbar_wait_drain(&kc_full[q % kRing], (q / kRing) & 1, p.limit, p.status);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer (whole warp; the elected lane issues: one thread
        // alone needs more cycles per tcgen05.mma issue)
        bool in_ok = nchunks > 0;
        const uint32_t q_addr = smem_u32(qh_s), w_addr = smem_u32(ring);   // projection operands
        for (int rd = 0; in_ok && rd < rounds_total; ++rd) {
            if (!mbar_wait_warp(&in_full, rd & 1, wc)) { in_ok = false; break; }
            tc_fence_after();
            // q~ (fp32, TMEM columns 0 .. DS-1) += Q half (128 x 64) * Wq slice (DS x 64)^T
            if (elect_one()) {
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    umma_bf16(tmem_base, smem_desc_sw128(q_addr + k * 32, 16, 1024),
                              smem_desc_sw128(w_addr + k * 32, 16, 1024), Cfg::IDESC_PROJ,
                              (rd > 0 || k > 0) ? 1u : 0u);
                umma_commit(rd + 1 < rounds_total ? &in_empty : &proj_done);   // Q half and Wq slice free
            }
            __syncwarp();
        }
        if (in_ok && mbar_wait_warp(&qt_ready, 0, wc)) {
            // S[gc&1] = q~ (128 x DS, bf16 in TMEM columns 0 .. DS/2) * Kt_chunk (32 x DS)^T,
            // for every chunk of every pass
            int gc = 0;
            bool ok = true;
            const int npass = resident ? 1 : npre;
            for (int ps = 0; ok && ps < npass + 1; ++ps) {
                if (resident && ps == npass) break;
                if (ps == npass) {
                    if (!pass_b) break;
                    if (!mbar_wait_warp(&plan_bar, 0, wc)) break;
                    if (!__all_sync(0xffffffffu, *reinterpret_cast<volatile int*>(&fail_flag) != 0)) break;
                }
                for (int c = 0; c < nchunks; ++c, ++gc) {
                    const int s = gc % kRing, b = gc & 1;
                    if (!mbar_wait_warp(&kc_full[s], (gc / kRing) & 1, wc)) { ok = false; break; }
                    if (!mbar_wait_warp(&s_free[b], ((gc >> 1) & 1) ^ 1u, wc)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t k_addr = smem_u32(ring + s * Cfg::KC_BYTES);
                    if (elect_one()) {
#pragma unroll
                        for (int k = 0; k < DS / 16; ++k) {
                            const uint32_t off_k = (k >> 2) * (kChunk * 128) + (k & 3) * 32;
                            umma_bf16_ta(tmem_base + Cfg::TMEM_S + b * kChunk, tmem_base + k * 8,
                                         smem_desc_sw128(k_addr + off_k, 16, 1024), Cfg::IDESC_S, k > 0);
                        }
                        umma_commit(&s_full[b]);
                        umma_commit(&kc_empty[s]);
                    }
                    __syncwarp();
                }
            }
        }
        if (elect_one()) {
            umma_commit(&drain_bar);
            mbar_wait_drain(&drain_bar, 0, p.limit, p.status);
        }
        __syncwarp();
    } else if (warp >= 2) {
        // ---------------- row threads
        const int q = warp & 3;
        const int r = q * 32 + lane;
        const int i = t * kRows + r;   // row within its sequence
        const bool valid = i < seq_n;
        const int Ci = valid ? (i >> 6) : 0;
        const int Kp = min(K, Ci);
        const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
        bool ok = true;
        if (nchunks > 0) {
            // q~ row: fp32 from TMEM columns 0 .. DS-1 -> bf16 pairs into columns
            // 0 .. DS/2-1 (element 2k in the low half of column k), the A operand
            // of the score products; each 64-column step reads its columns before
            // writing the 32 below them
            ok = mbar_wait_warp(&proj_done, 0, wc);
            if (ok) {
                tc_fence_after();
#pragma unroll 1
                for (int cc = 0; cc < DS / 64; ++cc) {
                    uint32_t u[32], o[32];
                    tmem_ld32(lane_addr + cc * 64, u);
                    tmem_wait_ld();
#pragma unroll
                    for (int k = 0; k < 16; ++k)
                        o[k] = pack_bf16x2(__uint_as_float(u[2 * k]), __uint_as_float(u[2 * k + 1]));
                    tmem_ld32(lane_addr + cc * 64 + 32, u);
                    tmem_wait_ld();
#pragma unroll
                    for (int k = 0; k < 16; ++k)
                        o[16 + k] = pack_bf16x2(__uint_as_float(u[2 * k]), __uint_as_float(u[2 * k + 1]));
                    tmem_st32(lane_addr + cc * 32, o);
                }
                tmem_wait_st();
                tc_fence_before();
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&qt_ready);
        }
        // this row's counters, over the Q half once the projection has read it
        uint32_t* my_hist = hist + r * Cfg::STRIDE;
        for (int w = 0; w < kBins; ++w) my_hist[w] = 0u;
        RowSel rs;
        rs.l = RowLse{-CUDART_INF_F, 0.f};
        rs.v0 = 0.f; rs.s1 = 0; rs.s2 = 0; rs.mn = CUDART_INF_F;
        row_set_all(rs);
        rs.nabove = 0; rs.pos = 0;
        rs.ws = -CUDART_INF_F; rs.wpos = 0;
        // the products u are selected on directly (s = u scale); with noise the
        // pass works on s~ = s + eps itself
        const float c_exp = noisy ? kLog2e : p.score_scale * kLog2e;
        const float emit_scale = noisy ? 1.f : p.score_scale;
        const long long row_off = static_cast<long long>(bh) * p.N + geo.base + i;
        const RowAddr ra{smem_u32(st.idx + r * st.stride), smem_u32(my_hist) - kBinMagicBits * 4u};
        int gc = 0;
        for (int ps = 0; ok && ps < npre + 1; ++ps) {
            int kind;
            if (ps == npre) {
                if (!pass_b) break;
                if (!mbar_wait_warp(&plan_bar, 0, wc)) { ok = false; break; }
                if (!*reinterpret_cast<volatile int*>(&fail_flag)) break;
                kind = kPassD;
            } else if (full) {
                kind = ps == 0 ? kPassA : kPassW;
            } else {
                kind = ps == 0 ? kPassA : (ps == npre - 1 ? kPassC : kPassB);
            }
            for (int c = 0; c < nchunks; ++c, ++gc) {
                const int b = resident ? c : (gc & 1);
                if ((!resident || ps == 0) && !mbar_wait_warp(&s_full[b], resident ? 0 : ((gc >> 1) & 1), wc)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                uint32_t uu[32];
                tmem_ld32(lane_addr + Cfg::TMEM_S + b * kChunk, uu);
                tmem_wait_ld();
                if (!resident) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&s_free[b]);
                }
                const int m0 = kChunk * c;
                const int lim = Ci - m0;
                if (noisy) {
                    const float* nrow = p.noise + row_off * p.C + m0;
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (j < lim)
                            uu[j] = __float_as_uint(
                                __fadd_rn(__fmul_rn(__uint_as_float(uu[j]), p.score_scale), __ldg(nrow + j)));
                }
                const float* u = reinterpret_cast<const float*>(uu);
                if (kind == kPassW) {
                    float* dst = p.full_table + row_off * p.C + m0;
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (j < lim) dst[j] = __fmul_rn(u[j], p.score_scale);
                } else {
                    // the vote comes before any lane leaves; the lanes meet again
                    // before the next warp-collective TMEM load
                    const bool whole = __all_sync(0xffffffffu, lim >= 32);
                    if (kind == kPassB || kind == kPassC) {
                        if (!whole) {
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (j >= lim) uu[j] = 0x7fc00000u;   // NaN: past the history
                        }
                        row_pass<true, Cfg::OFF_LG>(rs, kind, u, m0, lim, Kp, ra, st, r, c_exp);
                    } else if (whole) {
                        row_pass<true, Cfg::OFF_LG>(rs, kind, u, m0, lim, Kp, ra, st, r, c_exp);
                    } else if (lim > 0) {
                        row_pass<false, Cfg::OFF_LG>(rs, kind, u, m0, lim, Kp, ra, st, r, c_exp);
                    }
                }
                __syncwarp();
            }
            if (!ok) break;
            if (kind == kPassA) {
                row_after_a(rs, Ci, K);
            } else if (kind == kPassB) {
                row_after_b(rs, my_hist, Kp);
                // whether pass D runs (some row failed), for the producer, the MMA
                // issuer and the row warps: flag first, then one arrive per warp
                if (rs.mode == kRowFail) atomicOr(&fail_flag, 1);
                __syncwarp();
                if (lane == 0) mbar_arrive(&plan_bar);
            } else if (kind == kPassC) {
                row_after_c(rs, st, r, Kp);
            } else {
                staged_sort_by_block(st, r, rs.pos);
            }
        }
        ok = ok && !abort_flag;
        if (full) {
            // full scope: the row's log-sum-exp of its scores (the table is written)
            if (valid && ok) p.full_lse[row_off] = Ci > 0 ? __fmul_rn(rs.l.mx, p.score_scale) + logf(rs.l.sum) : 0.f;
        } else if (valid && ok) {
            // log-gates from s = u / sqrt(d_sel), -1 padding, tile-union bits
            const float lse = Ci > 0 ? __fmul_rn(rs.l.mx, emit_scale) + logf(rs.l.sum) : 0.f;
            for (int e = 0; e < K; ++e) {
                if (e < Kp) {
                    const int m = st.idx[r * st.stride + e * st.es];
                    const float sc = __fmul_rn(st.lg[r * st.stride + e * st.es], emit_scale);
                    st.lg[r * st.stride + e * st.es] = staged_gate(sc, lse, p.gate_act);
                    if (static_cast<unsigned>(m) < static_cast<unsigned>(diag)) umap[m] = 1;   // same value from any row
                } else {
                    st.idx[r * st.stride + e * st.es] = -1;
                    st.lg[r * st.stride + e * st.es] = 0.f;
                }
            }
        }
        if (!full) {
            named_bar_sync(1, 128);
            if (ok)
                copy_out(st, p, bh, static_cast<long long>(geo.base) + t * kRows, min(kRows, seq_n - t * kRows),
                         static_cast<int>(threadIdx.x) - 64, 128);
            if (warp == 2)
                compact_union_bytes(umap, diag, p.union_idx + (static_cast<long long>(bh) * p.T + geo.slot) * p.C,
                                    p.union_cnt + static_cast<long long>(bh) * p.T + geo.slot);
        }
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, 128);
    }
}

template <int D, int DS, bool BIGK>
cudaError_t launch_proj_k(const SelectArgs& a, const SelParams& p, const KernelEnv& env, const char** err) {
    const size_t smem = 1024 + proj_smem_bytes<D, DS, BIGK>(a.C);
    if (smem > 227 * 1024) { *err = "selection: too many blocks for shared memory"; return cudaErrorInvalidValue; }
    cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(select_proj_kernel<D, DS, BIGK>), smem, true);
    if (e != cudaSuccess) { *err = "cudaFuncSetAttribute(select)"; return e; }
    CUtensorMap mq, mw, mk;
    // Q of all query heads; Wq [H][DS][G D] (a group's gate-query projection)
    if (make_tmap_bf16_3d(&mq, a.Q, D, a.N, a.BH * a.G, 64, kRows) != 0) { *err = "tensor map Q"; return cudaErrorInvalidValue; }
    if (make_tmap_bf16_3d(&mw, a.Wq, static_cast<uint64_t>(a.G) * D, DS, a.H, 64, DS) != 0) { *err = "tensor map Wq"; return cudaErrorInvalidValue; }
    if (make_tmap_bf16_3d(&mk, a.Kt, DS, a.F > 0 ? a.F : 1, a.BH, 64, kChunk) != 0) { *err = "tensor map Kt"; return cudaErrorInvalidValue; }
    const dim3 grid(a.BH * a.T);
    select_proj_kernel<D, DS, BIGK><<<grid, 192, smem, env.stream>>>(mq, mw, mk, p, a.H, a.G);
    e = cudaGetLastError();
    if (e != cudaSuccess) *err = "select launch";
    return e;
}

// K + kBoundaryMax list entries per row: within the histogram words up to K = 36
template <int D, int DS>
cudaError_t launch_proj(const SelectArgs& a, const SelParams& p, const KernelEnv& env, const char** err) {
    if (a.topk + kBoundaryMax <= kListSmall) return launch_proj_k<D, DS, false>(a, p, env, err);
    if (a.topk + kBoundaryMax <= kListBig) return launch_proj_k<D, DS, true>(a, p, env, err);
    *err = "selection: top-K too large";
    return cudaErrorInvalidValue;
}

template <bool REG, bool NOISE>
cudaError_t launch_given(const SelectArgs& a, const SelParams& p, const KernelEnv& env, const char** err) {
    const size_t smem = smem_topk_bytes(a.topk) + staging_bytes(a.topk) + bitmap_bytes(a.C);
    if (smem > 200 * 1024) { *err = "selection: top-K too large for shared memory"; return cudaErrorInvalidValue; }
    cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(select_given_kernel<REG, NOISE>), smem);
    if (e != cudaSuccess) { *err = "cudaFuncSetAttribute(select_given)"; return e; }
    const dim3 grid(a.BH * a.T);
    select_given_kernel<REG, NOISE><<<grid, 128, smem, env.stream>>>(p);
    e = cudaGetLastError();
    if (e != cudaSuccess) *err = "select launch";
    return e;
}


// Full training scope with given scores: each row's log-sum-exp over its C_i
// scores (Eq. normalized_log_gate's normaliser), one warp per row, reading the
// row twice (maximum, then the sum; the second read hits the cache).
__global__ void __launch_bounds__(256) row_lse_kernel(const float* scores, int N, int C, long long rows,
                                                      float* out) {
    const long long w = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (w >= rows) return;
    const int i = static_cast<int>(w % N);
    const int Ci = i >> 6;
    const float* s = scores + w * C;
    float mx = -CUDART_INF_F;
    for (int m = lane; m < Ci; m += 32) mx = fmaxf(mx, __ldg(s + m));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float sum = 0.f;
    for (int m = lane; m < Ci; m += 32) sum += fast_exp2((__ldg(s + m) - mx) * kLog2e);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (lane == 0) out[w] = Ci > 0 ? mx + logf(sum) : 0.f;
}

constexpr int kStatusBadInput = 1;   // == SAS_ERR_INVALID_ARG

// Tile table of packed sequences (one CTA).  Sequence s holds rows
// cu[s] .. cu[s+1]-1 and T_s = ceil(n_s / 128) tiles; an entry is
// {first row cu[s], tile index within the sequence, n_s, s}.  Entries are ordered by
// the tile's index within its sequence, descending (longest key history
// first): tile t of every sequence with T_s > t sits at off(t) + rank(s),
// off(t) = number of tiles with a larger index, rank(s) = the sequence's place
// when sequences are ordered by T_s descending (ties in arrival order: the
// order only schedules work).  Bad offsets set the status word and leave no
// tiles.
__global__ void __launch_bounds__(1024) varlen_tiles_kernel(const int32_t* cu, int S, int Ncap, int max_len,
                                                            int tmax, int4* tiles, int* ntiles, int* tile_off,
                                                            int* status) {
    extern __shared__ int vsh[];   // hist[tmax + 2], cnt_gt[tmax + 2], off[tmax + 2], next[tmax + 2]
    int* hist = vsh;
    int* gt = hist + tmax + 2;     // gt[t] = number of sequences with T_s > t
    int* off = gt + tmax + 2;
    int* nxt = off + tmax + 2;
    __shared__ int bad;
    const int tid = threadIdx.x;
    for (int k = tid; k < tmax + 2; k += blockDim.x) { hist[k] = 0; nxt[k] = 0; }
    if (tid == 0) bad = (S < 1 || __ldg(cu) != 0 || __ldg(cu + S) > Ncap) ? 1 : 0;
    __syncthreads();
    for (int s = tid; s < S; s += blockDim.x) {
        const int n = __ldg(cu + s + 1) - __ldg(cu + s);
        if (n < 0 || n > max_len) { bad = 1; continue; }
        atomicAdd(&hist[(n + kRows - 1) / kRows], 1);
    }
    __syncthreads();
    if (bad) {
        if (tid == 0) {
            *ntiles = 0;
            atomicExch(status, kStatusBadInput);
        }
        return;
    }
    if (tid == 0) {
        // gt[t] = sum_{T > t} hist[T]; off[t] = sum_{t' > t} gt[t']
        int g = 0, o = 0;
        for (int t = tmax; t >= 0; --t) {
            g += hist[t + 1];
            gt[t] = g;
            off[t] = o;
            o += g;
        }
        *ntiles = o;
    }
    __syncthreads();
    // first slot of every local tile index: sequence s of rank r keeps its
    // tile t at slot tile_off[t] + r (the backward maps tiles of a sequence
    // to one another through it)
    for (int t = tid; t <= tmax; t += blockDim.x) tile_off[t] = off[t];
    for (int s = tid; s < S; s += blockDim.x) {
        const int b0 = __ldg(cu + s), n = __ldg(cu + s + 1) - b0;
        const int T = (n + kRows - 1) / kRows;
        if (T == 0) continue;
        const int rank = gt[T] + atomicAdd(&nxt[T], 1);   // sequences with more tiles come first
        for (int t = 0; t < T; ++t) tiles[off[t] + rank] = make_int4(b0, t, n, s);
    }
}

}  // namespace

cudaError_t launch_varlen_tiles(const int32_t* cu, int S, int Ncap, int max_len, int4* tiles, int* ntiles,
                                int* tile_off, const KernelEnv& env) {
    const int tmax = (max_len + kRows - 1) / kRows;
    const size_t smem = static_cast<size_t>(4) * (tmax + 2) * sizeof(int);
    if (smem > 200 * 1024) return cudaErrorInvalidValue;
    if (smem > 48 * 1024) {
        cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(varlen_tiles_kernel), smem);
        if (e != cudaSuccess) return e;
    }
    varlen_tiles_kernel<<<1, 1024, smem, env.stream>>>(cu, S, Ncap, max_len, tmax, tiles, ntiles, tile_off,
                                                       env.status);
    return cudaGetLastError();
}

namespace {

// Head-packed GQA tiles: per (KV group, segment of R tokens) the sorted union
// of the tokens' kept blocks, from the kept lists.  One warp per segment; its
// tokens share one current block c (R <= 64, segments aligned), and kept
// blocks are < c.  cap: row stride of the output lists (>= min(C, R topk)).
// Packed sequences: segment sg is part sg % G of tile slot sg / G (G = 128 / R).
__global__ void __launch_bounds__(256) seg_union_kernel(const int32_t* sel_idx, int BHkv, int N, int C, int topk,
                                                        int R, int nseg, int cap, int32_t* out_idx,
                                                        int32_t* out_cnt, const int4* tiles, const int* ntiles) {
    extern __shared__ uint32_t segbits[];   // per warp: ceil(C / 32) words
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long item = static_cast<long long>(blockIdx.x) * (blockDim.x >> 5) + warp;
    if (item >= static_cast<long long>(BHkv) * nseg) return;   // no block-wide synchronisation below
    const int kv = static_cast<int>(item / nseg), sg = static_cast<int>(item - static_cast<long long>(kv) * nseg);
    const int nw = (C + 31) >> 5;
    uint32_t* bits = segbits + warp * nw;
    for (int w = lane; w < nw; w += 32) bits[w] = 0u;
    __syncwarp();
    // the segment's first token within its sequence, the sequence's first row and length
    int i0 = sg * R, base = 0, n = N;
    if (tiles != nullptr) {
        const int G = kRows / R;
        if (sg / G >= __ldg(ntiles)) return;   // an unused slot: the attention does not read it
        const int4 v = __ldg(tiles + sg / G);
        i0 = v.y * kRows + (sg % G) * R;
        base = v.x;
        n = v.z;
    }
    for (int rr = lane; rr < R; rr += 32) {
        const int i = i0 + rr;
        if (i >= n) break;
        const int c = i >> 6;
        const int ne = min(topk, c);
        const int32_t* idx = sel_idx + (static_cast<long long>(kv) * N + base + i) * topk;
        for (int e = 0; e < ne; ++e) {
            const int m = __ldg(idx + e);
            if (static_cast<unsigned>(m) < static_cast<unsigned>(c)) atomicOr(&bits[m >> 5], 1u << (m & 31));
        }
    }
    __syncwarp();
    compact_union(bits, i0 >> 6, out_idx + item * cap, out_cnt + item);
}

}  // namespace

cudaError_t launch_seg_unions(const int32_t* sel_idx, int BHkv, int N, int C, int topk, int seg_rows, int nseg,
                              int32_t* seg_union_idx, int32_t* seg_union_cnt, const KernelEnv& env, const int4* tiles,
                              const int* ntiles) {
    const long long items = static_cast<long long>(BHkv) * nseg;
    const size_t smem = static_cast<size_t>(8) * ((C + 31) / 32) * 4;
    if (smem > 48 * 1024) {
        cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(seg_union_kernel), smem);
        if (e != cudaSuccess) return e;
    }
    const int cap = min(C, seg_rows * max(topk, 1));
    seg_union_kernel<<<static_cast<unsigned>((items + 7) / 8), 256, smem, env.stream>>>(
        sel_idx, BHkv, N, C, topk, seg_rows, nseg, cap, seg_union_idx, seg_union_cnt, tiles, ntiles);
    return cudaGetLastError();
}

cudaError_t launch_row_lse(const float* scores, int N, int C, long long rows, float* out, const KernelEnv& env) {
    const long long blocks = (rows * 32 + 255) / 256;
    row_lse_kernel<<<static_cast<unsigned>(blocks), 256, 0, env.stream>>>(scores, N, C, rows, out);
    return cudaGetLastError();
}

cudaError_t launch_select(const SelectArgs& a, const KernelEnv& env, const char** err) {
    SelParams p;
    p.BH = a.BH; p.N = a.N; p.C = a.C; p.T = a.T; p.F = a.F; p.topk = a.topk;
    p.gate_act = a.gate_act;
    p.score_scale = a.score_scale;
    p.scores = a.scores;
    p.sel_idx = a.sel_idx; p.sel_logg = a.sel_logg;
    p.union_idx = a.union_idx; p.union_cnt = a.union_cnt;
    p.tiles = a.tiles; p.ntiles = a.ntiles;
    p.status = env.status; p.limit = env.limit;
    p.full_lse = a.full_lse; p.full_table = a.full_table; p.noise = a.noise;
    if (a.full_lse != nullptr && (a.tiles != nullptr || a.noise != nullptr)) {
        *err = "selection: the full scope takes neither packed sequences nor noise";
        return cudaErrorInvalidValue;
    }
    if (a.full_lse != nullptr && a.scores != nullptr) {
        // given scores: the attention kernel reads them directly; only the normalisers
        cudaError_t e = launch_row_lse(a.scores, a.N, a.C, static_cast<long long>(a.BH) * a.N, a.full_lse, env);
        if (e != cudaSuccess) *err = "row log-sum-exp launch";
        return e;
    }

    const bool reg = a.topk <= 32;
    if (a.scores != nullptr) {
        if (a.noise != nullptr)
            return reg ? launch_given<true, true>(a, p, env, err) : launch_given<false, true>(a, p, env, err);
        return reg ? launch_given<true, false>(a, p, env, err) : launch_given<false, false>(a, p, env, err);
    }
    if (a.d == 128 && a.d_sel == 128) return launch_proj<128, 128>(a, p, env, err);
    if (a.d == 128 && a.d_sel == 64) return launch_proj<128, 64>(a, p, env, err);
    if (a.d == 64 && a.d_sel == 64) return launch_proj<64, 64>(a, p, env, err);
    if (a.d == 64 && a.d_sel == 128) return launch_proj<64, 128>(a, p, env, err);
    *err = "selection: unsupported head / selector dims";
    return cudaErrorInvalidValue;
}

}  // namespace sas
