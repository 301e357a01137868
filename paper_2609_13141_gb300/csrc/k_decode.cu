// Decode step of SAS (Alg. 2): one new token per sequence, grouped-query
// attention with one block selection per query group (Sec. 5, inference
// implementation), over a paged KV cache holding one 64-token block per page.
//
//   dec_prep_kernel    appends k_new / v_new at position n-1, summarises the block
//                      that position closes (K~ = bf16(Wk mean K), App. B) and
//                      forms the group's gate query q~ = bf16(Wq_g [q_0; ...]).
//   dec_score_kernel   s_m = q~ . K~_m / sqrt(d_sel) for the C historical blocks
//                      (Alg. 2 step 1), CTAs of 256 blocks whose summary rows are
//                      staged in shared memory by bulk async copies.  Each CTA keeps
//                      the exact Top-K of its own blocks (rank by counting); the
//                      last CTA of a group selects the Top-K of those candidates
//                      (step 2) by a radix select on the scores' order-preserving
//                      bit patterns, ties to the lower block, and writes the kept
//                      list in ascending order.
//   dec_attn_kernel    split-KV attention over B_0 and the kept blocks (steps 3-4):
//                      each CTA streams one or a few pages (K and V slices of 16 KB
//                      at d = 128, bulk async copies into a ring), keeps an online
//                      softmax per head, and the last CTA of a group merges the
//                      partial (max, sum, output) triples.
// The three kernels are chained with programmatic dependent launch: each one
// starts while its predecessor runs, does the work that needs none of the
// predecessor's results (barrier set-up, reading lengths and queries, the page
// of the current block) and then waits on the grid dependency.
// A decode step moves bytes, not flops (a few FMAs per cached element), so the
// arithmetic runs on CUDA cores with packed fp32x2 FMAs; there is no tensor-core
// contraction on this path.
#include <math_constants.h>

#include "internal.h"
#include "ptx.cuh"

namespace sas {
namespace {

constexpr int kBlk = 64;
constexpr int kStatusBadInput = 1;   // == SAS_ERR_INVALID_ARG
constexpr int kPrepThreads = 256;
constexpr int kScoreThreads = 256;
constexpr int kAttnThreads = 256;
constexpr int kStages = 3;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ bool bad_len(int n, const DecodeArgs& a) { return n < 1 || n > a.max_blocks * kBlk; }

// Programmatic dependent launch: wait until the preceding grid has completed
// and its writes are visible; allow the next grid to start launching.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Exclusive prefix sum over the 256 threads of a CTA (scan: 16 shared ints).
__device__ int block_excl_scan(int v, int* scan) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) scan[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = lane < 8 ? scan[lane] : 0;
        const int own = w;
#pragma unroll
        for (int o = 1; o < 8; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        if (lane < 8) scan[8 + lane] = w - own;
    }
    __syncthreads();
    const int r = x - v + scan[8 + warp];
    __syncthreads();
    return r;
}

// One full block's summary (App. B): the mean of its 64 keys in fp32, projected
// by the KV head's Wk [d_sel][d] and rounded to bf16.  256 threads.
// red: 512 floats, kbar: 128 floats of shared memory.
__device__ void summarize_block(const bf16* Kt, const bf16* Wk, bf16* out, int d, int d_sel, float* red,
                                float* kbar) {
    const int t = threadIdx.x;
    const int nw = d >> 1;                    // bf16 pairs per key row
    const int groups = kPrepThreads / nw;     // 4 (d = 128) or 8 (d = 64) row groups
    const int rows = kBlk / groups;
    const int wi = t % nw, rg = t / nw;
    const uint32_t* K32 = reinterpret_cast<const uint32_t*>(Kt);
    float a0 = 0.f, a1 = 0.f;
    for (int r = rg * rows; r < (rg + 1) * rows; ++r) {
        const uint32_t w = __ldg(K32 + r * nw + wi);
        a0 += bf_lo(w);
        a1 += bf_hi(w);
    }
    red[rg * d + 2 * wi] = a0;
    red[rg * d + 2 * wi + 1] = a1;
    __syncthreads();
    if (t < d) {
        float s = 0.f;
        for (int g = 0; g < groups; ++g) s += red[g * d + t];
        kbar[t] = s * (1.f / kBlk);
    }
    __syncthreads();
    const int warp = t >> 5, lane = t & 31;
    for (int o = warp; o < d_sel; o += kPrepThreads / 32) {
        const uint32_t* row = reinterpret_cast<const uint32_t*>(Wk + static_cast<size_t>(o) * d);
        float acc = 0.f;
        for (int e = lane; e < nw; e += 32) {
            const uint32_t w = __ldg(row + e);
            acc = fmaf(bf_lo(w), kbar[2 * e], acc);
            acc = fmaf(bf_hi(w), kbar[2 * e + 1], acc);
        }
        acc = warp_sum(acc);
        if (lane == 0) out[o] = __float2bfloat16_rn(acc);
    }
}

// grid (B*Hkv, 1 + d_sel/8): y = 0 appends the token and updates the summary
// cache, y >= 1 computes 8 entries of the group's gate query (one per warp).
__global__ void __launch_bounds__(kPrepThreads) dec_prep_kernel(DecodeArgs a, int* status) {
    __shared__ float red[512];
    __shared__ __align__(16) float vec[1024];
    grid_dep_launch();   // the score kernel may start its set-up
    const int bh = blockIdx.x;
    const int b = bh / a.Hkv, g = bh - b * a.Hkv;
    const int n = __ldg(a.seq_lens + b);
    const int t = threadIdx.x;
    if (bad_len(n, a)) {
        if (t == 0 && blockIdx.y == 0) atomicExch(status, kStatusBadInput);
        return;
    }
    if (blockIdx.y == 0) {
        const int pos = n - 1, blk = pos / kBlk, slot = pos - blk * kBlk;
        const int32_t* row = a.block_table + static_cast<size_t>(b) * a.max_blocks;
        const int page = __ldg(row + blk);
        if (page < 0 || page >= a.num_pages) {
            if (t == 0) atomicExch(status, kStatusBadInput);
            return;
        }
        if (a.k_new != nullptr) {
            const int nu = a.d / 8;   // 16-byte units per row
            if (t < 2 * nu) {
                const bool isv = t >= nu;
                const int u = isv ? t - nu : t;
                const uint4* src =
                    reinterpret_cast<const uint4*>(static_cast<const bf16*>(isv ? a.v_new : a.k_new) +
                                                   static_cast<size_t>(bh) * a.d) + u;
                uint4* dst = reinterpret_cast<uint4*>(static_cast<bf16*>(isv ? a.V_cache : a.K_cache) +
                                                      ((static_cast<size_t>(page) * a.Hkv + g) * kBlk + slot) * a.d) + u;
                *dst = __ldg(src);
            }
        }
        if (!a.dense && slot == 0 && blk >= 1) {
            const int pp = __ldg(row + blk - 1);
            if (pp < 0 || pp >= a.num_pages) {
                if (t == 0) atomicExch(status, kStatusBadInput);
                return;
            }
            summarize_block(static_cast<const bf16*>(a.K_cache) + (static_cast<size_t>(pp) * a.Hkv + g) * kBlk * a.d,
                            static_cast<const bf16*>(a.Wk) + static_cast<size_t>(g) * a.d_sel * a.d,
                            static_cast<bf16*>(a.Ksum) + (static_cast<size_t>(bh) * a.max_blocks + blk - 1) * a.d_sel,
                            a.d, a.d_sel, red, vec);
        }
        return;
    }
    // gate query q~[o] = bf16(sum_e Wq_g[o][e] q_cat[e]), o = 8 (y-1) + warp.  The
    // warp's row of Wq_g (G*d <= 1024 bf16) is loaded in one go, 32 bytes a lane.
    const int GD = a.G * a.d;
    const int warp = t >> 5, lane = t & 31;
    const int o = (blockIdx.y - 1) * 8 + warp;
    const bool has_row = o < a.d_sel;
    const bf16* wrow = static_cast<const bf16*>(a.Wq) + (static_cast<size_t>(g) * a.d_sel + (has_row ? o : 0)) * GD;
    uint4 w[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int e = (k * 32 + lane) * 8;
        w[k] = (has_row && e < GD) ? __ldg(reinterpret_cast<const uint4*>(wrow + e)) : make_uint4(0, 0, 0, 0);
    }
    const bf16* qg = static_cast<const bf16*>(a.q) + (static_cast<size_t>(b) * a.Hq + static_cast<size_t>(g) * a.G) * a.d;
    for (int e = t; e < GD; e += kPrepThreads) vec[e] = __bfloat162float(qg[e]);
    __syncthreads();
    if (!has_row) return;
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int e = (k * 32 + lane) * 8;
        if (e < GD) {
            const float4 x0 = *reinterpret_cast<const float4*>(vec + e);
            const float4 x1 = *reinterpret_cast<const float4*>(vec + e + 4);
            acc = fmaf(bf_lo(w[k].x), x0.x, acc);
            acc = fmaf(bf_hi(w[k].x), x0.y, acc);
            acc = fmaf(bf_lo(w[k].y), x0.z, acc);
            acc = fmaf(bf_hi(w[k].y), x0.w, acc);
            acc = fmaf(bf_lo(w[k].z), x1.x, acc);
            acc = fmaf(bf_hi(w[k].z), x1.y, acc);
            acc = fmaf(bf_lo(w[k].w), x1.z, acc);
            acc = fmaf(bf_hi(w[k].w), x1.w, acc);
        }
    }
    acc = warp_sum(acc);
    if (lane == 0) static_cast<bf16*>(a.qt)[static_cast<size_t>(bh) * a.d_sel + o] = __float2bfloat16_rn(acc);
}

// grid (max_blocks, B*Hkv): summary of full block m of every sequence (after a prefill).
__global__ void __launch_bounds__(kPrepThreads) dec_summarize_kernel(DecodeArgs a, int* status) {
    __shared__ float red[512];
    __shared__ float kbar[128];
    const int m = blockIdx.x, bh = blockIdx.y;
    const int b = bh / a.Hkv, g = bh - b * a.Hkv;
    const int n = __ldg(a.seq_lens + b);
    if (n < 0 || n > a.max_blocks * kBlk) {
        if (threadIdx.x == 0 && m == 0) atomicExch(status, kStatusBadInput);
        return;
    }
    if (m >= n / kBlk) return;
    const int page = __ldg(a.block_table + static_cast<size_t>(b) * a.max_blocks + m);
    if (page < 0 || page >= a.num_pages) {
        if (threadIdx.x == 0) atomicExch(status, kStatusBadInput);
        return;
    }
    summarize_block(static_cast<const bf16*>(a.K_cache) + (static_cast<size_t>(page) * a.Hkv + g) * kBlk * a.d,
                    static_cast<const bf16*>(a.Wk) + static_cast<size_t>(g) * a.d_sel * a.d,
                    static_cast<bf16*>(a.Ksum) + (static_cast<size_t>(bh) * a.max_blocks + m) * a.d_sel, a.d, a.d_sel,
                    red, kbar);
}

// ------------------------------------------------------------ scores + Top-K

struct ScoreSmem {
    size_t r0;   // staged summary rows; in the last CTA the candidates (keys, blocks)
    size_t qs, bars, misc, xchg, hist, scan, total;
};
__host__ __device__ inline ScoreSmem score_smem_layout(int nsplit, int topk, int d_sel) {
    ScoreSmem L;
    const size_t slab = static_cast<size_t>(8) * 32 * d_sel * 2;
    const size_t cand = static_cast<size_t>(nsplit) * (topk > 0 ? topk : 1) * 8;
    L.r0 = ((slab > cand ? slab : cand) + 127) / 128 * 128;
    L.qs = L.r0;                  // d_sel bf16 (<= 256 bytes)
    L.bars = L.qs + 256;          // 8 mbarriers
    L.misc = L.bars + 64;         // flag, radix broadcast, per-warp counts (16 ints)
    L.xchg = L.misc + 64;         // 256 64-bit sort keys
    L.hist = L.xchg + 256 * 8;    // 4096 ints
    L.scan = L.hist + 4096 * 4;   // 16 ints
    L.total = L.scan + 128;
    return L;
}

// Order-preserving map of a finite float to uint32 (larger float, larger key);
// -0 is mapped like +0 so that equal scores stay ties.  Every finite float maps
// above 0, so 0 marks an empty candidate slot.
__device__ __forceinline__ uint32_t order_key(float f) {
    const uint32_t u = __float_as_uint(f == 0.f ? 0.f : f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Descending bitonic sort of 256 distinct 64-bit keys, one per thread of the
// CTA; returns the key that ends at position threadIdx.x.  Exchanges within a
// warp use shuffles, wider ones the 256-entry shared buffer xchg.
__device__ uint64_t bitonic256_desc(uint64_t c, uint64_t* xchg) {
    const int t = threadIdx.x;
#pragma unroll
    for (int k = 2; k <= 256; k <<= 1) {
#pragma unroll
        for (int j = k >> 1; j > 0; j >>= 1) {
            uint64_t o;
            if (j >= 32) {
                xchg[t] = c;
                __syncthreads();
                o = xchg[t ^ j];
                __syncthreads();
            } else {
                o = __shfl_xor_sync(0xffffffffu, c, j);
            }
            const bool keep_max = ((t & j) == 0) == ((t & k) == 0);
            c = keep_max ? (c > o ? c : o) : (c < o ? c : o);
        }
    }
    return c;
}

// Exact Top-K of M candidates (keys[i], block idx[i]) listed in ascending block
// order, ties to the lower block: radix select of the K-th largest key tau in
// digits of 12, 10 and 10 bits, then every key > tau plus the first keys == tau,
// emitted in list order.  256 threads; K < number of non-empty candidates.
__device__ void select_candidates(const DecodeArgs& a, int bh, int M, const uint32_t* keys, const int32_t* idx,
                                  int* hist, int* scan, int* bc) {
    const int K = a.topk;
    const int t = threadIdx.x, lane = t & 31;
    int32_t* lst = a.list + static_cast<size_t>(bh) * 64;
    int32_t* so = a.sel_idx ? a.sel_idx + static_cast<size_t>(bh) * K : nullptr;
    uint32_t prefix = 0, mask = 0;
    int r = K;
#pragma unroll 1
    for (int pass = 0; pass < 3; ++pass) {
        const int width = pass == 0 ? 12 : 10;
        const int sh = pass == 0 ? 20 : (pass == 1 ? 10 : 0);
        const int nb = 1 << width;
        for (int i = t; i < nb; i += kScoreThreads) hist[i] = 0;
        __syncthreads();
        for (int base = 0; base < M; base += kScoreThreads) {
            const int i = base + t;
            bool in = false;
            int bin = 0;
            if (i < M) {
                const uint32_t k = keys[i];
                in = (k & mask) == prefix;
                bin = static_cast<int>((k >> sh) & static_cast<uint32_t>(nb - 1));
            }
            // lanes with the same bin add once (the first pass sees few distinct bins)
            const uint32_t peers = __match_any_sync(0xffffffffu, in ? bin : -1 - lane);
            if (in && lane == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
        }
        __syncthreads();
        const int per = nb / kScoreThreads;   // 16 or 4 bins per thread, highest digits first
        int s = 0;
        for (int j = 0; j < per; ++j) s += hist[nb - 1 - (t * per + j)];
        const int excl = block_excl_scan(s, scan);
        if (excl < r && excl + s >= r) {
            int cum = excl;
            for (int j = 0; j < per; ++j) {
                const int bin = nb - 1 - (t * per + j);
                const int c = hist[bin];
                if (cum + c >= r) {
                    bc[0] = bin;
                    bc[1] = r - cum;
                    break;
                }
                cum += c;
            }
        }
        __syncthreads();
        prefix |= static_cast<uint32_t>(bc[0]) << sh;
        mask |= static_cast<uint32_t>(nb - 1) << sh;
        r = bc[1];
    }
    const uint32_t tau = prefix;   // the K-th largest key; take the first r keys equal to it
    // list-order emission: contiguous ranges of odd length per thread (conflict-free reads)
    const int per = ((M + kScoreThreads - 1) / kScoreThreads) | 1;
    const int lo = min(t * per, M), hi = min(lo + per, M);
    int eq = 0;
    for (int i = lo; i < hi; ++i) eq += keys[i] == tau;
    const int eq_base = block_excl_scan(eq, scan);
    int cnt = 0, er = eq_base;
    for (int i = lo; i < hi; ++i) {
        const uint32_t k = keys[i];
        if (k > tau) {
            ++cnt;
        } else if (k == tau) {
            if (er < r) ++cnt;
            ++er;
        }
    }
    int pos = block_excl_scan(cnt, scan);
    er = eq_base;
    for (int i = lo; i < hi; ++i) {
        const uint32_t k = keys[i];
        bool take = k > tau;
        if (k == tau) {
            take = er < r;
            ++er;
        }
        if (take) {
            lst[pos] = idx[i];
            if (so) so[pos] = idx[i];
            ++pos;
        }
    }
    if (t == 0) a.list_n[bh] = K;
}

// grid (nsplit_s, B*Hkv), launched as a programmatic dependent of the prep kernel.
template <int DSEL>
__global__ void __launch_bounds__(kScoreThreads) dec_score_kernel(DecodeArgs a, int* status, long long limit,
                                                                  float score_scale) {
    extern __shared__ __align__(128) uint8_t smem[];
    constexpr int kRowBytes = DSEL * 2;
    constexpr int kSlab = 32 * kRowBytes;
    const ScoreSmem L = score_smem_layout(a.nsplit_s, a.topk, DSEL);
    uint8_t* stage = smem;
    uint4* qs = reinterpret_cast<uint4*>(smem + L.qs);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L.bars);
    int* misc = reinterpret_cast<int*>(smem + L.misc);
    uint64_t* xchg = reinterpret_cast<uint64_t*>(smem + L.xchg);
    const int bh = blockIdx.y;
    const int b = bh / a.Hkv;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    if (t == 0) {
        for (int w = 0; w < 8; ++w) mbar_init(&bars[w], 1);
        fence_barrier_init();
    }
    const int n = __ldg(a.seq_lens + b);
    grid_dep_wait();     // q~ and the summary of a block closed by this step
    grid_dep_launch();   // the attention kernel may start its set-up
    if (bad_len(n, a)) return;   // recorded by the prep kernel
    const int C = (n - 1) / kBlk;
    const int K = a.topk;
    const int Kc = K > 0 ? K : 1;
    const int m0 = blockIdx.x * kDecScoreChunk;
    const int rows_cta = max(0, min(kDecScoreChunk, C - m0));
    __syncthreads();
    uint32_t key = 0;
    if (rows_cta > 0 && K > 0 && C > K) {
        if (t < DSEL / 8) qs[t] = __ldg(reinterpret_cast<const uint4*>(a.qt) + static_cast<size_t>(bh) * (DSEL / 8) + t);
        const int r0 = m0 + warp * 32;
        const int rows = max(0, min(32, C - r0));
        if (rows > 0 && lane == 0) {
            const uint32_t bytes = static_cast<uint32_t>(rows) * kRowBytes;
            mbar_arrive_expect_tx(&bars[warp], bytes);
            bulk_load(stage + warp * kSlab,
                      static_cast<const bf16*>(a.Ksum) + (static_cast<size_t>(bh) * a.max_blocks + r0) * DSEL, bytes,
                      &bars[warp]);
        }
        __syncthreads();   // q~ in shared memory
        if (rows > 0) {
            const bool ok = mbar_wait_drain(&bars[warp], 0, limit, status);
            if (ok && lane < rows) {
                const uint4* krow = reinterpret_cast<const uint4*>(stage + warp * kSlab + lane * kRowBytes);
                constexpr int NCH = DSEL / 8;
                uint64_t acc = 0;
#pragma unroll
                for (int j = 0; j < NCH; ++j) {
                    const int c = (j + lane) & (NCH - 1);   // rotated: a quarter warp hits distinct banks
                    const uint4 kv = krow[c], qv = qs[c];
                    acc = fma_f32x2(f32x2(bf_lo(kv.x), bf_hi(kv.x)), f32x2(bf_lo(qv.x), bf_hi(qv.x)), acc);
                    acc = fma_f32x2(f32x2(bf_lo(kv.y), bf_hi(kv.y)), f32x2(bf_lo(qv.y), bf_hi(qv.y)), acc);
                    acc = fma_f32x2(f32x2(bf_lo(kv.z), bf_hi(kv.z)), f32x2(bf_lo(qv.z), bf_hi(qv.z)), acc);
                    acc = fma_f32x2(f32x2(bf_lo(kv.w), bf_hi(kv.w)), f32x2(bf_lo(qv.w), bf_hi(qv.w)), acc);
                }
                float s0, s1;
                f32x2_split(acc, s0, s1);
                key = order_key((s0 + s1) * score_scale);
            }
        }
        // local Top-K of this CTA's blocks: sort the distinct keys (score key, then
        // the lower block first) and keep those at or above the K-th
        bool take = t < rows_cta && key != 0;
        if (rows_cta > K) {
            const uint64_t comp = (static_cast<uint64_t>(key) << 32) | (0xffffffffu - static_cast<uint32_t>(t));
            const uint64_t sorted = bitonic256_desc(comp, xchg);
            __syncthreads();
            if (t == K - 1) xchg[0] = sorted;
            __syncthreads();
            take = take && comp >= xchg[0];
        }
        // compact the kept blocks in block order into this CTA's K candidate slots
        const unsigned bal = __ballot_sync(0xffffffffu, take);
        if (lane == 0) misc[8 + warp] = __popc(bal);
        __syncthreads();
        int off = 0, total = 0;
#pragma unroll
        for (int w = 0; w < 8; ++w) {
            const int c = misc[8 + w];
            off += w < warp ? c : 0;
            total += c;
        }
        const size_t cbase = (static_cast<size_t>(bh) * a.nsplit_s + blockIdx.x) * Kc;
        if (take) {
            const int pos = off + __popc(bal & ((1u << lane) - 1u));
            a.cand_key[cbase + pos] = key;
            a.cand_idx[cbase + pos] = m0 + t;
        }
        for (int e = total + t; e < Kc; e += kScoreThreads) {
            a.cand_key[cbase + e] = 0;
            a.cand_idx[cbase + e] = -1;
        }
    } else if (K > 0 && C > K) {
        // no blocks in this CTA's range: empty candidate slots
        const size_t cbase = (static_cast<size_t>(bh) * a.nsplit_s + blockIdx.x) * Kc;
        for (int e = t; e < Kc; e += kScoreThreads) {
            a.cand_key[cbase + e] = 0;
            a.cand_idx[cbase + e] = -1;
        }
    }
    // the last CTA of the group to finish selects
    __threadfence();
    __syncthreads();
    if (t == 0) {
        const int old = atomicAdd(a.cnt_sel + bh, 1);
        misc[0] = old == static_cast<int>(gridDim.x) - 1;
    }
    __syncthreads();
    if (!misc[0]) return;
    __threadfence();
    if (t == 0) a.cnt_sel[bh] = 0;   // zero again for the next launch
    int32_t* lst = a.list + static_cast<size_t>(bh) * 64;
    int32_t* so = a.sel_idx ? a.sel_idx + static_cast<size_t>(bh) * K : nullptr;
    if (C <= K) {   // short history: every historical block is kept
        for (int e = t; e < K; e += kScoreThreads) {
            if (e < C) lst[e] = e;
            if (so) so[e] = e < C ? e : -1;
        }
        if (t == 0) a.list_n[bh] = C;
        return;
    }
    if (K == 0) {
        if (t == 0) a.list_n[bh] = 0;
        return;
    }
    const size_t gbase = static_cast<size_t>(bh) * a.nsplit_s * Kc;
    if (C <= kDecScoreChunk) {
        // one CTA held every block: its local Top-K is the group's, already in block order
        for (int e = t; e < K; e += kScoreThreads) {
            const int m = __ldcg(a.cand_idx + gbase + e);
            lst[e] = m;
            if (so) so[e] = m;
        }
        if (t == 0) a.list_n[bh] = K;
        return;
    }
    const int M = ((C + kDecScoreChunk - 1) / kDecScoreChunk) * Kc;   // the splits that held blocks
    uint32_t* ckeys = reinterpret_cast<uint32_t*>(stage);
    int32_t* cidx = reinterpret_cast<int32_t*>(stage) + M;
    for (int i = t; i < M; i += kScoreThreads) {
        ckeys[i] = __ldcg(a.cand_key + gbase + i);
        cidx[i] = __ldcg(a.cand_idx + gbase + i);
    }
    select_candidates(a, bh, M, ckeys, cidx, reinterpret_cast<int*>(smem + L.hist),
                      reinterpret_cast<int*>(smem + L.scan), misc + 1);
}

// ---------------------------------------------------------------- attention

// Shared-memory layout of the attention kernel for a ring of nst stages.
struct AttnLayout {
    size_t tile, q32, ps, red, alpha, lsum, bars, misc, ent, total;
};
__host__ __device__ inline AttnLayout attn_layout(int D, int G, int nst, int bpc) {
    AttnLayout L;
    L.tile = static_cast<size_t>(kBlk) * D * 2;     // one K or V page slice
    L.q32 = nst * 2 * L.tile;                        // fp32 queries [G][D]
    L.ps = L.q32 + static_cast<size_t>(G) * D * 4;   // probabilities [G][64]
    L.red = L.ps + static_cast<size_t>(G) * 64 * 4;  // [8 warps][8]
    L.alpha = L.red + 64 * 4;                        // [8], then merge max [8] and sum [8]
    L.lsum = L.alpha + 32 * 4;                       // [8 warps][8]
    L.bars = L.lsum + 64 * 4;                        // nst mbarriers
    L.misc = L.bars + 64;                            // flag
    L.ent = L.misc + 64;                             // entries: block, page (2 ints each)
    L.total = L.ent + static_cast<size_t>(bpc) * 8;
    return L;
}

// grid (nsplit_a, B*Hkv), a programmatic dependent of the score kernel (of the
// prep kernel in dense mode).  The group's list is the current block c first,
// then the kept blocks in ascending order (dense: blocks 0 .. c-1); this CTA
// takes entries [x*bpc, (x+1)*bpc).
template <int D, int G>
__global__ void __launch_bounds__(kAttnThreads) dec_attn_kernel(DecodeArgs a, int* status, long long limit,
                                                                float scale_log2) {
    constexpr int kNW = D / 2;                          // bf16 pairs per row
    constexpr int NQG = kAttnThreads / 64;              // head groups in the score step
    constexpr int HP = (G + NQG - 1) / NQG;             // heads per thread in the score step
    constexpr int NHG = kAttnThreads / kNW;             // head groups in the PV step
    constexpr int HPV = (G + NHG - 1) / NHG;            // heads per thread in the PV step
    constexpr int NCH = D / 8;                          // 16-byte chunks per row
    extern __shared__ __align__(128) uint8_t smem[];
    const int nst = a.nst;
    const AttnLayout Ly = attn_layout(D, G, nst, a.bpc);
    const int kTile = static_cast<int>(Ly.tile);
    float* q32 = reinterpret_cast<float*>(smem + Ly.q32);
    float* Ps = reinterpret_cast<float*>(smem + Ly.ps);
    float* red = reinterpret_cast<float*>(smem + Ly.red);
    float* alpha_s = reinterpret_cast<float*>(smem + Ly.alpha);
    float* lsum = reinterpret_cast<float*>(smem + Ly.lsum);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + Ly.bars);
    int* misc = reinterpret_cast<int*>(smem + Ly.misc);
    int* ent = reinterpret_cast<int*>(smem + Ly.ent);

    const int bh = blockIdx.y;
    const int b = bh / a.Hkv, g = bh - b * a.Hkv;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int n = __ldg(a.seq_lens + b);
    const bool bad = bad_len(n, a);   // recorded by the prep kernel
    const int c = bad ? 0 : (n - 1) / kBlk;
    const int j0 = blockIdx.x * a.bpc;
    const size_t head_off = static_cast<size_t>(g) * kBlk * D;   // this KV head's slice inside a page
    auto issue = [&](int jj) {
        const int s = jj % nst;
        const int page = ent[2 * jj + 1];
        uint8_t* dst = smem + s * 2 * kTile;
        if (page < 0) {
            mbar_arrive(&full[s]);
            return;
        }
        const size_t off = static_cast<size_t>(page) * a.Hkv * kBlk * D + head_off;
        mbar_arrive_expect_tx(&full[s], 2 * kTile);
        bulk_load(dst, static_cast<const bf16*>(a.K_cache) + off, kTile, &full[s]);
        bulk_load(dst + kTile, static_cast<const bf16*>(a.V_cache) + off, kTile, &full[s]);
    };

    // --- set-up that needs nothing from the preceding kernel
    if (t == 0) {
        for (int s = 0; s < nst; ++s) mbar_init(&full[s], 1);
        fence_barrier_init();
    }
    const bf16* qg = static_cast<const bf16*>(a.q) + (static_cast<size_t>(b) * a.Hq + static_cast<size_t>(g) * G) * D;
    for (int e = t; e < G * D; e += kAttnThreads) q32[e] = __bfloat162float(qg[e]);
    grid_dep_wait();   // the kept list
    if (bad) return;
    const int L = (a.dense ? c : __ldg(a.list_n + bh)) + 1;
    const int cnt = max(0, min(j0 + a.bpc, L) - j0);
    // (the current block, entry 0, is written by the preceding kernel, so every
    // page load waits for the grid dependency)
    const int first = 0;
    for (int jj = first + t; jj < cnt; jj += kAttnThreads) {
        const int j = j0 + jj;
        const int blk = j == 0 ? c : (a.dense ? j - 1 : __ldg(a.list + static_cast<size_t>(bh) * 64 + j - 1));
        int page = __ldg(a.block_table + static_cast<size_t>(b) * a.max_blocks + blk);
        if (page < 0 || page >= a.num_pages) {
            atomicExch(status, kStatusBadInput);
            page = -1;
        }
        ent[2 * jj] = blk;
        ent[2 * jj + 1] = page;
    }
    __syncthreads();
    int issued = first;
    if (t == 0) {
        for (; issued < min(cnt, nst); ++issued) issue(issued);
    }

    const int k = t & 63, hh = t >> 6;           // score step: key k, heads hh*HP + u (keys of a head in warps 2hh, 2hh+1)
    const int wi = t % kNW, hg = t / kNW;        // PV step: column pair wi, heads hg*HPV + u
    float m_run[HP], l_part[HP];
#pragma unroll
    for (int u = 0; u < HP; ++u) {
        m_run[u] = -CUDART_INF_F;
        l_part[u] = 0.f;
    }
    uint64_t acc[HPV];
#pragma unroll
    for (int u = 0; u < HPV; ++u) acc[u] = 0;

    bool ok = true;
    int jj = 0;
    for (; jj < cnt; ++jj) {
        const int s = jj % nst;
        const bool got = mbar_wait_drain(&full[s], (jj / nst) & 1, limit, status);
        if (!__syncthreads_and(got)) {
            ok = false;
            break;
        }
        const int page = ent[2 * jj + 1];
        const int nvalid = page < 0 ? 0 : (ent[2 * jj] == c ? n - c * kBlk : kBlk);
        const uint8_t* Kt = smem + s * 2 * kTile;
        const uint8_t* Vt = Kt + kTile;

        // z = scale * q_h . k for this thread's key and heads (log2 units)
        float z[HP];
        {
            uint64_t az[HP];
#pragma unroll
            for (int u = 0; u < HP; ++u) az[u] = 0;
            const uint4* krow = reinterpret_cast<const uint4*>(Kt + k * D * 2);
#pragma unroll
            for (int jc = 0; jc < NCH; ++jc) {
                const int cc = (jc + k) & (NCH - 1);    // rotated chunk: no bank conflicts across keys
                const uint4 kv = krow[cc];
                const uint64_t k01 = f32x2(bf_lo(kv.x), bf_hi(kv.x));
                const uint64_t k23 = f32x2(bf_lo(kv.y), bf_hi(kv.y));
                const uint64_t k45 = f32x2(bf_lo(kv.z), bf_hi(kv.z));
                const uint64_t k67 = f32x2(bf_lo(kv.w), bf_hi(kv.w));
#pragma unroll
                for (int u = 0; u < HP; ++u) {
                    const int h = hh * HP + u;
                    if (h < G) {
                        const float4 qa = *reinterpret_cast<const float4*>(q32 + h * D + cc * 8);
                        const float4 qb = *reinterpret_cast<const float4*>(q32 + h * D + cc * 8 + 4);
                        az[u] = fma_f32x2(k01, f32x2(qa.x, qa.y), az[u]);
                        az[u] = fma_f32x2(k23, f32x2(qa.z, qa.w), az[u]);
                        az[u] = fma_f32x2(k45, f32x2(qb.x, qb.y), az[u]);
                        az[u] = fma_f32x2(k67, f32x2(qb.z, qb.w), az[u]);
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < HP; ++u) {
                float z0, z1;
                f32x2_split(az[u], z0, z1);
                z[u] = k < nvalid ? (z0 + z1) * scale_log2 : -CUDART_INF_F;
            }
        }
#pragma unroll
        for (int u = 0; u < HP; ++u) {
            const float mx = warp_max(z[u]);
            if (lane == 0) red[warp * 8 + u] = mx;
        }
        __syncthreads();
#pragma unroll
        for (int u = 0; u < HP; ++u) {
            const int h = hh * HP + u;
            if (h < G) {
                const float mb = fmaxf(red[(2 * hh) * 8 + u], red[(2 * hh + 1) * 8 + u]);
                const float m_new = fmaxf(m_run[u], mb);
                const float alpha = m_run[u] == -CUDART_INF_F ? 0.f : fast_exp2(m_run[u] - m_new);
                const float p = z[u] == -CUDART_INF_F ? 0.f : fast_exp2(z[u] - m_new);
                l_part[u] = l_part[u] * alpha + p;
                m_run[u] = m_new;
                Ps[h * 64 + k] = p;
                if (k == 0) alpha_s[h] = alpha;
            }
        }
        __syncthreads();
        // O_h = alpha_h O_h + sum_k p_hk v_k for this thread's column pair
#pragma unroll
        for (int u = 0; u < HPV; ++u) {
            const int h = hg * HPV + u;
            if (h < G) {
                const float al = alpha_s[h];
                acc[u] = fma_f32x2(acc[u], f32x2(al, al), 0ull);
            }
        }
        const uint32_t* V32 = reinterpret_cast<const uint32_t*>(Vt);
#pragma unroll 4
        for (int kk = 0; kk < nvalid; ++kk) {
            const uint32_t w = V32[kk * kNW + wi];
            const uint64_t v2 = f32x2(bf_lo(w), bf_hi(w));
#pragma unroll
            for (int u = 0; u < HPV; ++u) {
                const int h = hg * HPV + u;
                if (h < G) {
                    const float p = Ps[h * 64 + kk];
                    acc[u] = fma_f32x2(f32x2(p, p), v2, acc[u]);
                }
            }
        }
        __syncthreads();   // the stage, Ps and red are free
        if (t == 0 && issued < cnt) {
            fence_proxy_async_smem();
            issue(issued);
            ++issued;
        }
    }
    if (!ok) {
        // let copies still in flight land before the CTA exits; report nothing
        if (t == 0)
            for (int q = jj; q < issued; ++q) mbar_wait_drain(&full[q % nst], (q / nst) & 1, limit, status);
#pragma unroll
        for (int u = 0; u < HP; ++u) {
            m_run[u] = -CUDART_INF_F;
            l_part[u] = 0.f;
        }
#pragma unroll
        for (int u = 0; u < HPV; ++u) acc[u] = 0;
    }

    // partial (max, sum, output) of this CTA per head
#pragma unroll
    for (int u = 0; u < HP; ++u) {
        const float ls = warp_sum(l_part[u]);
        if (lane == 0) lsum[warp * 8 + u] = ls;
    }
    __syncthreads();
    float* part = a.part + (static_cast<size_t>(bh) * a.nsplit_a + blockIdx.x) * G * (D + 2);
    if (k == 0) {
#pragma unroll
        for (int u = 0; u < HP; ++u) {
            const int h = hh * HP + u;
            if (h < G) {
                part[h * (D + 2)] = m_run[u];
                part[h * (D + 2) + 1] = lsum[(2 * hh) * 8 + u] + lsum[(2 * hh + 1) * 8 + u];
            }
        }
    }
#pragma unroll
    for (int u = 0; u < HPV; ++u) {
        const int h = hg * HPV + u;
        if (h < G) {
            float o0, o1;
            f32x2_split(acc[u], o0, o1);
            part[h * (D + 2) + 2 + 2 * wi] = o0;
            part[h * (D + 2) + 3 + 2 * wi] = o1;
        }
    }
    __threadfence();
    __syncthreads();
    if (t == 0) {
        const int old = atomicAdd(a.cnt_attn + bh, 1);
        misc[0] = old == static_cast<int>(gridDim.x) - 1;
    }
    __syncthreads();
    if (!misc[0]) return;
    __threadfence();
    if (t == 0) a.cnt_attn[bh] = 0;   // zero again for the next launch

    // Merge the partials of every head (only the splits the list reached).  The
    // (max, sum) pairs are staged in the free ring first, turned into weights
    // exp2(m_x - M) per head, then every thread sums its columns over the splits
    // with all loads independent.
    const int used = (L + a.bpc - 1) / a.bpc;
    const float* pg = a.part + static_cast<size_t>(bh) * a.nsplit_a * G * (D + 2);
    float* mw = reinterpret_cast<float*>(smem);    // [used][G][2]
    float* mM = alpha_s + 8;                       // [G] max
    float* mL = alpha_s + 16;                      // [G] sum
    for (int i = t; i < used * G; i += kAttnThreads) {
        const float* px = pg + static_cast<size_t>(i) * (D + 2);
        mw[2 * i] = __ldcg(px);
        mw[2 * i + 1] = __ldcg(px + 1);
    }
    __syncthreads();
    if (t < G) {
        float M = -CUDART_INF_F;
        for (int x = 0; x < used; ++x) M = fmaxf(M, mw[2 * (x * G + t)]);
        float ls = 0.f;
        for (int x = 0; x < used; ++x) {
            const float mx = mw[2 * (x * G + t)];
            const float w = mx == -CUDART_INF_F ? 0.f : fast_exp2(mx - M);
            ls = fmaf(w, mw[2 * (x * G + t) + 1], ls);
            mw[2 * (x * G + t)] = w;
        }
        mM[t] = M;
        mL[t] = ls;
    }
    __syncthreads();
#pragma unroll
    for (int u = 0; u < HPV; ++u) {
        const int h = hg * HPV + u;
        if (h >= G) continue;
        float o0 = 0.f, o1 = 0.f;
#pragma unroll 16
        for (int x = 0; x < used; ++x) {
            const float2 v = __ldcg(reinterpret_cast<const float2*>(pg + (static_cast<size_t>(x) * G + h) * (D + 2) + 2) + wi);
            const float w = mw[2 * (x * G + h)];
            o0 = fmaf(w, v.x, o0);
            o1 = fmaf(w, v.y, o1);
        }
        const float inv = 1.f / mL[h];
        const size_t orow = (static_cast<size_t>(b) * a.Hq + static_cast<size_t>(g) * G + h) * D;
        reinterpret_cast<uint32_t*>(static_cast<bf16*>(a.O) + orow)[wi] = pack_bf16x2(o0 * inv, o1 * inv);
        if (a.LSE != nullptr && wi == 0)
            a.LSE[static_cast<size_t>(b) * a.Hq + static_cast<size_t>(g) * G + h] = (mM[h] + log2f(mL[h])) / kLog2e;
    }
}

// -------------------------------------------------- attention on tensor cores (d = 128)
//
// A step takes two pages (128 keys) of the CTA's list:
//   S^T[128 keys][16] = Kpair[128 x 128] . Qpad[16 x 128]^T          tcgen05, M=128 N=16, K-major A and B
//   softmax over the 128 keys of every head (TMEM lane = key)
//   O^T[128 d][16]    = Vpair^T[128 d x 128 keys] . Ppad[16 x 128]^T  tcgen05, A MN-major (V as stored)
// Q and P are padded from G <= 8 heads to N = 16 rows of zeros.  K and V tiles
// sit in shared memory as [d half][128 keys][128 B] with the 128-byte swizzle,
// written by four 64 x 64 TMA boxes each (page 0 in rows 0-63, page 1 in
// rows 64-127); Q is [d half][16][128 B], P [key half][16][128 B], both
// swizzled by the threads that write them.  Every step's O^T is a fresh
// accumulator that the threads fold into registers (thread t owns row d = t)
// with the online-softmax rescale.

constexpr int kTcThreads = 128;
constexpr int kTcTile = 2 * 128 * 128;          // bytes of one K (or V) tile of a step
constexpr int kTcStage = 2 * kTcTile;           // K and V
constexpr uint32_t kTcTmemCols = 64;            // S^T in columns 0-15, O^T in 32-47

struct TcLayout {
    size_t q, p, red, alpha, lsum, bars, misc, ent, total;
};
__host__ __device__ inline TcLayout tc_layout(int nst, int bpc) {
    TcLayout L;
    L.q = static_cast<size_t>(nst) * kTcStage;   // 4096: [2][16][128 B]
    L.p = L.q + 4096;                            // 4096: [2][16][128 B]
    L.red = L.p + 4096;                          // [4 warps][16]
    L.alpha = L.red + 64 * 4;                    // [16] alpha, then merge max [16] and sum [16]
    L.lsum = L.alpha + 48 * 4;                   // [4 warps][16]
    L.bars = L.lsum + 64 * 4;                    // full[4], qk, pv
    L.misc = L.bars + 64;                        // flag, TMEM base
    L.ent = L.misc + 64;                         // entries: block, page
    L.total = L.ent + static_cast<size_t>(bpc) * 8 + 1024;   // + alignment slack
    return L;
}

// TMA loads of list entry e (a page of step e/2) into the step's stage: K and V,
// two 64 x 64 boxes each (the two halves of d); nothing for a missing page.
__device__ __forceinline__ void tc_load_page(uint8_t* smem, int nst, const int* ent, int e, const CUtensorMap* mapK,
                                             const CUtensorMap* mapV, uint64_t* full, int Hkv, int g) {
    const int page = ent[2 * e + 1];
    if (page < 0) return;
    const int s = (e >> 1) % nst, pg = e & 1;
    uint8_t* st = smem + static_cast<size_t>(s) * kTcStage;
    const int row = page * Hkv + g;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        tma_load_3d(st + h * 16384 + pg * 8192, mapK, &full[s], h * 64, 0, row);
        tma_load_3d(st + kTcTile + h * 16384 + pg * 8192, mapV, &full[s], h * 64, 0, row);
    }
}
__device__ __forceinline__ uint32_t tc_page_bytes(const int* ent, int e) {
    return ent[2 * e + 1] >= 0 ? 4u * 8192u : 0u;
}

template <int G>
__global__ void __launch_bounds__(kTcThreads) dec_attn_tc_kernel(const __grid_constant__ CUtensorMap mapK,
                                                                 const __grid_constant__ CUtensorMap mapV,
                                                                 DecodeArgs a, int* status, long long limit,
                                                                 float scale_log2) {
    constexpr int D = 128;
    constexpr uint32_t IDESC_S = idesc_bf16(128, 16, 0, 0);
    constexpr uint32_t IDESC_O = idesc_bf16(128, 16, 1, 0);
    extern __shared__ __align__(1024) uint8_t dsm[];
    // the swizzled tiles need 1024-byte alignment
    uint8_t* smem = dsm + ((1024u - (smem_u32(dsm) & 1023u)) & 1023u);
    const int nst = a.nst;
    const TcLayout Ly = tc_layout(nst, a.bpc);
    uint8_t* qs = smem + Ly.q;
    uint8_t* ps = smem + Ly.p;
    float* red = reinterpret_cast<float*>(smem + Ly.red);
    float* mM = reinterpret_cast<float*>(smem + Ly.alpha) + 16;
    float* mL = reinterpret_cast<float*>(smem + Ly.alpha) + 32;
    float* lsum = reinterpret_cast<float*>(smem + Ly.lsum);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + Ly.bars);
    uint64_t* qk_bar = full + 4;
    uint64_t* pv_bar = full + 5;
    int* misc = reinterpret_cast<int*>(smem + Ly.misc);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc + 4);
    int* ent = reinterpret_cast<int*>(smem + Ly.ent);

    const int bh = blockIdx.y;
    const int b = bh / a.Hkv, g = bh - b * a.Hkv;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int n = __ldg(a.seq_lens + b);
    const bool bad = bad_len(n, a);   // recorded by the prep kernel
    const int c = bad ? 0 : (n - 1) / kBlk;
    const int j0 = blockIdx.x * a.bpc;

#define SAS_TC_LOAD(e) tc_load_page(smem, nst, ent, (e), &mapK, &mapV, full, a.Hkv, g)

    // --- set-up that needs nothing from the preceding kernel
    if (t == 0) {
        for (int s = 0; s < nst; ++s) mbar_init(&full[s], 1);
        mbar_init(qk_bar, 1);
        mbar_init(pv_bar, 1);
        fence_barrier_init();
        tma_prefetch_desc(&mapK);
        tma_prefetch_desc(&mapV);
        // the current block (entry 0) was appended by the prep kernel, which the
        // score kernel waited for before letting this grid start, so its page can
        // load now (dense mode: the prep kernel precedes this one directly)
        if (!bad && j0 == 0 && !a.dense) {
            int page = __ldg(a.block_table + static_cast<size_t>(b) * a.max_blocks + c);
            if (page < 0 || page >= a.num_pages) page = -1;   // recorded by the prep kernel
            ent[0] = c;
            ent[1] = page;
            mbar_expect_tx(&full[0], tc_page_bytes(ent, 0));
            SAS_TC_LOAD(0);
        }
    }
    if (warp == 0) {
        tmem_alloc(tmem_slot, kTcTmemCols);
        tmem_relinquish();
    }
    // Q rows (zero past G) and P (rows past G stay zero), 16-byte chunks swizzled
    const bf16* qg = static_cast<const bf16*>(a.q) + (static_cast<size_t>(b) * a.Hq + static_cast<size_t>(g) * G) * D;
    for (int i = t; i < 2 * 16 * 8; i += kTcThreads) {
        const int h = i >> 7, row = (i >> 3) & 15, ch = i & 7;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (row < G) v = __ldg(reinterpret_cast<const uint4*>(qg + row * D + h * 64 + ch * 8));
        *reinterpret_cast<uint4*>(qs + h * 2048 + row * 128 + ((ch ^ (row & 7)) << 4)) = v;
        *reinterpret_cast<uint4*>(ps + h * 2048 + row * 128 + (ch << 4)) = make_uint4(0, 0, 0, 0);
    }
    grid_dep_wait();   // the kept list
    const int L = bad ? 0 : (a.dense ? c : __ldg(a.list_n + bh)) + 1;
    const int cnt = bad ? 0 : max(0, min(j0 + a.bpc, L) - j0);
    const int first = (j0 == 0 && !a.dense) ? 1 : 0;   // entries set up before the wait
    for (int jj = first + t; jj < cnt; jj += kTcThreads) {
        const int j = j0 + jj;
        const int blk = j == 0 ? c : (a.dense ? j - 1 : __ldg(a.list + static_cast<size_t>(bh) * 64 + j - 1));
        int page = __ldg(a.block_table + static_cast<size_t>(b) * a.max_blocks + blk);
        if (page < 0 || page >= a.num_pages) {
            atomicExch(status, kStatusBadInput);
            page = -1;
        }
        ent[2 * jj] = blk;
        ent[2 * jj + 1] = page;
    }
    fence_proxy_async_smem();   // Q and P writes before the tensor cores read them
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const int steps = (cnt + 1) >> 1;
    int issued = 0;   // steps whose loads are issued (thread 0)
    if (t == 0) {
        for (; issued < min(steps, nst); ++issued) {
            const int e0 = 2 * issued, e1 = e0 + 1;
            uint32_t bytes = 0;
            if (e0 >= first) bytes += tc_page_bytes(ent, e0);
            if (e1 < cnt) bytes += tc_page_bytes(ent, e1);
            mbar_arrive_expect_tx(&full[issued], bytes);
            if (e0 >= first) SAS_TC_LOAD(e0);
            if (e1 < cnt) SAS_TC_LOAD(e1);
        }
    }

    float m_run[G], l_part[G], o[G];
#pragma unroll
    for (int h = 0; h < G; ++h) {
        m_run[h] = -CUDART_INF_F;
        l_part[h] = 0.f;
        o[h] = 0.f;
    }
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    bool ok = true;
    int j = 0;
    int pending = 0;   // 1: a QK commit outstanding, 2: a PV commit outstanding
    for (; j < steps; ++j) {
        const int s = j % nst;
        uint8_t* st = smem + static_cast<size_t>(s) * kTcStage;
        const bool got = mbar_wait_drain(&full[s], (j / nst) & 1, limit, status);
        if (!__syncthreads_and(got)) {
            ok = false;
            break;
        }
        // rows of a page past its valid keys (or of a missing page) get zero values,
        // so P = 0 there cannot meet a non-finite V
        const int e0 = 2 * j, e1 = e0 + 1;
        const int nv0 = ent[2 * e0 + 1] < 0 ? 0 : (ent[2 * e0] == c ? n - c * kBlk : kBlk);
        const int nv1 = (e1 >= cnt || ent[2 * e1 + 1] < 0) ? 0 : (ent[2 * e1] == c ? n - c * kBlk : kBlk);
        if (nv0 < kBlk || nv1 < kBlk) {
            for (int i = t; i < 2 * 2 * 64 * 8; i += kTcThreads) {   // (page, half, row, chunk)
                const int pg = i >> 10, h = (i >> 9) & 1, row = (i >> 3) & 63, ch = i & 7;
                if (row >= (pg ? nv1 : nv0))
                    *reinterpret_cast<uint4*>(st + kTcTile + h * 16384 + pg * 8192 + row * 128 + (ch << 4)) =
                        make_uint4(0, 0, 0, 0);
            }
            fence_proxy_async_smem();
            __syncthreads();
        }
        if (t == 0) {
            tc_fence_after();
            const uint32_t kb = smem_u32(st), qb = smem_u32(qs);
#pragma unroll
            for (int k = 0; k < D / 16; ++k) {
                const uint64_t da = smem_desc_sw128(kb + (k >> 2) * 16384 + (k & 3) * 32, 16, 1024);
                const uint64_t db = smem_desc_sw128(qb + (k >> 2) * 2048 + (k & 3) * 32, 16, 1024);
                umma_bf16(tmem, da, db, IDESC_S, k > 0);
            }
            umma_commit(qk_bar);
        }
        pending = 1;
        if (!mbar_wait_drain(qk_bar, j & 1, limit, status)) ok = false;
        if (!__syncthreads_and(ok)) break;
        pending = 0;
        tc_fence_after();
        uint32_t sr[16];
        tmem_ld16(lane_base, sr);
        tmem_wait_ld();
        const int key = t;                           // TMEM lane = key of the pair
        const bool valid = key < 64 ? key < nv0 : key - 64 < nv1;
        float z[G];
#pragma unroll
        for (int h = 0; h < G; ++h) {
            z[h] = valid ? __uint_as_float(sr[h]) * scale_log2 : -CUDART_INF_F;
            const float mx = warp_max(z[h]);
            if (lane == 0) red[warp * 16 + h] = mx;
        }
        __syncthreads();
        float alpha[G];
#pragma unroll
        for (int h = 0; h < G; ++h) {
            const float mb = fmaxf(fmaxf(red[h], red[16 + h]), fmaxf(red[32 + h], red[48 + h]));
            const float m_new = fmaxf(m_run[h], mb);
            alpha[h] = m_run[h] == -CUDART_INF_F ? 0.f : fast_exp2(m_run[h] - m_new);
            const float pr = z[h] == -CUDART_INF_F ? 0.f : fast_exp2(z[h] - m_new);
            l_part[h] = l_part[h] * alpha[h] + pr;
            m_run[h] = m_new;
            const int kh = key >> 6, ch = (key & 63) >> 3;
            *reinterpret_cast<bf16*>(ps + kh * 2048 + h * 128 + ((ch ^ (h & 7)) << 4) + ((key & 7) << 1)) =
                __float2bfloat16_rn(pr);
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (t == 0) {
            tc_fence_after();
            const uint32_t vb = smem_u32(st + kTcTile), pb = smem_u32(ps);
#pragma unroll
            for (int k = 0; k < 128 / 16; ++k) {
                const uint64_t da = smem_desc_sw128(vb + k * 2048, 16384, 1024);
                const uint64_t db = smem_desc_sw128(pb + (k >> 2) * 2048 + (k & 3) * 32, 16, 1024);
                umma_bf16(tmem + 32, da, db, IDESC_O, k > 0);
            }
            umma_commit(pv_bar);
        }
        pending = 2;
        if (!mbar_wait_drain(pv_bar, j & 1, limit, status)) ok = false;
        if (!__syncthreads_and(ok)) break;
        pending = 0;
        tc_fence_after();
        uint32_t orr[16];
        tmem_ld16(lane_base + 32, orr);
        tmem_wait_ld();
#pragma unroll
        for (int h = 0; h < G; ++h) o[h] = fmaf(o[h], alpha[h], __uint_as_float(orr[h]));
        tc_fence_before();
        __syncthreads();   // the stage, P and the TMEM columns are free
        if (t == 0 && issued < steps) {
            const int e0 = 2 * issued, e1 = e0 + 1;
            const int s2 = issued % nst;
            uint32_t bytes = tc_page_bytes(ent, e0);
            if (e1 < cnt) bytes += tc_page_bytes(ent, e1);
            mbar_arrive_expect_tx(&full[s2], bytes);
            SAS_TC_LOAD(e0);
            if (e1 < cnt) SAS_TC_LOAD(e1);
            ++issued;
        }
    }
    if (!ok) {
        // let the tensor cores and the copies in flight finish before leaving
        if (t == 0) {
            if (pending == 1) mbar_wait_drain(qk_bar, j & 1, limit, status);
            if (pending == 2) mbar_wait_drain(pv_bar, j & 1, limit, status);
            for (int q = j; q < issued; ++q) mbar_wait_drain(&full[q % nst], (q / nst) & 1, limit, status);
        }
#pragma unroll
        for (int h = 0; h < G; ++h) {
            m_run[h] = -CUDART_INF_F;
            l_part[h] = 0.f;
            o[h] = 0.f;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, kTcTmemCols);
    }

    // partial (max, sum, output) of this CTA per head
#pragma unroll
    for (int h = 0; h < G; ++h) {
        const float ls = warp_sum(l_part[h]);
        if (lane == 0) lsum[warp * 16 + h] = ls;
    }
    __syncthreads();
    float* part = a.part + (static_cast<size_t>(bh) * a.nsplit_a + blockIdx.x) * G * (D + 2);
#pragma unroll
    for (int h = 0; h < G; ++h) {
        if (t == 0) {
            part[h * (D + 2)] = m_run[h];
            part[h * (D + 2) + 1] = lsum[h] + lsum[16 + h] + lsum[32 + h] + lsum[48 + h];
        }
        part[h * (D + 2) + 2 + t] = o[h];
    }
    __threadfence();
    __syncthreads();
    if (t == 0) {
        const int old = atomicAdd(a.cnt_attn + bh, 1);
        misc[0] = old == static_cast<int>(gridDim.x) - 1;
    }
    __syncthreads();
    if (!misc[0]) return;
    __threadfence();
    if (t == 0) a.cnt_attn[bh] = 0;   // zero again for the next launch
    if (bad) return;

    // merge the partials of the splits the list reached
    const int used = (L + a.bpc - 1) / a.bpc;
    const float* pgp = a.part + static_cast<size_t>(bh) * a.nsplit_a * G * (D + 2);
    float* mw = reinterpret_cast<float*>(smem);    // [used][G][2], in the free stage
    for (int i = t; i < used * G; i += kTcThreads) {
        const float* px = pgp + static_cast<size_t>(i) * (D + 2);
        mw[2 * i] = __ldcg(px);
        mw[2 * i + 1] = __ldcg(px + 1);
    }
    __syncthreads();
    if (t < G) {
        float M = -CUDART_INF_F;
        for (int x = 0; x < used; ++x) M = fmaxf(M, mw[2 * (x * G + t)]);
        float ls = 0.f;
        for (int x = 0; x < used; ++x) {
            const float mx = mw[2 * (x * G + t)];
            const float w = mx == -CUDART_INF_F ? 0.f : fast_exp2(mx - M);
            ls = fmaf(w, mw[2 * (x * G + t) + 1], ls);
            mw[2 * (x * G + t)] = w;
        }
        mM[t] = M;
        mL[t] = ls;
    }
    __syncthreads();
#pragma unroll
    for (int h = 0; h < G; ++h) {
        float acc = 0.f;
#pragma unroll 8
        for (int x = 0; x < used; ++x)
            acc = fmaf(mw[2 * (x * G + h)], __ldcg(pgp + (static_cast<size_t>(x) * G + h) * (D + 2) + 2 + t), acc);
        const size_t orow = (static_cast<size_t>(b) * a.Hq + static_cast<size_t>(g) * G + h) * D;
        static_cast<bf16*>(a.O)[orow + t] = __float2bfloat16_rn(acc / mL[h]);
        if (a.LSE != nullptr && t == 0)
            a.LSE[static_cast<size_t>(b) * a.Hq + static_cast<size_t>(g) * G + h] = (mM[h] + log2f(mL[h])) / kLog2e;
    }
#undef SAS_TC_LOAD
}

// Launch with programmatic stream serialization: the kernel may start while
// the preceding kernel on the stream still runs (it waits with griddepcontrol).
template <class... KArgs, class... Args>
cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                             Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// Raises the kernel's dynamic shared-memory limit to what these arguments need
// (called when a handle is created, so that a captured step sets nothing).
template <int D, int G>
cudaError_t prepare_attn_dg(const DecodeArgs& a) {
    const size_t smem = attn_layout(D, G, a.nst, a.bpc).total;
    return ensure_smem_attr(reinterpret_cast<const void*>(dec_attn_kernel<D, G>), smem);
}

template <int D, int G>
cudaError_t launch_attn_dg(const DecodeArgs& a, const KernelEnv& env) {
    const size_t smem = attn_layout(D, G, a.nst, a.bpc).total;
    cudaError_t e = prepare_attn_dg<D, G>(a);
    if (e != cudaSuccess) return e;
    dim3 grid(a.nsplit_a, a.B * a.Hkv);
    return launch_dependent(dec_attn_kernel<D, G>, grid, dim3(kAttnThreads), smem, env.stream, a, env.status,
                            env.limit, a.sm_scale * kLog2e);
}

template <int G>
cudaError_t prepare_attn_tc(const DecodeArgs& a) {
    const size_t smem = tc_layout(a.nst, a.bpc).total;
    return ensure_smem_attr(reinterpret_cast<const void*>(dec_attn_tc_kernel<G>), smem);
}

template <int G>
cudaError_t launch_attn_tc(const DecodeArgs& a, const KernelEnv& env) {
    cudaError_t e = prepare_attn_tc<G>(a);
    if (e != cudaSuccess) return e;
    CUtensorMap mk, mv;
    const uint64_t rows = static_cast<uint64_t>(a.num_pages) * a.Hkv;
    if (make_tmap_bf16_3d(&mk, a.K_cache, 128, kBlk, rows, 64, kBlk) != 0) return cudaErrorInvalidValue;
    if (make_tmap_bf16_3d(&mv, a.V_cache, 128, kBlk, rows, 64, kBlk) != 0) return cudaErrorInvalidValue;
    dim3 grid(a.nsplit_a, a.B * a.Hkv);
    return launch_dependent(dec_attn_tc_kernel<G>, grid, dim3(kTcThreads), tc_layout(a.nst, a.bpc).total, env.stream,
                            mk, mv, a, env.status, env.limit, a.sm_scale * kLog2e);
}

template <int D>
cudaError_t launch_attn_d(const DecodeArgs& a, const KernelEnv& env) {
    if constexpr (D == 128) {
        switch (a.G) {
            case 1: return launch_attn_tc<1>(a, env);
            case 2: return launch_attn_tc<2>(a, env);
            case 4: return launch_attn_tc<4>(a, env);
            case 8: return launch_attn_tc<8>(a, env);
        }
    } else {
        switch (a.G) {
            case 1: return launch_attn_dg<D, 1>(a, env);
            case 2: return launch_attn_dg<D, 2>(a, env);
            case 4: return launch_attn_dg<D, 4>(a, env);
            case 8: return launch_attn_dg<D, 8>(a, env);
        }
    }
    return cudaErrorInvalidValue;
}

template <int D>
cudaError_t prepare_attn_d(const DecodeArgs& a) {
    if constexpr (D == 128) {
        switch (a.G) {
            case 1: return prepare_attn_tc<1>(a);
            case 2: return prepare_attn_tc<2>(a);
            case 4: return prepare_attn_tc<4>(a);
            case 8: return prepare_attn_tc<8>(a);
        }
    } else {
        switch (a.G) {
            case 1: return prepare_attn_dg<D, 1>(a);
            case 2: return prepare_attn_dg<D, 2>(a);
            case 4: return prepare_attn_dg<D, 4>(a);
            case 8: return prepare_attn_dg<D, 8>(a);
        }
    }
    return cudaErrorInvalidValue;
}

template <int DSEL>
cudaError_t prepare_score_d(const DecodeArgs& a) {
    const size_t smem = score_smem_layout(a.nsplit_s, a.topk, DSEL).total;
    return ensure_smem_attr(reinterpret_cast<const void*>(dec_score_kernel<DSEL>), smem);
}

template <int DSEL>
cudaError_t launch_score_d(const DecodeArgs& a, const KernelEnv& env) {
    const size_t smem = score_smem_layout(a.nsplit_s, a.topk, DSEL).total;
    cudaError_t e = prepare_score_d<DSEL>(a);
    if (e != cudaSuccess) return e;
    dim3 grid(a.nsplit_s, a.B * a.Hkv);
    return launch_dependent(dec_score_kernel<DSEL>, grid, dim3(kScoreThreads), smem, env.stream, a, env.status,
                            env.limit, static_cast<float>(1.0 / sqrt(static_cast<double>(DSEL))));
}

}  // namespace

void decode_attn_split(int max_len, int d, int* nsplit, int* bpc, int* nst) {
    int per;
    if (d == 128) {
        // tensor-core kernel: two pages (one 128-key step) per CTA for a SAS list;
        // long dense lists cut into at most 64 (128 past 2048 pages) pieces of
        // whole steps.  One stage, so that three CTAs share an SM and overlap one
        // another's loads (two stages and one CTA per SM measured slower).
        const int pieces = max_len <= 2048 ? 64 : 128;   // long lists: more CTAs pay for the larger merge
        per = max_len <= 96 ? 2 : 2 * ((max_len + 2 * pieces - 1) / (2 * pieces));
        *nst = 1;
    } else {
        // CUDA-core kernel: one page per CTA for a SAS list; long dense lists in
        // at most 64 pieces streamed through a 3-stage ring
        per = max_len <= 96 ? 1 : (max_len + 63) / 64;
        *nst = per < kStages ? per : kStages;
    }
    *bpc = per;
    *nsplit = (max_len + per - 1) / per;
}

size_t decode_score_smem(int nsplit, int topk, int d_sel) { return score_smem_layout(nsplit, topk, d_sel).total; }

size_t decode_attn_smem(int d, int G, int nst, int bpc) {
    return d == 128 ? tc_layout(nst, bpc).total : attn_layout(d, G, nst, bpc).total;
}

cudaError_t decode_prepare(const DecodeArgs& a) {
    cudaError_t e = cudaSuccess;
    if (!a.dense) e = a.d_sel == 128 ? prepare_score_d<128>(a) : prepare_score_d<64>(a);
    if (e == cudaSuccess) e = a.d == 128 ? prepare_attn_d<128>(a) : prepare_attn_d<64>(a);
    return e;
}

cudaError_t launch_decode_prep(const DecodeArgs& a, const KernelEnv& env) {
    dim3 grid(a.B * a.Hkv, a.dense ? 1 : 1 + (a.d_sel + 7) / 8);
    dec_prep_kernel<<<grid, kPrepThreads, 0, env.stream>>>(a, env.status);
    return cudaGetLastError();
}

cudaError_t launch_decode_summarize(const DecodeArgs& a, const KernelEnv& env) {
    dim3 grid(a.max_blocks, a.B * a.Hkv);
    dec_summarize_kernel<<<grid, kPrepThreads, 0, env.stream>>>(a, env.status);
    return cudaGetLastError();
}

cudaError_t launch_decode_score(const DecodeArgs& a, const KernelEnv& env) {
    if (a.d_sel == 128) return launch_score_d<128>(a, env);
    if (a.d_sel == 64) return launch_score_d<64>(a, env);
    return cudaErrorInvalidValue;
}

cudaError_t launch_decode_attn(const DecodeArgs& a, const KernelEnv& env) {
    if (a.d == 128) return launch_attn_d<128>(a, env);
    if (a.d == 64) return launch_attn_d<64>(a, env);
    return cudaErrorInvalidValue;
}

}  // namespace sas
