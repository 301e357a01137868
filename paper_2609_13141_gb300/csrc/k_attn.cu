// a5: fused gated block-sparse attention forward (Eq. ours_train; Alg. 3).
//
// For query row i with current block c = floor(i/64) the logits are
//   z_ij = sm_scale q_i.k_j + beta_ij,
//   beta_ij = 0                for j in block c with j <= i   (unit gate, causal)
//           = log g_{i,m}      for j in a kept historical block m (0 in Alg. 2 mode)
//           = -inf             otherwise,
// and O_i = sum_j softmax(z_i)_j v_j, LSE_i = log sum_j exp(z_ij).
//
// One CTA handles one 128-row query tile t (query blocks 2t and 2t+1) of one
// (batch, head).  It visits only the key blocks some row of the tile needs:
// the tile's union list from the selection pass (blocks < 2t, ascending),
// then the diagonal blocks 2t and 2t+1.  Per visited 64-key block:
//   * warp 0 TMA-loads K (two-stage ring), warp 1 TMA-loads V (own ring);
//   * warp 2 issues S = Q K^T into the TMEM score buffer (tcgen05.mma M=128
//     N=64 K=16 steps); warp 3 issues O += P V into the TMEM output
//     accumulator (M=128 N=d, P read from TMEM, V as an MN-major operand).
//     Each walks its loop as a whole warp and issues from the elect.sync
//     lane; the two streams use different accumulators and are issued
//     independently: one thread cannot issue the small score MMAs as fast
//     as the tensor pipe runs them;
//   * warps 4-7, one thread per query row (TMEM lane), read the score row,
//     add the row's gate or mask (each thread walks its own ascending list of
//     kept blocks), run the online softmax in the log2 domain, write P as
//     packed bf16 into one of two TMEM P buffers and rescale the TMEM output
//     row when the running maximum grows by more than 2^8.
// The score buffer is released as soon as the softmax warps have loaded it,
// so the next block's QK runs during this block's softmax; a P buffer is
// reused once the PV two blocks back has read it.
// The epilogue divides by the row sum and writes bf16 O and fp32 LSE.
// GQA: K, V and the kept lists of query head bh are those of KV group bh / G.
// Head-packed GQA tiles (G >= 2, 128 = G R): a tile takes R consecutive
// tokens of all G query heads of a KV group (rows h R .. h R + R - 1 are head
// h), which share one kept list per token, so the tile visits the union of R
// tokens' kept blocks (one query block's worth at most) instead of two query
// blocks' for each head; the segment unions come from seg_union_kernel.
// Packed sequences: each tile's first row, tile index within its sequence and
// sequence length come from the selection pass's tile table.
#include <math_constants.h>

#include "internal.h"
#include "ptx.cuh"

namespace sas {
namespace {

constexpr int kBM = 128;          // query rows per tile
constexpr int kBN = 64;           // keys per block
constexpr int kThreads = 256;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.69314718055994531f;
constexpr float kRescaleThreshold = 8.0f;   // log2 units
constexpr int kMaxStages = 4;                // capacity of the K / V ring barrier arrays
constexpr int kItemSlots = 4;                // work items in flight between the fetching thread and the other roles
constexpr int kItemReaders = 8;              // K and V producers, QK and PV issuers, four softmax warps
constexpr int kRing = 8;                     // kept-list entries staged ahead per row

template <int D>
struct AttnCfg {
    static constexpr int Q_BYTES = kBM * D * 2;
    static constexpr int KV_BYTES = kBN * D * 2;
    static constexpr int KST = 2;
    static constexpr int VST = 2;
    static_assert(KST <= kMaxStages && VST <= kMaxStages, "ring barrier arrays");
    static constexpr int OFF_K = Q_BYTES;
    static constexpr int OFF_V = OFF_K + KST * KV_BYTES;
    // per row, the next kRing kept blocks and log-gates: int/float [kRing][kBM] each
    static constexpr int OFF_RING = OFF_V + VST * KV_BYTES;
    static constexpr int OFF_CTL = OFF_RING + 2 * kRing * kBM * 4;
    // All shared state lives in the dynamic region (no static shared memory),
    // so that two CTAs fit on one SM.
    static constexpr int SMEM = OFF_CTL + 512;
    static constexpr int TMEM_COLS = 256;    // O [0,D)  S [128,192)  P0 [192,224)  P1 [224,256)
    static constexpr int TMEM_O = 0;
    static constexpr int TMEM_S = 128;
    static constexpr int TMEM_P = 192;       // P buffer b at TMEM_P + 32 b (64 keys packed in pairs)
    static constexpr uint32_t IDESC_S = idesc_bf16(kBM, kBN, 0, 0);
    static constexpr uint32_t IDESC_O = idesc_bf16(kBM, D, 0, 1);
};

// Barriers and flags at the end of the dynamic shared-memory region.
struct AttnCtl {
    uint64_t q_full, q_empty, k_full[kMaxStages], k_empty[kMaxStages], v_full[kMaxStages], v_empty[kMaxStages];
    uint64_t s_full, s_free, p_full[2], pv_done[2], drain_bar;
    uint64_t item_full[kItemSlots], item_empty[kItemSlots];
    int item[kItemSlots];   // work item (or -1: no more work) published to the other roles
    uint32_t tmem_base;
    int abort_flag;
};
static_assert(sizeof(AttnCtl) <= 512, "control block");

constexpr int kStatusLayout = 3;   // == SAS_ERR_CUDA: shared-memory base not 1024-byte aligned

struct AttnParams {
    bf16* O;
    float* LSE;
    const int32_t* union_idx;
    const int32_t* union_cnt;
    const int32_t* sel_idx;
    const float* sel_logg;
    int N, C, T, BH, topk, mode;
    int G;                  // query heads per KV group: K, V and the lists of head bh are group bh / G
    int group;              // heads per group of the work list (a multiple of G)
    const int4* tiles;      // packed sequences: {first row, tile in sequence, length} per slot (else null)
    const int* ntiles;      // slots in use (device)
    int* sched;             // [0] next work item, [1] CTAs finished; both zero between launches
    const float* full_table;   // full training scope: scores [BHkv][N][C] and normalisers [BHkv][N]
    const float* full_lse;
    int seg_rows;              // head-packed tiles: tokens per head R (0: tiles of 128 rows of one head)
    const int32_t* seg_union_idx;   // head-packed: [BHkv][T][C] segment unions (T = segments)
    const int32_t* seg_union_cnt;
    float scale_log2;
    int* status;
    long long limit;
};

// The work list: heads are taken in groups whose K and V fit in about half of
// L2 together (all heads at once when they fit), and within a group the tiles
// with the longest key histories come first, the head varying fastest.  The
// grid is persistent and the list is handed out dynamically: a CTA's K
// producer takes the next item from a global counter when it starts a tile
// (tile costs vary with their union lists, so a fixed split would leave SMs
// idle) and passes it to the CTA's other roles through a small shared ring.
// With GQA the G query heads of a KV group are adjacent in that order, so they
// run the same tile at about the same time over the same K, V blocks.

struct TileRef {
    int t, bh, kv;          // tile (within its sequence), query head (head-packed: the first), KV group
    int base, n;            // the sequence's first row in the token axis and its length
    int row0;               // the tile's first token row within the sequence
    int diag0, ndiag;       // its diagonal blocks: diag0 .. diag0 + ndiag - 1
    const int32_t* ulist;   // the tile's union list (ascending historical blocks)
    int U;                  // its length
};

// T: tile slots in use (p.T, or the packed sequences' tile count; head-packed: segments).
__device__ __forceinline__ TileRef tile_ref(const AttnParams& p, int w, int T) {
    TileRef x;
    if (p.seg_rows > 0) {
        // head-packed: items over (KV group, segment), the group varying fastest
        // within L2-sized groups of KV groups, longest history first.  Packed
        // sequences: segment sg is part sg % G of the table's tile slot sg / G.
        const int BHkv = p.BH / p.G;
        const int Ts = p.tiles == nullptr ? T : T * p.G;   // segments in use
        const int gkv = max(1, p.group / p.G);
        const int per_group = gkv * Ts;
        const int g0 = w / per_group;
        const int k0 = g0 * gkv;
        const int gs = min(gkv, BHkv - k0);
        const int wi = w - g0 * per_group;
        const int sg = p.tiles == nullptr ? Ts - 1 - wi / gs : wi / gs;
        x.kv = k0 + wi % gs;
        x.bh = x.kv * p.G;
        x.t = sg;
        if (p.tiles == nullptr) {
            x.base = 0;
            x.n = p.N;
            x.row0 = sg * p.seg_rows;
        } else {
            const int4 v = __ldg(p.tiles + sg / p.G);
            x.base = v.x;
            x.n = v.z;
            x.row0 = v.y * kBM + (sg % p.G) * p.seg_rows;
        }
        x.diag0 = x.row0 >> 6;   // all R <= 64 tokens share one block
        x.ndiag = 1;
        const long long tb = static_cast<long long>(x.kv) * p.T + sg;   // p.T: segment slots per KV group
        x.ulist = p.seg_union_idx + tb * min(p.C, p.seg_rows * max(p.topk, 1));   // rows of min(C, R K) entries
        x.U = p.full_table != nullptr ? x.diag0 : __ldg(p.seg_union_cnt + tb);
        return x;
    }
    const int per_group = p.group * T;                    // items of a full group
    const int g0 = w / per_group;                         // group index
    const int h0 = g0 * p.group;                          // its first head
    const int gs = min(p.group, p.BH - h0);               // heads in this group
    const int wi = w - g0 * per_group;
    int slot;
    if (p.tiles == nullptr) {
        x.t = T - 1 - wi / gs;
        x.base = 0;
        x.n = p.N;
        slot = x.t;
    } else {
        slot = wi / gs;                                   // the table is ordered longest history first
        const int4 v = __ldg(p.tiles + slot);
        x.base = v.x;
        x.t = v.y;
        x.n = v.z;
    }
    x.bh = h0 + wi % gs;
    x.kv = x.bh / p.G;
    x.row0 = x.t * kBM;
    x.diag0 = 2 * x.t;
    x.ndiag = (2 * x.t + 1) * kBN < x.n ? 2 : 1;
    const long long tb = static_cast<long long>(x.kv) * p.T + slot;
    x.ulist = p.union_idx + tb * p.C;
    // full scope: every historical block of the tile (blocks 0 .. 2t-1, all full)
    x.U = p.full_table != nullptr ? 2 * x.t : __ldg(p.union_cnt + tb);
    return x;
}

// Reader side of the item ring: the r-th work item of this CTA, or -1.
// The caller arrives on item_empty once its lanes have read the value.
__device__ __forceinline__ bool read_item(AttnCtl& ctl, int r, const WaitCtl& wc, int& w) {
    const int slot = r % kItemSlots;
    if (!mbar_wait(&ctl.item_full[slot], (r / kItemSlots) & 1, wc)) return false;
    w = *reinterpret_cast<volatile int*>(&ctl.item[slot]);
    return true;
}

// visited blocks of a tile: its union list, then the diagonal block(s)
__device__ __forceinline__ int tile_blocks(const AttnParams& p, const TileRef& x) {
    return x.U + x.ndiag;
}

template <bool FULL>
__device__ __forceinline__ int block_at(const TileRef& x, int j) {
    return j < x.U ? (FULL ? j : __ldg(x.ulist + j)) : x.diag0 + (j - x.U);
}

// OUTER: the gate of a kept block multiplies its probabilities after the
// softmax (gate position "outer" of Sec. 4.2) instead of adding log g to its
// logits; the row sum and LSE then stay those of the ungated logits.
// FULL: the full training scope (Table 1 setting 9): no kept lists, every
// historical block m of a row enters with log g_m = s_m - LSE of the row's
// scores, read from a [N][C] score table and a per-row normaliser.
template <int D, bool OUTER, bool FULL>
__global__ void __launch_bounds__(kThreads, 2)
attn_kernel(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK,
            const __grid_constant__ CUtensorMap mapV, AttnParams p) {
    using Cfg = AttnCfg<D>;
    extern __shared__ __align__(1024) uint8_t smem[];
    if ((smem_u32(smem) & 1023u) != 0) {
        // The 128-byte swizzle atoms need 1024-byte alignment; report, never fault.
        if (threadIdx.x == 0) atomicExch(p.status, kStatusLayout);
        return;
    }
    AttnCtl& ctl = *reinterpret_cast<AttnCtl*>(smem + Cfg::OFF_CTL);
    uint64_t& q_full = ctl.q_full;
    uint64_t& q_empty = ctl.q_empty;
    uint64_t* k_full = ctl.k_full;
    uint64_t* k_empty = ctl.k_empty;
    uint64_t* v_full = ctl.v_full;
    uint64_t* v_empty = ctl.v_empty;
    uint64_t& s_full = ctl.s_full;     // QK of block g done
    uint64_t& s_free = ctl.s_free;     // all four softmax warps have loaded the scores of block g
    uint64_t* p_full = ctl.p_full;     // P of block g written to P buffer g % 2
    uint64_t* pv_done = ctl.pv_done;   // PV of block g done (O updated, P buffer g % 2 read)
    uint64_t& drain_bar = ctl.drain_bar;
    uint32_t& tmem_base_sh = ctl.tmem_base;
    int& abort_flag = ctl.abort_flag;

    const uint32_t warp = warp_id(), lane = lane_id();
    const int Tn = p.tiles == nullptr ? p.T : __ldg(p.ntiles);   // tile slots in use (head-packed: segments)
    // head-packed: G segments per tile slot of packed sequences
    const int W = p.seg_rows > 0 ? (p.tiles == nullptr ? Tn : Tn * p.G) * (p.BH / p.G) : Tn * p.BH;

    if (threadIdx.x == 0) {
        mbar_init(&q_full, 1);
        mbar_init(&q_empty, 1);
        for (int s = 0; s < Cfg::KST; ++s) { mbar_init(&k_full[s], 1); mbar_init(&k_empty[s], 1); }
        for (int s = 0; s < Cfg::VST; ++s) { mbar_init(&v_full[s], 1); mbar_init(&v_empty[s], 1); }
        mbar_init(&s_full, 1);
        mbar_init(&s_free, 4);
        for (int s = 0; s < 2; ++s) {
            mbar_init(&pv_done[s], 1);
            mbar_init(&p_full[s], 4);
        }
        mbar_init(&drain_bar, 2);   // both MMA issuers
        for (int s = 0; s < kItemSlots; ++s) {
            mbar_init(&ctl.item_full[s], 1);
            mbar_init(&ctl.item_empty[s], kItemReaders);
        }
        abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 3) {
        tmem_alloc(&tmem_base_sh, Cfg::TMEM_COLS);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = tmem_base_sh;
    const WaitCtl wc{&abort_flag, p.status, p.limit};

    // Every role walks the same work items and counts visited blocks over all of
    // them (g): ring slots, score buffers and barrier phases follow g, so the
    // pipeline runs on across tile boundaries.
    if (warp == 0 && lane == 0) {
        // ---------------- K producer
        tma_prefetch_desc(&mapK);
        int g = 0, nk = 0;
        bool ok = true;
        for (int r = 0; ok; ++r) {
            // take the next item and publish it (the slot is free once all readers
            // have taken the item published kItemSlots tiles earlier)
            const int slot = r % kItemSlots;
            if (!mbar_wait(&ctl.item_empty[slot], ((r / kItemSlots) & 1) ^ 1u, wc)) { ok = false; break; }
            int w = atomicAdd(p.sched, 1);
            if (w >= W) w = -1;
            *reinterpret_cast<volatile int*>(&ctl.item[slot]) = w;
            mbar_arrive(&ctl.item_full[slot]);
            mbar_arrive(&ctl.item_empty[slot]);   // this thread has read it too
            if (w < 0) break;
            const TileRef x = tile_ref(p, w, Tn);
            const int n = tile_blocks(p, x);
            for (int j = 0; j < n; ++j) {
                const int gb = g + j;
                const int s = gb % Cfg::KST;
                const int m = block_at<FULL>(x, j);
                if (!mbar_wait(&k_empty[s], ((gb / Cfg::KST) & 1) ^ 1u, wc)) { ok = false; break; }
                uint8_t* dst = smem + Cfg::OFF_K + s * Cfg::KV_BYTES;
                mbar_arrive_expect_tx(&k_full[s], Cfg::KV_BYTES);
#pragma unroll
                for (int a = 0; a < D / 64; ++a)
                    tma_load_3d(dst + a * (kBN * 128), &mapK, &k_full[s], a * 64, x.base + m * kBN, x.kv);
                ++nk;
            }
            g += n;
        }
        if (!ok) {
            // loads are issued in block order, one per block: the last KST may be in flight
            for (int q = nk - 1; q >= 0 && q >= nk - Cfg::KST; --q)
                mbar_wait_drain(&k_full[q % Cfg::KST], (q / Cfg::KST) & 1, p.limit, p.status);
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- V producer and the Q tile.  Q_{i+1} waits until the last
        // QK of tile i has run; that falls between the V slots it waits on, so
        // neither stream holds the other up.
        tma_prefetch_desc(&mapQ);
        tma_prefetch_desc(&mapV);
        int g = 0, tc = 0;
        int nv = 0, nq = 0;
        bool ok = true;
        for (int r = 0; ok; ++r) {
            int w;
            if (!read_item(ctl, r, wc, w)) { ok = false; break; }
            mbar_arrive(&ctl.item_empty[r % kItemSlots]);
            if (w < 0) break;
            const TileRef x = tile_ref(p, w, Tn);
            const int n = tile_blocks(p, x);
            if (!mbar_wait(&q_empty, (tc & 1) ^ 1u, wc)) { ok = false; break; }
            mbar_arrive_expect_tx(&q_full, Cfg::Q_BYTES);
            if (p.seg_rows > 0) {
                // R rows of each of the G heads (the Q map's box is R rows high)
                for (int hq = 0; hq < p.G; ++hq)
#pragma unroll
                    for (int a = 0; a < D / 64; ++a)
                        tma_load_3d(smem + a * (kBM * 128) + hq * p.seg_rows * 128, &mapQ, &q_full, a * 64,
                                    x.base + x.row0, x.bh + hq);
            } else {
#pragma unroll
                for (int a = 0; a < D / 64; ++a)
                    tma_load_3d(smem + a * (kBM * 128), &mapQ, &q_full, a * 64, x.base + x.row0, x.bh);
            }
            ++nq;
            for (int j = 0; j < n; ++j) {
                const int gb = g + j;
                const int s = gb % Cfg::VST;
                const int m = block_at<FULL>(x, j);
                if (!mbar_wait(&v_empty[s], ((gb / Cfg::VST) & 1) ^ 1u, wc)) { ok = false; break; }
                uint8_t* dst = smem + Cfg::OFF_V + s * Cfg::KV_BYTES;
                mbar_arrive_expect_tx(&v_full[s], Cfg::KV_BYTES);
#pragma unroll
                for (int a = 0; a < D / 64; ++a)
                    tma_load_3d(dst + a * (kBN * 128), &mapV, &v_full[s], a * 64, x.base + m * kBN, x.kv);
                ++nv;
            }
            g += n;
            ++tc;
        }
        if (!ok) {
            if (nq > 0) mbar_wait_drain(&q_full, (nq - 1) & 1, p.limit, p.status);
            for (int q = nv - 1; q >= 0 && q >= nv - Cfg::VST; --q)
                mbar_wait_drain(&v_full[q % Cfg::VST], (q / Cfg::VST) & 1, p.limit, p.status);
        }
    } else if (warp == 2) {
        // ---------------- QK issuer (whole warp; the elected lane issues): S = Q K_g^T
        // for every visited block g, once the softmax warps have loaded S_{g-1}
        const uint64_t dq0 = smem_desc_sw128(smem_u32(smem), 16, 1024);
        const uint64_t dk0 = smem_desc_sw128(smem_u32(smem + Cfg::OFF_K), 16, 1024);
        int g = 0, tc = 0;
        bool ok = true;
        for (int r = 0; ok; ++r) {
            int w;
            if (!__all_sync(0xffffffffu, read_item(ctl, r, wc, w))) { ok = false; break; }
            __syncwarp();
            if (lane == 0) mbar_arrive(&ctl.item_empty[r % kItemSlots]);
            if (w < 0) break;
            const int n = tile_blocks(p, tile_ref(p, w, Tn));
            if (!mbar_wait_warp(&q_full, tc & 1, wc)) { ok = false; break; }
            for (int j = 0; j < n; ++j) {
                const int gb = g + j;
                const int s = gb % Cfg::KST;
                if (!mbar_wait_warp(&k_full[s], (gb / Cfg::KST) & 1, wc)) { ok = false; break; }
                if (gb >= 1 && !mbar_wait_warp(&s_free, (gb - 1) & 1, wc)) { ok = false; break; }
                tc_fence_after();
                // descriptors advance by (byte offset >> 4) in their start-address field
                const uint64_t dk = dk0 + static_cast<uint64_t>((s * Cfg::KV_BYTES) >> 4);
                if (elect_one()) {
#pragma unroll
                    for (int k = 0; k < D / 16; ++k) {
                        const uint32_t off_q = (k >> 2) * (kBM * 128) + (k & 3) * 32;
                        const uint32_t off_k = (k >> 2) * (kBN * 128) + (k & 3) * 32;
                        umma_bf16(tmem_base + Cfg::TMEM_S, dq0 + (off_q >> 4), dk + (off_k >> 4), Cfg::IDESC_S,
                                  k > 0);
                    }
                    umma_commit(&s_full);
                    umma_commit(&k_empty[s]);
                    if (j == n - 1) umma_commit(&q_empty);   // Q slot free for the next tile
                }
                __syncwarp();
            }
            g += n;
            ++tc;
        }
        if (elect_one()) {
            umma_commit(&drain_bar);
            mbar_wait_drain(&drain_bar, 0, p.limit, p.status);
        }
        __syncwarp();
    } else if (warp == 3) {
        // ---------------- PV issuer (whole warp; the elected lane issues): O += P_g V_g
        // for every visited block g; the first block of a tile starts a new accumulator
        const uint64_t dv0 = smem_desc_sw128(smem_u32(smem + Cfg::OFF_V), kBN * 128, 1024);
        int g = 0;
        bool ok = true;
        for (int r = 0; ok; ++r) {
            int w;
            if (!__all_sync(0xffffffffu, read_item(ctl, r, wc, w))) { ok = false; break; }
            __syncwarp();
            if (lane == 0) mbar_arrive(&ctl.item_empty[r % kItemSlots]);
            if (w < 0) break;
            const int n = tile_blocks(p, tile_ref(p, w, Tn));
            for (int j = 0; j < n; ++j) {
                const int gb = g + j;
                const int vs = gb % Cfg::VST;
                // p_full[gb&1] cannot run two phases ahead: the softmax writes P_{gb+2}
                // only after PV_gb (issued after this wait) has read the buffer.
                if (!mbar_wait_warp(&p_full[gb & 1], (gb >> 1) & 1, wc)) { ok = false; break; }
                if (!mbar_wait_warp(&v_full[vs], (gb / Cfg::VST) & 1, wc)) { ok = false; break; }
                tc_fence_after();
                const uint64_t dv = dv0 + static_cast<uint64_t>((vs * Cfg::KV_BYTES) >> 4);
                if (elect_one()) {
#pragma unroll
                    for (int k = 0; k < kBN / 16; ++k) {
                        // P_gb sits in P buffer gb & 1 (16 keys = 8 packed columns per step).
                        // V is MN-major (d contiguous): 16 keys = two 8-row atoms (2048 bytes);
                        // the two 64-wide d halves sit kBN*128 bytes apart.
                        umma_bf16_ta(tmem_base + Cfg::TMEM_O, tmem_base + Cfg::TMEM_P + (gb & 1) * 32 + k * 8,
                                     dv + ((k * 2048) >> 4), Cfg::IDESC_O, (j > 0 || k > 0) ? 1u : 0u);
                    }
                    umma_commit(&pv_done[gb & 1]);
                    umma_commit(&v_empty[vs]);
                }
                __syncwarp();
            }
            g += n;
        }
        if (elect_one()) {
            umma_commit(&drain_bar);
            mbar_wait_drain(&drain_bar, 0, p.limit, p.status);
        }
        __syncwarp();
    } else if (warp >= 4) {
        // ---------------- softmax / correction / epilogue: one thread per row
        const int q = warp - 4;
        const int r_row = q * 32 + lane;
        const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
        const uint64_t scale2 = f32x2(p.scale_log2, p.scale_log2);
        const bool train = p.mode == 0;
        int g = 0;
        bool ok = true;
        for (int r = 0; ok; ++r) {
            const int slot = r % kItemSlots;
            if (!mbar_wait_warp(&ctl.item_full[slot], (r / kItemSlots) & 1, wc)) { ok = false; break; }
            const int w = *reinterpret_cast<volatile int*>(&ctl.item[slot]);
            __syncwarp();
            if (lane == 0) mbar_arrive(&ctl.item_empty[slot]);
            if (w < 0) break;
            const TileRef x = tile_ref(p, w, Tn);
            const int n = tile_blocks(p, x);
            // the row's query head and token (within its sequence)
            const int hq = p.seg_rows > 0 ? r_row / p.seg_rows : 0;
            const int i = x.row0 + (p.seg_rows > 0 ? r_row - hq * p.seg_rows : r_row);
            const bool valid = i < x.n;
            const int c = i >> 6;
            const int nsel = (valid && !FULL) ? min(p.topk, c) : 0;
            const long long row_off = static_cast<long long>(x.bh + hq) * p.N + x.base + i;   // O, LSE
            const long long sel_off = static_cast<long long>(x.kv) * p.N + x.base + i;   // the group's kept list
            const int32_t* my_idx = p.sel_idx + sel_off * p.topk;
            const float* my_lg = p.sel_logg + sel_off * p.topk;
            // The row's kept list is staged kRing entries ahead in a shared ring
            // (entry e in slot e % kRing, one commit group per entry), so the walk
            // below only reads entries that have landed long ago.  Every entry of
            // the list is consumed within the tile (each kept block is visited).
            int* ring_i = reinterpret_cast<int*>(smem + Cfg::OFF_RING) + r_row;
            float* ring_l = reinterpret_cast<float*>(smem + Cfg::OFF_RING + kRing * kBM * 4) + r_row;
#pragma unroll
            for (int e = 0; e < kRing; ++e) {
                if (e < nsel) {
                    cp_async4(ring_i + e * kBM, my_idx + e);
                    cp_async4(ring_l + e * kBM, my_lg + e);
                }
                cp_async_commit();
            }
            int sp = 0;   // current entry; groups issued so far = sp + kRing
            int km0 = 0x7fffffff;
            float kl0 = 0.f;
            if (nsel > 0) {
                cp_async_wait<kRing - 1>();
                km0 = ring_i[0];
                kl0 = ring_l[0];
            }

            float m_use = -CUDART_INF_F;
            float l = 0.f;
            // raw list entry for the next iteration (entries past the union are the diagonal blocks)
            int raw_next = 0;
            if (!FULL && x.U > 0) raw_next = __ldg(x.ulist);
            // full scope: the row's score of the next historical block, loaded one block ahead
            const float* tbl = nullptr;
            float lse_row = 0.f, t_next = 0.f;
            if constexpr (FULL) {
                tbl = p.full_table + sel_off * p.C;
                if (valid) lse_row = __ldg(p.full_lse + sel_off);
                if (valid && c > 0 && n > 0) t_next = __ldg(tbl);   // the first visited block is 0
            }
            for (int j = 0; j < n; ++j) {
                const int gb = g + j;
                const int pb = gb & 1;
                const int m = FULL ? block_at<true>(x, j) : (j < x.U ? raw_next : x.diag0 + (j - x.U));
                if (!FULL && j + 1 < x.U) raw_next = __ldg(x.ulist + j + 1);
                // gate (log2 units) and the last visible key column of block m for this row
                float bias = 0.f;
                float gsc = 1.f;   // outer position: gate applied to the probabilities
                int lim;
                if constexpr (FULL) {
                    const float t_cur = t_next;
                    if (j + 1 < n) {
                        const int m1 = block_at<true>(x, j + 1);
                        t_next = (valid && m1 < c) ? __ldg(tbl + m1) : 0.f;
                    }
                    if (m < c) {
                        bias = train ? (t_cur - lse_row) * kLog2e : 0.f;
                        lim = kBN - 1;
                    } else if (m == c) {
                        lim = i & (kBN - 1);
                    } else {
                        lim = -1;
                    }
                } else if (m < c) {
                    if (m == km0) {
                        if constexpr (OUTER) gsc = train ? fast_exp2(kl0 * kLog2e) : 1.f;
                        else bias = train ? kl0 * kLog2e : 0.f;
                        lim = kBN - 1;
                        // refill the finished slot with entry sp + kRing, then step to sp + 1
                        const int e = sp + kRing;
                        if (e < nsel) {
                            cp_async4(ring_i + (sp % kRing) * kBM, my_idx + e);
                            cp_async4(ring_l + (sp % kRing) * kBM, my_lg + e);
                        }
                        cp_async_commit();
                        ++sp;
                        km0 = 0x7fffffff;
                        if (sp < nsel) {
                            cp_async_wait<kRing - 1>();
                            km0 = ring_i[(sp % kRing) * kBM];
                            kl0 = ring_l[(sp % kRing) * kBM];
                        }
                    } else {
                        lim = -1;
                    }
                } else if (m == c) {
                    lim = i & (kBN - 1);
                } else {
                    lim = -1;
                }
                const bool active = lim >= 0;

                // s_full cannot run a phase ahead: QK_{gb+1} waits for this warp's s_free arrival
                if (!mbar_wait_warp(&s_full, gb & 1, wc)) { ok = false; break; }
                // P buffer gb & 1 is free once PV_{gb-2} has read it
                if (gb >= 2 && !mbar_wait_warp(&pv_done[pb], ((gb - 2) >> 1) & 1, wc)) { ok = false; break; }
                tc_fence_after();
                const bool warp_active = __any_sync(0xffffffffu, active);
                bool need = false;
                float m_new = m_use;
                float rs = 0.f;
                uint32_t pk[32];   // P row as packed bf16 pairs
                if (warp_active) {
                    float xs[64];
                    {
                        uint32_t u0[32], u1[32];
                        tmem_ld32(lane_addr + Cfg::TMEM_S, u0);
                        tmem_ld32(lane_addr + Cfg::TMEM_S + 32, u1);
                        tmem_wait_ld();
#pragma unroll
                        for (int k = 0; k < 32; ++k) {
                            xs[k] = __uint_as_float(u0[k]);
                            xs[k + 32] = __uint_as_float(u1[k]);
                        }
                    }
                    // the score buffer is free for the next block's QK
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&s_free);
                    // causal mask on the diagonal block only
                    if (__any_sync(0xffffffffu, lim >= 0 && lim < kBN - 1)) {
#pragma unroll
                        for (int k = 0; k < 64; ++k) xs[k] = k <= lim ? xs[k] : -CUDART_INF_F;
                    }
                    float mx0 = -CUDART_INF_F, mx1 = -CUDART_INF_F;
#pragma unroll
                    for (int k = 0; k < 64; k += 4) {
                        mx0 = max3f(mx0, xs[k], xs[k + 1]);
                        mx1 = max3f(mx1, xs[k + 2], xs[k + 3]);
                    }
                    const float mx = fmaxf(mx0, mx1);
                    // max of the gated logits (log2 units): the gate is constant over the block
                    const float mb = active ? fmaf(mx, p.scale_log2, bias) : -CUDART_INF_F;
                    need = mb > m_use + kRescaleThreshold;
                    m_new = need ? mb : m_use;
                    const float base = m_new == -CUDART_INF_F ? 0.f : m_new;
                    const float off = active ? bias - base : -CUDART_INF_F;
                    const uint64_t off2 = f32x2(off, off);
                    uint64_t acc[4] = {0, 0, 0, 0};
#pragma unroll
                    for (int k = 0; k < 64; k += 2) {
                        float a0, a1;
                        f32x2_split(fma_f32x2(f32x2(xs[k], xs[k + 1]), scale2, off2), a0, a1);
                        const float e0 = fast_exp2(a0), e1 = fast_exp2(a1);
                        acc[(k >> 1) & 3] = add_f32x2(acc[(k >> 1) & 3], f32x2(e0, e1));
                        if constexpr (OUTER) pk[k >> 1] = pack_bf16x2(e0 * gsc, e1 * gsc);
                        else pk[k >> 1] = pack_bf16x2(e0, e1);
                    }
                    float s0, s1, s2, s3, s4, s5, s6, s7;
                    f32x2_split(acc[0], s0, s1);
                    f32x2_split(acc[1], s2, s3);
                    f32x2_split(acc[2], s4, s5);
                    f32x2_split(acc[3], s6, s7);
                    rs = ((s0 + s1) + (s2 + s3)) + ((s4 + s5) + (s6 + s7));
                } else {
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&s_free);
#pragma unroll
                    for (int k = 0; k < 32; ++k) pk[k] = 0u;
                }
                float factor = 1.f;
                if (need) factor = m_use == -CUDART_INF_F ? 0.f : fast_exp2(m_use - m_new);

                if (j > 0 && __any_sync(0xffffffffu, need)) {
                    // Rescaling O needs PV_{gb-1} done.  PV_{gb-1} is the ((gb-1)/2)-th phase of
                    // pv_done[(gb-1)&1]; that barrier cannot move past it before p_full(gb+1).
                    if (!mbar_wait_warp(&pv_done[(gb - 1) & 1], ((gb - 1) >> 1) & 1, wc)) { ok = false; break; }
                    tc_fence_after();
#pragma unroll 1
                    for (int cc = 0; cc < D / 32; ++cc) {
                        uint32_t o[32];
                        tmem_ld32(lane_addr + Cfg::TMEM_O + cc * 32, o);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * factor);
                        tmem_st32(lane_addr + Cfg::TMEM_O + cc * 32, o);
                    }
                    tmem_wait_st();
                }
                l = l * factor + rs;
                m_use = m_new;

                // P row (64 bf16, packed in pairs) into P buffer gb & 1
                tmem_st32(lane_addr + Cfg::TMEM_P + pb * 32, pk);
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&p_full[pb]);
            }
            if (!ok) break;

            // Epilogue.  The next tile's first PV overwrites O; it is issued only after
            // this warp has arrived on p_full for that tile's first block, i.e. after
            // the reads below have completed.  (Its first QK may already run.)
            const int gl = g + n - 1;
            if (!mbar_wait_warp(&pv_done[gl & 1], (gl >> 1) & 1, wc)) { ok = false; break; }
            tc_fence_after();
            const float inv = 1.f / l;
            bf16* orow = p.O + row_off * D;
#pragma unroll 1
            for (int cc = 0; cc < D / 32; ++cc) {
                uint32_t o[32];
                tmem_ld32(lane_addr + Cfg::TMEM_O + cc * 32, o);
                tmem_wait_ld();
                if (valid) {
                    uint4* dst = reinterpret_cast<uint4*>(orow + cc * 32);
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        uint4 v;
                        v.x = pack_bf16x2(__uint_as_float(o[8 * e + 0]) * inv, __uint_as_float(o[8 * e + 1]) * inv);
                        v.y = pack_bf16x2(__uint_as_float(o[8 * e + 2]) * inv, __uint_as_float(o[8 * e + 3]) * inv);
                        v.z = pack_bf16x2(__uint_as_float(o[8 * e + 4]) * inv, __uint_as_float(o[8 * e + 5]) * inv);
                        v.w = pack_bf16x2(__uint_as_float(o[8 * e + 6]) * inv, __uint_as_float(o[8 * e + 7]) * inv);
                        dst[e] = v;
                    }
                }
            }
            if (valid && p.LSE != nullptr) p.LSE[row_off] = m_use * kLn2 + logf(l);
            tc_fence_before();
            g += n;
        }
        // a row that stopped early may still have kept-list copies in flight
        cp_async_wait<0>();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        // This CTA takes no more items.  The last CTA to get here returns the
        // counters to zero for the next launch.
        __threadfence();
        if (atomicAdd(p.sched + 1, 1) == static_cast<int>(gridDim.x) - 1) {
            atomicExch(p.sched, 0);
            atomicExch(p.sched + 1, 0);
        }
    }
    if (warp == 3) {
        tc_fence_after();
        tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
    }
}

template <int D, bool OUTER, bool FULL>
cudaError_t launch_d(const AttnArgs& a, const KernelEnv& env, const char** err) {
    using Cfg = AttnCfg<D>;
    {
        cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(attn_kernel<D, OUTER, FULL>), Cfg::SMEM);
        if (e != cudaSuccess) { *err = "cudaFuncSetAttribute(attn)"; return e; }
    }
    int dev = 0, sms = 0, l2 = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev);
    if (e != cudaSuccess) { *err = "device attributes"; return e; }
    CUtensorMap mq, mk, mv;
    const bool hp = a.seg_rows > 0;   // head-packed tiles: the Q box is one head's seg_rows rows
    if (make_tmap_bf16_3d(&mq, a.Q, D, a.N, a.BH, 64, hp ? a.seg_rows : kBM) != 0) {
        *err = "tensor map Q";
        return cudaErrorInvalidValue;
    }
    const int BHkv = a.BH / a.G;
    if (make_tmap_bf16_3d(&mk, a.K, D, a.N, BHkv, 64, kBN) != 0) { *err = "tensor map K"; return cudaErrorInvalidValue; }
    if (make_tmap_bf16_3d(&mv, a.V, D, a.N, BHkv, 64, kBN) != 0) { *err = "tensor map V"; return cudaErrorInvalidValue; }
    AttnParams p;
    p.O = static_cast<bf16*>(a.O);
    p.LSE = a.LSE;
    p.union_idx = a.union_idx;
    p.union_cnt = a.union_cnt;
    p.sel_idx = a.sel_idx;
    p.sel_logg = a.sel_logg;
    p.N = a.N; p.C = a.C; p.T = hp ? a.nseg : a.T; p.BH = a.BH; p.topk = a.topk; p.mode = a.mode;
    p.seg_rows = hp ? a.seg_rows : 0;
    p.seg_union_idx = a.seg_union_idx;
    p.seg_union_cnt = a.seg_union_cnt;
    p.G = a.G;
    p.tiles = a.tiles;
    p.ntiles = a.ntiles;
    // KV groups whose K and V (2 * N * d bf16 each) fit in half of L2 together,
    // at least one; the work list takes their G query heads each
    const long long kv_head = 4LL * a.N * D;
    const long long fit = kv_head > 0 ? (static_cast<long long>(l2) / 2) / kv_head : BHkv;
    const long long groups = fit < 1 ? 1 : (fit > BHkv ? BHkv : fit);
    p.group = static_cast<int>(groups * a.G);
    p.scale_log2 = a.sm_scale * kLog2e;
    p.status = env.status;
    p.limit = env.limit;
    p.sched = a.sched;
    p.full_table = a.full_table;
    p.full_lse = a.full_lse;
    // persistent grid: two CTAs per SM (their shared memory and TMEM both fit twice)
    // head-packed: segments (packed sequences: G per tile slot; the slot count caps the grid)
    const long long items = hp ? static_cast<long long>(a.nseg) * BHkv : static_cast<long long>(a.T) * a.BH;
    const int G = static_cast<int>(items < 2LL * sms ? items : 2LL * sms);
    attn_kernel<D, OUTER, FULL><<<G, kThreads, Cfg::SMEM, env.stream>>>(mq, mk, mv, p);
    e = cudaGetLastError();
    if (e != cudaSuccess) *err = "attention launch";
    return e;
}

}  // namespace

cudaError_t launch_attn(const AttnArgs& a, const KernelEnv& env, const char** err) {
    if (a.G < 1 || a.BH % a.G != 0) {
        *err = "attention: query heads must fill whole KV groups";
        return cudaErrorInvalidValue;
    }
    if (a.seg_rows > 0 && (a.G < 2 || a.seg_rows * a.G != kBM || a.seg_rows % 8 != 0 || a.full_table != nullptr ||
                           a.seg_union_idx == nullptr || a.seg_union_cnt == nullptr)) {
        *err = "attention: head-packed tiles need G >= 2 with 128 = G x seg_rows (a multiple of 8) and the sparse scope";
        return cudaErrorInvalidValue;
    }
    const bool outer = a.gate_pos == 1;
    if (a.full_table != nullptr) {
        if (outer || a.tiles != nullptr || a.full_lse == nullptr) {
            *err = "attention: the full scope takes the inner gate position and [B, H, N] inputs";
            return cudaErrorInvalidValue;
        }
        if (a.d == 128) return launch_d<128, false, true>(a, env, err);
        if (a.d == 64) return launch_d<64, false, true>(a, env, err);
    }
    if (a.d == 128) return outer ? launch_d<128, true, false>(a, env, err) : launch_d<128, false, false>(a, env, err);
    if (a.d == 64) return outer ? launch_d<64, true, false>(a, env, err) : launch_d<64, false, false>(a, env, err);
    *err = "attention: unsupported head dim";
    return cudaErrorInvalidValue;
}

}  // namespace sas
