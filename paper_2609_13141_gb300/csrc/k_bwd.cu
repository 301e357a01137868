// Backward of the SAS training forward (Alg. 4, App. E; gate and score
// gradients of App. D), d = 128, gate position inner, softmax gates.
//
//   bwd_dq_kernel     pass 1, one CTA per (head, 128-row tile) over the tile's
//                     visited blocks (union of kept blocks + its diagonal
//                     blocks, the forward's lists): S = Q K^T and dP = dO V^T
//                     on the tensor cores, P = exp(S + log g - LSE) and
//                     dS = P (dP - Delta) per row, dS into TMEM as the A
//                     operand of dQ += dS K; the row sum of dS over a kept
//                     block is that row's log-gate gradient.  Also writes
//                     Delta and, per (visited block, row), log g - LSE for
//                     pass 2 (slots from bwd_slots + a scan).
//   bwd_inv_*         the forward's per-tile block lists inverted into, per
//                     key pair (blocks 2p, 2p+1), the query tiles that visit
//                     them (count, scan, fill).
//   bwd_dkv_kernel    pass 2, one CTA per (head, key pair) over those query
//                     tiles, 64 rows at a time: S^T = K Q^T, dP^T = V dO^T
//                     into two TMEM buffers, P^T and dS^T written in place
//                     over them, dV += P^T dO and dK += dS^T Q.
//   bwd_ds_kernel     score gradient of given scores (sparse scope):
//                     ds_m = dlogg_m [m kept] - g_m sum dlogg.
//   bwd_dense_*       kept lists and tile unions of every historical block:
//                     with them the same passes give the backward of the
//                     full training scope (every block kept and gated) and,
//                     pass 1 alone with the soft log-gates and the hard
//                     forward's LSE, the gate gradient of the hard Top-K gate
//                     under the straight-through estimator (x_m = g_m dg_m,
//                     whose score gradient x - g sum x is g (dg - sum g dg)).
// GQA: a KV group's K, V, kept lists and log-gates feed its G query heads, so
// pass 1 runs per query head on its group's K, V and lists and writes the
// head's log-gate gradient, bwd_dlogg_sum adds the G heads (in head order:
// deterministic), pass 2 runs per (group, key pair) over every visiting query
// tile of each of the G heads, accumulating dK, dV of the group, and the score
// gradient applies the gate softmax's Jacobian to the summed d(log g).
// Roles, pass 1: warps 0-7 are the rows (two threads per TMEM lane, half a
// block of keys each), warp 8 issues S and dQ, warp 9 issues dP, warp 10
// issues the TMA loads.  Pass 2: warps 0-3 are the keys (one thread per TMEM
// lane), warps 4 and 7 issue the MMAs, warp 5 stages the query tiles' per-row
// information, warp 6 issues the TMA loads.
#include <math_constants.h>

#include "internal.h"
#include "ptx.cuh"

namespace sas {
namespace {

constexpr int kRows = 128;          // query rows per tile
constexpr int kKeys = 64;           // keys per block
constexpr int kD = 128;             // head dim
constexpr int kWorkers = 128;       // key threads (pass 2)
constexpr int kRowThreads = 256;    // pass 1: two threads per row, 32 keys of a block each
constexpr int kThreadsB = 352;      // + two MMA-issuing warps (one thread cannot feed N = 64 MMAs fast enough) + a loader
constexpr float kLog2eB = 1.4426950408889634f;
// Waiting threads sleep (woken when the phase completes) instead of spinning:
// the issuing and row-information warps wait most of the time and would
// otherwise take issue slots from the row / key warps.
constexpr uint32_t kSleepNs = 1000;

__device__ __forceinline__ float bfl(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bfh(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// 16 packed bf16 pairs into 16 TMEM columns of this thread's lane.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}

// Delta_i = dO_i . O_i for one row (bf16 rows of d = 128).
__device__ __forceinline__ float row_delta(const bf16* O, const bf16* dO) {
    const uint4* o4 = reinterpret_cast<const uint4*>(O);
    const uint4* g4 = reinterpret_cast<const uint4*>(dO);
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < kD / 8; ++i) {
        const uint4 a = __ldg(o4 + i), b = __ldg(g4 + i);
        acc = fmaf(bfl(a.x), bfl(b.x), acc); acc = fmaf(bfh(a.x), bfh(b.x), acc);
        acc = fmaf(bfl(a.y), bfl(b.y), acc); acc = fmaf(bfh(a.y), bfh(b.y), acc);
        acc = fmaf(bfl(a.z), bfl(b.z), acc); acc = fmaf(bfh(a.z), bfh(b.z), acc);
        acc = fmaf(bfl(a.w), bfl(b.w), acc); acc = fmaf(bfh(a.w), bfh(b.w), acc);
    }
    return acc;
}

// ------------------------------------------------------------------ pass 1

struct DqCtl {
    uint64_t q_full, kv_full[4], kv_empty[4], sdp_full[2], ds_full[2], dq_done[2], fin;
    uint32_t tmem_base;
    int abort_flag;
};

constexpr int kQBytes = kRows * kD * 2;                 // 32 KB
constexpr int kKVBytes = kKeys * kD * 2;                // 16 KB
constexpr int kDqOffDO = kQBytes;
// K, V ring: the load of block j + 4 goes out once dQ of block j has read K, so
// three blocks of loads are in flight behind the one being multiplied
constexpr int kKvStages = 4;
constexpr int kDqOffKV = 2 * kQBytes;                   // kKvStages x (K, V)
constexpr int kDqOffCtl = kDqOffKV + kKvStages * 2 * kKVBytes;
constexpr int kDqSmem = kDqOffCtl + 256 + 1024;         // + alignment slack
// TMEM: dQ [0,128); S and dP of block j in buffer j & 1: S [128 + 128 b, +64),
// dP [192 + 128 b, +64); dS buffers [384,416), [416,448)
constexpr uint32_t kTmemDQ = 0, kTmemS = 128, kTmemDP = 192, kTmemDS = 384;

struct BwdParams {
    const bf16* O;
    const bf16* dO;
    const float* LSE;
    const int32_t* union_idx;
    const int32_t* union_cnt;
    const int32_t* sel_idx;
    const float* sel_logg;
    bf16* dQ;
    bf16* dK;
    bf16* dV;
    float* dlogg;
    float* delta;
    const int32_t* inv_off;
    const int32_t* inv_tiles;
    const int32_t* inv_pos;     // per inverted entry: positions of blocks 2p, 2p+1 in the tile's list (+1; 0: absent)
    const int32_t* slot_off;    // per tile: first slot of its visited blocks in offs
    float* offs;                // per (tile, visited block) slot: 128 rows of log g - LSE (log2), -inf if not attended
    const int4* tiles;          // packed sequences: {first row of the sequence, local tile, length, sequence} per slot
    const int* ntiles;          // slots in use (device)
    const int* tile_off;        // first slot of each local tile index
    // head-packed tiles (the forward's): R tokens x G heads of a KV group per
    // tile, segments sg = 0 .. nseg - 1 of R tokens per group, their unions
    // (row stride seg_cap); 0 = tiles of 128 rows of one head.  Packed
    // sequences: segment slot sg is sub-segment sg % G of tile slot sg / G
    // (nseg = G T); a segment's index within its sequence is G t + sg % G for
    // the slot's local tile t
    int seg_rows, nseg, seg_cap;
    const int32_t* seg_union_idx;
    const int32_t* seg_union_cnt;
    int N, C, T, BH, topk, mode;
    int G;                      // query heads per KV group (BH counts query heads)
    float sm_scale, scale_log2;
    int* status;
    long long limit;
};

// A tile slot's place in its sequence: the local tile index t (rows 128 t ..
// 128 t + 127 of the sequence, key blocks 2t, 2t + 1), the sequence's first
// row in the head's token axis and its length.  [B, H, N, d] batches: one
// sequence of N rows, slot = tile.
struct BwdTile {
    int t, base, n;
};
__device__ __forceinline__ BwdTile bwd_tile(const BwdParams& p, int slot) {
    if (p.tiles == nullptr) return {slot, 0, p.N};
    const int4 v = __ldg(p.tiles + slot);
    return {v.y, v.x, v.z};
}
__device__ __forceinline__ int bwd_slots_in_use(const int4* tiles, const int* ntiles, int T) {
    return tiles == nullptr ? T : __ldg(ntiles);
}
// Head-packed segment slot sg: t = the segment's index within its sequence
// (rows R t .. R t + R - 1 of it), the sequence's first row and length; t = -1
// for a slot past the tiles in use or a segment past its sequence's end.
__device__ __forceinline__ BwdTile bwd_seg(const BwdParams& p, int sg) {
    if (p.tiles == nullptr) return {sg, 0, p.N};
    const int ts = sg / p.G;
    if (ts >= __ldg(p.ntiles)) return {-1, 0, 0};
    const int4 v = __ldg(p.tiles + ts);
    const int t = v.y * p.G + (sg - ts * p.G);
    return {t * p.seg_rows < v.z ? t : -1, v.x, v.z};
}

template <bool HP, bool OUTER>
__global__ void __launch_bounds__(kThreadsB, 1)
bwd_dq_kernel(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapDO,
              const __grid_constant__ CUtensorMap mapK, const __grid_constant__ CUtensorMap mapV, BwdParams p) {
    extern __shared__ __align__(1024) uint8_t dsm[];
    uint8_t* smem = dsm + ((1024u - (smem_u32(dsm) & 1023u)) & 1023u);
    DqCtl& ctl = *reinterpret_cast<DqCtl*>(smem + kDqOffCtl);
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    // per-head tiles: CTA (query head bh, tile slot); head-packed (HP): (KV group, segment)
    constexpr bool hp = HP;
    const int nsl = hp ? p.nseg : p.T;
    const int slot = blockIdx.x % nsl, bh = blockIdx.x / nsl;
    if (!hp && slot >= bwd_slots_in_use(p.tiles, p.ntiles, p.T)) return;   // an unused slot (packed sequences)
    const BwdTile tg = hp ? bwd_seg(p, slot) : bwd_tile(p, slot);
    if (hp && tg.t < 0) return;                                  // no rows (packed sequences)
    const int tile = tg.t;                                       // local tile index (head-packed: segment)
    const int kv = hp ? bh : bh / p.G;                           // the KV group
    const int row0 = tg.base + tile * (hp ? p.seg_rows : kRows);   // first token row in the token axis
    const long long tb = static_cast<long long>(bh) * nsl + slot;   // this tile's offset slots
    const long long tbk = static_cast<long long>(kv) * nsl + slot;  // its union
    const int32_t* ulist = hp ? p.seg_union_idx + tbk * p.seg_cap : p.union_idx + tbk * p.C;
    const int U = __ldg((hp ? p.seg_union_cnt : p.union_cnt) + tbk);
    const int cseq = (tg.n + kKeys - 1) / kKeys;                 // blocks of the sequence
    // visited blocks: the union, then the diagonal one(s)
    const int diag0 = hp ? (tile * p.seg_rows) >> 6 : 2 * tile;
    const int nb = U + (hp ? 1 : ((2 * tile + 1 < cseq) ? 2 : 1));
    if (t == 0) {
        mbar_init(&ctl.q_full, 1);
        for (int s = 0; s < kKvStages; ++s) {
            mbar_init(&ctl.kv_full[s], 1);
            mbar_init(&ctl.kv_empty[s], 2);   // dQ (reads K) and dP (reads V)
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&ctl.ds_full[s], kRowThreads / 32);   // one arrive per row warp
            mbar_init(&ctl.dq_done[s], 1);
            mbar_init(&ctl.sdp_full[s], 2);   // S from one issuer, dP from the other
        }
        mbar_init(&ctl.fin, 2);
        ctl.abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0) {
        tmem_alloc(&ctl.tmem_base, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = ctl.tmem_base;
    const WaitCtl wc{&ctl.abort_flag, p.status, p.limit};

    if (warp == 10) {
        if (lane == 0) {
            // ---- loader: Q and dO once, then K and V of block j into stage
            // j % kKvStages as soon as dQ and dP of block j - kKvStages are done
            mbar_arrive_expect_tx(&ctl.q_full, 2 * kQBytes);
            if (hp) {
                // R rows of each of the G heads (the Q / dO maps' box is R rows high)
                for (int hq = 0; hq < p.G; ++hq)
                    for (int h = 0; h < 2; ++h) {
                        const int so = h * (kRows * 128) + hq * p.seg_rows * 128;
                        tma_load_3d(smem + so, &mapQ, &ctl.q_full, h * 64, row0, bh * p.G + hq);
                        tma_load_3d(smem + kDqOffDO + so, &mapDO, &ctl.q_full, h * 64, row0, bh * p.G + hq);
                    }
            } else {
                for (int h = 0; h < 2; ++h) {
                    tma_load_3d(smem + h * (kRows * 128), &mapQ, &ctl.q_full, h * 64, row0, bh);
                    tma_load_3d(smem + kDqOffDO + h * (kRows * 128), &mapDO, &ctl.q_full, h * 64, row0, bh);
                }
            }
            for (int j = 0; j < nb; ++j) {
                const int s = j % kKvStages;
                if (j >= kKvStages && !mbar_wait(&ctl.kv_empty[s], ((j / kKvStages) - 1) & 1, wc, kSleepNs)) break;
                const int m = j < U ? __ldg(ulist + j) : diag0 + (j - U);
                uint8_t* st = smem + kDqOffKV + s * 2 * kKVBytes;
                mbar_arrive_expect_tx(&ctl.kv_full[s], 2 * kKVBytes);
                for (int h = 0; h < 2; ++h) {
                    tma_load_3d(st + h * (kKeys * 128), &mapK, &ctl.kv_full[s], h * 64, tg.base + m * kKeys, kv);
                    tma_load_3d(st + kKVBytes + h * (kKeys * 128), &mapV, &ctl.kv_full[s], h * 64,
                                tg.base + m * kKeys, kv);
                }
            }
        }
    } else if (warp == 8) {
        {
            // ---- issuer of S = Q K^T and dQ += dS K (whole warp; the elected lane issues)
            constexpr uint32_t IDESC_S = idesc_bf16(kRows, kKeys, 0, 0);
            constexpr uint32_t IDESC_DQ = idesc_bf16(kRows, kD, 0, 1);
            const uint32_t qb = smem_u32(smem);
            bool ok = mbar_wait_warp(&ctl.q_full, 0, wc, kSleepNs);
            // S and dP of block j go to TMEM buffer j & 1 while the rows still work
            // on block j - 1; dQ += dS K of block j - 1 follows once its dS is in.
            for (int j = 0; ok && j <= nb; ++j) {
                if (j < nb) {
                    const int s = j & 1, ks = j % kKvStages;
                    if (!mbar_wait_warp(&ctl.kv_full[ks], (j / kKvStages) & 1, wc, kSleepNs)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t kb = smem_u32(smem + kDqOffKV + ks * 2 * kKVBytes);
                    if (elect_one()) {
#pragma unroll
                        for (int k = 0; k < kD / 16; ++k) {
                            const uint32_t oq = (k >> 2) * (kRows * 128) + (k & 3) * 32;
                            const uint32_t ok2 = (k >> 2) * (kKeys * 128) + (k & 3) * 32;
                            umma_bf16(tmem + kTmemS + s * 128, smem_desc_sw128(qb + oq, 16, 1024),
                                      smem_desc_sw128(kb + ok2, 16, 1024), IDESC_S, k > 0);
                        }
                        umma_commit(&ctl.sdp_full[s]);
                    }
                    __syncwarp();
                }
                if (j >= 1) {
                    const int jp = j - 1, sp = jp & 1, kp = jp % kKvStages;
                    // dS of block jp is in TMEM buffer sp once every row has written it
                    if (!mbar_wait_warp(&ctl.ds_full[sp], (jp >> 1) & 1, wc, kSleepNs)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t kb = smem_u32(smem + kDqOffKV + kp * 2 * kKVBytes);
                    if (elect_one()) {
#pragma unroll
                        for (int k = 0; k < kKeys / 16; ++k)
                            umma_bf16_ta(tmem + kTmemDQ, tmem + kTmemDS + sp * 32 + k * 8,
                                         smem_desc_sw128(kb + k * 2048, kKeys * 128, 1024), IDESC_DQ,
                                         (jp > 0 || k > 0) ? 1u : 0u);
                        umma_commit(&ctl.dq_done[sp]);
                        umma_commit(&ctl.kv_empty[kp]);
                    }
                    __syncwarp();
                }
            }
            if (elect_one()) {
                umma_commit(&ctl.fin);
                mbar_wait_drain(&ctl.fin, 0, p.limit, p.status);
            }
            __syncwarp();
        }
    } else if (warp == 9) {
        {
            // ---- second issuer: dP = dO V^T of every block into TMEM buffer j & 1,
            // once the rows are done with block j - 2 (which used that buffer)
            constexpr uint32_t IDESC_S = idesc_bf16(kRows, kKeys, 0, 0);
            const uint32_t gb = smem_u32(smem + kDqOffDO);
            bool ok = mbar_wait_warp(&ctl.q_full, 0, wc, kSleepNs);
            for (int j = 0; ok && j < nb; ++j) {
                const int s = j & 1, ks = j % kKvStages;
                if (!mbar_wait_warp(&ctl.kv_full[ks], (j / kKvStages) & 1, wc, kSleepNs)) { ok = false; break; }
                if (j >= 2 && !mbar_wait_warp(&ctl.ds_full[s], ((j - 2) >> 1) & 1, wc, kSleepNs)) { ok = false; break; }
                tc_fence_after();
                const uint32_t vb = smem_u32(smem + kDqOffKV + ks * 2 * kKVBytes) + kKVBytes;
                if (elect_one()) {
#pragma unroll
                    for (int k = 0; k < kD / 16; ++k) {
                        const uint32_t oq = (k >> 2) * (kRows * 128) + (k & 3) * 32;
                        const uint32_t ok2 = (k >> 2) * (kKeys * 128) + (k & 3) * 32;
                        umma_bf16(tmem + kTmemDP + s * 128, smem_desc_sw128(gb + oq, 16, 1024),
                                  smem_desc_sw128(vb + ok2, 16, 1024), IDESC_S, k > 0);
                    }
                    umma_commit(&ctl.sdp_full[s]);
                    umma_commit(&ctl.kv_empty[ks]);
                }
                __syncwarp();
            }
            if (elect_one()) {
                umma_commit(&ctl.fin);
                mbar_wait_drain(&ctl.fin, 0, p.limit, p.status);
            }
            __syncwarp();
        }
    } else {
        // ---- rows: thread t takes row t % 128 (its TMEM lane) and keys
        // 32 hk .. 32 hk + 31 of every block, hk = t / 128
        const int r = t & (kRows - 1), hk = t >> 7;
        // the row's query head and token (head-packed: row r is head r / R, token r % R of the segment)
        const int hq = hp ? r / p.seg_rows : 0;
        const int rt = hp ? r - hq * p.seg_rows : r;
        const int i = row0 - tg.base + rt;     // row index within the sequence
        const bool valid = i < tg.n;
        const int c = i >> 6;                  // the row's current block
        const uint32_t lane_addr = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
        const long long roff = static_cast<long long>(hp ? bh * p.G + hq : bh) * p.N + row0 + rt;
        const long long kvoff = static_cast<long long>(kv) * p.N + row0 + rt;   // the group's kept list
        float delta = 0.f, lse2 = 0.f;
        if (valid) {
            delta = row_delta(p.O + roff * kD, p.dO + roff * kD);
            lse2 = __ldg(p.LSE + roff) * kLog2eB;
            if (hk == 0) p.delta[roff] = delta;
        }
        // the per-block offsets for pass 2 (a gate-only pass has no pass 2: offs null)
        const int slot0 = p.offs != nullptr ? __ldg(p.slot_off + tb) : 0;
        const int nsel = valid ? min(p.topk, c) : 0;
        const int32_t* my_idx = p.sel_idx + kvoff * p.topk;
        const float* my_lg = p.sel_logg + kvoff * p.topk;
        float* my_dlg = p.dlogg + roff * p.topk;   // this head's (zeroed before this kernel; both halves add)
        int e = 0;                             // next kept entry (ascending)
        int km = nsel > 0 ? __ldg(my_idx) : 0x7fffffff;
        float kl = nsel > 0 ? __ldg(my_lg) : 0.f;
        // the entry after it, loaded one step early
        int km_n = nsel > 1 ? __ldg(my_idx + 1) : 0x7fffffff;
        float kl_n = nsel > 1 ? __ldg(my_lg + 1) : 0.f;
        const bool train = p.mode == 0;
        bool ok = true;
        for (int j = 0; j < nb; ++j) {
            const int m = j < U ? __ldg(ulist + j) : diag0 + (j - U);
            float bias = 0.f;
            int lim = -1;
            bool kept = false;
            if (valid) {
                if (m < c) {
                    if (m == km) {
                        kept = true;
                        bias = train ? kl * kLog2eB : 0.f;
                        lim = kKeys - 1;
                    }
                } else if (m == c) {
                    lim = i & (kKeys - 1);
                }
            }
            if (!mbar_wait_warp(&ctl.sdp_full[j & 1], (j >> 1) & 1, wc, kSleepNs)) { ok = false; break; }
            // the dS buffer j & 1 is free once dQ of block j - 2 has read it
            if (j >= 2 && !mbar_wait_warp(&ctl.dq_done[j & 1], ((j - 2) >> 1) & 1, wc, kSleepNs)) { ok = false; break; }
            tc_fence_after();
            float sum = 0.f;
            {
                uint32_t sv[32], dv[32];
                tmem_ld32(lane_addr + kTmemS + (j & 1) * 128 + hk * 32, sv);
                tmem_ld32(lane_addr + kTmemDP + (j & 1) * 128 + hk * 32, dv);
                tmem_wait_ld();
                // P = exp2(S scale + (log g - LSE)) in log2 units; exp2(-inf) = 0 for a
                // block the row does not attend; the causal limit only on its own block.
                // Outer gate position: P is the plain softmax (no bias) and the block's
                // gate w multiplies dP: dS = P (w dP - Delta); pass 2 gets w (-1: not
                // attended) in place of the offset
                const float boff = lim >= 0 ? (OUTER ? -lse2 : bias - lse2) : -CUDART_INF_F;
                const float wg = OUTER ? fast_exp2(bias) : 1.f;
                const bool causal = lim >= 0 && lim < kKeys - 1;
                if (hk == 0 && p.offs != nullptr)
                    p.offs[(static_cast<long long>(slot0) + j) * kRows + r] = OUTER ? (lim >= 0 ? wg : -1.f) : boff;
                const uint64_t sc2 = f32x2(p.scale_log2, p.scale_log2), bo2 = f32x2(boff, boff);
                const uint64_t nd2 = f32x2(-delta, -delta), w2 = f32x2(wg, wg);
                uint64_t acc = 0;
                uint32_t pk[16];
#pragma unroll
                for (int k = 0; k < 32; k += 2) {
                    float z0, z1;
                    f32x2_split(fma_f32x2(f32x2(__uint_as_float(sv[k]), __uint_as_float(sv[k + 1])), sc2, bo2), z0, z1);
                    float p0 = fast_exp2(z0), p1 = fast_exp2(z1);
                    if (causal) {
                        p0 = hk * 32 + k <= lim ? p0 : 0.f;
                        p1 = hk * 32 + k + 1 <= lim ? p1 : 0.f;
                    }
                    const uint64_t dv2 = f32x2(__uint_as_float(dv[k]), __uint_as_float(dv[k + 1]));
                    const uint64_t d2 = OUTER ? fma_f32x2(dv2, w2, nd2) : add_f32x2(dv2, nd2);
                    const uint64_t ds2 = fma_f32x2(f32x2(p0, p1), d2, 0ull);
                    // the block's d(log g): row sum of dS (inner), w times that of P dP (outer)
                    acc = OUTER ? fma_f32x2(f32x2(p0, p1), dv2, acc) : add_f32x2(acc, ds2);
                    float a0, a1;
                    f32x2_split(ds2, a0, a1);
                    pk[k >> 1] = pack_bf16x2(a0, a1);
                }
                float s0, s1;
                f32x2_split(acc, s0, s1);
                sum = OUTER ? wg * (s0 + s1) : s0 + s1;
                tmem_st16(lane_addr + kTmemDS + (j & 1) * 32 + hk * 16, pk);
            }
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive_warp(&ctl.ds_full[j & 1]);
            if (kept) {
                if (train) atomicAdd(my_dlg + e, sum);   // two halves: a + b, order-independent
                ++e;
                km = km_n;
                kl = kl_n;
                km_n = e + 1 < nsel ? __ldg(my_idx + e + 1) : 0x7fffffff;
                kl_n = e + 1 < nsel ? __ldg(my_lg + e + 1) : 0.f;
            }
        }
        // dQ: columns 64 hk .. 64 hk + 63 of the row
        if (ok && mbar_wait_warp(&ctl.fin, 0, wc, kSleepNs)) {
            tc_fence_after();
#pragma unroll 1
            for (int cc = 2 * hk; cc < 2 * hk + 2; ++cc) {
                uint32_t o[32];
                tmem_ld32(lane_addr + kTmemDQ + cc * 32, o);
                tmem_wait_ld();
                if (valid && p.dQ != nullptr) {   // null: a gate-only pass
                    uint4* dst = reinterpret_cast<uint4*>(p.dQ + roff * kD + cc * 32);
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        dst[q] = make_uint4(pack_bf16x2(__uint_as_float(o[8 * q + 0]) * p.sm_scale, __uint_as_float(o[8 * q + 1]) * p.sm_scale),
                                            pack_bf16x2(__uint_as_float(o[8 * q + 2]) * p.sm_scale, __uint_as_float(o[8 * q + 3]) * p.sm_scale),
                                            pack_bf16x2(__uint_as_float(o[8 * q + 4]) * p.sm_scale, __uint_as_float(o[8 * q + 5]) * p.sm_scale),
                                            pack_bf16x2(__uint_as_float(o[8 * q + 6]) * p.sm_scale, __uint_as_float(o[8 * q + 7]) * p.sm_scale));
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// ------------------------------------------------------- inverted block lists

// Slot of the key pair (blocks 2 pr, 2 pr + 1) of the sequence whose local
// tile tq sits at slot g: the pair's keys are the rows of local tile pr, and a
// sequence of rank r keeps its tile t at tile_off[t] + r.  [B, H, N, d]: pr.
__device__ __forceinline__ int pair_slot(const int4* tiles, const int* tile_off, int g, int pr) {
    if (tiles == nullptr) return pr;
    const int tq = __ldg(tiles + g).y;
    return g - __ldg(tile_off + tq) + __ldg(tile_off + pr);
}

// A source of the inverted lists: a tile slot g, or (head-packed, hg = G) a
// segment slot g.  ts = its tile slot, entry = its index within the sequence
// (tile or segment), own = the key pair of its diagonal block when that pair
// visits it as a diagonal item (head-packed: segments of block 2p + 1 may keep
// block 2p), else -1; ts = -1 for an unused slot.
struct InvSrc {
    int ts, entry, own;
};
__device__ __forceinline__ InvSrc inv_src(int g, int hg, const int4* tiles, const int* ntiles) {
    const int ts = hg > 0 ? g / hg : g;
    // every source of a [B, H, N, d] batch is live (its last tile may hold fewer than G segments)
    if (tiles != nullptr && ts >= __ldg(ntiles)) return {-1, 0, -1};
    const int tq = tiles == nullptr ? ts : __ldg(tiles + ts).y;   // local tile
    if (hg == 0) return {ts, tq, -1};
    return {ts, tq * hg + (g - ts * hg), tq};
}

// count: for every tile (head-packed: segment), the key pairs (2p, 2p+1) its
// union list touches, but its own pair; nsrc tiles or segments per group,
// union rows of ustride; hg = G for head-packed segments, else 0
__global__ void bwd_inv_count_kernel(const int32_t* union_idx, const int32_t* union_cnt, int32_t* cnt, int BH,
                                     int T, int nsrc, int ustride, const int4* tiles, const int* ntiles,
                                     const int* tile_off, int hg) {
    const long long tb = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (tb >= static_cast<long long>(BH) * nsrc) return;
    const int bh = static_cast<int>(tb / nsrc);
    const int g = static_cast<int>(tb - static_cast<long long>(bh) * nsrc);
    const InvSrc src = inv_src(g, hg, tiles, ntiles);
    if (src.ts < 0) return;
    const int32_t* u = union_idx + tb * ustride;
    const int U = union_cnt[tb];
    int last = -1;
    for (int k = 0; k < U; ++k) {
        const int pr = u[k] >> 1;
        if (pr == last || pr == src.own) continue;
        last = pr;
        atomicAdd(cnt + static_cast<long long>(bh) * T + pair_slot(tiles, tile_off, src.ts, pr), 1);
    }
}

// exclusive scan of n counts into off[0..n] (one CTA of 1024 threads)
__global__ void __launch_bounds__(1024) bwd_inv_scan_kernel(const int32_t* cnt, int32_t* off, int32_t* cursor,
                                                            long long n) {
    __shared__ int part[1024];
    const int t = threadIdx.x;
    const long long per = (n + 1023) / 1024;
    const long long lo = min(static_cast<long long>(t) * per, n), hi = min(lo + per, n);
    int s = 0;
    for (long long k = lo; k < hi; ++k) s += cnt[k];
    part[t] = s;
    __syncthreads();
    for (int o = 1; o < 1024; o <<= 1) {
        const int v = t >= o ? part[t - o] : 0;
        __syncthreads();
        part[t] += v;
        __syncthreads();
    }
    int run = part[t] - s;
    for (long long k = lo; k < hi; ++k) {
        off[k] = run;
        if (cursor) cursor[k] = run;
        run += cnt[k];
    }
    if (t == 1023) off[n] = part[1023];
}

// fill: entry = the visiting tile's index within its sequence (head-packed: the
// segment's) and the positions of the pair's blocks in its list
__global__ void bwd_inv_fill_kernel(const int32_t* union_idx, const int32_t* union_cnt, int32_t* cursor,
                                    int32_t* tiles, int32_t* pos, int BH, int T, int nsrc, int ustride,
                                    const int4* ttab, const int* ntiles, const int* tile_off, int hg) {
    const long long tb = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (tb >= static_cast<long long>(BH) * nsrc) return;
    const int bh = static_cast<int>(tb / nsrc);
    const int g = static_cast<int>(tb - static_cast<long long>(bh) * nsrc);
    const InvSrc src = inv_src(g, hg, ttab, ntiles);
    if (src.ts < 0) return;
    const int32_t* u = union_idx + tb * ustride;
    const int U = union_cnt[tb];
    int last = -1;
    for (int k = 0; k < U; ++k) {
        const int m = u[k], pr = m >> 1;
        if (pr == last || pr == src.own) continue;
        last = pr;
        // positions (+1) of blocks 2pr and 2pr+1 in this tile's list (ascending)
        const int j0 = m == 2 * pr ? k + 1 : 0;
        const int j1 = m == 2 * pr + 1 ? k + 1 : (k + 1 < U && u[k + 1] == 2 * pr + 1 ? k + 2 : 0);
        const int slot = atomicAdd(cursor + static_cast<long long>(bh) * T + pair_slot(ttab, tile_off, src.ts, pr), 1);
        tiles[slot] = src.entry;
        pos[slot] = j0 | (j1 << 16);
    }
}

// visited blocks per (query head, tile): its group's union list plus one or two
// diagonal blocks; head-packed (seg_cnt non-null): per (KV group, segment slot),
// its union plus its one diagonal block (none for an unused slot or a segment
// past its sequence's end: seg_R rows per segment)
__global__ void bwd_slots_kernel(const int32_t* union_cnt, int32_t* cnt, int BH, int T, int N, int G,
                                 const int4* tiles, const int* ntiles, const int32_t* seg_cnt, long long nseg_total,
                                 int nseg, int seg_R) {
    const long long tb = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (seg_cnt != nullptr) {
        if (tb >= nseg_total) return;
        bool live = true;
        if (tiles != nullptr) {
            const int sg = static_cast<int>(tb % nseg), ts = sg / G;
            live = ts < __ldg(ntiles);
            if (live) {
                const int4 v = __ldg(tiles + ts);
                live = (v.y * G + (sg - ts * G)) * seg_R < v.z;
            }
        }
        cnt[tb] = live ? seg_cnt[tb] + 1 : 0;
        return;
    }
    if (tb >= static_cast<long long>(BH) * T) return;
    const int g = static_cast<int>(tb % T);
    if (g >= bwd_slots_in_use(tiles, ntiles, T)) {
        cnt[tb] = 0;
        return;
    }
    int t = g, n = N;
    if (tiles != nullptr) {
        const int4 v = __ldg(tiles + g);
        t = v.y;
        n = v.z;
    }
    const long long tbk = (tb / T) / G * T + g;
    cnt[tb] = union_cnt[tbk] + ((2 * t + 1 < (n + kKeys - 1) / kKeys) ? 2 : 1);
}

// GQA: the log-gate gradient of a KV group is the sum of its G query heads'
// (Eq. ours_train: the group's log-gates enter the logits of all G heads),
// added in head order so the result does not depend on scheduling.
__global__ void bwd_dlogg_sum_kernel(const float* heads, float* out, long long per_group, long long total, int G) {
    const long long x = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (x >= total) return;
    const long long g = x / per_group, k = x - g * per_group;
    const float* src = heads + g * G * per_group + k;
    float s = 0.f;
    for (int h = 0; h < G; ++h) s += __ldg(src + h * per_group);
    out[x] = s;
}

// ------------------------------------------------------------------ pass 2

struct DkvCtl {
    uint64_t kv_full, q_full[2], q_empty[2], info_full[4], info_empty[4];
    uint64_t sdp_full[2], pds_full[2], fin;   // per TMEM buffer
    uint32_t tmem_base;
    int abort_flag;
};

constexpr int kThreadsD = 256;                           // keys (4 warps), two issuers, a row-info warp, a loader
constexpr int kInfoLanes = 32;
constexpr int kPairBytes = 2 * kKeys * kD * 2;           // 32 KB: K (or V) of the key pair
constexpr int kDkvOffV = kPairBytes;
constexpr int kDkvOffQ = 2 * kPairBytes;                 // 2 stages x (Q, dO) tiles
constexpr int kInfoStages = 4;                           // row information computed up to 3 tiles ahead
constexpr int kDkvOffInfo = kDkvOffQ + 2 * 2 * kQBytes;  // stages x [4][128] floats: lse2, delta, bias0, bias1
constexpr int kDkvOffList = kDkvOffInfo + kInfoStages * 4 * kRows * 4;
// query tiles of a key pair (sorted list, then the unsorted copy); the host
// refuses heads of more than kBwdMaxTiles tiles
constexpr int kDkvListCap = 2048;
constexpr int kDkvOffCtl = kDkvOffList + 3 * kDkvListCap * 4;   // order, tiles, positions
constexpr int kDkvSmem = kDkvOffCtl + 256 + 1024;
// TMEM: dV [0,128), dK [128,256), then two buffers b of 128 columns at 256 + 128 b:
// S^T in the first 64, dP^T in the last 64.  The keys write P^T (dS^T) in place
// over the first 32 columns of the S^T (dP^T) they have read.
constexpr uint32_t kTmemDV = 0, kTmemDK = 128, kTmemBuf = 256, kTmemST = 0, kTmemDPT = 64;

template <bool HP, bool OUTER>
__global__ void __launch_bounds__(kThreadsD, 1)
bwd_dkv_kernel(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapDO,
               const __grid_constant__ CUtensorMap mapK2, const __grid_constant__ CUtensorMap mapV2, BwdParams p) {
    extern __shared__ __align__(1024) uint8_t dsm[];
    uint8_t* smem = dsm + ((1024u - (smem_u32(dsm) & 1023u)) & 1023u);
    DkvCtl& ctl = *reinterpret_cast<DkvCtl*>(smem + kDkvOffCtl);
    int* list = reinterpret_cast<int*>(smem + kDkvOffList);
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    // key pair = blocks 2pr, 2pr+1 (keys 128 pr .. of the sequence) of group kv; its
    // slot is that of the sequence's local tile pr
    const int pslot = blockIdx.x % p.T, kv = blockIdx.x / p.T;
    if (pslot >= bwd_slots_in_use(p.tiles, p.ntiles, p.T)) return;   // an unused slot (packed sequences)
    const BwdTile ptg = bwd_tile(p, pslot);
    const int pr = ptg.t;
    const int cseq = (ptg.n + kKeys - 1) / kKeys;
    const long long pb = static_cast<long long>(kv) * p.T + pslot;
    constexpr bool hp = HP;   // head-packed tiles
    // diagonal query tiles first: per-head tiles, tile pr; head-packed, the
    // segments of tokens 128 pr .. 128 pr + 127 that exist
    const int ndg = hp ? min(p.G, (ptg.n - pr * kRows + p.seg_rows - 1) / p.seg_rows) : 1;
    const int off = __ldg(p.inv_off + pb);
    const int cnt = min(__ldg(p.inv_off + pb + 1) - off, kDkvListCap - 1 - ndg);
    const int nq = cnt + ndg;
    // work items: per-head tiles, every visiting query tile once for each of the
    // group's G query heads (item k: tile list[k / G] of head kv G + k % G);
    // head-packed, every visiting segment once (its 128 rows hold all G heads)
    const int G = hp ? 1 : p.G;
    const int nitems = nq * G;
    if (t == 0) {
        mbar_init(&ctl.kv_full, 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(&ctl.q_full[s], 1);
            mbar_init(&ctl.q_empty[s], 2);    // both issuers' products of the tile
        }
        for (int s = 0; s < kInfoStages; ++s) {
            mbar_init(&ctl.info_full[s], 1);                // the row-information warp
            mbar_init(&ctl.info_empty[s], kWorkers / 32);   // one arrive per key warp
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&ctl.sdp_full[b], 2);   // S^T from the first issuer, dP^T from the second
            mbar_init(&ctl.pds_full[b], kWorkers / 32);
        }
        mbar_init(&ctl.fin, 2);
        ctl.abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0) {
        tmem_alloc(&ctl.tmem_base, 512);
        tmem_relinquish();
    }
    // the query tiles: diagonal first, then the others in ascending order (a
    // fixed summation order); rank sort of the inverted list in shared memory
    // list[q]: index into raw / rawpos of the q-th query tile (slot 0: the diagonal
    // tile, which visits 2pr, 2pr+1 right after its union list); raw holds the
    // tiles' indices within the sequence (so packed sequences sum in the order of
    // a batch of the same data)
    int* raw = list + kDkvListCap;
    int* rawpos = raw + kDkvListCap;
    if (t == 0) {
        if (!hp) {
            list[0] = 0;
            raw[0] = pr;
            const int Upr = __ldg(p.union_cnt + pb);
            rawpos[0] = (Upr + 1) | ((2 * pr + 1 < cseq ? Upr + 2 : 0) << 16);
        } else {
            // segment sg of block c visits c right after its union (position U); a
            // segment of block 2 pr + 1 may also keep block 2 pr (its union's last entry)
            for (int k = 0; k < ndg; ++k) {
                const int sg = pr * p.G + k;   // within the sequence; its slot: pslot G + k (packed)
                const long long sb = static_cast<long long>(kv) * p.nseg + (p.tiles == nullptr ? sg : pslot * p.G + k);
                const int Us = __ldg(p.seg_union_cnt + sb);
                const int cb = (sg * p.seg_rows) >> 6;
                int pos;
                if (cb == 2 * pr) {
                    pos = Us + 1;
                } else {
                    const bool has0 = Us > 0 && __ldg(p.seg_union_idx + sb * p.seg_cap + Us - 1) == 2 * pr;
                    pos = (has0 ? Us : 0) | ((Us + 1) << 16);
                }
                list[k] = k;
                raw[k] = sg;
                rawpos[k] = pos;
            }
        }
    }
    for (int k = t; k < cnt; k += kThreadsD) {
        raw[ndg + k] = __ldg(p.inv_tiles + off + k);
        rawpos[ndg + k] = __ldg(p.inv_pos + off + k);
    }
    __syncthreads();
    for (int k = t; k < cnt; k += kThreadsD) {
        const int v = raw[ndg + k];
        int rank = 0;
        for (int q = 0; q < cnt; ++q) rank += raw[ndg + q] < v;
        list[ndg + rank] = ndg + k;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = ctl.tmem_base;
    const WaitCtl wc{&ctl.abort_flag, p.status, p.limit};
    float* info = reinterpret_cast<float*>(smem + kDkvOffInfo);
    const int nh = 2 * nitems;   // 64-row halves of the items

    if (warp == 5) {
        // ---- row information of query tile q, up to three tiles ahead: per row
        // the offsets (log g - LSE) of blocks 2pr, 2pr+1 that pass 1 wrote, and -Delta
        const int il = lane;
        for (int it = 0; it < nitems; ++it) {
            const int s = it % kInfoStages;
            if (it >= kInfoStages &&
                !mbar_wait(&ctl.info_empty[s], ((it - kInfoStages) / kInfoStages) & 1, wc, kSleepNs))
                break;
            float* inf = info + s * 4 * kRows;
            const int q = it / G;
            const int bhq = kv * G + it % G;   // the item's query head (per-head tiles)
            const int tq = raw[list[q]];       // the query tile within the sequence (head-packed: segment), and its slot
            int gq = tq;
            if (p.tiles != nullptr) {
                const int tt = hp ? tq / p.G : tq;   // the local tile
                gq = pslot - __ldg(p.tile_off + pr) + __ldg(p.tile_off + tt);
                if (hp) gq = gq * p.G + (tq - tt * p.G);
            }
            const int ps = rawpos[list[q]];
            const int j0 = (ps & 0xffff) - 1, j1 = (ps >> 16) - 1;
            const long long tbq = hp ? static_cast<long long>(kv) * p.nseg + gq : static_cast<long long>(bhq) * p.T + gq;
            const long long so = static_cast<long long>(__ldg(p.slot_off + tbq)) * kRows;
#pragma unroll
            for (int rr = 0; rr < kRows / kInfoLanes; ++rr) {
                const int r = il + rr * kInfoLanes;
                // the row's head and token within the sequence
                const int hr = hp ? r / p.seg_rows : 0;
                const int i = hp ? tq * p.seg_rows + (r - hr * p.seg_rows) : tq * kRows + r;
                const long long drow = static_cast<long long>(hp ? kv * p.G + hr : bhq) * p.N + ptg.base + i;
                // outer gate position: the blocks' gates w (-1: not attended) and -LSE
                const float kAbsent = OUTER ? -1.f : -CUDART_INF_F;
                inf[r] = j0 >= 0 ? __ldcg(p.offs + so + static_cast<long long>(j0) * kRows + r) : kAbsent;
                inf[kRows + r] = j1 >= 0 ? __ldcg(p.offs + so + static_cast<long long>(j1) * kRows + r) : kAbsent;
                inf[2 * kRows + r] = i < ptg.n ? -__ldcg(p.delta + drow) : 0.f;
                if (OUTER) inf[3 * kRows + r] = i < ptg.n ? -__ldg(p.LSE + drow) * kLog2eB : -CUDART_INF_F;
            }
            mbar_arrive_warp(&ctl.info_full[s]);
        }
    } else if (warp == 6) {
        if (lane == 0) {
            // ---- loader: K and V of the pair once, then the (Q, dO) rows of
            // query tile q into stage q & 1 once both products of tile q - 2 are done
            mbar_arrive_expect_tx(&ctl.kv_full, 2 * kPairBytes);
            for (int h = 0; h < 2; ++h) {
                tma_load_3d(smem + h * (2 * kKeys * 128), &mapK2, &ctl.kv_full, h * 64, ptg.base + pr * 2 * kKeys, kv);
                tma_load_3d(smem + kDkvOffV + h * (2 * kKeys * 128), &mapV2, &ctl.kv_full, h * 64,
                            ptg.base + pr * 2 * kKeys, kv);
            }
            for (int it = 0; it < nitems; ++it) {
                const int s = it & 1;
                if (it >= 2 && !mbar_wait(&ctl.q_empty[s], ((it - 2) >> 1) & 1, wc, kSleepNs)) break;
                const int tq = raw[list[it / G]];
                uint8_t* st = smem + kDkvOffQ + s * 2 * kQBytes;
                mbar_arrive_expect_tx(&ctl.q_full[s], 2 * kQBytes);
                if (hp) {
                    // the segment's R rows of each of the G heads
                    const int row = ptg.base + tq * p.seg_rows;
                    for (int hq = 0; hq < p.G; ++hq)
                        for (int h = 0; h < 2; ++h) {
                            const int so = h * (kRows * 128) + hq * p.seg_rows * 128;
                            tma_load_3d(st + so, &mapQ, &ctl.q_full[s], h * 64, row, kv * p.G + hq);
                            tma_load_3d(st + kQBytes + so, &mapDO, &ctl.q_full[s], h * 64, row, kv * p.G + hq);
                        }
                } else {
                    const int row = ptg.base + tq * kRows;
                    const int bhq = kv * G + it % G;
                    for (int h = 0; h < 2; ++h) {
                        tma_load_3d(st + h * (kRows * 128), &mapQ, &ctl.q_full[s], h * 64, row, bhq);
                        tma_load_3d(st + kQBytes + h * (kRows * 128), &mapDO, &ctl.q_full[s], h * 64, row, bhq);
                    }
                }
            }
        }
    } else if (warp == 4 || warp == 7) {
        {
            // ---- issuers (whole warp; the elected lane issues): warp 4 issues
            // S^T = K Q^T and dV += P^T dO; warp 7 issues dP^T = V dO^T and
            // dK += dS^T Q.  Half x uses TMEM buffer x & 1: its products go in
            // two halves ahead, right behind the accumulation of half x - 2
            // (which reads P^T / dS^T from that buffer); its accumulation once
            // the keys have written P^T, dS^T.
            const bool first = warp == 4;
            constexpr uint32_t IDESC_T = idesc_bf16(2 * kKeys, 64, 0, 0);   // M = 128 keys, N = 64 rows
            constexpr uint32_t IDESC_ACC = idesc_bf16(2 * kKeys, kD, 0, 1);
            // A operand (K or V of the pair) and this issuer's columns of the buffers
            const uint32_t ab = smem_u32(smem + (first ? 0 : kDkvOffV));
            const uint32_t t_own = tmem + kTmemBuf + (first ? kTmemST : kTmemDPT);
            const uint32_t t_acc = tmem + (first ? kTmemDV : kTmemDK);
            bool ok = mbar_wait_warp(&ctl.kv_full, 0, wc, kSleepNs);
            auto issue_prod = [&](int x) -> bool {
                const int q = x >> 1, h = x & 1, s = q & 1;
                if (h == 0 && !mbar_wait_warp(&ctl.q_full[s], (q >> 1) & 1, wc, kSleepNs)) return false;
                tc_fence_after();
                // B operand: Q (first issuer) or dO rows of this half, K-major
                const uint32_t bb = smem_u32(smem + kDkvOffQ + s * 2 * kQBytes) + (first ? 0 : kQBytes);
                const uint32_t dst = t_own + (x & 1) * 128;
                if (elect_one()) {
#pragma unroll
                    for (int k = 0; k < kD / 16; ++k) {
                        const uint32_t oa = (k >> 2) * (2 * kKeys * 128) + (k & 3) * 32;
                        const uint32_t ob = (k >> 2) * (kRows * 128) + h * 64 * 128 + (k & 3) * 32;
                        umma_bf16(dst, smem_desc_sw128(ab + oa, 16, 1024), smem_desc_sw128(bb + ob, 16, 1024),
                                  IDESC_T, k > 0);
                    }
                    umma_commit(&ctl.sdp_full[x & 1]);
                }
                __syncwarp();
                return true;
            };
            if (ok) ok = issue_prod(0);
            if (ok && nh > 1) ok = issue_prod(1);
            for (int x = 0; ok && x < nh; ++x) {
                const int q = x >> 1, h = x & 1, s = q & 1, b = x & 1;
                if (!mbar_wait_warp(&ctl.pds_full[b], (x >> 1) & 1, wc, kSleepNs)) { ok = false; break; }
                tc_fence_after();
                // B operand: dO (first issuer, for dV) or Q (for dK) rows of this half, MN-major
                const uint32_t bb = smem_u32(smem + kDkvOffQ + s * 2 * kQBytes) + (first ? kQBytes : 0);
                const uint32_t a2 = t_own + b * 128;   // P^T or dS^T, in place
                if (elect_one()) {
#pragma unroll
                    for (int k = 0; k < 64 / 16; ++k) {
                        const uint32_t ob = h * 64 * 128 + k * 2048;   // 16 rows = two 8-row atoms
                        umma_bf16_ta(t_acc, a2 + k * 8, smem_desc_sw128(bb + ob, kRows * 128, 1024), IDESC_ACC,
                                     (x > 0 || k > 0) ? 1u : 0u);
                    }
                    if (h == 1) umma_commit(&ctl.q_empty[s]);
                }
                __syncwarp();
                // The products of half x + 2 overwrite the columns this accumulation
                // reads: MMAs of one thread (elect.sync of a full warp always picks
                // its lowest lane) run in issue order through the tensor pipe, so
                // they are issued right behind it without a wait.
                if (x + 2 < nh && !issue_prod(x + 2)) { ok = false; break; }
            }
            if (elect_one()) {
                umma_commit(&ctl.fin);
                mbar_wait_drain(&ctl.fin, 0, p.limit, p.status);
            }
            __syncwarp();
        }
    } else {
        // ---- keys: thread = key of the pair (TMEM lane)
        const int key = t;
        const int kl = pr * 2 * kKeys + key;      // key index within the sequence
        const int kblk = key >> 6;                // 0: block 2pr, 1: block 2pr + 1
        const uint32_t lane_addr = tmem + (static_cast<uint32_t>(warp * 32) << 16);
        bool ok = true;
        for (int x = 0; x < nh; ++x) {
            const int q = x >> 1, h = x & 1, si = q % kInfoStages, b = x & 1;
            const float* inf = info + si * 4 * kRows;
            const uint32_t buf = lane_addr + kTmemBuf + b * 128;
            if (h == 0 && !mbar_wait_warp(&ctl.info_full[si], (q / kInfoStages) & 1, wc, kSleepNs)) { ok = false; break; }
            if (!mbar_wait_warp(&ctl.sdp_full[b], (x >> 1) & 1, wc, kSleepNs)) { ok = false; break; }
            tc_fence_after();
            uint32_t sv[64], dv[64];
            tmem_ld32(buf + kTmemST, *reinterpret_cast<uint32_t(*)[32]>(sv));
            tmem_ld32(buf + kTmemST + 32, *reinterpret_cast<uint32_t(*)[32]>(sv + 32));
            tmem_ld32(buf + kTmemDPT, *reinterpret_cast<uint32_t(*)[32]>(dv));
            tmem_ld32(buf + kTmemDPT + 32, *reinterpret_cast<uint32_t(*)[32]>(dv + 32));
            tmem_wait_ld();
            uint32_t pp[32], dd[32];
            // In a diagonal tile the rows whose own block is this key's block see
            // only the keys up to themselves.  Per-head tiles (the first item of
            // the list, items 0 .. G-1): the rows of half h have block 2pr + h, and
            // column k is token k of it.  Head-packed: all rows of diagonal segment
            // sg are in block (sg R) / 64, column k is token (sg R) % 64 + k % R.
            const int qi = q / G;
            bool causal;
            int toff0 = 0, rmask = 63;
            if constexpr (HP) {
                const int sg = raw[list[qi]];
                causal = qi < ndg && ((sg * p.seg_rows) >> 6) == 2 * pr + kblk;
                toff0 = (sg * p.seg_rows) & 63;
                rmask = p.seg_rows - 1;
            } else {
                causal = qi == 0 && h == kblk;
            }
            const float2* off2 = reinterpret_cast<const float2*>(inf + kblk * kRows + h * 64);
            const float2* nd2p = reinterpret_cast<const float2*>(inf + 2 * kRows + h * 64);
            const float2* ul2p = reinterpret_cast<const float2*>(inf + 3 * kRows + h * 64);   // outer: -LSE
            const uint64_t sc2 = f32x2(p.scale_log2, p.scale_log2);
            const int kin = key & 63;
#pragma unroll
            for (int k = 0; k < 64; k += 2) {
                // inner: o = the offset (log g - LSE); outer: o = the gate w (-1: not
                // attended), P unweighted from -LSE, P^T = P w, dS^T = P (w dP - Delta)
                const float2 o = off2[k >> 1], nd = nd2p[k >> 1];
                const float2 zo = OUTER ? ul2p[k >> 1] : o;
                float z0, z1;
                f32x2_split(fma_f32x2(f32x2(__uint_as_float(sv[k]), __uint_as_float(sv[k + 1])), sc2, f32x2(zo.x, zo.y)),
                            z0, z1);
                float p0 = fast_exp2(z0), p1 = fast_exp2(z1);
                if (OUTER) {
                    p0 = o.x >= 0.f ? p0 : 0.f;
                    p1 = o.y >= 0.f ? p1 : 0.f;
                }
                if (causal) {
                    p0 = kin <= toff0 + (k & rmask) ? p0 : 0.f;
                    p1 = kin <= toff0 + ((k + 1) & rmask) ? p1 : 0.f;
                }
                const uint64_t dv2 = f32x2(__uint_as_float(dv[k]), __uint_as_float(dv[k + 1]));
                const uint64_t d2 = OUTER ? fma_f32x2(dv2, f32x2(o.x, o.y), f32x2(nd.x, nd.y))
                                          : add_f32x2(dv2, f32x2(nd.x, nd.y));
                float a0, a1;
                f32x2_split(fma_f32x2(f32x2(p0, p1), d2, 0ull), a0, a1);
                pp[k >> 1] = OUTER ? pack_bf16x2(p0 * o.x, p1 * o.y) : pack_bf16x2(p0, p1);
                dd[k >> 1] = pack_bf16x2(a0, a1);
            }
            // P^T and dS^T over the S^T and dP^T columns just read
            tmem_st32(buf + kTmemST, pp);
            tmem_st32(buf + kTmemDPT, dd);
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive_warp(&ctl.pds_full[b]);
            if (h == 1) mbar_arrive_warp(&ctl.info_empty[si]);
        }
        if (ok && mbar_wait_warp(&ctl.fin, 0, wc, kSleepNs)) {
            tc_fence_after();
            const bool kv_in = kl < ptg.n;
            const long long koff = static_cast<long long>(kv) * p.N + ptg.base + kl;
#pragma unroll 1
            for (int which = 0; which < 2; ++which) {
                bf16* dst_row = (which == 0 ? p.dV : p.dK) + koff * kD;
                const float sc = which == 0 ? 1.f : p.sm_scale;
#pragma unroll 1
                for (int cc = 0; cc < kD / 32; ++cc) {
                    uint32_t o[32];
                    tmem_ld32(lane_addr + (which == 0 ? kTmemDV : kTmemDK) + cc * 32, o);
                    tmem_wait_ld();
                    if (kv_in) {
                        uint4* dst = reinterpret_cast<uint4*>(dst_row + cc * 32);
#pragma unroll
                        for (int q2 = 0; q2 < 4; ++q2)
                            dst[q2] = make_uint4(pack_bf16x2(__uint_as_float(o[8 * q2 + 0]) * sc, __uint_as_float(o[8 * q2 + 1]) * sc),
                                                 pack_bf16x2(__uint_as_float(o[8 * q2 + 2]) * sc, __uint_as_float(o[8 * q2 + 3]) * sc),
                                                 pack_bf16x2(__uint_as_float(o[8 * q2 + 4]) * sc, __uint_as_float(o[8 * q2 + 5]) * sc),
                                                 pack_bf16x2(__uint_as_float(o[8 * q2 + 6]) * sc, __uint_as_float(o[8 * q2 + 7]) * sc));
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// ----------------------------------------------------- dense block lists

// Kept lists and tile unions holding every historical block, for the
// backwards that gate all of them: the full training scope (Sec. 4.2; log g =
// s - LSE of the row's scores) and the gate pass of the hard Top-K gate under
// the straight-through estimator (the soft log g of every block).  Row i keeps
// blocks 0 .. C_i - 1 in order with log g_m = s_m - lse_i (0 past its
// history); one warp per row.
__global__ void __launch_bounds__(256) bwd_dense_rows_kernel(const float* s, const float* lse, int N, int C,
                                                             long long rows, int32_t* idx, float* lg) {
    const long long w = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (w >= rows) return;
    const int c = min(static_cast<int>(w % N) >> 6, C);
    const float l = c > 0 ? __ldg(lse + w) : 0.f;
    const float* sr = s + w * C;
    for (int m = lane; m < C; m += 32) {
        idx[w * C + m] = m;
        lg[w * C + m] = m < c ? __ldg(sr + m) - l : 0.f;
    }
}

// Tile t's union: blocks 0 .. 2t - 1 (its diagonal blocks are visited apart).
// One warp per (group, tile).
__global__ void __launch_bounds__(256) bwd_dense_unions_kernel(int32_t* uidx, int32_t* ucnt, int T, int C,
                                                               long long tiles) {
    const long long w = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (w >= tiles) return;
    const int n = min(2 * static_cast<int>(w % T), C);
    for (int k = lane; k < n; k += 32) uidx[w * C + k] = k;
    if (lane == 0) ucnt[w] = n;
}

// --------------------------------------------------------- score gradient

// ds_m = dlogg_m [m kept] - g_m sum_kept dlogg, g = softmax of the row's C_i
// given scores; 0 past the history.  The other gate activations have
// independent gates: ds_m = dlogg_m d(log g_m)/ds_m on kept blocks only
// (act 1, sigmoid: dlogg_m (1 - g_m) = -dlogg_m expm1(log g_m); act 2, raw
// logit: dlogg_m).  One warp per row, every load of the row
// issued first (the row's scores are held in registers when C <= 32 NCH):
// the log-normaliser comes back from the first kept entry (log g_m = s_m -
// LSE of the scores, Eq. normalized_log_gate), the kept dlogg values are
// scattered into the warp's C floats of shared memory.
template <int NCH>
__global__ void __launch_bounds__(256)
bwd_ds_kernel(const float* scores, const int32_t* sel_idx, const float* sel_logg, const float* dlogg, float* ds,
              int N, int C, int topk, int train, int act, int chunks, const int4* tiles, const int* ntiles) {
    extern __shared__ float dsh[];   // per warp: C floats (the row's kept dlogg, scattered)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // CTA = (head, run of blockDim / 32 rows of it): one division per CTA.
    // Packed sequences: chunks = tile slots x runs per 128-row tile, and i is
    // the row's index within its sequence (its blocks count from there).
    const int bh = static_cast<int>(blockIdx.x / static_cast<unsigned>(chunks));
    const int run = static_cast<int>(blockIdx.x - static_cast<unsigned>(bh) * chunks);
    int i, row;
    if (tiles == nullptr) {
        i = run * (blockDim.x >> 5) + warp;
        row = i;
        if (i >= N) return;          // no block-wide synchronisation below
    } else {
        const int per_tile = kRows / (blockDim.x >> 5);
        const int g = run / per_tile;
        if (g >= __ldg(ntiles)) return;
        const int4 v = __ldg(tiles + g);
        const int r = (run - g * per_tile) * (blockDim.x >> 5) + warp;
        i = v.y * kRows + r;
        row = v.x + i;
        if (i >= v.z) return;
    }
    const long long w = static_cast<long long>(bh) * N + row;
    float* add = dsh + warp * C;
    const int c = i >> 6;
    const int nsel = train ? min(topk, c) : 0;
    const float* s = scores + w * C;
    float* out = ds + w * C;
    float sv[NCH > 0 ? NCH : 1];
    if (NCH > 0) {
#pragma unroll
        for (int q = 0; q < NCH; ++q) {
            const int m = lane + 32 * q;
            sv[q] = m < c ? __ldg(s + m) : 0.f;
        }
    }
    const int32_t* ix = sel_idx + w * topk;
    const float* dl = dlogg + w * topk;
    // a kept entry's d(log g)/ds: sigmoid 1 - g, else 1 (softmax couples through the sum below)
    const float* lgr = sel_logg + w * topk;
    auto dlds = [&](int e) { return act == 1 ? -expm1f(__ldg(lgr + e)) : 1.f; };
    const float v0 = lane < nsel ? __ldg(dl + lane) * dlds(lane) : 0.f;
    const int i0 = lane < nsel ? __ldg(ix + lane) : 0;
    const float lg0 = nsel > 0 ? __ldg(lgr) : 0.f;
    for (int m = lane; m < C; m += 32) add[m] = 0.f;
    __syncwarp();
    float sum = v0;
    if (lane < nsel) add[i0] = v0;   // kept blocks are distinct
    for (int e = lane + 32; e < nsel; e += 32) {
        const float v = __ldg(dl + e) * dlds(e);
        sum += v;
        add[__ldg(ix + e)] = v;
    }
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (act != 0) sum = 0.f;   // independent gates: no coupling term
    // LSE = s_m0 - log g_m0 for the first kept block m0 (< c, so in registers)
    const int m0 = __shfl_sync(0xffffffffu, i0, 0);
    float s0;
    if (NCH > 0) {
        float mine = 0.f;
#pragma unroll
        for (int q = 0; q < NCH; ++q)
            if (q == (m0 >> 5)) mine = sv[q];
        s0 = __shfl_sync(0xffffffffu, mine, m0 & 31);
    } else {
        s0 = nsel > 0 ? __ldg(s + m0) : 0.f;
    }
    const float lse = s0 - lg0;
    __syncwarp();
    if (NCH > 0) {
#pragma unroll
        for (int q = 0; q < NCH; ++q) {
            const int m = lane + 32 * q;
            if (m < C) {
                float v = 0.f;
                if (m < c) {
                    v = add[m];
                    if (sum != 0.f) v -= __expf(sv[q] - lse) * sum;
                }
                out[m] = v;
            }
        }
    } else {
        for (int m = lane; m < C; m += 32) {
            float v = 0.f;
            if (m < c) {
                v = add[m];
                if (sum != 0.f) v -= __expf(__ldg(s + m) - lse) * sum;
            }
            out[m] = v;
        }
    }
}

}  // namespace

const int kBwdMaxTiles = kDkvListCap - 1;

// Slots of the per-tile visited-block offsets pass 1 writes for pass 2: one per
// visited block of every tile; returns their total in *total (synchronises).
cudaError_t launch_bwd_slots(const AttnBwdArgs& a, const KernelEnv& env, long long* total) {
    // offset slots per (query head, tile), head-packed per (KV group, segment)
    const long long tiles = a.seg_rows > 0 ? static_cast<long long>(a.BH / a.G) * a.nseg : static_cast<long long>(a.BH) * a.T;
    const unsigned gb = static_cast<unsigned>((tiles + 255) / 256);
    bwd_slots_kernel<<<gb, 256, 0, env.stream>>>(a.union_cnt, a.inv_cnt, a.BH, a.T, a.N, a.G, a.tiles, a.ntiles,
                                                 a.seg_rows > 0 ? a.seg_union_cnt : nullptr, tiles, a.nseg, a.seg_rows);
    bwd_inv_scan_kernel<<<1, 1024, 0, env.stream>>>(a.inv_cnt, a.slot_off, nullptr, tiles);
    if (total == nullptr) return cudaGetLastError();   // the caller's buffer holds the upper bound
    int32_t host = 0;
    cudaError_t e = cudaMemcpyAsync(&host, a.slot_off + tiles, 4, cudaMemcpyDeviceToHost, env.stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(env.stream);
    *total = host;
    return e;
}

cudaError_t launch_bwd_dense_lists(const float* s, const float* lse, int BHkv, int N, int C, int T, int32_t* idx,
                                   float* lg, int32_t* uidx, int32_t* ucnt, const KernelEnv& env) {
    const long long rows = static_cast<long long>(BHkv) * N;
    const long long tiles = static_cast<long long>(BHkv) * T;
    bwd_dense_rows_kernel<<<static_cast<unsigned>((rows * 32 + 255) / 256), 256, 0, env.stream>>>(s, lse, N, C, rows,
                                                                                                  idx, lg);
    bwd_dense_unions_kernel<<<static_cast<unsigned>((tiles * 32 + 255) / 256), 256, 0, env.stream>>>(uidx, ucnt, T, C,
                                                                                                    tiles);
    return cudaGetLastError();
}

cudaError_t launch_attn_bwd(const AttnBwdArgs& a, const KernelEnv& env, const char** err) {
    if (a.d != kD) {
        *err = "backward: head dim must be 128";
        return cudaErrorInvalidValue;
    }
    const int G = a.G > 0 ? a.G : 1;
    if (a.BH % G != 0 || (G > 1 && a.dlogg_heads == nullptr)) {
        *err = "backward: query heads must fill whole KV groups";
        return cudaErrorInvalidValue;
    }
    // segments of one sequence: a key pair's inverted list holds at most that many, plus its diagonal ones
    const long long seq_segs = a.tiles != nullptr ? static_cast<long long>(G) * ((a.C + 1) / 2) : a.nseg;
    if (a.seg_rows > 0 && (G < 2 || a.seg_rows * G != kRows || a.seg_rows % 8 != 0 ||
                           a.seg_union_idx == nullptr || a.seg_union_cnt == nullptr ||
                           (a.tiles != nullptr && a.nseg != G * a.T) || seq_segs + G > kDkvListCap - 1)) {
        *err = "backward: head-packed tiles need 128 = G x seg_rows, segment unions and short enough sequences";
        return cudaErrorInvalidValue;
    }
    const int BHkv = a.BH / G;   // KV groups x batch
    {
        const void* dq[4] = {reinterpret_cast<const void*>(bwd_dq_kernel<false, false>),
                             reinterpret_cast<const void*>(bwd_dq_kernel<true, false>),
                             reinterpret_cast<const void*>(bwd_dq_kernel<false, true>),
                             reinterpret_cast<const void*>(bwd_dq_kernel<true, true>)};
        const void* dkv[4] = {reinterpret_cast<const void*>(bwd_dkv_kernel<false, false>),
                              reinterpret_cast<const void*>(bwd_dkv_kernel<true, false>),
                              reinterpret_cast<const void*>(bwd_dkv_kernel<false, true>),
                              reinterpret_cast<const void*>(bwd_dkv_kernel<true, true>)};
        cudaError_t e = cudaSuccess;
        for (int v = 0; v < 4 && e == cudaSuccess; ++v) {
            e = ensure_smem_attr(dq[v], kDqSmem);
            if (e == cudaSuccess) e = ensure_smem_attr(dkv[v], kDkvSmem);
        }
        if (e != cudaSuccess) { *err = "cudaFuncSetAttribute(bwd)"; return e; }
    }
    CUtensorMap mq, mdo, mk, mv, mk2, mv2;
    const bool hp = a.seg_rows > 0;   // head-packed tiles: the Q / dO boxes are one head's seg_rows rows
    if (make_tmap_bf16_3d(&mq, a.Q, kD, a.N, a.BH, 64, hp ? a.seg_rows : kRows) != 0 ||
        make_tmap_bf16_3d(&mdo, a.dO, kD, a.N, a.BH, 64, hp ? a.seg_rows : kRows) != 0 ||
        make_tmap_bf16_3d(&mk, a.K, kD, a.N, BHkv, 64, kKeys) != 0 ||
        make_tmap_bf16_3d(&mv, a.V, kD, a.N, BHkv, 64, kKeys) != 0 ||
        make_tmap_bf16_3d(&mk2, a.K, kD, a.N, BHkv, 64, 2 * kKeys) != 0 ||
        make_tmap_bf16_3d(&mv2, a.V, kD, a.N, BHkv, 64, 2 * kKeys) != 0) {
        *err = "backward tensor maps";
        return cudaErrorInvalidValue;
    }
    BwdParams p{};
    p.O = static_cast<const bf16*>(a.O);
    p.dO = static_cast<const bf16*>(a.dO);
    p.LSE = a.LSE;
    p.union_idx = a.union_idx;
    p.union_cnt = a.union_cnt;
    p.sel_idx = a.sel_idx;
    p.sel_logg = a.sel_logg;
    p.dQ = static_cast<bf16*>(a.dQ);
    p.dK = static_cast<bf16*>(a.dK);
    p.dV = static_cast<bf16*>(a.dV);
    p.dlogg = G > 1 ? a.dlogg_heads : a.dlogg;   // pass 1 writes per query head
    p.delta = a.delta;
    p.inv_off = a.inv_off;
    p.inv_tiles = a.inv_tiles;
    p.inv_pos = a.inv_pos;
    p.slot_off = a.slot_off;
    p.offs = a.offs;
    p.tiles = a.tiles;
    p.ntiles = a.ntiles;
    p.tile_off = a.tile_off;
    p.seg_rows = a.seg_rows;
    p.nseg = a.nseg;
    p.seg_cap = a.seg_cap;
    p.seg_union_idx = a.seg_union_idx;
    p.seg_union_cnt = a.seg_union_cnt;
    p.N = a.N; p.C = a.C; p.T = a.T; p.BH = a.BH; p.topk = a.topk; p.mode = a.mode;
    p.G = G;
    p.sm_scale = a.sm_scale;
    p.scale_log2 = a.sm_scale * kLog2eB;
    p.status = env.status;
    p.limit = env.limit;
    // pass 1 tiles: (query head, tile), head-packed (KV group, segment)
    const long long tiles = hp ? static_cast<long long>(BHkv) * a.nseg : static_cast<long long>(a.BH) * a.T;
    const long long gtiles = static_cast<long long>(BHkv) * a.T;       // (KV group, key pair)
    const int nsrc = hp ? a.nseg : a.T;                                 // union lists per group
    const long long srcs = static_cast<long long>(BHkv) * nsrc;
    if (tiles > 0x7fffffffLL) { *err = "backward: too many tiles"; return cudaErrorInvalidValue; }
    // pass 1 (also writes Delta for pass 2); both halves of a row add into dlogg
    const long long per_head = static_cast<long long>(a.N) * (a.topk > 0 ? a.topk : 1);
    cudaError_t e0 = cudaMemsetAsync(p.dlogg, 0, static_cast<size_t>(a.BH) * per_head * 4, env.stream);
    if (e0 != cudaSuccess) { *err = "backward dlogg"; return e0; }
    // outer gate position with gates (training mode); without gates it is the inner form
    const bool outer = a.pos == 1 && a.mode == 0;
    {
        const dim3 g1(static_cast<unsigned>(tiles));
        if (hp && outer) bwd_dq_kernel<true, true><<<g1, kThreadsB, kDqSmem, env.stream>>>(mq, mdo, mk, mv, p);
        else if (hp) bwd_dq_kernel<true, false><<<g1, kThreadsB, kDqSmem, env.stream>>>(mq, mdo, mk, mv, p);
        else if (outer) bwd_dq_kernel<false, true><<<g1, kThreadsB, kDqSmem, env.stream>>>(mq, mdo, mk, mv, p);
        else bwd_dq_kernel<false, false><<<g1, kThreadsB, kDqSmem, env.stream>>>(mq, mdo, mk, mv, p);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) { *err = "backward pass 1"; return e; }
    if (!a.gate_only) {   // a gate-only pass (the STE gate gradient) has no pass 2
        // inverted lists of the KV groups' union lists
        e = cudaMemsetAsync(a.inv_cnt, 0, static_cast<size_t>(gtiles) * 4, env.stream);
        if (e != cudaSuccess) { *err = "backward list counts"; return e; }
        const unsigned gb = static_cast<unsigned>((srcs + 255) / 256);
        const int32_t* uidx = hp ? a.seg_union_idx : a.union_idx;
        const int32_t* ucnt = hp ? a.seg_union_cnt : a.union_cnt;
        const int ustride = hp ? a.seg_cap : a.C;
        bwd_inv_count_kernel<<<gb, 256, 0, env.stream>>>(uidx, ucnt, a.inv_cnt, BHkv, a.T, nsrc, ustride, a.tiles,
                                                          a.ntiles, a.tile_off, hp ? G : 0);
        bwd_inv_scan_kernel<<<1, 1024, 0, env.stream>>>(a.inv_cnt, a.inv_off, a.inv_cursor, gtiles);
        bwd_inv_fill_kernel<<<gb, 256, 0, env.stream>>>(uidx, ucnt, a.inv_cursor, a.inv_tiles, a.inv_pos, BHkv, a.T,
                                                         nsrc, ustride, a.tiles, a.ntiles, a.tile_off, hp ? G : 0);
        e = cudaGetLastError();
        if (e != cudaSuccess) { *err = "backward inverted lists"; return e; }
        // pass 2: one CTA per (KV group, key pair)
        const dim3 g2(static_cast<unsigned>(gtiles));
        if (hp && outer) bwd_dkv_kernel<true, true><<<g2, kThreadsD, kDkvSmem, env.stream>>>(mq, mdo, mk2, mv2, p);
        else if (hp) bwd_dkv_kernel<true, false><<<g2, kThreadsD, kDkvSmem, env.stream>>>(mq, mdo, mk2, mv2, p);
        else if (outer) bwd_dkv_kernel<false, true><<<g2, kThreadsD, kDkvSmem, env.stream>>>(mq, mdo, mk2, mv2, p);
        else bwd_dkv_kernel<false, false><<<g2, kThreadsD, kDkvSmem, env.stream>>>(mq, mdo, mk2, mv2, p);
        e = cudaGetLastError();
        if (e != cudaSuccess) { *err = "backward pass 2"; return e; }
    }
    if (G > 1 && a.topk > 0) {
        const long long total = static_cast<long long>(BHkv) * per_head;
        bwd_dlogg_sum_kernel<<<static_cast<unsigned>((total + 255) / 256), 256, 0, env.stream>>>(
            a.dlogg_heads, a.dlogg, per_head, total, G);
        e = cudaGetLastError();
        if (e != cudaSuccess) { *err = "backward gate-gradient sum"; return e; }
    } else if (G > 1) {
        e = cudaMemsetAsync(a.dlogg, 0, static_cast<size_t>(BHkv) * per_head * 4, env.stream);
        if (e != cudaSuccess) { *err = "backward dlogg"; return e; }
    }
    if (a.scores != nullptr && a.ds != nullptr && a.topk > 0) {
        // one warp per row, at most 32 KB of shared memory per CTA; packed
        // sequences: a power of two of warps, so that runs tile 128 rows
        int wpc = max(1, min(8, 8192 / a.C));
        if (a.tiles != nullptr) wpc = 1 << (31 - __builtin_clz(static_cast<unsigned>(wpc)));
        const size_t sh = static_cast<size_t>(wpc) * a.C * sizeof(float);
        const int chunks = a.tiles != nullptr ? a.T * (kRows / wpc) : (a.N + wpc - 1) / wpc;
        const unsigned grid = static_cast<unsigned>(static_cast<long long>(BHkv) * chunks);
        const int train = a.mode == 0 ? 1 : 0;
        if (a.C <= 128)
            bwd_ds_kernel<4><<<grid, 32 * wpc, sh, env.stream>>>(a.scores, a.sel_idx, a.sel_logg, a.dlogg, a.ds, a.N,
                                                                 a.C, a.topk, train, a.act, chunks, a.tiles, a.ntiles);
        else if (a.C <= 384)
            bwd_ds_kernel<12><<<grid, 32 * wpc, sh, env.stream>>>(a.scores, a.sel_idx, a.sel_logg, a.dlogg, a.ds, a.N,
                                                                  a.C, a.topk, train, a.act, chunks, a.tiles, a.ntiles);
        else
            bwd_ds_kernel<0><<<grid, 32 * wpc, sh, env.stream>>>(a.scores, a.sel_idx, a.sel_logg, a.dlogg, a.ds, a.N,
                                                                 a.C, a.topk, train, a.act, chunks, a.tiles, a.ntiles);
        e = cudaGetLastError();
        if (e != cudaSuccess) { *err = "backward score gradient"; return e; }
    } else if (a.ds != nullptr) {
        e = cudaMemsetAsync(a.ds, 0, static_cast<size_t>(BHkv) * a.N * a.C * 4, env.stream);
        if (e != cudaSuccess) { *err = "backward score gradient"; return e; }
    }
    return cudaSuccess;
}

}  // namespace sas
