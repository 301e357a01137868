// a1: block summaries for the learned selector.
//
//   Kbar_m = (1/64) sum_{j in B_m} k_j            (pooled block summary)
//   K~_m   = bf16(Wk[h] Kbar_m)                    (selector key projection)
//
// for the F = floor(N/64) full blocks of every (batch, head): a partial last
// block is never historical for any query, so it is never summarised.  One
// CTA handles 8 consecutive blocks of one head: warp w streams block w's 64
// key rows with coalesced 16-byte loads (sixteen in flight per lane) and
// keeps fp32 column sums in registers; the CTA then projects the 8 summaries
// with Wk[h] staged row-major in shared memory (rows padded by one word so
// that the 32 threads of a warp, one output each, hit distinct banks).  The pass is HBM-bound: it
// reads every full-block key once and writes 2*d_sel bytes per block.
//
// Packed sequences: blocks restart at every sequence's first token.  Block m
// of sequence s (tokens cu[s] + 64 m .. + 63) goes to summary slot
// floor(cu[s] / 64) + s + m: the slots of different sequences never overlap
// (floor((a + b) / 64) >= floor(a / 64) + floor(b / 64)), and a head needs at
// most N / 64 + max_seqs of them.  The CTAs walk the selection pass's tile
// table: tile t of a sequence covers its blocks 2t and 2t + 1.
#include "internal.h"
#include "ptx.cuh"

namespace sas {
namespace {

constexpr int kGroup = 8;   // blocks per CTA == warps per CTA

template <int D, int DS>
__global__ void __launch_bounds__(256) pool_kernel(const bf16* __restrict__ K, const bf16* __restrict__ Wk,
                                                    bf16* __restrict__ Kt, int H, int N, int F,
                                                    const int4* __restrict__ tiles, const int* __restrict__ ntiles) {
    __shared__ float kbar[kGroup][D];
    __shared__ __align__(16) bf16 ws[DS][D + 2];   // ws[j][k] = Wk[h][j][k]; rows 4-byte aligned
    __shared__ int slot_of[kGroup];                // summary slot of each warp's block, -1 if none

    const int bh = blockIdx.y;
    const int h = bh % H;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // this warp's block: its first key row in the head's token axis and its slot
    int first = -1, slot = -1;
    if (tiles == nullptr) {
        const int m = blockIdx.x * kGroup + warp;
        if (m < F) { first = 64 * m; slot = m; }
    } else {
        const int g = blockIdx.x * (kGroup / 2) + warp / 2;   // tile slot: its blocks 2t, 2t + 1
        if (g < __ldg(ntiles)) {
            const int4 v = __ldg(tiles + g);                    // {first row, tile, length, sequence}
            const int lb = 2 * v.y + (warp & 1);
            if (64 * (lb + 1) <= v.z) { first = v.x + 64 * lb; slot = v.x / 64 + v.w + lb; }
        }
    }
    if (lane == 0) slot_of[warp] = slot;

    // Wk[h] rows (D bf16 = D/8 16-byte pieces each) into the padded shared copy
    const bf16* w = Wk + static_cast<long long>(h) * DS * D;
    for (int e = threadIdx.x; e < DS * (D / 8); e += blockDim.x) {
        const int j = e / (D / 8), k8 = (e - j * (D / 8)) * 8;
        const uint4 u = __ldg(reinterpret_cast<const uint4*>(w + j * D + k8));
        const uint32_t* uw = reinterpret_cast<const uint32_t*>(&u);
#pragma unroll
        for (int q = 0; q < 4; ++q) *reinterpret_cast<uint32_t*>(&ws[j][k8 + 2 * q]) = uw[q];
    }

    // Warp w sums block m0 + w.  A key row is D * 2 bytes: D / 8 lanes cover it
    // with 16-byte loads, so one warp instruction reads LPR = 256 / D rows and
    // each lane keeps fp32 sums of 8 dims over its rows.
    constexpr int LANES_PER_ROW = D / 8;
    constexpr int ROWS_PER_STEP = 32 / LANES_PER_ROW;
    if (slot >= 0) {
        const int sub = lane / LANES_PER_ROW;            // which of the step's rows
        const int dl = (lane % LANES_PER_ROW) * 8;       // first of this lane's 8 dims
        float acc[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] = 0.f;
        const bf16* base = K + (static_cast<long long>(bh) * N + first + sub) * D + dl;
        // issue all of the lane's row loads before summing (16 in flight)
        constexpr int STEPS = 64 / ROWS_PER_STEP;
#pragma unroll
        for (int t0 = 0; t0 < STEPS; t0 += 16) {
            uint4 u[16];
#pragma unroll
            for (int t = 0; t < 16; ++t)
                u[t] = __ldg(reinterpret_cast<const uint4*>(base + static_cast<long long>(t0 + t) * ROWS_PER_STEP * D));
#pragma unroll
            for (int t = 0; t < 16; ++t) {
                const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&u[t]);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    acc[2 * q] += __low2float(h2[q]);
                    acc[2 * q + 1] += __high2float(h2[q]);
                }
            }
        }
        // fold the partial sums of the lanes that share dims
#pragma unroll
        for (int off = LANES_PER_ROW; off < 32; off <<= 1) {
#pragma unroll
            for (int q = 0; q < 8; ++q) acc[q] += __shfl_xor_sync(0xffffffffu, acc[q], off);
        }
        if (sub == 0) {
#pragma unroll
            for (int q = 0; q < 8; ++q) kbar[warp][dl + q] = acc[q] * (1.0f / 64.0f);
        }
    }
    __syncthreads();

    for (int o = threadIdx.x; o < kGroup * DS; o += blockDim.x) {
        const int g = o / DS, j = o - g * DS;
        const int sl = slot_of[g];
        if (sl < 0) continue;
        float s = 0.f;
#pragma unroll 8
        for (int k = 0; k < D; ++k) s = fmaf(kbar[g][k], __bfloat162float(ws[j][k]), s);
        Kt[(static_cast<long long>(bh) * F + sl) * DS + j] = __float2bfloat16_rn(s);
    }
}

// F: summary slots per head (N / 64, or N / 64 + max_seqs for packed sequences);
// tiles / ntiles / T: the packed sequences' tile table and its slot count (null otherwise).
template <int D, int DS>
cudaError_t launch_dd(const void* K, const void* Wk, void* Kt, int BH, int H, int N, int F, const int4* tiles,
                      const int* ntiles, int T, const KernelEnv& env) {
    if (F == 0) return cudaSuccess;
    const int gx = tiles == nullptr ? (F + kGroup - 1) / kGroup : (T + kGroup / 2 - 1) / (kGroup / 2);
    if (gx == 0) return cudaSuccess;
    dim3 grid(gx, BH);
    pool_kernel<D, DS><<<grid, 256, 0, env.stream>>>(static_cast<const bf16*>(K), static_cast<const bf16*>(Wk),
                                                     static_cast<bf16*>(Kt), H, N, F, tiles, ntiles);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_pool(const void* K, const void* Wk, void* Kt, int BH, int H, int N, int d, int d_sel,
                        const KernelEnv& env, int F, const int4* tiles, const int* ntiles, int T) {
    if (F < 0) F = N / 64;
    if (d == 128 && d_sel == 128) return launch_dd<128, 128>(K, Wk, Kt, BH, H, N, F, tiles, ntiles, T, env);
    if (d == 128 && d_sel == 64) return launch_dd<128, 64>(K, Wk, Kt, BH, H, N, F, tiles, ntiles, T, env);
    if (d == 64 && d_sel == 64) return launch_dd<64, 64>(K, Wk, Kt, BH, H, N, F, tiles, ntiles, T, env);
    if (d == 64 && d_sel == 128) return launch_dd<64, 128>(K, Wk, Kt, BH, H, N, F, tiles, ntiles, T, env);
    return cudaErrorInvalidValue;
}

}  // namespace sas
