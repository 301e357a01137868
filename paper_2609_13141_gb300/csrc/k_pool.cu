// a1: block summaries for the learned selector.
//
//   Kbar_m = (1/64) sum_{j in B_m} k_j            (pooled block summary)
//   K~_m   = bf16(Wk[h] Kbar_m)                    (selector key projection)
//
// for the F = floor(N/64) full blocks of every (batch, head): a partial last
// block is never historical for any query, so it is never summarised.  One
// CTA handles 8 consecutive blocks of one head: warp w streams block w's 64
// key rows with coalesced 8-byte loads (a warp covers one 256-byte row) and
// keeps fp32 column sums in registers; the CTA then projects the 8 summaries
// with Wk[h] staged row-major in shared memory (rows padded by one word so
// that the 32 threads of a warp, one output each, hit distinct banks).  The pass is HBM-bound: it
// reads every full-block key once and writes 2*d_sel bytes per block.
#include "internal.h"
#include "ptx.cuh"

namespace sas {
namespace {

constexpr int kGroup = 8;   // blocks per CTA == warps per CTA

template <int D, int DS>
__global__ void __launch_bounds__(256) pool_kernel(const bf16* __restrict__ K, const bf16* __restrict__ Wk,
                                                    bf16* __restrict__ Kt, int H, int N, int F) {
    __shared__ float kbar[kGroup][D];
    __shared__ __align__(16) bf16 ws[DS][D + 2];   // ws[j][k] = Wk[h][j][k]

    const int bh = blockIdx.y;
    const int h = bh % H;
    const int m0 = blockIdx.x * kGroup;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const bf16* w = Wk + static_cast<long long>(h) * DS * D;
    for (int e = threadIdx.x; e < DS * D; e += blockDim.x) {
        const int j = e / D, k = e - j * D;
        ws[j][k] = w[e];
    }

    const int m = m0 + warp;
    constexpr int PER = D / 32;
    if (m < F) {
        float acc[PER];
#pragma unroll
        for (int q = 0; q < PER; ++q) acc[q] = 0.f;
        const bf16* base = K + (static_cast<long long>(bh) * N + static_cast<long long>(m) * 64) * D + lane * PER;
#pragma unroll 4
        for (int t = 0; t < 64; ++t) {
            const bf16* rp = base + static_cast<long long>(t) * D;
            if constexpr (PER == 4) {
                const uint2 u = *reinterpret_cast<const uint2*>(rp);
                const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&u.x);
                const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162*>(&u.y);
                acc[0] += __low2float(a);
                acc[1] += __high2float(a);
                acc[2] += __low2float(b);
                acc[3] += __high2float(b);
            } else {
                const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(rp);
                acc[0] += __low2float(a);
                acc[1] += __high2float(a);
            }
        }
#pragma unroll
        for (int q = 0; q < PER; ++q) kbar[warp][lane * PER + q] = acc[q] * (1.0f / 64.0f);
    }
    __syncthreads();

    for (int o = threadIdx.x; o < kGroup * DS; o += blockDim.x) {
        const int g = o / DS, j = o - g * DS;
        const int mm = m0 + g;
        if (mm >= F) continue;
        float s = 0.f;
#pragma unroll 8
        for (int k = 0; k < D; ++k) s = fmaf(kbar[g][k], __bfloat162float(ws[j][k]), s);
        Kt[(static_cast<long long>(bh) * F + mm) * DS + j] = __float2bfloat16_rn(s);
    }
}

template <int D, int DS>
cudaError_t launch_dd(const void* K, const void* Wk, void* Kt, int BH, int H, int N, const KernelEnv& env) {
    const int F = N / 64;
    if (F == 0) return cudaSuccess;
    dim3 grid((F + kGroup - 1) / kGroup, BH);
    pool_kernel<D, DS><<<grid, 256, 0, env.stream>>>(static_cast<const bf16*>(K), static_cast<const bf16*>(Wk),
                                                     static_cast<bf16*>(Kt), H, N, F);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_pool(const void* K, const void* Wk, void* Kt, int BH, int H, int N, int d, int d_sel,
                        const KernelEnv& env) {
    if (d == 128 && d_sel == 128) return launch_dd<128, 128>(K, Wk, Kt, BH, H, N, env);
    if (d == 128 && d_sel == 64) return launch_dd<128, 64>(K, Wk, Kt, BH, H, N, env);
    if (d == 64 && d_sel == 64) return launch_dd<64, 64>(K, Wk, Kt, BH, H, N, env);
    if (d == 64 && d_sel == 128) return launch_dd<64, 128>(K, Wk, Kt, BH, H, N, env);
    return cudaErrorInvalidValue;
}

}  // namespace sas
