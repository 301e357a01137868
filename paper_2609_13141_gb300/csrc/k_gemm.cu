// Persistent warp-specialised bf16 GEMM on the 5th-generation tensor cores.
//
//   C[b] = epi(A[b] @ B[b % b_mod]^T + bias)        (fp32 accumulate, bf16 out)
//
// Used for the dense MLP sublayer (up-projection with an exact-GELU epilogue,
// then the down-projection) and for the selector's batched per-head query
// projection.  Design:
//   * one CTA per SM, static round-robin over 128 x BN output tiles, grouped
//     along M so that concurrently running CTAs share operand tiles in L2;
//   * warp 0 streams 128x64 A and BNx64 B tiles with TMA (128-byte swizzle)
//     into a ring of shared-memory stages guarded by mbarriers;
//   * warp 1 (one lane) issues tcgen05.mma (M=128, N=BN, K=16) into one of
//     two TMEM accumulators and releases stages with tcgen05.commit;
//   * warps 2-5 drain the other accumulator (tcgen05.ld), apply bias/GELU in
//     fp32, write bf16 into a per-warp 128-byte-swizzled staging tile and send
//     each 32 x 64 block out with a TMA tensor store (per-thread row stores
//     scattered over 32 rows cost 6% of the GEMM), overlapping the next tile's
//     main loop.
#include "internal.h"
#include "ptx.cuh"

namespace sas {
namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kThreads = 192;

template <int BN>
struct GemmCfg {
    static constexpr int A_BYTES = kBM * kBK * 2;
    static constexpr int B_BYTES = BN * kBK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int STAGES = BN == 256 ? 4 : (BN == 128 ? 6 : 8);
    static constexpr int TMEM_COLS = 2 * BN;
    // per epilogue warp two 32-row x 64-column bf16 staging tiles (4 KB each)
    static constexpr int OFF_STAGING = STAGES * STAGE_BYTES;
    static constexpr int STAGING_BYTES = 4 * 2 * 4096;
    static constexpr int SMEM = OFF_STAGING + STAGING_BYTES + 1024;
    static constexpr uint32_t IDESC = idesc_bf16(kBM, BN, 0, 0);
};

struct GemmParams {
    bf16* C;
    const bf16* bias;
    int M, N, K;
    int batches, b_mod;
    long long c_batch_stride;
    int ldc;
    int gelu;
    int* status;
    long long limit;
};

constexpr int kGroupM = 16;
// Every wait in this kernel sleeps while it waits (measured: 4.5% faster for the
// up-projection than polling, which takes issue slots from the epilogue warps).
constexpr uint32_t kSuspendNs = 1000;

__device__ __forceinline__ void tile_coords(int t, int m_tiles, int n_tiles, int& b, int& m, int& n) {
    const int per_batch = m_tiles * n_tiles;
    b = t / per_batch;
    const int r = t - b * per_batch;
    const int group_span = kGroupM * n_tiles;
    const int g = r / group_span;
    const int first_m = g * kGroupM;
    const int gsize = min(m_tiles - first_m, kGroupM);
    const int rr = r - g * group_span;
    m = first_m + rr % gsize;
    n = rr / gsize;
}

__device__ __forceinline__ float gelu_erf(float x) {
    return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}

template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
gemm_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
            const __grid_constant__ CUtensorMap mapC, GemmParams p) {
    using Cfg = GemmCfg<BN>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    __shared__ uint64_t full_bar[Cfg::STAGES], empty_bar[Cfg::STAGES];
    __shared__ uint64_t tfull_bar[2], tempty_bar[2], drain_bar;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int abort_flag;

    const uint32_t warp = warp_id(), lane = lane_id();
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + ((1024u - (raw & 1023u)) & 1023u);

    const int m_tiles = (p.M + kBM - 1) / kBM;
    const int n_tiles = p.N / BN;
    const int total = p.batches * m_tiles * n_tiles;
    const int kblocks = p.K / kBK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < Cfg::STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull_bar[a], 1);
            mbar_init(&tempty_bar[a], 128);
        }
        mbar_init(&drain_bar, 1);
        abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc(&tmem_base_sh, Cfg::TMEM_COLS);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = tmem_base_sh;
    const WaitCtl wc{&abort_flag, p.status, p.limit};

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer
        tma_prefetch_desc(&mapA);
        tma_prefetch_desc(&mapB);
        int s = 0;
        uint32_t ph = 0;
        long long issued = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < total && ok; t += gridDim.x) {
            int b, m, n;
            tile_coords(t, m_tiles, n_tiles, b, m, n);
            for (int kb = 0; kb < kblocks; ++kb) {
                if (!mbar_wait(&empty_bar[s], ph ^ 1u, wc, kSuspendNs)) { ok = false; break; }
                uint8_t* sa = smem + s * Cfg::STAGE_BYTES;
                mbar_arrive_expect_tx(&full_bar[s], Cfg::STAGE_BYTES);
                tma_load_3d(sa, &mapA, &full_bar[s], kb * kBK, m * kBM, b);
                tma_load_3d(sa + Cfg::A_BYTES, &mapB, &full_bar[s], kb * kBK, n * BN, b % p.b_mod);
                ++issued;
                if (++s == Cfg::STAGES) { s = 0; ph ^= 1u; }
            }
        }
        if (!ok) {
            // Let every load already issued land before the CTA can exit.
            for (long long q = issued - 1; q >= 0 && q >= issued - Cfg::STAGES; --q)
                mbar_wait_drain(&full_bar[q % Cfg::STAGES], static_cast<uint32_t>((q / Cfg::STAGES) & 1),
                                p.limit, p.status);
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer
        int s = 0;
        uint32_t ph = 0;
        int it = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < total && ok; t += gridDim.x, ++it) {
            const int acc = it & 1;
            const uint32_t aph = (it >> 1) & 1;
            if (!mbar_wait(&tempty_bar[acc], aph ^ 1u, wc, kSuspendNs)) break;
            tc_fence_after();
            const uint32_t d_tmem = tmem_base + acc * BN;
            for (int kb = 0; kb < kblocks; ++kb) {
                if (!mbar_wait(&full_bar[s], ph, wc, kSuspendNs)) { ok = false; break; }
                tc_fence_after();
                const uint32_t a_addr = smem_u32(smem + s * Cfg::STAGE_BYTES);
                const uint32_t b_addr = a_addr + Cfg::A_BYTES;
#pragma unroll
                for (int k = 0; k < kBK / 16; ++k) {
                    const uint64_t ad = smem_desc_sw128(a_addr + k * 32, 16, 1024);
                    const uint64_t bd = smem_desc_sw128(b_addr + k * 32, 16, 1024);
                    umma_bf16(d_tmem, ad, bd, Cfg::IDESC, (kb | k) != 0);
                }
                umma_commit(&empty_bar[s]);
                if (++s == Cfg::STAGES) { s = 0; ph ^= 1u; }
            }
            if (!ok) break;
            umma_commit(&tfull_bar[acc]);
        }
        umma_commit(&drain_bar);
        mbar_wait_drain(&drain_bar, 0, p.limit, p.status);
    } else if (warp >= 2) {
        // ---------------- epilogue: TMEM -> registers -> bias/GELU -> bf16 -> staging -> TMA store
        const int q = warp & 3;
        const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
        uint8_t* staging = smem + Cfg::OFF_STAGING + q * 2 * 4096;
        if (lane == 0) tma_prefetch_desc(&mapC);
        int it = 0;
        int nst = 0;   // stores issued by this warp (staging buffer = nst & 1)
        for (int t = blockIdx.x; t < total; t += gridDim.x, ++it) {
            const int acc = it & 1;
            const uint32_t aph = (it >> 1) & 1;
            if (!mbar_wait_warp(&tfull_bar[acc], aph, wc, kSuspendNs)) break;
            tc_fence_after();
            int b, m, n;
            tile_coords(t, m_tiles, n_tiles, b, m, n);
#pragma unroll 1
            for (int cg = 0; cg < BN / 64; ++cg, ++nst) {
                uint8_t* buf = staging + (nst & 1) * 4096;
                // the store issued from this buffer two groups ago has finished reading it
                if (lane == 0) bulk_wait_read<1>();
                __syncwarp();
#pragma unroll 1
                for (int hh = 0; hh < 2; ++hh) {
                    const int c = cg * 2 + hh;
                    uint32_t r[32];
                    tmem_ld32(lane_addr + acc * BN + c * 32, r);
                    tmem_wait_ld();
                    float v[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
                    if (p.bias != nullptr) {
                        const bf16* bp = p.bias + n * BN + c * 32;
#pragma unroll
                        for (int j = 0; j < 32; ++j) v[j] += __bfloat162float(bp[j]);
                    }
                    if (p.gelu) {
#pragma unroll
                        for (int j = 0; j < 32; ++j) v[j] = gelu_erf(v[j]);
                    }
                    // row `lane` of the staging tile: 16-byte chunk k of the row at k ^ (lane & 7)
                    uint8_t* row = buf + lane * 128;
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        uint4 w;
                        w.x = pack_bf16x2(v[8 * j + 0], v[8 * j + 1]);
                        w.y = pack_bf16x2(v[8 * j + 2], v[8 * j + 3]);
                        w.z = pack_bf16x2(v[8 * j + 4], v[8 * j + 5]);
                        w.w = pack_bf16x2(v[8 * j + 6], v[8 * j + 7]);
                        const int k = hh * 4 + j;
                        *reinterpret_cast<uint4*>(row + ((k ^ (lane & 7)) << 4)) = w;
                    }
                }
                fence_proxy_async_smem();
                __syncwarp();
                // rows past M are clipped by the tensor store
                if (lane == 0) {
                    tma_store_3d(&mapC, buf, n * BN + cg * 64, m * kBM + q * 32, b);
                    bulk_commit();
                }
            }
            tc_fence_before();
            mbar_arrive(&tempty_bar[acc]);
        }
        if (lane == 0) bulk_wait_all();
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
    }
}

template <int BN>
cudaError_t launch_bn(const GemmProblem& p, const KernelEnv& env, const char** err) {
    using Cfg = GemmCfg<BN>;
    {
        cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(gemm_kernel<BN>), Cfg::SMEM);
        if (e != cudaSuccess) { *err = "cudaFuncSetAttribute(gemm)"; return e; }
    }
    if (p.ldc != p.N || (p.batches > 1 && p.c_batch_stride != static_cast<long long>(p.M) * p.N)) {
        *err = "gemm: C must be a dense [batches][M][N] tensor";
        return cudaErrorInvalidValue;
    }
    CUtensorMap ma, mb, mc;
    const int nb = p.b_mod;
    if (make_tmap_bf16_3d(&ma, p.A, p.K, p.M, p.batches, kBK, kBM) != 0) { *err = "tensor map A"; return cudaErrorInvalidValue; }
    if (make_tmap_bf16_3d(&mb, p.B, p.K, p.N, nb, kBK, BN) != 0) { *err = "tensor map B"; return cudaErrorInvalidValue; }
    if (make_tmap_bf16_3d(&mc, p.C, p.N, p.M, p.batches, 64, 32) != 0) { *err = "tensor map C"; return cudaErrorInvalidValue; }
    GemmParams gp;
    gp.C = static_cast<bf16*>(p.C);
    gp.bias = static_cast<const bf16*>(p.bias);
    gp.M = p.M; gp.N = p.N; gp.K = p.K;
    gp.batches = p.batches; gp.b_mod = p.b_mod;
    gp.c_batch_stride = p.c_batch_stride; gp.ldc = p.ldc; gp.gelu = p.gelu;
    gp.status = env.status; gp.limit = env.limit;
    const long long tiles = static_cast<long long>(p.batches) * ((p.M + kBM - 1) / kBM) * (p.N / BN);
    int grid = p.max_ctas > 0 ? p.max_ctas : device_sm_count();
    if (tiles < grid) grid = static_cast<int>(tiles);
    gemm_kernel<BN><<<grid, kThreads, Cfg::SMEM, env.stream>>>(ma, mb, mc, gp);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) *err = "gemm launch";
    return e;
}

}  // namespace

cudaError_t launch_gemm(const GemmProblem& p, const KernelEnv& env, const char** err) {
    switch (p.bn) {
        case 256: return launch_bn<256>(p, env, err);
        case 128: return launch_bn<128>(p, env, err);
        case 64: return launch_bn<64>(p, env, err);
        default: *err = "gemm: unsupported tile width"; return cudaErrorInvalidValue;
    }
}

}  // namespace sas
