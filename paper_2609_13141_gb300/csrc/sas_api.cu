// C ABI of the SAS library: argument checking, workspace ownership, launch
// sequencing on the caller's stream, per-kernel event timing and the device
// status word.  All arithmetic happens in the kernels of k_*.cu.
#include <cmath>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <string>
#include <algorithm>
#include <vector>

#include <cudaTypedefs.h>

#include "../../include/sas.h"
#include "internal.h"
#include "ptx.cuh"

namespace sas {

// ------------------------------------------------------------ tensor maps

namespace {
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

void resolve_encode() {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
        g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
}
}  // namespace

int make_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows, uint64_t outer,
                      uint32_t box_inner, uint32_t box_rows) {
    std::call_once(g_encode_once, resolve_encode);
    if (g_encode == nullptr) return -1;
    cuuint64_t dims[3] = {inner, rows, outer};
    cuuint64_t strides[2] = {inner * 2, inner * rows * 2};
    cuuint32_t box[3] = {box_inner, box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return static_cast<int>(r);
}

// --------------------------------------------- per-device launch attributes

namespace {
std::mutex g_attr_mutex;
std::map<std::pair<const void*, int>, size_t> g_smem_attr;   // (kernel, device) -> limit set
std::map<int, int> g_sms;                                     // device -> SM count
}  // namespace

cudaError_t ensure_smem_attr(const void* func, size_t bytes, bool max_carveout) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(g_attr_mutex);
    size_t& set = g_smem_attr[{func, dev}];
    if (bytes <= set) return cudaSuccess;
    e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes));
    if (e == cudaSuccess && max_carveout)
        e = cudaFuncSetAttribute(func, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
    if (e == cudaSuccess) set = bytes;
    return e;
}

int device_sm_count() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    std::lock_guard<std::mutex> lock(g_attr_mutex);
    int& n = g_sms[dev];
    if (n <= 0) {
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        if (n <= 0) n = 1;
    }
    return n;
}

// ------------------------------------------------------- failure self test

namespace {
__global__ void wait_selftest_kernel(int* status, long long limit) {
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);   // nothing ever arrives
        abort_flag = 0;
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const WaitCtl wc{&abort_flag, status, limit};
        mbar_wait(&bar, 0, wc);
    }
}
}  // namespace

cudaError_t launch_wait_selftest(int* status, long long limit, cudaStream_t stream) {
    wait_selftest_kernel<<<1, 32, 0, stream>>>(status, limit);
    return cudaGetLastError();
}

}  // namespace sas

// ================================================================ handle

namespace {

constexpr long long kDefaultWaitLimit = 4000000000LL;   // ~2 s of SM clock per wait

struct TimeRec {
    int kind;
    cudaEvent_t a, b;
};

}  // namespace

struct sas_handle {
    sas_config cfg;
    int device = 0;
    int d_sel = 0;
    float sm_scale = 0.f;
    int BH = 0, C = 0, T = 0, F = 0;
    int Hkv = 0, G = 1, BHkv = 0;   // KV heads, query heads per group, KV groups x batch
    bool varlen = false;            // packed sequences: T = tile slots, C from max_seqlen
    // head-packed GQA attention tiles (G >= 2, 128 = G seg_rows): segment unions
    int seg_rows = 0, nseg = 0, seg_cap = 0;
    int32_t* seg_union_idx = nullptr;   // [BHkv][nseg][seg_cap]
    int32_t* seg_union_cnt = nullptr;   // [BHkv][nseg]
    int last_fwd = 0;                   // tiles of the last forward: 0 per head, 1 head-packed, 2 packed sequences
    int4* tiles = nullptr;          // packed sequences' tile table [T] and its count
    int* ntiles = nullptr;
    int* tile_off = nullptr;    // first slot of every local tile index (see launch_varlen_tiles)
    // workspace
    void* Kt = nullptr;         // bf16 [BH][max(F,1)][d_sel]
    int32_t* union_idx = nullptr;
    int32_t* union_cnt = nullptr;
    int32_t* sel_idx = nullptr;
    float* sel_logg = nullptr;
    int* status = nullptr;
    int* sched = nullptr;       // attention work counters (zero between launches)
    bool full = false;          // full training scope
    float* full_lse = nullptr;  // [BHkv][N] row normalisers of the scores
    float* full_table = nullptr;   // learned selector, full scope: scores [BHkv][N][C]
    // MLP hidden activation
    void* hidden = nullptr;
    size_t hidden_bytes = 0;
    // backward workspace (allocated by the first sas_attention_bwd)
    float* bwd_delta = nullptr;
    int32_t* bwd_inv = nullptr;     // counts, cursors, offsets, slot offsets
    int32_t* bwd_tiles = nullptr;   // inverted lists: tiles, then block positions
    float* bwd_dlogg = nullptr;     // GQA: per query head [BH][N][topk], then per group [BHkv][N][topk]
    float* bwd_offs = nullptr;      // per-row offsets of every visited block (pass 1 -> pass 2)
    // full scope and hard-STE backwards: lists of every historical block
    int32_t* dense_idx = nullptr;   // [BHkv][N][C] block indices 0 .. C_i - 1
    float* dense_lg = nullptr;      // [BHkv][N][C] their log-gates s - LSE
    int32_t* dense_uidx = nullptr;  // [BHkv][T][C] tile unions (every block below the diagonal)
    int32_t* dense_ucnt = nullptr;  // [BHkv][T]
    float* dense_lse = nullptr;     // [BHkv][N] soft normalisers of the given scores (hard-STE)
    size_t bwd_offs_bytes = 0;
    bool bwd_offs_bound = false;    // sized for the upper bound: no per-call read-back
    // timing
    bool timing = false;
    std::vector<TimeRec> recs;
    std::vector<cudaEvent_t> events;
    size_t events_used = 0;
    int64_t launches = 0;
    long long limit = kDefaultWaitLimit;
    std::string last_error;
};

namespace {

sas_status fail(sas_handle* h, sas_status s, const std::string& msg) {
    if (h) h->last_error = msg;
    return s;
}

sas_status cuda_fail(sas_handle* h, cudaError_t e, const char* what) {
    std::string m = std::string(what ? what : "cuda") + ": " + cudaGetErrorString(e);
    return fail(h, e == cudaErrorMemoryAllocation ? SAS_ERR_OOM : SAS_ERR_CUDA, m);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Gate form the forward kernels run: the hard-STE mode's forward is the hard one.
int kernel_mode(const sas_config& c) { return c.mode == SAS_MODE_TRAIN_HARD_STE ? SAS_MODE_INFER_HARD : c.mode; }
bool aligned4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }

cudaEvent_t next_event(sas_handle* h) {
    if (h->events_used == h->events.size()) {
        cudaEvent_t e;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        h->events.push_back(e);
    }
    return h->events[h->events_used++];
}

// Runs one kernel launch, bracketed by events when timing is on.
template <class Fn>
cudaError_t timed_launch(sas_handle* h, int kind, cudaStream_t s, Fn&& fn) {
    cudaEvent_t a = nullptr, b = nullptr;
    if (h->timing) {
        a = next_event(h);
        b = next_event(h);
        if (a) cudaEventRecord(a, s);
    }
    cudaError_t e = fn();
    if (e == cudaSuccess) ++h->launches;
    if (h->timing && a && b) {
        cudaEventRecord(b, s);
        h->recs.push_back({kind, a, b});
    }
    return e;
}

template <class T>
cudaError_t alloc(T** p, size_t bytes) {
    void* v = nullptr;
    cudaError_t e = cudaMalloc(&v, bytes < 16 ? 16 : bytes);
    *p = static_cast<T*>(v);
    return e;
}

sas_status check_device(sas_handle* h) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaGetDevice");
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (major != 10 || minor != 3)
        return fail(h, SAS_ERR_UNSUPPORTED, "device is not sm_103 (GB300); the kernels are built for sm_103a only");
    return SAS_OK;
}

}  // namespace

// ================================================================ C ABI

extern "C" {

const char* sas_status_str(sas_status s) {
    switch (s) {
        case SAS_OK: return "ok";
        case SAS_ERR_INVALID_ARG: return "invalid argument";
        case SAS_ERR_UNSUPPORTED: return "unsupported";
        case SAS_ERR_CUDA: return "cuda error";
        case SAS_ERR_TIMEOUT: return "device wait timed out";
        case SAS_ERR_OOM: return "out of device memory";
    }
    return "unknown status";
}

const char* sas_last_error(const sas_handle* h) { return h ? h->last_error.c_str() : ""; }

sas_status sas_create(const sas_config* cfg, sas_handle** out) {
    if (out == nullptr || cfg == nullptr) return SAS_ERR_INVALID_ARG;
    *out = nullptr;
    const sas_config& c = *cfg;
    if (c.B < 1 || c.H < 1 || c.N < 1) return SAS_ERR_INVALID_ARG;
    if (c.N > (1 << 30)) return SAS_ERR_UNSUPPORTED;   // block indices stay below 2^24
    if (c.block != 64) return SAS_ERR_UNSUPPORTED;
    if (c.d != 64 && c.d != 128) return SAS_ERR_UNSUPPORTED;
    if (c.topk < 0) return SAS_ERR_INVALID_ARG;
    if (c.topk > 64) return SAS_ERR_UNSUPPORTED;
    if (c.mode != SAS_MODE_TRAIN_SOFT && c.mode != SAS_MODE_INFER_HARD && c.mode != SAS_MODE_TRAIN_HARD_STE)
        return SAS_ERR_INVALID_ARG;
    if (c.selector != SAS_SEL_SCORES_GIVEN && c.selector != SAS_SEL_MEANPOOL_PROJ) return SAS_ERR_INVALID_ARG;
    if (c.gate_act != SAS_GATE_SOFTMAX && c.gate_act != SAS_GATE_SIGMOID && c.gate_act != SAS_GATE_LOGIT)
        return SAS_ERR_INVALID_ARG;
    if (c.gate_pos != SAS_GATE_INNER && c.gate_pos != SAS_GATE_OUTER) return SAS_ERR_INVALID_ARG;
    if (!(c.sm_scale >= 0.f) || !std::isfinite(c.sm_scale)) return SAS_ERR_INVALID_ARG;
    if (c.scope != SAS_SCOPE_SPARSE && c.scope != SAS_SCOPE_FULL) return SAS_ERR_INVALID_ARG;
    if (c.scope == SAS_SCOPE_FULL &&
        (c.gate_act != SAS_GATE_SOFTMAX || c.gate_pos != SAS_GATE_INNER || c.max_seqs > 0))
        return SAS_ERR_UNSUPPORTED;
    // the straight-through estimator of the hard gate stands the softmax gates in
    if (c.mode == SAS_MODE_TRAIN_HARD_STE &&
        (c.scope != SAS_SCOPE_SPARSE || c.gate_act != SAS_GATE_SOFTMAX || c.gate_pos != SAS_GATE_INNER))
        return SAS_ERR_UNSUPPORTED;
    const int d_sel = c.d_sel == 0 ? c.d : c.d_sel;
    if (d_sel != 64 && d_sel != 128) return SAS_ERR_UNSUPPORTED;
    const int Hkv = c.Hkv == 0 ? c.H : c.Hkv;
    if (Hkv < 1 || Hkv > c.H || c.H % Hkv != 0) return SAS_ERR_INVALID_ARG;
    if (c.max_seqs < 0 || c.max_seqlen < 0 || c.max_seqlen > c.N) return SAS_ERR_INVALID_ARG;
    const bool varlen = c.max_seqs > 0;
    if (varlen && c.B != 1) return SAS_ERR_INVALID_ARG;
    if (varlen && c.max_seqs > (1 << 20)) return SAS_ERR_UNSUPPORTED;
    const long long BH = static_cast<long long>(c.B) * c.H;
    const long long BHkv = static_cast<long long>(c.B) * Hkv;
    if (BH > (1LL << 30) || BH * c.N > (1LL << 40)) return SAS_ERR_UNSUPPORTED;
    if (BH * ((c.N + 127) / 128) > 0x7fffffffLL) return SAS_ERR_UNSUPPORTED;   // (head, tile) pairs index a 1-D grid

    sas_handle* h = new sas_handle();
    h->cfg = c;
    h->d_sel = d_sel;
    h->sm_scale = c.sm_scale > 0.f ? c.sm_scale : 1.0f / std::sqrt(static_cast<float>(c.d));
    h->BH = static_cast<int>(BH);
    h->Hkv = Hkv;
    h->G = c.H / Hkv;
    h->BHkv = static_cast<int>(BHkv);
    h->varlen = varlen;
    h->full = c.scope == SAS_SCOPE_FULL;
    const int max_len = varlen && c.max_seqlen > 0 ? c.max_seqlen : c.N;
    h->C = (max_len + 63) / 64;
    // packed sequences: at most N / 128 + max_seqs tiles (each sequence adds one partial tile)
    h->T = (c.N + 127) / 128 + (varlen ? c.max_seqs : 0);
    // summary slots per KV group: N / 64 blocks, and with packed sequences one
    // more per sequence (block m of sequence s sits at floor(cu[s] / 64) + s + m)
    h->F = c.N / 64 + (varlen ? c.max_seqs : 0);
    sas_status st = check_device(h);
    if (st != SAS_OK) { delete h; return st; }
    cudaGetDevice(&h->device);

    cudaError_t e = cudaSuccess;
    const size_t rows = static_cast<size_t>(BHkv) * c.N;   // selection rows: one per group and token
    if (c.selector == SAS_SEL_MEANPOOL_PROJ) {
        if (e == cudaSuccess) e = alloc(&h->Kt, static_cast<size_t>(BHkv) * (h->F > 0 ? h->F : 1) * d_sel * 2);
    }
    if (e == cudaSuccess) e = alloc(&h->union_idx, static_cast<size_t>(BHkv) * h->T * h->C * 4);
    if (e == cudaSuccess) e = alloc(&h->union_cnt, static_cast<size_t>(BHkv) * h->T * 4);
    if (e == cudaSuccess) e = alloc(&h->sel_idx, rows * (c.topk > 0 ? c.topk : 1) * 4);
    if (e == cudaSuccess) e = alloc(&h->sel_logg, rows * (c.topk > 0 ? c.topk : 1) * 4);
    if (varlen) {
        if (e == cudaSuccess) e = alloc(&h->tiles, static_cast<size_t>(h->T) * sizeof(int4));
        if (e == cudaSuccess) e = alloc(&h->ntiles, 16);
        if (e == cudaSuccess) e = cudaMemset(h->ntiles, 0, 16);
        if (e == cudaSuccess) e = alloc(&h->tile_off, static_cast<size_t>((max_len + 127) / 128 + 2) * 4);
    }
    // head-packed attention tiles: G query heads x 128 / G tokens share one kept
    // list per token (sparse scope; packed sequences: G segments per tile slot)
    if (!h->full && h->G >= 2 && 128 % h->G == 0 && (128 / h->G) % 8 == 0 && c.topk > 0) {
        h->seg_rows = 128 / h->G;
        h->nseg = varlen ? h->T * h->G : (c.N + h->seg_rows - 1) / h->seg_rows;
        h->seg_cap = std::min(h->C, h->seg_rows * c.topk);
        if (e == cudaSuccess)
            e = alloc(&h->seg_union_idx, static_cast<size_t>(BHkv) * h->nseg * std::max(h->seg_cap, 1) * 4);
        if (e == cudaSuccess) e = alloc(&h->seg_union_cnt, static_cast<size_t>(BHkv) * h->nseg * 4);
    }
    if (h->full) {
        if (e == cudaSuccess) e = alloc(&h->full_lse, rows * 4);
        if (e == cudaSuccess && c.selector == SAS_SEL_MEANPOOL_PROJ)
            e = alloc(&h->full_table, rows * static_cast<size_t>(h->C) * 4);
    }
    if (e == cudaSuccess) e = alloc(&h->status, 16);
    if (e == cudaSuccess) e = cudaMemset(h->status, 0, 16);
    if (e == cudaSuccess) e = alloc(&h->sched, 16);
    if (e == cudaSuccess) e = cudaMemset(h->sched, 0, 16);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        sas_status s = e == cudaErrorMemoryAllocation ? SAS_ERR_OOM : SAS_ERR_CUDA;
        sas_destroy(h);
        return s;
    }
    *out = h;
    return SAS_OK;
}

void sas_destroy(sas_handle* h) {
    if (h == nullptr) return;
    cudaDeviceSynchronize();
    cudaFree(h->Kt);
    cudaFree(h->union_idx);
    cudaFree(h->union_cnt);
    cudaFree(h->sel_idx);
    cudaFree(h->sel_logg);
    cudaFree(h->tiles);
    cudaFree(h->ntiles);
    cudaFree(h->tile_off);
    cudaFree(h->status);
    cudaFree(h->sched);
    cudaFree(h->full_lse);
    cudaFree(h->full_table);
    cudaFree(h->seg_union_idx);
    cudaFree(h->seg_union_cnt);
    cudaFree(h->hidden);
    cudaFree(h->bwd_delta);
    cudaFree(h->bwd_inv);
    cudaFree(h->bwd_tiles);
    cudaFree(h->bwd_dlogg);
    cudaFree(h->bwd_offs);
    cudaFree(h->dense_idx);
    cudaFree(h->dense_lg);
    cudaFree(h->dense_uidx);
    cudaFree(h->dense_ucnt);
    cudaFree(h->dense_lse);
    for (cudaEvent_t ev : h->events) cudaEventDestroy(ev);
    delete h;
}

}  // extern "C"

namespace {

sas_status attention_fwd(sas_handle* h, const void* Q, const void* K, const void* V, const float* scores,
                         const void* Wq, const void* Wk, const float* noise, void* O, float* LSE, int32_t* sel_idx,
                         float* sel_logg, void* stream) {
    if (h == nullptr) return SAS_ERR_INVALID_ARG;
    const sas_config& c = h->cfg;
    if (h->varlen) return fail(h, SAS_ERR_INVALID_ARG, "packed-sequence handle: use sas_attention_fwd_varlen");
    if (noise != nullptr && h->full) return fail(h, SAS_ERR_INVALID_ARG, "noise belongs to the sparse scope (full*)");
    if (noise != nullptr && !aligned4(noise)) return fail(h, SAS_ERR_INVALID_ARG, "noise must be 4-byte aligned");
    if (h->full && (sel_idx != nullptr || sel_logg != nullptr))
        return fail(h, SAS_ERR_INVALID_ARG, "the full scope keeps no Top-K: sel_idx and sel_logg must be NULL");
    if (!Q || !K || !V || !O) return fail(h, SAS_ERR_INVALID_ARG, "Q, K, V and O are required");
    if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O))
        return fail(h, SAS_ERR_INVALID_ARG, "Q, K, V and O must be 16-byte aligned");
    if (c.selector == SAS_SEL_SCORES_GIVEN) {
        if (!scores || !aligned4(scores)) return fail(h, SAS_ERR_INVALID_ARG, "scores required (4-byte aligned)");
        if (Wq || Wk) return fail(h, SAS_ERR_INVALID_ARG, "Wq/Wk must be NULL with given scores");
    } else {
        if (scores) return fail(h, SAS_ERR_INVALID_ARG, "scores must be NULL with the learned selector");
        if (!Wq || !Wk || !aligned16(Wq) || !aligned16(Wk))
            return fail(h, SAS_ERR_INVALID_ARG, "Wq and Wk required (16-byte aligned)");
    }
    if ((LSE && !aligned4(LSE)) || (sel_idx && !aligned4(sel_idx)) || (sel_logg && !aligned4(sel_logg)))
        return fail(h, SAS_ERR_INVALID_ARG, "LSE / sel_idx / sel_logg must be 4-byte aligned");

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const sas::KernelEnv env{s, h->status, h->limit};
    const char* err = "";
    int32_t* out_idx = sel_idx ? sel_idx : h->sel_idx;
    float* out_lg = sel_logg ? sel_logg : h->sel_logg;
    cudaError_t e = cudaSuccess;

    if (c.selector == SAS_SEL_MEANPOOL_PROJ) {
        // a1: block summaries -> projected summaries
        if (h->F > 0) {
            e = timed_launch(h, 0, s, [&] {
                return sas::launch_pool(K, Wk, h->Kt, h->BHkv, h->Hkv, c.N, c.d, h->d_sel, env, h->F);   // per KV group
            });
            if (e != cudaSuccess) return cuda_fail(h, e, "block summaries");
        }
    }
    // a2-a4: query projection (learned selector), scores, log-gates, Top-K, tile unions
    sas::SelectArgs sa{};
    sa.BH = h->BHkv; sa.H = h->Hkv; sa.N = c.N; sa.C = h->C; sa.T = h->T; sa.topk = c.topk; sa.d_sel = h->d_sel;
    sa.G = h->G;
    sa.gate_act = c.gate_act;
    sa.score_scale = c.selector == SAS_SEL_MEANPOOL_PROJ ? 1.0f / std::sqrt(static_cast<float>(h->d_sel)) : 1.0f;
    sa.scores = scores;
    sa.Q = Q; sa.Wq = Wq; sa.d = c.d; sa.Kt = h->Kt; sa.F = h->F;
    sa.sel_idx = out_idx; sa.sel_logg = out_lg;
    sa.union_idx = h->union_idx; sa.union_cnt = h->union_cnt;
    sa.noise = noise;
    if (h->full) {
        sa.full_lse = h->full_lse;
        sa.full_table = h->full_table;
    }
    e = timed_launch(h, 2, s, [&] { return sas::launch_select(sa, env, &err); });
    if (e != cudaSuccess) return cuda_fail(h, e, err);
    if (h->seg_rows > 0) {
        // the segment unions of the head-packed attention tiles (timed with the selection)
        e = timed_launch(h, 2, s, [&] {
            return sas::launch_seg_unions(out_idx, h->BHkv, c.N, h->C, c.topk, h->seg_rows, h->nseg, h->seg_union_idx,
                                          h->seg_union_cnt, env);
        });
        if (e != cudaSuccess) return cuda_fail(h, e, "segment unions");
    }
    // a5: gated sparse attention
    sas::AttnArgs aa{};
    aa.Q = Q; aa.K = K; aa.V = V; aa.O = O; aa.LSE = LSE;
    aa.union_idx = h->union_idx; aa.union_cnt = h->union_cnt;
    aa.sel_idx = out_idx; aa.sel_logg = out_lg;
    aa.BH = h->BH; aa.N = c.N; aa.d = c.d; aa.C = h->C; aa.T = h->T; aa.topk = c.topk; aa.mode = kernel_mode(c);
    aa.G = h->G;
    aa.gate_pos = c.gate_pos;
    aa.sm_scale = h->sm_scale;
    aa.sched = h->sched;
    if (h->full) {
        aa.full_table = c.selector == SAS_SEL_SCORES_GIVEN ? scores : h->full_table;
        aa.full_lse = h->full_lse;
    }
    if (h->seg_rows > 0) {
        aa.seg_rows = h->seg_rows;
        aa.nseg = h->nseg;
        aa.seg_union_idx = h->seg_union_idx;
        aa.seg_union_cnt = h->seg_union_cnt;
    }
    h->last_fwd = h->seg_rows > 0 ? 1 : 0;
    e = timed_launch(h, 3, s, [&] { return sas::launch_attn(aa, env, &err); });
    if (e != cudaSuccess) return cuda_fail(h, e, err);
    return SAS_OK;
}

}  // namespace

extern "C" {

sas_status sas_attention_fwd(sas_handle* h, const void* Q, const void* K, const void* V, const float* scores,
                             const void* Wq, const void* Wk, void* O, float* LSE, int32_t* sel_idx,
                             float* sel_logg, void* stream) {
    return attention_fwd(h, Q, K, V, scores, Wq, Wk, nullptr, O, LSE, sel_idx, sel_logg, stream);
}

sas_status sas_attention_fwd_noisy(sas_handle* h, const void* Q, const void* K, const void* V, const float* scores,
                                   const void* Wq, const void* Wk, const float* noise, void* O, float* LSE,
                                   int32_t* sel_idx, float* sel_logg, void* stream) {
    if (h != nullptr && noise == nullptr) return fail(h, SAS_ERR_INVALID_ARG, "noise is required");
    return attention_fwd(h, Q, K, V, scores, Wq, Wk, noise, O, LSE, sel_idx, sel_logg, stream);
}

sas_status sas_attention_fwd_varlen(sas_handle* h, const int32_t* cu_seqlens, int32_t num_seqs, const void* Q,
                                    const void* K, const void* V, const float* scores, const void* Wq, const void* Wk,
                                    void* O, float* LSE, int32_t* sel_idx, float* sel_logg, void* stream) {
    if (h == nullptr) return SAS_ERR_INVALID_ARG;
    const sas_config& c = h->cfg;
    if (!h->varlen) return fail(h, SAS_ERR_INVALID_ARG, "handle not created for packed sequences (max_seqs = 0)");
    if (num_seqs < 1 || num_seqs > c.max_seqs)
        return fail(h, SAS_ERR_INVALID_ARG, "num_seqs must be in 1 .. max_seqs");
    if (!cu_seqlens || !aligned4(cu_seqlens)) return fail(h, SAS_ERR_INVALID_ARG, "cu_seqlens required (4-byte aligned)");
    if (!Q || !K || !V || !O) return fail(h, SAS_ERR_INVALID_ARG, "Q, K, V and O are required");
    if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O))
        return fail(h, SAS_ERR_INVALID_ARG, "Q, K, V and O must be 16-byte aligned");
    const bool learned = c.selector == SAS_SEL_MEANPOOL_PROJ;
    if (!learned) {
        if (!scores || !aligned4(scores)) return fail(h, SAS_ERR_INVALID_ARG, "scores required (4-byte aligned)");
        if (Wq || Wk) return fail(h, SAS_ERR_INVALID_ARG, "Wq/Wk must be NULL with given scores");
    } else {
        if (scores) return fail(h, SAS_ERR_INVALID_ARG, "scores must be NULL with the learned selector");
        if (!Wq || !Wk || !aligned16(Wq) || !aligned16(Wk))
            return fail(h, SAS_ERR_INVALID_ARG, "Wq and Wk required (16-byte aligned)");
    }
    if ((LSE && !aligned4(LSE)) || (sel_idx && !aligned4(sel_idx)) || (sel_logg && !aligned4(sel_logg)))
        return fail(h, SAS_ERR_INVALID_ARG, "LSE / sel_idx / sel_logg must be 4-byte aligned");

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const sas::KernelEnv env{s, h->status, h->limit};
    const char* err = "";
    int32_t* out_idx = sel_idx ? sel_idx : h->sel_idx;
    float* out_lg = sel_logg ? sel_logg : h->sel_logg;
    const int max_len = c.max_seqlen > 0 ? c.max_seqlen : c.N;
    // the tile table of the packed sequences (device offsets, checked on the device)
    cudaError_t e =
        sas::launch_varlen_tiles(cu_seqlens, num_seqs, c.N, max_len, h->tiles, h->ntiles, h->tile_off, env);
    if (e != cudaSuccess) return cuda_fail(h, e, "packed-sequence tile table");
    h->launches += 1;
    if (learned) {
        // a1: each sequence's block summaries (blocks restart at its first token)
        e = timed_launch(h, 0, s, [&] {
            return sas::launch_pool(K, Wk, h->Kt, h->BHkv, h->Hkv, c.N, c.d, h->d_sel, env, h->F, h->tiles,
                                    h->ntiles, h->T);
        });
        if (e != cudaSuccess) return cuda_fail(h, e, "block summaries");
    }
    // a2-a4 over the tiles of every sequence
    sas::SelectArgs sa{};
    sa.BH = h->BHkv; sa.H = h->Hkv; sa.N = c.N; sa.C = h->C; sa.T = h->T; sa.topk = c.topk; sa.d_sel = h->d_sel;
    sa.G = h->G;
    sa.gate_act = c.gate_act;
    sa.score_scale = learned ? 1.0f / std::sqrt(static_cast<float>(h->d_sel)) : 1.0f;
    sa.scores = scores;
    sa.Q = Q; sa.Wq = Wq; sa.Kt = h->Kt; sa.F = h->F;
    sa.d = c.d;
    sa.sel_idx = out_idx; sa.sel_logg = out_lg;
    sa.union_idx = h->union_idx; sa.union_cnt = h->union_cnt;
    sa.tiles = h->tiles; sa.ntiles = h->ntiles;
    e = timed_launch(h, 2, s, [&] { return sas::launch_select(sa, env, &err); });
    if (e != cudaSuccess) return cuda_fail(h, e, err);
    if (h->seg_rows > 0) {
        // the segment unions of the head-packed attention tiles (timed with the selection)
        e = timed_launch(h, 2, s, [&] {
            return sas::launch_seg_unions(out_idx, h->BHkv, c.N, h->C, c.topk, h->seg_rows, h->nseg, h->seg_union_idx,
                                          h->seg_union_cnt, env, h->tiles, h->ntiles);
        });
        if (e != cudaSuccess) return cuda_fail(h, e, "segment unions");
    }
    // a5 over the same tiles
    sas::AttnArgs aa{};
    aa.Q = Q; aa.K = K; aa.V = V; aa.O = O; aa.LSE = LSE;
    aa.union_idx = h->union_idx; aa.union_cnt = h->union_cnt;
    aa.sel_idx = out_idx; aa.sel_logg = out_lg;
    aa.BH = h->BH; aa.N = c.N; aa.d = c.d; aa.C = h->C; aa.T = h->T; aa.topk = c.topk; aa.mode = kernel_mode(c);
    aa.G = h->G;
    aa.tiles = h->tiles; aa.ntiles = h->ntiles;
    aa.gate_pos = c.gate_pos;
    aa.sm_scale = h->sm_scale;
    aa.sched = h->sched;
    if (h->seg_rows > 0) {
        aa.seg_rows = h->seg_rows;
        aa.nseg = h->nseg;
        aa.seg_union_idx = h->seg_union_idx;
        aa.seg_union_cnt = h->seg_union_cnt;
    }
    h->last_fwd = h->seg_rows > 0 ? 1 : 0;
    e = timed_launch(h, 3, s, [&] { return sas::launch_attn(aa, env, &err); });
    if (e != cudaSuccess) return cuda_fail(h, e, err);
    return SAS_OK;
}

sas_status sas_mlp_fwd(sas_handle* h, const void* X, const void* W1, const void* b1, const void* W2, const void* b2,
                       void* Y, int64_t T, int64_t D, int64_t F, void* stream) {
    if (h == nullptr) return SAS_ERR_INVALID_ARG;
    if (!X || !W1 || !W2 || !Y) return fail(h, SAS_ERR_INVALID_ARG, "X, W1, W2 and Y are required");
    if (!aligned16(X) || !aligned16(W1) || !aligned16(W2) || !aligned16(Y) || (b1 && !aligned16(b1)) ||
        (b2 && !aligned16(b2)))
        return fail(h, SAS_ERR_INVALID_ARG, "MLP tensors must be 16-byte aligned");
    if (T < 1 || D < 64 || F < 64) return fail(h, SAS_ERR_INVALID_ARG, "T >= 1, D >= 64, F >= 64 required");
    if (D % 64 != 0 || F % 64 != 0) return fail(h, SAS_ERR_UNSUPPORTED, "D and F must be multiples of 64");
    if (T > (1LL << 31) - 1 || D > 65536 || F > 262144) return fail(h, SAS_ERR_UNSUPPORTED, "MLP size too large");

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const size_t need = static_cast<size_t>(T) * F * 2;
    if (need > h->hidden_bytes) {
        cudaError_t e = cudaStreamSynchronize(s);
        if (e == cudaSuccess) {
            cudaFree(h->hidden);
            h->hidden = nullptr;
            h->hidden_bytes = 0;
            e = cudaMalloc(&h->hidden, need);
        }
        if (e != cudaSuccess) return cuda_fail(h, e, "MLP hidden buffer");
        h->hidden_bytes = need;
    }
    const sas::KernelEnv env{s, h->status, h->limit};
    const char* err = "";
    auto pick_bn = [](int64_t n) { return n % 256 == 0 ? 256 : (n % 128 == 0 ? 128 : 64); };

    sas::GemmProblem g1{};
    g1.A = X; g1.B = W1; g1.C = h->hidden; g1.bias = b1;
    g1.M = static_cast<int>(T); g1.N = static_cast<int>(F); g1.K = static_cast<int>(D);
    g1.batches = 1; g1.b_mod = 1; g1.c_batch_stride = 0; g1.ldc = static_cast<int>(F);
    g1.gelu = 1; g1.bn = pick_bn(F); g1.max_ctas = 0;
    cudaError_t e = timed_launch(h, 4, s, [&] { return sas::launch_gemm(g1, env, &err); });
    if (e != cudaSuccess) return cuda_fail(h, e, err);

    sas::GemmProblem g2{};
    g2.A = h->hidden; g2.B = W2; g2.C = Y; g2.bias = b2;
    g2.M = static_cast<int>(T); g2.N = static_cast<int>(D); g2.K = static_cast<int>(F);
    g2.batches = 1; g2.b_mod = 1; g2.c_batch_stride = 0; g2.ldc = static_cast<int>(D);
    g2.gelu = 0; g2.bn = pick_bn(D); g2.max_ctas = 0;
    e = timed_launch(h, 5, s, [&] { return sas::launch_gemm(g2, env, &err); });
    if (e != cudaSuccess) return cuda_fail(h, e, err);
    return SAS_OK;
}

sas_status sas_attention_bwd(sas_handle* h, const void* Q, const void* K, const void* V, const float* scores,
                             const void* O, const float* LSE, const void* dO, const int32_t* sel_idx,
                             const float* sel_logg, void* dQ, void* dK, void* dV, float* dlogg, float* dscores,
                             void* stream) {
    if (h == nullptr) return SAS_ERR_INVALID_ARG;
    const sas_config& c = h->cfg;
    if (!Q || !K || !V || !O || !LSE || !dO || !dQ || !dK || !dV)
        return fail(h, SAS_ERR_INVALID_ARG, "Q, K, V, O, LSE, dO, dQ, dK and dV are required");
    if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O) || !aligned16(dO) || !aligned16(dQ) ||
        !aligned16(dK) || !aligned16(dV) || !aligned4(LSE) || (sel_idx && !aligned4(sel_idx)) ||
        (sel_logg && !aligned4(sel_logg)) || (dlogg && !aligned4(dlogg)) || (dscores && !aligned4(dscores)) ||
        (scores && !aligned4(scores)))
        return fail(h, SAS_ERR_INVALID_ARG, "misaligned pointer");
    if (c.d != 128) return fail(h, SAS_ERR_UNSUPPORTED, "the backward supports d = 128");
    // the full scope and the hard gate's estimator gate every historical block
    const bool ste = c.mode == SAS_MODE_TRAIN_HARD_STE;
    const bool dense = h->full || ste;
    if (dense) {
        if (h->varlen) return fail(h, SAS_ERR_UNSUPPORTED, "the full-scope and hard-STE backwards take [B, H, N, d] inputs");
        if (ste && c.selector != SAS_SEL_SCORES_GIVEN)
            return fail(h, SAS_ERR_UNSUPPORTED, "the hard-STE backward needs given scores (SCORES_GIVEN)");
        if (c.selector == SAS_SEL_SCORES_GIVEN && !scores)
            return fail(h, SAS_ERR_INVALID_ARG, "the full-scope and hard-STE backwards need the given scores");
    }
    // query tiles of one sequence (a key pair's inverted list holds at most that many)
    const int tseq = h->varlen ? (h->C + 1) / 2 : h->T;
    if (tseq > sas::kBwdMaxTiles)
        return fail(h, SAS_ERR_UNSUPPORTED, "the backward supports sequences of at most 262016 tokens");
    if (dscores) {
        if (c.selector != SAS_SEL_SCORES_GIVEN || !scores)
            return fail(h, SAS_ERR_INVALID_ARG, "dscores needs given scores (SCORES_GIVEN)");
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const size_t rows = static_cast<size_t>(h->BH) * c.N;
    const size_t tiles = static_cast<size_t>(h->BH) * h->T;
    // gate-gradient entries per row: the kept blocks, or every block (dense)
    const size_t dl_w = std::max<size_t>(1, std::max(c.topk, dense ? h->C : 0));
    if (h->bwd_delta == nullptr) {
        // first backward on this handle: workspace (synchronous)
        cudaError_t e = cudaStreamSynchronize(s);
        const size_t pairs = static_cast<size_t>(h->T < h->C ? h->T : h->C);
        if (e == cudaSuccess) e = alloc(&h->bwd_delta, rows * 4);
        if (e == cudaSuccess) e = alloc(&h->bwd_inv, (4 * tiles + 2) * 4);
        if (e == cudaSuccess) e = alloc(&h->bwd_tiles, 2 * tiles * pairs * 4);
        const size_t dl_rows = rows + (h->G > 1 ? static_cast<size_t>(h->BHkv) * c.N : 0);
        if (e == cudaSuccess) e = alloc(&h->bwd_dlogg, dl_rows * dl_w * 4);
        // offsets of pass 1 for pass 2: local tile t visits at most 2t + 2 blocks, so a
        // head needs at most T (T + 1) slots of 128 rows (packed sequences: 2 tseq per
        // tile slot); held whole when that fits in 8 GiB
        const size_t per_tile = h->varlen ? 2 * static_cast<size_t>(tseq) : static_cast<size_t>(h->T + 1);
        const size_t bound = tiles * per_tile * 128 * 4;
        if (e == cudaSuccess && bound <= (static_cast<size_t>(8) << 30)) {
            cudaError_t eb = alloc(&h->bwd_offs, bound);
            if (eb == cudaSuccess) {
                h->bwd_offs_bytes = bound;
                h->bwd_offs_bound = true;
            } else if (eb == cudaErrorMemoryAllocation) {
                // no room for the bound: clear the error and size the buffer from the
                // slot count each call reads back (the path used above 8 GiB)
                cudaGetLastError();
                h->bwd_offs = nullptr;
            } else {
                e = eb;
            }
        }
        if (e != cudaSuccess) {
            cudaFree(h->bwd_delta); cudaFree(h->bwd_inv); cudaFree(h->bwd_tiles); cudaFree(h->bwd_dlogg);
            h->bwd_delta = nullptr; h->bwd_inv = nullptr; h->bwd_tiles = nullptr; h->bwd_dlogg = nullptr;
            return cuda_fail(h, e, "backward workspace");
        }
    }
    if (dense && h->dense_idx == nullptr) {
        // lists of every historical block (first dense backward on this handle; synchronous)
        cudaError_t e = cudaStreamSynchronize(s);
        const size_t cells = static_cast<size_t>(h->BHkv) * c.N * h->C;
        const size_t utiles = static_cast<size_t>(h->BHkv) * h->T;
        if (e == cudaSuccess) e = alloc(&h->dense_idx, cells * 4);
        if (e == cudaSuccess) e = alloc(&h->dense_lg, cells * 4);
        if (e == cudaSuccess) e = alloc(&h->dense_uidx, utiles * h->C * 4);
        if (e == cudaSuccess) e = alloc(&h->dense_ucnt, utiles * 4);
        if (e == cudaSuccess) e = alloc(&h->dense_lse, static_cast<size_t>(h->BHkv) * c.N * 4);
        if (e != cudaSuccess) {
            cudaFree(h->dense_idx); cudaFree(h->dense_lg); cudaFree(h->dense_uidx); cudaFree(h->dense_ucnt);
            cudaFree(h->dense_lse);
            h->dense_idx = nullptr; h->dense_lg = nullptr; h->dense_uidx = nullptr; h->dense_ucnt = nullptr;
            h->dense_lse = nullptr;
            return cuda_fail(h, e, "backward block lists");
        }
    }
    sas::AttnBwdArgs a{};
    a.Q = Q; a.K = K; a.V = V; a.O = O; a.dO = dO; a.LSE = LSE;
    a.union_idx = h->union_idx; a.union_cnt = h->union_cnt;
    a.sel_idx = sel_idx ? sel_idx : h->sel_idx;
    a.sel_logg = sel_logg ? sel_logg : h->sel_logg;
    a.scores = dscores ? scores : nullptr;
    a.dQ = dQ; a.dK = dK; a.dV = dV;
    // GQA: pass 1 writes each query head's d(log g); the group's is their sum
    a.dlogg_heads = h->G > 1 ? h->bwd_dlogg : nullptr;
    float* dlogg_scratch = h->bwd_dlogg + (h->G > 1 ? rows * dl_w : 0);   // the group sums when dlogg is NULL
    a.dlogg = dlogg ? dlogg : dlogg_scratch;
    a.ds = dscores;
    a.delta = h->bwd_delta;
    a.inv_cnt = h->bwd_inv;
    a.inv_cursor = h->bwd_inv + tiles;
    a.inv_off = h->bwd_inv + 2 * tiles;
    a.slot_off = h->bwd_inv + 3 * tiles + 1;
    a.inv_tiles = h->bwd_tiles;
    a.inv_pos = h->bwd_tiles + tiles * static_cast<size_t>(h->T < h->C ? h->T : h->C);
    a.N = c.N; a.C = h->C; a.T = h->T; a.BH = h->BH; a.topk = c.topk; a.mode = c.mode; a.d = c.d;
    a.G = h->G;
    a.act = c.gate_act;
    a.pos = c.gate_pos;
    a.sm_scale = h->sm_scale;
    if (h->varlen) {
        // the tile table of the last sas_attention_fwd_varlen (its union lists are per slot)
        a.tiles = h->tiles;
        a.ntiles = h->ntiles;
        a.tile_off = h->tile_off;
    }
    // segments of one sequence, each a possible entry of a key pair's inverted list
    const long long seq_segs = h->varlen ? static_cast<long long>(h->G) * tseq : h->nseg;
    if (h->seg_rows > 0 && h->last_fwd == 1 && seq_segs + h->G <= sas::kBwdMaxTiles) {
        // head-packed tiles over the forward's segment unions
        a.seg_rows = h->seg_rows;
        a.nseg = h->nseg;
        a.seg_cap = h->seg_cap;
        a.seg_union_idx = h->seg_union_idx;
        a.seg_union_cnt = h->seg_union_cnt;
    }
    const sas::KernelEnv env{s, h->status, h->limit};
    const char* err = "";
    sas::AttnBwdArgs ag{};   // hard-STE: the gate pass over every historical block
    if (dense) {
        // log g = s - LSE of every historical block: the full scope's own
        // normalisers, or (hard-STE) the soft ones of the given scores
        const float* sv = c.selector == SAS_SEL_SCORES_GIVEN ? scores : h->full_table;
        const float* lse = h->full_lse;
        cudaError_t e = cudaSuccess;
        if (ste) {
            e = sas::launch_row_lse(scores, c.N, h->C, static_cast<long long>(h->BHkv) * c.N, h->dense_lse, env);
            lse = h->dense_lse;
        }
        if (e == cudaSuccess)
            e = sas::launch_bwd_dense_lists(sv, lse, h->BHkv, c.N, h->C, h->T, h->dense_idx, h->dense_lg,
                                            h->dense_uidx, h->dense_ucnt, env);
        if (e != cudaSuccess) return cuda_fail(h, e, "backward block lists");
        h->launches += 2 + (ste ? 1 : 0);
        if (ste) {
            // the gate pass: pass 1 alone over every block, the soft log-gates as
            // biases under the hard forward's LSE; its row sums are x = g dg
            ag = a;
            ag.mode = SAS_MODE_TRAIN_SOFT;
            ag.sel_idx = h->dense_idx; ag.sel_logg = h->dense_lg;
            ag.union_idx = h->dense_uidx; ag.union_cnt = h->dense_ucnt;
            ag.topk = h->C;
            ag.seg_rows = 0; ag.nseg = 0; ag.seg_cap = 0; ag.seg_union_idx = nullptr; ag.seg_union_cnt = nullptr;
            ag.gate_only = true;
            ag.dQ = nullptr;
            ag.offs = nullptr;
            // the hard pass: no gate gradient (its zeros go to the scratch), no score gradient
            a.mode = SAS_MODE_INFER_HARD;
            a.dlogg = dlogg_scratch;
            a.ds = nullptr;
            a.scores = nullptr;
        } else {
            a.sel_idx = h->dense_idx; a.sel_logg = h->dense_lg;
            a.union_idx = h->dense_uidx; a.union_cnt = h->dense_ucnt;
            a.topk = h->C;
        }
    }
    // slots of the per-row offsets pass 1 hands to pass 2: their number depends on
    // the forward's tile lists; a buffer of the upper bound needs no read-back,
    // otherwise it is read back (synchronously) to size the buffer
    long long slots = 0;
    cudaError_t e = sas::launch_bwd_slots(a, env, h->bwd_offs_bound ? nullptr : &slots);
    if (e != cudaSuccess) return cuda_fail(h, e, "backward slots");
    const size_t need = static_cast<size_t>(slots) * 128 * 4;
    if (!h->bwd_offs_bound && need > h->bwd_offs_bytes) {
        cudaFree(h->bwd_offs);
        h->bwd_offs = nullptr;
        h->bwd_offs_bytes = 0;
        e = alloc(&h->bwd_offs, need);
        if (e != cudaSuccess) return cuda_fail(h, e, "backward offsets");
        h->bwd_offs_bytes = need;
    }
    a.offs = h->bwd_offs;
    e = timed_launch(h, 6, s, [&] { return sas::launch_attn_bwd(a, env, &err); });
    if (e != cudaSuccess) return cuda_fail(h, e, err);
    // all its kernels: slot count and scan, pass 1, the inverted lists (count, scan,
    // fill), pass 2, the group sum of d(log g) and the score gradient
    h->launches += 7 + ((h->G > 1 && a.topk > 0) ? 1 : 0) +
                   ((a.ds != nullptr && a.scores != nullptr && a.topk > 0) ? 1 : 0);
    if (ste) {
        e = timed_launch(h, 6, s, [&] { return sas::launch_attn_bwd(ag, env, &err); });
        if (e != cudaSuccess) return cuda_fail(h, e, err);
        h->launches += 1 + ((h->G > 1 && ag.topk > 0) ? 1 : 0) +
                       ((ag.ds != nullptr && ag.scores != nullptr && ag.topk > 0) ? 1 : 0);
    }
    return SAS_OK;
}

sas_status sas_get_device_status(sas_handle* h, int32_t* out_status) {
    if (h == nullptr || out_status == nullptr) return SAS_ERR_INVALID_ARG;
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(h, e, "synchronize");
    int v = 0;
    e = cudaMemcpy(&v, h->status, sizeof(int), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess) e = cudaMemset(h->status, 0, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(h, e, "status word");
    *out_status = v;
    return SAS_OK;
}

sas_status sas_set_timing(sas_handle* h, int32_t enable) {
    if (h == nullptr) return SAS_ERR_INVALID_ARG;
    cudaDeviceSynchronize();
    h->timing = enable != 0;
    h->recs.clear();
    h->events_used = 0;
    return SAS_OK;
}

sas_status sas_get_timings(sas_handle* h, int64_t* launches, double* total_ms, int32_t n_kinds) {
    if (h == nullptr || launches == nullptr || total_ms == nullptr || n_kinds < 0 || n_kinds > SAS_NUM_KERNEL_KINDS)
        return SAS_ERR_INVALID_ARG;
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(h, e, "synchronize");
    for (int k = 0; k < n_kinds; ++k) { launches[k] = 0; total_ms[k] = 0.0; }
    for (const TimeRec& r : h->recs) {
        if (r.kind >= n_kinds) continue;
        float ms = 0.f;
        if (cudaEventElapsedTime(&ms, r.a, r.b) == cudaSuccess) {
            launches[r.kind] += 1;
            total_ms[r.kind] += ms;
        }
    }
    return SAS_OK;
}

int64_t sas_launch_count(const sas_handle* h) { return h ? h->launches : 0; }

sas_status sas_set_wait_limit(sas_handle* h, int64_t cycles) {
    if (h == nullptr || cycles < 0) return SAS_ERR_INVALID_ARG;
    h->limit = cycles == 0 ? kDefaultWaitLimit : cycles;
    return SAS_OK;
}

sas_status sas_get_tile_union_counts(sas_handle* h, int32_t* host_out, int64_t n) {
    if (h == nullptr || host_out == nullptr) return SAS_ERR_INVALID_ARG;
    const int64_t total = static_cast<int64_t>(h->BHkv) * h->T;   // one union list per KV group and tile
    if (n < total) return fail(h, SAS_ERR_INVALID_ARG, "output too small");
    cudaError_t e = cudaDeviceSynchronize();
    if (e == cudaSuccess) e = cudaMemcpy(host_out, h->union_cnt, total * 4, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(h, e, "union counts");
    return SAS_OK;
}

sas_status sas_get_attention_work(sas_handle* h, int64_t* tiles, int64_t* tile_blocks) {
    if (h == nullptr || tiles == nullptr || tile_blocks == nullptr) return SAS_ERR_INVALID_ARG;
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(h, e, "synchronize");
    const int N = h->cfg.N;
    int64_t nt = 0, nb = 0;
    auto ndiag = [](int t, int n) { return (2 * t + 1) * 64 < n ? 2 : 1; };
    if (h->last_fwd == 1) {
        // head-packed: one tile per (KV group, segment in use), its union and one diagonal block
        std::vector<int32_t> cnt(static_cast<size_t>(h->BHkv) * h->nseg);
        e = cudaMemcpy(cnt.data(), h->seg_union_cnt, cnt.size() * 4, cudaMemcpyDeviceToHost);
        int used = h->nseg;
        if (e == cudaSuccess && h->varlen) {
            e = cudaMemcpy(&used, h->ntiles, 4, cudaMemcpyDeviceToHost);
            used *= h->G;
        }
        if (e != cudaSuccess) return cuda_fail(h, e, "segment union counts");
        for (int kv = 0; kv < h->BHkv; ++kv)
            for (int sg = 0; sg < used; ++sg) nb += cnt[static_cast<size_t>(kv) * h->nseg + sg] + 1;
        nt = static_cast<int64_t>(h->BHkv) * used;
    } else {
        // one tile per (query head, tile slot): its group's union and one or two diagonal blocks
        std::vector<int32_t> cnt(static_cast<size_t>(h->BHkv) * h->T);
        e = cudaMemcpy(cnt.data(), h->union_cnt, cnt.size() * 4, cudaMemcpyDeviceToHost);
        if (e != cudaSuccess) return cuda_fail(h, e, "union counts");
        std::vector<int4> tl;
        int used = h->T;
        if (h->varlen) {
            e = cudaMemcpy(&used, h->ntiles, 4, cudaMemcpyDeviceToHost);
            tl.resize(static_cast<size_t>(std::max(used, 0)));
            if (e == cudaSuccess && used > 0)
                e = cudaMemcpy(tl.data(), h->tiles, tl.size() * sizeof(int4), cudaMemcpyDeviceToHost);
            if (e != cudaSuccess) return cuda_fail(h, e, "tile table");
        }
        for (int kv = 0; kv < h->BHkv; ++kv)
            for (int g = 0; g < used; ++g) {
                const int t = h->varlen ? tl[g].y : g;
                const int n = h->varlen ? tl[g].z : N;
                const int u = h->full ? 2 * t : cnt[static_cast<size_t>(kv) * h->T + g];
                nb += static_cast<int64_t>(h->G) * (u + ndiag(t, n));
                nt += h->G;
            }
    }
    *tiles = nt;
    *tile_blocks = nb;
    return SAS_OK;
}

sas_status sas_selftest_wait_timeout(int64_t limit_cycles, int32_t* host_status) {
    if (host_status == nullptr || limit_cycles < 0) return SAS_ERR_INVALID_ARG;
    if (check_device(nullptr) != SAS_OK) return SAS_ERR_UNSUPPORTED;
    int* d = nullptr;
    cudaError_t e = cudaMalloc(&d, 16);
    if (e == cudaSuccess) e = cudaMemset(d, 0, 16);
    if (e == cudaSuccess) e = sas::launch_wait_selftest(d, limit_cycles, nullptr);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    int v = 0;
    if (e == cudaSuccess) e = cudaMemcpy(&v, d, sizeof(int), cudaMemcpyDeviceToHost);
    cudaFree(d);
    if (e != cudaSuccess) return SAS_ERR_CUDA;
    *host_status = v;
    return SAS_OK;
}

}  // extern "C"
