// C ABI of the SAS decode step: argument checking, workspace ownership, launch
// sequencing on the caller's stream, event timing and the device status word.
// The arithmetic is in k_decode.cu.
#include <cmath>
#include <string>
#include <vector>

#include "../../include/sas.h"
#include "internal.h"

namespace {

constexpr long long kDecodeWaitLimit = 4000000000LL;   // ~2 s of SM clock per wait

struct DecTimeRec {
    int kind;
    cudaEvent_t a, b;
};

}  // namespace

struct sas_decode_handle {
    sas_decode_config cfg;
    int G = 1, d_sel = 0;
    float sm_scale = 0.f;
    int nsplit_s = 0, nsplit_a = 0, bpc = 0, nst = 0;
    // workspace
    void* qt = nullptr;
    uint32_t* cand_key = nullptr;
    int32_t* cand_idx = nullptr;
    int32_t* list = nullptr;
    int32_t* list_n = nullptr;
    float* part = nullptr;
    int* counters = nullptr;   // [2][B*Hkv]
    int* status = nullptr;
    // timing
    bool timing = false;
    std::vector<DecTimeRec> recs;
    std::vector<cudaEvent_t> events;
    size_t events_used = 0;
    int64_t launches = 0;
    long long limit = kDecodeWaitLimit;
    std::string last_error;
};

namespace {

sas_status dfail(sas_decode_handle* h, sas_status s, const std::string& msg) {
    if (h) h->last_error = msg;
    return s;
}

sas_status dcuda_fail(sas_decode_handle* h, cudaError_t e, const char* what) {
    std::string m = std::string(what) + ": " + cudaGetErrorString(e);
    return dfail(h, e == cudaErrorMemoryAllocation ? SAS_ERR_OOM : SAS_ERR_CUDA, m);
}

bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool al4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }

template <class T>
cudaError_t dalloc(T** p, size_t bytes) {
    void* v = nullptr;
    cudaError_t e = cudaMalloc(&v, bytes < 16 ? 16 : bytes);
    *p = static_cast<T*>(v);
    return e;
}

cudaEvent_t dnext_event(sas_decode_handle* h) {
    if (h->events_used == h->events.size()) {
        cudaEvent_t e;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        h->events.push_back(e);
    }
    return h->events[h->events_used++];
}

// Brackets one launch with events when timing is on.  The events are recorded
// as external event nodes when the stream is being captured, so a replayed
// graph re-records them and sas_decode_get_timings reads the latest replay.
template <class Fn>
cudaError_t dtimed(sas_decode_handle* h, int kind, cudaStream_t s, Fn&& fn) {
    cudaEvent_t a = nullptr, b = nullptr;
    unsigned flags = cudaEventRecordDefault;
    if (h->timing) {
        a = dnext_event(h);
        b = dnext_event(h);
        cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
        if (cudaStreamIsCapturing(s, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusActive)
            flags = cudaEventRecordExternal;
        if (a && cudaEventRecordWithFlags(a, s, flags) != cudaSuccess) a = nullptr;
    }
    cudaError_t e = fn();
    if (e == cudaSuccess) ++h->launches;
    if (h->timing && a && b && cudaEventRecordWithFlags(b, s, flags) == cudaSuccess) h->recs.push_back({kind, a, b});
    return e;
}

sas::DecodeArgs base_args(const sas_decode_handle* h) {
    const sas_decode_config& c = h->cfg;
    sas::DecodeArgs a{};
    a.B = c.B; a.Hq = c.Hq; a.Hkv = c.Hkv; a.G = h->G; a.d = c.d; a.d_sel = h->d_sel; a.topk = c.topk;
    a.max_blocks = c.max_blocks; a.num_pages = c.num_pages; a.dense = c.dense; a.sm_scale = h->sm_scale;
    a.qt = h->qt; a.cand_key = h->cand_key; a.cand_idx = h->cand_idx; a.list = h->list; a.list_n = h->list_n; a.part = h->part;
    a.cnt_sel = h->counters;
    a.cnt_attn = h->counters + static_cast<size_t>(c.B) * c.Hkv;
    a.nsplit_s = h->nsplit_s; a.nsplit_a = h->nsplit_a; a.bpc = h->bpc; a.nst = h->nst;
    return a;
}

}  // namespace

extern "C" {

sas_status sas_decode_create(const sas_decode_config* cfg, sas_decode_handle** out) {
    if (out == nullptr || cfg == nullptr) return SAS_ERR_INVALID_ARG;
    *out = nullptr;
    const sas_decode_config& c = *cfg;
    if (c.B < 1 || c.Hq < 1 || c.Hkv < 1 || c.max_blocks < 1 || c.num_pages < 1) return SAS_ERR_INVALID_ARG;
    if (c.Hq % c.Hkv != 0) return SAS_ERR_INVALID_ARG;
    const int G = c.Hq / c.Hkv;
    if (G != 1 && G != 2 && G != 4 && G != 8) return SAS_ERR_UNSUPPORTED;
    if (c.block != 64) return SAS_ERR_UNSUPPORTED;
    if (c.d != 64 && c.d != 128) return SAS_ERR_UNSUPPORTED;
    const int d_sel = c.d_sel == 0 ? c.d : c.d_sel;
    if (d_sel != 64 && d_sel != 128) return SAS_ERR_UNSUPPORTED;
    if (c.topk < 0) return SAS_ERR_INVALID_ARG;
    if (c.topk > 64) return SAS_ERR_UNSUPPORTED;
    if (c.max_blocks > 32768) return SAS_ERR_UNSUPPORTED;
    if (c.dense != 0 && c.dense != 1) return SAS_ERR_INVALID_ARG;
    if (!(c.sm_scale >= 0.f) || !std::isfinite(c.sm_scale)) return SAS_ERR_INVALID_ARG;
    const long long BH = static_cast<long long>(c.B) * c.Hkv;
    if (BH > 65535) return SAS_ERR_UNSUPPORTED;   // (sequence, KV head) pairs index grid.y

    sas_decode_handle* h = new sas_decode_handle();
    h->cfg = c;
    h->G = G;
    h->d_sel = d_sel;
    h->sm_scale = c.sm_scale > 0.f ? c.sm_scale : 1.0f / std::sqrt(static_cast<float>(c.d));
    h->nsplit_s = (c.max_blocks + sas::kDecScoreChunk - 1) / sas::kDecScoreChunk;
    sas::decode_attn_split(c.dense ? c.max_blocks : c.topk + 1, c.d, &h->nsplit_a, &h->bpc, &h->nst);

    int dev = 0, major = 0, minor = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (e != cudaSuccess) {
        delete h;
        return SAS_ERR_CUDA;
    }
    if (major != 10 || minor != 3) {
        delete h;
        return SAS_ERR_UNSUPPORTED;
    }
    if (e == cudaSuccess) e = dalloc(&h->qt, static_cast<size_t>(BH) * d_sel * 2);
    const size_t ncand = static_cast<size_t>(BH) * h->nsplit_s * (c.topk > 0 ? c.topk : 1);
    if (e == cudaSuccess) e = dalloc(&h->cand_key, ncand * 4);
    if (e == cudaSuccess) e = dalloc(&h->cand_idx, ncand * 4);
    if (e == cudaSuccess) e = dalloc(&h->list, static_cast<size_t>(BH) * 64 * 4);
    if (e == cudaSuccess) e = dalloc(&h->list_n, static_cast<size_t>(BH) * 4);
    if (e == cudaSuccess) e = dalloc(&h->part, static_cast<size_t>(BH) * h->nsplit_a * G * (c.d + 2) * 4);
    if (e == cudaSuccess) e = dalloc(&h->counters, static_cast<size_t>(BH) * 2 * 4);
    if (e == cudaSuccess) e = cudaMemset(h->counters, 0, static_cast<size_t>(BH) * 2 * 4);
    if (e == cudaSuccess) e = dalloc(&h->status, 16);
    if (e == cudaSuccess) e = cudaMemset(h->status, 0, 16);
    if (e == cudaSuccess) e = sas::decode_prepare(base_args(h));
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        const sas_status s = e == cudaErrorMemoryAllocation ? SAS_ERR_OOM : SAS_ERR_CUDA;
        sas_decode_destroy(h);
        return s;
    }
    *out = h;
    return SAS_OK;
}

void sas_decode_destroy(sas_decode_handle* h) {
    if (h == nullptr) return;
    cudaDeviceSynchronize();
    cudaFree(h->qt);
    cudaFree(h->cand_key);
    cudaFree(h->cand_idx);
    cudaFree(h->list);
    cudaFree(h->list_n);
    cudaFree(h->part);
    cudaFree(h->counters);
    cudaFree(h->status);
    for (cudaEvent_t ev : h->events) cudaEventDestroy(ev);
    delete h;
}

sas_status sas_decode_summarize(sas_decode_handle* h, const void* K_cache, const int32_t* block_table,
                                const int32_t* seq_lens, const void* Wk, void* Ksum, void* stream) {
    if (h == nullptr) return SAS_ERR_INVALID_ARG;
    if (h->cfg.dense) return dfail(h, SAS_ERR_INVALID_ARG, "a dense decode handle keeps no summaries");
    if (!K_cache || !block_table || !seq_lens || !Wk || !Ksum)
        return dfail(h, SAS_ERR_INVALID_ARG, "K_cache, block_table, seq_lens, Wk and Ksum are required");
    if (!al16(K_cache) || !al16(Wk) || !al16(Ksum) || !al4(block_table) || !al4(seq_lens))
        return dfail(h, SAS_ERR_INVALID_ARG, "misaligned pointer");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const sas::KernelEnv env{s, h->status, h->limit};
    sas::DecodeArgs a = base_args(h);
    a.K_cache = const_cast<void*>(K_cache);
    a.block_table = block_table;
    a.seq_lens = seq_lens;
    a.Wk = Wk;
    a.Ksum = Ksum;
    cudaError_t e = dtimed(h, 3, s, [&] { return sas::launch_decode_summarize(a, env); });
    if (e != cudaSuccess) return dcuda_fail(h, e, "summary fill");
    return SAS_OK;
}

sas_status sas_decode_step(sas_decode_handle* h, const void* q, const void* k_new, const void* v_new,
                           void* K_cache, void* V_cache, const int32_t* block_table, const int32_t* seq_lens,
                           const void* Wq, const void* Wk, void* Ksum, void* O, float* LSE, int32_t* sel_idx,
                           void* stream) {
    if (h == nullptr) return SAS_ERR_INVALID_ARG;
    const sas_decode_config& c = h->cfg;
    if (!q || !K_cache || !V_cache || !block_table || !seq_lens || !O)
        return dfail(h, SAS_ERR_INVALID_ARG, "q, K_cache, V_cache, block_table, seq_lens and O are required");
    if ((k_new == nullptr) != (v_new == nullptr))
        return dfail(h, SAS_ERR_INVALID_ARG, "k_new and v_new are given together or not at all");
    if (!al16(q) || !al16(K_cache) || !al16(V_cache) || !al16(O) || (k_new && (!al16(k_new) || !al16(v_new))) ||
        !al4(block_table) || !al4(seq_lens) || (LSE && !al4(LSE)) || (sel_idx && !al4(sel_idx)))
        return dfail(h, SAS_ERR_INVALID_ARG, "misaligned pointer");
    if (c.dense) {
        if (sel_idx) return dfail(h, SAS_ERR_INVALID_ARG, "sel_idx must be NULL in dense mode");
    } else {
        if (!Wq || !Wk || !Ksum || !al16(Wq) || !al16(Wk) || !al16(Ksum))
            return dfail(h, SAS_ERR_INVALID_ARG, "Wq, Wk and Ksum required (16-byte aligned)");
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const sas::KernelEnv env{s, h->status, h->limit};
    sas::DecodeArgs a = base_args(h);
    a.q = q; a.k_new = k_new; a.v_new = v_new; a.K_cache = K_cache; a.V_cache = V_cache;
    a.block_table = block_table; a.seq_lens = seq_lens; a.Wq = Wq; a.Wk = Wk; a.Ksum = Ksum;
    a.O = O; a.LSE = LSE; a.sel_idx = sel_idx;
    cudaError_t e = dtimed(h, 0, s, [&] { return sas::launch_decode_prep(a, env); });
    if (e != cudaSuccess) return dcuda_fail(h, e, "decode prep");
    if (!c.dense) {
        e = dtimed(h, 1, s, [&] { return sas::launch_decode_score(a, env); });
        if (e != cudaSuccess) return dcuda_fail(h, e, "decode scores + Top-K");
    }
    e = dtimed(h, 2, s, [&] { return sas::launch_decode_attn(a, env); });
    if (e != cudaSuccess) return dcuda_fail(h, e, "decode attention");
    return SAS_OK;
}

const char* sas_decode_last_error(const sas_decode_handle* h) { return h ? h->last_error.c_str() : ""; }

sas_status sas_decode_get_device_status(sas_decode_handle* h, int32_t* out_status) {
    if (h == nullptr || out_status == nullptr) return SAS_ERR_INVALID_ARG;
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return dcuda_fail(h, e, "synchronize");
    int v = 0;
    e = cudaMemcpy(&v, h->status, sizeof(int), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess) e = cudaMemset(h->status, 0, sizeof(int));
    if (e != cudaSuccess) return dcuda_fail(h, e, "status word");
    *out_status = v;
    return SAS_OK;
}

sas_status sas_decode_set_timing(sas_decode_handle* h, int32_t enable) {
    if (h == nullptr) return SAS_ERR_INVALID_ARG;
    cudaDeviceSynchronize();
    h->timing = enable != 0;
    if (h->timing) {   // a new recording starts; stopping keeps the records
        h->recs.clear();
        h->events_used = 0;
    }
    return SAS_OK;
}

sas_status sas_decode_get_timings(sas_decode_handle* h, int64_t* launches, double* total_ms, int32_t n_kinds) {
    if (h == nullptr || launches == nullptr || total_ms == nullptr || n_kinds < 0 ||
        n_kinds > SAS_DECODE_NUM_KERNEL_KINDS)
        return SAS_ERR_INVALID_ARG;
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return dcuda_fail(h, e, "synchronize");
    for (int k = 0; k < n_kinds; ++k) {
        launches[k] = 0;
        total_ms[k] = 0.0;
    }
    for (const DecTimeRec& r : h->recs) {
        if (r.kind >= n_kinds) continue;
        float ms = 0.f;
        if (cudaEventElapsedTime(&ms, r.a, r.b) == cudaSuccess) {
            launches[r.kind] += 1;
            total_ms[r.kind] += ms;
        }
    }
    return SAS_OK;
}

int64_t sas_decode_launch_count(const sas_decode_handle* h) { return h ? h->launches : 0; }

}  // extern "C"
