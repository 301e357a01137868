// Handle-free MLP entry point that allocates no device memory.
//
// sas_mlp_fwd keeps the hidden activation GELU(X W1^T + b1) in memory its
// handle allocates with cudaMalloc.  Some callers cannot do that: code that
// runs while a CUDA graph is being captured on its stream (an allocation
// there fails or breaks the capture), plug-ins whose host framework owns all
// device memory and forbids allocations on its hot path, and callers that
// must keep a fixed, known device-memory footprint.  For them the hidden
// activation lives here instead, in a fixed-size array that is part of this
// library's device image: every GPU that loads the library reserves it until
// the process exits, whether or not this entry point is ever called.
#include <mutex>

#include "../../include/sas.h"
#include "internal.h"

namespace {

constexpr size_t kScratchBytes = size_t(32) << 20;   // SAS_MLP_NOALLOC_MAX_HIDDEN_BYTES
static_assert(kScratchBytes == SAS_MLP_NOALLOC_MAX_HIDDEN_BYTES, "header and array must agree");

// Hidden activation of the handle-free MLP, bf16 [T][F] with T*F*2 <= 32 MiB.
static __device__ __align__(256) unsigned char g_mlp_hidden[kScratchBytes];
// Status word of the GEMM kernels (written only when a bounded wait runs out,
// or when a CTA finds its shared memory misaligned); read and cleared by
// sas_mlp_noalloc_get_device_status.
static __device__ __align__(256) int g_mlp_wait_status[64];

constexpr int kMaxDevices = 128;
void* g_hidden_addr[kMaxDevices] = {};
int* g_status_addr[kMaxDevices] = {};
std::mutex g_setup_mutex;

// Looks up, once per device and with that device current, the device
// addresses of the two arrays above.  In host code their names only stand
// in for them; a kernel must be given the address cudaGetSymbolAddress returns.
cudaError_t device_arrays(int dev, void** hidden, int** status) {
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (g_hidden_addr[dev] == nullptr || g_status_addr[dev] == nullptr) {
        void* h = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&h, g_mlp_hidden);
        if (e != cudaSuccess) return e;
        void* s = nullptr;
        e = cudaGetSymbolAddress(&s, g_mlp_wait_status);
        if (e != cudaSuccess) return e;
        g_hidden_addr[dev] = h;
        g_status_addr[dev] = static_cast<int*>(s);
    }
    *hidden = g_hidden_addr[dev];
    *status = g_status_addr[dev];
    return cudaSuccess;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" sas_status sas_mlp_fwd_noalloc(const void* X, const void* W1, const void* b1, const void* W2,
                                          const void* b2, void* Y, int64_t T, int64_t D, int64_t F,
                                          void* stream) {
    if (!X || !W1 || !W2 || !Y) return SAS_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(W1) || !aligned16(W2) || !aligned16(Y) || (b1 && !aligned16(b1)) ||
        (b2 && !aligned16(b2)))
        return SAS_ERR_INVALID_ARG;
    if (T < 1 || D < 64 || F < 64) return SAS_ERR_INVALID_ARG;
    if (D % 64 != 0 || F % 64 != 0 || D > 65536 || F > 262144) return SAS_ERR_UNSUPPORTED;
    // The hidden activation must fit the fixed array: T * F * 2 bytes.
    if (T > static_cast<int64_t>(kScratchBytes / 2) / F) return SAS_ERR_UNSUPPORTED;

    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SAS_ERR_CUDA;
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (major != 10 || minor != 3) return SAS_ERR_UNSUPPORTED;

    void* hidden = nullptr;
    int* status = nullptr;
    if (device_arrays(dev, &hidden, &status) != cudaSuccess) return SAS_ERR_CUDA;

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const sas::KernelEnv env{s, status, 4000000000LL};
    const char* err = "";
    auto pick_bn = [](int64_t n) { return n % 256 == 0 ? 256 : (n % 128 == 0 ? 128 : 64); };

    // Nothing in the shared array has to start at zero: the up-projection
    // writes every hidden value the down-projection reads.
    sas::GemmProblem g1{};
    g1.A = X; g1.B = W1; g1.C = hidden; g1.bias = b1;
    g1.M = static_cast<int>(T); g1.N = static_cast<int>(F); g1.K = static_cast<int>(D);
    g1.batches = 1; g1.b_mod = 1; g1.c_batch_stride = 0; g1.ldc = static_cast<int>(F);
    g1.gelu = 1; g1.bn = pick_bn(F); g1.max_ctas = 0;
    if (sas::launch_gemm(g1, env, &err) != cudaSuccess) return SAS_ERR_CUDA;

    sas::GemmProblem g2{};
    g2.A = hidden; g2.B = W2; g2.C = Y; g2.bias = b2;
    g2.M = static_cast<int>(T); g2.N = static_cast<int>(D); g2.K = static_cast<int>(F);
    g2.batches = 1; g2.b_mod = 1; g2.c_batch_stride = 0; g2.ldc = static_cast<int>(D);
    g2.gelu = 0; g2.bn = pick_bn(D); g2.max_ctas = 0;
    if (sas::launch_gemm(g2, env, &err) != cudaSuccess) return SAS_ERR_CUDA;
    return SAS_OK;
}

extern "C" sas_status sas_mlp_noalloc_get_device_status(int32_t* out_status) {
    if (out_status == nullptr) return SAS_ERR_INVALID_ARG;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SAS_ERR_CUDA;
    // every call's kernels have finished once the device is idle
    if (cudaDeviceSynchronize() != cudaSuccess) return SAS_ERR_CUDA;
    int v = 0;
    // reads and clears the current device's copy of the word; neither copy allocates
    if (cudaMemcpyFromSymbol(&v, g_mlp_wait_status, sizeof(int)) != cudaSuccess) return SAS_ERR_CUDA;
    const int zero = 0;
    if (cudaMemcpyToSymbol(g_mlp_wait_status, &zero, sizeof(int)) != cudaSuccess) return SAS_ERR_CUDA;
    *out_status = v;
    return SAS_OK;
}
