// aq_gemv_static_scratch: the GEMV of aq_gemv for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc when they run a layer: a plugin inside a host program
// that owns every byte of device memory and offers no allocator, a serving loop that must not
// allocate after start-up (an allocation can synchronise the device or fail under memory
// pressure), or code whose device footprint has to be fixed and known in advance. They cannot
// provide the workspace that aq_gemv needs either. This entry point takes that scratch
// (status word and per-slice partial sums) from a fixed buffer that lives
// in this file as a device array, so a call allocates nothing.
#include <mutex>

#include "aq_internal.cuh"

namespace {

// The fixed scratch buffer. Being a file-scope device array, it is created on every GPU that
// loads this library and stays there until the process exits.
constexpr size_t kStaticScratchBytes = AQ_STATIC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

// In host code, g_static_scratch names a host-side stand-in, not the device buffer; the device
// address is looked up once per device (with that device current) and cached here. The cache
// belongs to the device's primary context: after cudaDeviceReset the address is stale, so
// this entry point must not be used across a reset.
std::mutex g_mu;
void* g_scratch_addr[64] = {};

aq_status static_scratch_address(void** out) {
    int dev = 0;
    if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return aq::cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= 64) return AQ_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        if (cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch); e != cudaSuccess)
            return aq::cuda_fail(e, "cudaGetSymbolAddress");
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return AQ_OK;
}

}  // namespace

extern "C" aq_status aq_gemv_static_scratch(const aq_layout* layout, int m, const void* planes,
                                            const void* books, const void* scales,
                                            const void* x, int x_dtype, int batch, void* y,
                                            int y_dtype, void* stream) {
    // Same argument checks as aq_gemv: run them with no workspace. Any answer other than
    // "workspace missing" (an argument error, or success for empty work) is final.
    const aq_status pre = aq_gemv(layout, m, planes, books, scales, x, x_dtype, batch, y,
                                  y_dtype, nullptr, 0, stream);
    if (pre != AQ_ERR_WORKSPACE) return pre;

    const size_t need = aq_gemv_workspace_bytes(layout, batch);
    if (need == 0 || need > kStaticScratchBytes) return AQ_ERR_WORKSPACE;  // beyond the fixed buffer

    void* scratch = nullptr;
    if (aq_status e = static_scratch_address(&scratch); e != AQ_OK) return e;
    // Nothing is cleared here: the partial sums are always written before they are read, and
    // the status word (zero when the library is loaded) is set only when a device-side wait
    // gives up; it stays set until aq_gemv_static_scratch_status reads and clears it. So a
    // call enqueues the GEMV kernels alone, which keeps the overlap of consecutive calls
    // (programmatic dependent launch) that a memset between them would break.
    return aq_gemv(layout, m, planes, books, scales, x, x_dtype, batch, y, y_dtype, scratch,
                   kStaticScratchBytes, stream);
}

extern "C" aq_status aq_gemv_static_scratch_status(void* stream) {
    void* scratch = nullptr;
    if (aq_status e = static_scratch_address(&scratch); e != AQ_OK) return e;
    return aq_workspace_status(scratch, stream);
}
