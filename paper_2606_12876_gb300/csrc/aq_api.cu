// Host side of the C ABI declared in include/aq.h: argument validation, size queries and
// dispatch to the kernel launchers. Nothing here allocates device memory.
#include <cstdio>
#include <mutex>

#include "aq_internal.cuh"

namespace aq {

aq_status make_dims(const aq_layout* L, Dims* d) {
    if (!L || !d) return AQ_ERR_INVALID_ARG;
    if (L->out_features < 0 || L->in_features <= 0 || L->group_size <= 0 || L->num_books <= 0 ||
        L->code_bits <= 0 || L->code_bits > 16)
        return AQ_ERR_INVALID_ARG;
    if (L->in_features % L->group_size) return AQ_ERR_INVALID_ARG;
    if ((L->book_dtype != AQ_F16 && L->book_dtype != AQ_BF16) ||
        (L->scale_dtype != AQ_F16 && L->scale_dtype != AQ_BF16))
        return AQ_ERR_INVALID_ARG;
    if (L->group_size != 8) return AQ_ERR_UNSUPPORTED;
    if (L->code_bits != 4 && L->code_bits != 8 && L->code_bits != 16) return AQ_ERR_UNSUPPORTED;
    if (L->num_books > 8) return AQ_ERR_UNSUPPORTED;
    d->out = L->out_features;
    d->in = L->in_features;
    d->G = L->group_size;
    d->M = L->num_books;
    d->B = L->code_bits;
    d->book_dt = L->book_dtype;
    d->scale_dt = L->scale_dtype;
    if (L->flags & ~AQ_LAYOUT_STATIC_WEIGHTS) return AQ_ERR_INVALID_ARG;
    d->flags = L->flags;
    d->ng = d->in / 8;
    d->ng_pad = (d->ng + 31) / 32 * 32;
    d->S = d->ng_pad / 32;
    d->rows_pad = (int)(((long long)d->out + 31) / 32 * 32);
    d->RBc = d->rows_pad / 32;
    d->esz = d->B / 8;                  // 0 for 4-bit codes (two per byte)
    d->plane_elems = (size_t)d->rows_pad * (size_t)d->ng_pad;
    d->plane_bytes = d->plane_elems * (size_t)d->B / 8;
    return AQ_OK;
}

namespace {
thread_local char g_last_error[256] = "";
}

aq_status cuda_fail(cudaError_t e, const char* what) {
    snprintf(g_last_error, sizeof(g_last_error), "%s: %s (%s)", what, cudaGetErrorName(e),
             cudaGetErrorString(e));
    // A failed launch or runtime call leaves its error as the thread's last error; take it
    // back, so that a later launch checked with cudaGetLastError is not blamed for it (a sticky
    // error, one that corrupted the context, is reported again by every later call anyway).
    (void)cudaGetLastError();
    return AQ_ERR_CUDA;
}

aq_status driver_fail(int result, const char* name, const char* what) {
    snprintf(g_last_error, sizeof(g_last_error), "%s: CUresult %d (%s)", what, result,
             name ? name : "unknown");
    return AQ_ERR_CUDA;
}

aq_status device_info(DeviceInfo* info) {
    static std::mutex mu;
    static DeviceInfo cache[64];
    static bool have[64] = {};
    int dev = 0;
    if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= 64) return AQ_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(mu);
    if (!have[dev]) {
        DeviceInfo di{};
        if (cudaError_t e = cudaDeviceGetAttribute(&di.sms, cudaDevAttrMultiProcessorCount, dev);
            e != cudaSuccess)
            return cuda_fail(e, "cudaDeviceGetAttribute");
        if (cudaError_t e = cudaDeviceGetAttribute(&di.smem_optin,
                                                   cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
            e != cudaSuccess)
            return cuda_fail(e, "cudaDeviceGetAttribute");
        cache[dev] = di;
        have[dev] = true;
    }
    *info = cache[dev];
    return AQ_OK;
}

}  // namespace aq

using aq::Dims;

namespace {

inline bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

inline cudaStream_t as_stream(void* s) { return (cudaStream_t)s; }

aq_status check_m(const Dims& d, int m) { return (m < 1 || m > d.M) ? AQ_ERR_INVALID_ARG : AQ_OK; }

aq_status check_ptrs(std::initializer_list<const void*> ps) {
    for (const void* p : ps)
        if (!p) return AQ_ERR_INVALID_ARG;
    for (const void* p : ps)
        if (!aligned16(p)) return AQ_ERR_ALIGNMENT;
    return AQ_OK;
}

// GEMM workspace: status word, then room for an fp16 copy of bf16 activations.
size_t gemm_ws_bytes(const Dims& d, int tokens) { return aq::gemm_ws_need(d, tokens); }

size_t gemv_ws_bytes(const Dims& d, int batch) {
    // Partial planes: S per token, or S per book and token for the largest prefix the
    // table-lookup kernel serves at this batch.
    size_t planes = (size_t)d.S * (size_t)batch;
    const int lm = aq::lut_max_m(batch), mt = d.M < lm ? d.M : lm;
    if (mt > 0 && aq::uses_lut(d, mt, batch)) planes = (size_t)d.S * (size_t)batch * (size_t)mt;
    return aq::ws_partial_offset(d) + planes * (size_t)d.rows_pad * 4;
}

}  // namespace

extern "C" {

int aq_abi_version(void) { return AQ_ABI_VERSION; }

const char* aq_last_error(void) { return aq::g_last_error; }

const char* aq_status_string(int status) {
    switch (status) {
        case AQ_OK: return "ok";
        case AQ_ERR_INVALID_ARG: return "invalid argument";
        case AQ_ERR_UNSUPPORTED: return "unsupported configuration";
        case AQ_ERR_ALIGNMENT: return "pointer not 16-byte aligned";
        case AQ_ERR_CUDA: return "CUDA error";
        case AQ_ERR_TIMEOUT: return "device-side wait timed out";
        case AQ_ERR_WORKSPACE: return "workspace missing or too small";
        default: return "unknown status";
    }
}

size_t aq_plane_bytes(const aq_layout* layout) {
    Dims d;
    return aq::make_dims(layout, &d) == AQ_OK ? d.plane_bytes : 0;
}

size_t aq_packed_bytes(const aq_layout* layout, int m) {
    Dims d;
    if (aq::make_dims(layout, &d) != AQ_OK || check_m(d, m) != AQ_OK) return 0;
    return (size_t)m * d.plane_bytes;
}

aq_status aq_pack(const aq_layout* layout, const void* codes, void* planes, void* stream) {
    Dims d;
    aq_status st = aq::make_dims(layout, &d);
    if (st != AQ_OK) return st;
    if ((st = check_ptrs({planes})) != AQ_OK) return st;
    if (d.out > 0 && (st = check_ptrs({codes})) != AQ_OK) return st;
    return aq::launch_pack(d, codes, planes, as_stream(stream));
}

aq_status aq_decode(const aq_layout* layout, int m, const void* planes, const void* books,
                    const void* scales, void* w, void* stream) {
    Dims d;
    aq_status st = aq::make_dims(layout, &d);
    if (st != AQ_OK) return st;
    if ((st = check_m(d, m)) != AQ_OK) return st;
    if (d.out == 0) return AQ_OK;
    if ((st = check_ptrs({planes, books, scales, w})) != AQ_OK) return st;
    return aq::launch_decode(d, m, planes, books, scales, w, as_stream(stream));
}

size_t aq_gemv_workspace_bytes(const aq_layout* layout, int batch) {
    Dims d;
    if (aq::make_dims(layout, &d) != AQ_OK || batch < 0 || batch > 16) return 0;
    return gemv_ws_bytes(d, batch < 1 ? 1 : batch);
}

aq_status aq_gemv(const aq_layout* layout, int m, const void* planes, const void* books,
                  const void* scales, const void* x, int x_dtype, int batch, void* y,
                  int y_dtype, void* workspace, size_t workspace_bytes, void* stream) {
    Dims d;
    aq_status st = aq::make_dims(layout, &d);
    if (st != AQ_OK) return st;
    if ((st = check_m(d, m)) != AQ_OK) return st;
    if (batch < 0 || batch > 16) return AQ_ERR_INVALID_ARG;
    if (x_dtype != AQ_F16 && x_dtype != AQ_BF16) return AQ_ERR_INVALID_ARG;
    if (y_dtype != AQ_F16 && y_dtype != AQ_BF16 && y_dtype != AQ_F32) return AQ_ERR_INVALID_ARG;
    if (batch == 0 || d.out == 0) return AQ_OK;
    if ((st = check_ptrs({planes, books, scales, x, y})) != AQ_OK) return st;
    if (!workspace || workspace_bytes < gemv_ws_bytes(d, batch)) return AQ_ERR_WORKSPACE;
    if (!aligned16(workspace)) return AQ_ERR_ALIGNMENT;
    return aq::launch_gemv(d, m, planes, books, scales, x, x_dtype, batch, y, y_dtype, workspace,
                           as_stream(stream));
}

// Layouts of a group: 1..4 valid layouts with the same in_features, code width and codebook
// and scale types; fills ds.
static aq_status group_dims(int n, const aq_layout* layouts, Dims* ds) {
    if (n < 1 || n > 4 || !layouts) return AQ_ERR_INVALID_ARG;
    for (int l = 0; l < n; ++l) {
        if (aq_status st = aq::make_dims(&layouts[l], &ds[l]); st != AQ_OK) return st;
        if (ds[l].in != ds[0].in || ds[l].B != ds[0].B || ds[l].book_dt != ds[0].book_dt ||
            ds[l].scale_dt != ds[0].scale_dt)
            return AQ_ERR_INVALID_ARG;
    }
    return AQ_OK;
}

size_t aq_gemv_group_workspace_bytes(int n, const aq_layout* layouts, int batch) {
    Dims ds[4];
    if (group_dims(n, layouts, ds) != AQ_OK || batch < 0 || batch > 16) return 0;
    size_t total = 0;
    for (int l = 0; l < n; ++l) total += aq::round_up(gemv_ws_bytes(ds[l], batch), 256);
    return total;
}

aq_status aq_gemv_group(int n, const aq_layout* layouts, int m, const void* const* planes,
                        const void* const* books, const void* const* scales, const void* x,
                        int x_dtype, int batch, void* const* y, int y_dtype, void* workspace,
                        size_t workspace_bytes, void* stream) {
    Dims ds[4];
    aq_status st = group_dims(n, layouts, ds);
    if (st != AQ_OK) return st;
    for (int l = 0; l < n; ++l)
        if ((st = check_m(ds[l], m)) != AQ_OK) return st;
    if (batch < 0 || batch > 16) return AQ_ERR_INVALID_ARG;
    if (x_dtype != AQ_F16 && x_dtype != AQ_BF16) return AQ_ERR_INVALID_ARG;
    if (y_dtype != AQ_F16 && y_dtype != AQ_BF16 && y_dtype != AQ_F32) return AQ_ERR_INVALID_ARG;
    if (!planes || !books || !scales || !y) return AQ_ERR_INVALID_ARG;
    if (batch == 0) return AQ_OK;
    for (int l = 0; l < n; ++l)
        if (ds[l].out > 0)
            if ((st = check_ptrs({planes[l], books[l], scales[l], x, y[l]})) != AQ_OK) return st;
    if (!workspace || workspace_bytes < aq_gemv_group_workspace_bytes(n, layouts, batch))
        return AQ_ERR_WORKSPACE;
    if (!aligned16(workspace)) return AQ_ERR_ALIGNMENT;
    void* ws[4];
    size_t off = 0;
    for (int l = 0; l < n; ++l) {
        ws[l] = (char*)workspace + off;
        off += aq::round_up(gemv_ws_bytes(ds[l], batch), 256);
    }
    return aq::launch_gemv_group(ds, n, m, planes, books, scales, x, x_dtype, batch, y, y_dtype, ws,
                                 as_stream(stream));
}

aq_status aq_gemv_refine(const aq_layout* layout, int m, const void* planes, const void* books,
                         const void* scales, const void* x, int x_dtype, int batch,
                         const void* y_prev, void* y, int y_dtype, void* workspace,
                         size_t workspace_bytes, void* stream) {
    Dims d;
    aq_status st = aq::make_dims(layout, &d);
    if (st != AQ_OK) return st;
    if ((st = check_m(d, m)) != AQ_OK) return st;
    if (batch < 0 || batch > 16) return AQ_ERR_INVALID_ARG;
    if (x_dtype != AQ_F16 && x_dtype != AQ_BF16) return AQ_ERR_INVALID_ARG;
    if (y_dtype != AQ_F16 && y_dtype != AQ_BF16 && y_dtype != AQ_F32) return AQ_ERR_INVALID_ARG;
    if (batch == 0 || d.out == 0) return AQ_OK;
    if ((st = check_ptrs({planes, books, scales, x, y})) != AQ_OK) return st;
    if (y_prev && !aligned16(y_prev)) return AQ_ERR_ALIGNMENT;
    if (!workspace || workspace_bytes < gemv_ws_bytes(d, batch)) return AQ_ERR_WORKSPACE;
    if (!aligned16(workspace)) return AQ_ERR_ALIGNMENT;
    // The increment of book m-1 is a one-book product: plane m-1 and book m-1 are the whole
    // code planes and codebooks of a one-book layout (the partial planes it needs fit in the
    // workspace of the full layout).
    const char* plane1 = (const char*)planes + (size_t)(m - 1) * d.plane_bytes;
    const char* book1 = (const char*)books + (size_t)(m - 1) * ((size_t)1 << d.B) * d.G * 2;
    return aq::launch_gemv(d, 1, plane1, book1, scales, x, x_dtype, batch, y, y_dtype, workspace,
                           as_stream(stream), y_prev);
}

size_t aq_wmse_workspace_bytes(const aq_layout* layout) {
    Dims d;
    if (aq::make_dims(layout, &d) != AQ_OK) return 0;
    return aq::wmse_ws_bytes(d);
}

aq_status aq_wmse(const aq_layout* layout, const void* w, const void* planes, const void* books,
                  const void* scales, const void* h, int h_dtype, const double* lambda, double* d_out,
                  void* workspace, size_t workspace_bytes, void* stream) {
    Dims d;
    aq_status st = aq::make_dims(layout, &d);
    if (st != AQ_OK) return st;
    if (h_dtype != AQ_F32 && h_dtype != AQ_BF16) return AQ_ERR_INVALID_ARG;
    if (!d_out) return AQ_ERR_INVALID_ARG;
    if (((uintptr_t)d_out & 7u) != 0) return AQ_ERR_ALIGNMENT;
    if (d.out > 0) {
        if ((st = check_ptrs({w, planes, books, scales, h})) != AQ_OK) return st;
        if (!workspace || workspace_bytes < aq::wmse_ws_bytes(d)) return AQ_ERR_WORKSPACE;
        if (!aligned16(workspace)) return AQ_ERR_ALIGNMENT;
    }
    return aq::launch_wmse(d, w, planes, books, scales, h, h_dtype, lambda, d_out, workspace,
                           as_stream(stream));
}

size_t aq_beam_workspace_bytes(const aq_layout* layout) {
    Dims d;
    if (aq::make_dims(layout, &d) != AQ_OK) return 0;
    return aq::beam_ws_bytes(d);
}

aq_status aq_beam_search(const aq_layout* layout, const void* w, const void* codes,
                         const void* books, const void* scales, const void* h, int h_dtype,
                         const double* lambda, int beam, void* codes_out, void* workspace,
                         size_t workspace_bytes, void* stream) {
    Dims d;
    aq_status st = aq::make_dims(layout, &d);
    if (st != AQ_OK) return st;
    if (d.B == 16) return AQ_ERR_UNSUPPORTED;          // 2^16-entry books do not fit on chip
    if (h_dtype != AQ_F32 && h_dtype != AQ_BF16) return AQ_ERR_INVALID_ARG;
    if (beam < 1 || beam > 16) return AQ_ERR_INVALID_ARG;
    if (lambda)
        for (int k = 0; k < d.M; ++k)
            if (!(lambda[k] >= 0.0)) return AQ_ERR_INVALID_ARG;
    if (d.out == 0) return AQ_OK;
    if ((st = check_ptrs({w, codes, books, scales, h, codes_out})) != AQ_OK) return st;
    if (!workspace || workspace_bytes < aq::beam_ws_bytes(d)) return AQ_ERR_WORKSPACE;
    if (!aligned16(workspace)) return AQ_ERR_ALIGNMENT;
    return aq::launch_beam(d, w, codes, books, scales, h, h_dtype, lambda, beam, codes_out,
                           workspace, as_stream(stream));
}

size_t aq_gemm_workspace_bytes(const aq_layout* layout, int tokens) {
    Dims d;
    if (aq::make_dims(layout, &d) != AQ_OK || tokens < 0) return 0;
    return gemm_ws_bytes(d, tokens);
}

aq_status aq_gemm(const aq_layout* layout, int m, const void* planes, const void* books,
                  const void* scales, const void* x, int x_dtype, int tokens, void* y,
                  int y_dtype, void* workspace, size_t workspace_bytes, void* stream) {
    Dims d;
    aq_status st = aq::make_dims(layout, &d);
    if (st != AQ_OK) return st;
    if ((st = check_m(d, m)) != AQ_OK) return st;
    if (tokens < 0) return AQ_ERR_INVALID_ARG;
    if (x_dtype != AQ_F16 && x_dtype != AQ_BF16) return AQ_ERR_INVALID_ARG;
    if (y_dtype != AQ_F16 && y_dtype != AQ_BF16 && y_dtype != AQ_F32) return AQ_ERR_INVALID_ARG;
    if (tokens == 0 || d.out == 0) return AQ_OK;
    if ((st = check_ptrs({planes, books, scales, x, y})) != AQ_OK) return st;
    if (!workspace || workspace_bytes < gemm_ws_bytes(d, tokens)) return AQ_ERR_WORKSPACE;
    if (!aligned16(workspace)) return AQ_ERR_ALIGNMENT;
    return aq::launch_gemm(d, m, planes, books, scales, x, x_dtype, tokens, y, y_dtype, workspace,
                           as_stream(stream));
}

aq_status aq_selftest_wait(void* workspace, size_t workspace_bytes, void* stream) {
    if (!workspace) return AQ_ERR_INVALID_ARG;
    if (workspace_bytes < aq::kWsStatusBytes) return AQ_ERR_WORKSPACE;
    if (!aligned16(workspace)) return AQ_ERR_ALIGNMENT;
    return aq::launch_selftest_wait((unsigned int*)workspace, as_stream(stream));
}

aq_status aq_selftest_read(const void* src, size_t bytes, void* sink, void* stream) {
    if (!sink || (!src && bytes > 0)) return AQ_ERR_INVALID_ARG;
    if (!aligned16(src) || ((uintptr_t)sink & 3u) || bytes % 16) return AQ_ERR_ALIGNMENT;
    return aq::launch_selftest_read(src, bytes, (unsigned int*)sink, as_stream(stream));
}

aq_status aq_workspace_init(void* workspace, size_t bytes, void* stream) {
    if (!workspace) return AQ_ERR_INVALID_ARG;
    if (!aligned16(workspace)) return AQ_ERR_ALIGNMENT;
    return aq::cuda_ok(cudaMemsetAsync(workspace, 0, bytes, as_stream(stream)), "cudaMemsetAsync");
}

aq_status aq_workspace_status(void* workspace, void* stream) {
    if (!workspace) return AQ_ERR_INVALID_ARG;
    if (!aligned16(workspace)) return AQ_ERR_ALIGNMENT;
    unsigned int word = 0;
    const cudaStream_t st = as_stream(stream);
    aq_status rc = aq::cuda_ok(cudaMemcpyAsync(&word, workspace, 4, cudaMemcpyDeviceToHost, st),
                               "cudaMemcpyAsync");
    if (rc == AQ_OK) rc = aq::cuda_ok(cudaStreamSynchronize(st), "cudaStreamSynchronize");
    if (rc != AQ_OK || word == 0) return rc;
    rc = aq::cuda_ok(cudaMemsetAsync(workspace, 0, 4, st), "cudaMemsetAsync");
    if (rc == AQ_OK) rc = aq::cuda_ok(cudaStreamSynchronize(st), "cudaStreamSynchronize");
    if (rc != AQ_OK) return rc;
    return (aq_status)word;
}

}  // extern "C"
