// Internal declarations shared by the translation units of libaq (not part of the ABI).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "aq.h"

namespace aq {

// Derived sizes of a validated layout (see the packed-plane description in aq.h).
struct Dims {
    int out, in, G, M, B, book_dt, scale_dt;
    int ng;        // groups per row, in/8
    int ng_pad;    // ng rounded up to 32
    int S;         // slices of 32 groups
    int rows_pad;  // out rounded up to 32
    int RBc;       // 32-row blocks, rows_pad/32
    int esz;       // bytes per code (1 or 2)
    size_t plane_elems, plane_bytes;
};

// Validates a layout; returns AQ_OK and fills d, or the status to report.
aq_status make_dims(const aq_layout* layout, Dims* d);

// Per-device facts cached on first use (SM count, opt-in shared memory).
struct DeviceInfo {
    int sms;
    int smem_optin;
};
aq_status device_info(DeviceInfo* info);

// Workspace layout shared by the split-K kernels: [status 256 B][counters][partials].
constexpr size_t kWsStatusBytes = 256;
inline size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }
inline size_t ws_counter_bytes(const Dims& d) { return round_up((size_t)d.RBc * 4, 256); }
inline size_t ws_partial_offset(const Dims& d) { return kWsStatusBytes + ws_counter_bytes(d); }

// ---- launchers (each returns AQ_OK or AQ_ERR_CUDA; arguments are already validated) ----
aq_status launch_pack(const Dims& d, const void* codes, void* planes, cudaStream_t st);
aq_status launch_decode(const Dims& d, int m, const void* planes, const void* books,
                        const void* scales, void* w, cudaStream_t st);
aq_status launch_gemv(const Dims& d, int m, const void* planes, const void* books,
                      const void* scales, const void* x, int x_dt, int batch, void* y,
                      int y_dt, void* ws, cudaStream_t st);

// ---- device helpers ---------------------------------------------------------------------
template <int DT>
__device__ __forceinline__ float bits_to_f32(uint16_t v) {
    if constexpr (DT == AQ_F16) return __half2float(__ushort_as_half(v));
    else return __bfloat162float(__ushort_as_bfloat16(v));
}

__device__ __forceinline__ float bits_to_f32_rt(uint16_t v, int dt) {
    return dt == AQ_F16 ? __half2float(__ushort_as_half(v))
                        : __bfloat162float(__ushort_as_bfloat16(v));
}

template <int DT>
__device__ __forceinline__ uint16_t f32_to_bits(float v) {
    if constexpr (DT == AQ_F16) return __half_as_ushort(__float2half_rn(v));
    else return __bfloat16_as_ushort(__float2bfloat16_rn(v));
}

// Eight packed 16-bit values (one uint4) -> eight floats.
template <int DT>
__device__ __forceinline__ void unpack8(const uint4& v, float* f) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        f[2 * i] = bits_to_f32<DT>((uint16_t)(w[i] & 0xffffu));
        f[2 * i + 1] = bits_to_f32<DT>((uint16_t)(w[i] >> 16));
    }
}

// 16-byte streaming load of data read exactly once (codes): no L1 allocation.
__device__ __forceinline__ uint4 ld_stream_v4(const void* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

// Byte permute (PTX prmt, generic mode): selector nibbles pick bytes of {b:a}; a nibble
// with bit 3 set replicates the sign bit of the picked byte.
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// Split-K epilogue shared by the GEMV kernels: the CTA that finishes last for a row chunk
// sums the per-slice partials in slice order (deterministic), applies the row scale and
// stores y. Counters are left at zero for the next call.
template <int SDT>
__device__ __forceinline__ void splitk_finish(unsigned int* counters, const float* partials,
                                              const uint16_t* scales, void* y, int y_dt,
                                              int out, int rows_pad, int S, int batch,
                                              int chunk, int row0, int row1) {
    __shared__ int s_last;
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const unsigned prev = atomicAdd(&counters[chunk], 1u);
        s_last = (prev == (unsigned)(S - 1));
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    const int r1 = min(row1, out);
    const int nrows = r1 - row0;
    for (int idx = threadIdx.x; idx < nrows * batch; idx += blockDim.x) {
        const int t = idx / nrows;
        const int r = row0 + (idx - t * nrows);
        float sum = 0.0f;
        for (int s = 0; s < S; ++s) sum += __ldcg(partials + ((size_t)s * batch + t) * rows_pad + r);
        const float v = sum * bits_to_f32<SDT>(scales[r]);
        const size_t yi = (size_t)t * out + r;
        if (y_dt == AQ_F32) ((float*)y)[yi] = v;
        else if (y_dt == AQ_F16) ((uint16_t*)y)[yi] = f32_to_bits<AQ_F16>(v);
        else ((uint16_t*)y)[yi] = f32_to_bits<AQ_BF16>(v);
    }
    if (threadIdx.x == 0) counters[chunk] = 0u;
}

}  // namespace aq
