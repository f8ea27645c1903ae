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
    int flags;     // AQ_LAYOUT_* bits
    int ng;        // groups per row, in/8
    int ng_pad;    // ng rounded up to 32
    int S;         // slices of 32 groups
    int rows_pad;  // out rounded up to 32
    int RBc;       // 32-row blocks, rows_pad/32
    int esz;       // bytes per code (1 or 2; 0 for 4-bit codes, two per byte)
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

// Workspace layout of the split-K GEMV: [status word, 256 B][fp32 partials
// [units][batch][rows_pad]], written by the product kernel and read by the reduction.
constexpr size_t kWsStatusBytes = 256;
inline size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }
inline size_t ws_partial_offset(const Dims&) { return kWsStatusBytes; }

// The table-lookup GEMV (2^8-entry books; batch 1 and 2 with prefixes up to kLutMaxM, batch
// 3..4 with prefixes up to kLutMultiM: their two 64 KiB tables and five or more codebooks
// leave room for a single code stage; batch 5..8 with prefixes up to kLut8M and fp16 tables,
// when the layer has at least kLut8MinItems (slice, book, 32-row block) items, about 30 per SM:
// below that an eight-token table build costs more than the tensor-core kernel's decode)
// writes one partial plane per (slice, book, token); every other GEMV one per (slice, token).
constexpr int kLutMaxM = 8, kLutMultiM = 4, kLut8M = 6;
constexpr long long kLut8MinItems = 4560;
inline int lut_max_m(int batch) {
    return batch <= 2 ? kLutMaxM : batch <= 4 ? kLutMultiM : batch <= 8 ? kLut8M : 0;
}
inline bool uses_lut(const Dims& d, int m, int batch) {
    if (d.B != 8 || m > lut_max_m(batch)) return false;
    return batch <= 4 || (long long)d.S * m * d.RBc >= kLut8MinItems;
}

// Prefill GEMM workspace: [status block, 256 B: status word at 0, the dense form's weight
// factor (float) at kWsWfacOffset][per-token activation factors, float][fp16 copy of bf16
// activations][dense W_m, fp16]. From kGemmDenseTokens tokens, prefixes of two or more books
// decode W_m once into the workspace and run the pair MMAs on it (decoding in the GEMM's inner
// loop is bound by shared-memory gathers, and at that length every weight tile is decoded
// again for every 512 tokens). 4-bit layouts always take the dense form (the in-loop decoders
// read 8-bit codes).
constexpr int kGemmDenseTokens = 2048;
constexpr size_t kWsWfacOffset = 128;
inline bool gemm_uses_dense(const Dims& d, int m, int tokens) {
    return d.B == 4 || (m >= 2 && tokens >= kGemmDenseTokens);
}
inline size_t gemm_xfac_offset() { return kWsStatusBytes; }
inline size_t gemm_x16_offset(int tokens) { return kWsStatusBytes + round_up((size_t)tokens * 4, 256); }
inline size_t gemm_w16_offset(const Dims& d, int tokens) {
    return round_up(gemm_x16_offset(tokens) + (size_t)tokens * (size_t)d.in * 2, 1024);
}
inline size_t gemm_ws_need(const Dims& d, int tokens) {
    if (d.B == 4 || (d.B == 8 && d.M >= 2 && tokens >= kGemmDenseTokens))
        return gemm_w16_offset(d, tokens) + (size_t)d.out * (size_t)d.in * 2;
    return gemm_x16_offset(tokens) + (size_t)tokens * (size_t)d.in * 2;
}

// Records a failed CUDA call (thread-local text for aq_last_error) and returns AQ_ERR_CUDA.
aq_status cuda_fail(cudaError_t e, const char* what);
// AQ_OK if e is cudaSuccess, else cuda_fail(e, what).
inline aq_status cuda_ok(cudaError_t e, const char* what) {
    return e == cudaSuccess ? AQ_OK : cuda_fail(e, what);
}
// Records a failed CUDA driver call (its CUresult code and, when known, name) for
// aq_last_error and returns AQ_ERR_CUDA.
aq_status driver_fail(int result, const char* name, const char* what);

// ---- launchers (each returns AQ_OK or AQ_ERR_CUDA; arguments are already validated) ----
aq_status launch_pack(const Dims& d, const void* codes, void* planes, cudaStream_t st);
aq_status launch_decode(const Dims& d, int m, const void* planes, const void* books,
                        const void* scales, void* w, cudaStream_t st);
// y_prev (optional): added to the product (y = y_prev + product), read in y's type.
aq_status launch_gemv(const Dims& d, int m, const void* planes, const void* books,
                      const void* scales, const void* x, int x_dt, int batch, void* y,
                      int y_dt, void* ws, cudaStream_t st, const void* y_prev = nullptr);
// aq_gemv_group: n (<= 4) layers sharing x; ws[l] = layer l's workspace region.
aq_status launch_gemv_group(const Dims* ds, int n, int m, const void* const* planes,
                            const void* const* books, const void* const* scales, const void* x,
                            int x_dt, int batch, void* const* y, int y_dt, void* const* ws,
                            cudaStream_t st);
aq_status launch_gemm(const Dims& d, int m, const void* planes, const void* books,
                      const void* scales, const void* x, int x_dt, int tokens, void* y, int y_dt,
                      void* ws, cudaStream_t st);
// aq_selftest_wait: one bounded wait that nothing completes (records AQ_ERR_TIMEOUT).
aq_status launch_selftest_wait(unsigned int* status, cudaStream_t st);
// Read probe (aq_selftest_read): reads bytes at src with the GEMV's launch shape.
aq_status launch_selftest_read(const void* src, size_t bytes, unsigned int* sink, cudaStream_t st);
// Beam-search code update (aq_beam_search): workspace bytes, and the launch (validated
// arguments; codes natural [out][in/8][M], uint8 for B <= 8).
size_t beam_ws_bytes(const Dims& d);
aq_status launch_beam(const Dims& d, const void* w, const void* codes, const void* books,
                      const void* scales, const void* h, int h_dt, const double* lambda, int K,
                      void* codes_out, void* ws, cudaStream_t st);
// Per-prefix distortion (aq_wmse): workspace bytes, and the launch (validated arguments).
size_t wmse_ws_bytes(const Dims& d);
aq_status launch_wmse(const Dims& d, const void* w, const void* planes, const void* books,
                      const void* scales, const void* h, int h_dt, const double* lambda,
                      double* out_d, void* ws, cudaStream_t st);

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
// Both halves of a packed pair of 16-bit floats, widened exactly to fp32 (low half first).
// bf16 is the top half of an fp32, so widening is a shift. fp16 is widened by the mixed-type
// add of sm_100 and later (fp16 operand, fp32 operand and result) with -0.0, which returns
// the fp16 value exactly and runs on the fp32 pipe, unlike the conversion instruction.
template <int DT>
__device__ __forceinline__ void widen2(uint32_t w, float& lo, float& hi) {
    if constexpr (DT == AQ_F16) {
        asm("{.reg .b16 l, h;\n\tmov.b32 {l, h}, %2;\n\t"
            "add.rn.f32.f16 %0, l, 0f80000000;\n\tadd.rn.f32.f16 %1, h, 0f80000000;}"
            : "=f"(lo), "=f"(hi) : "r"(w));
    } else {
        lo = __uint_as_float(w << 16);
        hi = __uint_as_float(w & 0xffff0000u);
    }
}

// lo += low half of w, hi += high half of w (16-bit floats of type DT), each with one
// mixed-type add (16-bit operand, fp32 sum and result, sm_100 and later): the same result as
// widening exactly and adding in fp32.
template <int DT>
__device__ __forceinline__ void add_widen2(uint32_t w, float& lo, float& hi) {
    if constexpr (DT == AQ_F16) {
        asm("{.reg .b16 l, h;\n\tmov.b32 {l, h}, %2;\n\t"
            "add.rn.f32.f16 %0, l, %0;\n\tadd.rn.f32.f16 %1, h, %1;}"
            : "+f"(lo), "+f"(hi) : "r"(w));
    } else {
        asm("{.reg .b16 l, h;\n\tmov.b32 {l, h}, %2;\n\t"
            "add.rn.f32.bf16 %0, l, %0;\n\tadd.rn.f32.bf16 %1, h, %1;}"
            : "+f"(lo), "+f"(hi) : "r"(w));
    }
}

template <int DT>
__device__ __forceinline__ void unpack8(const uint4& v, float* f) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) widen2<DT>(w[i], f[2 * i], f[2 * i + 1]);
}

// 16-byte streaming load of data read exactly once (codes): no L1 allocation.
__device__ __forceinline__ uint4 ld_stream_v4(const void* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

// 32-bit shared-window address of a pointer into shared memory, and plain shared loads and
// stores through it (no generic-address conversion per access).
__device__ __forceinline__ float lds_f32(uint32_t addr) {
    float v;
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(addr));
    return v;
}

// Byte permute (PTX prmt, generic mode): selector nibbles pick bytes of {b:a}; a nibble
// with bit 3 set replicates the sign bit of the picked byte.
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// ---- shared-memory barriers, bulk copies and programmatic dependent launch (sm_90+) -------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
                 : "memory");
}

// Make barrier initialisation visible to the async (TMA) proxy and the other threads.
__device__ __forceinline__ void mbar_fence_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// How long one try_wait may park the waiting thread (ns). The thread resumes as soon as the
// phase completes; without a hint try_wait returns almost at once when the phase is still
// open, and a waiting warp then spends issue slots polling that the working warps need.
constexpr uint32_t kSuspendHintNs = 1u << 20;   // about 1 ms

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(kSuspendHintNs)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Every wait in this library is bounded: after kWaitLimitNs of elapsed time it gives up and
// the caller records AQ_ERR_TIMEOUT instead of hanging.
constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s

__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    do {
        if (mbar_try_wait(bar, parity)) return true;
    } while (global_ns() - t0 < kWaitLimitNs);
    return false;
}

// The 32 code bytes of row o of a slice as stored (position p holds group (p + o) mod 32),
// returned in group order: byte q of word j of u is the code of group 4j + q. A rotation by
// o bytes: whole words by o / 4 in three conditional steps (no dynamically indexed register
// array), then the byte part with funnel shifts.
__device__ __forceinline__ void unrotate_codes(const uint32_t (&w)[8], int o, uint32_t (&u)[8]) {
    const int r = o & 31, rw = r >> 2, rb = (r & 3) * 8;
    uint32_t t[8], v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) t[i] = (rw & 1) ? w[(i + 7) & 7] : w[i];
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = (rw & 2) ? t[(i + 6) & 7] : t[i];
#pragma unroll
    for (int i = 0; i < 8; ++i) t[i] = (rw & 4) ? v[(i + 4) & 7] : v[i];
#pragma unroll
    for (int j = 0; j < 8; ++j) u[j] = rb ? __funnelshift_l(t[(j + 7) & 7], t[j], rb) : t[j];
}

// Shared-memory accesses through 32-bit shared-window addresses. lds128 is for data that no
// thread writes while it may be read (codebooks): the compiler may reorder it freely.
// lds128_ordered stays after the barrier wait that precedes it.
__device__ __forceinline__ uint4 lds128(uint32_t a) {
    uint4 v;
    asm("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}
__device__ __forceinline__ uint4 lds128_ordered(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a) : "memory");
    return v;
}
__device__ __forceinline__ void sts128(uint32_t a, uint4 v) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(v.x), "r"(v.y), "r"(v.z),
                 "r"(v.w)
                 : "memory");
}

// 16-byte asynchronous copy global -> shared (cp.async, L2 only), its group commit and wait.
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Interleaved copies (log2) of staged codebooks for the decoders that write a dense W_m
// (aq_decode, and the prefill GEMM's dense form): copy c of codeword j at 16-byte slot
// j * 2^copies + c, read by the lanes L with L mod 2^copies = c. With eight copies the eight
// lanes of a quarter-warp phase of a 16-byte load reach eight different bank groups whatever
// their codes; fewer where m books of 2^8 entries would not fit eight times next to the
// decoders' code buffers.
inline int book_copies_log2(int B, int m) {
    if (B <= 4) return 3;
    return m <= 4 ? 3 : m <= 6 ? 2 : 1;
}

// Bytes of one (row, slice) unit of a code plane: 32 codes of B bits (B = 4, 8 or 16).
constexpr int unit_bytes(int B) { return 32 * B / 8; }
// Bytes of shared memory for the first m codebooks when they are staged there (B <= 8:
// 2^B codewords of 16 bytes each); 16-bit codebooks are read through L2.
constexpr size_t staged_books_bytes(int B, int m) { return B <= 8 ? (size_t)m * (16u << B) : 0; }

// The code at position p (0..31) of a staged (row, slice) unit. B = 4 packs two codes per
// byte: position p in byte p / 2, low four bits for even p, high four bits for odd p.
template <int B>
__device__ __forceinline__ uint32_t unit_code(const unsigned char* u, int p) {
    if constexpr (B == 4) return (uint32_t)(u[p >> 1] >> ((p & 1) * 4)) & 15u;
    else if constexpr (B == 8) return u[p];
    else return ((const uint16_t*)u)[p];
}

// floor(log2(v)) for a finite v > 0 (subnormals count as 2^-126), from the exponent field.
__device__ __forceinline__ int exponent_of(float v) {
    const int e = (int)((__float_as_uint(v) >> 23) & 0xffu);
    return (e == 0 ? 1 : e) - 127;
}
// 2^e as a float, for -126 <= e <= 127.
__device__ __forceinline__ float pow2f(int e) { return __uint_as_float((uint32_t)(e + 127) << 23); }

// Record a device-side failure in the workspace status word (first error wins).
__device__ __forceinline__ void record_status(unsigned int* status, unsigned int code) {
    if (status) atomicCAS(status, 0u, code);
}

// 1-D bulk copy global -> shared (TMA engine), completing on an mbarrier transaction count.
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

// Prefetch `bytes` of global memory into L2 (no data returned to the SM). src 16-byte
// aligned, bytes a multiple of 16.
__device__ __forceinline__ void prefetch_l2(const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// Programmatic dependent launch: wait for the preceding grid's results / allow the next grid
// to start launching. Both are no-ops when the launch has no programmatic dependency.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Named barrier over a subset of the CTA's warps.
__device__ __forceinline__ void named_barrier(int id, int threads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// Packed fp32 pair add (each lane rounded to nearest, as a scalar add): d = a + b.
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
    unsigned long long ar, br, dr;
    asm("mov.b64 %0, {%1, %2};" : "=l"(ar) : "f"(a.x), "f"(a.y));
    asm("mov.b64 %0, {%1, %2};" : "=l"(br) : "f"(b.x), "f"(b.y));
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(dr) : "l"(ar), "l"(br));
    float2 d;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(d.x), "=f"(d.y) : "l"(dr));
    return d;
}

// Packed fp32 pair FMA (one instruction for two lanes of work): d = a * b + c.
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
    unsigned long long ar = *(unsigned long long*)&a, br = *(unsigned long long*)&b,
                       cr = *(unsigned long long*)&c, dr;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(dr) : "l"(ar), "l"(br), "l"(cr));
    return *(float2*)&dr;
}

// Two fp32 values rounded to nearest-even into a packed pair of 16-bit floats of type DT (low
// half first): the same per-value rounding as f32_to_bits.
template <int DT>
__device__ __forceinline__ uint32_t round_pack2(float lo, float hi) {
    uint32_t d;
    if constexpr (DT == AQ_F16) asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
    else asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
    return d;
}

}  // namespace aq
