// aq_gemm: prefill product y = x * W_m^T for many tokens on the tcgen05 tensor cores, with W_m
// (the prefix-m additive reconstruction of Sec. 3.2 / Sec. 5) decoded tile by tile into shared
// memory and never written to HBM.
//
// Tile: 512 tokens x 128 output rows, K in steps of 64 inputs (one 128-byte swizzle row of
// 16-bit values). The four 128x128 fp32 accumulators fill the 512 columns of tensor memory, so
// every decoded weight tile feeds 512 tokens. Roles (12 warps):
//   warp 0      TMA producer: activation tiles (2-D tensor map, 128-byte swizzle, two
//               256-token boxes per stage) and, once per 256-input slice, the slice's code rows
//               of the first m planes (1-D bulk copies; a tile's rows of a slice are contiguous
//               in every plane).
//   warp 1      allocates tensor memory; lane 0 issues tcgen05.mma (4 token blocks x 4 K=16
//               steps per stage) and commits stage-release / accumulator-ready barriers.
//   warps 4-11  decoders: each thread owns one weight row and four groups of every stage; it
//               sums the m codewords in fp32 (book order), rounds once to the book type and
//               writes the 16-byte group into the B tile in the UMMA K-major 128-byte-swizzle
//               layout. Afterwards the same warps are the epilogue: tcgen05.ld from tensor
//               memory, times the row scale (R1), round, store.
// Operands are fp16 (kind::f16, fp32 accumulation): the summed weights are rounded once to
// fp16 (about 2^-11 relative), which keeps the product inside the stated per-element bound;
// bf16 activations are first converted to fp16 into the workspace (exact for normal-range
// values, which bf16's 8-bit significand always fits; saturating beyond +-65504).
// Every mbarrier wait is bounded; a timeout records AQ_ERR_TIMEOUT in the workspace status
// word and the CTA winds down without waiting further.
#include <cuda.h>

#include <cstring>
#include <mutex>

#include "aq_internal.cuh"

namespace aq {
namespace {

constexpr int kBM = 128;                      // tokens per MMA
constexpr int kMT = 4;                        // token blocks per tile (512 tokens)
constexpr int kBN = 128;                      // output rows per tile
constexpr int kBK = 64;                       // inputs per stage
constexpr int kStages = 2;
constexpr int kGemmThreads = 384;
constexpr int kDecWarp0 = 4, kDecWarps = 8;
constexpr int kGemmMaxM = 4;

constexpr int kAStage = kMT * kBM * 128;      // 64 KiB
constexpr int kBStage = kBN * 128;            // 16 KiB
constexpr int kCodeBuf = kGemmMaxM * kBN * 32;   // one slice of codes, all planes (16 KiB)

// Shared-memory map (offsets from a 1024-byte aligned base).
constexpr int kOffA = 0;
constexpr int kOffB = kOffA + kStages * kAStage;
constexpr int kOffCodes = kOffB + kStages * kBStage;
constexpr int kOffBooks = kOffCodes + 2 * kCodeBuf;
constexpr int kOffScale = kOffBooks + kGemmMaxM * 4096;
constexpr int kOffBar = kOffScale + kBN * 4;
constexpr int kNumBars = 3 * kStages + 4 + 1;   // full_a, full_b, empty, codes_full[2], codes_empty[2], acc
constexpr int kOffTmem = kOffBar + kNumBars * 8;
constexpr int kSmemUsed = kOffTmem + 16;
constexpr int kGemmSmem = kSmemUsed + 1024;     // slack for aligning the base to 1024 bytes

// ---- tcgen05 / TMA helpers (PTX) -----------------------------------------------------------

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int c0, int c1,
                                            uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
        "l"((uint64_t)map), "r"(c0), "r"(c1), "r"(smem_u32(bar))
        : "memory");
}

// UMMA shared-memory descriptor: K-major operand, 128-byte swizzle, 8-row atoms 1024 bytes
// apart (SBO), version 1, leading offset unused (16 bytes).
__device__ __forceinline__ uint64_t umma_desc_sw128(uint32_t saddr) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)64 << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

__device__ __forceinline__ void umma_f16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                         uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void umma_commit(uint64_t* bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// 32 consecutive fp32 columns of this warp's 32 tensor-memory lanes (one lane per thread).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
        "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ uint32_t pack2(float lo, float hi, int dt) {
    if (dt == AQ_BF16) {
        __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
        return *(uint32_t*)&h;
    }
    __half2 h = __floats2half2_rn(lo, hi);
    return *(uint32_t*)&h;
}

// Bounded wait that gives up at once after a failure anywhere in the CTA.
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort,
                                              unsigned int* status) {
    if (*abort) return false;
    if (mbar_wait(bar, parity)) return true;
    record_status(status, AQ_ERR_TIMEOUT);
    *abort = 1;
    return false;
}

template <int BDT>
__global__ void __launch_bounds__(kGemmThreads, 1)
gemm_kernel(const __grid_constant__ CUtensorMap xmap, const uint8_t* __restrict__ planes,
            const uint16_t* __restrict__ books, const uint16_t* __restrict__ scales, void* y,
            int y_dt, int scale_dt, unsigned int* __restrict__ status, int m, int tokens, int out,
            int in, int ng, int rows_pad, size_t plane_bytes) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* bars = (uint64_t*)(smem + kOffBar);
    uint64_t* full_a = bars;
    uint64_t* full_b = bars + kStages;
    uint64_t* empty = bars + 2 * kStages;
    uint64_t* codes_full = bars + 3 * kStages;
    uint64_t* codes_empty = codes_full + 2;
    uint64_t* acc_full = codes_empty + 2;
    uint32_t* tmem_slot = (uint32_t*)(smem + kOffTmem);
    float* scale_s = (float*)(smem + kOffScale);
    const uint4* books_s = (const uint4*)(smem + kOffBooks);
    __shared__ volatile int s_abort;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int n0 = blockIdx.x * kBN;          // first output row of the tile
    const int t0 = blockIdx.y * (kMT * kBM);  // first token of the tile
    const int nk = (in + kBK - 1) / kBK;      // K steps
    const int nsl = (nk + 3) / 4;             // 256-input slices
    const int rows_valid = min(kBN, rows_pad - n0);   // packed rows present (multiple of 32)

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full_a[s], 1);             // producer arrival + TMA bytes
            mbar_init(&full_b[s], kDecWarps);     // one arrival per decoder warp
            mbar_init(&empty[s], 1);              // tcgen05.commit
        }
        for (int c = 0; c < 2; ++c) {
            mbar_init(&codes_full[c], 1);
            mbar_init(&codes_empty[c], kDecWarps);
        }
        mbar_init(acc_full, 1);
        mbar_fence_init();
        s_abort = 0;
    }
    if (warp == 1) {   // tensor memory: 512 columns = four 128x128 fp32 accumulators
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(
                         smem_u32(tmem_slot))
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    pdl_wait();

    if (warp == 0) {
        // ---------------- producer
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&xmap) : "memory");
            int issued_a = 0, issued_c = 0;
            for (int ks = 0; ks < nk && !s_abort; ++ks) {
                const int st = ks % kStages;
                if (ks % 4 == 0) {                        // codes of slice ks/4
                    const int sl = ks / 4, cb = sl & 1;
                    if (sl >= 2 && !wait_or_abort(&codes_empty[cb], ((sl >> 1) - 1) & 1, &s_abort, status))
                        break;
                    mbar_arrive_expect_tx(&codes_full[cb], (uint32_t)(m * rows_valid * 32));
                    for (int k = 0; k < m; ++k)
                        bulk_g2s(smem + kOffCodes + cb * kCodeBuf + k * (kBN * 32),
                                 planes + (size_t)k * plane_bytes + ((size_t)sl * rows_pad + n0) * 32,
                                 (uint32_t)(rows_valid * 32), &codes_full[cb]);
                    ++issued_c;
                }
                if (ks >= kStages &&
                    !wait_or_abort(&empty[st], ((ks / kStages) - 1) & 1, &s_abort, status))
                    break;
                mbar_arrive_expect_tx(&full_a[st], (uint32_t)kAStage);
                unsigned char* a = smem + kOffA + st * kAStage;
                tma_load_2d(a, &xmap, ks * kBK, t0, &full_a[st]);
                tma_load_2d(a + kAStage / 2, &xmap, ks * kBK, t0 + 2 * kBM, &full_a[st]);
                ++issued_a;
            }
            // No copy may still be in flight when the CTA exits.
            for (int j = max(0, issued_a - kStages); j < issued_a; ++j)
                mbar_wait(&full_a[j % kStages], (j / kStages) & 1);
            for (int j = max(0, issued_c - 2); j < issued_c; ++j)
                mbar_wait(&codes_full[j & 1], (j >> 1) & 1);
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer
        if (lane == 0) {
            // kind::f16 instruction descriptor: fp32 accumulator, fp16 A and B, both K-major,
            // N = 128, M = 128.
            const uint32_t idesc = (1u << 4) | ((uint32_t)(kBN >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);
            for (int ks = 0; ks < nk; ++ks) {
                const int st = ks % kStages;
                const uint32_t par = (ks / kStages) & 1;
                if (!wait_or_abort(&full_a[st], par, &s_abort, status)) break;
                if (!wait_or_abort(&full_b[st], par, &s_abort, status)) break;
                tc_fence_after();
                const uint32_t a0 = smem_u32(smem + kOffA + st * kAStage);
                const uint32_t b0 = smem_u32(smem + kOffB + st * kBStage);
#pragma unroll
                for (int i = 0; i < kMT; ++i)
#pragma unroll
                    for (int kk = 0; kk < kBK / 16; ++kk)
                        umma_f16(tmem + i * kBN, umma_desc_sw128(a0 + i * (kBM * 128) + kk * 32),
                                 umma_desc_sw128(b0 + kk * 32), idesc, (ks > 0 || kk > 0) ? 1u : 0u);
                umma_commit(&empty[st]);
            }
            umma_commit(acc_full);
        }
    } else if (warp >= kDecWarp0) {
        // ---------------- decoders, then epilogue
        const int dt = tid - kDecWarp0 * 32;        // 0..255
        const int n = dt & (kBN - 1);               // tile row owned by this thread
        const int cs = dt >> 7;                     // groups 4cs..4cs+3 of every stage
        const int row = n0 + n;
        for (int i = dt; i < m * 256; i += kDecWarps * 32)
            ((uint4*)books_s)[i] = __ldg((const uint4*)books + i);
        if (dt < kBN) scale_s[dt] = (n0 + dt < out) ? bits_to_f32_rt(scales[n0 + dt], scale_dt) : 0.0f;
        named_barrier(1, kDecWarps * 32);

        const int r = row & 31;                     // rotation of this row's codes
        for (int sl = 0; sl < nsl; ++sl) {
            const int cb = sl & 1;
            uint32_t cw[kGemmMaxM][8];              // this row's 32 codes of the slice, per plane
            const bool have = wait_or_abort(&codes_full[cb], (sl >> 1) & 1, &s_abort, status);
#pragma unroll
            for (int k = 0; k < kGemmMaxM; ++k) {
                uint32_t w[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
                if (have && k < m && n < rows_valid) {
                    const uint4* src = (const uint4*)(smem + kOffCodes + cb * kCodeBuf + k * (kBN * 32) + n * 32);
                    const uint4 lo = src[0], hi = src[1];
                    w[0] = lo.x; w[1] = lo.y; w[2] = lo.z; w[3] = lo.w;
                    w[4] = hi.x; w[5] = hi.y; w[6] = hi.z; w[7] = hi.w;
                }
                // Undo the row rotation: byte q of the result is the code of group q of the
                // slice (position p holds group (p + row) mod 32, i.e. rotate left by r bytes).
                // Word rotation V[i] = W[i - rw] as three conditional steps (rw is per thread,
                // so no dynamically indexed register array), then the byte part with funnel
                // shifts: out word i = bytes of V[i-1]:V[i] shifted left by 8*(r mod 4).
                const int rw = r >> 2, rb = (r & 3) * 8;
                uint32_t v[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) v[i] = w[i];
                {
                    uint32_t t[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) t[i] = (rw & 1) ? v[(i + 7) & 7] : v[i];
#pragma unroll
                    for (int i = 0; i < 8; ++i) v[i] = (rw & 2) ? t[(i + 6) & 7] : t[i];
#pragma unroll
                    for (int i = 0; i < 8; ++i) t[i] = (rw & 4) ? v[(i + 4) & 7] : v[i];
#pragma unroll
                    for (int i = 0; i < 8; ++i) v[i] = t[i];
                }
#pragma unroll
                for (int i = 0; i < 8; ++i) cw[k][i] = rb ? __funnelshift_l(v[(i + 7) & 7], v[i], rb) : v[i];
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&codes_empty[cb]);

#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int ks = sl * 4 + j;
                if (ks >= nk) break;
                const int st = ks % kStages;
                if (ks >= kStages) wait_or_abort(&empty[st], ((ks / kStages) - 1) & 1, &s_abort, status);
                unsigned char* bt = smem + kOffB + st * kBStage + (n >> 3) * 1024 + (n & 7) * 128;
#pragma unroll
                for (int cc = 0; cc < 4; ++cc) {
                    const int c = cs * 4 + cc;                  // group within the stage
                    const int g = sl * 32 + j * 8 + c;          // group within the row
                    float acc[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[e] = 0.0f;
#pragma unroll
                    for (int k = 0; k < kGemmMaxM; ++k) {
                        if (k < m) {
                            // group j*8 + 4*cs + cc of the slice: word 2j + cs, byte cc
                            const uint32_t word = cs ? cw[k][2 * j + 1] : cw[k][2 * j];
                            const uint32_t code = (word >> (cc * 8)) & 0xffu;
                            const uint4 q = books_s[k * 256 + code];
                            float f[8];
                            unpack8<BDT>(q, f);
#pragma unroll
                            for (int e = 0; e < 8; ++e) acc[e] += f[e];
                        }
                    }
                    const bool valid = g < ng && row < out;
                    uint4 o;
                    o.x = valid ? pack2(acc[0], acc[1], AQ_F16) : 0u;
                    o.y = valid ? pack2(acc[2], acc[3], AQ_F16) : 0u;
                    o.z = valid ? pack2(acc[4], acc[5], AQ_F16) : 0u;
                    o.w = valid ? pack2(acc[6], acc[7], AQ_F16) : 0u;
                    *(uint4*)(bt + ((c ^ (n & 7)) << 4)) = o;
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(&full_b[st]);
            }
        }

        // ---------------- epilogue: accumulators -> scale -> y
        const bool ready = __all_sync(0xffffffffu, wait_or_abort(acc_full, 0, &s_abort, status));
        tc_fence_after();
        __syncwarp();
        // Vector stores need 16-byte aligned row segments: out a multiple of 8 (the output
        // pointer itself is 16-byte aligned by contract).
        const bool vec = (out & 7) == 0;
        if (ready) {
            const int q = warp & 3;                       // tensor-memory lane quarter
            const int half = (warp - kDecWarp0) >> 2;     // token blocks 2*half, 2*half+1
            for (int i = 2 * half; i < 2 * half + 2; ++i) {
                const int t = t0 + i * kBM + q * 32 + lane;
                for (int nc = 0; nc < kBN; nc += 32) {
                    float v[32];
                    tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + i * kBN + nc, v);
                    if (t < tokens) {
                        const size_t base = (size_t)t * out + n0 + nc;
                        if (vec && n0 + nc + 32 <= out) {
                            if (y_dt == AQ_F32) {
                                float4* yp = (float4*)((float*)y + base);
#pragma unroll
                                for (int e = 0; e < 32; e += 4)
                                    yp[e / 4] = make_float4(v[e] * scale_s[nc + e], v[e + 1] * scale_s[nc + e + 1],
                                                            v[e + 2] * scale_s[nc + e + 2], v[e + 3] * scale_s[nc + e + 3]);
                            } else {
                                uint4* yp = (uint4*)((uint16_t*)y + base);
#pragma unroll
                                for (int e = 0; e < 32; e += 8)
                                    yp[e / 8] = make_uint4(pack2(v[e] * scale_s[nc + e], v[e + 1] * scale_s[nc + e + 1], y_dt),
                                                           pack2(v[e + 2] * scale_s[nc + e + 2], v[e + 3] * scale_s[nc + e + 3], y_dt),
                                                           pack2(v[e + 4] * scale_s[nc + e + 4], v[e + 5] * scale_s[nc + e + 5], y_dt),
                                                           pack2(v[e + 6] * scale_s[nc + e + 6], v[e + 7] * scale_s[nc + e + 7], y_dt));
                            }
                        } else {
#pragma unroll
                            for (int e = 0; e < 32; ++e) {
                                if (n0 + nc + e < out) {
                                    const float val = v[e] * scale_s[nc + e];
                                    if (y_dt == AQ_F32) ((float*)y)[base + e] = val;
                                    else if (y_dt == AQ_BF16) ((uint16_t*)y)[base + e] = f32_to_bits<AQ_BF16>(val);
                                    else ((uint16_t*)y)[base + e] = f32_to_bits<AQ_F16>(val);
                                }
                            }
                        }
                    }
                }
            }
        }
    }

    // ---------------- teardown: release tensor memory once every reader is done
    tc_fence_before();
    __syncthreads();
    pdl_launch_dependents();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem) : "memory");
    }
}

// bf16 -> fp16 copy of the activations (8 values per thread; saturating at +-65504).
__global__ void __launch_bounds__(256) bf16_to_f16_kernel(const uint4* __restrict__ src,
                                                          uint4* __restrict__ dst, size_t n8) {
    pdl_wait();
    pdl_launch_dependents();
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n8;
         i += (size_t)gridDim.x * blockDim.x) {
        const uint4 v = src[i];
        float f[8];
        unpack8<AQ_BF16>(v, f);
        uint32_t o[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            uint32_t h;
            asm("cvt.rn.satfinite.f16x2.f32 %0, %1, %2;" : "=r"(h) : "f"(f[2 * e + 1]), "f"(f[2 * e]));
            o[e] = h;
        }
        dst[i] = make_uint4(o[0], o[1], o[2], o[3]);
    }
}

// ---- host side ------------------------------------------------------------------------------

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

aq_status get_encode_fn(EncodeTiledFn* fn) {
    static std::mutex mu;
    static EncodeTiledFn cached = nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!cached) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                                             cudaEnableDefault, &q);
            e != cudaSuccess)
            return cuda_fail(e, "cudaGetDriverEntryPointByVersion");
        if (q != cudaDriverEntryPointSuccess || !p) return AQ_ERR_CUDA;
        cached = (EncodeTiledFn)p;
    }
    *fn = cached;
    return AQ_OK;
}

template <int BDT>
aq_status run_gemm(const Dims& d, int m, const void* planes, const void* books,
                   const void* scales, const void* x, int tokens, void* y, int y_dt, void* ws,
                   cudaStream_t st) {   // x: fp16 [tokens][in]
    EncodeTiledFn encode;
    if (aq_status e = get_encode_fn(&encode); e != AQ_OK) return e;
    CUtensorMap map;
    std::memset(&map, 0, sizeof(map));
    const cuuint64_t dims[2] = {(cuuint64_t)d.in, (cuuint64_t)tokens};
    const cuuint64_t strides[1] = {(cuuint64_t)d.in * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)(2 * kBM)};
    const cuuint32_t estr[2] = {1, 1};
    if (encode(&map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(x), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return AQ_ERR_CUDA;

    auto kern = gemm_kernel<BDT>;
    static std::mutex mu;
    static bool attr_done[64] = {};
    int dev = 0;
    if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    {
        std::lock_guard<std::mutex> lock(mu);
        if (dev >= 0 && dev < 64 && !attr_done[dev]) {
            if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kGemmSmem);
                e != cudaSuccess)
                return cuda_fail(e, "cudaFuncSetAttribute");
            if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout,
                                                     (int)cudaSharedmemCarveoutMaxShared);
                e != cudaSuccess)
                return cuda_fail(e, "cudaFuncSetAttribute");
            attr_done[dev] = true;
        }
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((d.out + kBN - 1) / kBN, (tokens + kMT * kBM - 1) / (kMT * kBM));
    cfg.blockDim = dim3(kGemmThreads);
    cfg.dynamicSmemBytes = kGemmSmem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cuda_ok(cudaLaunchKernelEx(&cfg, kern, map, (const uint8_t*)planes,
                                      (const uint16_t*)books, (const uint16_t*)scales, y, y_dt,
                                      d.scale_dt, (unsigned int*)ws, m, tokens, d.out, d.in, d.ng,
                                      d.rows_pad, d.plane_bytes),
                   "cudaLaunchKernelEx");
}

}  // namespace

aq_status launch_gemm(const Dims& d, int m, const void* planes, const void* books,
                      const void* scales, const void* x, int x_dt, int tokens, void* y, int y_dt,
                      void* ws, cudaStream_t st) {
    if (d.out == 0 || tokens == 0) return AQ_OK;
    if (d.B != 8 || m > kGemmMaxM) return AQ_ERR_UNSUPPORTED;
    const void* xh = x;
    if (x_dt == AQ_BF16) {
        // fp16 copy of the activations after the status word of the workspace
        void* dst = (char*)ws + kWsStatusBytes;
        const size_t n8 = (size_t)tokens * d.in / 8;
        DeviceInfo di;
        if (aq_status e = device_info(&di); e != AQ_OK) return e;
        const size_t want = (n8 + 255) / 256;
        const int blocks = (int)(want < (size_t)di.sms * 8 ? want : (size_t)di.sms * 8);
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(blocks);
        cfg.blockDim = dim3(256);
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (aq_status e = cuda_ok(cudaLaunchKernelEx(&cfg, bf16_to_f16_kernel, (const uint4*)x,
                                                     (uint4*)dst, n8),
                                  "cudaLaunchKernelEx");
            e != AQ_OK)
            return e;
        xh = dst;
    }
    return d.book_dt == AQ_BF16
               ? run_gemm<AQ_BF16>(d, m, planes, books, scales, xh, tokens, y, y_dt, ws, st)
               : run_gemm<AQ_F16>(d, m, planes, books, scales, xh, tokens, y, y_dt, ws, st);
}

}  // namespace aq
