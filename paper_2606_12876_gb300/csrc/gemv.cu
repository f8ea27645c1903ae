// aq_gemv: y = x * W_m^T for 1..16 tokens, W_m the prefix-m additive reconstruction
// (Sec. 3.2 group sums, restricted to the first m codebooks as in Sec. 5; Y = W X of Sec. 2.2).
//
// Work split (split-K): the grid is (row chunks) x (slices of 32 groups = 256 inputs). Each
// CTA reads the first m code planes of its (slice, rows) region once, writes one fp32
// partial per (row, token), and the last CTA of a row chunk sums the slices in order, scales
// the row (R1: s[o] multiplies the codebook sum, so it factors out of the dot product) and
// stores y.
//
// Two kernels:
//  * gemv_lut (B = 8, one token, m <= 4). By linearity, x_g . (sum_k C_k[b_k]) =
//    sum_k T_k[g][b_k] with T_k[g][j] = x_g . C_k[j]. The CTA builds T for its 32 groups and
//    m books in shared memory (32 KiB per book), then every code byte costs one shared-memory
//    lookup and one fp32 add. Lane L owns row 32*rb+L; because each row's 32 codes are stored
//    rotated by the row index, at step p all 32 lanes look up 32 different groups, i.e. 32
//    different banks, so the lookups are conflict-free and no cross-lane reduction is needed.
//  * gemv_direct (any B, 1..16 tokens). Decode each group in fp32 (sum of m codewords), then
//    multiply by the tokens' 8 activations. Lane L owns row 32*rb+L and walks the 32 groups
//    of the slice in a common order, so the activation loads are warp-uniform broadcasts.
#include <mutex>

#include "aq_internal.cuh"

namespace aq {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

// ------------------------------------------------------------------ LUT kernel (B = 8, b = 1)

// Table layout: pairs of books share 256-byte rows, T[k/2][j][k%2][32 groups] (fp32), so the
// byte offset of entry (k, j, g) is (k/2)*65536 + j*256 + (k%2)*128 + g*4 and j*256 + g*4 is
// produced from a code byte by one prmt.
template <int MM, int BDT, int XDT, int SDT>
__global__ void __launch_bounds__(kThreads)
gemv_lut_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
                const uint16_t* __restrict__ x, const uint16_t* __restrict__ scales,
                float* __restrict__ partials, unsigned int* __restrict__ counters, void* y,
                int y_dt, int out, int ng, int rows_pad, int S, int RBc, int rb_per_chunk,
                size_t plane_bytes) {
    constexpr int NP = (MM + 1) / 2;
    extern __shared__ __align__(16) unsigned char smem[];
    unsigned char* T = smem;                                   // NP * 64 KiB
    float* Cf = (float*)(smem + NP * 65536);                   // [MM][256][8] fp32

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int s = blockIdx.y, chunk = blockIdx.x;

    // Stage the first MM codebooks as fp32.
    for (int i = tid; i < MM * 256; i += kThreads) {
        const uint4 v = __ldg((const uint4*)books + i);
        float f[8];
        unpack8<BDT>(v, f);
        float4* d = (float4*)(Cf + (size_t)i * 8);
        d[0] = make_float4(f[0], f[1], f[2], f[3]);
        d[1] = make_float4(f[4], f[5], f[6], f[7]);
    }
    // Activations of group s*32+lane (zero for padding groups).
    float xv[8];
    {
        const int g = s * 32 + lane;
        if (g < ng) {
            unpack8<XDT>(__ldg((const uint4*)x + g), xv);
        } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) xv[e] = 0.0f;
        }
    }
    __syncthreads();

    // T_k[j][lane] = x_{s*32+lane} . C_k[j]
    for (int j = warp; j < 256; j += kWarps) {
#pragma unroll
        for (int k = 0; k < MM; ++k) {
            const float4 c0 = *(const float4*)(Cf + ((size_t)k * 256 + j) * 8);
            const float4 c1 = *(const float4*)(Cf + ((size_t)k * 256 + j) * 8 + 4);
            float t = xv[0] * c0.x;
            t = fmaf(xv[1], c0.y, t);
            t = fmaf(xv[2], c0.z, t);
            t = fmaf(xv[3], c0.w, t);
            t = fmaf(xv[4], c1.x, t);
            t = fmaf(xv[5], c1.y, t);
            t = fmaf(xv[6], c1.z, t);
            t = fmaf(xv[7], c1.w, t);
            *(float*)(T + (k >> 1) * 65536 + j * 256 + (k & 1) * 128 + lane * 4) = t;
        }
    }
    __syncthreads();

    // goff[q] byte i = 4 * group-in-slice read at position 4q+i by this lane: (4q+i+lane) mod 32.
    uint32_t goff[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        uint32_t v = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i) v |= (uint32_t)(((4 * q + i + lane) & 31) * 4) << (8 * i);
        goff[q] = v;
    }

    const int rb0 = chunk * rb_per_chunk;
    const int rb1 = min(rb0 + rb_per_chunk, RBc);
    for (int rb = rb0 + warp; rb < rb1; rb += kWarps) {
        const int o = rb * 32 + lane;
        uint4 cw[MM][2];
#pragma unroll
        for (int k = 0; k < MM; ++k) {
            const uint8_t* src = planes + k * plane_bytes + ((size_t)s * rows_pad + o) * 32;
            cw[k][0] = ld_stream_v4(src);
            cw[k][1] = ld_stream_v4(src + 16);
        }
        float acc = 0.0f;
#pragma unroll
        for (int k = 0; k < MM; ++k) {
            const unsigned char* Tk = T + (k >> 1) * 65536 + (k & 1) * 128;
            const uint32_t wd[8] = {cw[k][0].x, cw[k][0].y, cw[k][0].z, cw[k][0].w,
                                    cw[k][1].x, cw[k][1].y, cw[k][1].z, cw[k][1].w};
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                // byte0 = goff byte i, byte1 = code byte i, bytes 2-3 = sign of goff byte (0)
                acc += *(const float*)(Tk + prmt(wd[q], goff[q], 0xCC04u));
                acc += *(const float*)(Tk + prmt(wd[q], goff[q], 0xDD15u));
                acc += *(const float*)(Tk + prmt(wd[q], goff[q], 0xEE26u));
                acc += *(const float*)(Tk + prmt(wd[q], goff[q], 0xFF37u));
            }
        }
        partials[(size_t)s * rows_pad + o] = acc;
    }
    splitk_finish<SDT>(counters, partials, scales, y, y_dt, out, rows_pad, S, 1, chunk,
                       rb0 * 32, rb1 * 32);
}

// ------------------------------------------------------------------ direct kernel (any B, b <= 16)

template <int NB, int B, int BDT, int SDT>
__global__ void __launch_bounds__(kThreads)
gemv_direct_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
                   const uint16_t* __restrict__ x, int x_dt, const uint16_t* __restrict__ scales,
                   float* __restrict__ partials, unsigned int* __restrict__ counters, void* y,
                   int y_dt, int m, int batch, int out, int in, int ng, int rows_pad, int S,
                   int RBc, int rb_per_chunk, size_t plane_bytes) {
    constexpr int ESZ = B / 8;
    constexpr int UNIT = 32 * ESZ;
    extern __shared__ __align__(16) unsigned char smem[];
    float* xs = (float*)smem;                                        // [NB][256]
    uint16_t* books_s = (uint16_t*)(smem + NB * 1024);               // B = 8: [m][256][8]
    const size_t books_bytes = (B == 8) ? (size_t)m * 4096 : 0;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    unsigned char* codes_s = smem + NB * 1024 + books_bytes + (size_t)warp * m * 32 * UNIT;
    const int s = blockIdx.y, chunk = blockIdx.x;

    for (int i = tid; i < NB * 256; i += kThreads) {
        const int t = i >> 8, c = i & 255;
        const int col = s * 256 + c;
        float v = 0.0f;
        if (t < batch && col < in) v = bits_to_f32_rt(x[(size_t)t * in + col], x_dt);
        xs[i] = v;
    }
    if constexpr (B == 8) {
        for (int i = tid; i < m * 256; i += kThreads)
            ((uint4*)books_s)[i] = __ldg((const uint4*)books + i);
    }
    __syncthreads();

    const int rb0 = chunk * rb_per_chunk;
    const int rb1 = min(rb0 + rb_per_chunk, RBc);
    for (int rb = rb0 + warp; rb < rb1; rb += kWarps) {
        const int o = rb * 32 + lane;
        for (int k = 0; k < m; ++k) {
            const uint4* src = (const uint4*)(planes + k * plane_bytes + ((size_t)s * rows_pad + o) * UNIT);
            uint4* dst = (uint4*)(codes_s + ((size_t)k * 32 + lane) * UNIT);
#pragma unroll
            for (int q = 0; q < UNIT / 16; ++q) dst[q] = ld_stream_v4(src + q);
        }
        __syncwarp();
        float acc[NB];
#pragma unroll
        for (int t = 0; t < NB; ++t) acc[t] = 0.0f;
        for (int gl = 0; gl < 32; ++gl) {
            const int p = (gl - lane) & 31;        // position of group gl in row o (o mod 32 = lane)
            float wv[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) wv[e] = 0.0f;
            for (int k = 0; k < m; ++k) {
                uint32_t code;
                if constexpr (B == 8) code = codes_s[((size_t)k * 32 + lane) * UNIT + p];
                else code = ((const uint16_t*)(codes_s + ((size_t)k * 32 + lane) * UNIT))[p];
                uint4 cwv;
                if constexpr (B == 8) cwv = ((const uint4*)books_s)[k * 256 + code];
                else cwv = __ldg((const uint4*)books + ((size_t)k << 16) + code);
                float c[8];
                unpack8<BDT>(cwv, c);
#pragma unroll
                for (int e = 0; e < 8; ++e) wv[e] += c[e];
            }
#pragma unroll
            for (int t = 0; t < NB; ++t) {
                const float4 x0 = *(const float4*)(xs + t * 256 + gl * 8);
                const float4 x1 = *(const float4*)(xs + t * 256 + gl * 8 + 4);
                float a = acc[t];
                a = fmaf(x0.x, wv[0], a);
                a = fmaf(x0.y, wv[1], a);
                a = fmaf(x0.z, wv[2], a);
                a = fmaf(x0.w, wv[3], a);
                a = fmaf(x1.x, wv[4], a);
                a = fmaf(x1.y, wv[5], a);
                a = fmaf(x1.z, wv[6], a);
                a = fmaf(x1.w, wv[7], a);
                acc[t] = a;
            }
        }
        __syncwarp();
#pragma unroll
        for (int t = 0; t < NB; ++t)
            if (t < batch) partials[((size_t)s * batch + t) * rows_pad + o] = acc[t];
    }
    splitk_finish<SDT>(counters, partials, scales, y, y_dt, out, rows_pad, S, batch, chunk,
                       rb0 * 32, rb1 * 32);
}

// ------------------------------------------------------------------ host side

struct Grid {
    int chunks, rb_per_chunk;
};

Grid plan_grid(const Dims& d, int sms, int ctas_per_sm) {
    const int target = sms * (ctas_per_sm > 0 ? ctas_per_sm : 1);
    int chunks = (target + d.S - 1) / d.S;
    if (chunks < 1) chunks = 1;
    if (chunks > d.RBc) chunks = d.RBc;
    const int rbpc = (d.RBc + chunks - 1) / chunks;
    return Grid{(d.RBc + rbpc - 1) / rbpc, rbpc};
}

// Raises the kernel's dynamic shared-memory limit and returns its occupancy. Both are cached
// per (kernel, device, slot), slot being the prefix m where the shared-memory size depends on
// it, so the CUDA attribute calls happen once, before any stream capture that later calls
// reuse.
struct PrepCache {
    std::mutex mu;
    int occ[64][9] = {};
};

template <typename K>
aq_status prepare(K kern, size_t smem, int slot, int* ctas_per_sm) {
    static PrepCache cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64 || slot < 0 || slot > 8)
        return AQ_ERR_CUDA;
    std::lock_guard<std::mutex> lock(cache.mu);
    if (cache.occ[dev][slot] > 0) {
        *ctas_per_sm = cache.occ[dev][slot];
        return AQ_OK;
    }
    DeviceInfo di;
    if (device_info(&di) != AQ_OK) return AQ_ERR_CUDA;
    cudaFuncAttributes fa;
    if (cudaFuncGetAttributes(&fa, kern) != cudaSuccess) return AQ_ERR_CUDA;
    const int dyn_max = di.smem_optin - (int)fa.sharedSizeBytes;
    if ((int)smem > dyn_max) return AQ_ERR_UNSUPPORTED;
    // Allow the largest size any slot of this kernel may need (the attribute is per kernel).
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn_max) !=
        cudaSuccess)
        return AQ_ERR_CUDA;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas_per_sm, kern, kThreads, smem) != cudaSuccess)
        return AQ_ERR_CUDA;
    if (*ctas_per_sm < 1) return AQ_ERR_UNSUPPORTED;
    cache.occ[dev][slot] = *ctas_per_sm;
    return AQ_OK;
}

template <int MM, int BDT, int XDT, int SDT>
aq_status run_lut(const Dims& d, const void* planes, const void* books, const void* scales,
                  const void* x, void* y, int y_dt, void* ws, cudaStream_t st) {
    DeviceInfo di;
    if (device_info(&di) != AQ_OK) return AQ_ERR_CUDA;
    const size_t smem = (size_t)((MM + 1) / 2) * 65536 + (size_t)MM * 8192;
    auto kern = gemv_lut_kernel<MM, BDT, XDT, SDT>;
    int occ = 0;
    if (aq_status e = prepare(kern, smem, 0, &occ); e != AQ_OK) return e;
    const Grid g = plan_grid(d, di.sms, occ);
    unsigned int* counters = (unsigned int*)((char*)ws + kWsStatusBytes);
    float* partials = (float*)((char*)ws + ws_partial_offset(d));
    kern<<<dim3(g.chunks, d.S), kThreads, smem, st>>>(
        (const uint8_t*)planes, (const uint16_t*)books, (const uint16_t*)x,
        (const uint16_t*)scales, partials, counters, y, y_dt, d.out, d.ng, d.rows_pad, d.S,
        d.RBc, g.rb_per_chunk, d.plane_bytes);
    return cudaGetLastError() == cudaSuccess ? AQ_OK : AQ_ERR_CUDA;
}

template <int NB, int B, int BDT, int SDT>
aq_status run_direct(const Dims& d, int m, const void* planes, const void* books,
                     const void* scales, const void* x, int x_dt, int batch, void* y, int y_dt,
                     void* ws, cudaStream_t st) {
    DeviceInfo di;
    if (device_info(&di) != AQ_OK) return AQ_ERR_CUDA;
    const size_t smem = (size_t)NB * 1024 + (B == 8 ? (size_t)m * 4096 : 0) +
                        (size_t)kWarps * m * 32 * 32 * (B / 8);
    auto kern = gemv_direct_kernel<NB, B, BDT, SDT>;
    int occ = 0;
    if (aq_status e = prepare(kern, smem, m, &occ); e != AQ_OK) return e;
    const Grid g = plan_grid(d, di.sms, occ);
    unsigned int* counters = (unsigned int*)((char*)ws + kWsStatusBytes);
    float* partials = (float*)((char*)ws + ws_partial_offset(d));
    kern<<<dim3(g.chunks, d.S), kThreads, smem, st>>>(
        (const uint8_t*)planes, (const uint16_t*)books, (const uint16_t*)x, x_dt,
        (const uint16_t*)scales, partials, counters, y, y_dt, m, batch, d.out, d.in, d.ng,
        d.rows_pad, d.S, d.RBc, g.rb_per_chunk, d.plane_bytes);
    return cudaGetLastError() == cudaSuccess ? AQ_OK : AQ_ERR_CUDA;
}

template <int BDT, int XDT, int SDT>
aq_status dispatch_lut(const Dims& d, int m, const void* planes, const void* books,
                       const void* scales, const void* x, void* y, int y_dt, void* ws,
                       cudaStream_t st) {
    switch (m) {
        case 1: return run_lut<1, BDT, XDT, SDT>(d, planes, books, scales, x, y, y_dt, ws, st);
        case 2: return run_lut<2, BDT, XDT, SDT>(d, planes, books, scales, x, y, y_dt, ws, st);
        case 3: return run_lut<3, BDT, XDT, SDT>(d, planes, books, scales, x, y, y_dt, ws, st);
        default: return run_lut<4, BDT, XDT, SDT>(d, planes, books, scales, x, y, y_dt, ws, st);
    }
}

template <int B, int BDT, int SDT>
aq_status dispatch_direct(const Dims& d, int m, const void* planes, const void* books,
                          const void* scales, const void* x, int x_dt, int batch, void* y,
                          int y_dt, void* ws, cudaStream_t st) {
    if (batch <= 1) return run_direct<1, B, BDT, SDT>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
    if (batch <= 2) return run_direct<2, B, BDT, SDT>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
    if (batch <= 4) return run_direct<4, B, BDT, SDT>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
    if (batch <= 8) return run_direct<8, B, BDT, SDT>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
    return run_direct<16, B, BDT, SDT>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
}

}  // namespace

aq_status launch_gemv(const Dims& d, int m, const void* planes, const void* books,
                      const void* scales, const void* x, int x_dt, int batch, void* y,
                      int y_dt, void* ws, cudaStream_t st) {
    if (d.out == 0 || batch == 0) return AQ_OK;
    const bool bb = d.book_dt == AQ_BF16, sb = d.scale_dt == AQ_BF16, xb = x_dt == AQ_BF16;
    if (d.B == 8 && batch == 1 && m <= 4) {
        const int key = bb * 4 + xb * 2 + sb;
        switch (key) {
            case 0: return dispatch_lut<AQ_F16, AQ_F16, AQ_F16>(d, m, planes, books, scales, x, y, y_dt, ws, st);
            case 1: return dispatch_lut<AQ_F16, AQ_F16, AQ_BF16>(d, m, planes, books, scales, x, y, y_dt, ws, st);
            case 2: return dispatch_lut<AQ_F16, AQ_BF16, AQ_F16>(d, m, planes, books, scales, x, y, y_dt, ws, st);
            case 3: return dispatch_lut<AQ_F16, AQ_BF16, AQ_BF16>(d, m, planes, books, scales, x, y, y_dt, ws, st);
            case 4: return dispatch_lut<AQ_BF16, AQ_F16, AQ_F16>(d, m, planes, books, scales, x, y, y_dt, ws, st);
            case 5: return dispatch_lut<AQ_BF16, AQ_F16, AQ_BF16>(d, m, planes, books, scales, x, y, y_dt, ws, st);
            case 6: return dispatch_lut<AQ_BF16, AQ_BF16, AQ_F16>(d, m, planes, books, scales, x, y, y_dt, ws, st);
            default: return dispatch_lut<AQ_BF16, AQ_BF16, AQ_BF16>(d, m, planes, books, scales, x, y, y_dt, ws, st);
        }
    }
    const int key = (d.B == 16) * 4 + bb * 2 + sb;
    switch (key) {
        case 0: return dispatch_direct<8, AQ_F16, AQ_F16>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
        case 1: return dispatch_direct<8, AQ_F16, AQ_BF16>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
        case 2: return dispatch_direct<8, AQ_BF16, AQ_F16>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
        case 3: return dispatch_direct<8, AQ_BF16, AQ_BF16>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
        case 4: return dispatch_direct<16, AQ_F16, AQ_F16>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
        case 5: return dispatch_direct<16, AQ_F16, AQ_BF16>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
        case 6: return dispatch_direct<16, AQ_BF16, AQ_F16>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
        default: return dispatch_direct<16, AQ_BF16, AQ_BF16>(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
    }
}

}  // namespace aq
