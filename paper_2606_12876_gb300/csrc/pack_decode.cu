// aq_pack and aq_decode kernels.
//
// Packing turns the natural code tensor b (Sec. 3.2: one B-bit index per output row, group
// of 8 inputs and codebook) into codebook-major planes so that a prefix of m codebooks
// (Sec. 5) is a prefix of the buffer. Decoding writes the partial reconstruction W_m densely.
#include "aq_internal.cuh"

namespace aq {
namespace {

// One thread per packed code. Output index = ((k*S + s)*rows_pad + o)*32 + p.
template <typename CT>
__global__ void pack_kernel(const CT* __restrict__ codes, CT* __restrict__ planes, int out,
                            int ng, int M, int rows_pad, int S, size_t total) {
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int p = (int)(idx & 31);
        size_t rest = idx >> 5;
        const int o = (int)(rest % rows_pad);
        rest /= rows_pad;
        const int s = (int)(rest % S);
        const int k = (int)(rest / S);
        const int g = s * 32 + ((p + o) & 31);
        CT v = 0;
        if (o < out && g < ng) v = codes[((size_t)o * ng + g) * M + k];
        planes[idx] = v;
    }
}

// 4-bit codes: one thread per packed byte (positions 2b and 2b + 1 of a unit). Output byte
// index = ((k*S + s)*rows_pad + o)*16 + b; even positions in the low four bits.
__global__ void pack4_kernel(const uint8_t* __restrict__ codes, uint8_t* __restrict__ planes,
                             int out, int ng, int M, int rows_pad, int S, size_t total) {
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int b = (int)(idx & 15);
        size_t rest = idx >> 4;
        const int o = (int)(rest % rows_pad);
        rest /= rows_pad;
        const int s = (int)(rest % S);
        const int k = (int)(rest / S);
        uint32_t v = 0;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int g = s * 32 + ((2 * b + h + o) & 31);
            if (o < out && g < ng) v |= ((uint32_t)codes[((size_t)o * ng + g) * M + k] & 15u) << (4 * h);
        }
        planes[idx] = (uint8_t)v;
    }
}

constexpr int kDecWarps = 8;

// Decode: each warp owns one 32-row block of one slice. Lane L stages its own row's codes
// for the m planes in shared memory, then the warp walks the 32 rows with lane L producing
// group s*32+L of that row, so each output row segment is written as 512 contiguous bytes.
// Bit-exact contract (aq.h): fp32 adds in book order from +0.0f, one fp32 multiply by the
// scale, one round-to-nearest-even to the book type.
template <int B, int BDT, int SDT>
__global__ void __launch_bounds__(kDecWarps * 32)
decode_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
              const uint16_t* __restrict__ scales, uint16_t* __restrict__ w, int m, int out,
              int in, int ng, int rows_pad, int RBc, size_t plane_bytes) {
    constexpr int UNIT = unit_bytes(B);              // bytes of one (row, slice) unit
    extern __shared__ __align__(16) unsigned char smem[];
    uint16_t* books_s = (uint16_t*)smem;             // B <= 8: [m][2^B][8]
    const size_t books_bytes = staged_books_bytes(B, m);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    unsigned char* codes_s = smem + books_bytes + (size_t)warp * m * 32 * UNIT;

    if constexpr (B <= 8) {
        const uint4* src = (const uint4*)books;
        uint4* dst = (uint4*)books_s;
        for (int i = threadIdx.x; i < (m << B); i += blockDim.x) dst[i] = src[i];
    }
    const int s = blockIdx.y;
    const int rb = blockIdx.x * kDecWarps + warp;
    const bool active = rb < RBc;
    if (active) {
        const int o = rb * 32 + lane;
        for (int k = 0; k < m; ++k) {
            const uint4* src =
                (const uint4*)(planes + k * plane_bytes + ((size_t)s * rows_pad + o) * UNIT);
            uint4* dst = (uint4*)(codes_s + ((size_t)k * 32 + lane) * UNIT);
#pragma unroll
            for (int q = 0; q < UNIT / 16; ++q) dst[q] = ld_stream_v4(src + q);
        }
    }
    __syncthreads();
    if (!active) return;

    const int g = s * 32 + lane;
    for (int r = 0; r < 32; ++r) {
        const int o = rb * 32 + r;
        if (o >= out) break;
        const float sc = bits_to_f32<SDT>(scales[o]);
        const int p = (lane - r) & 31;               // position of group `lane` in row o
        float acc[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = 0.0f;
        for (int k = 0; k < m; ++k) {
            const uint32_t code = unit_code<B>(codes_s + ((size_t)k * 32 + r) * UNIT, p);
            uint4 cw;
            if constexpr (B <= 8) cw = ((const uint4*)books_s)[(k << B) + code];
            else cw = __ldg((const uint4*)books + ((size_t)k << 16) + code);
            float c[8];
            unpack8<BDT>(cw, c);
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[e] = __fadd_rn(acc[e], c[e]);
        }
        if (g < ng) {
            uint32_t pk[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint32_t lo = f32_to_bits<BDT>(__fmul_rn(acc[2 * i], sc));
                const uint32_t hi = f32_to_bits<BDT>(__fmul_rn(acc[2 * i + 1], sc));
                pk[i] = lo | (hi << 16);
            }
            *(uint4*)(w + (size_t)o * in + (size_t)g * 8) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        }
    }
}

template <int B, int BDT, int SDT>
aq_status run_decode(const Dims& d, int m, const void* planes, const void* books,
                     const void* scales, void* w, cudaStream_t st) {
    const size_t smem = staged_books_bytes(B, m) + (size_t)kDecWarps * m * 32 * unit_bytes(B);
    auto kern = decode_kernel<B, BDT, SDT>;
    if (smem > 48 * 1024)
        if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)smem);
            e != cudaSuccess)
            return cuda_fail(e, "cudaFuncSetAttribute");
    dim3 grid((d.RBc + kDecWarps - 1) / kDecWarps, d.S);
    kern<<<grid, kDecWarps * 32, smem, st>>>((const uint8_t*)planes, (const uint16_t*)books,
                                             (const uint16_t*)scales, (uint16_t*)w, m, d.out,
                                             d.in, d.ng, d.rows_pad, d.RBc, d.plane_bytes);
    return cuda_ok(cudaGetLastError(), "kernel launch");
}

}  // namespace

namespace {

// Self-test of the bounded waits: thread 0 waits, through the same bounded wait the compute
// kernels use, on a shared-memory mbarrier that nothing arrives at; when the wait gives up it
// records AQ_ERR_TIMEOUT in the status word and the kernel returns.
__global__ void selftest_wait_kernel(unsigned int* status) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_fence_init();
    }
    __syncthreads();
    if (threadIdx.x == 0 && !mbar_wait(&bar, 0)) record_status(status, AQ_ERR_TIMEOUT);
}

}  // namespace

aq_status launch_selftest_wait(unsigned int* status, cudaStream_t st) {
    selftest_wait_kernel<<<1, 32, 0, st>>>(status);
    return cuda_ok(cudaGetLastError(), "kernel launch");
}

namespace {

// Read probe: the launch shape of the one-token GEMV (one CTA per SM, sixteen warps,
// programmatic dependent launch, source requested before the grid wait) doing nothing but
// reading. CTA b takes 1 KiB chunks [c0, c1); warp w takes chunks c0 + w, c0 + w + 16, ...,
// four in flight; lane L reads bytes 16 L and 512 + 16 L of a chunk (each load instruction
// covers 512 contiguous bytes). The 32-bit words are XOR-folded, and each CTA XORs its fold
// into *sink once. A tail of bytes % 1024 is read by CTA 0, 16 bytes per thread.
constexpr int kReadWarps = 16, kReadDepth = 4;

__global__ void __launch_bounds__(kReadWarps * 32, 1)
selftest_read_kernel(const uint8_t* __restrict__ src, size_t chunks, size_t tail, int q, int r,
                     unsigned int* sink) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, b = blockIdx.x;
    const size_t c0 = (size_t)b * q + min(b, r), c1 = c0 + q + (b < r ? 1 : 0);
    uint4 v[kReadDepth][2];
    size_t c = c0 + warp;
#pragma unroll
    for (int d = 0; d < kReadDepth; ++d) {
        const size_t cd = c + (size_t)d * kReadWarps;
        v[d][0] = v[d][1] = make_uint4(0u, 0u, 0u, 0u);
        if (cd < c1) {
            v[d][0] = ld_stream_v4(src + cd * 1024 + lane * 16);
            v[d][1] = ld_stream_v4(src + cd * 1024 + 512 + lane * 16);
        }
    }
    pdl_wait();
    pdl_launch_dependents();
    uint32_t acc = 0;
    for (; c < c1; c += (size_t)kReadDepth * kReadWarps) {
#pragma unroll
        for (int d = 0; d < kReadDepth; ++d) {
            acc ^= v[d][0].x ^ v[d][0].y ^ v[d][0].z ^ v[d][0].w ^ v[d][1].x ^ v[d][1].y ^
                   v[d][1].z ^ v[d][1].w;
            v[d][0] = v[d][1] = make_uint4(0u, 0u, 0u, 0u);
            const size_t cn = c + (size_t)(d + kReadDepth) * kReadWarps;
            if (cn < c1) {
                v[d][0] = ld_stream_v4(src + cn * 1024 + lane * 16);
                v[d][1] = ld_stream_v4(src + cn * 1024 + 512 + lane * 16);
            }
        }
    }
    if (b == 0)
        for (size_t i = (size_t)threadIdx.x * 16; i < tail; i += (size_t)kReadWarps * 32 * 16) {
            const uint4 t = ld_stream_v4(src + chunks * 1024 + i);
            acc ^= t.x ^ t.y ^ t.z ^ t.w;
        }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc ^= __shfl_xor_sync(0xffffffffu, acc, o);
    __shared__ uint32_t red[kReadWarps];
    if (lane == 0) red[warp] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t f = 0;
        for (int w = 0; w < kReadWarps; ++w) f ^= red[w];
        atomicXor(sink, f);
    }
}

}  // namespace

aq_status launch_selftest_read(const void* src, size_t bytes, unsigned int* sink, cudaStream_t st) {
    DeviceInfo di;
    if (aq_status e = device_info(&di); e != AQ_OK) return e;
    const size_t chunks = bytes / 1024, tail = bytes % 1024;
    const size_t grid = chunks < (size_t)di.sms ? (chunks > 0 ? chunks : 1) : (size_t)di.sms;
    const int q = (int)(chunks / grid), r = (int)(chunks % grid);
    if (chunks / grid > 0x7fffffffULL) return AQ_ERR_UNSUPPORTED;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kReadWarps * 32);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cuda_ok(cudaLaunchKernelEx(&cfg, selftest_read_kernel, (const uint8_t*)src, chunks, tail,
                                      q, r, sink),
                   "cudaLaunchKernelEx");
}

aq_status launch_pack(const Dims& d, const void* codes, void* planes, cudaStream_t st) {
    const size_t total = (size_t)d.M * d.plane_elems;
    if (total == 0) return AQ_OK;
    const int threads = 256;
    const size_t want = (total + threads - 1) / threads;
    const int blocks = (int)(want < 65535 * 16 ? want : 65535 * 16);
    if (d.B == 4) {
        const size_t bytes = total / 2;
        const size_t want4 = (bytes + threads - 1) / threads;
        const int blocks4 = (int)(want4 < 65535 * 16 ? want4 : 65535 * 16);
        pack4_kernel<<<blocks4, threads, 0, st>>>((const uint8_t*)codes, (uint8_t*)planes, d.out,
                                                  d.ng, d.M, d.rows_pad, d.S, bytes);
    } else if (d.esz == 1)
        pack_kernel<uint8_t><<<blocks, threads, 0, st>>>((const uint8_t*)codes, (uint8_t*)planes,
                                                         d.out, d.ng, d.M, d.rows_pad, d.S, total);
    else
        pack_kernel<uint16_t><<<blocks, threads, 0, st>>>((const uint16_t*)codes,
                                                          (uint16_t*)planes, d.out, d.ng, d.M,
                                                          d.rows_pad, d.S, total);
    return cuda_ok(cudaGetLastError(), "kernel launch");
}

aq_status launch_decode(const Dims& d, int m, const void* planes, const void* books,
                        const void* scales, void* w, cudaStream_t st) {
    if (d.out == 0) return AQ_OK;
    const int key = (d.B == 16) * 4 + (d.book_dt == AQ_BF16) * 2 + (d.scale_dt == AQ_BF16);
    if (d.B == 4) {
        switch (key) {
            case 0: return run_decode<4, AQ_F16, AQ_F16>(d, m, planes, books, scales, w, st);
            case 1: return run_decode<4, AQ_F16, AQ_BF16>(d, m, planes, books, scales, w, st);
            case 2: return run_decode<4, AQ_BF16, AQ_F16>(d, m, planes, books, scales, w, st);
            default: return run_decode<4, AQ_BF16, AQ_BF16>(d, m, planes, books, scales, w, st);
        }
    }
    switch (key) {
        case 0: return run_decode<8, AQ_F16, AQ_F16>(d, m, planes, books, scales, w, st);
        case 1: return run_decode<8, AQ_F16, AQ_BF16>(d, m, planes, books, scales, w, st);
        case 2: return run_decode<8, AQ_BF16, AQ_F16>(d, m, planes, books, scales, w, st);
        case 3: return run_decode<8, AQ_BF16, AQ_BF16>(d, m, planes, books, scales, w, st);
        case 4: return run_decode<16, AQ_F16, AQ_F16>(d, m, planes, books, scales, w, st);
        case 5: return run_decode<16, AQ_F16, AQ_BF16>(d, m, planes, books, scales, w, st);
        case 6: return run_decode<16, AQ_BF16, AQ_F16>(d, m, planes, books, scales, w, st);
        default: return run_decode<16, AQ_BF16, AQ_BF16>(d, m, planes, books, scales, w, st);
    }
}

}  // namespace aq
