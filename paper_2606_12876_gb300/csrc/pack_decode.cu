// aq_pack and aq_decode kernels.
//
// Packing turns the natural code tensor b (Sec. 3.2: one B-bit index per output row, group
// of 8 inputs and codebook) into codebook-major planes so that a prefix of m codebooks
// (Sec. 5) is a prefix of the buffer. Decoding writes the partial reconstruction W_m densely.
#include <mutex>

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

constexpr int kDecMaxWarps = 16;

// Decode: one CTA per SM (or as many as fit) walks the (32-row block, slice) items, a warp at a
// time (grid-stride; row blocks fastest, so a warp's code loads are one contiguous 1 KiB per
// plane for 8-bit codes and its stores 512 contiguous bytes per row). For B <= 8 the CTA stages
// the first m codebooks once, in 2^cshift interleaved copies (book_copies_log2: with eight the
// codeword gathers are free of bank conflicts); 16-bit codebooks are read through L2. Each
// lane copies its row's codes of the m planes into the warp's staging buffer (cp.async), the
// next item's while the current one is decoded; then lane L walks the rows, four at a time,
// producing group s*32 + L of each.
// Bit-exact contract (aq.h): fp32 adds in book order from +0.0f, one fp32 multiply by the
// scale, one round-to-nearest-even to the book type.
template <int B, int BDT, int SDT>
__global__ void __launch_bounds__(kDecMaxWarps * 32, 1)
decode_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
              const uint16_t* __restrict__ scales, uint16_t* __restrict__ w, int m, int cshift,
              int out, int in, int ng, int rows_pad, int RBc, int S, size_t plane_bytes) {
    constexpr int UNIT = unit_bytes(B);              // bytes of one (row, slice) unit
    constexpr bool STAGED = B <= 8;
    extern __shared__ __align__(16) unsigned char smem[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (int)(blockDim.x >> 5);
    const size_t books_bytes = STAGED ? ((size_t)m << B << cshift) * 16 : 0;   // [m][2^B][2^cshift]
    unsigned char* cbuf = smem + books_bytes + (size_t)warp * 2 * m * 32 * UNIT;   // [2][m][32][UNIT]
    const long long items = (long long)RBc * S;
    const long long stride = (long long)gridDim.x * nw;
    auto issue = [&](long long item, int buf) {   // the item's codes into buffer buf
        if (item < items) {
            const int s = (int)(item / RBc), rb = (int)(item - (long long)s * RBc);
            const size_t src = ((size_t)s * rows_pad + (size_t)rb * 32 + lane) * UNIT;
            unsigned char* dst = cbuf + ((size_t)buf * m * 32 + lane) * UNIT;
            for (int k = 0; k < m; ++k)
#pragma unroll
                for (int q = 0; q < UNIT / 16; ++q)
                    cp_async16(dst + (size_t)k * 32 * UNIT + q * 16, planes + k * plane_bytes + src + q * 16);
        }
        cp_async_commit();
    };
    long long item = (long long)blockIdx.x * nw + warp;
    issue(item, 0);   // the first codes travel while the books are staged
    if constexpr (STAGED) {
        uint4* dst = (uint4*)smem;
        for (int i = threadIdx.x; i < (m << B) << cshift; i += blockDim.x)
            dst[i] = __ldg((const uint4*)books + (i >> cshift));
    }
    __syncthreads();
    const uint32_t books_u = smem_u32(smem) + ((uint32_t)(lane & ((1 << cshift) - 1)) << 4);
    // lane L holds the scale of row 32 rb + L of an item; the next item's is requested one item
    // ahead, with its codes
    auto scale_of = [&](long long it) -> uint16_t {
        if (it >= items) return 0;
        const int row = (int)(it % RBc) * 32 + lane;
        return row < out ? scales[row] : (uint16_t)0;
    };
    uint16_t sc_next = scale_of(item);
    int buf = 0;
    for (; item < items; item += stride) {
        issue(item + stride, buf ^ 1);
        const float sc_l = bits_to_f32<SDT>(sc_next);
        sc_next = scale_of(item + stride);
        const int s = (int)(item / RBc), rb = (int)(item - (long long)s * RBc);
        const int g = s * 32 + lane;
        cp_async_wait<1>();      // this lane's copies of the current item landed
        __syncwarp();            // ... and every lane's
        const unsigned char* cb = cbuf + (size_t)buf * m * 32 * UNIT;
        {
            // every lane computes (padding groups beyond ng have code 0); lanes g < ng store
            for (int r0 = 0; r0 < 32 && rb * 32 + r0 < out; r0 += 4) {
                float acc[4][8];
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[i][e] = 0.0f;
                for (int k = 0; k < m; ++k) {
                    uint4 cw[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int r = r0 + i;
                        // position of group `lane` in row rb*32 + r
                        const uint32_t code = unit_code<B>(cb + ((size_t)k * 32 + r) * UNIT, (lane - r) & 31);
                        if constexpr (STAGED)
                            cw[i] = lds128(books_u + ((((uint32_t)k << B) + code) << (cshift + 4)));
                        else
                            cw[i] = __ldg((const uint4*)books + ((size_t)k << 16) + code);
                    }
#pragma unroll
                    for (int i = 0; i < 4; ++i) {   // exact widening, one fp32 rounding per add
                        add_widen2<BDT>(cw[i].x, acc[i][0], acc[i][1]);
                        add_widen2<BDT>(cw[i].y, acc[i][2], acc[i][3]);
                        add_widen2<BDT>(cw[i].z, acc[i][4], acc[i][5]);
                        add_widen2<BDT>(cw[i].w, acc[i][6], acc[i][7]);
                    }
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int o = rb * 32 + r0 + i;
                    const float sc = __shfl_sync(0xffffffffu, sc_l, r0 + i);
                    if (o < out && g < ng) {
                        // times the scale (a packed fma with -0.0 added: the rounded product,
                        // signed zeros included), then one rounding to the book type per value
                        uint32_t pk[4];
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const float2 v = ffma2(make_float2(acc[i][2 * j], acc[i][2 * j + 1]),
                                                   make_float2(sc, sc), make_float2(-0.0f, -0.0f));
                            pk[j] = round_pack2<BDT>(v.x, v.y);
                        }
                        *(uint4*)(w + (size_t)o * in + (size_t)g * 8) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                    }
                }
            }
        }
        __syncwarp();            // every lane has read the buffer before it is refilled
        buf ^= 1;
    }
    cp_async_wait<0>();
}

template <int B, int BDT, int SDT>
aq_status run_decode(const Dims& d, int m, const void* planes, const void* books,
                     const void* scales, void* w, cudaStream_t st) {
    auto kern = decode_kernel<B, BDT, SDT>;
    DeviceInfo di;
    if (aq_status e = device_info(&di); e != AQ_OK) return e;
    // the kernel's shared-memory limit raised once per device (the attribute is per kernel)
    static std::mutex mu;
    static int dyn_max[64] = {};
    int dev = 0;
    if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= 64) return AQ_ERR_UNSUPPORTED;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (dyn_max[dev] == 0) {
            cudaFuncAttributes fa;
            if (cudaError_t e = cudaFuncGetAttributes(&fa, kern); e != cudaSuccess)
                return cuda_fail(e, "cudaFuncGetAttributes");
            const int lim = di.smem_optin - (int)fa.sharedSizeBytes;
            if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, lim);
                e != cudaSuccess)
                return cuda_fail(e, "cudaFuncSetAttribute");
            dyn_max[dev] = lim;
        }
    }
    const int cshift = B <= 8 ? book_copies_log2(B, m) : 0;
    const size_t books_bytes = B <= 8 ? ((size_t)m << B << cshift) * 16 : 0;
    const size_t per_warp = (size_t)2 * m * 32 * unit_bytes(B);
    // warps per CTA: the choice (16, 12, 8, 6 or 4) with the most resident warps per SM (the
    // code buffers are per warp), found once per device and prefix
    static int choice[64][9][2] = {};   // [dev][m] -> {warps, CTAs per SM}
    int nw = 0, occ = 0;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (choice[dev][m][0] == 0) {
            int best_w = 0;
            for (int w : {16, 12, 8, 6, 4}) {
                const size_t sm_bytes = books_bytes + w * per_warp;
                if (sm_bytes > (size_t)dyn_max[dev]) continue;
                int o = 0;
                if (cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, kern, w * 32, sm_bytes);
                    e != cudaSuccess)
                    return cuda_fail(e, "cudaOccupancyMaxActiveBlocksPerMultiprocessor");
                if (o * w > best_w) {
                    best_w = o * w;
                    choice[dev][m][0] = w;
                    choice[dev][m][1] = o;
                }
            }
            if (best_w == 0) return AQ_ERR_UNSUPPORTED;
        }
        nw = choice[dev][m][0];
        occ = choice[dev][m][1];
    }
    const size_t smem = books_bytes + nw * per_warp;
    const long long items = (long long)d.RBc * d.S;
    long long grid = (long long)di.sms * occ;
    const long long need = (items + nw - 1) / nw;
    if (grid > need) grid = need;
    kern<<<(unsigned)grid, nw * 32, smem, st>>>((const uint8_t*)planes, (const uint16_t*)books,
                                                (const uint16_t*)scales, (uint16_t*)w, m, cshift, d.out,
                                                d.in, d.ng, d.rows_pad, d.RBc, d.S, d.plane_bytes);
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
