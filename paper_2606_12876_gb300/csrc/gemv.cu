// aq_gemv: y = x * W_m^T for 1..16 tokens, W_m the prefix-m additive reconstruction
// (Sec. 3.2 group sums, restricted to the first m codebooks as in Sec. 5; Y = W X of Sec. 2.2).
//
// Work split (split-K): the input dimension is cut into slices of 32 groups (256 inputs).
// A work item is (slice, 32-row block). Each item reads the first m code planes of its rows
// once and writes one fp32 partial per (row, token). A second, small kernel (splitk_reduce,
// launched right behind with programmatic dependent launch, so its CTAs are already resident
// when the product finishes) sums each row's partials in slice order (deterministic), scales
// the row and stores y, with the rows spread evenly over the GPU.
//
// Two product kernels:
//  * gemv_lut (B = 8, one token, m <= 4). By linearity, x_g . (sum_k C_k[b_k]) =
//    sum_k T_k[g][b_k] with T_k[g][j] = x_g . C_k[j]. A persistent CTA (one per SM) walks a
//    contiguous range of work items; for each slice it builds T for the 32 groups and m books
//    in shared memory (32 KiB per book), then every code byte costs one shared-memory lookup
//    and one fp32 add. Lane L owns row 32*rb+L; because each row's 32 codes are stored
//    rotated by the row index, at step p all 32 lanes look up 32 different groups, i.e. 32
//    different banks, so the lookups are conflict-free and no cross-lane reduction is needed.
//    One producer warp streams the code planes into a shared-memory ring with TMA bulk copies
//    (the CTA's rows of a slice are contiguous in every plane), overlapping HBM reads with
//    the table build and the lookups of the eight consumer warps.
//  * gemv_direct (any B, 1..16 tokens). Decode each group in fp32 (sum of m codewords), then
//    multiply by the tokens' 8 activations. Lane L owns row 32*rb+L and walks the 32 groups
//    of the slice in a common order, so the activation loads are warp-uniform broadcasts.
#include <map>
#include <mutex>
#include <tuple>

#include "aq_internal.cuh"

namespace aq {
namespace {

// ------------------------------------------------------------------ LUT kernel (B = 8, b = 1)

constexpr int kCons = 16;                         // consumer warps (one 32-row block each per stage)
constexpr int kLutThreads = (kCons + 1) * 32;     // + one producer warp
constexpr int kStageRb = 16;                      // 32-row blocks per stage: a 16 KiB plane copy
constexpr int kSlot = kStageRb * 1024;            // one ring slot = one plane of one stage
constexpr int kSlots = 8;                         // largest ring depth (128 KiB)
constexpr int kXSlices = 8;                       // activation slices staged up front
constexpr int kTBytes = 65536;                    // table of one book pair
constexpr int kLutMaxM = 8;

// Shared memory: [T 64 KiB][codebooks m x 4 KiB][activations 8 x 512 B][ring][barriers]
inline size_t lut_smem_bytes(int m, int slots) {
    return (size_t)kTBytes + (size_t)m * 4096 + kXSlices * 512 + (size_t)slots * kSlot +
           2 * kSlots * 8;
}

// The m books are processed in passes of at most two (pass p: books 2p, 2p+1), so the table
// never exceeds 64 KiB: T[j][k%2][32 groups] (fp32), entry (k, j, g) at byte
// j*256 + (k%2)*128 + g*4; j*256 + g*4 is produced from a code byte by one prmt.
//
// A CTA owns the items [i0, i1) (item = slice * RBc + 32-row block). In every pass it walks
// them in stages of up to 16 items that never cross a slice. For each stage and each book of
// the pass the producer warp copies the stage's rows of that book's plane into one ring slot
// with a TMA bulk copy (16 KiB; the CTA's rows of a slice are contiguous in every plane), and
// consumer warp w looks up item w of the stage. A row's sum over the pass's books stays in a
// register; pass 0 stores it as the fp32 partial and later passes add to it. The codebooks
// and the activations of the CTA's first slices are requested before any code.
template <int BDT, int XDT, int SDT>
__global__ void __launch_bounds__(kLutThreads, 1)
gemv_lut_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
                const uint16_t* __restrict__ x, float* __restrict__ partials, unsigned int* __restrict__ status, int m, int in,
                int ng, int rows_pad, int RBc, int S, int total_items, size_t plane_bytes,
                int nslots, int cps, int static_weights) {
    extern __shared__ __align__(128) unsigned char smem[];
    unsigned char* T = smem;
    uint4* Cb = (uint4*)(smem + kTBytes);                          // [m][256] codewords
    unsigned char* xs = smem + kTBytes + (size_t)m * 4096;         // [kXSlices][256] activations
    unsigned char* ring = xs + kXSlices * 512;                     // nslots x 16 KiB
    uint64_t* full = (uint64_t*)(ring + (size_t)nslots * kSlot);
    uint64_t* empty = full + kSlots;
    __shared__ volatile int s_abort;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // Item range of this CTA: slice-aligned (cps CTAs per slice) or balanced over the grid.
    // Item indices fit in 32 bits (checked by the host); the per-stage bookkeeping below is
    // incremental, without divisions (an integer division is a long instruction sequence).
    int i0, i1;
    if (cps > 0) {
        const int s = blockIdx.x / cps, c = blockIdx.x % cps;
        i0 = s * RBc + c * RBc / cps;
        i1 = s * RBc + (c + 1) * RBc / cps;
    } else {
        i0 = (int)((long long)blockIdx.x * total_items / gridDim.x);
        i1 = (int)((long long)(blockIdx.x + 1) * total_items / gridDim.x);
    }
    const int s_first = i0 / RBc, rb_first = i0 - s_first * RBc;
    // A walk over the CTA's items in stages: up to kStageRb items, never crossing a slice.
    struct Walk {
        int it, s, rb, n;
    };
    auto walk_start = [&]() {
        Walk w{i0, s_first, rb_first, 0};
        w.n = min(min(kStageRb, RBc - w.rb), i1 - w.it);
        return w;
    };
    auto walk_next = [&](Walk& w) {
        w.it += w.n;
        w.rb += w.n;
        if (w.rb == RBc) {
            w.rb = 0;
            ++w.s;
        }
        w.n = min(min(kStageRb, RBc - w.rb), i1 - w.it);
    };
    const int npass = (m + 1) / 2;

    // Producer state (warp kCons, lane 0): the next copy is book 2*p_pass + p_k of stage p_w,
    // into ring slot p_slot (use parity p_phase); p_q copies issued so far.
    int p_q = 0, p_slot = 0, p_pass = 0, p_k = 0;
    uint32_t p_phase = 0;
    Walk p_w = walk_start();
    if (i0 >= i1) p_pass = npass;
    auto issue_next = [&]() {
        const int mp = min(2, m - 2 * p_pass);
        const size_t src = ((size_t)p_w.s * rows_pad + (size_t)p_w.rb * 32) * 32;
        mbar_arrive_expect_tx(&full[p_slot], (uint32_t)(p_w.n * 1024));
        bulk_g2s(ring + (size_t)p_slot * kSlot,
                 planes + (size_t)(2 * p_pass + p_k) * plane_bytes + src,
                 (uint32_t)(p_w.n * 1024), &full[p_slot]);
        ++p_q;
        if (++p_slot == nslots) {
            p_slot = 0;
            p_phase ^= 1u;
        }
        if (++p_k == mp) {
            p_k = 0;
            walk_next(p_w);
            if (p_w.it >= i1) {
                ++p_pass;
                p_w = walk_start();
            }
        }
    };
    if (tid == 0) {
        for (int d = 0; d < nslots; ++d) {
            mbar_init(&full[d], 1);
            mbar_init(&empty[d], kCons);
        }
        mbar_fence_init();
        s_abort = 0;
    }
    __syncthreads();            // barriers initialised before the first copy
    // Codebooks and activations are requested first (into registers); the producer starts
    // its copies only after every thread has issued these loads (the barrier below).
    // (consumer threads only: they are the ones that store the codebooks below)
    uint4 cb_r[4];
    auto load_books = [&]() {
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int i = tid + r * kCons * 32;
            cb_r[r] = (tid < kCons * 32 && i < m * 256) ? __ldg((const uint4*)books + i)
                                                          : make_uint4(0u, 0u, 0u, 0u);
        }
    };
    if (static_weights) {
        // The weights are read-only while calls run (AQ_LAYOUT_STATIC_WEIGHTS): request the
        // codebooks before waiting for the preceding kernel.
        load_books();
        // The code planes are read-only too: fill the ring before waiting for the preceding
        // kernel, so the first stages overlap its tail.
        if (warp == kCons && lane == 0)
            while (p_q < nslots && p_pass < npass) issue_next();
    }
    pdl_wait();                 // inputs may come from the preceding kernel in the stream
    pdl_launch_dependents();    // the split-K reduction may become resident (it waits for us)
    if (!static_weights) load_books();
    uint2 x_r = make_uint2(0u, 0u);
    if (tid < kXSlices * 64) {
        const int col = (s_first + (tid >> 6)) * 256 + (tid & 63) * 4;
        if (col < in) x_r = __ldg((const uint2*)(x + col));
    }
    __syncthreads();

    // Stage sequence shared by the producer and the consumers: pass, then the walk's stages;
    // one ring slot per (stage, book of the pass).

    if (warp == kCons) {
        // ---- producer (lane 0 issues; the warp stays converged for the final barriers)
        if (lane == 0) {
            while (p_pass < npass) {
                if (s_abort) break;
                if (p_q >= nslots && !mbar_wait(&empty[p_slot], p_phase ^ 1u)) {
                    record_status(status, AQ_ERR_TIMEOUT);
                    s_abort = 1;
                    break;
                }
                issue_next();
            }
            // No copy may be in flight when the CTA exits (bounded wait on the last slots).
            for (int j = max(0, p_q - nslots); j < p_q; ++j) mbar_wait(&full[j % nslots], (j / nslots) & 1);
        }
        __syncwarp();
    } else {
        // ---- consumers
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int i = tid + r * kCons * 32;
            if (i < m * 256) Cb[i] = cb_r[r];
        }
        if (tid < kXSlices * 64) *(uint2*)(xs + (tid >> 6) * 512 + (tid & 63) * 8) = x_r;
        named_barrier(1, kCons * 32);   // staged codebooks and activations visible to all consumers

        // Each lane reads its row's 32 code bytes as two 16-byte halves; lanes 4-7 of every
        // eight read the second half first (no bank conflicts between the two reads).
        // goff[q] byte i = 4 * group at byte 4q+i of what this lane read, in its read order
        // (position p of row o holds group (p + o) mod 32).
        const int c0 = (lane >> 2) & 1;
        uint32_t goff[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            uint32_t v = 0;
#pragma unroll
            for (int i = 0; i < 4; ++i)
                v |= (uint32_t)((((4 * q + i + (c0 ? 16 : 0)) + lane) & 31) * 4) << (8 * i);
            goff[q] = v;
        }

        int slot = 0;
        uint32_t phase = 0;                     // parity of the slot's current use
        for (int pass = 0; pass < npass; ++pass) {
            const int mp = min(2, m - 2 * pass);
            int cur_s = -1;
            for (Walk w = walk_start(); w.it < i1; walk_next(w)) {
                const int n = w.n, s = w.s, rb = w.rb;
                if (s != cur_s) {
                    // Table of the pass's books for slice s. Lane L = 8*ph + gq computes groups
                    // 4gq..4gq+3 for codewords j = 16*warp + ph + 4i: one 16-byte codeword read
                    // serves four entries, stored as one 16-byte piece.
                    const int ph = lane >> 3, gq = lane & 7, sl = s - s_first;
                    float2 xv[4][4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int g = s * 32 + gq * 4 + u;
                        uint4 xr = make_uint4(0u, 0u, 0u, 0u);
                        if (sl < kXSlices) xr = *(const uint4*)(xs + sl * 512 + (gq * 4 + u) * 16);
                        else if (g < ng) xr = __ldg((const uint4*)x + g);
                        float f[8];
                        unpack8<XDT>(xr, f);
#pragma unroll
                        for (int e = 0; e < 4; ++e) xv[u][e] = make_float2(f[2 * e], f[2 * e + 1]);
                    }
                    named_barrier(1, kCons * 32);   // old table no longer read; Cb / xs staged
                    for (int k = 0; k < mp; ++k) {
                        const int kb = 2 * pass + k;
                        unsigned char* Tk = T + k * 128 + gq * 16;
                        uint4 cw[4];
#pragma unroll
                        for (int i = 0; i < 4; ++i) cw[i] = Cb[kb * 256 + warp * 16 + ph + 4 * i];
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            float c[8];
                            unpack8<BDT>(cw[i], c);
                            float r[4];
#pragma unroll
                            for (int u = 0; u < 4; ++u) {
                                float2 t = make_float2(xv[u][0].x * c[0], xv[u][0].y * c[1]);
                                t = ffma2(xv[u][1], make_float2(c[2], c[3]), t);
                                t = ffma2(xv[u][2], make_float2(c[4], c[5]), t);
                                t = ffma2(xv[u][3], make_float2(c[6], c[7]), t);
                                r[u] = t.x + t.y;
                            }
                            *(float4*)(Tk + (warp * 16 + ph + 4 * i) * 256) =
                                make_float4(r[0], r[1], r[2], r[3]);
                        }
                    }
                    named_barrier(1, kCons * 32);
                    cur_s = s;
                }
                float part = 0.0f;
                for (int k = 0; k < mp; ++k) {
                    bool ok = !s_abort;
                    if (ok && !mbar_wait(&full[slot], phase)) {
                        record_status(status, AQ_ERR_TIMEOUT);
                        s_abort = 1;
                        ok = false;
                    }
                    if (ok && warp < n) {
                        const unsigned char* row = ring + (size_t)slot * kSlot + warp * 1024 + lane * 32;
                        const uint4 a = *(const uint4*)(row + c0 * 16);
                        const uint4 b = *(const uint4*)(row + (c0 ^ 1) * 16);
                        const uint32_t wd[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
                        const uint32_t Tk = smem_u32(T) + k * 128;
                        float2 acc = make_float2(0.0f, 0.0f);
#pragma unroll
                        for (int qq = 0; qq < 8; ++qq) {
                            // byte0 = goff byte i, byte1 = code byte i, bytes 2-3 = sign of goff byte (0)
                            const uint32_t w = wd[qq], g = goff[qq];
                            const float v0 = lds_f32(Tk + prmt(w, g, 0xCC04u));
                            const float v1 = lds_f32(Tk + prmt(w, g, 0xDD15u));
                            const float v2 = lds_f32(Tk + prmt(w, g, 0xEE26u));
                            const float v3 = lds_f32(Tk + prmt(w, g, 0xFF37u));
                            acc = add2(acc, add2(make_float2(v0, v1), make_float2(v2, v3)));
                        }
                        part += acc.x + acc.y;
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&empty[slot]);
                    if (++slot == nslots) {
                        slot = 0;
                        phase ^= 1u;
                    }
                }
                if (!s_abort && warp < n) {
                    float* dst = partials + (size_t)s * rows_pad + (size_t)(rb + warp) * 32 + lane;
                    if (pass > 0) part += *dst;     // this thread wrote it in the previous pass
                    *dst = part;
                }
            }
        }
    }
}

// ------------------------------------------------------------------ direct kernel (any B, b <= 16)

template <int NB, int B, int BDT, int SDT>
__global__ void __launch_bounds__(256)
gemv_direct_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
                   const uint16_t* __restrict__ x, int x_dt, float* __restrict__ partials, int m, int batch, int in, int rows_pad, int RBc,
                   int rb_per_chunk, size_t plane_bytes) {
    constexpr int ESZ = B / 8;
    constexpr int UNIT = 32 * ESZ;
    constexpr int kWarps = 8;
    extern __shared__ __align__(128) unsigned char smem[];
    float* xs = (float*)smem;                                        // [NB][256]
    uint16_t* books_s = (uint16_t*)(smem + NB * 1024);               // B = 8: [m][256][8]
    const size_t books_bytes = (B == 8) ? (size_t)m * 4096 : 0;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    unsigned char* codes_s = smem + NB * 1024 + books_bytes + (size_t)warp * m * 32 * UNIT;
    const int s = blockIdx.y, chunk = blockIdx.x;

    pdl_wait();
    pdl_launch_dependents();
    for (int i = tid; i < NB * 256; i += 256) {
        const int t = i >> 8, c = i & 255;
        const int col = s * 256 + c;
        float v = 0.0f;
        if (t < batch && col < in) v = bits_to_f32_rt(x[(size_t)t * in + col], x_dt);
        xs[i] = v;
    }
    if constexpr (B == 8) {
        for (int i = tid; i < m * 256; i += 256)
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
}

// ------------------------------------------------------------------ split-K reduction

// y[t][r] = s[r] * sum over the S slices of partials[s][t][r], in slice order (R1: the row
// scale multiplies the codebook sum, so it factors out of the dot product). One thread per
// (row, token); all of a thread's loads are issued before the additions.
template <int SDT>
__global__ void __launch_bounds__(256)
splitk_reduce_kernel(const float* __restrict__ partials, const uint16_t* __restrict__ scales,
                     void* y, int y_dt, int out, int rows_pad, int S, int batch) {
    pdl_wait();                 // the product kernel's partials
    pdl_launch_dependents();
    const int r = blockIdx.x * blockDim.x + threadIdx.x, t = blockIdx.y;
    if (r >= out) return;
    const size_t stride = (size_t)batch * rows_pad;
    const float* p = partials + (size_t)t * rows_pad + r;
    float sum = 0.0f;
    int sl = 0;
    for (; sl + 16 <= S; sl += 16) {
        float v[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) v[q] = __ldcg(p + (size_t)(sl + q) * stride);
#pragma unroll
        for (int q = 0; q < 16; ++q) sum += v[q];
    }
    for (; sl < S; ++sl) sum += __ldcg(p + (size_t)sl * stride);
    const float v = sum * bits_to_f32<SDT>(scales[r]);
    const size_t yi = (size_t)t * out + r;
    if (y_dt == AQ_F32) ((float*)y)[yi] = v;
    else if (y_dt == AQ_F16) ((uint16_t*)y)[yi] = f32_to_bits<AQ_F16>(v);
    else ((uint16_t*)y)[yi] = f32_to_bits<AQ_BF16>(v);
}

// ------------------------------------------------------------------ host side

// Launch with the programmatic-stream-serialization attribute (PDL), so the kernel's CTAs may
// become resident while the preceding kernel in the stream drains; every kernel launched this
// way calls griddepcontrol.wait before it reads anything another kernel may have written.
template <typename... KArgs, typename... Args>
aq_status launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                     Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cuda_ok(cudaLaunchKernelEx(&cfg, kern, (KArgs)args...), "cudaLaunchKernelEx");
}

// Raises the kernel's dynamic shared-memory limit and returns its occupancy. Both are cached
// per (kernel, device, slot), slot being the prefix m where the shared-memory size depends on
// it, so the CUDA attribute calls happen once, before any stream capture that later calls
// reuse.
template <typename K>
aq_status prepare(K kern, size_t smem, int threads, int slot, int* ctas_per_sm) {
    static std::mutex mu;
    static std::map<std::tuple<const void*, int, int>, int> cache;
    int dev = 0;
    if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    const auto key = std::make_tuple((const void*)kern, dev, slot);
    std::lock_guard<std::mutex> lock(mu);
    if (auto it = cache.find(key); it != cache.end()) {
        *ctas_per_sm = it->second;
        return AQ_OK;
    }
    DeviceInfo di;
    if (aq_status e = device_info(&di); e != AQ_OK) return e;
    cudaFuncAttributes fa;
    if (cudaError_t e = cudaFuncGetAttributes(&fa, kern); e != cudaSuccess)
        return cuda_fail(e, "cudaFuncGetAttributes");
    const int dyn_max = di.smem_optin - (int)fa.sharedSizeBytes;
    if ((int)smem > dyn_max) return AQ_ERR_UNSUPPORTED;
    // Allow the largest size any slot of this kernel may need (the attribute is per kernel).
    if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             dyn_max);
        e != cudaSuccess)
        return cuda_fail(e, "cudaFuncSetAttribute");
    // Every kernel of the library asks for the same (largest) shared-memory carve-out, so
    // consecutive launches never force an SM to re-split its L1 / shared-memory storage.
    if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout,
                                             (int)cudaSharedmemCarveoutMaxShared);
        e != cudaSuccess)
        return cuda_fail(e, "cudaFuncSetAttribute");
    if (cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas_per_sm, kern, threads,
                                                                      smem);
        e != cudaSuccess)
        return cuda_fail(e, "cudaOccupancyMaxActiveBlocksPerMultiprocessor");
    if (*ctas_per_sm < 1) return AQ_ERR_UNSUPPORTED;
    cache[key] = *ctas_per_sm;
    return AQ_OK;
}

struct GemvArgs {
    const void *planes, *books, *scales, *x;
    int x_dt, batch;
    void* y;
    int y_dt;
    float* partials;
    unsigned int* status;
};

template <int BDT, int XDT, int SDT>
aq_status run_lut(const Dims& d, int m, const GemvArgs& a, cudaStream_t st) {
    DeviceInfo di;
    if (aq_status e = device_info(&di); e != AQ_OK) return e;
    auto kern = gemv_lut_kernel<BDT, XDT, SDT>;
    // As many 16 KiB ring slots as fit next to the table, codebooks and activations (<= 8).
    const size_t fixed = lut_smem_bytes(m, 0) + 8192;   // + static shared memory and slack
    int nslots = di.smem_optin > (int)fixed ? (int)((di.smem_optin - fixed) / kSlot) : 0;
    if (nslots > kSlots) nslots = kSlots;
    if (nslots < 2) return AQ_ERR_UNSUPPORTED;
    const size_t smem = lut_smem_bytes(m, nslots);
    int occ = 0;
    if (aq_status e = prepare(kern, smem, kLutThreads, m, &occ); e != AQ_OK) return e;
    const long long items = (long long)d.S * d.RBc;
    if (items > 0x7fffffffLL) return AQ_ERR_UNSUPPORTED;   // item indices are 32-bit
    // One CTA per SM. If whole slices per CTA keep at least 90% of the SMs busy, every CTA
    // gets a single slice (one table build per book); otherwise items are balanced evenly
    // and a CTA may span two slices.
    int cps = di.sms / d.S;
    if (cps > d.RBc) cps = d.RBc;
    int grid;
    if (cps >= 1 && (long long)cps * d.S * 10 >= (long long)di.sms * 9) {
        grid = cps * d.S;
    } else {
        cps = 0;
        grid = (int)(items < di.sms ? items : di.sms);
    }
    return launch_pdl(kern, dim3(grid), dim3(kLutThreads), smem, st, (const uint8_t*)a.planes,
                      (const uint16_t*)a.books, (const uint16_t*)a.x, a.partials, a.status, m,
                      d.in, d.ng,
                      d.rows_pad, d.RBc, d.S, items, d.plane_bytes, nslots, cps,
                      (d.flags & AQ_LAYOUT_STATIC_WEIGHTS) ? 1 : 0);
}

template <int NB, int B, int BDT, int SDT>
aq_status run_direct(const Dims& d, int m, const GemvArgs& a, cudaStream_t st) {
    DeviceInfo di;
    if (aq_status e = device_info(&di); e != AQ_OK) return e;
    const size_t smem = (size_t)NB * 1024 + (B == 8 ? (size_t)m * 4096 : 0) +
                        (size_t)8 * m * 32 * 32 * (B / 8);
    auto kern = gemv_direct_kernel<NB, B, BDT, SDT>;
    int occ = 0;
    if (aq_status e = prepare(kern, smem, 256, m, &occ); e != AQ_OK) return e;
    const int target = di.sms * occ;
    int chunks = (target + d.S - 1) / d.S;
    chunks = chunks < 1 ? 1 : (chunks > d.RBc ? d.RBc : chunks);
    const int rbpc = (d.RBc + chunks - 1) / chunks;
    chunks = (d.RBc + rbpc - 1) / rbpc;
    return launch_pdl(kern, dim3(chunks, d.S), dim3(256), smem, st, (const uint8_t*)a.planes,
                      (const uint16_t*)a.books, (const uint16_t*)a.x, a.x_dt,
                      a.partials, m, a.batch, d.in, d.rows_pad, d.RBc, rbpc, d.plane_bytes);
}

template <int B, int BDT, int SDT>
aq_status dispatch_direct(const Dims& d, int m, const GemvArgs& a, cudaStream_t st) {
    if (a.batch <= 1) return run_direct<1, B, BDT, SDT>(d, m, a, st);
    if (a.batch <= 2) return run_direct<2, B, BDT, SDT>(d, m, a, st);
    if (a.batch <= 4) return run_direct<4, B, BDT, SDT>(d, m, a, st);
    if (a.batch <= 8) return run_direct<8, B, BDT, SDT>(d, m, a, st);
    return run_direct<16, B, BDT, SDT>(d, m, a, st);
}

}  // namespace

// The product kernel of aq_gemv: fp32 partial sums per (slice, token, row) into the workspace.
static aq_status launch_product(const Dims& d, int m, const void* planes, const void* books,
                                const void* scales, const void* x, int x_dt, int batch, void* y,
                                int y_dt, void* ws, cudaStream_t st) {
    if (d.out == 0 || batch == 0) return AQ_OK;
    GemvArgs a{planes, books, scales, x, x_dt, batch, y, y_dt,
               (float*)((char*)ws + ws_partial_offset(d)), (unsigned int*)ws};
    const int bb = d.book_dt == AQ_BF16, xb = x_dt == AQ_BF16, sb = d.scale_dt == AQ_BF16;
    if (d.B == 8 && batch == 1 && m <= kLutMaxM) {
        switch (bb * 4 + xb * 2 + sb) {
            case 0: return run_lut<AQ_F16, AQ_F16, AQ_F16>(d, m, a, st);
            case 1: return run_lut<AQ_F16, AQ_F16, AQ_BF16>(d, m, a, st);
            case 2: return run_lut<AQ_F16, AQ_BF16, AQ_F16>(d, m, a, st);
            case 3: return run_lut<AQ_F16, AQ_BF16, AQ_BF16>(d, m, a, st);
            case 4: return run_lut<AQ_BF16, AQ_F16, AQ_F16>(d, m, a, st);
            case 5: return run_lut<AQ_BF16, AQ_F16, AQ_BF16>(d, m, a, st);
            case 6: return run_lut<AQ_BF16, AQ_BF16, AQ_F16>(d, m, a, st);
            default: return run_lut<AQ_BF16, AQ_BF16, AQ_BF16>(d, m, a, st);
        }
    }
    switch ((d.B == 16) * 4 + bb * 2 + sb) {
        case 0: return dispatch_direct<8, AQ_F16, AQ_F16>(d, m, a, st);
        case 1: return dispatch_direct<8, AQ_F16, AQ_BF16>(d, m, a, st);
        case 2: return dispatch_direct<8, AQ_BF16, AQ_F16>(d, m, a, st);
        case 3: return dispatch_direct<8, AQ_BF16, AQ_BF16>(d, m, a, st);
        case 4: return dispatch_direct<16, AQ_F16, AQ_F16>(d, m, a, st);
        case 5: return dispatch_direct<16, AQ_F16, AQ_BF16>(d, m, a, st);
        case 6: return dispatch_direct<16, AQ_BF16, AQ_F16>(d, m, a, st);
        default: return dispatch_direct<16, AQ_BF16, AQ_BF16>(d, m, a, st);
    }
}

template <int SDT>
static aq_status launch_reduce(const Dims& d, const GemvArgs& a, cudaStream_t st) {
    return launch_pdl(splitk_reduce_kernel<SDT>, dim3((d.out + 255) / 256, a.batch), dim3(256),
                      0, st, (const float*)a.partials, (const uint16_t*)a.scales, a.y, a.y_dt,
                      d.out, d.rows_pad, d.S, a.batch);
}

aq_status launch_gemv(const Dims& d, int m, const void* planes, const void* books,
                      const void* scales, const void* x, int x_dt, int batch, void* y,
                      int y_dt, void* ws, cudaStream_t st) {
    if (d.out == 0 || batch == 0) return AQ_OK;
    if (aq_status e = launch_product(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
        e != AQ_OK)
        return e;
    GemvArgs a{planes, books, scales, x, x_dt, batch, y, y_dt,
               (float*)((char*)ws + ws_partial_offset(d)), (unsigned int*)ws};
    return d.scale_dt == AQ_BF16 ? launch_reduce<AQ_BF16>(d, a, st) : launch_reduce<AQ_F16>(d, a, st);
}

}  // namespace aq
