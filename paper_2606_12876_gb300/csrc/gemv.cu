// aq_gemv: y = x * W_m^T for 1..16 tokens, W_m the prefix-m additive reconstruction
// (Sec. 3.2 group sums, restricted to the first m codebooks as in Sec. 5; Y = W X of Sec. 2.2).
//
// Work split (split-K): the input dimension is cut into slices of 32 groups (256 inputs).
// A work item is (slice, 32-row block) for the direct and tensor-core kernels and (slice,
// codebook, 32-row block) for the table-lookup kernel. Each item reads its code planes once
// and writes one fp32 partial per (row, token). A second, small kernel (splitk_reduce,
// launched right behind with programmatic dependent launch, so its CTAs are already resident
// when the product finishes) sums each row's partials in a fixed order (deterministic),
// scales the row and stores y, with the rows spread evenly over the GPU.
//
// Three product kernels, chosen by batch, code width and prefix:
//  * gemv_lut (B = 8; 1 or 2 tokens with m <= 8, or 3..4 tokens with m <= 4). By linearity,
//    x_g . (sum_k C_k[b_k]) = sum_k T_k[g][b_k] with T_k[g][j] = x_g . C_k[j]. A persistent
//    CTA (one per SM) walks a contiguous range of work items; for each (slice, book) it builds
//    that book's T for the 32 groups in shared memory (32 KiB per token), then every code
//    byte costs one shared-memory lookup and one fp32 add per token. Lane L owns row
//    32*rb+L; because each row's 32 codes are stored rotated by the row index, at step p all
//    32 lanes look up 32 different groups, i.e. 32 different banks, so the lookups are
//    conflict-free and no cross-lane reduction is needed. One producer warp streams the code
//    planes into a shared-memory ring with TMA bulk copies (the CTA's rows of a slice are
//    contiguous in every plane), overlapping HBM reads with the table build and the lookups
//    of the sixteen consumer warps.
//  * gemv_mma (B = 8, 5..16 tokens, any m <= 8). The decoded group (fp32 sum of the m
//    codewords, rounded once to tf32) is an A fragment of a tensor-core multiply with 8 or
//    16 tokens of activations (mma.sync m16n8k8).
//  * gemv_lut4 (B = 4, 1 token): the whole product in one kernel; each warp builds the
//    16-entry tables of its slices and looks up one entry per 4-bit code.
//  * gemv_direct (any other case: 4- and 16-bit codes, larger m). Decode each group in fp32 (sum of
//    m codewords), then multiply by the tokens' 8 activations. Lane L owns row 32*rb+L and
//    walks the 32 groups of the slice in a common order, so the activation loads are
//    warp-uniform broadcasts.
#include <map>
#include <mutex>
#include <tuple>
#include <type_traits>

#include "aq_internal.cuh"

namespace aq {
namespace {

// ------------------------------------------------------------------ LUT kernel (B = 8, b <= 4)

constexpr int kCons = 16;                         // consumer warps (two 32-row blocks each per stage)
constexpr int kLutThreads = (kCons + 1) * 32;     // + one producer warp
constexpr int kStageRb = 2 * kCons;               // 32-row blocks per stage: a 32 KiB plane copy
constexpr int kSlot = kStageRb * 1024;            // one ring slot = one plane of one stage
constexpr int kSlots = 4;                         // largest ring depth (128 KiB)
constexpr int kXStage = 8;                        // (token, slice) activation rows staged up front

// Tables: 64 KiB per two tokens (NT = 1 uses the two halves for consecutive units).
constexpr int lut_table_bytes(int nt) { return nt == 4 ? 131072 : 65536; }

// Shared memory: [T][codebooks m x 4 KiB][activations 8 x 1 KiB fp32][ring][barriers]
inline size_t lut_smem_bytes(int nt, int m, int slots, int nsets = 1) {
    return (size_t)lut_table_bytes(nt) + (size_t)nsets * m * 4096 + kXStage * 1024 +
           (size_t)slots * kSlot + 2 * kSlots * 8;
}

// Work is split by slice and by codebook: by linearity in the books (the successive-refinement
// form of Sec. 5, y_m = sum over k < m of x . (s o C_k[b_k])^T), the product over slice s and
// book k is a separate term. A unit is such a (slice s, book k) pair, numbered u = s*m + k;
// an item is (unit, 32-row block), numbered u*RBc + rb. Each item writes one fp32 partial per
// row into plane u of the partial sums, and the reduction adds the m*S planes of a row. So a
// CTA builds the table of one book for every unit it touches (one or two units in general),
// and looks it up for all of that unit's rows it owns, instead of building m tables for a
// third as many rows.
//
// Table of a unit: T[j][h][32 groups] (fp32), entry (j, g) of the unit's book at byte
// j*256 + h*128 + g*4, h alternating between the CTA's consecutive units, so a unit's table is
// built while the other half still serves the previous unit; j*256 + g*4 is produced from a
// code byte by one prmt.
//
// NT = 2 or 4 tokens (batch 2..4): one table per token, token t in the 64 KiB table t/2 at
// half t%2, so the same prmt offset serves every token and the token is a constant of the
// load: a code byte costs one prmt plus one load and one add per token. The tables are
// rebuilt in place (a barrier first) and the partial planes are per (unit, token).
//
// A CTA owns the items [i0, i1) and walks them in stages of up to 32 items that never cross a
// unit. For each stage the producer warp copies the stage's rows of the unit's book plane into
// one ring slot with a TMA bulk copy (32 KiB; the CTA's rows of a slice are contiguous in
// every plane), and consumer warp w looks up items w and w + 16 of the stage, so each wait on
// the ring serves two row blocks. The codebooks and the activations of the CTA's first slices
// are requested before any code.
// The layers of one call: one layer, or up to kGroupMax layers that share the activations
// (aq_gemv_group). Items are numbered layer after layer: layer l holds the items
// [base[l], base[l+1]), numbered within the layer as above (unit u = s*m + k, then row block).
// A CTA's items lie in at most two layers (checked by the host), whose first m codebooks it
// stages.
constexpr int kGroupMax = 4;
struct LutLayers {
    const uint8_t* planes[kGroupMax];
    const uint16_t* books[kGroupMax];
    float* partials[kGroupMax];
    size_t plane_bytes[kGroupMax];
    int rows_pad[kGroupMax], RBc[kGroupMax], base[kGroupMax + 1];
    int n;
};

template <int BDT, int XDT, int NT, bool GROUP>
__global__ void __launch_bounds__(kLutThreads, 1)
gemv_lut_kernel(const __grid_constant__ LutLayers L, const uint16_t* __restrict__ x,
                unsigned int* __restrict__ status, int m, int in, int ng, int nslots, int cpu,
                int q, int r, int static_weights, int batch) {
    constexpr int kTB = lut_table_bytes(NT);
    constexpr int kXSlices = kXStage / NT;      // activation slices staged per token
    extern __shared__ __align__(128) unsigned char smem[];
    unsigned char* T = smem;
    const int nl = GROUP ? L.n : 1;             // layers (a single call: one, known at compile time)
    const int nsets = nl > 1 ? 2 : 1;           // codebook sets staged (layers per CTA)
    uint4* Cb = (uint4*)(smem + kTB);                              // [nsets][m][256] codewords
    // [NT][kXSlices][256] activations in fp32; group g of a slice at 128-byte line g/4, its
    // two 16-byte halves at quads (2*(g%4) + half) ^ (g/4 mod 8), so the table build's reads
    // (eight lanes at eight different lines) hit eight different bank quads.
    unsigned char* xs = smem + kTB + (size_t)nsets * m * 4096;
    unsigned char* ring = xs + kXStage * 1024;                     // nslots x 32 KiB
    uint64_t* full = (uint64_t*)(ring + (size_t)nslots * kSlot);
    uint64_t* empty = full + kSlots;
    __shared__ volatile int s_abort;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // Item range of this CTA: a share of one unit (cpu CTAs per unit: RBc = q*cpu + r) or a
    // share of all items (total = q*gridDim.x + r); the first r shares are one item longer.
    // Item indices fit in 32 bits (checked by the host); the per-stage bookkeeping below is
    // incremental, without divisions (an integer division is a long instruction sequence).
    int i0, i1;
    {
        int b = blockIdx.x, base = 0;
        if (cpu > 0) {                          // single layer only
            const int u = b / cpu;
            b -= u * cpu;
            base = u * L.RBc[0];
        }
        i0 = base + b * q + min(b, r);
        i1 = i0 + q + (b < r ? 1 : 0);
    }
    const int S = (ng + 31) >> 5;
    int l_first = 0;
    while (l_first + 1 < nl && i0 >= L.base[l_first + 1]) ++l_first;
    const int u_first = (i0 - (GROUP ? L.base[l_first] : 0)) / L.RBc[l_first], s_first = u_first / m;
    // A walk over the CTA's items in stages: up to kStageRb items, never crossing a unit
    // (nor, therefore, a layer). rbc, rp: row blocks and padded rows of layer l.
    struct Walk {
        int it, l, s, k, rb, n, rbc, rp;
    };
    auto walk_start = [&]() {
        const int rbc = L.RBc[l_first];
        Walk w{i0, l_first, s_first, u_first - s_first * m, i0 - (GROUP ? L.base[l_first] : 0) - u_first * rbc, 0,
               rbc, L.rows_pad[l_first]};
        w.n = min(min(kStageRb, rbc - w.rb), i1 - w.it);
        return w;
    };
    auto walk_next = [&](Walk& w) {
        w.it += w.n;
        w.rb += w.n;
        if (w.rb == w.rbc) {
            w.rb = 0;
            if (++w.k == m) {
                w.k = 0;
                if (++w.s == S && w.l + 1 < nl) {
                    w.s = 0;
                    ++w.l;
                    w.rbc = L.RBc[w.l];
                    w.rp = L.rows_pad[w.l];
                }
            }
        }
        w.n = min(min(kStageRb, w.rbc - w.rb), i1 - w.it);
    };

    // Producer state (warp kCons, lane 0): the next copy is stage p_w into ring slot p_slot
    // (use parity p_phase); p_q copies issued so far.
    int p_q = 0, p_slot = 0;
    uint32_t p_phase = 0;
    Walk p_w = walk_start();
    auto issue_next = [&]() {
        const size_t src = ((size_t)p_w.s * p_w.rp + (size_t)p_w.rb * 32) * 32;
        mbar_arrive_expect_tx(&full[p_slot], (uint32_t)(p_w.n * 1024));
        bulk_g2s(ring + (size_t)p_slot * kSlot,
                 L.planes[GROUP ? p_w.l : 0] + (size_t)p_w.k * L.plane_bytes[GROUP ? p_w.l : 0] + src,
                 (uint32_t)(p_w.n * 1024), &full[p_slot]);
        ++p_q;
        if (++p_slot == nslots) {
            p_slot = 0;
            p_phase ^= 1u;
        }
        walk_next(p_w);
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
    // Codebooks and activations are requested first (into registers) by the consumer threads,
    // which store them below.
    // codebook sets: layer l_first, and l_first + 1 when the CTA's items reach into it
    int l_last = l_first;
    while (l_last + 1 < nl && i1 - 1 >= L.base[l_last + 1]) ++l_last;
    uint4 cb_r[2][4];
    auto load_books = [&]() {
#pragma unroll
        for (int set = 0; set < 2; ++set)
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int i = tid + r * kCons * 32;
                cb_r[set][r] = (l_first + set <= l_last && tid < kCons * 32 && i < m * 256)
                                   ? __ldg((const uint4*)L.books[l_first + set] + i)
                                   : make_uint4(0u, 0u, 0u, 0u);
            }
    };
    if (static_weights) {
        // The weights are read-only while calls run (AQ_LAYOUT_STATIC_WEIGHTS): request the
        // codebooks and the first code stage before waiting for the preceding kernel, so they
        // overlap its tail. Only one stage: the activations are requested right after the
        // wait and queue behind whatever code copies are still in flight (measured on the
        // 14336 x 4096 layer: one stage 4-7 % faster per call than a full ring).
        load_books();
        if (warp == kCons && lane == 0 && p_w.it < i1) issue_next();
    }
    pdl_wait();                 // inputs may come from the preceding kernel in the stream
    pdl_launch_dependents();    // the split-K reduction may become resident (it waits for us)
    if (!static_weights) load_books();
    uint2 x_r = make_uint2(0u, 0u);
    if (tid < kXStage * 64) {                   // row tid/64 = token * kXSlices + slice
        const int xt = (tid >> 6) / kXSlices, col = (s_first + (tid >> 6) % kXSlices) * 256 + (tid & 63) * 4;
        if (xt < batch && col < in) x_r = __ldg((const uint2*)(x + (size_t)xt * in + col));
    }

    if (warp == kCons) {
        // ---- producer (lane 0 issues; the warp stays converged for the final barriers)
        if (lane == 0) {
            while (p_w.it < i1) {
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
        for (int set = 0; set < 2; ++set)
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int i = tid + r * kCons * 32;
                if (set < nsets && i < m * 256) Cb[set * m * 256 + i] = cb_r[set][r];
            }
        if (tid < kXStage * 64) {
            const int e = tid & 63, g = e >> 1;
            float4 f;
            widen2<XDT>(x_r.x, f.x, f.y);
            widen2<XDT>(x_r.y, f.z, f.w);
            *(float4*)(xs + (tid >> 6) * 1024 + (g >> 2) * 128 + ((((g & 3) * 2) + (e & 1)) ^ ((g >> 2) & 7)) * 16) = f;
        }
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

        // Table build: lane L = 8*ph + gq computes groups 4gq..4gq+3 for codewords
        // j = 16*warp + ph + 4i; one 16-byte codeword read serves four entries, stored as one
        // 16-byte piece. xv holds the four groups' activations of the current slice.
        const int ph = lane >> 3, gq = lane & 7;
        float2 xv[4][4];
        int slot = 0;
        uint32_t phase = 0;                     // parity of the slot's current use
        int cur_s = -1, cur_k = -1, cur_l = -1, h = 1;
        for (Walk w = walk_start(); w.it < i1; walk_next(w)) {
            const int n = w.n, s = w.s, rb = w.rb;
            if (s != cur_s || w.k != cur_k || w.l != cur_l) {
                // Activations of the four groups 4gq..4gq+3 of slice s for token t.
                auto load_xv = [&](int t) {
                    // (the activations are shared by the layers of a group: slice s of x
                    // whatever the layer)
                    const int sl = s - s_first;
                    if ((unsigned)sl < (unsigned)kXSlices) {
                        const unsigned char* xb = xs + (t * kXSlices + sl) * 1024 + gq * 128;
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            const float4 lo = *(const float4*)(xb + (((2 * u) ^ gq) & 7) * 16);
                            const float4 hi = *(const float4*)(xb + (((2 * u + 1) ^ gq) & 7) * 16);
                            xv[u][0] = make_float2(lo.x, lo.y);
                            xv[u][1] = make_float2(lo.z, lo.w);
                            xv[u][2] = make_float2(hi.x, hi.y);
                            xv[u][3] = make_float2(hi.z, hi.w);
                        }
                    } else {
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            const int g = s * 32 + gq * 4 + u;
                            uint4 xr = make_uint4(0u, 0u, 0u, 0u);
                            if (t < batch && g < ng) xr = __ldg((const uint4*)(x + (size_t)t * in) + g);
                            float f[8];
                            unpack8<XDT>(xr, f);
#pragma unroll
                            for (int e = 0; e < 4; ++e) xv[u][e] = make_float2(f[2 * e], f[2 * e + 1]);
                        }
                    }
                };
                // Entries j = 16*warp + ph + 4i, groups 4gq..4gq+3 of the unit's book, for the
                // activations in xv, stored as 16-byte pieces at Th.
                auto build = [&](unsigned char* Th) {
                    uint4 cw[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        cw[i] = Cb[((GROUP ? w.l - l_first : 0) * m + w.k) * 256 + warp * 16 + ph + 4 * i];
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
                        *(float4*)(Th + (warp * 16 + ph + 4 * i) * 256) = make_float4(r[0], r[1], r[2], r[3]);
                    }
                };
                if constexpr (NT == 1) {
                    if (s != cur_s) load_xv(0);
                    h ^= 1;
                    // The other half served the previous unit; this half was last read two
                    // units ago, before every consumer passed the previous unit's barrier.
                    build(T + h * 128 + gq * 16);
                } else {
                    if (cur_k >= 0) named_barrier(1, kCons * 32);   // previous unit looked up
#pragma unroll 1
                    for (int t = 0; t < NT; ++t) {
                        load_xv(t);
                        build(T + (t >> 1) * 65536 + (t & 1) * 128 + gq * 16);
                    }
                }
                cur_s = s;
                cur_k = w.k;
                cur_l = w.l;
                named_barrier(1, kCons * 32);
            }
            float part0[NT], part1[NT];
#pragma unroll
            for (int t = 0; t < NT; ++t) part0[t] = part1[t] = 0.0f;
            bool ok = !s_abort;
            if (ok && !mbar_wait(&full[slot], phase)) {
                record_status(status, AQ_ERR_TIMEOUT);
                s_abort = 1;
                ok = false;
            }
            if (ok && warp < n) {
                // Each lane reads its row's 32 code bytes of item warp (and warp + 16) as two
                // 16-byte halves. The prmt forms the table offset of a code byte: byte0 = goff
                // byte i, byte1 = code byte i, bytes 2-3 = sign of the goff byte (0). The
                // table half (and for NT > 1 the token) is a constant of the load, so a lookup
                // is prmt, then a load and an add per token.
                const unsigned char* row0 = ring + (size_t)slot * kSlot + warp * 1024 + lane * 32;
                const uint4 a0 = *(const uint4*)(row0 + c0 * 16);
                const uint4 b0 = *(const uint4*)(row0 + (c0 ^ 1) * 16);
                const uint32_t w0[8] = {a0.x, a0.y, a0.z, a0.w, b0.x, b0.y, b0.z, b0.w};
                const bool two = warp + kCons < n;
                uint32_t w1[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
                if (two) {
                    const unsigned char* row1 = row0 + kCons * 1024;
                    const uint4 a1 = *(const uint4*)(row1 + c0 * 16);
                    const uint4 b1 = *(const uint4*)(row1 + (c0 ^ 1) * 16);
                    w1[0] = a1.x; w1[1] = a1.y; w1[2] = a1.z; w1[3] = a1.w;
                    w1[4] = b1.x; w1[5] = b1.y; w1[6] = b1.z; w1[7] = b1.w;
                }
                auto look = [&](auto half) {
                    const unsigned char* Tb = T + decltype(half)::value;
                    // token t of the table entry at offset o (token 0 when NT = 1)
                    auto ld = [&](uint32_t o, int t) {
                        return *(const float*)(Tb + (t >> 1) * 65536 + (t & 1) * 128 + o);
                    };
                    if (two) {
#pragma unroll
                        for (int qq = 0; qq < 8; ++qq) {
                            const uint32_t g = goff[qq];
                            const uint32_t o0 = prmt(w0[qq], g, 0xCC04u), p0 = prmt(w1[qq], g, 0xCC04u);
                            const uint32_t o1 = prmt(w0[qq], g, 0xDD15u), p1 = prmt(w1[qq], g, 0xDD15u);
                            const uint32_t o2 = prmt(w0[qq], g, 0xEE26u), p2 = prmt(w1[qq], g, 0xEE26u);
                            const uint32_t o3 = prmt(w0[qq], g, 0xFF37u), p3 = prmt(w1[qq], g, 0xFF37u);
#pragma unroll
                            for (int t = 0; t < NT; ++t) {
                                const float v0 = ld(o0, t), u0 = ld(p0, t), v1 = ld(o1, t), u1 = ld(p1, t);
                                const float v2 = ld(o2, t), u2 = ld(p2, t), v3 = ld(o3, t), u3 = ld(p3, t);
                                part0[t] += (v0 + v1) + (v2 + v3);
                                part1[t] += (u0 + u1) + (u2 + u3);
                            }
                        }
                    } else {
#pragma unroll
                        for (int qq = 0; qq < 8; ++qq) {
                            const uint32_t g = goff[qq];
                            const uint32_t o0 = prmt(w0[qq], g, 0xCC04u), o1 = prmt(w0[qq], g, 0xDD15u);
                            const uint32_t o2 = prmt(w0[qq], g, 0xEE26u), o3 = prmt(w0[qq], g, 0xFF37u);
#pragma unroll
                            for (int t = 0; t < NT; ++t) {
                                const float v0 = ld(o0, t), v1 = ld(o1, t), v2 = ld(o2, t), v3 = ld(o3, t);
                                part0[t] += (v0 + v1) + (v2 + v3);
                            }
                        }
                    }
                };
                if (NT == 1 && h) look(std::integral_constant<int, 128>());
                else look(std::integral_constant<int, 0>());
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[slot]);
            if (++slot == nslots) {
                slot = 0;
                phase ^= 1u;
            }
            if (ok && warp < n) {
#pragma unroll
                for (int t = 0; t < NT; ++t) {
                    if (t >= batch) break;
                    float* dst = L.partials[GROUP ? w.l : 0] + (((size_t)s * m + cur_k) * batch + t) * w.rp +
                                 (size_t)(rb + warp) * 32 + lane;
                    dst[0] = part0[t];
                    if (warp + kCons < n) dst[kCons * 32] = part1[t];
                }
            }
        }
    }
}

// ------------------------------------------------------------------ 8-token LUT kernel (B = 8)
//
// gemv_lut8 (a pass of up to 8 tokens, B = 8, m <= kLut8MaxM; 9..16 tokens take two passes):
// the table form for several tokens with fp16 table entries. The table of a (slice s, book k)
// unit holds, for every codeword j and group g, the eight tokens' products x_t,g . C_k[j],
// four tokens to an 8-byte entry: sub-table h (tokens 4h..4h+3) at byte h*65536 + j*256 + 8g.
// A code byte then costs one prmt (offset j*256 + 8g), two 8-byte shared loads and eight
// mixed-type adds into fp32 sums; the 32 lanes of a warp hit 32 different groups (the row
// rotation), i.e. 32 different 8-byte words: two wavefronts per load, conflict-free.
// Range: the entries of token t in unit (s, k) are scaled by 2^f with
// f = 12 - floor(log2(8 max|x_t over slice s| max|C_k|)), so every entry is below 2^13 in
// magnitude and the largest ones use fp16's full precision; the item's sum is multiplied by
// 2^-f when it is stored. Both scalings are exact. The entries of two consecutive code bytes
// are first added in fp16 (packed adds; a sum of two stays below 2^14), then widened once
// into the fp32 sums: one extra fp16 rounding per pair of entries (a longer window measured
// per-element errors beyond the product tolerance on long rows), half the widening work.
// Work split, code ring, producer warp, bounded waits and partial planes as gemv_lut (one
// partial plane per (slice, book, token)); the tables are rebuilt in place behind a barrier.
constexpr int kLut8MaxM = 6;       // 128 KiB of tables, m codebooks and two 32 KiB code stages

// Packed fp16 pair add, each half rounded to nearest.
__device__ __forceinline__ uint32_t hadd2(uint32_t a, uint32_t b) {
    uint32_t d;
    asm("add.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

inline size_t lut8_smem_bytes(int m, int slots) {
    return 131072 + (size_t)m * 4096 + (size_t)slots * kSlot + 2 * kSlots * 8;
}

template <int BDT, int XDT>
__global__ void __launch_bounds__(kLutThreads, 1)
gemv_lut8_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
                 const uint16_t* __restrict__ x, float* __restrict__ partials,
                 unsigned int* __restrict__ status, int m, int in, int ng, int rows_pad, int RBc,
                 size_t plane_bytes, int nslots, int cpu, int q, int r, int static_weights,
                 int batch, int t_base) {
    extern __shared__ __align__(128) unsigned char smem[];
    unsigned char* T = smem;                                       // two 64 KiB sub-tables
    uint4* Cb = (uint4*)(smem + 131072);                           // [m][256] codewords
    unsigned char* ring = smem + 131072 + (size_t)m * 4096;        // nslots x 32 KiB
    uint64_t* full = (uint64_t*)(ring + (size_t)nslots * kSlot);
    uint64_t* empty = full + kSlots;
    __shared__ volatile int s_abort;
    __shared__ unsigned int s_cmax[kLut8MaxM];   // bits of max |C_k| (non-negative floats order as ints)

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    int i0, i1;
    {
        int b = blockIdx.x, base = 0;
        if (cpu > 0) {
            const int u = b / cpu;
            b -= u * cpu;
            base = u * RBc;
        }
        i0 = base + b * q + min(b, r);
        i1 = i0 + q + (b < r ? 1 : 0);
    }
    const int u_first = i0 / RBc, s_first = u_first / m;
    struct Walk {
        int it, s, k, rb, n;
    };
    auto walk_start = [&]() {
        Walk w{i0, s_first, u_first - s_first * m, i0 - u_first * RBc, 0};
        w.n = min(min(kStageRb, RBc - w.rb), i1 - w.it);
        return w;
    };
    auto walk_next = [&](Walk& w) {
        w.it += w.n;
        w.rb += w.n;
        if (w.rb == RBc) {
            w.rb = 0;
            if (++w.k == m) {
                w.k = 0;
                ++w.s;
            }
        }
        w.n = min(min(kStageRb, RBc - w.rb), i1 - w.it);
    };

    int p_q = 0, p_slot = 0;
    uint32_t p_phase = 0;
    Walk p_w = walk_start();
    auto issue_next = [&]() {
        const size_t src = ((size_t)p_w.s * rows_pad + (size_t)p_w.rb * 32) * 32;
        mbar_arrive_expect_tx(&full[p_slot], (uint32_t)(p_w.n * 1024));
        bulk_g2s(ring + (size_t)p_slot * kSlot, planes + (size_t)p_w.k * plane_bytes + src,
                 (uint32_t)(p_w.n * 1024), &full[p_slot]);
        ++p_q;
        if (++p_slot == nslots) {
            p_slot = 0;
            p_phase ^= 1u;
        }
        walk_next(p_w);
    };
    if (tid == 0) {
        for (int d = 0; d < nslots; ++d) {
            mbar_init(&full[d], 1);
            mbar_init(&empty[d], kCons);
        }
        mbar_fence_init();
        s_abort = 0;
    }
    if (tid < kLut8MaxM) s_cmax[tid] = 0u;
    __syncthreads();
    uint4 cb_r[3];
    auto load_books = [&]() {
#pragma unroll
        for (int i = 0; i < 3; ++i) {
            const int c = tid + i * kCons * 32;
            cb_r[i] = (tid < kCons * 32 && c < m * 256) ? __ldg((const uint4*)books + c)
                                                         : make_uint4(0u, 0u, 0u, 0u);
        }
    };
    if (static_weights) {
        // read-only weights (AQ_LAYOUT_STATIC_WEIGHTS): codebooks and the first code stage
        // are requested before waiting for the preceding kernel
        load_books();
        if (warp == kCons && lane == 0 && p_w.it < i1) issue_next();
    }
    pdl_wait();
    pdl_launch_dependents();
    if (!static_weights) load_books();

    if (warp == kCons) {
        // ---- producer
        if (lane == 0) {
            while (p_w.it < i1) {
                if (s_abort) break;
                if (p_q >= nslots && !mbar_wait(&empty[p_slot], p_phase ^ 1u)) {
                    record_status(status, AQ_ERR_TIMEOUT);
                    s_abort = 1;
                    break;
                }
                issue_next();
            }
            for (int j = max(0, p_q - nslots); j < p_q; ++j) mbar_wait(&full[j % nslots], (j / nslots) & 1);
        }
        __syncwarp();
        return;
    }

    // ---- consumers: stage the codebooks and each book's largest magnitude
#pragma unroll
    for (int i = 0; i < 3; ++i) {
        const int c = tid + i * kCons * 32;
        float mx = 0.0f;
        if (c < m * 256) {
            Cb[c] = cb_r[i];
            float f[8];
            unpack8<BDT>(cb_r[i], f);
#pragma unroll
            for (int e = 0; e < 8; ++e) mx = fmaxf(mx, fabsf(f[e]));
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        // the 32 codewords of a warp belong to one book (256 per book)
        if (lane == 0 && c < m * 256) atomicMax(&s_cmax[c >> 8], __float_as_uint(mx));
    }
    named_barrier(1, kCons * 32);

    // Code bytes: each lane reads its row's 32 bytes as two 16-byte halves, lanes 4-7 of every
    // eight the second half first (conflict-free ring reads). Read position r (0..31) is row
    // position p = (r + 16 c0) mod 32, group (p + lane) mod 32. gz[v] bytes 0..2 = 8 * group of
    // read positions 3v..3v+2, byte 3 = 0 (the zero that fills the offset's upper half).
    const int c0 = (lane >> 2) & 1;
    uint32_t gz[11];
#pragma unroll
    for (int v = 0; v < 11; ++v) {
        uint32_t z = 0;
#pragma unroll
        for (int i = 0; i < 3; ++i) {
            const int rr = 3 * v + i;
            if (rr < 32) z |= (uint32_t)((((rr + (c0 ? 16 : 0)) + lane) & 31) * 8) << (8 * i);
        }
        gz[v] = z;
    }

    // Table of unit (s, k) for this pass's tokens: lane g (group g of slice s) computes, for
    // codewords j = 16*warp .. 16*warp + 15, the entries of all eight tokens from its group's
    // activations, pre-multiplied by 2^f (exact: f is also limited so that no scaled
    // activation exceeds 2^100).
    float sinv[8];      // 2^-f of each token for the current unit
    auto build = [&](int s, int k) {
        const int g = s * 32 + lane;
        const float cmax = __uint_as_float(s_cmax[k]);
        float xv[8][8];
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            uint4 xr = make_uint4(0u, 0u, 0u, 0u);
            if (t_base + t < batch && g < ng) xr = __ldg((const uint4*)(x + (size_t)(t_base + t) * in) + g);
            unpack8<XDT>(xr, xv[t]);
        }
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            float mx = 0.0f;
#pragma unroll
            for (int e = 0; e < 8; ++e) mx = fmaxf(mx, fabsf(xv[t][e]));
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            const float bound = 8.0f * mx * cmax;
            int f = 0;
            if (bound > 0.0f) f = min(min(126, 100 - exponent_of(mx)), max(-126, 12 - exponent_of(bound)));
            const float sc = pow2f(f);
#pragma unroll
            for (int e = 0; e < 8; ++e) xv[t][e] *= sc;
            sinv[t] = pow2f(-f);
        }
        unsigned char* Tl = T + lane * 8;
#pragma unroll 2
        for (int i = 0; i < 16; ++i) {
            const int j = warp * 16 + i;
            float c[8];
            unpack8<BDT>(Cb[k * 256 + j], c);
            float v[8];
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                float2 a = make_float2(xv[t][0] * c[0], xv[t][1] * c[1]);
                a = ffma2(make_float2(xv[t][2], xv[t][3]), make_float2(c[2], c[3]), a);
                a = ffma2(make_float2(xv[t][4], xv[t][5]), make_float2(c[4], c[5]), a);
                a = ffma2(make_float2(xv[t][6], xv[t][7]), make_float2(c[6], c[7]), a);
                v[t] = a.x + a.y;
            }
            uint32_t h[4];
#pragma unroll
            for (int u = 0; u < 4; ++u)
                asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(h[u]) : "f"(v[2 * u + 1]), "f"(v[2 * u]));
            *(uint2*)(Tl + j * 256) = make_uint2(h[0], h[1]);
            *(uint2*)(Tl + 65536 + j * 256) = make_uint2(h[2], h[3]);
        }
    };

    int slot = 0;
    uint32_t phase = 0;
    int cur_s = -1, cur_k = -1;
    for (Walk w = walk_start(); w.it < i1; walk_next(w)) {
        const int n = w.n, s = w.s, rb = w.rb;
        if (s != cur_s || w.k != cur_k) {
            if (cur_k >= 0) named_barrier(1, kCons * 32);   // the previous unit looked up
            build(s, w.k);
            cur_s = s;
            cur_k = w.k;
            named_barrier(1, kCons * 32);                    // the unit's table built
        }
        float acc0[8], acc1[8];
#pragma unroll
        for (int t = 0; t < 8; ++t) acc0[t] = acc1[t] = 0.0f;
        bool ok = !s_abort;
        if (ok && !mbar_wait(&full[slot], phase)) {
            record_status(status, AQ_ERR_TIMEOUT);
            s_abort = 1;
            ok = false;
        }
        const bool two = warp + kCons < n;
        if (ok && warp < n) {
            const unsigned char* row0 = ring + (size_t)slot * kSlot + warp * 1024 + lane * 32;
            const uint4 a0 = *(const uint4*)(row0 + c0 * 16);
            const uint4 b0 = *(const uint4*)(row0 + (c0 ^ 1) * 16);
            const uint32_t w0[8] = {a0.x, a0.y, a0.z, a0.w, b0.x, b0.y, b0.z, b0.w};
            uint32_t w1[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
            if (two) {
                const unsigned char* row1 = row0 + kCons * 1024;
                const uint4 a1 = *(const uint4*)(row1 + c0 * 16);
                const uint4 b1 = *(const uint4*)(row1 + (c0 ^ 1) * 16);
                w1[0] = a1.x; w1[1] = a1.y; w1[2] = a1.z; w1[3] = a1.w;
                w1[4] = b1.x; w1[5] = b1.y; w1[6] = b1.z; w1[7] = b1.w;
            }
            // The four code bytes of word qq: offsets j*256 + 8g; the entries (fp16 pairs of
            // tokens 0-1, 2-3, 4-5, 6-7) of bytes 0+1 and of bytes 2+3 are added in fp16, then
            // widened into the fp32 sums.
            auto look4 = [&](uint32_t code_word, int qq, float (&acc)[8]) {
#pragma unroll
                for (int i = 0; i < 4; i += 2) {
                    uint32_t sum[4];
#pragma unroll
                    for (int ii = 0; ii < 2; ++ii) {
                        const int rr = 4 * qq + i + ii;
                        const uint32_t sel =
                            0x7700u | ((uint32_t)(i + ii) << 4) | (uint32_t)(4 + rr % 3);
                        const uint32_t o = prmt(code_word, gz[rr / 3], sel);
                        const uint2 lo = *(const uint2*)(T + o);
                        const uint2 hi = *(const uint2*)(T + 65536 + o);
                        if (ii == 0) {
                            sum[0] = lo.x; sum[1] = lo.y; sum[2] = hi.x; sum[3] = hi.y;
                        } else {
                            sum[0] = hadd2(sum[0], lo.x);
                            sum[1] = hadd2(sum[1], lo.y);
                            sum[2] = hadd2(sum[2], hi.x);
                            sum[3] = hadd2(sum[3], hi.y);
                        }
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u) add_widen2<AQ_F16>(sum[u], acc[2 * u], acc[2 * u + 1]);
                }
            };
#pragma unroll
            for (int qq = 0; qq < 8; ++qq) {
                look4(w0[qq], qq, acc0);
                if (two) look4(w1[qq], qq, acc1);
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[slot]);
        if (++slot == nslots) {
            slot = 0;
            phase ^= 1u;
        }
        if (ok && warp < n) {
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                if (t_base + t >= batch) break;
                float* dst = partials + (((size_t)s * m + cur_k) * batch + t_base + t) * rows_pad +
                             (size_t)(rb + warp) * 32 + lane;
                dst[0] = acc0[t] * sinv[t];
                if (two) dst[kCons * 32] = acc1[t] * sinv[t];
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
    constexpr int UNIT = unit_bytes(B);
    constexpr int kWarps = 8;
    extern __shared__ __align__(128) unsigned char smem[];
    float* xs = (float*)smem;                                        // [NB][256]
    uint16_t* books_s = (uint16_t*)(smem + NB * 1024);               // B <= 8: [m][2^B][8]
    const size_t books_bytes = staged_books_bytes(B, m);
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
    if constexpr (B <= 8) {
        for (int i = tid; i < (m << B); i += 256)
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
                const uint32_t code = unit_code<B>(codes_s + ((size_t)k * 32 + lane) * UNIT, p);
                uint4 cwv;
                if constexpr (B <= 8) cwv = ((const uint4*)books_s)[(k << B) + code];
                else cwv = ld_stream_v4((const uint4*)books + ((size_t)k << 16) + code);
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

// ------------------------------------------------------------------ tensor-core kernel (B = 8, 2..16 tokens)

// Partials for 2..16 tokens with the multiply on the tensor cores (mma.sync m16n8k8, tf32
// operands, fp32 accumulation). Each warp takes one 32-row block of the CTA's slice: the
// block's code rows (first MB planes) are staged in shared memory in group order, and for
// every group the lanes gather the codeword elements of their A-fragment positions (rows g,
// g+8, g+16, g+24 of the block, elements c and c+4 of the group), sum them over the MB books
// in fp32 in book order, round the sum once to tf32 and multiply with the activations (B
// fragments: 8 or 16 tokens, exact in tf32). The codebooks are staged with the elements of
// every codeword interleaved (0,4,1,5,2,6,3,7), so a lane's two elements are one 32-bit word;
// each element is added to its fp32 sum by one mixed-type add (16-bit operand, fp32 sum).
// (Eight bank-disjoint copies of each book, which make the gathers conflict-free, measured
// slower: at m = 3, 4 their 32 KiB per book leave one CTA per SM.)
constexpr int kMmaMaxM = 8;       // prefixes compiled for this kernel
constexpr int kMmaXStride = 260;   // floats per staged token row (4 of padding: conflict-free)
constexpr int kMmaCodeRow = 36;    // bytes per staged code row (4 of padding: conflict-free)

inline size_t mma_smem_bytes(int nt, int mb) {
    return (size_t)8 * nt * kMmaXStride * 4 + (size_t)mb * 4096 + (size_t)8 * mb * 32 * kMmaCodeRow;
}

__device__ __forceinline__ uint32_t to_tf32(float v) {
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(v));
    return r;
}

__device__ __forceinline__ void mma_tf32(float (&d)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
    asm volatile(
        "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
        "{%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

template <int NT, int BDT, int MB>
__global__ void __launch_bounds__(256)
gemv_mma_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
                const uint16_t* __restrict__ x, int x_dt, float* __restrict__ partials, int batch,
                int in, int rows_pad, int RBc, int rb_per_chunk, size_t plane_bytes) {
    constexpr int NBT = 8 * NT;                 // tokens held (missing ones are zero)
    extern __shared__ __align__(16) unsigned char smem[];
    float* xs = (float*)smem;                                            // [NBT][260]
    uint32_t* books_s = (uint32_t*)(smem + NBT * kMmaXStride * 4);      // [MB][256][4]
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    unsigned char* codes_w =
        smem + NBT * kMmaXStride * 4 + MB * 4096 + warp * (MB * 32 * kMmaCodeRow);
    const int s = blockIdx.y, chunk = blockIdx.x;

    pdl_wait();
    pdl_launch_dependents();
    for (int i = tid; i < NBT * 256; i += 256) {
        const int t = i >> 8, c = i & 255, col = s * 256 + c;
        float v = 0.0f;
        if (t < batch && col < in) v = bits_to_f32_rt(x[(size_t)t * in + col], x_dt);
        xs[t * kMmaXStride + c] = v;
    }
    for (int i = tid; i < MB * 256; i += 256) {
        const uint4 w = __ldg((const uint4*)books + i);   // halves 0..7 of codeword i
        *(uint4*)(books_s + i * 4) = make_uint4(prmt(w.x, w.z, 0x5410u), prmt(w.x, w.z, 0x7632u),
                                                prmt(w.y, w.w, 0x5410u), prmt(w.y, w.w, 0x7632u));
    }
    __syncthreads();

    const int g = lane >> 2, c = lane & 3;
    const int rb0 = chunk * rb_per_chunk;
    const int rb1 = min(rb0 + rb_per_chunk, RBc);
    for (int rb = rb0 + warp; rb < rb1; rb += 8) {
        // the block's code rows, in group order (lane = row)
#pragma unroll
        for (int k = 0; k < MB; ++k) {
            const uint4* src = (const uint4*)(planes + k * plane_bytes +
                                              ((size_t)s * rows_pad + (size_t)rb * 32 + lane) * 32);
            const uint4 lo = ld_stream_v4(src), hi = ld_stream_v4(src + 1);
            const uint32_t w[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
            uint32_t u[8];
            unrotate_codes(w, lane, u);
            uint32_t* dst = (uint32_t*)(codes_w + (k * 32 + lane) * kMmaCodeRow);
#pragma unroll
            for (int j = 0; j < 8; ++j) dst[j] = u[j];
        }
        __syncwarp();
        float acc[2][NT][4];
#pragma unroll
        for (int mt = 0; mt < 2; ++mt)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[mt][nt][e] = 0.0f;
#pragma unroll 1
        for (int q = 0; q < 8; ++q) {           // groups 4q .. 4q+3
            uint32_t cw[4][MB];                 // codes of rows g + 8rr, one byte per group
#pragma unroll
            for (int rr = 0; rr < 4; ++rr)
#pragma unroll
                for (int k = 0; k < MB; ++k)
                    cw[rr][k] = *(const uint32_t*)(codes_w + (k * 32 + g + 8 * rr) * kMmaCodeRow + 4 * q);
#pragma unroll
            for (int gg = 0; gg < 4; ++gg) {
                const int G = 4 * q + gg;
                uint32_t bf[NT][2];
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                    const float* xr = xs + (8 * nt + g) * kMmaXStride + 8 * G + c;
                    bf[nt][0] = __float_as_uint(xr[0]);
                    bf[nt][1] = __float_as_uint(xr[4]);
                }
                uint32_t af[4][2];
#pragma unroll
                for (int rr = 0; rr < 4; ++rr) {
                    float lo = -0.0f, hi = -0.0f;   // -0 + v = v exactly, so the first add widens
#pragma unroll
                    for (int k = 0; k < MB; ++k) {
                        const uint32_t code = (cw[rr][k] >> (8 * gg)) & 0xffu;
                        add_widen2<BDT>(books_s[(k * 256 + code) * 4 + c], lo, hi);
                    }
                    af[rr][0] = to_tf32(lo);
                    af[rr][1] = to_tf32(hi);
                }
#pragma unroll
                for (int mt = 0; mt < 2; ++mt) {
                    const uint32_t a[4] = {af[2 * mt][0], af[2 * mt + 1][0], af[2 * mt][1], af[2 * mt + 1][1]};
#pragma unroll
                    for (int nt = 0; nt < NT; ++nt) mma_tf32(acc[mt][nt], a, bf[nt]);
                }
            }
        }
        __syncwarp();                           // the code buffer is refilled next
#pragma unroll
        for (int mt = 0; mt < 2; ++mt)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const int r0 = rb * 32 + mt * 16 + g, t0 = 8 * nt + 2 * c;
                float* p0 = partials + ((size_t)s * batch + t0) * rows_pad + r0;
                if (t0 < batch) {
                    p0[0] = acc[mt][nt][0];
                    p0[8] = acc[mt][nt][2];
                }
                if (t0 + 1 < batch) {
                    p0[rows_pad] = acc[mt][nt][1];
                    p0[rows_pad + 8] = acc[mt][nt][3];
                }
            }
    }
}

// ------------------------------------------------------------------ 2^16-entry books, one token
//
// gemv_gather16 (B = 16, 1 token, m <= 2): the codewords come from 1 MiB books read through L2,
// so the kernel is bound by the number of random 16-byte gathers in flight. Lane L owns row
// 32*rb + L of a slice; its 32 codes per book (64 bytes, position p holding group
// (p + L) mod 32) are loaded into registers, then for every eight positions the lane issues all
// 8*m codeword gathers (not allocated in L1: the hit rate there is nil) before it adds and
// multiplies any of them. Activations are staged per slice in shared memory as fp32 and read
// per lane (group (p + L) mod 32). Partials per (slice, row) as gemv_direct.
constexpr int kG16Warps = 8;

template <int BDT, int XDT, int MB>
__global__ void __launch_bounds__(kG16Warps * 32)
gemv_gather16_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
                     const uint16_t* __restrict__ x, float* __restrict__ partials, int in,
                     int rows_pad, int RBc, int rb_per_chunk, size_t plane_bytes) {
    __shared__ __align__(16) float xs[256];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int s = blockIdx.y, chunk = blockIdx.x;
    const int rb0 = chunk * rb_per_chunk, rb1 = min(rb0 + rb_per_chunk, RBc);
    pdl_wait();
    pdl_launch_dependents();
    for (int i = tid; i < 256; i += kG16Warps * 32) {
        const int col = s * 256 + i;
        xs[i] = col < in ? bits_to_f32<XDT>(x[col]) : 0.0f;
    }
    __syncthreads();
    for (int rb = rb0 + warp; rb < rb1; rb += kG16Warps) {
        const int o = rb * 32 + lane;
        uint4 cr[MB][4];                          // 32 codes per book, 8 per uint4
#pragma unroll
        for (int k = 0; k < MB; ++k) {
            const uint4* src = (const uint4*)(planes + (size_t)k * plane_bytes + ((size_t)s * rows_pad + o) * 64);
#pragma unroll
            for (int q = 0; q < 4; ++q) cr[k][q] = ld_stream_v4(src + q);
        }
        float acc = 0.0f;
#pragma unroll
        for (int p0 = 0; p0 < 32; p0 += 8) {
            uint4 cw[MB][8];
#pragma unroll
            for (int k = 0; k < MB; ++k) {
                const uint4 w4 = cr[k][p0 >> 3];
                const uint32_t wv[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const uint32_t code = (wv[i >> 1] >> (16 * (i & 1))) & 0xffffu;
                    cw[k][i] = ld_stream_v4((const uint4*)books + ((size_t)k << 16) + code);
                }
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int g = (p0 + i + lane) & 31;
                const float4 x0 = *(const float4*)(xs + g * 8);
                const float4 x1 = *(const float4*)(xs + g * 8 + 4);
                float w[8];
                unpack8<BDT>(cw[0][i], w);
#pragma unroll
                for (int k = 1; k < MB; ++k) {
                    float c[8];
                    unpack8<BDT>(cw[k][i], c);
#pragma unroll
                    for (int e = 0; e < 8; ++e) w[e] += c[e];
                }
                acc = fmaf(x0.x, w[0], acc);
                acc = fmaf(x0.y, w[1], acc);
                acc = fmaf(x0.z, w[2], acc);
                acc = fmaf(x0.w, w[3], acc);
                acc = fmaf(x1.x, w[4], acc);
                acc = fmaf(x1.y, w[5], acc);
                acc = fmaf(x1.z, w[6], acc);
                acc = fmaf(x1.w, w[7], acc);
            }
        }
        partials[(size_t)s * rows_pad + o] = acc;
    }
}

// ------------------------------------------------------------------ split-K reduction

// y[t][r] = s[r] * sum over the P partial planes p of partials[p*batch + t][r] (R1: the row
// scale multiplies the codebook sum, so it factors out of the dot product). A CTA of eight
// warps takes 32 * 8 / wpr rows of one token; the wpr warps (1, 2, 4 or 8) of a 32-row group
// split its planes: warp j of the group adds planes j, j + wpr, ... in order (up to sixteen
// loads in flight, coalesced over the rows), then the group's first warp adds the wpr sums in
// order, so the summation order is fixed. With static weights the row scales are read before
// waiting for the product kernel. With y_prev (a refinement, Sec. 4 successive
// reconstruction) the scaled sum is added to y_prev[t][r], read in y's type (y_prev may be y).
// The kernel is kept small: it runs once per CTA, so its instructions are fetched cold.
// The layers a reduction finishes: one, or the layers of a group (blockIdx.z = layer).
struct ReduceLayers {
    const float* partials[kGroupMax];
    const uint16_t* scales[kGroupMax];
    void* y[kGroupMax];
    int out[kGroupMax], rows_pad[kGroupMax];
};

template <int SDT, bool GROUP>
__global__ void __launch_bounds__(256)
splitk_reduce_kernel(const __grid_constant__ ReduceLayers R, int y_dt, int P, int batch, int wpr,
                     int static_weights, const void* y_prev) {
    const int z = GROUP ? blockIdx.z : 0;
    const float* __restrict__ partials = R.partials[z];
    const uint16_t* __restrict__ scales = R.scales[z];
    void* y = R.y[z];
    const int out = R.out[z], rows_pad = R.rows_pad[z];
    __shared__ float red[8][32];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int j = w & (wpr - 1), rg = w - j;     // rg: first warp of the row group
    const int r = blockIdx.x * (256 / wpr) + (rg / wpr) * 32 + lane, t = blockIdx.y;
    const bool lead = j == 0 && r < out;
    uint16_t sc = 0;
    if (static_weights && lead) sc = scales[r];
    pdl_wait();                 // the product kernel's partials
    pdl_launch_dependents();
    if (!static_weights && lead) sc = scales[r];
    float sum = 0.0f;
    if (r < out) {
        const size_t step = (size_t)wpr * batch * rows_pad;   // plane p to plane p + wpr
        const float* p = partials + ((size_t)j * batch + t) * rows_pad + r;
#pragma unroll 1
        for (int q = j; q < P; q += 16 * wpr, p += 16 * step) {
            float v[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = q + i * wpr < P ? __ldcg(p + i * step) : 0.0f;
#pragma unroll
            for (int i = 0; i < 16; ++i) sum += v[i];
        }
    }
    if (wpr > 1) {
        red[w][lane] = sum;
        __syncthreads();
        if (lead)
            for (int i = 1; i < wpr; ++i) sum += red[w + i][lane];
    }
    if (lead) {
        float v = sum * bits_to_f32<SDT>(sc);
        const size_t yi = (size_t)t * out + r;
        if (y_prev)
            v = (y_dt == AQ_F32 ? ((const float*)y_prev)[yi]
                                : bits_to_f32_rt(((const uint16_t*)y_prev)[yi], y_dt)) + v;
        if (y_dt == AQ_F32) ((float*)y)[yi] = v;
        else ((uint16_t*)y)[yi] = y_dt == AQ_F16 ? f32_to_bits<AQ_F16>(v) : f32_to_bits<AQ_BF16>(v);
    }
}

// ------------------------------------------------------------------ 4-bit codes, one token

// y = x W_m^T for one token with 4-bit codes in one kernel (no split-K partials): a CTA owns
// 32 rows (lane L is row 32*blockIdx.x + L) and its warp w walks the slices w, w+8, ... For a
// slice the warp first builds the tables T_k[j][g] = x_g . C_k[j] of every book k < m (16
// entries x 32 groups, 2 KiB per book): lane g computes group g's 16m entries from its own
// eight activations. Then each lane reads its row's 16-byte code unit per book and adds one
// table entry per code; position p of row o holds group (p + o) mod 32, so at every step the
// 32 lanes read 32 different groups, word g of a 128-byte table row: no bank conflicts. At the
// end the warps' sums are added in a fixed order (warp 0, 1, ...), scaled by s[o] and, for a
// refinement, added to y_prev in fp32 before the one rounding to y's type.
// Warps per CTA: 16 while their tables fit (up to six books), else 8.
inline int lut4_warps(int m) { return m <= 6 ? 16 : 8; }

template <int BDT, int XDT, int SDT>
__global__ void __launch_bounds__(512)
gemv_lut4_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
                 const uint16_t* __restrict__ scales, const uint16_t* __restrict__ x, void* y,
                 int y_dt, const void* y_prev, int m, int out, int in, int ng, int S,
                 int rows_pad, size_t plane_bytes) {
    // [warps][m][16][32] tables, [warps][32] sums, [m][16] codewords
    extern __shared__ __align__(16) float t4[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    float* T = t4 + (size_t)warp * m * 512;
    float* red = t4 + (size_t)nw * m * 512;
    uint4* books_s = (uint4*)(red + nw * 32);
    const int o = blockIdx.x * 32 + lane;
    pdl_wait();
    pdl_launch_dependents();
    for (int i = threadIdx.x; i < m * 16; i += blockDim.x) books_s[i] = __ldg((const uint4*)books + i);
    __syncthreads();
    // four accumulators (code words q = 0..3 of a unit) keep the adds independent
    float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    for (int s = warp; s < S; s += nw) {
        // the row's code units of this slice, requested before the tables are built
        uint4 u[8];
#pragma unroll
        for (int k = 0; k < 8; ++k)
            if (k < m) u[k] = ld_stream_v4(planes + (size_t)k * plane_bytes + ((size_t)s * rows_pad + o) * 16);
        const int g = s * 32 + lane;                 // this lane's group for the table build
        float xv[8];
        if (g < ng) unpack8<XDT>(__ldg((const uint4*)(x + (size_t)g * 8)), xv);
        else
#pragma unroll
            for (int e = 0; e < 8; ++e) xv[e] = 0.0f;
        __syncwarp();                                // the previous slice's lookups are done
        for (int k = 0; k < m; ++k) {
            uint4 cw[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) cw[j] = books_s[k * 16 + j];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                float c[8];
                unpack8<BDT>(cw[j], c);
                float t = xv[0] * c[0];
#pragma unroll
                for (int e = 1; e < 8; ++e) t = fmaf(xv[e], c[e], t);
                T[(k * 16 + j) * 32 + lane] = t;
            }
        }
        __syncwarp();
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            if (k >= m) break;
            const uint32_t wd[4] = {u[k].x, u[k].y, u[k].z, u[k].w};
            const float* Tk = T + k * 512;
#pragma unroll
            for (int b = 0; b < 8; ++b)              // position p = 8q + b: nibble b of word q
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int p = 8 * q + b;
                    const uint32_t j = (wd[q] >> (4 * b)) & 15u;
                    acc[q] += Tk[j * 32 + ((p + lane) & 31)];
                }
        }
    }
    red[warp * 32 + lane] = (acc[0] + acc[1]) + (acc[2] + acc[3]);
    __syncthreads();
    if (warp == 0 && o < out) {
        float sum = 0.0f;
        for (int w = 0; w < nw; ++w) sum += red[w * 32 + lane];
        float v = sum * bits_to_f32<SDT>(scales[o]);
        if (y_prev)
            v = (y_dt == AQ_F32 ? ((const float*)y_prev)[o]
                                : bits_to_f32_rt(((const uint16_t*)y_prev)[o], y_dt)) + v;
        if (y_dt == AQ_F32) ((float*)y)[o] = v;
        else ((uint16_t*)y)[o] = y_dt == AQ_F16 ? f32_to_bits<AQ_F16>(v) : f32_to_bits<AQ_BF16>(v);
    }
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

// The table-lookup product for n layers sharing the activations (n = 1: an ordinary call):
// layer l's dims ds[l], pointers as[l] (x, batch and the status word are taken from as[0]).
// Returns AQ_ERR_UNSUPPORTED without launching when a group cannot be served by one launch
// (a CTA's items would reach into more than two layers).
template <int BDT, int XDT, int NT>
aq_status run_lut_layers(const Dims* ds, const GemvArgs* as, int n, int m, cudaStream_t st) {
    DeviceInfo di;
    if (aq_status e = device_info(&di); e != AQ_OK) return e;
    auto kern = gemv_lut_kernel<BDT, XDT, NT, false>;
    if constexpr (NT == 1) {                    // groups: one token only
        if (n > 1) kern = gemv_lut_kernel<BDT, XDT, NT, true>;
    } else if (n > 1) {
        return AQ_ERR_UNSUPPORTED;
    }
    const int nsets = n > 1 ? 2 : 1;
    // As many 32 KiB ring slots as fit next to the tables, codebooks and activations (<= 4).
    const size_t fixed = lut_smem_bytes(NT, m, 0, nsets) + 8192;   // + static shared memory and slack
    int nslots = di.smem_optin > (int)fixed ? (int)((di.smem_optin - fixed) / kSlot) : 0;
    if (nslots > kSlots) nslots = kSlots;
    if (nslots < 2) return AQ_ERR_UNSUPPORTED;
    const size_t smem = lut_smem_bytes(NT, m, nslots, nsets);
    int occ = 0;
    if (aq_status e = prepare(kern, smem, kLutThreads, m * nsets, &occ); e != AQ_OK) return e;
    LutLayers L = {};
    L.n = n;
    long long items = 0;
    for (int l = 0; l < n; ++l) {
        L.planes[l] = (const uint8_t*)as[l].planes;
        L.books[l] = (const uint16_t*)as[l].books;
        L.partials[l] = as[l].partials;
        L.plane_bytes[l] = ds[l].plane_bytes;
        L.rows_pad[l] = ds[l].rows_pad;
        L.RBc[l] = ds[l].RBc;
        L.base[l] = (int)items;
        items += (long long)ds[l].S * m * ds[l].RBc;
        if (items > 0x7fffffffLL) return AQ_ERR_UNSUPPORTED;   // item indices are 32-bit
    }
    L.base[n] = (int)items;
    const Dims& d = ds[0];
    const long long units = (long long)d.S * m;       // (slice, book) pairs of one layer
    // One CTA per SM at most. Two ways to share the items of a single layer: whole shares of
    // single units (cpu CTAs per unit, one table build each), or an even split of all items
    // over the SMs, where a CTA may straddle units and build two or more tables. Every call
    // waits for its slowest CTA, so the choice takes the smaller worst-CTA cost, one table
    // build being worth kTableItems row blocks of streaming (about 0.8 us against 23 ns per
    // 1 KiB block at the per-SM share of HBM bandwidth). A group always takes the even split.
    // In the whole-share form a grid of more than kLutCpuMaxCtas CTAs costs about 0.6 us more
    // (kGridItems / NT row blocks of NT-token lookups): one CTA on each of 144 SMs measured
    // slower than 128 or 96 CTAs with larger shares (4096 x 4096 at m = 3: 6.60 against
    // 5.85 us with two CTAs per unit; 14336 x 4096 at m = 1: 6.33 against 5.55 us with
    // eight), unless the larger shares cost more (14336 x 4096 at m = 3: 10.17 against
    // 11.19 us; four tokens, 4096 x 4096 at m = 3: 10.7 against 12.2 us).
    constexpr long long kTableItems = 35;
    constexpr long long kLutCpuMaxCtas = 128, kGridItems = 25;
    long long cpu = 0, cost_cpu = -1;
    if (n == 1)
        for (long long c = 1; c * units <= di.sms && c <= d.RBc; ++c) {
            const long long cost = kTableItems + (d.RBc + c - 1) / c +
                                   (c * units > kLutCpuMaxCtas ? kGridItems / NT : 0);
            if (cost_cpu < 0 || cost < cost_cpu) {
                cost_cpu = cost;
                cpu = c;
            }
        }
    const long long grid_b = items < di.sms ? items : di.sms;
    const long long qb = items / grid_b, rb = items % grid_b;
    long long cost_b = 0;
    if (n == 1)
        for (long long b = 0; b < grid_b; ++b) {
            const long long i0 = b * qb + (b < rb ? b : rb), i1 = i0 + qb + (b < rb ? 1 : 0);
            const long long tables = (i1 - 1) / d.RBc - i0 / d.RBc + 1;
            const long long c = tables * kTableItems + (i1 - i0);
            if (c > cost_b) cost_b = c;
        }
    else
        for (int l = 0; l < n; ++l)   // a CTA (at most qb + 1 items) then meets at most two layers
            if ((long long)ds[l].S * m * ds[l].RBc < qb + 1) return AQ_ERR_UNSUPPORTED;
    int grid, q, r;   // a CTA's share: q items, one more for the first r shares
    if (cost_cpu >= 0 && cost_cpu <= cost_b) {
        grid = (int)(cpu * units);
        q = d.RBc / (int)cpu;
        r = d.RBc % (int)cpu;
    } else {
        cpu = 0;
        grid = (int)grid_b;
        q = (int)qb;
        r = (int)rb;
    }
    return launch_pdl(kern, dim3(grid), dim3(kLutThreads), smem, st, L, (const uint16_t*)as[0].x,
                      as[0].status, m, d.in, d.ng, nslots, (int)cpu, q, r,
                      (d.flags & AQ_LAYOUT_STATIC_WEIGHTS) ? 1 : 0, as[0].batch);
}

template <int BDT, int XDT, int NT>
aq_status run_lut(const Dims& d, int m, const GemvArgs& a, cudaStream_t st) {
    return run_lut_layers<BDT, XDT, NT>(&d, &a, 1, m, st);
}

// One pass of gemv_lut8 over tokens [t_base, t_base + 8): the work split of run_lut.
template <int BDT, int XDT>
aq_status run_lut8(const Dims& d, int m, const GemvArgs& a, int t_base, cudaStream_t st) {
    DeviceInfo di;
    if (aq_status e = device_info(&di); e != AQ_OK) return e;
    auto kern = gemv_lut8_kernel<BDT, XDT>;
    const size_t fixed = lut8_smem_bytes(m, 0) + 8192;
    int nslots = di.smem_optin > (int)fixed ? (int)((di.smem_optin - fixed) / kSlot) : 0;
    if (nslots > kSlots) nslots = kSlots;
    if (nslots < 2) return AQ_ERR_UNSUPPORTED;
    const size_t smem = lut8_smem_bytes(m, nslots);
    int occ = 0;
    if (aq_status e = prepare(kern, smem, kLutThreads, m, &occ); e != AQ_OK) return e;
    const long long units = (long long)d.S * m;
    const long long items = units * d.RBc;
    if (items > 0x7fffffffLL) return AQ_ERR_UNSUPPORTED;
    // An 8-token table build costs about eight times a one-token build.
    constexpr long long kTableItems = 280;
    long long cpu = di.sms / units;
    if (cpu > d.RBc) cpu = d.RBc;
    long long cost_cpu = -1;
    if (cpu >= 1) cost_cpu = kTableItems + (d.RBc + cpu - 1) / cpu;
    const long long grid_b = items < di.sms ? items : di.sms;
    const long long qb = items / grid_b, rb = items % grid_b;
    long long cost_b = 0;
    for (long long b = 0; b < grid_b; ++b) {
        const long long i0 = b * qb + (b < rb ? b : rb), i1 = i0 + qb + (b < rb ? 1 : 0);
        const long long tables = (i1 - 1) / d.RBc - i0 / d.RBc + 1;
        const long long c = tables * kTableItems + (i1 - i0);
        if (c > cost_b) cost_b = c;
    }
    int grid, q, r;
    if (cost_cpu >= 0 && cost_cpu <= cost_b) {
        grid = (int)(cpu * units);
        q = d.RBc / (int)cpu;
        r = d.RBc % (int)cpu;
    } else {
        cpu = 0;
        grid = (int)grid_b;
        q = (int)qb;
        r = (int)rb;
    }
    return launch_pdl(kern, dim3(grid), dim3(kLutThreads), smem, st, (const uint8_t*)a.planes,
                      (const uint16_t*)a.books, (const uint16_t*)a.x, a.partials, a.status, m,
                      d.in, d.ng, d.rows_pad, d.RBc, d.plane_bytes, nslots, (int)cpu, q, r,
                      (d.flags & AQ_LAYOUT_STATIC_WEIGHTS) ? 1 : 0, a.batch, t_base);
}

template <int BDT, int XDT>
aq_status run_lut8_all(const Dims& d, int m, const GemvArgs& a, cudaStream_t st) {
    for (int t = 0; t < a.batch; t += 8)
        if (aq_status e = run_lut8<BDT, XDT>(d, m, a, t, st); e != AQ_OK) return e;
    return AQ_OK;
}

template <int NB, int B, int BDT, int SDT>
aq_status run_direct(const Dims& d, int m, const GemvArgs& a, cudaStream_t st) {
    DeviceInfo di;
    if (aq_status e = device_info(&di); e != AQ_OK) return e;
    const size_t smem = (size_t)NB * 1024 + staged_books_bytes(B, m) +
                        (size_t)8 * m * 32 * unit_bytes(B);
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

template <int BDT, int XDT, int MB>
aq_status run_gather16(const Dims& d, const GemvArgs& a, cudaStream_t st) {
    DeviceInfo di;
    if (aq_status e = device_info(&di); e != AQ_OK) return e;
    auto kern = gemv_gather16_kernel<BDT, XDT, MB>;
    int occ = 0;
    if (aq_status e = prepare(kern, 0, kG16Warps * 32, MB, &occ); e != AQ_OK) return e;
    const int target = di.sms * occ;
    int chunks = (target + d.S - 1) / d.S;
    chunks = chunks < 1 ? 1 : (chunks > d.RBc ? d.RBc : chunks);
    const int rbpc = (d.RBc + chunks - 1) / chunks;
    chunks = (d.RBc + rbpc - 1) / rbpc;
    return launch_pdl(kern, dim3(chunks, d.S), dim3(kG16Warps * 32), 0, st,
                      (const uint8_t*)a.planes, (const uint16_t*)a.books, (const uint16_t*)a.x,
                      a.partials, d.in, d.rows_pad, d.RBc, rbpc, d.plane_bytes);
}

template <int NT, int BDT, int MB>
aq_status run_mma(const Dims& d, const GemvArgs& a, cudaStream_t st) {
    DeviceInfo di;
    if (aq_status e = device_info(&di); e != AQ_OK) return e;
    const size_t smem = mma_smem_bytes(NT, MB);
    auto kern = gemv_mma_kernel<NT, BDT, MB>;
    int occ = 0;
    if (aq_status e = prepare(kern, smem, 256, 0, &occ); e != AQ_OK) return e;
    const int target = di.sms * occ;
    int chunks = (target + d.S - 1) / d.S;
    chunks = chunks < 1 ? 1 : (chunks > d.RBc ? d.RBc : chunks);
    const int rbpc = (d.RBc + chunks - 1) / chunks;
    chunks = (d.RBc + rbpc - 1) / rbpc;
    return launch_pdl(kern, dim3(chunks, d.S), dim3(256), smem, st, (const uint8_t*)a.planes,
                      (const uint16_t*)a.books, (const uint16_t*)a.x, a.x_dt, a.partials, a.batch,
                      d.in, d.rows_pad, d.RBc, rbpc, d.plane_bytes);
}

template <int NT, int BDT>
aq_status dispatch_mma_nt(const Dims& d, int m, const GemvArgs& a, cudaStream_t st) {
    switch (m) {
        case 1: return run_mma<NT, BDT, 1>(d, a, st);
        case 2: return run_mma<NT, BDT, 2>(d, a, st);
        case 3: return run_mma<NT, BDT, 3>(d, a, st);
        case 4: return run_mma<NT, BDT, 4>(d, a, st);
        case 5: return run_mma<NT, BDT, 5>(d, a, st);
        case 6: return run_mma<NT, BDT, 6>(d, a, st);
        case 7: return run_mma<NT, BDT, 7>(d, a, st);
        default: return run_mma<NT, BDT, 8>(d, a, st);
    }
}

template <int BDT>
aq_status dispatch_mma(const Dims& d, int m, const GemvArgs& a, cudaStream_t st) {
    return a.batch <= 8 ? dispatch_mma_nt<1, BDT>(d, m, a, st) : dispatch_mma_nt<2, BDT>(d, m, a, st);
}

template <int B, int BDT, int SDT>
aq_status dispatch_direct(const Dims& d, int m, const GemvArgs& a, cudaStream_t st) {
    if constexpr (B == 16) {
        if (a.batch == 1 && m <= 2) {   // 2^16-entry books, one token: gathers in flight
            const bool xb = a.x_dt == AQ_BF16;
            if (m == 1) return xb ? run_gather16<BDT, AQ_BF16, 1>(d, a, st) : run_gather16<BDT, AQ_F16, 1>(d, a, st);
            return xb ? run_gather16<BDT, AQ_BF16, 2>(d, a, st) : run_gather16<BDT, AQ_F16, 2>(d, a, st);
        }
    }
    if (a.batch <= 1) return run_direct<1, B, BDT, SDT>(d, m, a, st);
    if (a.batch <= 2) return run_direct<2, B, BDT, SDT>(d, m, a, st);
    if (a.batch <= 4) return run_direct<4, B, BDT, SDT>(d, m, a, st);
    if (a.batch <= 8) return run_direct<8, B, BDT, SDT>(d, m, a, st);
    return run_direct<16, B, BDT, SDT>(d, m, a, st);
}

}  // namespace

template <int BDT, int XDT, int SDT>
aq_status run_lut4(const Dims& d, int m, const void* planes, const void* books,
                   const void* scales, const void* x, void* y, int y_dt, const void* y_prev,
                   cudaStream_t st) {
    const int nw = lut4_warps(m);
    const size_t smem = ((size_t)nw * m * 512 + nw * 32) * 4 + (size_t)m * 16 * 16;
    auto kern = gemv_lut4_kernel<BDT, XDT, SDT>;
    int occ = 0;
    if (aq_status e = prepare(kern, smem, nw * 32, m, &occ); e != AQ_OK) return e;
    return launch_pdl(kern, dim3(d.RBc), dim3(nw * 32), smem, st, (const uint8_t*)planes,
                      (const uint16_t*)books, (const uint16_t*)scales, (const uint16_t*)x, y,
                      y_dt, y_prev, m, d.out, d.in, d.ng, d.S, d.rows_pad, d.plane_bytes);
}

// 4-bit codes, one token: the whole product in one kernel (tables per slice and warp).
static aq_status launch_lut4(const Dims& d, int m, const void* planes, const void* books,
                             const void* scales, const void* x, int x_dt, void* y, int y_dt,
                             const void* y_prev, cudaStream_t st) {
    const int key = (d.book_dt == AQ_BF16) * 4 + (x_dt == AQ_BF16) * 2 + (d.scale_dt == AQ_BF16);
    switch (key) {
        case 0: return run_lut4<AQ_F16, AQ_F16, AQ_F16>(d, m, planes, books, scales, x, y, y_dt, y_prev, st);
        case 1: return run_lut4<AQ_F16, AQ_F16, AQ_BF16>(d, m, planes, books, scales, x, y, y_dt, y_prev, st);
        case 2: return run_lut4<AQ_F16, AQ_BF16, AQ_F16>(d, m, planes, books, scales, x, y, y_dt, y_prev, st);
        case 3: return run_lut4<AQ_F16, AQ_BF16, AQ_BF16>(d, m, planes, books, scales, x, y, y_dt, y_prev, st);
        case 4: return run_lut4<AQ_BF16, AQ_F16, AQ_F16>(d, m, planes, books, scales, x, y, y_dt, y_prev, st);
        case 5: return run_lut4<AQ_BF16, AQ_F16, AQ_BF16>(d, m, planes, books, scales, x, y, y_dt, y_prev, st);
        case 6: return run_lut4<AQ_BF16, AQ_BF16, AQ_F16>(d, m, planes, books, scales, x, y, y_dt, y_prev, st);
        default: return run_lut4<AQ_BF16, AQ_BF16, AQ_BF16>(d, m, planes, books, scales, x, y, y_dt, y_prev, st);
    }
}

// The product kernel of aq_gemv: fp32 partial sums per (slice, token, row) into the workspace.
static aq_status launch_product(const Dims& d, int m, const void* planes, const void* books,
                                const void* scales, const void* x, int x_dt, int batch, void* y,
                                int y_dt, void* ws, cudaStream_t st) {
    if (d.out == 0 || batch == 0) return AQ_OK;
    GemvArgs a{planes, books, scales, x, x_dt, batch, y, y_dt,
               (float*)((char*)ws + ws_partial_offset(d)), (unsigned int*)ws};
    const int bb = d.book_dt == AQ_BF16, xb = x_dt == AQ_BF16, sb = d.scale_dt == AQ_BF16;
    if (uses_lut(d, m, batch)) {
        if (batch == 1) {
            switch (bb * 2 + xb) {
                case 0: return run_lut<AQ_F16, AQ_F16, 1>(d, m, a, st);
                case 1: return run_lut<AQ_F16, AQ_BF16, 1>(d, m, a, st);
                case 2: return run_lut<AQ_BF16, AQ_F16, 1>(d, m, a, st);
                default: return run_lut<AQ_BF16, AQ_BF16, 1>(d, m, a, st);
            }
        }
        if (batch == 2) {
            switch (bb * 2 + xb) {
                case 0: return run_lut<AQ_F16, AQ_F16, 2>(d, m, a, st);
                case 1: return run_lut<AQ_F16, AQ_BF16, 2>(d, m, a, st);
                case 2: return run_lut<AQ_BF16, AQ_F16, 2>(d, m, a, st);
                default: return run_lut<AQ_BF16, AQ_BF16, 2>(d, m, a, st);
            }
        }
        if (batch > 4) {
            switch (bb * 2 + xb) {
                case 0: return run_lut8_all<AQ_F16, AQ_F16>(d, m, a, st);
                case 1: return run_lut8_all<AQ_F16, AQ_BF16>(d, m, a, st);
                case 2: return run_lut8_all<AQ_BF16, AQ_F16>(d, m, a, st);
                default: return run_lut8_all<AQ_BF16, AQ_BF16>(d, m, a, st);
            }
        }
        switch (bb * 2 + xb) {
            case 0: return run_lut<AQ_F16, AQ_F16, 4>(d, m, a, st);
            case 1: return run_lut<AQ_F16, AQ_BF16, 4>(d, m, a, st);
            case 2: return run_lut<AQ_BF16, AQ_F16, 4>(d, m, a, st);
            default: return run_lut<AQ_BF16, AQ_BF16, 4>(d, m, a, st);
        }
    }
    if (d.B == 8 && batch >= 2 && m <= kMmaMaxM)
        return bb ? dispatch_mma<AQ_BF16>(d, m, a, st) : dispatch_mma<AQ_F16>(d, m, a, st);
    if (d.B == 4) {
        switch (bb * 2 + sb) {
            case 0: return dispatch_direct<4, AQ_F16, AQ_F16>(d, m, a, st);
            case 1: return dispatch_direct<4, AQ_F16, AQ_BF16>(d, m, a, st);
            case 2: return dispatch_direct<4, AQ_BF16, AQ_F16>(d, m, a, st);
            default: return dispatch_direct<4, AQ_BF16, AQ_BF16>(d, m, a, st);
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

// P partial planes per token: one per (slice, book) for the LUT kernel, one per slice for the
// direct kernel.
// The reduction of n layers (P partial planes per row and token in each), one launch.
template <int SDT>
static aq_status launch_reduce_layers(const Dims* ds, const GemvArgs* as, int n, int P,
                                      const void* y_prev, int static_weights, cudaStream_t st) {
    int occ = 0;
    auto kern = n > 1 ? splitk_reduce_kernel<SDT, true> : splitk_reduce_kernel<SDT, false>;
    if (aq_status e = prepare(kern, 0, 256, 0, &occ); e != AQ_OK) return e;
    // Warps per 32-row group: one while a warp's sixteen loads cover the planes (no shared
    // memory step, a small grid), else eight (measured: 1 at P = 16, 8 at P >= 32 are the
    // fastest choices on the layer shapes of the benchmark).
    const int wpr = P <= 16 ? 1 : 8;
    const int rows_per_cta = 256 / wpr;
    ReduceLayers R = {};
    int out_max = 0;
    for (int l = 0; l < n; ++l) {
        R.partials[l] = as[l].partials;
        R.scales[l] = (const uint16_t*)as[l].scales;
        R.y[l] = as[l].y;
        R.out[l] = ds[l].out;
        R.rows_pad[l] = ds[l].rows_pad;
        if (ds[l].out > out_max) out_max = ds[l].out;
    }
    return launch_pdl(kern, dim3((out_max + rows_per_cta - 1) / rows_per_cta, as[0].batch, n), dim3(256), 0,
                      st, R, as[0].y_dt, P, as[0].batch, wpr, static_weights, y_prev);
}

template <int SDT>
static aq_status launch_reduce(const Dims& d, int P, const GemvArgs& a, const void* y_prev,
                               cudaStream_t st) {
    return launch_reduce_layers<SDT>(&d, &a, 1, P, y_prev,
                                     (d.flags & AQ_LAYOUT_STATIC_WEIGHTS) ? 1 : 0, st);
}

aq_status launch_gemv(const Dims& d, int m, const void* planes, const void* books,
                      const void* scales, const void* x, int x_dt, int batch, void* y,
                      int y_dt, void* ws, cudaStream_t st, const void* y_prev) {
    if (d.out == 0 || batch == 0) return AQ_OK;
    if (d.B == 4 && batch == 1)
        return launch_lut4(d, m, planes, books, scales, x, x_dt, y, y_dt, y_prev, st);
    if (aq_status e = launch_product(d, m, planes, books, scales, x, x_dt, batch, y, y_dt, ws, st);
        e != AQ_OK)
        return e;
    GemvArgs a{planes, books, scales, x, x_dt, batch, y, y_dt,
               (float*)((char*)ws + ws_partial_offset(d)), (unsigned int*)ws};
    const int P = uses_lut(d, m, batch) ? d.S * m : d.S;
    return d.scale_dt == AQ_BF16 ? launch_reduce<AQ_BF16>(d, P, a, y_prev, st)
                                 : launch_reduce<AQ_F16>(d, P, a, y_prev, st);
}

// aq_gemv_group: n layers that share the activations x. ws[l] is layer l's workspace region
// (status word and partial planes, laid out as for aq_gemv). At batch 1 with 2^8-entry books
// the n products are one launch of the table-lookup kernel (the items of all layers in one
// numbering) and the n reductions one launch; otherwise, or when a CTA's items would reach
// into more than two layers, the layers run as n ordinary calls. Either way each layer's
// partial sums and their order are those of its own call, so the results are identical.
aq_status launch_gemv_group(const Dims* ds, int n, int m, const void* const* planes,
                            const void* const* books, const void* const* scales, const void* x,
                            int x_dt, int batch, void* const* y, int y_dt, void* const* ws,
                            cudaStream_t st) {
    if (batch == 0) return AQ_OK;
    bool any_rows = false;
    for (int l = 0; l < n; ++l) any_rows |= ds[l].out > 0;
    if (!any_rows) return AQ_OK;
    bool fused = n >= 2 && batch == 1 && uses_lut(ds[0], m, 1);
    for (int l = 0; l < n && fused; ++l) fused = ds[l].out > 0;
    if (fused) {
        Dims dd[kGroupMax];
        GemvArgs as[kGroupMax];
        int flags = AQ_LAYOUT_STATIC_WEIGHTS;
        for (int l = 0; l < n; ++l) {
            dd[l] = ds[l];
            flags &= ds[l].flags;
            as[l] = GemvArgs{planes[l], books[l], scales[l], x, x_dt, batch, y[l], y_dt,
                             (float*)((char*)ws[l] + ws_partial_offset(ds[l])), (unsigned int*)ws[0]};
        }
        dd[0].flags = flags;   // prefetch before the grid wait only if every layer's weights are static
        const int bb = ds[0].book_dt == AQ_BF16, xb = x_dt == AQ_BF16;
        aq_status e;
        switch (bb * 2 + xb) {
            case 0: e = run_lut_layers<AQ_F16, AQ_F16, 1>(dd, as, n, m, st); break;
            case 1: e = run_lut_layers<AQ_F16, AQ_BF16, 1>(dd, as, n, m, st); break;
            case 2: e = run_lut_layers<AQ_BF16, AQ_F16, 1>(dd, as, n, m, st); break;
            default: e = run_lut_layers<AQ_BF16, AQ_BF16, 1>(dd, as, n, m, st); break;
        }
        if (e == AQ_OK) {
            const int P = ds[0].S * m, sw = flags ? 1 : 0;
            return ds[0].scale_dt == AQ_BF16 ? launch_reduce_layers<AQ_BF16>(dd, as, n, P, nullptr, sw, st)
                                             : launch_reduce_layers<AQ_F16>(dd, as, n, P, nullptr, sw, st);
        }
        if (e != AQ_ERR_UNSUPPORTED) return e;   // nothing was launched for UNSUPPORTED
    }
    for (int l = 0; l < n; ++l)
        if (aq_status e = launch_gemv(ds[l], m, planes[l], books[l], scales[l], x, x_dt, batch, y[l],
                                      y_dt, ws[l], st, nullptr);
            e != AQ_OK)
            return e;
    return AQ_OK;
}

}  // namespace aq
