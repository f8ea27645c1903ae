// aq_wmse: the per-prefix distortion of Drop-by-Drop (Sec. 5) with the weighted MSE of Sec. 2.2
// (Eq. wmse-task, trace form), for every prefix k = 1..M of a packed layer in one call:
//
//     D^(k) = (1/d_out) tr[E_k H E_k^T],   E_k = W - W^(k),   W^(k) = s o sum_{j<k} C_j[b_j],
//
// and, given weights lambda_k, the Drop-by-Drop objective L = sum_k lambda_k D^(k) (Sec. 5).
//
// Symmetric folding. tr[E H E^T] = sum_o e_o H e_o^T depends only on the symmetric part S of H.
// Cut the inputs into blocks of 256 and let P[t][k] = S[t][k] when block(k) < block(t),
// S[t][k] / 2 when block(k) = block(t), and 0 above the block diagonal. Then for every pair of
// blocks the folded weights of (t, k) and (k, t) add up to S[t][k], so
//     e H e^T = sum_t e[t] * sum_{k <= end of block(t)} P[t][k] e[k].
// The inner sums are a contraction Z = E P^T whose K range stops at the end of t's block: the
// tensor-core work is half that of E H, and H is read only through P (bf16).
//
// Kernels:
//   wmse_prep_kernel  P from H (fp32 or bf16, any square matrix; only its symmetric part is
//                     used), written in bf16 into the workspace, lower block triangle only.
//   wmse_kernel       one CTA pair per tile of 256 values of t (H rows) x 128 rows of E.
//                     Pair MMAs (tcgen05.mma.cta_group::2, kind::f16 with bf16 operands,
//                     M = 256 t, N = 128 rows, K = 16) accumulate Z^T for up to four prefixes
//                     at once, one 128-column accumulator per prefix in tensor memory (512
//                     columns). A operand: P rows by TMA (128-byte swizzle). B operand: E_k
//                     decoded in shared memory from W (TMA) and the codes: each decoder thread
//                     owns one row and two groups per stage, sums the codewords of the books in
//                     order (fp32) and writes E_k = W - s*sum for every prefix of the pass,
//                     rounded once to bf16, into that prefix's tile. Epilogue: the E_k values
//                     at (row, t) for the tile are decoded again into shared memory (bf16),
//                     multiplied with the accumulators read from tensor memory and summed per
//                     CTA and prefix into the workspace.
//   wmse_reduce_kernel sums the per-CTA partial sums in a fixed order in fp64, divides by
//                     d_out, and forms L.
// Prefixes beyond four take a second pass of wmse_kernel (books 0..3 are summed again, their
// prefixes are not stored). Every mbarrier wait is bounded; a timeout records AQ_ERR_TIMEOUT
// in the workspace status word.
#include <cstring>
#include <mutex>

#include "aq_internal.cuh"
#include "tc_ptx.cuh"

namespace aq {
namespace {

constexpr int kWBM = 128;          // values of t (rows of P) per CTA; M = 256 per pair
constexpr int kWTB = 2 * kWBM;     // t per pair tile, and the block size of the folding
constexpr int kWRows = 64;         // rows of E decoded by one CTA
constexpr int kWBN = 2 * kWRows;   // rows of E per pair tile (N of the MMA)
constexpr int kWBK = 64;           // inputs per stage
constexpr int kWThreads = 384;
constexpr int kWDec0 = 4, kWDecWarps = 8;
constexpr int kWMaxPf = 4;         // prefixes per pass: 4 accumulators x 128 columns

// Shared-memory map. NB (books summed in the pass) up to 4 in the first pass; the second pass
// (books 5..8) keeps twice the codes and codebooks and shortens the rings.
template <bool BIG>
struct WL {
    static constexpr int kStagesA = BIG ? 3 : 4;
    static constexpr int kStagesB = BIG ? 2 : 3;
    static constexpr int kBooks = BIG ? 8 : 4;
    static constexpr int kPStage = kWBM * 128;           // 128 rows of P x 64 inputs, bf16
    static constexpr int kWStage = kWRows * 128;         // 64 rows of W x 64 inputs, 16-bit
    static constexpr int kAStage = kPStage + kWStage;    // 24 KiB
    static constexpr int kBTile = kWRows * 128;          // one prefix's E tile, 8 KiB
    static constexpr int kBStage = kWMaxPf * kBTile;     // 32 KiB
    static constexpr int kCodeBuf = kBooks * kWRows * 32;
    static constexpr int kOffA = 0;
    static constexpr int kOffB = kOffA + kStagesA * kAStage;
    static constexpr int kOffCodes = kOffB + kStagesB * kBStage;
    static constexpr int kOffBooks = kOffCodes + 2 * kCodeBuf;
    static constexpr int kOffScale = kOffBooks + kBooks * 4096;
    static constexpr int kOffBar = kOffScale + kWRows * 4;
    // full_a, empty_a (per A stage); full_b, empty_b, ready (per B stage); codes_full[2],
    // codes_empty[2], acc_full
    static constexpr int kNumBars = 2 * kStagesA + 3 * kStagesB + 5;
    static constexpr int kOffTmem = kOffBar + kNumBars * 8;
    static constexpr int kOffAbort = kOffTmem + 16;
    static constexpr int kOffRed = kOffAbort + 16;       // [8 warps][4 prefixes] floats
    static constexpr int kSmem = kOffRed + kWDecWarps * kWMaxPf * 4;
    static constexpr int kPatch = kWBN * kWBM * 2;       // one prefix's epilogue E patch, bf16
};
static_assert(WL<false>::kSmem <= 227 * 1024 && WL<true>::kSmem <= 227 * 1024,
              "shared memory map exceeds the per-CTA limit");
static_assert(kWMaxPf * WL<false>::kPatch <= WL<false>::kOffCodes &&
                  kWMaxPf * WL<true>::kPatch <= WL<true>::kOffCodes,
              "epilogue patches must fit in the rings");

// 16 consecutive fp32 columns of this warp's 32 tensor-memory lanes.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
        "%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ uint32_t bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *(uint32_t*)&h;
}

// E = w - s * acc for eight values, rounded once to bf16 (packed, low element first).
__device__ __forceinline__ uint4 residual8(const float (&w)[8], const float (&acc)[8], float s) {
    float e[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) e[i] = w[i] - s * acc[i];
    return make_uint4(bf16x2(e[0], e[1]), bf16x2(e[2], e[3]), bf16x2(e[4], e[5]), bf16x2(e[6], e[7]));
}

// acc += codeword (eight 16-bit values of type BDT at shared address a), exactly widened.
template <int BDT>
__device__ __forceinline__ void add_codeword(uint32_t a, float (&acc)[8]) {
    const uint4 c = lds128(a);
    add_widen2<BDT>(c.x, acc[0], acc[1]);
    add_widen2<BDT>(c.y, acc[2], acc[3]);
    add_widen2<BDT>(c.z, acc[4], acc[5]);
    add_widen2<BDT>(c.w, acc[6], acc[7]);
}

// One pass: books 0..NB-1 are summed; prefixes NB-NPF+1 .. NB (NPF of them) are evaluated.
// BDT is the element type of the codebooks and of W.
template <int BDT, int NB>
__global__ void __launch_bounds__(kWThreads, 1)
wmse_kernel(const __grid_constant__ CUtensorMap pmap, const __grid_constant__ CUtensorMap wmap,
            const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
            const uint16_t* __restrict__ scales, const uint16_t* __restrict__ w,
            float* __restrict__ partials, unsigned int* __restrict__ status, int M, int out,
            int in, int ng, int rows_pad, size_t plane_bytes, int tblocks, int oblocks,
            int scale_dt) {
    constexpr bool BIG = NB > kWMaxPf;
    constexpr int NPF = BIG ? NB - kWMaxPf : NB;
    constexpr int K0 = NB - NPF;                 // books summed before the first evaluated prefix
    using L = WL<BIG>;
    extern __shared__ __align__(1024) unsigned char smem[];
    uint64_t* bars = (uint64_t*)(smem + L::kOffBar);
    uint64_t* full_a = bars;                     // P and W tiles of the stage landed
    uint64_t* empty_a = bars + L::kStagesA;      // the pair MMAs reading the A stage completed
    uint64_t* full_b = empty_a + L::kStagesA;    // (peer) its decoders wrote the E tiles
    uint64_t* empty_b = full_b + L::kStagesB;    // the pair MMAs reading the B stage completed
    uint64_t* ready = empty_b + L::kStagesB;     // (leader) both halves of the stage in place
    uint64_t* codes_full = ready + L::kStagesB;
    uint64_t* codes_empty = codes_full + 2;
    uint64_t* acc_full = codes_empty + 2;
    uint32_t* tmem_slot = (uint32_t*)(smem + L::kOffTmem);
    float* scale_s = (float*)(smem + L::kOffScale);
    uint4* books_s = (uint4*)(smem + L::kOffBooks);
    float* red = (float*)(smem + L::kOffRed);
    volatile int& s_abort = *(volatile int*)(smem + L::kOffAbort);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t rank = cluster_rank() & 1u;  // 0: leader (issues the MMAs), 1: peer
    // Heaviest tiles first: the K range of t-block tb is (tb + 1) * 256 inputs.
    const int pi = blockIdx.x >> 1;
    const int tb = tblocks - 1 - pi / oblocks;
    const int n0 = (pi % oblocks) * kWBN;        // first row of E of the pair tile
    const int t0 = tb * kWTB;                    // first t of the pair tile
    const int rd0 = n0 + (int)rank * kWRows;     // first row decoded by this CTA
    const int ta0 = t0 + (int)rank * kWBM;       // first t of this CTA
    const int kend = min((tb + 1) * kWTB, in);
    const int nk = (kend + kWBK - 1) / kWBK;     // K steps
    const int nsl = (nk + 3) / 4;                // 256-input slices
    const int rows_valid = max(0, min(kWRows, rows_pad - rd0));

    if (smem_u32(smem) & 1023u) {
        if (tid == 0) record_status(status, AQ_ERR_ALIGNMENT);
        return;
    }
    if (tid == 0) {
        for (int s = 0; s < L::kStagesA; ++s) {
            mbar_init(&full_a[s], 1);
            mbar_init(&empty_a[s], 1);
        }
        for (int s = 0; s < L::kStagesB; ++s) {
            mbar_init(&full_b[s], kWDecWarps);
            mbar_init(&empty_b[s], 1);
            mbar_init(&ready[s], kWDecWarps + 2);
        }
        for (int c = 0; c < 2; ++c) {
            mbar_init(&codes_full[c], 1);
            mbar_init(&codes_empty[c], kWDecWarps);
        }
        mbar_init(acc_full, 1);
        mbar_fence_init();
        s_abort = 0;
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(
                         smem_u32(tmem_slot))
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    cluster_sync();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    pdl_wait();

    if (warp == 0) {
        // ---------------- producer: per slice the code rows of the NB planes; per stage the
        // P tile (this CTA's 128 values of t) and the W tile (its 64 rows)
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&pmap) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&wmap) : "memory");
            int issued_a = 0, issued_c = 0;
            bool stop = false;
            for (int sl = 0; sl < nsl && !stop; ++sl) {
                const int cb = sl & 1;
                if (sl >= 2 && !wait_or_abort(&codes_empty[cb], ((sl >> 1) - 1) & 1, &s_abort, status))
                    break;
                mbar_arrive_expect_tx(&codes_full[cb], (uint32_t)(NB * rows_valid * 32));
                if (rows_valid > 0)
                    for (int k = 0; k < NB; ++k)
                        bulk_g2s(smem + L::kOffCodes + cb * L::kCodeBuf + k * (kWRows * 32),
                                 planes + (size_t)k * plane_bytes + ((size_t)sl * rows_pad + rd0) * 32,
                                 (uint32_t)(rows_valid * 32), &codes_full[cb]);
                ++issued_c;
                const int nj = min(4, nk - sl * 4);
                for (int j = 0; j < nj; ++j) {
                    const int it = issued_a, st = it % L::kStagesA;
                    if (it >= L::kStagesA &&
                        !wait_or_abort(&empty_a[st], ((it / L::kStagesA) - 1) & 1, &s_abort, status)) {
                        stop = true;
                        break;
                    }
                    mbar_arrive_expect_tx(&full_a[st], (uint32_t)L::kAStage);
                    unsigned char* a = smem + L::kOffA + st * L::kAStage;
                    const int kx = (sl * 4 + j) * kWBK;
                    tma_load_2d(a, &pmap, kx, ta0, &full_a[st]);
                    tma_load_2d(a + L::kPStage, &wmap, kx, rd0, &full_a[st]);
                    ++issued_a;
                }
            }
            for (int j = max(0, issued_a - L::kStagesA); j < issued_a; ++j)
                mbar_wait(&full_a[j % L::kStagesA], (j / L::kStagesA) & 1);
            for (int j = max(0, issued_c - 2); j < issued_c; ++j)
                mbar_wait(&codes_full[j & 1], (j >> 1) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0 && rank == 0) {
            // ---------------- MMA issuer (leader)
            // kind::f16 instruction descriptor: fp32 accumulator, bf16 A and B, both K-major,
            // N = 128, M = 256 (pair).
            const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) |
                                   ((uint32_t)(kWBN >> 3) << 17) | ((uint32_t)((2 * kWBM) >> 4) << 24);
            for (int it = 0; it < nk; ++it) {
                const int sa = it % L::kStagesA, sb = it % L::kStagesB;
                if (s_abort || !mbar_wait_cluster(&ready[sb], (it / L::kStagesB) & 1)) {
                    record_status(status, AQ_ERR_TIMEOUT);
                    s_abort = 1;
                    break;
                }
                tc_fence_after();
                const uint32_t a0 = smem_u32(smem + L::kOffA + sa * L::kAStage);
                const uint32_t b0 = smem_u32(smem + L::kOffB + sb * L::kBStage);
#pragma unroll
                for (int p = 0; p < NPF; ++p)
#pragma unroll
                    for (int kk = 0; kk < kWBK / 16; ++kk)
                        umma_f16_pair(tmem + p * kWBN, umma_desc_sw128(a0 + kk * 32),
                                      umma_desc_sw128(b0 + p * L::kBTile + kk * 32), idesc,
                                      (it > 0 || kk > 0) ? 1u : 0u);
                umma_commit_pair(&empty_a[sa], (uint16_t)0x3u);
                umma_commit_pair(&empty_b[sb], (uint16_t)0x3u);
            }
            umma_commit_pair(acc_full, (uint16_t)0x3u);
        } else if (lane == 0) {
            // ---------------- relay (peer): this CTA's half of a stage is ready
            const uint32_t leader_ready = map_to_rank(smem_u32(ready), 0);
            for (int it = 0; it < nk; ++it) {
                const int sa = it % L::kStagesA, sb = it % L::kStagesB;
                if (!wait_or_abort(&full_a[sa], (it / L::kStagesA) & 1, &s_abort, status)) break;
                if (!wait_or_abort(&full_b[sb], (it / L::kStagesB) & 1, &s_abort, status)) break;
                mbar_arrive_cluster(leader_ready + sb * 8);
            }
        }
    } else if (warp == 2) {
        if (lane == 0 && rank == 0) {
            // ---------------- P relay (leader): its A stage landed. The A ring is deeper than
            // the stage barrier's ring: before counting stage it, wait until the barrier's
            // previous phase (stage it - kStagesB) is done.
            for (int it = 0; it < nk; ++it) {
                const int sa = it % L::kStagesA, sb = it % L::kStagesB;
                if (it >= L::kStagesB &&
                    !wait_or_abort(&ready[sb], ((it / L::kStagesB) - 1) & 1, &s_abort, status))
                    break;
                if (!wait_or_abort(&full_a[sa], (it / L::kStagesA) & 1, &s_abort, status)) break;
                mbar_arrive(&ready[sb]);
            }
        }
    } else if (warp >= kWDec0) {
        // ---------------- decoders, then epilogue
        const int dt = tid - kWDec0 * 32;        // 0..255
        const int n = dt & (kWRows - 1);         // decoded row owned by the thread
        const int c0 = (dt >> 6) * 2;            // its groups c0, c0 + 1 of every stage
        const int row = rd0 + n;
        for (int i = dt; i < NB * 256; i += kWDecWarps * 32) books_s[i] = __ldg((const uint4*)books + i);
        for (int i = dt; i < kWRows; i += kWDecWarps * 32)
            scale_s[i] = (rd0 + i < out) ? bits_to_f32_rt(scales[rd0 + i], scale_dt) : 0.0f;
        named_barrier(1, kWDecWarps * 32);

        const float s = scale_s[n];
        const int r = row & 31;                  // rotation of this row's codes
        const int rw = r >> 2, rb = (r & 3) * 8;
        const bool row_ok = row < out;
        const uint32_t books_u = smem_u32(books_s);
        const uint32_t b_row = smem_u32(smem + L::kOffB) + (n >> 3) * 1024 + (n & 7) * 128;
        const uint32_t w_row = smem_u32(smem + L::kOffA + L::kPStage) + n * 128;
        int it = 0;
        for (int sl = 0; sl < nsl; ++sl) {
            const int cb = sl & 1;
            // q[k][j]: the word holding the codes (one byte each) of the thread's groups
            // 8j + c0, 8j + c0 + 1 of the slice in plane k (from byte c0 & 3); the front entry
            // always belongs to the next stage.
            uint32_t q[NB][4];
            const bool have = wait_or_abort(&codes_full[cb], (sl >> 1) & 1, &s_abort, status);
#pragma unroll
            for (int k = 0; k < NB; ++k) {
                uint32_t wd[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
                if (have && n < rows_valid) {
                    const uint32_t src = smem_u32(smem + L::kOffCodes + cb * L::kCodeBuf + k * (kWRows * 32) + n * 32);
                    const uint4 lo = lds128_ordered(src), hi = lds128_ordered(src + 16);
                    wd[0] = lo.x; wd[1] = lo.y; wd[2] = lo.z; wd[3] = lo.w;
                    wd[4] = hi.x; wd[5] = hi.y; wd[6] = hi.z; wd[7] = hi.w;
                }
                // Undo the row rotation (position p holds group (p + row) mod 32): words by
                // rw in three conditional steps, then bytes by funnel shifts.
                uint32_t v[8], t[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) t[i] = (rw & 1) ? wd[(i + 7) & 7] : wd[i];
#pragma unroll
                for (int i = 0; i < 8; ++i) v[i] = (rw & 2) ? t[(i + 6) & 7] : t[i];
#pragma unroll
                for (int i = 0; i < 8; ++i) t[i] = (rw & 4) ? v[(i + 4) & 7] : v[i];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const uint32_t cur = (c0 >> 2) ? t[2 * j + 1] : t[2 * j];
                    const uint32_t prev = (c0 >> 2) ? t[2 * j] : t[(2 * j + 7) & 7];
                    q[k][j] = rb ? __funnelshift_l(prev, cur, rb) : cur;
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&codes_empty[cb]);

            const int nj = min(4, nk - sl * 4);
#pragma unroll 1
            for (int j = 0; j < nj; ++j) {
                const int sa = it % L::kStagesA, sb = it % L::kStagesB;
                wait_or_abort(&full_a[sa], (it / L::kStagesA) & 1, &s_abort, status);   // W tile
                if (it >= L::kStagesB)
                    wait_or_abort(&empty_b[sb], ((it / L::kStagesB) - 1) & 1, &s_abort, status);
                const uint32_t bt = b_row + sb * L::kBStage;
                const uint32_t wt = w_row + sa * L::kAStage;
                const int g0 = sl * 32 + j * 8 + c0;
#pragma unroll
                for (int cc = 0; cc < 2; ++cc) {
                    const int c = c0 + cc;
                    const uint32_t sw = (uint32_t)((c ^ (n & 7)) << 4);
                    const bool ok = row_ok && g0 + cc < ng;
                    float wv[8], acc[8];
                    {
                        const uint4 wq = lds128_ordered(wt + sw);
                        widen2<BDT>(wq.x, wv[0], wv[1]);
                        widen2<BDT>(wq.y, wv[2], wv[3]);
                        widen2<BDT>(wq.z, wv[4], wv[5]);
                        widen2<BDT>(wq.w, wv[6], wv[7]);
                    }
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[e] = -0.0f;
#pragma unroll
                    for (int k = 0; k < NB; ++k) {
                        const uint32_t code = (q[k][0] >> (((c0 & 3) + cc) * 8)) & 0xffu;
                        add_codeword<BDT>(books_u + ((uint32_t)k << 12) + (code << 4), acc);
                        if (k >= K0) {
                            uint4 o = residual8(wv, acc, s);
                            if (!ok) o = make_uint4(0u, 0u, 0u, 0u);
                            sts128(bt + (k - K0) * L::kBTile + sw, o);
                        }
                    }
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(rank == 0 ? &ready[sb] : &full_b[sb]);
                ++it;
#pragma unroll
                for (int k = 0; k < NB; ++k) {
                    q[k][0] = q[k][1];
                    q[k][1] = q[k][2];
                    q[k][2] = q[k][3];
                }
            }
        }

        // ---------------- epilogue
        const bool done = __all_sync(0xffffffffu, wait_or_abort(acc_full, 0, &s_abort, status));
        tc_fence_after();
        // (1) E_k at (row o of the pair tile, t of this CTA) for every prefix of the pass,
        // bf16, into [prefix][o][t] over the rings (no MMA or copy reads them any more).
        // Items: 128 rows x 16 groups of t; row and codes read from global memory (L2).
        const int gbase = ta0 >> 3;
        for (int item = dt; item < kWBN * 16; item += kWDecWarps * 32) {
            const int ol = item >> 4, gl = item & 15;
            const int o = n0 + ol, g = gbase + gl;
            uint4 res[NPF];
#pragma unroll
            for (int p = 0; p < NPF; ++p) res[p] = make_uint4(0u, 0u, 0u, 0u);
            if (done && o < out && g < ng) {
                float wv[8], acc[8];
                const uint4 wq = *(const uint4*)(w + (size_t)o * in + (size_t)g * 8);
                widen2<BDT>(wq.x, wv[0], wv[1]);
                widen2<BDT>(wq.y, wv[2], wv[3]);
                widen2<BDT>(wq.z, wv[4], wv[5]);
                widen2<BDT>(wq.w, wv[6], wv[7]);
                const float so = bits_to_f32_rt(scales[o], scale_dt);
                const size_t cpos = ((size_t)(g >> 5) * rows_pad + o) * 32 + (((g & 31) - o) & 31);
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[e] = -0.0f;
#pragma unroll
                for (int k = 0; k < NB; ++k) {
                    const uint32_t code = planes[(size_t)k * plane_bytes + cpos];
                    add_codeword<BDT>(books_u + ((uint32_t)k << 12) + (code << 4), acc);
                    if (k >= K0) res[k - K0] = residual8(wv, acc, so);
                }
            }
#pragma unroll
            for (int p = 0; p < NPF; ++p)
                sts128(smem_u32(smem + p * L::kPatch + ol * (kWBM * 2) + gl * 16), res[p]);
        }
        named_barrier(1, kWDecWarps * 32);
        // (2) sum over the tile of Z^T[t, o] * E_k[o, t]: thread = one t (tensor-memory lane),
        // half the rows of the tile.
        const int qd = warp & 3;                       // tensor-memory lane quarter
        const int h = (warp - kWDec0) >> 2;            // rows 64h .. 64h + 63 of the tile
        const int tl = qd * 32 + lane;
        float sum[NPF];
#pragma unroll
        for (int p = 0; p < NPF; ++p) {
            sum[p] = 0.0f;
            if (!done) continue;
            for (int oc = 0; oc < kWRows; oc += 16) {
                float z[16];
                tmem_ld16(tmem + ((uint32_t)(qd * 32) << 16) + p * kWBN + h * kWRows + oc, z);
                const unsigned char* pe = smem + p * L::kPatch + (h * kWRows + oc) * (kWBM * 2) + tl * 2;
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const float e = __uint_as_float((uint32_t)(*(const uint16_t*)(pe + i * (kWBM * 2))) << 16);
                    sum[p] = fmaf(z[i], e, sum[p]);
                }
            }
        }
#pragma unroll
        for (int p = 0; p < NPF; ++p) {
            float v = sum[p];
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
            if (lane == 0) red[(warp - kWDec0) * kWMaxPf + p] = v;
        }
        named_barrier(1, kWDecWarps * 32);
        if (dt < NPF) {
            float v = 0.0f;
            for (int wi = 0; wi < kWDecWarps; ++wi) v += red[wi * kWMaxPf + dt];
            partials[(size_t)blockIdx.x * M + K0 + dt] = v;
        }
    }

    // ---------------- teardown (as in the GEMM: the pair MMAs touch both CTAs)
    if (warp == 1 && lane == 0 && rank == 0) mbar_wait(acc_full, 0);
    tc_fence_before();
    cluster_sync();
    pdl_launch_dependents();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, 512;" ::"r"(tmem) : "memory");
    }
}

// P from H (n x n), lower block triangle only (blocks of kWTB): P[t][k] = (H[t][k] + H[k][t])
// times 1 below the block diagonal and 1/2 on it, rounded once to bf16. 32 x 32 tiles, the
// transposed operand staged through shared memory.
template <int HDT>
__global__ void __launch_bounds__(256) wmse_prep_kernel(const void* __restrict__ h,
                                                        uint16_t* __restrict__ P, int n) {
    __shared__ float tr[32][33];
    const int kt = blockIdx.x, tt = blockIdx.y;
    pdl_wait();
    pdl_launch_dependents();
    if ((kt * 32) / kWTB > (tt * 32) / kWTB) return;   // above the block diagonal: never read
    const bool diag = (kt * 32) / kWTB == (tt * 32) / kWTB;
    auto ld = [&](long idx) -> float {
        if constexpr (HDT == AQ_F32) return ((const float*)h)[idx];
        else return __uint_as_float((uint32_t)((const uint16_t*)h)[idx] << 16);
    };
    const int x = threadIdx.x & 31, y0 = threadIdx.x >> 5;
    for (int y = y0; y < 32; y += 8) {                 // H[k][t]: k = kt*32 + y, t = tt*32 + x
        const int k = kt * 32 + y, t = tt * 32 + x;
        tr[y][x] = (k < n && t < n) ? ld((long)k * n + t) : 0.0f;
    }
    __syncthreads();
    for (int y = y0; y < 32; y += 8) {                 // P[t][k]: t = tt*32 + y, k = kt*32 + x
        const int t = tt * 32 + y, k = kt * 32 + x;
        if (t < n && k < n) {
            float v = ld((long)t * n + k) + tr[x][y];
            if (diag) v *= 0.5f;
            P[(long)t * n + k] = __bfloat16_as_ushort(__float2bfloat16_rn(v));
        }
    }
}

struct Lambda {
    double v[8];
};

// d[k] = (sum over CTAs of partials[c][k]) / d_out in fp64, in a fixed order; d[M] = L.
__global__ void __launch_bounds__(256) wmse_reduce_kernel(const float* __restrict__ partials,
                                                          int nctas, int M, double inv_out,
                                                          Lambda lam, int has_lambda,
                                                          double* __restrict__ d) {
    __shared__ double red[256];
    pdl_wait();
    double loss = 0.0;
    for (int k = 0; k < M; ++k) {
        double s = 0.0;
        for (int c = threadIdx.x; c < nctas; c += 256) s += (double)partials[(size_t)c * M + k];
        red[threadIdx.x] = s;
        __syncthreads();
        for (int w = 128; w > 0; w >>= 1) {
            if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
            __syncthreads();
        }
        if (threadIdx.x == 0) {
            const double dk = red[0] * inv_out;
            d[k] = dk;
            loss += lam.v[k] * dk;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0 && has_lambda) d[M] = loss;
    pdl_launch_dependents();
}

aq_status launch_cfg(cudaLaunchConfig_t* cfg, cudaLaunchAttribute* attr, int cluster) {
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg->attrs = attr;
    cfg->numAttrs = 1;
    if (cluster > 1) {
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = (unsigned)cluster;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        cfg->numAttrs = 2;
    }
    return AQ_OK;
}

using WKern = void (*)(const CUtensorMap, const CUtensorMap, const uint8_t*, const uint16_t*,
                       const uint16_t*, const uint16_t*, float*, unsigned int*, int, int, int,
                       int, int, size_t, int, int, int);

template <int BDT>
WKern wmse_kernel_for(int nb) {
    switch (nb) {
        case 1: return wmse_kernel<BDT, 1>;
        case 2: return wmse_kernel<BDT, 2>;
        case 3: return wmse_kernel<BDT, 3>;
        case 4: return wmse_kernel<BDT, 4>;
        case 5: return wmse_kernel<BDT, 5>;
        case 6: return wmse_kernel<BDT, 6>;
        case 7: return wmse_kernel<BDT, 7>;
        default: return wmse_kernel<BDT, 8>;
    }
}

aq_status encode_2d(CUtensorMap* map, const void* base, int inner, int rows, int box_inner,
                    int box_rows) {
    EncodeTiledFn encode;
    if (aq_status e = get_encode_fn(&encode); e != AQ_OK) return e;
    std::memset(map, 0, sizeof(*map));
    const cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)inner * 2};
    const cuuint32_t box[2] = {(cuuint32_t)box_inner, (cuuint32_t)box_rows};
    const cuuint32_t estr[2] = {1, 1};
    // bf16 and fp16 tiles are moved as 16-bit words (the kernel reads the bits).
    if (encode(map, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return AQ_ERR_CUDA;
    return AQ_OK;
}

template <int BDT>
aq_status run_wmse(const Dims& d, const void* w, const void* planes, const void* books,
                   const void* scales, const void* P, float* partials, unsigned int* status,
                   cudaStream_t st) {
    const int tblocks = (d.in + kWTB - 1) / kWTB, oblocks = (d.out + kWBN - 1) / kWBN;
    CUtensorMap pmap, wmap;
    if (aq_status e = encode_2d(&pmap, P, d.in, d.in, kWBK, kWBM); e != AQ_OK) return e;
    if (aq_status e = encode_2d(&wmap, w, d.in, d.out, kWBK, kWRows); e != AQ_OK) return e;
    static std::mutex mu;
    static bool attr_done[9][64] = {};
    int dev = 0;
    if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    for (int k0 = 0; k0 < d.M; k0 += kWMaxPf) {
        const int nb = d.M < k0 + kWMaxPf ? d.M : k0 + kWMaxPf;
        const WKern kern = wmse_kernel_for<BDT>(nb);
        const int smem = nb > kWMaxPf ? WL<true>::kSmem : WL<false>::kSmem;
        {
            std::lock_guard<std::mutex> lock(mu);
            if (dev >= 0 && dev < 64 && !attr_done[nb][dev]) {
                if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
                    e != cudaSuccess)
                    return cuda_fail(e, "cudaFuncSetAttribute");
                attr_done[nb][dev] = true;
            }
        }
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[2];
        cfg.gridDim = dim3(2 * tblocks * oblocks);
        cfg.blockDim = dim3(kWThreads);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = st;
        launch_cfg(&cfg, attr, 2);
        if (aq_status e = cuda_ok(cudaLaunchKernelEx(&cfg, kern, pmap, wmap, (const uint8_t*)planes,
                                                     (const uint16_t*)books, (const uint16_t*)scales,
                                                     (const uint16_t*)w, partials, status, d.M, d.out,
                                                     d.in, d.ng, d.rows_pad, d.plane_bytes, tblocks,
                                                     oblocks, d.scale_dt),
                                  "cudaLaunchKernelEx");
            e != AQ_OK)
            return e;
    }
    return AQ_OK;
}

}  // namespace

size_t wmse_p_offset() { return 1024; }

size_t wmse_ws_bytes(const Dims& d) {
    const size_t tb = (size_t)(d.in + kWTB - 1) / kWTB, ob = (size_t)(d.out + kWBN - 1) / kWBN;
    return wmse_p_offset() + round_up((size_t)d.in * d.in * 2, 1024) + 2 * tb * ob * d.M * 4;
}

aq_status launch_wmse(const Dims& d, const void* w, const void* planes, const void* books,
                      const void* scales, const void* h, int h_dt, const double* lambda,
                      double* out_d, void* ws, cudaStream_t st) {
    const size_t out_bytes = (size_t)(d.M + (lambda ? 1 : 0)) * sizeof(double);
    if (d.out == 0) return cuda_ok(cudaMemsetAsync(out_d, 0, out_bytes, st), "cudaMemsetAsync");
    unsigned int* status = (unsigned int*)ws;
    uint16_t* P = (uint16_t*)((char*)ws + wmse_p_offset());
    float* partials = (float*)((char*)P + round_up((size_t)d.in * d.in * 2, 1024));
    const int tblocks = (d.in + kWTB - 1) / kWTB, oblocks = (d.out + kWBN - 1) / kWBN;

    {   // P from H
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[2];
        const int nt = (d.in + 31) / 32;
        cfg.gridDim = dim3(nt, nt);
        cfg.blockDim = dim3(256);
        cfg.stream = st;
        launch_cfg(&cfg, attr, 1);
        const cudaError_t e = h_dt == AQ_F32
                                  ? cudaLaunchKernelEx(&cfg, wmse_prep_kernel<AQ_F32>, h, P, d.in)
                                  : cudaLaunchKernelEx(&cfg, wmse_prep_kernel<AQ_BF16>, h, P, d.in);
        if (aq_status s = cuda_ok(e, "cudaLaunchKernelEx"); s != AQ_OK) return s;
    }
    if (aq_status e = d.book_dt == AQ_BF16
                          ? run_wmse<AQ_BF16>(d, w, planes, books, scales, P, partials, status, st)
                          : run_wmse<AQ_F16>(d, w, planes, books, scales, P, partials, status, st);
        e != AQ_OK)
        return e;
    Lambda lam = {};
    for (int k = 0; k < d.M; ++k) lam.v[k] = lambda ? lambda[k] : 0.0;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    cfg.gridDim = dim3(1);
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    launch_cfg(&cfg, attr, 1);
    return cuda_ok(cudaLaunchKernelEx(&cfg, wmse_reduce_kernel, (const float*)partials,
                                      2 * tblocks * oblocks, d.M, 1.0 / (double)d.out, lam,
                                      lambda ? 1 : 0, out_d),
                   "cudaLaunchKernelEx");
}

}  // namespace aq
