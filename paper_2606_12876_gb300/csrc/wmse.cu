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
// Kernels (in stream order):
//   wmse_prep_kernel   P from H (fp32 or bf16, any square matrix; only its symmetric part is
//                      used), bf16, lower block triangle only, into the workspace.
//   wmse_resid_kernel  E_k for every prefix, written once to the workspace in bf16
//                      ([M][d_out][d_in]): per (row, group) the codewords are summed in book
//                      order in fp32 and each prefix's E_k = W - s*sum is rounded once. Every
//                      contraction tile needs E_k again (each row block meets every block of
//                      t), so decoding it once and streaming it through L2 costs one HBM pass
//                      instead of a shared-memory decode per tile.
//   wmse_kernel        one CTA pair per tile of 256 values of t (rows of P) x 256 rows of E,
//                      for two prefixes (one pass; all passes in one grid). TMA brings per
//                      stage a 128 x 64 tile of P and, in one 3-D box, the CTA's 128 x 64
//                      tiles of E_k for both prefixes (128-byte swizzle). Pair MMAs
//                      (tcgen05.mma.cta_group::2, kind::f16, bf16 operands, M = 256, N = 256,
//                      K = 16) accumulate Z^T, one 256-column tensor-memory accumulator per
//                      prefix (512 columns). N = 256 reads each P slab for 256 rows of E, which
//                      keeps the shared-memory traffic per MMA (operand reads plus TMA writes)
//                      well under the port's bandwidth; with four prefixes of N = 128 it was
//                      the limit. Epilogue: TMA brings the tile's E_k[o][t] (256 x 128 per
//                      prefix) into the freed ring, each thread (one t) multiplies it with its
//                      accumulator row and the CTA sums per prefix into the workspace.
//   wmse_reduce_kernel sums the per-CTA partial sums in a fixed order, divides by d_out,
//                      and forms L.
// Every mbarrier wait is bounded; a timeout records AQ_ERR_TIMEOUT in the workspace status word.
#include <cstring>
#include <mutex>

#include "aq_internal.cuh"
#include "tc_ptx.cuh"

namespace aq {
namespace {

constexpr int kWBM = 128;          // values of t (rows of P) per CTA; M = 256 per pair
constexpr int kWTB = 2 * kWBM;     // t per pair tile, and the block size of the folding
constexpr int kWRows = 128;        // rows of E per CTA (its half of the MMA's N)
constexpr int kWBN = 2 * kWRows;   // rows of E per pair tile (N of the MMA)
constexpr int kWBK = 64;           // inputs per stage
constexpr int kWThreads = 384;
constexpr int kWEpi0 = 4, kWEpiWarps = 8;
constexpr int kWMaxPf = 2;         // prefixes per pass: 2 accumulators x 256 columns
constexpr int kWStages = 4;
constexpr int kWGroup = 4;         // row blocks per group of the tile order

// Shared-memory map (identical in both CTAs of a pair: the pair MMA reads the peer's operands
// at the same offsets). The epilogue reuses the ring for the E patches.
constexpr int kWAStage = kWBM * 128;               // 128 rows of P x 64 inputs, 16 KiB
constexpr int kWBTile = kWRows * 128;              // 128 rows of one E_k x 64 inputs, 16 KiB
constexpr int kWStage = kWAStage + kWMaxPf * kWBTile;   // 48 KiB
constexpr int kWOffBar = kWStages * kWStage;
// full, empty, ready (per stage), acc_full, patch_full
constexpr int kWNumBars = 3 * kWStages + 2;
constexpr int kWOffTmem = kWOffBar + kWNumBars * 8;
constexpr int kWOffAbort = kWOffTmem + 16;
constexpr int kWOffRed = kWOffAbort + 16;          // [8 warps][2 prefixes] floats
constexpr int kWSmem = kWOffRed + kWEpiWarps * kWMaxPf * 4;
constexpr int kWPatch = kWBN * kWBM * 2;           // one prefix's E_k[o][t] patch, 64 KiB
static_assert(kWSmem <= 227 * 1024, "shared memory map exceeds the per-CTA limit");
static_assert(kWMaxPf * kWPatch <= kWOffBar, "epilogue patches must fit in the ring");

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

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int c0, int c1,
                                            int c2, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_u32(dst)),
        "l"((uint64_t)map), "r"(c0), "r"(c1), "r"(c2), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ uint32_t bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *(uint32_t*)&h;
}

// ---------------------------------------------------------------- E_k = W - W^(k), bf16
// Each warp owns one 32-row block of one 256-input slice: lane L stages its row's codes of the
// M planes in shared memory, then the warp walks the 32 rows with lane L producing group
// s*32 + L of the row, so every store of a prefix is 512 contiguous bytes.
constexpr int kRWarps = 8;

template <int B, int BDT, int SDT>
__global__ void __launch_bounds__(kRWarps * 32)
wmse_resid_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
                  const uint16_t* __restrict__ scales, const uint16_t* __restrict__ w,
                  uint16_t* __restrict__ e_out, int M, int out, int in, int ng, int rows_pad,
                  int RBc, size_t plane_bytes) {
    constexpr int UNIT = unit_bytes(B);              // bytes of one (row, slice) code unit
    extern __shared__ __align__(16) unsigned char smem[];
    uint16_t* books_s = (uint16_t*)smem;             // B <= 8: [M][2^B][8]
    const size_t books_bytes = staged_books_bytes(B, M);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    unsigned char* codes_s = smem + books_bytes + (size_t)warp * M * 32 * UNIT;
    pdl_wait();
    pdl_launch_dependents();
    if constexpr (B <= 8) {
        const uint4* src = (const uint4*)books;
        uint4* dst = (uint4*)books_s;
        for (int i = threadIdx.x; i < (M << B); i += blockDim.x) dst[i] = src[i];
    }
    const int s = blockIdx.y;
    const int rb = blockIdx.x * kRWarps + warp;
    const bool active = rb < RBc;
    if (active) {
        const int o = rb * 32 + lane;
        for (int k = 0; k < M; ++k) {
            const uint4* src = (const uint4*)(planes + k * plane_bytes + ((size_t)s * rows_pad + o) * UNIT);
            uint4* dst = (uint4*)(codes_s + ((size_t)k * 32 + lane) * UNIT);
#pragma unroll
            for (int q = 0; q < UNIT / 16; ++q) dst[q] = ld_stream_v4(src + q);
        }
    }
    __syncthreads();
    if (!active) return;
    const int g = s * 32 + lane;
    if (g >= ng) return;
    const size_t plane_e = (size_t)out * in;
    constexpr int kAhead = 4;                        // rows whose W loads are in flight together
    for (int r0 = 0; r0 < 32; r0 += kAhead) {
        uint4 wq[kAhead];
#pragma unroll
        for (int j = 0; j < kAhead; ++j) {
            const int o = rb * 32 + r0 + j;
            wq[j] = o < out ? ld_stream_v4(w + (size_t)o * in + (size_t)g * 8) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int j = 0; j < kAhead; ++j) {
        const int r = r0 + j, o = rb * 32 + r;
        if (o >= out) break;
        const float sc = bits_to_f32<SDT>(scales[o]);
        const int p = (lane - r) & 31;               // position of group `lane` in row o
        float wv[8], acc[8];
        unpack8<BDT>(wq[j], wv);
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = -0.0f;
        for (int k = 0; k < M; ++k) {
            const uint32_t code = unit_code<B>(codes_s + ((size_t)k * 32 + r) * UNIT, p);
            uint4 cw;
            if constexpr (B <= 8) cw = ((const uint4*)books_s)[(k << B) + code];
            else cw = __ldg((const uint4*)books + ((size_t)k << 16) + code);
            add_widen2<BDT>(cw.x, acc[0], acc[1]);
            add_widen2<BDT>(cw.y, acc[2], acc[3]);
            add_widen2<BDT>(cw.z, acc[4], acc[5]);
            add_widen2<BDT>(cw.w, acc[6], acc[7]);
            float ev[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) ev[e] = wv[e] - sc * acc[e];
            *(uint4*)(e_out + (size_t)k * plane_e + (size_t)o * in + (size_t)g * 8) =
                make_uint4(bf16x2(ev[0], ev[1]), bf16x2(ev[2], ev[3]), bf16x2(ev[4], ev[5]),
                           bf16x2(ev[6], ev[7]));
        }
        }
    }
}

// ---------------------------------------------------------------- the contraction
// All passes in one grid: pass q covers prefixes 2q+1 and 2q+2 (E_k planes 2q, 2q+1; the
// second absent when M is odd), with its own set of tiles.
__global__ void __launch_bounds__(kWThreads, 1)
wmse_kernel(const __grid_constant__ CUtensorMap pmap, const __grid_constant__ CUtensorMap emap,
            const __grid_constant__ CUtensorMap patch_map, float* __restrict__ partials,
            unsigned int* __restrict__ status, int M, int out, int in, int tblocks,
            int oblocks) {
    extern __shared__ __align__(1024) unsigned char smem[];
    uint64_t* bars = (uint64_t*)(smem + kWOffBar);
    uint64_t* full = bars;                       // this CTA's P and E tiles of the stage landed
    uint64_t* empty = bars + kWStages;           // the pair MMAs reading the stage completed
    uint64_t* ready = empty + kWStages;          // (leader) both CTAs' halves landed
    uint64_t* acc_full = ready + kWStages;
    uint64_t* patch_full = acc_full + 1;
    uint32_t* tmem_slot = (uint32_t*)(smem + kWOffTmem);
    float* red = (float*)(smem + kWOffRed);
    volatile int& s_abort = *(volatile int*)(smem + kWOffAbort);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t rank = cluster_rank() & 1u;  // 0: leader (issues the MMAs), 1: peer
    // Tile order: groups of kWGroup row blocks (the E rows that the resident tiles stream stay
    // few enough to be reused from L2 by the tiles of the other t-blocks), heaviest t-block
    // first within a group (the K range of t-block tb is (tb + 1) * 256 inputs), so the tail
    // of the grid is made of short tiles.
    const int tiles = tblocks * oblocks;
    const int pass = (blockIdx.x >> 1) / tiles;
    const int K0 = pass * kWMaxPf;                // first E_k plane of the pass
    const int npf = min(kWMaxPf, M - K0);         // prefixes of the pass
    const int pi = (blockIdx.x >> 1) - pass * tiles;
    const int grp = pi / (kWGroup * tblocks);
    const int gsz = min(kWGroup, oblocks - grp * kWGroup);
    const int rr = pi - grp * kWGroup * tblocks;
    const int tb = tblocks - 1 - rr / gsz;
    const int n0 = (grp * kWGroup + rr % gsz) * kWBN;   // first row of E of the pair tile
    const int rd0 = n0 + (int)rank * kWRows;     // first row of this CTA's E operand
    const int ta0 = tb * kWTB + (int)rank * kWBM;   // first t of this CTA
    const int nk = (min((tb + 1) * kWTB, in) + kWBK - 1) / kWBK;   // K steps
    // The E box always spans kWMaxPf planes (a plane past M is filled with zeros).
    constexpr uint32_t kStageBytes = kWStage;

    if (smem_u32(smem) & 1023u) {
        if (tid == 0) record_status(status, AQ_ERR_ALIGNMENT);
        return;
    }
    if (tid == 0) {
        for (int s = 0; s < kWStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
            mbar_init(&ready[s], 2);             // the leader's relay and the peer's relay
        }
        mbar_init(acc_full, 1);
        mbar_init(patch_full, 1);
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
        // ---------------- producer: per stage the P tile of this CTA's 128 values of t and,
        // in one 3-D box, its 64 rows of E_k for the pass's prefixes
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&pmap) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&emap) : "memory");
            int issued = 0;
            for (int it = 0; it < nk; ++it) {
                const int st = it % kWStages;
                if (it >= kWStages &&
                    !wait_or_abort(&empty[st], ((it / kWStages) - 1) & 1, &s_abort, status))
                    break;
                mbar_arrive_expect_tx(&full[st], kStageBytes);
                unsigned char* a = smem + st * kWStage;
                tma_load_2d(a, &pmap, it * kWBK, ta0, &full[st]);
                tma_load_3d(a + kWAStage, &emap, it * kWBK, rd0, K0, &full[st]);
                ++issued;
            }
            for (int j = max(0, issued - kWStages); j < issued; ++j)
                mbar_wait(&full[j % kWStages], (j / kWStages) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0 && rank == 0) {
            // ---------------- MMA issuer (leader)
            // kind::f16 instruction descriptor: fp32 accumulator, bf16 A and B, both K-major,
            // N = 256, M = 256 (pair).
            const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) |
                                   ((uint32_t)(kWBN >> 3) << 17) | ((uint32_t)((2 * kWBM) >> 4) << 24);
            for (int it = 0; it < nk; ++it) {
                const int st = it % kWStages;
                if (s_abort || !mbar_wait_cluster(&ready[st], (it / kWStages) & 1)) {
                    record_status(status, AQ_ERR_TIMEOUT);
                    s_abort = 1;
                    break;
                }
                tc_fence_after();
                const uint32_t a0 = smem_u32(smem + st * kWStage);
                const uint32_t b0 = a0 + kWAStage;
                for (int p = 0; p < npf; ++p)
#pragma unroll
                    for (int kk = 0; kk < kWBK / 16; ++kk)
                        umma_f16_pair(tmem + p * kWBN, umma_desc_sw128(a0 + kk * 32),
                                      umma_desc_sw128(b0 + p * kWBTile + kk * 32), idesc,
                                      (it > 0 || kk > 0) ? 1u : 0u);
                umma_commit_pair(&empty[st], (uint16_t)0x3u);
            }
            umma_commit_pair(acc_full, (uint16_t)0x3u);
        } else if (lane == 0) {
            // ---------------- relay (peer): its half of a stage landed
            const uint32_t leader_ready = map_to_rank(smem_u32(ready), 0);
            for (int it = 0; it < nk; ++it) {
                const int st = it % kWStages;
                if (!wait_or_abort(&full[st], (it / kWStages) & 1, &s_abort, status)) break;
                mbar_arrive_cluster(leader_ready + st * 8);
            }
        }
    } else if (warp == 2) {
        if (lane == 0 && rank == 0) {
            // ---------------- relay (leader): its half of a stage landed
            for (int it = 0; it < nk; ++it) {
                const int st = it % kWStages;
                if (!wait_or_abort(&full[st], (it / kWStages) & 1, &s_abort, status)) break;
                mbar_arrive(&ready[st]);
            }
        }
    } else if (warp >= kWEpi0) {
        // ---------------- epilogue
        const int et = tid - kWEpi0 * 32;        // 0..255
        const bool done = __all_sync(0xffffffffu, wait_or_abort(acc_full, 0, &s_abort, status));
        tc_fence_after();
        // (1) E_k[o][t] for the tile's 128 rows and this CTA's 128 values of t, one 32 KiB box
        // per prefix, into the ring (no MMA or copy touches it any more).
        if (et == 0) {
            if (done) {
                mbar_arrive_expect_tx(patch_full, (uint32_t)(npf * kWPatch));
                for (int p = 0; p < npf; ++p)
                    tma_load_3d(smem + p * kWPatch, &patch_map, ta0, n0, K0 + p, patch_full);
            } else {
                mbar_arrive(patch_full);
            }
        }
        const bool have = __all_sync(0xffffffffu, wait_or_abort(patch_full, 0, &s_abort, status)) && done;
        // (2) sum over the tile of Z^T[t, o] * E_k[o, t]: thread = one t (tensor-memory lane),
        // half the rows of the tile.
        const int qd = warp & 3;                       // tensor-memory lane quarter
        const int h = (warp - kWEpi0) >> 2;            // rows 128h .. 128h + 127 of the tile
        const int tl = qd * 32 + lane;
        float sum[kWMaxPf];
#pragma unroll
        for (int p = 0; p < kWMaxPf; ++p) {
            sum[p] = 0.0f;
            if (!have || p >= npf) continue;
            for (int oc = 0; oc < kWRows; oc += 16) {
                float z[16];
                tmem_ld16(tmem + ((uint32_t)(qd * 32) << 16) + p * kWBN + h * kWRows + oc, z);
                const unsigned char* pe = smem + p * kWPatch + (h * kWRows + oc) * (kWBM * 2) + tl * 2;
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const float e = __uint_as_float((uint32_t)(*(const uint16_t*)(pe + i * (kWBM * 2))) << 16);
                    sum[p] = fmaf(z[i], e, sum[p]);
                }
            }
        }
#pragma unroll
        for (int p = 0; p < kWMaxPf; ++p) {
            float v = sum[p];
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
            if (lane == 0) red[(warp - kWEpi0) * kWMaxPf + p] = v;
        }
        named_barrier(1, kWEpiWarps * 32);
        if (et < npf) {     // one entry per (CTA of the pass, prefix): written exactly once
            float v = 0.0f;
            for (int wi = 0; wi < kWEpiWarps; ++wi) v += red[wi * kWMaxPf + et];
            partials[(size_t)(blockIdx.x - pass * 2 * tiles) * M + K0 + et] = v;
        }
    }

    // ---------------- teardown (the pair MMAs touch both CTAs)
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
// times 1 below the block diagonal and 1/2 on it, rounded once to bf16. One 64 x 64 tile per
// CTA; the transposed operand is staged through shared memory. Rows are read four values at a
// time (n is a multiple of 8, so a row of four never crosses the end of a row).
template <int HDT>
__global__ void __launch_bounds__(256) wmse_prep_kernel(const void* __restrict__ h,
                                                        uint16_t* __restrict__ P, int n) {
    __shared__ float tr[64][65];
    const int kt = blockIdx.x, tt = blockIdx.y;
    pdl_wait();
    pdl_launch_dependents();
    if ((kt * 64) / kWTB > (tt * 64) / kWTB) return;   // above the block diagonal: never read
    const bool diag = (kt * 64) / kWTB == (tt * 64) / kWTB;
    auto ld4 = [&](long idx, float* v) {              // four consecutive values of H
        if constexpr (HDT == AQ_F32) {
            const float4 q = *(const float4*)((const float*)h + idx);
            v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
        } else {
            const uint2 q = *(const uint2*)((const uint16_t*)h + idx);
            v[0] = __uint_as_float(q.x << 16); v[1] = __uint_as_float(q.x & 0xffff0000u);
            v[2] = __uint_as_float(q.y << 16); v[3] = __uint_as_float(q.y & 0xffff0000u);
        }
    };
    const int x4 = (threadIdx.x & 15) * 4, y0 = threadIdx.x >> 4;   // 16 x 16 threads
    float a[4][4], b[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {                     // rows y0 + 16i of both tiles
        const int y = y0 + 16 * i;
        const int k = kt * 64 + y, t = tt * 64 + x4;  // H[k][t..t+3]
        if (k < n && t < n) ld4((long)k * n + t, a[i]);
        else a[i][0] = a[i][1] = a[i][2] = a[i][3] = 0.0f;
        const int t2 = tt * 64 + y, k2 = kt * 64 + x4;   // H[t2][k2..k2+3]
        if (t2 < n && k2 < n) ld4((long)t2 * n + k2, b[i]);
        else b[i][0] = b[i][1] = b[i][2] = b[i][3] = 0.0f;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) tr[y0 + 16 * i][x4 + j] = a[i][j];   // tr[k][t]
    __syncthreads();
#pragma unroll
    for (int i = 0; i < 4; ++i) {                     // P[t][k..k+3], t = tt*64 + y
        const int y = y0 + 16 * i;
        const int t = tt * 64 + y, k = kt * 64 + x4;
        if (t >= n || k >= n) continue;
        float v[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            v[j] = b[i][j] + tr[x4 + j][y];
            if (diag) v[j] *= 0.5f;
        }
        *(uint2*)(P + (long)t * n + k) = make_uint2(bf16x2(v[0], v[1]), bf16x2(v[2], v[3]));
    }
}

struct Lambda {
    double v[8];
};

// d[k] = (sum over CTAs of partials[c][k]) / d_out; d[M] = L. Fixed order: each thread adds
// its CTAs' entries (fp32), a shuffle tree adds the 32 lanes of each warp (fp32), one thread
// adds the 8 warps in fp64 (the fp64 pipe of this GPU is slow, so the wide part stays fp32:
// for 2 x 512 entries the fp32 tree adds about 10 roundings of 2^-24 relative to the sum of
// magnitudes).
__global__ void __launch_bounds__(256) wmse_reduce_kernel(const float* __restrict__ partials,
                                                          int nctas, int M, double inv_out,
                                                          Lambda lam, int has_lambda,
                                                          double* __restrict__ d) {
    __shared__ float red[8][8];
    pdl_wait();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float s[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) s[k] = 0.0f;
    for (int c = threadIdx.x; c < nctas; c += 256) {
        float v[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) v[k] = k < M ? partials[(size_t)c * M + k] : 0.0f;
#pragma unroll
        for (int k = 0; k < 8; ++k) s[k] += v[k];
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) s[k] += __shfl_xor_sync(0xffffffffu, s[k], off);
        if (lane == 0) red[warp][k] = s[k];
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double loss = 0.0;
        for (int k = 0; k < M; ++k) {
            double t = 0.0;
            for (int w = 0; w < 8; ++w) t += (double)red[w][k];
            const double dk = t * inv_out;
            d[k] = dk;
            loss += lam.v[k] * dk;
        }
        if (has_lambda) d[M] = loss;
    }
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

aq_status encode(CUtensorMap* map, const void* base, int rank, const cuuint64_t* dims,
                 const cuuint64_t* strides, const cuuint32_t* box, CUtensorMapSwizzle swz) {
    EncodeTiledFn enc;
    if (aq_status e = get_encode_fn(&enc); e != AQ_OK) return e;
    std::memset(map, 0, sizeof(*map));
    const cuuint32_t estr[3] = {1, 1, 1};
    // bf16 tiles moved as 16-bit words (the MMA and the epilogue read the bits as bf16).
    if (enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT16, (cuuint32_t)rank, const_cast<void*>(base), dims,
            strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return AQ_ERR_CUDA;
    return AQ_OK;
}

template <int B, int BDT, int SDT>
aq_status run_resid(const Dims& d, const void* w, const void* planes, const void* books,
                    const void* scales, uint16_t* E, cudaStream_t st) {
    const size_t smem = staged_books_bytes(B, d.M) + (size_t)kRWarps * d.M * 32 * unit_bytes(B);
    auto kern = wmse_resid_kernel<B, BDT, SDT>;
    if (smem > 48 * 1024)
        if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)smem);
            e != cudaSuccess)
            return cuda_fail(e, "cudaFuncSetAttribute");
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    cfg.gridDim = dim3((d.RBc + kRWarps - 1) / kRWarps, d.S);
    cfg.blockDim = dim3(kRWarps * 32);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    launch_cfg(&cfg, attr, 1);
    return cuda_ok(cudaLaunchKernelEx(&cfg, kern, (const uint8_t*)planes, (const uint16_t*)books,
                                      (const uint16_t*)scales, (const uint16_t*)w, E, d.M, d.out,
                                      d.in, d.ng, d.rows_pad, d.RBc, d.plane_bytes),
                   "cudaLaunchKernelEx");
}

aq_status launch_resid(const Dims& d, const void* w, const void* planes, const void* books,
                       const void* scales, uint16_t* E, cudaStream_t st) {
    const int key = (d.B == 16) * 4 + (d.book_dt == AQ_BF16) * 2 + (d.scale_dt == AQ_BF16);
    if (d.B == 4) {
        switch (key) {
            case 0: return run_resid<4, AQ_F16, AQ_F16>(d, w, planes, books, scales, E, st);
            case 1: return run_resid<4, AQ_F16, AQ_BF16>(d, w, planes, books, scales, E, st);
            case 2: return run_resid<4, AQ_BF16, AQ_F16>(d, w, planes, books, scales, E, st);
            default: return run_resid<4, AQ_BF16, AQ_BF16>(d, w, planes, books, scales, E, st);
        }
    }
    switch (key) {
        case 0: return run_resid<8, AQ_F16, AQ_F16>(d, w, planes, books, scales, E, st);
        case 1: return run_resid<8, AQ_F16, AQ_BF16>(d, w, planes, books, scales, E, st);
        case 2: return run_resid<8, AQ_BF16, AQ_F16>(d, w, planes, books, scales, E, st);
        case 3: return run_resid<8, AQ_BF16, AQ_BF16>(d, w, planes, books, scales, E, st);
        case 4: return run_resid<16, AQ_F16, AQ_F16>(d, w, planes, books, scales, E, st);
        case 5: return run_resid<16, AQ_F16, AQ_BF16>(d, w, planes, books, scales, E, st);
        case 6: return run_resid<16, AQ_BF16, AQ_F16>(d, w, planes, books, scales, E, st);
        default: return run_resid<16, AQ_BF16, AQ_BF16>(d, w, planes, books, scales, E, st);
    }
}

aq_status run_contraction(const Dims& d, const uint16_t* P, const uint16_t* E, float* partials,
                          unsigned int* status, cudaStream_t st) {
    const int tblocks = (d.in + kWTB - 1) / kWTB, oblocks = (d.out + kWBN - 1) / kWBN;
    CUtensorMap pmap;
    {
        const cuuint64_t dims[2] = {(cuuint64_t)d.in, (cuuint64_t)d.in};
        const cuuint64_t strides[1] = {(cuuint64_t)d.in * 2};
        const cuuint32_t box[2] = {(cuuint32_t)kWBK, (cuuint32_t)kWBM};
        if (aq_status e = encode(&pmap, P, 2, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B); e != AQ_OK)
            return e;
    }
    const cuuint64_t edims[3] = {(cuuint64_t)d.in, (cuuint64_t)d.out, (cuuint64_t)d.M};
    const cuuint64_t estrides[2] = {(cuuint64_t)d.in * 2, (cuuint64_t)d.out * d.in * 2};
    CUtensorMap patch_map;
    {
        const cuuint32_t box[3] = {(cuuint32_t)kWBM, (cuuint32_t)kWBN, 1};
        if (aq_status e = encode(&patch_map, E, 3, edims, estrides, box, CU_TENSOR_MAP_SWIZZLE_NONE);
            e != AQ_OK)
            return e;
    }
    CUtensorMap emap;
    {
        const cuuint32_t box[3] = {(cuuint32_t)kWBK, (cuuint32_t)kWRows, (cuuint32_t)kWMaxPf};
        if (aq_status e = encode(&emap, E, 3, edims, estrides, box, CU_TENSOR_MAP_SWIZZLE_128B); e != AQ_OK)
            return e;
    }
    static std::mutex mu;
    static bool attr_done[64] = {};
    int dev = 0;
    if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    {
        std::lock_guard<std::mutex> lock(mu);
        if (dev >= 0 && dev < 64 && !attr_done[dev]) {
            if (cudaError_t e = cudaFuncSetAttribute(wmse_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kWSmem);
                e != cudaSuccess)
                return cuda_fail(e, "cudaFuncSetAttribute");
            attr_done[dev] = true;
        }
    }
    const int passes = (d.M + kWMaxPf - 1) / kWMaxPf;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    cfg.gridDim = dim3(2 * passes * tblocks * oblocks);
    cfg.blockDim = dim3(kWThreads);
    cfg.dynamicSmemBytes = kWSmem;
    cfg.stream = st;
    launch_cfg(&cfg, attr, 2);
    if (aq_status e = cuda_ok(cudaLaunchKernelEx(&cfg, wmse_kernel, pmap, emap, patch_map, partials,
                                                 status, d.M, d.out, d.in, tblocks, oblocks),
                              "cudaLaunchKernelEx");
        e != AQ_OK)
        return e;
    return AQ_OK;
}

// Workspace: [status, 1 KiB][P: d_in^2 bf16][E: M * d_out * d_in bf16][partials: CTAs x M fp32]
size_t p_bytes(const Dims& d) { return round_up((size_t)d.in * d.in * 2, 1024); }
size_t e_bytes(const Dims& d) { return round_up((size_t)d.M * d.out * d.in * 2, 1024); }

}  // namespace

size_t wmse_ws_bytes(const Dims& d) {
    const size_t tb = (size_t)(d.in + kWTB - 1) / kWTB, ob = (size_t)(d.out + kWBN - 1) / kWBN;
    return 1024 + p_bytes(d) + e_bytes(d) + 2 * tb * ob * d.M * 4;   // partials: CTAs of one pass
}

aq_status launch_wmse(const Dims& d, const void* w, const void* planes, const void* books,
                      const void* scales, const void* h, int h_dt, const double* lambda,
                      double* out_d, void* ws, cudaStream_t st) {
    const size_t out_bytes = (size_t)(d.M + (lambda ? 1 : 0)) * sizeof(double);
    if (d.out == 0) return cuda_ok(cudaMemsetAsync(out_d, 0, out_bytes, st), "cudaMemsetAsync");
    unsigned int* status = (unsigned int*)ws;
    uint16_t* P = (uint16_t*)((char*)ws + 1024);
    uint16_t* E = (uint16_t*)((char*)P + p_bytes(d));
    float* partials = (float*)((char*)E + e_bytes(d));
    const int tblocks = (d.in + kWTB - 1) / kWTB, oblocks = (d.out + kWBN - 1) / kWBN;

    {   // P from H
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[2];
        const int nt = (d.in + 63) / 64;
        cfg.gridDim = dim3(nt, nt);
        cfg.blockDim = dim3(256);
        cfg.stream = st;
        launch_cfg(&cfg, attr, 1);
        const cudaError_t e = h_dt == AQ_F32
                                  ? cudaLaunchKernelEx(&cfg, wmse_prep_kernel<AQ_F32>, h, P, d.in)
                                  : cudaLaunchKernelEx(&cfg, wmse_prep_kernel<AQ_BF16>, h, P, d.in);
        if (aq_status s = cuda_ok(e, "cudaLaunchKernelEx"); s != AQ_OK) return s;
    }
    if (aq_status e = launch_resid(d, w, planes, books, scales, E, st); e != AQ_OK) return e;
    if (aq_status e = run_contraction(d, P, E, partials, status, st); e != AQ_OK) return e;
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
