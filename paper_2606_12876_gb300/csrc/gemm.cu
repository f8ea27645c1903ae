// aq_gemm: prefill product y = x * W_m^T for many tokens on the tcgen05 tensor cores, with W_m
// (the prefix-m additive reconstruction of Sec. 3.2 / Sec. 5) decoded tile by tile into shared
// memory and never written to HBM.
//
// A CTA pair (two CTAs, one per SM) computes a 512-token x 256-row tile with pair MMAs
// (tcgen05.mma.cta_group::2, M = 256 tokens, N = 256 rows, K = 16): each CTA holds 128 tokens
// of every A block and 128 of the 256 weight rows, and the MMA reads both halves of both
// operands, so every SM supplies half the operand bytes of what a single-CTA MMA of the same
// work would read from its shared memory. A cluster holds NP = 1, 2 or 4 such pairs with the
// same rows and consecutive token tiles. The CTAs with the same role in the other pairs (the
// partners) need the same 128 weight rows: each of the NP decodes 128/NP of them and sends its
// slab to the others with one shared-memory bulk copy per partner and stage, which divides the
// codeword gathers (the decoders' shared-memory traffic, what bounds the kernel at larger m)
// by NP.
// Each CTA's tensor memory holds its 128 tokens x 256 rows for two token blocks (512 columns).
// Roles (12 warps per CTA):
//   warp 0      TMA producer: activation tiles (2-D tensor map, 128-byte swizzle, two
//               128-token boxes per stage) and, once per 256-input slice, the code rows this
//               CTA decodes, of the first m planes (1-D bulk copies).
//   warp 1      allocates the pair's tensor memory (together with the peer's warp 1). In the
//               leader CTA of a pair lane 0 issues the pair MMAs (2 token blocks x 4 K=16
//               steps per stage) after one barrier wait per stage, and commits the
//               activation-stage release and accumulator-ready barriers to its pair and the
//               weight-stage release to every CTA of the cluster. In the peer CTA lane 0 relays "stage
//               ready" (its activations landed, its weight operand complete) to the leader
//               with a remote mbarrier arrive.
//   warp 2      (leader) lane 0 counts the leader's landed activation stages on the stage
//               barrier.
//   warp 3      lane 0 copies this CTA's decoded slab of each stage to the partners.
//   warps 4-11  decoders: each thread owns one weight row and 4/NP groups of every stage; it
//               sums the m codewords in fp32 (book order), rounds once to fp16 and writes the
//               16-byte group into the B tile in the UMMA K-major 128-byte-swizzle layout.
//               Afterwards the same warps are the epilogue: tcgen05.ld from tensor memory,
//               times the row scale (R1), round; a 16-bit y is staged in the freed operand
//               rings and written by bulk tensor stores (per-thread stores otherwise).
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
#include "tc_ptx.cuh"

namespace aq {
namespace {

constexpr int kBM = 128;                      // tokens per CTA per MMA (M = 256 per pair)
constexpr int kAcc = 2;                       // token blocks (accumulators) per CTA
constexpr int kPairTokens = 2 * kAcc * kBM;   // 512 tokens per pair tile
constexpr int kRows = 128;                    // weight rows decoded by one CTA
constexpr int kBN = 2 * kRows;                // weight rows per pair tile (N of the MMA)
constexpr int kBK = 64;                       // inputs per stage
constexpr int kGemmThreads = 384;
constexpr int kDecWarp0 = 4, kDecWarps = 8;
constexpr int kGemmMaxM = 8;

constexpr int kABlock = kBM * 128;            // one 128-token x 64-input block (16 KiB)
constexpr int kAStage = kAcc * kABlock;       // 32 KiB
constexpr int kBStage = kRows * 128;          // 16 KiB

// Shared-memory map for prefix length MB (offsets from a 1024-byte aligned base; identical in
// both CTAs of a pair, which the pair MMA relies on: it reads the peer's operands at the same
// offsets). One or two books: four activation and four weight stages, room for MB planes of
// codes and MB codebooks; three or four books: three weight stages, room for four of each.
// Longer prefixes need more room for codes and codebooks (MB planes of 128 rows per slice, MB
// codebooks of 4 KiB): the activation ring drops to three stages, and from seven books the
// weight ring to two. The dense form has no codes or books in shared memory: four stages of
// each ring.
template <int MB, bool DENSE = false>
struct GemmLayout {
    static constexpr int kBooks = DENSE ? 0 : MB <= 2 ? MB : MB <= 4 ? 4 : MB;
    static constexpr int kStagesA = DENSE || MB <= 4 ? 4 : 3;
    static constexpr int kStagesB = DENSE || MB <= 2 ? 4 : MB <= 6 ? 3 : 2;
    static constexpr int kCodeBuf = kBooks * kRows * 32;   // one slice of codes, all planes
    static constexpr int kOffA = 0;
    static constexpr int kOffB = kOffA + kStagesA * kAStage;
    static constexpr int kOffCodes = kOffB + kStagesB * kBStage;
    static constexpr int kOffBooks = kOffCodes + 2 * kCodeBuf;
    static constexpr int kOffScale = kOffBooks + kBooks * 4096;
    static constexpr int kOffBar = kOffScale + kBN * 4;
    // full_a, empty_a (per A stage), full_b, empty_b, ready, dec_done (per B stage),
    // codes_full[2], codes_empty[2], acc_full
    static constexpr int kNumBars = 2 * kStagesA + 4 * kStagesB + 4 + 1;
    static constexpr int kOffTmem = kOffBar + kNumBars * 8;
    static constexpr int kOffAbort = kOffTmem + 16;
    static constexpr int kOffWmax = kOffAbort + 16;        // per-book largest |entry| (8 words)
    // The kernel has no static shared memory, so its dynamic shared memory starts on a
    // 1024-byte boundary (checked at run time: the 128-byte swizzled tiles need it).
    static constexpr int kSmem = kOffWmax + 32;
    static_assert(kSmem <= 227 * 1024, "shared memory map exceeds the per-CTA limit");
    // the epilogue's 16-bit staging (eight warps x 32 tokens x 256 rows) reuses the operand rings
    static_assert(kOffCodes - kOffA >= kDecWarps * 32 * kBN * 2, "operand rings too small for y staging");
};

__device__ __forceinline__ uint32_t pack2(float lo, float hi, int dt) {
    if (dt == AQ_BF16) {
        __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
        return *(uint32_t*)&h;
    }
    __half2 h = __floats2half2_rn(lo, hi);
    return *(uint32_t*)&h;
}

__device__ __forceinline__ uint32_t f16x2(float2 v) {   // {lo, hi} -> packed fp16 pair, RN
    uint32_t h;
    asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(h) : "f"(v.y), "f"(v.x));
    return h;
}

// fp16 range for any input (R9). The MMA operands are fp16; bf16 activations and bf16
// codebooks can hold values far outside fp16's range (and fp16 books' sums can exceed it).
// Both are therefore scaled by powers of two, which is exact: each token row of bf16
// activations by 2^-e_t so that its largest |x| lies in [2^14, 2^15) (bf16_rows_to_f16_kernel),
// and the codebooks by 2^-f so that the largest possible |sum of m codewords| (the sum over
// the books of their largest |entry|) lies below 2^15 (for bf16 books also at least 2^14, so
// that small weights do not fall into fp16's subnormal range; fp16 books are only scaled down,
// and a single fp16 book not at all). The epilogue multiplies by 2^(e_t + f). Where nothing
// was out of range the result is bit-identical to the unscaled computation.

// Largest |entry| of a codeword of eight 16-bit values, as the bits of a non-negative float
// (monotonic in the value, so unsigned maxima of them are maxima of the values).
template <int BDT>
__device__ __forceinline__ unsigned int codeword_max_bits(const uint4& c) {
    float f[8];
    unpack8<BDT>(c, f);
    float mx = 0.0f;
#pragma unroll
    for (int e = 0; e < 8; ++e) mx = fmaxf(mx, fabsf(f[e]));
    return __float_as_uint(mx);
}

// f of the codebooks of prefix m from the per-book largest |entry| (float bits).
template <int BDT>
__device__ __forceinline__ int book_exponent(const unsigned int* wmax, int m) {
    if (BDT == AQ_F16 && m == 1) return 0;   // one fp16 codeword is an fp16 value already
    float tot = 0.0f;
    for (int k = 0; k < m; ++k) tot += __uint_as_float(wmax[k]);
    if (!(tot > 0.0f)) return 0;             // all-zero books (or NaN entries)
    int f = exponent_of(fminf(tot, 3.0e38f)) - 14;
    if (BDT == AQ_F16 && f < 0) f = 0;
    return max(-100, min(100, f));
}

// A codeword times sc (a power of two), back in its own type.
template <int BDT>
__device__ __forceinline__ uint4 scale_codeword(const uint4& c, float sc) {
    float f[8];
    unpack8<BDT>(c, f);
    uint16_t h[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) h[e] = f32_to_bits<BDT>(f[e] * sc);
    return make_uint4(h[0] | ((uint32_t)h[1] << 16), h[2] | ((uint32_t)h[3] << 16),
                      h[4] | ((uint32_t)h[5] << 16), h[6] | ((uint32_t)h[7] << 16));
}

// Decoded group (eight fp16 weights): sum of the MB codewords in fp32, in book order, rounded
// once to fp16. code[k] is the group's code in plane k; book k starts at books + k*4096.
template <int BDT, int MB>
__device__ __forceinline__ uint4 decode_group(uint32_t books, const uint32_t (&code)[MB]) {
    const uint4 c0 = lds128(books + (code[0] << 4));
    if constexpr (MB == 1 && BDT == AQ_F16) {
        return c0;   // one fp16 codeword: widening to fp32 and rounding back is exact
    } else {
        // one mixed-type add per element (16-bit operand into the fp32 sum); -0 + v = v
        // exactly, so the first book is widened by the same instruction
        float a[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) a[e] = -0.0f;
        add_widen2<BDT>(c0.x, a[0], a[1]);
        add_widen2<BDT>(c0.y, a[2], a[3]);
        add_widen2<BDT>(c0.z, a[4], a[5]);
        add_widen2<BDT>(c0.w, a[6], a[7]);
#pragma unroll
        for (int k = 1; k < MB; ++k) {
            const uint4 ck = lds128(books + ((uint32_t)k << 12) + (code[k] << 4));
            add_widen2<BDT>(ck.x, a[0], a[1]);
            add_widen2<BDT>(ck.y, a[2], a[3]);
            add_widen2<BDT>(ck.z, a[4], a[5]);
            add_widen2<BDT>(ck.w, a[6], a[7]);
        }
        return make_uint4(f16x2(make_float2(a[0], a[1])), f16x2(make_float2(a[2], a[3])),
                          f16x2(make_float2(a[4], a[5])), f16x2(make_float2(a[6], a[7])));
    }
}

// One instantiation per book type and prefix length MB (= m): the decoders' code holds exactly
// the lookups of that prefix. NP: pairs per cluster (launched with cluster size 2*NP) that
// split the decode of each weight operand between partners; with NP = 1 each CTA decodes its
// own 128 rows. Sharing pays when the gathers bound the kernel (m >= 2) and every pair has
// tokens; larger clusters leave more SMs idle (36 clusters of four, or fewer of eight, fit on
// the 152 SMs), which at m = 1 costs more than the decode they save.
//
// DENSE: the weights were decoded beforehand (dense_w_kernel: fp16 sums of the m codewords,
// the same values the decoders would write) and each CTA's weight tile arrives by TMA (wmap,
// 128-byte swizzle, the layout the decoders write) like the activations; the decoder warps
// only run the epilogue. Instantiated with MB = NP = 1.
template <int BDT, int MB, int NP, bool DENSE = false>
__global__ void __launch_bounds__(kGemmThreads, 1)
gemm_kernel(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap wmap,
            const __grid_constant__ CUtensorMap ymap, int y_tma, const uint8_t* __restrict__ planes,
            const uint16_t* __restrict__ books, const uint16_t* __restrict__ scales, void* y,
            int y_dt, int scale_dt, unsigned int* __restrict__ status,
            const float* __restrict__ xfac, int tokens, int out, int in, int ng, int rows_pad,
            size_t plane_bytes) {
    static_assert(!DENSE || (MB == 1 && NP == 1), "dense tiles: one instantiation");
    using GL = GemmLayout<MB, DENSE>;
    constexpr int kStagesA = GL::kStagesA, kStagesB = GL::kStagesB, kCodeBuf = GL::kCodeBuf;
    constexpr int kOffA = GL::kOffA, kOffB = GL::kOffB, kOffCodes = GL::kOffCodes;
    extern __shared__ __align__(1024) unsigned char smem[];
    uint64_t* bars = (uint64_t*)(smem + GL::kOffBar);
    uint64_t* full_a = bars;                    // this CTA's activation copies landed
    uint64_t* empty_a = bars + kStagesA;        // the pair MMAs reading the A stage completed
    uint64_t* full_b = bars + 2 * kStagesA;     // this CTA's decoders wrote its weight half
    uint64_t* empty_b = full_b + kStagesB;      // the pair MMAs reading the B stage completed
    // ready (leader only): both CTAs' A and B halves of the stage are in place. Arrivals: the
    // leader's decoder warps (or, when sharing, its copier with the partner's bytes), the
    // leader's activation relay and the peer's relay.
    uint64_t* ready = empty_b + kStagesB;
    uint64_t* dec_done = ready + kStagesB;      // this CTA's decoders wrote their half
    uint64_t* codes_full = dec_done + kStagesB;
    uint64_t* codes_empty = codes_full + 2;
    uint64_t* acc_full = codes_empty + 2;
    uint32_t* tmem_slot = (uint32_t*)(smem + GL::kOffTmem);
    float* scale_s = (float*)(smem + GL::kOffScale);
    uint4* books_s = (uint4*)(smem + GL::kOffBooks);
    constexpr int m = MB;
    volatile int& s_abort = *(volatile int*)(smem + GL::kOffAbort);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // rank = role in the pair (0: leader, issues the MMAs; 1: peer). A cluster = NP CTA pairs
    // with the same 256 weight rows and different 512-token tiles; pair = which token tile.
    // The CTAs with the same rank in the other pairs are the partners: all need the same 128
    // weight rows, and each decodes 128/NP of them.
    static_assert(NP == 1 || NP == 2 || NP == 4, "pairs per cluster");
    constexpr bool SHARE = NP > 1;
    constexpr int kClusterLog = NP == 1 ? 1 : NP == 2 ? 2 : 3;
    constexpr int DR = kRows / NP;              // rows decoded by one CTA
    constexpr int kSlab = DR * 128;             // their 64-input slab of a weight stage
    const uint32_t rank4 = cluster_rank();
    const uint32_t rank = rank4 & 1u, pair = SHARE ? rank4 >> 1 : 0u;
    // Tile of the cluster: row tile tn, token tile tt. With decoding in the loop the grid runs
    // all row tiles of one token tile together (blockIdx.x fastest); the dense variant reads
    // 2 bytes of weight per element instead of m/8 of codes, so there the clusters of one row
    // tile run together and its weight tiles are read from HBM once and then from L2.
    int tn, tt;
    if constexpr (DENSE) {
        const int ntt = (int)gridDim.y;
        const int cid = (int)blockIdx.y * (int)(gridDim.x >> kClusterLog) + (int)(blockIdx.x >> kClusterLog);
        tn = cid / ntt;
        tt = cid - tn * ntt;
    } else {
        tn = (int)(blockIdx.x >> kClusterLog);
        tt = (int)blockIdx.y;
    }
    const int n0 = tn * kBN;                    // first output row of the pair tile
    const int r0 = n0 + (int)rank * kRows;      // first row of this CTA's weight operand
    const int rd0 = r0 + (int)pair * DR;        // first row decoded by this CTA
    const int t0 = (tt * NP + (int)pair) * kPairTokens;   // first token
    const int nk = (in + kBK - 1) / kBK;        // K steps
    const int nsl = (nk + 3) / 4;               // 256-input slices
    const int rows_valid = max(0, min(DR, rows_pad - rd0));   // packed rows present
    // Pairs that run at the same time share their token tile; if they all walked K in the same
    // order they would request the same activation lines from L2 at the same moment. Each
    // pair therefore starts at its own 256-input slice and wraps around (only the fp32
    // accumulation order differs). Every role walks the slices in this order; `it` counts
    // stages in processing order and drives the ring.
    const int rot = tn % nsl;                   // the same in both pairs of a cluster

    // Same answer in both CTAs of the pair (identical layouts), so both leave before any
    // cluster-wide step.
    if (smem_u32(smem) & 1023u) {
        if (tid == 0) record_status(status, AQ_ERR_ALIGNMENT);
        return;
    }
    if (tid == 0) {
        for (int s = 0; s < kStagesA; ++s) {
            mbar_init(&full_a[s], 1);             // producer arrival + TMA bytes
            mbar_init(&empty_a[s], 1);            // the leader's multicast commit
        }
        for (int s = 0; s < kStagesB; ++s) {
            // (peer) the copier with the partner's bytes, or the decoder warps
            mbar_init(&full_b[s], (SHARE || DENSE) ? 1 : kDecWarps);
            mbar_init(&empty_b[s], NP);           // commits of the pairs writing the stage
            // (leader) the copier or the decoder warps, plus the two relays
            mbar_init(&ready[s], DENSE ? 2 : SHARE ? 3 : kDecWarps + 2);
            mbar_init(&dec_done[s], kDecWarps);   // (SHARE) one arrival per decoder warp
        }
        for (int c = 0; c < 2; ++c) {
            mbar_init(&codes_full[c], 1);
            mbar_init(&codes_empty[c], kDecWarps);
        }
        mbar_init(acc_full, 1);
        mbar_fence_init();
        s_abort = 0;
    }
    if (warp == 1) {   // tensor memory of the pair: 512 columns in each CTA, allocated jointly
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(
                         smem_u32(tmem_slot))
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    cluster_sync();    // barriers of every CTA initialised before any cross-CTA arrival
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    pdl_wait();

    if (warp == 0) {
        // ---------------- producer
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&xmap) : "memory");
            if constexpr (DENSE) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&wmap) : "memory");
            int issued_a = 0, issued_c = 0;
            bool stop = false;
            for (int js = 0; js < nsl && !stop; ++js) {
                const int sl = rot + js < nsl ? rot + js : rot + js - nsl;
                if constexpr (!DENSE) {
                    const int cb = js & 1;                // codes of slice sl
                    if (js >= 2 && !wait_or_abort(&codes_empty[cb], ((js >> 1) - 1) & 1, &s_abort, status))
                        break;
                    mbar_arrive_expect_tx(&codes_full[cb], (uint32_t)(m * rows_valid * 32));
                    if (rows_valid > 0)
                        for (int k = 0; k < m; ++k)
                            bulk_g2s(smem + kOffCodes + cb * kCodeBuf + k * (DR * 32),
                                     planes + (size_t)k * plane_bytes + ((size_t)sl * rows_pad + rd0) * 32,
                                     (uint32_t)(rows_valid * 32), &codes_full[cb]);
                    ++issued_c;
                }
                const int nj = min(4, nk - sl * 4);
                for (int j = 0; j < nj; ++j) {
                    const int it = issued_a, st = it % kStagesA;
                    if (it >= kStagesA &&
                        !wait_or_abort(&empty_a[st], ((it / kStagesA) - 1) & 1, &s_abort, status)) {
                        stop = true;
                        break;
                    }
                    mbar_arrive_expect_tx(&full_a[st], (uint32_t)kAStage);
                    unsigned char* a = smem + kOffA + st * kAStage;
#pragma unroll
                    for (int i = 0; i < kAcc; ++i)
                        tma_load_2d(a + i * kABlock, &xmap, (sl * 4 + j) * kBK,
                                    t0 + i * 2 * kBM + (int)rank * kBM, &full_a[st]);
                    if constexpr (DENSE) {
                        // this CTA's 128 weight rows of the stage, into the weight ring
                        const int sb = it % kStagesB;
                        if (it >= kStagesB &&
                            !wait_or_abort(&empty_b[sb], ((it / kStagesB) - 1) & 1, &s_abort, status)) {
                            stop = true;
                            ++issued_a;
                            break;
                        }
                        mbar_arrive_expect_tx(&full_b[sb], (uint32_t)kBStage);
                        tma_load_2d(smem + kOffB + sb * kBStage, &wmap, (sl * 4 + j) * kBK, r0, &full_b[sb]);
                    }
                    ++issued_a;
                }
            }
            // No copy may still be in flight when the CTA exits.
            for (int j = max(0, issued_a - kStagesA); j < issued_a; ++j)
                mbar_wait(&full_a[j % kStagesA], (j / kStagesA) & 1);
            if constexpr (DENSE)
                for (int j = max(0, issued_a - kStagesB); j < issued_a; ++j)
                    mbar_wait(&full_b[j % kStagesB], (j / kStagesB) & 1);
            for (int j = max(0, issued_c - 2); j < issued_c; ++j)
                mbar_wait(&codes_full[j & 1], (j >> 1) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0 && rank == 0) {
            // ---------------- MMA issuer (leader)
            // kind::f16 instruction descriptor: fp32 accumulator, fp16 A and B, both K-major,
            // N = 256, M = 256 (pair).
            const uint32_t idesc = (1u << 4) | ((uint32_t)(kBN >> 3) << 17) | ((uint32_t)((2 * kBM) >> 4) << 24);
            for (int it = 0; it < nk; ++it) {
                const int sa = it % kStagesA, sb = it % kStagesB;
                if (s_abort || !mbar_wait_cluster(&ready[sb], (it / kStagesB) & 1)) {
                    record_status(status, AQ_ERR_TIMEOUT);
                    s_abort = 1;
                    break;
                }
                tc_fence_after();
                const uint32_t a0 = smem_u32(smem + kOffA + sa * kAStage);
                const uint32_t b0 = smem_u32(smem + kOffB + sb * kBStage);
#pragma unroll
                for (int i = 0; i < kAcc; ++i)
#pragma unroll
                    for (int kk = 0; kk < kBK / 16; ++kk)
                        umma_f16_pair(tmem + i * kBN, umma_desc_sw128(a0 + i * kABlock + kk * 32),
                                      umma_desc_sw128(b0 + kk * 32), idesc, (it > 0 || kk > 0) ? 1u : 0u);
                // The activation stage belongs to this pair; when sharing, the weight stage is
                // also written by the partners, so its release goes to every CTA of the cluster.
                umma_commit_pair(&empty_a[sa], (uint16_t)(0x3u << (2 * pair)));
                umma_commit_pair(&empty_b[sb], (uint16_t)((1u << (2 * NP)) - 1u));
            }
            umma_commit_pair(acc_full, (uint16_t)(0x3u << (2 * pair)));
        } else if (lane == 0) {
            // ---------------- relay (peer): this CTA's half of a stage is ready
            const uint32_t leader_ready = map_to_rank(smem_u32(ready), pair << 1);
            for (int it = 0; it < nk; ++it) {
                const int sa = it % kStagesA, sb = it % kStagesB;
                if (!wait_or_abort(&full_a[sa], (it / kStagesA) & 1, &s_abort, status)) break;
                if (!wait_or_abort(&full_b[sb], (it / kStagesB) & 1, &s_abort, status)) break;
                mbar_arrive_cluster(leader_ready + sb * 8);
            }
        }
    } else if (warp == 2) {
        if (lane == 0 && rank == 0) {
            // ---------------- activation relay (leader): its A stage landed
            // The A ring is deeper than the stage barrier's ring, so before counting stage it
            // the relay waits until the barrier's previous phase (stage it - kStagesB) is done.
            for (int it = 0; it < nk; ++it) {
                const int sa = it % kStagesA, sb = it % kStagesB;
                if (it >= kStagesB &&
                    !wait_or_abort(&ready[sb], ((it / kStagesB) - 1) & 1, &s_abort, status))
                    break;
                if (!wait_or_abort(&full_a[sa], (it / kStagesA) & 1, &s_abort, status)) break;
                if constexpr (DENSE)
                    if (!wait_or_abort(&full_b[sb], (it / kStagesB) & 1, &s_abort, status)) break;
                mbar_arrive(&ready[sb]);
            }
        }
    } else if (warp == 3) {
        if (SHARE && lane == 0) {
            // ---------------- copier: once this CTA's decoders have written their slab of a
            // weight stage, copy it into each partner's stage (same offset) with a bulk copy
            // that completes on that partner's stage barrier, and count this CTA's slab on its
            // own stage barrier together with the partners' incoming bytes. The copies'
            // source is free again once every pair released the stage, which needs the copies
            // to have landed.
            uint64_t* stage_bar = rank == 0 ? ready : full_b;
            const uint32_t slab0 = smem_u32(smem + kOffB) + pair * kSlab;
            for (int it = 0; it < nk; ++it) {
                const int sb = it % kStagesB;
                if (!wait_or_abort(&dec_done[sb], (it / kStagesB) & 1, &s_abort, status)) break;
#pragma unroll
                for (int pp = 1; pp < NP; ++pp) {
                    const uint32_t partner = ((((int)pair + pp) % NP) << 1) | rank;
                    bulk_to_peer(map_to_rank(slab0, partner) + sb * kBStage, slab0 + sb * kBStage,
                                 kSlab, map_to_rank(smem_u32(stage_bar), partner) + sb * 8);
                }
                mbar_arrive_expect_tx(&stage_bar[sb], (NP - 1) * kSlab);
            }
        }
    } else if (warp >= kDecWarp0) {
        // ---------------- decoders, then epilogue
        const int dt = tid - kDecWarp0 * 32;        // 0..255
        constexpr int GPT = DR * 8 / 256;           // groups per thread and stage
        const int n = dt & (DR - 1);                // decoded row owned by the thread
        const int cs = dt / DR;                     // groups GPT*cs .. GPT*cs + GPT-1 of a stage
        const int c0 = cs * GPT;
        const int row = rd0 + n;
        const int nn = (int)pair * DR + n;          // its row in the weight operand tile
        // Books staged times 2^-f (fp16 range, above), 2^f folded into the row scales; the
        // dense variant's writer staged its books the same way and left 2^f in the workspace.
        float wfac = 1.0f;
        if constexpr (!DENSE) {
            unsigned int* wmax_s = (unsigned int*)(smem + GL::kOffWmax);
            if (dt < 8) wmax_s[dt] = 0u;
            named_barrier(1, kDecWarps * 32);
            uint4 cw[MB];               // codeword dt of every book (256 per book, 256 threads)
#pragma unroll
            for (int k = 0; k < MB; ++k) {
                cw[k] = __ldg((const uint4*)books + k * 256 + dt);
                atomicMax(&wmax_s[k], codeword_max_bits<BDT>(cw[k]));
            }
            named_barrier(1, kDecWarps * 32);
            const int f = book_exponent<BDT>(wmax_s, MB);
            wfac = pow2f(f);
#pragma unroll
            for (int k = 0; k < MB; ++k)
                books_s[k * 256 + dt] = f ? scale_codeword<BDT>(cw[k], pow2f(-f)) : cw[k];
        } else {
            wfac = *(const volatile float*)((const char*)status + kWsWfacOffset);
        }
        for (int i = dt; i < kBN; i += kDecWarps * 32)
            scale_s[i] = (n0 + i < out) ? bits_to_f32_rt(scales[n0 + i], scale_dt) * wfac : 0.0f;
        named_barrier(1, kDecWarps * 32);

        const int r = row & 31;                     // rotation of this row's codes
        const int rw = r >> 2, rb = (r & 3) * 8;
        const bool row_ok = row < out;
        const uint32_t books_u = smem_u32(books_s);
        const uint32_t b_tile = smem_u32(smem + kOffB) + (nn >> 3) * 1024 + (nn & 7) * 128;
        int it = 0;                                 // stages decoded so far (ring position)
        for (int js = 0; js < (DENSE ? 0 : nsl); ++js) {
            const int sl = rot + js < nsl ? rot + js : rot + js - nsl;
            const int cb = js & 1;
            // q[k][j]: the word holding the codes (one byte each) of the thread's groups
            // 8j + c0 .. 8j + c0 + GPT-1 of the slice in plane k (from byte c0 & 3); the
            // front entry always belongs to the next stage.
            uint32_t q[MB][4];
            const bool have = wait_or_abort(&codes_full[cb], (js >> 1) & 1, &s_abort, status);
#pragma unroll
            for (int k = 0; k < MB; ++k) {
                uint32_t w[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
                if (have && n < rows_valid) {
                    const uint32_t src = smem_u32(smem + kOffCodes + cb * kCodeBuf + k * (DR * 32) + n * 32);
                    const uint4 lo = lds128_ordered(src), hi = lds128_ordered(src + 16);
                    w[0] = lo.x; w[1] = lo.y; w[2] = lo.z; w[3] = lo.w;
                    w[4] = hi.x; w[5] = hi.y; w[6] = hi.z; w[7] = hi.w;
                }
                // Undo the row rotation: byte q of the result is the code of group q of the
                // slice (position p holds group (p + row) mod 32, i.e. rotate left by r bytes).
                // Word rotation V[i] = W[i - rw] as three conditional steps (rw is per thread,
                // so no dynamically indexed register array), then the byte part with funnel
                // shifts: out word i = bytes of V[i-1]:V[i] shifted left by 8*(r mod 4).
                uint32_t v[8], t[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) t[i] = (rw & 1) ? w[(i + 7) & 7] : w[i];
#pragma unroll
                for (int i = 0; i < 8; ++i) v[i] = (rw & 2) ? t[(i + 6) & 7] : t[i];
#pragma unroll
                for (int i = 0; i < 8; ++i) t[i] = (rw & 4) ? v[(i + 4) & 7] : v[i];
#pragma unroll
                for (int j = 0; j < 4; ++j) {           // output word 2j + (c0 >> 2)
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
                const int st = it % kStagesB;
                if (it >= kStagesB) wait_or_abort(&empty_b[st], ((it / kStagesB) - 1) & 1, &s_abort, status);
                const uint32_t bt = b_tile + st * kBStage;
                const int g0 = sl * 32 + j * 8 + c0;         // first group of the thread's GPT
#pragma unroll
                for (int cc = 0; cc < GPT; ++cc) {
                    uint32_t code[MB];
#pragma unroll
                    for (int k = 0; k < MB; ++k) code[k] = (q[k][0] >> (((c0 & 3) + cc) * 8)) & 0xffu;
                    uint4 o = decode_group<BDT, MB>(books_u, code);
                    if (!(row_ok && g0 + cc < ng)) o = make_uint4(0u, 0u, 0u, 0u);
                    sts128(bt + (((c0 + cc) ^ (nn & 7)) << 4), o);
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(SHARE ? &dec_done[st] : rank == 0 ? &ready[st] : &full_b[st]);
                ++it;
#pragma unroll
                for (int k = 0; k < MB; ++k) {
                    q[k][0] = q[k][1];
                    q[k][1] = q[k][2];
                    q[k][2] = q[k][3];
                }
            }
        }

        // ---------------- epilogue: accumulators -> scale -> y
        const bool ready = __all_sync(0xffffffffu, wait_or_abort(acc_full, 0, &s_abort, status));
        tc_fence_after();
        __syncwarp();
        // Vector stores need 16-byte aligned row segments: out a multiple of 8 (the output
        // pointer itself is 16-byte aligned by contract).
        const bool vec = (out & 7) == 0;
        if (ready && y_tma) {
            // 16-bit y by TMA stores: every MMA has completed, so the operand rings are free;
            // each warp stages its 32 tokens x 256 rows as eight 32 x 32 chunks (2 KiB each, a
            // token's 64 bytes per row of the chunk, 16-byte pieces placed by the 64-byte
            // swizzle of the store's tensor map: piece j of token row r at j ^ ((r >> 1) & 3),
            // conflict-free) and stores each chunk with one bulk tensor store.
            const int q = warp & 3;                       // tensor-memory lane quarter
            const int i = (warp - kDecWarp0) >> 2;        // token block (accumulator)
            const int tw = t0 + i * 2 * kBM + (int)rank * kBM + q * 32;   // the warp's first token
            const int t = tw + lane;
            const float xf = (xfac && t < tokens) ? xfac[t] : 1.0f;   // 2^e_t (bf16 activations)
            const uint32_t stage = smem_u32(smem + kOffA) + (uint32_t)(warp - kDecWarp0) * (kBN / 32) * 2048u;
            const uint32_t sw = (uint32_t)(lane >> 1) & 3u;
            for (int nc = 0; nc < kBN; nc += 32) {
                float v[32];
                tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + i * kBN + nc, v);
                if (xf != 1.0f)
#pragma unroll
                    for (int e = 0; e < 32; ++e) v[e] *= xf;   // exact: a power of two
                const uint32_t chunk = stage + (uint32_t)(nc / 32) * 2048u;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int e = 8 * j;
                    sts128(chunk + (uint32_t)lane * 64u + (((uint32_t)j ^ sw) << 4),
                           make_uint4(pack2(v[e] * scale_s[nc + e], v[e + 1] * scale_s[nc + e + 1], y_dt),
                                      pack2(v[e + 2] * scale_s[nc + e + 2], v[e + 3] * scale_s[nc + e + 3], y_dt),
                                      pack2(v[e + 4] * scale_s[nc + e + 4], v[e + 5] * scale_s[nc + e + 5], y_dt),
                                      pack2(v[e + 6] * scale_s[nc + e + 6], v[e + 7] * scale_s[nc + e + 7], y_dt)));
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0 && tw < tokens && n0 + nc < out) tma_store_2d(&ymap, n0 + nc, tw, chunk);
            }
            if (lane == 0) {   // the staged chunks are read before the CTA leaves
                bulk_commit();
                bulk_wait_read_all();
            }
            __syncwarp();
        } else if (ready) {
            const int q = warp & 3;                       // tensor-memory lane quarter
            const int i = (warp - kDecWarp0) >> 2;        // token block (accumulator)
            const int t = t0 + i * 2 * kBM + (int)rank * kBM + q * 32 + lane;
            const float xf = (xfac && t < tokens) ? xfac[t] : 1.0f;   // 2^e_t (bf16 activations)
            for (int nc = 0; nc < kBN; nc += 32) {
                float v[32];
                tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + i * kBN + nc, v);
                if (xf != 1.0f)
#pragma unroll
                    for (int e = 0; e < 32; ++e) v[e] *= xf;   // exact: a power of two
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

    // ---------------- teardown
    // The pair MMAs read both CTAs' shared memory and write both CTAs' tensor memory: the
    // leader makes sure every MMA it issued has completed (the final commit always fires) and
    // neither CTA leaves or frees tensor memory before the other is done with it.
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

// bf16 -> fp16 copy of the activations, one token row per CTA (grid-stride over the rows): the
// row is multiplied by 2^-e_t, e_t chosen so that its largest |x| lies in [2^14, 2^15), which is
// exact (a power of two; bf16's 8 significant bits fit fp16's 11 wherever the scaled value is
// in fp16's normal range), and 2^e_t is stored for the epilogue. An all-zero row keeps e_t = 0.
__global__ void __launch_bounds__(256) bf16_rows_to_f16_kernel(const uint16_t* __restrict__ src,
                                                               uint16_t* __restrict__ dst,
                                                               float* __restrict__ xfac, int in,
                                                               int tokens) {
    __shared__ unsigned int red[8];
    pdl_wait();
    pdl_launch_dependents();
    const int n8 = in / 8, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int t = blockIdx.x; t < tokens; t += gridDim.x) {
        const uint4* row = (const uint4*)(src + (size_t)t * in);
        unsigned int mx = 0;            // largest |bf16| bit pattern of the row
        for (int i = threadIdx.x; i < n8; i += blockDim.x) {
            const uint4 v = row[i];
            const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) mx = max(mx, max(w[e] & 0x7fffu, (w[e] >> 16) & 0x7fffu));
        }
        mx = __reduce_max_sync(0xffffffffu, mx);
        if (lane == 0) red[warp] = mx;
        __syncthreads();
        mx = red[0];
        for (int w = 1; w < 8; ++w) mx = max(mx, red[w]);
        __syncthreads();                // red is reused by the next row
        int et = 0;
        if (mx != 0) {
            const int eb = (int)((mx >> 7) & 0xffu);           // biased bf16 exponent
            et = max(-100, min(100, (eb == 0 ? 1 : eb) - 127 - 14));
        }
        const float sc = pow2f(-et);
        uint4* out = (uint4*)(dst + (size_t)t * in);
        for (int i = threadIdx.x; i < n8; i += blockDim.x) {
            const uint4 v = row[i];
            float f[8];
            unpack8<AQ_BF16>(v, f);
            uint32_t o[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                uint32_t h;
                asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(h) : "f"(f[2 * e + 1] * sc), "f"(f[2 * e] * sc));
                o[e] = h;
            }
            out[i] = make_uint4(o[0], o[1], o[2], o[3]);
        }
        if (threadIdx.x == 0) xfac[t] = pow2f(et);
    }
}

// ---- host side ------------------------------------------------------------------------------

// Four pairs per cluster (clusters of eight) measured slower than two at every m: only 16
// clusters of eight fit at once (128 of the 152 SMs), which costs more than the halved
// gathers save.
int gemm_pairs_per_cluster(int m, int tokens) {
    return m >= 2 && tokens > kPairTokens ? 2 : 1;
}

// Tensor map of a 16-bit y [tokens][out] for the epilogue's bulk stores: 32 x 32 boxes, 64-byte
// swizzle. *use = 0 (the per-thread stores) for fp32 y or rows that are not a multiple of 16
// bytes long.
aq_status make_y_map(CUtensorMap* map, int* use, void* y, int y_dt, int out, int tokens) {
    std::memset(map, 0, sizeof(*map));
    *use = 0;
    if (y_dt == AQ_F32 || (out & 7) != 0 || ((uintptr_t)y & 15u) != 0) return AQ_OK;
    EncodeTiledFn encode;
    if (aq_status e = get_encode_fn(&encode); e != AQ_OK) return e;
    const cuuint64_t dims[2] = {(cuuint64_t)out, (cuuint64_t)tokens};
    const cuuint64_t strides[1] = {(cuuint64_t)out * 2};
    const cuuint32_t box[2] = {32, 32};
    const cuuint32_t estr[2] = {1, 1};
    if (encode(map, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, y, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return AQ_ERR_CUDA;
    *use = 1;
    return AQ_OK;
}

template <int BDT>
aq_status run_gemm(const Dims& d, int m, const void* planes, const void* books,
                   const void* scales, const void* x, const float* xfac, int tokens, void* y,
                   int y_dt, void* ws, cudaStream_t st) {   // x: fp16 [tokens][in]
    EncodeTiledFn encode;
    if (aq_status e = get_encode_fn(&encode); e != AQ_OK) return e;
    CUtensorMap map;
    std::memset(&map, 0, sizeof(map));
    const cuuint64_t dims[2] = {(cuuint64_t)d.in, (cuuint64_t)tokens};
    const cuuint64_t strides[1] = {(cuuint64_t)d.in * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)kBM};
    const cuuint32_t estr[2] = {1, 1};
    if (encode(&map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(x), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return AQ_ERR_CUDA;

    // Pairs per cluster sharing the decode: sharing pays where the gathers bound the kernel
    // (m >= 2) and every pair of a cluster has tokens (one 512-token tile per pair).
    const int np = gemm_pairs_per_cluster(m, tokens);
    using Kern = void (*)(const CUtensorMap, const CUtensorMap, const CUtensorMap, int, const uint8_t*,
                          const uint16_t*, const uint16_t*,
                          void*, int, int, unsigned int*, const float*, int, int, int, int, int, size_t);
    const Kern k1[kGemmMaxM] = {gemm_kernel<BDT, 1, 1>, gemm_kernel<BDT, 2, 1>, gemm_kernel<BDT, 3, 1>,
                                gemm_kernel<BDT, 4, 1>, gemm_kernel<BDT, 5, 1>, gemm_kernel<BDT, 6, 1>,
                                gemm_kernel<BDT, 7, 1>, gemm_kernel<BDT, 8, 1>};
    const Kern k2[kGemmMaxM] = {nullptr, gemm_kernel<BDT, 2, 2>, gemm_kernel<BDT, 3, 2>,
                                gemm_kernel<BDT, 4, 2>, gemm_kernel<BDT, 5, 2>, gemm_kernel<BDT, 6, 2>,
                                gemm_kernel<BDT, 7, 2>, gemm_kernel<BDT, 8, 2>};
    const int smem_sizes[kGemmMaxM] = {GemmLayout<1>::kSmem, GemmLayout<2>::kSmem, GemmLayout<3>::kSmem,
                                       GemmLayout<4>::kSmem, GemmLayout<5>::kSmem, GemmLayout<6>::kSmem,
                                       GemmLayout<7>::kSmem, GemmLayout<8>::kSmem};
    const Kern kern = (np == 2 ? k2 : k1)[m - 1];
    const int smem = smem_sizes[m - 1];
    const int csize = 2 * np;         // CTAs per cluster
    static std::mutex mu;
    static bool attr_done[2 * kGemmMaxM][64] = {};
    const int slot = (m - 1) + (np == 2 ? kGemmMaxM : 0);
    int dev = 0;
    if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    {
        std::lock_guard<std::mutex> lock(mu);
        if (dev >= 0 && dev < 64 && !attr_done[slot][dev]) {
            if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
                e != cudaSuccess)
                return cuda_fail(e, "cudaFuncSetAttribute");
            if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout,
                                                     (int)cudaSharedmemCarveoutMaxShared);
                e != cudaSuccess)
                return cuda_fail(e, "cudaFuncSetAttribute");
            attr_done[slot][dev] = true;
        }
    }
    cudaLaunchConfig_t cfg = {};
    // x: one cluster per 256-row tile, y: one token tile per pair of the cluster
    const int tok_tile = np * kPairTokens;
    cfg.gridDim = dim3(csize * ((d.out + kBN - 1) / kBN), (tokens + tok_tile - 1) / tok_tile);
    cfg.blockDim = dim3(kGemmThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)csize;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    CUtensorMap unused;                 // the weight map is read only by the dense variant
    std::memset(&unused, 0, sizeof(unused));
    CUtensorMap ym;
    int y_tma = 0;
    if (aq_status e = make_y_map(&ym, &y_tma, y, y_dt, d.out, tokens); e != AQ_OK) return e;
    return cuda_ok(cudaLaunchKernelEx(&cfg, kern, map, unused, ym, y_tma, (const uint8_t*)planes,
                                      (const uint16_t*)books, (const uint16_t*)scales, y, y_dt,
                                      d.scale_dt, (unsigned int*)ws, xfac, tokens, d.out, d.in, d.ng,
                                      d.rows_pad, d.plane_bytes),
                   "cudaLaunchKernelEx (GEMM)");
}

// ---- dense variant: W_m decoded once into the workspace, then TMA-fed pair MMAs -----------

// W16[o][i] = fp16(sum_{k<m} C_k[b_k[o, i/8]][i mod 8]): the unscaled fp32 sum of the m
// codewords in book order, rounded once to fp16 (the values the GEMM's decoders write; the
// epilogue applies the row scale).
// One CTA per SM walks the (32-row block, 256-input slice) items, a warp at a time
// (grid-stride; row blocks fastest, so a warp's code loads are one contiguous 1 KiB per plane
// and its stores 512 contiguous bytes per row). The CTA stages the first m codebooks once, in
// 2^cshift interleaved copies (book_copies_log2), so the gathers are free of bank conflicts
// with eight copies (with one copy random codes cost about 2.4 times the conflict-free
// wavefronts). Each lane
// copies its row's codes of the m planes into the warp's staging buffer (cp.async, 16 bytes
// at a time), the next item's while the current one is decoded; then lane L walks the 32 rows
// producing group s*32 + L of each.
constexpr int kDenseMaxWarps = 16;

// Shared memory of a writer CTA of nw warps: the staged books and each warp's two code buffers.
inline size_t dense_w_smem(int B, int m, int nw) {
    return (size_t)m * ((size_t)16 << B << book_copies_log2(B, m)) + (size_t)nw * 2 * m * 32 * unit_bytes(B);
}

template <int B, int BDT>
__global__ void __launch_bounds__(kDenseMaxWarps * 32, 1)
dense_w_kernel(const uint8_t* __restrict__ planes, const uint16_t* __restrict__ books,
               uint16_t* __restrict__ w16, float* __restrict__ wfac_out, int m, int cshift, int out,
               int in, int ng, int rows_pad, int RBc, int S, size_t plane_bytes) {
    constexpr int UNIT = unit_bytes(B);
    constexpr int NC = 1 << B;
    extern __shared__ __align__(16) unsigned char smem_d[];
    uint4* books_s = (uint4*)smem_d;                 // [m][NC][2^cshift] codewords
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (int)(blockDim.x >> 5);
    // this warp's code buffers: [2][m][32 rows][UNIT]
    unsigned char* cbuf = smem_d + ((size_t)m * NC << cshift) * 16 + (size_t)warp * 2 * m * 32 * UNIT;
    __shared__ unsigned int wmax[8];
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
    pdl_wait();
    pdl_launch_dependents();
    long long item = (long long)blockIdx.x * nw + warp;
    issue(item, 0);   // the first codes travel while the books are staged
    // Books staged times 2^-f (fp16 range, as in the GEMM's decoders); 2^f goes to the
    // workspace for the GEMM's epilogue (every CTA finds the same f; CTA 0 writes it).
    if (threadIdx.x < 8) wmax[threadIdx.x] = 0u;
    __syncthreads();
    for (int i = threadIdx.x; i < m * NC; i += blockDim.x)
        atomicMax(&wmax[i >> B], codeword_max_bits<BDT>(__ldg((const uint4*)books + i)));
    __syncthreads();
    const int f = book_exponent<BDT>(wmax, m);
    for (int i = threadIdx.x; i < (m * NC) << cshift; i += blockDim.x) {
        const uint4 c = __ldg((const uint4*)books + (i >> cshift));
        books_s[i] = f ? scale_codeword<BDT>(c, pow2f(-f)) : c;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) *wfac_out = pow2f(f);
    __syncthreads();
    const uint32_t books_u = smem_u32(books_s) + ((uint32_t)(lane & ((1 << cshift) - 1)) << 4);
    int buf = 0;
    for (; item < items; item += stride) {
        issue(item + stride, buf ^ 1);
        cp_async_wait<1>();      // this lane's copies of the current item landed
        __syncwarp();            // ... and every lane's
        const int s = (int)(item / RBc), rb = (int)(item - (long long)s * RBc);
        const int g = s * 32 + lane;
        const unsigned char* cb = cbuf + (size_t)buf * m * 32 * UNIT;
        if (g < ng) {
            // four rows at a time: four independent gathers per book in flight
            for (int r0 = 0; r0 < 32 && rb * 32 + r0 < out; r0 += 4) {
                float a[4][8];
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int e = 0; e < 8; ++e) a[i][e] = -0.0f;
                for (int k = 0; k < m; ++k) {
                    uint4 c[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int r = r0 + i;
                        // position of group `lane` in row rb*32 + r
                        const uint32_t code = unit_code<B>(cb + ((size_t)k * 32 + r) * UNIT, (lane - r) & 31);
                        c[i] = lds128(books_u + ((((uint32_t)k << B) + code) << (cshift + 4)));
                    }
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        add_widen2<BDT>(c[i].x, a[i][0], a[i][1]);
                        add_widen2<BDT>(c[i].y, a[i][2], a[i][3]);
                        add_widen2<BDT>(c[i].z, a[i][4], a[i][5]);
                        add_widen2<BDT>(c[i].w, a[i][6], a[i][7]);
                    }
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int o = rb * 32 + r0 + i;
                    if (o < out)
                        *(uint4*)(w16 + (size_t)o * in + (size_t)g * 8) =
                            make_uint4(f16x2(make_float2(a[i][0], a[i][1])), f16x2(make_float2(a[i][2], a[i][3])),
                                       f16x2(make_float2(a[i][4], a[i][5])), f16x2(make_float2(a[i][6], a[i][7])));
                }
            }
        }
        __syncwarp();            // every lane has read the buffer before it is refilled
        buf ^= 1;
    }
    cp_async_wait<0>();
}

template <int B, int BDT>
aq_status run_gemm_dense(const Dims& d, int m, const void* planes, const void* books,
                         const void* scales, const void* x, const float* xfac, int tokens, void* y,
                         int y_dt, void* ws, uint16_t* w16, cudaStream_t st) {   // x: fp16 [tokens][in]
    {   // decode W_m once
        auto kern = dense_w_kernel<B, BDT>;
        DeviceInfo di;
        if (aq_status e = device_info(&di); e != AQ_OK) return e;
        // the kernel's shared-memory limit raised once per device; per prefix the warps per CTA
        // (16, 12, 8, 6 or 4) with the most resident warps per SM
        static std::mutex mu_w;
        static int dyn_max[64] = {};
        static int choice[64][kGemmMaxM + 1][2] = {};   // [dev][m] -> {warps, CTAs per SM}
        int dev = 0;
        if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
        if (dev < 0 || dev >= 64 || m < 1 || m > kGemmMaxM) return AQ_ERR_UNSUPPORTED;
        int nw = 0, occ = 0;
        {
            std::lock_guard<std::mutex> lock(mu_w);
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
            if (choice[dev][m][0] == 0) {
                int best_w = 0;
                for (int w : {16, 12, 8, 6, 4}) {
                    const size_t sm_bytes = dense_w_smem(B, m, w);
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
        const size_t smem = dense_w_smem(B, m, nw);
        const long long items = (long long)d.RBc * d.S;
        long long grid = (long long)di.sms * occ;
        const long long need = (items + nw - 1) / nw;
        if (grid > need) grid = need;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)grid);
        cfg.blockDim = dim3(nw * 32);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (aq_status e = cuda_ok(cudaLaunchKernelEx(&cfg, kern, (const uint8_t*)planes, (const uint16_t*)books,
                                                     w16, (float*)((char*)ws + kWsWfacOffset), m,
                                                     book_copies_log2(B, m), d.out, d.in, d.ng, d.rows_pad,
                                                     d.RBc, d.S, d.plane_bytes),
                                  "cudaLaunchKernelEx (dense W_m)");
            e != AQ_OK)
            return e;
    }
    EncodeTiledFn encode;
    if (aq_status e = get_encode_fn(&encode); e != AQ_OK) return e;
    CUtensorMap xm, wm;
    std::memset(&xm, 0, sizeof(xm));
    std::memset(&wm, 0, sizeof(wm));
    const cuuint64_t strides[1] = {(cuuint64_t)d.in * 2};
    const cuuint32_t estr[2] = {1, 1};
    {
        const cuuint64_t dims[2] = {(cuuint64_t)d.in, (cuuint64_t)tokens};
        const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)kBM};
        if (encode(&xm, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(x), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return AQ_ERR_CUDA;
    }
    {
        const cuuint64_t dims[2] = {(cuuint64_t)d.in, (cuuint64_t)d.out};
        const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)kRows};
        if (encode(&wm, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, (void*)w16, dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return AQ_ERR_CUDA;
    }
    auto kern = gemm_kernel<BDT, 1, 1, true>;
    constexpr int smem = GemmLayout<1, true>::kSmem;
    static std::mutex mu;
    static bool attr_done[64] = {};
    int dev = 0;
    if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    {
        std::lock_guard<std::mutex> lock(mu);
        if (dev >= 0 && dev < 64 && !attr_done[dev]) {
            if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
                e != cudaSuccess)
                return cuda_fail(e, "cudaFuncSetAttribute");
            attr_done[dev] = true;
        }
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * ((d.out + kBN - 1) / kBN), (tokens + kPairTokens - 1) / kPairTokens);
    cfg.blockDim = dim3(kGemmThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = 2;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    CUtensorMap ym;
    int y_tma = 0;
    if (aq_status e = make_y_map(&ym, &y_tma, y, y_dt, d.out, tokens); e != AQ_OK) return e;
    return cuda_ok(cudaLaunchKernelEx(&cfg, kern, xm, wm, ym, y_tma, (const uint8_t*)planes, (const uint16_t*)books,
                                      (const uint16_t*)scales, y, y_dt, d.scale_dt, (unsigned int*)ws,
                                      xfac, tokens, d.out, d.in, d.ng, d.rows_pad, d.plane_bytes),
                   "cudaLaunchKernelEx (dense GEMM)");
}

}  // namespace

aq_status launch_gemm(const Dims& d, int m, const void* planes, const void* books,
                      const void* scales, const void* x, int x_dt, int tokens, void* y, int y_dt,
                      void* ws, cudaStream_t st) {
    if (d.out == 0 || tokens == 0) return AQ_OK;
    if ((d.B != 8 && d.B != 4) || m > kGemmMaxM) return AQ_ERR_UNSUPPORTED;
    const void* xh = x;
    const float* xfac = nullptr;
    if (x_dt == AQ_BF16) {
        // fp16 copy of the activations, each token row scaled into fp16's range, and the
        // per-token factors, in the workspace
        void* dst = (char*)ws + gemm_x16_offset(tokens);
        float* fac = (float*)((char*)ws + gemm_xfac_offset());
        DeviceInfo di;
        if (aq_status e = device_info(&di); e != AQ_OK) return e;
        const int blocks = tokens < di.sms * 8 ? tokens : di.sms * 8;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(blocks);
        cfg.blockDim = dim3(256);
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (aq_status e = cuda_ok(cudaLaunchKernelEx(&cfg, bf16_rows_to_f16_kernel, (const uint16_t*)x,
                                                     (uint16_t*)dst, fac, d.in, tokens),
                                  "cudaLaunchKernelEx (activation copy)");
            e != AQ_OK)
            return e;
        xh = dst;
        xfac = fac;
    }
    if (gemm_uses_dense(d, m, tokens)) {
        uint16_t* w16 = (uint16_t*)((char*)ws + gemm_w16_offset(d, tokens));
        if (d.B == 4)   // the in-loop decoders read 8-bit codes; 4-bit layouts always go dense
            return d.book_dt == AQ_BF16
                       ? run_gemm_dense<4, AQ_BF16>(d, m, planes, books, scales, xh, xfac, tokens, y, y_dt, ws, w16, st)
                       : run_gemm_dense<4, AQ_F16>(d, m, planes, books, scales, xh, xfac, tokens, y, y_dt, ws, w16, st);
        return d.book_dt == AQ_BF16
                   ? run_gemm_dense<8, AQ_BF16>(d, m, planes, books, scales, xh, xfac, tokens, y, y_dt, ws, w16, st)
                   : run_gemm_dense<8, AQ_F16>(d, m, planes, books, scales, xh, xfac, tokens, y, y_dt, ws, w16, st);
    }
    return d.book_dt == AQ_BF16
               ? run_gemm<AQ_BF16>(d, m, planes, books, scales, xh, xfac, tokens, y, y_dt, ws, st)
               : run_gemm<AQ_F16>(d, m, planes, books, scales, xh, xfac, tokens, y, y_dt, ws, st);
}

}  // namespace aq
