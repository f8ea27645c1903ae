/*
 * aq.h - C ABI of the multi-bitwidth additive-codebook dequantize-and-multiply library
 * (GB300 / sm_103a). Drop-by-Drop, arxiv 2606.12876.
 *
 * A linear layer W (d_out x d_in) is stored once as M additive codebooks C_0..C_{M-1}
 * (each 2^B codewords of g = 8 values), per-output-row scales s, and one B-bit code per
 * (row, group of g inputs, codebook). At call time a prefix length m (1 <= m <= M) selects
 * how many codebooks are summed (Sec. 5: the weights are rebuilt from the leading k
 * codebooks only, and how many are active is chosen at deployment):
 *
 *     W_m[o, g*8 + e] = s[o] * sum_{k<m} C_k[ b_k[o, g] ][e]         (Sec. 3.2 and Sec. 5)
 *     y[t, o]         = sum_i x[t, i] * W_m[o, i]                     (Sec. 2.2, Y = W X)
 *
 * Conventions that hold for every entry point:
 *   - All data pointers are DEVICE pointers, 16-byte aligned, owned by the caller. Apart
 *     from the aq_store_* entry points (dynamic loading, below), the library allocates and
 *     frees nothing and keeps no pointer after a call returns.
 *   - stream is a cudaStream_t passed as void* (NULL = the legacy default stream). All work
 *     is enqueued asynchronously on it; no call synchronises unless its comment says so.
 *   - Argument errors are detected on the host before anything is launched; the call then
 *     returns a non-zero aq_status and the device is untouched. A failed launch returns
 *     AQ_ERR_CUDA.
 *   - Readings of points the paper leaves open: the scale multiplies the codebook sum of its
 *     row (R1); a codebook is stored [2^B][g], codeword-contiguous (R2); books are numbered
 *     0..M-1 and "prefix m" means books 0..m-1.
 */
#ifndef AQ_H
#define AQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define AQ_ABI_VERSION 1

typedef enum {
    AQ_OK = 0,
    AQ_ERR_INVALID_ARG = 1,   /* null pointer, m outside 1..M, bad sizes, bad dtype */
    AQ_ERR_UNSUPPORTED = 2,   /* valid in principle but not implemented (e.g. g != 8) */
    AQ_ERR_ALIGNMENT = 3,     /* a pointer is not 16-byte aligned */
    AQ_ERR_CUDA = 4,          /* a CUDA launch or runtime call failed */
    AQ_ERR_TIMEOUT = 5,       /* a bounded device-side wait gave up (reported via workspace) */
    AQ_ERR_WORKSPACE = 6      /* workspace missing or smaller than the *_workspace_bytes query */
} aq_status;

typedef enum { AQ_F16 = 0, AQ_BF16 = 1, AQ_F32 = 2 } aq_dtype;

/* Shape and storage types of one quantized layer (App. C lists the three stored parts:
 * codebooks, codes, per-output-unit scales). */
typedef struct aq_layout {
    int32_t out_features;   /* d_out >= 0 */
    int32_t in_features;    /* d_in >= 8, a multiple of group_size */
    int32_t group_size;     /* g; only 8 is supported */
    int32_t num_books;      /* M, 1..8 */
    int32_t code_bits;      /* B; 4 (two codes per byte), 8 (uint8 codes) or 16 (uint16) */
    int32_t book_dtype;     /* AQ_F16 or AQ_BF16: element type of the codebooks */
    int32_t scale_dtype;    /* AQ_F16 or AQ_BF16: element type of the scales */
    int32_t flags;          /* 0 or AQ_LAYOUT_STATIC_WEIGHTS */
} aq_layout;

/* Layout flag: the layer's codes, codebooks and scales are not written by any kernel that
 * may still be running when a GEMV or GEMM call on them starts (in inference they are written
 * once, then only read). A call may then begin reading them - prefetching the first code
 * stages into L2 and staging the codebooks - before the kernel that precedes it on the stream
 * has finished, which overlaps that traffic with the preceding kernel's tail. Activations are
 * always read only after the preceding kernel has finished. Without the flag (0) every read
 * waits for the preceding kernel. */
#define AQ_LAYOUT_STATIC_WEIGHTS 1

/* ABI version of the loaded library (AQ_ABI_VERSION). */
int aq_abi_version(void);

/* Static English text for a status code; never NULL. */
const char* aq_status_string(int status);

/* Text of the last CUDA failure seen by this thread inside the library (the call that
 * failed, the CUDA error name and message), or "" if none. Valid until the next call. */
const char* aq_last_error(void);

/* ---------------------------------------------------------------- packed code planes
 * Codes are stored codebook-major ("planes"), so a prefix m reads only the first m planes:
 *   rows_pad = d_out rounded up to 32; ng = d_in/8 groups, ng_pad = ng rounded up to 32;
 *   S = ng_pad/32 slices of 32 groups. Plane k (k = 0..M-1) is rows_pad*ng_pad codes of
 *   B/8 bytes each, laid out [slice][row][position] with 32 positions per (slice,row).
 *   Position p of row o in slice s holds the code of group s*32 + ((p + o) mod 32): each
 *   row's 32 codes of a slice are rotated by the row index, so 32 consecutive rows read a
 *   position p together touch 32 different groups. Padding rows/groups hold code 0.
 *   Plane k starts at byte k*aq_plane_bytes(); the first m planes are a contiguous prefix.
 *   4-bit codes (B = 4, the 16-entry codebooks of the paper's 4x4-bit ablation, App. G.1)
 *   share bytes: position p of a (slice, row) unit is in byte p/2, in the low four bits for
 *   even p and the high four bits for odd p, so a unit is 16 bytes and a plane
 *   rows_pad*ng_pad/2 bytes. */

/* Bytes of one code plane (the codes b of one codebook, Sec. 3.2; App. C counts them as
 * d_out*(d_in/g)*B bits per codebook, the codes term of Eq. avg_bits); 0 if the layout is
 * invalid. */
size_t aq_plane_bytes(const aq_layout* layout);

/* Bytes of the first m planes (m*aq_plane_bytes): the codes a prefix-m call reads (Sec. 5,
 * the first k codebooks); 0 if the layout or m is invalid. */
size_t aq_packed_bytes(const aq_layout* layout, int m);

/* Pack natural codes into planes (the codes b_{i,j,m} of Sec. 3.2).
 *   codes  : device, (d_out, d_in/8, M) row-major, uint8 (B = 4, 8) or uint16 (B = 16);
 *            code values must be < 2^B.
 *   planes : device, aq_packed_bytes(layout, M) bytes, fully written (padding = 0). */
aq_status aq_pack(const aq_layout* layout, const void* codes, void* planes, void* stream);

/* ---------------------------------------------------------------- decode
 * W_m written out densely (Sec. 5 partial reconstruction with the scale of R1).
 * Bit-exact contract: for each element, acc = +0.0f; for k = 0..m-1: acc += (float)C_k[...][e]
 * (fp32 adds, in that order); v = acc * (float)s[o] (one fp32 multiply); the output is v
 * rounded once, to nearest-even, to book_dtype.
 *   planes : device, at least the first m planes (aq_packed_bytes(layout, m) bytes)
 *   books  : device, [M][2^B][8] of book_dtype (only the first m books are read)
 *   scales : device, [d_out] of scale_dtype
 *   w      : device, [d_out][d_in] of book_dtype, row-major. */
aq_status aq_decode(const aq_layout* layout, int m, const void* planes, const void* books,
                    const void* scales, void* w, void* stream);

/* ---------------------------------------------------------------- GEMV (batch 1..16)
 * y[t, o] = sum_i x[t, i] * W_m[o, i] for t < batch (Sec. 2.2 Y = W X, with W_m the prefix-m
 * reconstruction of Sec. 3.2 / Sec. 5), accumulated in fp32. The kernel reads the first m
 * planes once (HBM-bound at batch 1); 8-bit codebooks are staged on chip. At batch 5..8 with
 * up to six 2^8-entry books, on layers of at least 4560 (256-input slice, codebook, 32-row
 * block) items, the products are taken from per-(slice, codebook) tables of fp16 values (each
 * token's scaled by a power of two, so the range of the activations is kept); elsewhere every
 * intermediate is fp32 or a tf32 operand.
 *   x         : device, [batch][d_in] of x_dtype (AQ_F16 or AQ_BF16), row-major
 *   y         : device, [batch][d_out] of y_dtype (AQ_F16, AQ_BF16 or AQ_F32), row-major
 *   workspace : device scratch of at least aq_gemv_workspace_bytes(layout, batch) bytes:
 *               a status word and fp32 partial sums for every row: one per 256-input
 *               slice and token, or, with 2^8-entry books at batch 1..2 (batch 3..4, batch
 *               5..8 on the layers above), one per slice, token and codebook of the largest
 *               prefix up to 8 (up to 4, up to 6) served that way. Zero-fill it once before its first use (aq_workspace_init); every
 *               call leaves it ready for the next one.
 *               Calls that may overlap on the GPU must not share a workspace.
 * Two kernels are enqueued, both with programmatic dependent launch: the product (fp32
 * partial sums per 256-input slice, and per codebook at batch 1..8 with 2^8-entry books, into
 * the workspace) and a split-K reduction that sums each row's partials, scales it and
 * writes y (4-bit codes at batch 1: one kernel that writes y itself). Each waits for the
 * preceding grid before reading memory. The partials of each
 * row are summed in a fixed order, so the result does not depend on scheduling.
 * Accuracy: relative Frobenius error <= 2e-3 and |y - y_exact| <= 1e-2*(1+|y_exact|) per
 * element, with y_exact the fp64 product of the exactly widened stored values, on unit-scale
 * inputs (activations of order 1, codebook entries of the order of N(0, 0.02^2), as in the
 * benchmark layers). Batch 1..4 add fp32 table entries (fp32 roundings only); batch 5..16
 * round each decoded weight to a tf32 operand, or each table entry to fp16 and pairs of
 * entries once more, so their per-element error is bounded by about
 * 2^-10 * |s[o]| * sum_i |x_i| sum_k |C_k[b_k]_i|, which scales with the inputs. */
size_t aq_gemv_workspace_bytes(const aq_layout* layout, int batch);
aq_status aq_gemv(const aq_layout* layout, int m, const void* planes, const void* books,
                  const void* scales, const void* x, int x_dtype, int batch, void* y,
                  int y_dtype, void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------- GEMV of a group of layers
 * (No counterpart in the paper: a way to call the product of Sec. 2.2 with the prefix-m
 * reconstruction of Sec. 3.2 / Sec. 5 for several layers that read the same activations,
 * such as a decoder block's query, key and value projections, or its gate and up projections.)
 * y_l = x * W_m,l^T for l < n, each as aq_gemv would compute it, bit for bit: every layer's
 * partial sums and their summation order are those of its own call. At batch 1 with 2^8-entry
 * codebooks the n products run as one kernel over the items of all layers and the n
 * reductions as one kernel, so the group pays the fixed cost of a call (two kernel boundaries,
 * the activation load, the first table build) once instead of n times; otherwise the layers
 * are computed one after the other, as n calls of aq_gemv.
 *   n        : 1..4 layers
 *   layouts  : n layouts with the same in_features, code_bits, book_dtype and scale_dtype
 *   m        : 1 <= m <= num_books of every layer
 *   planes, books, scales : host arrays of n device pointers, as for aq_gemv
 *   x        : device, [batch][d_in], shared by the layers
 *   y        : host array of n device pointers, layer l's [batch][d_out_l] of y_dtype
 *   workspace: aq_gemv_group_workspace_bytes(n, layouts, batch) bytes, 16-byte aligned,
 *              zero-filled before first use: layer l's aq_gemv workspace at the sum of the
 *              earlier layers' sizes, each rounded up to 256 bytes; a device-side status is
 *              recorded in layer 0's status word (aq_workspace_status(workspace, ...)).
 * Errors: as aq_gemv; AQ_ERR_INVALID_ARG also for n outside 1..4, NULL pointer arrays or
 * layouts that differ in in_features, code_bits, book_dtype or scale_dtype. */
size_t aq_gemv_group_workspace_bytes(int n, const aq_layout* layouts, int batch);
aq_status aq_gemv_group(int n, const aq_layout* layouts, int m, const void* const* planes,
                        const void* const* books, const void* const* scales, const void* x,
                        int x_dtype, int batch, void* const* y, int y_dtype, void* workspace,
                        size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------- GEMV refinement (prefix m-1 -> m)
 * y = y_prev + x * (s o C_{m-1}[b_{m-1}])^T: the increment that raises a product computed with
 * the first m-1 codebooks to the product with the first m (the successive reconstruction of
 * Sec. 4, y^(k) = y^(k-1) + increment, applied to the codebook prefixes of Sec. 5; by the
 * linearity of the product in the books, y_prev = the prefix-(m-1) product gives the prefix-m
 * product). Only plane m-1 of the codes and codebook m-1 are read, so raising the precision
 * of a result at run time costs one plane of HBM traffic.
 *   m       : 1 <= m <= num_books; the book whose increment is added is m-1
 *   planes  : device, at least the first m planes (only plane m-1 is read)
 *   y_prev  : device, [batch][d_out] of y_dtype, 16-byte aligned, or NULL (read as zero: y is
 *             then the increment alone). It may be y itself (in-place refinement).
 *   all other arguments, the workspace size and the error behaviour are those of aq_gemv.
 * Each element is y_prev + (the increment in fp32), rounded once to y_dtype; with
 * y_dtype = AQ_F32 a chain of refinements from m = 1 (y_prev = NULL) to m stays within the
 * aq_gemv accuracy bounds of the prefix-m product. */
aq_status aq_gemv_refine(const aq_layout* layout, int m, const void* planes, const void* books,
                         const void* scales, const void* x, int x_dtype, int batch,
                         const void* y_prev, void* y, int y_dtype, void* workspace,
                         size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------- GEMV without a workspace
 * (This entry point has no counterpart in the paper.) The GEMV of aq_gemv for callers that
 * cannot allocate device memory when they run a layer, and so cannot pass a workspace: for
 * example a plugin inside a host program that owns all device memory and offers no
 * allocator, or a serving loop that must not allocate after start-up because an allocation
 * can synchronise the device or fail under memory pressure. Nothing is allocated: the scratch
 * comes from a fixed AQ_STATIC_SCRATCH_BYTES buffer that the library holds, as a device
 * array, on every GPU that loads it, until the process exits.
 *   - Arguments and host-side status codes are those of aq_gemv (same checks).
 *   - Returns AQ_ERR_WORKSPACE when aq_gemv_workspace_bytes(layout, batch) is larger than
 *     AQ_STATIC_SCRATCH_BYTES; use aq_gemv with a workspace for such sizes.
 *   - The first call on a device looks up the buffer's device address; make that first call
 *     on each device before capturing any stream on it. The address is cached for the life of
 *     the device's primary context: do not use this entry point after cudaDeviceReset.
 *   - Each call enqueues the GEMV kernels only (nothing is cleared in between).
 *   - A device-side failure (a bounded wait that gave up, AQ_ERR_TIMEOUT) is recorded in the
 *     buffer's status word and stays there, across later calls, until
 *     aq_gemv_static_scratch_status reads and clears it.
 *   - Every call on a device shares the one buffer, which keeps the last call's contents:
 *     calls that may overlap on the GPU (other streams, other host threads) race on it and
 *     must be ordered by the caller. */
#define AQ_STATIC_SCRATCH_BYTES ((size_t)16 << 20)
aq_status aq_gemv_static_scratch(const aq_layout* layout, int m, const void* planes,
                                 const void* books, const void* scales, const void* x,
                                 int x_dtype, int batch, void* y, int y_dtype, void* stream);

/* The device-side status of the aq_gemv_static_scratch calls on the current device: as
 * aq_workspace_status for the library's fixed buffer. SYNCHRONISES stream, returns the status
 * a kernel recorded (AQ_OK if none) and clears it. (No counterpart in the paper.) */
aq_status aq_gemv_static_scratch_status(void* stream);

/* ---------------------------------------------------------------- GEMM (prefill)
 * Same product for many tokens (Sec. 2.2 Y = W X with W_m of Sec. 3.2 / Sec. 5):
 * y[t, o] = sum_i x[t, i] * W_m[o, i], t < tokens. Decoded weight tiles are built in shared
 * memory and multiplied on the tcgen05 tensor cores with fp32 accumulation in tensor memory
 * (up to 2047 tokens, or m = 1, W_m is never written to HBM; see workspace below). The MMA
 * operands are fp16, over the whole range of the inputs: each decoded weight (fp32 sum of the
 * m codewords) is rounded once to fp16 after the codebooks were scaled by a power of two
 * 2^-f that keeps the largest possible sum below 2^15; bf16 activations are copied to fp16 in
 * the workspace, each token row scaled by a power of two 2^-e_t that puts its largest |x| in
 * [2^14, 2^15); the epilogue multiplies by 2^(e_t + f). The scalings are exact, so inputs
 * already inside fp16's range give the same bits as without them, and bf16 values far outside
 * it (activation outliers, large codebook entries) are multiplied with fp16's 11-bit
 * significand instead of saturating. Supported: code_bits = 8 and 4 (4-bit layouts always
 * decode W_m into the workspace first), any m <= num_books <= 8.
 *   x : device, [tokens][d_in] of x_dtype (AQ_F16 or AQ_BF16); y : device, [tokens][d_out]
 *       of y_dtype (AQ_F16, AQ_BF16 or AQ_F32).
 *   workspace : aq_gemm_workspace_bytes(layout, tokens) bytes (a 256-byte status block, one
 *               float per token for the activation factors, room for the fp16 activation
 *               copy and, from 2048 tokens when num_books >= 2 (for 4-bit codes always), room
 *               for W_m decoded once in fp16, d_out*d_in*2 bytes: at that length calls with
 *               m >= 2 decode W_m into it and multiply by TMA-fed tensor-core tiles, which is
 *               faster than decoding every weight tile again for every 512 tokens),
 *               zero-filled before first use; its first word receives a device-side status
 *               (see aq_workspace_status).
 * Accuracy: as aq_gemv for fp32 outputs; fp16/bf16 outputs add one rounding of y. */
size_t aq_gemm_workspace_bytes(const aq_layout* layout, int tokens);
aq_status aq_gemm(const aq_layout* layout, int m, const void* planes, const void* books,
                  const void* scales, const void* x, int x_dtype, int tokens, void* y,
                  int y_dtype, void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------- distortion of every prefix
 * The weighted MSE of Sec. 2.2 (Eq. wmse-task, trace form) for every prefix, as Drop-by-Drop
 * measures its partial reconstructions (Sec. 5), and the Drop-by-Drop objective:
 *     D[k-1] = (1/d_out) * tr[(W - W^(k)) H (W - W^(k))^T],   k = 1..M,
 *     W^(k)[o, g*8+e] = s[o] * sum_{j<k} C_j[b_j[o,g]][e]   (unrounded; fp32 on the GPU),
 *     L = sum_k lambda[k-1] * D[k-1]                        (when lambda is given).
 * H is the proxy Hessian X X^T / n of the layer's calibration inputs; only its symmetric part
 * enters the trace, so any square H is accepted and evaluated as (H + H^T)/2.
 *   w       : device, [d_out][d_in] of book_dtype (the original weight)
 *   h       : device, [d_in][d_in] of h_dtype (AQ_F32 or AQ_BF16), row-major
 *   lambda  : HOST, M doubles (the weight of prefix k at index k-1), or NULL
 *   d       : device, M doubles, 8-byte aligned (M + 1 when lambda is given: d[M] = L);
 *             written, not accumulated; d_out = 0 gives zeros
 *   workspace : device, aq_wmse_workspace_bytes(layout) bytes, 16-byte aligned: a status word,
 *             a bf16 copy of the folded H (d_in^2 * 2 bytes), the residuals E_k of every
 *             prefix in bf16 (M * d_out * d_in * 2 bytes) and per-CTA partial sums. Zero-fill
 *             it once before first use (aq_workspace_init); device-side waits that time out
 *             are reported through it (aq_workspace_status).
 * Computation: E_k = W - W^(k) (fp32, then rounded once to bf16, written to the workspace)
 * times H folded to its block-lower-triangular symmetric form (bf16) on the tcgen05 tensor
 * cores with fp32 accumulation, two prefixes per pass; per-tile sums are added in a fixed
 * order. Accuracy: |D - D_exact| <= 1.25e-2 * D_abs with
 * D_abs = (1/d_out) sum_o |e_o||H||e_o|^T (three bf16 roundings, first order), typically far
 * smaller. Errors: as aq_gemv. */
size_t aq_wmse_workspace_bytes(const aq_layout* layout);
aq_status aq_wmse(const aq_layout* layout, const void* w, const void* planes, const void* books,
                  const void* scales, const void* h, int h_dtype, const double* lambda, double* d,
                  void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------- code update (beam search)
 * The code update of Alg. 1 (Sec. 5, "update assignments b using beam search"; App. C calls it
 * a search for the codeword combinations that minimise the error of the layer's outputs). The
 * paper gives no further detail; this is the reading implemented: every (row o, group g), with
 * the row's other groups held at their current codes, chooses its M codes by a beam search of
 * width K over the books in order k = 0..M-1, minimising the row's Drop-by-Drop objective
 *     sum_k lambda[k-1] * e^(k) S e^(k)^T,  e^(k) = W[o] - W^(k)[o],  S = (H + H^T)/2
 * (the trace form of aq_wmse above, restricted to the row). Every group is updated from the
 * same current codes (a Jacobi step: the groups' new codes are not combined while searching).
 * With delta_k the group's block of e^(k) and h_k = (S e^(k))_g - S_gg e^(k)_g its cross term
 * with the rest of the row, the group's terms are delta_k^T S_gg delta_k + 2 delta_k^T h_k;
 * book t extends each kept state (P = sum of its chosen codewords) by every codeword c of
 * C_t, scoring the parent's score + lambda[t] * (d^T S_gg d + 2 d^T h_{t+1}) with
 * d = w_g - s[o] (P + C_t[c]), and the K best extensions are kept, ordered by score, then the
 * parent's rank, then c. The result is the best state after book M-1. K = 2^(B(M-1)) makes the
 * search exhaustive (the exact minimiser per group).
 *   w        : device, [d_out][d_in] of book_dtype (the original weight)
 *   codes    : device, the current codes, natural layout [d_out][d_in/8][M], uint8 (B = 4 or
 *              8; B = 16 returns AQ_ERR_UNSUPPORTED: the 2^16-entry books do not fit on chip)
 *   books, scales : as aq_decode
 *   h        : device, [d_in][d_in] of h_dtype (AQ_F32 or AQ_BF16), row-major; any square H
 *   lambda   : HOST, M non-negative doubles (the weight of prefix k at index k-1), or NULL for
 *              all ones
 *   beam     : K, 1..16
 *   codes_out: device, same layout as codes, 16-byte aligned; may be codes (in place: codes
 *              are read only before any is written)
 *   workspace: device, aq_beam_workspace_bytes(layout) bytes, 16-byte aligned: a status word,
 *              S (d_in^2 floats), the residuals E_k and the products E_k S of every prefix
 *              (2 * M * d_out * d_in floats). No initialisation needed.
 * Arithmetic: fp32 throughout (residuals, E_k S on the CUDA cores, scores); with inputs whose
 * sums are exact in fp32 the codes equal the fp64 search's exactly. Stream-ordered; errors:
 * as aq_gemv. */
size_t aq_beam_workspace_bytes(const aq_layout* layout);
aq_status aq_beam_search(const aq_layout* layout, const void* w, const void* codes,
                         const void* books, const void* scales, const void* h, int h_dtype,
                         const double* lambda, int beam, void* codes_out, void* workspace,
                         size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------- dynamic loading
 * Device storage for one layer that holds only a prefix of its codebooks. One stored model
 * serves every bit width, and each deployment keeps as many codebooks on the device as its
 * memory or latency budget allows, loading more (or dropping some) at run time (Sec. 1 and
 * Sec. 5). Since the planes are codebook-major, a prefix is one contiguous byte range.
 * A store reserves device address space for the whole layer once and backs with physical
 * memory only the scales, the codebooks and the planes of the resident prefix (in whole
 * allocation granules, the device's minimum for virtual-memory mappings, 2 MiB on current
 * GPUs). Raising the prefix maps memory behind the resident planes and copies the new planes
 * in; lowering it releases the memory of the dropped planes. The device addresses never
 * move: pointers taken from a store stay valid for its life and may be passed to every
 * compute entry point with any m up to the resident prefix. A call with a larger m would read
 * unmapped addresses: the caller must not make one. These entry points allocate and free
 * device memory; a store is used by one host thread at a time. */
typedef struct aq_store aq_store;   /* opaque */

/* Create an empty store (prefix 0) for layout on the current device: reserves the address
 * range and maps memory for the scales and all M codebooks (2^B*16 bytes per codebook), none
 * for planes. Synchronous.
 *   store : receives the handle (NULL on failure).
 * Errors: AQ_ERR_INVALID_ARG / AQ_ERR_UNSUPPORTED (null store or a bad layout, as aq_pack),
 * AQ_ERR_CUDA (a runtime or driver call failed, e.g. out of memory; see aq_last_error). */
aq_status aq_store_create(const aq_layout* layout, aq_store** store);

/* Make planes 0..m-1 and codebooks 0..m-1 resident, 0 <= m <= M; m0 = the current prefix.
 * Raising (m > m0) maps memory for planes m0..m-1, then enqueues on stream the copies of
 * planes m0..m-1 and codebooks m0..m-1, and of the scales when m0 = 0, from:
 *   src_planes : the packed planes of all M codebooks, aq_packed_bytes(layout, M) bytes laid
 *                out as aq_pack writes them (only planes m0..m-1 are read)
 *   src_books  : [M][2^B][8] of book_dtype (only codebooks m0..m-1 are read)
 *   src_scales : [d_out] of scale_dtype (read only when m0 = 0)
 * Each may be host memory (pinned, for a copy that runs asynchronously) or device memory, and
 * must stay valid until the copies have run. Work that reads the new prefix must be ordered
 * after them: enqueue it on stream, or make its stream wait for an event recorded there.
 * Lowering (m < m0) is ordered on stream and does not wait: the memory that only planes
 * m..m0-1 use (the granule that plane m-1 shares with plane m stays) is released once the
 * work enqueued on stream before the call has finished. Work that reads the dropped planes
 * must therefore be enqueued on stream before the call (or be ordered before it), and no
 * later work may read them. The release itself happens in a later call on the store that
 * finds that work finished (aq_store_set_prefix, aq_store_device_bytes, aq_store_destroy);
 * a raise that needs the addresses again first takes the allocations back instead. No other
 * stream of the process is made to wait. The src pointers are not used and may be NULL. m = m0
 * does nothing.
 * Errors: AQ_ERR_INVALID_ARG (null store, m outside 0..M, a NULL src pointer that a raise
 * needs), AQ_ERR_CUDA (mapping, copy or event failed; the prefix then stays m0). */
aq_status aq_store_set_prefix(aq_store* store, int m, const void* src_planes,
                              const void* src_books, const void* src_scales, void* stream);

/* The resident prefix (0 for a NULL store). */
int aq_store_prefix(const aq_store* store);
/* Device addresses of the store's planes ([M planes], plane k at k*aq_plane_bytes), codebooks
 * ([M][2^B][8]) and scales ([d_out]); fixed for the store's life, 16-byte aligned, readable
 * for the resident prefix only. NULL for a NULL store. */
void* aq_store_planes(const aq_store* store);
void* aq_store_books(const aq_store* store);
void* aq_store_scales(const aq_store* store);
/* Bytes of device memory the store holds (0 for a NULL store): the scales, the codebooks, the
 * resident planes and dropped planes whose release still waits for their stream. Dropped
 * planes whose stream work has finished are released first, so after the caller's stream has
 * been synchronised the count is that of the resident prefix. */
size_t aq_store_device_bytes(aq_store* store);

/* Synchronise the device, release the store's memory and address range, free the handle.
 * NULL: nothing (AQ_OK). Errors: AQ_ERR_CUDA if the synchronisation reported an error (the
 * store is released all the same). */
aq_status aq_store_destroy(aq_store* store);

/* ---------------------------------------------------------------- workspace helpers
 * aq_selftest_wait: self-test of the library's failure detection (no counterpart in the
 * paper). Enqueues a one-thread kernel that waits, through the same time-bounded mbarrier wait
 * the compute kernels use (about 2 s), for a barrier phase that nothing completes; when the
 * wait gives up it records AQ_ERR_TIMEOUT in the workspace status word and returns, leaving
 * the context usable. aq_workspace_status then reports AQ_ERR_TIMEOUT once.
 *   workspace : device, at least 256 bytes, 16-byte aligned, zero-filled.
 * aq_workspace_init: enqueue a zero-fill of bytes at workspace (cudaMemsetAsync).
 * aq_workspace_status: SYNCHRONISES stream, then returns the device-side status a kernel
 * recorded in the workspace (AQ_OK if none) and clears it. */
aq_status aq_selftest_wait(void* workspace, size_t workspace_bytes, void* stream);

/* aq_selftest_read: a read probe for measurement (no counterpart in the paper). Enqueues one
 * kernel with the launch shape of the one-token GEMV (one CTA per SM, programmatic dependent
 * launch, the source requested before waiting for the preceding kernel) that only reads:
 * the XOR of all 32-bit words of src[0, bytes) is XORed into *sink. Timed back to back, it
 * gives the per-call cost of reading the same bytes with nothing computed, the floor that a
 * GEMV call of the same size is compared with.
 *   src   : device, 16-byte aligned, bytes a multiple of 16 (read only)
 *   sink  : device, one 32-bit word, 4-byte aligned (the caller zeroes it to check the fold)
 * Errors: AQ_ERR_INVALID_ARG (sink NULL, or src NULL with bytes > 0), AQ_ERR_ALIGNMENT. */
aq_status aq_selftest_read(const void* src, size_t bytes, void* sink, void* stream);
aq_status aq_workspace_init(void* workspace, size_t bytes, void* stream);
aq_status aq_workspace_status(void* workspace, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* AQ_H */
