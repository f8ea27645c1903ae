// aq_beam_search: the code update of Alg. 1 ("update assignments b using beam search"; App. C:
// the search for codeword combinations that minimise the error of the layer's outputs), in
// the reading stated in aq.h: every (row o, group g), with the row's other groups at their
// current codes, chooses its M codes by a beam search of width K over the books in order,
// minimising the row's Drop-by-Drop objective sum_k lambda_k e^(k) S e^(k)^T (Sec. 5, the
// trace form of Sec. 2.2 with S the symmetric part of H). The terms that depend on the
// group's codes are delta_k^T S_gg delta_k + 2 delta_k^T h_k, with
// delta_k = w_g - s_o * (sum_{j<k} C_j[b_j]) and h_k = (S e^(k))_g - S_gg e^(k)_g.
//
// Kernels (all fp32):
//   beam_resid_kernel  E_k[o][i] = W[o][i] - s_o * (sum_{j<k} C_j[b_j])  (current codes)
//   beam_sym_kernel    S = (H + H^T) / 2
//   beam_gemm_kernel   V_k = E_k S (tiled, CUDA cores: the cross terms need fp32)
//   beam_kernel        one warp per (row, group): h_k, then the beam over the books
#include <cfloat>

#include "aq_internal.cuh"

namespace aq {
namespace {

constexpr int kBeamMaxK = 16;
constexpr int kBeamWarps = 8;

// The prefix weights lambda_1..lambda_M, passed by value.
struct Lambdas {
    float v[8];
};

// Workspace: [status 256 B][S: in*in][E: M*out*in][V: M*out*in] (fp32)
inline size_t beam_s_off() { return kWsStatusBytes; }
inline size_t beam_e_off(const Dims& d) { return round_up(beam_s_off() + (size_t)d.in * d.in * 4, 256); }
inline size_t beam_v_off(const Dims& d) {
    return round_up(beam_e_off(d) + (size_t)d.M * d.out * d.in * 4, 256);
}

template <int BDT, int SDT>
__global__ void beam_resid_kernel(const uint16_t* __restrict__ w, const void* __restrict__ codes,
                                  const uint16_t* __restrict__ books,
                                  const uint16_t* __restrict__ scales, float* __restrict__ E,
                                  int out, int in, int ng, int M, int B) {
    pdl_wait();
    pdl_launch_dependents();
    const size_t n = (size_t)out * ng;
    for (size_t t = (size_t)blockIdx.x * blockDim.x + threadIdx.x; t < n;
         t += (size_t)gridDim.x * blockDim.x) {
        const int o = (int)(t / ng), g = (int)(t % ng);
        const float s = bits_to_f32<SDT>(scales[o]);
        float wv[8], P[8];
        unpack8<BDT>(*(const uint4*)(w + (size_t)o * in + (size_t)g * 8), wv);
#pragma unroll
        for (int e = 0; e < 8; ++e) P[e] = 0.0f;
        for (int k = 0; k < M; ++k) {
            const size_t ci = ((size_t)o * ng + g) * M + k;
            const uint32_t c = B == 16 ? ((const uint16_t*)codes)[ci] : ((const uint8_t*)codes)[ci];
            float cv[8];
            unpack8<BDT>(*(const uint4*)(books + (((size_t)k << B) + c) * 8), cv);
            float* dst = E + ((size_t)k * out + o) * in + (size_t)g * 8;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                P[e] += cv[e];
                dst[e] = wv[e] - s * P[e];
            }
        }
    }
}

__global__ void beam_sym_kernel(const void* __restrict__ h, int h_dt, float* __restrict__ S, int in) {
    pdl_wait();
    pdl_launch_dependents();
    const size_t n = (size_t)in * in;
    for (size_t t = (size_t)blockIdx.x * blockDim.x + threadIdx.x; t < n;
         t += (size_t)gridDim.x * blockDim.x) {
        const size_t i = t / in, j = t % in;
        float a, b;
        if (h_dt == AQ_F32) {
            a = ((const float*)h)[i * in + j];
            b = ((const float*)h)[j * in + i];
        } else {
            a = bits_to_f32<AQ_BF16>(((const uint16_t*)h)[i * in + j]);
            b = bits_to_f32<AQ_BF16>(((const uint16_t*)h)[j * in + i]);
        }
        S[t] = (a + b) * 0.5f;
    }
}

// C[r][j] = sum_i A[r][i] * S[i][j] for r < rows, j < in (A = E of every prefix, rows = M*out).
// 64 x 64 tiles, 16-deep k steps through shared memory, 4 x 4 outputs per thread; the row
// tiles beyond gridDim.y are taken in turn by the same CTAs.
__global__ void __launch_bounds__(256) beam_gemm_kernel(const float* __restrict__ A,
                                                        const float* __restrict__ S,
                                                        float* __restrict__ C, int rows, int in) {
    __shared__ float As[16][65], Bs[16][64];
    pdl_wait();
    pdl_launch_dependents();
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int c0 = blockIdx.x * 64;
    for (int r0 = blockIdx.y * 64; r0 < rows; r0 += gridDim.y * 64) {
        float acc[4][4] = {};
        for (int k0 = 0; k0 < in; k0 += 16) {
            for (int i = threadIdx.x; i < 64 * 16; i += 256) {
                const int r = i / 16, kk = i % 16;
                As[kk][r] = (r0 + r < rows && k0 + kk < in) ? A[(size_t)(r0 + r) * in + k0 + kk] : 0.0f;
                const int kb = i / 64, cc = i % 64;
                Bs[kb][cc] = (k0 + kb < in && c0 + cc < in) ? S[(size_t)(k0 + kb) * in + c0 + cc] : 0.0f;
            }
            __syncthreads();
#pragma unroll
            for (int kk = 0; kk < 16; ++kk) {
                float a[4], b[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    a[u] = As[kk][ty * 4 + u];
                    b[u] = Bs[kk][tx * 4 + u];
                }
#pragma unroll
                for (int u = 0; u < 4; ++u)
#pragma unroll
                    for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(a[u], b[v], acc[u][v]);
            }
            __syncthreads();
        }
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int v = 0; v < 4; ++v) {
                const int r = r0 + ty * 4 + u, c = c0 + tx * 4 + v;
                if (r < rows && c < in) C[(size_t)r * in + c] = acc[u][v];
            }
    }
}

// Candidate order: smaller score first, then smaller index (parent rank * 2^B + codeword).
__device__ __forceinline__ bool before(float a, int ia, float b, int ib) {
    return a < b || (a == b && ia < ib);
}

// One warp per (row, group), the rows of one group handled by the warps of a CTA (the group's
// block S_gg and the codebooks are staged once per CTA). Per book t, the candidates are every
// (state, codeword) pair, index j = rank * 2^B + c; lane L scores j = L, L + 32, ... and keeps
// its K best in a sorted list; K rounds of a warp-wide minimum over the lists' heads then give
// the K best overall.
template <int BDT, int SDT>
__global__ void __launch_bounds__(kBeamWarps * 32)
beam_kernel(const uint16_t* __restrict__ w, const uint16_t* __restrict__ books,
            const uint16_t* __restrict__ scales, const float* __restrict__ S,
            const float* __restrict__ E, const float* __restrict__ V, void* __restrict__ codes_out,
            Lambdas lam, int out, int in, int ng, int M, int B, int K) {
    extern __shared__ __align__(16) float bsm[];
    const int nb = 1 << B;
    float* Cs = bsm;                                   // [M][nb][8] codebooks, fp32
    float* Sgg = Cs + (size_t)M * nb * 8;              // [8][8]
    float* wsh = Sgg + 64;                             // per warp: [M][8] h, then two beams
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    constexpr int kBeamFloats = kBeamMaxK * 9 + kBeamMaxK * 8;   // P[8] + score, codes as ints
    float* my = wsh + (size_t)warp * (8 * 8 + 2 * kBeamFloats + 32 * kBeamMaxK * 2);
    float* hv = my;                                    // [M][8]
    float* beamA = hv + 64;
    float* beamB = beamA + kBeamFloats;
    float* lst = beamB + kBeamFloats;                  // per lane: K (score, index) pairs
    pdl_wait();
    pdl_launch_dependents();
    const int g = blockIdx.y;
    for (int i = threadIdx.x; i < M * nb; i += blockDim.x) {
        float cv[8];
        unpack8<BDT>(*(const uint4*)(books + (size_t)i * 8), cv);
#pragma unroll
        for (int e = 0; e < 8; ++e) Cs[(size_t)i * 8 + e] = cv[e];
    }
    for (int i = threadIdx.x; i < 64; i += blockDim.x)
        Sgg[i] = S[(size_t)(g * 8 + i / 8) * in + g * 8 + i % 8];
    __syncthreads();

    for (int o = blockIdx.x * kBeamWarps + warp; o < out; o += gridDim.x * kBeamWarps) {
        const float s = bits_to_f32<SDT>(scales[o]);
        float wg[8];
        unpack8<BDT>(*(const uint4*)(w + (size_t)o * in + (size_t)g * 8), wg);
        // h_k = (S e^(k))_g - S_gg e^(k)_g, lane (k, e) for k < M, e < 8 (M <= 4 here per
        // pass of 32 lanes; two passes for more books)
        for (int idx = lane; idx < M * 8; idx += 32) {
            const int k = idx / 8, e = idx % 8;
            const float* ek = E + ((size_t)k * out + o) * in + (size_t)g * 8;
            float v = V[((size_t)k * out + o) * in + (size_t)g * 8 + e];
#pragma unroll
            for (int f = 0; f < 8; ++f) v -= Sgg[e * 8 + f] * ek[f];
            hv[idx] = v;
        }
        // the single empty state
        if (lane < 8) beamA[lane] = 0.0f;
        if (lane == 0) beamA[kBeamMaxK * 8] = 0.0f;    // score
        __syncwarp();
        int nstates = 1;
        float* cur = beamA;
        float* nxt = beamB;
        for (int t = 0; t < M; ++t) {
            const float lt = lam.v[t];
            const float* ht = hv + t * 8;
            float* myl = lst + (size_t)lane * kBeamMaxK * 2;
            int cnt = 0;
            const int ncand = nstates * nb;
            for (int j = lane; j < ncand; j += 32) {
                const int r = j / nb, c = j % nb;
                const float* P = cur + r * 8;
                const float* cw = Cs + ((size_t)t * nb + c) * 8;
                float d[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) d[e] = wg[e] - s * (P[e] + cw[e]);
                float q = 0.0f, l = 0.0f;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    float sd = 0.0f;
#pragma unroll
                    for (int f = 0; f < 8; ++f) sd += Sgg[e * 8 + f] * d[f];
                    q += d[e] * sd;
                    l += d[e] * ht[e];
                }
                float sc = cur[kBeamMaxK * 8 + r] + lt * (q + 2.0f * l);
                if (!(sc <= FLT_MAX)) sc = FLT_MAX;   // NaN and +inf last: keeps the order total
                // insert into this lane's sorted list of at most K
                if (cnt < K || before(sc, j, myl[(K - 1) * 2], __float_as_int(myl[(K - 1) * 2 + 1]))) {
                    int p = cnt < K ? cnt : K - 1;
                    while (p > 0 && before(sc, j, myl[(p - 1) * 2], __float_as_int(myl[(p - 1) * 2 + 1]))) {
                        myl[p * 2] = myl[(p - 1) * 2];
                        myl[p * 2 + 1] = myl[(p - 1) * 2 + 1];
                        --p;
                    }
                    myl[p * 2] = sc;
                    myl[p * 2 + 1] = __int_as_float(j);
                    if (cnt < K) ++cnt;
                }
            }
            // merge: K rounds of the warp-wide minimum of the lists' heads
            const int keep = ncand < K ? ncand : K;
            int head = 0;
            for (int i = 0; i < keep; ++i) {
                float bs = head < cnt ? myl[head * 2] : FLT_MAX;
                int bj = head < cnt ? __float_as_int(myl[head * 2 + 1]) : 0x7fffffff;
#pragma unroll
                for (int sh = 16; sh > 0; sh >>= 1) {
                    const float os = __shfl_xor_sync(0xffffffffu, bs, sh);
                    const int oj = __shfl_xor_sync(0xffffffffu, bj, sh);
                    if (before(os, oj, bs, bj)) {
                        bs = os;
                        bj = oj;
                    }
                }
                if (head < cnt && __float_as_int(myl[head * 2 + 1]) == bj) ++head;
                // new state i: parent rank bj / nb, codeword bj % nb
                // every round finds a real candidate (the lists hold at least `keep`), so bj
                // is one; the clamp only guards the shared-memory index
                const int r = min(bj / nb, nstates - 1), c = bj % nb;
                if (lane < 8) nxt[i * 8 + lane] = cur[r * 8 + lane] + Cs[((size_t)t * nb + c) * 8 + lane];
                if (lane == 0) nxt[kBeamMaxK * 8 + i] = bs;
                int* ncodes = (int*)(nxt + kBeamMaxK * 9);
                const int* ocodes = (const int*)(cur + kBeamMaxK * 9);
                if (lane < t) ncodes[i * 8 + lane] = ocodes[r * 8 + lane];
                if (lane == t) ncodes[i * 8 + t] = c;
            }
            __syncwarp();
            nstates = keep;
            float* tmp = cur;
            cur = nxt;
            nxt = tmp;
        }
        const int* best = (const int*)(cur + kBeamMaxK * 9);
        if (lane < M) {
            const size_t ci = ((size_t)o * ng + g) * M + lane;
            if (B == 16) ((uint16_t*)codes_out)[ci] = (uint16_t)best[lane];
            else ((uint8_t*)codes_out)[ci] = (uint8_t)best[lane];
        }
        __syncwarp();
    }
}

inline size_t beam_smem(int M, int B) {
    const int kBeamFloats = kBeamMaxK * 9 + kBeamMaxK * 8;
    return ((size_t)M * ((size_t)1 << B) * 8 + 64 +
            (size_t)kBeamWarps * (64 + 2 * kBeamFloats + 32 * kBeamMaxK * 2)) * 4;
}

template <int BDT, int SDT>
aq_status run_beam(const Dims& d, const void* w, const void* codes, const void* books,
                   const void* scales, const void* h, int h_dt, const Lambdas& lam, int K,
                   void* codes_out, void* ws, cudaStream_t st) {
    DeviceInfo di;
    if (aq_status e = device_info(&di); e != AQ_OK) return e;
    float* S = (float*)((char*)ws + beam_s_off());
    float* E = (float*)((char*)ws + beam_e_off(d));
    float* V = (float*)((char*)ws + beam_v_off(d));
    const int grid = di.sms * 8;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.stream = st;
    cfg.blockDim = dim3(256);
    cfg.gridDim = dim3(grid);
    if (aq_status e = cuda_ok(cudaLaunchKernelEx(&cfg, beam_resid_kernel<BDT, SDT>, (const uint16_t*)w, codes,
                                                 (const uint16_t*)books, (const uint16_t*)scales, E, d.out,
                                                 d.in, d.ng, d.M, d.B),
                              "cudaLaunchKernelEx (beam residuals)");
        e != AQ_OK)
        return e;
    if (aq_status e = cuda_ok(cudaLaunchKernelEx(&cfg, beam_sym_kernel, h, h_dt, S, d.in),
                              "cudaLaunchKernelEx (beam symmetric part)");
        e != AQ_OK)
        return e;
    const int row_tiles = (int)(((long long)d.M * d.out + 63) / 64);
    cfg.gridDim = dim3((d.in + 63) / 64, row_tiles < 65535 ? row_tiles : 65535);
    if (aq_status e = cuda_ok(cudaLaunchKernelEx(&cfg, beam_gemm_kernel, (const float*)E, (const float*)S, V,
                                                 d.M * d.out, d.in),
                              "cudaLaunchKernelEx (beam cross terms)");
        e != AQ_OK)
        return e;
    auto kern = beam_kernel<BDT, SDT>;
    const size_t smem = beam_smem(d.M, d.B);
    if (smem > (size_t)di.smem_optin) return AQ_ERR_UNSUPPORTED;
    if (cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        e != cudaSuccess)
        return cuda_fail(e, "cudaFuncSetAttribute");
    int xb = (d.out + kBeamWarps - 1) / kBeamWarps;
    const int want = (di.sms * 4 + d.ng - 1) / d.ng;   // enough CTAs to fill the SMs
    if (xb > want) xb = want < 1 ? 1 : want;
    cfg.gridDim = dim3(xb, d.ng);
    cfg.blockDim = dim3(kBeamWarps * 32);
    cfg.dynamicSmemBytes = smem;
    return cuda_ok(cudaLaunchKernelEx(&cfg, kern, (const uint16_t*)w, (const uint16_t*)books,
                                      (const uint16_t*)scales, (const float*)S, (const float*)E,
                                      (const float*)V, codes_out, lam, d.out, d.in, d.ng, d.M,
                                      d.B, K),
                   "cudaLaunchKernelEx (beam search)");
}

}  // namespace

size_t beam_ws_bytes(const Dims& d) { return beam_v_off(d) + (size_t)d.M * d.out * d.in * 4; }

aq_status launch_beam(const Dims& d, const void* w, const void* codes, const void* books,
                      const void* scales, const void* h, int h_dt, const double* lambda, int K,
                      void* codes_out, void* ws, cudaStream_t st) {
    if (d.out == 0) return AQ_OK;
    Lambdas lam = {};
    for (int k = 0; k < d.M; ++k) lam.v[k] = lambda ? (float)lambda[k] : 1.0f;
    const int key = (d.book_dt == AQ_BF16) * 2 + (d.scale_dt == AQ_BF16);
    switch (key) {
        case 0: return run_beam<AQ_F16, AQ_F16>(d, w, codes, books, scales, h, h_dt, lam, K, codes_out, ws, st);
        case 1: return run_beam<AQ_F16, AQ_BF16>(d, w, codes, books, scales, h, h_dt, lam, K, codes_out, ws, st);
        case 2: return run_beam<AQ_BF16, AQ_F16>(d, w, codes, books, scales, h, h_dt, lam, K, codes_out, ws, st);
        default: return run_beam<AQ_BF16, AQ_BF16>(d, w, codes, books, scales, h, h_dt, lam, K, codes_out, ws, st);
    }
}

}  // namespace aq
