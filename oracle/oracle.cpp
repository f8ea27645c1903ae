// CPU oracle for the multi-bitwidth additive-codebook dequantize-and-multiply.
//
// TEST INFRASTRUCTURE ONLY. This file is the plain, slow, obviously correct statement of
// what the GPU library computes. Only the test-suite, the smoke check and the CPU-baseline
// leg of the benchmark may load it. It shares no code, header, table or helper with the
// CUDA library: every conversion below is written here from the IEEE-754 definitions.
//
// What it follows (Drop-by-Drop, arxiv 2606.12876):
//   * Sec. 3.2 ("Additive Quantization and AQLM"): a weight row is split into groups of g
//     consecutive inputs; group j of row i is the sum over the M codebooks of the codeword
//     that the one-hot code b_{ijm} selects, and the row is the concatenation of its groups.
//   * Sec. 5 (Drop-by-Drop, the partial reconstruction W^(k)): the same sum restricted to the
//     first k codebooks; at inference a prefix of k <= M books is chosen as a deployment knob.
//     This file calls that prefix length m and numbers books 0..m-1.
//   * Sec. 2.2 (Y = W X): the layer output is the product of the (reconstructed) weight with
//     the input activations. Here activations are row vectors, y[t,o] = sum_i x[t,i] W[o,i].
//   * App. C ("Estimating Model Size", Eq. avg_bits): storage cost of codebooks, codes and
//     per-output-unit scales.
//   * Sec. 5 partial reconstruction W^(k) in fp64, the input of the per-prefix distortion
//     D^(k) (Sec. 2.2 Eq. wmse-task; evaluated in oracle/__init__.py).
//
// Readings where the paper is silent (each is listed in the design notes of the repository):
//   R1 the per-output-row scale s[o] multiplies the codebook sum: W[o, group] = s[o]*sum_k C_k[b].
//   R2 a codebook is stored as [2^B][g]: codeword j is g contiguous values.
//   R3 decode sums in fp32, in the fixed order k = 0..m-1, starting from +0.0f, then
//      multiplies by s[o] in fp32 and rounds once (round-to-nearest-even) to the book type.
//   R4 the codes term of Eq. avg_bits carries a factor M (the paper's own worked example,
//      approximately 2.002 bits for the 70B gate projection, holds only with it).
//
// Build: g++ -O2 -std=c++17 -ffp-contract=off -fopenmp -shared -fPIC (see oracle/build.py).
// -ffp-contract=off keeps a*b+c from being fused, which R3's bit-exact contract needs.

#include <cmath>
#include <cstdint>
#include <cstring>

namespace {

enum { DT_F16 = 0, DT_BF16 = 1 };

// ---- IEEE-754 binary16 / bfloat16 <-> binary32, written from the format definitions ----

// binary16: 1 sign bit, 5 exponent bits (bias 15), 10 fraction bits.
double f16_bits_to_double(uint16_t h) {
    const int sign = (h >> 15) & 1;
    const int expo = (h >> 10) & 0x1f;
    const int frac = h & 0x3ff;
    double v;
    if (expo == 0) {
        v = std::ldexp((double)frac, -24);                  // subnormal: frac * 2^-24
    } else if (expo == 31) {
        v = frac ? NAN : INFINITY;
    } else {
        v = std::ldexp((double)(1024 + frac), expo - 25);   // (1.frac) * 2^(expo-15)
    }
    return sign ? -v : v;
}

// bfloat16: the upper 16 bits of a binary32.
double bf16_bits_to_double(uint16_t b) {
    uint32_t u = (uint32_t)b << 16;
    float f;
    std::memcpy(&f, &u, 4);
    return (double)f;
}

double bits_to_double(uint16_t v, int dtype) {
    return dtype == DT_F16 ? f16_bits_to_double(v) : bf16_bits_to_double(v);
}

// Widening to float is exact for both formats (their value sets are subsets of binary32).
float bits_to_float(uint16_t v, int dtype) { return (float)bits_to_double(v, dtype); }

// binary32 -> binary16, round to nearest, ties to even.
uint16_t float_to_f16_rne(float x) {
    uint32_t f;
    std::memcpy(&f, &x, 4);
    const uint16_t sign = (uint16_t)((f >> 16) & 0x8000u);
    const uint32_t a = f & 0x7fffffffu;
    if (a >= 0x7f800000u) return (uint16_t)(sign | (a > 0x7f800000u ? 0x7e00u : 0x7c00u));
    const int e = (int)(a >> 23) - 127;          // unbiased exponent of a normal binary32
    const uint32_t mant = a & 0x7fffffu;
    if (e >= -14) {                               // lands in the binary16 normal range (or overflows)
        if (e > 15) return (uint16_t)(sign | 0x7c00u);
        uint32_t h = ((uint32_t)(e + 15) << 10) | (mant >> 13);
        const uint32_t rem = mant & 0x1fffu;      // the 13 dropped fraction bits
        if (rem > 0x1000u || (rem == 0x1000u && (h & 1u))) h += 1;  // a carry may reach 0x7c00 = inf
        return (uint16_t)(sign | h);
    }
    if (e < -25) return sign;                     // below half the smallest subnormal: rounds to 0
    // Subnormal result: count units of 2^-24. The value is sig * 2^(e-23), sig has 24 bits.
    const uint32_t sig = mant | 0x800000u;
    const int shift = -1 - e;                     // 14..24
    uint32_t q = sig >> shift;
    const uint32_t rem = sig & ((1u << shift) - 1u);
    const uint32_t half = 1u << (shift - 1);
    if (rem > half || (rem == half && (q & 1u))) q += 1;  // q == 1024 is the smallest normal
    return (uint16_t)(sign | q);
}

// binary32 -> bfloat16, round to nearest, ties to even (drop the low 16 bits).
uint16_t float_to_bf16_rne(float x) {
    uint32_t f;
    std::memcpy(&f, &x, 4);
    if ((f & 0x7fffffffu) > 0x7f800000u) return (uint16_t)(((f >> 16) & 0x8000u) | 0x7fc0u);
    uint32_t keep = f >> 16;
    const uint32_t rem = f & 0xffffu;
    if (rem > 0x8000u || (rem == 0x8000u && (keep & 1u))) keep += 1;  // carry into inf is correct
    return (uint16_t)keep;
}

uint16_t float_to_bits_rne(float x, int dtype) {
    return dtype == DT_F16 ? float_to_f16_rne(x) : float_to_bf16_rne(x);
}

// Code b_{o,g,k} from the natural (out, in/G, M) code tensor; element type u8 for B <= 8,
// u16 for 8 < B <= 16.
inline uint32_t code_at(const void* codes, int B, long idx) {
    return B <= 8 ? (uint32_t)((const uint8_t*)codes)[idx] : (uint32_t)((const uint16_t*)codes)[idx];
}

int check_shape(int out, int in, int G, int M, int B, int m) {
    if (out < 0 || in < 0 || G <= 0 || M <= 0 || B <= 0 || B > 16) return 1;
    if (in % G != 0) return 1;
    if (m < 1 || m > M) return 1;
    return 0;
}

}  // namespace

extern "C" {

// App. C, Eq. avg_bits, with reading R4 (codes term times M):
//   bits = 16*g*M*2^B + M*d_out*(d_in/g)*B + 16*d_out, divided by d_out*d_in.
double oracle_avg_bits(long d_out, long d_in, int g, int M, int B) {
    const double codebooks = 16.0 * g * M * std::ldexp(1.0, B);
    const double codes = (double)M * (double)d_out * ((double)d_in / g) * B;
    const double scales = 16.0 * (double)d_out;
    return (codebooks + codes + scales) / ((double)d_out * (double)d_in);
}

// Bits per weight of the codes alone for a prefix of m books: m*B/g (Sec. 5 prefix, App. C).
double oracle_prefix_code_bits(int g, int m, int B) { return (double)m * B / g; }

// Decode (Sec. 3.2 group reconstruction restricted to the first m books as in Sec. 5), under
// readings R1-R3. books: [M][2^B][G] values of book_dtype (bit patterns); codes: natural
// (out, in/G, M); scales: [out] of scale_dtype; w_out: [out][in] bit patterns of book_dtype.
int oracle_decode(int out, int in, int G, int M, int B, int m, const void* codes,
                  const uint16_t* books, int book_dtype, const uint16_t* scales, int scale_dtype,
                  uint16_t* w_out) {
    if (check_shape(out, in, G, M, B, m)) return 1;
    const long ng = in / G;
    const long book_stride = (1L << B) * G;
#pragma omp parallel for schedule(static)
    for (long o = 0; o < out; ++o) {
        const float s = bits_to_float(scales[o], scale_dtype);
        for (long g = 0; g < ng; ++g) {
            for (int e = 0; e < G; ++e) {
                float acc = 0.0f;
                for (int k = 0; k < m; ++k) {
                    const uint32_t j = code_at(codes, B, (o * ng + g) * M + k);
                    acc = acc + bits_to_float(books[k * book_stride + (long)j * G + e], book_dtype);
                }
                const float v = acc * s;
                w_out[o * in + g * G + e] = float_to_bits_rne(v, book_dtype);
            }
        }
    }
    return 0;
}

// Exact product (the parity reference): W_m in fp64 from the stored values widened exactly,
// W_m[o, g*G+e] = s[o] * sum_{k<m} C_k[b_{o,g,k}][e], then y[t,o] = sum_i x[t,i] * W_m[o,i]
// accumulated in fp64 in the order i = 0..in-1. x: [batch][in] of x_dtype; y: [batch][out].
int oracle_product_exact(int out, int in, int G, int M, int B, int m, const void* codes,
                         const uint16_t* books, int book_dtype, const uint16_t* scales,
                         int scale_dtype, const uint16_t* x, int x_dtype, int batch, double* y) {
    if (check_shape(out, in, G, M, B, m) || batch < 0) return 1;
    const long ng = in / G;
    const long book_stride = (1L << B) * G;
#pragma omp parallel
    {
        double* wrow = new double[in > 0 ? in : 1];
#pragma omp for schedule(static)
        for (long o = 0; o < out; ++o) {
            const double s = bits_to_double(scales[o], scale_dtype);
            for (long g = 0; g < ng; ++g) {
                for (int e = 0; e < G; ++e) {
                    double acc = 0.0;
                    for (int k = 0; k < m; ++k) {
                        const uint32_t j = code_at(codes, B, (o * ng + g) * M + k);
                        acc += bits_to_double(books[k * book_stride + (long)j * G + e], book_dtype);
                    }
                    wrow[g * G + e] = s * acc;
                }
            }
            for (long t = 0; t < batch; ++t) {
                double sum = 0.0;
                for (long i = 0; i < in; ++i) sum += bits_to_double(x[t * in + i], x_dtype) * wrow[i];
                y[t * out + o] = sum;
            }
        }
        delete[] wrow;
    }
    return 0;
}

// Exact partial reconstruction W^(m) of Sec. 5 in fp64 (no rounding): the stored values
// widened exactly, w_out[o][g*G+e] = s[o] * sum_{k<m} C_k[b_{o,g,k}][e], summed in book order.
// This is the reconstruction inside the distortion D^(k) of Sec. 5.
int oracle_reconstruct_exact(int out, int in, int G, int M, int B, int m, const void* codes,
                             const uint16_t* books, int book_dtype, const uint16_t* scales,
                             int scale_dtype, double* w_out) {
    if (check_shape(out, in, G, M, B, m)) return 1;
    const long ng = in / G;
    const long book_stride = (1L << B) * G;
#pragma omp parallel for schedule(static)
    for (long o = 0; o < out; ++o) {
        const double s = bits_to_double(scales[o], scale_dtype);
        for (long g = 0; g < ng; ++g)
            for (int e = 0; e < G; ++e) {
                double acc = 0.0;
                for (int k = 0; k < m; ++k) {
                    const uint32_t j = code_at(codes, B, (o * ng + g) * M + k);
                    acc += bits_to_double(books[k * book_stride + (long)j * G + e], book_dtype);
                }
                w_out[o * in + g * G + e] = s * acc;
            }
    }
    return 0;
}

// Diagnostic product with the rounded weights that oracle_decode stores:
// y[t,o] = sum_i x[t,i] * w[o,i] in fp64, w given as [out][in] bit patterns of w_dtype.
int oracle_product_dense(int out, int in, const uint16_t* w, int w_dtype, const uint16_t* x,
                         int x_dtype, int batch, double* y) {
    if (out < 0 || in < 0 || batch < 0) return 1;
#pragma omp parallel for schedule(static)
    for (long o = 0; o < out; ++o) {
        for (long t = 0; t < batch; ++t) {
            double sum = 0.0;
            for (long i = 0; i < in; ++i)
                sum += bits_to_double(x[t * in + i], x_dtype) * bits_to_double(w[o * in + i], w_dtype);
            y[t * out + o] = sum;
        }
    }
    return 0;
}

// Packed code-plane layout, stated as a plain index map (the layout is this library's own
// storage choice for the codes b of Sec. 3.2; the paper fixes only their meaning).
//   rows_pad = out rounded up to 32, ng_pad = in/G rounded up to 32, S = ng_pad/32 slices.
//   Plane k (k = 0..M-1) holds rows_pad*ng_pad codes; planes are contiguous, so the first m
//   planes are a prefix of the buffer. Inside a plane the order is [slice][row][position],
//   32 positions per (slice,row); position p of row o in slice s holds the code of group
//   s*32 + ((p + o) mod 32). Padding rows and groups hold code 0.
// Element size is 1 byte for 4 < B <= 8 and 2 bytes for B <= 16; for B <= 4 two codes
// share a byte: position p lives in byte p / 2 of its (slice, row) unit, in the low four bits
// for even p and the high four bits for odd p (a unit is then 16 bytes). planes must hold
// M*rows_pad*ng_pad codes.
int oracle_pack(int out, int in, int G, int M, int B, const void* codes, void* planes) {
    if (out < 0 || in < 0 || G <= 0 || M <= 0 || B <= 0 || B > 16 || in % G) return 1;
    const long ng = in / G;
    const long rows_pad = (out + 31) / 32 * 32;
    const long ng_pad = (ng + 31) / 32 * 32;
    const long plane = rows_pad * ng_pad;
    const long S = ng_pad / 32;
    if (B <= 4) std::memset(planes, 0, (size_t)(M * plane / 2));
    for (long k = 0; k < M; ++k)
        for (long s = 0; s < S; ++s)
            for (long o = 0; o < rows_pad; ++o)
                for (long p = 0; p < 32; ++p) {
                    const long g = s * 32 + ((p + o) % 32);
                    uint32_t v = 0;
                    if (o < out && g < ng) v = code_at(codes, B, (o * ng + g) * M + k);
                    const long dst = k * plane + (s * rows_pad + o) * 32 + p;
                    if (B <= 4) ((uint8_t*)planes)[dst / 2] |= (uint8_t)((v & 15u) << (4 * (p % 2)));
                    else if (B <= 8) ((uint8_t*)planes)[dst] = (uint8_t)v;
                    else ((uint16_t*)planes)[dst] = (uint16_t)v;
                }
    return 0;
}

// Conversion entry points, exposed so the tests can pin them against independent libraries.
uint16_t oracle_f32_to_f16(float x) { return float_to_f16_rne(x); }
uint16_t oracle_f32_to_bf16(float x) { return float_to_bf16_rne(x); }
double oracle_f16_to_f64(uint16_t h) { return f16_bits_to_double(h); }
double oracle_bf16_to_f64(uint16_t b) { return bf16_bits_to_double(b); }
void oracle_f32_to_bits_array(const float* x, uint16_t* out, long n, int dtype) {
    for (long i = 0; i < n; ++i) out[i] = float_to_bits_rne(x[i], dtype);
}
void oracle_bits_to_f64_array(const uint16_t* v, double* out, long n, int dtype) {
    for (long i = 0; i < n; ++i) out[i] = bits_to_double(v[i], dtype);
}

int oracle_num_threads(void);
}

#ifdef _OPENMP
#include <omp.h>
extern "C" int oracle_num_threads(void) { return omp_get_max_threads(); }
extern "C" void oracle_set_num_threads(int n) { omp_set_num_threads(n > 0 ? n : 1); }
#else
extern "C" int oracle_num_threads(void) { return 1; }
extern "C" void oracle_set_num_threads(int) {}
#endif
