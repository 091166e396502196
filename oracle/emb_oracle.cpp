// Oracle for the block-quantised weight x bf16 activation matmul.
//
// TEST INFRASTRUCTURE ONLY. This file is a plain, slow, obviously-correct CPU
// restatement of what the GPU path computes. Only tests/, __graft_entry__.smoke()
// and bench.py's cpu_baseline / reference leg may build, load or call it. It shares
// no code, header, table or constant with the CUDA library and includes no CUDA
// header; every conversion below is written out from the IEEE-754 definition.
//
// What is computed (the paper's 8-, 6- and 4-bit weight configurations, Section 4,
// Table 3; the paper fixes no byte format, so the block formats below are the readings
// listed in the design notes):
//   Q8_0: per 32 consecutive weights along K of one output row,
//         d = fp16(max|w| / 127), q = clamp(round_half_away(w / d), -127, 127), w' = d*q
//   Q4_0: m = the signed weight of largest magnitude (lowest index on ties),
//         d = fp16(m / -8), q = clamp(round_half_away(w / d), -8, 7) + 8, w' = d*(q-8)
//   Q6_0: the same with 6-bit codes: d = fp16(m / -32),
//         q = clamp(round_half_away(w / d), -32, 31) + 32 in 0..63, w' = d*(q-32)
//   matmul: Y[m][n] = sum_k w'[n][k] * x[m][k], accumulated in fp64, with the
//         per-element tolerance bound B[m][n] = 1e-3 * sum_k |w'[n][k] x[m][k]| + 1e-6.
//
// Packed image (restated here from the layout definition, not shared with the GPU code):
//   codes plane at byte 0: Q8_0 int8 [N][K]; Q4_0 uint8 [N][K/2] where, inside each
//     32-block, byte j (0..15) holds code j in its low nibble and code j+16 in its high one;
//     Q6_0: the low 4 bits of each code in a plane laid out like Q4_0's ([N][K/2]), then at
//     byte roundup(N*K/2, 256) the high 2 bits, uint8 [N][K/4], where inside each 32-block
//     byte j (0..7) holds the high bits of codes j, j+8, j+16, j+24 at bits 0-1, 2-3, 4-5, 6-7;
//   scales plane at byte roundup(codes_bytes, 256) (Q6_0: roundup of the end of the
//     high-bits plane): fp16 [N][ldS], ldS = roundup(K/32, 8);
//   every padding byte is zero.

#include <cmath>
#include <cstdint>
#include <cstring>
#include <thread>
#include <vector>
#include <sched.h>

namespace {

uint32_t f32_bits(float f) { uint32_t u; std::memcpy(&u, &f, 4); return u; }
float bits_f32(uint32_t u) { float f; std::memcpy(&f, &u, 4); return f; }

int64_t roundup(int64_t a, int64_t b) { return (a + b - 1) / b * b; }

// Shift a non-negative integer right by s bits, rounding to nearest, ties to even.
uint64_t shift_rne(uint64_t v, int s) {
    if (s <= 0) return v << (-s);
    if (s >= 64) return 0;
    uint64_t q = v >> s;
    uint64_t rem = v & ((uint64_t(1) << s) - 1);
    uint64_t half = uint64_t(1) << (s - 1);
    if (rem > half || (rem == half && (q & 1))) q += 1;
    return q;
}

}  // namespace

extern "C" {

// binary32 -> binary16, round to nearest even (IEEE-754 2008, 4.3.1 / 7.4 overflow to inf).
uint16_t ref_f32_to_f16(float f) {
    uint32_t u = f32_bits(f);
    uint16_t sign = uint16_t((u >> 16) & 0x8000u);
    int32_t e = int32_t((u >> 23) & 0xFF);
    uint32_t mant = u & 0x7FFFFFu;
    if (e == 0xFF) return uint16_t(sign | 0x7C00u | (mant ? 0x200u : 0u));  // inf / quiet NaN
    if (e == 0 && mant == 0) return sign;                                       // signed zero
    // value = sig * 2^(exp2 - 23) with sig the 24-bit significand (binary32 subnormals too)
    uint64_t sig = (e == 0) ? mant : (mant | 0x800000u);
    int32_t exp2 = (e == 0) ? -126 : e - 127;
    // binary16: normal when exp2 >= -14 (10 fraction bits), else subnormal with unit 2^-24
    uint64_t h;
    if (exp2 >= -14) {
        // keep 11 significant bits: shift by 13, then rebuild (carry may bump the exponent)
        uint64_t r = shift_rne(sig, 13);               // 11 or 12 bits
        int32_t he = exp2 + 15;
        if (r >= (1u << 11)) { r >>= 1; he += 1; }     // rounding carried out of the significand
        if (he >= 31) return uint16_t(sign | 0x7C00u); // overflow -> inf
        h = (uint64_t(he) << 10) | (r & 0x3FFu);
    } else {
        // subnormal result: round(sig * 2^(exp2-23) / 2^-24) = round(sig * 2^(exp2+1))
        int s = -(exp2 + 1);
        uint64_t r = shift_rne(sig, s);
        h = r;  // r == 1024 means it rounded up to the smallest normal: encoding is the same
    }
    return uint16_t(sign | h);
}

float ref_f16_to_f32(uint16_t h) {
    uint32_t sign = uint32_t(h & 0x8000u) << 16;
    uint32_t e = (h >> 10) & 0x1F;
    uint32_t mant = h & 0x3FFu;
    if (e == 0x1F) return bits_f32(sign | 0x7F800000u | (mant << 13));
    if (e == 0) {
        // subnormal: mant * 2^-24, exact in binary32
        float v = float(mant) * std::ldexp(1.0f, -24);
        return sign ? -v : v;
    }
    return bits_f32(sign | ((e - 15 + 127) << 23) | (mant << 13));
}

// binary32 -> bfloat16 (the top 16 bits of binary32), round to nearest even.
uint16_t ref_f32_to_bf16(float f) {
    uint32_t u = f32_bits(f);
    if (((u >> 23) & 0xFF) == 0xFF && (u & 0x7FFFFFu)) return uint16_t((u >> 16) | 0x40u);
    uint64_t r = shift_rne(u & 0x7FFFFFFFu, 16);     // magnitude; carry into the exponent is correct
    return uint16_t(((u >> 16) & 0x8000u) | r);
}

float ref_bf16_to_f32(uint16_t b) { return bits_f32(uint32_t(b) << 16); }

// Element-wise array forms of the four conversions above (for bulk tests).
void ref_f32_to_f16_n(const float* in, uint16_t* out, int64_t n) {
    for (int64_t i = 0; i < n; ++i) out[i] = ref_f32_to_f16(in[i]);
}
void ref_f16_to_f32_n(const uint16_t* in, float* out, int64_t n) {
    for (int64_t i = 0; i < n; ++i) out[i] = ref_f16_to_f32(in[i]);
}
void ref_f32_to_bf16_n(const float* in, uint16_t* out, int64_t n) {
    for (int64_t i = 0; i < n; ++i) out[i] = ref_f32_to_bf16(in[i]);
}

// Q6_0: byte offset of the high-bits plane.
static int64_t q6_high_offset(int64_t N, int64_t K) { return roundup(N * K / 2, 256); }

static int64_t scales_offset(int fmt, int64_t N, int64_t K) {
    if (fmt == 2) return roundup(q6_high_offset(N, K) + N * K / 4, 256);
    return roundup((fmt == 0) ? N * K : N * K / 2, 256);
}

// Byte size of the packed image (see header comment); 0 when the shape is invalid.
int64_t ref_packed_bytes(int fmt, int64_t N, int64_t K) {
    if ((fmt != 0 && fmt != 1 && fmt != 2) || N < 1 || K < 32 || K % 32) return 0;
    return scales_offset(fmt, N, K) + N * roundup(K / 32, 8) * 2;
}

// Quantise fp32 W [N][K] into a zero-initialised packed image. Returns 0, or -1 if invalid.
int ref_quantize(int fmt, const float* W, int64_t N, int64_t K, uint8_t* out) {
    int64_t total = ref_packed_bytes(fmt, N, K);
    if (!total) return -1;
    std::memset(out, 0, size_t(total));
    const int64_t nb = K / 32, ldS = roundup(nb, 8);
    uint16_t* scales = reinterpret_cast<uint16_t*>(out + scales_offset(fmt, N, K));
    for (int64_t n = 0; n < N; ++n) {
        for (int64_t b = 0; b < nb; ++b) {
            const float* w = W + n * K + b * 32;
            int q[32];
            uint16_t dh;
            if (fmt == 0) {
                float amax = 0.0f;
                for (int i = 0; i < 32; ++i) if (std::fabs(w[i]) > amax) amax = std::fabs(w[i]);
                float d32 = amax / 127.0f;
                dh = ref_f32_to_f16(d32);
                float d = ref_f16_to_f32(dh);
                for (int i = 0; i < 32; ++i) {
                    if (d == 0.0f) { q[i] = 0; continue; }
                    float t = std::round(w[i] / d);           // std::round: half away from zero
                    q[i] = int(t < -127.0f ? -127.0f : (t > 127.0f ? 127.0f : t));
                }
                int8_t* codes = reinterpret_cast<int8_t*>(out) + n * K + b * 32;
                for (int i = 0; i < 32; ++i) codes[i] = int8_t(q[i]);
            } else {
                // Q4_0 (half = 8) and Q6_0 (half = 32): codes q - half in [-half, half - 1]
                const float half = (fmt == 1) ? 8.0f : 32.0f;
                float amax = 0.0f, m = 0.0f;
                for (int i = 0; i < 32; ++i)
                    if (std::fabs(w[i]) > amax) { amax = std::fabs(w[i]); m = w[i]; }
                float d32 = m / -half;
                dh = ref_f32_to_f16(d32);
                float d = ref_f16_to_f32(dh);
                for (int i = 0; i < 32; ++i) {
                    if (d == 0.0f) { q[i] = int(half); continue; }
                    float t = std::round(w[i] / d);
                    q[i] = int(t < -half ? -half : (t > half - 1.0f ? half - 1.0f : t)) + int(half);
                }
                uint8_t* codes = out + n * (K / 2) + b * 16;
                for (int j = 0; j < 16; ++j) codes[j] = uint8_t((q[j] & 15) | ((q[j + 16] & 15) << 4));
                if (fmt == 2) {
                    uint8_t* high = out + q6_high_offset(N, K) + n * (K / 4) + b * 8;
                    for (int j = 0; j < 8; ++j)
                        high[j] = uint8_t((q[j] >> 4) | ((q[j + 8] >> 4) << 2) | ((q[j + 16] >> 4) << 4) |
                                          ((q[j + 24] >> 4) << 6));
                }
            }
            scales[n * ldS + b] = dh;
        }
    }
    return 0;
}

// Read back code i (0..K-1) of row n and its block scale as binary32.
static void load_code(int fmt, const uint8_t* img, int64_t N, int64_t K, int64_t n, int64_t k,
                      int* q, float* d) {
    const uint16_t* scales = reinterpret_cast<const uint16_t*>(img + scales_offset(fmt, N, K));
    *d = ref_f16_to_f32(scales[n * roundup(K / 32, 8) + k / 32]);
    if (fmt == 0) {
        *q = int(reinterpret_cast<const int8_t*>(img)[n * K + k]);
    } else {
        int64_t b = k / 32, i = k % 32;
        uint8_t byte = img[n * (K / 2) + b * 16 + (i % 16)];
        *q = (i < 16) ? (byte & 0xF) : (byte >> 4);
        if (fmt == 2) {  // high 2 bits: byte i % 8 of the block, bit pair i / 8
            uint8_t hb = img[q6_high_offset(N, K) + n * (K / 4) + b * 8 + (i % 8)];
            *q |= ((hb >> (2 * (i / 8))) & 3) << 4;
        }
    }
}

// w' as binary32: d*q (Q8_0), d*(q-8) (Q4_0) or d*(q-32) (Q6_0). The product of an 11-bit
// and an at most 8-bit significand is exact in binary32.
static float deq_value(int fmt, int q, float d) {
    return fmt == 0 ? d * float(q) : fmt == 1 ? d * float(q - 8) : d * float(q - 32);
}

int ref_dequant_f32(int fmt, const uint8_t* img, int64_t N, int64_t K, float* out) {
    if (!ref_packed_bytes(fmt, N, K)) return -1;
    for (int64_t n = 0; n < N; ++n)
        for (int64_t k = 0; k < K; ++k) {
            int q; float d;
            load_code(fmt, img, N, K, n, k, &q, &d);
            out[n * K + k] = deq_value(fmt, q, d);
        }
    return 0;
}

// bf16 staging value: one round-to-nearest-even of the exact binary32 dequantised weight.
int ref_dequant_bf16(int fmt, const uint8_t* img, int64_t N, int64_t K, uint16_t* out) {
    if (!ref_packed_bytes(fmt, N, K)) return -1;
    for (int64_t n = 0; n < N; ++n)
        for (int64_t k = 0; k < K; ++k) {
            int q; float d;
            load_code(fmt, img, N, K, n, k, &q, &d);
            out[n * K + k] = ref_f32_to_bf16(deq_value(fmt, q, d));
        }
    return 0;
}

static void matmul_rows(int fmt, const uint8_t* img, const uint16_t* X, int64_t M, int64_t N,
                        int64_t K, int64_t n0, int64_t n1, double* Y, double* B) {
    std::vector<double> w(static_cast<size_t>(K));
    for (int64_t n = n0; n < n1; ++n) {
        for (int64_t k = 0; k < K; ++k) {
            int q; float d;
            load_code(fmt, img, N, K, n, k, &q, &d);
            w[size_t(k)] = double(deq_value(fmt, q, d));
        }
        for (int64_t m = 0; m < M; ++m) {
            double acc = 0.0, mag = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                double p = w[size_t(k)] * double(ref_bf16_to_f32(X[m * K + k]));
                acc += p;
                mag += std::fabs(p);
            }
            Y[m * N + n] = acc;
            if (B) B[m * N + n] = 1e-3 * mag + 1e-6;
        }
    }
}

// Host threads this process may run on (the affinity mask, not the machine's core count).
int ref_host_threads(void) {
    cpu_set_t set;
    if (sched_getaffinity(0, sizeof(set), &set) == 0) return CPU_COUNT(&set);
    unsigned h = std::thread::hardware_concurrency();
    return h ? int(h) : 1;
}

// Y [M][N] fp64 = X [M][K] (bf16 bits) x w'^T; B (optional) gets the tolerance bound.
// nthreads <= 0 uses every thread of the affinity mask; rows n are split across threads,
// each output element is still a plain sequential sum over k.
int ref_qmatmul(int fmt, const uint8_t* img, const uint16_t* X, int64_t M, int64_t N, int64_t K,
                double* Y, double* B, int nthreads) {
    if (!ref_packed_bytes(fmt, N, K) || M < 1) return -1;
    if (nthreads <= 0) nthreads = ref_host_threads();
    if (nthreads > N) nthreads = int(N);
    if (nthreads <= 1) { matmul_rows(fmt, img, X, M, N, K, 0, N, Y, B); return 0; }
    std::vector<std::thread> pool;
    for (int t = 0; t < nthreads; ++t) {
        int64_t n0 = N * t / nthreads, n1 = N * (t + 1) / nthreads;
        pool.emplace_back(matmul_rows, fmt, img, X, M, N, K, n0, n1, Y, B);
    }
    for (auto& th : pool) th.join();
    return 0;
}

// Selected elements only: Y[i] = sum_k w'[ns[i]][k] * x[ms[i]][k] (fp64), B[i] its bound.
int ref_qmatmul_sampled(int fmt, const uint8_t* img, const uint16_t* X, int64_t M, int64_t N,
                        int64_t K, const int64_t* ms, const int64_t* ns, int64_t count,
                        double* Y, double* B) {
    if (!ref_packed_bytes(fmt, N, K) || M < 1) return -1;
    for (int64_t i = 0; i < count; ++i) {
        if (ms[i] < 0 || ms[i] >= M || ns[i] < 0 || ns[i] >= N) return -1;
        double acc = 0.0, mag = 0.0;
        for (int64_t k = 0; k < K; ++k) {
            int q; float d;
            load_code(fmt, img, N, K, ns[i], k, &q, &d);
            double p = double(deq_value(fmt, q, d)) * double(ref_bf16_to_f32(X[ms[i] * K + k]));
            acc += p;
            mag += std::fabs(p);
        }
        Y[i] = acc;
        if (B) B[i] = 1e-3 * mag + 1e-6;
    }
    return 0;
}

}  // extern "C"
