// Exact in-register dequantisation and dot products of one 16-byte unit of packed codes
// with fp32 activations, used by the GEMV kernels (gemv.cu). Each code becomes an exact fp32 value through a "magic number"
// (the code placed in the mantissa of a float with a fixed exponent, the offset subtracted
// exactly); products and their sums are fp32 FMAs on packed pairs (FFMA2) in a fixed order.
#pragma once

#include "common.cuh"

namespace emb {
namespace dq {

__device__ __forceinline__ float lo_bf16(uint32_t h) { return __uint_as_float(h << 16); }
__device__ __forceinline__ float hi_bf16(uint32_t h) { return __uint_as_float(h & 0xFFFF0000u); }
// (a & mask) | bits in one LOP3 (written out: the compiler otherwise emits an AND and
// an OR when both constants are immediates).
__device__ __forceinline__ uint32_t and_or(uint32_t a, uint32_t mask, uint32_t bits) {
    uint32_t d;
    asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(d) : "r"(a), "r"(mask), "r"(bits));
    return d;
}
// Nibble field of v selected by mask, as the binary32 2^23 + field (exact).
__device__ __forceinline__ float magic(uint32_t v, uint32_t mask) { return __uint_as_float(and_or(v, mask, 0x4B000000u)); }

// 16 Q8_0 codes (one unit) times 16 fp32 activations -> fp32 partial sum.
// __byte_perm(v ^ 0x80808080, 0x4B000000, 0x7540 + i) is the binary32 2^23 + (q_i + 128)
// exactly; subtracting 2^23 + 128 leaves q_i exactly.
__device__ __forceinline__ float dot_q8_unit(const uint4 c, const float* x) {
    const uint32_t w[4] = {c.x, c.y, c.z, c.w};
    const float2 off = make_float2(-8388736.0f, -8388736.0f);  // -(2^23 + 128)
    float2 acc = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const uint32_t v = w[j] ^ 0x80808080u;
        const float2 q01 = __fadd2_rn(make_float2(__uint_as_float(__byte_perm(v, 0x4B000000u, 0x7540u)),
                                                  __uint_as_float(__byte_perm(v, 0x4B000000u, 0x7541u))),
                                      off);
        const float2 q23 = __fadd2_rn(make_float2(__uint_as_float(__byte_perm(v, 0x4B000000u, 0x7542u)),
                                                  __uint_as_float(__byte_perm(v, 0x4B000000u, 0x7543u))),
                                      off);
        acc = __ffma2_rn(q01, make_float2(x[4 * j + 0], x[4 * j + 1]), acc);
        acc = __ffma2_rn(q23, make_float2(x[4 * j + 2], x[4 * j + 3]), acc);
    }
    return acc.x + acc.y;
}

// 32 Q4_0 codes (one block, 16 bytes) times 32 fp32 activations -> sum of (q-8)*x.
// Word j holds codes 4j..4j+3 in its low nibbles and 16+4j..16+4j+3 in its high nibbles.
// A nibble at bit s (s <= 16) OR-ed into 0x4B000000 is 2^23 + q*2^s; one FMA with
// (2^-s, -(2^(23-s) + 8)) turns it into q - 8 exactly. Nibbles at bits 20..28 are
// first shifted down by 12.
__device__ __forceinline__ float dot_q4_unit(const uint4 c, const float* x) {
    const uint32_t w[4] = {c.x, c.y, c.z, c.w};
    const float2 s_a = make_float2(1.0f, 0x1p-8f), o_a = make_float2(-(0x1p23f + 8.0f), -(0x1p15f + 8.0f));
    const float2 s_b = make_float2(0x1p-4f, 0x1p-12f), o_b = make_float2(-(0x1p19f + 8.0f), -(0x1p11f + 8.0f));
    const float2 s_c = make_float2(0x1p-16f, 0x1p-12f), o_c = make_float2(-(0x1p7f + 8.0f), -(0x1p11f + 8.0f));
    const float2 s_d = make_float2(0x1p-8f, 0x1p-16f), o_d = make_float2(-(0x1p15f + 8.0f), -(0x1p7f + 8.0f));
    float2 acc = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const uint32_t v = w[j], v2 = w[j] >> 12;
        // codes 4j, 4j+1 (bits 0..3, 8..11)
        const float2 a = __ffma2_rn(make_float2(magic(v, 0xFu), magic(v, 0xF00u)), s_a, o_a);
        // codes 16+4j, 16+4j+1 (bits 4..7, 12..15)
        const float2 b = __ffma2_rn(make_float2(magic(v, 0xF0u), magic(v, 0xF000u)), s_b, o_b);
        // codes 4j+2, 4j+3 (bits 16..19, 24..27 -> 12..15 after the shift)
        const float2 cc = __ffma2_rn(make_float2(magic(v, 0xF0000u), magic(v2, 0xF000u)), s_c, o_c);
        // codes 16+4j+2, 16+4j+3 (bits 20..23 -> 8..11, 28..31 -> 16..19)
        const float2 d = __ffma2_rn(make_float2(magic(v2, 0xF00u), magic(v2, 0xF0000u)), s_d, o_d);
        acc = __ffma2_rn(a, make_float2(x[4 * j + 0], x[4 * j + 1]), acc);
        acc = __ffma2_rn(cc, make_float2(x[4 * j + 2], x[4 * j + 3]), acc);
        acc = __ffma2_rn(b, make_float2(x[16 + 4 * j + 0], x[16 + 4 * j + 1]), acc);
        acc = __ffma2_rn(d, make_float2(x[16 + 4 * j + 2], x[16 + 4 * j + 3]), acc);
    }
    return acc.x + acc.y;
}

// 32 Q6_0 codes (one block: 16 bytes of low nibbles c, 8 bytes of high bits h) times 32
// fp32 activations -> sum of (q-32)*x. Low word j holds the low nibbles of codes 4j..4j+3
// (bits 0-3 of its bytes) and 16+4j..16+4j+3 (bits 4-7); high word j&1 shifted right by
// 2*(j>>1) holds their high bits at bits 0-1 and 4-5 of the same bytes. So every byte of
// a = (c & 0x0F..) | (h & 0x03..) << 4 and of b = (c >> 4 & 0x0F..) | (h & 0x30..) is a
// whole 6-bit code; __byte_perm(., 0x4B000000, 0x7540 + i) is 2^23 + q exactly and
// subtracting 2^23 + 32 leaves q - 32 exactly.
__device__ __forceinline__ float dot_q6_unit(const uint4 c, const uint2 h, const float* x) {
    const uint32_t w[4] = {c.x, c.y, c.z, c.w};
    const float2 off = make_float2(-8388640.0f, -8388640.0f);  // -(2^23 + 32)
    float2 acc = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const uint32_t hh = ((j & 1) ? h.y : h.x) >> (2 * (j >> 1));
        const uint32_t a = and_or(w[j], 0x0F0F0F0Fu, (hh & 0x03030303u) << 4);
        const uint32_t b = and_or(w[j] >> 4, 0x0F0F0F0Fu, hh & 0x30303030u);
        const float2 a01 = __fadd2_rn(make_float2(__uint_as_float(__byte_perm(a, 0x4B000000u, 0x7540u)),
                                                  __uint_as_float(__byte_perm(a, 0x4B000000u, 0x7541u))), off);
        const float2 a23 = __fadd2_rn(make_float2(__uint_as_float(__byte_perm(a, 0x4B000000u, 0x7542u)),
                                                  __uint_as_float(__byte_perm(a, 0x4B000000u, 0x7543u))), off);
        const float2 b01 = __fadd2_rn(make_float2(__uint_as_float(__byte_perm(b, 0x4B000000u, 0x7540u)),
                                                  __uint_as_float(__byte_perm(b, 0x4B000000u, 0x7541u))), off);
        const float2 b23 = __fadd2_rn(make_float2(__uint_as_float(__byte_perm(b, 0x4B000000u, 0x7542u)),
                                                  __uint_as_float(__byte_perm(b, 0x4B000000u, 0x7543u))), off);
        acc = __ffma2_rn(a01, make_float2(x[4 * j + 0], x[4 * j + 1]), acc);
        acc = __ffma2_rn(a23, make_float2(x[4 * j + 2], x[4 * j + 3]), acc);
        acc = __ffma2_rn(b01, make_float2(x[16 + 4 * j + 0], x[16 + 4 * j + 1]), acc);
        acc = __ffma2_rn(b23, make_float2(x[16 + 4 * j + 2], x[16 + 4 * j + 3]), acc);
    }
    return acc.x + acc.y;
}

}  // namespace dq
}  // namespace emb
