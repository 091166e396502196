// Quantisation (offline packing) and test-support dequantisation kernels.
//
// Formats: the library's definitions of the paper's 8-, 6- and 4-bit weight
// configurations (Section 4, Table 3), written out in include/emb_qmm.h.
// Arithmetic is IEEE fp32 with explicit round-to-nearest intrinsics so that the
// packed bytes are reproducible bit for bit: max|w| (or the signed extreme),
// one correctly rounded division, one fp16 rounding of the scale, one correctly
// rounded division per weight and roundf (half away from zero).
#include "common.cuh"

namespace emb {
namespace {

constexpr unsigned kFull = 0xffffffffu;

// One warp per 32-weight block; lane i owns weight i of the block.
__global__ void __launch_bounds__(256) quantize_q8_0_kernel(const float* __restrict__ W,
                                                            int64_t N, int64_t K,
                                                            int8_t* __restrict__ codes,
                                                            __half* __restrict__ scales,
                                                            int64_t ldS) {
    const int lane = threadIdx.x & 31;
    const int64_t nb = K / kQBlock;
    const int64_t total = N * nb;
    int64_t warp = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = (int64_t(gridDim.x) * blockDim.x) >> 5;
    for (; warp < total; warp += nwarps) {
        const int64_t n = warp / nb, b = warp % nb;
        const float w = W[n * K + b * kQBlock + lane];
        const unsigned amax_bits = __reduce_max_sync(kFull, __float_as_uint(fabsf(w)));
        const float amax = __uint_as_float(amax_bits);
        const __half dh = __float2half_rn(__fdiv_rn(amax, 127.0f));
        const float d = __half2float(dh);
        int q = 0;
        if (d != 0.0f) {
            const float t = roundf(__fdiv_rn(w, d));
            q = int(fminf(fmaxf(t, -127.0f), 127.0f));
        }
        codes[n * K + b * kQBlock + lane] = int8_t(q);
        if (lane == 0) scales[n * ldS + b] = dh;
    }
}

// Q4_0 (HALF = 8) and Q6_0 (HALF = 32): codes q - HALF in [-HALF, HALF - 1] against the
// signed extreme m of the block; Q6_0 also writes the 2-bit high plane.
template <int HALF>
__global__ void __launch_bounds__(256) quantize_signed_kernel(const float* __restrict__ W,
                                                              int64_t N, int64_t K,
                                                              uint8_t* __restrict__ codes,
                                                              uint8_t* __restrict__ high,
                                                              __half* __restrict__ scales,
                                                              int64_t ldS) {
    const int lane = threadIdx.x & 31;
    const int64_t nb = K / kQBlock;
    const int64_t total = N * nb;
    int64_t warp = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = (int64_t(gridDim.x) * blockDim.x) >> 5;
    for (; warp < total; warp += nwarps) {
        const int64_t n = warp / nb, b = warp % nb;
        const float w = W[n * K + b * kQBlock + lane];
        const unsigned abits = __float_as_uint(fabsf(w));
        const unsigned amax_bits = __reduce_max_sync(kFull, abits);
        // the signed weight of largest magnitude, lowest lane on ties; +0 for a zero block
        const unsigned ties = __ballot_sync(kFull, abits == amax_bits);
        const float mw = __shfl_sync(kFull, w, __ffs(ties) - 1);
        const float m = (amax_bits == 0u) ? 0.0f : mw;
        const __half dh = __float2half_rn(__fdiv_rn(m, -float(HALF)));
        const float d = __half2float(dh);
        int q = HALF;
        if (d != 0.0f) {
            const float t = roundf(__fdiv_rn(w, d));
            q = int(fminf(fmaxf(t, -float(HALF)), float(HALF - 1))) + HALF;
        }
        // low plane: byte j = low nibble of code j | low nibble of code j + 16 << 4
        const int q_16 = __shfl_down_sync(kFull, q, 16);
        if (lane < 16) codes[n * (K / 2) + b * 16 + lane] = uint8_t((q & 15) | ((q_16 & 15) << 4));
        if constexpr (HALF == 32) {
            // high plane: byte j = high bits of codes j, j+8, j+16, j+24 at bit pairs 0..3
            const int q_8 = __shfl_down_sync(kFull, q, 8);
            const int q_24 = __shfl_down_sync(kFull, q, 24);
            if (lane < 8)
                high[n * (K / 4) + b * 8 + lane] =
                    uint8_t((q >> 4) | ((q_8 >> 4) << 2) | ((q_16 >> 4) << 4) | ((q_24 >> 4) << 6));
        }
        if (lane == 0) scales[n * ldS + b] = dh;
    }
}

__device__ __forceinline__ float deq_one(int fmt, const uint8_t* codes, const uint8_t* high,
                                         const __half* scales, int64_t K, int64_t ldS, int64_t n,
                                         int64_t k) {
    const float d = __half2float(scales[n * ldS + k / kQBlock]);
    int q;
    if (fmt == EMB_Q8_0) {
        q = int(reinterpret_cast<const int8_t*>(codes)[n * K + k]);
    } else {
        const int64_t b = k / kQBlock, i = k % kQBlock;
        const uint8_t byte = codes[n * (K / 2) + b * 16 + (i & 15)];
        q = int((i < 16) ? (byte & 0xF) : (byte >> 4));
        if (fmt == EMB_Q6_0) {
            const uint8_t hb = high[n * (K / 4) + b * 8 + (i & 7)];
            q = (q | (((hb >> (2 * (i >> 3))) & 3) << 4)) - 32;
        } else {
            q -= 8;
        }
    }
    return __fmul_rn(d, float(q));  // exact: 11-bit x at most 8-bit significands
}

__global__ void dequant_f32_kernel(int fmt, const uint8_t* __restrict__ codes,
                                   const uint8_t* __restrict__ high,
                                   const __half* __restrict__ scales, int64_t N, int64_t K,
                                   int64_t ldS, float* __restrict__ out) {
    const int64_t total = N * K;
    for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
         i += int64_t(gridDim.x) * blockDim.x)
        out[i] = deq_one(fmt, codes, high, scales, K, ldS, i / K, i % K);
}

__global__ void dequant_bf16_kernel(int fmt, const uint8_t* __restrict__ codes,
                                    const uint8_t* __restrict__ high,
                                    const __half* __restrict__ scales, int64_t N, int64_t K,
                                    int64_t ldS, __nv_bfloat16* __restrict__ out) {
    const int64_t total = N * K;
    for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
         i += int64_t(gridDim.x) * blockDim.x)
        out[i] = __float2bfloat16_rn(deq_one(fmt, codes, high, scales, K, ldS, i / K, i % K));
}

int grid_for(int64_t items, int per_block) {
    int64_t g = (items + per_block - 1) / per_block;
    if (g > 152 * 64) g = 152 * 64;
    return int(g < 1 ? 1 : g);
}

}  // namespace

cudaError_t launch_quantize(int fmt, const float* W, int64_t N, int64_t K, void* img,
                            cudaStream_t s) {
    const Layout L = layout_of(fmt, N, K);
    // zero the whole image first: the padding bytes are part of the format
    cudaError_t e = cudaMemsetAsync(img, 0, size_t(L.total), s);
    if (e != cudaSuccess) return e;
    uint8_t* base = static_cast<uint8_t*>(img);
    __half* scales = reinterpret_cast<__half*>(base + L.scales_off);
    const int grid = grid_for(N * (K / kQBlock), 8);  // 8 warps per 256-thread block
    if (fmt == EMB_Q8_0)
        quantize_q8_0_kernel<<<grid, 256, 0, s>>>(W, N, K, reinterpret_cast<int8_t*>(base),
                                                  scales, L.ldS);
    else if (fmt == EMB_Q4_0)
        quantize_signed_kernel<8><<<grid, 256, 0, s>>>(W, N, K, base, nullptr, scales, L.ldS);
    else
        quantize_signed_kernel<32><<<grid, 256, 0, s>>>(W, N, K, base, base + L.high_off, scales,
                                                        L.ldS);
    return cudaGetLastError();
}

cudaError_t launch_dequant_f32(int fmt, const void* img, int64_t N, int64_t K, float* out,
                               cudaStream_t s) {
    const Layout L = layout_of(fmt, N, K);
    const uint8_t* base = static_cast<const uint8_t*>(img);
    dequant_f32_kernel<<<grid_for(N * K, 256), 256, 0, s>>>(
        fmt, base, base + L.high_off, reinterpret_cast<const __half*>(base + L.scales_off), N, K,
        L.ldS, out);
    return cudaGetLastError();
}

cudaError_t launch_dequant_bf16(int fmt, const void* img, int64_t N, int64_t K, uint16_t* out,
                                cudaStream_t s) {
    const Layout L = layout_of(fmt, N, K);
    const uint8_t* base = static_cast<const uint8_t*>(img);
    dequant_bf16_kernel<<<grid_for(N * K, 256), 256, 0, s>>>(
        fmt, base, base + L.high_off, reinterpret_cast<const __half*>(base + L.scales_off), N, K,
        L.ldS, reinterpret_cast<__nv_bfloat16*>(out));
    return cudaGetLastError();
}

}  // namespace emb
