// Internal declarations shared by the library's translation units (not installed).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "../../include/emb_qmm.h"

namespace emb {

constexpr int kQBlock = 32;  // weights per quantisation block (both formats)

__host__ __device__ inline int64_t roundup(int64_t a, int64_t b) { return (a + b - 1) / b * b; }

// Byte layout of one packed image (the format comment of emb_qweight_bytes).
struct Layout {
    int64_t codes_bytes;  // codes plane size (Q6_0: the low-nibble plane)
    int64_t high_off;     // Q6_0: byte offset of the 2-bit high plane (256-aligned); else 0
    int64_t scales_off;   // byte offset of the fp16 scales plane (256-aligned)
    int64_t ldS;          // scales row pitch in halves (multiple of 8)
    int64_t total;        // total image size in bytes
};

__host__ __device__ inline Layout layout_of(int fmt, int64_t N, int64_t K) {
    Layout L;
    L.codes_bytes = (fmt == EMB_Q8_0) ? N * K : N * K / 2;
    L.high_off = (fmt == EMB_Q6_0) ? roundup(L.codes_bytes, 256) : 0;
    L.scales_off = (fmt == EMB_Q6_0) ? roundup(L.high_off + N * K / 4, 256) : roundup(L.codes_bytes, 256);
    L.ldS = roundup(K / kQBlock, 8);
    L.total = L.scales_off + N * L.ldS * 2;
    return L;
}

// ------------------------------------------------------------------ epilogues
// Activations of the gated epilogues, in fp32 with the CUDA math library.
__device__ __forceinline__ float act_gelu_tanh(float g) {
    return 0.5f * g * (1.0f + tanhf(0.7978845608028654f * (g + 0.044715f * g * g * g)));
}
__device__ __forceinline__ float act_silu(float g) { return g / (1.0f + expf(-g)); }

// Store one result v for element (m, n) of a Y with N columns.
__device__ __forceinline__ void epi_store(int epi, void* Y, int64_t m, int64_t n, int64_t N, float v) {
    const int64_t i = m * N + n;
    if (epi == EMB_EPI_BF16) {
        reinterpret_cast<__nv_bfloat16*>(Y)[i] = __float2bfloat16_rn(v);
    } else if (epi == EMB_EPI_ADD) {
        float* y = reinterpret_cast<float*>(Y);
        y[i] = __fadd_rn(y[i], v);
    } else {
        reinterpret_cast<float*>(Y)[i] = v;
    }
}

// Gated epilogues: gate row n (even) and up row n + 1 give element (m, n / 2) of a bf16 Y
// with N / 2 columns.
__device__ __forceinline__ void epi_store_gated(int epi, void* Y, int64_t m, int64_t n, int64_t N,
                                                float gate, float up) {
    const float a = (epi == EMB_EPI_GEGLU) ? act_gelu_tanh(gate) : act_silu(gate);
    reinterpret_cast<__nv_bfloat16*>(Y)[m * (N / 2) + n / 2] = __float2bfloat16_rn(__fmul_rn(a, up));
}

// Results v of elements (m, n .. n + 3), N % 4 == 0 and n % 4 == 0 (Y 16-byte aligned): one
// 16-byte (fp32, residual add), 8-byte (bf16) or 4-byte (gated: gate rows n, n + 2, up rows
// n + 1, n + 3) access, with the same roundings as epi_store / epi_store_gated.
__device__ __forceinline__ void epi_store4(int epi, void* Y, int64_t m, int64_t n, int64_t N, float4 v) {
    const int64_t i = m * N + n;
    if (epi == EMB_EPI_F32) {
        *reinterpret_cast<float4*>(reinterpret_cast<float*>(Y) + i) = v;
    } else if (epi == EMB_EPI_ADD) {
        float4* y = reinterpret_cast<float4*>(reinterpret_cast<float*>(Y) + i);
        const float4 o = *y;
        *y = make_float4(__fadd_rn(o.x, v.x), __fadd_rn(o.y, v.y), __fadd_rn(o.z, v.z),
                         __fadd_rn(o.w, v.w));
    } else if (epi == EMB_EPI_BF16) {
        const __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
        uint2 u;
        u.x = *reinterpret_cast<const uint32_t*>(&lo);
        u.y = *reinterpret_cast<const uint32_t*>(&hi);
        *reinterpret_cast<uint2*>(reinterpret_cast<__nv_bfloat16*>(Y) + i) = u;
    } else {
        const float a0 = (epi == EMB_EPI_GEGLU) ? act_gelu_tanh(v.x) : act_silu(v.x);
        const float a1 = (epi == EMB_EPI_GEGLU) ? act_gelu_tanh(v.z) : act_silu(v.z);
        *reinterpret_cast<__nv_bfloat162*>(reinterpret_cast<__nv_bfloat16*>(Y) + m * (N / 2) + n / 2) =
            __floats2bfloat162_rn(__fmul_rn(a0, v.y), __fmul_rn(a1, v.w));
    }
}

// Device status word values (bit flags, OR-ed by kernels).
constexpr int kStatusTimeout = 1;

// Default bound for every spin-wait inside the library's kernels (nanoseconds of
// %globaltimer). Long enough for any legitimate wait, short enough that a lost
// arrival turns into EMB_ETIMEOUT instead of a hung GPU.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// ------------------------------------------------------------------ launchers
// Each returns cudaSuccess or the launch error. `status` is the device address of
// the library's status word.

cudaError_t launch_quantize(int fmt, const float* W, int64_t N, int64_t K, void* img,
                            cudaStream_t s);
cudaError_t launch_dequant_f32(int fmt, const void* img, int64_t N, int64_t K, float* out,
                               cudaStream_t s);
cudaError_t launch_dequant_bf16(int fmt, const void* img, int64_t N, int64_t K, uint16_t* out,
                                cudaStream_t s);

// Up to kMaxGroup matrices that read the same X (fused q/k/v or gate/up).
constexpr int kMaxGroup = 4;

struct MatRef {
    const uint8_t* codes;   // Q6_0: the low-nibble plane
    const __half* scales;
    void* Y;                // as the group's epilogue says
    int64_t N;
    const uint8_t* high;    // Q6_0: the 2-bit high plane; else nullptr
};

struct GroupRef {
    int fmt;
    int epi;                // emb_epilogue kind of every member (flags stripped)
    bool precise;           // EMB_PRECISE_OPERAND: two-operand weights in the tensor-core GEMM
    int n_mats;
    MatRef mats[kMaxGroup];
    const __nv_bfloat16* X;
    int64_t M;
    int64_t K;
    int64_t ldS;
    void* ws;               // caller workspace for the tensor-core GEMM's stream-K schedule, or NULL
    size_t ws_bytes;
};

// Weight-streaming GEMV for small M (register dequant, shuffle reductions).
// pdl: launch with programmatic stream serialisation (the kernel reads X only after
// griddepcontrol.wait, weights before).
cudaError_t launch_gemv(const GroupRef& g, bool pdl, int* status, cudaStream_t s);

// Tensor-core GEMM (tcgen05 + TMEM) for larger M.
cudaError_t launch_gemm_tc(const GroupRef& g, bool pdl, int* status, cudaStream_t s);
bool gemm_tc_supported(const GroupRef& g);
// Bytes of zero-filled workspace the GEMM's stream-K schedule wants for this group on the
// current device (0: the group's plan needs none).
size_t gemm_tc_workspace(const GroupRef& g);

// Layer steps around the linears (csrc/layer_ops.cu): RMSNorm of the fp32 residual into
// bf16, rotary embedding in place, grouped-head attention over a prefix cache and the
// chunk's own keys. Arguments are validated by the caller (api.cu).
cudaError_t launch_rmsnorm(const float* x, const float* gamma, uint16_t* y, int64_t M, int64_t D,
                           float eps, cudaStream_t s);
cudaError_t launch_rope(uint16_t* x, int64_t n_heads, uint16_t* x2, int64_t n_heads2, int64_t M,
                        int64_t head_dim, int64_t pos0, double base, cudaStream_t s);
cudaError_t launch_attention(const uint16_t* Q, const uint16_t* K0, const uint16_t* V0, int64_t n0,
                             const uint16_t* K1, const uint16_t* V1, int64_t n1, uint16_t* O,
                             int64_t M, int64_t H, int64_t Hk, int64_t D, float scale, cudaStream_t s);

// Self-test kernel: waits on an mbarrier nobody arrives at, for timeout_ns.
cudaError_t launch_selftest_wait(uint64_t timeout_ns, int* status, cudaStream_t s);

}  // namespace emb
