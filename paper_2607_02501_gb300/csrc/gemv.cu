// Weight-streaming GEMV for small token counts (action-token decode, M = 1..4).
//
// The paper's batch-1 setting (Section 3.1, challenge 2) makes every linear layer a
// matrix-vector product whose cost is reading the packed weights once from HBM.
// Design for sm_103a:
//   * one CTA owns R consecutive weight rows (contiguous bytes in the codes plane);
//     its NT threads split K in 16-byte units: a Q8_0 unit is 16 codes (half a block),
//     a Q4_0 unit is one whole 32-code block; a warp reads 512 contiguous bytes;
//   * codes are loaded with 128-bit non-allocating loads, one unit ahead (register
//     double buffering), and dequantised in registers with exact integer->float
//     "magic number" conversions followed by packed fp32x2 FMAs (FFMA2);
//   * per-row partial sums are reduced with warp shuffles, then across warps in shared
//     memory; results are deterministic (fixed reduction order);
//   * the first unit's weights are fetched before griddepcontrol.wait, so under
//     programmatic dependent launch a layer's weight stream starts while the previous
//     layer is still finishing; X is read and Y written only after the wait.
// Up to kMaxGroup matrices that read the same X (q/k/v or gate/up) share one launch.
#include <mutex>

#include "ptx.cuh"

namespace emb {
namespace {

struct GemvParams {
    const uint8_t* codes[kMaxGroup];
    const __half* scales[kMaxGroup];
    float* Y[kMaxGroup];
    int32_t N[kMaxGroup];
    int32_t tile0[kMaxGroup + 1];  // first row tile of each matrix (prefix sums)
    int32_t n_mats;
    int32_t M, K, ldS, U;          // U = 16-byte code units per row
    const __nv_bfloat16* X;
};

__device__ __forceinline__ uint4 ld_stream_u4(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ void griddep_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void griddep_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ float lo_bf16(uint32_t h) { return __uint_as_float(h << 16); }
__device__ __forceinline__ float hi_bf16(uint32_t h) { return __uint_as_float(h & 0xFFFF0000u); }
__device__ __forceinline__ float magic(uint32_t bits) { return __uint_as_float(bits | 0x4B000000u); }

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
        const float2 a = __ffma2_rn(make_float2(magic(v & 0xFu), magic(v & 0xF00u)), s_a, o_a);
        // codes 16+4j, 16+4j+1 (bits 4..7, 12..15)
        const float2 b = __ffma2_rn(make_float2(magic(v & 0xF0u), magic(v & 0xF000u)), s_b, o_b);
        // codes 4j+2, 4j+3 (bits 16..19, 24..27 -> 12..15 after the shift)
        const float2 cc = __ffma2_rn(make_float2(magic(v & 0xF0000u), magic(v2 & 0xF000u)), s_c, o_c);
        // codes 16+4j+2, 16+4j+3 (bits 20..23 -> 8..11, 28..31 -> 16..19)
        const float2 d = __ffma2_rn(make_float2(magic(v2 & 0xF00u), magic(v2 & 0xF0000u)), s_d, o_d);
        acc = __ffma2_rn(a, make_float2(x[4 * j + 0], x[4 * j + 1]), acc);
        acc = __ffma2_rn(cc, make_float2(x[4 * j + 2], x[4 * j + 3]), acc);
        acc = __ffma2_rn(b, make_float2(x[16 + 4 * j + 0], x[16 + 4 * j + 1]), acc);
        acc = __ffma2_rn(d, make_float2(x[16 + 4 * j + 2], x[16 + 4 * j + 3]), acc);
    }
    return acc.x + acc.y;
}

template <int FMT, int R, int NT, int MT>
__global__ void __launch_bounds__(NT) gemv_kernel(const __grid_constant__ GemvParams p) {
    constexpr int UW = (FMT == EMB_Q8_0) ? 16 : 32;  // weights per 16-byte unit
    constexpr int NWARP = NT / 32;
    const int tile = blockIdx.x;
    int g = 0;
#pragma unroll
    for (int i = 1; i < kMaxGroup; ++i)
        if (i < p.n_mats && tile >= p.tile0[i]) g = i;
    const int row0 = (tile - p.tile0[g]) * R;
    const int N = p.N[g];
    const int m0 = blockIdx.y * MT;
    const int t = threadIdx.x;
    const int64_t row_bytes = (FMT == EMB_Q8_0) ? int64_t(p.K) : int64_t(p.K) / 2;
    const uint8_t* cbase = p.codes[g] + int64_t(row0) * row_bytes;
    const __half* sbase = p.scales[g] + int64_t(row0) * p.ldS;
    const int U = p.U;

    griddep_launch_dependents();

    uint4 c[R];
    float d[R];
    auto load_unit = [&](int u, uint4* cc, float* dd) {
#pragma unroll
        for (int r = 0; r < R; ++r) {
            if (row0 + r < N) {
                cc[r] = ld_stream_u4(cbase + r * row_bytes + int64_t(u) * 16);
                dd[r] = __half2float(sbase[int64_t(r) * p.ldS + ((FMT == EMB_Q8_0) ? (u >> 1) : u)]);
            } else {
                cc[r] = make_uint4(0, 0, 0, 0);
                dd[r] = 0.0f;
            }
        }
    };

    int u = t;
    if (u < U) load_unit(u, c, d);
    // weights do not depend on earlier launches; X and Y may
    griddep_wait();

    float acc[R][MT];
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
        for (int j = 0; j < MT; ++j) acc[r][j] = 0.0f;

    for (; u < U; u += NT) {
        uint4 cn[R];
        float dn[R];
        const int un = u + NT;
        if (un < U) load_unit(un, cn, dn);
#pragma unroll
        for (int j = 0; j < MT; ++j) {
            const int m = m0 + j;
            if (m >= p.M) break;
            float x[UW];
            const uint4* xp = reinterpret_cast<const uint4*>(p.X + int64_t(m) * p.K + int64_t(u) * UW);
#pragma unroll
            for (int v = 0; v < UW / 8; ++v) {
                const uint4 h = __ldg(xp + v);
                x[8 * v + 0] = lo_bf16(h.x); x[8 * v + 1] = hi_bf16(h.x);
                x[8 * v + 2] = lo_bf16(h.y); x[8 * v + 3] = hi_bf16(h.y);
                x[8 * v + 4] = lo_bf16(h.z); x[8 * v + 5] = hi_bf16(h.z);
                x[8 * v + 6] = lo_bf16(h.w); x[8 * v + 7] = hi_bf16(h.w);
            }
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const float part = (FMT == EMB_Q8_0) ? dot_q8_unit(c[r], x) : dot_q4_unit(c[r], x);
                acc[r][j] = fmaf(d[r], part, acc[r][j]);
            }
        }
        if (un < U) {
#pragma unroll
            for (int r = 0; r < R; ++r) { c[r] = cn[r]; d[r] = dn[r]; }
        }
    }

    __shared__ float red[NWARP][R * MT];
    const int lane = t & 31, warp = t >> 5;
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
        for (int j = 0; j < MT; ++j) {
            float v = acc[r][j];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == 0) red[warp][r * MT + j] = v;
        }
    __syncthreads();
    if (t < R * MT) {
        const int r = t / MT, j = t % MT;
        float v = 0.0f;
#pragma unroll
        for (int w = 0; w < NWARP; ++w) v += red[w][t];
        const int n = row0 + r, m = m0 + j;
        if (n < N && m < p.M) p.Y[g][int64_t(m) * N + n] = v;
    }
}

template <int FMT, int R, int NT, int MT>
cudaError_t launch_one(const GemvParams& p, int grid_x, int grid_y, bool pdl, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid_x, grid_y, 1);
    cfg.blockDim = dim3(NT, 1, 1);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, gemv_kernel<FMT, R, NT, MT>, p);
}

template <int FMT, int R, int NT>
cudaError_t dispatch_mt(const GemvParams& p, int grid_x, int M, bool pdl, cudaStream_t s) {
    if (M == 1) return launch_one<FMT, R, NT, 1>(p, grid_x, 1, pdl, s);
    if (M == 2) return launch_one<FMT, R, NT, 2>(p, grid_x, 1, pdl, s);
    return launch_one<FMT, R, NT, 4>(p, grid_x, (M + 3) / 4, pdl, s);
}

template <int FMT, int R>
cudaError_t dispatch_nt(const GemvParams& p, int grid_x, int M, int NT, bool pdl, cudaStream_t s) {
    if (NT == 256) return dispatch_mt<FMT, R, 256>(p, grid_x, M, pdl, s);
    if (NT == 128) return dispatch_mt<FMT, R, 128>(p, grid_x, M, pdl, s);
    if (NT == 64) return dispatch_mt<FMT, R, 64>(p, grid_x, M, pdl, s);
    return dispatch_mt<FMT, R, 32>(p, grid_x, M, pdl, s);
}

// Threads per CTA (they split K): about 8 (Q8_0) or 4 (Q4_0) 16-byte units per thread
// and row, 32..128 threads, which amortises the per-thread prologue and reduction on large
// matrices (measured on GB300 at M=1, Q8_0 K=2048: 32 threads 5.6 TB/s, 128 threads
// 4.6 TB/s). Small matrices are latency-bound instead: there the count grows (up to one
// unit per thread, 256 threads) until about 152K threads put every byte in flight at once.
int pick_threads(int U, int fmt, int64_t tiles) {
    const int target = (fmt == EMB_Q8_0) ? U / 8 : U / 4;
    int nt = 32;
    while (nt < 128 && nt < target) nt *= 2;
    while (nt < 256 && nt < U && tiles * nt < int64_t(152) * 1024) nt *= 2;
    return nt;
}

}  // namespace

cudaError_t launch_gemv(const GroupRef& g, bool pdl, int* /*status*/, cudaStream_t s) {
    GemvParams p = {};
    const int U = int((g.fmt == EMB_Q8_0) ? g.K / 16 : g.K / 32);
    int64_t rows = 0;
    for (int i = 0; i < g.n_mats; ++i) rows += g.mats[i].N;
    // rows per CTA: 4 (activation reuse across rows) unless that leaves the GPU idle
    const int R = (rows >= 4 * 2 * 152) ? 4 : 1;
    int tiles = 0;
    for (int i = 0; i < g.n_mats; ++i) {
        p.codes[i] = g.mats[i].codes;
        p.scales[i] = g.mats[i].scales;
        p.Y[i] = g.mats[i].Y;
        p.N[i] = int32_t(g.mats[i].N);
        p.tile0[i] = tiles;
        tiles += int((g.mats[i].N + R - 1) / R);
    }
    p.tile0[g.n_mats] = tiles;
    p.n_mats = g.n_mats;
    p.M = int32_t(g.M);
    p.K = int32_t(g.K);
    p.ldS = int32_t(g.ldS);
    p.U = U;
    p.X = g.X;
    const int NT = pick_threads(U, g.fmt, tiles);
    const int M = int(g.M);
    if (g.fmt == EMB_Q8_0)
        return R == 4 ? dispatch_nt<EMB_Q8_0, 4>(p, tiles, M, NT, pdl, s)
                      : dispatch_nt<EMB_Q8_0, 1>(p, tiles, M, NT, pdl, s);
    return R == 4 ? dispatch_nt<EMB_Q4_0, 4>(p, tiles, M, NT, pdl, s)
                  : dispatch_nt<EMB_Q4_0, 1>(p, tiles, M, NT, pdl, s);
}

}  // namespace emb
