// GEMV for small token counts (action-token decode, M = 1..4).
//
// The paper's batch-1 setting (Section 3.1, challenge 2) makes every linear layer a
// matrix-vector product whose cost is reading the packed weights once from HBM.
// Three kernels:
//   * the staged kernel (large layers with short rows, and M > 1): each CTA pulls one
//     tile of rows plus its activations into shared memory with cp.async.bulk, so many
//     bytes are in flight per SM and the next layer's tiles load during this layer's
//     tail (programmatic dependent launch);
//   * the register kernel (small layers, and long rows at M = 1): one CTA owns R
//     consecutive weight rows; its NT threads split K in 16-byte units (a Q8_0 unit is
//     16 codes, half a block; a Q4_0 unit is one whole 32-code block; a warp reads 512
//     contiguous bytes), load codes with 128-bit non-allocating loads one unit ahead
//     (register double buffering) and reduce with warp shuffles, then across warps in
//     shared memory;
//   * the Q4_0 tensor-core kernel (large Q4_0 layers at M = 2..8): staged like the
//     first, with the dot products on mma.sync (described at its definition).
// The first two dequantise in registers with exact integer->float "magic number"
// conversions followed by packed fp32x2 FMAs (FFMA2). Every reduction runs in a fixed
// order, so results are deterministic. Weights are fetched before griddepcontrol.wait (they never depend
// on an earlier launch) with non-coherent streaming loads; X is read with ordinary
// (coherent, L1-cached) loads and Y written only after it: the previous launch may have
// just written X, and after griddepcontrol.wait its writes are visible to ordinary loads.
// Up to kMaxGroup matrices that read the same X (q/k/v or gate/up) share one launch.
#include <algorithm>
#include <mutex>

#include "dequant_dot.cuh"
#include "ptx.cuh"

namespace emb {
namespace {

using dq::and_or;
using dq::dot_q4_unit;
using dq::dot_q6_unit;
using dq::dot_q8_unit;
using dq::hi_bf16;
using dq::lo_bf16;

struct GemvParams {
    const uint8_t* codes[kMaxGroup];
    const uint8_t* high[kMaxGroup];  // Q6_0: 2-bit high plane of each matrix
    const __half* scales[kMaxGroup];
    void* Y[kMaxGroup];              // as the epilogue says
    int32_t N[kMaxGroup];
    int32_t tile0[kMaxGroup + 1];  // first row tile of each matrix (prefix sums)
    int32_t n_mats;
    int32_t M, K, ldS, U;          // U = 16-byte code units per row
    int32_t epi;                   // emb_epilogue (gated: R even, gate/up row pairs)
    const __nv_bfloat16* X;
};

__device__ __forceinline__ uint4 ld_stream_u4(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}
__device__ __forceinline__ uint2 ld_stream_u2(const void* p) {
    uint2 v;
    asm volatile("ld.global.nc.L1::no_allocate.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "l"(p));
    return v;
}

__device__ __forceinline__ void griddep_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void griddep_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// One 16-byte unit of codes (Q6_0: plus its 8 bytes of high bits) times its activations.
template <int FMT>
__device__ __forceinline__ float dot_unit(const uint4 c, const uint2 h, const float* x) {
    if constexpr (FMT == EMB_Q8_0) return dot_q8_unit(c, x);
    else if constexpr (FMT == EMB_Q4_0) return dot_q4_unit(c, x);
    else return dot_q6_unit(c, h, x);
}

// PF > 1 (M = 1 only, U <= PF * NT): every unit of the thread is loaded into registers
// before griddepcontrol.wait, so a layer with long rows has all of its weight bytes in
// flight while the previous launch drains; the products are summed in the same order as
// with PF = 1 (bitwise the same results).
template <int FMT, int R, int NT, int MT, int PF>
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
    const uint8_t* hbase = (FMT == EMB_Q6_0) ? p.high[g] + int64_t(row0) * (p.K / 4) : nullptr;
    const __half* sbase = p.scales[g] + int64_t(row0) * p.ldS;
    const int U = p.U;

    griddep_launch_dependents();
    // the activation rows towards L2 while the previous launch finishes (measured on GB300:
    // cold, they arrive ~2 us after the dependency wait, behind the weight stream); one CTA
    // per row block asks, since every CTA reads the same rows
    if (t == 0 && blockIdx.x == 0)
        ptx::prefetch_l2(p.X + int64_t(m0) * p.K, uint32_t(min(MT, p.M - m0)) * uint32_t(p.K) * 2u);

    uint4 c[R];
    uint2 h[R];  // Q6_0 high bits (unused otherwise)
    float d[R];
    auto load_unit = [&](int u, uint4* cc, uint2* hh, float* dd) {
#pragma unroll
        for (int r = 0; r < R; ++r) {
            if (row0 + r < N) {
                cc[r] = ld_stream_u4(cbase + r * row_bytes + int64_t(u) * 16);
                if constexpr (FMT == EMB_Q6_0) hh[r] = ld_stream_u2(hbase + int64_t(r) * (p.K / 4) + int64_t(u) * 8);
                else hh[r] = make_uint2(0, 0);
                dd[r] = __half2float(sbase[int64_t(r) * p.ldS + ((FMT == EMB_Q8_0) ? (u >> 1) : u)]);
            } else {
                cc[r] = make_uint4(0, 0, 0, 0);
                hh[r] = make_uint2(0, 0);
                dd[r] = 0.0f;
            }
        }
    };

    float acc[R][MT];
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
        for (int j = 0; j < MT; ++j) acc[r][j] = 0.0f;

    if constexpr (PF > 1) {
        static_assert(MT == 1, "whole-row prefetch is for one token");
        uint4 cp[PF][R];
        uint2 hp[PF][R];
        float dp[PF][R];
#pragma unroll
        for (int k = 0; k < PF; ++k)
            if (t + k * NT < U) load_unit(t + k * NT, cp[k], hp[k], dp[k]);
        // weights do not depend on earlier launches; X and Y may
        griddep_wait();
#pragma unroll
        for (int k = 0; k < PF; ++k) {
            const int uk = t + k * NT;
            if (uk >= U) break;
            float x[UW];
            const uint4* xp = reinterpret_cast<const uint4*>(p.X + int64_t(m0) * p.K + int64_t(uk) * UW);
#pragma unroll
            for (int v = 0; v < UW / 8; ++v) {
                const uint4 hx = xp[v];
                x[8 * v + 0] = lo_bf16(hx.x); x[8 * v + 1] = hi_bf16(hx.x);
                x[8 * v + 2] = lo_bf16(hx.y); x[8 * v + 3] = hi_bf16(hx.y);
                x[8 * v + 4] = lo_bf16(hx.z); x[8 * v + 5] = hi_bf16(hx.z);
                x[8 * v + 6] = lo_bf16(hx.w); x[8 * v + 7] = hi_bf16(hx.w);
            }
#pragma unroll
            for (int r = 0; r < R; ++r) acc[r][0] = fmaf(dp[k][r], dot_unit<FMT>(cp[k][r], hp[k][r], x), acc[r][0]);
        }
    }

    int u = (PF > 1) ? U : t;
    if (u < U) load_unit(u, c, h, d);
    // weights do not depend on earlier launches; X and Y may
    if constexpr (PF == 1) griddep_wait();

    for (; u < U; u += NT) {
        uint4 cn[R];
        uint2 hn[R];
        float dn[R];
        const int un = u + NT;
        if (un < U) load_unit(un, cn, hn, dn);
#pragma unroll
        for (int j = 0; j < MT; ++j) {
            const int m = m0 + j;
            if (m >= p.M) break;
            float x[UW];
            const uint4* xp = reinterpret_cast<const uint4*>(p.X + int64_t(m) * p.K + int64_t(u) * UW);
#pragma unroll
            for (int v = 0; v < UW / 8; ++v) {
                const uint4 h = xp[v];
                x[8 * v + 0] = lo_bf16(h.x); x[8 * v + 1] = hi_bf16(h.x);
                x[8 * v + 2] = lo_bf16(h.y); x[8 * v + 3] = hi_bf16(h.y);
                x[8 * v + 4] = lo_bf16(h.z); x[8 * v + 5] = hi_bf16(h.z);
                x[8 * v + 6] = lo_bf16(h.w); x[8 * v + 7] = hi_bf16(h.w);
            }
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const float part = dot_unit<FMT>(c[r], h[r], x);
                acc[r][j] = fmaf(d[r], part, acc[r][j]);
            }
        }
        if (un < U) {
#pragma unroll
            for (int r = 0; r < R; ++r) { c[r] = cn[r]; h[r] = hn[r]; d[r] = dn[r]; }
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
    if (p.epi >= EMB_EPI_GEGLU) {
        // gate row row0 + 2i and up row row0 + 2i + 1 (R is even) give one output
        if (t < (R / 2) * MT) {
            const int i = t / MT, j = t % MT;
            float gate = 0.0f, up = 0.0f;
#pragma unroll
            for (int w = 0; w < NWARP; ++w) {
                gate += red[w][(2 * i) * MT + j];
                up += red[w][(2 * i + 1) * MT + j];
            }
            const int n = row0 + 2 * i, m = m0 + j;
            if (n < N && m < p.M) epi_store_gated(p.epi, p.Y[g], m, n, N, gate, up);
        }
    } else if (t < R * MT) {
        const int r = t / MT, j = t % MT;
        float v = 0.0f;
#pragma unroll
        for (int w = 0; w < NWARP; ++w) v += red[w][t];
        const int n = row0 + r, m = m0 + j;
        if (n < N && m < p.M) epi_store(p.epi, p.Y[g], m, n, N, v);
    }
}

template <int FMT, int R, int NT, int MT, int PF = 1>
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
    return cudaLaunchKernelEx(&cfg, gemv_kernel<FMT, R, NT, MT, PF>, p);
}

template <int FMT, int R, int NT>
cudaError_t dispatch_mt(const GemvParams& p, int grid_x, int M, bool pdl, cudaStream_t s) {
    // Q8_0 rows longer than one pass of the CTA's threads (at most four) are loaded whole
    // before the wait (measured on GB300 on the Gemma-2B decode chain at M = 1, whose down
    // projection 2048 x 16384 took this path before the ring kernel: Q8_0 3899 -> 3987
    // GB/s). Not for Q4_0: its variant needs ~100 registers, halves the resident CTAs and
    // lost (2265 -> 2068).
    if constexpr (FMT == EMB_Q8_0 && R <= 2) {
        if (M == 1 && p.U > NT && p.U <= 4 * NT) return launch_one<FMT, R, NT, 1, 4>(p, grid_x, 1, pdl, s);
    }
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


// ------------------------------------------------------------------ staged GEMV
// One CTA owns a tile of TR consecutive rows of one matrix. Its codes (TR rows,
// contiguous in the codes plane) and scales (TR rows of the scales plane, contiguous
// too) arrive in shared memory through two cp.async.bulk copies that a single thread
// issues as soon as the CTA starts -- before griddepcontrol.wait, since weights never
// depend on an earlier launch -- and the CTA's activation rows (MT x K bf16, contiguous
// in X) through a third copy right after the wait. Up to kStageBytes of codes per CTA
// and several CTAs per SM keep far more bytes in flight than register double buffering
// can, and under programmatic dependent launch the next layer's tiles stream in while
// this layer's last CTAs finish. The four warps form a WR x WK grid (WR = 4 / WK): a
// warp owns RW rows of the tile and one K slice of U / WK units; its lanes stride the
// slice in 16-byte units and reuse each activation unit across the warp's RW rows.
constexpr int kStageWarps = 4;
constexpr int kStageThreads = 32 * kStageWarps;
constexpr int kStageBytes = 32 * 1024;     // codes of one tile, at most
constexpr int kStageXBytes = 32 * 1024;    // activation rows of one CTA, at most
constexpr int kStageHeader = 1152;         // mbarriers (0..15), cross-warp sums (128..1151)

struct StagedParams {
    const uint8_t* codes[kMaxGroup];
    const uint8_t* high[kMaxGroup];  // Q6_0: 2-bit high plane of each matrix
    const __half* scales[kMaxGroup];
    void* Y[kMaxGroup];              // as the epilogue says
    int32_t N[kMaxGroup];
    int32_t tile0[kMaxGroup + 1];  // first tile of each matrix (prefix sums)
    int32_t n_mats;
    int32_t M, K, ldS, U;
    int32_t TR, WK;                // rows per tile, warps along K
    int32_t epi;                   // emb_epilogue (gated: RW and TR even)
    const __nv_bfloat16* X;
    int* status;
};

template <int FMT, int RW, int MT>
__global__ void __launch_bounds__(kStageThreads) gemv_staged_kernel(const __grid_constant__ StagedParams p) {
    constexpr int UW = (FMT == EMB_Q8_0) ? 16 : 32;
    extern __shared__ __align__(128) uint8_t smem[];
    uint64_t* bar_w = reinterpret_cast<uint64_t*>(smem);      // weights landed
    uint64_t* bar_x = reinterpret_cast<uint64_t*>(smem + 8);  // activations landed
    float* red = reinterpret_cast<float*>(smem + 128);         // [WK][TR][MT]
    const int row_bytes = (FMT == EMB_Q8_0) ? p.K : p.K / 2;
    const int high_bytes = (FMT == EMB_Q6_0) ? p.K / 4 : 0;               // Q6_0 high bits per row
    uint8_t* x_s = smem + kStageHeader;                                    // [MT][K] bf16
    uint8_t* codes_s = x_s + MT * p.K * 2;                                 // [TR][row_bytes]
    uint8_t* high_s = codes_s + uint32_t(p.TR) * uint32_t(row_bytes);     // [TR][K/4] (Q6_0)
    uint8_t* scales_b = high_s + uint32_t(p.TR) * uint32_t(high_bytes);   // [TR][ldS] fp16
    const __half* scales_s = reinterpret_cast<const __half*>(scales_b);

    const int tile = blockIdx.x;
    int g = 0;
#pragma unroll
    for (int i = 1; i < kMaxGroup; ++i)
        if (i < p.n_mats && tile >= p.tile0[i]) g = i;
    const int N = p.N[g];
    const int row0 = (tile - p.tile0[g]) * p.TR;
    const int rows = min(p.TR, N - row0);
    const int m0 = blockIdx.y * MT;
    const int mt = min(MT, p.M - m0);  // activation rows of this CTA

    if (threadIdx.x == 0) {
        const uint32_t codes_bytes = uint32_t(rows) * uint32_t(row_bytes);
        const uint32_t hi_bytes = uint32_t(rows) * uint32_t(high_bytes);  // a multiple of 16 (K % 64 == 0)
        const uint32_t scales_bytes = uint32_t(rows) * uint32_t(p.ldS) * 2u;
        ptx::mbar_init(bar_w, 1);
        ptx::mbar_init(bar_x, 1);
        ptx::fence_mbar_init();
        ptx::mbar_arrive_expect_tx(bar_w, codes_bytes + hi_bytes + scales_bytes);
        ptx::bulk_load(codes_s, p.codes[g] + int64_t(row0) * row_bytes, codes_bytes, bar_w);
        if constexpr (FMT == EMB_Q6_0)
            ptx::bulk_load(high_s, p.high[g] + int64_t(row0) * high_bytes, hi_bytes, bar_w);
        ptx::bulk_load(scales_b, p.scales[g] + int64_t(row0) * p.ldS, scales_bytes, bar_w);
        // the activation rows towards L2 while the previous launch finishes (measured on
        // GB300: cold, they land ~2 us after the dependency wait, behind the weight stream);
        // one CTA per row block asks, since every CTA reads the same rows
        if (blockIdx.x == 0) ptx::prefetch_l2(p.X + int64_t(m0) * p.K, uint32_t(mt) * uint32_t(p.K) * 2u);
    }
    ptx::griddep_launch_dependents();
    // weights do not depend on earlier launches; X and Y may
    ptx::griddep_wait();
    if (threadIdx.x == 0) {
        const uint32_t x_bytes = uint32_t(mt) * uint32_t(p.K) * 2u;
        ptx::mbar_arrive_expect_tx(bar_x, x_bytes);
        ptx::bulk_load(x_s, p.X + int64_t(m0) * p.K, x_bytes, bar_x);
    }
    __syncthreads();  // the barriers' initialisation is visible to every waiting thread
    // both waits are bounded; the CTA leaves together if any of its threads gave up
    bool ok = ptx::mbar_wait(bar_w, 0, nullptr, p.status, kWaitLimitNs);
    ok = ok && ptx::mbar_wait(bar_x, 0, nullptr, p.status, kWaitLimitNs);
    if (__syncthreads_or(!ok)) return;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int WK = p.WK;
    const int wk = warp % WK, wr = warp / WK;
    const int r0 = wr * RW;                       // first tile row of this warp
    const int Uw = (p.U + WK - 1) / WK;
    const int u_lo = wk * Uw, u_hi = min(p.U, u_lo + Uw);

    float acc[RW][MT];
#pragma unroll
    for (int i = 0; i < RW; ++i)
#pragma unroll
        for (int t = 0; t < MT; ++t) acc[i][t] = 0.0f;

    if (r0 < rows) {
#pragma unroll 2
        for (int u = u_lo + lane; u < u_hi; u += 32) {
            uint4 c[RW];
            uint2 hq[RW];
            float d[RW];
#pragma unroll
            for (int i = 0; i < RW; ++i) {
                const int r = min(r0 + i, rows - 1);  // rows past the tile's end are never stored
                c[i] = *reinterpret_cast<const uint4*>(codes_s + r * row_bytes + u * 16);
                if constexpr (FMT == EMB_Q6_0)
                    hq[i] = *reinterpret_cast<const uint2*>(high_s + r * high_bytes + u * 8);
                else
                    hq[i] = make_uint2(0, 0);
                d[i] = __half2float(scales_s[r * p.ldS + ((FMT == EMB_Q8_0) ? (u >> 1) : u)]);
            }
#pragma unroll
            for (int t = 0; t < MT; ++t) {
                if (t >= mt) break;
                float x[UW];
                const uint4* xp = reinterpret_cast<const uint4*>(x_s + (t * p.K + u * UW) * 2);
#pragma unroll
                for (int v = 0; v < UW / 8; ++v) {
                    const uint4 h = xp[v];
                    x[8 * v + 0] = lo_bf16(h.x); x[8 * v + 1] = hi_bf16(h.x);
                    x[8 * v + 2] = lo_bf16(h.y); x[8 * v + 3] = hi_bf16(h.y);
                    x[8 * v + 4] = lo_bf16(h.z); x[8 * v + 5] = hi_bf16(h.z);
                    x[8 * v + 6] = lo_bf16(h.w); x[8 * v + 7] = hi_bf16(h.w);
                }
#pragma unroll
                for (int i = 0; i < RW; ++i) {
                    const float sdot = dot_unit<FMT>(c[i], hq[i], x);
                    acc[i][t] = fmaf(d[i], sdot, acc[i][t]);
                }
            }
        }
    }

    float mine = 0.0f;
#pragma unroll
    for (int i = 0; i < RW; ++i)
#pragma unroll
        for (int t = 0; t < MT; ++t) {
            float v = acc[i][t];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == i * MT + t) mine = v;
        }
    const bool gated = p.epi >= EMB_EPI_GEGLU;
    if (WK == 1) {
        // gated: the up row's sum sits MT lanes further on (RW is even)
        const float up = __shfl_down_sync(0xffffffffu, mine, MT);
        if (lane < RW * MT) {
            const int r = r0 + lane / MT, t = lane % MT;
            if (r < rows && t < mt) {
                if (!gated) epi_store(p.epi, p.Y[g], m0 + t, row0 + r, N, mine);
                else if ((r & 1) == 0) epi_store_gated(p.epi, p.Y[g], m0 + t, row0 + r, N, mine, up);
            }
        }
        return;
    }
    if (lane < RW * MT) red[(wk * p.TR + r0 + lane / MT) * MT + lane % MT] = mine;
    __syncthreads();
    // add the K slices in slice order
    if (gated) {
        for (int e = threadIdx.x; e < (rows / 2) * MT; e += kStageThreads) {
            const int i = e / MT, t = e % MT;
            float gate = 0.0f, up = 0.0f;
            for (int k = 0; k < WK; ++k) {
                gate += red[(k * p.TR + 2 * i) * MT + t];
                up += red[(k * p.TR + 2 * i + 1) * MT + t];
            }
            if (t < mt) epi_store_gated(p.epi, p.Y[g], m0 + t, row0 + 2 * i, N, gate, up);
        }
        return;
    }
    for (int e = threadIdx.x; e < rows * MT; e += kStageThreads) {
        float v = 0.0f;
        for (int k = 0; k < WK; ++k) v += red[k * p.TR * MT + e];
        const int r = e / MT, t = e % MT;
        if (t < mt) epi_store(p.epi, p.Y[g], m0 + t, row0 + r, N, v);
    }
}

template <int FMT, int RW, int MT>
cudaError_t launch_staged_one(const StagedParams& p, int tiles, size_t smem, bool pdl, cudaStream_t s) {
    static_assert(kStageHeader + kStageXBytes + kStageBytes + kStageBytes / 8 <= 227 * 1024, "smem");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(tiles, (p.M + MT - 1) / MT, 1);
    cfg.blockDim = dim3(kStageThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    if (smem > 48 * 1024) {
        // once per instantiation and device is enough, but the call is cheap and idempotent
        const cudaError_t e = cudaFuncSetAttribute(gemv_staged_kernel<FMT, RW, MT>,
                                                   cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   int(kStageHeader + kStageXBytes + kStageBytes + kStageBytes / 8));
        if (e != cudaSuccess) return e;
    }
    return cudaLaunchKernelEx(&cfg, gemv_staged_kernel<FMT, RW, MT>, p);
}

template <int FMT, int MT>
cudaError_t launch_staged_rw(const StagedParams& p, int RW, int tiles, size_t smem, bool pdl, cudaStream_t s) {
    if (RW == 4) return launch_staged_one<FMT, 4, MT>(p, tiles, smem, pdl, s);
    if (RW == 2) return launch_staged_one<FMT, 2, MT>(p, tiles, smem, pdl, s);
    return launch_staged_one<FMT, 1, MT>(p, tiles, smem, pdl, s);
}

// Tile shape: rows per warp RW and warps along K WK (TR = RW * 4 / WK rows per tile),
// in order of preference: Q8_0 favours activation reuse (4 rows per warp), Q4_0 unsplit
// K. Take the first whose tile fits `tile_bytes` and that makes at least 4 tiles per
// SM; for matrices too small for that, the fitting shape with the most tiles. A warp's
// K slice keeps at least 32 units (one per lane). Returns false when no tile fits.
// Measured on GB300 at M = 1 (graph-replayed chains): 16 KB tiles beat 32 KB ones by
// 3-6% (a shorter CTA lifetime shortens each launch's tail), e.g. Q8_0 32768 x 2048:
// 14.9 us (8 rows) vs 15.8 us (16 rows); at M = 4, 32 KB tiles win (22.7 vs 27.0 us).
bool pick_stage_shape(int fmt, int64_t rows_total, int64_t row_bytes, int U, int64_t tile_bytes,
                      bool even_rows, int& RW, int& WK) {
    static const int kQ8[5][2] = {{4, 1}, {4, 2}, {4, 4}, {2, 4}, {1, 4}};
    static const int kQ4[7][2] = {{4, 1}, {2, 1}, {1, 1}, {4, 2}, {4, 4}, {2, 4}, {1, 4}};
    const int n = (fmt == EMB_Q8_0) ? 5 : 7;
    bool found = false;
    for (int i = 0; i < n; ++i) {
        const int rw = (fmt == EMB_Q8_0) ? kQ8[i][0] : kQ4[i][0];
        const int wk = (fmt == EMB_Q8_0) ? kQ8[i][1] : kQ4[i][1];
        const int64_t tr = int64_t(rw) * kStageWarps / wk;
        if (tr * row_bytes > tile_bytes) continue;
        if (wk > 1 && U / wk < 32) continue;
        if (even_rows && (rw & 1)) continue;  // gated epilogues pair rows inside a warp
        RW = rw;
        WK = wk;
        found = true;
        if (rows_total / tr >= 4 * 152) break;
    }
    return found;
}

// Which layers take the staged path (measured on GB300, graph-replayed chains of one
// shape). Small layers are latency-bound: there the register kernel, whose threads issue
// their loads directly, finishes sooner than a bulk-copy round trip (5.6 MB q/k/v at
// M = 1: 2.1 us register, 3.2 us staged). Long rows at M = 1 leave a staged CTA one or two
// rows and re-stage the whole activation row per CTA; the register kernel with 2 rows
// per CTA is faster there (Q8_0 2048 x 16384: 9.6 us register, 12.0 us staged). Short
// rows favour the staged path (Q4_0 32768 x 2048: 13.4 us staged, 15.1 us register), and
// so does M > 1 (Q8_0 32768 x 2048 at M = 4: 22.6 us staged, 32.2 us register).
constexpr int64_t kStageMinBytes = 12ll << 20;
constexpr int64_t kStageMaxRowBytesM1 = 6 * 1024;

bool launch_staged(const GroupRef& g, bool pdl, int* status, cudaStream_t s, cudaError_t& err) {
    const int64_t row_bytes = (g.fmt == EMB_Q8_0) ? g.K : g.K / 2;
    // Q6_0 rows also carry K/4 bytes of high bits, copied as a second contiguous block
    // (16-byte multiples need K % 64 == 0; other K take the register path)
    const int64_t high_bytes = (g.fmt == EMB_Q6_0) ? g.K / 4 : 0;
    if (g.fmt == EMB_Q6_0 && g.K % 64 != 0) return false;
    const int64_t weight_row_bytes = row_bytes + high_bytes;
    const int U = int((g.fmt == EMB_Q8_0) ? g.K / 16 : g.K / 32);
    const int MT = (g.M == 1) ? 1 : (g.M == 2) ? 2 : 4;
    if (int64_t(MT) * g.K * 2 > kStageXBytes) return false;
    int64_t rows = 0;
    for (int i = 0; i < g.n_mats; ++i) rows += g.mats[i].N;
    if (rows * weight_row_bytes < kStageMinBytes) return false;
    if (g.M == 1 && weight_row_bytes > kStageMaxRowBytesM1) return false;
    int RW = 0, WK = 0;
    const int64_t tile_bytes = (g.M == 1) ? kStageBytes / 2 : kStageBytes;
    if (!pick_stage_shape(g.fmt, rows, weight_row_bytes, U, tile_bytes, g.epi >= EMB_EPI_GEGLU, RW, WK))
        return false;
    StagedParams p = {};
    const int TR = RW * kStageWarps / WK;
    int tiles = 0;
    for (int i = 0; i < g.n_mats; ++i) {
        p.high[i] = g.mats[i].high;
        p.codes[i] = g.mats[i].codes;
        p.scales[i] = g.mats[i].scales;
        p.Y[i] = g.mats[i].Y;
        p.N[i] = int32_t(g.mats[i].N);
        p.tile0[i] = tiles;
        tiles += int((g.mats[i].N + TR - 1) / TR);
    }
    p.tile0[g.n_mats] = tiles;
    p.n_mats = g.n_mats;
    p.M = int32_t(g.M);
    p.K = int32_t(g.K);
    p.ldS = int32_t(g.ldS);
    p.U = U;
    p.TR = TR;
    p.WK = WK;
    p.epi = g.epi;
    p.X = g.X;
    p.status = status;
    const size_t smem = kStageHeader + size_t(MT) * g.K * 2 + size_t(TR) * size_t(weight_row_bytes + g.ldS * 2);
    if (g.fmt == EMB_Q8_0) {
        if (MT == 1) err = launch_staged_rw<EMB_Q8_0, 1>(p, RW, tiles, smem, pdl, s);
        else if (MT == 2) err = launch_staged_rw<EMB_Q8_0, 2>(p, RW, tiles, smem, pdl, s);
        else err = launch_staged_rw<EMB_Q8_0, 4>(p, RW, tiles, smem, pdl, s);
    } else if (g.fmt == EMB_Q6_0) {
        if (MT == 1) err = launch_staged_rw<EMB_Q6_0, 1>(p, RW, tiles, smem, pdl, s);
        else if (MT == 2) err = launch_staged_rw<EMB_Q6_0, 2>(p, RW, tiles, smem, pdl, s);
        else err = launch_staged_rw<EMB_Q6_0, 4>(p, RW, tiles, smem, pdl, s);
    } else {
        if (MT == 1) err = launch_staged_rw<EMB_Q4_0, 1>(p, RW, tiles, smem, pdl, s);
        else if (MT == 2) err = launch_staged_rw<EMB_Q4_0, 2>(p, RW, tiles, smem, pdl, s);
        else err = launch_staged_rw<EMB_Q4_0, 4>(p, RW, tiles, smem, pdl, s);
    }
    return true;
}


// ------------------------------------------------------------ Q4_0 tensor-core GEMV
// For Q4_0 the dequantise-and-dot arithmetic, not HBM, bounds the kernels above. Here
// the dot products run on the tensor cores (mma.sync m16n8k16, bf16 x bf16 -> fp32) and
// the CUDA cores only unpack nibbles: a nibble OR-ed into the bf16 pattern 0x4300 is
// 128 + q exactly, and one packed bf16 subtraction of 136 leaves q - 8 exactly, so each
// pair of weights costs one LOP3 and one HSUB2. One MMA covers 16 rows x 16 consecutive
// K of one block (the tokens, M <= 8, are the MMA's 8 columns); a block's two MMAs
// accumulate into a fresh fragment that is then scaled by the block's fp32 scale, as in
// the plain definition. The MMA sums its 16 products in its own fixed order, so results
// are deterministic.
//
// Fragment mapping (any permutation of K inside a block is valid as long as A and B use
// the same one): lane (g, t) = (lane / 4, lane % 4) loads 32-bit word t of the block in
// rows g and g + 8. Word t holds q[4t + i] in the low nibble and q[16 + 4t + i] in the
// high nibble of its byte i. MMA 0 takes the low nibbles: (bytes 0, 2) -> k slots
// (2t, 2t + 1), (bytes 1, 3) -> (2t + 8, 2t + 9); MMA 1 the high nibbles likewise. The
// activation fragment of lane (g, t) is token g's x at the same four positions.
//
// The CTA's tile (TR rows, TR a multiple of 16) and its activations are staged in shared
// memory as in the staged kernel, but row by row into a padded layout (pitch = row
// bytes + 16) so that the eight rows a fragment load touches fall into distinct banks.
constexpr int kMmaWarps = 4;
constexpr int kMmaThreads = 32 * kMmaWarps;
constexpr int kMmaTileBytes = 32 * 1024;  // codes of one tile, at most
constexpr int kMmaMaxM = 8;
constexpr int kMmaHeader = 128 + 512 * 4;  // barriers, then cross-warp sums [WK][TR][8] (WK * TR <= 64)

struct MmaParams {
    const uint8_t* codes[kMaxGroup];
    const __half* scales[kMaxGroup];
    void* Y[kMaxGroup];              // as the epilogue says
    int32_t N[kMaxGroup];
    int32_t tile0[kMaxGroup + 1];
    int32_t n_mats;
    int32_t M, K, ldS;
    int32_t TR, WK;                // rows per tile (multiple of 16), warps along K
    int32_t pitch, spitch;         // padded shared-memory row pitch of codes / scales, bytes
    int32_t epi;                   // emb_epilogue (element-wise kinds only)
    const __nv_bfloat16* X;
    int* status;
};

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
        "{%8, %9}, {%10, %11, %12, %13};"
        : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(0.0f), "f"(0.0f), "f"(0.0f),
          "f"(0.0f));
}

// (128 + q) pairs from the nibbles at bits 0..3 and 16..19, then q - 8 (exact in bf16).
__device__ __forceinline__ uint32_t q4_pair(uint32_t v) {
    const uint32_t b = and_or(v, 0x000F000Fu, 0x43004300u);
    const __nv_bfloat162 r = __hsub2(*reinterpret_cast<const __nv_bfloat162*>(&b),
                                     __floats2bfloat162_rn(136.0f, 136.0f));
    return *reinterpret_cast<const uint32_t*>(&r);
}

__global__ void __launch_bounds__(kMmaThreads) gemv_q4_mma_kernel(const __grid_constant__ MmaParams p) {
    extern __shared__ __align__(128) uint8_t smem[];
    uint64_t* bar_w = reinterpret_cast<uint64_t*>(smem);
    uint64_t* bar_x = reinterpret_cast<uint64_t*>(smem + 8);
    float* red = reinterpret_cast<float*>(smem + 128);  // [WK][TR][8]
    const int row_bytes = p.K / 2;
    const int nb = p.K / kQBlock;
    uint8_t* x_s = smem + kMmaHeader;                  // [M][K] bf16
    uint8_t* codes_s = x_s + p.M * p.K * 2;            // [TR][pitch]
    uint8_t* scales_s = codes_s + p.TR * p.pitch;

    const int tile = blockIdx.x;
    int g_mat = 0;
#pragma unroll
    for (int i = 1; i < kMaxGroup; ++i)
        if (i < p.n_mats && tile >= p.tile0[i]) g_mat = i;
    const int N = p.N[g_mat];
    const int row0 = (tile - p.tile0[g_mat]) * p.TR;
    const int rows = min(p.TR, N - row0);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (warp == 0) {
        if (lane == 0) {
            ptx::mbar_init(bar_w, 1);
            ptx::mbar_init(bar_x, 1);
            ptx::fence_mbar_init();
            ptx::mbar_arrive_expect_tx(bar_w, uint32_t(rows) * uint32_t(row_bytes + p.ldS * 2));
        }
        __syncwarp();
        const uint8_t* src_c = p.codes[g_mat] + int64_t(row0) * row_bytes;
        const __half* src_s = p.scales[g_mat] + int64_t(row0) * p.ldS;
        for (int r = lane; r < rows; r += 32) {
            ptx::bulk_load(codes_s + r * p.pitch, src_c + int64_t(r) * row_bytes, uint32_t(row_bytes), bar_w);
            ptx::bulk_load(scales_s + r * p.spitch, src_s + int64_t(r) * p.ldS, uint32_t(p.ldS * 2), bar_w);
        }
        if (lane == 0 && blockIdx.x == 0) ptx::prefetch_l2(p.X, uint32_t(p.M) * uint32_t(p.K) * 2u);  // towards L2
    }
    ptx::griddep_launch_dependents();
    // weights do not depend on earlier launches; X and Y may
    ptx::griddep_wait();
    if (threadIdx.x == 0) {
        const uint32_t x_bytes = uint32_t(p.M) * uint32_t(p.K) * 2u;
        ptx::mbar_arrive_expect_tx(bar_x, x_bytes);
        ptx::bulk_load(x_s, p.X, x_bytes, bar_x);
    }
    __syncthreads();  // the barriers' initialisation is visible to every waiting thread
    // both waits are bounded; the CTA leaves together if any of its threads gave up
    bool ok = ptx::mbar_wait(bar_w, 0, nullptr, p.status, kWaitLimitNs);
    ok = ok && ptx::mbar_wait(bar_x, 0, nullptr, p.status, kWaitLimitNs);
    if (__syncthreads_or(!ok)) return;

    const int WK = p.WK;
    const int wk = warp % WK, rg = warp / WK;  // K slice, 16-row group
    const int gq = lane >> 2, t = lane & 3;
    const int bw = (nb + WK - 1) / WK;
    const int kb_lo = wk * bw, kb_hi = min(nb, kb_lo + bw);
    const uint8_t* c0 = codes_s + (rg * 16 + gq) * p.pitch + 4 * t;
    const uint8_t* c1 = c0 + 8 * p.pitch;
    const __half* s0 = reinterpret_cast<const __half*>(scales_s + (rg * 16 + gq) * p.spitch);
    const __half* s1 = reinterpret_cast<const __half*>(reinterpret_cast<const uint8_t*>(s0) + 8 * p.spitch);
    const bool has_x = gq < p.M;
    const uint8_t* xr = x_s + (gq * p.K + 4 * t) * 2;

    float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    if (rg * 16 < rows) {
#pragma unroll 4
        for (int kb = kb_lo; kb < kb_hi; ++kb) {
            uint32_t b[4] = {0u, 0u, 0u, 0u};
            if (has_x) {
                const uint2 lo = *reinterpret_cast<const uint2*>(xr + kb * 64);       // x[4t .. 4t+3]
                const uint2 hi = *reinterpret_cast<const uint2*>(xr + kb * 64 + 32);  // x[16+4t ..]
                b[0] = __byte_perm(lo.x, lo.y, 0x5410);
                b[1] = __byte_perm(lo.x, lo.y, 0x7632);
                b[2] = __byte_perm(hi.x, hi.y, 0x5410);
                b[3] = __byte_perm(hi.x, hi.y, 0x7632);
            }
            const uint32_t w0 = *reinterpret_cast<const uint32_t*>(c0 + kb * 16);
            const uint32_t w1 = *reinterpret_cast<const uint32_t*>(c1 + kb * 16);
            const uint32_t alo[4] = {q4_pair(w0), q4_pair(w1), q4_pair(w0 >> 8), q4_pair(w1 >> 8)};
            const uint32_t ahi[4] = {q4_pair(w0 >> 4), q4_pair(w1 >> 4), q4_pair(w0 >> 12), q4_pair(w1 >> 12)};
            float dlo[4], dhi[4];
            mma_bf16_16816(dlo, alo, b[0], b[1]);
            mma_bf16_16816(dhi, ahi, b[2], b[3]);
            const float sc0 = __half2float(s0[kb]), sc1 = __half2float(s1[kb]);
            acc[0] = fmaf(sc0, dlo[0] + dhi[0], acc[0]);
            acc[1] = fmaf(sc0, dlo[1] + dhi[1], acc[1]);
            acc[2] = fmaf(sc1, dlo[2] + dhi[2], acc[2]);
            acc[3] = fmaf(sc1, dlo[3] + dhi[3], acc[3]);
        }
    }
    // acc[0], acc[1]: row gq, tokens 2t, 2t+1; acc[2], acc[3]: row gq + 8, same tokens
    const int ra = rg * 16 + gq, rb = ra + 8, m0 = 2 * t;
    void* Yg = p.Y[g_mat];
    if (WK == 1) {
        if (m0 < p.M) {
            if (ra < rows) epi_store(p.epi, Yg, m0, row0 + ra, N, acc[0]);
            if (rb < rows) epi_store(p.epi, Yg, m0, row0 + rb, N, acc[2]);
        }
        if (m0 + 1 < p.M) {
            if (ra < rows) epi_store(p.epi, Yg, m0 + 1, row0 + ra, N, acc[1]);
            if (rb < rows) epi_store(p.epi, Yg, m0 + 1, row0 + rb, N, acc[3]);
        }
        return;
    }
    float* rw = red + wk * p.TR * 8;
    rw[ra * 8 + m0] = acc[0];
    rw[ra * 8 + m0 + 1] = acc[1];
    rw[rb * 8 + m0] = acc[2];
    rw[rb * 8 + m0 + 1] = acc[3];
    __syncthreads();
    // add the K slices in slice order
    for (int e = threadIdx.x; e < rows * p.M; e += kMmaThreads) {
        const int r = e / p.M, m = e % p.M;
        float v = 0.0f;
        for (int k = 0; k < WK; ++k) v += red[(k * p.TR + r) * 8 + m];
        epi_store(p.epi, Yg, m, row0 + r, N, v);
    }
}

// Q4_0 layers with 2..8 tokens, large enough for the staged path and with rows of at
// most 2 KB (K <= 4096). At M = 1 the FFMA2 staged kernel is faster (measured on GB300,
// Q4_0 32768 x 2048: 13.0 us FFMA2, 16.4 us MMA); from M = 2 the MMA's cost does not grow
// with the token count while FFMA2's does (M = 4: 17.0 us MMA, 29.5 us FFMA2).
// TR = 32 rows (2 row groups x 2 K slices) when that still gives 4 tiles per SM, else
// 16 rows (4 K slices).
bool launch_q4_mma(const GroupRef& g, bool pdl, int* status, cudaStream_t s, cudaError_t& err) {
    if (g.fmt != EMB_Q4_0 || g.M < 2 || g.M > kMmaMaxM || g.epi >= EMB_EPI_GEGLU) return false;
    const int64_t row_bytes = g.K / 2;
    if (row_bytes * 16 > kMmaTileBytes) return false;
    if (g.M * g.K * 2 > kStageXBytes) return false;
    int64_t rows = 0;
    for (int i = 0; i < g.n_mats; ++i) rows += g.mats[i].N;
    if (rows * row_bytes < kStageMinBytes) return false;
    const int nb = int(g.K / kQBlock);
    int TR = 16, WK = 4;
    if (row_bytes * 32 <= kMmaTileBytes && rows / 32 >= 4 * 152) { TR = 32; WK = 2; }
    if (nb < WK) WK = 1, TR = 16 * kMmaWarps;  // too few blocks to split K: 4 row groups
    if (TR * row_bytes > kMmaTileBytes) return false;
    MmaParams p = {};
    int tiles = 0;
    for (int i = 0; i < g.n_mats; ++i) {
        p.codes[i] = g.mats[i].codes;
        p.scales[i] = g.mats[i].scales;
        p.Y[i] = g.mats[i].Y;
        p.N[i] = int32_t(g.mats[i].N);
        p.tile0[i] = tiles;
        tiles += int((g.mats[i].N + TR - 1) / TR);
    }
    p.tile0[g.n_mats] = tiles;
    p.n_mats = g.n_mats;
    p.M = int32_t(g.M);
    p.K = int32_t(g.K);
    p.ldS = int32_t(g.ldS);
    p.TR = TR;
    p.WK = WK;
    p.pitch = int32_t(row_bytes + 16);
    p.spitch = int32_t(g.ldS * 2 + 16);
    p.epi = g.epi;
    p.X = g.X;
    p.status = status;
    const size_t smem = size_t(kMmaHeader) + size_t(g.M) * g.K * 2 + size_t(TR) * (p.pitch + p.spitch);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(tiles, 1, 1);
    cfg.blockDim = dim3(kMmaThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    if (smem > 48 * 1024) {
        err = cudaFuncSetAttribute(gemv_q4_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        if (err != cudaSuccess) return true;
    }
    err = cudaLaunchKernelEx(&cfg, gemv_q4_mma_kernel, p);
    return true;
}

// ------------------------------------------------------------------ ring GEMV
// Long rows at M = 1 (more than one pass of 256 threads; Gemma-2B's down projection,
// 2048 x 16384). The register kernel holds only as many bytes in flight as the resident
// CTAs' registers, so such a matrix streams in two waves of CTAs whose loads do not overlap,
// and the staged kernel re-stages the whole activation row for every tile of one or two
// rows. Here a CTA owns a run of consecutive rows (crossing
// matrix boundaries within the group) and keeps the activation row it needs in registers:
// each thread's units t + k*256 of X, loaded once after griddepcontrol.wait and reused for
// every row. The rows stream through a ring of shared-memory stages (one row of codes and
// its scales each; as many as kRingBudget holds, 2..8), filled by bulk copies that one
// thread issues -- a ring's worth before the wait -- and refills as soon as all eight warps
// have released a stage. The warps run on the ring's barriers alone (no CTA-wide barrier
// until the reduction). Each row is summed as in the register kernel (per thread over its
// units in order, shuffle tree, warps in order), so its bits equal that kernel's.
constexpr int kRingThreads = 256;
constexpr int kRingMaxStages = 8;
constexpr int kRingBudget = 56 * 1024;  // ring bytes per CTA: stages = budget / stage, 2..8
constexpr int kRingFlush = 16;  // rows whose per-warp sums are kept before a CTA-wide reduction
// barriers (0..127), abort flag (128), per-warp sums (144..655), then the ring
constexpr int kRingHeader = 144 + kRingFlush * (kRingThreads / 32) * 4;

struct RingParams {
    const uint8_t* codes[kMaxGroup];
    const uint8_t* high[kMaxGroup];  // Q6_0: 2-bit high plane of each matrix
    const __half* scales[kMaxGroup];
    void* Y[kMaxGroup];
    int32_t N[kMaxGroup];
    int32_t row0[kMaxGroup + 1];  // first row of each matrix in the group's row order
    int32_t n_mats;
    int32_t K, ldS, U;
    int32_t rows_per_cta, rows_total;
    int32_t stage_bytes;          // one row of codes (+ Q6_0 high bits) + its scales, rounded up to 16
    int32_t stages;               // ring depth (2..kRingMaxStages)
    int32_t epi;
    const __nv_bfloat16* X;
    int* status;
};

template <int FMT, int PF>
__global__ void __launch_bounds__(kRingThreads, 2) gemv_ring_kernel(const __grid_constant__ RingParams p) {
    constexpr int UW = (FMT == EMB_Q8_0) ? 16 : 32;
    constexpr int NT = kRingThreads, NWARP = NT / 32;
    extern __shared__ __align__(128) uint8_t smem[];
    uint64_t* full = reinterpret_cast<uint64_t*>(smem);              // [stages]
    uint64_t* empty = full + kRingMaxStages;                          // [stages]
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + 128);  // a wait gave up
    float* red = reinterpret_cast<float*>(smem + 144);               // [kRingFlush][NWARP]
    uint8_t* ring = smem + kRingHeader;                               // [stages][stage_bytes]
    const int S = p.stages;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int U = p.U;
    const int64_t row_bytes = (FMT == EMB_Q8_0) ? int64_t(p.K) : int64_t(p.K) / 2;
    const int64_t high_bytes = (FMT == EMB_Q6_0) ? int64_t(p.K) / 4 : 0;  // a multiple of 16
    const int r_begin = blockIdx.x * p.rows_per_cta;
    const int n_rows = min(p.rows_per_cta, p.rows_total - r_begin);
    // global row -> (matrix, row within it)
    auto locate = [&](int gr, int& g, int& n) {
        g = 0;
#pragma unroll
        for (int i = 1; i < kMaxGroup; ++i)
            if (i < p.n_mats && gr >= p.row0[i]) g = i;
        n = gr - p.row0[g];
    };
    auto issue = [&](int i, int stage) {  // row i of this CTA into a stage
        int g, n;
        locate(r_begin + i, g, n);
        uint8_t* st = ring + stage * p.stage_bytes;
        uint64_t* bar = &full[stage];
        const uint32_t cb = uint32_t(row_bytes), hb = uint32_t(high_bytes), sb = uint32_t(p.ldS) * 2u;
        ptx::mbar_arrive_expect_tx(bar, cb + hb + sb);
        ptx::bulk_load(st, p.codes[g] + int64_t(n) * row_bytes, cb, bar);
        if constexpr (FMT == EMB_Q6_0) ptx::bulk_load(st + row_bytes, p.high[g] + int64_t(n) * high_bytes, hb, bar);
        ptx::bulk_load(st + row_bytes + high_bytes, p.scales[g] + int64_t(n) * p.ldS, sb, bar);
    };
    if (t == 0) {
        *abort_flag = 0;
        for (int i = 0; i < S; ++i) {
            ptx::mbar_init(&full[i], 1);
            ptx::mbar_init(&empty[i], NWARP);
        }
        ptx::fence_mbar_init();
        for (int i = 0; i < S && i < n_rows; ++i) issue(i, i);
        // the activation row towards L2 while the previous launch finishes (one CTA asks)
        if (blockIdx.x == 0) ptx::prefetch_l2(p.X, uint32_t(p.K) * 2u);
    }
    griddep_launch_dependents();
    __syncthreads();  // the barriers' initialisation is visible to every waiting thread
    // weights do not depend on earlier launches; X and Y may
    griddep_wait();
    float x[PF][UW];
#pragma unroll
    for (int k = 0; k < PF; ++k) {
        const int uk = t + k * NT;
        const uint4* xp = reinterpret_cast<const uint4*>(p.X + int64_t(min(uk, U - 1)) * UW);
#pragma unroll
        for (int v = 0; v < UW / 8; ++v) {
            const uint4 hx = xp[v];
            x[k][8 * v + 0] = lo_bf16(hx.x); x[k][8 * v + 1] = hi_bf16(hx.x);
            x[k][8 * v + 2] = lo_bf16(hx.y); x[k][8 * v + 3] = hi_bf16(hx.y);
            x[k][8 * v + 4] = lo_bf16(hx.z); x[k][8 * v + 5] = hi_bf16(hx.z);
            x[k][8 * v + 6] = lo_bf16(hx.w); x[k][8 * v + 7] = hi_bf16(hx.w);
        }
    }
    const uint2 h0 = make_uint2(0, 0);
    bool ok = true;
    int flushed = 0;  // rows already reduced and stored
    // reduce and store rows [flushed, upto) of this CTA; false (the CTA leaves) if any of its
    // waits gave up. The only CTA-wide barriers: between them the warps run on the ring's
    // barriers alone, each wait bounded and abandoned as soon as another thread gave up.
    auto flush = [&](int upto) -> bool {
        if (__syncthreads_or(!ok)) return false;
        const int cnt = upto - flushed;
        if (p.epi >= EMB_EPI_GEGLU) {
            // gate row 2i and up row 2i + 1 of the CTA (runs start on even rows)
            if (t < cnt / 2) {
                float gate = 0.0f, up = 0.0f;
#pragma unroll
                for (int w = 0; w < NWARP; ++w) {
                    gate += red[(2 * t) * NWARP + w];
                    up += red[(2 * t + 1) * NWARP + w];
                }
                int g, n;
                locate(r_begin + flushed + 2 * t, g, n);
                epi_store_gated(p.epi, p.Y[g], 0, n, p.N[g], gate, up);
            }
        } else if (t < cnt) {
            float v = 0.0f;
#pragma unroll
            for (int w = 0; w < NWARP; ++w) v += red[t * NWARP + w];
            int g, n;
            locate(r_begin + flushed + t, g, n);
            epi_store(p.epi, p.Y[g], 0, n, p.N[g], v);
        }
        __syncthreads();
        flushed = upto;
        return true;
    };
    // stage and phase of row i, and of row i - 1, kept by increments (no integer division)
    int s = 0, sp = 0;
    uint32_t ph = 0, php = 0;
    for (int i = 0; i < n_rows; ++i) {
        // refill: the stage of row i - 1 once every warp has released it
        if (t == 0 && ok && i >= 1 && i - 1 + S < n_rows) {
            ok = ptx::mbar_wait(&empty[sp], php, abort_flag, p.status, kWaitLimitNs);
            if (ok) issue(i - 1 + S, sp);
        }
        ok = __all_sync(0xffffffffu, ok && ptx::mbar_wait(&full[s], ph, abort_flag, p.status, kWaitLimitNs));
        if (ok) {
            const uint8_t* cs = ring + s * p.stage_bytes;
            const __half* ss = reinterpret_cast<const __half*>(cs + row_bytes + high_bytes);
            float acc = 0.0f;
#pragma unroll
            for (int k = 0; k < PF; ++k) {
                const int uk = t + k * NT;
                if (uk < U) {
                    const uint4 c = *reinterpret_cast<const uint4*>(cs + int64_t(uk) * 16);
                    uint2 hq = h0;
                    if constexpr (FMT == EMB_Q6_0) hq = *reinterpret_cast<const uint2*>(cs + row_bytes + int64_t(uk) * 8);
                    const float d = __half2float(ss[(FMT == EMB_Q8_0) ? (uk >> 1) : uk]);
                    acc = fmaf(d, dot_unit<FMT>(c, hq, x[k]), acc);
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&empty[s]);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
            if (lane == 0) red[(i - flushed) * NWARP + warp] = acc;
        }
        if (i + 1 - flushed == kRingFlush && !flush(i + 1)) return;
        sp = s;
        php = ph;
        if (++s == S) {
            s = 0;
            ph ^= 1u;
        }
    }
    if (flushed < n_rows) flush(n_rows);  // (a CTA whose wait gave up leaves inside it)
}

template <int FMT, int PF>
cudaError_t launch_ring_one(const RingParams& p, int ctas, size_t smem, bool pdl, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(ctas, 1, 1);
    cfg.blockDim = dim3(kRingThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    const cudaError_t e = cudaFuncSetAttribute(gemv_ring_kernel<FMT, PF>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e != cudaSuccess) return e;
    return cudaLaunchKernelEx(&cfg, gemv_ring_kernel<FMT, PF>, p);
}

int gemv_sm_count() {
    static std::mutex mu;
    static int counts[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    std::lock_guard<std::mutex> lock(mu);
    if (!counts[dev] && cudaDeviceGetAttribute(&counts[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        counts[dev] = 0;
    return counts[dev];
}

// Which layers take the ring path: M = 1, Q8_0, Q4_0 or Q6_0 (K % 64 == 0, for its high
// plane's 16-byte rows), rows longer than the staged path takes at M = 1 and than one pass
// of 256 threads (2..4 units per thread), matrices of at least kStageMinBytes; two CTAs per
// SM, rows split evenly (even runs for gated epilogues).
// Measured on GB300, Gemma-2B decode step (paired runs on one box, 1000 steps): Q8_0 chain
// 0.507 -> 0.477 ms and Q4_0 0.457 -> 0.455 against a kernel with two rows per CTA in
// registers and two in shared memory; a 72 KB ring instead of 56 KB was slower for Q8_0,
// a CTA-wide barrier per row cost ~2 %, and stage indices by integer division ~4 %.
bool launch_ring(const GroupRef& g, bool pdl, int* status, cudaStream_t s, cudaError_t& err) {
    if (g.M != 1 || (g.fmt == EMB_Q6_0 && g.K % 64 != 0)) return false;
    const int64_t row_bytes = (g.fmt == EMB_Q8_0) ? g.K : g.K / 2;
    const int64_t high_bytes = (g.fmt == EMB_Q6_0) ? g.K / 4 : 0;
    const int64_t U = (g.fmt == EMB_Q8_0) ? g.K / 16 : g.K / 32;
    if (row_bytes + high_bytes <= kStageMaxRowBytesM1 || U <= kRingThreads || U > 4 * kRingThreads) return false;
    int64_t rows = 0;
    for (int i = 0; i < g.n_mats; ++i) rows += g.mats[i].N;
    if (rows * (row_bytes + high_bytes) < kStageMinBytes) return false;
    const int sms = gemv_sm_count();
    if (sms <= 0) return false;
    RingParams p = {};
    int64_t r0 = 0;
    for (int i = 0; i < g.n_mats; ++i) {
        p.codes[i] = g.mats[i].codes;
        p.high[i] = g.mats[i].high;
        p.scales[i] = g.mats[i].scales;
        p.Y[i] = g.mats[i].Y;
        p.N[i] = int32_t(g.mats[i].N);
        p.row0[i] = int32_t(r0);
        r0 += g.mats[i].N;
    }
    p.row0[g.n_mats] = int32_t(r0);
    p.n_mats = g.n_mats;
    p.K = int32_t(g.K);
    p.ldS = int32_t(g.ldS);
    p.U = int32_t(U);
    p.epi = g.epi;
    p.X = g.X;
    p.status = status;
    int64_t rpc = (rows + 2 * sms - 1) / (2 * sms);
    if (g.epi >= EMB_EPI_GEGLU) rpc = (rpc + 1) & ~int64_t(1);  // gate/up pairs stay in one CTA
    p.rows_per_cta = int32_t(rpc);
    p.rows_total = int32_t(rows);
    p.stage_bytes = int32_t((row_bytes + high_bytes + g.ldS * 2 + 15) & ~int64_t(15));
    p.stages = int32_t(std::min<int64_t>(kRingMaxStages, std::max<int64_t>(2, kRingBudget / p.stage_bytes)));
    const int ctas = int((rows + rpc - 1) / rpc);
    const size_t smem = kRingHeader + size_t(p.stages) * p.stage_bytes;
    const int pf = int((U + kRingThreads - 1) / kRingThreads);
    if (g.fmt == EMB_Q8_0)
        err = pf == 2 ? launch_ring_one<EMB_Q8_0, 2>(p, ctas, smem, pdl, s)
            : pf == 3 ? launch_ring_one<EMB_Q8_0, 3>(p, ctas, smem, pdl, s)
                      : launch_ring_one<EMB_Q8_0, 4>(p, ctas, smem, pdl, s);
    else if (g.fmt == EMB_Q4_0)
        err = pf == 2 ? launch_ring_one<EMB_Q4_0, 2>(p, ctas, smem, pdl, s)
            : pf == 3 ? launch_ring_one<EMB_Q4_0, 3>(p, ctas, smem, pdl, s)
                      : launch_ring_one<EMB_Q4_0, 4>(p, ctas, smem, pdl, s);
    else
        err = pf == 2 ? launch_ring_one<EMB_Q6_0, 2>(p, ctas, smem, pdl, s)
            : pf == 3 ? launch_ring_one<EMB_Q6_0, 3>(p, ctas, smem, pdl, s)
                      : launch_ring_one<EMB_Q6_0, 4>(p, ctas, smem, pdl, s);
    return true;
}

}  // namespace

cudaError_t launch_gemv_regs(const GroupRef& g, bool pdl, cudaStream_t s);

cudaError_t launch_gemv(const GroupRef& g, bool pdl, int* status, cudaStream_t s) {
    cudaError_t err = cudaSuccess;
    if (launch_q4_mma(g, pdl, status, s, err)) return err;
    if (launch_staged(g, pdl, status, s, err)) return err;
    if (launch_ring(g, pdl, status, s, err)) return err;
    return launch_gemv_regs(g, pdl, s);
}

// Register-streaming GEMV: every shape the staged path leaves out.
cudaError_t launch_gemv_regs(const GroupRef& g, bool pdl, cudaStream_t s) {
    GemvParams p = {};
    const int U = int((g.fmt == EMB_Q8_0) ? g.K / 16 : g.K / 32);
    int64_t rows = 0;
    for (int i = 0; i < g.n_mats; ++i) rows += g.mats[i].N;
    // rows per CTA: 4 (activation reuse across rows) unless that leaves the GPU idle;
    // 2 for long rows (U >= 320), where 4 rows leave too few CTAs per SM (measured on
    // GB300, M=1: Q8_0 2048 x 16384 10.8 us with 4 rows, 9.6 us with 2)
    int R = (rows < 4 * 2 * 152) ? 1 : (U >= 320) ? 2 : 4;
    if (g.epi >= EMB_EPI_GEGLU && R == 1) R = 2;  // gate/up row pairs inside one CTA
    int tiles = 0;
    for (int i = 0; i < g.n_mats; ++i) {
        p.codes[i] = g.mats[i].codes;
        p.high[i] = g.mats[i].high;
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
    p.epi = g.epi;
    p.X = g.X;
    const int NT = pick_threads(U, g.fmt, tiles);
    const int M = int(g.M);
    if (g.fmt == EMB_Q8_0)
        return R == 4 ? dispatch_nt<EMB_Q8_0, 4>(p, tiles, M, NT, pdl, s)
             : R == 2 ? dispatch_nt<EMB_Q8_0, 2>(p, tiles, M, NT, pdl, s)
                      : dispatch_nt<EMB_Q8_0, 1>(p, tiles, M, NT, pdl, s);
    if (g.fmt == EMB_Q4_0)
        return R == 4 ? dispatch_nt<EMB_Q4_0, 4>(p, tiles, M, NT, pdl, s)
             : R == 2 ? dispatch_nt<EMB_Q4_0, 2>(p, tiles, M, NT, pdl, s)
                      : dispatch_nt<EMB_Q4_0, 1>(p, tiles, M, NT, pdl, s);
    return R == 4 ? dispatch_nt<EMB_Q6_0, 4>(p, tiles, M, NT, pdl, s)
         : R == 2 ? dispatch_nt<EMB_Q6_0, 2>(p, tiles, M, NT, pdl, s)
                  : dispatch_nt<EMB_Q6_0, 1>(p, tiles, M, NT, pdl, s);
}

}  // namespace emb
