// The non-matmul steps of one transformer layer of the shared backbone and the action
// expert (the paper's single backbone execution path, Section 3.2): RMSNorm of the fp32
// residual stream into the bf16 activations of the next linear, rotary position
// embedding of q and k in place, and grouped-head attention of a chunk of queries over a
// prefix key/value cache plus the chunk's own keys. Definitions: RMSNorm (Zhang and
// Sennrich, 2019), rotary embedding with rotate-half pairs (Su et al., 2021), scaled
// dot-product attention (Vaswani et al., 2017); all keys are visible to every query.
//
// Every kernel is launched with programmatic stream serialisation and reads its inputs
// only after griddepcontrol.wait, so it chains behind the layer launches of emb_qlayer_seq.
#include <algorithm>
#include <cmath>
#include <mutex>

#include "ptx.cuh"

namespace emb {
namespace {

cudaError_t launch_pdl(const void* fn, dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       void** args, unsigned cluster_z = 1) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    int na = 1;
    if (cluster_z > 1) {
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = 1;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = cluster_z;
        na = 2;
    }
    cfg.attrs = attr;
    cfg.numAttrs = na;
    return cudaLaunchKernelExC(&cfg, fn, args);
}

// ------------------------------------------------------------------ RMSNorm
// One CTA per token: the sum of squares in fp32 (per-thread partial sums of 4-element
// groups, then a shuffle tree and the warps' sums in order), mean = sum / D, one correctly
// rounded square root and reciprocal, then y = bf16(x * inv * gamma).
constexpr int kNormThreads = 256;

// x is read with ordinary loads (not the read-only path): the previous launch wrote it
// while this grid was already resident (programmatic dependent launch); its writes are
// visible to ordinary loads after griddepcontrol.wait.
__global__ void __launch_bounds__(kNormThreads) rmsnorm_kernel(const float* x,
                                                               const float* __restrict__ gamma,
                                                               __nv_bfloat16* __restrict__ y,
                                                               int D, float eps) {
    ptx::griddep_launch_dependents();
    ptx::griddep_wait();  // x is the residual stream the previous launch wrote
    const int64_t row = blockIdx.x;
    const float* xr = x + row * D;
    float ss = 0.0f;
    for (int i = threadIdx.x * 4; i < D; i += kNormThreads * 4) {
        const float4 v = *reinterpret_cast<const float4*>(xr + i);
        ss = fmaf(v.x, v.x, ss);
        ss = fmaf(v.y, v.y, ss);
        ss = fmaf(v.z, v.z, ss);
        ss = fmaf(v.w, v.w, ss);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    __shared__ float warp_ss[kNormThreads / 32];
    __shared__ float inv_s;
    if ((threadIdx.x & 31) == 0) warp_ss[threadIdx.x >> 5] = ss;
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.0f;
        for (int w = 0; w < kNormThreads / 32; ++w) t += warp_ss[w];
        inv_s = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(__fdiv_rn(t, float(D)), eps)));
    }
    __syncthreads();
    const float inv = inv_s;
    __nv_bfloat16* yr = y + row * D;
    for (int i = threadIdx.x * 4; i < D; i += kNormThreads * 4) {
        const float4 v = *reinterpret_cast<const float4*>(xr + i);
        const float4 g = *reinterpret_cast<const float4*>(gamma + i);
        const __nv_bfloat162 lo = __floats2bfloat162_rn(__fmul_rn(__fmul_rn(v.x, inv), g.x),
                                                        __fmul_rn(__fmul_rn(v.y, inv), g.y));
        const __nv_bfloat162 hi = __floats2bfloat162_rn(__fmul_rn(__fmul_rn(v.z, inv), g.z),
                                                        __fmul_rn(__fmul_rn(v.w, inv), g.w));
        uint2 u;
        u.x = *reinterpret_cast<const uint32_t*>(&lo);
        u.y = *reinterpret_cast<const uint32_t*>(&hi);
        *reinterpret_cast<uint2*>(yr + i) = u;
    }
}

// ------------------------------------------------------------------ rotary embedding
// One thread per rotated pair (element i and i + d/2 of one head of one token). The host
// passes each pair's inverse frequency base^(-2i/d), computed in fp64, as two floats
// (hi + lo). The angle p * (hi + lo) is formed as an unevaluated sum A + a with one exact
// FMA residual (p < 2^24 is exact in fp32), its sine and cosine as sincosf(A) corrected to
// first order in a: error ~1e-7 at the positions of a prefix plus action chunk, against
// ~|angle| * 2^-24 for a plain fp32 angle.
constexpr int kRopeMaxPairs = 256;

struct RopeParams {
    __nv_bfloat16* x;   // [M][n_heads][head_dim]
    __nv_bfloat16* x2;  // [M][n_heads2][head_dim] at the same positions, or nothing (n_heads2 = 0)
    int64_t pairs1, pairs, pos0;
    int n_heads, n_heads2, head_dim;
    float inv_hi[kRopeMaxPairs], inv_lo[kRopeMaxPairs];
};

__global__ void __launch_bounds__(256) rope_kernel(const __grid_constant__ RopeParams p) {
    ptx::griddep_launch_dependents();
    ptx::griddep_wait();  // x was written by the previous launch
    const int half = p.head_dim / 2;
    for (int64_t t0 = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; t0 < p.pairs;
         t0 += int64_t(gridDim.x) * blockDim.x) {
        const bool second = t0 >= p.pairs1;  // the pairs of x come first, then those of x2
        const int64_t t = second ? t0 - p.pairs1 : t0;
        const int heads = second ? p.n_heads2 : p.n_heads;
        const int64_t per_token = int64_t(heads) * half;
        const int64_t m = t / per_token;
        const int r = int(t - m * per_token);
        const int h = r / half, i = r - h * half;
        const float pos = float(p.pos0 + m);
        const float A = __fmul_rn(pos, p.inv_hi[i]);
        const float a = __fadd_rn(fmaf(pos, p.inv_hi[i], -A), __fmul_rn(pos, p.inv_lo[i]));
        float sA, cA;
        sincosf(A, &sA, &cA);
        const float c = fmaf(-a, sA, cA), s = fmaf(a, cA, sA);
        __nv_bfloat16* xp = (second ? p.x2 : p.x) + m * (int64_t(heads) * p.head_dim) + int64_t(h) * p.head_dim + i;
        const float xa = __bfloat162float(xp[0]), xb = __bfloat162float(xp[half]);
        xp[0] = __float2bfloat16_rn(__fsub_rn(__fmul_rn(xa, c), __fmul_rn(xb, s)));
        xp[half] = __float2bfloat16_rn(__fadd_rn(__fmul_rn(xb, c), __fmul_rn(xa, s)));
    }
}

// ------------------------------------------------------------------ attention
// Tensor-core attention (mma.sync m16n8k16, bf16 operands, fp32 accumulation). The rows of
// one key/value head g are its (query m, head) pairs, row r = m * G + (h - g * G) with G the
// heads per key/value head, so every query head of a group shares the key and value tiles.
// CTA = (64 rows, key/value head, key split); warp w owns rows 16w..16w+15 of the CTA.
// Per 64-key tile (double-buffered in shared memory by cp.async, rows padded by 16 bytes so
// fragment loads are conflict-free): S = Q K^T (Q fragments held in registers for the whole
// kernel), scale, an online softmax on the accumulator fragments (row max and sums over the
// four lanes that share a row), then O += P V with P split into bf16 hi + lo parts (two MMAs,
// weight error 2^-16) and V fragments from ldmatrix.trans. The key splits of one row block
// form a cluster along z; their (max, sum, output) partials are combined through distributed
// shared memory in split order (deterministic).
constexpr int kAttnWarps = 4;
constexpr int kAttnThreads = 32 * kAttnWarps;
constexpr int kAttnRows = 16 * kAttnWarps;
constexpr int kKeyTile = 64;
constexpr int kMaxSplits = 16;      // cluster size along the keys (16: non-portable, opted in)
constexpr int kMinSplitKeys = 48;   // keys per split, at least

template <int D>
struct AttnSmem {
    static constexpr int kPitch = D + 8;                 // bf16 per padded key row
    __nv_bfloat16 k[2][kKeyTile][kPitch];
    __nv_bfloat16 v[2][kKeyTile][kPitch];
    float part_o[kAttnRows][D];
    float part_m[kAttnRows], part_l[kAttnRows];
};

struct AttnParams {
    const __nv_bfloat16* Q;
    const __nv_bfloat16* K0;
    const __nv_bfloat16* V0;
    const __nv_bfloat16* K1;
    const __nv_bfloat16* V1;
    __nv_bfloat16* O;
    int64_t n0, n1;
    int M, H, Hk;
    float scale;
};

__device__ __forceinline__ void mma_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
        "{%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t saddr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                              uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(saddr));
}

// 16-byte global -> shared copy; src_bytes 0 writes zeros (the source is not read).
__device__ __forceinline__ void cp_async16(uint32_t saddr, const void* g, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(saddr), "l"(g), "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&v);
}
__device__ __forceinline__ float2 unpack_bf16x2(uint32_t w) {
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}

template <int D>
__global__ void __launch_bounds__(kAttnThreads) attention_kernel(const __grid_constant__ AttnParams p) {
    constexpr int KS = D / 16;  // k-steps of the score MMAs (head dims)
    constexpr int NT = D / 8;   // n-tiles of the output (head dims)
    using SM = AttnSmem<D>;
    extern __shared__ __align__(128) uint8_t smem_raw[];
    SM& sm = *reinterpret_cast<SM*>(smem_raw);
    ptx::griddep_launch_dependents();
    ptx::griddep_wait();  // Q and the chunk's keys and values come from the previous launches

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quad = lane >> 2, qc = lane & 3;
    const int g = blockIdx.y, G = p.H / p.Hk;
    const int64_t rows_total = int64_t(p.M) * G;
    const int64_t row0 = int64_t(blockIdx.x) * kAttnRows;
    const int splits = gridDim.z, z = blockIdx.z;
    const int64_t n = p.n0 + p.n1;
    const int64_t k_lo = z * n / splits, k_hi = (z + 1) * n / splits;
    const int kv_stride = p.Hk * D;

    // global row -> (query, head) -> its Q / O row; nullptr past the last row
    auto q_row = [&](int64_t r) -> int64_t {
        return r < rows_total ? (r / G) * int64_t(p.H) * D + (int64_t(g) * G + r % G) * D : -1;
    };
    const int64_t rA = row0 + warp * 16 + quad, rB = rA + 8;
    const int64_t offA = q_row(rA), offB = q_row(rB);

    // Q fragments for the whole kernel (A operand, row-major 16 x D); ordinary loads, since
    // the previous launch wrote Q while this grid was already resident
    uint32_t qf[KS][4];
    auto ldq = [&](int64_t off) { return *reinterpret_cast<const uint32_t*>(p.Q + off); };
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
        const int c = ks * 16 + 2 * qc;
        qf[ks][0] = offA >= 0 ? ldq(offA + c) : 0u;
        qf[ks][1] = offB >= 0 ? ldq(offB + c) : 0u;
        qf[ks][2] = offA >= 0 ? ldq(offA + c + 8) : 0u;
        qf[ks][3] = offB >= 0 ? ldq(offB + c + 8) : 0u;
    }

    // tile loader: 64 keys x D of keys and of values, 16-byte chunks, zero past the split
    auto issue_tile = [&](int64_t t0, int stage) {
        constexpr int kChunksPerRow = D / 8;
        for (int e = threadIdx.x; e < kKeyTile * kChunksPerRow; e += kAttnThreads) {
            const int j = e / kChunksPerRow, c = e - j * kChunksPerRow;
            const int64_t key = t0 + j;
            const bool ok = key < k_hi;
            const int64_t kk = ok ? key : k_lo;  // any valid row when nothing is read
            const __nv_bfloat16* kp = kk < p.n0 ? p.K0 + kk * kv_stride : p.K1 + (kk - p.n0) * kv_stride;
            const __nv_bfloat16* vp = kk < p.n0 ? p.V0 + kk * kv_stride : p.V1 + (kk - p.n0) * kv_stride;
            cp_async16(ptx::smem_u32(&sm.k[stage][j][c * 8]), kp + g * D + c * 8, ok ? 16 : 0);
            cp_async16(ptx::smem_u32(&sm.v[stage][j][c * 8]), vp + g * D + c * 8, ok ? 16 : 0);
        }
    };

    float o[NT][4];
#pragma unroll
    for (int j = 0; j < NT; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.0f;
    float mA = -INFINITY, mB = -INFINITY, lA = 0.0f, lB = 0.0f;

    const int ntiles = int((k_hi - k_lo + kKeyTile - 1) / kKeyTile);
    if (ntiles > 0) issue_tile(k_lo, 0);
    cp_async_commit();
    for (int it = 0; it < ntiles; ++it) {
        const int stage = it & 1;
        const int64_t t0 = k_lo + int64_t(it) * kKeyTile;
        if (it + 1 < ntiles) issue_tile(t0 + kKeyTile, stage ^ 1);
        cp_async_commit();
        cp_async_wait1();  // this thread's copies of tile `it` have landed
        __syncthreads();   // and every thread's

        // S = Q K^T for 64 keys: 8 n-tiles of 8 keys
        float sc[8][4];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            sc[j][0] = sc[j][1] = sc[j][2] = sc[j][3] = 0.0f;
            const __nv_bfloat16* krow = &sm.k[stage][j * 8 + quad][0];
#pragma unroll
            for (int ks = 0; ks < KS; ++ks) {
                const uint32_t b0 = *reinterpret_cast<const uint32_t*>(krow + ks * 16 + 2 * qc);
                const uint32_t b1 = *reinterpret_cast<const uint32_t*>(krow + ks * 16 + 2 * qc + 8);
                mma_16816(sc[j], qf[ks], b0, b1);
            }
        }
        // scale, mask keys past the split, row maxima (rows A = quad, B = quad + 8)
        float tA = -INFINITY, tB = -INFINITY;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const bool ok = t0 + j * 8 + 2 * qc + e < k_hi;
                sc[j][e] = ok ? __fmul_rn(sc[j][e], p.scale) : -INFINITY;
                sc[j][2 + e] = ok ? __fmul_rn(sc[j][2 + e], p.scale) : -INFINITY;
                tA = fmaxf(tA, sc[j][e]);
                tB = fmaxf(tB, sc[j][2 + e]);
            }
        }
#pragma unroll
        for (int x = 1; x <= 2; x <<= 1) {
            tA = fmaxf(tA, __shfl_xor_sync(0xffffffffu, tA, x));
            tB = fmaxf(tB, __shfl_xor_sync(0xffffffffu, tB, x));
        }
        const float nA = fmaxf(mA, tA), nB = fmaxf(mB, tB);  // finite: the tile has a key
        const float cA = (mA == -INFINITY) ? 0.0f : expf(mA - nA);
        const float cB = (mB == -INFINITY) ? 0.0f : expf(mB - nB);
        mA = nA;
        mB = nB;
        float sA = 0.0f, sB = 0.0f;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                sc[j][e] = expf(sc[j][e] - nA);  // exp(-inf) = 0 for masked keys
                sc[j][2 + e] = expf(sc[j][2 + e] - nB);
                sA += sc[j][e];
                sB += sc[j][2 + e];
            }
        }
        lA = lA * cA + sA;  // lane-partial sums; the four lanes of a row are added at the end
        lB = lB * cB + sB;
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            o[j][0] *= cA;
            o[j][1] *= cA;
            o[j][2] *= cB;
            o[j][3] *= cB;
        }
        // O += P V: 4 k-steps of 16 keys; P as hi + lo bf16 A fragments
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            uint32_t ah[4], al[4];
            const float* s0 = sc[2 * kk];
            const float* s1 = sc[2 * kk + 1];
            const float src[4][2] = {{s0[0], s0[1]}, {s0[2], s0[3]}, {s1[0], s1[1]}, {s1[2], s1[3]}};
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                ah[r] = pack_bf16x2(src[r][0], src[r][1]);
                const float2 h = unpack_bf16x2(ah[r]);
                al[r] = pack_bf16x2(__fsub_rn(src[r][0], h.x), __fsub_rn(src[r][1], h.y));
            }
            // ldmatrix.trans: lanes 0-7 keys 16kk..+7, 8-15 keys +8..+15 (dims 8jj..),
            // lanes 16-31 the same keys at dims 8jj + 8
            const int key = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
            const int dcol = (lane >> 4) * 8;
#pragma unroll
            for (int jj = 0; jj < NT; jj += 2) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4_trans(ptx::smem_u32(&sm.v[stage][key][jj * 8 + dcol]), b0, b1, b2, b3);
                mma_16816(o[jj], ah, b0, b1);
                mma_16816(o[jj], al, b0, b1);
                mma_16816(o[jj + 1], ah, b2, b3);
                mma_16816(o[jj + 1], al, b2, b3);
            }
        }
        __syncthreads();  // every warp is done with this stage before it is refilled
    }
#pragma unroll
    for (int x = 1; x <= 2; x <<= 1) {
        lA += __shfl_xor_sync(0xffffffffu, lA, x);
        lB += __shfl_xor_sync(0xffffffffu, lB, x);
    }

    if (splits == 1) {
        const float iA = __fdiv_rn(1.0f, lA), iB = __fdiv_rn(1.0f, lB);
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            const int c = j * 8 + 2 * qc;
            if (offA >= 0)
                *reinterpret_cast<__nv_bfloat162*>(p.O + offA + c) =
                    __floats2bfloat162_rn(__fmul_rn(o[j][0], iA), __fmul_rn(o[j][1], iA));
            if (offB >= 0)
                *reinterpret_cast<__nv_bfloat162*>(p.O + offB + c) =
                    __floats2bfloat162_rn(__fmul_rn(o[j][2], iB), __fmul_rn(o[j][3], iB));
        }
        return;
    }
    // partials of this split into shared memory, then the cluster combines them
    const int lrA = warp * 16 + quad, lrB = lrA + 8;
#pragma unroll
    for (int j = 0; j < NT; ++j) {
        const int c = j * 8 + 2 * qc;
        sm.part_o[lrA][c] = o[j][0];
        sm.part_o[lrA][c + 1] = o[j][1];
        sm.part_o[lrB][c] = o[j][2];
        sm.part_o[lrB][c + 1] = o[j][3];
    }
    if (qc == 0) {
        sm.part_m[lrA] = mA;
        sm.part_l[lrA] = lA;
        sm.part_m[lrB] = mB;
        sm.part_l[lrB] = lB;
    }
    ptx::cluster_sync();
    // CTA z combines rows [z * 64 / splits, (z + 1) * 64 / splits): one thread per 4 dims
    const int rows_per = kAttnRows / splits;
    for (int e = threadIdx.x; e < rows_per * (D / 4); e += kAttnThreads) {
        const int lr = z * rows_per + e / (D / 4), c = (e % (D / 4)) * 4;
        const int64_t off = q_row(row0 + lr);
        if (off < 0) continue;
        const uint32_t am = ptx::smem_u32(&sm.part_m[lr]), al_ = ptx::smem_u32(&sm.part_l[lr]);
        const uint32_t ao = ptx::smem_u32(&sm.part_o[lr][c]);
        float qm[kMaxSplits], ql[kMaxSplits];
        float4 qo[kMaxSplits];
#pragma unroll
        for (int q = 0; q < kMaxSplits; ++q) {
            if (q < splits) {
                qm[q] = ptx::ld_dsmem_f32(ptx::map_dsmem(am, q));
                ql[q] = ptx::ld_dsmem_f32(ptx::map_dsmem(al_, q));
                qo[q] = ptx::ld_dsmem_f32x4(ptx::map_dsmem(ao, q));
            }
        }
        float mx = -INFINITY;
#pragma unroll
        for (int q = 0; q < kMaxSplits; ++q)
            if (q < splits) mx = fmaxf(mx, qm[q]);
        float L = 0.0f;
        float4 O = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
        for (int q = 0; q < kMaxSplits; ++q) {
            if (q < splits && qm[q] != -INFINITY) {  // a split without keys adds nothing
                const float w = expf(qm[q] - mx);
                L = fmaf(ql[q], w, L);
                O.x = fmaf(qo[q].x, w, O.x);
                O.y = fmaf(qo[q].y, w, O.y);
                O.z = fmaf(qo[q].z, w, O.z);
                O.w = fmaf(qo[q].w, w, O.w);
            }
        }
        const float inv = __fdiv_rn(1.0f, L);
        const __nv_bfloat162 lo = __floats2bfloat162_rn(__fmul_rn(O.x, inv), __fmul_rn(O.y, inv));
        const __nv_bfloat162 hi = __floats2bfloat162_rn(__fmul_rn(O.z, inv), __fmul_rn(O.w, inv));
        uint2 u;
        u.x = *reinterpret_cast<const uint32_t*>(&lo);
        u.y = *reinterpret_cast<const uint32_t*>(&hi);
        *reinterpret_cast<uint2*>(p.O + off + c) = u;
    }
    ptx::cluster_sync();  // remote shared memory must outlive its readers
}

template <int D>
cudaError_t launch_attention_d(const AttnParams& p, int splits, cudaStream_t s) {
    const size_t smem = sizeof(AttnSmem<D>);
    // the opt-in shared-memory size and cluster size are per-device function attributes
    static std::mutex mu;
    static bool attr_done[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    if (dev < 0 || dev >= 64 || !attr_done[dev]) {
        e = cudaFuncSetAttribute(attention_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        if (e != cudaSuccess) return e;
        if (kMaxSplits > 8) {
            e = cudaFuncSetAttribute(attention_kernel<D>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
            if (e != cudaSuccess) return e;
        }
        if (dev >= 0 && dev < 64) attr_done[dev] = true;
    }
    AttnParams pc = p;
    void* args[] = {&pc};
    const int64_t row_blocks = (int64_t(p.M) * (p.H / p.Hk) + kAttnRows - 1) / kAttnRows;
    return launch_pdl(reinterpret_cast<const void*>(attention_kernel<D>),
                      dim3(unsigned(row_blocks), unsigned(p.Hk), unsigned(splits)), dim3(kAttnThreads),
                      smem, s, args, unsigned(splits));
}

}  // namespace

cudaError_t launch_rmsnorm(const float* x, const float* gamma, uint16_t* y, int64_t M, int64_t D,
                           float eps, cudaStream_t s) {
    const float* xa = x;
    const float* ga = gamma;
    __nv_bfloat16* ya = reinterpret_cast<__nv_bfloat16*>(y);
    int Di = int(D);
    void* args[] = {&xa, &ga, &ya, &Di, &eps};
    return launch_pdl(reinterpret_cast<const void*>(rmsnorm_kernel), dim3(unsigned(M)),
                      dim3(kNormThreads), 0, s, args);
}

cudaError_t launch_rope(uint16_t* x, int64_t n_heads, uint16_t* x2, int64_t n_heads2, int64_t M,
                        int64_t head_dim, int64_t pos0, double base, cudaStream_t s) {
    RopeParams p;
    p.x = reinterpret_cast<__nv_bfloat16*>(x);
    p.x2 = reinterpret_cast<__nv_bfloat16*>(x2);
    p.pairs1 = M * n_heads * (head_dim / 2);
    p.pairs = p.pairs1 + M * n_heads2 * (head_dim / 2);
    p.pos0 = pos0;
    p.n_heads = int(n_heads);
    p.n_heads2 = int(n_heads2);
    p.head_dim = int(head_dim);
    for (int i = 0; i < kRopeMaxPairs; ++i) {
        const double v = i < head_dim / 2 ? std::pow(base, -2.0 * double(i) / double(head_dim)) : 0.0;
        p.inv_hi[i] = float(v);
        p.inv_lo[i] = float(v - double(p.inv_hi[i]));
    }
    const int64_t blocks = std::min<int64_t>((p.pairs + 255) / 256, 152 * 16);
    void* args[] = {&p};
    return launch_pdl(reinterpret_cast<const void*>(rope_kernel), dim3(unsigned(blocks)), dim3(256), 0,
                      s, args);
}

cudaError_t launch_attention(const uint16_t* Q, const uint16_t* K0, const uint16_t* V0, int64_t n0,
                             const uint16_t* K1, const uint16_t* V1, int64_t n1, uint16_t* O,
                             int64_t M, int64_t H, int64_t Hk, int64_t D, float scale, cudaStream_t s) {
    AttnParams p;
    p.Q = reinterpret_cast<const __nv_bfloat16*>(Q);
    p.K0 = reinterpret_cast<const __nv_bfloat16*>(K0);
    p.V0 = reinterpret_cast<const __nv_bfloat16*>(V0);
    p.K1 = reinterpret_cast<const __nv_bfloat16*>(K1);
    p.V1 = reinterpret_cast<const __nv_bfloat16*>(V1);
    p.O = reinterpret_cast<__nv_bfloat16*>(O);
    p.n0 = n0;
    p.n1 = n1;
    p.M = int(M);
    p.H = int(H);
    p.Hk = int(Hk);
    p.scale = scale;
    // key splits (one cluster): at least kMinSplitKeys keys each, at most kMaxSplits
    const int64_t n = n0 + n1;
    int splits = 1;
    while (splits < kMaxSplits && n >= int64_t(2 * splits) * kMinSplitKeys) splits *= 2;
    return D == 64 ? launch_attention_d<64>(p, splits, s) : launch_attention_d<128>(p, splits, s);
}

}  // namespace emb
