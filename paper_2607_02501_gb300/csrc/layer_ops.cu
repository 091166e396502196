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

#include "ptx.cuh"

namespace emb {
namespace {

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

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

__global__ void __launch_bounds__(kNormThreads) rmsnorm_kernel(const float* __restrict__ x,
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
    __nv_bfloat16* x;
    int64_t pairs, pos0;
    int n_heads, head_dim;
    float inv_hi[kRopeMaxPairs], inv_lo[kRopeMaxPairs];
};

__global__ void __launch_bounds__(256) rope_kernel(const __grid_constant__ RopeParams p) {
    ptx::griddep_launch_dependents();
    ptx::griddep_wait();  // x was written by the previous launch
    const int half = p.head_dim / 2;
    const int64_t per_token = int64_t(p.n_heads) * half;
    for (int64_t t = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; t < p.pairs;
         t += int64_t(gridDim.x) * blockDim.x) {
        const int64_t m = t / per_token;
        const int r = int(t - m * per_token);
        const int h = r / half, i = r - h * half;
        const float pos = float(p.pos0 + m);
        const float A = __fmul_rn(pos, p.inv_hi[i]);
        const float a = __fadd_rn(fmaf(pos, p.inv_hi[i], -A), __fmul_rn(pos, p.inv_lo[i]));
        float sA, cA;
        sincosf(A, &sA, &cA);
        const float c = fmaf(-a, sA, cA), s = fmaf(a, cA, sA);
        __nv_bfloat16* xp = p.x + m * (int64_t(p.n_heads) * p.head_dim) + int64_t(h) * p.head_dim + i;
        const float xa = __bfloat162float(xp[0]), xb = __bfloat162float(xp[half]);
        xp[0] = __float2bfloat16_rn(__fsub_rn(__fmul_rn(xa, c), __fmul_rn(xb, s)));
        xp[half] = __float2bfloat16_rn(__fadd_rn(__fmul_rn(xb, c), __fmul_rn(xa, s)));
    }
}

// ------------------------------------------------------------------ attention
// CTA = (query m, key/value head g with up to 8 of its query heads, key split z). Warp w
// computes query head g * G + sub * 8 + w over this split's keys: key tiles of 64 staged
// in shared memory by all 256 threads (bf16, key rows padded by one 32-bit word so that 32
// lanes reading 32 different keys hit 32 banks), scores in fp32 (lane L scores keys L and
// L + 32 of the tile), an online softmax per tile, and the weighted values accumulated in
// fp32 (lane L owns D/32 consecutive dims). The splits of one (m, g, sub) form a cluster
// along z; their (max, sum, output) triples are combined through distributed shared memory
// in split order by the CTA whose rank matches the head (fixed order: deterministic).
constexpr int kAttnWarps = 8;
constexpr int kAttnThreads = 32 * kAttnWarps;
constexpr int kKeyTile = 64;

template <int D>
struct AttnSmem {
    float q[kAttnWarps][D];
    uint32_t k[kKeyTile][D / 2 + 1];  // bf16 pairs, one pad word per key row
    uint32_t v[kKeyTile][D / 2];
    float part_m[kAttnWarps], part_l[kAttnWarps];
    float part_o[kAttnWarps][D];
};

struct AttnParams {
    const __nv_bfloat16* Q;
    const __nv_bfloat16* K0;
    const __nv_bfloat16* V0;
    const __nv_bfloat16* K1;
    const __nv_bfloat16* V1;
    __nv_bfloat16* O;
    int64_t n0, n1;
    int M, H, Hk, subgroups;  // subgroups: CTAs (of <= 8 heads) per key/value head
    float scale;
};

template <int D>
__global__ void __launch_bounds__(kAttnThreads) attention_kernel(const __grid_constant__ AttnParams p) {
    constexpr int DL = D / 32;  // dims per lane
    static_assert(DL == 2 || DL == 4, "head_dim 64 or 128");
    extern __shared__ __align__(16) uint8_t smem_raw[];
    AttnSmem<D>& sm = *reinterpret_cast<AttnSmem<D>*>(smem_raw);
    ptx::griddep_launch_dependents();
    ptx::griddep_wait();  // Q and the chunk's keys and values come from the previous launches

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m = blockIdx.x;
    const int g = blockIdx.y / p.subgroups, sub = blockIdx.y - g * p.subgroups;
    const int G = p.H / p.Hk;
    const int h0 = g * G + sub * kAttnWarps;
    const int nh = min(kAttnWarps, G - sub * kAttnWarps);  // heads of this CTA
    const int splits = gridDim.z, z = blockIdx.z;
    const int64_t n = p.n0 + p.n1;
    const int64_t k_lo = z * n / splits, k_hi = (z + 1) * n / splits;
    const int kv_stride = p.Hk * D;

    // the CTA's queries, fp32
    for (int e = threadIdx.x; e < nh * D; e += kAttnThreads) {
        const int w = e / D, i = e - w * D;
        sm.q[w][i] = __bfloat162float(p.Q[int64_t(m) * p.H * D + int64_t(h0 + w) * D + i]);
    }

    float run_m = -INFINITY, run_l = 0.0f;
    float acc[DL];
#pragma unroll
    for (int d = 0; d < DL; ++d) acc[d] = 0.0f;

    // Key/value tiles: each thread moves kChunks 16-byte chunks of keys and of values per
    // tile; the next tile's chunks are loaded into registers while this tile is computed.
    constexpr int kChunks = kKeyTile * (D / 8) / kAttnThreads;
    static_assert(kChunks * kAttnThreads == kKeyTile * (D / 8), "tile split");
    uint4 kr[kChunks], vr[kChunks];
    auto load_tile = [&](int64_t t0) {
#pragma unroll
        for (int u = 0; u < kChunks; ++u) {
            const int e = threadIdx.x + u * kAttnThreads;
            const int j = e / (D / 8), c = e - j * (D / 8);
            const int64_t key = t0 + j;
            if (key < k_hi) {
                const __nv_bfloat16* kp = key < p.n0 ? p.K0 + key * kv_stride : p.K1 + (key - p.n0) * kv_stride;
                const __nv_bfloat16* vp = key < p.n0 ? p.V0 + key * kv_stride : p.V1 + (key - p.n0) * kv_stride;
                kr[u] = *reinterpret_cast<const uint4*>(kp + g * D + c * 8);
                vr[u] = *reinterpret_cast<const uint4*>(vp + g * D + c * 8);
            }
        }
    };
    if (k_lo < k_hi) load_tile(k_lo);
    for (int64_t t0 = k_lo; t0 < k_hi; t0 += kKeyTile) {
        const int nt = int(k_hi - t0 < kKeyTile ? k_hi - t0 : int64_t(kKeyTile));
        __syncthreads();  // the previous tile (and, first time, the queries) are consumed / written
#pragma unroll
        for (int u = 0; u < kChunks; ++u) {
            const int e = threadIdx.x + u * kAttnThreads;
            const int j = e / (D / 8), c = e - j * (D / 8);
            if (j < nt) {
                sm.k[j][c * 4 + 0] = kr[u].x;
                sm.k[j][c * 4 + 1] = kr[u].y;
                sm.k[j][c * 4 + 2] = kr[u].z;
                sm.k[j][c * 4 + 3] = kr[u].w;
                *reinterpret_cast<uint4*>(&sm.v[j][c * 4]) = vr[u];
            }
        }
        __syncthreads();
        if (t0 + kKeyTile < k_hi) load_tile(t0 + kKeyTile);
        if (warp < nh) {
            // scores of keys lane and lane + 32
            float s0 = 0.0f, s1 = 0.0f;
            const bool has0 = lane < nt, has1 = lane + 32 < nt;
            const uint32_t* k0 = sm.k[has0 ? lane : 0];
            const uint32_t* k1 = sm.k[has1 ? lane + 32 : 0];
            const float* q = sm.q[warp];
#pragma unroll 8
            for (int i = 0; i < D / 2; ++i) {
                const float2 qq = *reinterpret_cast<const float2*>(q + 2 * i);
                const uint32_t a = k0[i], b = k1[i];
                s0 = fmaf(qq.x, bf16_lo(a), s0);
                s0 = fmaf(qq.y, bf16_hi(a), s0);
                s1 = fmaf(qq.x, bf16_lo(b), s1);
                s1 = fmaf(qq.y, bf16_hi(b), s1);
            }
            s0 = has0 ? __fmul_rn(s0, p.scale) : -INFINITY;
            s1 = has1 ? __fmul_rn(s1, p.scale) : -INFINITY;
            float tmax = fmaxf(s0, s1);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, o));
            const float new_m = fmaxf(run_m, tmax);  // finite: the tile has at least one key
            const float corr = (run_m == -INFINITY) ? 0.0f : expf(run_m - new_m);
            const float p0 = has0 ? expf(s0 - new_m) : 0.0f;
            const float p1 = has1 ? expf(s1 - new_m) : 0.0f;
            float psum = p0 + p1;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, o);
            run_l = run_l * corr + psum;
            run_m = new_m;
#pragma unroll
            for (int d = 0; d < DL; ++d) acc[d] *= corr;
            // weighted values: key j's weight comes from lane j % 32
            for (int j = 0; j < nt; ++j) {
                const float pj = __shfl_sync(0xffffffffu, j < 32 ? p0 : p1, j & 31);
                if constexpr (DL == 4) {
                    const uint2 vv = *reinterpret_cast<const uint2*>(&sm.v[j][lane * 2]);
                    acc[0] = fmaf(pj, bf16_lo(vv.x), acc[0]);
                    acc[1] = fmaf(pj, bf16_hi(vv.x), acc[1]);
                    acc[2] = fmaf(pj, bf16_lo(vv.y), acc[2]);
                    acc[3] = fmaf(pj, bf16_hi(vv.y), acc[3]);
                } else {
                    const uint32_t vv = sm.v[j][lane];
                    acc[0] = fmaf(pj, bf16_lo(vv), acc[0]);
                    acc[1] = fmaf(pj, bf16_hi(vv), acc[1]);
                }
            }
        }
    }

    const int64_t out_row = int64_t(m) * p.H * D;
    if (splits == 1) {
        if (warp < nh) {
            const float inv = __fdiv_rn(1.0f, run_l);
            __nv_bfloat16* o = p.O + out_row + int64_t(h0 + warp) * D + lane * DL;
#pragma unroll
            for (int d = 0; d < DL; d += 2)
                *reinterpret_cast<__nv_bfloat162*>(o + d) =
                    __floats2bfloat162_rn(__fmul_rn(acc[d], inv), __fmul_rn(acc[d + 1], inv));
        }
        return;
    }
    // split combine through distributed shared memory
    if (warp < nh) {
        if (lane == 0) {
            sm.part_m[warp] = run_m;
            sm.part_l[warp] = run_l;
        }
#pragma unroll
        for (int d = 0; d < DL; ++d) sm.part_o[warp][lane * DL + d] = acc[d];
    }
    ptx::cluster_sync();
    // CTA z combines the heads w with w % splits == z (warp w of this CTA does head w)
    if (warp < nh && warp % splits == z) {
        const uint32_t pm = ptx::smem_u32(&sm.part_m[warp]);
        const uint32_t pl = ptx::smem_u32(&sm.part_l[warp]);
        const uint32_t po = ptx::smem_u32(&sm.part_o[warp][lane * DL]);
        // every split's partials are read before any is used (one remote round trip)
        float qm[8], ql[8], qo[8][DL];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            if (q < splits) {
                qm[q] = ptx::ld_dsmem_f32(ptx::map_dsmem(pm, q));
                ql[q] = ptx::ld_dsmem_f32(ptx::map_dsmem(pl, q));
#pragma unroll
                for (int d = 0; d < DL; ++d) qo[q][d] = ptx::ld_dsmem_f32(ptx::map_dsmem(po + 4 * d, q));
            }
        }
        float mx = -INFINITY;
#pragma unroll
        for (int q = 0; q < 8; ++q)
            if (q < splits) mx = fmaxf(mx, qm[q]);
        float L = 0.0f, O[DL];
#pragma unroll
        for (int d = 0; d < DL; ++d) O[d] = 0.0f;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            if (q < splits && qm[q] != -INFINITY) {  // a split without keys adds nothing
                const float w = expf(qm[q] - mx);
                L = fmaf(ql[q], w, L);
#pragma unroll
                for (int d = 0; d < DL; ++d) O[d] = fmaf(qo[q][d], w, O[d]);
            }
        }
        const float inv = __fdiv_rn(1.0f, L);
        __nv_bfloat16* o = p.O + out_row + int64_t(h0 + warp) * D + lane * DL;
#pragma unroll
        for (int d = 0; d < DL; d += 2)
            *reinterpret_cast<__nv_bfloat162*>(o + d) =
                __floats2bfloat162_rn(__fmul_rn(O[d], inv), __fmul_rn(O[d + 1], inv));
    }
    ptx::cluster_sync();  // remote shared memory must outlive its readers
}

template <int D>
cudaError_t launch_attention_d(const AttnParams& p, int splits, cudaStream_t s) {
    const size_t smem = sizeof(AttnSmem<D>);
    static bool attr_done[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !attr_done[dev]) {
        e = cudaFuncSetAttribute(attention_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) attr_done[dev] = true;
    }
    AttnParams pc = p;
    void* args[] = {&pc};
    return launch_pdl(reinterpret_cast<const void*>(attention_kernel<D>),
                      dim3(p.M, p.Hk * p.subgroups, splits), dim3(kAttnThreads), smem, s, args,
                      unsigned(splits));
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

cudaError_t launch_rope(uint16_t* x, int64_t M, int64_t n_heads, int64_t head_dim, int64_t pos0,
                        double base, cudaStream_t s) {
    RopeParams p;
    p.x = reinterpret_cast<__nv_bfloat16*>(x);
    p.pairs = M * n_heads * (head_dim / 2);
    p.pos0 = pos0;
    p.n_heads = int(n_heads);
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
    const int G = int(H / Hk);
    p.subgroups = (G + kAttnWarps - 1) / kAttnWarps;
    p.scale = scale;
    // key splits (one cluster): at least 64 keys each, at most 8 (the portable cluster size)
    const int64_t n = n0 + n1;
    int splits = 1;
    while (splits < 8 && n >= int64_t(splits) * 2 * kKeyTile) splits *= 2;
    return D == 64 ? launch_attention_d<64>(p, splits, s) : launch_attention_d<128>(p, splits, s);
}

}  // namespace emb
