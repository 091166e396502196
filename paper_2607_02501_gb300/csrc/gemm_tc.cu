// Tensor-core GEMM for the larger token counts of one closed-loop step (M = 50 action
// chunk, M = 280..816 prefix prefill): packed Q8_0/Q4_0 weights are staged in shared
// memory by TMA, dequantised by eight warps into bf16 tiles held in tensor memory, and
// fed to tcgen05 MMAs (A operand from TMEM, B from shared memory) whose fp32
// accumulators also live in TMEM.
//
// "Swap AB": the MMA's M side is 128 weight rows (output features n), its N side is the
// CTA's T tokens, so one weight tile is dequantised once for up to 256 tokens and the
// accumulator D[n][m] sits in TMEM lanes = n. The epilogue reads TMEM lane n (one
// thread per output feature) and writes Y[m][n] with 128-byte coalesced stores.
//
// TMEM (512 columns, one CTA per SM): columns 0..255 the accumulator, 256..511 the ring
// of bf16 A tiles (32 columns = 64 k per tile, two values per column, row n in lane n).
// Keeping A out of shared memory leaves shared-memory bandwidth to the X tiles (written
// by TMA, read by the MMA), which bound this kernel (measured on GB300: 100 -> 70 KB of
// shared-memory traffic per 64-k step; M = 816 prefill 683 -> 736 TFLOP/s).
//
// Roles (352 threads):
//   warp 0 lane 0 : TMA producer. Raw stages (256 codes of 128 rows + their 8 scales)
//                   are fetched before griddepcontrol.wait (weights never depend on
//                   the previous launch); X tiles (64 k x T tokens) after it.
//   warp 1        : TMEM allocation; lane 0 issues the MMAs (4 x K=16 per 64-k stage).
//                   It never waits on an mbarrier while MMAs are in flight: warp 10
//                   waits for each stage and releases it through a named barrier.
//   warps 2..9    : dequantisation (two threads per weight row, tcgen05.st into the
//                   warp's lane quarter), then the epilogue.
// Grid: x = token tile (fastest: CTAs sharing a weight tile run together), y = weight-row
// tile, z = K split. With z > 1 the splits of one output tile form a thread-block cluster
// and are summed in a fixed order through distributed shared memory (deterministic).
// Every wait is bounded (ptx::mbar_wait); on expiry the kernel records EMB_ETIMEOUT,
// lets every copy and MMA it issued land, frees TMEM and returns.
//
// Precision: each operand value is bf16(w') -- one rounding of the exact fp32 w' -- so
// the products are exact and accumulate in fp32. For K < 1024, and for layers flagged
// EMB_PRECISE_OPERAND, the SPLIT variant also stages lo = bf16(w' - bf16(w')) and issues
// a second MMA per step, which brings the operand error from 2^-8 to 2^-16 relative (the
// 1e-3 * sum|w x| bound then holds for every input, not only statistically).
#include <cuda.h>
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>

#include "ptx.cuh"

namespace emb {
namespace {

constexpr int kBN = 128;                   // weight rows per CTA (MMA M)
constexpr int kKC = 64;                    // k per A/X stage: one 128-byte bf16 atom row
constexpr int kKR = 256;                   // k per raw stage
constexpr int kStepsPerRaw = kKR / kKC;    // 4
constexpr int kRawStages = 2;
constexpr int kDeqWarps = 8;               // dequantisation (then epilogue) warps
constexpr int kWaitWarp = 2 + kDeqWarps;   // waits on the MMA warp's behalf (see the kernel)
constexpr int kThreads = 32 * (kWaitWarp + 1);
constexpr int kAccCols = 256;              // TMEM columns [0, 256): one token tile's accumulator (T <= 256)
constexpr int kACols = kKC / 2;            // TMEM columns of one bf16 A tile (two values per column)
constexpr uint32_t kTmemCols = 512;        // accumulator + A stages
constexpr int kPlane = kBN * 128;          // 16 KB: 128 rows x 128 bytes of codes
constexpr int kScaleTile = kBN * 16;       // 2 KB: 128 rows x 8 fp16 scales
constexpr int kMaxStages = 8;              // A/X ring depth, at most

struct GemmParams {
    CUtensorMap x_map;                     // X [M][K] bf16, box {64, T}, 128B swizzle
    const __nv_bfloat16* X;                // the same X (for its L2 prefetch)
    CUtensorMap codes_map[kMaxGroup];      // codes [N][row bytes] u8, box {128, 128}, 128B swizzle
    CUtensorMap scales_map[kMaxGroup];     // scales [N][ldS] u16, box {8, 128}
    CUtensorMap high_map[kMaxGroup];       // Q6_0 high bits [N][K/4] u8, box {64, 128}, no swizzle
    void* Y[kMaxGroup];                    // as the epilogue says
    int32_t N[kMaxGroup];
    int32_t tile0[kMaxGroup + 1];
    int32_t n_mats;
    int32_t M, K;
    int32_t T;                             // tokens per token tile, multiple of 16, <= 256
    int32_t P;                             // token tiles per CTA (1, or 2 sharing each A tile)
    int32_t splits;                        // K splits (cluster size along z)
    int32_t epi;                           // emb_epilogue
    int32_t stages;                        // A/X ring depth
    int32_t a_gap0;                        // P = 2: TMEM column of the first A stage after tile 0's
    int32_t a_per_gap;                     //   accumulator, and A stages per gap (see pick_stages_pair)
    uint32_t tmem_cols;
    int32_t persist;                       // 1: CTAs loop over items (no K split)
    int32_t n_tt, n_items;                 // persistent: token tiles per weight tile, items
    int32_t streamk;                       // 1: the items' raw stages split evenly over the CTAs
    int32_t slot_floats;                   // stream-K: floats of one partial tile (P * T * 128)
    float* ws_part;                        // stream-K: one partial-tile slot per CTA
    uint32_t* ws_flag;                     // stream-K: one ready flag per CTA (zero between launches)
    int* status;
};

template <int FMT>
struct RawTraits {
    static constexpr int planes = (FMT == EMB_Q8_0) ? 2 : 1;  // 128-byte code chunks per raw stage
    static constexpr int bytes = planes * kPlane;
    // Q6_0: the high bits of a raw stage, 64 bytes per row (256 codes x 2 bits)
    static constexpr int hbytes = (FMT == EMB_Q6_0) ? kBN * 64 : 0;
    // w' = d*(f - bias) where f = 2^15 + byte is built by __byte_perm
    static constexpr float bias = (FMT == EMB_Q8_0) ? 32768.0f + 128.0f
                                : (FMT == EMB_Q4_0) ? 32768.0f + 8.0f : 32768.0f + 32.0f;
};

__device__ __forceinline__ uint4 lds128(const uint8_t* p) {
    return *reinterpret_cast<const uint4*>(p);
}

// bar.sync on a named barrier with `count` threads (whole warps).
__device__ __forceinline__ void named_sync(int id, int count) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
    __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&h);
}

// Four 8-bit values b_i (the bytes of u) -> w'_i = d*(b_i - bias) exactly, as two fp32 pairs.
// __byte_perm(u, 0x47000000, 0x7504 | i<<4) is the binary32 with exponent 15 whose
// fraction holds b_i at bits 8..15, i.e. 2^15 + b_i; one FMA with (d, -bias*d) gives
// d*(b_i - bias) exactly (the product has at most 19 significant bits; bias*d at most 24).
__device__ __forceinline__ void bytes_to_w(uint32_t u, float d, float nbd, float2& w01,
                                           float2& w23) {
    const float2 dd = make_float2(d, d), oo = make_float2(nbd, nbd);
    w01 = __ffma2_rn(make_float2(__uint_as_float(__byte_perm(u, 0x47000000u, 0x7504u)),
                                 __uint_as_float(__byte_perm(u, 0x47000000u, 0x7514u))),
                     dd, oo);
    w23 = __ffma2_rn(make_float2(__uint_as_float(__byte_perm(u, 0x47000000u, 0x7524u)),
                                 __uint_as_float(__byte_perm(u, 0x47000000u, 0x7534u))),
                     dd, oo);
}

// 8 consecutive w' (two input words) -> one 16-byte chunk of bf16 (hi), and for the split
// variant the residual chunk lo = bf16(w' - hi).
template <bool SPLIT>
__device__ __forceinline__ void make_chunk(uint32_t u0, uint32_t u1, float d, float nbd,
                                           uint4& hi, uint4& lo) {
    float2 a, b, c, e;
    bytes_to_w(u0, d, nbd, a, b);
    bytes_to_w(u1, d, nbd, c, e);
    hi = make_uint4(pack_bf16(a.x, a.y), pack_bf16(b.x, b.y), pack_bf16(c.x, c.y),
                    pack_bf16(e.x, e.y));
    if constexpr (SPLIT) {
        auto res = [](float2 v, uint32_t h) {
            const float2 hv = make_float2(__uint_as_float(h << 16), __uint_as_float(h & 0xFFFF0000u));
            const float2 r = __fadd2_rn(v, make_float2(-hv.x, -hv.y));  // exact
            return pack_bf16(r.x, r.y);
        };
        lo = make_uint4(res(a, hi.x), res(b, hi.y), res(c, hi.z), res(e, hi.w));
    }
}

// TMEM column of A stage s: after the accumulator (P = 1), or in the slots after each of
// the two accumulators at columns 0 and 256 (P = 2).
template <int P, bool SPLIT>
__device__ __forceinline__ uint32_t a_stage_col(int s, int gap0, int per_gap) {
    if constexpr (P == 1) return uint32_t(kAccCols + s * (SPLIT ? 2 : 1) * kACols);
    return uint32_t(s < per_gap ? gap0 + s * kACols : kAccCols + gap0 + (s - per_gap) * kACols);
}

template <int FMT, bool SPLIT, int P, bool SK>
__global__ void __launch_bounds__(kThreads, 1) gemm_tc_kernel(const __grid_constant__ GemmParams p) {
    using RT = RawTraits<FMT>;
    static_assert(P == 1 || (P == 2 && !SPLIT), "two token tiles only without the split operand");
    static_assert(!(SK && SPLIT), "stream-K only without the split operand");
    extern __shared__ uint8_t smem_dyn[];
    uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_dyn) + 1023) &
                                               ~uintptr_t(1023));
    const int S = p.stages, T = p.T;
    uint8_t* x_ring = base;                                     // S x P x T x 128 B
    uint8_t* r_ring = x_ring + S * P * T * 128;                 // 2 x RT::bytes
    uint8_t* s_ring = r_ring + kRawStages * RT::bytes;          // 2 x 2 KB
    uint8_t* h_ring = s_ring + kRawStages * kScaleTile;          // Q6_0: 2 x 8 KB of high bits
    uint64_t* bars = reinterpret_cast<uint64_t*>(h_ring + kRawStages * RT::hbytes);
    uint64_t* raw_full = bars;
    uint64_t* raw_empty = bars + kRawStages;
    uint64_t* x_full = bars + 2 * kRawStages;
    uint64_t* a_full = x_full + S;
    uint64_t* ax_empty = a_full + S;
    uint64_t* acc_full = ax_empty + S;
    uint64_t* acc_empty = acc_full + 1;  // the epilogue warps have read the accumulator
    uint64_t* sk_full = acc_empty + 1;   // stream-K head: a chunk of a tail is in the X ring
    uint64_t* sk_free = sk_full + 1;     // stream-K head: every epilogue warp has added it
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sk_free + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    volatile int* mma_stop = abort_flag + 1;  // set by the waiter warp when a wait gave up
    int* sk_cnt = const_cast<int*>(mma_stop) + 1;  // stream-K: epilogue warps done with the tail
    int* sk_seen = sk_cnt + 1;                     // stream-K: epilogue warps done with the head
    // split-K partial tile [T][128] fp32 (token-major): reuses the X ring once every MMA
    // has completed
    float* part = reinterpret_cast<float*>(x_ring);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int M = p.M, K = p.K;
    const int splits = gridDim.z, split = blockIdx.z;
    const int nr_all = (K + kKR - 1) / kKR, nk_all = (K + kKC - 1) / kKC;
    // Work items (weight tile, token tile), each over a range of raw stages (256 k) of its
    // row. Three schedules:
    //  * one item per CTA: grid x = token tile, y = weight tile, z = K split (a cluster
    //    along z shares one item; split s takes raw stages [s*nr/splits, (s+1)*nr/splits));
    //  * p.persist: CTA c takes whole items c, c + gridDim.x, ... in the order of token
    //    tiles within weight tiles, so the CTAs at work on a weight tile at one time read it
    //    once from HBM and then from L2;
    //  * SK (stream-K): the raw stages of all items, item after item, are cut into gridDim.x
    //    equal ranges, one per CTA, so every SM gets the same work whatever the tile count.
    //    A range starts inside an item (a "tail": its sum is left in the CTA's workspace
    //    slot, flagged ready) and/or ends inside one (a "head" holding k = 0: its CTA adds
    //    the tails of the CTAs after it, in CTA order, i.e. in k order, and runs the
    //    epilogue). Results are deterministic for a given grid.
    // With more than one item, rings and barrier phases run on across items; the next
    // item's codes and activations stream in while the current one's epilogue drains the
    // accumulator.
    const bool persist = p.persist != 0;
    constexpr bool streamk = SK;  // a separate instance: the plain schedules carry none of its code
    const int64_t sk_units = int64_t(p.n_items) * nr_all;  // stream-K: raw stages of all items
    // this CTA's segments j = 0 .. n_seg-1: item it0 + j*it_stride over raw stages [r0, r1),
    // r0 = 0 but for the first, r1 = nr_all but for the last
    int it0 = 0, it_stride = 1, r0_first = 0, r1_last = nr_all, n_seg = 1;
    if (streamk) {
        const int64_t u_beg = int64_t(blockIdx.x) * sk_units / gridDim.x;
        const int64_t u_end = int64_t(blockIdx.x + 1) * sk_units / gridDim.x;
        const int64_t last = (u_end - 1) / nr_all;
        it0 = int(u_beg / nr_all);
        r0_first = int(u_beg - int64_t(it0) * nr_all);
        r1_last = int(u_end - last * nr_all);
        n_seg = u_end > u_beg ? int(last) - it0 + 1 : 0;
    } else if (persist) {
        it0 = int(blockIdx.x);
        it_stride = int(gridDim.x);
        n_seg = int(blockIdx.x) < p.n_items ? (p.n_items - int(blockIdx.x) + int(gridDim.x) - 1) / int(gridDim.x) : 0;
    } else {
        r0_first = split * nr_all / splits;
        r1_last = (split + 1) * nr_all / splits;
    }
    // stream-K: a head (last segment holding k = 0 of an item that goes on) adds the tails of
    // CTAs [blockIdx.x + 1, sk_q_end): those whose ranges start inside that item
    int sk_q_end = int(blockIdx.x) + 1;
    if (streamk && n_seg > 0 && r1_last < nr_all && (n_seg > 1 || r0_first == 0)) {
        const int64_t item_end = int64_t(it0 + n_seg) * nr_all;
        while (sk_q_end < int(gridDim.x) && int64_t(sk_q_end) * sk_units / gridDim.x < item_end) ++sk_q_end;
    }
    struct Seg {
        int it, r0, r1;  // item, raw stages [r0, r1) of its row
    };
    auto seg_at = [&](int j) {
        Seg s;
        s.it = it0 + j * it_stride;
        s.r0 = j == 0 ? r0_first : 0;
        s.r1 = j == n_seg - 1 ? r1_last : nr_all;
        return s;
    };
    auto seg_nk = [&](const Seg& s) { return min(s.r1 * kStepsPerRaw, nk_all) - s.r0 * kStepsPerRaw; };
    struct Item {
        int g, n0, m0, N;
    };
    auto item_at = [&](int it) {
        const int tt = (persist || streamk) ? it % p.n_tt : int(blockIdx.x);
        const int tile = (persist || streamk) ? it / p.n_tt : int(blockIdx.y);
        Item r;
        r.g = 0;
#pragma unroll
        for (int i = 1; i < kMaxGroup; ++i)
            if (i < p.n_mats && tile >= p.tile0[i]) r.g = i;
        r.n0 = (tile - p.tile0[r.g]) * kBN;
        r.m0 = tt * P * T;  // first token of the item's first token tile
        r.N = p.N[r.g];
        return r;
    };

    if (threadIdx.x == 0) {
        for (int i = 0; i < kRawStages; ++i) {
            ptx::mbar_init(&raw_full[i], 1);
            ptx::mbar_init(&raw_empty[i], kDeqWarps);
        }
        for (int i = 0; i < S; ++i) {
            ptx::mbar_init(&x_full[i], 1);
            ptx::mbar_init(&a_full[i], kDeqWarps);
            ptx::mbar_init(&ax_empty[i], 1);
        }
        ptx::mbar_init(acc_full, 1);
        ptx::mbar_init(acc_empty, kDeqWarps);
        ptx::mbar_init(sk_full, 1);
        ptx::mbar_init(sk_free, kDeqWarps);
        *abort_flag = 0;
        *mma_stop = 0;
        *sk_cnt = 0;
        *sk_seen = 0;
        ptx::fence_mbar_init();
        ptx::prefetch_tmap(&p.x_map);
        for (int i = 0; i < p.n_mats; ++i) {
            ptx::prefetch_tmap(&p.codes_map[i]);
            ptx::prefetch_tmap(&p.scales_map[i]);
            if constexpr (FMT == EMB_Q6_0) ptx::prefetch_tmap(&p.high_map[i]);
        }
    }
    if (warp == 1) {
        // all 512 columns: one CTA per SM (see ptx::tmem_alloc for why this never waits)
        ptx::tmem_alloc(tmem_slot, p.tmem_cols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    ptx::griddep_launch_dependents();
    int items_done = 0;  // this CTA's items started by its role (phase of acc_full / acc_empty)

    if (warp == 0) {
        if (lane == 0) {
            // ---------------------------------------------------------------- producer
            const uint64_t pol_w = ptx::policy_evict_first();
            const uint64_t pol_x = ptx::policy_evict_last();
            int raw_issued = 0, x_issued = 0;  // over all items of the CTA
            bool stop = false, waited = false;
            int rbase = 0, xbase = 0;  // raw stages and steps of the earlier segments
            for (int j = 0; j < n_seg && !stop; ++j, ++items_done) {
                const Seg sg = seg_at(j);
                const Item I = item_at(sg.it);
                const int nr = sg.r1 - sg.r0, nk = seg_nk(sg), ks0 = sg.r0 * kStepsPerRaw;
                auto issue_raw = [&](int r) {  // raw stage r of this segment (global rbase + r)
                    const int rg_all = rbase + r;
                    const int slot = rg_all % kRawStages;
                    const int rg = sg.r0 + r;  // raw stage index within the whole row
                    ptx::mbar_arrive_expect_tx(&raw_full[slot], RT::bytes + RT::hbytes + kScaleTile);
#pragma unroll
                    for (int pl = 0; pl < RT::planes; ++pl)
                        ptx::tma_load_2d(r_ring + slot * RT::bytes + pl * kPlane, &p.codes_map[I.g],
                                         &raw_full[slot], (rg * RT::planes + pl) * 128, I.n0, pol_w);
                    if constexpr (FMT == EMB_Q6_0)  // x = 64 bytes per raw stage: 16-byte aligned
                        ptx::tma_load_2d(h_ring + slot * RT::hbytes, &p.high_map[I.g], &raw_full[slot],
                                         rg * 64, I.n0, pol_w);
                    ptx::tma_load_2d(s_ring + slot * kScaleTile, &p.scales_map[I.g], &raw_full[slot],
                                     rg * (kKR / kQBlock), I.n0, pol_w);
                };
                if (!waited) {
                    // the first raw stages before griddepcontrol.wait: weights never depend on
                    // the previous launch; X may be written by it, so only its rows' way towards
                    // L2 starts now (a hint: the TMA loads after the wait read the written values)
                    for (; raw_issued < nr && raw_issued < kRawStages; ++raw_issued) issue_raw(raw_issued);
                    const int x_rows = min(M - I.m0, P * T);
                    if (x_rows > 0 && I.n0 == 0 && I.g == 0 && sg.r0 == 0)  // one CTA per token tile
                        ptx::prefetch_l2(reinterpret_cast<const uint8_t*>(p.X) + int64_t(I.m0) * K * 2,
                                         uint32_t(min(int64_t(x_rows) * K * 2, int64_t(1) << 20)));
                    ptx::griddep_wait();
                    waited = true;
                }
                for (int i = 0; i < nk; ++i) {
                    if (i % kStepsPerRaw == 0) {
                        const int rg_all = rbase + i / kStepsPerRaw;
                        if (rg_all >= raw_issued) {
                            if (rg_all >= kRawStages &&
                                !ptx::mbar_wait(&raw_empty[rg_all % kRawStages], ((rg_all / kRawStages) - 1) & 1,
                                                abort_flag, p.status, kWaitLimitNs)) {
                                stop = true;
                                break;
                            }
                            issue_raw(i / kStepsPerRaw);
                            ++raw_issued;
                        }
                    }
                    const int xs = xbase + i;
                    const int s = xs % S;
                    if (xs >= S && !ptx::mbar_wait(&ax_empty[s], ((xs / S) - 1) & 1, abort_flag, p.status,
                                                   kWaitLimitNs)) {
                        stop = true;
                        break;
                    }
                    ptx::mbar_arrive_expect_tx(&x_full[s], uint32_t(P * T) * 128u);
#pragma unroll
                    for (int q = 0; q < P; ++q)  // a tile past M reads zeros (its outputs are not stored)
                        ptx::tma_load_2d(x_ring + (s * P + q) * T * 128, &p.x_map, &x_full[s],
                                         (ks0 + i) * kKC, I.m0 + q * T, pol_x);
                    ++x_issued;
                }
                rbase += nr;
                xbase += nk;
            }
            // every issued copy must land before this CTA's shared memory can be released
            for (int r = raw_issued - 1; r >= 0 && r >= raw_issued - kRawStages; --r)
                ptx::mbar_wait(&raw_full[r % kRawStages], (r / kRawStages) & 1, nullptr, p.status,
                               kWaitLimitNs);
            for (int i = x_issued - 1; i >= 0 && i >= x_issued - S; --i)
                ptx::mbar_wait(&x_full[i % S], (i / S) & 1, nullptr, p.status, kWaitLimitNs);
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------------- MMA issuer
        // Step i is released by the waiter warp through named barrier 1; this warp itself
        // runs no mbarrier wait while MMAs are in flight (see kWaitWarp below).
        const uint32_t idesc = ptx::idesc_bf16_f32(kBN, T);
        const uint32_t x0 = ptx::smem_u32(x_ring);
        bool stop = false;
        int commits = 0;  // accumulator commits (one per finished segment)
        int xbase = 0;
        for (int j = 0; j < n_seg && !stop; ++j, ++items_done) {
            const int nk = seg_nk(seg_at(j));
            for (int i = 0; i < nk; ++i) {
                named_sync(1, 64);
                if (*mma_stop) {
                    stop = true;
                    break;
                }
                if (lane == 0) {
                    const int s = (xbase + i) % S;
                    ptx::tc_fence_after();
                    const uint32_t a_tm = tmem + a_stage_col<P, SPLIT>(s, p.a_gap0, p.a_per_gap);
#pragma unroll
                    for (int q = 0; q < P; ++q) {
                        // token tile q: its own X tile and accumulator, the same A tile
                        const uint32_t x_addr = x0 + (s * P + q) * T * 128;
                        const uint32_t d_tm = tmem + uint32_t(q * kAccCols);
#pragma unroll
                        for (int k = 0; k < kKC / 16; ++k) {
                            const uint64_t bdesc = ptx::smem_desc_sw128(x_addr + 32 * k);
                            ptx::mma_bf16_ta(d_tm, a_tm + 8 * k, bdesc, idesc, (i | k) != 0);
                            if constexpr (SPLIT) ptx::mma_bf16_ta(d_tm, a_tm + kACols + 8 * k, bdesc, idesc, 1u);
                        }
                    }
                    ptx::mma_commit(&ax_empty[s]);
                }
                __syncwarp();
            }
            // the item's accumulator is complete once every MMA issued so far has finished
            if (stop) break;
            if (lane == 0) ptx::mma_commit(acc_full);
            ++commits;
            xbase += nk;
            __syncwarp();
        }
        if (lane == 0 && commits > 0)  // the last item's MMAs finish before TMEM is freed
            ptx::mbar_wait(acc_full, (commits - 1) & 1, nullptr, p.status, kWaitLimitNs);
    } else if (warp == kWaitWarp) {
        // ---------------------------------------------------------------- waiter
        // An mbarrier wait executed by the warp that issues tcgen05 MMAs is ordered behind
        // that warp's in-flight MMAs, which drains the tensor pipe at every step (measured
        // on GB300: 104 -> 330+ cycles per 128x208x16 MMA). This warp waits for step i's
        // X tile and A tile (and, at an item's first step, for the previous item's epilogue
        // to have read the accumulator) and then releases the MMA warp through named barrier 1.
        bool stop = false;
        int xbase = 0;
        for (int j = 0; j < n_seg && !stop; ++j, ++items_done) {
            const int nk = seg_nk(seg_at(j));
            for (int i = 0; i < nk; ++i) {
                const int xs = xbase + i;
                const int s = xs % S;
                const uint32_t ph = (xs / S) & 1;
                if (lane == 0) {
                    bool ok = true;
                    if (i == 0 && items_done > 0)
                        ok = ptx::mbar_wait(acc_empty, (items_done - 1) & 1, abort_flag, p.status, kWaitLimitNs);
                    ok = ok && ptx::mbar_wait(&x_full[s], ph, abort_flag, p.status, kWaitLimitNs) &&
                         ptx::mbar_wait(&a_full[s], ph, abort_flag, p.status, kWaitLimitNs);
                    if (!ok) *mma_stop = 1;
                }
                __syncwarp();
                named_sync(1, 64);
                if (*mma_stop) {
                    stop = true;
                    break;
                }
            }
            xbase += nk;
        }
    } else if (warp < 2 + kDeqWarps) {
        // ---------------------------------------------------------------- dequant
        // two threads per weight row: thread (row t, half h) produces 32 of the 64 bf16 of
        // each 64-k step (32-block 2j+h of step j) and stores them into its TMEM lane t,
        // 16 columns; a warp reaches only its lane quarter (warp % 4), so t = 32*(warp%4) + lane
        const int t = 32 * (warp & 3) + lane, h = (warp - 2) >> 2;
        const uint32_t a_lane = tmem + (uint32_t(32 * (warp & 3)) << 16) + uint32_t(16 * h);
        const unsigned full = 0xffffffffu;
        bool ok = true;
        int rbase = 0, xbase = 0;  // raw stages and steps of the earlier segments
        for (int j = 0; j < n_seg && ok; ++j, ++items_done) {
            const Seg sg = seg_at(j);
            const Item I = item_at(sg.it);
            const int nr = sg.r1 - sg.r0, nk = seg_nk(sg);
            // Software pipeline: step i's TMEM stores are completed (tcgen05.wait::st) and
            // signalled only after step i+1 has been computed, so the store latency overlaps
            // the next step's arithmetic instead of stalling this warp every step.
            int pending = -1;  // A stage whose stores are in flight, not yet signalled
            auto signal_pending = [&]() {
                if (pending >= 0) {
                    ptx::tmem_st_wait();
                    ptx::tc_fence_before();  // the stores are ordered before the arrive
                    __syncwarp();
                    if (lane == 0) ptx::mbar_arrive(&a_full[pending]);
                    pending = -1;
                }
            };
            for (int r = 0; r < nr && ok; ++r) {
                const int rg_all = rbase + r;
                const int rs = rg_all % kRawStages;
                ok = __all_sync(full, ptx::mbar_wait(&raw_full[rs], (rg_all / kRawStages) & 1, abort_flag,
                                                     p.status, kWaitLimitNs));
                if (!ok) break;
                const uint8_t* rbase_p = r_ring + rs * RT::bytes + t * 128;
                const uint4 sv = lds128(s_ring + rs * kScaleTile + t * 16);
                const uint32_t sw[4] = {sv.x, sv.y, sv.z, sv.w};
                float d[4], nbd[4];  // scale of block 2j + h (word j, half h), j = 0..3
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const uint16_t hb = uint16_t((sw[j] >> (16 * h)) & 0xFFFFu);
                    d[j] = __half2float(__ushort_as_half(hb));
                    nbd[j] = -RT::bias * d[j];  // exact (see bytes_to_w)
                }
#pragma unroll
                for (int j = 0; j < kStepsPerRaw; ++j) {
                    const int i = r * kStepsPerRaw + j;
                    if (i >= nk) break;
                    const int xs = xbase + i;
                    const int s = xs % S;
                    const uint32_t a_dst = a_lane + a_stage_col<P, SPLIT>(s, p.a_gap0, p.a_per_gap);
                    const int sx = t & 7;  // raw codes: 16-byte chunk c of row t lives at c ^ (t & 7)
                    uint32_t va[16], vl[16];  // this thread's 16 columns of the hi (and lo) tile
                    if constexpr (FMT == EMB_Q8_0) {
                        // atom j: codes 64j..64j+63 of the raw stage = plane j/2, chunks 4(j%2)..+3;
                        // this half: chunks 4(j%2)+2h, +1 (block 2j+h) -> output chunks 4h..4h+3
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int cc = 2 * h + e;
                            const int c = (j & 1) * 4 + cc;
                            const uint4 v = lds128(rbase_p + (j >> 1) * kPlane + ((c ^ sx) << 4));
                            uint4 h0, l0, h1, l1;
                            make_chunk<SPLIT>(v.x ^ 0x80808080u, v.y ^ 0x80808080u, d[j], nbd[j], h0, l0);
                            make_chunk<SPLIT>(v.z ^ 0x80808080u, v.w ^ 0x80808080u, d[j], nbd[j], h1, l1);
                            // output chunks 2cc, 2cc+1 (k = 16cc .. 16cc+15) -> columns 8e .. 8e+7
                            const int q = 8 * e;
                            va[q + 0] = h0.x; va[q + 1] = h0.y; va[q + 2] = h0.z; va[q + 3] = h0.w;
                            va[q + 4] = h1.x; va[q + 5] = h1.y; va[q + 6] = h1.z; va[q + 7] = h1.w;
                            if constexpr (SPLIT) {
                                vl[q + 0] = l0.x; vl[q + 1] = l0.y; vl[q + 2] = l0.z; vl[q + 3] = l0.w;
                                vl[q + 4] = l1.x; vl[q + 5] = l1.y; vl[q + 6] = l1.z; vl[q + 7] = l1.w;
                            }
                        }
                    } else {
                        // atom j: blocks 2j, 2j+1; this half: block 2j+h -> output chunks 4h..4h+3.
                        // A block's byte i holds code i (low nibble) and code i+16 (high nibble).
                        const int b = 2 * j + h;
                        const uint4 v = lds128(rbase_p + ((b ^ sx) << 4));
                        const uint32_t m = 0x0F0F0F0Fu;
                        // Q4_0: the nibbles are the codes. Q6_0: OR in the high bits so that every
                        // byte holds a whole code: high word (w & 1) >> 2(w >> 1) has the high bits
                        // of low word w's codes at bits 0-1 (codes 4w+i) and 4-5 (codes 16+4w+i).
                        uint32_t c0 = v.x & m, c1 = v.y & m, c2 = v.z & m, c3 = v.w & m;
                        uint32_t e0 = (v.x >> 4) & m, e1 = (v.y >> 4) & m, e2 = (v.z >> 4) & m, e3 = (v.w >> 4) & m;
                        if constexpr (FMT == EMB_Q6_0) {
                            const uint2 hv = *reinterpret_cast<const uint2*>(h_ring + rs * RT::hbytes + t * 64 + b * 8);
                            const uint32_t hw[4] = {hv.x, hv.y, hv.x >> 2, hv.y >> 2};
                            c0 |= (hw[0] & 0x03030303u) << 4; e0 |= hw[0] & 0x30303030u;
                            c1 |= (hw[1] & 0x03030303u) << 4; e1 |= hw[1] & 0x30303030u;
                            c2 |= (hw[2] & 0x03030303u) << 4; e2 |= hw[2] & 0x30303030u;
                            c3 |= (hw[3] & 0x03030303u) << 4; e3 |= hw[3] & 0x30303030u;
                        }
                        uint4 hh[4], ll[4];
                        make_chunk<SPLIT>(c0, c1, d[j], nbd[j], hh[0], ll[0]);  // codes 0..7
                        make_chunk<SPLIT>(c2, c3, d[j], nbd[j], hh[1], ll[1]);  // 8..15
                        make_chunk<SPLIT>(e0, e1, d[j], nbd[j], hh[2], ll[2]);  // 16..23
                        make_chunk<SPLIT>(e2, e3, d[j], nbd[j], hh[3], ll[3]);  // 24..31
#pragma unroll
                        for (int q = 0; q < 4; ++q) {  // output chunk 4h+q -> columns 4q .. 4q+3
                            va[4 * q + 0] = hh[q].x; va[4 * q + 1] = hh[q].y;
                            va[4 * q + 2] = hh[q].z; va[4 * q + 3] = hh[q].w;
                            if constexpr (SPLIT) {
                                vl[4 * q + 0] = ll[q].x; vl[4 * q + 1] = ll[q].y;
                                vl[4 * q + 2] = ll[q].z; vl[4 * q + 3] = ll[q].w;
                            }
                        }
                    }
                    signal_pending();
                    if (xs >= S) {
                        ok = __all_sync(full, ptx::mbar_wait(&ax_empty[s], ((xs / S) - 1) & 1, abort_flag,
                                                             p.status, kWaitLimitNs));
                        if (!ok) break;
                        ptx::tc_fence_after();  // the MMAs that read this A stage have completed
                    }
                    ptx::tmem_st_16(a_dst, va);
                    if constexpr (SPLIT) ptx::tmem_st_16(a_dst + kACols, vl);
                    pending = s;
                }
                if (!ok) break;
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(&raw_empty[rs]);
            }
            if (ok) signal_pending();
            ptx::tmem_st_wait();  // no store of this warp is left in flight, whatever happened

            // ---------------------------------------------------------------- epilogue
            ptx::griddep_wait();  // Y may be read or written by the previous launch
            ok = __all_sync(full, ok && ptx::mbar_wait(acc_full, items_done & 1, abort_flag, p.status,
                                                       kWaitLimitNs));
            // stream-K: a tail goes to this CTA's workspace slot; a head first adds the tails of
            // the CTAs after it (those whose ranges start inside this item), in CTA order
            const bool sk_tail = streamk && sg.r0 > 0;
            const bool sk_head = streamk && sg.r0 == 0 && sg.r1 < nr_all;
            if (ok) {
                ptx::tc_fence_after();
                // warps 2..9: TMEM lane quarter = warp % 4; the two warps of a quarter split the
                // columns of one token tile, or (P = 2) take one token tile each
                const int quarter = warp & 3, half = (warp - 2) >> 2;
                const int csplit = ((T >> 1) + 15) & ~15;
                const int tt = (P == 2) ? half : 0;  // token tile read by this warp
                const int cbeg = (P == 2 || !half) ? 0 : csplit;
                const int cend = (P == 2 || half) ? T : min(csplit, T);
                const int row = quarter * 32 + lane;
                const uint32_t taddr = tmem + (uint32_t(quarter * 32) << 16) + uint32_t(tt * kAccCols);
                const int n = I.n0 + row, N = I.N;
                const int mt = I.m0 + tt * T;  // first token of that tile
                void* Y = p.Y[I.g];
                const int epi = p.epi;
                // Emit 16 accumulator columns c0 .. c0+15 of this warp's rows, plus (stream-K
                // head) the staged last tail
                const uint32_t staged = ptx::smem_u32(x_ring);  // staged tail: [cols][128] fp32
                bool add_staged = false;
                auto emit = [&](uint32_t (&v)[16], int c0) {
                    if (add_staged) {
#pragma unroll
                        for (int e = 0; e < 16; ++e)
                            v[e] = __float_as_uint(__fadd_rn(
                                __uint_as_float(v[e]), ptx::ld_shared_f32(staged + uint32_t(((tt * T + c0 + e) * kBN + row) * 4))));
                    }
                    if (splits == 1) {
                        if (epi >= EMB_EPI_GEGLU) {
                            // gate row n (even lane) and up row n + 1 (the next lane): rows past N
                            // hold zeros (their weights were read as zeros), so every lane shuffles
#pragma unroll
                            for (int e = 0; e < 16; ++e) {
                                const float up = __shfl_down_sync(0xffffffffu, __uint_as_float(v[e]), 1);
                                const int m = mt + c0 + e;
                                if ((lane & 1) == 0 && n < N && m < M)
                                    epi_store_gated(epi, Y, m, n, N, __uint_as_float(v[e]), up);
                            }
                        } else if (epi == EMB_EPI_ADD && n < N) {
                            // reads four at a time ahead of their stores: a read after a store to
                            // the same buffer would otherwise wait for that store
                            float* y = reinterpret_cast<float*>(Y);
#pragma unroll
                            for (int e0 = 0; e0 < 16; e0 += 4) {
                                float old[4];
#pragma unroll
                                for (int e = 0; e < 4; ++e)
                                    old[e] = (mt + c0 + e0 + e < M) ? y[int64_t(mt + c0 + e0 + e) * N + n] : 0.0f;
#pragma unroll
                                for (int e = 0; e < 4; ++e)
                                    if (mt + c0 + e0 + e < M)
                                        y[int64_t(mt + c0 + e0 + e) * N + n] =
                                            __fadd_rn(old[e], __uint_as_float(v[e0 + e]));
                            }
                        } else if (n < N) {
#pragma unroll
                            for (int e = 0; e < 16; ++e) {
                                const int m = mt + c0 + e;
                                if (m < M) epi_store(epi, Y, m, n, N, __uint_as_float(v[e]));
                            }
                        }
                    } else {
                        // token-major partial tile part[m][row] (a warp writes 32 consecutive rows)
#pragma unroll
                        for (int e = 0; e < 16; ++e) part[(c0 + e) * kBN + row] = __uint_as_float(v[e]);
                    }
                };
                if (sk_head) {
                    // Workspace slots are token-major [P*T][128] fp32. Each tail is staged into the
                    // (now idle) X ring by bulk copies, in column chunks that fit it. Every tail but
                    // the last is added into the accumulator in TMEM; the last one, when it fits in
                    // one chunk, is added by the store pass below.
                    const int slot_cols = P * T;
                    const int chunk_cols = min(slot_cols, ((S * P * T) / 4) & ~15);  // X ring bytes / 512
                    int chunk_no = 0;
                    for (int q = int(blockIdx.x) + 1; q < sk_q_end && ok; ++q) {
                        for (int k0 = 0; k0 < slot_cols && ok; k0 += chunk_cols, ++chunk_no) {
                            const int k1 = min(slot_cols, k0 + chunk_cols);
                            if (warp == 2 && lane == 0) {
                                bool good = true;
                                if (k0 == 0) {
                                    good = ptx::flag_wait(p.ws_flag + q, abort_flag, p.status, kWaitLimitNs);
                                    ptx::fence_proxy_async_global();  // the tail's stores, seen by the copy
                                }
                                if (good && chunk_no > 0)  // every warp has read the previous chunk
                                    good = ptx::mbar_wait(sk_free, (chunk_no - 1) & 1, abort_flag, p.status,
                                                          kWaitLimitNs);
                                if (good) {
                                    const uint32_t bytes = uint32_t(k1 - k0) * uint32_t(kBN) * 4u;
                                    ptx::mbar_arrive_expect_tx(sk_full, bytes);
                                    ptx::bulk_load(x_ring, p.ws_part + int64_t(q) * p.slot_floats + int64_t(k0) * kBN,
                                                   bytes, sk_full);
                                }
                            }
                            ok = __all_sync(full, ptx::mbar_wait(sk_full, chunk_no & 1, abort_flag, p.status,
                                                                 kWaitLimitNs));
                            if (!ok) break;
                            if (q == sk_q_end - 1 && chunk_cols == slot_cols) {
                                add_staged = true;  // the store pass adds it
                                break;
                            }
                            for (int c0 = cbeg; c0 < cend; c0 += 16) {
                                const int sc = tt * T + c0;  // slot column (chunks are whole 16-column groups)
                                if (sc < k0 || sc >= k1) continue;
                                uint32_t v[16];
                                ptx::tmem_ld_16(taddr + uint32_t(c0), v);
                                ptx::tmem_ld_wait();
#pragma unroll
                                for (int e = 0; e < 16; ++e)
                                    v[e] = __float_as_uint(__fadd_rn(
                                        __uint_as_float(v[e]), ptx::ld_shared_f32(staged + uint32_t(((sc - k0 + e) * kBN + row) * 4))));
                                ptx::tmem_st_16(taddr + uint32_t(c0), v);
                            }
                            ptx::tmem_st_wait();
                            __syncwarp();
                            if (lane == 0) ptx::mbar_arrive(sk_free);
                        }
                    }
                }
                if (sk_tail) {
                    float* slot = p.ws_part + int64_t(blockIdx.x) * p.slot_floats;
                    for (int c0 = cbeg; c0 < cend; c0 += 16) {
                        uint32_t v[16];
                        ptx::tmem_ld_16(taddr + uint32_t(c0), v);
                        ptx::tmem_ld_wait();
                        float* dst = slot + int64_t(tt * T + c0) * kBN + row;  // a warp writes 32 consecutive rows
#pragma unroll
                        for (int e = 0; e < 16; ++e) __stcg(dst + e * kBN, __uint_as_float(v[e]));
                    }
                    // the last of the eight warps to finish publishes the tail
                    __threadfence();
                    __syncwarp();
                    if (lane == 0 && atomicAdd(sk_cnt, 1) == kDeqWarps - 1) {
                        __threadfence();
                        ptx::st_release_gpu(p.ws_flag + blockIdx.x, 1u);
                    }
                } else if (ok) {
                    // one TMEM load per wait (two per wait measured slower on GB300: the kernel's
                    // register count rose by 16 and the main loop lost 10-17 %)
                    for (int c0 = cbeg; c0 < cend; c0 += 16) {
                        uint32_t v[16];
                        ptx::tmem_ld_16(taddr + uint32_t(c0), v);
                        ptx::tmem_ld_wait();
                        emit(v, c0);
                    }
                }
                if (sk_head && ok) {
                    // the last of the eight warps to finish clears the flags it consumed
                    __syncwarp();
                    if (lane == 0 && atomicAdd(sk_seen, 1) == kDeqWarps - 1)
                        for (int q = int(blockIdx.x) + 1; q < sk_q_end; ++q) ptx::st_relaxed_gpu(p.ws_flag + q, 0u);
                }
                // the accumulator may be overwritten by the next item's MMAs
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(acc_empty);
            }
            rbase += nr;
            xbase += nk;
        }
    }
    // the split-K exchange below (never persistent: one item per CTA) sums that item's tile
    const Item I_one = item_at(0);
    const int n0 = I_one.n0, m0 = I_one.m0, N = I_one.N, g = I_one.g;

    __syncwarp();  // the producer / MMA warps reconverge before the block-wide barriers
    ptx::tc_fence_before();
    if (splits > 1) {
        // split-K: every CTA of the cluster holds its partial tile; CTA s sums rows
        // [s*128/splits, (s+1)*128/splits) over the cluster in a fixed order through
        // distributed shared memory and stores them (deterministic, no global scratch)
        ptx::cluster_sync();
        if (threadIdx.x >= 64 && !*abort_flag) {
            // one thread = 4 consecutive rows of one token: 16-byte remote loads and
            // 16-byte coalesced stores to Y[m][n..n+3]
            const int rows = kBN / splits, r0 = split * rows, q4 = rows / 4;
            const uint32_t pbase = ptx::smem_u32(part);
            void* Y = p.Y[g];
            const int epi = p.epi;
            const bool vec = (N % 4) == 0;
            for (int w = threadIdx.x - 64; w < q4 * T; w += kThreads - 64) {
                const int c = w / q4, row = r0 + 4 * (w - c * q4);
                const int m = m0 + c, n = n0 + row;
                const uint32_t off = pbase + uint32_t(c * kBN + row) * 4u;
                float4 acc = ptx::ld_dsmem_f32x4(ptx::map_dsmem(off, 0));
                for (int q = 1; q < splits; ++q) {
                    const float4 v = ptx::ld_dsmem_f32x4(ptx::map_dsmem(off, q));
                    acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
                }
                if (m < M) {
                    if (vec && n + 3 < N) {
                        epi_store4(epi, Y, m, n, N, acc);
                    } else if (epi >= EMB_EPI_GEGLU) {  // rows n, n + 2 are gate rows (n % 4 == 0)
                        if (n < N) epi_store_gated(epi, Y, m, n, N, acc.x, acc.y);
                        if (n + 2 < N) epi_store_gated(epi, Y, m, n + 2, N, acc.z, acc.w);
                    } else {
                        if (n < N) epi_store(epi, Y, m, n, N, acc.x);
                        if (n + 1 < N) epi_store(epi, Y, m, n + 1, N, acc.y);
                        if (n + 2 < N) epi_store(epi, Y, m, n + 2, N, acc.z);
                        if (n + 3 < N) epi_store(epi, Y, m, n + 3, N, acc.w);
                    }
                }
            }
        }
        ptx::cluster_sync();  // remote shared memory must outlive its readers
    } else {
        __syncthreads();
    }
    if (warp == 1) {
        __syncwarp();
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, p.tmem_cols);
    }
}

// ------------------------------------------------------------------ host side

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(f);
    });
    return fn;
}

bool encode_2d(CUtensorMap* m, CUtensorMapDataType dt, const void* base, uint64_t inner,
               uint64_t outer, uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_outer,
               CUtensorMapSwizzle sw, CUtensorMapL2promotion l2) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {inner, outer};
    const cuuint64_t strides[1] = {row_stride_bytes};
    const cuuint32_t box[2] = {box_inner, box_outer};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, dt, 2, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, sw, l2, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

constexpr int kSmemLimit = 227 * 1024;

// Every CTA allocates all 512 TMEM columns, so no two may share an SM (a second one
// would block in tcgen05.alloc, and inside a split-K cluster wait on the first forever):
// the dynamic shared memory is padded above half of the SM's.
constexpr int kOneCtaPerSm = 120 * 1024;

template <int FMT, bool SPLIT>
int smem_bytes(int T, int S, int P) {
    const int need = 1024 + S * P * T * 128 +
                     kRawStages * (RawTraits<FMT>::bytes + RawTraits<FMT>::hbytes + kScaleTile) +
                     (2 * kRawStages + 3 * S + 4) * 8 + 32;
    return need > kOneCtaPerSm ? need : kOneCtaPerSm;
}

// Ring depth: as many X stages as shared memory holds, at most as many A stages as fit
// in TMEM beside the accumulator (8 single tiles or 4 hi/lo pairs).
template <int FMT, bool SPLIT>
int pick_stages(int T) {
    int S = (int(kTmemCols) - kAccCols) / ((SPLIT ? 2 : 1) * kACols);
    while (S > 2 && smem_bytes<FMT, SPLIT>(T, S, 1) > kSmemLimit) --S;
    return S;
}

// Two token tiles per CTA (P = 2): the accumulators sit at TMEM columns 0 and 256 and the
// A stages in the 32-column slots after each (so T <= 224). Returns the ring depth that
// fits TMEM and shared memory (0 if fewer than two) and fills the stages' columns.
template <int FMT>
int pick_stages_pair(int T, int& gap0, int& per_gap) {
    gap0 = int(roundup(T, 32));
    per_gap = (kAccCols - gap0) / kACols;
    int S = std::min(2 * per_gap, kMaxStages);
    while (S > 2 && smem_bytes<FMT, false>(T, S, 2) > kSmemLimit) --S;
    if (S < 2 || smem_bytes<FMT, false>(T, S, 2) > kSmemLimit) return 0;
    return S;
}

template <int FMT, bool SPLIT, int P, bool SK = false>
cudaError_t launch_kernel(const GemmParams& p, int grid_x, int grid_y, bool pdl, cudaStream_t s) {
    // grid: x = token tile (fastest, so the CTAs sharing a weight tile run together and
    // read it from L2 after the first), y = weight-row tile, z = K split (one cluster)
    const int bytes = smem_bytes<FMT, SPLIT>(p.T, p.stages, p.P);
    // the opt-in shared-memory size is a per-device function attribute
    static std::mutex mu;
    static bool done[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (dev < 0 || dev >= 64 || !done[dev]) {
            e = cudaFuncSetAttribute(gemm_tc_kernel<FMT, SPLIT, P, SK>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit);
            if (e != cudaSuccess) return e;
            if (dev >= 0 && dev < 64) done[dev] = true;
        }
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid_x, grid_y, p.splits);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = size_t(bytes);
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    int na = 0;
    if (pdl) {
        attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[na].val.programmaticStreamSerializationAllowed = 1;
        ++na;
    }
    if (p.splits > 1) {
        attr[na].id = cudaLaunchAttributeClusterDimension;
        attr[na].val.clusterDim.x = 1;
        attr[na].val.clusterDim.y = 1;
        attr[na].val.clusterDim.z = unsigned(p.splits);
        ++na;
    }
    cfg.attrs = attr;
    cfg.numAttrs = na;
    return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<FMT, SPLIT, P, SK>, p);
}

int sm_count() {
    static std::mutex mu;
    static int counts[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    std::lock_guard<std::mutex> lock(mu);
    if (!counts[dev] && cudaDeviceGetAttribute(&counts[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        counts[dev] = 0;
    return counts[dev];
}

// K splits (1, 2, 4 or 8: one cluster of CTAs per output tile, 8 being the portable
// cluster size): the count minimising a simple time model -- waves of 148 CTAs, each
// costing a fixed ~3 us plus its share of the tile's MMA work at ~11.6 TFLOP/s per SM --
// subject to every split owning at least one 256-k raw stage and the partial tile fitting
// in the CTA's A/X rings. Eight-way splits lift the M = 50 action expert 48 -> 53 TFLOP/s.
int pick_splits(int64_t tiles, int T, int64_t K, int stages, bool split_operand) {
    const int64_t nr = (K + kKR - 1) / kKR;
    const double work_us = 2.0 * kBN * T * double(K) / 11.6e12 * 1e6 * (split_operand ? 2 : 1);
    const int64_t ring = int64_t(stages) * int64_t(T) * 128;
    const int64_t part = int64_t(kBN) * T * 4;
    int best = 1;
    double best_t = 1e30;
    for (int sp = 1; sp <= 8; sp *= 2) {
        if (sp > nr || (sp > 1 && part > ring)) break;
        const int64_t ctas = tiles * sp;
        const double t = double((ctas + 147) / 148) * (3.0 + work_us / sp);
        if (t < best_t * 0.97) { best_t = t; best = sp; }
    }
    return best;
}

}  // namespace

// Q6_0's high plane ([N][K/4] bytes) needs a 16-byte row pitch for its tensor map.
bool gemm_tc_supported(const GroupRef& g) {
    return g.M >= 1 && g.M <= int64_t(65535) * 256 && g.K <= (int64_t(1) << 30) &&
           (g.fmt != EMB_Q6_0 || g.K % 64 == 0) && encode_fn() != nullptr;
}

namespace {

struct GemmPlan {
    int T = 0, S = 0, P = 1, splits = 1;
    int grid_x = 0, grid_y = 0, persist = 0, streamk = 0;
    int a_gap0 = 0, a_per_gap = 0, n_tt = 0, n_items = 0;
    size_t ws_bytes = 0;  // stream-K workspace: flags, then grid_x partial-tile slots
};

// Stream-K workspace of a plan: one 32-bit flag per CTA in the first kSkFlagBytes, then one
// partial tile (P * T tokens x 128 rows, fp32) per CTA, each slot 256-byte aligned.
constexpr int kSkFlagBytes = 4096;  // room for 1024 CTAs
size_t sk_slot_bytes(int P, int T) { return size_t(roundup(int64_t(P) * T * kBN * 4, 256)); }
size_t sk_ws_bytes(int G, int P, int T) { return kSkFlagBytes + size_t(G) * sk_slot_bytes(P, T); }

// The launch shape of one group. With streamk_ok the plan may take the stream-K schedule,
// which needs plan.ws_bytes of zero-filled workspace.
GemmPlan plan_gemm(const GroupRef& g, bool streamk_ok) {
    GemmPlan pl;
    int tiles = 0;
    for (int i = 0; i < g.n_mats; ++i) tiles += int((g.mats[i].N + kBN - 1) / kBN);
    // one token tile per CTA: balanced tiles of at most 256, rounded up to the MMA's N granule
    int64_t t_tiles = (g.M + 255) / 256;
    int T = int(roundup((g.M + t_tiles - 1) / t_tiles, 16));
    const bool split = g.K < 1024 || g.precise;
    int S = g.fmt == EMB_Q8_0   ? (split ? pick_stages<EMB_Q8_0, true>(T) : pick_stages<EMB_Q8_0, false>(T))
            : g.fmt == EMB_Q4_0 ? (split ? pick_stages<EMB_Q4_0, true>(T) : pick_stages<EMB_Q4_0, false>(T))
                                : (split ? pick_stages<EMB_Q6_0, true>(T) : pick_stages<EMB_Q6_0, false>(T));
    int splits = pick_splits(int64_t(t_tiles) * tiles, T, g.K, S, split);
    // Prefill shapes whose weight tiles x token tiles leave SMs idle (narrow layers: the
    // vision tower's 1152-wide ones give 9-36 weight tiles) may take more, smaller token
    // tiles: per the cycle model below (per 64-k step the larger of the dequantisation,
    // ~1050 cycles, and the MMA work, ~5.2 cycles per token; ~3900 per CTA; times the
    // waves), up to three more tiles when that is at least 3 % faster. ViT M = 768: four
    // tiles of 192 instead of three of 256 (qkv 81 -> 108 CTAs, fc1 108 -> 144).
    if (!split && g.M >= 256) {
        const int sms = sm_count();
        if (sms > 0) {
            const double nk = double((g.K + kKC - 1) / kKC);
            auto cost = [&](int64_t tt, int Tc, int sp) {
                return double((tt * tiles * sp + sms - 1) / sms) *
                       (std::ceil(nk / sp) * std::max(1050.0, 5.2 * Tc) + 3900.0);
            };
            double best = cost(t_tiles, T, splits);
            const int64_t t0 = t_tiles;
            for (int64_t tt = t0 + 1; tt <= t0 + 3; ++tt) {
                const int Tc = int(roundup((g.M + tt - 1) / tt, 16));
                if (Tc < 64) break;
                const int Sc = g.fmt == EMB_Q8_0 ? pick_stages<EMB_Q8_0, false>(Tc)
                               : g.fmt == EMB_Q4_0 ? pick_stages<EMB_Q4_0, false>(Tc)
                                                   : pick_stages<EMB_Q6_0, false>(Tc);
                const int spc = pick_splits(tt * tiles, Tc, g.K, Sc, false);
                const double c = cost(tt, Tc, spc);
                if (c < 0.97 * best) {
                    best = c;
                    t_tiles = tt;
                    T = Tc;
                    S = Sc;
                    splits = spc;
                }
            }
        }
    }
    int P = 1, grid_x = int(t_tiles);
    // Two token tiles per CTA halve the dequantisation per token (each A tile feeds the MMAs
    // of both). Time model in cycles, fitted to GB300 measurements of both formats: per
    // 64-k step the larger of the dequantisation (~1050) and the MMA work (~5.2 per token
    // of the CTA), plus ~3900 of pipeline fill and drain per CTA, times the waves of CTAs
    // over the SMs. Pairs win where one tile per CTA is dequantisation-bound (T <= ~200)
    // and the pairs do not add a wave: Llama-7B qkv at M = 280, 455 -> 678 TFLOP/s; gate/up
    // 547 -> 610. At M = 816 (T = 208) one tile per CTA is already MMA-bound and pairs lose
    // (847 -> 772); narrow layers keep one tile per CTA and split K instead.
    if (!split && t_tiles >= 2) {
        const int64_t t2 = 2 * ((g.M + 447) / 448);  // even count of tiles of at most 224
        const int T2 = int(roundup((g.M + t2 - 1) / t2, 16));
        int gap0 = 0, per_gap = 0;
        const int S2 = (g.fmt == EMB_Q8_0)   ? pick_stages_pair<EMB_Q8_0>(T2, gap0, per_gap)
                       : (g.fmt == EMB_Q4_0) ? pick_stages_pair<EMB_Q4_0>(T2, gap0, per_gap)
                                             : pick_stages_pair<EMB_Q6_0>(T2, gap0, per_gap);
        const int sms = sm_count();
        if (S2 >= 2 && T2 <= 224 && sms > 0) {
            const double nk = double((g.K + kKC - 1) / kKC);
            auto waves = [&](int64_t ctas) { return double((ctas + sms - 1) / sms); };
            const double c1 = waves(int64_t(t_tiles) * tiles * splits) *
                              (std::ceil(nk / splits) * std::max(1050.0, 5.2 * T) + 3900.0);
            const double c2 = waves(int64_t(t2 / 2) * tiles) * (nk * std::max(1050.0, 5.2 * 2 * T2) + 3900.0);
            if (c2 < 0.95 * c1) {
                P = 2;
                T = T2;
                S = S2;
                splits = 1;
                grid_x = int(t2 / 2);
                pl.a_gap0 = gap0;
                pl.a_per_gap = per_gap;
            }
        }
    }
    // More items (weight tile x token tile) than SMs with one tile per CTA and no K split:
    // persistent CTAs, one per SM, each looping over items (barriers, TMEM and the first
    // copies' latency paid once per CTA; the next item's copies overlap this one's epilogue).
    int grid_y = tiles, persist = 0;
    {
        const int sms = sm_count();
        const int64_t items = int64_t(grid_x) * tiles;
        if (P == 1 && splits == 1 && sms > 0 && items > sms && items < (int64_t(1) << 30)) {
            persist = 1;
            pl.n_tt = grid_x;
            pl.n_items = int32_t(items);
            grid_x = sms;
            grid_y = 1;
        }
    }
    pl.T = T;
    pl.S = S;
    pl.P = P;
    pl.splits = splits;
    pl.grid_x = grid_x;
    pl.grid_y = grid_y;
    pl.persist = persist;
    // Stream-K: when the waves of whole items leave SMs idle (a last wave that is mostly
    // empty), cut the raw stages of all items into one equal range per SM. Both plans are
    // costed with per 64-k step max(900, 4.1 per token of the CTA) cycles (measured on
    // GB300: 922 at one tile of 208, 1170 at two of 144) plus ~3900 of fill per CTA (and
    // ~5000 for a K split's cluster exchange); stream-K adds ~17000 for writing, publishing,
    // staging and adding a partial tile and ~3300 for every further tail a head adds
    // (per-CTA %globaltimer stamps: 147 KB written in ~3 us, staged and added in ~1.7 us, a
    // slower store pass after it). So it is taken only where it is clearly faster (10 %):
    // Llama-7B gate/up at M = 280, 172 tiles on 152 SMs, 84 -> 61 us; the q/k/v, o and down
    // projections, whose tiles fill more of the SMs, gain nothing or lose.
    const int sms = sm_count();
    if (streamk_ok && !split && g.M >= 128 && sms > 0) {
        const int64_t nr_all = (g.K + kKR - 1) / kKR;
        const double nk = double((g.K + kKC - 1) / kKC);
        auto step = [](int Pc, int Tc) { return std::max(900.0, 4.1 * Pc * Tc); };
        double cur;
        if (pl.persist)
            cur = double((int64_t(pl.n_items) + sms - 1) / sms) * nk * step(P, T) + 3900.0;
        else
            cur = double((int64_t(grid_x) * grid_y * splits + sms - 1) / sms) *
                  (std::ceil(nk / splits) * step(P, T) + 3900.0 + (splits > 1 ? 5000.0 : 0.0));
        struct Cand { int P, T, S, gap0, per_gap; int64_t n_tt; };
        Cand cands[2];
        int nc = 0;
        {
            const int64_t tt1 = (g.M + 255) / 256;
            const int T1 = int(roundup((g.M + tt1 - 1) / tt1, 16));
            const int S1 = g.fmt == EMB_Q8_0   ? pick_stages<EMB_Q8_0, false>(T1)
                           : g.fmt == EMB_Q4_0 ? pick_stages<EMB_Q4_0, false>(T1)
                                               : pick_stages<EMB_Q6_0, false>(T1);
            cands[nc++] = Cand{1, T1, S1, 0, 0, tt1};
            const int64_t t2 = 2 * ((g.M + 447) / 448);
            const int T2 = int(roundup((g.M + t2 - 1) / t2, 16));
            int gap0 = 0, per_gap = 0;
            const int S2 = g.fmt == EMB_Q8_0   ? pick_stages_pair<EMB_Q8_0>(T2, gap0, per_gap)
                           : g.fmt == EMB_Q4_0 ? pick_stages_pair<EMB_Q4_0>(T2, gap0, per_gap)
                                               : pick_stages_pair<EMB_Q6_0>(T2, gap0, per_gap);
            if (S2 >= 2 && T2 <= 224) cands[nc++] = Cand{2, T2, S2, gap0, per_gap, t2 / 2};
        }
        double best = cur / 1.1;
        for (int c = 0; c < nc; ++c) {
            const Cand& cd = cands[c];
            const int64_t items = cd.n_tt * tiles;
            const int64_t U = items * nr_all;
            if (items >= (int64_t(1) << 30) || U >= (int64_t(1) << 31)) continue;
            const int64_t G = std::min<int64_t>(std::min(sms, kSkFlagBytes / 4), U);
            // a head adds the tails of the CTAs whose ranges start inside its item
            const int64_t per = std::max<int64_t>(1, U / G);
            const double tails = double(std::max<int64_t>(1, (nr_all + per - 1) / per));
            const double t = double((U + G - 1) / G) * kStepsPerRaw * step(cd.P, cd.T) + 3900.0 + 17000.0 +
                             3300.0 * (tails - 1.0);
            if (t < best) {
                best = t;
                pl.T = cd.T;
                pl.S = cd.S;
                pl.P = cd.P;
                pl.a_gap0 = cd.gap0;
                pl.a_per_gap = cd.per_gap;
                pl.splits = 1;
                pl.persist = 1;
                pl.streamk = 1;
                pl.n_tt = int(cd.n_tt);
                pl.n_items = int(items);
                pl.grid_x = int(G);
                pl.grid_y = 1;
                pl.ws_bytes = sk_ws_bytes(int(G), cd.P, cd.T);
            }
        }
    }
    return pl;
}

cudaError_t launch_plan(const GroupRef& g, const GemmPlan& pl, bool pdl, int* status, cudaStream_t s) {
    GemmParams p;
    memset(&p, 0, sizeof(p));
    const int T = pl.T, S = pl.S, P = pl.P, splits = pl.splits, grid_x = pl.grid_x, grid_y = pl.grid_y;
    const bool split = g.K < 1024 || g.precise;
    p.persist = pl.persist;
    p.streamk = pl.streamk;
    p.n_tt = pl.n_tt;
    p.n_items = pl.n_items;
    p.a_gap0 = pl.a_gap0;
    p.a_per_gap = pl.a_per_gap;
    if (pl.streamk) {
        p.slot_floats = int32_t(sk_slot_bytes(P, T) / 4);
        p.ws_flag = static_cast<uint32_t*>(g.ws);
        p.ws_part = reinterpret_cast<float*>(static_cast<uint8_t*>(g.ws) + kSkFlagBytes);
    }
    int tiles = 0;
    if (!encode_2d(&p.x_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, g.X, uint64_t(g.K), uint64_t(g.M),
                   uint64_t(g.K) * 2, kKC, uint32_t(T), CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_128B))
        return cudaErrorInvalidValue;
    tiles = 0;
    for (int i = 0; i < g.n_mats; ++i) {
        const MatRef& mr = g.mats[i];
        const uint64_t row_bytes = g.fmt == EMB_Q8_0 ? uint64_t(g.K) : uint64_t(g.K) / 2;
        if (!encode_2d(&p.codes_map[i], CU_TENSOR_MAP_DATA_TYPE_UINT8, mr.codes, row_bytes,
                       uint64_t(mr.N), row_bytes, 128, kBN, CU_TENSOR_MAP_SWIZZLE_128B,
                       CU_TENSOR_MAP_L2_PROMOTION_L2_256B))
            return cudaErrorInvalidValue;
        if (!encode_2d(&p.scales_map[i], CU_TENSOR_MAP_DATA_TYPE_UINT16, mr.scales,
                       uint64_t(g.ldS), uint64_t(mr.N), uint64_t(g.ldS) * 2, 8, kBN,
                       CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B))
            return cudaErrorInvalidValue;
        if (g.fmt == EMB_Q6_0 &&
            !encode_2d(&p.high_map[i], CU_TENSOR_MAP_DATA_TYPE_UINT8, mr.high, uint64_t(g.K) / 4,
                       uint64_t(mr.N), uint64_t(g.K) / 4, 64, kBN, CU_TENSOR_MAP_SWIZZLE_NONE,
                       CU_TENSOR_MAP_L2_PROMOTION_L2_256B))
            return cudaErrorInvalidValue;
        p.Y[i] = mr.Y;
        p.N[i] = int32_t(mr.N);
        p.tile0[i] = tiles;
        tiles += int((mr.N + kBN - 1) / kBN);
    }
    p.tile0[g.n_mats] = tiles;
    p.n_mats = g.n_mats;
    p.M = int32_t(g.M);
    p.K = int32_t(g.K);
    p.X = g.X;
    p.T = T;
    p.P = P;
    p.stages = S;
    p.splits = splits;
    p.epi = g.epi;
    p.tmem_cols = kTmemCols;
    p.status = status;
    if (pl.streamk) {
        if (g.fmt == EMB_Q8_0)
            return P == 2 ? launch_kernel<EMB_Q8_0, false, 2, true>(p, grid_x, grid_y, pdl, s)
                          : launch_kernel<EMB_Q8_0, false, 1, true>(p, grid_x, grid_y, pdl, s);
        if (g.fmt == EMB_Q4_0)
            return P == 2 ? launch_kernel<EMB_Q4_0, false, 2, true>(p, grid_x, grid_y, pdl, s)
                          : launch_kernel<EMB_Q4_0, false, 1, true>(p, grid_x, grid_y, pdl, s);
        return P == 2 ? launch_kernel<EMB_Q6_0, false, 2, true>(p, grid_x, grid_y, pdl, s)
                      : launch_kernel<EMB_Q6_0, false, 1, true>(p, grid_x, grid_y, pdl, s);
    }
    if (g.fmt == EMB_Q8_0)
        return split    ? launch_kernel<EMB_Q8_0, true, 1>(p, grid_x, grid_y, pdl, s)
               : P == 2 ? launch_kernel<EMB_Q8_0, false, 2>(p, grid_x, grid_y, pdl, s)
                        : launch_kernel<EMB_Q8_0, false, 1>(p, grid_x, grid_y, pdl, s);
    if (g.fmt == EMB_Q4_0)
        return split    ? launch_kernel<EMB_Q4_0, true, 1>(p, grid_x, grid_y, pdl, s)
               : P == 2 ? launch_kernel<EMB_Q4_0, false, 2>(p, grid_x, grid_y, pdl, s)
                        : launch_kernel<EMB_Q4_0, false, 1>(p, grid_x, grid_y, pdl, s);
    return split    ? launch_kernel<EMB_Q6_0, true, 1>(p, grid_x, grid_y, pdl, s)
           : P == 2 ? launch_kernel<EMB_Q6_0, false, 2>(p, grid_x, grid_y, pdl, s)
                    : launch_kernel<EMB_Q6_0, false, 1>(p, grid_x, grid_y, pdl, s);
}

}  // namespace

size_t gemm_tc_workspace(const GroupRef& g) {
    if (!gemm_tc_supported(g)) return 0;
    return plan_gemm(g, true).ws_bytes;
}

// The stream-K schedule runs only with a caller workspace large enough for it (its size
// is what gemm_tc_workspace reports); without one the group takes the plan without it.
cudaError_t launch_gemm_tc(const GroupRef& g, bool pdl, int* status, cudaStream_t s) {
    GemmPlan pl = plan_gemm(g, g.ws != nullptr);
    if (pl.streamk && g.ws_bytes < pl.ws_bytes) pl = plan_gemm(g, false);
    return launch_plan(g, pl, pdl, status, s);
}

}  // namespace emb
