// C ABI of libembqmm.so (declarations and contracts in include/emb_qmm.h).
//
// This file holds the host side of the library boundary: argument validation (every
// error is reported before anything is enqueued), dispatch by token count between the
// weight-streaming GEMV and the tcgen05 GEMM, fusion of consecutive layers that read the
// same activation, programmatic dependent launch between the launches of one layer
// chain (the paper's latency-first fused execution, Section 3.2, design principle 2),
// and the device status word that bounded device-side waits report into.
#include <algorithm>
#include <cmath>
#include <mutex>
#include <vector>

#include "ptx.cuh"

namespace emb {
namespace {

__device__ int g_status_word;  // OR of kStatus* flags; read and cleared by emb_device_status
__device__ int g_status_read;  // where emb_device_status's exchange leaves the value it read
// emb_qlayer_seq_noalloc's workspace: the library's own, zero at module load (4 KB of
// flags, then the partial tiles of one stream-K launch: room for ~190 SMs at the largest tile)
constexpr size_t kScratchBytes = size_t(48) << 20;
__device__ __align__(256) unsigned char g_scratch[kScratchBytes];

// Token counts up to this run the GEMV; above it, the tensor-core GEMM.
constexpr int64_t kGemvMaxM = 4;

int* status_ptr() {
    static std::mutex mu;
    static int* ptrs[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!ptrs[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
        ptrs[dev] = static_cast<int*>(p);
    }
    return ptrs[dev];
}

void* scratch_ptr() {
    static std::mutex mu;
    static void* ptrs[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!ptrs[dev] && cudaGetSymbolAddress(&ptrs[dev], g_scratch) != cudaSuccess) ptrs[dev] = nullptr;
    return ptrs[dev];
}

int* status_read_ptr() {
    static std::mutex mu;
    static int* ptrs[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!ptrs[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status_read) != cudaSuccess) return nullptr;
        ptrs[dev] = static_cast<int*>(p);
    }
    return ptrs[dev];
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

struct Range {
    uintptr_t lo, hi;  // [lo, hi)
};
bool overlap(Range a, Range b) { return a.lo < b.hi && b.lo < a.hi; }

bool valid_fmt(int fmt) { return fmt == EMB_Q8_0 || fmt == EMB_Q4_0 || fmt == EMB_Q6_0; }

bool valid_shape(int64_t M, int64_t N, int64_t K) {
    return M >= 1 && N >= 1 && K >= kQBlock && K % kQBlock == 0 && M < (int64_t(1) << 31) &&
           N < (int64_t(1) << 31) && K < (int64_t(1) << 30) && N * K < (int64_t(1) << 46) &&
           M * K < (int64_t(1) << 46) && M * N < (int64_t(1) << 46);
}

emb_status from_cuda(cudaError_t e) { return e == cudaSuccess ? EMB_OK : EMB_ECUDA; }

// An emb_qlayer.epilogue value: an emb_epilogue kind, optionally | EMB_PRECISE_OPERAND.
int epi_kind(int epi) { return epi & ~EMB_PRECISE_OPERAND; }
bool epi_precise(int epi) { return (epi & EMB_PRECISE_OPERAND) != 0; }
bool valid_epi(int epi) { return epi_kind(epi) >= EMB_EPI_F32 && epi_kind(epi) <= EMB_EPI_SWIGLU; }

// Bytes a layer's epilogue writes (and, for EMB_EPI_ADD, reads) at Y.
int64_t y_bytes(int epi, int64_t M, int64_t N) {
    epi = epi_kind(epi);
    if (epi == EMB_EPI_F32 || epi == EMB_EPI_ADD) return M * N * 4;
    if (epi == EMB_EPI_BF16) return M * N * 2;
    return M * (N / 2) * 2;  // gated: one bf16 per gate/up row pair
}

// Validation shared by emb_qmatmul and every layer of emb_qlayer_seq.
emb_status check_layer(int fmt, int epi, const void* W, const uint16_t* X, const void* Y, int64_t M,
                       int64_t N, int64_t K) {
    if (!valid_fmt(fmt) || !valid_epi(epi) || !valid_shape(M, N, K)) return EMB_EINVAL;
    if (epi_kind(epi) >= EMB_EPI_GEGLU && N % 2 != 0) return EMB_EINVAL;
    if (!W || !X || !Y) return EMB_EINVAL;
    if (!aligned(W, 256) || !aligned(X, 16) || !aligned(Y, 16)) return EMB_EALIGN;
    const Layout L = layout_of(fmt, N, K);
    const Range rw{uintptr_t(W), uintptr_t(W) + uintptr_t(L.total)};
    const Range rx{uintptr_t(X), uintptr_t(X) + uintptr_t(M * K * 2)};
    const Range ry{uintptr_t(Y), uintptr_t(Y) + uintptr_t(y_bytes(epi, M, N))};
    if (overlap(ry, rw) || overlap(ry, rx)) return EMB_EINVAL;
    return EMB_OK;
}

MatRef mat_ref(int fmt, const void* W, void* Y, int64_t N, int64_t K) {
    const Layout L = layout_of(fmt, N, K);
    const uint8_t* base = static_cast<const uint8_t*>(W);
    return MatRef{base, reinterpret_cast<const __half*>(base + L.scales_off), Y, N,
                  fmt == EMB_Q6_0 ? base + L.high_off : nullptr};
}

cudaError_t launch_group(const GroupRef& g, bool pdl, cudaStream_t s) {
    int* st = status_ptr();
    if (!st) return cudaErrorInvalidDevice;
    if (g.M <= kGemvMaxM) return launch_gemv(g, pdl, st, s);
    return launch_gemm_tc(g, pdl, st, s);
}

// Read and clear the status word in one atomic step, on the caller's stream: a flag that a
// kernel ORs in concurrently is either returned now or kept for the next read.
__global__ void status_exchange_kernel(int* status, int* out) { *out = atomicExch(status, 0); }

// ------------------------------------------------------------ self-test kernel
__global__ void selftest_wait_kernel(uint64_t timeout_ns, int* status) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        ptx::mbar_init(&bar, 1);
        ptx::fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        // nothing ever arrives on `bar`: the bounded wait must give up and report
        ptx::mbar_wait(&bar, 0, nullptr, status, timeout_ns);
    }
}

}  // namespace

cudaError_t launch_selftest_wait(uint64_t timeout_ns, int* status, cudaStream_t s) {
    selftest_wait_kernel<<<1, 32, 0, s>>>(timeout_ns, status);
    return cudaGetLastError();
}

}  // namespace emb

using namespace emb;

extern "C" {

size_t emb_qweight_bytes(emb_qfmt fmt, int64_t N, int64_t K) {
    if (!valid_fmt(fmt) || !valid_shape(1, N, K)) return 0;
    return size_t(layout_of(fmt, N, K).total);
}

static emb_status quantize_common(int fmt, const float* W, int64_t N, int64_t K, void* out,
                                  emb_stream_t stream) {
    if (!valid_shape(1, N, K) || !W || !out) return EMB_EINVAL;
    if (!aligned(W, 16) || !aligned(out, 256)) return EMB_EALIGN;
    const Layout L = layout_of(fmt, N, K);
    if (overlap(Range{uintptr_t(W), uintptr_t(W) + uintptr_t(N * K * 4)},
                Range{uintptr_t(out), uintptr_t(out) + uintptr_t(L.total)}))
        return EMB_EINVAL;
    return from_cuda(launch_quantize(fmt, W, N, K, out, reinterpret_cast<cudaStream_t>(stream)));
}

emb_status emb_quantize_q8_0(const float* W, int64_t N, int64_t K, void* W_blocks,
                             emb_stream_t stream) {
    return quantize_common(EMB_Q8_0, W, N, K, W_blocks, stream);
}

emb_status emb_quantize_q4_0(const float* W, int64_t N, int64_t K, void* W_blocks,
                             emb_stream_t stream) {
    return quantize_common(EMB_Q4_0, W, N, K, W_blocks, stream);
}

emb_status emb_quantize_q6_0(const float* W, int64_t N, int64_t K, void* W_blocks,
                             emb_stream_t stream) {
    return quantize_common(EMB_Q6_0, W, N, K, W_blocks, stream);
}

emb_status emb_qmatmul(emb_qfmt fmt, const void* W_blocks, const uint16_t* X, float* Y, int64_t M,
                       int64_t N, int64_t K, emb_stream_t stream) {
    const emb_status st = check_layer(fmt, EMB_EPI_F32, W_blocks, X, Y, M, N, K);
    if (st != EMB_OK) return st;
    GroupRef g = {};
    g.fmt = fmt;
    g.epi = EMB_EPI_F32;
    g.n_mats = 1;
    g.mats[0] = mat_ref(fmt, W_blocks, Y, N, K);
    g.X = reinterpret_cast<const __nv_bfloat16*>(X);
    g.M = M;
    g.K = K;
    g.ldS = layout_of(fmt, N, K).ldS;
    if (M > kGemvMaxM && !gemm_tc_supported(g)) return EMB_EUNSUPPORTED;
    return from_cuda(launch_group(g, false, reinterpret_cast<cudaStream_t>(stream)));
}

static Range y_range_of(const emb_qlayer& L, int64_t M) {
    return Range{uintptr_t(L.Y), uintptr_t(L.Y) + uintptr_t(y_bytes(L.epilogue, M, L.N))};
}

// Group consecutive layers that read the same X with the same format, K and epilogue,
// when no member's Y overlaps another member's W or Y (they then run in one launch).
static std::vector<std::pair<int, int>> plan_groups(const emb_qlayer* layers, int n, int64_t M) {
    std::vector<std::pair<int, int>> groups;  // [first, last)
    auto y_range = [&](int b) { return y_range_of(layers[b], M); };
    auto w_range = [&](int a) {
        const Layout La = layout_of(layers[a].fmt, layers[a].N, layers[a].K);
        return Range{uintptr_t(layers[a].W_blocks), uintptr_t(layers[a].W_blocks) + uintptr_t(La.total)};
    };
    int i = 0;
    while (i < n) {
        int j = i + 1;
        while (j < n && j - i < kMaxGroup && layers[j].X == layers[i].X &&
               layers[j].fmt == layers[i].fmt && layers[j].K == layers[i].K &&
               layers[j].epilogue == layers[i].epilogue) {
            bool clash = false;
            for (int a = i; a <= j && !clash; ++a)
                for (int b = i; b <= j && !clash; ++b)
                    if (a != b && (overlap(y_range(b), w_range(a)) || overlap(y_range(b), y_range(a))))
                        clash = true;
            if (clash) break;
            ++j;
        }
        groups.emplace_back(i, j);
        i = j;
    }
    return groups;
}

static emb_status check_seq(const emb_qlayer* layers, int n_layers, int64_t M) {
    if (!layers || n_layers < 1 || n_layers > EMB_MAX_LAYERS || M < 1) return EMB_EINVAL;
    for (int j = 0; j < n_layers; ++j) {
        const emb_qlayer& L = layers[j];
        const emb_status st = check_layer(L.fmt, L.epilogue, L.W_blocks, L.X, L.Y, M, L.N, L.K);
        if (st != EMB_OK) return st;
    }
    // a layer's weights may not be written by the same or an earlier layer: every launch
    // fetches its weights before waiting for the previous one. X may be an earlier layer's
    // output (read after that layer's launch has completed).
    for (int j = 0; j < n_layers; ++j) {
        const emb_qlayer& Lj = layers[j];
        const Range wj{uintptr_t(Lj.W_blocks),
                       uintptr_t(Lj.W_blocks) + uintptr_t(layout_of(Lj.fmt, Lj.N, Lj.K).total)};
        for (int i = 0; i < j; ++i)
            if (overlap(y_range_of(layers[i], M), wj)) return EMB_EINVAL;
    }
    return EMB_OK;
}

// Validation of one chain and its launch groups (nothing enqueued).
static emb_status prepare_seq(const emb_qlayer* layers, int n_layers, int64_t M,
                              std::vector<GroupRef>& refs) {
    const emb_status st = check_seq(layers, n_layers, M);
    if (st != EMB_OK) return st;
    const auto groups = plan_groups(layers, n_layers, M);
    refs.clear();
    refs.reserve(groups.size());
    for (const auto& gr : groups) {
        const emb_qlayer& L0 = layers[gr.first];
        GroupRef g = {};
        g.fmt = L0.fmt;
        g.epi = epi_kind(L0.epilogue);
        g.precise = epi_precise(L0.epilogue);
        g.n_mats = gr.second - gr.first;
        for (int k = 0; k < g.n_mats; ++k) {
            const emb_qlayer& L = layers[gr.first + k];
            g.mats[k] = mat_ref(L.fmt, L.W_blocks, L.Y, L.N, L.K);
        }
        g.X = reinterpret_cast<const __nv_bfloat16*>(L0.X);
        g.M = M;
        g.K = L0.K;
        g.ldS = layout_of(L0.fmt, 1, L0.K).ldS;
        if (M > kGemvMaxM && !gemm_tc_supported(g)) return EMB_EUNSUPPORTED;
        refs.push_back(g);
    }
    return EMB_OK;
}

size_t emb_qlayer_seq_workspace(const emb_qlayer* layers, int n_layers, int64_t M) {
    if (check_seq(layers, n_layers, M) != EMB_OK) return size_t(-1);
    std::vector<GroupRef> refs;
    if (prepare_seq(layers, n_layers, M, refs) != EMB_OK) return 0;  // unsupported here: the call fails anyway
    size_t need = 0;
    if (M > kGemvMaxM)
        for (const GroupRef& g : refs) need = std::max(need, gemm_tc_workspace(g));
    return need;
}

// The workspace of a chain: NULL (schedules that need none), else 256-byte aligned and at
// least emb_qlayer_seq_workspace() bytes; every group of the chain uses it in turn.
static emb_status attach_workspace(std::vector<GroupRef>& refs, int64_t M, void* workspace, size_t ws_bytes) {
    if (!workspace) return EMB_OK;
    if (!aligned(workspace, 256)) return EMB_EALIGN;
    size_t need = 0;
    if (M > kGemvMaxM)
        for (const GroupRef& g : refs) need = std::max(need, gemm_tc_workspace(g));
    if (ws_bytes < need) return EMB_ENOSPC;
    for (GroupRef& g : refs) {
        g.ws = workspace;
        g.ws_bytes = ws_bytes;
    }
    return EMB_OK;
}

static emb_status enqueue_seq(const std::vector<GroupRef>& refs, cudaStream_t s, bool first_pdl) {
    for (size_t i = 0; i < refs.size(); ++i) {
        // the first launch must not overlap whatever the caller enqueued before (it may
        // have produced the weights) unless the caller says it did not; later ones overlap
        // their weight fetch with the previous launch of this chain
        const cudaError_t e = launch_group(refs[i], i > 0 || first_pdl, s);
        if (e != cudaSuccess) return EMB_ECUDA;
    }
    return EMB_OK;
}

emb_status emb_qlayer_seq(const emb_qlayer* layers, int n_layers, int64_t M, void* workspace,
                          size_t ws_bytes, emb_stream_t stream) {
    std::vector<GroupRef> refs;
    emb_status st = prepare_seq(layers, n_layers, M, refs);
    if (st != EMB_OK) return st;
    st = attach_workspace(refs, M, workspace, ws_bytes);
    if (st != EMB_OK) return st;
    return enqueue_seq(refs, reinterpret_cast<cudaStream_t>(stream), false);
}

emb_status emb_qlayer_seq_chained(const emb_qlayer* layers, int n_layers, int64_t M,
                                  emb_stream_t stream) {
    std::vector<GroupRef> refs;
    const emb_status st = prepare_seq(layers, n_layers, M, refs);
    if (st != EMB_OK) return st;
    return enqueue_seq(refs, reinterpret_cast<cudaStream_t>(stream), true);
}

emb_status emb_qlayer_seq_noalloc(const emb_qlayer* layers, int n_layers, int64_t M,
                                  emb_stream_t stream) {
    std::vector<GroupRef> refs;
    emb_status st = prepare_seq(layers, n_layers, M, refs);
    if (st != EMB_OK) return st;
    size_t need = 0;
    if (M > kGemvMaxM)
        for (const GroupRef& g : refs) need = std::max(need, gemm_tc_workspace(g));
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (need > 0 && need <= kScratchBytes) {
        void* ws = scratch_ptr();
        if (!ws) return EMB_ECUDA;
        // the flags start at zero whatever an earlier call left (e.g. after EMB_ETIMEOUT)
        if (cudaMemsetAsync(ws, 0, 4096, s) != cudaSuccess) return EMB_ECUDA;
        st = attach_workspace(refs, M, ws, kScratchBytes);
        if (st != EMB_OK) return st;
    }
    return enqueue_seq(refs, s, false);
}

}  // extern "C"

// A recorded chain: the executable CUDA graph of one emb_qlayer_seq call.
struct emb_chain_st {
    cudaGraphExec_t exec;
};

extern "C" {

emb_status emb_chain_create(const emb_qlayer* layers, int n_layers, int64_t M, void* workspace,
                            size_t ws_bytes, emb_chain_t* chain) {
    if (!chain) return EMB_EINVAL;
    *chain = nullptr;
    std::vector<GroupRef> refs;
    emb_status st = prepare_seq(layers, n_layers, M, refs);
    if (st != EMB_OK) return st;
    st = attach_workspace(refs, M, workspace, ws_bytes);
    if (st != EMB_OK) return st;
    // capture the chain's launches on a private stream (thread-local capture mode, so other
    // threads' CUDA calls are unaffected), then instantiate the graph once
    cudaStream_t s = nullptr;
    if (cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking) != cudaSuccess) return EMB_ECUDA;
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    if (cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
        cudaStreamDestroy(s);
        return EMB_ECUDA;
    }
    st = enqueue_seq(refs, s, false);
    const cudaError_t ec = cudaStreamEndCapture(s, &graph);  // ends the capture in every case
    if (st == EMB_OK && ec != cudaSuccess) st = EMB_ECUDA;
    if (st == EMB_OK && cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess) st = EMB_ECUDA;
    if (graph) cudaGraphDestroy(graph);
    cudaStreamDestroy(s);
    if (st != EMB_OK) {
        if (exec) cudaGraphExecDestroy(exec);
        return st;
    }
    *chain = new emb_chain_st{exec};
    return EMB_OK;
}

emb_status emb_chain_launch(emb_chain_t chain, emb_stream_t stream) {
    if (!chain) return EMB_EINVAL;
    return from_cuda(cudaGraphLaunch(chain->exec, reinterpret_cast<cudaStream_t>(stream)));
}

emb_status emb_chain_destroy(emb_chain_t chain) {
    if (!chain) return EMB_OK;
    // an executable graph that is still running is freed once it completes
    const cudaError_t e = cudaGraphExecDestroy(chain->exec);
    delete chain;
    return from_cuda(e);
}

emb_status emb_chain_record_begin(emb_stream_t stream) {
    if (!stream) return EMB_EINVAL;  // the legacy default stream cannot be recorded
    return from_cuda(cudaStreamBeginCapture(reinterpret_cast<cudaStream_t>(stream),
                                            cudaStreamCaptureModeThreadLocal));
}

emb_status emb_chain_record_end(emb_stream_t stream, emb_chain_t* chain) {
    if (!stream || !chain) return EMB_EINVAL;
    *chain = nullptr;
    cudaGraph_t graph = nullptr;
    if (cudaStreamEndCapture(reinterpret_cast<cudaStream_t>(stream), &graph) != cudaSuccess || !graph) {
        if (graph) cudaGraphDestroy(graph);
        return EMB_ECUDA;
    }
    cudaGraphExec_t exec = nullptr;
    const cudaError_t e = cudaGraphInstantiate(&exec, graph, 0);
    cudaGraphDestroy(graph);
    if (e != cudaSuccess) return EMB_ECUDA;
    *chain = new emb_chain_st{exec};
    return EMB_OK;
}

emb_status emb_rmsnorm(const float* x, const float* gamma, uint16_t* y, int64_t M, int64_t D,
                       float eps, emb_stream_t stream) {
    if (!x || !gamma || !y || M < 1 || M >= (int64_t(1) << 31) || D < 8 || D % 8 != 0 ||
        D > 65536 || !(eps >= 0.0f) || !std::isfinite(eps))
        return EMB_EINVAL;
    if (!aligned(x, 16) || !aligned(gamma, 16) || !aligned(y, 16)) return EMB_EALIGN;
    const Range ry{uintptr_t(y), uintptr_t(y) + uintptr_t(M * D * 2)};
    if (overlap(ry, Range{uintptr_t(x), uintptr_t(x) + uintptr_t(M * D * 4)}) ||
        overlap(ry, Range{uintptr_t(gamma), uintptr_t(gamma) + uintptr_t(D * 4)}))
        return EMB_EINVAL;
    return from_cuda(launch_rmsnorm(x, gamma, y, M, D, eps, reinterpret_cast<cudaStream_t>(stream)));
}

emb_status emb_rope_qk(uint16_t* q, int64_t n_q_heads, uint16_t* k, int64_t n_k_heads, int64_t M,
                       int64_t head_dim, int64_t pos0, float base, emb_stream_t stream) {
    if (!q || M < 1 || n_q_heads < 1 || n_k_heads < 0 || (n_k_heads > 0 && !k) || head_dim < 2 ||
        head_dim % 2 != 0 || head_dim > 512 || pos0 < 0 || pos0 + M > (int64_t(1) << 24) ||
        M * (n_q_heads + n_k_heads) * head_dim >= (int64_t(1) << 46) || !(base > 0.0f) ||
        !std::isfinite(base))
        return EMB_EINVAL;
    if (!aligned(q, 16) || (n_k_heads > 0 && !aligned(k, 16))) return EMB_EALIGN;
    if (n_k_heads > 0 &&
        overlap(Range{uintptr_t(q), uintptr_t(q) + uintptr_t(M * n_q_heads * head_dim * 2)},
                Range{uintptr_t(k), uintptr_t(k) + uintptr_t(M * n_k_heads * head_dim * 2)}))
        return EMB_EINVAL;
    return from_cuda(launch_rope(q, n_q_heads, n_k_heads > 0 ? k : nullptr, n_k_heads, M, head_dim, pos0,
                                 double(base), reinterpret_cast<cudaStream_t>(stream)));
}

emb_status emb_rope(uint16_t* x, int64_t M, int64_t n_heads, int64_t head_dim, int64_t pos0,
                    float base, emb_stream_t stream) {
    return emb_rope_qk(x, n_heads, nullptr, 0, M, head_dim, pos0, base, stream);
}

emb_status emb_attention(const uint16_t* Q, const uint16_t* K0, const uint16_t* V0, int64_t n0,
                         const uint16_t* K1, const uint16_t* V1, int64_t n1, uint16_t* O, int64_t M,
                         int64_t n_heads, int64_t n_kv_heads, int64_t head_dim, float scale,
                         emb_stream_t stream) {
    if (!Q || !O || M < 1 || M >= (int64_t(1) << 31) || n0 < 0 || n1 < 0 || n0 + n1 < 1 ||
        n0 + n1 >= (int64_t(1) << 40) || n_heads < 1 || n_kv_heads < 1 || n_heads % n_kv_heads != 0 ||
        n_heads > 4096 || M * n_heads >= (int64_t(1) << 31) || !std::isfinite(scale))
        return EMB_EINVAL;
    if ((n0 > 0 && (!K0 || !V0)) || (n1 > 0 && (!K1 || !V1))) return EMB_EINVAL;
    if (head_dim != 64 && head_dim != 128) return EMB_EUNSUPPORTED;
    if (!aligned(Q, 16) || !aligned(O, 16) || (n0 > 0 && (!aligned(K0, 16) || !aligned(V0, 16))) ||
        (n1 > 0 && (!aligned(K1, 16) || !aligned(V1, 16))))
        return EMB_EALIGN;
    const int64_t row = n_heads * head_dim * 2, kv_row = n_kv_heads * head_dim * 2;
    const Range ro{uintptr_t(O), uintptr_t(O) + uintptr_t(M * row)};
    if (overlap(ro, Range{uintptr_t(Q), uintptr_t(Q) + uintptr_t(M * row)})) return EMB_EINVAL;
    const uint16_t* kv[4] = {K0, V0, K1, V1};
    const int64_t cnt[4] = {n0, n0, n1, n1};
    for (int i = 0; i < 4; ++i)
        if (cnt[i] > 0 && overlap(ro, Range{uintptr_t(kv[i]), uintptr_t(kv[i]) + uintptr_t(cnt[i] * kv_row)}))
            return EMB_EINVAL;
    return from_cuda(launch_attention(Q, K0, V0, n0, K1, V1, n1, O, M, n_heads, n_kv_heads, head_dim,
                                      scale, reinterpret_cast<cudaStream_t>(stream)));
}

emb_status emb_dequantize_f32(emb_qfmt fmt, const void* W_blocks, int64_t N, int64_t K,
                              float* out, emb_stream_t stream) {
    if (!valid_fmt(fmt) || !valid_shape(1, N, K) || !W_blocks || !out) return EMB_EINVAL;
    if (!aligned(W_blocks, 256) || !aligned(out, 16)) return EMB_EALIGN;
    return from_cuda(launch_dequant_f32(fmt, W_blocks, N, K, out, reinterpret_cast<cudaStream_t>(stream)));
}

emb_status emb_dequantize_bf16(emb_qfmt fmt, const void* W_blocks, int64_t N, int64_t K,
                               uint16_t* out, emb_stream_t stream) {
    if (!valid_fmt(fmt) || !valid_shape(1, N, K) || !W_blocks || !out) return EMB_EINVAL;
    if (!aligned(W_blocks, 256) || !aligned(out, 16)) return EMB_EALIGN;
    return from_cuda(launch_dequant_bf16(fmt, W_blocks, N, K, out, reinterpret_cast<cudaStream_t>(stream)));
}

emb_status emb_device_status(emb_stream_t stream) {
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    int* st = status_ptr();
    int* slot = status_read_ptr();
    if (!st || !slot) return EMB_ECUDA;
    // one read slot per device: concurrent callers take turns
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    status_exchange_kernel<<<1, 1, 0, s>>>(st, slot);
    if (cudaGetLastError() != cudaSuccess) return EMB_ECUDA;
    int host = 0;
    if (cudaMemcpyAsync(&host, slot, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess) return EMB_ECUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return EMB_ECUDA;
    return (host & kStatusTimeout) ? EMB_ETIMEOUT : EMB_OK;
}

emb_status emb_selftest_wait_timeout(int64_t timeout_ns, emb_stream_t stream) {
    if (timeout_ns < 1000 || timeout_ns > 1000000000) return EMB_EINVAL;
    int* st = status_ptr();
    if (!st) return EMB_ECUDA;
    return from_cuda(launch_selftest_wait(uint64_t(timeout_ns), st, reinterpret_cast<cudaStream_t>(stream)));
}

const char* emb_status_string(emb_status status) {
    switch (status) {
        case EMB_OK: return "EMB_OK";
        case EMB_EINVAL: return "EMB_EINVAL: invalid argument";
        case EMB_EALIGN: return "EMB_EALIGN: misaligned device pointer";
        case EMB_ENOSPC: return "EMB_ENOSPC: workspace too small";
        case EMB_ECUDA: return "EMB_ECUDA: CUDA runtime error";
        case EMB_ETIMEOUT: return "EMB_ETIMEOUT: device-side wait expired";
        case EMB_EUNSUPPORTED: return "EMB_EUNSUPPORTED: shape not supported by this build";
    }
    return "unknown emb_status";
}

const char* emb_build_info(void) {
    return "libembqmm: sm_103a; Q8_0/Q6_0/Q4_0; GEMV (M<=4: staged/ring/register FFMA2, Q4_0 mma.sync at M>=2) + "
           "tcgen05 GEMM (M>4: TMA, dequant to bf16 A tiles in TMEM, TMEM accumulators; one tile, persistent, "
           "cluster split-K or stream-K schedules); "
           "recorded chains (CUDA graphs); RMSNorm, rotary embedding, grouped-head attention";
}

}  // extern "C"
