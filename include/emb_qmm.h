/*
 * emb_qmm.h -- C ABI of libembqmm.so, the GB300 (sm_103a) block-quantised
 * weight x bf16 activation matmul that carries every linear layer of a
 * vision-language-action backbone and action head in batch-1 embodied inference.
 *
 * Paper: "Embodied.cpp: A Portable Inference Runtime of Embodied AI Models on
 * Heterogeneous Robots" (arXiv 2607.02501).
 *   - batch-1 execution where each control step's latency is what counts:
 *     Section 3.1, challenge 2; Section 3.2, design principle 2 (fusing the
 *     step's work, replaying it as a recorded graph, reusing its buffers and
 *     keeping host-device copies few);
 *   - the 8-, 6- and 4-bit weight configurations: Section 4, Table 3 (its
 *     8-bit, 6-bit and 4-bit C++ columns);
 *   - a stable deployment boundary behind one backend abstraction: abstract;
 *     Section 3.2 (Figure 2 description).
 * The paper gives no byte format; the three block formats below are this
 * library's definition of the 8-, 6- and 4-bit configurations.
 *
 * Conventions for every entry point
 *   - W is [N][K] (output features x input features, PyTorch Linear.weight
 *     layout), X is [M][K] row-major bf16 (passed as its 16-bit patterns),
 *     Y is [M][N] row-major fp32, and Y[m][n] = sum_k w'[n][k] * x[m][k].
 *   - Every pointer argument is DEVICE memory owned by the caller, except the
 *     `layers` arrays of emb_qlayer_seq / emb_chain_create, which are host memory
 *     read during the call only. The library allocates no device memory and keeps
 *     no per-call state (a recorded chain is a caller-owned handle); all calls are
 *     reentrant and thread-safe.
 *   - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) without any host synchronisation, except emb_device_status.
 *   - Argument errors are reported BEFORE anything is enqueued. Launch errors
 *     return EMB_ECUDA. Device-side failures (a bounded wait that expired) are
 *     recorded in a device status word read by emb_device_status. After
 *     EMB_ETIMEOUT the outputs of the calls enqueued since the last status read
 *     are undefined, residual-add (EMB_EPI_ADD) buffers included.
 *   - Outputs are fully overwritten. Inputs and outputs must not overlap.
 * Each entry point below names the paper passage it serves.
 */
#ifndef EMB_QMM_H
#define EMB_QMM_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define EMB_API __attribute__((visibility("default")))
#else
#define EMB_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t (the runtime's stream handle); NULL = default stream. */
typedef struct CUstream_st* emb_stream_t;

typedef enum {
    /* 32 consecutive weights of one row along K share one fp16 scale d;
     * each weight is an int8 code q in [-127, 127]; w' = d * q.
     * d = fp16_rne(max|w| / 127), q = clamp(round_half_away(w / d), -127, 127). */
    EMB_Q8_0 = 0,
    /* 32 consecutive weights share one fp16 scale d; each weight is a 4-bit code
     * q in [0, 15]; w' = d * (q - 8). With m the signed weight of largest
     * magnitude (lowest index on ties): d = fp16_rne(m / -8),
     * q = clamp(round_half_away(w / d), -8, 7) + 8. */
    EMB_Q4_0 = 1,
    /* As EMB_Q4_0 with 6-bit codes q in [0, 63]: w' = d * (q - 32),
     * d = fp16_rne(m / -32), q = clamp(round_half_away(w / d), -32, 31) + 32. */
    EMB_Q6_0 = 2
} emb_qfmt;

typedef enum {
    EMB_OK = 0,
    EMB_EINVAL = 1,        /* unknown format, M/N/K < 1, K % 32 != 0, NULL pointer,
                              overlapping buffers, too many layers */
    EMB_EALIGN = 2,        /* a device pointer is not 16-byte aligned
                              (W_blocks must be 256-byte aligned) */
    EMB_ENOSPC = 3,        /* workspace smaller than emb_qlayer_seq_workspace() */
    EMB_ECUDA = 4,         /* a CUDA runtime call or launch failed */
    EMB_ETIMEOUT = 5,      /* a device-side bounded wait expired (emb_device_status) */
    EMB_EUNSUPPORTED = 6   /* shape outside what this build supports (see limits) */
} emb_status;

/* ---------------------------------------------------------------- packed weights
 * Section 4, Table 3 (the 8-, 6- and 4-bit configurations whose weights these are).
 * Packed image of one [N][K] matrix (one caller allocation of
 * emb_qweight_bytes(fmt, N, K) bytes, 256-byte aligned, written only by
 * emb_quantize_*; callers may copy, save and reload it as plain bytes):
 *   codes plane at byte 0:
 *     Q8_0: int8  [N][K], row-major;
 *     Q4_0: uint8 [N][K/2]; in each 32-weight block, byte j (0..15) holds
 *           code j in its low nibble and code j+16 in its high nibble;
 *     Q6_0: the low 4 bits of every code in a [N][K/2] plane laid out as Q4_0's,
 *           then, at byte roundup(N*K/2, 256), the high 2 bits: uint8 [N][K/4]
 *           where in each block byte j (0..7) holds the high bits of codes j,
 *           j+8, j+16, j+24 at bits 0-1, 2-3, 4-5, 6-7;
 *   scales plane at byte roundup(codes_bytes, 256) (Q6_0: roundup of the end
 *     of the high plane, 256): fp16 [N][ldS] with ldS = roundup(K/32, 8)
 *     (16-byte row pitch);
 *   every padding byte is zero, so two images of the same weights compare equal
 *   byte for byte.
 * Returns the byte size, or 0 when fmt is unknown, N < 1, K < 32 or K % 32 != 0. */
EMB_API size_t emb_qweight_bytes(emb_qfmt fmt, int64_t N, int64_t K);

/* Section 4, Table 3 (8-bit column): the offline packing of one weight matrix.
 * Quantise fp32 W [N][K] (device, 16-byte aligned) into W_blocks (device,
 * 256-byte aligned, emb_qweight_bytes(EMB_Q8_0, N, K) bytes). Offline step of
 * the path (packing weights once per model). NaN/Inf weights, and weights so
 * large that max|w|/127 overflows fp16, are outside the contract. */
EMB_API emb_status emb_quantize_q8_0(const float* W, int64_t N, int64_t K, void* W_blocks,
                             emb_stream_t stream);

/* Section 4, Table 3 (4-bit column).
 * As emb_quantize_q8_0 for EMB_Q4_0 (m/-8 must not overflow fp16). */
EMB_API emb_status emb_quantize_q4_0(const float* W, int64_t N, int64_t K, void* W_blocks,
                             emb_stream_t stream);

/* Section 4, Table 3 (6-bit column; the paper gives no format, EMB_Q6_0 above is this
 * library's definition). As emb_quantize_q8_0 for EMB_Q6_0. */
EMB_API emb_status emb_quantize_q6_0(const float* W, int64_t N, int64_t K, void* W_blocks,
                             emb_stream_t stream);

/* ---------------------------------------------------------------------- matmul
 * Section 3.1, challenge 2 (batch-1, latency-first control steps: M = 1 decode, M = 50
 * action chunks, M = 250..820 prefix prefill) on the Table 3 weight formats.
 * Y [M][N] fp32 = X [M][K] bf16  x  w'^T, w' the dequantised weights of W_blocks.
 * X, Y: device, 16-byte aligned; W_blocks as produced by emb_quantize_*.
 * Small M (M <= 4, action-token decode) runs a weight-streaming GEMV that dequantises
 * in registers; larger M (action-chunk denoising, prefix prefill) runs a tcgen05
 * tensor-core GEMM that dequantises shared-memory tiles to bf16.
 * Accuracy, per element, with Y_exact from the same dequantised weights w' and the
 * same bf16 X, and S = sum_k |w'[n][k] x[m][k]|:
 *   - M <= 4, or K < 1024:  |Y - Y_exact| <= 1e-3 * S + 1e-6 for every input (the GEMV's
 *     products are exact; below K = 1024 the GEMM's operand is bf16(w') plus the bf16 of
 *     its rounding remainder, relative error <= 2^-16);
 *   - M > 4 and K >= 1024:  the GEMM's operand is bf16(w'), relative error <= 2^-8 per
 *     weight (bf16's unit roundoff), so |Y - Y_exact| <= (2^-8 + 2^-12) * S + 1e-6 always
 *     (operand rounding plus fp32 accumulation), and the 1e-3 * S + 1e-6 bound holds when
 *     S is spread over many terms (every workload shape: observed error / S below 2e-4)
 *     but can fail when a handful of terms dominate S. A layer whose epilogue
 *     carries EMB_PRECISE_OPERAND (emb_qlayer_seq) gets the two-operand form at every K
 *     and the 1e-3 * S + 1e-6 bound for every input, at about twice the tensor work.
 * Results are bitwise reproducible from call to call for a given shape. */
EMB_API emb_status emb_qmatmul(emb_qfmt fmt, const void* W_blocks, const uint16_t* X, float* Y,
                       int64_t M, int64_t N, int64_t K, emb_stream_t stream);

/* --------------------------------------------------------------- layer chains
 * One linear layer of a chain: Y = X x w'^T with its own X and Y (device). */
/* What a layer of a chain writes (its epilogue). acc[m][n] is the fp32 result
 * sum_k w'[n][k] x[m][k] with emb_qmatmul's accuracy.
 *   EMB_EPI_F32    Y fp32 [M][N] = acc                       (emb_qmatmul's output)
 *   EMB_EPI_BF16   Y bf16 [M][N] = bf16_rne(acc)             (input of a next layer)
 *   EMB_EPI_ADD    Y fp32 [M][N] += acc, one fp32 rounding   (residual add in place)
 *   EMB_EPI_GEGLU  W holds gate and up rows interleaved (row 2i = gate_i, row 2i+1 =
 *                  up_i; N even); Y bf16 [M][N/2] = bf16_rne(gelu(acc[2i]) * acc[2i+1])
 *                  with gelu(g) = 0.5 g (1 + tanh(sqrt(2/pi) (g + 0.044715 g^3)))
 *   EMB_EPI_SWIGLU as EMB_EPI_GEGLU with silu(g) = g / (1 + exp(-g))
 * The activations are evaluated in fp32 with the CUDA math library. */
typedef enum {
    EMB_EPI_F32 = 0,
    EMB_EPI_BF16 = 1,
    EMB_EPI_ADD = 2,
    EMB_EPI_GEGLU = 3,
    EMB_EPI_SWIGLU = 4
} emb_epilogue;

/* Flag OR-ed into emb_qlayer.epilogue: run this layer's tensor-core GEMM (M > 4) with the
 * two-operand weights bf16(w') + bf16(w' - bf16(w')) at every K, so that emb_qmatmul's
 * 1e-3 * S + 1e-6 accuracy holds for every input (see emb_qmatmul). No effect at M <= 4. */
#define EMB_PRECISE_OPERAND 0x100

typedef struct {
    int32_t fmt;            /* emb_qfmt */
    int32_t epilogue;       /* emb_epilogue, optionally | EMB_PRECISE_OPERAND */
    const void* W_blocks;   /* packed image of W [N][K] */
    int64_t N;
    int64_t K;
    const uint16_t* X;      /* [M][K] bf16 */
    void* Y;                /* as the epilogue says; 16-byte aligned */
} emb_qlayer;

#define EMB_MAX_LAYERS 4096

/* Section 3.2, principle 2 (buffer reuse: the caller owns every buffer of a chain,
 * the library allocates nothing).
 * Bytes of device workspace with which emb_qlayer_seq / emb_chain_create run these layers
 * at this M on the current device with their fastest schedule. 0 when no launch of the
 * chain wants one (every M <= 4 chain; prefill layers whose tiles already fill the SMs).
 * Otherwise some tensor-core launch (M >= 128) would split the k range of its tiles evenly
 * over all SMs ("stream-K") and add the partial tiles through the workspace: 4 KB of
 * flags, then one fp32 partial tile per SM, a few MB to about 35 MB in all. The answer
 * depends on the device's SM count. Returns (size_t)-1 for invalid arguments. */
EMB_API size_t emb_qlayer_seq_workspace(const emb_qlayer* layers, int n_layers, int64_t M);

/* Run n_layers linears in order on `stream`, all with M tokens (the paper's
 * fusion, graph replay and buffer reuse of Section 3.2, principle 2).
 * Semantics are those of n_layers single-layer calls in sequence, each with
 * its epilogue. Consecutive layers that read the same X with the same fmt, K
 * and epilogue (q/k/v, gate/up) are fused into one launch; each launch may
 * fetch its weights before the previous launch has finished (programmatic
 * dependent launch), and reads X and writes Y only after it. So a layer's X may
 * be the output of an earlier layer of the same call (a bf16 epilogue feeding
 * the next projection), and layers may add into the same residual buffer in
 * turn. A layer's W_blocks may not overlap the Y of the same or an earlier
 * layer, and its X may not overlap its own Y (EMB_EINVAL); an unknown epilogue,
 * or a gated one with odd N, is EMB_EINVAL. The call enqueues kernels only, so it may
 * be captured into a CUDA graph and replayed.
 * workspace / ws_bytes: NULL, or device memory of at least emb_qlayer_seq_workspace()
 * bytes (EMB_ENOSPC if smaller), 256-byte aligned (EMB_EALIGN), zero-filled before its
 * first use. A call leaves it ready for the next one (its first 4 KB, the flags, back at
 * zero) unless it reports EMB_ETIMEOUT: then zero it again before reusing it. With NULL
 * the launches take schedules that need none. The
 * results are deterministic either way, but the two schedules add the k range in different
 * pieces, so they agree within the accuracy bound, not bitwise. One workspace serves one
 * stream at a time: calls that may run concurrently need separate workspaces. */
EMB_API emb_status emb_qlayer_seq(const emb_qlayer* layers, int n_layers, int64_t M,
                          void* workspace, size_t ws_bytes, emb_stream_t stream);

/* Section 3.2, principle 2 (operator fusion across a layer's launches).
 * As emb_qlayer_seq, for a call inside a chain of this library's launches (a layer's
 * linears between its norm, rotary and attention launches): the first launch of the call
 * also overlaps its weight fetch with the end of the launch before it on `stream`, as
 * every later launch of a call does. Precondition: the weights of the call are not
 * written by the launch enqueued on `stream` just before the call (weights produced
 * further back, e.g. by emb_quantize_* followed by any other launch or a synchronisation,
 * are fine). No workspace: results are bitwise those of emb_qlayer_seq with a NULL
 * workspace. Errors as emb_qlayer_seq. */
EMB_API emb_status emb_qlayer_seq_chained(const emb_qlayer* layers, int n_layers, int64_t M,
                                          emb_stream_t stream);

/* Section 3.2, principle 2 has the caller own every buffer of a chain; this call is the
 * exception and has no counterpart in the paper. emb_qlayer_seq with a workspace that the
 * library owns: a static device array of 48 MB (zero at load) in this library's module on
 * each device, so a chain needs no allocation by the caller and still takes its stream-K
 * schedules (a chain wanting more than 48 MB runs as with a NULL workspace). Results are
 * bitwise those of emb_qlayer_seq with a caller workspace. Each call first zeroes the
 * array's 4 KB of flags on `stream` when a launch of the chain will use it. The array is
 * one per device: calls on different streams of one device must not run concurrently
 * (order them, e.g. with events); recording the call into a graph records the array's
 * address. Errors as emb_qlayer_seq; EMB_ECUDA if the array cannot be reached. */
EMB_API emb_status emb_qlayer_seq_noalloc(const emb_qlayer* layers, int n_layers, int64_t M,
                                          emb_stream_t stream);

/* ------------------------------------------------------------ recorded chains
 * Graph replay and buffer reuse (Section 3.2, design principle 2): the
 * launches that emb_qlayer_seq(layers, n_layers, M, workspace, ws_bytes, ...) enqueues
 * are recorded once into a CUDA graph and then replayed with one call, so a closed-loop
 * step costs one host call instead of one per launch group. */
typedef struct emb_chain_st* emb_chain_t;

/* Section 3.2, principle 2 (graph replay, buffer reuse).
 * Record the chain. Arguments, validation and error codes are those of emb_qlayer_seq
 * (nothing is launched: the launches are captured on a private stream of the current
 * device). The recording holds the layers' pointers: every replay reads the X buffers
 * and fully overwrites the Y buffers given here, so callers refill the X buffers between
 * replays and keep every buffer (and the workspace) alive until emb_chain_destroy.
 * Results of a replay are bitwise those of emb_qlayer_seq on the same inputs.
 * On success *chain receives a handle owned by the caller; on failure it is NULL.
 * Errors: EMB_EINVAL (also for a NULL chain pointer), EMB_EALIGN, EMB_EUNSUPPORTED,
 * EMB_ECUDA (stream capture or graph instantiation failed). */
EMB_API emb_status emb_chain_create(const emb_qlayer* layers, int n_layers, int64_t M,
                            void* workspace, size_t ws_bytes, emb_chain_t* chain);

/* Section 3.2, principle 2 (graph replay: one host call per closed-loop step).
 * Enqueue one replay of the recorded chain on `stream` (a stream of the device it was
 * recorded on). EMB_EINVAL for a NULL handle, EMB_ECUDA if the launch fails. */
EMB_API emb_status emb_chain_launch(emb_chain_t chain, emb_stream_t stream);

/* Section 3.2, principle 2 (graph replay). Free the recording (NULL is a no-op).
 * Replays already enqueued still complete. */
EMB_API emb_status emb_chain_destroy(emb_chain_t chain);

/* Section 3.2, principle 2: record any sequence of this library's calls as one chain
 * (graph replay of a whole layer or loop). After emb_chain_record_begin(stream), every library
 * call made by this thread on `stream` is recorded instead of run (CUDA stream capture in
 * thread-local mode) until emb_chain_record_end(stream, &chain) returns the recording,
 * which emb_chain_launch replays and emb_chain_destroy frees. The recording holds every
 * pointer the recorded calls were given; callers keep those buffers alive. Between begin
 * and end no call may synchronise (emb_device_status) and arguments are validated as
 * usual (an invalid call records nothing and returns its error; the recording goes on).
 * stream: a created (non-NULL) stream of the current device.
 * Errors: EMB_EINVAL (NULL stream or chain pointer), EMB_ECUDA (capture could not begin or
 * end, or instantiation failed; *chain is then NULL). */
EMB_API emb_status emb_chain_record_begin(emb_stream_t stream);
/* Section 3.2, principle 2 (graph replay): end the recording begun on `stream`. */
EMB_API emb_status emb_chain_record_end(emb_stream_t stream, emb_chain_t* chain);

/* ---------------------------------------------------------------- layer steps
 * The steps of one transformer layer of the shared backbone and the action expert around
 * its linears (the paper runs every model family through one backbone execution path,
 * Section 3.2, and defines none of these operators; the standard definitions are used).
 * All are enqueued on `stream` with programmatic dependent launch, like emb_qlayer_seq,
 * allocate nothing, and are deterministic. bf16 buffers hold bit patterns (uint16_t). */

/* Section 3.2 (the shared backbone layer around the linears).
 * RMSNorm (Zhang and Sennrich, 2019) of every token of the fp32 residual stream:
 * y[m][i] = bf16(x[m][i] / sqrt(mean_i x[m][i]^2 + eps) * gamma[i]), the mean and square
 * root in fp32 (correctly rounded square root and reciprocal), one bf16 rounding.
 * x: device fp32 [M][D]; gamma: device fp32 [D]; y: device bf16 [M][D]; 16-byte aligned.
 * 1 <= M < 2^31; D % 8 == 0, 8 <= D <= 65536; eps >= 0. y may not overlap x or gamma.
 * Errors: EMB_EINVAL, EMB_EALIGN, EMB_ECUDA. */
EMB_API emb_status emb_rmsnorm(const float* x, const float* gamma, uint16_t* y, int64_t M,
                               int64_t D, float eps, emb_stream_t stream);

/* Section 3.2 (the shared backbone layer around the linears).
 * Rotary position embedding (Su et al., 2021), rotate-half pairing, in place on bf16
 * x [M][n_heads][head_dim]: token m sits at position pos0 + m; in every head, element i
 * and element i + head_dim/2 (i < head_dim/2) are rotated by the angle
 * (pos0 + m) * base^(-2i/head_dim): (a, b) -> (a cos - b sin, b cos + a sin). The
 * inverse frequencies are formed in fp64 on the host, the angle as an exact two-float
 * product, its cosine and sine in fp32 (error ~1e-7), the rotation in fp32, one bf16
 * rounding. x: device, 16-byte aligned. head_dim even, 2..512; pos0 >= 0,
 * pos0 + M <= 2^24 (positions exact in fp32); base > 0.
 * Errors: EMB_EINVAL, EMB_EALIGN, EMB_ECUDA. */
EMB_API emb_status emb_rope(uint16_t* x, int64_t M, int64_t n_heads, int64_t head_dim,
                            int64_t pos0, float base, emb_stream_t stream);

/* Section 3.2 (the shared backbone layer), principle 2 (fusion: one launch for q and k).
 * emb_rope of q [M][n_q_heads][head_dim] and k [M][n_k_heads][head_dim] at the same
 * positions in one launch (results bitwise those of two emb_rope calls). k may be NULL
 * when n_k_heads == 0; q and k may not overlap. Errors as emb_rope. */
EMB_API emb_status emb_rope_qk(uint16_t* q, int64_t n_q_heads, uint16_t* k, int64_t n_k_heads,
                               int64_t M, int64_t head_dim, int64_t pos0, float base,
                               emb_stream_t stream);

/* Section 3.1 (the action chunk attends to the prefix cache: "prefix once, head many")
 * and Section 3.2 (the shared backbone layer).
 * Scaled dot-product attention (Vaswani et al., 2017) of M query tokens over n0 + n1 keys:
 * the prefix cache (K0, V0: [n0][n_kv_heads][head_dim]) followed by the chunk's own keys
 * (K1, V1: [n1][n_kv_heads][head_dim]), all visible to every query (no mask). Query head h
 * (Q: [M][n_heads][head_dim]) reads key/value head h / (n_heads / n_kv_heads);
 * O[m][h] = sum_j softmax_j(scale * q.k_j) v_j, in fp32, one bf16 rounding.
 * All bf16, device, 16-byte aligned; K0/V0 may be NULL when n0 == 0, K1/V1 when n1 == 0.
 * n_heads % n_kv_heads == 0; head_dim 64 or 128 (else EMB_EUNSUPPORTED); n0 + n1 >= 1.
 * O may not overlap any input. Errors: EMB_EINVAL, EMB_EALIGN, EMB_EUNSUPPORTED, EMB_ECUDA. */
EMB_API emb_status emb_attention(const uint16_t* Q, const uint16_t* K0, const uint16_t* V0,
                                 int64_t n0, const uint16_t* K1, const uint16_t* V1, int64_t n1,
                                 uint16_t* O, int64_t M, int64_t n_heads, int64_t n_kv_heads,
                                 int64_t head_dim, float scale, emb_stream_t stream);

/* ---------------------------------------------------------------- test support
 * Section 4, Table 3 (the weights of the 8-, 6- and 4-bit configurations, dequantised).
 * Dequantise W_blocks to fp32 [N][K] (w' exactly: the products are exact in fp32). */
EMB_API emb_status emb_dequantize_f32(emb_qfmt fmt, const void* W_blocks, int64_t N, int64_t K,
                              float* out, emb_stream_t stream);

/* Section 4, Table 3. Dequantise to bf16 bit patterns [N][K]: one round-to-nearest-even
 * of the exact fp32
 * w' -- the operand values the tensor-core GEMM feeds to its MMAs. */
EMB_API emb_status emb_dequantize_bf16(emb_qfmt fmt, const void* W_blocks, int64_t N, int64_t K,
                               uint16_t* out, emb_stream_t stream);

/* Section 3.2 (the deployment boundary reports device-side failures to the host).
 * Read and clear the device status word in one atomic exchange enqueued on `stream`,
 * then synchronise `stream` (only that stream): EMB_OK, or EMB_ETIMEOUT if a kernel's
 * bounded wait expired since the last call. A timeout recorded by work on another stream
 * that has not finished yet is reported by a later call. */
EMB_API emb_status emb_device_status(emb_stream_t stream);

/* Section 3.2 (deployment boundary; test support for the failure path above).
 * Launch one block that waits on a shared-memory barrier that nothing completes,
 * giving up after timeout_ns nanoseconds (1e3 .. 1e9): exercises the bounded-wait
 * error path; emb_device_status then returns EMB_ETIMEOUT. */
EMB_API emb_status emb_selftest_wait_timeout(int64_t timeout_ns, emb_stream_t stream);

/* Section 3.2 (deployment boundary). Human-readable name of a status code (static
 * string). */
EMB_API const char* emb_status_string(emb_status status);

/* Section 3.2 (backend abstraction: which backend this is). Static string describing
 * the build (target architecture, kernel variants). */
EMB_API const char* emb_build_info(void);

#ifdef __cplusplus
}
#endif

#endif /* EMB_QMM_H */
