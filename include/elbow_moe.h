/*
 * elbow_moe.h - C ABI of the GB300 (sm_103a) elbow-routed MoE layer.
 *
 * The method is "Elbow-based MoE Routing" (arxiv 2608.04401): per token, the
 * router's softmax probabilities are sorted in descending order, a
 * Kneedle-style elbow index e (0-based) is found on the curve normalised to
 * [0,1] (Alg. 1, which returns e + 1), and only k = min(e + 1, K) experts are
 * used instead of a fixed top-K (Sec. 2.1). This library runs that MoE layer
 * forward on one GPU.
 *
 * Conventions for every entry point:
 *   - All tensor pointers are DEVICE pointers owned by the caller; the library
 *     allocates no memory and never synchronises the stream (except
 *     moe_read_device_error, which says so).
 *   - Tensors are dense, row-major, with the shapes given per argument.
 *     bf16 tensors are passed as uint16_t bit patterns.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream). Work is
 *     enqueued on it and the call returns at once.
 *   - Every call returns a moe_status and never aborts the process. Argument
 *     errors are detected on the host before anything is enqueued.
 *   - Supported shapes: N (experts) in {64, 128}; 1 <= K <= 8 and K <= N;
 *     0 <= T < 2^28 tokens (T = 0 is a no-op; larger T returns
 *     MOE_ERR_INVALID_ARG, so that the T * K pair counts fit in int32); for
 *     the layer, d_model and the SwiGLU intermediate I multiples of 128,
 *     d, I <= 16384.
 *   - Pointers must be 16-byte aligned.
 *
 * Routing arithmetic is fp32 and fully specified (see elbow_route), so that
 * routing decisions are reproducible bit for bit by an independent
 * implementation of the same specification.
 */
#ifndef ELBOW_MOE_H
#define ELBOW_MOE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MOE_OK = 0,
  MOE_ERR_INVALID_ARG = 1,    /* null or misaligned pointer, negative size, bad params */
  MOE_ERR_UNSUPPORTED = 2,    /* shape outside the supported set above */
  MOE_ERR_WORKSPACE = 3,      /* workspace missing or smaller than the query says */
  MOE_ERR_CUDA = 4,           /* a CUDA runtime/driver call failed */
  MOE_ERR_DEVICE_TIMEOUT = 5  /* a kernel gave up a bounded wait (see moe_read_device_error) */
} moe_status;

typedef enum {
  MOE_ROUTE_ELBOW = 0,
  MOE_ROUTE_TOPK = 1,
  MOE_ROUTE_RAND_TAIL = 2,  /* elbow_route_randomized only */
  MOE_ROUTE_RAND_HEAD = 3   /* elbow_route_randomized only */
} moe_route_mode;

/* Routing parameters. K: the cap (top-K of the base router, Sec. 2.1).
 * eps: the epsilon of Alg. 1's normalisation (the paper leaves it unstated;
 * default 1e-8). mode: ELBOW (k = min(e, K)) or TOPK (k = K, the fixed top-K
 * baseline of Sec. 3 on the same kernels). renorm: 0 = gates are the selected
 * experts' softmax probabilities (default); 1 = divided by their sum. */
typedef struct {
  int K;
  float eps;
  int mode;
  int renorm;
} moe_route_params;

/* Human-readable name of a status code (static storage; "unknown moe_status"
 * for other values). No counterpart in the paper. */
const char* moe_status_string(moe_status s);

/*
 * elbow_route - Alg. 1 and the capped selection of Sec. 2.1, per token.
 *
 *   logits    [T, N] fp32      router logits l(x)
 *   k_out     [T]    int32     k = min(e + 1, K) (ELBOW) or K (TOPK), 1 <= k <= K
 *   ids_out   [T, K] int32     expert ids of the K largest probabilities in
 *                              descending order (ties: lower id first); all K
 *                              are written, the first k are the selection
 *   gates_out [T, K] fp32      p_(s) for s < k, 0 for s >= k (renorm: divided
 *                              by the sum of the first k, left to right)
 *
 * fp32 specification (every operation rounded to nearest even, no
 * contraction): m = max_j l_j; e_j = EXP(l_j - m) with EXP the library's
 * Cody-Waite/Taylor exponential (zero below 2^-126); s = balanced tree sum
 * (v_i += v_{i+h}, h = N/2 .. 1); p_j = e_j / s; sort p descending;
 * den = (p_max - p_min) + eps; p'_i = (p_(i) - p_min) / den (both quotients
 * correctly rounded, as the printed formulas divide);
 * x'_i = i/(N-1); D_i = (1 - p'_i) - x'_i (the deviation below the chord of
 * the descending curve; Alg. 1 prints the sign reversed, which would give
 * k = 1 always); e = smallest argmax_i D_i. Logits must be finite.
 */
moe_status elbow_route(const float* logits, int64_t T, int N, const moe_route_params* rp,
                       int32_t* k_out, int32_t* ids_out, float* gates_out, void* stream);

/* elbow_route (Alg. 1, Sec. 2.1) with one warp (instead of one thread) per token: lane l holds
 * experts l + 32c, the N (p, id) keys are sorted by a bitonic network of warp
 * shuffles and the argmax is a warp reduction. Same specification, same bits
 * as elbow_route; a much shorter critical path per token, at about three
 * times the instructions per token, so elbow_route uses it by itself for
 * T <= 16 (and moe_layer_forward's router, after a router GEMM split over d
 * and 16-token groups, for 3 <= T <= 64; for T <= 2 one cluster of CTAs computes
 * the logits and routes each token with one warp). Arguments and errors as elbow_route
 * (ids_out and gates_out need only 4-byte alignment). */
moe_status elbow_route_warp(const float* logits, int64_t T, int N, const moe_route_params* rp,
                            int32_t* k_out, int32_t* ids_out, float* gates_out, void* stream);

/* elbow_route (Alg. 1, Sec. 2.1) that also counts, for the dispatch (App. A.4), the selected pairs of each
 * expert in each chunk of 128 tokens: chunk_counts [N][ceil(T/128)] int32
 * (pass moe_dispatch_chunk_counts(ws) and follow with moe_dispatch_counted,
 * which then skips its own counting pass over k and ids). */
moe_status elbow_route_with_counts(const float* logits, int64_t T, int N,
                                   const moe_route_params* rp, int32_t* k_out, int32_t* ids_out,
                                   float* gates_out, int32_t* chunk_counts, void* stream);

/*
 * moe_dispatch - token-to-expert grouping of the selected (t, s < k_t) pairs,
 * as the MoE block of App. A.4 sends each token to its selected experts.
 *
 *   k        [T]      int32  selected counts (0 <= k_t <= K)
 *   ids      [T, K]   int32  expert ids (distinct within a token, < N)
 *   offsets  [N + 1]  int32  exclusive prefix sum of the per-expert counts;
 *                            offsets[N] = sum_t k_t
 *   perm     [T * K]  int32  capacity T*K; perm[offsets[e] .. offsets[e+1])
 *                            are the tokens routed to expert e, ascending
 *                            (stable); entries from offsets[N] on are untouched
 *   pair_pos [T, K]   int32  position in perm of pair (t, s), -1 for s >= k_t
 *   ws       device workspace of at least moe_dispatch_workspace_size bytes,
 *            256-byte aligned; its first int32 is a device error word
 * A pair whose id lies outside [0, N) is dropped: it is not counted, not in
 * perm, and its pair_pos is -1 (elbow_route never produces such ids). Ids
 * repeated within a token give unspecified positions, but no access outside
 * the arrays above.
 * moe_dispatch runs batches of more than 128 tokens whose per-block shared
 * memory fits as one cooperative kernel (each block reads its tokens' selections once,
 * counts, meets the others at one grid barrier, then places its pairs); that
 * barrier's wait is bounded, and when it runs out the error word is set and
 * moe_read_device_error(ws) returns MOE_ERR_DEVICE_TIMEOUT (the outputs are
 * then incomplete). The word is cleared by each such call.
 */
/* Bytes of moe_dispatch's workspace; 0 for unsupported sizes (T outside
 * [0, 2^28), N not 64 or 128). */
size_t moe_dispatch_workspace_size(int64_t T, int N, int K);
moe_status moe_dispatch(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                        int32_t* offsets, int32_t* perm, int32_t* pair_pos, void* ws,
                        size_t ws_bytes, void* stream);

/*
 * moe_dispatch_noalloc - moe_dispatch for callers that cannot allocate device
 * memory when they dispatch: for example a serving runtime that sizes all of
 * its device memory up front and allows no allocation on the request path
 * (an allocation can stall on the device or fragment its pool), or a plug-in
 * whose host framework passes it only input and output buffers. The paper has
 * no counterpart; this is a packaging variant of the same dispatch kernels.
 *
 * Arguments and results are those of moe_dispatch, without the workspace. The
 * scratch (per-chunk expert counts, 128 experts x 2048 chunks of 128 tokens,
 * plus totals and tile offsets: about 1 MB) is a fixed array inside the
 * library, which every GPU that loads the library keeps until the process
 * exits. Limits: T <= 262,144 tokens (larger T returns MOE_ERR_UNSUPPORTED),
 * N in {64, 128}, K <= 8.
 * No cudaMalloc, cudaFree or other allocating call is made.
 * The first call on each device looks up the array's device address (with
 * that device current) and caches it for the life of the process; make that
 * first call before any stream capture. cudaDeviceReset may move the array,
 * so this entry point must not be called again after a reset of a device it
 * has already been used on. All calls share the one array and each call
 * rewrites every part of it that it reads, so no clearing is needed; calls
 * whose kernels overlap on the GPU (different streams, or different host
 * threads) race on the array. Launch failures return MOE_ERR_CUDA (errors
 * left pending by earlier, unrelated calls are not read).
 */
moe_status moe_dispatch_noalloc(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                                int32_t* offsets, int32_t* perm, int32_t* pair_pos, void* stream);

/*
 * moe_layer_forward - one MoE layer forward under elbow routing (Sec. 2,
 * App. A.4): router logits l = W_r x (bf16 x bf16, fp32 accumulate), routing
 * as elbow_route, dispatch as moe_dispatch, per-expert SwiGLU
 *   h = silu(W_gate[e] x) * (W_up[e] x)   (bf16 tensor cores, fp32 accumulate,
 *                                          h stored as bf16; CUDA cores with fp32
 *                                          accumulation for T <= 2)
 *   o = W_down[e] h                       (stored as bf16)
 * and the combine y_t = sum_{s < k_t} g_{t,s} o_{t,s} (+ residual_t), summed
 * in s order in fp32 and rounded to bf16.
 *
 *   x          [T, d]       bf16   tokens
 *   w_router   [N, d]       bf16   router weight W_r
 *   w_gate_up  [N, 2I, d]   bf16   rows [0, I) = W_gate[e], rows [I, 2I) = W_up[e]
 *   w_down     [N, d, I]    bf16   W_down[e]
 *   residual   [T, d]       bf16   optional (NULL = none); may alias y
 *   y          [T, d]       bf16   output
 *   logits_out [T, N] fp32, k_out [T], ids_out [T, K], gates_out [T, K],
 *   offsets_out [N + 1]            optional copies of the intermediate
 *                                  results (NULL = not written)
 *   ws         device workspace of at least moe_layer_workspace_size bytes,
 *              256-byte aligned; it also holds the device error word read by
 *              moe_read_device_error.
 * TOPK mode runs the same kernels with k = K.
 * moe_layer_workspace_size returns 0 for unsupported sizes (T outside
 * [0, 2^28), N not 64 or 128, K outside [1, 8], d or I outside [1, 16384]).
 */
size_t moe_layer_workspace_size(int64_t T, int d, int N, int I, int K);
moe_status moe_layer_forward(const uint16_t* x, const uint16_t* w_router, const uint16_t* w_gate_up,
                             const uint16_t* w_down, int64_t T, int d, int N, int I,
                             const moe_route_params* rp, const uint16_t* residual, uint16_t* y,
                             float* logits_out, int32_t* k_out, int32_t* ids_out, float* gates_out,
                             int32_t* offsets_out, void* ws, size_t ws_bytes, void* stream);

/*
 * moe_read_device_error - SYNCHRONISES `stream`, then reads the error word
 * that the layer's kernels leave in `ws` (they clear it at the start of each
 * moe_layer_forward). Returns MOE_OK, or MOE_ERR_DEVICE_TIMEOUT if a kernel
 * gave up a bounded wait on its pipeline barriers (its outputs are then
 * invalid; the CUDA context stays usable).
 */
moe_status moe_read_device_error(const void* ws, void* stream);

/* ---- step-level entry points (the layer's stages, for testing and reuse) ----
 *
 * Errors, for each of them: MOE_ERR_INVALID_ARG for a null or misaligned
 * pointer (16 bytes for tensors, 4 bytes for int32 / fp32 arrays and the
 * error word) or a size out of range; MOE_ERR_UNSUPPORTED for N, K, d or I
 * outside the supported set; MOE_ERR_CUDA if a launch fails. A GEMM that gives
 * up a bounded wait writes a nonzero code into err_word (when given). */

/* Router logits l = W_r x (the router of Sec. 2): x [T, d] bf16, w_router [N, d] bf16 -> logits [T, N]
 * fp32 (tensor cores, fp32 accumulation). d a multiple of 64. err_word: a
 * device int32 that receives a nonzero code on a device timeout (may be NULL). */
moe_status moe_router_logits(const uint16_t* x, const uint16_t* w_router, int64_t T, int d, int N,
                             float* logits, int32_t* err_word, void* stream);

/* Router GEMM with the elbow routing fused into its epilogue (the layer's
 * first stage; Sec. 2, Alg. 1 and Sec. 2.1): the same logits as
 * moe_router_logits, routed exactly as
 * elbow_route routes them. logits_out [T, N] may be NULL (the logits then stay
 * on chip). chunk_counts [N][ceil(T/128)] int32 (may be NULL): the number of
 * selected pairs of each expert in each chunk of 128 tokens. */
moe_status moe_router_route(const uint16_t* x, const uint16_t* w_router, int64_t T, int d, int N,
                            const moe_route_params* rp, float* logits_out, int32_t* k_out,
                            int32_t* ids_out, float* gates_out, int32_t* chunk_counts,
                            int32_t* err_word, void* stream);

/* moe_expert_gate_up with the rows gathered from x [T, d] by perm (row r of
 * expert e is token perm[r]), without a gathered copy of x (App. A.4: each
 * expert applies its MLP to the tokens routed to it). */
moe_status moe_expert_gate_up_gathered(const uint16_t* x, int64_t T, const int32_t* perm,
                                       const uint16_t* w_gate_up, const int32_t* offsets,
                                       const int32_t* tile_off, int64_t P, int d, int N, int I,
                                       uint16_t* h, int32_t* err_word, void* stream);

/* Expert SwiGLU over dispatched rows (the expert MLP of App. A.4, in the
 * SwiGLU form of the OLMoE experts): for each expert e and each row r in
 * [offsets[e], offsets[e+1]): h[r] = silu(W_gate[e] xs[r]) * (W_up[e] xs[r]),
 * with xs [P, d] bf16 the tokens already gathered in dispatch order (P = the
 * row capacity, >= offsets[N]), h [P, I] bf16. `tile_off` [N + 1] int32 are
 * the exclusive prefix sums of ceil(count_e / 128) (moe_dispatch's workspace
 * holds them; see moe_dispatch_tile_offsets). */
moe_status moe_expert_gate_up(const uint16_t* xs, const uint16_t* w_gate_up, const int32_t* offsets,
                              const int32_t* tile_off, int64_t P, int d, int N, int I, uint16_t* h,
                              int32_t* err_word, void* stream);

/* Expert down projection (the second matrix of the expert MLP, App. A.4):
 * o[r] = W_down[e] h[r] for rows of expert e;
 * h [P, I] bf16 -> o [P, d] bf16. d a multiple of 128 (256-column output
 * tiles when d is a multiple of 256, else 128-column tiles), I of 64. */
moe_status moe_expert_down(const uint16_t* h, const uint16_t* w_down, const int32_t* offsets,
                           const int32_t* tile_off, int64_t P, int d, int N, int I, uint16_t* o,
                           int32_t* err_word, void* stream);

/* Decode-shaped expert contractions (App. A.4, in the small-batch latency
 * regime of Sec. 3) for batches of T <= 64 tokens, where an
 * expert has at most T rows (a token selects an expert at most once): the
 * same results as moe_expert_gate_up and moe_expert_down, computed with the
 * weights as the M operand (128 weight rows per tile, the expert's rows as N,
 * in a 16-, 32- or 64-column tile for T <= 16, <= 32, <= 64), so a tile
 * streams weights instead of a mostly empty 128-row token block.
 * moe_layer_forward takes this path by itself when 3 <= T <= 64. T is the token
 * count the rows came from (T > 64: MOE_ERR_UNSUPPORTED; rows of an expert
 * past T are not computed); xs [P, d] holds the dispatched rows
 * (moe_gather_rows), offsets [N + 1] the expert row offsets. I a multiple of
 * 64; d a multiple of 64 (gate/up) or 128 (down). */
moe_status moe_expert_gate_up_decode(const uint16_t* xs, const uint16_t* w_gate_up,
                                     const int32_t* offsets, int64_t T, int64_t P, int d, int N,
                                     int I, uint16_t* h, int32_t* err_word, void* stream);
moe_status moe_expert_down_decode(const uint16_t* h, const uint16_t* w_down, const int32_t* offsets,
                                  int64_t T, int64_t P, int d, int N, int I, uint16_t* o,
                                  int32_t* err_word, void* stream);

/* The expert contractions for batches of T <= 4 tokens (the expert MLP of
 * App. A.4 in the one-token latency regime of Sec. 3) on CUDA cores.
 * moe_layer_forward runs the same items, both contractions and the combine,
 * in one cooperative kernel for steps of T <= 2 tokens (d, I <= 4096; from
 * three tokens on the tensor-core decode tiles are faster): an expert then
 * has at most T rows, so its contraction is a few matrix-vector products that
 * spread the expert's weight rows over many blocks. The same results as
 * moe_expert_gate_up / moe_expert_down within fp32 accumulation (another
 * summation order), with the token rows read from x [T, d] through perm (row p
 * of expert e, p in [offsets[e], offsets[e+1]), is token perm[p]; no gathered
 * copy):
 *   moe_expert_gate_up_gemv: h [P, I] = silu(W_gate[e] x[perm[p]]) * (W_up[e] x[perm[p]])
 *   moe_expert_down_gemv:    o [P, d] = W_down[e] h[p]
 * K bounds the experts with rows (at most min(N, T * K)). T <= 4, d and I
 * multiples of 8 and at most 4096 (else MOE_ERR_UNSUPPORTED); x, h (for the
 * down step) and the weights 16-byte aligned. Rows of an expert past T or P
 * are not computed; tokens outside [0, T) are clamped into it. Each block
 * brings its weight rows into shared memory with bulk copies whose wait is
 * bounded: a block that gives up writes a nonzero code into err_word (device
 * int32, may be NULL) and leaves its outputs unwritten. */
moe_status moe_expert_gate_up_gemv(const uint16_t* x, int64_t T, const int32_t* perm,
                                   const int32_t* offsets, const uint16_t* w_gate_up, int64_t P,
                                   int d, int N, int I, int K, uint16_t* h, int32_t* err_word,
                                   void* stream);
moe_status moe_expert_down_gemv(const uint16_t* h, const int32_t* offsets, const uint16_t* w_down,
                                int64_t T, int64_t P, int d, int N, int I, int K, uint16_t* o,
                                int32_t* err_word, void* stream);

/* Device pointer, inside a moe_dispatch workspace, of the [N + 1] int32 tile
 * offsets (exclusive prefix sums of ceil(count_e / 128)) that the last
 * moe_dispatch on that workspace wrote. No counterpart in the paper (the
 * expert GEMMs' tile schedule). NULL for a NULL ws or unsupported N. */
const int32_t* moe_dispatch_tile_offsets(const void* ws, int64_t T, int N, int K);

/* Device pointer, inside a moe_dispatch workspace, of the [N][ceil(T/128)]
 * int32 per-chunk expert counts: pass it as moe_router_route's chunk_counts,
 * then call moe_dispatch_counted, which skips its own counting pass. The
 * first pass of the dispatch (App. A.4); NULL for a NULL ws or unsupported N. */
int32_t* moe_dispatch_chunk_counts(void* ws, int64_t T, int N, int K);

/* moe_dispatch (App. A.4) whose per-chunk expert counts are already in the
 * workspace (written there by moe_router_route or elbow_route_with_counts);
 * otherwise identical, errors included. */
moe_status moe_dispatch_counted(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                                int32_t* offsets, int32_t* perm, int32_t* pair_pos, void* ws,
                                size_t ws_bytes, void* stream);

/* Gather rows (sending each token to its experts, App. A.4):
 * xs[r] = x[perm[r]] for r < offsets[N] (x [T, d] bf16,
 * xs [P, d] bf16, P >= offsets[N]). Rows stop at P and tokens outside [0, T)
 * are clamped into it, so inconsistent arguments cannot reach outside x or
 * xs. */
moe_status moe_gather_rows(const uint16_t* x, const int32_t* perm, const int32_t* offsets, int64_t T,
                           int64_t P, int d, int N, uint16_t* xs, void* stream);

/* Combine (the gate-weighted sum of the selected experts' outputs that the MoE
 * block returns, Sec. 1 and App. A.4):
 * y_t = sum_{s < k_t} gates[t,s] * o[pair_pos[t,s]] (+ residual_t),
 * fp32 in s order, rounded to bf16. o [P, d] bf16; residual may be NULL.
 * Positions are clamped to the T * K rows of o. */
moe_status moe_combine(const uint16_t* o, const int32_t* k, const int32_t* pair_pos,
                       const float* gates, const uint16_t* residual, int64_t T, int d, int K,
                       uint16_t* y, void* stream);

/*
 * elbow_route_randomized - the tail-randomisation experiment of Sec. 2.2,
 * which keeps K experts per token but replaces part of the elbow-K selection
 * by random experts:
 *   rp->mode MOE_ROUTE_RAND_TAIL: slots s < k keep ranks 0..k-1 (k the elbow
 *     count of elbow_route); each slot s in [k, K) gets an expert drawn
 *     without replacement from those of rank >= k;
 *   rp->mode MOE_ROUTE_RAND_HEAD: slots s in [k, K) keep ranks k..K-1; each
 *     slot s < k gets an expert drawn without replacement from those of
 *     rank >= K.
 *   rand      [T, K] uint32   caller's random numbers; slot s of token t takes,
 *                             among the remaining experts in ascending id
 *                             order, the one at index rand[t, s] mod (number
 *                             remaining); slots that keep their rank ignore it
 *   k_out     [T]             K (every slot is used)
 *   ids_out, gates_out [T, K] the K experts and their own probabilities p
 *                             (renorm: divided by the sum over the K slots)
 * Routing arithmetic as elbow_route. Errors as elbow_route; rand NULL or a
 * mode other than the two above: MOE_ERR_INVALID_ARG. Pointers 4-byte
 * aligned (logits 16-byte).
 */
moe_status elbow_route_randomized(const float* logits, int64_t T, int N, const moe_route_params* rp,
                                  const uint32_t* rand, int32_t* k_out, int32_t* ids_out,
                                  float* gates_out, void* stream);

/* Bounds-check report of the debug build (the library compiled with
 * -DELBOW_MOE_DEBUG, paper_2608_04401_gb300.buildlib.build(debug=True), which
 * stands in for compute-sanitizer; no counterpart in the paper). In that build
 * every index a kernel takes from its inputs (k_t <= K, expert ids < N,
 * expert offsets and m-tile offsets consistent and within the row capacity,
 * permutation entries and token rows within [0, T), pair positions within
 * [0, T * K), finite logits) is checked on the device; a failed check counts
 * one violation and the kernel goes on with the clamp or skip of the release
 * build (it never traps). This call SYNCHRONISES the device, writes the
 * number of violations counted since the previous call into *out and resets
 * the count. Release build: *out = 0 and MOE_ERR_UNSUPPORTED. */
moe_status moe_debug_violations(uint32_t* out);

/* Self-check of the quotients the routing divides with (the softmax
 * p_j = e_j / s of Sec. 2 and Alg. 1's normalisation p'_i = (p_(i) - p_min) /
 * den, each a correctly rounded quotient): for i < n, out[3i] = the routing's
 * quotient a_i / b_i (one reciprocal per divisor, then Markstein's fused
 * multiply-add correction), out[3i + 1] = the same from the packed two-lane
 * form, out[3i + 2] = CUDA's __fdiv_rn(a_i, b_i). All three must be equal for
 * a_i >= 0 and b_i in [2^-32, 2^8]. a, b [n] and out [3n] fp32 device arrays,
 * 4-byte aligned; 0 <= n <= 2^30 (else MOE_ERR_INVALID_ARG). */
moe_status moe_check_quotients(const float* a, const float* b, int64_t n, float* out,
                               void* stream);

/* Exercises the bounded wait that every GEMM pipeline uses, on an mbarrier
 * that nothing arrives on: the kernel gives up after `seconds` (0 < seconds
 * <= 10) and writes the timeout code into err_word (device, 4-byte aligned;
 * cleared first), exactly as a GEMM whose producer never delivered would.
 * moe_read_device_error(err_word, stream) then returns MOE_ERR_DEVICE_TIMEOUT
 * and the context stays usable. */
moe_status moe_check_bounded_wait(int32_t* err_word, double seconds, void* stream);

/*
 * moe_route_diagnostics - routing diagnostics of Sec. 2.3 (elbow angle),
 * Sec. 2.4 and App. A.3 (expert-load changes of elbow-K against top-K).
 *
 * Per token, the whole sorted curve is evaluated with the fp32 steps of
 * elbow_route; e is the UNCAPPED elbow index (first argmax of D over all N
 * ranks, so k = min(e + 1, K)), and the elbow angle theta is the angle at the
 * elbow point (x'_e, 1 - p'_e) between the first (0,0) and the last (1,1)
 * point of the normalised curve, evaluated in fp64 and rounded to fp32
 * degrees (180 when the elbow is an end point).
 *
 *   logits     [T, N] fp32   router logits
 *   rp         K and eps are used; mode and renorm are ignored
 *   elbow_out  [T] int32     e per token (may be NULL)
 *   theta_out  [T] fp32      theta per token, degrees (may be NULL)
 *   diag       device pointer to one moe_route_diag, overwritten (8-byte
 *              aligned): integer histograms of the batch, and the normalised
 *              utilisations q = L / sum(L) of both selections reduced to
 *              delta = 1 - E[k]/K, the l1 change (bound 2 delta / (1 - delta),
 *              Theorem 1), the change of the largest share (Corollary 1, same
 *              bound), the change of CV^2 = N |q|^2 - 1 (bound
 *              2 N delta / (1 - delta)^2, Corollary 2), and the percentage
 *              changes of the top-1 share and of CV (Sec. 2.4).
 * Integer counts make every field independent of block order. Errors as
 * elbow_route; diag NULL or misaligned: MOE_ERR_INVALID_ARG.
 */
#define MOE_DIAG_MAX_N 128
typedef struct {
  int64_t tokens;                        /* T */
  int64_t sharp_elbows;                  /* tokens with theta <= 135 degrees */
  int64_t k_hist[9];                     /* tokens with k = 0..8 */
  int64_t elbow_hist[MOE_DIAG_MAX_N];    /* tokens with uncapped elbow index e */
  int64_t theta_hist[181];               /* tokens with floor(theta) = 0..180 */
  int64_t load_top[MOE_DIAG_MAX_N];      /* selected pairs per expert, top-K */
  int64_t load_elb[MOE_DIAG_MAX_N];      /* selected pairs per expert, elbow-K */
  double mean_k;                         /* E[k] */
  double delta;                          /* 1 - E[k] / K */
  double l1, l1_bound;                   /* |q_elb - q_top|_1 and 2 delta / (1 - delta) */
  double top1_change;                    /* | max q_elb - max q_top | */
  double cv2_change, cv2_bound;          /* |CV^2 change| and 2 N delta / (1 - delta)^2 */
  double top1_share_change_pct;          /* (max q_top - max q_elb) / max q_top * 100 */
  double cv_change_pct;                  /* (CV_top - CV_elb) / CV_top * 100 */
} moe_route_diag;

moe_status moe_route_diagnostics(const float* logits, int64_t T, int N, const moe_route_params* rp,
                                 int32_t* elbow_out, float* theta_out, moe_route_diag* diag,
                                 void* stream);

#ifdef __cplusplus
}
#endif

#endif /* ELBOW_MOE_H */
