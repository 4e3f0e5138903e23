// C ABI of the elbow-routed MoE layer: argument validation, the workspace
// layout, and the launch sequence of the layer forward. No allocation, no
// stream synchronisation (moe_read_device_error excepted, as documented).
#include <cstring>

#include "common.cuh"

namespace moe {
cudaError_t launch_elbow_route(const float* logits, int64_t T, int N, int K, float eps,
                               int topk_mode, int renorm, int32_t* k_out, int32_t* ids_out,
                               float* gates_out, int32_t* blk_cnt, const uint32_t* rand,
                               int rand_mode, cudaStream_t stream);
size_t dispatch_ws_bytes(int64_t T, int N);
int32_t* dispatch_tile_off(void* ws, int64_t T, int N);
int32_t* dispatch_counts(void* ws);
cudaError_t launch_dispatch(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                            int32_t* offsets, int32_t* perm, int32_t* pair_pos, void* ws,
                            int32_t* offsets_copy, bool counts_ready, int32_t* err,
                            unsigned int* arrive, cudaStream_t stream);
cudaError_t launch_dispatch_gather(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                                   int32_t* offsets, int32_t* perm, int32_t* pair_pos, void* ws,
                                   int32_t* offsets_copy, const uint16_t* x, int d, uint16_t* xs,
                                   int num_sms, cudaStream_t stream);
cudaError_t launch_gather(const uint16_t* x, int64_t T, const int32_t* perm, const int32_t* offsets,
                          int N, int64_t P, int d, uint16_t* xs, int num_sms, cudaStream_t stream);
cudaError_t launch_combine(const uint16_t* o, const int32_t* k, const int32_t* pair_pos,
                           const float* gates, const uint16_t* residual, int64_t T, int d, int K,
                           uint16_t* y, int num_sms, cudaStream_t stream);
cudaError_t launch_router_gemm(const uint16_t* x, const uint16_t* wr, int64_t T, int d, int N,
                               float* logits, int32_t* err, int num_sms, cudaStream_t stream);
cudaError_t launch_gateup_gemm(const uint16_t* xs, const uint16_t* wgu, const int32_t* offsets,
                               const int32_t* tile_off, int64_t P, int d, int N, int I, uint16_t* h,
                               int32_t* err, int num_sms, cudaStream_t stream);
cudaError_t launch_down_gemm(const uint16_t* h, const uint16_t* wd, const int32_t* offsets,
                             const int32_t* tile_off, int64_t P, int d, int N, int I, uint16_t* o,
                             int32_t* err, int num_sms, cudaStream_t stream);
cudaError_t launch_router_route(const uint16_t* x, const uint16_t* wr, int64_t T, int d, int N,
                                int K, float eps, int topk_mode, int renorm, float* logits_out,
                                int32_t* k_out, int32_t* ids_out, float* gates_out,
                                int32_t* blk_cnt, int32_t* err, int num_sms, cudaStream_t stream);
cudaError_t launch_gateup_decode_gemm(const uint16_t* xs, const uint16_t* wgu,
                                      const int32_t* offsets, int64_t P, int64_t max_rows, int d,
                                      int N, int I, uint16_t* h, int32_t* err, int num_sms,
                                      cudaStream_t stream);
cudaError_t launch_down_decode_gemm(const uint16_t* h, const uint16_t* wd, const int32_t* offsets,
                                    int64_t P, int64_t max_rows, int d, int N, int I, uint16_t* o,
                                    int32_t* err, int num_sms, cudaStream_t stream);
cudaError_t launch_gateup_gather_gemm_pair(const uint16_t* x, int64_t T, const int32_t* perm,
                                           const uint16_t* wgu, const int32_t* offsets, int64_t P,
                                           int d, int N, int I, uint16_t* h, int32_t* err,
                                           int num_sms, cudaStream_t stream);
cudaError_t launch_down_gemm_pair(const uint16_t* h, const uint16_t* wd, const int32_t* offsets,
                                  int64_t P, int d, int N, int I, uint16_t* o, int32_t* err,
                                  int num_sms, cudaStream_t stream);
cudaError_t launch_gate_up_gemv(const uint16_t* x, int64_t T, const int32_t* perm,
                                const int32_t* offsets, const uint16_t* wgu, int64_t P, int d,
                                int N, int I, int K, uint16_t* h, int32_t* err,
                                cudaStream_t stream);
cudaError_t launch_down_gemv(const uint16_t* h, const int32_t* offsets, const uint16_t* wd,
                             int64_t T, int64_t P, int d, int N, int I, int K, uint16_t* o,
                             int32_t* err, cudaStream_t stream);
cudaError_t launch_route_warp(const float* logits, int64_t T, int N, int K, float eps,
                              int topk_mode, int renorm, int32_t* k_out, int32_t* ids_out,
                              float* gates_out, cudaStream_t stream);
cudaError_t launch_router_small_route(const uint16_t* x, const uint16_t* w_router, int T, int d,
                                      int N, float* partial, unsigned int* ticket, int K, float eps,
                                      int topk_mode, int renorm, float* logits_out, int32_t* k_out,
                                      int32_t* ids_out, float* gates_out, cudaStream_t stream);
cudaError_t launch_router_few(const uint16_t* x, const uint16_t* w_router, int T, int d, int N,
                              int K, float eps, int topk_mode, int renorm, float* logits_out,
                              int32_t* k_out, int32_t* ids_out, float* gates_out, int32_t* offsets,
                              int32_t* perm, int32_t* pair_pos, int32_t* offsets_copy,
                              int32_t* clear, int nclear, cudaStream_t stream);
cudaError_t launch_expert_few_gemv(const uint16_t* x, int64_t T, const int32_t* perm,
                                   const int32_t* offsets, const uint16_t* wgu, const uint16_t* wd,
                                   int64_t P, int d, int N, int I, int K, uint16_t* h, uint16_t* o,
                                   int32_t* err, unsigned int* done, const int32_t* k,
                                   const int32_t* pair_pos, const float* gates,
                                   const uint16_t* residual, uint16_t* y, unsigned int* tickets,
                                   int num_sms, cudaStream_t stream);
cudaError_t launch_quotient_check(const float* a, const float* b, int64_t n, float* out,
                                  cudaStream_t stream);
cudaError_t launch_route_diagnostics(const float* logits, int64_t T, int N, int K, float eps,
                                     int32_t* elbow_out, float* theta_out, moe_route_diag* dg,
                                     cudaStream_t stream);
#ifdef ELBOW_MOE_DEBUG
cudaError_t debug_take_route(unsigned int* out);
cudaError_t debug_take_route_warp(unsigned int* out);
cudaError_t debug_take_dispatch(unsigned int* out);
cudaError_t debug_take_gemm(unsigned int* out);
cudaError_t debug_take_gemm2(unsigned int* out);
cudaError_t debug_take_gemv(unsigned int* out);
cudaError_t debug_take_diag(unsigned int* out);
#endif
}  // namespace moe

namespace {

// The bounded wait of the GEMM pipelines on an mbarrier that nothing arrives
// on: thread 0 gives up after limit_ns and writes the timeout code into *err.
__global__ void bounded_wait_check_kernel(int32_t* err, uint64_t limit_ns) {
  __shared__ alignas(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    moe::mbar_init(moe::smem_u32(&bar), 1);
    abort_flag = 0;
    moe::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 &&
      !moe::mbar_wait_bounded(moe::smem_u32(&bar), 0u, &abort_flag, limit_ns))
    atomicExch(err, moe::kDevErrTimeout);
}

// T < 2^28 keeps the pair counts and positions (up to T * K <= 2^31 - 8) in int32
constexpr int64_t kMaxTokens = (int64_t(1) << 28) - 1;
constexpr int kMaxDim = 16384;
// Batches of at most this many tokens take the decode-shaped expert GEMMs
// (weights as the M operand; every expert then has at most 64 rows).
constexpr int64_t kDecodeMaxTokens = 64;
// Batches of at most this many tokens route with one warp per token, after a
// router GEMM split over d (below it the fused router's one-thread-per-token
// routing chain dominates; above it the fused router is faster).
constexpr int64_t kWarpRouteMaxTokens = 16;
// Layer batches of at most this many tokens take the router GEMM split over d
// and over 16-token groups (each block a 64-column slice of one group; the
// last block of a group routes it, one warp per token) instead of the
// tensor-core router, whose single 128-row tile would stream all of x and W_r
// through one SM.
constexpr int64_t kSmallRouterMaxTokens = 64;
// The CUDA-core expert contractions take batches of at most kGemvMaxTokens
// tokens (d, I at most kGemvMaxDim). Layer steps of at most
// kGemvLayerMaxTokens tokens run as three kernels: the few-token cluster
// router (routing, dispatch, clearing the step's counters), then the expert
// MLP and combine in one cooperative kernel, which spreads each touched
// expert's weight rows over all SMs instead of paying the tensor-core decode
// tiles' fixed latency. Measured per step in graphs of 16 steps
// (d = 2048, N = 64, I = 1024): one token 15.3 us with two experts and 27.6
// us with eight (the tensor-core path 17.8 and 35.4), two tokens 32.7 and
// 50.6 us (38.9 and 59.8); from three tokens on the tensor-core tiles are
// faster (61.3 against 66.7 us).
constexpr int64_t kGemvMaxTokens = 4;
constexpr int64_t kGemvLayerMaxTokens = 2;
static_assert(kGemvLayerMaxTokens <= 4, "the few-token router serves the CUDA-core path");
constexpr int kGemvMaxDim = 4096;
constexpr int kSmallRouterSlice = 64;

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
// 4-byte alignment of int32 / fp32 arrays (a null pointer passes: optional
// arguments are checked for null separately)
bool aligned4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }

size_t up256(size_t b) { return (b + 255) & ~static_cast<size_t>(255); }

// SM count of the current device, or 0 if it cannot be queried (the entry
// points then return MOE_ERR_CUDA).
int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
    return 0;
  return n;
}

moe_status cuda_status(cudaError_t e) { return e == cudaSuccess ? MOE_OK : MOE_ERR_CUDA; }

// The prefill expert GEMMs: two-CTA (M = 256) tiles; the down projection needs
// d a multiple of 256 for them (else one-CTA 128-column tiles).
cudaError_t gate_up_gathered(const uint16_t* x, int64_t T, const int32_t* perm, const uint16_t* wgu,
                             const int32_t* offsets, const int32_t* tile_off, int64_t P, int d,
                             int N, int I, uint16_t* h, int32_t* err, int nsm, cudaStream_t s) {
  (void)tile_off;  // the two-CTA kernel derives its 256-row tiles from the offsets
  return moe::launch_gateup_gather_gemm_pair(x, T, perm, wgu, offsets, P, d, N, I, h, err, nsm, s);
}
cudaError_t expert_down(const uint16_t* h, const uint16_t* wd, const int32_t* offsets,
                        const int32_t* tile_off, int64_t P, int d, int N, int I, uint16_t* o,
                        int32_t* err, int nsm, cudaStream_t s) {
  if (d % 256 == 0)
    return moe::launch_down_gemm_pair(h, wd, offsets, P, d, N, I, o, err, nsm, s);
  return moe::launch_down_gemm(h, wd, offsets, tile_off, P, d, N, I, o, err, nsm, s);
}

moe_status check_route_params(const moe_route_params* rp, int N) {
  if (!rp) return MOE_ERR_INVALID_ARG;
  if (rp->mode != MOE_ROUTE_ELBOW && rp->mode != MOE_ROUTE_TOPK) return MOE_ERR_INVALID_ARG;
  if (rp->renorm != 0 && rp->renorm != 1) return MOE_ERR_INVALID_ARG;
  if (!(rp->eps >= 0.0f) || rp->eps > 1.0f) return MOE_ERR_INVALID_ARG;
  if (rp->K < 1 || rp->K > 8 || rp->K > N) return MOE_ERR_UNSUPPORTED;
  return MOE_OK;
}

bool supported_n(int N) { return N == 64 || N == 128; }

// Layer workspace layout (every region 256-byte aligned):
//   header (error word) | k [T] | ids [T,K] | gates [T,K] | offsets [N+1]
//   | dispatch scratch | perm [T*K] | pair_pos [T*K] | h [T*K, I] bf16
//   | o [T*K, d] bf16
struct LayerWs {
  int32_t* err;
  int32_t* k;
  int32_t* ids;
  float* gates;
  int32_t* offsets;
  void* disp;
  int32_t* perm;
  int32_t* pair_pos;
  uint16_t* h;
  uint16_t* o;
  float* partial;  // decode-sized batches: router partial sums [d/64][T][N]
  unsigned int* tickets;  // few-token steps: the combine's counters [ceil(d/16)], after err,
                          // then the expert kernel's 32 completion counters
  size_t bytes;
};

LayerWs layer_ws(void* base, int64_t T, int d, int N, int I, int K) {
  LayerWs w{};
  char* p = static_cast<char*>(base);
  size_t off = 0;
  auto take = [&](size_t b) {
    char* q = p ? p + off : nullptr;
    off += up256(b);
    return q;
  };
  const size_t P = static_cast<size_t>(T) * K;
  w.err = reinterpret_cast<int32_t*>(take(256));
  w.tickets = reinterpret_cast<unsigned int*>(take(sizeof(unsigned int) * ((d + 15) / 16 + 32)));
  w.k = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * T));
  w.ids = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * P));
  w.gates = reinterpret_cast<float*>(take(sizeof(float) * P));
  w.offsets = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * (N + 1)));
  w.disp = take(moe::dispatch_ws_bytes(T, N));
  w.perm = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * (P > 0 ? P : 1)));
  w.pair_pos = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * (P > 0 ? P : 1)));
  w.h = reinterpret_cast<uint16_t*>(take(sizeof(uint16_t) * P * I));
  w.o = reinterpret_cast<uint16_t*>(take(sizeof(uint16_t) * P * d));
  w.partial = reinterpret_cast<float*>(
      take(T <= kSmallRouterMaxTokens
               ? sizeof(float) * static_cast<size_t>(d / kSmallRouterSlice) * T * N
               : 0));
  w.bytes = off;
  return w;
}

}  // namespace

extern "C" {

const char* moe_status_string(moe_status s) {
  switch (s) {
    case MOE_OK: return "MOE_OK";
    case MOE_ERR_INVALID_ARG: return "MOE_ERR_INVALID_ARG: null/misaligned pointer or bad parameter";
    case MOE_ERR_UNSUPPORTED: return "MOE_ERR_UNSUPPORTED: shape outside the supported set";
    case MOE_ERR_WORKSPACE: return "MOE_ERR_WORKSPACE: workspace missing or too small";
    case MOE_ERR_CUDA: return "MOE_ERR_CUDA: a CUDA call failed";
    case MOE_ERR_DEVICE_TIMEOUT: return "MOE_ERR_DEVICE_TIMEOUT: a kernel gave up a bounded wait";
  }
  return "unknown moe_status";
}

moe_status elbow_route(const float* logits, int64_t T, int N, const moe_route_params* rp,
                       int32_t* k_out, int32_t* ids_out, float* gates_out, void* stream) {
  if (T < 0 || T > kMaxTokens) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N)) return MOE_ERR_UNSUPPORTED;
  moe_status st = check_route_params(rp, N);
  if (st != MOE_OK) return st;
  if (T == 0) return MOE_OK;
  if (!logits || !k_out || !ids_out || !gates_out) return MOE_ERR_INVALID_ARG;
  if (!aligned16(logits) || !aligned16(ids_out) || !aligned16(gates_out) ||
      (reinterpret_cast<uintptr_t>(k_out) & 3u))
    return MOE_ERR_INVALID_ARG;
  if (T <= kWarpRouteMaxTokens)  // a few tokens: one warp each has the shorter critical path
    return cuda_status(moe::launch_route_warp(logits, T, N, rp->K, rp->eps,
                                              rp->mode == MOE_ROUTE_TOPK, rp->renorm, k_out,
                                              ids_out, gates_out,
                                              static_cast<cudaStream_t>(stream)));
  return cuda_status(moe::launch_elbow_route(logits, T, N, rp->K, rp->eps, rp->mode == MOE_ROUTE_TOPK,
                                             rp->renorm, k_out, ids_out, gates_out, nullptr,
                                             nullptr, 0, static_cast<cudaStream_t>(stream)));
}

moe_status elbow_route_warp(const float* logits, int64_t T, int N, const moe_route_params* rp,
                            int32_t* k_out, int32_t* ids_out, float* gates_out, void* stream) {
  if (T < 0 || T > kMaxTokens) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N)) return MOE_ERR_UNSUPPORTED;
  moe_status st = check_route_params(rp, N);
  if (st != MOE_OK) return st;
  if (T == 0) return MOE_OK;
  if (!logits || !k_out || !ids_out || !gates_out) return MOE_ERR_INVALID_ARG;
  if (!aligned16(logits) || (reinterpret_cast<uintptr_t>(ids_out) & 3u) ||
      (reinterpret_cast<uintptr_t>(gates_out) & 3u) || (reinterpret_cast<uintptr_t>(k_out) & 3u))
    return MOE_ERR_INVALID_ARG;
  return cuda_status(moe::launch_route_warp(logits, T, N, rp->K, rp->eps,
                                            rp->mode == MOE_ROUTE_TOPK, rp->renorm, k_out, ids_out,
                                            gates_out, static_cast<cudaStream_t>(stream)));
}

moe_status elbow_route_randomized(const float* logits, int64_t T, int N, const moe_route_params* rp,
                                  const uint32_t* rand, int32_t* k_out, int32_t* ids_out,
                                  float* gates_out, void* stream) {
  if (T < 0 || T > kMaxTokens) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N)) return MOE_ERR_UNSUPPORTED;
  if (!rp || (rp->mode != MOE_ROUTE_RAND_TAIL && rp->mode != MOE_ROUTE_RAND_HEAD))
    return MOE_ERR_INVALID_ARG;
  moe_route_params base = *rp;
  base.mode = MOE_ROUTE_ELBOW;
  moe_status st = check_route_params(&base, N);
  if (st != MOE_OK) return st;
  if (T == 0) return MOE_OK;
  if (!logits || !rand || !k_out || !ids_out || !gates_out) return MOE_ERR_INVALID_ARG;
  if (!aligned16(logits) || (reinterpret_cast<uintptr_t>(rand) & 3u) ||
      (reinterpret_cast<uintptr_t>(k_out) & 3u) || (reinterpret_cast<uintptr_t>(ids_out) & 3u) ||
      (reinterpret_cast<uintptr_t>(gates_out) & 3u))
    return MOE_ERR_INVALID_ARG;
  return cuda_status(moe::launch_elbow_route(logits, T, N, rp->K, rp->eps, 0, rp->renorm, k_out,
                                             ids_out, gates_out, nullptr, rand, rp->mode,
                                             static_cast<cudaStream_t>(stream)));
}

moe_status moe_route_diagnostics(const float* logits, int64_t T, int N, const moe_route_params* rp,
                                 int32_t* elbow_out, float* theta_out, moe_route_diag* diag,
                                 void* stream) {
  if (T < 0 || T > kMaxTokens) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N)) return MOE_ERR_UNSUPPORTED;
  moe_status st = check_route_params(rp, N);
  if (st != MOE_OK) return st;
  if (!diag || (reinterpret_cast<uintptr_t>(diag) & 7u)) return MOE_ERR_INVALID_ARG;
  if (T > 0 && (!logits || !aligned16(logits))) return MOE_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(elbow_out) & 3u) || (reinterpret_cast<uintptr_t>(theta_out) & 3u))
    return MOE_ERR_INVALID_ARG;
  return cuda_status(moe::launch_route_diagnostics(logits, T, N, rp->K, rp->eps, elbow_out,
                                                   theta_out, diag,
                                                   static_cast<cudaStream_t>(stream)));
}

moe_status elbow_route_with_counts(const float* logits, int64_t T, int N,
                                   const moe_route_params* rp, int32_t* k_out, int32_t* ids_out,
                                   float* gates_out, int32_t* chunk_counts, void* stream) {
  if (T < 0 || T > kMaxTokens) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N)) return MOE_ERR_UNSUPPORTED;
  moe_status st = check_route_params(rp, N);
  if (st != MOE_OK) return st;
  if (T == 0) return MOE_OK;
  if (!logits || !k_out || !ids_out || !gates_out || !chunk_counts) return MOE_ERR_INVALID_ARG;
  if (!aligned16(logits) || !aligned16(ids_out) || !aligned16(gates_out) ||
      (reinterpret_cast<uintptr_t>(k_out) & 3u) || (reinterpret_cast<uintptr_t>(chunk_counts) & 3u))
    return MOE_ERR_INVALID_ARG;
  return cuda_status(moe::launch_elbow_route(logits, T, N, rp->K, rp->eps, rp->mode == MOE_ROUTE_TOPK,
                                             rp->renorm, k_out, ids_out, gates_out, chunk_counts,
                                             nullptr, 0, static_cast<cudaStream_t>(stream)));
}

size_t moe_dispatch_workspace_size(int64_t T, int N, int K) {
  (void)K;
  if (T < 0 || T > kMaxTokens || !supported_n(N)) return 0;
  return moe::dispatch_ws_bytes(T, N);
}

const int32_t* moe_dispatch_tile_offsets(const void* ws, int64_t T, int N, int K) {
  (void)K;
  if (!ws || T < 0 || !supported_n(N)) return nullptr;
  return moe::dispatch_tile_off(const_cast<void*>(ws), T, N);
}

int32_t* moe_dispatch_chunk_counts(void* ws, int64_t T, int N, int K) {
  (void)T;
  (void)K;
  if (!ws || !supported_n(N)) return nullptr;
  return moe::dispatch_counts(ws);
}

moe_status moe_dispatch_counted(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                                int32_t* offsets, int32_t* perm, int32_t* pair_pos, void* ws,
                                size_t ws_bytes, void* stream) {
  if (T < 0 || T > kMaxTokens) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N) || K < 1 || K > 8 || K > N) return MOE_ERR_UNSUPPORTED;
  if (!offsets || !ws) return MOE_ERR_INVALID_ARG;
  if (T > 0 && (!k || !ids || !perm || !pair_pos)) return MOE_ERR_INVALID_ARG;
  if (ws_bytes < moe::dispatch_ws_bytes(T, N)) return MOE_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u)) return MOE_ERR_INVALID_ARG;
  if (T > 0 && !aligned16(ids)) return MOE_ERR_INVALID_ARG;
  if (!aligned4(k) || !aligned4(offsets) || !aligned4(perm) || !aligned4(pair_pos))
    return MOE_ERR_INVALID_ARG;
  return cuda_status(moe::launch_dispatch(k, ids, T, N, K, offsets, perm, pair_pos, ws, nullptr,
                                          true, nullptr, nullptr,
                                          static_cast<cudaStream_t>(stream)));
}

moe_status moe_dispatch(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                        int32_t* offsets, int32_t* perm, int32_t* pair_pos, void* ws,
                        size_t ws_bytes, void* stream) {
  if (T < 0 || T > kMaxTokens) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N) || K < 1 || K > 8 || K > N) return MOE_ERR_UNSUPPORTED;
  if (!offsets || !ws) return MOE_ERR_INVALID_ARG;
  if (T > 0 && (!k || !ids || !perm || !pair_pos)) return MOE_ERR_INVALID_ARG;
  if (ws_bytes < moe::dispatch_ws_bytes(T, N)) return MOE_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u)) return MOE_ERR_INVALID_ARG;
  if (T > 0 && !aligned16(ids)) return MOE_ERR_INVALID_ARG;
  if (!aligned4(k) || !aligned4(offsets) || !aligned4(perm) || !aligned4(pair_pos))
    return MOE_ERR_INVALID_ARG;
  return cuda_status(moe::launch_dispatch(k, ids, T, N, K, offsets, perm, pair_pos, ws, nullptr,
                                          false, nullptr, nullptr,
                                          static_cast<cudaStream_t>(stream)));
}

size_t moe_layer_workspace_size(int64_t T, int d, int N, int I, int K) {
  if (T < 0 || T > kMaxTokens || d <= 0 || d > kMaxDim || I <= 0 || I > kMaxDim || K < 1 ||
      K > 8 || !supported_n(N))
    return 0;
  return layer_ws(nullptr, T, d, N, I, K).bytes;
}

moe_status moe_layer_forward(const uint16_t* x, const uint16_t* w_router, const uint16_t* w_gate_up,
                             const uint16_t* w_down, int64_t T, int d, int N, int I,
                             const moe_route_params* rp, const uint16_t* residual, uint16_t* y,
                             float* logits_out, int32_t* k_out, int32_t* ids_out, float* gates_out,
                             int32_t* offsets_out, void* ws, size_t ws_bytes, void* stream) {
  if (T < 0 || T > kMaxTokens) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N)) return MOE_ERR_UNSUPPORTED;
  if (d <= 0 || d > kMaxDim || d % 128 != 0 || I <= 0 || I > kMaxDim || I % 128 != 0)
    return MOE_ERR_UNSUPPORTED;
  moe_status st = check_route_params(rp, N);
  if (st != MOE_OK) return st;
  const int K = rp->K;
  if (!ws) return MOE_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(ws) & 255u) return MOE_ERR_INVALID_ARG;
  LayerWs w = layer_ws(ws, T, d, N, I, K);
  if (ws_bytes < w.bytes) return MOE_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (T > 0) {  // every argument is checked before anything is enqueued
    const void* need[] = {x, w_router, w_gate_up, w_down, y};
    for (const void* p : need)
      if (!p || !aligned16(p)) return MOE_ERR_INVALID_ARG;
    if (residual && !aligned16(residual)) return MOE_ERR_INVALID_ARG;
    if ((logits_out && !aligned16(logits_out)) || (ids_out && !aligned16(ids_out)) ||
        (gates_out && !aligned16(gates_out)) || !aligned4(k_out) || !aligned4(offsets_out))
      return MOE_ERR_INVALID_ARG;
  }
  // clear the device error word (and the small-batch router's four group
  // tickets beside it), so that a no-op call reads clean; on the few-token
  // path the router clears it, and the expert kernel's counters that follow
  const bool gemv_path = T >= 1 && T <= kGemvLayerMaxTokens && d <= kGemvMaxDim && I <= kGemvMaxDim;
  if (!gemv_path && cudaMemsetAsync(w.err, 0, 8 * sizeof(int32_t), s) != cudaSuccess)
    return MOE_ERR_CUDA;
  if (T == 0) return MOE_OK;

  int32_t* kk = k_out ? k_out : w.k;
  int32_t* ids = ids_out ? ids_out : w.ids;
  float* gates = gates_out ? gates_out : w.gates;
  const int64_t P = T * K;
  const int nsm = sm_count();
  if (nsm <= 0) return MOE_ERR_CUDA;

  cudaError_t e;
  if (gemv_path) {
    // a few tokens: router, routing and dispatch on one cluster, which also
    // clears the error word and the expert kernel's counters
    const int nclear = static_cast<int>((reinterpret_cast<char*>(w.tickets) -
                                         reinterpret_cast<char*>(w.err)) / sizeof(int32_t)) +
                       (d + 15) / 16 + 32;
    e = moe::launch_router_few(x, w_router, static_cast<int>(T), d, N, K, rp->eps,
                               rp->mode == MOE_ROUTE_TOPK, rp->renorm, logits_out, kk, ids, gates,
                               w.offsets, w.perm, w.pair_pos, offsets_out, w.err, nclear, s);
  } else if (T <= kSmallRouterMaxTokens) {
    // a few tokens: the router GEMM split over d on many SMs, then one warp per
    // token routes (the single-chunk dispatch counts the pairs itself)
    e = moe::launch_router_small_route(x, w_router, static_cast<int>(T), d, N, w.partial,
                                       reinterpret_cast<unsigned int*>(w.err + 1), K, rp->eps,
                                       rp->mode == MOE_ROUTE_TOPK, rp->renorm, logits_out, kk, ids,
                                       gates, s);
  } else {
    // router GEMM with the elbow routing in its epilogue; it also leaves the
    // per-chunk expert counts of the dispatch
    e = moe::launch_router_route(x, w_router, T, d, N, K, rp->eps, rp->mode == MOE_ROUTE_TOPK,
                                 rp->renorm, logits_out, kk, ids, gates,
                                 moe::dispatch_counts(w.disp), w.err, nsm, s);
  }
  if (e != cudaSuccess) return MOE_ERR_CUDA;
  if (gemv_path) {
    // a few tokens (dispatched by their router): the CUDA-core expert
    // contractions, which read the token rows through perm, and the combine,
    // in one cooperative launch
    e = moe::launch_expert_few_gemv(x, T, w.perm, w.offsets, w_gate_up, w_down, P, d, N, I, K, w.h,
                                    w.o, w.err, w.tickets + (d + 15) / 16, kk, w.pair_pos, gates,
                                    residual, y, w.tickets, nsm, s);
    if (e != cudaErrorCooperativeLaunchTooLarge) return e == cudaSuccess ? MOE_OK : MOE_ERR_CUDA;
    // SMs not all available to this context (MPS, green contexts): the
    // decode path below, which waits on nothing, serves this step
    (void)cudaGetLastError();
  }
  if (T <= kDecodeMaxTokens) {
    // decode-sized: the single-chunk dispatch also gathers the few token rows
    // (into o, which the down GEMM overwrites afterwards); the GEMMs stream
    // the weights as the M operand
    e = moe::launch_dispatch_gather(kk, ids, T, N, K, w.offsets, w.perm, w.pair_pos, w.disp,
                                    offsets_out, x, d, w.o, nsm, s);
    if (e != cudaSuccess) return MOE_ERR_CUDA;
    e = moe::launch_gateup_decode_gemm(w.o, w_gate_up, w.offsets, P, T, d, N, I, w.h, w.err, nsm,
                                       s);
    if (e != cudaSuccess) return MOE_ERR_CUDA;
    e = moe::launch_down_decode_gemm(w.h, w_down, w.offsets, P, T, d, N, I, w.o, w.err, nsm, s);
    if (e != cudaSuccess) return MOE_ERR_CUDA;
  } else {
    e = moe::launch_dispatch(kk, ids, T, N, K, w.offsets, w.perm, w.pair_pos, w.disp, offsets_out,
                             true, nullptr, nullptr, s);
    if (e != cudaSuccess) return MOE_ERR_CUDA;
    const int32_t* tile_off = moe::dispatch_tile_off(w.disp, T, N);
    // gate/up GEMM gathers its token rows itself (no dispatched copy of x)
    e = gate_up_gathered(x, T, w.perm, w_gate_up, w.offsets, tile_off, P, d, N, I, w.h, w.err, nsm,
                         s);
    if (e != cudaSuccess) return MOE_ERR_CUDA;
    e = expert_down(w.h, w_down, w.offsets, tile_off, P, d, N, I, w.o, w.err, nsm, s);
    if (e != cudaSuccess) return MOE_ERR_CUDA;
  }
  e = moe::launch_combine(w.o, kk, w.pair_pos, gates, residual, T, d, K, y, nsm, s);
  if (e != cudaSuccess) return MOE_ERR_CUDA;
  return MOE_OK;
}

moe_status moe_debug_violations(uint32_t* out) {
  if (!out) return MOE_ERR_INVALID_ARG;
  *out = 0;
#ifdef ELBOW_MOE_DEBUG
  if (cudaDeviceSynchronize() != cudaSuccess) return MOE_ERR_CUDA;
  unsigned int total = 0;
  for (auto take : {moe::debug_take_route, moe::debug_take_route_warp, moe::debug_take_dispatch,
                    moe::debug_take_gemm, moe::debug_take_gemm2, moe::debug_take_gemv,
                    moe::debug_take_diag}) {
    unsigned int v = 0;
    if (take(&v) != cudaSuccess) return MOE_ERR_CUDA;
    total += v;
  }
  *out = total;
  return MOE_OK;
#else
  return MOE_ERR_UNSUPPORTED;
#endif
}

moe_status moe_check_quotients(const float* a, const float* b, int64_t n, float* out,
                               void* stream) {
  if (n < 0 || n > (int64_t(1) << 30)) return MOE_ERR_INVALID_ARG;
  if (n == 0) return MOE_OK;
  if (!a || !b || !out || !aligned4(a) || !aligned4(b) || !aligned4(out)) return MOE_ERR_INVALID_ARG;
  return cuda_status(moe::launch_quotient_check(a, b, n, out, static_cast<cudaStream_t>(stream)));
}

moe_status moe_check_bounded_wait(int32_t* err_word, double seconds, void* stream) {
  if (!err_word || (reinterpret_cast<uintptr_t>(err_word) & 3u)) return MOE_ERR_INVALID_ARG;
  if (!(seconds > 0.0) || seconds > 10.0) return MOE_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(err_word, 0, sizeof(int32_t), s) != cudaSuccess) return MOE_ERR_CUDA;
  bounded_wait_check_kernel<<<1, 32, 0, s>>>(err_word, static_cast<uint64_t>(seconds * 1e9));
  return cuda_status(cudaGetLastError());
}

moe_status moe_read_device_error(const void* ws, void* stream) {
  if (!ws) return MOE_ERR_INVALID_ARG;
  int32_t v = 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return MOE_ERR_CUDA;
  if (cudaMemcpy(&v, ws, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return MOE_ERR_CUDA;
  return v == 0 ? MOE_OK : MOE_ERR_DEVICE_TIMEOUT;
}

moe_status moe_router_logits(const uint16_t* x, const uint16_t* w_router, int64_t T, int d, int N,
                             float* logits, int32_t* err_word, void* stream) {
  if (T < 0 || T > kMaxTokens) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N) || d <= 0 || d > kMaxDim || d % 64 != 0) return MOE_ERR_UNSUPPORTED;
  if (T == 0) return MOE_OK;
  if (!x || !w_router || !logits || !aligned16(x) || !aligned16(w_router) || !aligned16(logits) ||
      !aligned4(err_word))
    return MOE_ERR_INVALID_ARG;
  const int nsm = sm_count();
  if (nsm <= 0) return MOE_ERR_CUDA;
  return cuda_status(moe::launch_router_gemm(x, w_router, T, d, N, logits, err_word, nsm,
                                             static_cast<cudaStream_t>(stream)));
}

moe_status moe_expert_gate_up(const uint16_t* xs, const uint16_t* w_gate_up, const int32_t* offsets,
                              const int32_t* tile_off, int64_t P, int d, int N, int I, uint16_t* h,
                              int32_t* err_word, void* stream) {
  if (P < 0 || P > kMaxTokens * 8) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N) || d <= 0 || d > kMaxDim || d % 64 != 0 || I <= 0 || I > kMaxDim ||
      I % 128 != 0)
    return MOE_ERR_UNSUPPORTED;
  if (P == 0) return MOE_OK;
  if (!xs || !w_gate_up || !offsets || !tile_off || !h || !aligned16(xs) || !aligned16(w_gate_up) ||
      !aligned16(h) || !aligned4(offsets) || !aligned4(tile_off) || !aligned4(err_word))
    return MOE_ERR_INVALID_ARG;
  const int nsm = sm_count();
  if (nsm <= 0) return MOE_ERR_CUDA;
  return cuda_status(moe::launch_gateup_gemm(xs, w_gate_up, offsets, tile_off, P, d, N, I, h,
                                             err_word, nsm, static_cast<cudaStream_t>(stream)));
}

moe_status moe_expert_down(const uint16_t* h, const uint16_t* w_down, const int32_t* offsets,
                           const int32_t* tile_off, int64_t P, int d, int N, int I, uint16_t* o,
                           int32_t* err_word, void* stream) {
  if (P < 0 || P > kMaxTokens * 8) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N) || d <= 0 || d > kMaxDim || d % 128 != 0 || I <= 0 || I > kMaxDim ||
      I % 64 != 0)
    return MOE_ERR_UNSUPPORTED;
  if (P == 0) return MOE_OK;
  if (!h || !w_down || !offsets || !tile_off || !o || !aligned16(h) || !aligned16(w_down) ||
      !aligned16(o) || !aligned4(offsets) || !aligned4(tile_off) || !aligned4(err_word))
    return MOE_ERR_INVALID_ARG;
  const int nsm = sm_count();
  if (nsm <= 0) return MOE_ERR_CUDA;
  return cuda_status(expert_down(h, w_down, offsets, tile_off, P, d, N, I, o, err_word, nsm,
                                 static_cast<cudaStream_t>(stream)));
}

moe_status moe_expert_gate_up_decode(const uint16_t* xs, const uint16_t* w_gate_up,
                                     const int32_t* offsets, int64_t T, int64_t P, int d, int N,
                                     int I, uint16_t* h, int32_t* err_word, void* stream) {
  if (T < 0 || P < 0 || P > kMaxTokens * 8) return MOE_ERR_INVALID_ARG;
  if (T > kDecodeMaxTokens) return MOE_ERR_UNSUPPORTED;
  if (!supported_n(N) || d <= 0 || d > kMaxDim || d % 64 != 0 || I <= 0 || I > kMaxDim ||
      I % 64 != 0)
    return MOE_ERR_UNSUPPORTED;
  if (P == 0 || T == 0) return MOE_OK;
  if (!xs || !w_gate_up || !offsets || !h || !aligned16(xs) || !aligned16(w_gate_up) ||
      !aligned16(h) || !aligned4(offsets) || !aligned4(err_word))
    return MOE_ERR_INVALID_ARG;
  const int nsm = sm_count();
  if (nsm <= 0) return MOE_ERR_CUDA;
  return cuda_status(moe::launch_gateup_decode_gemm(xs, w_gate_up, offsets, P, T, d, N, I, h,
                                                    err_word, nsm,
                                                    static_cast<cudaStream_t>(stream)));
}

moe_status moe_expert_down_decode(const uint16_t* h, const uint16_t* w_down, const int32_t* offsets,
                                  int64_t T, int64_t P, int d, int N, int I, uint16_t* o,
                                  int32_t* err_word, void* stream) {
  if (T < 0 || P < 0 || P > kMaxTokens * 8) return MOE_ERR_INVALID_ARG;
  if (T > kDecodeMaxTokens) return MOE_ERR_UNSUPPORTED;
  if (!supported_n(N) || d <= 0 || d > kMaxDim || d % 128 != 0 || I <= 0 || I > kMaxDim ||
      I % 64 != 0)
    return MOE_ERR_UNSUPPORTED;
  if (P == 0 || T == 0) return MOE_OK;
  if (!h || !w_down || !offsets || !o || !aligned16(h) || !aligned16(w_down) || !aligned16(o) ||
      !aligned4(offsets) || !aligned4(err_word))
    return MOE_ERR_INVALID_ARG;
  const int nsm = sm_count();
  if (nsm <= 0) return MOE_ERR_CUDA;
  return cuda_status(moe::launch_down_decode_gemm(h, w_down, offsets, P, T, d, N, I, o, err_word,
                                                  nsm, static_cast<cudaStream_t>(stream)));
}

moe_status moe_expert_gate_up_gemv(const uint16_t* x, int64_t T, const int32_t* perm,
                                   const int32_t* offsets, const uint16_t* w_gate_up, int64_t P,
                                   int d, int N, int I, int K, uint16_t* h, int32_t* err_word,
                                   void* stream) {
  if (T < 0 || P < 0 || P > kMaxTokens * 8) return MOE_ERR_INVALID_ARG;
  if (T > kGemvMaxTokens || !supported_n(N) || K < 1 || K > 8 || d <= 0 || d > kGemvMaxDim ||
      d % 8 != 0 || I <= 0 || I > kGemvMaxDim || I % 8 != 0)
    return MOE_ERR_UNSUPPORTED;
  if (P == 0 || T == 0) return MOE_OK;
  if (!x || !perm || !offsets || !w_gate_up || !h || !aligned16(x) || !aligned16(w_gate_up) ||
      !aligned4(perm) || !aligned4(offsets) || (reinterpret_cast<uintptr_t>(h) & 1u) ||
      !aligned4(err_word))
    return MOE_ERR_INVALID_ARG;
  return cuda_status(moe::launch_gate_up_gemv(x, T, perm, offsets, w_gate_up, P, d, N, I, K, h,
                                              err_word, static_cast<cudaStream_t>(stream)));
}

moe_status moe_expert_down_gemv(const uint16_t* h, const int32_t* offsets, const uint16_t* w_down,
                                int64_t T, int64_t P, int d, int N, int I, int K, uint16_t* o,
                                int32_t* err_word, void* stream) {
  if (T < 0 || P < 0 || P > kMaxTokens * 8) return MOE_ERR_INVALID_ARG;
  if (T > kGemvMaxTokens || !supported_n(N) || K < 1 || K > 8 || d <= 0 || d > kGemvMaxDim ||
      d % 8 != 0 || I <= 0 || I > kGemvMaxDim || I % 8 != 0)
    return MOE_ERR_UNSUPPORTED;
  if (P == 0 || T == 0) return MOE_OK;
  if (!h || !offsets || !w_down || !o || !aligned16(h) || !aligned16(w_down) ||
      !aligned4(offsets) || (reinterpret_cast<uintptr_t>(o) & 1u) || !aligned4(err_word))
    return MOE_ERR_INVALID_ARG;
  return cuda_status(moe::launch_down_gemv(h, offsets, w_down, T, P, d, N, I, K, o, err_word,
                                           static_cast<cudaStream_t>(stream)));
}

moe_status moe_gather_rows(const uint16_t* x, const int32_t* perm, const int32_t* offsets, int64_t T,
                           int64_t P, int d, int N, uint16_t* xs, void* stream) {
  if (T < 0 || T > kMaxTokens || P < 0 || P > kMaxTokens * 8 || d <= 0 || d > kMaxDim ||
      d % 8 != 0)
    return MOE_ERR_INVALID_ARG;
  if (!supported_n(N)) return MOE_ERR_UNSUPPORTED;
  if (P == 0) return MOE_OK;
  if (!x || !perm || !offsets || !xs || !aligned16(x) || !aligned16(xs) || !aligned4(perm) ||
      !aligned4(offsets))
    return MOE_ERR_INVALID_ARG;
  const int nsm = sm_count();
  if (nsm <= 0) return MOE_ERR_CUDA;
  return cuda_status(moe::launch_gather(x, T, perm, offsets, N, P, d, xs, nsm,
                                        static_cast<cudaStream_t>(stream)));
}

moe_status moe_router_route(const uint16_t* x, const uint16_t* w_router, int64_t T, int d, int N,
                            const moe_route_params* rp, float* logits_out, int32_t* k_out,
                            int32_t* ids_out, float* gates_out, int32_t* chunk_counts,
                            int32_t* err_word, void* stream) {
  if (T < 0 || T > kMaxTokens) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N) || d <= 0 || d > kMaxDim || d % 64 != 0) return MOE_ERR_UNSUPPORTED;
  moe_status st = check_route_params(rp, N);
  if (st != MOE_OK) return st;
  if (T == 0) return MOE_OK;
  if (!x || !w_router || !k_out || !ids_out || !gates_out || !aligned16(x) || !aligned16(w_router) ||
      !aligned16(ids_out) || !aligned16(gates_out) || (logits_out && !aligned16(logits_out)) ||
      !aligned4(k_out) || !aligned4(chunk_counts) || !aligned4(err_word))
    return MOE_ERR_INVALID_ARG;
  const int nsm = sm_count();
  if (nsm <= 0) return MOE_ERR_CUDA;
  return cuda_status(moe::launch_router_route(x, w_router, T, d, N, rp->K, rp->eps,
                                              rp->mode == MOE_ROUTE_TOPK, rp->renorm, logits_out,
                                              k_out, ids_out, gates_out, chunk_counts, err_word,
                                              nsm, static_cast<cudaStream_t>(stream)));
}

moe_status moe_expert_gate_up_gathered(const uint16_t* x, int64_t T, const int32_t* perm,
                                       const uint16_t* w_gate_up, const int32_t* offsets,
                                       const int32_t* tile_off, int64_t P, int d, int N, int I,
                                       uint16_t* h, int32_t* err_word, void* stream) {
  if (T < 0 || P < 0 || P > kMaxTokens * 8) return MOE_ERR_INVALID_ARG;
  if (!supported_n(N) || d <= 0 || d > kMaxDim || d % 64 != 0 || I <= 0 || I > kMaxDim ||
      I % 128 != 0)
    return MOE_ERR_UNSUPPORTED;
  if (P == 0 || T == 0) return MOE_OK;
  if (!x || !perm || !w_gate_up || !offsets || !tile_off || !h || !aligned16(x) ||
      !aligned16(w_gate_up) || !aligned16(h) || !aligned4(perm) || !aligned4(offsets) ||
      !aligned4(tile_off) || !aligned4(err_word))
    return MOE_ERR_INVALID_ARG;
  const int nsm = sm_count();
  if (nsm <= 0) return MOE_ERR_CUDA;
  return cuda_status(gate_up_gathered(x, T, perm, w_gate_up, offsets, tile_off, P, d, N, I, h,
                                      err_word, nsm, static_cast<cudaStream_t>(stream)));
}

moe_status moe_combine(const uint16_t* o, const int32_t* k, const int32_t* pair_pos,
                       const float* gates, const uint16_t* residual, int64_t T, int d, int K,
                       uint16_t* y, void* stream) {
  if (T < 0 || T > kMaxTokens || d <= 0 || d > kMaxDim || d % 8 != 0 || K < 1 || K > 8)
    return MOE_ERR_INVALID_ARG;
  if (T == 0) return MOE_OK;
  if (!o || !k || !pair_pos || !gates || !y || !aligned16(o) || !aligned16(y) ||
      (residual && !aligned16(residual)) || !aligned4(k) || !aligned4(pair_pos) || !aligned4(gates))
    return MOE_ERR_INVALID_ARG;
  const int nsm = sm_count();
  if (nsm <= 0) return MOE_ERR_CUDA;
  return cuda_status(moe::launch_combine(o, k, pair_pos, gates, residual, T, d, K, y, nsm,
                                         static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
