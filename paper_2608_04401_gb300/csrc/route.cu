// Elbow router kernel: one thread per token (the device code is in
// route_impl.cuh, shared with the router GEMM's fused epilogue).
#include "route_impl.cuh"

namespace moe {
namespace route {

// Tail / head randomisation (Sec. 2.2) of one routed token, in place of its
// outputs: top[] holds the ids of ranks 0..K-1 and k the elbow count. mode 2
// keeps ranks 0..k-1 and fills slots k..K-1 with experts of rank >= k; mode 3
// keeps ranks k..K-1 and fills slots 0..k-1 with experts of rank >= K. Each
// draw takes, among the remaining experts in ascending id order, the one at
// index rand[t, s] mod (number remaining). Gates are the experts' own p (the
// row holds their e, and s is recomputed with the routing's tree order).
template <int N>
__device__ __noinline__ void randomize_token(const float* row, int64_t t, int K, int mode,
                                             int renorm, int k, const int* top,
                                             const uint32_t* __restrict__ rand,
                                             int32_t* __restrict__ k_out,
                                             int32_t* __restrict__ ids_out,
                                             float* __restrict__ gates_out) {
  float v[N];
#pragma unroll
  for (int j = 0; j < N; ++j) v[j] = row[j];
#pragma unroll
  for (int h = N / 2; h >= 1; h /= 2)
#pragma unroll
    for (int i = 0; i < h; ++i) v[i] = __fadd_rn(v[i], v[i + h]);
  const float sum = v[0], ys = __frcp_rn(sum);
  uint32_t taken[N / 32];
#pragma unroll
  for (int w = 0; w < N / 32; ++w) taken[w] = 0u;
  int ids[8];
  const int excl = mode == 2 ? k : K;
  for (int s = 0; s < K; ++s) {
    ids[s] = top[s];
    if (s < excl) taken[top[s] / 32] |= 1u << (top[s] % 32);
  }
  const int lo = mode == 2 ? k : 0, hi = mode == 2 ? K : k;
  int remaining = N - excl;
  for (int s = lo; s < hi; ++s) {
    uint32_t idx = rand[t * K + s] % static_cast<uint32_t>(remaining);
    int pick = 0;
    for (int w = 0; w < N / 32; ++w) {
      const uint32_t freew = ~taken[w];
      const uint32_t c = static_cast<uint32_t>(__popc(freew));
      if (idx < c) {
        uint32_t f = freew;
        for (uint32_t i = 0; i < idx; ++i) f &= f - 1u;  // drop the idx lowest free bits
        pick = w * 32 + __ffs(static_cast<int>(f)) - 1;
        break;
      }
      idx -= c;
    }
    taken[pick / 32] |= 1u << (pick % 32);
    ids[s] = pick;
    --remaining;
  }
  float S = 0.0f;
  for (int s = 0; s < K; ++s) S = __fadd_rn(S, quot(row[ids[s]], sum, ys));
  k_out[t] = K;
  for (int s = 0; s < K; ++s) {
    const float p = quot(row[ids[s]], sum, ys);
    ids_out[t * K + s] = ids[s];
    gates_out[t * K + s] = renorm ? __fdiv_rn(p, S) : p;
  }
}

// One thread per token; optionally (blk_cnt != nullptr) also the block's
// per-expert pair counts, written to blk_cnt[e * nblk + blockIdx.x] (the
// first pass of the dispatch, fused here so that the ids are not re-read).
template <int N, bool RAND>
__global__ void __launch_bounds__(kTok) elbow_route_kernel(
    const float* __restrict__ logits, int64_t T, int K, float eps, int topk_mode, int renorm,
    const __grid_constant__ RouteConsts<N> rc, int32_t* __restrict__ k_out,
    int32_t* __restrict__ ids_out, float* __restrict__ gates_out, int32_t* __restrict__ blk_cnt,
    int nblk, const uint32_t* __restrict__ rand, int rand_mode) {
  constexpr int kPitch = N + 4;
  extern __shared__ float4 smem4[];
  __shared__ int hist[N];
  float* tile = reinterpret_cast<float*>(smem4);

  const int64_t t0 = static_cast<int64_t>(blockIdx.x) * kTok;
  const int ntok = static_cast<int>(min_of<int64_t>(kTok, T - t0));
  const int tid = threadIdx.x;
  for (int e = tid; e < N; e += kTok) hist[e] = 0;

  // coalesced staging of the contiguous [ntok, N] logit block
  {
    const float4* src = reinterpret_cast<const float4*>(logits + t0 * N);
    const int nvec = ntok * (N / 4);
    for (int v = tid; v < nvec; v += kTok) {
      const float4 val = __ldcs(src + v);
      const int row = v / (N / 4), col = (v % (N / 4)) * 4;
      *reinterpret_cast<float4*>(tile + row * kPitch + col) = val;
    }
  }
  __syncthreads();
  int ids_sel[8];
  int k_sel = 0;
  float ssum = 0.0f;
  const bool valid = tid < ntok;
  if (valid)
    k_sel = route_token<N, RouteConsts<N>>(tile + tid * kPitch, t0 + tid, K, eps, topk_mode,
                                           renorm, rc, k_out, ids_out, gates_out, ids_sel, ssum);
  // tokens the fast path left undecided: routed by their whole warp
  const unsigned undecided = __ballot_sync(0xffffffffu, valid && k_sel < 0);
  if (undecided) {
    const float* wrow = tile + (tid & ~31) * kPitch;
    route_undecided<N>(undecided, [&](int l) { return wrow + l * kPitch; }, ssum, t0 + tid, K, eps,
                       topk_mode, renorm, k_out, ids_out, gates_out, k_sel, ids_sel);
  }
  if (valid) {
    if constexpr (RAND) {
      randomize_token<N>(tile + tid * kPitch, t0 + tid, K, rand_mode, renorm, k_sel, ids_sel, rand,
                         k_out, ids_out, gates_out);
      k_sel = K;
#pragma unroll
      for (int s = 0; s < 8; ++s)
        if (s < K) ids_sel[s] = ids_out[(t0 + tid) * K + s];
    }
  }
  if (blk_cnt != nullptr) {
#pragma unroll
    for (int s = 0; s < 8; ++s)
      if (s < k_sel) atomicAdd(&hist[ids_sel[s]], 1);
    __syncthreads();
    for (int e = tid; e < N; e += kTok) blk_cnt[static_cast<int64_t>(e) * nblk + blockIdx.x] = hist[e];
  }
}

template <int N>
cudaError_t launch(const float* logits, int64_t T, int K, float eps, int topk_mode, int renorm,
                   int32_t* k_out, int32_t* ids_out, float* gates_out, int32_t* blk_cnt,
                   const uint32_t* rand, int rand_mode, cudaStream_t stream) {
  RouteConsts<N> rc;
  fill_route_consts(rc, N);
  constexpr size_t smem = route_smem_bytes<N>();
  auto kern = rand_mode ? elbow_route_kernel<N, true> : elbow_route_kernel<N, false>;
  static std::atomic<uint64_t> attr_done{0};
  const cudaError_t ae = once_per_device(attr_done, [] {
    for (auto f : {elbow_route_kernel<N, true>, elbow_route_kernel<N, false>}) {
      const cudaError_t e =
          cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
  });
  if (ae != cudaSuccess) return ae;
  const int64_t blocks = (T + kTok - 1) / kTok;
  kern<<<static_cast<unsigned>(blocks), kTok, smem, stream>>>(
      logits, T, K, eps, topk_mode, renorm, rc, k_out, ids_out, gates_out, blk_cnt,
      static_cast<int>(blocks), rand, rand_mode);
  return cudaGetLastError();
}

// Self-check of the routing's quotients: out[3i .. 3i+2] = quot(a, b), the
// packed quot2 (both numerators of a pair at once; only where both qualify),
// and CUDA's __fdiv_rn, for a_i >= 0 and b_i in [2^-32, 2^8].
__global__ void quotient_check_kernel(const float* __restrict__ a, const float* __restrict__ b,
                                      int64_t n, float* __restrict__ out) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const float ai = a[i], bi = b[i], y = __frcp_rn(bi);
  const bool fast = ai == 0.0f || ai >= kQuotMin;
  const uint64_t q2 = quot2(pk(ai, fast ? ai : 0.0f), pk(-bi, -bi), pk(y, y));
  out[3 * i] = quot(ai, bi, y);
  out[3 * i + 1] = fast ? lo_of(q2) : __fdiv_rn(ai, bi);
  out[3 * i + 2] = __fdiv_rn(ai, bi);
}

}  // namespace route

cudaError_t launch_quotient_check(const float* a, const float* b, int64_t n, float* out,
                                  cudaStream_t stream) {
  if (n == 0) return cudaSuccess;
  const int64_t blocks = (n + 255) / 256;
  route::quotient_check_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(a, b, n, out);
  return cudaGetLastError();
}

// blk_cnt (nullable): per-128-token-chunk expert counts, [N][ceil(T/128)].
// rand (nullable) and rand_mode (0, or 2 / 3 for the tail / head randomisation).
cudaError_t launch_elbow_route(const float* logits, int64_t T, int N, int K, float eps,
                               int topk_mode, int renorm, int32_t* k_out, int32_t* ids_out,
                               float* gates_out, int32_t* blk_cnt, const uint32_t* rand,
                               int rand_mode, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  if (N == 64)
    return route::launch<64>(logits, T, K, eps, topk_mode, renorm, k_out, ids_out, gates_out,
                             blk_cnt, rand, rand_mode, stream);
  return route::launch<128>(logits, T, K, eps, topk_mode, renorm, k_out, ids_out, gates_out,
                            blk_cnt, rand, rand_mode, stream);
}

MOE_DEBUG_TU(route)

}  // namespace moe
