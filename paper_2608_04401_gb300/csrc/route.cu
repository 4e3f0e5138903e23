// Elbow router kernel: one thread per token (the device code is in
// route_impl.cuh, shared with the router GEMM's fused epilogue).
#include "route_impl.cuh"

namespace moe {
namespace route {

// One thread per token; optionally (blk_cnt != nullptr) also the block's
// per-expert pair counts, written to blk_cnt[e * nblk + blockIdx.x] (the
// first pass of the dispatch, fused here so that the ids are not re-read).
template <int N>
__global__ void __launch_bounds__(kTok) elbow_route_kernel(
    const float* __restrict__ logits, int64_t T, int K, float eps, int topk_mode, int renorm,
    const __grid_constant__ RouteConsts<N> rc, int32_t* __restrict__ k_out,
    int32_t* __restrict__ ids_out, float* __restrict__ gates_out, int32_t* __restrict__ blk_cnt,
    int nblk) {
  constexpr int kPitch = N + 4;
  extern __shared__ float4 smem4[];
  __shared__ int hist[N];
  float* tile = reinterpret_cast<float*>(smem4);
  uint64_t* keys64 = reinterpret_cast<uint64_t*>(tile + kTok * kPitch);  // [8][kTok]

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
  if (tid < ntok)
    k_sel = route_token<N, RouteConsts<N>>(tile + tid * kPitch, t0 + tid, tid, K, eps, topk_mode,
                                           renorm, rc, keys64, k_out, ids_out, gates_out, ids_sel);
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
                   cudaStream_t stream) {
  RouteConsts<N> rc;
  fill_route_consts(rc, N);
  constexpr size_t smem = smem_bytes<N>();
  static int attr_dev = -1;
  int dev = 0;
  cudaGetDevice(&dev);
  if (attr_dev != dev) {
    cudaError_t e = cudaFuncSetAttribute(elbow_route_kernel<N>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr_dev = dev;
  }
  const int64_t blocks = (T + kTok - 1) / kTok;
  elbow_route_kernel<N><<<static_cast<unsigned>(blocks), kTok, smem, stream>>>(
      logits, T, K, eps, topk_mode, renorm, rc, k_out, ids_out, gates_out, blk_cnt,
      static_cast<int>(blocks));
  return cudaGetLastError();
}

}  // namespace route

// blk_cnt (nullable): per-128-token-chunk expert counts, [N][ceil(T/128)].
cudaError_t launch_elbow_route(const float* logits, int64_t T, int N, int K, float eps,
                               int topk_mode, int renorm, int32_t* k_out, int32_t* ids_out,
                               float* gates_out, int32_t* blk_cnt, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  if (N == 64)
    return route::launch<64>(logits, T, K, eps, topk_mode, renorm, k_out, ids_out, gates_out,
                             blk_cnt, stream);
  return route::launch<128>(logits, T, K, eps, topk_mode, renorm, k_out, ids_out, gates_out,
                            blk_cnt, stream);
}

}  // namespace moe
