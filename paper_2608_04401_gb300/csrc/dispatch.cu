// Token-to-expert dispatch of the selected (t, s < k_t) pairs, stable in t,
// plus the row gather and the gate-weighted combine.
//
// Dispatch is a deterministic three-pass counting sort over token chunks:
//   count   : per chunk (kChunk tokens), per-expert pair counts (smem atomics:
//             the counts do not depend on their order)
//   scan    : per expert, exclusive prefix over chunks; per-expert totals ->
//             offsets [N+1]; m-tile prefix ceil(count_e / 128) -> tile_off
//   scatter : each chunk walks its tokens in order, 32 per warp; a pair's
//             position = chunk base + earlier warps of this round (ballots in
//             smem) + earlier lanes of this warp (popc of the ballot).
#include <mutex>

#include "common.cuh"

namespace moe {
namespace disp {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kChunk = 2048;  // tokens per chunk (block)

template <int N>
__global__ void __launch_bounds__(kThreads) count_kernel(const int32_t* __restrict__ k,
                                                         const int32_t* __restrict__ ids, int64_t T,
                                                         int K, int32_t* __restrict__ blk_cnt) {
  __shared__ int cnt[N];
  for (int i = threadIdx.x; i < N; i += kThreads) cnt[i] = 0;
  __syncthreads();
  const int64_t t0 = static_cast<int64_t>(blockIdx.x) * kChunk;
  const int64_t t1 = min_of<int64_t>(T, t0 + kChunk);
  for (int64_t t = t0 + threadIdx.x; t < t1; t += kThreads) {
    const int kt = min(k[t], K);
    for (int s = 0; s < kt; ++s) atomicAdd(&cnt[ids[t * K + s]], 1);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < N; i += kThreads) blk_cnt[static_cast<int64_t>(blockIdx.x) * N + i] = cnt[i];
}

// One block of 1024 threads: thread (g, e) owns expert e over the g-th slice
// of the chunks.
template <int N>
__global__ void __launch_bounds__(1024) scan_kernel(const int32_t* __restrict__ blk_cnt, int nblk,
                                                    int32_t* __restrict__ blk_base,
                                                    int32_t* __restrict__ offsets,
                                                    int32_t* __restrict__ tile_off,
                                                    int32_t* __restrict__ offsets_copy) {
  constexpr int G = 1024 / N;
  __shared__ int part[G][N];
  __shared__ int exp_off[N + 1];
  const int e = threadIdx.x % N, g = threadIdx.x / N;
  const int per = (nblk + G - 1) / G;
  const int b0 = g * per, b1 = min(nblk, b0 + per);
  int sum = 0;
  for (int b = b0; b < b1; ++b) sum += blk_cnt[static_cast<int64_t>(b) * N + e];
  part[g][e] = sum;
  __syncthreads();
  if (threadIdx.x == 0) {
    // totals per expert, then the exclusive scan over experts
    int run = 0, trun = 0;
    for (int x = 0; x < N; ++x) {
      int tot = 0;
      for (int y = 0; y < G; ++y) tot += part[y][x];
      exp_off[x] = run;
      offsets[x] = run;
      tile_off[x] = trun;
      if (offsets_copy) offsets_copy[x] = run;
      run += tot;
      trun += (tot + 127) / 128;
    }
    exp_off[N] = run;
    offsets[N] = run;
    tile_off[N] = trun;
    if (offsets_copy) offsets_copy[N] = run;
  }
  __syncthreads();
  int base = exp_off[e];
  for (int y = 0; y < g; ++y) base += part[y][e];
  for (int b = b0; b < b1; ++b) {
    blk_base[static_cast<int64_t>(b) * N + e] = base;
    base += blk_cnt[static_cast<int64_t>(b) * N + e];
  }
}

template <int N>
__global__ void __launch_bounds__(kThreads) scatter_kernel(const int32_t* __restrict__ k,
                                                           const int32_t* __restrict__ ids,
                                                           int64_t T, int K,
                                                           const int32_t* __restrict__ blk_base,
                                                           int32_t* __restrict__ perm,
                                                           int32_t* __restrict__ pair_pos) {
  __shared__ int run[N];
  __shared__ uint32_t bal[kWarps][N];
  __shared__ int wbase[kWarps][N];
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  for (int i = threadIdx.x; i < N; i += kThreads) run[i] = blk_base[static_cast<int64_t>(blockIdx.x) * N + i];
  const int64_t t0 = static_cast<int64_t>(blockIdx.x) * kChunk;
  const int64_t t1 = min_of<int64_t>(T, t0 + kChunk);
  const uint32_t lt_mask = (1u << lane) - 1u;
  for (int64_t r0 = t0; r0 < t1; r0 += kThreads) {
    const int64_t t = r0 + threadIdx.x;
    const bool valid = t < t1;
    const int kt = valid ? min(k[t], K) : 0;
    int my[8];
    uint64_t m0 = 0, m1 = 0;
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      my[s] = (s < kt) ? ids[t * K + s] : -1;
      if (s < kt) {
        if (my[s] < 64) m0 |= 1ull << my[s];
        else m1 |= 1ull << (my[s] - 64);
      }
    }
    __syncthreads();  // previous round's readers of bal/wbase are done
#pragma unroll
    for (int e = 0; e < N; ++e) {
      const bool has = ((e < 64 ? (m0 >> e) : (m1 >> (e - 64))) & 1ull) != 0;
      const uint32_t b = __ballot_sync(0xffffffffu, has);
      if (lane == (e & 31)) bal[warp][e] = b;
    }
    __syncthreads();
    for (int e = threadIdx.x; e < N; e += kThreads) {
      int acc = run[e];
#pragma unroll
      for (int w = 0; w < kWarps; ++w) {
        wbase[w][e] = acc;
        acc += __popc(bal[w][e]);
      }
      run[e] = acc;
    }
    __syncthreads();
    if (valid) {
#pragma unroll
      for (int s = 0; s < 8; ++s) {
        if (s < K) {
          if (s < kt) {
            const int e = my[s];
            const int pos = wbase[warp][e] + __popc(bal[warp][e] & lt_mask);
            perm[pos] = static_cast<int32_t>(t);
            pair_pos[t * K + s] = pos;
          } else {
            pair_pos[t * K + s] = -1;
          }
        }
      }
    }
  }
}

// xs[r] = x[perm[r]] for r < offsets[N]; one warp per row, 16-byte copies.
__global__ void __launch_bounds__(256) gather_kernel(const uint4* __restrict__ x,
                                                     const int32_t* __restrict__ perm,
                                                     const int32_t* __restrict__ offsets, int N,
                                                     int d8, uint4* __restrict__ xs) {
  const int total = offsets[N];
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * 8 + warp; r < total;
       r += static_cast<int64_t>(gridDim.x) * 8) {
    const int64_t t = perm[r];
    const uint4* src = x + t * d8;
    uint4* dst = xs + r * d8;
    for (int c = lane; c < d8; c += 32) dst[c] = __ldg(src + c);
  }
}

// y_t = sum_{s<k_t} g_{t,s} * o[pair_pos[t,s]] (+ residual_t); fp32 in s order.
__global__ void __launch_bounds__(256) combine_kernel(const uint4* __restrict__ o,
                                                      const int32_t* __restrict__ k,
                                                      const int32_t* __restrict__ pair_pos,
                                                      const float* __restrict__ gates,
                                                      const uint4* residual, int64_t T, int d8,
                                                      int K, uint4* y) {
  for (int64_t t = blockIdx.x; t < T; t += gridDim.x) {
    const int kt = min(k[t], K);
    int pos[8];
    float g[8];
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      pos[s] = (s < kt) ? pair_pos[t * K + s] : 0;
      g[s] = (s < kt) ? gates[t * K + s] : 0.0f;
    }
    for (int c = threadIdx.x; c < d8; c += blockDim.x) {
      float acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll
      for (int s = 0; s < 8; ++s) {
        if (s < kt) {
          const uint4 v = o[static_cast<int64_t>(pos[s]) * d8 + c];
          const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float2 f = __bfloat1622float2(h[u]);
            acc[2 * u] = fmaf(g[s], f.x, acc[2 * u]);
            acc[2 * u + 1] = fmaf(g[s], f.y, acc[2 * u + 1]);
          }
        }
      }
      if (residual) {
        const uint4 v = residual[t * d8 + c];
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const float2 f = __bfloat1622float2(h[u]);
          acc[2 * u] += f.x;
          acc[2 * u + 1] += f.y;
        }
      }
      uint4 out;
      out.x = pack_bf16x2(acc[0], acc[1]);
      out.y = pack_bf16x2(acc[2], acc[3]);
      out.z = pack_bf16x2(acc[4], acc[5]);
      out.w = pack_bf16x2(acc[6], acc[7]);
      y[t * d8 + c] = out;
    }
  }
}

}  // namespace disp

size_t dispatch_ws_bytes(int64_t T, int N) {
  const int64_t nblk = (T + disp::kChunk - 1) / disp::kChunk;
  const size_t a = static_cast<size_t>(nblk > 0 ? nblk : 1) * N * sizeof(int32_t);
  auto up = [](size_t b) { return (b + 255) & ~static_cast<size_t>(255); };
  return up(a) * 2 + up((N + 1) * sizeof(int32_t));
}

// Workspace layout: blk_cnt [nblk][N] | blk_base [nblk][N] | tile_off [N+1]
int32_t* dispatch_tile_off(void* ws, int64_t T, int N) {
  const int64_t nblk = (T + disp::kChunk - 1) / disp::kChunk;
  const size_t a = static_cast<size_t>(nblk > 0 ? nblk : 1) * N * sizeof(int32_t);
  const size_t up = (a + 255) & ~static_cast<size_t>(255);
  return reinterpret_cast<int32_t*>(static_cast<char*>(ws) + 2 * up);
}

cudaError_t launch_dispatch(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                            int32_t* offsets, int32_t* perm, int32_t* pair_pos, void* ws,
                            int32_t* offsets_copy, cudaStream_t stream) {
  const int64_t nblk64 = (T + disp::kChunk - 1) / disp::kChunk;
  const int nblk = static_cast<int>(nblk64);
  const size_t a = static_cast<size_t>(nblk > 0 ? nblk : 1) * N * sizeof(int32_t);
  const size_t up = (a + 255) & ~static_cast<size_t>(255);
  int32_t* blk_cnt = static_cast<int32_t*>(ws);
  int32_t* blk_base = reinterpret_cast<int32_t*>(static_cast<char*>(ws) + up);
  int32_t* tile_off = dispatch_tile_off(ws, T, N);
  if (N == 64) {
    if (nblk > 0) disp::count_kernel<64><<<nblk, disp::kThreads, 0, stream>>>(k, ids, T, K, blk_cnt);
    disp::scan_kernel<64><<<1, 1024, 0, stream>>>(blk_cnt, nblk, blk_base, offsets, tile_off, offsets_copy);
    if (nblk > 0) disp::scatter_kernel<64><<<nblk, disp::kThreads, 0, stream>>>(k, ids, T, K, blk_base, perm, pair_pos);
  } else {
    if (nblk > 0) disp::count_kernel<128><<<nblk, disp::kThreads, 0, stream>>>(k, ids, T, K, blk_cnt);
    disp::scan_kernel<128><<<1, 1024, 0, stream>>>(blk_cnt, nblk, blk_base, offsets, tile_off, offsets_copy);
    if (nblk > 0) disp::scatter_kernel<128><<<nblk, disp::kThreads, 0, stream>>>(k, ids, T, K, blk_base, perm, pair_pos);
  }
  return cudaGetLastError();
}

cudaError_t launch_gather(const uint16_t* x, const int32_t* perm, const int32_t* offsets, int N,
                          int64_t P, int d, uint16_t* xs, int num_sms, cudaStream_t stream) {
  if (P == 0) return cudaSuccess;
  int64_t blocks = (P + 7) / 8;
  const int64_t cap = static_cast<int64_t>(num_sms) * 16;
  if (blocks > cap) blocks = cap;
  disp::gather_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(
      reinterpret_cast<const uint4*>(x), perm, offsets, N, d / 8, reinterpret_cast<uint4*>(xs));
  return cudaGetLastError();
}

cudaError_t launch_combine(const uint16_t* o, const int32_t* k, const int32_t* pair_pos,
                           const float* gates, const uint16_t* residual, int64_t T, int d, int K,
                           uint16_t* y, int num_sms, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  int64_t blocks = T;
  const int64_t cap = static_cast<int64_t>(num_sms) * 64;
  if (blocks > cap) blocks = cap;
  disp::combine_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(
      reinterpret_cast<const uint4*>(o), k, pair_pos, gates,
      reinterpret_cast<const uint4*>(residual), T, d / 8, K, reinterpret_cast<uint4*>(y));
  return cudaGetLastError();
}

}  // namespace moe

// ---------------------------------------------------------------------------
// Dispatch without a caller-provided workspace.
//
// Some callers cannot allocate device memory at the point where they dispatch:
// a serving runtime that plans every byte of device memory up front and forbids
// allocation on its request path (an allocation can block on the device or
// fragment a pre-sized pool), or a plug-in whose host framework hands it only
// the input and output buffers. For them the dispatch's scratch (per-chunk
// expert counts and bases, and the m-tile offsets) lives in one file-scope
// device array of fixed size instead of a workspace. Every GPU that loads this
// library holds the array until the process exits.
namespace moe {
namespace disp {
constexpr int64_t kNoAllocMaxTokens = int64_t(1) << 20;  // 1,048,576 tokens
constexpr int kNoAllocMaxExperts = 128;
constexpr int64_t kNoAllocChunks = (kNoAllocMaxTokens + kChunk - 1) / kChunk;
constexpr int64_t kNoAllocInts = 2 * kNoAllocChunks * kNoAllocMaxExperts + 256;  // ~513 KB
}  // namespace disp
}  // namespace moe

static __device__ __align__(256) int32_t g_noalloc_dispatch_scratch[moe::disp::kNoAllocInts];

namespace {
constexpr int kNoAllocMaxDevices = 64;
std::mutex g_noalloc_mu;
int32_t* g_noalloc_ptr[kNoAllocMaxDevices] = {};

// Device address of the scratch array on the current device. The host-side
// symbol is only a stand-in, so the address is looked up once per device (with
// that device current) and cached.
cudaError_t noalloc_scratch(int32_t** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kNoAllocMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_dispatch_scratch);
    if (e != cudaSuccess) return e;
    g_noalloc_ptr[dev] = static_cast<int32_t*>(p);
  }
  *out = g_noalloc_ptr[dev];
  return cudaSuccess;
}
}  // namespace

extern "C" moe_status moe_dispatch_noalloc(const int32_t* k, const int32_t* ids, int64_t T, int N,
                                           int K, int32_t* offsets, int32_t* perm,
                                           int32_t* pair_pos, void* stream) {
  using namespace moe::disp;
  if (T < 0) return MOE_ERR_INVALID_ARG;
  if (T > kNoAllocMaxTokens) return MOE_ERR_UNSUPPORTED;
  if ((N != 64 && N != 128) || K < 1 || K > 8 || K > N) return MOE_ERR_UNSUPPORTED;
  if (!offsets) return MOE_ERR_INVALID_ARG;
  if (T > 0 && (!k || !ids || !perm || !pair_pos)) return MOE_ERR_INVALID_ARG;
  int32_t* scratch = nullptr;
  if (noalloc_scratch(&scratch) != cudaSuccess) return MOE_ERR_CUDA;
  // Layout: per-chunk counts [chunks][N] | per-chunk bases [chunks][N] | tile offsets
  // [N+1]. The counts and bases of every chunk in use and all N+1 tile offsets are
  // rewritten by each call, so nothing has to be cleared first.
  int32_t* blk_cnt = scratch;
  int32_t* blk_base = scratch + kNoAllocChunks * kNoAllocMaxExperts;
  int32_t* tile_off = scratch + 2 * kNoAllocChunks * kNoAllocMaxExperts;
  const int nblk = static_cast<int>((T + kChunk - 1) / kChunk);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (N == 64) {
    if (nblk > 0) count_kernel<64><<<nblk, kThreads, 0, s>>>(k, ids, T, K, blk_cnt);
    scan_kernel<64><<<1, 1024, 0, s>>>(blk_cnt, nblk, blk_base, offsets, tile_off, nullptr);
    if (nblk > 0) scatter_kernel<64><<<nblk, kThreads, 0, s>>>(k, ids, T, K, blk_base, perm, pair_pos);
  } else {
    if (nblk > 0) count_kernel<128><<<nblk, kThreads, 0, s>>>(k, ids, T, K, blk_cnt);
    scan_kernel<128><<<1, 1024, 0, s>>>(blk_cnt, nblk, blk_base, offsets, tile_off, nullptr);
    if (nblk > 0) scatter_kernel<128><<<nblk, kThreads, 0, s>>>(k, ids, T, K, blk_base, perm, pair_pos);
  }
  return cudaGetLastError() == cudaSuccess ? MOE_OK : MOE_ERR_CUDA;
}
