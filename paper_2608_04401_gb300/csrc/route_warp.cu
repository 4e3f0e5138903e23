// Small-batch routing: one WARP per token, for batches too small to hide the
// ~2500-instruction chain that one thread per token needs (decode steps).
//
// Lane l holds experts l + 32c (c < N/32). The arithmetic is the routing
// specification of route_impl.cuh, step for step, so the results are the same
// bits as the thread-per-token kernels and the oracle:
//   m = max l (warp reduction); e_j = EXP(l_j - m) (the packed spec
//   exponential); s = balanced tree sum (levels h >= 32 inside the lane, then
//   v_i += v_{i+h} by shuffles); p_j = e_j * (1/s);
//   a bitonic sort of the N keys (p bits << 32 | ~id) across the warp (64-bit
//   shuffles), which orders by p descending and ascending id on ties;
//   p'_i, D_i on each rank, the first argmax by a (max D, min index) warp
//   reduction, k = min(e + 1, K).
// The logits may arrive as `nslice` partial sums (the small-batch router GEMM
// splits d); they are added in slice order.
//
// router_small_route_kernel: the router GEMM for T <= 64 tokens on CUDA cores,
// split over d in slices of 64 columns (one block per slice) so that many SMs
// stream a slice of x and W_r instead of one SM streaming them all:
// partial[s][t][e] = sum_{k in slice s} x[t][k] w[e][k], fp32 fma in k order;
// the block that finishes last routes every token (slices added in order).
#include "route_impl.cuh"

namespace moe {
namespace rwarp {

using route::RouteConsts;

constexpr int kWarps = 4;        // tokens per block of the routing kernel
constexpr int kSlice = 64;       // d columns per block of the small router GEMM
constexpr int kSmallT = 64;      // largest batch of the small router GEMM
constexpr int kPitch2 = kSlice / 2 + 1;  // row pitch in bf16 pairs (odd: no bank conflicts)

template <int N>
MOE_DEV void router_small_body(const uint32_t* __restrict__ x, const uint32_t* __restrict__ w, int T,
                               int d, float* __restrict__ partial) {
  __shared__ uint32_t xs[kSmallT][kPitch2];  // bf16 pairs
  __shared__ uint32_t wsm[N][kPitch2];
  const int s = blockIdx.x;
  const int d2 = d / 2;
  const int c0 = s * (kSlice / 2);
  for (int i = threadIdx.x; i < kSmallT * (kSlice / 2); i += 256) {
    const int r = i / (kSlice / 2), c = i % (kSlice / 2);
    xs[r][c] = r < T ? x[static_cast<int64_t>(r) * d2 + c0 + c] : 0u;
  }
  for (int i = threadIdx.x; i < N * (kSlice / 2); i += 256) {
    const int r = i / (kSlice / 2), c = i % (kSlice / 2);
    wsm[r][c] = w[static_cast<int64_t>(r) * d2 + c0 + c];
  }
  __syncthreads();
  constexpr int kGroups = 256 / N;             // token groups
  constexpr int kTpg = kSmallT / kGroups;      // tokens per group
  const int e = threadIdx.x % N, g = threadIdx.x / N;
  float acc[kTpg];
#pragma unroll
  for (int i = 0; i < kTpg; ++i) acc[i] = 0.0f;
#pragma unroll 4
  for (int c = 0; c < kSlice / 2; ++c) {
    const float2 wv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&wsm[e][c]));
#pragma unroll
    for (int i = 0; i < kTpg; ++i) {
      const float2 xv =
          __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&xs[g * kTpg + i][c]));
      acc[i] = fmaf(xv.x, wv.x, acc[i]);
      acc[i] = fmaf(xv.y, wv.y, acc[i]);
    }
  }
#pragma unroll
  for (int i = 0; i < kTpg; ++i) {
    const int t = g * kTpg + i;
    if (t < T) partial[(static_cast<int64_t>(s) * T + t) * N + e] = acc[i];
  }
}

// Routes token t with the calling (whole, converged) warp. src holds the
// logits as nslice partial sums [nslice][T][N] (nslice = 1: the logits); with
// L2_ONLY they are read past L1 (written by other blocks of the same launch).
template <int N, bool L2_ONLY>
MOE_DEV void route_one_warp(const float* __restrict__ src, int64_t t, int64_t T, int nslice, int K,
                            float eps, int topk_mode, int renorm, float* __restrict__ logits_out,
                            int32_t* __restrict__ k_out, int32_t* __restrict__ ids_out,
                            float* __restrict__ gates_out) {
  constexpr int C = N / 32;
  const unsigned full = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  auto ld = [&](int64_t i) { return L2_ONLY ? __ldcg(src + i) : src[i]; };

  // logits, slices added in order
  float l[C];
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const int64_t off = t * N + 32 * c + lane;
    const int64_t stride = T * N;
    float a = ld(off);
    int s = 1;
    // eight slices' loads in flight at a time; the sum stays in slice order
    for (; s + 8 <= nslice; s += 8) {
      float q[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) q[u] = ld((s + u) * stride + off);
#pragma unroll
      for (int u = 0; u < 8; ++u) a = __fadd_rn(a, q[u]);
    }
    for (; s < nslice; ++s) a = __fadd_rn(a, ld(s * stride + off));
    l[c] = a;
    if (logits_out) logits_out[off] = a;
  }
  float m = l[0];
#pragma unroll
  for (int c = 1; c < C; ++c) m = fmaxf(m, l[c]);
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) m = fmaxf(m, __shfl_xor_sync(full, m, o));

  // e = EXP(l - m) on pairs
  float e[C];
  const uint64_t mm = route::pk(m, m);
#pragma unroll
  for (int c = 0; c < C; c += 2) {
    const uint64_t q = route::exp_spec2(route::sub2(route::pk(l[c], l[c + 1]), mm));
    e[c] = route::lo_of(q);
    e[c + 1] = route::hi_of(q);
  }

  // s: v_i += v_{i+h} for i < h, h = N/2 .. 1
  float v[C];
#pragma unroll
  for (int c = 0; c < C; ++c) v[c] = e[c];
#pragma unroll
  for (int h = N / 2; h >= 32; h >>= 1)
#pragma unroll
    for (int c = 0; c < h / 32; ++c) v[c] = __fadd_rn(v[c], v[c + h / 32]);
  float v0 = v[0];
#pragma unroll
  for (int h = 16; h >= 1; h >>= 1) {
    const float o = __shfl_down_sync(full, v0, h);
    if (lane < h) v0 = __fadd_rn(v0, o);
  }
  const float r = __frcp_rn(__shfl_sync(full, v0, 0));

  // keys: p bits above, ~id below; element j = 32 c + lane
  uint64_t key[C];
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const float p = __fmul_rn(e[c], r);
    key[c] = (static_cast<uint64_t>(__float_as_uint(p)) << 32) |
             static_cast<uint32_t>(~(32 * c + lane));
  }
  // bitonic sort, descending
#pragma unroll
  for (int k2 = 2; k2 <= N; k2 <<= 1) {
#pragma unroll
    for (int jj = k2 >> 1; jj > 0; jj >>= 1) {
      uint64_t nk[C];
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const int j = 32 * c + lane;
        const uint64_t other =
            jj >= 32 ? key[c ^ (jj / 32)] : __shfl_xor_sync(full, key[c], jj);
        const bool lower = (j & jj) == 0;
        const bool desc = (j & k2) == 0;
        const uint64_t hi = key[c] > other ? key[c] : other;
        const uint64_t lo = key[c] > other ? other : key[c];
        nk[c] = (lower == desc) ? hi : lo;
      }
#pragma unroll
      for (int c = 0; c < C; ++c) key[c] = nk[c];
    }
  }

  // the elbow over all ranks (rank of element j is j)
  const float pmax = __uint_as_float(static_cast<uint32_t>(__shfl_sync(full, key[0], 0) >> 32));
  const float pmin =
      __uint_as_float(static_cast<uint32_t>(__shfl_sync(full, key[C - 1], 31) >> 32));
  const float inv = __frcp_rn(__fadd_rn(__fsub_rn(pmax, pmin), eps));
  float best = 0.0f;
  int bi = 0;
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const int i = 32 * c + lane;
    const float p = __uint_as_float(static_cast<uint32_t>(key[c] >> 32));
    const float pn = __fmul_rn(__fsub_rn(p, pmin), inv);
    const float xi = __fdiv_rn(static_cast<float>(i), static_cast<float>(N - 1));
    const float D = __fsub_rn(__fsub_rn(1.0f, pn), xi);
    if (c == 0 || D > best) {
      best = D;
      bi = i;
    }
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    const float ob = __shfl_xor_sync(full, best, o);
    const int oi = __shfl_xor_sync(full, bi, o);
    if (ob > best || (ob == best && oi < bi)) {
      best = ob;
      bi = oi;
    }
  }
  const int k = topk_mode ? K : min(bi + 1, K);

  // ranks 0 .. K-1 are slot 0 of lanes 0 .. K-1
  const float p = __uint_as_float(static_cast<uint32_t>(key[0] >> 32));
  const int id = static_cast<int>(~static_cast<uint32_t>(key[0]));
  float S = 0.0f;
  if (renorm) {
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      const float ps = __shfl_sync(full, p, s);
      if (s < k) S = __fadd_rn(S, ps);
    }
  }
  if (lane < K) {
    ids_out[t * K + lane] = id;
    gates_out[t * K + lane] = lane < k ? (renorm ? __fdiv_rn(p, S) : p) : 0.0f;
  }
  if (lane == 0) k_out[t] = k;
}

template <int N>
__global__ void __launch_bounds__(32 * kWarps) route_warp_kernel(
    const float* __restrict__ src, int64_t T, int nslice, int K, float eps, int topk_mode,
    int renorm, float* __restrict__ logits_out, int32_t* __restrict__ k_out,
    int32_t* __restrict__ ids_out, float* __restrict__ gates_out) {
  const int64_t t = static_cast<int64_t>(blockIdx.x) * kWarps + threadIdx.x / 32;
  if (t >= T) return;  // uniform per warp
  route_one_warp<N, false>(src, t, T, nslice, K, eps, topk_mode, renorm, logits_out, k_out,
                           ids_out, gates_out);
}

// The small-batch router in one launch: every block writes its slice's
// partial sums; the block that finishes last (a ticket counter, after a
// memory fence: no block waits for another) routes all T tokens with its
// eight warps, reading the partials from L2, and resets the counter.
template <int N>
__global__ void __launch_bounds__(256) router_small_route_kernel(
    const uint32_t* __restrict__ x, const uint32_t* __restrict__ w, int T, int d,
    float* __restrict__ partial, unsigned int* __restrict__ ticket, int K, float eps, int topk_mode,
    int renorm, float* __restrict__ logits_out, int32_t* __restrict__ k_out,
    int32_t* __restrict__ ids_out, float* __restrict__ gates_out) {
  router_small_body<N>(x, w, T, d, partial);
  __threadfence();
  __syncthreads();
  __shared__ bool last;
  if (threadIdx.x == 0) last = atomicAdd(ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!last) return;
  __threadfence();
  for (int t = threadIdx.x / 32; t < T; t += 8)
    route_one_warp<N, true>(partial, t, T, static_cast<int>(gridDim.x), K, eps, topk_mode, renorm,
                            logits_out, k_out, ids_out, gates_out);
  if (threadIdx.x == 0) *ticket = 0u;
}

}  // namespace rwarp

// Warp-per-token routing of fp32 logits [T, N] (or of `nslice` partial sums
// of them, [nslice][T][N]); logits_out (nullable) receives the summed logits.
cudaError_t launch_route_warp(const float* src, int nslice, int64_t T, int N, int K, float eps,
                              int topk_mode, int renorm, float* logits_out, int32_t* k_out,
                              int32_t* ids_out, float* gates_out, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  const int64_t blocks = (T + rwarp::kWarps - 1) / rwarp::kWarps;
  if (N == 64)
    rwarp::route_warp_kernel<64><<<static_cast<unsigned>(blocks), 32 * rwarp::kWarps, 0, stream>>>(
        src, T, nslice, K, eps, topk_mode, renorm, logits_out, k_out, ids_out, gates_out);
  else
    rwarp::route_warp_kernel<128><<<static_cast<unsigned>(blocks), 32 * rwarp::kWarps, 0, stream>>>(
        src, T, nslice, K, eps, topk_mode, renorm, logits_out, k_out, ids_out, gates_out);
  return cudaGetLastError();
}

// Router logits of T <= 64 tokens (as d / 64 partial sums, partial [d/64][T][N])
// and their routing, in one launch; ticket: a zeroed device counter, left zero.
cudaError_t launch_router_small_route(const uint16_t* x, const uint16_t* w_router, int T, int d,
                                      int N, float* partial, unsigned int* ticket, int K, float eps,
                                      int topk_mode, int renorm, float* logits_out, int32_t* k_out,
                                      int32_t* ids_out, float* gates_out, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  const unsigned slices = static_cast<unsigned>(d / rwarp::kSlice);
  auto xx = reinterpret_cast<const uint32_t*>(x);
  auto ww = reinterpret_cast<const uint32_t*>(w_router);
  if (N == 64)
    rwarp::router_small_route_kernel<64><<<slices, 256, 0, stream>>>(
        xx, ww, T, d, partial, ticket, K, eps, topk_mode, renorm, logits_out, k_out, ids_out,
        gates_out);
  else
    rwarp::router_small_route_kernel<128><<<slices, 256, 0, stream>>>(
        xx, ww, T, d, partial, ticket, K, eps, topk_mode, renorm, logits_out, k_out, ids_out,
        gates_out);
  return cudaGetLastError();
}

}  // namespace moe
