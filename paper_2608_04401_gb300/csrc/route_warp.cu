// Small-batch routing: one WARP per token, for batches too small to hide the
// ~2500-instruction chain that one thread per token needs (decode steps).
//
// Lane l holds experts l + 32c (c < N/32). The arithmetic is the routing
// specification of route_impl.cuh, step for step, so the results are the same
// bits as the thread-per-token kernels and the oracle:
//   m = max l (warp reduction); e_j = EXP(l_j - m) (the packed spec
//   exponential); s = balanced tree sum (levels h >= 32 inside the lane, then
//   v_i += v_{i+h} by shuffles); p_j = e_j / s (correctly rounded);
//   a bitonic sort of the N keys (p bits << 32 | ~id) across the warp (64-bit
//   shuffles), which orders by p descending and ascending id on ties;
//   p'_i, D_i on each rank, the first argmax by a (max D, min index) warp
//   reduction, k = min(e + 1, K). The steps from p on are warp_route_from_e
//   (route_impl.cuh), which also routes the tokens that the thread-per-token
//   kernels leave undecided.
//
// router_small_route_kernel: the router GEMM for T <= 64 tokens on CUDA cores,
// split over d in slices of 64 columns and over tokens in groups of 16 (one
// block per slice and group) so that many SMs share the work instead of one
// SM streaming all of x and W_r:
// partial[s][t][e] = sum_{k in slice s} x[t][k] w[e][k], fp32 fma in k order;
// in each group the block that finishes last adds the slices in order and
// routes the group's tokens.
//
// router_few_kernel: the router of a step of at most 4 tokens with its routing
// and dispatch, on one cluster of 8 CTAs that add their column slices' sums
// through distributed shared memory (no global scratch, no counter).
#include "route_impl.cuh"

namespace moe {
namespace rwarp {

constexpr int kWarps = 4;            // tokens per block of the routing kernel
constexpr int kSlice = 64;           // d columns per block of the small router GEMM
constexpr int kGroupT = 16;          // tokens per block of the small router GEMM
constexpr int kSmallT = 64;          // largest batch of the small router
constexpr int kSmallThreads = 512;   // threads per block of the small router (16 warps)
constexpr int kPitch2 = kSlice / 2 + 1;  // row pitch in bf16 pairs (odd: no bank conflicts)

// acc[i] = sum over the slice's columns of x[t_i] w[e], t_i = g + G * i, fp32
// fma in column order (xs, wrow: bf16 pairs in shared memory).
template <int NT, int G>
MOE_DEV void slice_dots(const uint32_t (*xs)[kPitch2], const uint32_t* wrow, int g,
                        float (&acc)[NT]) {
#pragma unroll
  for (int i = 0; i < NT; ++i) acc[i] = 0.0f;
#pragma unroll 8
  for (int c = 0; c < kSlice / 2; ++c) {
    const float2 wv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&wrow[c]));
#pragma unroll
    for (int i = 0; i < NT; ++i) {
      const float2 xv =
          __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&xs[g + G * i][c]));
      acc[i] = fmaf(xv.x, wv.x, acc[i]);
      acc[i] = fmaf(xv.y, wv.y, acc[i]);
    }
  }
}

// Thread (e, g) of G = kSmallThreads / N groups: the partial sums of its NT
// tokens g, g + G, ... of the block's token group (NT is the thread's token
// count as a compile-time constant, so that no accumulator idles).
template <int N, int NT>
MOE_DEV void slice_tokens(const uint32_t (*xs)[kPitch2], const uint32_t* wrow, int g, int e,
                          float* __restrict__ out) {
  constexpr int G = kSmallThreads / N;
  float acc[NT];
  slice_dots<NT, G>(xs, wrow, g, acc);
#pragma unroll
  for (int i = 0; i < NT; ++i) out[(g + G * i) * N + e] = acc[i];
}

// Block (s, j): the partial sums of tokens t0 = 16 j .. t0 + nj - 1 over the
// d columns [64 s, 64 s + 64): partial[s][t0 + r][e].
template <int N>
MOE_DEV void router_small_body(const uint32_t* __restrict__ x, const uint32_t* __restrict__ w, int T,
                               int d, int t0, int nj, float* __restrict__ partial) {
  __shared__ uint32_t xs[kGroupT][kPitch2];  // bf16 pairs
  __shared__ uint32_t wsm[N][kPitch2];
  const int s = blockIdx.x;
  const int d2 = d / 2;
  const int c0 = s * (kSlice / 2);
  // 16-byte loads (four bf16 pairs), stored as single pairs into the odd pitch
  constexpr int kVec = kSlice / 8;  // uint4 per row slice
  for (int i = threadIdx.x; i < (nj + N) * kVec; i += kSmallThreads) {
    const int r = i / kVec, c = (i % kVec) * 4;
    const bool is_x = r < nj;
    const uint32_t* src = is_x ? x + static_cast<int64_t>(t0 + r) * d2
                               : w + static_cast<int64_t>(r - nj) * d2;
    const uint4 v = *reinterpret_cast<const uint4*>(src + c0 + c);
    uint32_t* dst = is_x ? &xs[r][c] : &wsm[r - nj][c];
    dst[0] = v.x; dst[1] = v.y; dst[2] = v.z; dst[3] = v.w;
  }
  __syncthreads();
  constexpr int G = kSmallThreads / N;
  const int e = threadIdx.x % N, g = threadIdx.x / N;
  if (g >= nj) return;  // whole warps (N >= 64)
  const int nt = (nj - g + G - 1) / G;  // 1 .. kGroupT / G
  float* out = partial + (static_cast<int64_t>(s) * T + t0) * N;
  switch (nt) {
    case 1: slice_tokens<N, 1>(xs, wsm[e], g, e, out); break;
    case 2: slice_tokens<N, 2>(xs, wsm[e], g, e, out); break;
    default:
      if constexpr (kGroupT / G > 2) {
        if (nt == 3) slice_tokens<N, 3>(xs, wsm[e], g, e, out);
        else slice_tokens<N, 4>(xs, wsm[e], g, e, out);
      }
  }
}

// Routes token t with the calling (whole, converged) warp from its logits
// row[0 .. N) (global or shared memory).
template <int N>
MOE_DEV void route_one_warp(const float* __restrict__ row, int64_t t, int K, float eps,
                            int topk_mode, int renorm, int32_t* __restrict__ k_out,
                            int32_t* __restrict__ ids_out, float* __restrict__ gates_out) {
  constexpr int C = N / 32;
  const unsigned full = 0xffffffffu;
  const int lane = threadIdx.x & 31;

  float l[C];
#pragma unroll
  for (int c = 0; c < C; ++c) l[c] = row[32 * c + lane];
  float m = l[0];
#pragma unroll
  for (int c = 1; c < C; ++c) m = fmaxf(m, l[c]);
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) m = fmaxf(m, __shfl_xor_sync(full, m, o));
  MOE_DCHECK(isfinite(m));

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
  const float s = __shfl_sync(full, v0, 0);

  int sel_id;
  route::warp_route_from_e<N>(e, s, t, K, eps, topk_mode, renorm, k_out, ids_out, gates_out,
                              sel_id);
}

template <int N>
__global__ void __launch_bounds__(32 * kWarps) route_warp_kernel(
    const float* __restrict__ logits, int64_t T, int K, float eps, int topk_mode, int renorm,
    int32_t* __restrict__ k_out, int32_t* __restrict__ ids_out, float* __restrict__ gates_out) {
  const int64_t t = static_cast<int64_t>(blockIdx.x) * kWarps + threadIdx.x / 32;
  if (t >= T) return;  // uniform per warp
  route_one_warp<N>(logits + t * N, t, K, eps, topk_mode, renorm, k_out, ids_out, gates_out);
}

// The small-batch router in one launch: block (s, j) writes the partial sums
// of slice s for token group j; the block of group j that finishes last (a
// ticket counter per group, taken by an acquire-release atomic after a block
// barrier: no block waits for another) adds them up in slice order with all its threads (two pairs'
// loads in flight per thread), keeps the group's logits in shared memory,
// routes its tokens with one warp each and resets the counter.
template <int N>
__global__ void __launch_bounds__(kSmallThreads) router_small_route_kernel(
    const uint32_t* __restrict__ x, const uint32_t* __restrict__ w, int T, int d,
    float* __restrict__ partial, unsigned int* __restrict__ ticket, int K, float eps, int topk_mode,
    int renorm, float* __restrict__ logits_out, int32_t* __restrict__ k_out,
    int32_t* __restrict__ ids_out, float* __restrict__ gates_out) {
  __shared__ float lg[kGroupT * N];
  __shared__ bool last;
  grid_dep_wait();
  grid_dep_launch();
  const int t0 = blockIdx.y * kGroupT;
  const int nj = min(kGroupT, T - t0);
  router_small_body<N>(x, w, T, d, t0, nj, partial);
  // the block's partial sums happen before thread 0's release (the barrier);
  // the acquire half makes every earlier block's sums visible to the last one
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned int prev;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;"
                 : "=r"(prev) : "l"(ticket + blockIdx.y) : "memory");
    last = prev == gridDim.x - 1;
  }
  __syncthreads();
  if (!last) return;
  const int nslice = static_cast<int>(gridDim.x);
  const int64_t stride = static_cast<int64_t>(T) * N;
  const float* src = partial + static_cast<int64_t>(t0) * N;
  float* dst = logits_out ? logits_out + static_cast<int64_t>(t0) * N : nullptr;
  const int npair = nj * N;
  auto sum_slices = [&](int i0, int i1) {  // pairs i0 and i1 (i1 may be past the end)
    const bool two = i1 < npair;
    float a0 = __ldcg(src + i0), a1 = two ? __ldcg(src + i1) : 0.0f;
    int sl = 1;
    for (; sl + 16 <= nslice; sl += 16) {
      float q0[16], q1[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        q0[u] = __ldcg(src + (sl + u) * stride + i0);
        q1[u] = two ? __ldcg(src + (sl + u) * stride + i1) : 0.0f;
      }
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        a0 = __fadd_rn(a0, q0[u]);
        a1 = __fadd_rn(a1, q1[u]);
      }
    }
    for (; sl < nslice; ++sl) {
      a0 = __fadd_rn(a0, __ldcg(src + sl * stride + i0));
      if (two) a1 = __fadd_rn(a1, __ldcg(src + sl * stride + i1));
    }
    lg[i0] = a0;
    if (dst) dst[i0] = a0;
    if (two) {
      lg[i1] = a1;
      if (dst) dst[i1] = a1;
    }
  };
  for (int i = threadIdx.x; i < npair; i += 2 * kSmallThreads) sum_slices(i, i + kSmallThreads);
  __syncthreads();
  const int wp = threadIdx.x / 32;
  if (wp < nj)
    route_one_warp<N>(lg + wp * N, t0 + wp, K, eps, topk_mode, renorm, k_out, ids_out, gates_out);
  if (threadIdx.x == 0) ticket[blockIdx.y] = 0u;
}

// ----------------------------------------------------- few-token router
// The router of a step of T <= 4 tokens on one cluster of kFewCtas CTAs, with
// the step's dispatch, and no global scratch or counter: CTA r forms the dots
// of columns [r cs, (r + 1) cs), cs = d / kFewCtas, thread (e, q) (q fastest)
// over the 16-byte chunks q, q + Q, ... of that range, for every token (each
// an fp32 fma chain in column order; the Q chains of an expert added by a
// shuffle tree); the cluster's CTA 0 adds the CTAs' sums in rank order through
// distributed shared memory, routes token t with warp t and writes the
// dispatch. Its rows are the selected pairs (t, s), s < k_t (a token selects
// an expert once), by expert id and then by token: offsets[e] = the number of
// pairs with an id below e; the row of pair (t, s) is that count for its id
// plus the pairs of the same expert from tokens before t; perm[row] = t;
// pair_pos[t, s] = the row, or -1 for s >= k_t. CTA 0 also zeroes
// clear[0 .. nclear) (the step's error word and counters) once the previous
// kernel has finished.
constexpr int kFewCtas = 8;
constexpr int kFewThreads = 512;
constexpr int kFewMaxT = 4;

struct FewTokenOut {
  float* logits;          // [T, N] or nullptr
  int32_t* k;             // [T]
  int32_t* ids;           // [T, K]
  float* gates;           // [T, K]
  int32_t* offsets;       // [N + 1]
  int32_t* perm;          // [T K]
  int32_t* pair_pos;      // [T, K]
  int32_t* offsets_copy;  // [N + 1] or nullptr
  int32_t* clear;         // [nclear]
  int nclear;
};

template <int N, int T>
__global__ void __launch_bounds__(kFewThreads) router_few_kernel(
    const uint4* __restrict__ x, const uint4* __restrict__ w, int d, int K, float eps,
    int topk_mode, int renorm, FewTokenOut out) {
  constexpr int Q = kFewThreads / N;  // chains per expert
  __shared__ float part[T][N];
  __shared__ float lg[T][N];
  grid_dep_wait();
  grid_dep_launch();
  const uint32_t rank = cluster_rank();
  const int d8 = d / 8;                // 16-byte chunks per row
  const int cs8 = d8 / kFewCtas;       // chunks per CTA
  const int q = threadIdx.x % Q, e = threadIdx.x / Q;
  const uint4* wr = w + static_cast<int64_t>(e) * d8 + rank * cs8;
  const uint4* xr = x + rank * cs8;
  float acc[T];
#pragma unroll
  for (int t = 0; t < T; ++t) acc[t] = 0.0f;
#pragma unroll 4
  for (int u = q; u < cs8; u += Q) {
    const uint4 wv = __ldg(wr + u);
    const uint32_t wa[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
    for (int t = 0; t < T; ++t) {
      const uint4 xv = __ldg(xr + static_cast<int64_t>(t) * d8 + u);
      const uint32_t xa[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        acc[t] = fmaf(__uint_as_float(xa[c] << 16), __uint_as_float(wa[c] << 16), acc[t]);
        acc[t] = fmaf(__uint_as_float(xa[c] & 0xFFFF0000u), __uint_as_float(wa[c] & 0xFFFF0000u),
                      acc[t]);
      }
    }
  }
#pragma unroll
  for (int t = 0; t < T; ++t) {
#pragma unroll
    for (int o = Q / 2; o >= 1; o >>= 1) acc[t] += __shfl_xor_sync(0xffffffffu, acc[t], o);
    if (q == 0) part[t][e] = acc[t];
  }
  if (rank == 0)
    for (int i = threadIdx.x; i < out.nclear; i += kFewThreads) out.clear[i] = 0;
  cluster_sync();  // every CTA's part[] is written
  if (rank == 0) {
    for (int i = threadIdx.x; i < T * N; i += kFewThreads) {
      const int t = i / N, ee = i % N;
      const uint32_t a = smem_u32(&part[t][ee]);
      float l = ld_cluster_f32(map_to_rank(a, 0));
      for (int r = 1; r < kFewCtas; ++r) l = __fadd_rn(l, ld_cluster_f32(map_to_rank(a, r)));
      lg[t][ee] = l;
      if (out.logits) out.logits[i] = l;
    }
  }
  cluster_sync();  // CTA 0 is done reading the others' part[]: they may leave
  if (rank != 0) return;
  const int wp = threadIdx.x / 32;
  if (wp < T) route_one_warp<N>(lg[wp], wp, K, eps, topk_mode, renorm, out.k, out.ids, out.gates);
  __syncthreads();  // k and ids are visible to the block
  // pair (t, s) is selected iff s < k_t
  auto kt = [&](int t) { return min(max(out.k[t], 0), K); };
  for (int ee = threadIdx.x; ee <= N; ee += kFewThreads) {
    int below = 0;
    for (int t = 0; t < T; ++t) {
      const int k1 = kt(t);
      for (int s2 = 0; s2 < k1; ++s2) below += out.ids[t * K + s2] < ee ? 1 : 0;
    }
    out.offsets[ee] = below;
    if (out.offsets_copy) out.offsets_copy[ee] = below;
  }
  if (threadIdx.x < T * K) {
    const int t = threadIdx.x / K, s2 = threadIdx.x % K;
    int pos = -1;
    if (s2 < kt(t)) {
      const int id = out.ids[t * K + s2];
      pos = 0;
      for (int t2 = 0; t2 < T; ++t2) {
        const int k2 = kt(t2);
        for (int s3 = 0; s3 < k2; ++s3) {
          const int id2 = out.ids[t2 * K + s3];
          pos += (id2 < id || (id2 == id && t2 < t)) ? 1 : 0;
        }
      }
      out.perm[pos] = t;
    }
    out.pair_pos[threadIdx.x] = pos;
  }
}

}  // namespace rwarp

// Warp-per-token routing of fp32 logits [T, N].
cudaError_t launch_route_warp(const float* logits, int64_t T, int N, int K, float eps,
                              int topk_mode, int renorm, int32_t* k_out, int32_t* ids_out,
                              float* gates_out, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  const int64_t blocks = (T + rwarp::kWarps - 1) / rwarp::kWarps;
  if (N == 64)
    rwarp::route_warp_kernel<64><<<static_cast<unsigned>(blocks), 32 * rwarp::kWarps, 0, stream>>>(
        logits, T, K, eps, topk_mode, renorm, k_out, ids_out, gates_out);
  else
    rwarp::route_warp_kernel<128><<<static_cast<unsigned>(blocks), 32 * rwarp::kWarps, 0, stream>>>(
        logits, T, K, eps, topk_mode, renorm, k_out, ids_out, gates_out);
  return cudaGetLastError();
}

// Router logits of T <= 64 tokens (as d / 64 partial sums, partial [d/64][T][N])
// and their routing, in one launch; ticket: ceil(T / 16) zeroed device
// counters, left zero.
cudaError_t launch_router_small_route(const uint16_t* x, const uint16_t* w_router, int T, int d,
                                      int N, float* partial, unsigned int* ticket, int K, float eps,
                                      int topk_mode, int renorm, float* logits_out, int32_t* k_out,
                                      int32_t* ids_out, float* gates_out, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  if (T > rwarp::kSmallT || d % rwarp::kSlice != 0) return cudaErrorInvalidValue;
  const dim3 grid(static_cast<unsigned>(d / rwarp::kSlice),
                  static_cast<unsigned>((T + rwarp::kGroupT - 1) / rwarp::kGroupT));
  auto xx = reinterpret_cast<const uint32_t*>(x);
  auto ww = reinterpret_cast<const uint32_t*>(w_router);
  auto kern = N == 64 ? rwarp::router_small_route_kernel<64> : rwarp::router_small_route_kernel<128>;
  return launch_pdl(kern, grid, dim3(rwarp::kSmallThreads), 0, stream, xx, ww, T, d, partial, ticket, K,
                    eps, topk_mode, renorm, logits_out, k_out, ids_out, gates_out);
}

// Router, routing and dispatch of T <= 4 tokens (d a multiple of 64): one
// cluster of 8 CTAs. Writes logits_out [T, N] (if not null), k_out [T],
// ids_out and gates_out [T, K], offsets [N + 1], perm [T K], pair_pos [T, K]
// and offsets_copy [N + 1] (if not null), and zeroes clear [nclear] after the
// previous kernel on the stream has finished.
cudaError_t launch_router_few(const uint16_t* x, const uint16_t* w_router, int T, int d, int N,
                              int K, float eps, int topk_mode, int renorm, float* logits_out,
                              int32_t* k_out, int32_t* ids_out, float* gates_out, int32_t* offsets,
                              int32_t* perm, int32_t* pair_pos, int32_t* offsets_copy,
                              int32_t* clear, int nclear, cudaStream_t stream) {
  if (T < 1 || T > rwarp::kFewMaxT || d % (8 * rwarp::kFewCtas) != 0 || (N != 64 && N != 128) ||
      nclear < 0 || T * K > rwarp::kFewThreads)
    return cudaErrorInvalidValue;
  const rwarp::FewTokenOut out{logits_out, k_out, ids_out, gates_out, offsets, perm,
                               pair_pos, offsets_copy, clear, nclear};
  auto xx = reinterpret_cast<const uint4*>(x);
  auto ww = reinterpret_cast<const uint4*>(w_router);
  using Kern = void (*)(const uint4*, const uint4*, int, int, float, int, int, rwarp::FewTokenOut);
  static const Kern kerns[2][rwarp::kFewMaxT] = {
      {rwarp::router_few_kernel<64, 1>, rwarp::router_few_kernel<64, 2>,
       rwarp::router_few_kernel<64, 3>, rwarp::router_few_kernel<64, 4>},
      {rwarp::router_few_kernel<128, 1>, rwarp::router_few_kernel<128, 2>,
       rwarp::router_few_kernel<128, 3>, rwarp::router_few_kernel<128, 4>}};
  return launch_cluster_pdl(kerns[N == 128][T - 1], dim3(rwarp::kFewCtas),
                            dim3(rwarp::kFewThreads), 0, stream, rwarp::kFewCtas, xx, ww, d, K,
                            eps, topk_mode, renorm, out);
}

MOE_DEBUG_TU(route_warp)

}  // namespace moe
