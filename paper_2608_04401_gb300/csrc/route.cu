// Elbow router (Alg. 1 + the capped selection of Sec. 2.1), one THREAD per token.
//
// A block routes 128 tokens. Its [128, N] fp32 logit tile is staged through
// shared memory with coalesced 16-byte loads (rows padded by 4 floats so that
// each thread's row reads are bank-conflict free). Each thread then keeps its
// token's N values in registers and runs, in fp32 with every operation
// rounded to nearest even (explicit __f*_rn intrinsics, no contraction):
//   m = max_j l_j; e_j = EXP(l_j - m); s = balanced tree sum; p_j = e_j * (1/s)
//   sort p descending (Batcher odd-even merge network, fmaxf/fminf: exact)
//   p' = (p_(i) - p_min) * (1 / ((p_max - p_min) + eps)); x' = i / (N-1)
//   D_i = (1 - p'_i) - x'_i ; e = smallest argmax ; k = min(e + 1, K)
// The ids of the K largest probabilities are recovered from the unsorted row
// in shared memory by a threshold scan (value > p_(K-1), plus the lowest-id
// ties at p_(K-1)), then ordered by (p desc, id asc) with an 8-key network.
#include <utility>

#include "common.cuh"

namespace moe {
namespace route {

// EXP: Cody & Waite (1980) argument reduction with ln 2 split in two (the high
// part has 16 significant bits, so n * kLn2Hi is exact), a degree-7 Taylor
// polynomial of exp on the reduced argument in Horner form with fused
// multiply-adds, and scaling by 2^n built from the exponent bits. Results
// below 2^-126 are flushed to zero.
constexpr float kLog2e = 0x1.715476p+0f;  // fp32(1 / ln 2)
constexpr float kLn2Hi = 0x1.62e4p-1f;    // ln 2 to 16 significant bits
constexpr float kLn2Lo = 0x1.7f7d1cp-20f; // fp32(ln 2 - kLn2Hi)
// Taylor coefficients 1/j!, each rounded once to fp32.
constexpr float kTay0 = static_cast<float>(1.0 / 1.0);
constexpr float kTay1 = static_cast<float>(1.0 / 1.0);
constexpr float kTay2 = static_cast<float>(1.0 / 2.0);
constexpr float kTay3 = static_cast<float>(1.0 / 6.0);
constexpr float kTay4 = static_cast<float>(1.0 / 24.0);
constexpr float kTay5 = static_cast<float>(1.0 / 120.0);
constexpr float kTay6 = static_cast<float>(1.0 / 720.0);
constexpr float kTay7 = static_cast<float>(1.0 / 5040.0);

MOE_DEV float exp_spec(float z) {
  if (!(z >= -104.0f)) return 0.0f;
  if (z > 88.0f) return __int_as_float(0x7f800000);
  const float n = rintf(__fmul_rn(z, kLog2e));
  float r = __fmaf_rn(-n, kLn2Hi, z);
  r = __fmaf_rn(-n, kLn2Lo, r);
  float q = kTay7;
  q = __fmaf_rn(q, r, kTay6);
  q = __fmaf_rn(q, r, kTay5);
  q = __fmaf_rn(q, r, kTay4);
  q = __fmaf_rn(q, r, kTay3);
  q = __fmaf_rn(q, r, kTay2);
  q = __fmaf_rn(q, r, kTay1);
  q = __fmaf_rn(q, r, kTay0);
  const int ni = static_cast<int>(n);
  if (ni < -126) return 0.0f;
  return __fmul_rn(q, __int_as_float((ni + 127) << 23));
}

// Batcher's odd-even merge sort network for N keys, as a flat comparator list
// built at compile time (so that every register index is a constant).
template <int N>
struct OddEvenMergeNet {
  static constexpr int count() {
    int c = 0;
    for (int p = 1; p < N; p <<= 1)
      for (int k = p; k >= 1; k >>= 1)
        for (int j = k % p; j + k < N; j += 2 * k)
          for (int i = 0; i < k && i + j + k < N; ++i)
            if ((i + j) / (2 * p) == (i + j + k) / (2 * p)) ++c;
    return c;
  }
  static constexpr int kCount = count();
  int lo[kCount];
  int hi[kCount];
  constexpr OddEvenMergeNet() : lo(), hi() {
    int c = 0;
    for (int p = 1; p < N; p <<= 1)
      for (int k = p; k >= 1; k >>= 1)
        for (int j = k % p; j + k < N; j += 2 * k)
          for (int i = 0; i < k && i + j + k < N; ++i)
            if ((i + j) / (2 * p) == (i + j + k) / (2 * p)) {
              lo[c] = i + j;
              hi[c] = i + j + k;
              ++c;
            }
  }
};

template <int N>
struct NetOf {
  static constexpr OddEvenMergeNet<N> net{};
};

template <int A, int B, int N>
MOE_DEV void cex_desc(float (&v)[N]) {
  const float a = v[A], b = v[B];
  v[A] = fmaxf(a, b);
  v[B] = fminf(a, b);
}

template <int N, size_t... C>
MOE_DEV void apply_net(float (&v)[N], std::index_sequence<C...>) {
  (cex_desc<NetOf<N>::net.lo[C], NetOf<N>::net.hi[C]>(v), ...);
}

// Sorts a register array in descending order (fmaxf/fminf are exact). The
// comparators are expanded at compile time: every index is a constant.
template <int N>
MOE_DEV void sort_desc(float (&v)[N]) {
  apply_net<N>(v, std::make_index_sequence<OddEvenMergeNet<N>::kCount>{});
}

// Balanced tree sum in place: v[i] += v[i + H] for i < H, then H/2, ..., 1;
// the total ends in v[0].
template <int H, int N>
MOE_DEV void tree_sum_level(float (&v)[N]) {
#pragma unroll
  for (int i = 0; i < H; ++i) v[i] = __fadd_rn(v[i], v[i + H]);
  if constexpr (H > 1) tree_sum_level<H / 2>(v);
}

MOE_DEV void cex_desc_u64(uint64_t& a, uint64_t& b) {
  const uint64_t hi = a > b ? a : b, lo = a > b ? b : a;
  a = hi;
  b = lo;
}

// 19-comparator sorting network for 8 keys (descending).
MOE_DEV void sort8_desc(uint64_t (&k)[8]) {
  cex_desc_u64(k[0], k[2]); cex_desc_u64(k[1], k[3]); cex_desc_u64(k[4], k[6]); cex_desc_u64(k[5], k[7]);
  cex_desc_u64(k[0], k[4]); cex_desc_u64(k[1], k[5]); cex_desc_u64(k[2], k[6]); cex_desc_u64(k[3], k[7]);
  cex_desc_u64(k[0], k[1]); cex_desc_u64(k[2], k[3]); cex_desc_u64(k[4], k[5]); cex_desc_u64(k[6], k[7]);
  cex_desc_u64(k[2], k[4]); cex_desc_u64(k[3], k[5]);
  cex_desc_u64(k[1], k[4]); cex_desc_u64(k[3], k[6]);
  cex_desc_u64(k[1], k[2]); cex_desc_u64(k[3], k[4]); cex_desc_u64(k[5], k[6]);
}

constexpr int kTok = 128;  // tokens (threads) per block

template <int N>
struct XGrid {
  float x[N];  // x'_i = i / (N - 1), computed on the host in fp32
};

template <int N>
constexpr size_t smem_bytes() {
  return sizeof(float) * kTok * (N + 4) + sizeof(uint64_t) * 8 * kTok;
}

template <int N>
__global__ void __launch_bounds__(kTok) elbow_route_kernel(
    const float* __restrict__ logits, int64_t T, int K, float eps, int topk_mode, int renorm,
    const __grid_constant__ XGrid<N> xg, int32_t* __restrict__ k_out, int32_t* __restrict__ ids_out,
    float* __restrict__ gates_out) {
  constexpr int kPitch = N + 4;
  extern __shared__ float4 smem4[];
  float* tile = reinterpret_cast<float*>(smem4);
  uint64_t* keys = reinterpret_cast<uint64_t*>(tile + kTok * kPitch);  // [8][kTok]

  const int64_t t0 = static_cast<int64_t>(blockIdx.x) * kTok;
  const int ntok = static_cast<int>(min_of<int64_t>(kTok, T - t0));
  const int tid = threadIdx.x;

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
  if (tid >= ntok) return;  // no block-wide barrier below this point

  float* row = tile + tid * kPitch;
  float v[N];
#pragma unroll
  for (int c = 0; c < N; c += 4) {
    const float4 q = *reinterpret_cast<const float4*>(row + c);
    v[c] = q.x; v[c + 1] = q.y; v[c + 2] = q.z; v[c + 3] = q.w;
  }

  // ---- p = softmax(l)
  float m = v[0];
#pragma unroll
  for (int j = 1; j < N; ++j) m = fmaxf(m, v[j]);
#pragma unroll
  for (int j = 0; j < N; ++j) v[j] = exp_spec(__fsub_rn(v[j], m));
#pragma unroll
  for (int c = 0; c < N; c += 4)
    *reinterpret_cast<float4*>(row + c) = make_float4(v[c], v[c + 1], v[c + 2], v[c + 3]);
  tree_sum_level<N / 2>(v);
  const float rs = __frcp_rn(v[0]);
#pragma unroll
  for (int c = 0; c < N; c += 4) {
    const float4 q = *reinterpret_cast<const float4*>(row + c);
    v[c] = __fmul_rn(q.x, rs); v[c + 1] = __fmul_rn(q.y, rs);
    v[c + 2] = __fmul_rn(q.z, rs); v[c + 3] = __fmul_rn(q.w, rs);
    *reinterpret_cast<float4*>(row + c) = make_float4(v[c], v[c + 1], v[c + 2], v[c + 3]);
  }

  // ---- p <- sort_desc(p)
  sort_desc<N>(v);

  // ---- Kneedle elbow and the capped count
  int k = K;
  if (!topk_mode) {
    const float p_min = v[N - 1];
    const float inv = __frcp_rn(__fadd_rn(__fsub_rn(v[0], p_min), eps));
    float best = -__int_as_float(0x7f800000), tail = -__int_as_float(0x7f800000);
    int e = 0;
#pragma unroll
    for (int i = 0; i < N; ++i) {
      const float pn = __fmul_rn(__fsub_rn(v[i], p_min), inv);
      const float D = __fsub_rn(__fsub_rn(1.0f, pn), xg.x[i]);
      if (i < 7) {
        // candidates for an elbow inside the cap (i < K - 1); the rest only
        // matter through their maximum
        if (i < K - 1) {
          if (D > best) { best = D; e = i; }
        } else {
          tail = fmaxf(tail, D);
        }
      } else {
        tail = fmaxf(tail, D);
      }
    }
    k = (best >= tail) ? e + 1 : K;
  }

  // ---- ids of the K largest: threshold scan of the unsorted row
  // p_(K-1), written as the minimum of the first K sorted values (a select on
  // s == K - 1 would be turned into a dynamic index into the register array)
  float thr = v[0];
#pragma unroll
  for (int s = 1; s < 8; ++s)
    if (s < K) thr = fminf(thr, v[s]);
  int above = 0;
#pragma unroll
  for (int s = 0; s < 8; ++s)
    if (s < K && v[s] > thr) ++above;
  const int need_eq = K - above;
  int cnt = 0, eq = 0;
#pragma unroll
  for (int c = 0; c < N; c += 4) {
    const float4 q = *reinterpret_cast<const float4*>(row + c);
    const float pq[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float pj = pq[u];
      const bool is_eq = pj == thr;
      const bool take = (pj > thr) || (is_eq && eq < need_eq);
      eq += is_eq ? 1 : 0;
      if (take && cnt < 8) {
        keys[cnt * kTok + tid] =
            (static_cast<uint64_t>(__float_as_uint(pj)) << 32) | static_cast<uint32_t>(~(c + u));
        ++cnt;
      }
    }
  }
  uint64_t key[8];
#pragma unroll
  for (int s = 0; s < 8; ++s) key[s] = (s < K) ? keys[s * kTok + tid] : 0ull;
  sort8_desc(key);

  // ---- gates
  float g[8];
  float S = 0.0f;
#pragma unroll
  for (int s = 0; s < 8; ++s)
    if (s < k) S = __fadd_rn(S, v[s]);
#pragma unroll
  for (int s = 0; s < 8; ++s) {
    const float p = renorm ? __fdiv_rn(v[s], S) : v[s];
    g[s] = (s < k) ? p : 0.0f;
  }

  const int64_t t = t0 + tid;
  k_out[t] = k;
  if (K == 8) {
    int4* ip = reinterpret_cast<int4*>(ids_out + t * 8);
    float4* gp = reinterpret_cast<float4*>(gates_out + t * 8);
    ip[0] = make_int4(~static_cast<int>(key[0]), ~static_cast<int>(key[1]),
                      ~static_cast<int>(key[2]), ~static_cast<int>(key[3]));
    ip[1] = make_int4(~static_cast<int>(key[4]), ~static_cast<int>(key[5]),
                      ~static_cast<int>(key[6]), ~static_cast<int>(key[7]));
    gp[0] = make_float4(g[0], g[1], g[2], g[3]);
    gp[1] = make_float4(g[4], g[5], g[6], g[7]);
  } else {
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if (s < K) {
        ids_out[t * K + s] = ~static_cast<int>(key[s]);
        gates_out[t * K + s] = g[s];
      }
    }
  }
}

template <int N>
cudaError_t launch(const float* logits, int64_t T, int K, float eps, int topk_mode, int renorm,
                   int32_t* k_out, int32_t* ids_out, float* gates_out, cudaStream_t stream) {
  XGrid<N> xg;
  for (int i = 0; i < N; ++i) xg.x[i] = static_cast<float>(i) / static_cast<float>(N - 1);
  constexpr size_t smem = smem_bytes<N>();
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(elbow_route_kernel<N>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const int64_t blocks = (T + kTok - 1) / kTok;
  elbow_route_kernel<N><<<static_cast<unsigned>(blocks), kTok, smem, stream>>>(
      logits, T, K, eps, topk_mode, renorm, xg, k_out, ids_out, gates_out);
  return cudaGetLastError();
}

}  // namespace route

cudaError_t launch_elbow_route(const float* logits, int64_t T, int N, int K, float eps,
                               int topk_mode, int renorm, int32_t* k_out, int32_t* ids_out,
                               float* gates_out, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  if (N == 64)
    return route::launch<64>(logits, T, K, eps, topk_mode, renorm, k_out, ids_out, gates_out, stream);
  return route::launch<128>(logits, T, K, eps, topk_mode, renorm, k_out, ids_out, gates_out, stream);
}

}  // namespace moe
