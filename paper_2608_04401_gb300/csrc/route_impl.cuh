// Elbow router (Alg. 1 + the capped selection of Sec. 2.1), one THREAD per token.
//
// A block routes 128 tokens. Its [128, N] fp32 logit tile is staged through
// shared memory with coalesced 16-byte loads (rows padded by 4 floats so that
// each thread's row reads are bank-conflict free). Each thread keeps its
// token's values in registers and evaluates, in fp32 with every operation
// rounded to nearest even (explicit .rn intrinsics / PTX, no contraction):
//   m = max_j l_j; e_j = EXP(l_j - m); s = balanced tree sum; p_j = e_j / s
//   sort p descending; p' = (p_(i) - p_min) / ((p_max - p_min) + eps);
//   x' = i / (N-1); D_i = (1 - p'_i) - x'_i; e = smallest argmax; k = min(e+1, K)
// Each quotient is the correctly rounded one (quot / quot2 below).
//
// Fast path. The elbow decision only needs the exact curve at the top ranks:
// for every rank i, D_i <= fl(1 - x'_i), so ranks i >= kTop - 1 cannot beat a
// head value >= fl(1 - x'_{kTop-1}). The thread therefore selects the kTop = 32
// largest values exactly, with the expert id carried in the low bits of a
// 32-bit key (the key orders by the truncated value, then by ascending id);
// exact values come back from the shared-memory row by id, and two checks
// prove that the selected ranks are the exact top ranks in exact order. Then:
//   M_head = max_{i < K-1} D_i (first argmax), M_mid = max_{K-1 <= i < kTop-1} D_i
//   M_head >= M_mid and M_head >= bound  ->  k = argmax + 1
//   M_mid > M_head                        ->  k = K (the elbow lies at or past K-1)
//   otherwise, or when a check fails      ->  undecided (rare)
// Sorting is by e, not p; p = fl(e / s) is monotone in e, so the curve is
// the same, and ids inside groups of equal p are re-ordered by ascending id.
// A p tie across the K boundary also leaves the token undecided.
//
// Undecided tokens (same arithmetic, every rank): the whole warp routes each
// of them in turn from its softmax numerators, sorting all N (p, id) keys by
// a bitonic network of shuffles (route_undecided / warp_route_from_e), instead
// of one lane running a full sort while the rest of its warp waits.
#pragma once

#include <utility>

#include "common.cuh"

namespace moe {
namespace route {

// EXP: Cody & Waite (1980) argument reduction with ln 2 split in two (the high
// part has 16 significant bits, so n * kLn2Hi is exact), a degree-7 Taylor
// polynomial of exp on the reduced argument in Horner form with fused
// multiply-adds, and scaling by 2^n built from the exponent bits. Results
// below 2^-126, and arguments below -104, give zero.
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
// Adding 1.5 * 2^23 to |t| < 2^22 rounds t to an integer (to nearest, ties to
// even) in the low mantissa bits: that sum minus the constant is rint(t), and
// its bit pattern minus kMagicBits is rint(t) as an integer.
constexpr float kMagic = 0x1.8p23f;
constexpr int32_t kMagicBits = 0x4B400000;

constexpr int kTok = 128;  // tokens (threads) per block
constexpr int kTop = 32;   // ranks selected exactly on the fast path

// ------------------------------------------------------- packed fp32 pairs
MOE_DEV uint64_t pk(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
MOE_DEV float lo_of(uint64_t v) { return __uint_as_float(static_cast<uint32_t>(v)); }
MOE_DEV float hi_of(uint64_t v) { return __uint_as_float(static_cast<uint32_t>(v >> 32)); }
MOE_DEV uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
MOE_DEV uint64_t sub2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
MOE_DEV uint64_t mul2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
MOE_DEV uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
MOE_DEV float max3f(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}
MOE_DEV float min3f(float a, float b, float c) {
  float r;
  asm("min.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// -------------------------------------------- correctly rounded quotients
// The softmax p_j = e_j / s and Alg. 1's p'_i = (p_(i) - p_min) / den are
// quotients rounded once. With y = RN(1/b) taken once per divisor b, each
// quotient a / b costs a product and four fused multiply-adds (Markstein's
// correction, IBM J. Res. Dev. 34(1), 1990):
//   q0 = RN(a y)                 within 2 ulp of a / b
//   q1 = RN(q0 + RN(a - b q0) y) within 1 ulp (a neighbour of a / b)
//   r  = a - b q1                exact in one fma
//   q  = RN(q1 + r y)            = RN(a / b)
// The last step's rounding cannot differ from RN(a / b): q1 + r y differs from
// a / b by (a / b - q1)(b y - 1), |b y - 1| <= B 2^-48 for the 24-bit
// significand B of b, while a / b lies at least 2^-24 ulp / B from any
// midpoint between floats (and never on one). Valid for a == 0 or
// a >= kQuotMin with b in [2^-32, 2^8] (no step underflows); other
// numerators take __fdiv_rn, which gives the same correctly rounded quotient.
constexpr float kQuotMin = 0x1p-90f;
MOE_DEV float quot(float a, float b, float y) {
  if (a != 0.0f && a < kQuotMin) return __fdiv_rn(a, b);
  float q = __fmul_rn(a, y);
  float r = __fmaf_rn(-q, b, a);
  q = __fmaf_rn(r, y, q);
  r = __fmaf_rn(-q, b, a);
  return __fmaf_rn(r, y, q);
}
// Two quotients at once with packed operations: a = (a0, a1), nb = (-b, -b),
// y = (RN(1/b), RN(1/b)). The caller guarantees that both numerators are 0 or
// at least kQuotMin.
MOE_DEV uint64_t quot2(uint64_t a, uint64_t nb, uint64_t y) {
  uint64_t q = mul2(a, y);
  uint64_t r = fma2(q, nb, a);
  q = fma2(r, y, q);
  r = fma2(q, nb, a);
  return fma2(r, y, q);
}

// EXP of two arguments z <= 0 at once with packed fp32 operations. z is
// clamped at -104.5 (every z < -104 gives n < -126, i.e. zero, either way),
// rint comes from the 1.5 * 2^23 addition, and an exponent below -126 is
// clamped to a zero scale.
MOE_DEV uint64_t exp_spec2(uint64_t z) {
  z = pk(fmaxf(lo_of(z), -104.5f), fmaxf(hi_of(z), -104.5f));
  const uint64_t t = mul2(z, pk(kLog2e, kLog2e));
  const uint64_t tm = add2(t, pk(kMagic, kMagic));
  const uint64_t n = sub2(tm, pk(kMagic, kMagic));
  uint64_t r = fma2(n, pk(-kLn2Hi, -kLn2Hi), z);
  r = fma2(n, pk(-kLn2Lo, -kLn2Lo), r);
  uint64_t q = fma2(pk(kTay7, kTay7), r, pk(kTay6, kTay6));
  q = fma2(q, r, pk(kTay5, kTay5));
  q = fma2(q, r, pk(kTay4, kTay4));
  q = fma2(q, r, pk(kTay3, kTay3));
  q = fma2(q, r, pk(kTay2, kTay2));
  q = fma2(q, r, pk(kTay1, kTay1));
  q = fma2(q, r, pk(kTay0, kTay0));
  // 2^n from the integer n = bits(tm) - kMagicBits; n < -126 -> +0.0
  const int32_t b0 = max(__float_as_int(lo_of(tm)), kMagicBits - 127);
  const int32_t b1 = max(__float_as_int(hi_of(tm)), kMagicBits - 127);
  const uint64_t scale = pk(__int_as_float((b0 - kMagicBits + 127) << 23),
                            __int_as_float((b1 - kMagicBits + 127) << 23));
  return mul2(q, scale);
}

// exp_spec2 for arguments z >= -87 (so that n >= -126): both clamps above are
// then no-ops, and this is the same sequence of operations without them.
MOE_DEV uint64_t exp_spec2_inrange(uint64_t z) {
  const uint64_t t = mul2(z, pk(kLog2e, kLog2e));
  const uint64_t tm = add2(t, pk(kMagic, kMagic));
  const uint64_t n = sub2(tm, pk(kMagic, kMagic));
  uint64_t r = fma2(n, pk(-kLn2Hi, -kLn2Hi), z);
  r = fma2(n, pk(-kLn2Lo, -kLn2Lo), r);
  uint64_t q = fma2(pk(kTay7, kTay7), r, pk(kTay6, kTay6));
  q = fma2(q, r, pk(kTay5, kTay5));
  q = fma2(q, r, pk(kTay4, kTay4));
  q = fma2(q, r, pk(kTay3, kTay3));
  q = fma2(q, r, pk(kTay2, kTay2));
  q = fma2(q, r, pk(kTay1, kTay1));
  q = fma2(q, r, pk(kTay0, kTay0));
  const int32_t b0 = __float_as_int(lo_of(tm)), b1 = __float_as_int(hi_of(tm));
  const uint64_t scale = pk(__int_as_float((b0 - kMagicBits + 127) << 23),
                            __int_as_float((b1 - kMagicBits + 127) << 23));
  return mul2(q, scale);
}

// -------------------------------------------------------- sorting networks
// Batcher's odd-even merge sort network for M keys, as a flat comparator list
// built at compile time (so that every register index is a constant).
template <int M>
struct OddEvenMergeNet {
  static constexpr int count() {
    int c = 0;
    for (int p = 1; p < M; p <<= 1)
      for (int k = p; k >= 1; k >>= 1)
        for (int j = k % p; j + k < M; j += 2 * k)
          for (int i = 0; i < k && i + j + k < M; ++i)
            if ((i + j) / (2 * p) == (i + j + k) / (2 * p)) ++c;
    return c;
  }
  static constexpr int kCount = count();
  int lo[kCount];
  int hi[kCount];
  constexpr OddEvenMergeNet() : lo(), hi() {
    int c = 0;
    for (int p = 1; p < M; p <<= 1)
      for (int k = p; k >= 1; k >>= 1)
        for (int j = k % p; j + k < M; j += 2 * k)
          for (int i = 0; i < k && i + j + k < M; ++i)
            if ((i + j) / (2 * p) == (i + j + k) / (2 * p)) {
              lo[c] = i + j;
              hi[c] = i + j + k;
              ++c;
            }
  }
};

// Bitonic merger (half-cleaners of stride M/2 .. 1): sorts a bitonic sequence.
template <int M>
struct BitonicMergeNet {
  static constexpr int count() {
    int c = 0;
    for (int s = M / 2; s >= 1; s >>= 1)
      for (int i = 0; i < M; ++i)
        if ((i & s) == 0) ++c;
    return c;
  }
  static constexpr int kCount = count();
  int lo[kCount];
  int hi[kCount];
  constexpr BitonicMergeNet() : lo(), hi() {
    int c = 0;
    for (int s = M / 2; s >= 1; s >>= 1)
      for (int i = 0; i < M; ++i)
        if ((i & s) == 0) {
          lo[c] = i;
          hi[c] = i + s;
          ++c;
        }
  }
};

template <typename Net>
struct NetHolder {
  static constexpr Net net{};
};

template <int A, int B, typename T, int N>
MOE_DEV void cex_desc(T (&v)[N]) {
  const T a = v[A], b = v[B];
  v[A] = max(a, b);
  v[B] = min(a, b);
}

template <typename Net, int OFF, typename T, int N, size_t... C>
MOE_DEV void apply_net(T (&v)[N], std::index_sequence<C...>) {
  (cex_desc<OFF + NetHolder<Net>::net.lo[C], OFF + NetHolder<Net>::net.hi[C]>(v), ...);
}

// v[OFF .. OFF+M) sorted descending.
template <int M, int OFF, typename T, int N>
MOE_DEV void sort_desc_at(T (&v)[N]) {
  apply_net<OddEvenMergeNet<M>, OFF>(v, std::make_index_sequence<OddEvenMergeNet<M>::kCount>{});
}

// v[A .. A+32) and v[B .. B+32) sorted descending -> v[A .. A+32) = the 32
// largest of both, sorted descending (the pairwise maxima of one run against
// the other reversed form a bitonic sequence holding the 32 largest).
template <int A, int B, typename T, int N, size_t... I>
MOE_DEV void keep_top32_first(T (&v)[N], std::index_sequence<I...>) {
  ((v[A + I] = max(v[A + I], v[B + 31 - I])), ...);
}
template <int A, int B, typename T, int N>
MOE_DEV void merge_keep_top32(T (&v)[N]) {
  keep_top32_first<A, B>(v, std::make_index_sequence<32>{});
  apply_net<BitonicMergeNet<32>, A>(v, std::make_index_sequence<BitonicMergeNet<32>::kCount>{});
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

// Balanced tree sum on packed pairs ep[a] = (v[2a], v[2a+1]): level H (even)
// adds element i + H to element i, i.e. pair a + H/2 to pair a; the last level
// (H = 1) is the sum of the two halves of ep[0].
template <int H, int NP>
MOE_DEV void tree_sum_level2(uint64_t (&ep)[NP]) {
#pragma unroll
  for (int a = 0; a < H / 2; ++a) ep[a] = add2(ep[a], ep[a + H / 2]);
  if constexpr (H > 2) tree_sum_level2<H / 2>(ep);
}

// ---------------------------------------------------------------- kernel
template <int N>
struct RouteConsts {
  float x[N];   // x'_i = fl(i / (N - 1))
  float bound;  // fl(1 - x'_{kTop-1}) >= D_i for every rank i >= kTop - 1
};

// Host: the constants of an N-expert curve, computed in fp32 (RN).
template <typename RC>
inline void fill_route_consts(RC& rc, int N) {
  for (int i = 0; i < N; ++i) rc.x[i] = static_cast<float>(i) / static_cast<float>(N - 1);
  rc.bound = 1.0f - rc.x[kTop - 1];
}

// Shared memory of a 128-token block: the [kTok][N + 4] row tile, plus eight
// 8-byte key slots per token for the full-sort helpers (topk_ids).
template <int N>
constexpr size_t smem_bytes() {
  return sizeof(float) * kTok * (N + 4) + sizeof(uint64_t) * 8 * kTok;
}
// ... and of the routing kernel, which needs the row tile only.
template <int N>
constexpr size_t route_smem_bytes() {
  return sizeof(float) * kTok * (N + 4);
}

MOE_DEV void write_outputs(int64_t t, int K, int k, const int (&ids)[8], const float (&g)[8],
                           int32_t* k_out, int32_t* ids_out, float* gates_out) {
  k_out[t] = k;
  if (K == 8) {
    int4* ip = reinterpret_cast<int4*>(ids_out + t * 8);
    float4* gp = reinterpret_cast<float4*>(gates_out + t * 8);
    ip[0] = make_int4(ids[0], ids[1], ids[2], ids[3]);
    ip[1] = make_int4(ids[4], ids[5], ids[6], ids[7]);
    gp[0] = make_float4(g[0], g[1], g[2], g[3]);
    gp[1] = make_float4(g[4], g[5], g[6], g[7]);
  } else {
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if (s < K) {
        ids_out[t * K + s] = ids[s];
        gates_out[t * K + s] = g[s];
      }
    }
  }
}

// The softmax sum s of a token and what its quotients e_j / s need: y = RN(1/s)
// (for quot / quot2), and `regular`: every logit lies within 40 of the maximum,
// so that every e_j >= EXP(-40) > 2^-58, every p_j > 2^-65, and every nonzero
// difference p_(i) - p_min is at least an ulp of p_min (> 2^-88): every
// numerator the routing divides is then 0 or at least kQuotMin.
struct Softmax {
  float s, y;
  bool regular;
};

// Softmax numerators of one token: e_j = EXP(l_j - m) for the N logits in
// row, written back into the row; the smallest e_j in emin; returns the sum s
// (the balanced tree sum of the e_j) with y = RN(1/s).
template <int N>
MOE_DEV Softmax softmax_row(float* row, float& emin) {
  float m, lmin;
  {
    float l[N];
#pragma unroll
    for (int c = 0; c < N; c += 4) {
      const float4 q = *reinterpret_cast<const float4*>(row + c);
      l[c] = q.x; l[c + 1] = q.y; l[c + 2] = q.z; l[c + 3] = q.w;
    }
    // four interleaved 3-input max (and min) chains over l[4 ..), two elements per step
    float acc[4] = {l[0], l[1], l[2], l[3]};
    float acn[4] = {l[0], l[1], l[2], l[3]};
#pragma unroll
    for (int j = 4; j < N; j += 2) {
      acc[(j / 2) % 4] = max3f(acc[(j / 2) % 4], l[j], l[j + 1]);
      acn[(j / 2) % 4] = min3f(acn[(j / 2) % 4], l[j], l[j + 1]);
    }
    m = fmaxf(max3f(acc[0], acc[1], acc[2]), acc[3]);
    lmin = fminf(min3f(acn[0], acn[1], acn[2]), acn[3]);
  }
  // the specification needs finite logits
  MOE_DCHECK(isfinite(m) && isfinite(lmin));
  const uint64_t mm = pk(m, m);
  // e_j = EXP(l_j - m), eight at a time in place in the row; the loop is not
  // unrolled, so its code is fetched once instead of N / 8 times. When every
  // l_j - m >= -87 (rounded as in the loop) the clamps of EXP cannot act, and
  // the same operations run without them.
  auto exp_pass = [&](auto ex) {
#pragma unroll 1
    for (int c = 0; c < N; c += 8) {
      const float4 q0 = *reinterpret_cast<const float4*>(row + c);
      const float4 q1 = *reinterpret_cast<const float4*>(row + c + 4);
      const uint64_t e0 = ex(sub2(pk(q0.x, q0.y), mm));
      const uint64_t e1 = ex(sub2(pk(q0.z, q0.w), mm));
      const uint64_t e2 = ex(sub2(pk(q1.x, q1.y), mm));
      const uint64_t e3 = ex(sub2(pk(q1.z, q1.w), mm));
      *reinterpret_cast<float4*>(row + c) = make_float4(lo_of(e0), hi_of(e0), lo_of(e1), hi_of(e1));
      *reinterpret_cast<float4*>(row + c + 4) =
          make_float4(lo_of(e2), hi_of(e2), lo_of(e3), hi_of(e3));
    }
  };
  const float zmin = __fsub_rn(lmin, m);
  if (zmin >= -87.0f)
    exp_pass([](uint64_t z) { return exp_spec2_inrange(z); });
  else
    exp_pass([](uint64_t z) { return exp_spec2(z); });
  uint64_t ep[N / 2];
#pragma unroll
  for (int c = 0; c < N; c += 4) {
    const float4 q = *reinterpret_cast<const float4*>(row + c);
    ep[c / 2] = pk(q.x, q.y);
    ep[c / 2 + 1] = pk(q.z, q.w);
  }
  {
    // four interleaved 3-input min chains over the pairs ep[2 ..)
    float acc[4] = {lo_of(ep[0]), hi_of(ep[0]), lo_of(ep[1]), hi_of(ep[1])};
#pragma unroll
    for (int a = 2; a < N / 2; ++a) acc[a % 4] = min3f(acc[a % 4], lo_of(ep[a]), hi_of(ep[a]));
    emin = fminf(min3f(acc[0], acc[1], acc[2]), acc[3]);
  }
  tree_sum_level2<N / 2>(ep);
  Softmax sm;
  sm.s = __fadd_rn(lo_of(ep[0]), hi_of(ep[0]));
  sm.y = __frcp_rn(sm.s);
  sm.regular = zmin >= -40.0f;
  return sm;
}

// v = all N probabilities p_j = e_j / s (row holds the e_j), sorted descending.
template <int N>
MOE_DEV void sorted_probs(const float* row, const Softmax& sm, float (&v)[N]) {
#pragma unroll
  for (int c = 0; c < N; c += 4) {
    const float4 q = *reinterpret_cast<const float4*>(row + c);
    v[c] = quot(q.x, sm.s, sm.y); v[c + 1] = quot(q.y, sm.s, sm.y);
    v[c + 2] = quot(q.z, sm.s, sm.y); v[c + 3] = quot(q.w, sm.s, sm.y);
  }
  sort_desc_at<N, 0>(v);
}

// ids of the K largest probabilities in sorted order (equal probabilities by
// ascending id), from the sorted values v and a threshold scan of the row:
// p_(K-1) is the minimum of the first K sorted values; every p above it is
// taken, and the equal ones in ascending id until K are taken. The (p, id)
// keys go through this thread's 8-byte slots keys[s * kTok + tid].
template <int N>
MOE_DEV void topk_ids(const float* row, const Softmax& sm, const float (&v)[N], int K,
                      uint64_t* keys, int tid, int (&ids)[8]) {
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
    const float pq[4] = {quot(q.x, sm.s, sm.y), quot(q.y, sm.s, sm.y), quot(q.z, sm.s, sm.y),
                         quot(q.w, sm.s, sm.y)};
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
#pragma unroll
  for (int s = 0; s < 8; ++s) ids[s] = ~static_cast<int>(key[s]);
}

// Routes token t with the calling (whole, converged) warp from the token's
// softmax numerators e (lane l holds experts l + 32c in e[c]) and their sum s,
// in the routing specification's arithmetic: p_j = e_j / s; a bitonic sort of
// the N keys (p bits << 32 | ~id) across the warp, which orders by p
// descending and ascending id on ties; p'_i and D_i on every rank; the first
// argmax by a (max D, min index) warp reduction; k = min(e + 1, K). Writes the
// token's outputs; returns k, and lane s < K gets the id of rank s in sel_id.
template <int N>
MOE_DEV int warp_route_from_e(const float (&e)[N / 32], float s, int64_t t, int K, float eps,
                              int topk_mode, int renorm, int32_t* __restrict__ k_out,
                              int32_t* __restrict__ ids_out, float* __restrict__ gates_out,
                              int& sel_id) {
  constexpr int C = N / 32;
  const unsigned full = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  uint64_t key[C];
  const float ys = __frcp_rn(s);
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const float p = quot(e[c], s, ys);
    key[c] = (static_cast<uint64_t>(__float_as_uint(p)) << 32) |
             static_cast<uint32_t>(~(32 * c + lane));
  }
  // bitonic sort, descending; element j = 32 c + lane
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
  const float den = __fadd_rn(__fsub_rn(pmax, pmin), eps);
  const float yd = __frcp_rn(den);
  float best = 0.0f;
  int bi = 0;
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const int i = 32 * c + lane;
    const float p = __uint_as_float(static_cast<uint32_t>(key[c] >> 32));
    const float pn = quot(__fsub_rn(p, pmin), den, yd);
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
    for (int s2 = 0; s2 < 8; ++s2) {
      const float ps = __shfl_sync(full, p, s2);
      if (s2 < k) S = __fadd_rn(S, ps);
    }
  }
  if (lane < K) {
    ids_out[t * K + lane] = id;
    gates_out[t * K + lane] = lane < k ? (renorm ? __fdiv_rn(p, S) : p) : 0.0f;
  }
  if (lane == 0) k_out[t] = k;
  sel_id = id;
  return k;
}

// The tokens of this warp that route_token left undecided (lane l's bit in
// `undecided`; its softmax numerators in row_of(l)[0 .. N), their sum in s,
// its token index in t) are routed one after another by the whole warp;
// their lanes receive k in k_sel and the selected ids in ids_sel. Every lane
// of the warp must call this.
template <int N, typename RowOf>
MOE_DEV void route_undecided(unsigned undecided, RowOf row_of, float s, int64_t t, int K,
                             float eps, int topk_mode, int renorm, int32_t* __restrict__ k_out,
                             int32_t* __restrict__ ids_out, float* __restrict__ gates_out,
                             int& k_sel, int (&ids_sel)[8]) {
  const unsigned full = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  while (undecided) {
    const int src = __ffs(static_cast<int>(undecided)) - 1;
    undecided &= undecided - 1u;
    const float* srow = row_of(src);
    float e[N / 32];
#pragma unroll
    for (int c = 0; c < N / 32; ++c) e[c] = srow[32 * c + lane];
    const float rs = __shfl_sync(full, s, src);
    const int64_t ts = __shfl_sync(full, t, src);
    int sel = 0;
    const int kf = warp_route_from_e<N>(e, rs, ts, K, eps, topk_mode, renorm, k_out, ids_out,
                                        gates_out, sel);
#pragma unroll
    for (int s2 = 0; s2 < 8; ++s2) {
      const int id_s = __shfl_sync(full, sel, s2);
      if (lane == src) ids_sel[s2] = id_s;
    }
    if (lane == src) k_sel = kf;
  }
}

// Routes the token of this thread (its logits are in `row`): writes its
// outputs and returns k, with the selected ids in ids_sel; or, when the fast
// path cannot settle the token, returns -1 and writes nothing (the row then
// holds the softmax numerators and s_out = s, for route_undecided).
template <int N, typename RC>
MOE_DEV int route_token(float* row, int64_t t, int K, float eps, int topk_mode, int renorm,
                        const RC& rc, int32_t* __restrict__ k_out, int32_t* __restrict__ ids_out,
                        float* __restrict__ gates_out, int (&ids_sel)[8], float& s_out) {
  constexpr uint32_t kIdMask = N - 1;

  // ---- e_j = EXP(l_j - m), stored back into the row; e_min; s; RN(1/s)
  float emin;
  const Softmax sm = softmax_row<N>(row, emin);
  s_out = sm.s;

  // ---- the kTop largest e, each key = truncated value | (N-1 - id): one
  // 32-key network (a loop, not unrolled, so its code is fetched once) sorts
  // each 32-expert slice into key[32..64); the running top 32 is key[0..32)
  uint32_t key[64];
#pragma unroll 1
  for (int h = 0; h < N / 32; ++h) {
#pragma unroll
    for (int c = 0; c < 32; c += 4) {
      const int j = 32 * h + c;
      const float4 q = *reinterpret_cast<const float4*>(row + j);
      key[32 + c] = (__float_as_uint(q.x) & ~kIdMask) | (kIdMask - j);
      key[32 + c + 1] = (__float_as_uint(q.y) & ~kIdMask) | (kIdMask - (j + 1));
      key[32 + c + 2] = (__float_as_uint(q.z) & ~kIdMask) | (kIdMask - (j + 2));
      key[32 + c + 3] = (__float_as_uint(q.w) & ~kIdMask) | (kIdMask - (j + 3));
    }
    sort_desc_at<32, 32>(key);
    if (h == 0) {
#pragma unroll
      for (int i = 0; i < 32; ++i) key[i] = key[32 + i];
    } else {
      merge_keep_top32<0, 32>(key);
    }
  }

  // ---- exact values of the selected ranks, and the proof that they are the
  // exact top ranks in exact order
  float ev[kTop];
  int idv[kTop];
#pragma unroll
  for (int i = 0; i < kTop; ++i) {
    idv[i] = static_cast<int>(kIdMask - (key[i] & kIdMask));
    ev[i] = row[idv[i]];
  }
  bool ok = ((key[kTop - 2] ^ key[kTop - 1]) & ~kIdMask) != 0u;
#pragma unroll
  for (int i = 0; i + 1 < kTop - 1; ++i) ok = ok && (ev[i] >= ev[i + 1]);

  // ---- probabilities of the top ranks: correctly rounded quotients e / s
  // (rows with a logit more than 40 below their maximum are left to the warp
  // path, which checks each numerator)
  ok = ok && sm.regular;
  float pv[kTop];
  {
    const uint64_t ys = pk(sm.y, sm.y), ns = pk(-sm.s, -sm.s);
#pragma unroll
    for (int i = 0; i < kTop; i += 2) {
      const uint64_t q = quot2(pk(ev[i], ev[i + 1]), ns, ys);
      pv[i] = lo_of(q);
      pv[i + 1] = hi_of(q);
    }
  }
  // ---- elbow decision
  int k = K;
  if (ok && !topk_mode) {
    const float p_min = quot(emin, sm.s, sm.y);
    const float den = __fadd_rn(__fsub_rn(pv[0], p_min), eps);
    const float yd = __frcp_rn(den);
    const uint64_t pmin2 = pk(p_min, p_min), nden2 = pk(-den, -den), yd2 = pk(yd, yd),
                   one2 = pk(1.0f, 1.0f);
    float best = -__int_as_float(0x7f800000), mid = -__int_as_float(0x7f800000);
    int e = 0;
#pragma unroll
    for (int i = 0; i < kTop; i += 2) {
      // p'_i = (p_(i) - p_min) / den; D_i = (1 - p'_i) - x'_i
      const uint64_t pn = quot2(sub2(pk(pv[i], pv[i + 1]), pmin2), nden2, yd2);
      const uint64_t D2 = sub2(sub2(one2, pn), pk(rc.x[i], rc.x[i + 1]));
      const float D[2] = {lo_of(D2), hi_of(D2)};
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int ii = i + u;
        if (ii >= kTop - 1) continue;
        if (ii < 7 && ii < K - 1) {
          if (D[u] > best) { best = D[u]; e = ii; }
        } else {
          mid = fmaxf(mid, D[u]);
        }
      }
    }
    if (best >= mid && best >= rc.bound) k = e + 1;
    else if (mid > best) k = K;
    else ok = false;
  }

  // ---- top-K ids and gates; equal probabilities are re-ordered by id
  // (p_(K) and p_(K-1) are written as a max and a min over sorted values: a
  // select on s == K would become a dynamic index into the register array)
  bool tie_in = false;
  float pK = 0.0f;
#pragma unroll
  for (int s = 0; s < 8; ++s)
    if (s + 1 < K && pv[s] == pv[s + 1]) tie_in = true;
#pragma unroll
  for (int s = 1; s <= 8; ++s)
    if (s >= K) pK = fmaxf(pK, pv[s]);
  float pKm1 = pv[0];
#pragma unroll
  for (int s = 1; s < 8; ++s)
    if (s < K) pKm1 = fminf(pKm1, pv[s]);
  if (pKm1 == pK) ok = false;  // a tie across the K boundary

  if (!ok) return -1;

  int ids[8];
  float g[8];
#pragma unroll
  for (int s = 0; s < 8; ++s) ids[s] = idv[s];
  if (tie_in) {
    uint64_t kk[8];
#pragma unroll
    for (int s = 0; s < 8; ++s)
      kk[s] = (s < K) ? ((static_cast<uint64_t>(__float_as_uint(pv[s])) << 32) |
                         static_cast<uint32_t>(~idv[s]))
                      : 0ull;
    sort8_desc(kk);
#pragma unroll
    for (int s = 0; s < 8; ++s) ids[s] = ~static_cast<int>(kk[s]);
  }
  float S = 0.0f;
#pragma unroll
  for (int s = 0; s < 8; ++s)
    if (s < k) S = __fadd_rn(S, pv[s]);
#pragma unroll
  for (int s = 0; s < 8; ++s) {
    const float p = renorm ? __fdiv_rn(pv[s], S) : pv[s];
    g[s] = (s < k) ? p : 0.0f;
  }
  write_outputs(t, K, k, ids, g, k_out, ids_out, gates_out);
#pragma unroll
  for (int s = 0; s < 8; ++s) ids_sel[s] = ids[s];
  return k;
}

}  // namespace route
}  // namespace moe
