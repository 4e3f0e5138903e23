/*
 * Elbow-routed MoE layer: plain, slow CPU oracle.
 *
 * TEST INFRASTRUCTURE. Only the test suite, the smoke check and the CPU-baseline
 * leg of the benchmark load this file's library. The product path (the CUDA
 * library and its Python binding) never calls it, and the two share no code,
 * headers, tables or constants.
 *
 * What it computes, in the paper's order and notation:
 *   - router logits l(x) = W_r x                                 (Sec. 2)
 *   - p = softmax(l), sorted descending p_(1) >= ... >= p_(N)    (Sec. 2; Alg. 1)
 *   - Kneedle normalisation p'_i, x'_i and deviation D_i, elbow e = argmax D_i,
 *     returned count e + 1                                       (Alg. 1)
 *   - capped selection k(x) = min(e(x), K)                       (Sec. 2.1)
 *   - stable token-to-expert dispatch                            (App. A.4: the
 *     patched OLMoE block sends each token to its selected experts)
 *   - SwiGLU experts and the gate-weighted combine, in fp64       (App. A.4)
 *
 * Readings of the paper (it is silent or garbled at these points):
 *   R1  Alg. 1 prints D_i = p'_i - x'_i. With p sorted descending that is
 *       strictly decreasing, so e = 0 and k = 1 for every token, which
 *       contradicts the reported k-mean of about 7.6 (Table 2) and the sample
 *       elbows k = 2..12 (App. A.2). The elbow-angle definition of Sec. 2.3
 *       places the normalised curve at (0,0) .. (1,1), i.e. it uses 1 - p'.
 *       Reading: D_i = (1 - p'_i) - x'_i.
 *   R2  Alg. 1 returns k = e + 1 while Sec. 2.1 writes k = min(e, K); the e of
 *       Sec. 2.1 is read as Alg. 1's returned count, so k = min(argmax + 1, K).
 *   R3  Ties: the sort puts equal probabilities in ascending expert id; the
 *       argmax takes the smallest index among equal D_i.
 *   R4  eps of Alg. 1 is unstated; it is a parameter (default 1e-8).
 *   R5  Gate weights are unstated; default: the selected experts' softmax
 *       probabilities, unrenormalised (renorm = 1 divides by their sum).
 *   R6  Precision of routing: the elbow decision is an integer taken from
 *       floating point, so it is specified here in fp32, step by step, with
 *       every operation of the printed formulas (the softmax of Sec. 2 and
 *       Alg. 1's normalisation and deviation) rounded once to nearest even
 *       and no contraction:
 *         m = max_j l_j;  z_j = l_j - m;  e_j = EXP(z_j) (spec below);
 *         s = balanced tree sum (v_i += v_{i+h}, h = N/2, ..., 1);
 *         p_j = e_j / s;
 *         den = (p_max - p_min) + eps;
 *         p'_i = (p_(i) - p_min) / den;  x'_i = i / (N - 1);
 *         D_i = (1 - p'_i) - x'_i.
 *   R7  Expert MLP: SwiGLU, y_e = W_down (silu(W_gate x) * (W_up x)),
 *       silu(z) = z / (1 + exp(-z)), evaluated in fp64 on the bf16 inputs.
 *   R11 Elbow angle (Sec. 2.3): the printed points (0,0), (x'_e, p'_e), (1,1)
 *       are read on the curve y' = 1 - p' that R1's chord uses (p' itself
 *       runs from (0,1) to (1,0)); theta is evaluated in fp64 from the fp32
 *       x'_e and p'_e, and is 180 degrees when the elbow is an end point.
 *   R12 Tail randomisation (Sec. 2.2): "experts of rank >= k" are drawn
 *       without replacement from the remaining experts in ascending id order,
 *       with caller-supplied uint32 random numbers; the head variant draws
 *       from ranks >= K so that the K slots stay distinct (see
 *       oracle_route_randomized).
 *
 * EXP, the routing exponential (written for this project from Cody & Waite's
 * argument reduction, 1980, and the Taylor series of exp):
 *   if !(z >= -104) return 0;  if z > 88 return +inf
 *   t = z * LOG2E;  n = rint(t)  (ties to even)
 *   r = fma(-n, LN2_HI, z);  r = fma(-n, LN2_LO, r)
 *   q = Horner(c7..c0; r) with fma, c_j = (float)(1 / j!)
 *   if n < -126 return 0;  return q * 2^n  (2^n built from its exponent bits)
 *   LOG2E = fp32(1/ln 2); LN2_HI = ln 2 rounded to 16 significant bits (so
 *   n * LN2_HI is exact); LN2_LO = fp32(ln 2 - LN2_HI).
 *
 * Build: gcc -O2 -std=c11 -ffp-contract=off (no fast-math), OpenMP over tokens.
 */
#include <math.h>
#include <omp.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_MAX_N 1024

/* OpenMP threads the oracle's parallel loops use, and setting them (timing
 * support: the CPU baseline is reported with all cores and with one). */
int oracle_max_threads(void) { return omp_get_max_threads(); }
void oracle_set_threads(int n) {
  if (n >= 1) omp_set_num_threads(n);
}

/* ---------------------------------------------------------------- EXP spec */
static const float LOG2E = 0x1.715476p+0f;
static const float LN2_HI = 0x1.62e4p-1f;
static const float LN2_LO = 0x1.7f7d1cp-20f;

/* c_j = 1/j!, evaluated in double and rounded once to fp32 */
static const float EXP_C[8] = {
    (float)(1.0 / 1.0),   (float)(1.0 / 1.0),   (float)(1.0 / 2.0),   (float)(1.0 / 6.0),
    (float)(1.0 / 24.0),  (float)(1.0 / 120.0), (float)(1.0 / 720.0), (float)(1.0 / 5040.0)};

float oracle_exp(float z) {
  if (!(z >= -104.0f)) return 0.0f;
  if (z > 88.0f) return INFINITY;
  float t = z * LOG2E;
  float n = rintf(t);
  float r = fmaf(-n, LN2_HI, z);
  r = fmaf(-n, LN2_LO, r);
  float q = EXP_C[7];
  for (int j = 6; j >= 0; --j) q = fmaf(q, r, EXP_C[j]);
  int ni = (int)n;
  if (ni < -126) return 0.0f;
  uint32_t bits = (uint32_t)(ni + 127) << 23;
  float two_n;
  memcpy(&two_n, &bits, sizeof two_n);
  return q * two_n;
}

/* Largest error of EXP, in units in the last place of the fp32 result, over
 * every fp32 z in [lo, hi] (lo <= hi <= 0), measured against double exp().
 * Results below the smallest normal float are skipped. Test support. */
double oracle_exp_max_ulp(float lo, float hi, float* worst_z) {
  uint32_t blo, bhi;
  memcpy(&blo, &lo, 4);
  memcpy(&bhi, &hi, 4);
  /* negative floats: larger magnitude has larger bit pattern */
  uint32_t b0 = (hi == 0.0f) ? 0x80000000u : bhi, b1 = blo;
  double worst = 0.0;
  float wz = 0.0f;
#pragma omp parallel
  {
    double lw = 0.0;
    float lz = 0.0f;
#pragma omp for schedule(static)
    for (int64_t b = (int64_t)b0; b <= (int64_t)b1; ++b) {
      uint32_t u = (uint32_t)b;
      float z;
      memcpy(&z, &u, 4);
      double ref = exp((double)z);
      if (ref < 0x1p-126) continue;
      int ex;
      frexp(ref, &ex); /* ref = f * 2^ex, f in [0.5, 1) */
      double ulp = ldexp(1.0, ex - 24);
      double err = fabs((double)oracle_exp(z) - ref) / ulp;
      if (err > lw) { lw = err; lz = z; }
    }
#pragma omp critical
    {
      if (lw > worst) { worst = lw; wz = lz; }
    }
  }
  if (worst_z) *worst_z = wz;
  return worst;
}

/* ------------------------------------------------------------- routing */

/* Algorithm 1 plus capped selection for one token. Returns k. Optional
 * outputs (NULL = not written): sorted_p [N], elbow_e, elbow_pn, p_out [N]
 * (unsorted p), pn_all [N] and d_all [N] (p'_i and D_i in sorted order). */
static int route_one(const float* l, int N, int K, float eps, int mode, int renorm,
                     int32_t* ids, float* gates, float* sorted_p, int32_t* elbow_e,
                     float* elbow_pn, float* p_out, float* pn_all, float* d_all) {
  float e[ORACLE_MAX_N], p[ORACLE_MAX_N], v[ORACLE_MAX_N];
  int idx[ORACLE_MAX_N];

  /* p = softmax(l) (R6) */
  float m = l[0];
  for (int j = 1; j < N; ++j)
    if (l[j] > m) m = l[j];
  for (int j = 0; j < N; ++j) e[j] = oracle_exp(l[j] - m);
  for (int j = 0; j < N; ++j) v[j] = e[j];
  for (int h = N / 2; h >= 1; h /= 2)
    for (int i = 0; i < h; ++i) v[i] = v[i] + v[i + h];
  float s = v[0];
  for (int j = 0; j < N; ++j) p[j] = e[j] / s;
  if (p_out)
    for (int j = 0; j < N; ++j) p_out[j] = p[j];

  /* p <- sort_desc(p): stable insertion sort of expert ids (R3) */
  for (int j = 0; j < N; ++j) idx[j] = j;
  for (int i = 1; i < N; ++i) {
    int key = idx[i], j = i - 1;
    while (j >= 0 && p[idx[j]] < p[key]) {
      idx[j + 1] = idx[j];
      --j;
    }
    idx[j + 1] = key;
  }
  if (sorted_p)
    for (int i = 0; i < N; ++i) sorted_p[i] = p[idx[i]];

  /* Kneedle: p'_i, x'_i, D_i (R1, R6); e = argmax D_i (R3) */
  float p_max = p[idx[0]], p_min = p[idx[N - 1]];
  float den = (p_max - p_min) + eps;
  int e_arg = 0;
  float d_best = 0.0f, pn_best = 0.0f;
  for (int i = 0; i < N; ++i) {
    float pn = (p[idx[i]] - p_min) / den;
    float xn = (float)i / (float)(N - 1);
    float D = (1.0f - pn) - xn;
    if (pn_all) pn_all[i] = pn;
    if (d_all) d_all[i] = D;
    if (i == 0 || D > d_best) {
      d_best = D;
      e_arg = i;
      pn_best = pn;
    }
  }
  if (elbow_e) *elbow_e = e_arg;
  if (elbow_pn) *elbow_pn = pn_best;

  /* k(x) = min(e(x), K) with e(x) = argmax + 1 (R2); fixed top-K: k = K */
  int k = (mode == 1) ? K : (e_arg + 1 < K ? e_arg + 1 : K);

  /* selected experts: the first K of the sorted order; gates (R5) */
  float S = 0.0f;
  for (int s = 0; s < k; ++s) S = S + p[idx[s]];
  for (int s = 0; s < K; ++s) {
    ids[s] = idx[s];
    float g = p[idx[s]];
    if (renorm) g = g / S;
    gates[s] = (s < k) ? g : 0.0f;
  }
  return k;
}

/* Route T tokens. logits [T,N] fp32; k_out [T]; ids_out/gates_out [T,K];
 * sorted_p_out [T,N] and elbow_out [T] may be NULL. mode 0 = elbow, 1 = top-K.
 * Returns 0, or -1 on an argument outside 2 <= N <= 1024 (power of two),
 * 1 <= K <= N. */
int oracle_route(const float* logits, int64_t T, int N, int K, float eps, int mode, int renorm,
                 int32_t* k_out, int32_t* ids_out, float* gates_out, float* sorted_p_out,
                 int32_t* elbow_out) {
  if (N < 2 || N > ORACLE_MAX_N || (N & (N - 1)) != 0 || K < 1 || K > N || T < 0) return -1;
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < T; ++t) {
    k_out[t] = route_one(logits + t * N, N, K, eps, mode, renorm, ids_out + t * K,
                         gates_out + t * K, sorted_p_out ? sorted_p_out + t * N : NULL,
                         elbow_out ? elbow_out + t : NULL, NULL, NULL, NULL, NULL);
  }
  return 0;
}

/* Per token, the normalised curve of Alg. 1 in sorted order: p_(i), p'_i and
 * D_i for i = 0..N-1, each [T, N] (test support: the pins check each printed
 * operation's rounding). Returns 0, or -1 on unsupported arguments. */
int oracle_elbow_curve(const float* logits, int64_t T, int N, float eps, float* sorted_p,
                       float* pn_out, float* d_out) {
  if (N < 2 || N > ORACLE_MAX_N || (N & (N - 1)) != 0 || T < 0) return -1;
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < T; ++t) {
    int32_t id1;
    float g1;
    route_one(logits + t * N, N, 1, eps, 0, 0, &id1, &g1, sorted_p + t * N, NULL, NULL, NULL,
              pn_out + t * N, d_out + t * N);
  }
  return 0;
}

/* Elbow angle (Sec. 2.3): the angle at the elbow point between the first and
 * the last point of the normalised curve. With the deviation read as below
 * the chord (R1), the normalised curve is (x'_i, y'_i) = (i/(N-1), 1 - p'_i),
 * from (0,0) to (1,1); at the elbow e, v1 = (0,0) - (x'_e, y'_e) and
 * v2 = (1,1) - (x'_e, y'_e), theta = arccos(v1.v2 / (|v1| |v2|)) (R11).
 * x'_e and p'_e are the fp32 values of the elbow step; the angle is evaluated
 * in fp64 and returned in degrees. A zero-length v1 or v2 (the elbow on an end
 * point) gives 180 degrees (no bend). */
static const double ORACLE_PI = 3.14159265358979323846;

double oracle_angle_deg(int e, int N, float pn_e) {
  double x = (double)((float)e / (float)(N - 1));
  double y = 1.0 - (double)pn_e;
  double ax = -x, ay = -y, bx = 1.0 - x, by = 1.0 - y;
  double na = sqrt(ax * ax + ay * ay), nb = sqrt(bx * bx + by * by);
  if (na == 0.0 || nb == 0.0) return 180.0;
  double c = (ax * bx + ay * by) / (na * nb);
  if (c > 1.0) c = 1.0;
  if (c < -1.0) c = -1.0;
  return acos(c) * (180.0 / ORACLE_PI);
}

/* Per token: the uncapped elbow index e (argmax of D over all N ranks) and
 * the elbow angle in degrees (rounded to fp32). Returns 0, or -1 on
 * unsupported arguments (as oracle_route). */
int oracle_elbow_angle(const float* logits, int64_t T, int N, float eps, int32_t* elbow_out,
                       float* theta_out) {
  if (N < 2 || N > ORACLE_MAX_N || (N & (N - 1)) != 0 || T < 0) return -1;
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < T; ++t) {
    int32_t id1, e;
    float g1, pn;
    route_one(logits + t * N, N, 1, eps, 0, 0, &id1, &g1, NULL, &e, &pn, NULL, NULL, NULL);
    elbow_out[t] = e;
    theta_out[t] = (float)oracle_angle_deg(e, N, pn);
  }
  return 0;
}

/* Tail randomisation (Sec. 2.2): the experiment that keeps K experts
 * but replaces part of the elbow-K selection by random experts.
 *   mode 2 (tail): slots s < k keep ranks 0..k-1; each slot s in [k, K) gets
 *     an expert drawn without replacement from those outside ranks 0..k-1
 *     (i.e. of rank >= k);
 *   mode 3 (head): slots s in [k, K) keep ranks k..K-1; each slot s < k gets
 *     an expert drawn without replacement from those of rank >= K (outside the
 *     top-K, so that the K experts stay distinct).
 * Draw (R12): the candidates are the remaining experts in ascending id order;
 * slot s takes the one at index rand[s] mod (number remaining), which is then
 * removed. rand [T, K] uint32 is an input. k_out = K (all K slots are used);
 * gates[s] = p of the expert in slot s, or with renorm its share of the sum
 * over the K slots, left to right. */
int oracle_route_randomized(const float* logits, int64_t T, int N, int K, float eps, int mode,
                            int renorm, const uint32_t* rand, int32_t* k_out, int32_t* ids_out,
                            float* gates_out) {
  if (N < 2 || N > ORACLE_MAX_N || (N & (N - 1)) != 0 || K < 1 || K > N || T < 0) return -1;
  if (mode != 2 && mode != 3) return -1;
  if (N - K < K) return -1; /* mode 3 needs k <= N - K candidates */
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < T; ++t) {
    int32_t ids[ORACLE_MAX_N];
    float gates[ORACLE_MAX_N], p[ORACLE_MAX_N];
    int taken[ORACLE_MAX_N];
    int k = route_one(logits + t * N, N, K, eps, 0, 0, ids, gates, NULL, NULL, NULL, p, NULL,
                      NULL);
    for (int j = 0; j < N; ++j) taken[j] = 0;
    int lo = (mode == 2) ? k : 0, hi = (mode == 2) ? K : k;
    int excl = (mode == 2) ? k : K; /* ranks 0..excl-1 are not candidates */
    for (int s = 0; s < excl; ++s) taken[ids[s]] = 1;
    int remaining = N - excl;
    for (int s = lo; s < hi; ++s) {
      uint32_t idx = rand[t * K + s] % (uint32_t)remaining;
      int pick = -1;
      for (int j = 0, c = 0; j < N; ++j) {
        if (taken[j]) continue;
        if ((uint32_t)c == idx) {
          pick = j;
          break;
        }
        ++c;
      }
      taken[pick] = 1;
      ids[s] = pick;
      --remaining;
    }
    float S = 0.0f;
    for (int s = 0; s < K; ++s) S = S + p[ids[s]];
    k_out[t] = K;
    for (int s = 0; s < K; ++s) {
      ids_out[t * K + s] = ids[s];
      gates_out[t * K + s] = renorm ? p[ids[s]] / S : p[ids[s]];
    }
  }
  return 0;
}

/* ------------------------------------------------------------ dispatch */

/* Token-to-expert dispatch of the (t, s < k_t) pairs: counts per expert,
 * exclusive offsets [N+1], and a stable scatter (ascending t within an
 * expert): perm[pos] = t, pair_pos[t,s] = pos, or -1 for s >= k_t.
 * Returns 0, or -1 on an expert id outside [0,N), a k outside [0,K], or an
 * expert selected twice by one token. */
int oracle_dispatch(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                    int32_t* offsets, int32_t* perm, int32_t* pair_pos) {
  int64_t* cnt = (int64_t*)calloc((size_t)N, sizeof(int64_t));
  if (!cnt) return -1;
  for (int64_t t = 0; t < T; ++t) {
    if (k[t] < 0 || k[t] > K) { free(cnt); return -1; }
    for (int s = 0; s < k[t]; ++s) {
      int e = ids[t * K + s];
      if (e < 0 || e >= N) { free(cnt); return -1; }
      for (int s2 = 0; s2 < s; ++s2)
        if (ids[t * K + s2] == e) { free(cnt); return -1; }
      cnt[e]++;
    }
  }
  offsets[0] = 0;
  for (int e = 0; e < N; ++e) offsets[e + 1] = offsets[e] + (int32_t)cnt[e];
  for (int e = 0; e < N; ++e) cnt[e] = offsets[e];
  for (int64_t t = 0; t < T; ++t) {
    for (int s = 0; s < K; ++s) {
      if (s < k[t]) {
        int e = ids[t * K + s];
        int64_t pos = cnt[e]++;
        perm[pos] = (int32_t)t;
        pair_pos[t * K + s] = (int32_t)pos;
      } else {
        pair_pos[t * K + s] = -1;
      }
    }
  }
  free(cnt);
  return 0;
}

/* --------------------------------------------------------------- layer */

static double bf16_to_double(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

/* round to fp32 (nearest), then to bf16 (nearest even) */
static double round_bf16(double v) {
  float f = (float)v;
  uint32_t u;
  memcpy(&u, &f, 4);
  u = (u + 0x7FFFu + ((u >> 16) & 1u)) & 0xFFFF0000u;
  memcpy(&f, &u, 4);
  return (double)f;
}

/* Router logits l = W_r x for the listed rows, accumulated in fp64 and
 * rounded once to fp32. x [T,d], w_router [N,d] bf16 bits; out [nrows,N]. */
void oracle_router_logits(const uint16_t* x, const uint16_t* w_router, int64_t T, int d, int N,
                          const int64_t* rows, int64_t nrows, float* out) {
  (void)T;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < nrows; ++r) {
    const uint16_t* xr = x + rows[r] * d;
    for (int j = 0; j < N; ++j) {
      double acc = 0.0;
      for (int c = 0; c < d; ++c) acc += bf16_to_double(xr[c]) * bf16_to_double(w_router[(int64_t)j * d + c]);
      out[r * N + j] = (float)acc;
    }
  }
}

/* One MoE layer forward for the listed token rows, in fp64:
 *   l = W_r x (rounded to fp32), routing as oracle_route,
 *   y = sum_{s<k} g_s * W_down[e_s] (silu(W_gate[e_s] x) * (W_up[e_s] x)) (+ residual).
 * w_gate_up [N,2I,d]: rows [0,I) gate, rows [I,2I) up; w_down [N,d,I].
 * flags bit 0: round h to bf16 before the down projection; bit 1: round each
 * expert output to bf16 before the combine (both mirror storage precisions).
 * Outputs per listed row: y [nrows,d] fp64, logits [nrows,N], k [nrows],
 * ids/gates [nrows,K] (any of the last four may be NULL). Returns 0 or -1. */
int oracle_layer_rows(const uint16_t* x, const uint16_t* w_router, const uint16_t* w_gate_up,
                      const uint16_t* w_down, int64_t T, int d, int N, int I, int K, float eps,
                      int mode, int renorm, const uint16_t* residual, const int64_t* rows,
                      int64_t nrows, int flags, double* y, float* logits_out, int32_t* k_out,
                      int32_t* ids_out, float* gates_out) {
  if (N < 2 || N > ORACLE_MAX_N || (N & (N - 1)) != 0 || K < 1 || K > N || d < 1 || I < 1) return -1;
  for (int64_t r = 0; r < nrows; ++r)
    if (rows[r] < 0 || rows[r] >= T) return -1;
  int bad = 0;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t r = 0; r < nrows; ++r) {
    int64_t t = rows[r];
    const uint16_t* xr = x + t * d;
    double* xd = (double*)malloc(sizeof(double) * (size_t)d);
    double* h = (double*)malloc(sizeof(double) * (size_t)I);
    float l[ORACLE_MAX_N];
    int32_t ids[ORACLE_MAX_N];
    float gates[ORACLE_MAX_N];
    if (!xd || !h) {
      free(xd);
      free(h);
#pragma omp atomic write
      bad = 1;
      continue;
    }
    for (int c = 0; c < d; ++c) xd[c] = bf16_to_double(xr[c]);
    for (int j = 0; j < N; ++j) {
      double acc = 0.0;
      for (int c = 0; c < d; ++c) acc += xd[c] * bf16_to_double(w_router[(int64_t)j * d + c]);
      l[j] = (float)acc;
    }
    int k = route_one(l, N, K, eps, mode, renorm, ids, gates, NULL, NULL, NULL, NULL, NULL, NULL);
    double* yr = y + r * d;
    for (int c = 0; c < d; ++c) yr[c] = 0.0;
    for (int s = 0; s < k; ++s) {
      int64_t e = ids[s];
      const uint16_t* wg = w_gate_up + e * 2 * (int64_t)I * d;
      const uint16_t* wu = wg + (int64_t)I * d;
      const uint16_t* wdn = w_down + e * (int64_t)d * I;
      for (int i = 0; i < I; ++i) {
        double g = 0.0, u = 0.0;
        for (int c = 0; c < d; ++c) {
          g += bf16_to_double(wg[(int64_t)i * d + c]) * xd[c];
          u += bf16_to_double(wu[(int64_t)i * d + c]) * xd[c];
        }
        double hv = g / (1.0 + exp(-g)) * u;
        h[i] = (flags & 1) ? round_bf16(hv) : hv;
      }
      for (int c = 0; c < d; ++c) {
        double o = 0.0;
        for (int i = 0; i < I; ++i) o += bf16_to_double(wdn[(int64_t)c * I + i]) * h[i];
        if (flags & 2) o = round_bf16(o);
        yr[c] += (double)gates[s] * o;
      }
    }
    if (residual)
      for (int c = 0; c < d; ++c) yr[c] += bf16_to_double(residual[t * d + c]);
    if (logits_out)
      for (int j = 0; j < N; ++j) logits_out[r * N + j] = l[j];
    if (k_out) k_out[r] = k;
    if (ids_out)
      for (int s = 0; s < K; ++s) ids_out[r * K + s] = ids[s];
    if (gates_out)
      for (int s = 0; s < K; ++s) gates_out[r * K + s] = gates[s];
    free(xd);
    free(h);
  }
  return bad ? -1 : 0;
}
