// Routing diagnostics (Sec. 2.3 elbow angle; Sec. 2.4 and App. A.3 load
// metrics): one thread per token evaluates the whole sorted curve exactly (the
// same fp32 steps as the routing), finds the uncapped elbow index e (first
// argmax of D over all N ranks) and the elbow angle, and counts into integer
// histograms: k = min(e + 1, K), e, floor(theta), and the per-expert loads of
// the elbow-K and the top-K selections. A one-thread finalize step turns the
// counts into the normalised utilisations and the quantities that Theorem 1
// and Corollaries 1-2 bound. Integer counts make every result independent of
// the order in which blocks finish.
#include "route_impl.cuh"

namespace moe {
namespace diag {

using route::kTok;
using route::RouteConsts;

constexpr int kThetaBins = 181;

// theta in degrees, fp64, for the elbow point (x'_e, y'_e = 1 - p'_e) of the
// normalised curve from (0,0) to (1,1): the angle between v1 = (0,0) - P and
// v2 = (1,1) - P; 180 degrees when P is an end point.
MOE_DEV float angle_deg(float xe, float pn) {
  const double x = static_cast<double>(xe), y = 1.0 - static_cast<double>(pn);
  const double ax = -x, ay = -y, bx = 1.0 - x, by = 1.0 - y;
  const double na = sqrt(ax * ax + ay * ay), nb = sqrt(bx * bx + by * by);
  if (na == 0.0 || nb == 0.0) return 180.0f;
  double c = (ax * bx + ay * by) / (na * nb);
  c = fmin(1.0, fmax(-1.0, c));
  constexpr double kDegPerRad = 180.0 / 3.14159265358979323846;
  return static_cast<float>(acos(c) * kDegPerRad);
}

template <int N>
__global__ void __launch_bounds__(kTok) diag_kernel(
    const float* __restrict__ logits, int64_t T, int K, float eps,
    const __grid_constant__ RouteConsts<N> rc, int32_t* __restrict__ elbow_out,
    float* __restrict__ theta_out, moe_route_diag* __restrict__ dg) {
  constexpr int kPitch = N + 4;
  extern __shared__ float4 smem4[];
  __shared__ int h_k[9], h_e[N], h_th[kThetaBins], h_top[N], h_elb[N], h_sharp;
  float* tile = reinterpret_cast<float*>(smem4);
  uint64_t* keys = reinterpret_cast<uint64_t*>(tile + kTok * kPitch);
  const int tid = threadIdx.x;
  const int64_t t0 = static_cast<int64_t>(blockIdx.x) * kTok;
  const int ntok = static_cast<int>(min_of<int64_t>(kTok, T - t0));
  for (int i = tid; i < 9; i += kTok) h_k[i] = 0;
  for (int i = tid; i < N; i += kTok) h_e[i] = h_top[i] = h_elb[i] = 0;
  for (int i = tid; i < kThetaBins; i += kTok) h_th[i] = 0;
  if (tid == 0) h_sharp = 0;
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
  if (tid < ntok) {
    float* row = tile + tid * kPitch;
    float emin;
    const route::Softmax sm = route::softmax_row<N>(row, emin);
    float v[N];
    route::sorted_probs<N>(row, sm, v);
    const float p_min = v[N - 1];
    const float den = __fadd_rn(__fsub_rn(v[0], p_min), eps);
    const float yd = __frcp_rn(den);
    float best = 0.0f, pn_e = 0.0f;
    int e = 0;
#pragma unroll
    for (int i = 0; i < N; ++i) {
      const float pn = route::quot(__fsub_rn(v[i], p_min), den, yd);
      const float D = __fsub_rn(__fsub_rn(1.0f, pn), rc.x[i]);
      if (i == 0 || D > best) {
        best = D;
        e = i;
        pn_e = pn;
      }
    }
    // x'_e = fl(e / (N - 1)), the same value as rc.x[e]
    const float th = angle_deg(__fdiv_rn(static_cast<float>(e), static_cast<float>(N - 1)), pn_e);
    const int64_t t = t0 + tid;
    if (elbow_out) elbow_out[t] = e;
    if (theta_out) theta_out[t] = th;
    const int k = min(e + 1, K);
    int ids[8];
    route::topk_ids<N>(row, sm, v, K, keys, tid, ids);
    atomicAdd(&h_k[k], 1);
    atomicAdd(&h_e[e], 1);
    atomicAdd(&h_th[min(kThetaBins - 1, max(0, static_cast<int>(floorf(th))))], 1);
    if (th <= 135.0f) atomicAdd(&h_sharp, 1);
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if (s < K) {
        atomicAdd(&h_top[ids[s]], 1);
        if (s < k) atomicAdd(&h_elb[ids[s]], 1);
      }
    }
  }
  __syncthreads();
  using ull = unsigned long long;
  auto add = [](int64_t* dst, int v) {
    if (v) atomicAdd(reinterpret_cast<ull*>(dst), static_cast<ull>(v));
  };
  for (int i = tid; i < 9; i += kTok) add(&dg->k_hist[i], h_k[i]);
  for (int i = tid; i < N; i += kTok) {
    add(&dg->elbow_hist[i], h_e[i]);
    add(&dg->load_top[i], h_top[i]);
    add(&dg->load_elb[i], h_elb[i]);
  }
  for (int i = tid; i < kThetaBins; i += kTok) add(&dg->theta_hist[i], h_th[i]);
  if (tid == 0) add(&dg->sharp_elbows, h_sharp);
}

// Counts -> utilisations and bounds (fp64, one thread, fixed summation order).
__global__ void diag_finalize(moe_route_diag* dg, int64_t T, int N, int K) {
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  dg->tokens = T;
  if (T == 0) return;
  double sum_k = 0.0, st = 0.0, se = 0.0;
  for (int k = 0; k <= 8; ++k) sum_k += static_cast<double>(k) * static_cast<double>(dg->k_hist[k]);
  for (int i = 0; i < N; ++i) {
    st += static_cast<double>(dg->load_top[i]);
    se += static_cast<double>(dg->load_elb[i]);
  }
  const double mean_k = sum_k / static_cast<double>(T);
  const double delta = 1.0 - mean_k / static_cast<double>(K);
  double l1 = 0.0, mt = 0.0, me = 0.0, q2t = 0.0, q2e = 0.0;
  for (int i = 0; i < N; ++i) {
    const double qt = static_cast<double>(dg->load_top[i]) / st;
    const double qe = static_cast<double>(dg->load_elb[i]) / se;
    l1 += fabs(qe - qt);
    mt = fmax(mt, qt);
    me = fmax(me, qe);
    q2t += qt * qt;
    q2e += qe * qe;
  }
  const double cv2t = N * q2t - 1.0, cv2e = N * q2e - 1.0;
  const double cvt = sqrt(fmax(cv2t, 0.0)), cve = sqrt(fmax(cv2e, 0.0));
  dg->mean_k = mean_k;
  dg->delta = delta;
  dg->l1 = l1;
  dg->l1_bound = 2.0 * delta / (1.0 - delta);
  dg->top1_change = fabs(me - mt);
  dg->cv2_change = fabs(cv2e - cv2t);
  dg->cv2_bound = 2.0 * N * delta / ((1.0 - delta) * (1.0 - delta));
  dg->top1_share_change_pct = (mt - me) / mt * 100.0;
  dg->cv_change_pct = cvt > 0.0 ? (cvt - cve) / cvt * 100.0 : 0.0;
}

template <int N>
cudaError_t launch(const float* logits, int64_t T, int K, float eps, int32_t* elbow_out,
                   float* theta_out, moe_route_diag* dg, cudaStream_t stream) {
  cudaError_t err = cudaMemsetAsync(dg, 0, sizeof(moe_route_diag), stream);
  if (err != cudaSuccess) return err;
  if (T > 0) {
    RouteConsts<N> rc;
    route::fill_route_consts(rc, N);
    constexpr size_t smem = route::smem_bytes<N>();
    static std::atomic<uint64_t> attr_done{0};
    err = once_per_device(attr_done, [&] {
      return cudaFuncSetAttribute(diag_kernel<N>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(smem));
    });
    if (err != cudaSuccess) return err;
    const int64_t blocks = (T + kTok - 1) / kTok;
    diag_kernel<N><<<static_cast<unsigned>(blocks), kTok, smem, stream>>>(
        logits, T, K, eps, rc, elbow_out, theta_out, dg);
    err = cudaGetLastError();
    if (err != cudaSuccess) return err;
  }
  diag_finalize<<<1, 32, 0, stream>>>(dg, T, N, K);
  return cudaGetLastError();
}

}  // namespace diag

cudaError_t launch_route_diagnostics(const float* logits, int64_t T, int N, int K, float eps,
                                     int32_t* elbow_out, float* theta_out, moe_route_diag* dg,
                                     cudaStream_t stream) {
  if (N == 64) return diag::launch<64>(logits, T, K, eps, elbow_out, theta_out, dg, stream);
  return diag::launch<128>(logits, T, K, eps, elbow_out, theta_out, dg, stream);
}

MOE_DEBUG_TU(diag)

}  // namespace moe
