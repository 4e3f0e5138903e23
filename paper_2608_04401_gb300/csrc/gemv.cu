// Expert contractions for the smallest batches (T <= 4 tokens; the expert MLP
// of App. A.4 in the one-token latency regime of Sec. 3), on CUDA cores.
//
// With at most four rows per expert an expert's contraction is a few
// matrix-vector products: the work is streaming the touched experts' weights
// from HBM, and what limits a tensor-core tile here is its fixed latency
// (pipeline set-up, TMEM, first bytes, epilogue) on the few SMs that hold
// tiles. These kernels spread each touched expert's weight rows over many
// blocks instead, read the token rows straight from x through the dispatch
// permutation (no gathered copy), and accumulate in fp32:
//
//   gemv_gate_up : h[p, i] = silu(sum_c Wg[e,i,c] x[t_p,c]) * (sum_c Wu[e,i,c] x[t_p,c])
//   gemv_down    : o[p, c] = sum_i Wd[e,c,i] h[p,i]
//
// for the rows p in [offsets[e], offsets[e+1]) of expert e, t_p = perm[p].
// Grid: (row blocks of the weight matrix, experts with rows); blockIdx.y = j
// selects the j-th expert with rows (found from the offsets in the prologue),
// so blocks of untouched experts do not exist beyond min(N, T K) columns of
// the grid and return at once. A block's weight rows (gate/up: the gate and
// the up rows of 8 output indices; down: 16 rows of W_down) are contiguous in
// memory, so one thread brings them into shared memory with one bulk copy per
// row (cp.async.bulk, completing on one mbarrier, whose wait is bounded) while
// the block stages the fp32 token rows; then each warp computes its outputs
// from shared memory (lane l takes the 16-byte chunks l, l + 32, ... of a row)
// and the lanes' partial sums meet in a butterfly reduction.
//
// gemv_expert_few_kernel does the same items, both contractions and the
// weighted combine, in one cooperative launch for the layer's steps of at
// most two tokens (see its comment).
#include "common.cuh"

#include <algorithm>

namespace moe {
namespace gemv {

constexpr int kMaxRows = 4;       // rows (tokens) per expert at most: T <= 4
constexpr int kMaxDim = 4096;     // d and I at most
constexpr int kThreads = 256;     // 8 warps
constexpr int kWarps = kThreads / 32;
constexpr int kGateUpOut = 8;     // gate/up: output indices per block (one per warp)
constexpr int kDownOut = 16;      // down: output columns per block (two per warp)

// The j-th expert (ascending id) whose row range is nonempty, or -1; all
// threads of the block get it. s_exp is one int of shared memory.
MOE_DEV int jth_expert(const int32_t* __restrict__ offsets, int N, int j, int* s_exp) {
  if (threadIdx.x < 32) {
    int base = 0, found = -1;
    for (int e0 = 0; e0 < N; e0 += 32) {
      const int e = e0 + threadIdx.x;
      const bool used = e < N && offsets[e + 1] > offsets[e];
      const unsigned m = __ballot_sync(0xffffffffu, used);
      const int n = __popc(m);
      if (found < 0 && j < base + n) {
        // the (j - base)-th set bit of m
        unsigned mm = m;
        for (int q = 0; q < j - base; ++q) mm &= mm - 1u;
        found = e0 + __ffs(static_cast<int>(mm)) - 1;
      }
      base += n;
    }
    if (threadIdx.x == 0) *s_exp = found;
  }
  __syncthreads();
  return *s_exp;
}

// 8 bf16 of a 16-byte chunk -> fp32
MOE_DEV void bf16x8_to_f32(const uint4& v, float (&f)[8]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    f[2 * q] = __uint_as_float(w[q] << 16);
    f[2 * q + 1] = __uint_as_float(w[q] & 0xFFFF0000u);
  }
}

MOE_DEV float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Bulk copy of `bytes` (a multiple of 16; both addresses 16-byte aligned) from
// global to this CTA's shared memory, completing on mbarrier `bar`.
MOE_DEV void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// Every thread waits (bounded) for the block's bulk copies; on a timeout the
// error word is set, and the copies still in flight are waited for again
// (bounded) so that none lands after the block has exited. Returns whether
// the data arrived.
MOE_DEV bool wait_rows(uint32_t bar, volatile int* abort_flag, int32_t* err, uint32_t parity = 0u) {
  const bool ok = mbar_wait_bounded(bar, parity, abort_flag);
  if (!ok) {
    if (threadIdx.x == 0 && err) atomicExch(err, kDevErrTimeout);
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait(bar, parity) && global_timer_ns() - t0 < 100000000ull) {
    }
  }
  return ok;
}

// h [P, I]: gate/up + SwiGLU. Dynamic shared memory: the 2 x kGateUpOut weight
// rows (d bf16 each), then the expert's token rows (T x d fp32).
__global__ void __launch_bounds__(kThreads) gemv_gate_up_kernel(
    const uint16_t* __restrict__ x, int64_t T, const int32_t* __restrict__ perm,
    const int32_t* __restrict__ offsets, const uint16_t* __restrict__ wgu, int64_t P, int d, int N,
    int I, uint16_t* __restrict__ h, int32_t* err) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ int s_exp;
  __shared__ alignas(8) uint64_t bar;
  __shared__ int abort_flag;
  const uint32_t bar_a = smem_u32(&bar);
  if (threadIdx.x == 0) {
    mbar_init(bar_a, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  grid_dep_wait();
  grid_dep_launch();
  const int e = jth_expert(offsets, N, blockIdx.y, &s_exp);  // (its barrier also orders the init)
  if (e < 0) return;
  const int i0 = blockIdx.x * kGateUpOut;
  const int nout = min(kGateUpOut, I - i0);
  if (nout <= 0) return;
  const uint32_t row_bytes = static_cast<uint32_t>(d) * 2;
  uint16_t* wrows = reinterpret_cast<uint16_t*>(smem);  // [2 * kGateUpOut][d]
  float* xs = reinterpret_cast<float*>(smem + 2 * kGateUpOut * row_bytes);
  if (threadIdx.x == 0) {
    // gate rows i0 .. i0 + nout - 1 into slots 0 .., up rows into slots kGateUpOut ..
    mbar_arrive_expect_tx(bar_a, 2 * nout * row_bytes);
    const uint16_t* wg = wgu + static_cast<int64_t>(e) * 2 * I * d;
    for (int u = 0; u < nout; ++u) {
      bulk_load(smem_u32(wrows) + u * row_bytes, wg + static_cast<int64_t>(i0 + u) * d, row_bytes,
                bar_a);
      bulk_load(smem_u32(wrows) + (kGateUpOut + u) * row_bytes,
                wg + static_cast<int64_t>(I + i0 + u) * d, row_bytes, bar_a);
    }
  }
  const int p0 = offsets[e];
  int rows = min(offsets[e + 1] - p0, kMaxRows);
  MOE_DCHECK(offsets[e + 1] - p0 <= kMaxRows && p0 >= 0 && p0 + rows <= P);
  // rows stay within P and within the T rows the shared staging holds
  rows = (p0 < 0 || p0 >= P) ? 0
                             : static_cast<int>(min_of<int64_t>(min_of<int64_t>(rows, P - p0), T));
  // the expert's token rows, fp32, in shared memory (while the weights stream in)
  const int d8 = d / 8;
  for (int idx = threadIdx.x; idx < rows * d8; idx += kThreads) {
    const int r = idx / d8, c = idx % d8;
    int tok = perm[p0 + r];
    MOE_DCHECK(tok >= 0 && tok < T);
    tok = min(max(tok, 0), static_cast<int>(T - 1));
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(x + static_cast<int64_t>(tok) * d) + c);
    float f[8];
    bf16x8_to_f32(v, f);
    float4* dst = reinterpret_cast<float4*>(xs + r * d + c * 8);
    dst[0] = make_float4(f[0], f[1], f[2], f[3]);
    dst[1] = make_float4(f[4], f[5], f[6], f[7]);
  }
  __syncthreads();
  if (!wait_rows(bar_a, &abort_flag, err)) return;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  if (warp >= nout || rows == 0) return;
  const uint4* grow = reinterpret_cast<const uint4*>(wrows + warp * d);
  const uint4* urow = reinterpret_cast<const uint4*>(wrows + (kGateUpOut + warp) * d);
  float g[kMaxRows] = {}, v[kMaxRows] = {};
  for (int c = lane; c < d8; c += 32) {
    float fg[8], fu[8];
    bf16x8_to_f32(grow[c], fg);
    bf16x8_to_f32(urow[c], fu);
#pragma unroll
    for (int r = 0; r < kMaxRows; ++r) {
      if (r < rows) {
        const float4 x0 = reinterpret_cast<const float4*>(xs + r * d + c * 8)[0];
        const float4 x1 = reinterpret_cast<const float4*>(xs + r * d + c * 8)[1];
        const float xv[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          g[r] = fmaf(fg[q], xv[q], g[r]);
          v[r] = fmaf(fu[q], xv[q], v[r]);
        }
      }
    }
  }
#pragma unroll
  for (int r = 0; r < kMaxRows; ++r) {
    if (r < rows) {
      const float gs = warp_sum(g[r]), us = warp_sum(v[r]);
      if (lane == 0)
        h[static_cast<int64_t>(p0 + r) * I + i0 + warp] =
            __bfloat16_as_ushort(__float2bfloat16_rn(silu(gs) * us));
    }
  }
}

// The weighted combine of a batch of T <= 4 tokens, done by the down
// projection itself (tickets == nullptr: not done):
// y[t, c] = sum_{s<k_t} g_{t,s} o[pair_pos[t,s], c] (+ residual[t, c]),
// accumulated in fp32 in s order, one bf16 rounding at the end.
struct Combine {
  const int32_t* k;          // [T]
  const int32_t* pair_pos;   // [T, K]
  const float* gates;        // [T, K]
  const uint16_t* residual;  // [T, d] or nullptr
  uint16_t* y;               // [T, d]
  unsigned int* tickets;     // one per column block, zero on entry, left zero
  int K;
  int T;
};

// The combine of one column block [c0, c0 + nout) by the last of the `count`
// blocks that wrote its slices of o (see Combine); called by all threads of
// each such block after its stores of o. T * nout <= kThreads.
MOE_DEV void combine_tail(const Combine& cmb, const uint16_t* o, int64_t P, int d, int c0, int nout,
                          int cb, int count, bool* last) {
  // the block's stores of o happen before thread 0's release (the barrier);
  // the acquire half makes every earlier block's stores visible to the last
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned int prev;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;"
                 : "=r"(prev) : "l"(cmb.tickets + cb) : "memory");
    *last = static_cast<int>(prev) == count - 1;
  }
  __syncthreads();
  if (!*last) return;
  if (threadIdx.x < cmb.T * nout) {
    const int t = threadIdx.x / nout, c = c0 + threadIdx.x % nout;
    const int kt = min(max(cmb.k[t], 0), cmb.K);
    MOE_DCHECK(cmb.k[t] >= 0 && cmb.k[t] <= cmb.K);
    float acc = 0.0f;
    for (int s2 = 0; s2 < kt; ++s2) {
      const int pos = cmb.pair_pos[t * cmb.K + s2];
      MOE_DCHECK(pos >= 0 && pos < P);
      const int pc = static_cast<int>(min_of<int64_t>(max(pos, 0), P - 1));
      const uint16_t ov = __ldcg(o + static_cast<int64_t>(pc) * d + c);
      acc = fmaf(cmb.gates[t * cmb.K + s2], __uint_as_float(static_cast<uint32_t>(ov) << 16), acc);
    }
    const int64_t yi = static_cast<int64_t>(t) * d + c;
    if (cmb.residual) acc += __uint_as_float(static_cast<uint32_t>(cmb.residual[yi]) << 16);
    cmb.y[yi] = __bfloat16_as_ushort(__float2bfloat16_rn(acc));
  }
  if (threadIdx.x == 0) cmb.tickets[cb] = 0u;
}

// o [P, d]: down projection. Dynamic shared memory: kDownOut rows of W_down
// (I bf16 each), then the expert's rows of h (T x I fp32).
__global__ void __launch_bounds__(kThreads) gemv_down_kernel(
    const uint16_t* __restrict__ h, const int32_t* __restrict__ offsets,
    const uint16_t* __restrict__ wd, int64_t T, int64_t P, int d, int N, int I,
    uint16_t* __restrict__ o, int32_t* err) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ int s_exp;
  __shared__ alignas(8) uint64_t bar;
  __shared__ int abort_flag;
  const uint32_t bar_a = smem_u32(&bar);
  if (threadIdx.x == 0) {
    mbar_init(bar_a, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  grid_dep_wait();
  grid_dep_launch();
  const int e = jth_expert(offsets, N, blockIdx.y, &s_exp);
  if (e < 0) return;
  const int c0 = blockIdx.x * kDownOut;
  const int nout = min(kDownOut, d - c0);
  if (nout <= 0) return;
  const uint32_t row_bytes = static_cast<uint32_t>(I) * 2;
  uint16_t* wrows = reinterpret_cast<uint16_t*>(smem);  // [kDownOut][I]
  float* hs = reinterpret_cast<float*>(smem + kDownOut * row_bytes);
  if (threadIdx.x == 0) {
    // rows c0 .. c0 + nout - 1 of W_down[e] are contiguous: one copy
    mbar_arrive_expect_tx(bar_a, nout * row_bytes);
    bulk_load(smem_u32(wrows), wd + (static_cast<int64_t>(e) * d + c0) * I, nout * row_bytes, bar_a);
  }
  const int p0 = offsets[e];
  int rows = min(offsets[e + 1] - p0, kMaxRows);
  MOE_DCHECK(offsets[e + 1] - p0 <= kMaxRows && p0 >= 0 && p0 + rows <= P);
  rows = (p0 < 0 || p0 >= P) ? 0
                             : static_cast<int>(min_of<int64_t>(min_of<int64_t>(rows, P - p0), T));
  const int i8 = I / 8;
  for (int idx = threadIdx.x; idx < rows * i8; idx += kThreads) {
    const int r = idx / i8, c = idx % i8;
    const uint4 v = reinterpret_cast<const uint4*>(h + static_cast<int64_t>(p0 + r) * I)[c];
    float f[8];
    bf16x8_to_f32(v, f);
    float4* dst = reinterpret_cast<float4*>(hs + r * I + c * 8);
    dst[0] = make_float4(f[0], f[1], f[2], f[3]);
    dst[1] = make_float4(f[4], f[5], f[6], f[7]);
  }
  __syncthreads();
  // one decision for the whole block (a thread may see the copy land just
  // after another gave up)
  if (__syncthreads_or(!wait_rows(bar_a, &abort_flag, err) ? 1 : 0)) return;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  for (int u = warp; rows > 0 && u < nout; u += kWarps) {
    const uint4* row = reinterpret_cast<const uint4*>(wrows + u * I);
    float acc[kMaxRows] = {};
    for (int q8 = lane; q8 < i8; q8 += 32) {
      float fw[8];
      bf16x8_to_f32(row[q8], fw);
#pragma unroll
      for (int r = 0; r < kMaxRows; ++r) {
        if (r < rows) {
          const float4 h0 = reinterpret_cast<const float4*>(hs + r * I + q8 * 8)[0];
          const float4 h1 = reinterpret_cast<const float4*>(hs + r * I + q8 * 8)[1];
          const float hv[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
#pragma unroll
          for (int q = 0; q < 8; ++q) acc[r] = fmaf(fw[q], hv[q], acc[r]);
        }
      }
    }
#pragma unroll
    for (int r = 0; r < kMaxRows; ++r) {
      if (r < rows) {
        const float sum = warp_sum(acc[r]);
        if (lane == 0)
          o[static_cast<int64_t>(p0 + r) * d + c0 + u] = __bfloat16_as_ushort(__float2bfloat16_rn(sum));
      }
    }
  }
}

// ------------------------------------------- few-token expert MLP, fused
// The gate/up and down contractions of a step of T <= 4 tokens (and its
// combine) in one cooperative launch, so that no kernel boundary separates
// them and the first down weights stream in while the last gate/up rows are
// computed. The work items are those of the two kernels above: gate/up items
// (j, output block of 8) and down items (j, block of dn_rows columns) over the
// j < n experts with rows (ascending id), each item covering all of expert j's
// rows (at most T). Block b takes the gate/up items b, b + G, ... and then the
// down items G - 1 - b, 2G - 1 - b, ... (G blocks, all resident: the launch is
// cooperative), so that the blocks with fewer gate/up items take the second
// round of down items. After a gate/up item's h stores, thread 0 adds one to
// done[j] (release); a down item starts its weight copy, then thread 0 waits
// (acquire, bounded) until done[j] counts all of expert j's gate/up items
// before the block reads h. Every block finishes its gate/up items before it
// waits, and all blocks are resident, so every wait ends; a wait that runs
// out sets the error word and the block leaves once its copy has landed. The
// last block of each column block combines (combine_tail).
constexpr int kFewMaxT = 4;
constexpr int kFewMaxExperts = 32;  // experts with rows: at most T K

MOE_DEV bool wait_count(const unsigned int* ctr, unsigned int target, volatile int* abort) {
  const uint64_t t0 = global_timer_ns();
  for (uint32_t spins = 1;; ++spins) {
    unsigned int v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
    if (v >= target) return true;
    if (spins % 64u == 0u) {
      if (*abort) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        *abort = 1;
        return false;
      }
    }
    __nanosleep(32);
  }
}

// Dynamic shared memory: wbytes of weight rows (the gate/up item's 2 x 8 rows
// of d, or the down item's dn_rows rows of I, bf16), then the T token rows of
// x (bf16, d each) in the gate/up items, and the expert's rows of h (bf16, I
// each) in the down items. A down item takes 16 rows, or more when the
// experts' down items outnumber the blocks, up to dn_max rows: as many as the
// gate/up item's space holds (a multiple of 8, 16 to 64).
// MT: rows per expert at most (1, 2 or 4; T <= MT); with MT = 1 every row
// holds token 0.
template <int MT>
__global__ void __launch_bounds__(kThreads) gemv_expert_few_kernel(
    const uint16_t* __restrict__ x, int T, const int32_t* __restrict__ perm,
    const int32_t* __restrict__ offsets, const uint16_t* __restrict__ wgu,
    const uint16_t* __restrict__ wd, int64_t P, int d, int N, int I, uint32_t wbytes, int dn_max,
    uint16_t* h, uint16_t* o, int32_t* err, unsigned int* done, Combine cmb) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ int s_used[kFewMaxExperts];
  __shared__ int s_n, s_ok;
  __shared__ int s_tok[MT];
  __shared__ alignas(8) uint64_t bar;
  __shared__ int abort_flag;
  __shared__ bool last;
  const uint32_t bar_a = smem_u32(&bar);
  if (threadIdx.x == 0) {
    mbar_init(bar_a, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  grid_dep_wait();
  grid_dep_launch();
  if (threadIdx.x < 32) {  // the experts with rows, ascending id
    const int lane = threadIdx.x;
    int base = 0;
    for (int e0 = 0; e0 < N; e0 += 32) {
      const int e = e0 + lane;
      const bool used = e < N && offsets[e + 1] > offsets[e];
      const unsigned m = __ballot_sync(0xffffffffu, used);
      const int idx = base + __popc(m & ((1u << lane) - 1u));
      if (used && idx < kFewMaxExperts) s_used[idx] = e;
      base += __popc(m);
    }
    MOE_DCHECK(base <= kFewMaxExperts);
    if (lane == 0) s_n = min(base, kFewMaxExperts);
  }
  uint16_t* wrows = reinterpret_cast<uint16_t*>(smem);
  uint16_t* vec = reinterpret_cast<uint16_t*>(smem + wbytes);  // x rows, then h rows (bf16)
  const int d8 = d / 8, i8 = I / 8;
  for (int c = threadIdx.x; c < T * d8; c += kThreads)  // the T token rows
    reinterpret_cast<uint4*>(vec)[c] = __ldg(reinterpret_cast<const uint4*>(x) + c);
  __syncthreads();  // s_used, s_n, x, barrier init
  const int n = s_n;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int ngu = (I + kGateUpOut - 1) / kGateUpOut;
  // down items: the fewest rows (16, 24, ... up to dn_max) that give each
  // block at most one item, so that few experts still spread over all blocks
  int dn_rows = 16;
  while (dn_rows < dn_max && n * ((d + dn_rows - 1) / dn_rows) > static_cast<int>(gridDim.x))
    dn_rows += 8;
  const int ndn = (d + dn_rows - 1) / dn_rows;
  uint32_t parity = 0;
  // expert e's rows: [p0, p0 + rows), rows <= T
  auto rows_of = [&](int e, int& p0) {
    p0 = offsets[e];
    const int r = offsets[e + 1] - p0;
    MOE_DCHECK(r >= 1 && r <= T && p0 >= 0 && p0 + r <= P);
    if (p0 < 0 || p0 >= P) return 0;
    return static_cast<int>(min_of<int64_t>(min(max(r, 0), min(T, MT)), P - p0));
  };

  for (int it = blockIdx.x; it < n * ngu; it += gridDim.x) {
    const int j = it / ngu, i0 = (it % ngu) * kGateUpOut;
    const int e = s_used[j];
    const int nout = min(kGateUpOut, I - i0);
    const uint32_t row_bytes = static_cast<uint32_t>(d) * 2;
    int p0;
    const int rows = rows_of(e, p0);
    if (threadIdx.x == 0) {
      mbar_arrive_expect_tx(bar_a, 2 * nout * row_bytes);
      const uint16_t* wg = wgu + static_cast<int64_t>(e) * 2 * I * d;
      for (int u = 0; u < nout; ++u) {
        bulk_load(smem_u32(wrows) + u * row_bytes, wg + static_cast<int64_t>(i0 + u) * d, row_bytes,
                  bar_a);
        bulk_load(smem_u32(wrows) + (kGateUpOut + u) * row_bytes,
                  wg + static_cast<int64_t>(I + i0 + u) * d, row_bytes, bar_a);
      }
    }
    if (MT > 1 && threadIdx.x < rows) {
      const int tok = perm[p0 + threadIdx.x];
      MOE_DCHECK(tok >= 0 && tok < T);
      s_tok[threadIdx.x] = min(max(tok, 0), T - 1);
    }
    const bool ok = !__syncthreads_or(!wait_rows(bar_a, &abort_flag, err, parity) ? 1 : 0);
    parity ^= 1u;
    if (!ok) return;
    if (warp < nout) {
      const uint4* grow = reinterpret_cast<const uint4*>(wrows + warp * d);
      const uint4* urow = reinterpret_cast<const uint4*>(wrows + (kGateUpOut + warp) * d);
      const uint4* xr[MT];
#pragma unroll
      for (int r = 0; r < MT; ++r)
        xr[r] = reinterpret_cast<const uint4*>(vec) + (MT > 1 && r < rows ? s_tok[r] : 0) * d8;
      float g[MT] = {}, v[MT] = {};
      for (int c = lane; c < d8; c += 32) {
        float fg[8], fu[8];
        bf16x8_to_f32(grow[c], fg);
        bf16x8_to_f32(urow[c], fu);
#pragma unroll
        for (int r = 0; r < MT; ++r) {
          if (r < rows) {
            float xv[8];
            bf16x8_to_f32(xr[r][c], xv);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              g[r] = fmaf(fg[q], xv[q], g[r]);
              v[r] = fmaf(fu[q], xv[q], v[r]);
            }
          }
        }
      }
#pragma unroll
      for (int r = 0; r < MT; ++r) {
        if (r < rows) {
          const float gs = warp_sum(g[r]), us = warp_sum(v[r]);
          if (lane == 0)
            h[static_cast<int64_t>(p0 + r) * I + i0 + warp] =
                __bfloat16_as_ushort(__float2bfloat16_rn(silu(gs) * us));
        }
      }
    }
    // the item's h stores happen before the release; the weight rows are free
    __syncthreads();
    if (threadIdx.x == 0)
      asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(done + j) : "memory");
  }

  for (int it = gridDim.x - 1 - blockIdx.x; it < n * ndn; it += gridDim.x) {
    const int j = it / ndn, cb = it % ndn, c0 = cb * dn_rows;
    const int e = s_used[j];
    const int nout = min(dn_rows, d - c0);
    const uint32_t row_bytes = static_cast<uint32_t>(I) * 2;
    if (threadIdx.x == 0) {
      // rows c0 .. c0 + nout - 1 of W_down[e] are contiguous: one copy
      mbar_arrive_expect_tx(bar_a, nout * row_bytes);
      bulk_load(smem_u32(wrows), wd + (static_cast<int64_t>(e) * d + c0) * I, nout * row_bytes,
                bar_a);
      s_ok = wait_count(done + j, static_cast<unsigned int>(ngu), &abort_flag) ? 1 : 0;
      if (!s_ok && err) atomicExch(err, kDevErrTimeout);
    }
    __syncthreads();
    int p0;
    const int rows = s_ok ? rows_of(e, p0) : 0;
    for (int c = threadIdx.x; c < rows * i8; c += kThreads)  // expert j's h rows
      reinterpret_cast<uint4*>(vec)[c] =
          __ldcg(reinterpret_cast<const uint4*>(h + static_cast<int64_t>(p0) * I) + c);
    const bool ok = !__syncthreads_or(!wait_rows(bar_a, &abort_flag, err, parity) ? 1 : 0);
    parity ^= 1u;
    if (!ok || !s_ok) return;  // uniform: s_ok is shared, the copy has landed or was waited for
    for (int u = warp; u < nout; u += kWarps) {
      const uint4* row = reinterpret_cast<const uint4*>(wrows + u * I);
      float acc[MT] = {};
      for (int q8 = lane; q8 < i8; q8 += 32) {
        float fw[8];
        bf16x8_to_f32(row[q8], fw);
#pragma unroll
        for (int r = 0; r < MT; ++r) {
          if (r < rows) {
            float hv[8];
            bf16x8_to_f32(reinterpret_cast<const uint4*>(vec)[r * i8 + q8], hv);
#pragma unroll
            for (int q = 0; q < 8; ++q) acc[r] = fmaf(fw[q], hv[q], acc[r]);
          }
        }
      }
#pragma unroll
      for (int r = 0; r < MT; ++r) {
        if (r < rows) {
          const float sum = warp_sum(acc[r]);
          if (lane == 0)
            o[static_cast<int64_t>(p0 + r) * d + c0 + u] =
                __bfloat16_as_ushort(__float2bfloat16_rn(sum));
        }
      }
    }
    combine_tail(cmb, o, P, d, c0, nout, cb, n, &last);
    __syncthreads();  // the weight rows and h are free for the next item
  }
}

}  // namespace gemv

MOE_DEBUG_TU(gemv)

// Expert columns of the grid: at most min(N, T * K) experts have rows.
static unsigned gemv_experts(int64_t T, int K, int N) {
  const int64_t m = T * K < N ? T * K : N;
  return static_cast<unsigned>(m > 0 ? m : 1);
}

cudaError_t launch_gate_up_gemv(const uint16_t* x, int64_t T, const int32_t* perm,
                                const int32_t* offsets, const uint16_t* wgu, int64_t P, int d,
                                int N, int I, int K, uint16_t* h, int32_t* err,
                                cudaStream_t stream) {
  using namespace gemv;
  if (P == 0 || T == 0) return cudaSuccess;
  if (T > kMaxRows || d > kMaxDim || I > kMaxDim || d % 8 != 0) return cudaErrorInvalidValue;
  const size_t smem = static_cast<size_t>(2 * kGateUpOut) * d * 2 + sizeof(float) * T * d;
  static std::atomic<uint64_t> attr_done{0};
  const cudaError_t e = once_per_device(attr_done, [] {
    return cudaFuncSetAttribute(
        gemv_gate_up_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
        static_cast<int>(2 * kGateUpOut * kMaxDim * 2 + sizeof(float) * kMaxRows * kMaxDim));
  });
  if (e != cudaSuccess) return e;
  const dim3 grid(static_cast<unsigned>((I + kGateUpOut - 1) / kGateUpOut), gemv_experts(T, K, N));
  return launch_pdl(gemv_gate_up_kernel, grid, dim3(kThreads), smem, stream, x, T, perm, offsets,
                    wgu, P, d, N, I, h, err);
}

cudaError_t launch_down_gemv(const uint16_t* h, const int32_t* offsets, const uint16_t* wd,
                             int64_t T, int64_t P, int d, int N, int I, int K, uint16_t* o,
                             int32_t* err, cudaStream_t stream) {
  using namespace gemv;
  if (P == 0 || T == 0) return cudaSuccess;
  if (T > kMaxRows || d > kMaxDim || I > kMaxDim || I % 8 != 0) return cudaErrorInvalidValue;
  const size_t smem = static_cast<size_t>(kDownOut) * I * 2 + sizeof(float) * T * I;
  static std::atomic<uint64_t> attr_done{0};
  const cudaError_t e = once_per_device(attr_done, [] {
    return cudaFuncSetAttribute(
        gemv_down_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
        static_cast<int>(kDownOut * kMaxDim * 2 + sizeof(float) * kMaxRows * kMaxDim));
  });
  if (e != cudaSuccess) return e;
  const dim3 grid(static_cast<unsigned>((d + kDownOut - 1) / kDownOut), gemv_experts(T, K, N));
  return launch_pdl(gemv_down_kernel, grid, dim3(kThreads), smem, stream, h, offsets, wd, T, P, d,
                    N, I, o, err);
}


// The expert MLP and combine of a step of T <= 4 tokens (see
// gemv_expert_few_kernel): h [P, I] and o [P, d] scratch, done: 32 zeroed
// counters (left counting), tickets: ceil(d / 16) zeroed counters (left zero).
cudaError_t launch_expert_few_gemv(const uint16_t* x, int64_t T, const int32_t* perm,
                                   const int32_t* offsets, const uint16_t* wgu, const uint16_t* wd,
                                   int64_t P, int d, int N, int I, int K, uint16_t* h, uint16_t* o,
                                   int32_t* err, unsigned int* done, const int32_t* k,
                                   const int32_t* pair_pos, const float* gates,
                                   const uint16_t* residual, uint16_t* y, unsigned int* tickets,
                                   int num_sms, cudaStream_t stream) {
  using namespace gemv;
  if (P == 0 || T == 0) return cudaSuccess;
  if (T > kFewMaxT || d > kMaxDim || I > kMaxDim || d % 8 != 0 || I % 8 != 0 ||
      T * K > kFewMaxExperts || num_sms <= 0 || !done || !tickets || !k || !pair_pos || !gates ||
      !y)
    return cudaErrorInvalidValue;
  const int dn_max = std::min(64, std::max(16, (2 * kGateUpOut * d / I) / 8 * 8));
  // T * 64 combine threads at most
  static_assert(kFewMaxT * 64 <= kThreads, "combine threads");
  const uint32_t wbytes = static_cast<uint32_t>(
      std::max(2 * kGateUpOut * d * 2, dn_max * I * 2));
  const size_t smem = wbytes + 2 * static_cast<size_t>(T) * std::max(d, I);
  using Kern = void (*)(const uint16_t*, int, const int32_t*, const int32_t*, const uint16_t*,
                       const uint16_t*, int64_t, int, int, int, uint32_t, int, uint16_t*,
                       uint16_t*, int32_t*, unsigned int*, Combine);
  static const Kern kerns[3] = {gemv_expert_few_kernel<1>, gemv_expert_few_kernel<2>,
                                gemv_expert_few_kernel<4>};
  const Kern kern = kerns[T == 1 ? 0 : T == 2 ? 1 : 2];
  static std::atomic<uint64_t> attr_done{0};
  cudaError_t e = once_per_device(attr_done, [] {
    // (dn_max * I <= max(16 I, 16 d): at most 2 x 8 rows of kMaxDim)
    for (Kern k : kerns) {
      const cudaError_t r = cudaFuncSetAttribute(
          k, cudaFuncAttributeMaxDynamicSharedMemorySize,
          static_cast<int>(2 * kGateUpOut * kMaxDim * 2 + 2 * kFewMaxT * kMaxDim));
      if (r != cudaSuccess) return r;
    }
    return cudaSuccess;
  });
  if (e != cudaSuccess) return e;
  // resident blocks per SM for this kernel and size (cached: the last asked)
  static thread_local size_t cached_smem = 0;
  static thread_local Kern cached_kern = nullptr;
  static thread_local int cached_dev = -1, cached_blocks = 0;
  int dev = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if (cached_smem != smem || cached_dev != dev || cached_kern != kern) {
    int nb = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kern, kThreads, smem);
    if (e != cudaSuccess) return e;
    if (nb <= 0) return cudaErrorInvalidConfiguration;
    cached_smem = smem;
    cached_kern = kern;
    cached_dev = dev;
    cached_blocks = nb;
  }
  const int nexp = static_cast<int>(std::min<int64_t>(N, T * K));
  const int items = nexp * std::max((I + kGateUpOut - 1) / kGateUpOut, (d + 15) / 16);
  const int grid = std::min(items, cached_blocks * num_sms);
  const Combine cmb{k, pair_pos, gates, residual, y, tickets, K, static_cast<int>(T)};
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, x, static_cast<int>(T), perm, offsets, wgu, wd, P, d, N, I,
                            wbytes, dn_max, h, o, err, done, cmb);
}

}  // namespace moe
