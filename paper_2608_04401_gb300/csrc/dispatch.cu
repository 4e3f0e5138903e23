// Token-to-expert dispatch of the selected (t, s < k_t) pairs, stable in t,
// plus the row gather and the gate-weighted combine.
//
// Dispatch is a deterministic counting sort over chunks of 128 tokens:
//   count   : per chunk, per-expert pair counts (shared-memory increments), stored
//             expert-major: cnt[e][chunk]. The elbow router can write these
//             itself, in which case this pass is skipped.
//   scan    : one block per expert: exclusive prefix over the chunks, in
//             place, and the expert's total.
//   scatter : each chunk recomputes the expert offsets from the totals, then
//             places its pairs: position = offsets[e] + chunk base + earlier
//             warps of the chunk (per-expert warp masks in smem) + earlier lanes
//             of the warp (popc of the mask). Chunk 0 also writes offsets [N+1] and the
//             m-tile prefix sums ceil(count_e / 128) [N+1].
// A pair whose expert id lies outside [0, N) is dropped by every pass (not
// counted, not placed, pair_pos -1), so no id indexes outside the arrays.
#include <atomic>
#include <mutex>

#include "common.cuh"

namespace moe {
namespace disp {

constexpr int kChunk = 128;  // tokens per chunk = threads per block
constexpr int kWarps = kChunk / 32;
constexpr int kScanThreads = 1024;

// Expert-membership bit masks of one token's selection (experts 0..63,
// 64..127); ids outside [0, N) set no bit (their pairs are dropped).
template <int N>
MOE_DEV void load_selection(const int32_t* __restrict__ k, const int32_t* __restrict__ ids,
                            int64_t t, bool valid, int K, int& kt, int (&my)[8], uint64_t& m0,
                            uint64_t& m1) {
  kt = valid ? min(k[t], K) : 0;
  MOE_DCHECK(!valid || (k[t] >= 0 && k[t] <= K));
  if (valid && K == 8) {
    const int4 a = reinterpret_cast<const int4*>(ids + t * 8)[0];
    const int4 b = reinterpret_cast<const int4*>(ids + t * 8)[1];
    my[0] = a.x; my[1] = a.y; my[2] = a.z; my[3] = a.w;
    my[4] = b.x; my[5] = b.y; my[6] = b.z; my[7] = b.w;
  } else {
#pragma unroll
    for (int s = 0; s < 8; ++s) my[s] = (s < kt) ? ids[t * K + s] : 0;
  }
  m0 = 0;
  m1 = 0;
#pragma unroll
  for (int s = 0; s < 8; ++s) {
    MOE_DCHECK(s >= kt || static_cast<unsigned>(my[s]) < static_cast<unsigned>(N));
    if (s < kt && static_cast<unsigned>(my[s]) < static_cast<unsigned>(N)) {
      if (my[s] < 64) m0 |= 1ull << my[s];
      else m1 |= 1ull << (my[s] - 64);
    }
  }
}

// 32 x 32 bit-matrix transpose across a warp: lane i holds row i in x; lane j
// gets column j (bit i of the result = bit j of lane i's x). Five stages swap
// the off-diagonal blocks of width 16, 8, 4, 2, 1 with the partner lane
// (Warren, Hacker's Delight, sec. 7-3, with lanes as rows). Applied to the
// lanes' expert masks it gives lane e the ballot of expert e for the warp's 32
// tokens, in five shuffles instead of 32 ballots.
MOE_DEV uint32_t transpose32(uint32_t x, int lane) {
#pragma unroll
  for (int s = 16; s >= 1; s >>= 1) {
    const uint32_t m = s == 16 ? 0x0000FFFFu
                     : s == 8  ? 0x00FF00FFu
                     : s == 4  ? 0x0F0F0F0Fu
                     : s == 2  ? 0x33333333u
                               : 0x55555555u;
    const uint32_t y = __shfl_xor_sync(0xffffffffu, x, s);
    x = (lane & s) ? ((x & ~m) | ((y & ~m) >> s)) : ((x & m) | ((y & m) << s));
  }
  return x;
}

// The expert masks as 32-bit words: experts 32q .. 32q + 31 in word q.
MOE_DEV uint32_t mask_word(int q, uint64_t m0, uint64_t m1) {
  const uint64_t m = q < 2 ? m0 : m1;
  return static_cast<uint32_t>((q & 1) ? (m >> 32) : m);
}

template <int N>
__global__ void __launch_bounds__(kChunk) count_kernel(const int32_t* __restrict__ k,
                                                       const int32_t* __restrict__ ids, int64_t T,
                                                       int K, int nblk, int32_t* __restrict__ cnt) {
  // one shared-memory increment per selected pair (ids outside [0, N) are
  // not counted: they cannot come from the router)
  __shared__ int hist[N];
  grid_dep_wait();
  grid_dep_launch();
  for (int e = threadIdx.x; e < N; e += kChunk) hist[e] = 0;
  const int64_t t = static_cast<int64_t>(blockIdx.x) * kChunk + threadIdx.x;
  const bool valid = t < T;
  const int kt = valid ? min(k[t], K) : 0;
  MOE_DCHECK(!valid || (k[t] >= 0 && k[t] <= K));
  int my[8];
  if (valid && K == 8) {
    const int4 a = reinterpret_cast<const int4*>(ids + t * 8)[0];
    const int4 b = reinterpret_cast<const int4*>(ids + t * 8)[1];
    my[0] = a.x; my[1] = a.y; my[2] = a.z; my[3] = a.w;
    my[4] = b.x; my[5] = b.y; my[6] = b.z; my[7] = b.w;
  } else {
#pragma unroll
    for (int s = 0; s < 8; ++s) my[s] = (s < kt) ? ids[t * K + s] : 0;
  }
  __syncthreads();
#pragma unroll
  for (int s = 0; s < 8; ++s) {
    MOE_DCHECK(s >= kt || static_cast<unsigned>(my[s]) < static_cast<unsigned>(N));
    if (s < kt && static_cast<unsigned>(my[s]) < static_cast<unsigned>(N)) atomicAdd(&hist[my[s]], 1);
  }
  __syncthreads();
  for (int e = threadIdx.x; e < N; e += kChunk)
    cnt[static_cast<int64_t>(e) * nblk + blockIdx.x] = hist[e];
}

// ------------------------------------------------ single-pass dispatch
// The whole dispatch in one cooperative launch of G blocks (all resident),
// reading each selection once: block b owns the TB tokens [b TB, (b+1) TB)
// (TB a multiple of 32; unit u = its tokens 32u .. 32u + 31).
//   1. Each warp loads its units' k and ids (the next unit's loads in flight
//      while the current one is stored), keeps the ids as bytes (0xFF for
//      s >= k_t and ids outside [0, N)) and the unit's expert bit masks
//      mask[u][e] (bit l: token 32u + l selected e; a 32 x 32 transpose of
//      the tokens' expert masks) in shared memory, then counts its range of
//      units per expert. The block's per-expert count goes to agg[b][e].
//   2. One grid barrier (an arrival counter, zero on entry; the wait is
//      bounded and sets the error word when it runs out).
//   3. Every block adds the counts of the blocks before it and of all blocks
//      (its base and the expert totals); block 0 writes offsets, the m-tile
//      prefix sums and offsets_copy.
//   4. pair_pos: each warp walks its units in order with per-expert running
//      positions (in shared memory) and ranks each pair in its unit by the
//      popcount of the mask bits below its lane; a token's K positions leave
//      as 16-byte stores.
//   5. perm: each warp takes whole experts and walks their units 32 at a
//      time (lane = unit), a warp scan of the units' counts placing each
//      unit's tokens in ascending order.
// The result equals the counting sort above: rows by expert, then token.
constexpr int kCoopThreads = 1024;
constexpr int kCoopWarps = kCoopThreads / 32;

struct CoopSel {
  int kt;
  int id[8];
};

MOE_DEV CoopSel coop_load(const int32_t* __restrict__ k, const int32_t* __restrict__ ids,
                          int64_t t, bool valid, int K, bool vec) {
  CoopSel c;
  c.kt = valid ? min(max(k[t], 0), K) : 0;
  MOE_DCHECK(!valid || (k[t] >= 0 && k[t] <= K));
  if (valid && vec) {
    const int4 a = __ldg(reinterpret_cast<const int4*>(ids + t * 8));
    const int4 b = __ldg(reinterpret_cast<const int4*>(ids + t * 8) + 1);
    c.id[0] = a.x; c.id[1] = a.y; c.id[2] = a.z; c.id[3] = a.w;
    c.id[4] = b.x; c.id[5] = b.y; c.id[6] = b.z; c.id[7] = b.w;
  } else {
#pragma unroll
    for (int s = 0; s < 8; ++s) c.id[s] = (valid && s < K) ? __ldg(ids + t * K + s) : 0;
  }
  return c;
}

template <int N>
__global__ void __launch_bounds__(kCoopThreads, 1) dispatch_coop_kernel(
    const int32_t* __restrict__ k, const int32_t* __restrict__ ids, int64_t T, int K, int TB,
    int32_t* agg, unsigned int* arrive, int32_t* err, int32_t* __restrict__ perm,
    int32_t* __restrict__ pair_pos, int32_t* __restrict__ offsets, int32_t* __restrict__ tile_off,
    int32_t* __restrict__ offsets_copy) {
  constexpr int C = N / 32;      // mask words per unit (lane l: experts l + 32c)
  constexpr int kPitch = N + 1;  // mask row pitch (odd: lane-per-unit reads hit distinct banks)
  extern __shared__ __align__(16) uint8_t smem[];
  uint2* ids8 = reinterpret_cast<uint2*>(smem);                       // [TB] 8 id bytes
  uint32_t* mask = reinterpret_cast<uint32_t*>(smem + static_cast<size_t>(TB) * 8);  // [U][kPitch]
  __shared__ int rc[kCoopWarps][N];  // per warp range: count, then global start per expert
  __shared__ int s_base[N], s_tot[N], s_off[N], s_gbase[N];
  __shared__ int s_part[kCoopThreads / N][N];
  __shared__ int s_ok;
  grid_dep_wait();
  grid_dep_launch();
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int G = static_cast<int>(gridDim.x), b = static_cast<int>(blockIdx.x);
  const int64_t t0 = static_cast<int64_t>(b) * TB;
  const int U = TB / 32;
  const int UR = (U + kCoopWarps - 1) / kCoopWarps;  // units per warp range
  const int u0 = min(U, warp * UR), u1 = min(U, u0 + UR);
  const bool vec = K == 8 && (reinterpret_cast<uintptr_t>(ids) & 15u) == 0;
  const uint32_t lt_mask = (1u << lane) - 1u;

  // 1. selections -> id bytes and unit masks (each warp its own range of units)
  {
    int64_t t = t0 + static_cast<int64_t>(u0) * 32 + lane;
    CoopSel cur = coop_load(k, ids, t, u0 < u1 && t < T, K, vec);
    for (int u = u0; u < u1; ++u) {
      const int64_t tn = t + 32;
      const CoopSel nxt = coop_load(k, ids, tn, u + 1 < u1 && tn < T, K, vec);
      uint32_t lo = 0, hi = 0;
      uint64_t m0 = 0, m1 = 0;
#pragma unroll
      for (int s = 0; s < 8; ++s) {
        const bool ok = s < cur.kt && static_cast<unsigned>(cur.id[s]) < static_cast<unsigned>(N);
        MOE_DCHECK(s >= cur.kt || static_cast<unsigned>(cur.id[s]) < static_cast<unsigned>(N));
        const uint32_t byte = ok ? static_cast<uint32_t>(cur.id[s]) : 0xFFu;
        if (s < 4) lo |= byte << (8 * s);
        else hi |= byte << (8 * (s - 4));
        if (ok) {
          if (cur.id[s] < 64) m0 |= 1ull << cur.id[s];
          else m1 |= 1ull << (cur.id[s] - 64);
        }
      }
      ids8[u * 32 + lane] = make_uint2(lo, hi);
#pragma unroll
      for (int c = 0; c < C; ++c)
        mask[u * kPitch + 32 * c + lane] = transpose32(mask_word(c, m0, m1), lane);
      cur = nxt;
      t = tn;
    }
    __syncwarp();
    // the range's count per expert
#pragma unroll
    for (int c = 0; c < C; ++c) {
      int n = 0;
      for (int u = u0; u < u1; ++u) n += __popc(mask[u * kPitch + 32 * c + lane]);
      rc[warp][32 * c + lane] = n;
    }
  }
  __syncthreads();
  if (threadIdx.x < N) {
    const int e = threadIdx.x;
    int run = 0;
    for (int w = 0; w < kCoopWarps; ++w) {
      const int n = rc[w][e];
      rc[w][e] = run;  // exclusive within the block, for now
      run += n;
    }
    agg[static_cast<int64_t>(b) * N + e] = run;
  }
  // 2. grid barrier: the block's counts (the barrier) before thread 0's release
  __syncthreads();
  if (threadIdx.x == 0) {
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(arrive) : "memory");
    const uint64_t w0 = global_timer_ns();
    bool ok = true;
    for (uint32_t spins = 1;; ++spins) {
      unsigned int v;
      asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(arrive) : "memory");
      if (v >= static_cast<unsigned int>(G)) break;
      if (spins % 64u == 0u && global_timer_ns() - w0 > kWaitLimitNs) {
        ok = false;
        break;
      }
      __nanosleep(64);
    }
    if (!ok && err) atomicExch(err, kDevErrTimeout);
    s_ok = ok ? 1 : 0;
  }
  __syncthreads();
  if (!s_ok) return;
  // 3. this block's base and the expert totals
  {
    constexpr int kParts = kCoopThreads / N;
    const int e = threadIdx.x % N, part = threadIdx.x / N;
    int below = 0, tot = 0;
    for (int bb = part; bb < G; bb += kParts) {
      const int v = __ldcg(agg + static_cast<int64_t>(bb) * N + e);
      tot += v;
      below += bb < b ? v : 0;
    }
    s_part[part][e] = below;
    __syncthreads();
    if (part == 0) {
      int sb = below;
      for (int pp = 1; pp < kParts; ++pp) sb += s_part[pp][e];
      s_base[e] = sb;
    }
    __syncthreads();
    s_part[part][e] = tot;
    __syncthreads();
    if (part == 0) {
      int st = tot;
      for (int pp = 1; pp < kParts; ++pp) st += s_part[pp][e];
      s_tot[e] = st;
    }
    __syncthreads();
  }
  if (warp == 0) {  // exclusive scans over the experts: offsets and m-tile counts
    int run = 0, trun = 0;
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const int e = 32 * c + lane;
      const int v = s_tot[e], tv = (v + 127) / 128;
      int x = v, tx = tv;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o), ty = __shfl_up_sync(0xffffffffu, tx, o);
        if (lane >= o) {
          x += y;
          tx += ty;
        }
      }
      const int off = run + x - v, toff = trun + tx - tv;
      s_off[e] = off;
      s_gbase[e] = off + s_base[e];
      if (b == 0) {
        offsets[e] = off;
        tile_off[e] = toff;
        if (offsets_copy) offsets_copy[e] = off;
      }
      run += __shfl_sync(0xffffffffu, x, 31);
      trun += __shfl_sync(0xffffffffu, tx, 31);
    }
    if (b == 0 && lane == 0) {
      MOE_DCHECK(static_cast<int64_t>(run) <= T * K);
      offsets[N] = run;
      tile_off[N] = trun;
      if (offsets_copy) offsets_copy[N] = run;
    }
  }
  __syncthreads();
  // 4. pair_pos, each warp over its units in order; rc[warp][e] becomes the
  // running position of expert e (global)
#pragma unroll
  for (int c = 0; c < C; ++c) rc[warp][32 * c + lane] += s_gbase[32 * c + lane];
  __syncwarp();
  {
    int* run = rc[warp];
    for (int u = u0; u < u1; ++u) {
      const int64_t t = t0 + static_cast<int64_t>(u) * 32 + lane;
      const uint2 w8 = ids8[u * 32 + lane];
      const uint32_t* mrow = mask + u * kPitch;
      int pp[8];
#pragma unroll
      for (int s = 0; s < 8; ++s) {
        const uint32_t byte = __byte_perm(s < 4 ? w8.x : w8.y, 0u, 0x4440u | (s & 3));
        const int e = static_cast<int>(byte & (N - 1));  // 0xFF: an in-range index, unused
        const int v = run[e] + __popc(mrow[e] & lt_mask);
        pp[s] = byte == 0xFFu ? -1 : v;
      }
      __syncwarp();
#pragma unroll
      for (int c = 0; c < C; ++c) run[32 * c + lane] += __popc(mrow[32 * c + lane]);
      __syncwarp();
      if (t < T) {
        int32_t* dst = pair_pos + t * K;
        if (K == 8 && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
          reinterpret_cast<int4*>(dst)[0] = make_int4(pp[0], pp[1], pp[2], pp[3]);
          reinterpret_cast<int4*>(dst)[1] = make_int4(pp[4], pp[5], pp[6], pp[7]);
        } else {
#pragma unroll
          for (int s = 0; s < 8; ++s)
            if (s < K) dst[s] = pp[s];
        }
      }
    }
  }
  // 5. perm, each warp over whole experts (units 32 at a time, lane = unit):
  // a warp scan of the units' counts places each unit's tokens in ascending
  // order (consecutive lanes write neighbouring runs). A unit holds at most K
  // bits per token and only ids below N, so the block's positions stay below
  // the total pair count <= T K: no store leaves perm.
  for (int e = warp; e < N; e += kCoopWarps) {
    int run = s_gbase[e];
    for (int ub = 0; ub < U; ub += 32) {
      const int u = ub + lane;
      uint32_t m = u < U ? mask[u * kPitch + e] : 0u;
      const int c = __popc(m);
      int x = c;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      MOE_DCHECK(m == 0u || (run + x - c >= 0 && static_cast<int64_t>(run + x) <= T * K));
      int32_t* dst = perm + (run + x - c);
      const int32_t tu = static_cast<int32_t>(t0) + u * 32;
      while (m) {
        *dst++ = tu + (__ffs(static_cast<int>(m)) - 1);
        m &= m - 1u;
      }
      run += __shfl_sync(0xffffffffu, x, 31);
    }
  }
}

// Block e: exclusive prefix sum of cnt[e][0 .. nblk) in place; total -> totals[e].
// Warp w owns a contiguous segment of the chunks, read in coalesced 32-chunk
// slices: a first pass sums the segment, the block scans the warp sums, and a
// second pass rescans each slice (eight slices loaded ahead) with the carry.
__global__ void __launch_bounds__(kScanThreads) scan_kernel(int32_t* __restrict__ cnt, int nblk,
                                                            int32_t* __restrict__ totals) {
  constexpr int kW = kScanThreads / 32;
  __shared__ int warp_sum[kW];
  grid_dep_wait();
  grid_dep_launch();
  int32_t* col = cnt + static_cast<int64_t>(blockIdx.x) * nblk;
  const int lane = threadIdx.x % 32, warp = threadIdx.x / 32;
  const int seg = (((nblk + kW - 1) / kW) + 31) & ~31;
  const int s0 = warp * seg;
  const int s1 = min(nblk, s0 + seg);
  int sum = 0;
  for (int b = s0 + lane; b < s1; b += 32) sum += col[b];
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  if (lane == 0) warp_sum[warp] = sum;
  __syncthreads();
  int carry = 0, total = 0;
#pragma unroll
  for (int w = 0; w < kW; ++w) {
    if (w < warp) carry += warp_sum[w];
    total += warp_sum[w];
  }
  for (int base = s0; base < s1; base += 8 * 32) {
    int v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int b = base + 32 * j + lane;
      v[j] = b < s1 ? col[b] : 0;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      int x = v[j];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      const int b = base + 32 * j + lane;
      if (b < s1) col[b] = carry + x - v[j];
      carry += __shfl_sync(0xffffffffu, x, 31);
    }
  }
  if (threadIdx.x == 0) totals[blockIdx.x] = total;
}

// Exclusive scan of N <= 128 values held by threads 0..N-1 of a 128-thread
// block; every thread gets the scan of its own index (0 beyond N) and the total.
template <int N>
MOE_DEV int block_exclusive_scan_small(int v, int* warp_tmp, int& total) {
  const int lane = threadIdx.x % 32, warp = threadIdx.x / 32;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tmp[warp] = x;
  __syncthreads();
  int before = 0;
  total = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    if (w < warp) before += warp_tmp[w];
    total += warp_tmp[w];
  }
  __syncthreads();
  return before + x - v;
}

// SINGLE: the batch is one chunk (T <= 128); its own counts are the expert
// totals and its scan the expert offsets, so no count or scan pass runs.
// GATHER (with SINGLE): every block of the grid computes the chunk's dispatch
// in shared memory, block 0 writes it out, and all blocks copy the dispatched
// token rows xs[r] = x[perm[r]] (one warp per row, rows strided over the grid),
// so the gather needs no launch of its own.
template <int N, bool SINGLE, bool GATHER = false>
__global__ void __launch_bounds__(kChunk) scatter_kernel(
    const int32_t* __restrict__ k, const int32_t* __restrict__ ids, int64_t T, int K, int nblk,
    const int32_t* __restrict__ base, const int32_t* __restrict__ totals,
    int32_t* __restrict__ perm, int32_t* __restrict__ pair_pos, int32_t* __restrict__ offsets,
    int32_t* __restrict__ tile_off, int32_t* __restrict__ offsets_copy,
    const uint4* __restrict__ x = nullptr, int d8 = 0, uint4* __restrict__ xs = nullptr) {
  static_assert(SINGLE || !GATHER, "the fused gather needs the single-chunk dispatch");
  grid_dep_wait();
  grid_dep_launch();
  const bool writer = !GATHER || blockIdx.x == 0;
  __shared__ int exp_off[N];
  __shared__ uint32_t bal[kWarps][N];
  __shared__ int wbase[kWarps][N];   // global position of each warp's first pair per expert
  __shared__ int lbase[kWarps][N];   // the same inside this chunk's expert-sorted pair list
  __shared__ int warp_tmp[kWarps];
  __shared__ int s_tok[kChunk * 8];  // the chunk's pairs sorted by expert: token
  __shared__ int s_gpos[kChunk * 8]; //                                     and global position
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int tid = threadIdx.x;

  // expert offsets [N + 1] and m-tile prefix sums [N + 1], written by block 0
  auto write_offsets = [&](int tot, int off, int total_pairs) {
    int total_tiles;
    const int toff = block_exclusive_scan_small<N>(tid < N ? (tot + 127) / 128 : 0, warp_tmp,
                                                   total_tiles);
    if (tid < N) {
      offsets[tid] = off;
      tile_off[tid] = toff;
      if (offsets_copy) offsets_copy[tid] = off;
    }
    if (tid == 0) {
      MOE_DCHECK(total_pairs >= 0 && static_cast<int64_t>(total_pairs) <= T * K);
      offsets[N] = total_pairs;
      tile_off[N] = total_tiles;
      if (offsets_copy) offsets_copy[N] = total_pairs;
    }
  };
  // every global input of the block is requested first, so that their
  // latencies overlap: the tokens' selections, the expert totals and this
  // chunk's per-expert base counts
  // (with GATHER every block works on the one chunk)
  const int64_t t = (GATHER ? 0 : static_cast<int64_t>(blockIdx.x) * kChunk) + tid;
  const bool valid = t < T;
  int kt, my[8];
  uint64_t m0, m1;
  load_selection<N>(k, ids, t, valid, K, kt, my, m0, m1);
  int chunk_base = 0;
  if constexpr (!SINGLE) {
    if (tid < N) chunk_base = base[static_cast<int64_t>(tid) * nblk + blockIdx.x];
    // expert offsets from the totals (every chunk recomputes them)
    const int tot = tid < N ? totals[tid] : 0;
    int total_pairs;
    const int off = block_exclusive_scan_small<N>(tot, warp_tmp, total_pairs);
    if (tid < N) exp_off[tid] = off;
    if (blockIdx.x == 0) write_offsets(tot, off, total_pairs);
  }
#pragma unroll
  for (int q = 0; q < N / 32; ++q) bal[warp][32 * q + lane] = transpose32(mask_word(q, m0, m1), lane);
  __syncthreads();
  // this chunk's count per expert, and its exclusive scan over the experts
  int c_e = 0;
  if (tid < N) {
#pragma unroll
    for (int w = 0; w < kWarps; ++w) c_e += __popc(bal[w][tid]);
  }
  int chunk_pairs;
  const int chunk_off = block_exclusive_scan_small<N>(c_e, warp_tmp, chunk_pairs);
  if constexpr (SINGLE) {
    if (writer) write_offsets(c_e, chunk_off, chunk_pairs);  // block-uniform condition
  }
  if (tid < N) {
    int acc = SINGLE ? chunk_off : exp_off[tid] + chunk_base;
    int lacc = chunk_off;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      wbase[w][tid] = acc;
      lbase[w][tid] = lacc;
      const int c = __popc(bal[w][tid]);
      acc += c;
      lacc += c;
    }
  }
  __syncthreads();
  if (valid) {
    const uint32_t lt_mask = (1u << lane) - 1u;
    int pp[8];
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      pp[s] = -1;
      if (s < kt && static_cast<unsigned>(my[s]) < static_cast<unsigned>(N)) {
        const int e = my[s];
        const int below = __popc(bal[warp][e] & lt_mask);
        const int pos = wbase[warp][e] + below;
        const int lpos = lbase[warp][e] + below;
        s_tok[lpos] = static_cast<int32_t>(t);
        s_gpos[lpos] = pos;
        pp[s] = pos;
      }
    }
    if (writer) {
      // the token's K positions are contiguous: whole 16-byte stores where
      // they fit (one store per pair would touch a sector per lane)
      int32_t* dst = pair_pos + t * K;
      if (K == 8 && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
        reinterpret_cast<int4*>(dst)[0] = make_int4(pp[0], pp[1], pp[2], pp[3]);
        reinterpret_cast<int4*>(dst)[1] = make_int4(pp[4], pp[5], pp[6], pp[7]);
      } else if (K == 4 && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
        reinterpret_cast<int4*>(dst)[0] = make_int4(pp[0], pp[1], pp[2], pp[3]);
      } else {
#pragma unroll
        for (int s = 0; s < 8; ++s)
          if (s < K) dst[s] = pp[s];
      }
    }
  }
  __syncthreads();
  // write perm from the expert-sorted list: consecutive threads write
  // consecutive positions inside each expert's run
  if (writer) {
    for (int i = tid; i < chunk_pairs; i += kChunk) {
      const int pos = s_gpos[i];
      // positions stay below T*K when the counts match the ids
      MOE_DCHECK(pos >= 0 && static_cast<int64_t>(pos) < T * K);
      if (pos >= 0 && static_cast<int64_t>(pos) < T * K) perm[pos] = s_tok[i];
    }
  }
  if constexpr (GATHER) {
    // single chunk: the global position of list entry r is r itself
    for (int r = blockIdx.x * kWarps + warp; r < chunk_pairs; r += gridDim.x * kWarps) {
      const uint4* src = x + static_cast<int64_t>(s_tok[r]) * d8;
      uint4* dst = xs + static_cast<int64_t>(r) * d8;
      for (int c = lane; c < d8; c += 32) dst[c] = __ldg(src + c);
    }
  }
}

// xs[r] = x[perm[r]] for r < offsets[N]; one warp per row, 16-byte copies.
// Rows stop at the capacity P and tokens are clamped to [0, T), so that
// inconsistent arguments cannot reach outside x or xs.
__global__ void __launch_bounds__(256) gather_kernel(const uint4* __restrict__ x,
                                                     const int32_t* __restrict__ perm,
                                                     const int32_t* __restrict__ offsets, int N,
                                                     int64_t T, int64_t P, int d8,
                                                     uint4* __restrict__ xs) {
  const int64_t total = min_of<int64_t>(offsets[N], P);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  MOE_DCHECK(offsets[N] >= 0 && offsets[N] <= P);
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * 8 + warp; r < total;
       r += static_cast<int64_t>(gridDim.x) * 8) {
    const int64_t pt = perm[r];
    MOE_DCHECK(pt >= 0 && pt < T);
    const int64_t t = pt < 0 ? 0 : (pt >= T ? T - 1 : pt);
    const uint4* src = x + t * d8;
    uint4* dst = xs + r * d8;
    for (int c = lane; c < d8; c += 32) dst[c] = __ldg(src + c);
  }
}

// y_t = sum_{s<k_t} g_{t,s} * o[pair_pos[t,s]] (+ residual_t); fp32 in s order.
// One warp per unit: a whole token, or for small batches (SPLIT) one slab of a
// token so that they still spread over many warps. A slab is 32 * CH
// sixteen-byte chunks (lane l owns chunks l + 32c, c < CH; CH = 2 without a
// residual, 1 with one). The k rows of a slab (and the residual) are copied
// with cp.async into this warp's two-stage shared-memory ring while the
// previous slab is accumulated, so a warp keeps up to two slabs (16 KB) in
// flight without holding them in registers. Each lane reads back only the
// chunks it copied itself, so no barrier is needed between the lanes; the
// next unit's k, positions and gates are read a unit ahead.
constexpr int kCombineWarps = 4;

template <bool RES>
struct CombineCfg {
  static constexpr int CH = RES ? 1 : 2;
  static constexpr int kSlabChunks = 32 * CH;
  static constexpr int kRows = 8 + (RES ? 1 : 0);                 // k rows (+ residual)
  static constexpr int kStage = kRows * CH * 32;                  // uint4 per stage
  static constexpr int kWarpBytes = 2 * kStage * 16;              // two stages
  static constexpr int kBlockBytes = kCombineWarps * kWarpBytes;
};

MOE_DEV void combine_cp16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src)
               : "memory");
}

struct CombineUnit {
  int64_t t;
  int s0, s1, kt, pos;
  float g;
  bool valid;
};

template <bool RES, bool SPLIT>
__global__ void __launch_bounds__(32 * kCombineWarps) combine_kernel(
    const uint4* __restrict__ o, const int32_t* __restrict__ k, const int32_t* __restrict__ pair_pos,
    const float* __restrict__ gates, const uint4* residual, int64_t T, int d8, int K, uint4* y) {
  using C = CombineCfg<RES>;
  constexpr int CH = C::CH;
  extern __shared__ uint4 cmb_smem[];
  grid_dep_wait();
  grid_dep_launch();
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x / 32;
  uint4* ring = cmb_smem + static_cast<size_t>(warp) * 2 * C::kStage;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kCombineWarps;
  const int64_t cap = T * K;
  const int nslab = (d8 + C::kSlabChunks - 1) / C::kSlabChunks;
  const int64_t units = SPLIT ? T * nslab : T;

  auto unit_at = [&](int64_t u) {
    CombineUnit m;
    m.valid = u < units;
    if (!m.valid) {
      m.t = 0; m.s0 = m.s1 = 0; m.kt = 0; m.pos = 0; m.g = 0.0f;
      return m;
    }
    m.t = SPLIT ? u / nslab : u;
    m.s0 = SPLIT ? static_cast<int>(u % nslab) * C::kSlabChunks : 0;
    m.s1 = SPLIT ? m.s0 + C::kSlabChunks : d8;
    m.kt = min(k[m.t], K);
    MOE_DCHECK(k[m.t] >= 0 && k[m.t] <= K);
    MOE_DCHECK(lane >= m.kt || (pair_pos[m.t * K + lane] >= 0 &&
                                static_cast<int64_t>(pair_pos[m.t * K + lane]) < cap));
    m.pos = lane < m.kt ? static_cast<int>(min_of<int64_t>(max(pair_pos[m.t * K + lane], 0), cap - 1))
                        : 0;
    m.g = lane < m.kt ? gates[m.t * K + lane] : 0.0f;
    return m;
  };
  // copies of one slab of unit m into stage st (rows s >= kt are not read back)
  auto issue = [&](const CombineUnit& m, int slab, int st) {
    uint4* b = ring + st * C::kStage;
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      const int p = __shfl_sync(0xffffffffu, m.pos, s);
#pragma unroll
      for (int c = 0; c < CH; ++c) {
        const int ci = slab + lane + 32 * c;
        if (s < m.kt && ci < d8)
          combine_cp16(b + (s * CH + c) * 32 + lane, o + static_cast<int64_t>(p) * d8 + ci);
      }
    }
    if constexpr (RES) {
#pragma unroll
      for (int c = 0; c < CH; ++c) {
        const int ci = slab + lane + 32 * c;
        if (ci < d8) combine_cp16(b + (8 * CH + c) * 32 + lane, residual + m.t * d8 + ci);
      }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };

  int64_t u = static_cast<int64_t>(blockIdx.x) * kCombineWarps + warp;
  CombineUnit cur = unit_at(u);
  if (!cur.valid) return;  // uniform per warp
  CombineUnit nxt = unit_at(u + nwarps);
  int slab = cur.s0;
  int st = 0;
  issue(cur, slab, 0);
  while (true) {
    // the next slab: the rest of this unit, else the next unit's first
    const bool more_here = slab + C::kSlabChunks < cur.s1;
    if (more_here) {
      issue(cur, slab + C::kSlabChunks, st ^ 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else if (nxt.valid) {
      issue(nxt, nxt.s0, st ^ 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    // accumulate this slab from the ring, in s order
    const uint4* b = ring + st * C::kStage;
    float acc[CH][8];
#pragma unroll
    for (int c = 0; c < CH; ++c)
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[c][q] = 0.0f;
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      const float g = __shfl_sync(0xffffffffu, cur.g, s);
      if (s < cur.kt) {
#pragma unroll
        for (int c = 0; c < CH; ++c) {
          const uint4 v = b[(s * CH + c) * 32 + lane];
          const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float2 f = __bfloat1622float2(h[q]);
            acc[c][2 * q] = fmaf(g, f.x, acc[c][2 * q]);
            acc[c][2 * q + 1] = fmaf(g, f.y, acc[c][2 * q + 1]);
          }
        }
      }
    }
#pragma unroll
    for (int c = 0; c < CH; ++c) {
      const int ci = slab + lane + 32 * c;
      if (ci >= d8) continue;
      if constexpr (RES) {
        const uint4 rv = b[(8 * CH + c) * 32 + lane];
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&rv);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 f = __bfloat1622float2(h[q]);
          acc[c][2 * q] += f.x;
          acc[c][2 * q + 1] += f.y;
        }
      }
      uint4 out;
      out.x = pack_bf16x2(acc[c][0], acc[c][1]);
      out.y = pack_bf16x2(acc[c][2], acc[c][3]);
      out.z = pack_bf16x2(acc[c][4], acc[c][5]);
      out.w = pack_bf16x2(acc[c][6], acc[c][7]);
      y[cur.t * d8 + ci] = out;
    }
    // advance
    if (more_here) {
      slab += C::kSlabChunks;
    } else {
      if (!nxt.valid) break;
      cur = nxt;
      slab = cur.s0;
      u += nwarps;
      nxt = unit_at(u + nwarps);
    }
    st ^= 1;
  }
}

}  // namespace disp

MOE_DEBUG_TU(dispatch)

static int num_chunks(int64_t T) { return static_cast<int>((T + disp::kChunk - 1) / disp::kChunk); }

// Workspace layout: header (256 bytes: error word, the single-pass
// dispatch's barrier counter) | cnt/base [N][nchunks] int32 (the single-pass
// dispatch's per-block counts [G][N], G <= nchunks) | totals [N] | tile_off [N+1]
constexpr size_t kWsHeader = 256;

size_t dispatch_ws_bytes(int64_t T, int N) {
  auto up = [](size_t b) { return (b + 255) & ~static_cast<size_t>(255); };
  const size_t nblk = static_cast<size_t>(num_chunks(T) > 0 ? num_chunks(T) : 1);
  return kWsHeader + up(nblk * N * sizeof(int32_t)) + up(N * sizeof(int32_t)) +
         up((N + 1) * sizeof(int32_t));
}

int32_t* dispatch_counts(void* ws) {
  return reinterpret_cast<int32_t*>(static_cast<char*>(ws) + kWsHeader);
}

static int32_t* dispatch_totals(void* ws, int64_t T, int N) {
  auto up = [](size_t b) { return (b + 255) & ~static_cast<size_t>(255); };
  const size_t nblk = static_cast<size_t>(num_chunks(T) > 0 ? num_chunks(T) : 1);
  return reinterpret_cast<int32_t*>(reinterpret_cast<char*>(dispatch_counts(ws)) +
                                    up(nblk * N * sizeof(int32_t)));
}

int32_t* dispatch_tile_off(void* ws, int64_t T, int N) {
  auto up = [](size_t b) { return (b + 255) & ~static_cast<size_t>(255); };
  return reinterpret_cast<int32_t*>(reinterpret_cast<char*>(dispatch_totals(ws, T, N)) +
                                    up(N * sizeof(int32_t)));
}

// The single-pass dispatch's shape: G blocks of TB tokens and the dynamic
// shared memory of one block; false when it does not fit (one block per SM,
// at most kCoopMaxSmem bytes) or the batch is too small to need it.
constexpr size_t kCoopMaxSmem = 200 * 1024;

static bool coop_shape(int64_t T, int N, int num_sms, int& G, int& TB, size_t& smem) {
  if (T <= disp::kChunk || num_sms <= 0) return false;
  const int64_t nblk = num_chunks(T);  // the counts region holds nblk x N ints
  int64_t g = num_sms < nblk ? num_sms : nblk;
  int64_t tb = ((T + g - 1) / g + 31) / 32 * 32;
  g = (T + tb - 1) / tb;
  smem = static_cast<size_t>(tb) * 8 + static_cast<size_t>(tb / 32) * (N + 1) * sizeof(uint32_t);
  if (smem > kCoopMaxSmem) return false;
  G = static_cast<int>(g);
  TB = static_cast<int>(tb);
  return true;
}

// The single-pass dispatch (see dispatch_coop_kernel). arrive: a zeroed
// counter; err: the word a barrier timeout sets.
static cudaError_t launch_dispatch_coop(const int32_t* k, const int32_t* ids, int64_t T, int N,
                                        int K, int G, int TB, size_t smem, int32_t* agg,
                                        unsigned int* arrive, int32_t* err, int32_t* perm,
                                        int32_t* pair_pos, int32_t* offsets, int32_t* tile_off,
                                        int32_t* offsets_copy, cudaStream_t stream) {
  using Kern = void (*)(const int32_t*, const int32_t*, int64_t, int, int, int32_t*, unsigned int*,
                        int32_t*, int32_t*, int32_t*, int32_t*, int32_t*, int32_t*);
  const Kern kern = N == 64 ? disp::dispatch_coop_kernel<64> : disp::dispatch_coop_kernel<128>;
  static std::atomic<uint64_t> attr_done{0};
  const cudaError_t e = once_per_device(attr_done, [] {
    for (Kern f : {disp::dispatch_coop_kernel<64>, disp::dispatch_coop_kernel<128>}) {
      const cudaError_t r = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 static_cast<int>(kCoopMaxSmem));
      if (r != cudaSuccess) return r;
    }
    return cudaSuccess;
  });
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(G));
  cfg.blockDim = dim3(disp::kCoopThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, k, ids, T, K, TB, agg, arrive, err, perm, pair_pos, offsets,
                            tile_off, offsets_copy);
}

// SM count of the current device (cached per device ordinal below 64).
static int sm_count_cached() {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (dev >= 0 && dev < 64) {
    const int c = cache[dev].load(std::memory_order_relaxed);
    if (c > 0) return c;
  }
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  if (dev >= 0 && dev < 64) cache[dev].store(n, std::memory_order_relaxed);
  return n;
}

// counts_ready: the elbow router already wrote the per-chunk counts into cnt
// (then the scan and scatter passes run: faster than the single pass, which
// would count again). Otherwise arrive, a zeroed counter, enables the
// single-pass dispatch (err: the word its barrier timeout sets); nullptr
// gives the count / scan / scatter passes.
static cudaError_t run_dispatch(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                                int32_t* offsets, int32_t* perm, int32_t* pair_pos, int32_t* cnt,
                                int32_t* totals, int32_t* tile_off, int32_t* offsets_copy,
                                bool counts_ready, int32_t* err, unsigned int* arrive,
                                cudaStream_t stream) {
  const int nblk = num_chunks(T);
  const uint4* no_x = nullptr;
  uint4* no_xs = nullptr;
  if (nblk == 1) {
    auto kern = N == 64 ? disp::scatter_kernel<64, true> : disp::scatter_kernel<128, true>;
    return launch_pdl(kern, dim3(1), dim3(disp::kChunk), 0, stream, k, ids, T, K, nblk, cnt, totals,
                      perm, pair_pos, offsets, tile_off, offsets_copy, no_x, 0, no_xs);
  }
  cudaError_t e;
  int G = 0, TB = 0;
  size_t smem = 0;
  if (arrive && !counts_ready && coop_shape(T, N, sm_count_cached(), G, TB, smem)) {
    e = launch_dispatch_coop(k, ids, T, N, K, G, TB, smem, cnt, arrive, err, perm, pair_pos,
                             offsets, tile_off, offsets_copy, stream);
    // a device whose SMs are not all available to this context (MPS, green
    // contexts) may refuse the co-resident grid: the passes below need none
    if (e != cudaErrorCooperativeLaunchTooLarge) return e;
    (void)cudaGetLastError();
  }
  if (nblk > 0 && !counts_ready) {
    auto kern = N == 64 ? disp::count_kernel<64> : disp::count_kernel<128>;
    e = launch_pdl(kern, dim3(nblk), dim3(disp::kChunk), 0, stream, k, ids, T, K, nblk, cnt);
    if (e != cudaSuccess) return e;
  }
  if (nblk > 0) {
    e = launch_pdl(disp::scan_kernel, dim3(N), dim3(disp::kScanThreads), 0, stream, cnt, nblk, totals);
  } else {
    e = cudaMemsetAsync(totals, 0, N * sizeof(int32_t), stream);
  }
  if (e != cudaSuccess) return e;
  const int grid = nblk > 0 ? nblk : 1;
  auto kern = N == 64 ? disp::scatter_kernel<64, false> : disp::scatter_kernel<128, false>;
  return launch_pdl(kern, dim3(grid), dim3(disp::kChunk), 0, stream, k, ids, T, K, nblk, cnt, totals,
                    perm, pair_pos, offsets, tile_off, offsets_copy, no_x, 0, no_xs);
}

// err / arrive: the error word and a zeroed counter for the single-pass
// dispatch, or nullptr to use the workspace header's two words, which are
// cleared here when the single-pass dispatch runs.
cudaError_t launch_dispatch(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                            int32_t* offsets, int32_t* perm, int32_t* pair_pos, void* ws,
                            int32_t* offsets_copy, bool counts_ready, int32_t* err,
                            unsigned int* arrive, cudaStream_t stream) {
  int G = 0, TB = 0;
  size_t smem = 0;
  if (!arrive && !counts_ready && num_chunks(T) > 1 &&
      coop_shape(T, N, sm_count_cached(), G, TB, smem)) {
    err = static_cast<int32_t*>(ws);
    arrive = reinterpret_cast<unsigned int*>(err + 1);
    const cudaError_t e = cudaMemsetAsync(ws, 0, 2 * sizeof(int32_t), stream);
    if (e != cudaSuccess) return e;
  }
  return run_dispatch(k, ids, T, N, K, offsets, perm, pair_pos, dispatch_counts(ws),
                      dispatch_totals(ws, T, N), dispatch_tile_off(ws, T, N), offsets_copy,
                      counts_ready, err, arrive, stream);
}

// Single-chunk dispatch (T <= 128) fused with the row gather xs[r] = x[perm[r]].
cudaError_t launch_dispatch_gather(const int32_t* k, const int32_t* ids, int64_t T, int N, int K,
                                   int32_t* offsets, int32_t* perm, int32_t* pair_pos, void* ws,
                                   int32_t* offsets_copy, const uint16_t* x, int d, uint16_t* xs,
                                   int num_sms, cudaStream_t stream) {
  if (num_chunks(T) != 1) return cudaErrorInvalidValue;
  // one warp per dispatched row: T * K rows at most
  int64_t blocks = (T * K + disp::kWarps - 1) / disp::kWarps;
  if (blocks > num_sms) blocks = num_sms;
  auto kern = N == 64 ? disp::scatter_kernel<64, true, true> : disp::scatter_kernel<128, true, true>;
  return launch_pdl(kern, dim3(static_cast<unsigned>(blocks)), dim3(disp::kChunk), 0, stream, k, ids,
                    T, K, 1, static_cast<const int32_t*>(dispatch_counts(ws)),
                    static_cast<const int32_t*>(dispatch_totals(ws, T, N)), perm, pair_pos, offsets,
                    dispatch_tile_off(ws, T, N), offsets_copy, reinterpret_cast<const uint4*>(x),
                    d / 8, reinterpret_cast<uint4*>(xs));
}

cudaError_t launch_gather(const uint16_t* x, int64_t T, const int32_t* perm, const int32_t* offsets,
                          int N, int64_t P, int d, uint16_t* xs, int num_sms, cudaStream_t stream) {
  if (P == 0 || T == 0) return cudaSuccess;
  int64_t blocks = (P + 7) / 8;
  const int64_t cap = static_cast<int64_t>(num_sms) * 16;
  if (blocks > cap) blocks = cap;
  disp::gather_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(
      reinterpret_cast<const uint4*>(x), perm, offsets, N, T, P, d / 8, reinterpret_cast<uint4*>(xs));
  return cudaGetLastError();
}

cudaError_t launch_combine(const uint16_t* o, const int32_t* k, const int32_t* pair_pos,
                           const float* gates, const uint16_t* residual, int64_t T, int d, int K,
                           uint16_t* y, int num_sms, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  const int ch = residual ? 32 : 64;  // sixteen-byte chunks per slab
  const int nslab = (d / 8 + ch - 1) / ch;
  // whole tokens per warp once the batch alone fills the GPU; slabs otherwise
  const bool split = T < static_cast<int64_t>(num_sms) * 16;
  const int64_t units = split ? T * nslab : T;
  const int smem = residual ? disp::CombineCfg<true>::kBlockBytes : disp::CombineCfg<false>::kBlockBytes;
  auto kern = residual ? (split ? disp::combine_kernel<true, true> : disp::combine_kernel<true, false>)
                       : (split ? disp::combine_kernel<false, true> : disp::combine_kernel<false, false>);
  static std::atomic<uint64_t> attr_done{0};
  const cudaError_t ae = once_per_device(attr_done, [] {
    for (auto f : {disp::combine_kernel<true, true>, disp::combine_kernel<true, false>,
                   disp::combine_kernel<false, true>, disp::combine_kernel<false, false>}) {
      const cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 disp::CombineCfg<false>::kBlockBytes);
      if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
  });
  if (ae != cudaSuccess) return ae;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 32 * disp::kCombineWarps, smem) !=
          cudaSuccess ||
      per_sm < 1)
    per_sm = 1;
  int64_t blocks = (units + disp::kCombineWarps - 1) / disp::kCombineWarps;
  const int64_t cap = static_cast<int64_t>(num_sms) * per_sm;
  if (blocks > cap) blocks = cap;
  return launch_pdl(kern, dim3(static_cast<unsigned>(blocks)), dim3(32 * disp::kCombineWarps), smem,
                    stream, reinterpret_cast<const uint4*>(o), k, pair_pos, gates,
                    reinterpret_cast<const uint4*>(residual), T, d / 8, K,
                    reinterpret_cast<uint4*>(y));
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
constexpr int64_t kNoAllocMaxTokens = int64_t(1) << 18;  // 262,144 tokens
constexpr int kNoAllocMaxExperts = 128;
constexpr int64_t kNoAllocChunks = (kNoAllocMaxTokens + kChunk - 1) / kChunk;
// counts [experts][chunks], totals [experts], tile offsets [experts + 1]: ~1 MB
constexpr int64_t kNoAllocInts = kNoAllocChunks * kNoAllocMaxExperts + 2 * kNoAllocMaxExperts + 64;
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
  if (T > 0 && (reinterpret_cast<uintptr_t>(ids) & 15u)) return MOE_ERR_INVALID_ARG;
  for (const void* p : {static_cast<const void*>(k), static_cast<const void*>(offsets),
                        static_cast<const void*>(perm), static_cast<const void*>(pair_pos)})
    if (reinterpret_cast<uintptr_t>(p) & 3u) return MOE_ERR_INVALID_ARG;
  int32_t* scratch = nullptr;
  if (noalloc_scratch(&scratch) != cudaSuccess) return MOE_ERR_CUDA;
  // Layout: per-chunk counts [N][chunks] | totals [N] | tile offsets [N+1]. The
  // counts of every chunk in use, the totals and all N+1 tile offsets are
  // rewritten by each call before they are read, so nothing has to be cleared.
  int32_t* cnt = scratch;
  int32_t* totals = scratch + kNoAllocChunks * kNoAllocMaxExperts;
  int32_t* tile_off = totals + kNoAllocMaxExperts;
  return moe::run_dispatch(k, ids, T, N, K, offsets, perm, pair_pos, cnt, totals, tile_off, nullptr,
                           false, nullptr, nullptr, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? MOE_OK
             : MOE_ERR_CUDA;
}
