// Persistent tcgen05 GEMMs with TMA-fed shared-memory pipelines and TMEM
// accumulators, one CTA per tile, for the contractions of the layer (the
// prefill layer's gathered gate/up and down GEMMs use the two-CTA kernels of
// gemm2.cu; kDown here serves d not a multiple of 256):
//
//   kRouter       : logits[T, N] = x[T, d] . W_r[N, d]^T             (fp32 out)
//   kRouterFused  : the same, with the elbow routing of each token run in the
//                   epilogue (one epilogue thread per token row, the logits
//                   staged in shared memory), plus the dispatch's per-chunk
//                   expert counts; the logits need not leave the chip
//   kGateUp       : h[P, I] = silu(xs W_gate[e]^T) * (xs W_up[e]^T), per expert
//                   e over its dispatched rows [offsets[e], offsets[e+1]) (bf16)
//   kDown         : o[P, d] = h W_down[e]^T, per expert                 (bf16 out)
//   kDecGateUp, kDecDown : the same two expert contractions for decode-sized
//                   batches (every expert has at most 64 rows), with the roles
//                   of the operands swapped: A = 128 weight rows (M), B = the
//                   expert's <= 64 token rows (N = 64), so a tile streams
//                   weights instead of padding 128-row token tiles. For
//                   kDecGateUp the A tile is 64 gate rows and the matching 64
//                   up rows; the epilogue pairs them through shared memory.
//
// Both operands are K-major bf16 tiles of 64 columns (128 bytes) moved by TMA
// with 128-byte swizzle; the MMA is tcgen05.mma.cta_group::1.kind::f16 with
// M = 128 and N = BN (64/128 for the router, 256 for the experts), fp32
// accumulation in TMEM. For kGateUp the 256-row B tile is the 128 gate rows
// and the matching 128 up rows of the expert, so one accumulator holds both
// halves of the SwiGLU and the epilogue fuses silu(g) * u.
//
// Warp roles (192 threads, one CTA per SM):
//   warp 0     : TMA producer (one elected lane)
//   warp 1     : TMEM allocator + MMA issuer (one elected lane)
//   warps 2..5 : epilogue; warp w reads TMEM lanes [32 (w % 4), +32)
// Two TMEM accumulators (2 x BN columns) let the epilogue of tile i overlap
// the main loop of tile i + 1. Tiles are scheduled statically
// (tile = blockIdx.x + i * gridDim.x); for the grouped modes a tile index maps
// to (expert, n-block, m-block) through the device-side m-tile prefix sums, so
// the ragged expert sizes never travel to the host. Consecutive tiles share
// an expert's weight block (m-block fastest), which keeps it in L2.
//
// Every barrier wait is bounded (kWaitLimitNs); a timed-out CTA raises a flag
// that stops its other roles, drains what it has in flight, frees its TMEM and
// writes an error code into the caller's error word.
#include "common.cuh"
#include "route_impl.cuh"

namespace moe {
namespace gemm {

constexpr int BM = 128;
constexpr int BK = 64;
// Warps: kProdWarps producers, one MMA warp, four epilogue warps.
template <int MODE>
struct Roles {
  static constexpr int kProdWarps = 1;
  static constexpr int kMmaWarp = kProdWarps;
  static constexpr int kEpiWarp0 = kProdWarps + 1;
  static constexpr int kThreads = 32 * (kProdWarps + 5);
};
enum Mode {
  kRouter = 0,
  kGateUp = 1,
  kDown = 2,
  kRouterFused = 4,
  kDecGateUp = 5,
  kDecDown = 6
};

template <int MODE>
__host__ __device__ constexpr bool is_router() { return MODE == kRouter || MODE == kRouterFused; }
template <int MODE>
__host__ __device__ constexpr bool is_gateup() { return MODE == kGateUp; }
template <int MODE>
__host__ __device__ constexpr bool is_decode() { return MODE == kDecGateUp || MODE == kDecDown; }

// Routing constants for the fused router epilogue (x'_i for i < N, and the
// fast-path bound), in the layout route_token expects.
struct RouteX {
  float x[128];
  float bound;
};

template <int MODE, int BN>
struct Cfg {
  static constexpr int kABytes = BM * BK * 2;
  static constexpr int kBBytes = BN * BK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  // fused routing: logit rows [128][BN + 4] fp32, histogram
  static constexpr int kRouteTileBytes = 128 * (BN + 4) * 4;
  static constexpr int kRouteBytes = MODE == kRouterFused ? kRouteTileBytes + BN * 4 : 0;
  // kDown: per epilogue warp two 32 x 32 bf16 staging tiles for TMA stores;
  // kDecGateUp: the up half of the accumulator, [64 rows][65] fp32
  static constexpr int kEpiBytes =
      MODE == kDown ? 4 * 2 * 32 * 64 : (MODE == kDecGateUp ? 64 * 65 * 4 : 0);
  static constexpr int kStages = (208 * 1024 - kRouteBytes - kEpiBytes) / kStageBytes;
  // TMEM columns per accumulator: at least 32, so that a 32-column load of one
  // accumulator never reaches into the other
  static constexpr int kAccStride = BN < 32 ? 32 : BN;
  static constexpr int kTmemCols = (2 * kAccStride <= 64) ? 64
                                 : (2 * kAccStride <= 128 ? 128 : (2 * kAccStride <= 256 ? 256 : 512));
  static constexpr int kBarOff = kStages * kStageBytes;
  // barriers: full[S], empty[S], tfull[2], tempty[2], drain
  static constexpr int kNumBars = 2 * kStages + 5;
  static constexpr int kMiscOff = kBarOff + kNumBars * 8;
  static constexpr int kTableOff = kMiscOff + 16;
  static constexpr int kMaxGroups = 128;
  static constexpr int kRouteOff = (kTableOff + 2 * (kMaxGroups + 1) * 4 + 15) & ~15;
  static constexpr int kEpiOff = (kRouteOff + kRouteBytes + 127) & ~127;
  static constexpr int kSmemBytes = kEpiOff + kEpiBytes + 1024;  // + align slack
  static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
};

struct Args {
  const int32_t* offsets;   // [G + 1] row offsets per group (grouped modes)
  const int32_t* tile_off;  // [G + 1] prefix sums of ceil(rows_g / 128)
  int groups;               // G
  int64_t m_rows;           // router: T
  int64_t p_rows;           // grouped and decode modes: the row capacity P of the
                            // dispatched operand and the output
  int n_tiles;              // n-blocks per group
  int k_blocks;             // K / 64
  int b_rows;               // rows of B per group (2I for gate/up, d for down)
  int b_half;               // gate/up: I (row offset of the up half)
  void* out;
  int64_t ldo;              // output row stride, elements
  int32_t* err;             // device error word (may be null)
  // kRouterFused
  RouteX rx;
  int K, topk_mode, renorm, nblk;
  float eps;
  int32_t* k_out;
  int32_t* ids_out;
  float* gates_out;
  int32_t* blk_cnt;         // [N][nblk] per-128-token-chunk expert counts (may be null)
};

struct Tile {
  int g, nb, row0, rows;
};

template <int MODE>
MOE_DEV Tile decode(int tile, const Args& a, const int* s_off, const int* s_toff) {
  Tile t;
  if (is_router<MODE>()) {
    t.g = 0;
    t.nb = 0;
    t.row0 = tile * BM;
    t.rows = static_cast<int>(min_of<int64_t>(BM, a.m_rows - t.row0));
    return t;
  }
  if (is_decode<MODE>()) {
    // tile = j * n_tiles + weight-row block, j indexing the experts that have
    // rows (s_toff holds their ids in ascending order); the expert's rows are
    // its B columns
    t.g = s_toff[tile / a.n_tiles];
    t.nb = tile % a.n_tiles;
    t.row0 = s_off[t.g];
    t.rows = s_off[t.g + 1] - t.row0;
    MOE_DCHECK(t.rows >= 0 && t.row0 >= 0 && static_cast<int64_t>(t.row0) + t.rows <= a.p_rows);
    // rows stay inside [0, P) whatever the offsets say
    t.rows = (t.row0 < 0 || t.row0 >= a.p_rows)
                 ? 0
                 : static_cast<int>(min_of<int64_t>(t.rows, a.p_rows - t.row0));
    return t;
  }
  int lo = 0, hi = a.groups;  // s_toff[lo] * n_tiles <= tile < s_toff[hi] * n_tiles
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (s_toff[mid] * a.n_tiles <= tile) lo = mid; else hi = mid;
  }
  const int mt = s_toff[lo + 1] - s_toff[lo];
  const int local = tile - s_toff[lo] * a.n_tiles;
  const int mb = local % mt;
  t.g = lo;
  t.nb = local / mt;
  t.row0 = s_off[lo] + mb * BM;
  t.rows = min(BM, s_off[lo + 1] - t.row0);
  MOE_DCHECK(s_off[lo + 1] >= s_off[lo] && t.row0 >= 0 &&
             static_cast<int64_t>(t.row0) + t.rows <= a.p_rows);
  MOE_DCHECK(mt == (s_off[lo + 1] - s_off[lo] + BM - 1) / BM);
  // rows stay inside [0, P) whatever the offsets say
  t.rows = (t.row0 < 0 || t.row0 >= a.p_rows)
               ? 0
               : static_cast<int>(min_of<int64_t>(t.rows, a.p_rows - t.row0));
  return t;
}

template <int MODE, int BN>
__global__ void __launch_bounds__(Roles<MODE>::kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ CUtensorMap tmC,
                const __grid_constant__ Args args) {
  using C = Cfg<MODE, BN>;
  using R = Roles<MODE>;
  constexpr int kThreads = R::kThreads;
  constexpr int S = C::kStages;
  constexpr uint32_t kIdesc = idesc_bf16_f32(BM, BN);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + C::kBarOff;
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (S + s); };
  auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * S + a); };
  auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * S + 2 + a); };
  const uint32_t drain_bar = bar0 + 8u * (2 * S + 4);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::kMiscOff);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kMiscOff + 4);
  int* s_off = reinterpret_cast<int*>(smem + C::kTableOff);
  int* s_toff = s_off + (C::kMaxGroups + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull_bar(a), 1);
      mbar_init(tempty_bar(a), 4);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&tmA);
    prefetch_tensormap(&tmB);
  }
  // everything above touches no global memory; from here on the preceding
  // kernels' results are read (and TMEM is taken only once they have ended)
  grid_dep_wait();
  grid_dep_launch();
  if (!is_router<MODE>()) {  // grouped schedule tables (router modes have none)
    for (int i = threadIdx.x; i <= args.groups; i += kThreads) {
      s_off[i] = args.offsets[i];
      // the decode modes schedule by expert and need no m-tile prefix sums
      // (their tile_off is null)
      s_toff[i] = is_decode<MODE>() ? 0 : args.tile_off[i];
    }
  }
  if constexpr (is_decode<MODE>()) {
    // the experts with rows, in ascending order, into s_toff[0 ..), their
    // count into s_toff[kMaxGroups]: tiles are numbered over these experts
    // only, so the round-robin over CTAs stays balanced however many are empty
    __syncthreads();
    if (warp == 0) {
      int base = 0;
      for (int e0 = 0; e0 < args.groups; e0 += 32) {
        const int e = e0 + lane;
        const bool used = e < args.groups && s_off[e + 1] > s_off[e];
        const unsigned m = __ballot_sync(0xffffffffu, used);
        if (used) s_toff[base + __popc(m & ((1u << lane) - 1u))] = e;
        base += __popc(m);
      }
      if (lane == 0) s_toff[C::kMaxGroups] = base;
    }
  }
  if (warp == R::kMmaWarp) {
    __syncwarp();
    tmem_alloc<C::kTmemCols>(smem_u32(tmem_slot));
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int total = is_router<MODE>()   ? static_cast<int>((args.m_rows + BM - 1) / BM)
                    : is_decode<MODE>() ? s_toff[C::kMaxGroups] * args.n_tiles
                                        : s_toff[args.groups] * args.n_tiles;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      for (int tile = blockIdx.x; tile < total && !*abort_flag; tile += gridDim.x) {
        const Tile t = decode<MODE>(tile, args, s_off, s_toff);
        if (is_decode<MODE>() && t.rows <= 0) continue;
        for (int kb = 0; kb < args.k_blocks; ++kb) {
          if (!mbar_wait_bounded(empty_bar(stage), phase ^ 1u, abort_flag)) break;
          const uint32_t a_dst = sbase + stage * C::kStageBytes;
          const uint32_t b_dst = a_dst + C::kABytes;
          mbar_arrive_expect_tx(full_bar(stage), C::kStageBytes);
          if (MODE == kDecGateUp) {
            // 64 gate rows, then the matching 64 up rows, of the expert's W_gate/up
            const int arow = t.g * args.b_rows + t.nb * 64;
            tma_load_2d(a_dst, &tmA, full_bar(stage), kb * BK, arow);
            tma_load_2d(a_dst + 64 * BK * 2, &tmA, full_bar(stage), kb * BK, arow + args.b_half);
          } else if (MODE == kDecDown) {
            tma_load_2d(a_dst, &tmA, full_bar(stage), kb * BK, t.g * args.b_rows + t.nb * BM);
          } else {
            tma_load_2d(a_dst, &tmA, full_bar(stage), kb * BK, t.row0);
          }
          if (is_decode<MODE>()) {
            // the expert's token rows (rows past them belong to other experts
            // or lie past the end: their columns are never stored)
            tma_load_2d(b_dst, &tmB, full_bar(stage), kb * BK, t.row0);
          } else if (is_gateup<MODE>()) {
            const int brow = t.g * args.b_rows + t.nb * 128;
            tma_load_2d(b_dst, &tmB, full_bar(stage), kb * BK, brow);
            tma_load_2d(b_dst + 128 * BK * 2, &tmB, full_bar(stage), kb * BK, brow + args.b_half);
          } else {
            tma_load_2d(b_dst, &tmB, full_bar(stage), kb * BK, t.g * args.b_rows + t.nb * BN);
          }
          ++issued;
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (*abort_flag) {
        // let the copies this thread started land before the CTA exits
        int st = stage;
        uint32_t ph = phase;
        const int n = issued < S ? issued : S;
        for (int i = 0; i < n; ++i) {
          if (--st < 0) { st = S - 1; ph ^= 1u; }
          const uint64_t t0 = global_timer_ns();
          while (!mbar_try_wait(full_bar(st), ph) && global_timer_ns() - t0 < 100000000ull) {
          }
        }
      }
    }
  } else if (warp == R::kMmaWarp) {
    // ----------------------------------------------------------------- MMA
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int local = 0;
      bool issued_any = false;
      for (int tile = blockIdx.x; tile < total && !*abort_flag; tile += gridDim.x, ++local) {
        if (is_decode<MODE>() && decode<MODE>(tile, args, s_off, s_toff).rows <= 0) {
          --local;  // an empty expert uses no accumulator (the loop step adds it back)
          continue;
        }
        const int acc = local & 1;
        const uint32_t acc_phase = (local >> 1) & 1;
        if (!mbar_wait_bounded(tempty_bar(acc), acc_phase ^ 1u, abort_flag)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * C::kAccStride;
        bool ok = true;
        for (int kb = 0; kb < args.k_blocks; ++kb) {
          if (!mbar_wait_bounded(full_bar(stage), phase, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a_addr = sbase + stage * C::kStageBytes;
          const uint64_t adesc = smem_desc_sw128(a_addr);
          const uint64_t bdesc = smem_desc_sw128(a_addr + C::kABytes);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            // advance 16 bf16 (32 bytes) along K inside the swizzled rows
            umma_bf16(d_tmem, adesc + 2 * k, bdesc + 2 * k, kIdesc, (kb | k) != 0 ? 1u : 0u);
          }
          issued_any = true;
          umma_commit(empty_bar(stage));
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(tfull_bar(acc));
      }
      if (*abort_flag && issued_any) {
        // wait for the MMAs in flight before TMEM is released
        umma_commit(drain_bar);
        const uint64_t t0 = global_timer_ns();
        while (!mbar_try_wait(drain_bar, 0) && global_timer_ns() - t0 < 100000000ull) {
        }
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;  // the four epilogue warps cover the four TMEM lane quarters
    int epi_buf = 0;         // kDown: which of this warp's two staging tiles is next
    const int r = q * 32 + lane;
    int local = 0;
    for (int tile = blockIdx.x; tile < total; tile += gridDim.x, ++local) {
      const Tile t = decode<MODE>(tile, args, s_off, s_toff);
      if (is_decode<MODE>() && t.rows <= 0) {
        --local;  // as in the MMA loop
        continue;
      }
      const int acc = local & 1;
      const uint32_t acc_phase = (local >> 1) & 1;
      const bool ok = mbar_wait_bounded(tfull_bar(acc), acc_phase, abort_flag);
      if (MODE == kRouterFused || MODE == kDecGateUp) {
        // all four epilogue warps take the same decision (they meet at named
        // barriers below), and each warp reconverges
        if (!epilogue_all(ok)) break;
        __syncwarp();
      } else {
        // all lanes agree (and reconverge) before the warp-collective TMEM loads
        if (!__all_sync(0xffffffffu, ok)) break;
      }
      tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + acc * C::kAccStride;
      const bool valid = r < t.rows;
      const int64_t grow = static_cast<int64_t>(t.row0) + r;
      if (MODE == kRouter) {
        float* out = static_cast<float*>(args.out) + grow * args.ldo;
#pragma unroll
        for (int c = 0; c < BN; c += 32) {
          uint32_t v[32];
          tmem_ld_32x32b_x32(taddr + c, v);
          tmem_ld_wait();
          if (valid) {
            float4* o4 = reinterpret_cast<float4*>(out + c);
#pragma unroll
            for (int u = 0; u < 8; ++u)
              o4[u] = make_float4(__uint_as_float(v[4 * u]), __uint_as_float(v[4 * u + 1]),
                                  __uint_as_float(v[4 * u + 2]), __uint_as_float(v[4 * u + 3]));
          }
        }
      } else if (MODE == kRouterFused) {
        // logits -> this thread's row in shared memory (and to global if asked)
        float* rtile = reinterpret_cast<float*>(smem + C::kRouteOff);
        int* hist = reinterpret_cast<int*>(smem + C::kRouteOff + C::kRouteTileBytes);
        float* row = rtile + r * (BN + 4);
        float* gout = args.out ? static_cast<float*>(args.out) + grow * args.ldo : nullptr;
#pragma unroll
        for (int c = 0; c < BN; c += 32) {
          uint32_t v[32];
          tmem_ld_32x32b_x32(taddr + c, v);
          tmem_ld_wait();
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const float4 f = make_float4(__uint_as_float(v[4 * u]), __uint_as_float(v[4 * u + 1]),
                                         __uint_as_float(v[4 * u + 2]), __uint_as_float(v[4 * u + 3]));
            reinterpret_cast<float4*>(row + c)[u] = f;
            if (valid && gout) reinterpret_cast<float4*>(gout + c)[u] = f;
          }
        }
        // the accumulator is free once read: release it before routing
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(tempty_bar(acc));
        if (args.blk_cnt) {
          for (int e = r; e < BN; e += 128) hist[e] = 0;
          epilogue_sync();
        }
        int ids_sel[8];
        int k_sel = 0;
        float ssum = 0.0f;
        if (valid)
          k_sel = route::route_token<BN, RouteX>(row, grow, args.K, args.eps, args.topk_mode,
                                                 args.renorm, args.rx, args.k_out, args.ids_out,
                                                 args.gates_out, ids_sel, ssum);
        // tokens the fast path left undecided: routed by their whole warp
        const unsigned undecided = __ballot_sync(0xffffffffu, valid && k_sel < 0);
        if constexpr (BN >= 64) if (undecided) {
          const float* wrow = rtile + q * 32 * (BN + 4);
          route::route_undecided<BN>(
              undecided, [&](int l) { return wrow + l * (BN + 4); }, ssum, grow, args.K, args.eps,
              args.topk_mode, args.renorm, args.k_out, args.ids_out, args.gates_out, k_sel,
              ids_sel);
        }
        if (args.blk_cnt) {
#pragma unroll
          for (int s2 = 0; s2 < 8; ++s2)
            if (s2 < k_sel && ids_sel[s2] >= 0 && ids_sel[s2] < BN) atomicAdd(&hist[ids_sel[s2]], 1);
          epilogue_sync();
          for (int e = r; e < BN; e += 128)
            args.blk_cnt[static_cast<int64_t>(e) * args.nblk + tile] = hist[e];
          epilogue_sync();
        }
        continue;
      } else if (is_decode<MODE>()) {
        // TMEM lane r = weight row of the tile, column c = the expert's c-th row
        // (BN = 16, 32 or 64 columns; only columns below the expert's rows are stored)
        static_assert(!is_decode<MODE>() || BN == 16 || BN == 32 || BN == 64, "decode tile width");
        uint32_t v0[32], v1[32];
        tmem_ld_32x32b_x32(taddr, v0);
        if constexpr (BN > 32) tmem_ld_32x32b_x32(taddr + 32, v1);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(tempty_bar(acc));
        const int ncols = min(t.rows, BN);
        __nv_bfloat16* out = static_cast<__nv_bfloat16*>(args.out) +
                             static_cast<int64_t>(t.row0) * args.ldo;
        if (MODE == kDecGateUp) {
          // rows 64..127 hold up(i0 + r - 64): hand them to the warps holding gate(i0 + r)
          float* xch = reinterpret_cast<float*>(smem + C::kEpiOff);
          if (q >= 2) {
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              xch[(r - 64) * 65 + c] = __uint_as_float(v0[c]);
              if constexpr (BN > 32) xch[(r - 64) * 65 + 32 + c] = __uint_as_float(v1[c]);
            }
          }
          epilogue_sync();
          if (q < 2) {
            __nv_bfloat16* o = out + t.nb * 64 + r;
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              if (c < ncols)
                o[c * args.ldo] = __float2bfloat16_rn(silu(__uint_as_float(v0[c])) * xch[r * 65 + c]);
              if constexpr (BN > 32) {
                if (32 + c < ncols)
                  o[(32 + c) * args.ldo] =
                      __float2bfloat16_rn(silu(__uint_as_float(v1[c])) * xch[r * 65 + 32 + c]);
              }
            }
          }
          epilogue_sync();  // the exchange buffer is reused by the next tile
        } else {
          __nv_bfloat16* o = out + t.nb * BM + r;
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            if (c < ncols) o[c * args.ldo] = __float2bfloat16_rn(__uint_as_float(v0[c]));
            if constexpr (BN > 32) {
              if (32 + c < ncols) o[(32 + c) * args.ldo] = __float2bfloat16_rn(__uint_as_float(v1[c]));
            }
          }
        }
        continue;
      } else if (is_gateup<MODE>()) {
        __nv_bfloat16* out = static_cast<__nv_bfloat16*>(args.out) + grow * args.ldo + t.nb * 128;
#pragma unroll 1
        for (int c = 0; c < 128; c += 32) {
          uint32_t gv[32], uv[32];
          tmem_ld_32x32b_x32(taddr + c, gv);
          tmem_ld_32x32b_x32(taddr + 128 + c, uv);
          tmem_ld_wait();
          if (valid) {
            uint4* o4 = reinterpret_cast<uint4*>(out + c);
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              uint32_t w[4];
#pragma unroll
              for (int z = 0; z < 4; ++z) {
                const int i0 = 8 * u + 2 * z;
                w[z] = pack_bf16x2(silu(__uint_as_float(gv[i0])) * __uint_as_float(uv[i0]),
                                   silu(__uint_as_float(gv[i0 + 1])) * __uint_as_float(uv[i0 + 1]));
              }
              o4[u] = make_uint4(w[0], w[1], w[2], w[3]);
            }
          }
        }
      } else {
        // Output rows are written 32 x 32 at a time: when all 32 rows of this
        // warp belong to the tile's expert, through a staging tile in shared
        // memory and a TMA store (coalesced, asynchronous); otherwise (the
        // ragged last tile of an expert) row by row from registers.
        __nv_bfloat16* out = static_cast<__nv_bfloat16*>(args.out) + grow * args.ldo + t.nb * BN;
        const bool full_warp = __all_sync(0xffffffffu, valid);
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          uint32_t v[32];
          tmem_ld_32x32b_x32(taddr + c, v);
          tmem_ld_wait();
          uint4 w4[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            uint32_t w[4];
#pragma unroll
            for (int z = 0; z < 4; ++z) {
              const int i0 = 8 * u + 2 * z;
              w[z] = pack_bf16x2(__uint_as_float(v[i0]), __uint_as_float(v[i0 + 1]));
            }
            w4[u] = make_uint4(w[0], w[1], w[2], w[3]);
          }
          if (MODE == kDown && full_warp) {
            uint8_t* sb = smem + C::kEpiOff + (q * 2 + epi_buf) * 2048;
            // the store issued from this buffer two chunks ago has read it
            if (lane == 0) bulk_wait_read<1>();
            __syncwarp();
#pragma unroll
            for (int u = 0; u < 4; ++u) reinterpret_cast<uint4*>(sb + lane * 64)[u] = w4[u];
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&tmC, smem_u32(sb), t.nb * BN + c, t.row0 + q * 32);
              bulk_commit();
            }
            epi_buf ^= 1;
          } else if (valid) {
            uint4* o4 = reinterpret_cast<uint4*>(out + c);
#pragma unroll
            for (int u = 0; u < 4; ++u) o4[u] = w4[u];
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty_bar(acc));
    }
    if (MODE == kDown && lane == 0) bulk_wait<0>();  // every TMA store has completed
  }

  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag && args.err) atomicExch(args.err, kDevErrTimeout);
  if (warp == R::kMmaWarp) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc<C::kTmemCols>(tmem_base);
  }
}

// ---------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn lookup_encode_fn() {
  void* p = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
          cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    return reinterpret_cast<EncodeTiledFn>(p);
  return nullptr;
}

// The driver's tensor-map encoder, looked up once (a function-local static is
// initialised exactly once even when several host threads call at the same time).
static EncodeTiledFn encode_fn() {
  static const EncodeTiledFn fn = lookup_encode_fn();
  return fn;
}

// 2-D bf16 tensor [outer, inner] (row-major), box [box_outer, 64], 128B swizzle.
bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                     uint32_t box_outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), box_outer};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2-D bf16 tensor [outer, inner], box [box_outer, box_inner], no swizzle.
bool make_map_plain(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                           uint32_t box_inner, uint32_t box_outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int MODE, int BN>
static cudaError_t launch_mode(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                               const Args& args, int grid, cudaStream_t stream) {
  using C = Cfg<MODE, BN>;
  static std::atomic<uint64_t> attr_done{0};
  const cudaError_t e = once_per_device(attr_done, [] {
    return cudaFuncSetAttribute(gemm_kernel<MODE, BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                C::kSmemBytes);
  });
  if (e != cudaSuccess) return e;
  return launch_pdl(gemm_kernel<MODE, BN>, dim3(grid), dim3(Roles<MODE>::kThreads), C::kSmemBytes,
                    stream, a, b, c, args);
}

}  // namespace gemm

MOE_DEBUG_TU(gemm)

// logits[T, N] = x[T, d] W_r[N, d]^T
cudaError_t launch_router_gemm(const uint16_t* x, const uint16_t* wr, int64_t T, int d, int N,
                               float* logits, int32_t* err, int num_sms, cudaStream_t stream) {
  using namespace gemm;
  if (T == 0) return cudaSuccess;
  CUtensorMap ma, mb;
  if (!make_map(&ma, x, d, T, BM) || !make_map(&mb, wr, d, N, N)) return cudaErrorInvalidValue;
  Args a{};
  a.groups = 1;
  a.m_rows = T;
  a.n_tiles = 1;
  a.k_blocks = d / BK;
  a.out = logits;
  a.ldo = N;
  a.err = err;
  const int64_t tiles = (T + BM - 1) / BM;
  const int grid = static_cast<int>(tiles < num_sms ? tiles : num_sms);
  if (N == 64) return launch_mode<kRouter, 64>(ma, mb, ma, a, grid, stream);
  return launch_mode<kRouter, 128>(ma, mb, ma, a, grid, stream);
}

// Router GEMM with the elbow routing in its epilogue: k/ids/gates per token and
// the dispatch's per-chunk expert counts ([N][ceil(T/128)], may be null);
// logits_out may be null.
cudaError_t launch_router_route(const uint16_t* x, const uint16_t* wr, int64_t T, int d, int N,
                                int K, float eps, int topk_mode, int renorm, float* logits_out,
                                int32_t* k_out, int32_t* ids_out, float* gates_out,
                                int32_t* blk_cnt, int32_t* err, int num_sms, cudaStream_t stream) {
  using namespace gemm;
  if (T == 0) return cudaSuccess;
  CUtensorMap ma, mb;
  if (!make_map(&ma, x, d, T, BM) || !make_map(&mb, wr, d, N, N)) return cudaErrorInvalidValue;
  Args a{};
  a.groups = 1;
  a.m_rows = T;
  a.n_tiles = 1;
  a.k_blocks = d / BK;
  a.out = logits_out;
  a.ldo = N;
  a.err = err;
  route::fill_route_consts(a.rx, N);
  a.K = K;
  a.eps = eps;
  a.topk_mode = topk_mode;
  a.renorm = renorm;
  a.k_out = k_out;
  a.ids_out = ids_out;
  a.gates_out = gates_out;
  a.blk_cnt = blk_cnt;
  const int64_t tiles = (T + BM - 1) / BM;
  a.nblk = static_cast<int>(tiles);
  const int grid = static_cast<int>(tiles < num_sms ? tiles : num_sms);
  if (N == 64) return launch_mode<kRouterFused, 64>(ma, mb, ma, a, grid, stream);
  return launch_mode<kRouterFused, 128>(ma, mb, ma, a, grid, stream);
}

// h[P, I] = silu(xs W_g^T) * (xs W_u^T) per expert
cudaError_t launch_gateup_gemm(const uint16_t* xs, const uint16_t* wgu, const int32_t* offsets,
                               const int32_t* tile_off, int64_t P, int d, int N, int I, uint16_t* h,
                               int32_t* err, int num_sms, cudaStream_t stream) {
  using namespace gemm;
  if (P == 0) return cudaSuccess;
  CUtensorMap ma, mb;
  if (!make_map(&ma, xs, d, P, BM) ||
      !make_map(&mb, wgu, d, static_cast<uint64_t>(N) * 2 * I, 128))
    return cudaErrorInvalidValue;
  Args a{};
  a.offsets = offsets;
  a.tile_off = tile_off;
  a.groups = N;
  a.p_rows = P;
  a.n_tiles = I / 128;
  a.k_blocks = d / BK;
  a.b_rows = 2 * I;
  a.b_half = I;
  a.out = h;
  a.ldo = I;
  a.err = err;
  return launch_mode<kGateUp, 256>(ma, mb, ma, a, num_sms, stream);
}

// o[P, d] = h W_d[e]^T per expert
cudaError_t launch_down_gemm(const uint16_t* h, const uint16_t* wd, const int32_t* offsets,
                             const int32_t* tile_off, int64_t P, int d, int N, int I, uint16_t* o,
                             int32_t* err, int num_sms, cudaStream_t stream) {
  using namespace gemm;
  if (P == 0) return cudaSuccess;
  // d a multiple of 256: 256-column output tiles; otherwise (d a multiple of
  // 128) 128-column tiles
  const int bn = d % 256 == 0 ? 256 : 128;
  CUtensorMap ma, mb;
  if (!make_map(&ma, h, I, P, BM) ||
      !make_map(&mb, wd, I, static_cast<uint64_t>(N) * d, static_cast<uint32_t>(bn)))
    return cudaErrorInvalidValue;
  Args a{};
  a.offsets = offsets;
  a.tile_off = tile_off;
  a.groups = N;
  a.p_rows = P;
  a.n_tiles = d / bn;
  a.k_blocks = I / BK;
  a.b_rows = d;
  a.out = o;
  a.ldo = d;
  a.err = err;
  CUtensorMap mc;  // o [P, d], boxes of 32 x 32, no swizzle (TMA stores)
  if (!make_map_plain(&mc, o, d, P, 32, 32)) return cudaErrorInvalidValue;
  if (bn == 128) return launch_mode<kDown, 128>(ma, mb, mc, a, num_sms, stream);
  return launch_mode<kDown, 256>(ma, mb, mc, a, num_sms, stream);
}

// Decode-sized batches (every expert has at most 64 rows):
// Width of the decode GEMMs' token operand: an expert of a T-token batch has at
// most T rows, so 16, 32 or 64 columns cover it.
static int decode_width(int64_t max_rows) { return max_rows <= 16 ? 16 : (max_rows <= 32 ? 32 : 64); }

// h[P, I] = silu(xs W_g^T) * (xs W_u^T) per expert, weights as the M operand;
// max_rows (<= 64) bounds the rows of any expert (the batch's token count).
cudaError_t launch_gateup_decode_gemm(const uint16_t* xs, const uint16_t* wgu,
                                      const int32_t* offsets, int64_t P, int64_t max_rows, int d,
                                      int N, int I, uint16_t* h, int32_t* err, int num_sms,
                                      cudaStream_t stream) {
  using namespace gemm;
  if (P == 0) return cudaSuccess;
  if (max_rows > 64) return cudaErrorInvalidValue;
  const int bn = decode_width(max_rows);
  CUtensorMap ma, mb;
  if (!make_map(&ma, wgu, d, static_cast<uint64_t>(N) * 2 * I, 64) ||
      !make_map(&mb, xs, d, P, static_cast<uint32_t>(bn)))
    return cudaErrorInvalidValue;
  Args a{};
  a.offsets = offsets;
  a.groups = N;
  a.p_rows = P;
  a.n_tiles = I / 64;
  a.k_blocks = d / BK;
  a.b_rows = 2 * I;
  a.b_half = I;
  a.out = h;
  a.ldo = I;
  a.err = err;
  const int tiles = N * a.n_tiles;
  const int grid = tiles < num_sms ? tiles : num_sms;
  if (bn == 16) return launch_mode<kDecGateUp, 16>(ma, mb, ma, a, grid, stream);
  if (bn == 32) return launch_mode<kDecGateUp, 32>(ma, mb, ma, a, grid, stream);
  return launch_mode<kDecGateUp, 64>(ma, mb, ma, a, grid, stream);
}

// o[P, d] = h W_d[e]^T per expert, weights as the M operand; max_rows as above
cudaError_t launch_down_decode_gemm(const uint16_t* h, const uint16_t* wd, const int32_t* offsets,
                                    int64_t P, int64_t max_rows, int d, int N, int I, uint16_t* o,
                                    int32_t* err, int num_sms, cudaStream_t stream) {
  using namespace gemm;
  if (P == 0) return cudaSuccess;
  if (max_rows > 64) return cudaErrorInvalidValue;
  const int bn = decode_width(max_rows);
  CUtensorMap ma, mb;
  if (!make_map(&ma, wd, I, static_cast<uint64_t>(N) * d, BM) ||
      !make_map(&mb, h, I, P, static_cast<uint32_t>(bn)))
    return cudaErrorInvalidValue;
  Args a{};
  a.offsets = offsets;
  a.groups = N;
  a.p_rows = P;
  a.n_tiles = d / BM;
  a.k_blocks = I / BK;
  a.b_rows = d;
  a.out = o;
  a.ldo = d;
  a.err = err;
  const int tiles = N * a.n_tiles;
  const int grid = tiles < num_sms ? tiles : num_sms;
  if (bn == 16) return launch_mode<kDecDown, 16>(ma, mb, ma, a, grid, stream);
  if (bn == 32) return launch_mode<kDecDown, 32>(ma, mb, ma, a, grid, stream);
  return launch_mode<kDecDown, 64>(ma, mb, ma, a, grid, stream);
}

}  // namespace moe
