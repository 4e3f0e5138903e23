// Two-CTA grouped expert GEMMs (tcgen05.mma.cta_group::2, M = 256) for the
// prefill layer's two expert contractions (the expert MLP of App. A.4):
//
//   kGateUpGather : h[P, I] = silu(x[perm] W_gate[e]^T) * (x[perm] W_up[e]^T)
//                   per expert e over its dispatched rows, the rows gathered
//                   from x by the dispatch permutation (cp.async)
//   kDown         : o[P, d] = h W_down[e]^T per expert
//
// A cluster of two CTAs (on two SMs) computes one 256 x 256 output tile: CTA r
// holds rows 128 r .. 128 r + 127 of the tile's A operand and half of its B
// operand (gate/up: CTA 0 the 128 gate rows, CTA 1 the matching 128 up rows;
// down: 128 of the 256 W_down rows each), so one pipeline stage is 32 KB per
// CTA instead of the 48 KB of a one-CTA 128 x 256 tile, and the L2 -> SM
// operand traffic per MMA drops by a third. The MMA is issued by one thread of
// CTA 0 (the leader) and reads the A and B halves of both CTAs' shared memory;
// each CTA's TMEM holds its 128 rows x 256 fp32 columns of the accumulator,
// which its own epilogue drains.
//
// Barriers. The TMA copies of both CTAs complete on the leader's `full`
// barrier of the stage (the peer's copies with the .cta_group::2 form, which
// may signal the peer's barrier); the leader's producer expects both CTAs'
// bytes. Gathered rows (cp.async) complete on their own CTA's barrier: in CTA
// 1 a relay thread waits for them, fences the async proxy and arrives on the
// leader's barrier of the same stage. The leader's MMA thread waits there
// (acquire at cluster scope) for everything the stage holds in both CTAs.
// MMA completion is committed to the `empty` barriers of both CTAs (multicast)
// and to both CTAs' `tfull` barriers; both epilogues release an accumulator on
// the leader's `tempty` barrier (the peer's warps remotely). Every wait is
// bounded (kWaitLimitNs): a CTA that gives up raises its abort flag, drains what
// it has in flight and writes the timeout code into the caller's error word.
// Both CTAs meet at a cluster barrier after setting up their barriers and TMEM
// and again before they release TMEM and exit, so neither exits while the other
// (or the MMA) may still touch its shared memory.
//
// Tiles. Per expert, 256-row pair blocks (the prefix sums of ceil(rows / 256)
// are computed in the prologue from the expert offsets), times the n-blocks;
// tile = cluster index + i * number of clusters, m-block fastest within an
// expert so concurrent clusters share the expert's weight block in L2.
#include "common.cuh"

namespace moe {
namespace gemm2 {

constexpr int BM = 128;  // rows of A per CTA (256 per pair)
constexpr int BN = 256;  // output columns per tile
constexpr int BK = 64;   // K per stage (128 bytes of bf16: one swizzle row)
enum Mode { kGateUpGather = 0, kDown = 1 };

template <int MODE>
struct Cfg {
  static constexpr int kProdWarps = MODE == kGateUpGather ? 4 : 1;
  static constexpr int kMmaWarp = kProdWarps;   // MMA issuer (leader), relay (peer)
  static constexpr int kEpiWarp0 = kProdWarps + 1;
  static constexpr int kThreads = 32 * (kProdWarps + 5);
  static constexpr int kABytes = BM * BK * 2;          // this CTA's 128 rows
  static constexpr int kBBytes = (BN / 2) * BK * 2;    // this CTA's half of B
  static constexpr int kStageBytes = kABytes + kBBytes;
  // kDown: per epilogue warp two 32 x 32 bf16 staging tiles for TMA stores
  static constexpr int kEpiBytes = MODE == kDown ? 4 * 2 * 32 * 64 : 0;
  static constexpr int kStages = (208 * 1024 - kEpiBytes) / kStageBytes;
  static constexpr int kTmemCols = 2 * BN;  // two accumulators
  static constexpr int kBarOff = kStages * kStageBytes;
  // barriers: full[S], empty[S], tfull[2], tempty[2], drain
  static constexpr int kNumBars = 2 * kStages + 5;
  static constexpr int kMiscOff = kBarOff + kNumBars * 8;
  static constexpr int kMaxGroups = 128;
  static constexpr int kTableOff = kMiscOff + 16;
  static constexpr int kEpiOff = (kTableOff + 2 * (kMaxGroups + 1) * 4 + 127) & ~127;
  static constexpr int kSmemBytes = kEpiOff + kEpiBytes + 1024;  // + align slack
  static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
};

// ---------------------------------------------------------- cluster helpers
// Arrive once on an mbarrier of the other CTA of the pair (the address from
// map_to_rank). The default semantics of the remote arrive (release at CTA
// scope) are those production two-SM kernels use for cross-CTA arrivals: a
// release at cluster scope here costs about a microsecond per arrival, which
// measured as a 2x slower GEMM. What the arrival publishes is data already
// complete in the arriving CTA's shared memory (its barrier phase was
// observed first) or TMEM reads already waited for (tcgen05.wait::ld and
// tcgen05.fence::before_thread_sync).
MOE_DEV void mbar_arrive_remote(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// TMA load into this CTA's shared memory whose completion (transaction bytes)
// is signalled on an mbarrier of either CTA of the pair (cluster address).
MOE_DEV void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, uint32_t bar_cluster, int c0,
                              int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(c0), "r"(c1)
      : "memory");
}

MOE_DEV bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// mbar_wait_bounded with acquire at cluster scope (for arrivals of the peer CTA).
MOE_DEV bool mbar_wait_cluster_bounded(uint32_t bar, uint32_t parity, volatile int* abort) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  uint32_t spins = 0;
  while (true) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if (++spins % 64u == 0u) {
      if (*abort) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        *abort = 1;
        return false;
      }
    }
  }
}


// ------------------------------------------------------------ tcgen05, pair
// TMEM allocation of the pair: one warp of each CTA, the same columns in both.
template <int kCols>
MOE_DEV void tmem_alloc_pair(uint32_t dst_smem) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "n"(kCols)
               : "memory");
}
MOE_DEV void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
template <int kCols>
MOE_DEV void tmem_dealloc_pair(uint32_t taddr) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "n"(kCols)
               : "memory");
}

// D[tmem of both CTAs] (+)= A[smem of both CTAs] * B[smem of both CTAs]^T,
// M = 256 (128 rows per CTA), bf16 inputs, fp32 accumulation.
MOE_DEV void umma_pair_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on the mbarrier at local offset `bar` in every CTA of the pair
// when the MMAs this thread issued so far have completed.
MOE_DEV void umma_commit_pair_both(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(bar),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}

// The same, on this CTA's barrier only.
MOE_DEV void umma_commit_pair_self(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   bar)
               : "memory");
}

struct Args {
  const int32_t* offsets;  // [G + 1] row offsets per expert
  int groups;              // G
  int64_t p_rows;          // row capacity P of the dispatched operand and the output
  int n_tiles;             // n-blocks per expert (gate/up: I / 128; down: d / 256)
  int k_blocks;            // K / 64
  int b_rows;              // rows of B per expert (2I for gate/up, d for down)
  int b_half;              // gate/up: I (row offset of the up half)
  void* out;
  int64_t ldo;             // output row stride, elements
  int32_t* err;            // device error word (may be null)
  const int32_t* perm;     // kGateUpGather: token of each dispatched row
  const void* a_src;       // kGateUpGather: x [m_rows, lda] bf16
  int64_t lda;
  int64_t m_rows;          // kGateUpGather: rows of x (tokens clamped into it)
};

struct Tile {
  int g, nb, row0, rows;  // expert, n-block, this CTA's first row and row count
};

// Pair tile -> (expert, n-block, rows of CTA `rank`): s_tp holds the prefix
// sums of ceil(rows_e / 256). The second CTA of an expert's last pair block
// may get no rows (its results are computed and never stored).
MOE_DEV Tile decode_pair(int tile, const Args& a, const int* s_off, const int* s_tp, uint32_t rank) {
  int lo = 0, hi = a.groups;  // s_tp[lo] * n_tiles <= tile < s_tp[hi] * n_tiles
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (s_tp[mid] * a.n_tiles <= tile) lo = mid; else hi = mid;
  }
  const int mt = s_tp[lo + 1] - s_tp[lo];
  const int local = tile - s_tp[lo] * a.n_tiles;
  Tile t;
  t.g = lo;
  t.nb = local / mt;
  t.row0 = s_off[lo] + (local % mt) * (2 * BM) + static_cast<int>(rank) * BM;
  const int rows = min(BM, s_off[lo + 1] - t.row0);
  MOE_DCHECK(s_off[lo + 1] >= s_off[lo] && s_off[lo] >= 0 && s_off[lo + 1] <= a.p_rows);
  // rows stay inside [0, P) whatever the offsets say
  t.rows = (rows <= 0 || t.row0 < 0 || t.row0 >= a.p_rows)
               ? 0
               : static_cast<int>(min_of<int64_t>(rows, a.p_rows - t.row0));
  return t;
}

template <int MODE>
__global__ void __launch_bounds__(Cfg<MODE>::kThreads, 1)
    gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     const __grid_constant__ CUtensorMap tmC, const __grid_constant__ Args args) {
  using C = Cfg<MODE>;
  constexpr int S = C::kStages;
  constexpr uint32_t kIdesc = idesc_bf16_f32(2 * BM, BN);
  constexpr bool kGather = MODE == kGateUpGather;

  extern __shared__ uint8_t smem_raw[];
  // the same offsets in both CTAs: the MMA reads both at the leader's addresses
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + C::kBarOff;
  auto full_bar = [&](int st) { return bar0 + 8u * st; };
  auto empty_bar = [&](int st) { return bar0 + 8u * (S + st); };
  auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * S + a); };
  auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * S + 2 + a); };
  const uint32_t drain_bar = bar0 + 8u * (2 * S + 4);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::kMiscOff);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kMiscOff + 4);
  int* s_off = reinterpret_cast<int*>(smem + C::kTableOff);
  int* s_tp = s_off + (C::kMaxGroups + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;

  if (threadIdx.x == 0) {
    // The leader's full barrier of a stage completes when the TMA bytes of both
    // CTAs have landed (its producer's expect-tx arrival counts them; the peer's
    // copies complete on it directly) and, for gathered rows, when its own 128
    // producer lanes' copies have landed and the peer's relay has arrived. The
    // peer's own full barrier counts only its gathered rows (for the relay).
    const uint32_t full_count = leader ? (kGather ? 2 + 32 * C::kProdWarps : 1)
                                       : (kGather ? 32 * C::kProdWarps : 1);
    for (int st = 0; st < S; ++st) {
      mbar_init(full_bar(st), full_count);
      mbar_init(empty_bar(st), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull_bar(a), 1);
      mbar_init(tempty_bar(a), 8);  // four epilogue warps of each CTA (leader's barrier)
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&tmA);
    prefetch_tensormap(&tmB);
  }
  // everything above touches no global memory
  grid_dep_wait();
  grid_dep_launch();
  for (int i = threadIdx.x; i <= args.groups; i += C::kThreads) s_off[i] = args.offsets[i];
  __syncthreads();
  if (warp == 0) {
    // prefix sums of the experts' 256-row pair blocks
    int carry = 0;
    for (int e0 = 0; e0 < args.groups; e0 += 32) {
      const int e = e0 + lane;
      const int c = e < args.groups ? max(s_off[e + 1] - s_off[e], 0) : 0;
      const int nblk = (c + 2 * BM - 1) / (2 * BM);
      int x = nblk;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      if (e < args.groups) s_tp[e] = carry + x - nblk;
      carry += __shfl_sync(0xffffffffu, x, 31);
    }
    if (lane == 0) s_tp[args.groups] = carry;
  }
  if (warp == C::kMmaWarp) {
    __syncwarp();
    tmem_alloc_pair<C::kTmemCols>(smem_u32(tmem_slot));
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers and TMEM are set up
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int total = s_tp[args.groups] * args.n_tiles;
  const int cluster = static_cast<int>(blockIdx.x >> 1);
  const int nclusters = static_cast<int>(gridDim.x >> 1);

  if (kGather && warp < C::kProdWarps) {
    // ------------------------------------- producers: gathered A rows + B
    // A: cp.async, 16 bytes per lane, straight into the 128B-swizzled K-major
    // layout (chunk c of row r at r * 128 + ((c ^ (r & 7)) << 4)); producer
    // warp w owns rows 32w .. 32w + 31, four full 128-byte lines per copy;
    // each lane arms an arrival on the stage's full barrier that fires when its
    // copies have landed. Lane 0 of warp 0 brings this CTA's half of B by TMA.
    const __nv_bfloat16* xg = static_cast<const __nv_bfloat16*>(args.a_src);
    const int chunk = lane & 7;
    int stage = 0;
    uint32_t phase = 0;
    for (int tile = cluster; tile < total && !*abort_flag; tile += nclusters) {
      const Tile t = decode_pair(tile, args, s_off, s_tp, rank);
      int64_t roff[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int r = 32 * warp + 4 * i + (lane >> 3);
        // rows past the expert's end (never stored) repeat its first token; a
        // CTA without rows reads token 0
        int tok = t.rows > 0 ? args.perm[t.row0 + (r < t.rows ? r : 0)] : 0;
        MOE_DCHECK(tok >= 0 && tok < args.m_rows);
        tok = min(max(tok, 0), static_cast<int>(args.m_rows - 1));
        roff[i] = static_cast<int64_t>(tok) * args.lda + chunk * 8;
      }
      bool ok_tile = true;
      for (int kb = 0; kb < args.k_blocks; ++kb) {
        int ok = 1;
        if (lane == 0) ok = mbar_wait_cluster_bounded(empty_bar(stage), phase ^ 1u, abort_flag) ? 1 : 0;
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) {
          ok_tile = false;
          break;
        }
        const uint32_t a_dst = sbase + stage * C::kStageBytes;
        const uint32_t b_dst = a_dst + C::kABytes;
        if (warp == 0 && lane == 0) {
          // CTA 0: the 128 gate rows of the n-block; CTA 1: the matching up
          // rows, whose bytes complete on the leader's barrier
          const int brow = t.g * args.b_rows + (leader ? 0 : args.b_half) + t.nb * (BN / 2);
          if (leader) {
            mbar_arrive_expect_tx(full_bar(stage), 2 * C::kBBytes);
            tma_load_2d(b_dst, &tmB, full_bar(stage), kb * BK, brow);
          } else {
            tma_load_2d_pair(b_dst, &tmB, map_to_rank(full_bar(stage), 0), kb * BK, brow);
          }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int r = 32 * warp + 4 * i + (lane >> 3);
          const uint32_t dst = a_dst + r * 128 + ((chunk ^ (r & 7)) << 4);
          cp_async_16(dst, xg + roff[i] + kb * BK);
        }
        cp_async_arrive_noinc(full_bar(stage));
        if (++stage == S) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok_tile) break;
    }
    cp_async_wait_group<0>();  // nothing of this thread in flight at exit
  } else if (!kGather && warp == 0) {
    // ------------------------------------------- producer: A and B by TMA
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      for (int tile = cluster; tile < total && !*abort_flag; tile += nclusters) {
        const Tile t = decode_pair(tile, args, s_off, s_tp, rank);
        for (int kb = 0; kb < args.k_blocks; ++kb) {
          if (!mbar_wait_cluster_bounded(empty_bar(stage), phase ^ 1u, abort_flag)) break;
          const uint32_t a_dst = sbase + stage * C::kStageBytes;
          const uint32_t b_dst = a_dst + C::kABytes;
          // rows past P (a CTA without rows) are zero-filled by the copy; both
          // CTAs' copies complete on the leader's barrier
          const int brow = t.g * args.b_rows + t.nb * BN + static_cast<int>(rank) * (BN / 2);
          if (leader) {
            mbar_arrive_expect_tx(full_bar(stage), 2 * C::kStageBytes);
            tma_load_2d(a_dst, &tmA, full_bar(stage), kb * BK, t.row0);
            tma_load_2d(b_dst, &tmB, full_bar(stage), kb * BK, brow);
          } else {
            const uint32_t lb = map_to_rank(full_bar(stage), 0);
            tma_load_2d_pair(a_dst, &tmA, lb, kb * BK, t.row0);
            tma_load_2d_pair(b_dst, &tmB, lb, kb * BK, brow);
          }
          ++issued;
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (*abort_flag) {
        // let the copies this thread started land before the CTA exits: the
        // leader waits (bounded) for its stages, which count both CTAs'
        // bytes; the peer, whose copies complete on the leader's barriers,
        // waits a fixed 2 ms (a tile of copies lands in microseconds)
        if (leader) {
          int st = stage;
          uint32_t ph = phase;
          const int n = issued < S ? issued : S;
          for (int i = 0; i < n; ++i) {
            if (--st < 0) {
              st = S - 1;
              ph ^= 1u;
            }
            const uint64_t t0 = global_timer_ns();
            while (!mbar_try_wait(full_bar(st), ph) && global_timer_ns() - t0 < 100000000ull) {
            }
          }
        } else if (issued > 0) {
          const uint64_t t0 = global_timer_ns();
          while (global_timer_ns() - t0 < 2000000ull) {
          }
        }
      }
    }
  } else if (warp == C::kMmaWarp) {
    if (leader && lane == 0) {
      // ------------------------------------------------ MMA (leader CTA)
      int stage = 0;
      uint32_t phase = 0;
      int local = 0;
      bool issued_any = false;
      for (int tile = cluster; tile < total && !*abort_flag; tile += nclusters, ++local) {
        const int acc = local & 1;
        const uint32_t acc_phase = (local >> 1) & 1;
        if (!mbar_wait_cluster_bounded(tempty_bar(acc), acc_phase ^ 1u, abort_flag)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        bool ok = true;
        for (int kb = 0; kb < args.k_blocks; ++kb) {
          // both halves of the stage: this CTA's loads and the peer's relay
          if (!mbar_wait_cluster_bounded(full_bar(stage), phase, abort_flag)) {
            ok = false;
            break;
          }
          // A rows written by cp.async (generic proxy) are read by the tensor core
          if (kGather) fence_proxy_async_smem();
          tc_fence_after();
          const uint32_t a_addr = sbase + stage * C::kStageBytes;
          const uint64_t adesc = smem_desc_sw128(a_addr);
          const uint64_t bdesc = smem_desc_sw128(a_addr + C::kABytes);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            // advance 16 bf16 (32 bytes) along K inside the swizzled rows
            umma_pair_bf16(d_tmem, adesc + 2 * k, bdesc + 2 * k, kIdesc, (kb | k) != 0 ? 1u : 0u);
          }
          issued_any = true;
          umma_commit_pair_both(empty_bar(stage));
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit_pair_both(tfull_bar(acc));
      }
      if (*abort_flag && issued_any) {
        // wait for the MMAs in flight before TMEM is released
        umma_commit_pair_self(drain_bar);
        const uint64_t t0 = global_timer_ns();
        while (!mbar_try_wait(drain_bar, 0) && global_timer_ns() - t0 < 100000000ull) {
        }
      }
    } else if (kGather && !leader && lane == 0) {
      // ------------------------------------------------ relay (peer CTA)
      // each stage's gathered rows of this CTA, once they have landed, count
      // as one arrival on the leader's barrier of the same stage
      int stage = 0;
      uint32_t phase = 0;
      for (int tile = cluster; tile < total && !*abort_flag; tile += nclusters) {
        bool ok = true;
        for (int kb = 0; kb < args.k_blocks; ++kb) {
          if (!mbar_wait_bounded(full_bar(stage), phase, abort_flag)) {
            ok = false;
            break;
          }
          // this CTA's cp.async rows are read by the leader's tensor core
          if (kGather) fence_proxy_async_smem();
          mbar_arrive_remote(map_to_rank(full_bar(stage), 0));
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;  // the four epilogue warps cover the four TMEM lane quarters
    int epi_buf = 0;         // kDown: which of this warp's two staging tiles is next
    const int r = q * 32 + lane;
    int local = 0;
    for (int tile = cluster; tile < total; tile += nclusters, ++local) {
      const Tile t = decode_pair(tile, args, s_off, s_tp, rank);
      const int acc = local & 1;
      const uint32_t acc_phase = (local >> 1) & 1;
      const bool ok = mbar_wait_cluster_bounded(tfull_bar(acc), acc_phase, abort_flag);
      // all lanes agree (and reconverge) before the warp-collective TMEM loads
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + acc * BN;
      const bool valid = r < t.rows;
      const int64_t grow = static_cast<int64_t>(t.row0) + r;
      if constexpr (kGather) {
        // columns [0, 128) gate, [128, 256) up of h's columns nb * 128 ..
        __nv_bfloat16* out =
            static_cast<__nv_bfloat16*>(args.out) + grow * args.ldo + t.nb * (BN / 2);
#pragma unroll 1
        for (int c = 0; c < BN / 2; c += 32) {
          uint32_t gv[32], uv[32];
          tmem_ld_32x32b_x32(taddr + c, gv);
          tmem_ld_32x32b_x32(taddr + BN / 2 + c, uv);
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
        // 32 x 32 output groups: through a staging tile and a TMA store when all
        // 32 rows of this warp belong to the tile's expert, else row by row
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
          if (full_warp) {
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
      // release the accumulator on the leader's barrier
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (leader) mbar_arrive(tempty_bar(acc));
        else mbar_arrive_remote(map_to_rank(tempty_bar(acc), 0));
      }
    }
    if (!kGather && lane == 0) bulk_wait<0>();  // every TMA store has completed
  }

  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag && args.err) atomicExch(args.err, kDevErrTimeout);
  tc_fence_before();
  cluster_sync();  // neither CTA leaves while the pair's MMAs or arrivals may touch it
  if (warp == C::kMmaWarp) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc_pair<C::kTmemCols>(tmem_base);
  }
}
// ---------------------------------------------------------------- host side
template <int MODE>
cudaError_t launch_pair(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                        const Args& args, int num_sms, cudaStream_t stream) {
  using C = Cfg<MODE>;
  static std::atomic<uint64_t> attr_done{0};
  cudaError_t e = once_per_device(attr_done, [] {
    return cudaFuncSetAttribute(gemm_pair_kernel<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                C::kSmemBytes);
  });
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(C::kThreads);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  // persistent grid: as many CTA pairs as can be resident at once (tiles are
  // assigned statically, so every cluster must run from the start), found once
  // per device
  static std::atomic<int> resident[64];
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  int clusters = dev < 64 ? resident[dev].load(std::memory_order_acquire) : 0;
  if (clusters <= 0) {
    cfg.gridDim = dim3(static_cast<unsigned>(num_sms & ~1));
    cfg.numAttrs = 1;
    e = cudaOccupancyMaxActiveClusters(&clusters, gemm_pair_kernel<MODE>, &cfg);
    if (e != cudaSuccess) return e;
    if (clusters <= 0) return cudaErrorInvalidConfiguration;
    if (dev < 64) resident[dev].store(clusters, std::memory_order_release);
  }
  clusters = min(clusters, num_sms / 2);
  cfg.gridDim = dim3(static_cast<unsigned>(2 * clusters));
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, gemm_pair_kernel<MODE>, a, b, c, args);
}

}  // namespace gemm2

namespace gemm {
bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint32_t box_outer);
bool make_map_plain(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                    uint32_t box_inner, uint32_t box_outer);
}  // namespace gemm

MOE_DEBUG_TU(gemm2)

// h[P, I] = silu(x[perm] W_g^T) * (x[perm] W_u^T) per expert, two-CTA tiles;
// I a multiple of 128, d of 64, N <= 128.
cudaError_t launch_gateup_gather_gemm_pair(const uint16_t* x, int64_t T, const int32_t* perm,
                                           const uint16_t* wgu, const int32_t* offsets, int64_t P,
                                           int d, int N, int I, uint16_t* h, int32_t* err,
                                           int num_sms, cudaStream_t stream) {
  using namespace gemm2;
  if (P == 0 || T == 0) return cudaSuccess;
  if (I % 128 != 0 || d % BK != 0 || N > Cfg<kGateUpGather>::kMaxGroups) return cudaErrorInvalidValue;
  CUtensorMap mb;
  if (!gemm::make_map(&mb, wgu, d, static_cast<uint64_t>(N) * 2 * I, BN / 2))
    return cudaErrorInvalidValue;
  Args a{};
  a.offsets = offsets;
  a.groups = N;
  a.p_rows = P;
  a.n_tiles = I / (BN / 2);
  a.k_blocks = d / BK;
  a.b_rows = 2 * I;
  a.b_half = I;
  a.out = h;
  a.ldo = I;
  a.err = err;
  a.perm = perm;
  a.a_src = x;
  a.lda = d;
  a.m_rows = T;
  return launch_pair<kGateUpGather>(mb, mb, mb, a, num_sms, stream);
}

// o[P, d] = h W_d[e]^T per expert, two-CTA tiles; d a multiple of 256, I of
// 64, N <= 128.
cudaError_t launch_down_gemm_pair(const uint16_t* h, const uint16_t* wd, const int32_t* offsets,
                                  int64_t P, int d, int N, int I, uint16_t* o, int32_t* err,
                                  int num_sms, cudaStream_t stream) {
  using namespace gemm2;
  if (P == 0) return cudaSuccess;
  if (d % BN != 0 || I % BK != 0 || N > Cfg<kDown>::kMaxGroups) return cudaErrorInvalidValue;
  CUtensorMap ma, mb, mc;
  if (!gemm::make_map(&ma, h, I, P, BM) ||
      !gemm::make_map(&mb, wd, I, static_cast<uint64_t>(N) * d, BN / 2) ||
      !gemm::make_map_plain(&mc, o, d, P, 32, 32))
    return cudaErrorInvalidValue;
  Args a{};
  a.offsets = offsets;
  a.groups = N;
  a.p_rows = P;
  a.n_tiles = d / BN;
  a.k_blocks = I / BK;
  a.b_rows = d;
  a.out = o;
  a.ldo = d;
  a.err = err;
  return launch_pair<kDown>(ma, mb, mc, a, num_sms, stream);
}

}  // namespace moe
