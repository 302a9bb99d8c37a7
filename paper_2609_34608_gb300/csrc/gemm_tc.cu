// Dense projections of the DiT block on the fifth-generation tensor cores (sm_103a).
//
// C[M,N] = A[M,K] . Wt[N,K]^T with bf16 operands and an fp32 accumulator held in TMEM, and the
// block's elementwise tail fused into the accumulator read-back (bias, GELU, adaLN-gated
// residual).  Persistent, warp-specialised CTAs:
//   warp 0      TMA producer: a stage holds KA K-atoms (64 bf16 = one 128-byte swizzle row each)
//               of the 128-row A tile and the BN-row B tile, each operand fetched by 3-D boxes
//               {64, rows, KA}; with KA = 2 one request moves 32 KB.  The single producer
//               thread's round trip per stage (barrier wait, expect-tx, copy issue) rather than
//               bandwidth bounds small projections, so fewer, larger requests are faster
//   warp 1      MMA issuer: one thread issues tcgen05.mma (M=128, N=BN for one-atom stages, else
//               N=min(BN,128), K=16) and commits
//               smem-slot / accumulator-ready mbarriers; also owns the TMEM allocation
//   warps 2..5  epilogue: tcgen05.ld 32x32b per TMEM lane quarter (one row per lane), fused
//               tail, then each warp's 32 x 32 block goes through a swizzled shared-memory
//               transpose so that 8 (fp32) or 4 (bf16) lanes store each 32-column row segment.
//               What the tail reads besides the accumulator (bias, the gate row, the residual)
//               is fetched while the main loop still runs.
// The accumulator is double buffered in TMEM (2 x BN columns) so the epilogue of one tile
// overlaps the main loop of the next.
//
// CTA pairs (CG = 2, no K split; chosen by the shape rule from four waves of tiles on): a cluster
// of two CTAs computes a 256-row x BN unit with one tcgen05.mma.cta_group::2 per K step, M = 256.
// Each CTA loads its 128 rows of A and BN / 2 rows of the weight tile to the same shared-memory
// offsets, and both CTAs' copies signal the first CTA's full barrier (TMA .cta_group::2), which
// that CTA arms with the bytes of both.  Only the first CTA issues MMAs; its commits arrive on
// both CTAs' stage and accumulator barriers by multicast.  Each CTA's epilogue reads its own
// 128 x BN accumulator, and the second CTA releases it to the MMA thread by a remote arrival.
// Per output tile an SM thus receives half the weight rows of a single-CTA tile.  The TMEM
// allocation is collective over the pair.
//
// Clusters of two (MC = 2, no K split; explicit plans only): the two CTAs of a cluster take the
// same 128-row block and adjacent column tiles, so they read the same A tile.  Each loads one
// 64-row half of it with TMA multicast into both CTAs' shared memory (the L2 serves A once per
// pair); a stage is refilled only after both CTAs' MMAs consumed it (their commits arrive on both
// CTAs' empty barriers).
//
// K split: a projection with too few output tiles to fill the GPU is cut into `splits` work units
// per tile, each over a contiguous range of K.  A unit's epilogue stores its fp32 partial tile to
// a workspace and takes a ticket from the tile's counter; the unit that takes the last ticket
// (no CTA ever waits for another) fetches all partials into its (now idle) stage buffers with
// bulk asynchronous copies, sums them in split order, which makes the result independent of
// which unit finishes last, applies the fused tail and resets the counter.  Splitting is only
// planned in one wave (one unit per CTA) and when the partials fit the stage buffers.  Every mbarrier wait is bounded (%globaltimer); on
// timeout the CTA raises an abort flag, sets the context's device error word, drains what it
// issued and frees TMEM before returning.
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "gemm_epilogue.cuh"
#include "tcgen05.cuh"

namespace wam {
namespace {

// ---- cluster helpers ----
WAM_DEV uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
WAM_DEV void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// 2-D TMA load delivered to the same shared-memory offset (and mbarrier offset) of every CTA in
// cta_mask.
WAM_DEV void tma_load_2d_mc(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar, uint16_t cta_mask) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.multicast::cluster"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "h"(cta_mask)
      : "memory");
}
// Arrive on the mbarrier at this offset in every CTA of cta_mask once this thread's MMAs completed.
WAM_DEV void umma_commit_mc(uint32_t bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
      "h"(cta_mask)
      : "memory");
}

// ---- two-SM (CTA pair) MMA helpers ----
// The shared::cluster address of offset `saddr` in the shared memory of cluster CTA `rank`.
WAM_DEV uint32_t cluster_addr(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
// TMA loads into this CTA's shared memory whose completion is signalled on an mbarrier of either
// CTA of the pair (`bar`: a shared::cluster address), so the pair's first CTA sees both halves.
WAM_DEV void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
WAM_DEV void tma_load_3d_pair(uint32_t dst, const CUtensorMap* map, int x, int y, int z, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar)
      : "memory");
}
// One MMA of the pair, issued by its first CTA: D is 256 x N, rows 0..127 in the first CTA's TMEM
// and rows 128..255 in the second's (same TMEM address); A rows 0..127 / 128..255 and B columns
// 0..N/2-1 / N/2..N-1 are read at the same shared-memory offsets of the first / second CTA.
WAM_DEV void umma_bf16_pair(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
// Arrive on the mbarrier at offset `bar` of every CTA in cta_mask once the pair's MMAs issued by
// this thread completed.
WAM_DEV void umma_commit_pair_mc(uint32_t bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
      "h"(cta_mask)
      : "memory");
}
WAM_DEV void umma_commit_pair(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
// Arrive (release, cluster scope) on an mbarrier given by its shared::cluster address.
WAM_DEV void mbar_arrive_cluster(uint32_t cbar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cbar) : "memory");
}
// Bounded wait (as mbar_wait) with cluster-scope acquire: for barriers the peer CTA arrives on.
WAM_DEV bool mbar_wait_cluster(uint32_t bar, uint32_t parity, volatile int* abort_flag, int* dev_err) {
  auto try_wait = [&]() -> bool {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
  };
  if (try_wait()) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (try_wait()) return true;
    if ((i & 63u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer_ns() - t0 > kWaitLimitNs) {
        *abort_flag = 1;
        if (dev_err != nullptr) atomicOr(dev_err, kDevErrTimeout);
        return false;
      }
    }
  }
}

constexpr int kBM = 128;
constexpr int kBK = 64;           // 64 bf16 = 128 bytes = one swizzle row
constexpr int kThreads = 192;
constexpr int kTileBytesA = kBM * kBK * 2;  // 16 KB
constexpr int kBoxRows = 128;               // TMA box rows of the A operand and wide B tiles

// CG = 2: a CTA pair runs one 256-row MMA (tcgen05 cta_group::2); each CTA holds 128 rows of A,
// BN / 2 rows of B and its 128 rows x BN columns of the accumulator.
template <int BN, int KA, int CG = 1>
struct TileCfg {
  static constexpr int kBRows = BN / CG;                        // B rows this CTA loads
  static constexpr int kBoxB = kBRows < kBoxRows ? kBRows : kBoxRows;  // rows per B request
  // One atom per stage: the B boxes lie back to back, so one MMA spans all BN columns.  Two atoms:
  // each box holds both atoms of its rows ([atom][rows]), so each box gets its own MMA.  A pair's
  // B half is one box, and one MMA spans both halves.
  static constexpr int kMmaN = (KA == 1 || CG == 2) ? BN : kBoxB;
  static constexpr int kBytesA = KA * kTileBytesA;              // [KA atoms][128 rows][128 B]
  static constexpr int kBoxBytesB = KA * kBoxB * kBK * 2;       // [KA atoms][kBoxB rows][128 B]
  static constexpr int kStageBytes = kBytesA + (kBRows / kBoxB) * kBoxBytesB;
  static_assert(CG == 1 || (CG == 2 && kBRows == kBoxB && BN <= 256), "a pair's B half is one box");
  static constexpr int kStages = (192 * 1024) / kStageBytes;    // 2 .. 8
  static constexpr int kTmemCols = 2 * BN;
  static constexpr int kBarrierBytes = 256;
  // the epilogue's staged bias and gate row of a tile, one copy per TMEM accumulator, and each
  // epilogue warp's 32 x 32 fp32 block for the transpose ahead of the coalesced stores
  static constexpr int kEpiStageBytes = 2 * 2 * BN * 4;
  static constexpr int kEpiScratchBytes = 4 * 4096;
  static constexpr int kSmemBytes = kStages * kStageBytes + kBarrierBytes + kEpiStageBytes + kEpiScratchBytes + 1024;
  static_assert(kStages >= 2 && kStages <= 8, "stage count");
  static_assert((2 * kStages + 7) * 8 + 12 <= kBarrierBytes, "barrier block");
};

struct SplitArgs {
  int splits;       // K ranges per output tile (1 = no split)
  float* ws;        // [tiles][splits][BN / 4][kBM][4] fp32 partials
  int* counters;    // [tiles] tickets, zero between launches
};

template <int BN, int EPI, int KA, int MC, int CG = 1>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   int M, int N, int K, EpiArgs e, SplitArgs sp, int* dev_err) {
  using C = TileCfg<BN, KA, CG>;
  static_assert(MC == 1 || MC == 2, "cluster size");
  static_assert(CG == 1 || (CG == 2 && MC == 1), "CTA-pair MMAs do not combine with multicast clusters");
  constexpr bool kPair = CG == 2;
  constexpr int kRowsPerUnit = kBM * CG;   // output rows of a work unit
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* tiles = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::kStages * C::kStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + C::kStages;
  uint64_t* tfull = bars + 2 * C::kStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* epbar = drain + 1;   // the 128 epilogue threads, once per split-K hand-off
  uint64_t* rbar = epbar + 1;    // bulk copies of a tile's partials landed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(rbar + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* last_flag = abort_flag + 1;
  float* epi_stage = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + C::kBarrierBytes);
  uint8_t* epi_scratch = reinterpret_cast<uint8_t*>(epi_stage) + C::kEpiStageBytes;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int num_m = (M + kRowsPerUnit - 1) / kRowsPerUnit;
  const int num_n = N / BN;
  const int num_mn = num_m * num_n;
  const int splits = sp.splits;
  const int num_k = K / (kBK * KA) / splits;   // stages per work unit
  // With clusters a unit is a pair of adjacent column tiles of one row block, one per CTA; the
  // cluster walks the units (first = cluster index, stride = clusters), both CTAs in lockstep.
  // With CTA pairs (CG = 2) a unit is a 256-row x BN tile: this CTA holds its rows
  // [128 rank, 128 rank + 128) and loads B rows [rank BN/2, (rank + 1) BN/2) of the column tile;
  // the pair walks the units in lockstep like a cluster.
  const int rank = (MC == 2 || kPair) ? static_cast<int>(cluster_rank()) : 0;
  const int num_units = MC == 2 ? num_mn / 2 : num_mn * splits;
  const int unit0 = (MC == 2 || kPair) ? static_cast<int>(blockIdx.x) / 2 : static_cast<int>(blockIdx.x);
  const int unit_stride = (MC == 2 || kPair) ? static_cast<int>(gridDim.x) / 2 : static_cast<int>(gridDim.x);
  const bool leader = !kPair || rank == 0;   // the CTA that issues a pair's MMAs
  const int b_row_off = kPair ? rank * C::kBRows : 0;
  // first output (and A) row of unit tile row mt held by this CTA
  auto tile_row = [&](int mt) { return mt * kRowsPerUnit + (kPair ? rank * kBM : 0); };
  // unit u: output tile mn = u % num_mn, K range u / num_mn.  Column tiles vary fastest, so the
  // CTAs running at the same time share A row blocks (each read from DRAM about once) while the
  // weight matrix, a few MB, stays in L2; with rows fastest a tall activation operand was
  // streamed from DRAM once per column tile.
  auto unit_mt = [&](int u) { return MC == 2 ? u / (num_n / 2) : (u % num_mn) / num_n; };
  auto unit_nt = [&](int u) { return MC == 2 ? 2 * (u % (num_n / 2)) + rank : (u % num_mn) % num_n; };
  auto unit_kb0 = [&](int u) { return MC == 2 ? 0 : (u / num_mn) * num_k; };
  // A tile of a stage: one request per operand (MC = 1), or this CTA's 64-row half of each K-atom
  // multicast to both CTAs (the other half arrives from the peer)
  auto load_a = [&](uint32_t dst, const CUtensorMap* map, int row, int atom, uint32_t bar) {
    if constexpr (kPair) {
      if constexpr (KA == 1)
        tma_load_2d_pair(dst, map, atom * kBK, row, bar);
      else
        tma_load_3d_pair(dst, map, 0, row, atom, bar);
    } else if constexpr (MC == 1) {
      if constexpr (KA == 1)
        tma_load_2d(dst, map, atom * kBK, row, bar);
      else
        tma_load_3d(dst, map, 0, row, atom, bar);
    } else {
#pragma unroll
      for (int a = 0; a < KA; ++a)
        tma_load_2d_mc(dst + a * kTileBytesA + rank * (kTileBytesA / 2), map, (atom + a) * kBK, row + rank * 64, bar,
                       0x3);
    }
  };
  // K-atoms [atom, atom + KA) of rows [row, row + box): one 2-D box {64, rows} for one atom, one
  // 3-D box {64, rows, 2} for two
  auto load_k = [&](uint32_t dst, const CUtensorMap* map, int row, int atom, uint32_t bar) {
    if constexpr (kPair) {
      if constexpr (KA == 1)
        tma_load_2d_pair(dst, map, atom * kBK, row, bar);
      else
        tma_load_3d_pair(dst, map, 0, row, atom, bar);
    } else if constexpr (KA == 1) {
      tma_load_2d(dst, map, atom * kBK, row, bar);
    } else {
      tma_load_3d(dst, map, 0, row, atom, bar);
    }
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), MC);   // with clusters: both CTAs' MMAs release the stage
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), 128 * CG);   // pairs: both CTAs' epilogue threads
    }
    mbar_init(smem_u32(drain), 1);
    mbar_init(smem_u32(epbar), 128);
    mbar_init(smem_u32(rbar), 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    if constexpr (kPair) {
      // one warp of each CTA of the pair allocates the same columns in both CTAs' TMEM
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                       smem_u32(tmem_slot)),
                   "r"(C::kTmemCols)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                       smem_u32(tmem_slot)),
                   "r"(C::kTmemCols)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  // the peer's barriers exist before any multicast or any copy signalling them
  if constexpr (MC == 2 || kPair) cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_launch_dependents();

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer ----------------
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
    // The weight operand does not depend on earlier kernels: its first stages are requested
    // before waiting for them, overlapping the previous kernel's tail.
    const int u0 = unit0;
    const int pre = u0 < num_units ? (num_k < C::kStages ? num_k : C::kStages) : 0;
    // A stage's copies signal its full barrier; with CTA pairs both CTAs' copies signal the first
    // CTA's barrier, whose MMA thread consumes the stage of both, and only that CTA arms it (with
    // the bytes of both CTAs).
    auto full_bar = [&](int st) -> uint32_t {
      return kPair ? cluster_addr(smem_u32(&full[st]), 0) : smem_u32(&full[st]);
    };
    for (int s = 0; s < pre; ++s) {
      const uint32_t fb = full_bar(s);
      const uint32_t b_dst = smem_u32(tiles + s * C::kStageBytes) + C::kBytesA;
      if (leader) mbar_expect_tx(smem_u32(&full[s]), CG * C::kStageBytes);
#pragma unroll
      for (int h = 0; h < C::kBRows / C::kBoxB; ++h)
        load_k(b_dst + h * C::kBoxBytesB, &tmB, unit_nt(u0) * BN + b_row_off + h * C::kBoxB, (unit_kb0(u0) + s) * KA,
               fb);
    }
    pdl_wait();
    int stage = 0;
    uint32_t phase = 0;
    int issued[C::kStages];
    uint32_t issued_phase[C::kStages];
    for (int s = 0; s < C::kStages; ++s) issued[s] = 0, issued_phase[s] = 0;
    bool ok = true;
    bool first = true;
    for (int unit = unit0; ok && unit < num_units; unit += unit_stride) {
      const int mt = unit_mt(unit);
      const int nt = unit_nt(unit);
      const int kb0 = unit_kb0(unit);
      for (int kb = 0; kb < num_k; ++kb) {
        if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1u, abort_flag, dev_err)) {
          ok = false;
          break;
        }
        const uint32_t fb = full_bar(stage);
        const uint32_t a_dst = smem_u32(tiles + stage * C::kStageBytes);
        const uint32_t b_dst = a_dst + C::kBytesA;
        if (!(first && kb < pre)) {
          if (leader) mbar_expect_tx(smem_u32(&full[stage]), CG * C::kStageBytes);
#pragma unroll
          for (int h = 0; h < C::kBRows / C::kBoxB; ++h)
            load_k(b_dst + h * C::kBoxBytesB, &tmB, nt * BN + b_row_off + h * C::kBoxB, (kb0 + kb) * KA, fb);
        }
        load_a(a_dst, &tmA, tile_row(mt), (kb0 + kb) * KA, fb);
        issued[stage] = 1;
        issued_phase[stage] = phase;
        if (++stage == C::kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      first = false;
    }
    if (!ok && !leader) {
      // The second CTA of a pair cannot observe its copies (they signal the first CTA's barriers):
      // give them time to land before the CTA releases its shared memory.
      const uint64_t t0 = globaltimer_ns();
      while (globaltimer_ns() - t0 < 200000ull) {
      }
    } else if (!ok) {
      // Drain: let every copy this thread issued land before the CTA releases its smem.
      for (int s = 0; s < C::kStages; ++s) {
        if (!issued[s]) continue;
        const uint32_t fb = smem_u32(&full[s]);
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(fb, issued_phase[s]) && globaltimer_ns() - t0 < kWaitLimitNs) {
        }
      }
    }
  } else if (warp == 1 && lane == 0 && leader) {
    // ---------------- MMA issuer (with CTA pairs: the first CTA's, for both) ----------------
    pdl_wait();
    const uint32_t idesc = idesc_bf16(kRowsPerUnit, C::kMmaN);
    int stage = 0;
    uint32_t phase = 0;
    int it = 0;
    bool ok = true;
    bool issued_any = false;
    for (int unit = unit0; ok && unit < num_units; unit += unit_stride, ++it) {
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      const bool drained = kPair ? mbar_wait_cluster(smem_u32(&tempty[acc]), acc_phase ^ 1u, abort_flag, dev_err)
                                 : mbar_wait(smem_u32(&tempty[acc]), acc_phase ^ 1u, abort_flag, dev_err);
      if (!drained) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + acc * BN;
      for (int kb = 0; kb < num_k; ++kb) {
        if (!mbar_wait(smem_u32(&full[stage]), phase, abort_flag, dev_err)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = smem_u32(tiles + stage * C::kStageBytes);
        // One descriptor per operand and stage; the address field holds addr >> 4 and shared
        // memory stays below 256 KB, so an offset is one add of (offset >> 4).
        const uint64_t da = sw128_desc(a0), db = sw128_desc(a0 + C::kBytesA);
#pragma unroll
        for (int a = 0; a < KA; ++a) {
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
#pragma unroll
            for (int h = 0; h < BN / C::kMmaN; ++h) {
              if constexpr (kPair)
                umma_bf16_pair(d_tmem, da + ((a * kTileBytesA + k * 32) >> 4), db + ((a * C::kBoxB * 128 + k * 32) >> 4),
                               idesc, (kb | a | k) != 0 ? 1u : 0u);
              else
                umma_bf16(d_tmem + h * C::kMmaN, da + ((a * kTileBytesA + k * 32) >> 4),
                          db + ((h * C::kBoxBytesB + a * C::kBoxB * 128 + k * 32) >> 4), idesc,
                          (kb | a | k) != 0 ? 1u : 0u);
            }
          }
        }
        issued_any = true;
        if constexpr (kPair)
          umma_commit_pair_mc(smem_u32(&empty[stage]), 0x3);   // both CTAs' stage buffers are free
        else if constexpr (MC == 2)
          umma_commit_mc(smem_u32(&empty[stage]), 0x3);
        else
          umma_commit(smem_u32(&empty[stage]));
        if (++stage == C::kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) break;
      if constexpr (kPair)
        umma_commit_pair_mc(smem_u32(&tfull[acc]), 0x3);   // both CTAs' halves of the accumulator
      else
        umma_commit(smem_u32(&tfull[acc]));
    }
    if (!ok && issued_any) {
      // Drain: wait for every MMA this thread issued before TMEM is released.
      if constexpr (kPair)
        umma_commit_pair(smem_u32(drain));
      else
        umma_commit(smem_u32(drain));
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(smem_u32(drain), 0) && globaltimer_ns() - t0 < kWaitLimitNs) {
      }
    }
  } else if (warp >= 2) {
    // ---------------- epilogue ----------------
    pdl_wait();
    const int quarter = warp & 3;  // TMEM lanes this warp may access
    int it = 0;
    uint32_t ep_phase = 0;
    uint32_t rb_phase = 0;
    // All 128 epilogue threads meet on an mbarrier (bounded wait, unlike a named barrier).
    auto ep_sync = [&]() -> bool {
      mbar_arrive(smem_u32(epbar));
      const bool r = mbar_wait(smem_u32(epbar), ep_phase, abort_flag, dev_err);
      ep_phase ^= 1u;
      return r;
    };
    const int r_local = quarter * 32 + lane;   // tile row of this thread
    const int t_epi = static_cast<int>(threadIdx.x) - 64;   // 0 .. 127
    for (int unit = unit0; unit < num_units; unit += unit_stride, ++it) {
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      const int mt = unit_mt(unit);
      const int nt = unit_nt(unit);
      const int row = tile_row(mt) + r_local;
      // Everything the tail reads besides the accumulator is fetched while the main loop runs:
      // the tile's bias and (gated residual) the gate row of its first row's item into shared
      // memory, and the residual values this thread stores in the first 64 columns into registers
      // (in the layout of the coalesced stores: 8 lanes per 32-column row segment).
      float* sb = epi_stage + acc * 2 * BN;   // [bias BN][gate BN]
      int item0 = 0;
      float4 hb0[8], hb1[8];
      if (splits == 1) {
        if constexpr (EPI == kEpiResidF32) {
          // (the second CTA of a pair may hold only rows past M: clamp to a real row's item)
          item0 = (tile_row(mt) < M ? tile_row(mt) : M - 1) / e.rows_per_item;
          if (e.item_map != nullptr) item0 = e.item_map[item0];
        }
        for (int c = t_epi; c < BN; c += 128) {
          if (e.bias != nullptr) sb[c] = e.bias[nt * BN + c];
          if constexpr (EPI == kEpiResidF32) sb[BN + c] = e.gate[item0 * e.gate_stride + nt * BN + c];
        }
        if constexpr (EPI == kEpiResidF32) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int trow = tile_row(mt) + quarter * 32 + i * 4 + (lane >> 3);
            if (trow < M) {
              const float4* h4 = reinterpret_cast<const float4*>(static_cast<const float*>(e.C) +
                                                                 static_cast<int64_t>(trow) * N + nt * BN) + (lane & 7);
              hb0[i] = h4[0];
              hb1[i] = h4[8];
            }
          }
        }
        if (!ep_sync()) break;   // the staged values are visible to every epilogue thread
      }
      // One lane waits; the warp then proceeds together (tcgen05.ld is warp-collective).
      int ok = 1;
      if (lane == 0) ok = mbar_wait(smem_u32(&tfull[acc]), acc_phase, abort_flag, dev_err) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      __syncwarp();
      if (!ok) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN;
      if (splits == 1) {
        EpiArgs es = e;
        es.bias = e.bias != nullptr ? sb - nt * BN : nullptr;          // es.bias + col hits the stage
        uint8_t* wscr = epi_scratch + (warp - 2) * 4096;               // this warp's transpose block
        const int row0 = tile_row(mt) + quarter * 32;                       // first row of this warp
        // every row of this warp belongs to the item whose gate row was staged
        bool one_item = true;
        if constexpr (EPI == kEpiResidF32) {
          const int last = (row0 + 31 < M ? row0 + 31 : M - 1);
          one_item = (tile_row(mt)) / e.rows_per_item == last / e.rows_per_item;
        }
        // The tail of one 32-column chunk.  The accumulator arrives one row per lane; the stores
        // leave one 32 x 32 block per warp through shared memory so that 8 (fp32) or 4 (bf16)
        // lanes write each row segment, i.e. whole cache lines per store instruction.  Both
        // shared-memory passes use a 16-byte-piece XOR swizzle: conflict-free.  hb = the residual
        // values of this chunk in the store layout.
        auto chunk = [&](int c, const float4 (&hb)[8]) {
          uint32_t r[32];
          tmem_ld32(taddr + c * 32, r);
          const int col_c = nt * BN + c * 32;
          if constexpr (EPI == kEpiResidF32 || EPI == kEpiF32) {
#pragma unroll
            for (int pc = 0; pc < 8; ++pc)
              *reinterpret_cast<uint4*>(wscr + lane * 128 + ((pc ^ (lane & 7)) * 16)) =
                  make_uint4(r[4 * pc], r[4 * pc + 1], r[4 * pc + 2], r[4 * pc + 3]);
            __syncwarp();
            const int pc = lane & 7;
            float4 vv[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const int rr = i * 4 + (lane >> 3);
              vv[i] = *reinterpret_cast<const float4*>(wscr + rr * 128 + ((pc ^ (rr & 7)) * 16));
            }
            __syncwarp();   // the block is free for the next chunk
            float4 b4 = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            if (es.bias != nullptr) b4 = *reinterpret_cast<const float4*>(es.bias + col_c + pc * 4);
            float4 g0 = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            if constexpr (EPI == kEpiResidF32) g0 = *reinterpret_cast<const float4*>(sb + BN + c * 32 + pc * 4);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const int grow = row0 + i * 4 + (lane >> 3);
              float4 v = vv[i];
              if (grow < M) {
                if (es.bias != nullptr) {
                  v.x += b4.x;
                  v.y += b4.y;
                  v.z += b4.z;
                  v.w += b4.w;
                }
                float4* dst = reinterpret_cast<float4*>(static_cast<float*>(e.C) + static_cast<int64_t>(grow) * N + col_c) + pc;
                if constexpr (EPI == kEpiResidF32) {
                  float4 g = g0;
                  if (!one_item) {
                    int item = grow / e.rows_per_item;
                    if (e.item_map != nullptr) item = e.item_map[item];
                    if (item != item0) g = __ldg(reinterpret_cast<const float4*>(e.gate + item * e.gate_stride + col_c) + pc);
                  }
                  float4 h = hb[i];
                  h.x = fmaf(g.x, v.x, h.x);
                  h.y = fmaf(g.y, v.y, h.y);
                  h.z = fmaf(g.z, v.z, h.z);
                  h.w = fmaf(g.w, v.w, h.w);
                  *dst = h;
                } else {
                  *dst = v;
                }
              }
            }
          } else {
            const int d3 = N / 3;
            if (EPI == kEpiQkvVt && col_c >= 2 * d3) {
              // V columns: written transposed into V^T straight from the row layout (lanes hold
              // consecutive tokens, so each store instruction covers 64 contiguous bytes)
              if (row < M) {
#pragma unroll
                for (int half = 0; half < 2; ++half) {
                  EpiIn in;
                  if (es.bias != nullptr) {
#pragma unroll
                    for (int j = 0; j < 4; ++j) in.b[j] = reinterpret_cast<const float4*>(es.bias + col_c + half * 16)[j];
                  }
                  epi_store16<EPI>(es, N, row, col_c + half * 16, r + half * 16, in);
                }
              }
              return;
            }
            float v[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
            if (es.bias != nullptr) {
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                const float4 b = reinterpret_cast<const float4*>(es.bias + col_c)[j];
                v[4 * j] += b.x;
                v[4 * j + 1] += b.y;
                v[4 * j + 2] += b.z;
                v[4 * j + 3] += b.w;
              }
            }
            if constexpr (EPI == kEpiGeluBf16) {
#pragma unroll
              for (int i = 0; i < 32; ++i) v[i] = gelu_tanh_bf16tail(v[i]);
            }
#pragma unroll
            for (int pc = 0; pc < 4; ++pc)
              *reinterpret_cast<uint4*>(wscr + lane * 64 + ((pc ^ ((lane >> 1) & 3)) * 16)) = pack_bf16x8(v + 8 * pc);
            __syncwarp();
            const int pc = lane & 3;
            uint4 uu[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int rr = i * 8 + (lane >> 2);
              uu[i] = *reinterpret_cast<const uint4*>(wscr + rr * 64 + ((pc ^ ((rr >> 1) & 3)) * 16));
            }
            __syncwarp();   // the block is free for the next chunk
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int grow = row0 + i * 8 + (lane >> 2);
              if (grow < M)
                reinterpret_cast<uint4*>(static_cast<bf16*>(e.C) + static_cast<int64_t>(grow) * N + col_c)[pc] = uu[i];
            }
          }
        };
        auto reload = [&](int c, float4 (&hb)[8]) {
          if constexpr (EPI == kEpiResidF32) {
            if (c < BN / 32) {
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                const int trow = row0 + i * 4 + (lane >> 3);
                if (trow < M)
                  hb[i] = reinterpret_cast<const float4*>(static_cast<const float*>(e.C) + static_cast<int64_t>(trow) * N +
                                                          nt * BN + c * 32)[lane & 7];
              }
            }
          }
        };
#pragma unroll 1
        for (int c = 0; c < BN / 32; c += 2) {
          chunk(c, hb0);
          reload(c + 2, hb0);
          chunk(c + 1, hb1);
          reload(c + 3, hb1);
        }
        tc_fence_before();
        if constexpr (kPair)
          mbar_arrive_cluster(cluster_addr(smem_u32(&tempty[acc]), 0));   // the MMA thread's barrier
        else
          mbar_arrive(smem_u32(&tempty[acc]));
        continue;
      }
      if constexpr (kPair) break;   // pairs never split K
      // ---- K split: publish this unit's partial, then the last unit of the tile finishes it ----
      const int mn = unit % num_mn;
      const int ks = unit / num_mn;
      float4* part = reinterpret_cast<float4*>(sp.ws) + (static_cast<size_t>(mn) * splits + ks) * (kBM * BN / 4);
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(taddr + c * 32, r);
#pragma unroll
        for (int j = 0; j < 8; ++j)   // [BN/4][kBM][4]: a warp's 32 rows of one column quad are contiguous
          __stcg(part + (c * 8 + j) * kBM + r_local,
                 make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                             __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3])));
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&tempty[acc]));
      __threadfence();
      if (!ep_sync()) break;
      if (threadIdx.x == 64) *last_flag = (atomicAdd(sp.counters + mn, 1) == splits - 1) ? 1 : 0;
      if (!ep_sync()) break;
      if (*last_flag == 0) continue;
      // Last unit of the tile: bulk-copy every partial ([splits][BN/4][kBM][4] fp32, contiguous in
      // the workspace) into the stage buffers, which this CTA's finished main loop left idle.
      const uint32_t bytes = static_cast<uint32_t>(splits) * kBM * BN * 4;
      if (threadIdx.x == 64) {
        __threadfence();
        sp.counters[mn] = 0;   // every unit of the tile has taken its ticket
        asm volatile("fence.proxy.async.global;" ::: "memory");   // partials written by other CTAs
        const uint8_t* src = reinterpret_cast<const uint8_t*>(sp.ws) + static_cast<size_t>(mn) * bytes;
        mbar_expect_tx(smem_u32(rbar), bytes);
        for (uint32_t off = 0; off < bytes; off += 32768u) {
          const uint32_t n = bytes - off < 32768u ? bytes - off : 32768u;
          asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                       ::"r"(smem_u32(tiles) + off), "l"(src + off), "r"(n), "r"(smem_u32(rbar))
                       : "memory");
        }
      }
      if (!mbar_wait(smem_u32(rbar), rb_phase, abort_flag, dev_err)) break;
      rb_phase ^= 1u;
      const float4* parts = reinterpret_cast<const float4*>(tiles);
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        float v[32];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          float4 a = parts[(c * 8 + j) * kBM + r_local];
          for (int q = 1; q < splits; ++q) {
            const float4 b = parts[(q * (BN / 4) + c * 8 + j) * kBM + r_local];
            a.x += b.x;
            a.y += b.y;
            a.z += b.z;
            a.w += b.w;
          }
          v[4 * j] = a.x;
          v[4 * j + 1] = a.y;
          v[4 * j + 2] = a.z;
          v[4 * j + 3] = a.w;
        }
        uint32_t r[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(v[i]);
        if (row < M) epilogue32<EPI>(e, N, row, nt * BN + c * 32, r);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  // no CTA of a cluster leaves while its peer may still multicast into it or arrive on its barriers
  // (pairs: nor while the first CTA's MMAs may still write the second CTA's TMEM)
  if constexpr (MC == 2 || kPair) cluster_sync();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    if constexpr (kPair)
      asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(C::kTmemCols)
                   : "memory");
    else
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(C::kTmemCols)
                   : "memory");
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

template <int BN, int EPI, int KA, int MC, int CG = 1>
cudaError_t launch(const CUtensorMap& ta, const CUtensorMap& tb, int M, int N, int K,
                   const EpiArgs& e, const SplitArgs& sp, int num_sms, int* dev_err, cudaStream_t s) {
  using C = TileCfg<BN, KA, CG>;
  static PerDeviceSmem smem_rec;  // contexts may run on several host threads and devices
  const cudaError_t err = ensure_max_smem(smem_rec, gemm_tc_kernel<BN, EPI, KA, MC, CG>, C::kSmemBytes);
  if (err != cudaSuccess) return err;
  const int units = ((M + kBM * CG - 1) / (kBM * CG)) * (N / BN) * sp.splits;
  if constexpr (CG == 2) {
    // one cluster (the CTA pair) per 256-row unit, at most one CTA per SM
    const int grid = 2 * (units < num_sms / 2 ? units : num_sms / 2);
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = 2;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = C::kSmemBytes;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<BN, EPI, KA, 1, 2>, ta, tb, M, N, K, e, sp, dev_err);
  } else if constexpr (MC == 1) {
    const int grid = units < num_sms ? units : num_sms;
    return launch_pdl(gemm_tc_kernel<BN, EPI, KA, 1>, dim3(grid), dim3(kThreads), C::kSmemBytes, s, ta, tb, M, N,
                      K, e, sp, dev_err);
  } else {
    // one cluster of two CTAs per pair of column tiles, at most one CTA per SM
    const int pairs = units / 2;
    const int grid = 2 * (pairs < num_sms / 2 ? pairs : num_sms / 2);
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = 2;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = C::kSmemBytes;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<BN, EPI, KA, 2>, ta, tb, M, N, K, e, sp, dev_err);
  }
}

template <int BN, int KA, int MC, int CG = 1>
cudaError_t dispatch_epi(const CUtensorMap& ta, const CUtensorMap& tb, int M, int N, int K, int epi,
                         const EpiArgs& e, const SplitArgs& sp, int num_sms, int* dev_err, cudaStream_t s) {
  switch (epi) {
    case kEpiBf16: return launch<BN, kEpiBf16, KA, MC, CG>(ta, tb, M, N, K, e, sp, num_sms, dev_err, s);
    case kEpiGeluBf16: return launch<BN, kEpiGeluBf16, KA, MC, CG>(ta, tb, M, N, K, e, sp, num_sms, dev_err, s);
    case kEpiResidF32: return launch<BN, kEpiResidF32, KA, MC, CG>(ta, tb, M, N, K, e, sp, num_sms, dev_err, s);
    case kEpiF32: return launch<BN, kEpiF32, KA, MC, CG>(ta, tb, M, N, K, e, sp, num_sms, dev_err, s);
    case kEpiQkvVt: return launch<BN, kEpiQkvVt, KA, MC, CG>(ta, tb, M, N, K, e, sp, num_sms, dev_err, s);
    default: return cudaErrorInvalidValue;
  }
}

int pick_ka(int bn, int K) { return (bn <= 128 && K % (2 * kBK) == 0) ? 2 : 1; }

// Bytes of stage buffers of a tile shape: the most partials the last unit of a split tile can
// gather (splits x 128 x bn fp32).
long split_capacity(int bn, int ka) {
  if (bn == 64) return ka == 2 ? TileCfg<64, 2>::kStages * TileCfg<64, 2>::kStageBytes
                               : TileCfg<64, 1>::kStages * TileCfg<64, 1>::kStageBytes;
  if (bn == 128) return ka == 2 ? TileCfg<128, 2>::kStages * TileCfg<128, 2>::kStageBytes
                                : TileCfg<128, 1>::kStages * TileCfg<128, 1>::kStageBytes;
  return TileCfg<256, 1>::kStages * TileCfg<256, 1>::kStageBytes;
}

}  // namespace

// Maps of one K-major bf16 operand [rows][K]: for one-atom boxes the plain 2-D {K, rows} with box
// {64, box_rows}; for two-atom boxes {64 (one swizzle row), rows, K/64} with the atom dimension
// 128 bytes apart and box {64, box_rows, 2}.
static int encode_kmajor_3d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t K, uint32_t box_rows,
                            uint32_t ka) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (fn == nullptr) return -1;
  if ((reinterpret_cast<uintptr_t>(base) & 15u) != 0 || K % kBK != 0) return -2;
  if (ka == 1) return tc_encode_bf16_box(map, base, rows, K, K, static_cast<uint32_t>(kBK), box_rows);
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(kBK), rows, K / kBK};
  cuuint64_t strides[2] = {K * 2, static_cast<cuuint64_t>(kBK) * 2};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(kBK), box_rows, ka};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : -3;
}

int tc_encode_gemm_operand(GemmOperand* op, const void* base, uint64_t rows, uint64_t K, bool rows64) {
  op->k2 = K % (2 * kBK) == 0;
  op->r64 = rows64;
  int r = encode_kmajor_3d(&op->r128_k1, base, rows, K, kBoxRows, 1);
  if (r == 0 && op->k2) r = encode_kmajor_3d(&op->r128_k2, base, rows, K, kBoxRows, 2);
  if (r == 0 && rows64) r = encode_kmajor_3d(&op->r64_k1, base, rows, K, 64, 1);
  if (r == 0 && rows64 && op->k2) r = encode_kmajor_3d(&op->r64_k2, base, rows, K, 64, 2);
  return r;
}

size_t tc_gemm_workspace_bytes(int num_sms) {
  // Splitting is only planned when all units fit in one wave: at most num_sms partial tiles of
  // 128 x 256 fp32, plus one counter per output tile.
  return static_cast<size_t>(num_sms) * kBM * 256 * sizeof(float) + static_cast<size_t>(num_sms) * sizeof(int);
}

// Tile width from the shape alone, so a plan never depends on timing: measured across the
// projections of the three model sizes at 1 to 32 episodes, 64-wide tiles win while the 128-wide
// ones cannot fill the SMs (more CTAs in flight hide the operand latency), 256-wide tiles win once
// they fill four waves (fewest operand bytes per flop), 128-wide tiles in between.  K splitting
// changes the summation order, so it is only used when asked for.
// Where the rule picks 256-wide tiles (and K % 128 == 0), CTA pairs run them as 256 x 256 units on
// one two-SM MMA: each SM then receives 128 weight rows per unit instead of 256 (serving scale,
// 78848 x {1024, 3072, 4096} projections: 1565 / 1537 / 1567 -> 1801 / 1574 / 1595 TFLOP/s).  At one
// episode the pairs gain nothing (fixed per-launch costs dominate), and the rule keeps single CTAs.
// Multicast clusters are not chosen by the rule: measured on the three models' projections at 1 to
// 32 episodes, they never beat the best single-CTA plan.  Both stay available through explicit
// plans.
GemmPlan tc_gemm_plan(int M, int N, int K, bool allow64, bool pairs64, int num_sms) {
  const long m_tiles = (M + kBM - 1) / kBM;
  const long tiles128 = m_tiles * (N / 128);
  int bn = 128;
  if (allow64 && tiles128 < num_sms)
    bn = 64;
  else if (N % 256 == 0 && (tiles128 / 2) >= 4L * num_sms)
    bn = 256;
  if (bn == 256 && K % (2 * kBK) == 0 && num_sms >= 2) return GemmPlan{256, 1, 3};
  // 128-wide tiles over many waves (N not a multiple of 256, e.g. the d1152 model's QKV and
  // MLP down-projection at 8 episodes: 1226 / 1214 -> 1294 / 1386 TFLOP/s) run as pairs too
  if (bn == 128 && pairs64 && K % (2 * kBK) == 0 && tiles128 >= 4L * num_sms && num_sms >= 2) return GemmPlan{128, 1, 3};
  return GemmPlan{bn, 1, 1};
}

cudaError_t tc_gemm(const GemmOperand& a, const GemmOperand& b, int M, int N, int K, int epi, const EpiArgs& e,
                    int num_sms, int* dev_err, cudaStream_t s, const SplitWorkspace* ws, GemmPlan plan) {
  if (M <= 0) return cudaSuccess;
  if (K % kBK != 0 || N % 128 != 0) return cudaErrorInvalidValue;
  if (plan.bn == 0) plan = tc_gemm_plan(M, N, K, b.r64, b.r64, num_sms);
  const int bn = plan.bn;
  // clusters need a K split of 1, two K-atoms per stage, an even number of column tiles and the
  // A operand's 64-row boxes; otherwise the plan runs without
  int mc = plan.mc == 0 ? tc_gemm_plan(M, N, K, b.r64, b.r64, num_sms).mc : plan.mc;
  if (plan.mc == 0) plan.mc = mc;
  if (mc == 2 && !(plan.splits <= 1 && bn <= 128 && K % (2 * kBK) == 0 && (N / bn) % 2 == 0 && a.r64 &&
                   num_sms >= 2))
    mc = 1;
  if ((bn != 64 && bn != 128 && bn != 256) || N % bn != 0 || (bn == 64 && !b.r64)) return cudaErrorInvalidValue;
  const int ka = pick_ka(bn, K);
  if (ka == 2 && !(a.k2 && b.k2)) return cudaErrorInvalidValue;
  SplitArgs sp{plan.splits < 1 ? 1 : plan.splits, nullptr, nullptr};
  if (sp.splits > 1) {
    const long units = static_cast<long>((M + kBM - 1) / kBM) * (N / bn) * sp.splits;
    if (ws == nullptr || ws->ws == nullptr || (K / (kBK * ka)) % sp.splits != 0 || units > num_sms ||
        static_cast<size_t>(units) * kBM * bn * sizeof(float) > ws->ws_bytes ||
        static_cast<long>(sp.splits) * kBM * bn * 4 > split_capacity(bn, ka))
      return cudaErrorInvalidValue;
    sp.ws = ws->ws;
    sp.counters = ws->counters;
  }
  if (plan.mc == 3) {
    // CTA pairs on one 256-row MMA: each CTA loads 128 rows of A and bn / 2 rows of B (one box)
    if (sp.splits != 1 || (bn != 128 && bn != 256) || N % bn != 0 || K % (2 * kBK) != 0 || !(a.k2 && b.k2) ||
        (bn == 128 && !b.r64) || num_sms < 2)
      return cudaErrorInvalidValue;
    if (bn == 256) return dispatch_epi<256, 2, 1, 2>(a.r128_k2, b.r128_k2, M, N, K, epi, e, sp, num_sms, dev_err, s);
    return dispatch_epi<128, 2, 1, 2>(a.r128_k2, b.r64_k2, M, N, K, epi, e, sp, num_sms, dev_err, s);
  }
  if (mc == 2) {   // A halves through the 64-row one-atom boxes
    if (bn == 64) return dispatch_epi<64, 2, 2>(a.r64_k1, b.r64_k2, M, N, K, epi, e, sp, num_sms, dev_err, s);
    return dispatch_epi<128, 2, 2>(a.r64_k1, b.r128_k2, M, N, K, epi, e, sp, num_sms, dev_err, s);
  }
  const CUtensorMap& ta = ka == 2 ? a.r128_k2 : a.r128_k1;
  if (bn == 64) {
    const CUtensorMap& tb = ka == 2 ? b.r64_k2 : b.r64_k1;
    return ka == 2 ? dispatch_epi<64, 2, 1>(ta, tb, M, N, K, epi, e, sp, num_sms, dev_err, s)
                   : dispatch_epi<64, 1, 1>(ta, tb, M, N, K, epi, e, sp, num_sms, dev_err, s);
  }
  if (bn == 256) return dispatch_epi<256, 1, 1>(ta, b.r128_k1, M, N, K, epi, e, sp, num_sms, dev_err, s);
  const CUtensorMap& tb = ka == 2 ? b.r128_k2 : b.r128_k1;
  return ka == 2 ? dispatch_epi<128, 2, 1>(ta, tb, M, N, K, epi, e, sp, num_sms, dev_err, s)
                 : dispatch_epi<128, 1, 1>(ta, tb, M, N, K, epi, e, sp, num_sms, dev_err, s);
}

int tc_encode_bf16_box(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t ld,
                       uint32_t box_cols, uint32_t box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (fn == nullptr) return -1;
  if ((reinterpret_cast<uintptr_t>(base) & 15u) != 0 || (ld * 2) % 16 != 0) return -2;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : -3;
}

int tc_encode_bf16_3d(CUtensorMap* map, const void* base, const uint64_t (&dims)[3], const uint64_t (&strides)[2],
                      const uint32_t (&box)[3], int swizzle_bytes) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (fn == nullptr) return -1;
  if ((reinterpret_cast<uintptr_t>(base) & 15u) != 0 || strides[0] % 16 != 0 || strides[1] % 16 != 0) return -2;
  const CUtensorMapSwizzle sw = swizzle_bytes == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
                                : swizzle_bytes == 32 ? CU_TENSOR_MAP_SWIZZLE_32B : CU_TENSOR_MAP_SWIZZLE_NONE;
  cuuint64_t d[3] = {dims[0], dims[1], dims[2]};
  cuuint64_t st[2] = {strides[0], strides[1]};
  cuuint32_t bx[3] = {box[0], box[1], box[2]};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), d, st, bx, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : -3;
}

}  // namespace wam
