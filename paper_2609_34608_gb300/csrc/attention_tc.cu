// Full bidirectional attention on the fifth-generation tensor cores (head dim 64 or 72).
//
// Head dim 72 (the bimanual model): tcgen05 K and N come in steps of 16, so the head is padded to
// 80.  Q and K arrive as a 128-byte-swizzled atom of columns 0..63 plus a 32-byte-swizzled atom of
// columns 64..79, fetched through a 3-D view {72, 3 heads, rows} of the QKV buffer whose
// out-of-range columns 72..79 TMA fills with zeros, so the fifth K step of Q K^T adds nothing
// spurious.  The P.V product runs with N = 80 over V^T rows of the head and the next eight
// (or zero fill at the end); O columns 72..79 are never read.  Two S buffers instead of three keep
// S and both padded O accumulators within the 512 TMEM columns.  The description below is for
// head dim 64; with 72 the O accumulators sit at columns 256..335 and 336..415.
//
// One CTA owns 128 queries of one (item, head); TMEM lane r is query r.  Per block of 128 keys:
//   S = Q K^T    tcgen05.mma M=128 N=128 K=64 into one of three TMEM S buffers (cols 0/128/256)
//   softmax      warps 4-11, two threads per query row, each an independent online-softmax
//                stream over its half (64 keys) of every block: tcgen05.ld of its S half-row,
//                running max / sum in the log2 domain, then P (bf16 pairs) stored with tcgen05.st
//                over the first 32 columns of the same half-row, so P needs no TMEM of its own.
//                Each half accumulates into its own O, rescaled only when its running max grows
//                by more than 2^8 (the stale max keeps every P <= 256); the two streams are merged
//                once, at the end, so the halves never wait on each other per block
//   O_h += P_h V_h  tcgen05.mma M=128 N=64 K=64 per half with the A operand P read from TMEM
//                and V^T (written by the QKV projection's epilogue) as the K-major B operand
//                from shared memory; O_0 in TMEM cols 384..447, O_1 in cols 448..511
// Warp 0 streams Q once and K / V^T tiles through a six-stage TMA ring (one barrier per stage
// for both tiles; a stage is released when the P.V of its block finished).  Warp 1 issues
// S = Q K^T, warps 2 and 3 issue the P.V of the two halves; each of these warps waits as a
// whole and issues its MMAs and their commit from one elected lane (warp-uniform operands keep
// the issue fast next to the busy softmax warps).  tcgen05.commit tracks the MMAs of the
// issuing thread only, so the streams complete independently.  An S buffer is reused once both
// P.V that read its P finished, so S runs up to two blocks ahead of the softmax.  Softmax
// arrivals are one per warp.  Every wait is bounded.
#include "common.cuh"
#include "tcgen05.cuh"

namespace wam {
namespace {

constexpr int kQ = 128;
constexpr int kKV = 128;
constexpr int kThreadsAttn = 384;
constexpr float kRescaleLog2 = 8.0f;  // lazy-rescale threshold (log2 units)
constexpr uint32_t kTmemCols = 512;
constexpr int kSoftmaxWarps = 8;

// Shape of one head dimension.  Q / K tiles: a 128-byte-swizzled atom (head columns 0..63) plus,
// for 72, a 32-byte-swizzled atom (columns 64..79); V^T tiles: kDHP rows of 128 keys as two atom
// columns of 64 keys.
template <int DH>
struct AttnShape {
  static constexpr int kDHP = DH == 64 ? 64 : 80;       // head dim padded to the MMA's N / K step
  static constexpr int kTailRow = DH == 64 ? 0 : 32;    // bytes per row of the 32-byte-swizzled atom
  static constexpr int kKVStages = DH == 64 ? 6 : 5;
  static constexpr int kSBuf = DH == 64 ? 3 : 2;        // TMEM S buffers (each also holds its P)
  static constexpr int kQBytes = kQ * (128 + kTailRow);
  static constexpr int kKBytes = kKV * (128 + kTailRow);
  static constexpr int kVBytes = kDHP * kKV * 2;        // two atom columns of 64 keys
  static constexpr int kOffQ = 0;
  static constexpr int kOffK = kOffQ + kQBytes;
  static constexpr int kOffV = kOffK + kKVStages * kKBytes;
  static constexpr int kOffX = kOffV + kKVStages * kVBytes;   // max / sum exchange [2][2][128] floats
  static constexpr int kOffBar = kOffX + 2048;
  static constexpr int kNumBars = 1 + 2 * kKVStages + 3 * kSBuf + 8;
  static constexpr int kSmem = kOffBar + 512 + 1024;   // barriers, TMEM slot, abort flag; alignment slack
  static constexpr uint32_t kColO = kSBuf * kKV;        // O_0 at kColO, O_1 at kColO + kDHP
  static_assert(kNumBars * 8 + 8 <= 512, "barrier block exceeds its reservation");
  static_assert(kColO + 2 * kDHP <= kTmemCols, "TMEM columns");
  static_assert(kSmem <= 232448, "shared memory");
  static_assert(kOffK % 1024 == 0 && kKBytes % 1024 == 0 && kVBytes % 2048 == 0, "swizzle alignment");
};

WAM_DEV float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

WAM_DEV float max3(float a, float b, float c) {
  float y;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(y) : "f"(a), "f"(b), "f"(c));
  return y;
}

template <int DH>
__global__ void __launch_bounds__(kThreadsAttn, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQK, const __grid_constant__ CUtensorMap tmQKTail,
                   const __grid_constant__ CUtensorMap tmVt, bf16* __restrict__ out, int N, int d, int H,
                   float scale_log2, int* dev_err) {
  using S = AttnShape<DH>;
  constexpr int kDHP = S::kDHP, kKVStages = S::kKVStages, kSBuf = S::kSBuf;
  constexpr int kQBytes = S::kQBytes, kKBytes = S::kKBytes, kVBytes = S::kVBytes;
  constexpr int kOffQ = S::kOffQ, kOffK = S::kOffK, kOffV = S::kOffV, kOffX = S::kOffX, kOffBar = S::kOffBar;
  constexpr uint32_t kColO = S::kColO;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint64_t* q_full = bars + 0;
  uint64_t* kv_full = bars + 1;                   // [kKVStages]: K and V^T tiles of the stage landed
  uint64_t* kv_empty = kv_full + kKVStages;       // [kKVStages]: P.V of the stage's block finished
  uint64_t* s_full = kv_empty + kKVStages;        // [kSBuf]: S of the buffer's block computed
  uint64_t* s_free = s_full + kSBuf;              // [kSBuf]: P.V that read the buffer's P finished
  uint64_t* p_full = s_free + kSBuf;              // [kSBuf]: P of the buffer's block stored
  uint64_t* xpair = p_full + kSBuf;               // [4 quarters][2]: the two threads of a row exchanged values
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(xpair + 8);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* xch = reinterpret_cast<float*>(smem + kOffX);  // [2 buffers][2 halves][128 rows]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int q0 = blockIdx.x * kQ;
  const int h = blockIdx.y;
  const int b = blockIdx.z;
  const int row_base = b * N;
  const int nkv = (N + kKV - 1) / kKV;

  if (threadIdx.x == 0) {
    mbar_init(smem_u32(q_full), 1);
    for (int i = 0; i < kKVStages; ++i) {
      mbar_init(smem_u32(&kv_full[i]), 1);
      mbar_init(smem_u32(&kv_empty[i]), 2);   // one commit from each P.V thread
    }
    for (int i = 0; i < kSBuf; ++i) {
      mbar_init(smem_u32(&s_full[i]), 1);
      mbar_init(smem_u32(&s_free[i]), 2);
      mbar_init(smem_u32(&p_full[i]), kSoftmaxWarps);   // one arrival per softmax warp
    }
    for (int i = 0; i < 8; ++i) mbar_init(smem_u32(&xpair[i]), 64);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_launch_dependents();

  if (warp == 0 && lane == 0) {
    // ---------------- TMA: Q once, then K and V^T tiles ----------------
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmQK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmVt)) : "memory");
    pdl_wait();
    // Q (or K) rows [row, row + 128) of head hh: head dim 64 through the 2-D map {3d, rows};
    // 72 through the 3-D map {72, 3H, rows}, columns 0..63 and 64..79 (72..79 zero-filled)
    auto load_qk = [&](uint32_t dst, int hh, int row, uint32_t bar) {
      if constexpr (DH == 64) {
        tma_load_2d(dst, &tmQK, hh * 64, row, bar);
      } else {
        tma_load_3d(dst, &tmQK, 0, hh, row, bar);
        tma_load_3d(dst + kQ * 128, &tmQKTail, 64, hh, row, bar);
      }
    };
    mbar_expect_tx(smem_u32(q_full), kQBytes);
    load_qk(smem_u32(smem + kOffQ), h, row_base + q0, smem_u32(q_full));
    const int vt_row = (b * H + h) * DH;
    for (int j = 0; j < nkv; ++j) {
      const int s = j % kKVStages;
      if (!mbar_wait(smem_u32(&kv_empty[s]), ((j / kKVStages) & 1) ^ 1u, abort_flag, dev_err)) break;
      const uint32_t fb = smem_u32(&kv_full[s]);
      mbar_expect_tx(fb, kKBytes + kVBytes);
      load_qk(smem_u32(smem + kOffK + s * kKBytes), H + h, row_base + j * kKV, fb);
      tma_load_2d(smem_u32(smem + kOffV + s * kVBytes), &tmVt, j * kKV, vt_row, fb);
      tma_load_2d(smem_u32(smem + kOffV + s * kVBytes + kVBytes / 2), &tmVt, j * kKV + 64, vt_row, fb);
    }
  } else if (warp == 1) {
    // ---------------- S = Q K^T issue (whole warp waits, one elected lane issues) ----------------
    // Warps 2 and 3 issue P.V: tcgen05.commit tracks the MMAs of the issuing thread only, so
    // the streams complete independently and none waits behind another's barriers.
    const uint32_t idS = idesc_bf16(kQ, kKV);
    bool ok = warp_all_wait(smem_u32(q_full), 0, abort_flag, dev_err);
    const uint64_t dq = sw128_desc(smem_u32(smem + kOffQ));
    for (int j = 0; ok && j < nkv; ++j) {
      const int s = j % kSBuf;
      const int ks = j % kKVStages;
      if (!warp_all_wait(smem_u32(&kv_full[ks]), (j / kKVStages) & 1, abort_flag, dev_err)) break;
      if (!warp_all_wait(smem_u32(&s_free[s]), ((j / kSBuf) & 1) ^ 1u, abort_flag, dev_err)) break;
      tc_fence_after();
      const uint64_t dk = sw128_desc(smem_u32(smem + kOffK + ks * kKBytes));
      if (elect_one()) {
#pragma unroll
        for (int t = 0; t < 4; ++t)   // descriptor address field is addr >> 4: +32 B = +2
          umma_bf16(tmem + s * kKV, dq + 2 * t, dk + 2 * t, idS, t > 0 ? 1u : 0u);
        if constexpr (DH != 64)        // head columns 64..79 from the 32-byte-swizzled atoms
          umma_bf16(tmem + s * kKV, sw32_desc(smem_u32(smem + kOffQ) + kQ * 128),
                    sw32_desc(smem_u32(smem + kOffK + ks * kKBytes) + kKV * 128), idS, 1u);
        umma_commit(smem_u32(&s_full[s]));   // same lane as the MMAs it tracks
      }
      __syncwarp();
    }
  } else if (warp == 2 || warp == 3) {
    // ---------------- O_h += P_h V_h issue, h = warp - 2 (as for S) ----------------
    // Each half's four MMAs come from their own thread.  kv_empty[stage] completes (two commits)
    // when both halves of the stage's block finished: it releases the K and V^T tiles to the
    // producer and tells the softmax that O is up to date; s_free[buffer] hands the S buffer (and
    // the P inside it) back to the S thread.
    const int hv = warp - 2;
    const uint32_t idO = idesc_bf16(kQ, kDHP);
    for (int j = 0; j < nkv; ++j) {
      const int sb = j % kSBuf;
      const int vs = j % kKVStages;
      if (!warp_all_wait(smem_u32(&p_full[sb]), (j / kSBuf) & 1, abort_flag, dev_err)) break;
      if (!warp_all_wait(smem_u32(&kv_full[vs]), (j / kKVStages) & 1, abort_flag, dev_err)) break;
      tc_fence_after();
      // keys 64 hv + 16t .. +15: P in columns 64 hv + 8t .. +7 of the buffer, V^T in atom column hv
      const uint32_t tp = tmem + sb * kKV + hv * 64;
      const uint64_t dv = sw128_desc(smem_u32(smem + kOffV + vs * kVBytes) + hv * (kVBytes / 2));
      if (elect_one()) {
#pragma unroll
        for (int t = 0; t < 4; ++t)
          umma_bf16_ta(tmem + kColO + hv * kDHP, tp + t * 8, dv + 2 * t, idO, (j > 0 || t > 0) ? 1u : 0u);
        umma_commit(smem_u32(&s_free[sb]));   // same lane as the MMAs they track
        umma_commit(smem_u32(&kv_empty[vs]));
      }
      __syncwarp();
    }
  } else if (warp >= 4) {
    // ---------------- softmax: two threads per query row ----------------
    const int quarter = warp & 3;
    const int half = (warp - 4) >> 2;         // keys [64 half, 64 half + 64), O cols [32 half, +32)
    const int r = quarter * 32 + lane;
    const uint32_t lane_addr = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    // Exchange with the partner thread of the same row (the other warp of this quarter) through
    // a double-buffered slot guarded by an mbarrier of the 64 threads of the two warps; use u
    // of the exchange goes to buffer u & 1 and completes phase u >> 1 of its barrier (used
    // twice, to merge the two half streams at the end).
    auto exchange = [&](int u, float v, float& partner) -> bool {
      float* slot = xch + (u & 1) * 2 * kQ;
      slot[half * kQ + r] = v;
      const uint32_t bar = smem_u32(&xpair[quarter * 2 + (u & 1)]);
      mbar_arrive(bar);
      if (!mbar_wait(bar, (u >> 1) & 1, abort_flag, dev_err)) return false;
      partner = slot[(half ^ 1) * kQ + r];
      return true;
    };
    // The running max starts at a finite floor far above the mask value (-1e30 before scaling),
    // so a half whose keys are all masked (N <= 64) keeps P = 0 and l = 0.
    float m = -1e20f, l = 0.0f;
    bool ok = true;
    for (int j = 0; j < nkv; ++j) {
      const int s = j % kSBuf;
      if (!warp_wait(smem_u32(&s_full[s]), (j / kSBuf) & 1, abort_flag, dev_err)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float p[64];
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        uint32_t v[32];
        tmem_ld32(lane_addr + s * kKV + half * 64 + c * 32, v);
#pragma unroll
        for (int i = 0; i < 32; ++i) p[c * 32 + i] = __uint_as_float(v[i]);
      }
      const int kv0 = j * kKV + half * 64;
      if (kv0 + 64 > N) {
#pragma unroll
        for (int i = 0; i < 64; ++i)
          if (kv0 + i >= N) p[i] = -1e30f;
      }
      // Row max with three-input max (four independent chains), then the exponentials with
      // packed f32x2 FMA / add: the softmax warps share their SM sub-partitions with the MMA
      // issuing threads, so fewer instructions here means faster MMA issue there.
      float mx4[4] = {p[0], p[1], p[2], p[3]};
#pragma unroll
      for (int i = 4; i < 64; i += 8) {
#pragma unroll
        for (int k = 0; k < 4; ++k) mx4[k] = max3(mx4[k], p[i + 2 * k], p[i + 2 * k + 1]);
      }
      const float mx = max3(mx4[0], mx4[1], fmaxf(mx4[2], mx4[3]));
      const float cand = mx * scale_log2;
      // Lazy rescale: keep the stale max unless the new one exceeds it by more than 2^8.
      const bool grow = j == 0 || cand > m + kRescaleLog2;
      const float m_use = grow ? fmaxf(m, cand) : m;
      const float corr = grow ? ex2(m - m_use) : 1.0f;
      const float2 sc2 = make_float2(scale_log2, scale_log2);
      const float2 nm2 = make_float2(-m_use, -m_use);
      float2 rs2[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) rs2[k] = make_float2(0.0f, 0.0f);
#pragma unroll
      for (int c = 0; c < 32; ++c) {
        float2 x = __ffma2_rn(make_float2(p[2 * c], p[2 * c + 1]), sc2, nm2);
        x.x = ex2(x.x);
        x.y = ex2(x.y);
        p[2 * c] = x.x;
        p[2 * c + 1] = x.y;
        rs2[c & 3] = __fadd2_rn(rs2[c & 3], x);
      }
      const float2 rs = __fadd2_rn(__fadd2_rn(rs2[0], rs2[1]), __fadd2_rn(rs2[2], rs2[3]));
      l = l * corr + (rs.x + rs.y);
      m = m_use;
      if (j > 0 && __any_sync(0xffffffffu, corr != 1.0f)) {
        // Rescale this thread's 32 O columns once every earlier P.V has landed.
        if (!warp_wait(smem_u32(&kv_empty[(j - 1) % kKVStages]), ((j - 1) / kKVStages) & 1, abort_flag, dev_err)) {
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          uint32_t v[32];
          tmem_ld32(lane_addr + kColO + half * kDHP + c * 32, v);
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * corr);
          tmem_st32(lane_addr + kColO + half * kDHP + c * 32, v);
        }
        if constexpr (DH != 64) {   // head columns 64..71 (72..79 are padding, never read)
          uint32_t v[8];
          tmem_ld8(lane_addr + kColO + half * kDHP + 64, v);
#pragma unroll
          for (int i = 0; i < 8; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * corr);
          tmem_st8(lane_addr + kColO + half * kDHP + 64, v);
        }
      }
      // 32 bf16 pairs over the first 32 columns of this thread's S half-row (already read).
      uint32_t pk[32];
#pragma unroll
      for (int c = 0; c < 32; ++c) pk[c] = pack_bf16x2(p[2 * c], p[2 * c + 1]);
      tmem_st32(lane_addr + s * kKV + half * 64, pk);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&p_full[s]));
    }
    // Merge the two half streams: O = sum_h O_h 2^(m_h - M), l = sum_h l_h 2^(m_h - M).
    float m_partner = 0.0f, l_partner = 0.0f;
    if (ok && exchange(0, m, m_partner) && exchange(1, l, l_partner)) {
      const float M = fmaxf(m, m_partner);
      const float f_own = ex2(m - M), f_par = ex2(m_partner - M);
      const float inv = 1.0f / (l * f_own + l_partner * f_par);
      const float w0 = (half == 0 ? f_own : f_par) * inv;   // weight of O_0
      const float w1 = (half == 0 ? f_par : f_own) * inv;   // weight of O_1
      if (warp_wait(smem_u32(&kv_empty[(nkv - 1) % kKVStages]), ((nkv - 1) / kKVStages) & 1, abort_flag, dev_err)) {
        tc_fence_after();
        const int q = q0 + r;
        uint32_t v0[32], v1[32];
        tmem_ld32(lane_addr + kColO + half * 32, v0);         // O_0, this thread's 32 columns
        tmem_ld32(lane_addr + kColO + kDHP + half * 32, v1);  // O_1, same columns
        if constexpr (DH != 64) {   // head columns 64..71, written by the first thread of the row
          uint32_t t0[8], t1[8];
          tmem_ld8(lane_addr + kColO + 64, t0);
          tmem_ld8(lane_addr + kColO + kDHP + 64, t1);
          if (q < N && half == 0) {
            float o[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) o[e] = fmaf(__uint_as_float(t0[e]), w0, __uint_as_float(t1[e]) * w1);
            uint4 u;
            u.x = pack_bf16x2(o[0], o[1]);
            u.y = pack_bf16x2(o[2], o[3]);
            u.z = pack_bf16x2(o[4], o[5]);
            u.w = pack_bf16x2(o[6], o[7]);
            *reinterpret_cast<uint4*>(out + static_cast<int64_t>(row_base + q) * d + h * DH + 64) = u;
          }
        }
        if (q < N) {
          uint4* dst = reinterpret_cast<uint4*>(out + static_cast<int64_t>(row_base + q) * d + h * DH + half * 32);
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            float o[8];
#pragma unroll
            for (int e = 0; e < 8; ++e)
              o[e] = fmaf(__uint_as_float(v0[8 * k + e]), w0, __uint_as_float(v1[8 * k + e]) * w1);
            uint4 u;
            u.x = pack_bf16x2(o[0], o[1]);
            u.y = pack_bf16x2(o[2], o[3]);
            u.z = pack_bf16x2(o[4], o[5]);
            u.w = pack_bf16x2(o[6], o[7]);
            dst[k] = u;
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace

int attention_tc_encode(AttnMaps* m, const void* qkv, const void* vt, int items, int N, int d, int H, int vt_ld) {
  const int dh = H > 0 ? d / H : 0;
  const uint64_t rows = static_cast<uint64_t>(items) * N;
  if (H <= 0 || d != dh * H || (dh != 64 && dh != 72)) return -1;
  m->dh = dh;
  if (dh == 64) {
    if (tc_encode_bf16_box(&m->qk, qkv, rows, 3 * d, 3 * d, 64, 128) != 0) return -2;
    m->qk_tail = m->qk;
  } else {
    // {72 head columns, 3H heads of q | k | v, rows}: box columns past 72 are zero-filled
    const uint64_t dims[3] = {72, static_cast<uint64_t>(3 * H), rows};
    const uint64_t strides[2] = {72 * 2, static_cast<uint64_t>(3 * d) * 2};
    const uint32_t box0[3] = {64, 1, 128}, box1[3] = {16, 1, 128};
    if (tc_encode_bf16_3d(&m->qk, qkv, dims, strides, box0, 128) != 0 ||
        tc_encode_bf16_3d(&m->qk_tail, qkv, dims, strides, box1, 32) != 0)
      return -2;
  }
  const uint32_t vrows = dh == 64 ? 64 : 80;
  if (tc_encode_bf16_box(&m->vt, vt, static_cast<uint64_t>(items) * d, vt_ld, vt_ld, 64, vrows) != 0) return -3;
  return 0;
}

cudaError_t attention_tc(const AttnMaps& m, bf16* out, int B, int N, int d, int H, int* dev_err, cudaStream_t s) {
  if (B <= 0 || N <= 0) return cudaSuccess;
  if (d / H != m.dh) return cudaErrorInvalidValue;
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(m.dh));  // log2(e) / sqrt(dh)
  dim3 grid((N + kQ - 1) / kQ, H, B);
  if (m.dh == 64) {
    static PerDeviceSmem smem_rec;  // contexts may run on several host threads and devices
    const cudaError_t e = ensure_max_smem(smem_rec, attn_tc_kernel<64>, AttnShape<64>::kSmem);
    if (e != cudaSuccess) return e;
    return launch_pdl(attn_tc_kernel<64>, grid, dim3(kThreadsAttn), AttnShape<64>::kSmem, s, m.qk, m.qk_tail, m.vt,
                      out, N, d, H, scale_log2, dev_err);
  }
  static PerDeviceSmem smem_rec72;
  const cudaError_t e = ensure_max_smem(smem_rec72, attn_tc_kernel<72>, AttnShape<72>::kSmem);
  if (e != cudaSuccess) return e;
  return launch_pdl(attn_tc_kernel<72>, grid, dim3(kThreadsAttn), AttnShape<72>::kSmem, s, m.qk, m.qk_tail, m.vt,
                    out, N, d, H, scale_log2, dev_err);
}

int attention_tc_vt_ld(int N) { return (N + 7) / 8 * 8; }

}  // namespace wam
