// Full bidirectional attention on the fifth-generation tensor cores (head dim 64).
//
// One CTA owns 128 queries of one (item, head); TMEM lane r is query r.  Per block of 128 keys:
//   S = Q K^T    tcgen05.mma M=128 N=128 K=64 into one of two TMEM S buffers (cols 0 / 128)
//   softmax      warps 4-7, one thread per query row: tcgen05.ld of the S row, online max /
//                sum in the log2 domain, rescale of the O row in TMEM when the max grew,
//                P (bf16) written to shared memory in the 128-byte-swizzled K-major layout
//   O += P V     tcgen05.mma M=128 N=64 K=128 with P from shared memory and V^T (written by the
//                QKV projection's epilogue) as the K-major B operand; O in TMEM cols 256..319
// Warp 0 streams Q once and K / V^T tiles through a two-stage TMA ring; warp 1 issues the MMAs,
// computing S of block j+1 while the softmax works on block j.  Every wait is bounded.
#include "common.cuh"
#include "tcgen05.cuh"

namespace wam {
namespace {

constexpr int kQ = 128;
constexpr int kKV = 128;
constexpr int kDH = 64;
constexpr int kThreadsAttn = 256;
constexpr int kQBytes = kQ * kDH * 2;    // 16 KB
constexpr int kKBytes = kKV * kDH * 2;   // 16 KB
constexpr int kVBytes = kDH * kKV * 2;   // 16 KB: two 8 KB atom columns (64 keys each)
constexpr int kPBytes = kQ * kKV * 2;    // 32 KB: two 16 KB atom columns (64 keys each)
constexpr int kOffQ = 0;
constexpr int kOffK = kOffQ + kQBytes;
constexpr int kOffV = kOffK + 2 * kKBytes;
constexpr int kOffP = kOffV + 2 * kVBytes;
constexpr int kOffBar = kOffP + kPBytes;
constexpr int kSmemAttn = kOffBar + 256 + 1024;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColO = 256;

WAM_DEV float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__global__ void __launch_bounds__(kThreadsAttn, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQK, const __grid_constant__ CUtensorMap tmVt,
                   bf16* __restrict__ out, int N, int d, int H, float scale_log2, int* dev_err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint64_t* q_full = bars + 0;
  uint64_t* kv_full = bars + 1;   // [2]
  uint64_t* kv_empty = bars + 3;  // [2]
  uint64_t* s_full = bars + 5;    // [2]
  uint64_t* s_empty = bars + 7;   // [2]
  uint64_t* p_full = bars + 9;
  uint64_t* o_done = bars + 10;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 11);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int q0 = blockIdx.x * kQ;
  const int h = blockIdx.y;
  const int b = blockIdx.z;
  const int row_base = b * N;
  const int nkv = (N + kKV - 1) / kKV;

  if (threadIdx.x == 0) {
    mbar_init(smem_u32(q_full), 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&kv_full[i]), 1);
      mbar_init(smem_u32(&kv_empty[i]), 1);
      mbar_init(smem_u32(&s_full[i]), 1);
      mbar_init(smem_u32(&s_empty[i]), 128);
    }
    mbar_init(smem_u32(p_full), 128);
    mbar_init(smem_u32(o_done), 1);
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
    mbar_expect_tx(smem_u32(q_full), kQBytes);
    tma_load_2d(smem_u32(smem + kOffQ), &tmQK, h * kDH, row_base + q0, smem_u32(q_full));
    const int vt_row = (b * H + h) * kDH;
    for (int j = 0; j < nkv; ++j) {
      const int s = j & 1;
      if (!mbar_wait(smem_u32(&kv_empty[s]), ((j >> 1) & 1) ^ 1u, abort_flag, dev_err)) break;
      const uint32_t fb = smem_u32(&kv_full[s]);
      mbar_expect_tx(fb, kKBytes + kVBytes);
      tma_load_2d(smem_u32(smem + kOffK + s * kKBytes), &tmQK, d + h * kDH, row_base + j * kKV, fb);
      tma_load_2d(smem_u32(smem + kOffV + s * kVBytes), &tmVt, j * kKV, vt_row, fb);
      tma_load_2d(smem_u32(smem + kOffV + s * kVBytes + kVBytes / 2), &tmVt, j * kKV + 64, vt_row, fb);
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issue ----------------
    const uint32_t idS = idesc_bf16(kQ, kKV);
    const uint32_t idO = idesc_bf16(kQ, kDH);
    bool ok = mbar_wait(smem_u32(q_full), 0, abort_flag, dev_err);
    const uint32_t sq = smem_u32(smem + kOffQ);
    const uint32_t sp = smem_u32(smem + kOffP);
    for (int j = 0; ok && j <= nkv; ++j) {
      if (j < nkv) {
        const int s = j & 1;
        if (!mbar_wait(smem_u32(&kv_full[s]), (j >> 1) & 1, abort_flag, dev_err)) break;
        if (!mbar_wait(smem_u32(&s_empty[s]), ((j >> 1) & 1) ^ 1u, abort_flag, dev_err)) break;
        tc_fence_after();
        const uint32_t sk = smem_u32(smem + kOffK + s * kKBytes);
#pragma unroll
        for (int t = 0; t < kDH / 16; ++t)
          umma_bf16(tmem + s * kKV, sw128_desc(sq + t * 32), sw128_desc(sk + t * 32), idS, t > 0 ? 1u : 0u);
        umma_commit(smem_u32(&s_full[s]));
      }
      if (j >= 1) {
        const int jj = j - 1;
        if (!mbar_wait(smem_u32(p_full), jj & 1, abort_flag, dev_err)) break;
        tc_fence_after();
        const uint32_t sv = smem_u32(smem + kOffV + (jj & 1) * kVBytes);
#pragma unroll
        for (int t = 0; t < kKV / 16; ++t) {
          const uint32_t a = sp + (t >> 2) * (kPBytes / 2) + (t & 3) * 32;
          const uint32_t bb = sv + (t >> 2) * (kVBytes / 2) + (t & 3) * 32;
          umma_bf16(tmem + kColO, sw128_desc(a), sw128_desc(bb), idO, (jj > 0 || t > 0) ? 1u : 0u);
        }
        umma_commit(smem_u32(o_done));
        umma_commit(smem_u32(&kv_empty[jj & 1]));
      }
    }
  } else if (warp >= 4) {
    // ---------------- softmax: one query row per thread ----------------
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t lane_addr = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    uint8_t* prow = smem + kOffP + r * 128;
    float m = -1e30f, l = 0.0f;
    bool ok = true;
    for (int j = 0; j < nkv; ++j) {
      const int s = j & 1;
      if (!warp_wait(smem_u32(&s_full[s]), (j >> 1) & 1, abort_flag, dev_err)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float p[kKV];
#pragma unroll
      for (int c = 0; c < kKV / 32; ++c) {
        uint32_t v[32];
        tmem_ld32(lane_addr + s * kKV + c * 32, v);
#pragma unroll
        for (int i = 0; i < 32; ++i) p[c * 32 + i] = __uint_as_float(v[i]);
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&s_empty[s]));
      const int kv0 = j * kKV;
      if (kv0 + kKV > N) {
#pragma unroll
        for (int i = 0; i < kKV; ++i)
          if (kv0 + i >= N) p[i] = -1e30f;
      }
      float mx = p[0];
#pragma unroll
      for (int i = 1; i < kKV; ++i) mx = fmaxf(mx, p[i]);
      const float m_new = fmaxf(m, mx * scale_log2);
      float rs = 0.0f;
#pragma unroll
      for (int i = 0; i < kKV; ++i) {
        p[i] = ex2(fmaf(p[i], scale_log2, -m_new));
        rs += p[i];
      }
      const float corr = ex2(m - m_new);
      l = l * corr + rs;
      m = m_new;
      if (j > 0) {
        // P.V of the previous block must be complete: O is then stable and P's buffer free.
        if (!warp_wait(smem_u32(o_done), (j - 1) & 1, abort_flag, dev_err)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (__any_sync(0xffffffffu, corr != 1.0f)) {
#pragma unroll
          for (int c = 0; c < kDH / 32; ++c) {
            uint32_t v[32];
            tmem_ld32(lane_addr + kColO + c * 32, v);
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * corr);
            tmem_st32(lane_addr + kColO + c * 32, v);
          }
        }
      }
      // P row -> shared memory: 16 chunks of 8 bf16; chunk c of atom column c/8 lands at
      // 16-byte slot (c%8) xor (r%8) of the row (128-byte swizzle).
#pragma unroll
      for (int c = 0; c < kKV / 8; ++c) {
        uint4 u;
        u.x = pack_bf16x2(p[8 * c + 0], p[8 * c + 1]);
        u.y = pack_bf16x2(p[8 * c + 2], p[8 * c + 3]);
        u.z = pack_bf16x2(p[8 * c + 4], p[8 * c + 5]);
        u.w = pack_bf16x2(p[8 * c + 6], p[8 * c + 7]);
        *reinterpret_cast<uint4*>(prow + (c >> 3) * (kPBytes / 2) + (((c & 7) ^ (r & 7)) << 4)) = u;
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      tc_fence_before();
      mbar_arrive(smem_u32(p_full));
    }
    if (ok && warp_wait(smem_u32(o_done), (nkv - 1) & 1, abort_flag, dev_err)) {
      tc_fence_after();
      const float inv = 1.0f / l;
      const int q = q0 + r;
      uint4* dst = reinterpret_cast<uint4*>(out + static_cast<int64_t>(row_base + q) * d + h * kDH);
#pragma unroll
      for (int c = 0; c < kDH / 32; ++c) {
        uint32_t v[32];
        tmem_ld32(lane_addr + kColO + c * 32, v);
        if (q < N) {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            uint4 u;
            u.x = pack_bf16x2(__uint_as_float(v[8 * k + 0]) * inv, __uint_as_float(v[8 * k + 1]) * inv);
            u.y = pack_bf16x2(__uint_as_float(v[8 * k + 2]) * inv, __uint_as_float(v[8 * k + 3]) * inv);
            u.z = pack_bf16x2(__uint_as_float(v[8 * k + 4]) * inv, __uint_as_float(v[8 * k + 5]) * inv);
            u.w = pack_bf16x2(__uint_as_float(v[8 * k + 6]) * inv, __uint_as_float(v[8 * k + 7]) * inv);
            dst[c * 4 + k] = u;
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

cudaError_t attention_tc(const CUtensorMap& tm_qk, const CUtensorMap& tm_vt, bf16* out, int B, int N, int d,
                         int H, int* dev_err, cudaStream_t s) {
  if (B <= 0 || N <= 0) return cudaSuccess;
  if (d / H != kDH) return cudaErrorInvalidValue;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemAttn);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const float scale_log2 = 1.4426950408889634f / 8.0f;  // log2(e) / sqrt(64)
  dim3 grid((N + kQ - 1) / kQ, H, B);
  return launch_pdl(attn_tc_kernel, grid, dim3(kThreadsAttn), kSmemAttn, s, tm_qk, tm_vt, out, N, d, H,
                    scale_log2, dev_err);
}

int attention_tc_vt_ld(int N) { return (N + 7) / 8 * 8; }

}  // namespace wam
