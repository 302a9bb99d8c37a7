// Dense projections of the DiT block on the fifth-generation tensor cores (sm_103a).
//
// C[M,N] = A[M,K] . Wt[N,K]^T with bf16 operands and an fp32 accumulator held in TMEM, and the
// block's elementwise tail fused into the accumulator read-back (bias, GELU, adaLN-gated
// residual).  Persistent, warp-specialised CTAs:
//   warp 0      TMA producer: 128x64 A and BNx64 B tiles, 128-byte swizzle, STAGES-deep ring
//   warp 1      MMA issuer: one thread issues tcgen05.mma (M=128, N=BN, K=16) and commits
//               smem-slot / accumulator-ready mbarriers; also owns the TMEM allocation
//   warps 2..5  epilogue: tcgen05.ld 32x32b per TMEM lane quarter, fused tail, 16-byte stores
// The accumulator is double buffered in TMEM (2 x BN columns) so the epilogue of one tile
// overlaps the main loop of the next.  Every mbarrier wait is bounded (%globaltimer); on
// timeout the CTA raises an abort flag, sets the context's device error word, drains what it
// issued and frees TMEM before returning.
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "tcgen05.cuh"

namespace wam {
namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;           // 64 bf16 = 128 bytes = one swizzle row
constexpr int kThreads = 192;
constexpr int kTileBytesA = kBM * kBK * 2;  // 16 KB
constexpr int kBoxRows = 128;               // TMA box rows of the A operand and wide B tiles

template <int BN>
struct TileCfg {
  static constexpr int kStages = (BN == 256) ? 4 : (BN == 128 ? 6 : 8);
  static constexpr int kBoxB = BN < kBoxRows ? BN : kBoxRows;  // rows per B load
  static constexpr int kTileBytesB = BN * kBK * 2;
  static constexpr int kStageBytes = kTileBytesA + kTileBytesB;
  static constexpr int kTmemCols = 2 * BN;
  static constexpr int kBarrierBytes = 256;
  static constexpr int kSmemBytes = kStages * kStageBytes + kBarrierBytes + 1024;
};

// Fused accumulator read-back for one row segment of 32 columns.
template <int EPI>
WAM_DEV void epilogue32(const EpiArgs& e, int N, int row, int col0, const uint32_t (&r)[32]) {
  float v[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
  if (e.bias != nullptr) {
    const float4* b4 = reinterpret_cast<const float4*>(e.bias + col0);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float4 b = __ldg(b4 + j);
      v[4 * j] += b.x;
      v[4 * j + 1] += b.y;
      v[4 * j + 2] += b.z;
      v[4 * j + 3] += b.w;
    }
  }
  if constexpr (EPI == kEpiGeluBf16) {
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = gelu_tanh_f(v[i]);
  }
  if constexpr (EPI == kEpiBf16 || EPI == kEpiGeluBf16) {
    uint4* dst = reinterpret_cast<uint4*>(static_cast<bf16*>(e.C) + static_cast<int64_t>(row) * N + col0);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      uint4 u;
      __nv_bfloat162 p0 = __floats2bfloat162_rn(v[8 * j + 0], v[8 * j + 1]);
      __nv_bfloat162 p1 = __floats2bfloat162_rn(v[8 * j + 2], v[8 * j + 3]);
      __nv_bfloat162 p2 = __floats2bfloat162_rn(v[8 * j + 4], v[8 * j + 5]);
      __nv_bfloat162 p3 = __floats2bfloat162_rn(v[8 * j + 6], v[8 * j + 7]);
      u.x = *reinterpret_cast<uint32_t*>(&p0);
      u.y = *reinterpret_cast<uint32_t*>(&p1);
      u.z = *reinterpret_cast<uint32_t*>(&p2);
      u.w = *reinterpret_cast<uint32_t*>(&p3);
      dst[j] = u;
    }
  } else if constexpr (EPI == kEpiQkvVt) {
    // q | k columns as bf16 rows; v columns transposed per (item, head) into V^T so that the
    // attention's P.V product reads a K-major operand.  Lanes hold consecutive tokens, so each
    // of the 32 stores of a warp writes 64 contiguous bytes.
    const int d = N / 3;
    if (col0 < 2 * d) {
      uint4* dst = reinterpret_cast<uint4*>(static_cast<bf16*>(e.C) + static_cast<int64_t>(row) * N + col0);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        uint4 u;
        __nv_bfloat162 p0 = __floats2bfloat162_rn(v[8 * j + 0], v[8 * j + 1]);
        __nv_bfloat162 p1 = __floats2bfloat162_rn(v[8 * j + 2], v[8 * j + 3]);
        __nv_bfloat162 p2 = __floats2bfloat162_rn(v[8 * j + 4], v[8 * j + 5]);
        __nv_bfloat162 p3 = __floats2bfloat162_rn(v[8 * j + 6], v[8 * j + 7]);
        u.x = *reinterpret_cast<uint32_t*>(&p0);
        u.y = *reinterpret_cast<uint32_t*>(&p1);
        u.z = *reinterpret_cast<uint32_t*>(&p2);
        u.w = *reinterpret_cast<uint32_t*>(&p3);
        dst[j] = u;
      }
    } else {
      const int cc = col0 - 2 * d;
      const int item = row / e.rows_per_item;
      const int n = row - item * e.rows_per_item;
      bf16* dst = e.vt + (static_cast<int64_t>(item) * d + cc) * e.vt_ld + n;
#pragma unroll
      for (int i = 0; i < 32; ++i) dst[static_cast<int64_t>(i) * e.vt_ld] = __float2bfloat16(v[i]);
    }
  } else if constexpr (EPI == kEpiF32) {
    float4* dst = reinterpret_cast<float4*>(static_cast<float*>(e.C) + static_cast<int64_t>(row) * N + col0);
#pragma unroll
    for (int j = 0; j < 8; ++j) dst[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
  } else {  // kEpiResidF32: h += gate * (acc + bias)
    int item = row / e.rows_per_item;
    if (e.item_map != nullptr) item = e.item_map[item];
    const float4* g4 = reinterpret_cast<const float4*>(e.gate + item * e.gate_stride + col0);
    float4* h4 = reinterpret_cast<float4*>(static_cast<float*>(e.C) + static_cast<int64_t>(row) * N + col0);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float4 g = __ldg(g4 + j);
      float4 h = h4[j];
      h.x = fmaf(g.x, v[4 * j], h.x);
      h.y = fmaf(g.y, v[4 * j + 1], h.y);
      h.z = fmaf(g.z, v[4 * j + 2], h.z);
      h.w = fmaf(g.w, v[4 * j + 3], h.w);
      h4[j] = h;
    }
  }
}

template <int BN, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   int M, int N, int K, EpiArgs e, int* dev_err) {
  using C = TileCfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* tiles = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::kStages * C::kStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + C::kStages;
  uint64_t* tfull = bars + 2 * C::kStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int num_m = (M + kBM - 1) / kBM;
  const int num_n = N / BN;
  const int num_tiles = num_m * num_n;
  const int num_k = K / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), 128);
    }
    mbar_init(smem_u32(drain), 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(C::kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_launch_dependents();

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer ----------------
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
    // The weight operand does not depend on earlier kernels: its first stages are requested
    // before waiting for them, overlapping the previous kernel's tail.
    const int pre = blockIdx.x < num_tiles ? (num_k < C::kStages ? num_k : C::kStages) : 0;
    for (int s = 0; s < pre; ++s) {
      const uint32_t fb = smem_u32(&full[s]);
      const uint32_t b_dst = smem_u32(tiles + s * C::kStageBytes) + kTileBytesA;
      mbar_expect_tx(fb, C::kStageBytes);
#pragma unroll
      for (int h = 0; h < BN / C::kBoxB; ++h)
        tma_load_2d(b_dst + h * C::kBoxB * 128, &tmB, s * kBK, (blockIdx.x / num_m) * BN + h * C::kBoxB, fb);
    }
    pdl_wait();
    int stage = 0;
    uint32_t phase = 0;
    int issued[C::kStages];
    uint32_t issued_phase[C::kStages];
    for (int s = 0; s < C::kStages; ++s) issued[s] = 0, issued_phase[s] = 0;
    bool ok = true;
    bool first = true;
    for (int tile = blockIdx.x; ok && tile < num_tiles; tile += gridDim.x) {
      const int mt = tile % num_m;
      const int nt = tile / num_m;
      for (int kb = 0; kb < num_k; ++kb) {
        if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1u, abort_flag, dev_err)) {
          ok = false;
          break;
        }
        const uint32_t fb = smem_u32(&full[stage]);
        const uint32_t a_dst = smem_u32(tiles + stage * C::kStageBytes);
        const uint32_t b_dst = a_dst + kTileBytesA;
        if (!(first && kb < pre)) {
          mbar_expect_tx(fb, C::kStageBytes);
#pragma unroll
          for (int h = 0; h < BN / C::kBoxB; ++h)
            tma_load_2d(b_dst + h * C::kBoxB * 128, &tmB, kb * kBK, nt * BN + h * C::kBoxB, fb);
        }
        tma_load_2d(a_dst, &tmA, kb * kBK, mt * kBM, fb);
        issued[stage] = 1;
        issued_phase[stage] = phase;
        if (++stage == C::kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      first = false;
    }
    if (!ok) {
      // Drain: let every copy this thread issued land before the CTA releases its smem.
      for (int s = 0; s < C::kStages; ++s) {
        if (!issued[s]) continue;
        const uint32_t fb = smem_u32(&full[s]);
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(fb, issued_phase[s]) && globaltimer_ns() - t0 < kWaitLimitNs) {
        }
      }
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    pdl_wait();
    const uint32_t idesc = idesc_bf16(kBM, BN);
    int stage = 0;
    uint32_t phase = 0;
    int it = 0;
    bool ok = true;
    bool issued_any = false;
    for (int tile = blockIdx.x; ok && tile < num_tiles; tile += gridDim.x, ++it) {
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      if (!mbar_wait(smem_u32(&tempty[acc]), acc_phase ^ 1u, abort_flag, dev_err)) {
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
        const uint32_t b0 = a0 + kTileBytesA;
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k) {
          umma_bf16(d_tmem, sw128_desc(a0 + k * 32), sw128_desc(b0 + k * 32), idesc,
                    (kb | k) != 0 ? 1u : 0u);
        }
        issued_any = true;
        umma_commit(smem_u32(&empty[stage]));
        if (++stage == C::kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) break;
      umma_commit(smem_u32(&tfull[acc]));
    }
    if (!ok && issued_any) {
      // Drain: wait for every MMA this thread issued before TMEM is released.
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
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++it) {
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      // One lane waits; the warp then proceeds together (tcgen05.ld is warp-collective).
      int ok = 1;
      if (lane == 0) ok = mbar_wait(smem_u32(&tfull[acc]), acc_phase, abort_flag, dev_err) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      __syncwarp();
      if (!ok) break;
      tc_fence_after();
      const int mt = tile % num_m;
      const int nt = tile / num_m;
      const int row = mt * kBM + quarter * 32 + lane;
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN;
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(taddr + c * 32, r);
        if (row < M) epilogue32<EPI>(e, N, row, nt * BN + c * 32, r);
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&tempty[acc]));
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(C::kTmemCols)
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

template <int BN, int EPI>
cudaError_t launch(const CUtensorMap& ta, const CUtensorMap& tb, int M, int N, int K,
                   const EpiArgs& e, int num_sms, int* dev_err, cudaStream_t s) {
  using C = TileCfg<BN>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t err = cudaFuncSetAttribute(gemm_tc_kernel<BN, EPI>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
    if (err != cudaSuccess) return err;
    attr_set = true;
  }
  const int tiles = ((M + kBM - 1) / kBM) * (N / BN);
  const int grid = tiles < num_sms ? tiles : num_sms;
  return launch_pdl(gemm_tc_kernel<BN, EPI>, dim3(grid), dim3(kThreads), C::kSmemBytes, s, ta, tb, M, N, K, e,
                    dev_err);
}

template <int BN>
cudaError_t dispatch_epi(const CUtensorMap& ta, const CUtensorMap& tb, int M, int N, int K,
                         int epi, const EpiArgs& e, int num_sms, int* dev_err, cudaStream_t s) {
  switch (epi) {
    case kEpiBf16: return launch<BN, kEpiBf16>(ta, tb, M, N, K, e, num_sms, dev_err, s);
    case kEpiGeluBf16: return launch<BN, kEpiGeluBf16>(ta, tb, M, N, K, e, num_sms, dev_err, s);
    case kEpiResidF32: return launch<BN, kEpiResidF32>(ta, tb, M, N, K, e, num_sms, dev_err, s);
    case kEpiF32: return launch<BN, kEpiF32>(ta, tb, M, N, K, e, num_sms, dev_err, s);
    case kEpiQkvVt: return launch<BN, kEpiQkvVt>(ta, tb, M, N, K, e, num_sms, dev_err, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

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

int tc_encode_kmajor_bf16_box64(CUtensorMap* map, const void* base, uint64_t rows, uint64_t K) {
  return tc_encode_bf16_box(map, base, rows, K, K, kBK, 64);
}

int tc_encode_kmajor_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t K) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (fn == nullptr) return -1;
  if ((reinterpret_cast<uintptr_t>(base) & 15u) != 0 || (K * 2) % 16 != 0) return -2;
  cuuint64_t dims[2] = {K, rows};
  cuuint64_t strides[1] = {K * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(kBoxRows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : -3;
}

cudaError_t tc_gemm(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap* tb64, int M, int N, int K,
                    int epi, const EpiArgs& e, int num_sms, int* dev_err, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  if (K % kBK != 0 || N % 128 != 0) return cudaErrorInvalidValue;
  // Tile width: each CTA's operand delivery (about 17 cycles per KB of A + B tile per K block)
  // bounds these kernels, so pick the width that minimises waves x bytes per K block:
  // narrow tiles spread a small projection over more SMs, wide ones halve the A re-reads.
  const int m_tiles = (M + kBM - 1) / kBM;
  auto cost = [&](int bn) {
    const long tiles = static_cast<long>(m_tiles) * (N / bn);
    return ((tiles + num_sms - 1) / num_sms) * (16 + bn / 8);
  };
  int bn = 128;
  if (N % 256 == 0 && cost(256) <= cost(bn)) bn = 256;
  if (tb64 != nullptr && cost(64) < cost(bn)) bn = 64;
  if (bn == 64) return dispatch_epi<64>(ta, *tb64, M, N, K, epi, e, num_sms, dev_err, s);
  if (bn == 256) return dispatch_epi<256>(ta, tb, M, N, K, epi, e, num_sms, dev_err, s);
  return dispatch_epi<128>(ta, tb, M, N, K, epi, e, num_sms, dev_err, s);
}

}  // namespace wam
