// Full bidirectional multi-head attention over the joint [obs ; video ; action] sequence.
//
// bf16 path: flash-style single pass with an online softmax.  A 128-thread CTA owns 64 query
// rows of one (item, head); each warp owns 16 rows.  K/V tiles of 64 keys are double
// buffered in shared memory with cp.async; Q K^T and P V run on m16n8k16 bf16 tensor-core
// MMAs with fp32 accumulation; P never leaves registers.  Head dims 64 and 72 are supported
// (72 = the bimanual workload) by zero-padding the contraction to a multiple of 16.
//
// fp32 path: one warp per (query row, head, item), lanes splitting the head dimension, a
// streaming online softmax over the keys.  Used by the fp32 precision mode only.
#include <math_constants.h>

#include "common.cuh"

namespace wam {
namespace {

WAM_DEV uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

WAM_DEV void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n)
               : "memory");
}
WAM_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
WAM_DEV void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

WAM_DEV void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
WAM_DEV void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
WAM_DEV void ldsm_x2_t(uint32_t addr, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];"
               : "=r"(r0), "=r"(r1)
               : "r"(addr));
}

WAM_DEV void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

WAM_DEV uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

template <int DH>
struct AttnCfg {
  static constexpr int kDHP = (DH + 15) / 16 * 16;  // contraction width of Q K^T
  static constexpr int kLds = kDHP + 8;             // smem row stride (odd number of 16 B)
  static constexpr int kBQ = 64;
  static constexpr int kBKV = 64;
  static constexpr int kChunks = DH / 8;            // 16-byte chunks per row
  static constexpr int kKS = kDHP / 16;             // k-steps of Q K^T
  static constexpr int kNTO = DH / 8;               // n-tiles of O
  static constexpr int kTile = kBKV * kLds;
  static constexpr int kSmem = (kBQ * kLds + 4 * kTile) * 2;
};

template <int DH>
__global__ void __launch_bounds__(128) attn_bf16_kernel(const bf16* __restrict__ qkv,
                                                        bf16* __restrict__ out, int N, int d,
                                                        float scale_log2) {
  using C = AttnCfg<DH>;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  bf16* sQ = reinterpret_cast<bf16*>(smem_raw);
  bf16* sK = sQ + C::kBQ * C::kLds;
  bf16* sV = sK + 2 * C::kTile;
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int q0 = blockIdx.x * C::kBQ;
  pdl_wait();
  pdl_launch_dependents();
  const int h = blockIdx.y;
  const int b = blockIdx.z;
  const int64_t ld = 3 * static_cast<int64_t>(d);
  const bf16* base = qkv + static_cast<int64_t>(b) * N * ld + h * DH;

  if constexpr (C::kDHP > DH) {
    // Zero the contraction padding of Q and both K buffers; the tile loads never touch it.
    for (int i = tid; i < 3 * C::kBQ; i += 128) {
      const int t = i / C::kBQ, r = i % C::kBQ;
      bf16* row = (t == 0 ? sQ : sK + (t - 1) * C::kTile) + r * C::kLds;
      for (int c = DH; c < C::kDHP; ++c) row[c] = __float2bfloat16(0.0f);
    }
  }

  auto load_tile = [&](bf16* dst, int row0, int col_off) {
    for (int i = tid; i < 64 * C::kChunks; i += 128) {
      const int r = i / C::kChunks, c = i % C::kChunks;
      const int gr = row0 + r;
      const bool valid = gr < N;
      const bf16* src = base + static_cast<int64_t>(valid ? gr : 0) * ld + col_off + c * 8;
      cp_async16(smem_u32(dst + r * C::kLds + c * 8), src, valid);
    }
  };

  const int nkv = (N + C::kBKV - 1) / C::kBKV;
  load_tile(sQ, q0, 0);
  load_tile(sK, 0, d);
  load_tile(sV, 0, 2 * d);
  cp_async_commit();

  float o[C::kNTO][4];
#pragma unroll
  for (int i = 0; i < C::kNTO; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.0f;
  float m0 = -CUDART_INF_F, m1 = -CUDART_INF_F, l0 = 0.0f, l1 = 0.0f;
  uint32_t qf[C::kKS][4];

  for (int j = 0; j < nkv; ++j) {
    const int buf = j & 1;
    if (j + 1 < nkv) {
      load_tile(sK + (buf ^ 1) * C::kTile, (j + 1) * C::kBKV, d);
      load_tile(sV + (buf ^ 1) * C::kTile, (j + 1) * C::kBKV, 2 * d);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (j == 0) {
#pragma unroll
      for (int ks = 0; ks < C::kKS; ++ks) {
        const int r = warp * 16 + (lane & 15);
        const int c = ks * 16 + (lane >> 4) * 8;
        ldsm_x4(smem_u32(sQ + r * C::kLds + c), qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3]);
      }
    }
    const bf16* ks_ = sK + buf * C::kTile;
    const bf16* vs_ = sV + buf * C::kTile;

    float s[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.0f;
#pragma unroll
    for (int ks = 0; ks < C::kKS; ++ks) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        const int key = np * 16 + (lane >> 4) * 8 + (lane & 7);
        const int col = ks * 16 + ((lane >> 3) & 1) * 8;
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(ks_ + key * C::kLds + col), b0, b1, b2, b3);
        mma16816(s[2 * np], qf[ks], b0, b1);
        mma16816(s[2 * np + 1], qf[ks], b2, b3);
      }
    }
    if ((j + 1) * C::kBKV > N) {
#pragma unroll
      for (int nt = 0; nt < 8; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = j * C::kBKV + nt * 8 + 2 * (lane & 3) + (e & 1);
          if (key >= N) s[nt][e] = -CUDART_INF_F;
        }
    }
    float mx0 = -CUDART_INF_F, mx1 = -CUDART_INF_F;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      mx0 = fmaxf(mx0, fmaxf(s[nt][0], s[nt][1]));
      mx1 = fmaxf(mx1, fmaxf(s[nt][2], s[nt][3]));
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float mn0 = fmaxf(m0, mx0 * scale_log2);
    const float mn1 = fmaxf(m1, mx1 * scale_log2);
    const float c0 = exp2f(m0 - mn0);
    const float c1 = exp2f(m1 - mn1);
    m0 = mn0;
    m1 = mn1;
    float rs0 = 0.0f, rs1 = 0.0f;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      s[nt][0] = exp2f(fmaf(s[nt][0], scale_log2, -mn0));
      s[nt][1] = exp2f(fmaf(s[nt][1], scale_log2, -mn0));
      s[nt][2] = exp2f(fmaf(s[nt][2], scale_log2, -mn1));
      s[nt][3] = exp2f(fmaf(s[nt][3], scale_log2, -mn1));
      rs0 += s[nt][0] + s[nt][1];
      rs1 += s[nt][2] + s[nt][3];
    }
    l0 = l0 * c0 + rs0;
    l1 = l1 * c1 + rs1;
#pragma unroll
    for (int nt = 0; nt < C::kNTO; ++nt) {
      o[nt][0] *= c0;
      o[nt][1] *= c0;
      o[nt][2] *= c1;
      o[nt][3] *= c1;
    }
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {
      const uint32_t a[4] = {pack_bf16(s[2 * ks][0], s[2 * ks][1]),
                             pack_bf16(s[2 * ks][2], s[2 * ks][3]),
                             pack_bf16(s[2 * ks + 1][0], s[2 * ks + 1][1]),
                             pack_bf16(s[2 * ks + 1][2], s[2 * ks + 1][3])};
      const int key = ks * 16 + ((lane >> 3) & 1) * 8 + (lane & 7);
#pragma unroll
      for (int np = 0; np < C::kNTO / 2; ++np) {
        const int col = np * 16 + (lane >> 4) * 8;
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(smem_u32(vs_ + key * C::kLds + col), b0, b1, b2, b3);
        mma16816(o[2 * np], a, b0, b1);
        mma16816(o[2 * np + 1], a, b2, b3);
      }
      if constexpr ((C::kNTO & 1) != 0) {
        uint32_t b0, b1;
        ldsm_x2_t(smem_u32(vs_ + key * C::kLds + (C::kNTO - 1) * 8), b0, b1);
        mma16816(o[C::kNTO - 1], a, b0, b1);
      }
    }
    __syncthreads();
  }

  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const float inv0 = 1.0f / l0;
  const float inv1 = 1.0f / l1;
  const int r0 = q0 + warp * 16 + (lane >> 2);
  const int r1 = r0 + 8;
  bf16* ob = out + static_cast<int64_t>(b) * N * d + h * DH;
#pragma unroll
  for (int nt = 0; nt < C::kNTO; ++nt) {
    const int col = nt * 8 + 2 * (lane & 3);
    if (r0 < N)
      *reinterpret_cast<uint32_t*>(ob + static_cast<int64_t>(r0) * d + col) =
          pack_bf16(o[nt][0] * inv0, o[nt][1] * inv0);
    if (r1 < N)
      *reinterpret_cast<uint32_t*>(ob + static_cast<int64_t>(r1) * d + col) =
          pack_bf16(o[nt][2] * inv1, o[nt][3] * inv1);
  }
}

__global__ void __launch_bounds__(256) attn_f32_kernel(const float* __restrict__ qkv,
                                                       float* __restrict__ out, int B, int N,
                                                       int d, int H, float scale) {
  pdl_wait();
  pdl_launch_dependents();
  const int64_t gw = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (gw >= static_cast<int64_t>(B) * H * N) return;
  const int i = static_cast<int>(gw % N);
  const int h = static_cast<int>((gw / N) % H);
  const int b = static_cast<int>(gw / (static_cast<int64_t>(N) * H));
  const int dh = d / H;
  const int64_t ld = 3 * static_cast<int64_t>(d);
  const float* qrow = qkv + (static_cast<int64_t>(b) * N + i) * ld + h * dh;
  const float* kbase = qkv + static_cast<int64_t>(b) * N * ld + d + h * dh;
  const float* vbase = kbase + d;
  float q[4], o[4];
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int c = lane + 32 * r;
    q[r] = c < dh ? qrow[c] : 0.0f;
    o[r] = 0.0f;
  }
  float m = -CUDART_INF_F, l = 0.0f;
  for (int j = 0; j < N; ++j) {
    const float* kr = kbase + static_cast<int64_t>(j) * ld;
    const float* vr = vbase + static_cast<int64_t>(j) * ld;
    float p = 0.0f;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int c = lane + 32 * r;
      if (c < dh) p = fmaf(q[r], kr[c], p);
    }
    p = warp_sum(p) * scale;
    const float mn = fmaxf(m, p);
    const float corr = expf(m - mn);
    const float e = expf(p - mn);
    l = l * corr + e;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int c = lane + 32 * r;
      if (c < dh) o[r] = fmaf(o[r], corr, e * vr[c]);
    }
    m = mn;
  }
  float* orow = out + (static_cast<int64_t>(b) * N + i) * d + h * dh;
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int c = lane + 32 * r;
    if (c < dh) orow[c] = o[r] / l;
  }
}

template <int DH>
cudaError_t launch_bf16(const bf16* qkv, bf16* out, int B, int N, int d, int H, cudaStream_t s) {
  using C = AttnCfg<DH>;
  static PerDeviceSmem smem_rec;  // contexts may run on several host threads and devices
  const cudaError_t e = ensure_max_smem(smem_rec, attn_bf16_kernel<DH>, C::kSmem);
  if (e != cudaSuccess) return e;
  dim3 grid((N + C::kBQ - 1) / C::kBQ, H, B);
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(DH));
  return launch_pdl(attn_bf16_kernel<DH>, grid, dim3(128), C::kSmem, s, qkv, out, N, d, scale_log2);
}

}  // namespace

bool attention_bf16_supported(int head_dim) { return head_dim == 64 || head_dim == 72; }

cudaError_t attention_bf16(const bf16* qkv, bf16* out, int B, int N, int d, int H,
                           cudaStream_t s) {
  if (B <= 0 || N <= 0) return cudaSuccess;
  switch (d / H) {
    case 64: return launch_bf16<64>(qkv, out, B, N, d, H, s);
    case 72: return launch_bf16<72>(qkv, out, B, N, d, H, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t attention_f32(const float* qkv, float* out, int B, int N, int d, int H,
                          cudaStream_t s) {
  if (B <= 0 || N <= 0) return cudaSuccess;
  if (d / H > 128) return cudaErrorInvalidValue;
  const int64_t warps = static_cast<int64_t>(B) * H * N;
  const int64_t blocks = (warps * 32 + 255) / 256;
  return launch_pdl(attn_f32_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, s, qkv, out, B, N, d, H,
                    1.0f / sqrtf(static_cast<float>(d / H)));
}

}  // namespace wam
