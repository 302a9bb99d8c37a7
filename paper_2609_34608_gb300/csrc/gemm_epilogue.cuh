// Accumulator read-back of the tensor-core GEMMs: the DiT block's elementwise tail applied to
// one 32-column segment of an output row (bias, GELU, adaLN-gated residual, the V^T transpose of
// the QKV projection), shared by the per-projection GEMM and the fused row-chain kernel.
#pragma once

#include "common.cuh"

namespace wam {
namespace {

// GELU (tanh form) for the bf16 tail: 0.5 x (1 + tanh(u)) = x / (1 + exp(-2u)) with
// u = sqrt(2/pi) (x + 0.044715 x^3), evaluated with the hardware base-2 exponential and
// reciprocal (two MUFU operations; relative error a few 1e-6, far below the bf16 rounding of
// the result).  Large negative x gives exp -> inf and the result -> -0, large positive x gives x.
WAM_DEV float gelu_tanh_bf16tail(float x) {
  constexpr float kC = -2.302208198144325f;   // -2 log2(e) sqrt(2/pi)
  const float t = kC * x * fmaf(0.044715f, x * x, 1.0f);
  float e, r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(t));
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(1.0f + e));
  return x * r;
}

// What the fused tail of one 16-column row segment reads from memory besides the accumulator:
// the bias, and for the gated residual the gate and the residual itself.  The GEMM loads it one
// segment pair ahead of the accumulator read-back (the first pair before the accumulator is
// ready), so these loads' latency overlaps the main loop and the previous segments' tail.
struct EpiIn {
  float4 b[4];
  float4 g[4];
  float4 h[4];
};

template <int EPI>
WAM_DEV void epi_load16(const EpiArgs& e, int N, int row, int col0, EpiIn& in) {
  if (e.bias != nullptr) {
    // a plain load: the fused row-chain kernel passes a staged copy in shared memory
    const float4* b4 = reinterpret_cast<const float4*>(e.bias + col0);
#pragma unroll
    for (int j = 0; j < 4; ++j) in.b[j] = b4[j];
  }
  if constexpr (EPI == kEpiResidF32) {
    int item = row / e.rows_per_item;
    if (e.item_map != nullptr) item = e.item_map[item];
    const float4* g4 = reinterpret_cast<const float4*>(e.gate + item * e.gate_stride + col0);
    const float4* h4 = reinterpret_cast<const float4*>(static_cast<const float*>(e.C) + static_cast<int64_t>(row) * N + col0);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      in.g[j] = __ldg(g4 + j);
      in.h[j] = h4[j];
    }
  }
}

WAM_DEV uint4 pack_bf16x8(const float* v) {
  uint4 u;
  __nv_bfloat162 p0 = __floats2bfloat162_rn(v[0], v[1]);
  __nv_bfloat162 p1 = __floats2bfloat162_rn(v[2], v[3]);
  __nv_bfloat162 p2 = __floats2bfloat162_rn(v[4], v[5]);
  __nv_bfloat162 p3 = __floats2bfloat162_rn(v[6], v[7]);
  u.x = *reinterpret_cast<uint32_t*>(&p0);
  u.y = *reinterpret_cast<uint32_t*>(&p1);
  u.z = *reinterpret_cast<uint32_t*>(&p2);
  u.w = *reinterpret_cast<uint32_t*>(&p3);
  return u;
}

// The fused tail of one 16-column row segment: r = the fp32 accumulator, in = its epi_load16.
template <int EPI>
WAM_DEV void epi_store16(const EpiArgs& e, int N, int row, int col0, const uint32_t* r, const EpiIn& in) {
  float v[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
  if (e.bias != nullptr) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      v[4 * j] += in.b[j].x;
      v[4 * j + 1] += in.b[j].y;
      v[4 * j + 2] += in.b[j].z;
      v[4 * j + 3] += in.b[j].w;
    }
  }
  if constexpr (EPI == kEpiGeluBf16) {
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = gelu_tanh_bf16tail(v[i]);
  }
  if constexpr (EPI == kEpiBf16 || EPI == kEpiGeluBf16) {
    uint4* dst = reinterpret_cast<uint4*>(static_cast<bf16*>(e.C) + static_cast<int64_t>(row) * N + col0);
    dst[0] = pack_bf16x8(v);
    dst[1] = pack_bf16x8(v + 8);
  } else if constexpr (EPI == kEpiQkvVt) {
    // q | k columns as bf16 rows; v columns transposed per (item, head) into V^T so that the
    // attention's P.V product reads a K-major operand.  Lanes hold consecutive tokens, so each
    // of the 16 stores of a warp writes 64 contiguous bytes.
    const int d = N / 3;
    if (col0 < 2 * d) {
      uint4* dst = reinterpret_cast<uint4*>(static_cast<bf16*>(e.C) + static_cast<int64_t>(row) * N + col0);
      dst[0] = pack_bf16x8(v);
      dst[1] = pack_bf16x8(v + 8);
    } else {
      const int cc = col0 - 2 * d;
      const int item = row / e.rows_per_item;
      const int n = row - item * e.rows_per_item;
      bf16* dst = e.vt + (static_cast<int64_t>(item) * d + cc) * e.vt_ld + n;
#pragma unroll
      for (int i = 0; i < 16; ++i) dst[static_cast<int64_t>(i) * e.vt_ld] = __float2bfloat16(v[i]);
    }
  } else if constexpr (EPI == kEpiF32) {
    float4* dst = reinterpret_cast<float4*>(static_cast<float*>(e.C) + static_cast<int64_t>(row) * N + col0);
#pragma unroll
    for (int j = 0; j < 4; ++j) dst[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
  } else {  // kEpiResidF32: h += gate * (acc + bias)
    float4* h4 = reinterpret_cast<float4*>(static_cast<float*>(e.C) + static_cast<int64_t>(row) * N + col0);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float4 g = in.g[j];
      float4 h = in.h[j];
      h.x = fmaf(g.x, v[4 * j], h.x);
      h.y = fmaf(g.y, v[4 * j + 1], h.y);
      h.z = fmaf(g.z, v[4 * j + 2], h.z);
      h.w = fmaf(g.w, v[4 * j + 3], h.w);
      h4[j] = h;
    }
  }
}

// Fused accumulator read-back for one row segment of 32 columns (loads, then the tail).
template <int EPI>
WAM_DEV void epilogue32(const EpiArgs& e, int N, int row, int col0, const uint32_t (&r)[32]) {
  EpiIn a, b;
  epi_load16<EPI>(e, N, row, col0, a);
  epi_load16<EPI>(e, N, row, col0 + 16, b);
  epi_store16<EPI>(e, N, row, col0, r, a);
  epi_store16<EPI>(e, N, row, col0 + 16, r + 16, b);
}

}  // namespace
}  // namespace wam
