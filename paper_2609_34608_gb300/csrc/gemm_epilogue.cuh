// Accumulator read-back of the tensor-core GEMMs: the DiT block's elementwise tail applied to
// one 32-column segment of an output row (bias, GELU, adaLN-gated residual, the V^T transpose of
// the QKV projection), shared by the per-projection GEMM and the fused row-chain kernel.
#pragma once

#include "common.cuh"

namespace wam {
namespace {

// Fused accumulator read-back for one row segment of 32 columns.
template <int EPI>
WAM_DEV void epilogue32(const EpiArgs& e, int N, int row, int col0, const uint32_t (&r)[32]) {
  float v[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
  if (e.bias != nullptr) {
    // a plain load: the fused row-chain kernel passes a staged copy in shared memory
    const float4* b4 = reinterpret_cast<const float4*>(e.bias + col0);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float4 b = b4[j];
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

}  // namespace
}  // namespace wam
