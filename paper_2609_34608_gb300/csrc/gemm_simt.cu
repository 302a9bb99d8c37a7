// float32 SIMT projection for the library's fp32 precision mode (tcgen05 has no exact fp32
// kind).  C = A[M,K] . Wt[N,K]^T with the same fused epilogues as the tensor-core GEMM.
// 64x64 output tile per 256-thread block, 4x4 register micro-tile, K staged 16 at a time.
#include "common.cuh"

namespace wam {
namespace {

constexpr int kT = 64;
constexpr int kKc = 16;

template <int EPI>
WAM_DEV void store_one(const EpiArgs& e, int N, int row, int col, float acc) {
  float v = acc + (e.bias != nullptr ? e.bias[col] : 0.0f);
  if constexpr (EPI == kEpiGeluBf16) v = gelu_tanh_f(v);
  float* C = static_cast<float*>(e.C);
  if constexpr (EPI == kEpiResidF32) {
    int item = row / e.rows_per_item;
    if (e.item_map != nullptr) item = e.item_map[item];
    const float g = e.gate[item * e.gate_stride + col];
    C[static_cast<int64_t>(row) * N + col] = fmaf(g, v, C[static_cast<int64_t>(row) * N + col]);
  } else {
    C[static_cast<int64_t>(row) * N + col] = v;
  }
}

// In fp32 mode the "bf16" epilogues store float32 (the activation type of that mode).
template <int EPI>
__global__ void __launch_bounds__(256) simt_gemm_kernel(const float* __restrict__ A,
                                                        const float* __restrict__ Wt, int M, int N,
                                                        int K, EpiArgs e) {
  __shared__ float As[kKc][kT + 4];
  __shared__ float Bs[kKc][kT + 4];
  pdl_wait();
  pdl_launch_dependents();
  const int tx = threadIdx.x & 15;
  const int ty = threadIdx.x >> 4;
  const int m0 = blockIdx.y * kT;
  const int n0 = blockIdx.x * kT;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;

  for (int k0 = 0; k0 < K; k0 += kKc) {
    for (int i = threadIdx.x; i < kT * kKc; i += 256) {
      const int r = i / kKc, c = i % kKc;
      const int gm = m0 + r, gn = n0 + r, gk = k0 + c;
      As[c][r] = (gm < M && gk < K) ? A[static_cast<int64_t>(gm) * K + gk] : 0.0f;
      Bs[c][r] = (gn < N && gk < K) ? Wt[static_cast<int64_t>(gn) * K + gk] : 0.0f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kKc; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int row = m0 + ty * 4 + i;
    if (row >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int col = n0 + tx * 4 + j;
      if (col < N) store_one<EPI>(e, N, row, col, acc[i][j]);
    }
  }
}

}  // namespace

cudaError_t simt_gemm(const float* A, const float* Wt, int M, int N, int K, int epi,
                      const EpiArgs& e, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  dim3 grid((N + kT - 1) / kT, (M + kT - 1) / kT);
  switch (epi) {
    case kEpiBf16: return launch_pdl(simt_gemm_kernel<kEpiBf16>, grid, dim3(256), 0, s, A, Wt, M, N, K, e);
    case kEpiGeluBf16: return launch_pdl(simt_gemm_kernel<kEpiGeluBf16>, grid, dim3(256), 0, s, A, Wt, M, N, K, e);
    case kEpiResidF32: return launch_pdl(simt_gemm_kernel<kEpiResidF32>, grid, dim3(256), 0, s, A, Wt, M, N, K, e);
    case kEpiF32: return launch_pdl(simt_gemm_kernel<kEpiF32>, grid, dim3(256), 0, s, A, Wt, M, N, K, e);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace wam
