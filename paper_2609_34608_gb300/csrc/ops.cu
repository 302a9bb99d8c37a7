// Kernel-level entry points (wam_ops.h): single hot-path kernels on caller-owned device
// buffers, for parity tests and kernel benchmarks.  They allocate no device memory.
#include <string>

#include "kernels.cuh"
#include "wam.h"
#include "wam_ops.h"

using namespace wam;

namespace {

thread_local std::string g_op_err;

int op_fail(int code, const std::string& msg) {
  g_op_err = msg;
  return code;
}

int op_cuda(const char* what, cudaError_t e) {
  return op_fail(WAM_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

EpiArgs make_epi(const float* bias, void* C, const float* gate, int64_t gstride, int rpi) {
  EpiArgs e;
  e.bias = bias;
  e.C = C;
  e.gate = gate;
  e.gate_stride = gstride;
  e.rows_per_item = rpi > 0 ? rpi : 1;
  e.item_map = nullptr;
  e.vt = nullptr;
  e.vt_ld = 0;
  return e;
}

int check_gemm_args(const void* A, const void* Wt, void* C, int M, int N, int K, int epi,
                    const float* gate, int rpi) {
  if (A == nullptr || Wt == nullptr || C == nullptr) return op_fail(WAM_ERR_INVALID_ARG, "null operand");
  if (M < 0 || N <= 0 || K <= 0) return op_fail(WAM_ERR_INVALID_ARG, "bad GEMM shape");
  if (epi < WAM_EPI_BF16 || epi > WAM_EPI_F32) return op_fail(WAM_ERR_INVALID_ARG, "unknown epilogue");
  if (epi == WAM_EPI_RESID_F32 && (gate == nullptr || rpi <= 0)) return op_fail(WAM_ERR_INVALID_ARG, "RESID needs gate and rows_per_item");
  return WAM_OK;
}

}  // namespace

namespace wam {
void set_op_error(const std::string& msg) { g_op_err = msg; }
}  // namespace wam

extern "C" {

const char* wam_op_last_error(void) { return g_op_err.c_str(); }

int wam_op_gemm_bf16(const void* A, const void* Wt, const float* bias, void* C, int32_t M, int32_t N,
                     int32_t K, int32_t epilogue, const float* gate, int64_t gate_stride,
                     int32_t rows_per_item, void* stream) {
  return wam_op_gemm_bf16_plan(A, Wt, bias, C, M, N, K, epilogue, gate, gate_stride, rows_per_item, 0, 0, 0, nullptr,
                               0, stream);
}

size_t wam_op_gemm_workspace_bytes(void) {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 0;
  return tc_gemm_workspace_bytes(sms);
}

int wam_op_gemm_plan(int32_t M, int32_t N, int32_t K, int32_t residual, int32_t num_sms, int32_t* tile_n,
                     int32_t* cta_pairs) {
  if (M < 1 || N < 128 || N % 128 != 0 || K < 64 || K % 64 != 0 || num_sms < 1 || tile_n == nullptr ||
      cta_pairs == nullptr)
    return op_fail(WAM_ERR_INVALID_ARG, "bad GEMM plan query");
  // a context's projections: 64-wide tiles for the residual ones, 64-row boxes on every weight
  const GemmPlan p = tc_gemm_plan(M, N, K, residual != 0, true, num_sms);
  *tile_n = p.bn;
  *cta_pairs = p.mc == 3 ? 1 : 0;
  return WAM_OK;
}

int wam_op_gemm_bf16_plan(const void* A, const void* Wt, const float* bias, void* C, int32_t M, int32_t N,
                          int32_t K, int32_t epilogue, const float* gate, int64_t gate_stride,
                          int32_t rows_per_item, int32_t tile_n, int32_t k_splits, int32_t cluster,
                          void* workspace, size_t workspace_bytes, void* stream) {
  int r = check_gemm_args(A, Wt, C, M, N, K, epilogue, gate, rows_per_item);
  if (r != WAM_OK) return r;
  if (K % 64 != 0 || N % 128 != 0) return op_fail(WAM_ERR_UNSUPPORTED, "needs K % 64 == 0 and N % 128 == 0");
  if (!aligned16(A) || !aligned16(Wt) || !aligned16(C) || (bias && !aligned16(bias)) || (gate && !aligned16(gate)) ||
      (gate && gate_stride % 4 != 0))
    return op_fail(WAM_ERR_INVALID_ARG, "operands must be 16-byte aligned");
  if (tile_n != 0 && tile_n != 64 && tile_n != 128 && tile_n != 256)
    return op_fail(WAM_ERR_INVALID_ARG, "tile_n must be 0, 64, 128 or 256");
  if (k_splits < 0 || k_splits > 4) return op_fail(WAM_ERR_INVALID_ARG, "k_splits must be 0 .. 4");
  if (cluster < 0 || cluster > 3) return op_fail(WAM_ERR_INVALID_ARG, "cluster must be 0, 1, 2 or 3");
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return op_cuda("device query", e);
  const size_t need = tc_gemm_workspace_bytes(sms);
  if (workspace != nullptr && (workspace_bytes < need || !aligned16(workspace)))
    return op_fail(WAM_ERR_INVALID_ARG, "workspace smaller than wam_op_gemm_workspace_bytes() or unaligned");
  GemmOperand ta, tb;
  if (tc_encode_gemm_operand(&ta, A, static_cast<uint64_t>(M > 0 ? M : 1), K, true) != 0 ||
      tc_encode_gemm_operand(&tb, Wt, N, K, true) != 0)
    return op_fail(WAM_ERR_CUDA, "cuTensorMapEncodeTiled failed");
  SplitWorkspace ws{nullptr, nullptr, 0};
  if (workspace != nullptr) {
    const size_t counters_bytes = static_cast<size_t>(sms) * sizeof(int);
    ws = SplitWorkspace{static_cast<float*>(workspace),
                        reinterpret_cast<int*>(static_cast<uint8_t*>(workspace) + need - counters_bytes),
                        need - counters_bytes};
  }
  const GemmPlan plan{tile_n, tile_n == 0 ? 0 : (k_splits < 1 ? 1 : k_splits), cluster};
  if (plan.bn == 0 && k_splits > 1) return op_fail(WAM_ERR_INVALID_ARG, "k_splits needs an explicit tile_n");
  e = tc_gemm(ta, tb, M, N, K, epilogue, make_epi(bias, C, gate, gate_stride, rows_per_item), sms, nullptr,
              static_cast<cudaStream_t>(stream), workspace != nullptr ? &ws : nullptr, plan);
  if (e == cudaErrorInvalidValue)
    return op_fail(WAM_ERR_UNSUPPORTED, "tile width / K split not possible for this shape (K ranges must divide "
                                        "the K stages, all units must fit one wave, a split needs a workspace)");
  return e == cudaSuccess ? WAM_OK : op_cuda("tcgen05 GEMM launch", e);
}

int wam_op_gemm_f32(const float* A, const float* Wt, const float* bias, float* C, int32_t M, int32_t N,
                    int32_t K, int32_t epilogue, const float* gate, int64_t gate_stride,
                    int32_t rows_per_item, void* stream) {
  int r = check_gemm_args(A, Wt, C, M, N, K, epilogue, gate, rows_per_item);
  if (r != WAM_OK) return r;
  cudaError_t e = simt_gemm(A, Wt, M, N, K, epilogue, make_epi(bias, C, gate, gate_stride, rows_per_item),
                            static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? WAM_OK : op_cuda("SIMT GEMM launch", e);
}

int wam_op_attention(const void* qkv, void* out, int32_t B, int32_t N, int32_t d, int32_t n_heads,
                     int32_t precision, void* stream) {
  if (qkv == nullptr || out == nullptr || B < 0 || N < 0 || d <= 0 || n_heads <= 0 || d % n_heads != 0)
    return op_fail(WAM_ERR_INVALID_ARG, "bad attention arguments");
  cudaError_t e;
  if (precision == WAM_PREC_BF16) {
    if (!attention_bf16_supported(d / n_heads)) return op_fail(WAM_ERR_UNSUPPORTED, "head dim must be 64 or 72");
    if (!aligned16(qkv) || !aligned16(out)) return op_fail(WAM_ERR_INVALID_ARG, "16-byte alignment required");
    e = attention_bf16(static_cast<const bf16*>(qkv), static_cast<bf16*>(out), B, N, d, n_heads,
                       static_cast<cudaStream_t>(stream));
  } else if (precision == WAM_PREC_FP32) {
    if (d / n_heads > 128) return op_fail(WAM_ERR_UNSUPPORTED, "head dim must be <= 128");
    e = attention_f32(static_cast<const float*>(qkv), static_cast<float*>(out), B, N, d, n_heads,
                      static_cast<cudaStream_t>(stream));
  } else {
    return op_fail(WAM_ERR_INVALID_ARG, "unknown precision");
  }
  return e == cudaSuccess ? WAM_OK : op_cuda("attention launch", e);
}

int wam_op_ln_modulate(const float* h, const float* shift, const float* scale, int64_t mod_stride, void* out,
                       int32_t M, int32_t d, int32_t rows_per_item, int32_t precision, void* stream) {
  if (h == nullptr || shift == nullptr || scale == nullptr || out == nullptr || M < 0 || rows_per_item <= 0)
    return op_fail(WAM_ERR_INVALID_ARG, "bad LN arguments");
  if (d % 128 != 0 || d > 1536) return op_fail(WAM_ERR_UNSUPPORTED, "d must be a multiple of 128, at most 1536");
  // shift and scale are addressed as offsets from a common base (the modulation row)
  const int64_t so = static_cast<int64_t>(shift - scale);
  const float* base = so >= 0 ? scale : shift;
  const int shift_off = static_cast<int>(shift - base), scale_off = static_cast<int>(scale - base);
  cudaError_t e = ln_modulate(h, nullptr, base, mod_stride, shift_off, scale_off, nullptr, out,
                              precision == WAM_PREC_BF16, M, d, rows_per_item, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? WAM_OK : op_cuda("LN-modulate launch", e);
}

int wam_op_gemm_qkv_vt(const void* A, const void* Wt, const float* bias, void* qkv, void* vt, int32_t M,
                       int32_t d, int32_t rows_per_item, int32_t vt_ld, void* stream) {
  const int N = 3 * d, K = d;
  int r = check_gemm_args(A, Wt, qkv, M, N, K, WAM_EPI_BF16, nullptr, rows_per_item);
  if (r != WAM_OK) return r;
  if (vt == nullptr || rows_per_item <= 0 || vt_ld < rows_per_item || vt_ld % 8 != 0 || d % 128 != 0)
    return op_fail(WAM_ERR_INVALID_ARG, "bad V^T arguments");
  if (!aligned16(A) || !aligned16(Wt) || !aligned16(qkv) || (bias && !aligned16(bias)))
    return op_fail(WAM_ERR_INVALID_ARG, "operands must be 16-byte aligned");
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return op_cuda("device query", e);
  GemmOperand ta, tb;
  if (tc_encode_gemm_operand(&ta, A, static_cast<uint64_t>(M > 0 ? M : 1), K, false) != 0 ||
      tc_encode_gemm_operand(&tb, Wt, N, K, false) != 0)
    return op_fail(WAM_ERR_CUDA, "cuTensorMapEncodeTiled failed");
  EpiArgs ep = make_epi(bias, qkv, nullptr, 0, rows_per_item);
  ep.vt = static_cast<bf16*>(vt);
  ep.vt_ld = vt_ld;
  e = tc_gemm(ta, tb, M, N, K, kEpiQkvVt, ep, sms, nullptr, static_cast<cudaStream_t>(stream), nullptr,
              GemmPlan{0, 0});
  return e == cudaSuccess ? WAM_OK : op_cuda("tcgen05 QKV GEMM launch", e);
}

int wam_op_attention_tc(const void* qkv, const void* vt, void* out, int32_t B, int32_t N, int32_t d,
                        int32_t n_heads, void* stream) {
  if (qkv == nullptr || vt == nullptr || out == nullptr || B < 0 || N < 0 || n_heads <= 0 ||
      (d != 64 * n_heads && d != 72 * n_heads))
    return op_fail(WAM_ERR_INVALID_ARG, "tcgen05 attention needs head dim 64 or 72");
  if (!aligned16(qkv) || !aligned16(vt) || !aligned16(out)) return op_fail(WAM_ERR_INVALID_ARG, "16-byte alignment required");
  if (B == 0 || N == 0) return WAM_OK;
  const int vt_ld = attention_tc_vt_ld(N);
  AttnMaps maps;
  if (attention_tc_encode(&maps, qkv, vt, B, N, d, n_heads, vt_ld) != 0)
    return op_fail(WAM_ERR_CUDA, "cuTensorMapEncodeTiled failed");
  cudaError_t e = attention_tc(maps, static_cast<bf16*>(out), B, N, d, n_heads, nullptr,
                               static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? WAM_OK : op_cuda("tcgen05 attention launch", e);
}

}  // extern "C"
