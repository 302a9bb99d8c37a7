// Shared helpers of the WAMachine CUDA library (device utilities, launch bookkeeping and the
// internal interfaces between translation units).  Nothing here is part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "wam.h"

#include <atomic>
#include <mutex>

#define WAM_DEV __device__ __forceinline__

namespace wam {

using bf16 = __nv_bfloat16;

// Bits of the device error word a context hands to kernels with bounded waits.
constexpr int kDevErrTimeout = 1;
// A bounded wait gives up after this long (ns of %globaltimer).
constexpr uint64_t kWaitLimitNs = 2000000000ull;

WAM_DEV uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Programmatic dependent launch: every hot-path kernel is launched so that the next kernel in
// the stream may be scheduled while it runs.  A kernel calls pdl_wait() before it touches data
// written by earlier work in the stream (the wait returns once that work has completed and its
// memory is visible), and pdl_launch_dependents() to let the next kernel start its prologue.
WAM_DEV void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
WAM_DEV void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Kernel attributes (the dynamic shared-memory limit) and device properties belong to one device,
// and a process may drive contexts on several GPUs (wam_continue_many switches devices per
// context), so "already set" is recorded per device index.  Devices beyond 64 are simply set on
// every launch.
constexpr int kMaxTrackedDevices = 64;

inline int current_device() {
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess) d = -1;
  return d;
}

// Largest dynamic shared-memory size already granted to one kernel, per device.
struct PerDeviceSmem {
  std::atomic<int> granted[kMaxTrackedDevices] = {};
};

// Raises the kernel's limit to at least `bytes` on the current device.  The limit never shrinks:
// another host thread may launch the same kernel with a larger size between this set and its own
// launch.  Sets are serialised so the recorded value is always the attribute's value.
inline std::mutex& smem_attr_mutex() {
  static std::mutex m;
  return m;
}

template <typename Kernel>
inline cudaError_t ensure_max_smem(PerDeviceSmem& rec, Kernel kernel, int bytes) {
  const int dev = current_device();
  const bool tracked = dev >= 0 && dev < kMaxTrackedDevices;
  if (tracked && rec.granted[dev].load(std::memory_order_acquire) >= bytes) return cudaSuccess;
  std::lock_guard<std::mutex> lock(smem_attr_mutex());
  if (!tracked) {
    // untracked device: never lower the limit below what the function already allows
    int cur = 0;
    cudaFuncAttributes fa;
    if (cudaFuncGetAttributes(&fa, kernel) == cudaSuccess) cur = fa.maxDynamicSharedSizeBytes;
    return cur >= bytes ? cudaSuccess : cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  }
  if (rec.granted[dev].load(std::memory_order_relaxed) >= bytes) return cudaSuccess;
  const cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return e;
  rec.granted[dev].store(bytes, std::memory_order_release);
  return cudaSuccess;
}

// Streaming-multiprocessor count of the current device, looked up once per device.
inline int device_sm_count() {
  static std::atomic<int> cached[kMaxTrackedDevices] = {};
  const int dev = current_device();
  const bool tracked = dev >= 0 && dev < kMaxTrackedDevices;
  int n = tracked ? cached[dev].load(std::memory_order_relaxed) : 0;
  if (n > 0) return n;
  if (dev < 0 || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
  if (tracked) cached[dev].store(n, std::memory_order_relaxed);
  return n;
}

WAM_DEV float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

WAM_DEV double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Mean and reciprocal standard deviation (eps 1e-6) of one d-wide row held by a warp as NV4
// float4s per lane (d = 128 NV4): the LayerNorm statistics of every LN kernel.
template <int NV4>
WAM_DEV void row_stats(const float4 (&v)[NV4], int d, float& mean, float& rstd) {
  float s = 0.0f;
#pragma unroll
  for (int i = 0; i < NV4; ++i) s += (v[i].x + v[i].y) + (v[i].z + v[i].w);
  mean = warp_sum(s) / d;
  float q = 0.0f;
#pragma unroll
  for (int i = 0; i < NV4; ++i) {
    const float a = v[i].x - mean, b = v[i].y - mean, c = v[i].z - mean, e = v[i].w - mean;
    q += (a * a + b * b) + (c * c + e * e);
  }
  rstd = rsqrtf(warp_sum(q) / d + 1e-6f);
}

// ---- double-float accumulation (float32 pairs) ----------------------------------------
// GB300 runs float64 at a small fraction of its float32 rate, which made float64 reductions the
// bottleneck of the TR direction sums.  A sum of squares kept as an unevaluated pair hi + lo of
// floats, with the exact error of every product (fma) and addition (two-sum) carried in lo, is
// accurate to about 2^-44 relative, enough for the float32 results those sums scale.
WAM_DEV void two_sum(float a, float b, float& s, float& e) {
  s = a + b;
  const float bb = s - a;
  e = (a - (s - bb)) + (b - bb);
}

// x_b + g (x_r - x_b) for a float64 gain g given as gh = float(g), gl = float(g - gh): the
// difference split exactly by two_sum, the product's rounding error recovered by fma, one final
// rounding.  Within one float32 ulp of the float64 evaluation (Eq. 2's remap), on the float32 pipe.
WAM_DEV float df_remap(float xr, float xb, float gh, float gl) {
  float dh, dl;
  two_sum(xr, -xb, dh, dl);
  const float ph = __fmul_rn(gh, dh);   // never contracted into the sum below
  const float pl = fmaf(gh, dl, fmaf(gl, dh, fmaf(gh, dh, -ph)));
  float sh, se;
  two_sum(xb, ph, sh, se);
  return sh + (se + pl);
}

// (hi, lo) += v^2 for v = x - y, with x - y itself split exactly into vh + vl.
WAM_DEV void df_add_sq_diff(float x, float y, float& hi, float& lo) {
  float vh, vl;
  two_sum(x, -y, vh, vl);
  const float ph = vh * vh;
  const float pl = fmaf(vh, vh, -ph) + fmaf(2.0f * vh, vl, vl * vl);
  float sh, se;
  two_sum(hi, ph, sh, se);
  const float sl = lo + (se + pl);
  hi = sh + sl;                 // renormalise: |sl| is far below |sh|
  lo = sl - (hi - sh);
}

// (hi, lo) += (bh, bl)
WAM_DEV void df_add(float& hi, float& lo, float bh, float bl) {
  float sh, se;
  two_sum(hi, bh, sh, se);
  const float sl = lo + bl + se;
  hi = sh + sl;
  lo = sl - (hi - sh);
}

// Warp sum of double-float values; every lane ends with the total.
WAM_DEV void warp_sum_df(float& hi, float& lo) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float oh = __shfl_xor_sync(0xffffffffu, hi, o);
    const float ol = __shfl_xor_sync(0xffffffffu, lo, o);
    df_add(hi, lo, oh, ol);
  }
}

WAM_DEV float silu_f(float x) { return x / (1.0f + expf(-x)); }

WAM_DEV float gelu_tanh_f(float x) {
  // 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))
  const float k0 = 0.7978845608028654f;
  return 0.5f * x * (1.0f + tanhf(k0 * (x + 0.044715f * x * x * x)));
}

// ---- activation storage type helpers ---------------------------------------------------
template <typename T> struct Act;
template <> struct Act<float> {
  static WAM_DEV void store4(float* p, float a, float b, float c, float d) {
    *reinterpret_cast<float4*>(p) = make_float4(a, b, c, d);
  }
  static WAM_DEV float load(const float* p) { return *p; }
};
template <> struct Act<bf16> {
  static WAM_DEV void store4(bf16* p, float a, float b, float c, float d) {
    __nv_bfloat162 lo = __floats2bfloat162_rn(a, b);
    __nv_bfloat162 hi = __floats2bfloat162_rn(c, d);
    uint2 u;
    u.x = *reinterpret_cast<uint32_t*>(&lo);
    u.y = *reinterpret_cast<uint32_t*>(&hi);
    *reinterpret_cast<uint2*>(p) = u;
  }
  static WAM_DEV float load(const bf16* p) { return __bfloat162float(*p); }
};

// ---- GEMM epilogue description (shared by the tensor-core and SIMT GEMMs) ---------------
enum EpiMode { kEpiBf16 = 0, kEpiGeluBf16 = 1, kEpiResidF32 = 2, kEpiF32 = 3, kEpiQkvVt = 4 };

// Every field has a default, so an EpiArgs that names only what its epilogue uses is complete.
struct EpiArgs {
  const float* bias = nullptr;    // [N] or null
  void* C = nullptr;              // output (bf16 or f32, row-major, leading dim N)
  const float* gate = nullptr;    // RESID: gate rows
  int64_t gate_stride = 0;        // floats between gate rows of consecutive items
  int rows_per_item = 1;          // rows of one item (tokens of one episode)
  const int* item_map = nullptr;  // nullable: gate row of local item i = item_map[i]
  bf16* vt = nullptr;             // QKV_VT: V^T destination [items * heads * 64, vt_ld]
  int vt_ld = 0;                  // QKV_VT: padded token count (row length of V^T)
};

// ---- internal interfaces -----------------------------------------------------------------
// tcgen05 GEMM (gemm_tc.cu).  CUtensorMap is the driver's 128-byte opaque descriptor.
// Tensor maps of one K-major bf16 GEMM operand [rows][K] for every tile shape the GEMM may pick:
// boxes of 128 rows (the A operand and 128- / 256-wide B tiles) and of 64 rows (64-wide B tiles),
// one or two 64-column K-atoms deep (two only when K % 128 == 0).
struct GemmOperand {
  CUtensorMap r128_k1, r128_k2, r64_k1, r64_k2;
  bool k2;    // two-atom maps encoded
  bool r64;   // 64-row maps encoded
};
int tc_encode_gemm_operand(GemmOperand* op, const void* base, uint64_t rows, uint64_t K, bool rows64);
// Output tile width (64 / 128 / 256) and number of K ranges per tile; {0, 0} = choose.
struct GemmPlan {
  int bn;
  int splits;
  int mc = 0;   // CTAs per cluster sharing the A tile by multicast: 1 or 2; 0 = by the shape rule
};
// Device scratch of split-K: fp32 partial tiles, then one int ticket counter per output tile.
// The counters must be zero before the first use; every GEMM leaves them zero.
struct SplitWorkspace {
  float* ws;
  int* counters;
  size_t ws_bytes;
};
size_t tc_gemm_workspace_bytes(int num_sms);
// allow64: 64-wide tiles may be chosen; pairs64: the weight has 64-row boxes (128-wide CTA pairs)
GemmPlan tc_gemm_plan(int M, int N, int K, bool allow64, bool pairs64, int num_sms);
// ws == nullptr: no K split.  plan.bn == 0: chosen by tc_gemm_plan.
cudaError_t tc_gemm(const GemmOperand& a, const GemmOperand& b, int M, int N, int K, int epi, const EpiArgs& e,
                    int num_sms, int* dev_err, cudaStream_t s, const SplitWorkspace* ws, GemmPlan plan);

// Row-local chain of DiT blocks as one persistent tcgen05 kernel (dit_chain.cu): the "tail" of
// block l (out-projection + gated residual, LN, MLP up, MLP down + gated residual) followed by the
// "head" of block l+1 (LN + modulation, QKV projection with V^T), either part optional.
struct ChainParams {
  int M, Mt, d, dff;          // rows, 128-row blocks, model width, MLP width
  int has_tail, has_head;
  EpiArgs e_out, e_up, e_down, e_qkv;
  const float* mods;          // per-item modulation rows
  int64_t mod_stride;
  const int* item_map;        // nullable: modulation row of local item i = item_map[i]
  int rows_per_item;
  int shift2_off, scale2_off;  // tail: LN before the MLP
  int shift1_off, scale1_off;  // head: LN before attention
  float* h;                   // fp32 residual stream [M, d]
  float* hq;                  // nullable: the head's LN also copies h here
  bf16* xln;                  // LN output [M, d]
  int* ctr;                   // dit_chain_counters(max rows) ints, zero before the first launch
  int* dev_err;
  wam_chain_task* trace;      // nullable: per-task timestamps (profiling), task t at trace[t]
  int trace_cap;              // tasks beyond it are not recorded
  int trace_launch;           // launch number written into the records
  int phase_barrier;          // 1: each kind waits for all of the previous kind (grid-wide)
};
// Two-atom, 128-row tensor maps of the operands (unused ones may repeat any valid map).
struct ChainMaps {
  const CUtensorMap *att, *xln, *u, *out_w, *up_w, *down_w, *qkv_w;
};
int dit_chain_counters(int max_rows);
int dit_chain_tasks(const ChainParams& p);
bool dit_chain_supported(int d, int dff);
cudaError_t dit_chain(const ChainMaps& maps, const ChainParams& p, int num_sms, cudaStream_t s);

// float32 SIMT GEMM (gemm_simt.cu): C = A[M,K] Wt[N,K]^T
cudaError_t simt_gemm(const float* A, const float* Wt, int M, int N, int K, int epi,
                      const EpiArgs& e, cudaStream_t s);

// attention (attention.cu)
cudaError_t attention_bf16(const bf16* qkv, bf16* out, int B, int N, int d, int H,
                           cudaStream_t s);
cudaError_t attention_f32(const float* qkv, float* out, int B, int N, int d, int H,
                          cudaStream_t s);
bool attention_bf16_supported(int head_dim);
// tcgen05 attention (attention_tc.cu), head dim 64 or 72: Q / K read from the qkv buffer
// [items * N, 3d], V^T [items * d, vt_ld] as written by the QKV projection's epilogue.
struct AttnMaps {
  CUtensorMap qk, qk_tail, vt;
  int dh;
};
// 0 on success; negative when the head dim is unsupported or an encoding failed.
int attention_tc_encode(AttnMaps* m, const void* qkv, const void* vt, int items, int N, int d, int H, int vt_ld);
cudaError_t attention_tc(const AttnMaps& m, bf16* out, int B, int N, int d, int H, int* dev_err, cudaStream_t s);
int attention_tc_vt_ld(int N);
int tc_encode_bf16_box(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t ld,
                       uint32_t box_cols, uint32_t box_rows);
// 3-D bf16 map: dims (innermost first), byte strides of dims 1 and 2, box, swizzle 128 or 32 bytes.
int tc_encode_bf16_3d(CUtensorMap* map, const void* base, const uint64_t (&dims)[3], const uint64_t (&strides)[2],
                      const uint32_t (&box)[3], int swizzle_bytes);

}  // namespace wam
