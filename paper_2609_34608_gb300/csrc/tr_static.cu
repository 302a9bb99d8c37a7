// Trajectory Remapping for callers that cannot allocate device memory.
//
// Robot controllers often run their control loop under a no-allocation rule: everything is
// allocated at start-up so that each control step has bounded latency, and some embed this
// library inside a host runtime that owns all device memory and gives it none.  Such callers
// cannot create a context (which allocates its scratch with cudaMalloc), so this entry point
// remaps a batch of finished trajectories using only the caller's buffers and a fixed array
// compiled into the library for the float64 partial sums of the direction's RMS.
//
// The array holds kStaticPartials doubles (64 KiB) and exists on every GPU that loads the
// library until the process exits.  All calls share it and it keeps the last call's contents;
// every slot a call reads is written by the same call first, so nothing needs clearing, but
// two calls that overlap on the GPU (different streams, or different host threads) race on it
// and must be serialised by the caller.  The first call on a device looks up the array's
// device address (cudaGetSymbolAddress, with that device current); make that first call before
// any stream capture begins.
#include <climits>
#include <mutex>
#include <string>

#include "common.cuh"
#include "wam.h"
#include "wam_ops.h"

namespace wam {
void set_op_error(const std::string& msg);  // ops.cu

namespace {

constexpr int kStaticChunk = 2048;     // trajectory values per reduction block
constexpr int kStaticPartials = 8192;  // float64 partial sums: 64 KiB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) double g_tr_partials[kStaticPartials];

std::mutex g_mu;
double* g_partials_ptr[kMaxDevices] = {};

// Sum over one chunk of one branch of (x^r - x_bar)^2 / sigma_r^2, with the same operations in
// the same order as the remap of wam_adapt_state (thread t of the block takes elements t, t + 256,
// ... of the chunk into a double-float sum; then the warp and block sums; the block total is
// scaled by 1 / sigma_r^2 once), so the two entry points agree bit for bit.
__global__ void __launch_bounds__(256) tr_static_partial_kernel(const float* __restrict__ x_bar,
                                                                const float* __restrict__ x_r,
                                                                int T, int V, double sigma_r,
                                                                int nch, double* __restrict__ partial) {
  __shared__ float red[2][8];
  const int b = blockIdx.z, br = blockIdx.y, ch = blockIdx.x;
  const int beg = br == 0 ? 0 : V;
  const int len = br == 0 ? V : T - V;
  const int64_t bo = static_cast<int64_t>(b) * T + beg;
  const int end = min(len, (ch + 1) * kStaticChunk);
  float hi = 0.0f, lo = 0.0f;
  for (int u = 0; u < kStaticChunk / 256; ++u) {
    const int i = ch * kStaticChunk + u * 256 + threadIdx.x;
    const float a = i < end ? x_r[bo + i] : 0.0f;
    const float c = i < end ? x_bar[bo + i] : 0.0f;
    df_add_sq_diff(a, c, hi, lo);
  }
  warp_sum_df(hi, lo);
  const int warp = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) {
    red[0][warp] = hi;
    red[1][warp] = lo;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int w = 0; w < 8; ++w) s += static_cast<double>(red[0][w]) + static_cast<double>(red[1][w]);
    partial[(static_cast<int64_t>(b) * 2 + br) * nch + ch] = s * (1.0 / (sigma_r * sigma_r));
  }
}

// Remapped init: retained slots get x_bar + sigma_b0 * unit-RMS direction, computed as
// x_bar + g (x_r - x_bar) with the branch gain g = sigma_b0 / (sigma_r rms) in double-float
// arithmetic (the same operations as the remap of wam_adapt_state); the action slots move by the
// executed shift and the slots left uncovered (and, in video mode 1, every video slot) get
// sigma_b0 * eps.
__global__ void __launch_bounds__(256) tr_static_apply_kernel(
    const float* __restrict__ x_bar, const float* __restrict__ x_r, const float* __restrict__ eps,
    float* __restrict__ out, int T, int V, int Na, int ad, int shift, double sigma_r,
    double sigma_b0, int normalize, int video_mode, int nch, const double* __restrict__ partial) {
  __shared__ float gain_hi[2], gain_lo[2];
  const int b = blockIdx.y;
  if (threadIdx.x < 2) {
    double s = 0.0;
    for (int c = 0; c < nch; ++c) s += partial[(static_cast<int64_t>(b) * 2 + threadIdx.x) * nch + c];
    const double ms = s / (threadIdx.x == 0 ? V : T - V);
    const double rms = normalize ? sqrt(ms) : 1.0;
    const bool zero = normalize && !(ms > 0.0);
    const double gain = zero ? 0.0 : sigma_b0 / (sigma_r * rms);
    gain_hi[threadIdx.x] = static_cast<float>(gain);
    gain_lo[threadIdx.x] = static_cast<float>(gain - static_cast<double>(gain_hi[threadIdx.x]));
  }
  __syncthreads();
  const int64_t bo = static_cast<int64_t>(b) * T;
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < T; j += gridDim.x * blockDim.x) {
    int src = -1, br = 0;
    if (j < V) {
      if (video_mode == 0) src = j;
    } else {
      br = 1;
      const int ja = j - V;
      const int row = ja / ad, col = ja - row * ad;
      if (row + shift < Na) src = V + (row + shift) * ad + col;
    }
    float val;
    if (src >= 0) {
      val = df_remap(x_r[bo + src], x_bar[bo + src], gain_hi[br], gain_lo[br]);
    } else {
      val = static_cast<float>(sigma_b0 * static_cast<double>(eps[bo + j]));
    }
    out[bo + j] = val;
  }
}

// Device address of the partial-sum array on the current device, looked up once per device.
int partials_on_current_device(double** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    set_op_error(std::string("cudaGetDevice: ") + cudaGetErrorString(e));
    return WAM_ERR_CUDA;
  }
  if (dev < 0 || dev >= kMaxDevices) {
    set_op_error("device index beyond the 64 devices this entry point tracks");
    return WAM_ERR_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_partials_ptr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_tr_partials);
    if (e != cudaSuccess || p == nullptr) {
      set_op_error(std::string("cudaGetSymbolAddress of the static partial sums: ") + cudaGetErrorString(e));
      return WAM_ERR_CUDA;
    }
    g_partials_ptr[dev] = static_cast<double*>(p);
  }
  *out = g_partials_ptr[dev];
  return WAM_OK;
}

}  // namespace
}  // namespace wam

extern "C" int wam_tr_remap_static(const float* x_bar, const float* x_r, const float* eps, float* out,
                                   int32_t batch, int32_t n_video, int32_t video_dim, int32_t n_action,
                                   int32_t action_dim, int32_t shift, double sigma_r, double sigma_b0,
                                   int32_t normalize, int32_t video_mode, void* stream) {
  using namespace wam;
  if (x_bar == nullptr || x_r == nullptr || out == nullptr || batch < 1 || n_video < 1 || video_dim < 1 ||
      n_action < 1 || action_dim < 1 || shift < 0 || !(sigma_r > 0.0) || !(sigma_b0 >= 0.0) ||
      (video_mode != 0 && video_mode != 1)) {
    set_op_error("invalid argument: null buffer, non-positive size, negative shift or sigma_r <= 0");
    return WAM_ERR_INVALID_ARG;
  }
  const int64_t V64 = static_cast<int64_t>(n_video) * video_dim;
  const int64_t T64 = V64 + static_cast<int64_t>(n_action) * action_dim;
  if (T64 > INT_MAX || static_cast<int64_t>(batch) * T64 > (int64_t(1) << 40)) {
    set_op_error("trajectory length n_video*video_dim + n_action*action_dim above 2^31 - 1 values");
    return WAM_ERR_INVALID_ARG;
  }
  const int V = static_cast<int>(V64);
  const int T = static_cast<int>(T64);
  if (eps == nullptr && (video_mode == 1 || shift > 0)) {
    set_op_error("eps is required when any slot receives fresh noise");
    return WAM_ERR_INVALID_ARG;
  }
  const int nv = (V + kStaticChunk - 1) / kStaticChunk;
  const int na = (T - V + kStaticChunk - 1) / kStaticChunk;
  const int nch = nv > na ? nv : na;
  if (static_cast<int64_t>(batch) * 2 * nch > kStaticPartials) {
    set_op_error("batch * 2 * ceil(max(video, action values) / 2048) exceeds the 8192 static partial sums");
    return WAM_ERR_UNSUPPORTED;
  }
  double* partials = nullptr;
  const int r = partials_on_current_device(&partials);
  if (r != WAM_OK) return r;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  tr_static_partial_kernel<<<dim3(nch, 2, batch), 256, 0, s>>>(x_bar, x_r, T, V, sigma_r, nch, partials);
  const int blocks = (T + 255) / 256 < 64 ? (T + 255) / 256 : 64;
  tr_static_apply_kernel<<<dim3(blocks, batch), 256, 0, s>>>(x_bar, x_r, eps, out, T, V, n_action, action_dim,
                                                            shift, sigma_r, sigma_b0, normalize, video_mode, nch,
                                                            partials);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_op_error(std::string("static-scratch remap launch: ") + cudaGetErrorString(e));
    return WAM_ERR_CUDA;
  }
  return WAM_OK;
}
