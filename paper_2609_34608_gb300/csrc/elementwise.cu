// Memory-bound kernels of the denoising step and of the state adaptation:
//   conditioning GEMVs (timestep features -> MLP -> every layer's adaLN modulation),
//   token embedding, adaLN modulate (LN without affine, *(1+scale)+shift),
//   final modulated norm + output heads fused with the Euler update,
//   Trajectory Remapping (Eqs. 1-2, 12), Observation Rebinding score (Eq. 4),
//   Residual Rescaling probe / gate / injection-or-refresh (Eqs. 5-9),
//   and weight preparation.
// Row kernels use one warp per token row with float4 traffic and warp-shuffle reductions;
// every reduction that feeds a decision accumulates in float64 in a fixed order.
#include <math_constants.h>

#include "kernels.cuh"

namespace wam {
namespace {

constexpr int kRowWarps = 8;  // warps per block of the row kernels

WAM_DEV double block_sum_d(double v, double* red) {
  v = warp_sum_d(v);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  double s = 0.0;
  if (threadIdx.x == 0) {
    for (int w = 0; w < (blockDim.x >> 5); ++w) s += red[w];
  }
  __syncthreads();
  return s;  // valid in thread 0
}

// ---------------------------------------------------------------- conditioning GEMV
template <typename TW>
WAM_DEV float2 load_w2(const TW* W, int64_t idx);
template <>
WAM_DEV float2 load_w2<float>(const float* W, int64_t idx) {
  return *reinterpret_cast<const float2*>(W + idx);
}
template <>
WAM_DEV float2 load_w2<bf16>(const bf16* W, int64_t idx) {
  return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(W + idx));
}

// out[b, n] = post(sum_k pre(x[b, k]) W[k, n] + bias[n]).  64 output columns per block
// (2 per lane), the 8 warps split K and combine through shared memory; inputs are staged
// 8 items at a time so each weight row is read once per group of items.
template <typename TW, int PRE, int POST>
__global__ void __launch_bounds__(256) cond_gemv_kernel(const float* __restrict__ x,
                                                        const StepItem* __restrict__ items,
                                                        const TW* __restrict__ W,
                                                        const float* __restrict__ bias,
                                                        float* __restrict__ out, int Bw, int K,
                                                        int Nout) {
  constexpr int kB = 8;
  extern __shared__ float sx[];  // [kB][K]
  __shared__ float red[8][kB][64];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = blockIdx.x * 64 + lane * 2;
  const int kper = (K + 7) / 8;
  const int k0 = warp * kper;
  const int k1 = min(K, k0 + kper);
  for (int b0 = 0; b0 < Bw; b0 += kB) {
    const int nb = min(kB, Bw - b0);
    for (int i = threadIdx.x; i < nb * K; i += 256) {
      const int bi = i / K, k = i % K;
      float v;
      if constexpr (PRE == kPreFeatures) {
        // cos / sin of 1000 sigma 10000^(-j/half), argument formed in float64
        const int half = K / 2;
        const int j = k < half ? k : k - half;
        const double f = exp(-log(10000.0) * static_cast<double>(j) / half);
        const double a = 1000.0 * items[b0 + bi].sigma * f;
        v = static_cast<float>(k < half ? cos(a) : sin(a));
      } else {
        v = x[static_cast<int64_t>(b0 + bi) * K + k];
        if constexpr (PRE == kPreSilu) v = silu_f(v);
      }
      sx[bi * K + k] = v;
    }
    __syncthreads();
    float acc[kB][2];
#pragma unroll
    for (int bi = 0; bi < kB; ++bi) acc[bi][0] = acc[bi][1] = 0.0f;
    if (n < Nout) {
      for (int k = k0; k < k1; ++k) {
        const float2 w = load_w2<TW>(W, static_cast<int64_t>(k) * Nout + n);
#pragma unroll
        for (int bi = 0; bi < kB; ++bi) {
          const float xv = sx[bi * K + k];
          acc[bi][0] = fmaf(xv, w.x, acc[bi][0]);
          acc[bi][1] = fmaf(xv, w.y, acc[bi][1]);
        }
      }
    }
#pragma unroll
    for (int bi = 0; bi < kB; ++bi) {
      red[warp][bi][lane * 2] = acc[bi][0];
      red[warp][bi][lane * 2 + 1] = acc[bi][1];
    }
    __syncthreads();
    for (int i = threadIdx.x; i < nb * 64; i += 256) {
      const int bi = i / 64, c = i % 64;
      const int col = blockIdx.x * 64 + c;
      if (col < Nout) {
        float s = 0.0f;
#pragma unroll
        for (int w = 0; w < 8; ++w) s += red[w][bi][c];
        s += bias[col];
        if constexpr (POST == 1) s = silu_f(s);
        out[static_cast<int64_t>(b0 + bi) * Nout + col] = s;
      }
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------- token embedding
__global__ void __launch_bounds__(256) embed_kernel(
    float* __restrict__ h, float* __restrict__ xhist, int64_t stage_stride,
    const StepItem* __restrict__ items, const float* __restrict__ x, int T,
    const float* __restrict__ obs_emb, const float* __restrict__ vid_w,
    const float* __restrict__ vid_b, const float* __restrict__ act_w,
    const float* __restrict__ act_b, const float* __restrict__ pos, int Bw, int No, int Nv,
    int vd, int Na, int ad, int d) {
  const int N = No + Nv + Na;
  const int64_t gw = static_cast<int64_t>(blockIdx.x) * kRowWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (gw >= static_cast<int64_t>(Bw) * N) return;
  const int w = static_cast<int>(gw / N), n = static_cast<int>(gw % N);
  const StepItem it = items[w];
  float4* hr = reinterpret_cast<float4*>(h + gw * d);
  const float4* pr = reinterpret_cast<const float4*>(pos + static_cast<int64_t>(n) * d);
  const int d4 = d / 4;
  if (n < No) {
    const float4* src = reinterpret_cast<const float4*>(obs_emb + (static_cast<int64_t>(it.ep) * No + n) * d);
    for (int c = lane; c < d4; c += 32) {
      const float4 a = src[c], p = pr[c];
      hr[c] = make_float4(a.x + p.x, a.y + p.y, a.z + p.z, a.w + p.w);
    }
    return;
  }
  const bool video = n < No + Nv;
  const int in_dim = video ? vd : ad;
  const int64_t xoff = static_cast<int64_t>(it.ep) * T +
                       (video ? static_cast<int64_t>(n - No) * vd
                              : static_cast<int64_t>(Nv) * vd + static_cast<int64_t>(n - No - Nv) * ad);
  const float* xin = x + xoff;
  // Record the latent entering this stage (the retained trajectory at stage k).
  if (lane < in_dim) xhist[static_cast<int64_t>(it.stage) * stage_stride + xoff + lane] = xin[lane];
  float xi[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) xi[i] = i < in_dim ? xin[i] : 0.0f;
  const float4* W4 = reinterpret_cast<const float4*>(video ? vid_w : act_w);
  const float4* b4 = reinterpret_cast<const float4*>(video ? vid_b : act_b);
  for (int c = lane; c < d4; c += 32) {
    float4 acc = b4[c];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      if (i < in_dim) {
        const float4 wv = W4[static_cast<int64_t>(i) * d4 + c];
        acc.x = fmaf(xi[i], wv.x, acc.x);
        acc.y = fmaf(xi[i], wv.y, acc.y);
        acc.z = fmaf(xi[i], wv.z, acc.z);
        acc.w = fmaf(xi[i], wv.w, acc.w);
      }
    }
    const float4 p = pr[c];
    hr[c] = make_float4(acc.x + p.x, acc.y + p.y, acc.z + p.z, acc.w + p.w);
  }
}

// ---------------------------------------------------------------- LN modulate
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

template <int NV4, typename TO>
__global__ void __launch_bounds__(256) ln_mod_kernel(const float* __restrict__ h,
                                                     float* __restrict__ hcopy,
                                                     const float* __restrict__ mods,
                                                     int64_t mod_stride, int shift_off,
                                                     int scale_off,
                                                     const int* __restrict__ item_map,
                                                     TO* __restrict__ out, int M, int d,
                                                     int rows_per_item) {
  const int64_t row = static_cast<int64_t>(blockIdx.x) * kRowWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= M) return;
  const float4* hr = reinterpret_cast<const float4*>(h + row * d);
  float4 v[NV4];
#pragma unroll
  for (int i = 0; i < NV4; ++i) v[i] = hr[lane + 32 * i];
  if (hcopy != nullptr) {
    float4* cr = reinterpret_cast<float4*>(hcopy + row * d);
#pragma unroll
    for (int i = 0; i < NV4; ++i) cr[lane + 32 * i] = v[i];
  }
  float mean, rstd;
  row_stats<NV4>(v, d, mean, rstd);
  int item = static_cast<int>(row / rows_per_item);
  if (item_map != nullptr) item = item_map[item];
  const float* shift = mods + item * mod_stride + shift_off;
  const float* scale = mods + item * mod_stride + scale_off;
#pragma unroll
  for (int i = 0; i < NV4; ++i) {
    const int c = (lane + 32 * i) * 4;
    const float4 sh = *reinterpret_cast<const float4*>(shift + c);
    const float4 sc = *reinterpret_cast<const float4*>(scale + c);
    Act<TO>::store4(out + row * d + c, fmaf((v[i].x - mean) * rstd, 1.0f + sc.x, sh.x),
                    fmaf((v[i].y - mean) * rstd, 1.0f + sc.y, sh.y),
                    fmaf((v[i].z - mean) * rstd, 1.0f + sc.z, sh.z),
                    fmaf((v[i].w - mean) * rstd, 1.0f + sc.w, sh.w));
  }
}

// ---------------------------------------------------------------- final layer + Euler
template <int NV4>
__global__ void __launch_bounds__(256) final_euler_kernel(
    const float* __restrict__ h, const StepItem* __restrict__ items,
    const float* __restrict__ mods, int64_t mod_stride, int fin_off,
    const float* __restrict__ vout_w, const float* __restrict__ vout_b,
    const float* __restrict__ aout_w, const float* __restrict__ aout_b, float* __restrict__ x,
    float* __restrict__ xhist, float* __restrict__ vhist, int64_t stage_stride, int T, int Bw,
    int No, int Nv, int vd, int Na, int ad, int d) {
  const int rows = Nv + Na;
  const int64_t gw = static_cast<int64_t>(blockIdx.x) * kRowWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (gw >= static_cast<int64_t>(Bw) * rows) return;
  const int w = static_cast<int>(gw / rows), r = static_cast<int>(gw % rows);
  const StepItem it = items[w];
  const int N = No + Nv + Na;
  const float4* hr = reinterpret_cast<const float4*>(h + (static_cast<int64_t>(w) * N + No + r) * d);
  float4 v[NV4];
#pragma unroll
  for (int i = 0; i < NV4; ++i) v[i] = hr[lane + 32 * i];
  float mean, rstd;
  row_stats<NV4>(v, d, mean, rstd);
  const float* shift = mods + w * mod_stride + fin_off;
  const float* scale = shift + d;
  const bool video = r < Nv;
  const int od = video ? vd : ad;
  const float* Wo = video ? vout_w : aout_w;
  float acc[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) acc[j] = 0.0f;
#pragma unroll
  for (int i = 0; i < NV4; ++i) {
    const int c = (lane + 32 * i) * 4;
    const float4 sh = *reinterpret_cast<const float4*>(shift + c);
    const float4 sc = *reinterpret_cast<const float4*>(scale + c);
    const float y[4] = {fmaf((v[i].x - mean) * rstd, 1.0f + sc.x, sh.x),
                        fmaf((v[i].y - mean) * rstd, 1.0f + sc.y, sh.y),
                        fmaf((v[i].z - mean) * rstd, 1.0f + sc.z, sh.z),
                        fmaf((v[i].w - mean) * rstd, 1.0f + sc.w, sh.w)};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float* wr = Wo + static_cast<int64_t>(c + e) * od;
#pragma unroll
      for (int j = 0; j < 16; ++j)
        if (j < od) acc[j] = fmaf(y[e], wr[j], acc[j]);
    }
  }
  float mine = 0.0f;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    if (j < od) {
      const float s = warp_sum(acc[j]);
      if (lane == j) mine = s;
    }
  }
  if (lane < od) {
    const float vel = mine + (video ? vout_b : aout_b)[lane];
    const int64_t idx = static_cast<int64_t>(it.ep) * T +
                        (video ? static_cast<int64_t>(r) * vd
                               : static_cast<int64_t>(Nv) * vd + static_cast<int64_t>(r - Nv) * ad) +
                        lane;
    const float xn = static_cast<float>(static_cast<double>(x[idx]) + it.dsigma * static_cast<double>(vel));
    x[idx] = xn;
    xhist[static_cast<int64_t>(it.stage + 1) * stage_stride + idx] = xn;
    vhist[static_cast<int64_t>(it.stage) * stage_stride + idx] = vel;
  }
}

// ---------------------------------------------------------------- Trajectory Remapping
__global__ void __launch_bounds__(256) tr_rms_partial_kernel(const AdaptItem* __restrict__ items,
                                                             const float* __restrict__ xhist,
                                                             int64_t stage_stride, int K, int T,
                                                             int V, int nch,
                                                             double* __restrict__ partial) {
  __shared__ double red[8];
  const int b = blockIdx.z, br = blockIdx.y, ch = blockIdx.x;
  const AdaptItem it = items[b];
  double s = 0.0;
  if (it.op == kAdaptTR) {
    const int beg = br == 0 ? 0 : V;
    const int len = br == 0 ? V : T - V;
    const float* xr = xhist + it.r * stage_stride + static_cast<int64_t>(b) * T + beg;
    const float* xb = xhist + K * stage_stride + static_cast<int64_t>(b) * T + beg;
    const int end = min(len, (ch + 1) * kTrChunk);
    for (int i = ch * kTrChunk + threadIdx.x; i < end; i += blockDim.x) {
      const double u = (static_cast<double>(xr[i]) - static_cast<double>(xb[i])) / it.sigma_r;
      s += u * u;
    }
  }
  s = block_sum_d(s, red);
  if (threadIdx.x == 0) partial[(static_cast<int64_t>(b) * 2 + br) * nch + ch] = s;
}

// Remapped initialisation (Eq. 2), cold init, restart, and binding of the new condition.
// Reads x_bar (stage K) and x^r from the stage history, writes the current latent and the
// retained init x^{b0}; blocks past the trajectory range copy the new observation tokens.
__global__ void __launch_bounds__(256) adapt_apply_kernel(
    const AdaptItem* __restrict__ items, const double* __restrict__ partial, int nch,
    float* __restrict__ x, float* __restrict__ xb0, const float* __restrict__ xhist,
    int64_t stage_stride, int K, const float* __restrict__ eps,
    const float* __restrict__ obs_new, float* __restrict__ obs, int T, int V, int Na, int ad,
    int64_t obs_elems, int normalize, int video_mode, int traj_blocks) {
  __shared__ double rms[2];
  __shared__ int zero[2];
  const int b = blockIdx.y;
  const AdaptItem it = items[b];
  if (it.op == kAdaptNone && !it.bind_obs) return;
  if (static_cast<int>(blockIdx.x) >= traj_blocks) {
    if (!it.bind_obs) return;
    const int64_t base = static_cast<int64_t>(b) * obs_elems;
    const int64_t start = static_cast<int64_t>(blockIdx.x - traj_blocks) * blockDim.x + threadIdx.x;
    const int64_t stride = static_cast<int64_t>(gridDim.x - traj_blocks) * blockDim.x;
    for (int64_t i = start; i < obs_elems; i += stride) obs[base + i] = obs_new[base + i];
    return;
  }
  if (it.op == kAdaptNone) return;
  if (threadIdx.x < 2) {
    double ms = 0.0;
    if (it.op == kAdaptTR) {
      double s = 0.0;
      for (int c = 0; c < nch; ++c) s += partial[(static_cast<int64_t>(b) * 2 + threadIdx.x) * nch + c];
      ms = s / (threadIdx.x == 0 ? V : T - V);
    }
    rms[threadIdx.x] = normalize ? sqrt(ms) : 1.0;
    zero[threadIdx.x] = normalize && !(ms > 0.0);
  }
  __syncthreads();
  const int64_t bo = static_cast<int64_t>(b) * T;
  const float* xr = xhist + it.r * stage_stride + bo;
  const float* xb = xhist + K * stage_stride + bo;
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < T; j += traj_blocks * blockDim.x) {
    float val;
    if (it.op == kAdaptCold) {
      val = eps[bo + j];
    } else if (it.op == kAdaptRestart) {
      val = xb0[bo + j];
    } else {
      int src = -1;
      int br = 0;
      if (j < V) {
        if (video_mode == 0) src = j;
      } else {
        br = 1;
        const int ja = j - V;
        const int row = ja / ad, col = ja - row * ad;
        const int srow = row + it.shift;
        if (srow < Na) src = V + srow * ad + col;
      }
      if (src >= 0) {
        const double u = (static_cast<double>(xr[src]) - static_cast<double>(xb[src])) / it.sigma_r;
        const double dir = zero[br] ? 0.0 : u / rms[br];
        val = static_cast<float>(static_cast<double>(xb[src]) + it.sigma_b0 * dir);
      } else {
        val = static_cast<float>(it.sigma_b0 * static_cast<double>(eps[bo + j]));
      }
    }
    x[bo + j] = val;
    if (it.op != kAdaptRestart) xb0[bo + j] = val;
  }
}

// ---------------------------------------------------------------- Observation Rebinding
__global__ void __launch_bounds__(256) or_partial_kernel(const float* __restrict__ pred,
                                                         const float* __restrict__ real,
                                                         int64_t obs_elems, int M,
                                                         float4 inv_delta, int nch,
                                                         double* __restrict__ partial) {
  __shared__ double red[8];
  const int b = blockIdx.z, m = blockIdx.y, ch = blockIdx.x;
  const int64_t comp = obs_elems / M;
  const int64_t base = static_cast<int64_t>(b) * obs_elems + m * comp;
  const float idl = m == 0 ? inv_delta.x : m == 1 ? inv_delta.y : m == 2 ? inv_delta.z : inv_delta.w;
  const int64_t end = min(comp, static_cast<int64_t>(ch + 1) * kOrChunk);
  double s = 0.0;
  for (int64_t i = static_cast<int64_t>(ch) * kOrChunk + threadIdx.x; i < end; i += blockDim.x) {
    const double dv = (static_cast<double>(pred[base + i]) - static_cast<double>(real[base + i])) * idl;
    s += dv * dv;
  }
  s = block_sum_d(s, red);
  if (threadIdx.x == 0) partial[(static_cast<int64_t>(b) * M + m) * nch + ch] = s;
}

// ---------------------------------------------------------------- Residual Rescaling
// Per (item, branch, chunk): sum p_i p_a, sum p_a^2, sum p_i^2 with p_i = h_s - h_q.
__global__ void __launch_bounds__(256) rr_probe_kernel(const float* __restrict__ h,
                                                       const float* __restrict__ hq,
                                                       const float* __restrict__ pa,
                                                       const StepItem* __restrict__ items,
                                                       int N, int d, int split_row, int nch,
                                                       double* __restrict__ partial) {
  __shared__ double red[8];
  const int w = blockIdx.z, br = blockIdx.y, ch = blockIdx.x;
  const int ep = items[w].ep;
  const int64_t row0 = br == 0 ? 0 : split_row;
  const int64_t n_el = (br == 0 ? static_cast<int64_t>(split_row) : static_cast<int64_t>(N - split_row)) * d;
  const int64_t off_w = (static_cast<int64_t>(w) * N + row0) * d;
  const int64_t off_e = (static_cast<int64_t>(ep) * N + row0) * d;
  const float4* h4 = reinterpret_cast<const float4*>(h + off_w);
  const float4* q4 = reinterpret_cast<const float4*>(hq + off_w);
  const float4* a4 = reinterpret_cast<const float4*>(pa + off_e);
  const int64_t beg4 = static_cast<int64_t>(ch) * (kProbeChunk / 4);
  const int64_t end4 = min(n_el / 4, beg4 + kProbeChunk / 4);
  float sia = 0.0f, saa = 0.0f, sii = 0.0f;
  for (int64_t i = beg4 + threadIdx.x; i < end4; i += blockDim.x) {
    const float4 hv = h4[i], qv = q4[i], av = a4[i];
    const float p0 = hv.x - qv.x, p1 = hv.y - qv.y, p2 = hv.z - qv.z, p3 = hv.w - qv.w;
    sia += (p0 * av.x + p1 * av.y) + (p2 * av.z + p3 * av.w);
    saa += (av.x * av.x + av.y * av.y) + (av.z * av.z + av.w * av.w);
    sii += (p0 * p0 + p1 * p1) + (p2 * p2 + p3 * p3);
  }
  const double t0 = block_sum_d(sia, red);
  const double t1 = block_sum_d(saa, red);
  const double t2 = block_sum_d(sii, red);
  if (threadIdx.x == 0) {
    double* out = partial + ((static_cast<int64_t>(w) * 2 + br) * nch + ch) * 3;
    out[0] = t0;
    out[1] = t1;
    out[2] = t2;
  }
}

// alpha (Eq. 7), cosine and relative fit (Eq. 8) per (item, branch).
__global__ void rr_gate_kernel(const double* __restrict__ partial, int Bw, int nch, int64_t n0,
                               int64_t n1, double amin, double amax, double eps, double gcos,
                               double gfit, RRGate* __restrict__ out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= Bw * 2) return;
  const double* p = partial + static_cast<int64_t>(i) * nch * 3;
  double sia = 0.0, saa = 0.0, sii = 0.0;
  for (int c = 0; c < nch; ++c) {
    sia += p[3 * c];
    saa += p[3 * c + 1];
    sii += p[3 * c + 2];
  }
  const double n = static_cast<double>((i & 1) ? n1 : n0);
  double alpha = (sia / n) / fmax(saa / n, eps);
  alpha = fmin(fmax(alpha, amin), amax);
  RRGate g;
  g.alpha = alpha;
  g.pad = 0;
  if (sii > 0.0 && saa > 0.0) {
    g.cos = sia / (sqrt(sii) * sqrt(saa));
    g.fit = sqrt(fmax(sii - 2.0 * alpha * sia + alpha * alpha * saa, 0.0)) / sqrt(sii);
    g.pass = (g.cos >= gcos && g.fit <= gfit) ? 1 : 0;
  } else {
    g.cos = 0.0;
    g.fit = CUDART_INF;
    g.pass = 0;
  }
  out[i] = g;
}

// Accepted: h_e = h_s + alpha_branch R_a (Eq. 9).  Refresh: R_a = h_e - h_s, p_a = h_s - h_q,
// h = h_e.  Copy-back: h = h_e (item not on an RR path).
__global__ void __launch_bounds__(256) rr_apply_kernel(float* __restrict__ h,
                                                       const float* __restrict__ hm,
                                                       const float* __restrict__ hq,
                                                       float* __restrict__ pa,
                                                       float* __restrict__ ra,
                                                       const StepItem* __restrict__ items,
                                                       const RRApply* __restrict__ ap, int N,
                                                       int d, int split_row) {
  const int w = blockIdx.y;
  const RRApply a = ap[w];
  if (a.mode == kRRNone) return;
  const int ep = items[w].ep;
  const int64_t n4 = static_cast<int64_t>(N) * d / 4;
  const int64_t split4 = static_cast<int64_t>(split_row) * d / 4;
  float4* h4 = reinterpret_cast<float4*>(h + static_cast<int64_t>(w) * N * d);
  const float4* m4 = reinterpret_cast<const float4*>(hm + static_cast<int64_t>(a.cidx) * N * d);
  const float4* q4 = reinterpret_cast<const float4*>(hq + static_cast<int64_t>(w) * N * d);
  float4* p4 = reinterpret_cast<float4*>(pa + static_cast<int64_t>(ep) * N * d);
  float4* r4 = reinterpret_cast<float4*>(ra + static_cast<int64_t>(ep) * N * d);
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    if (a.mode == kRRInject) {
      const float al = i < split4 ? a.alpha0 : a.alpha1;
      float4 hv = h4[i];
      const float4 rv = r4[i];
      hv.x = fmaf(al, rv.x, hv.x);
      hv.y = fmaf(al, rv.y, hv.y);
      hv.z = fmaf(al, rv.z, hv.z);
      hv.w = fmaf(al, rv.w, hv.w);
      h4[i] = hv;
    } else if (a.mode == kRRRefresh) {
      const float4 hs = h4[i], he = m4[i], hqv = q4[i];
      r4[i] = make_float4(he.x - hs.x, he.y - hs.y, he.z - hs.z, he.w - hs.w);
      p4[i] = make_float4(hs.x - hqv.x, hs.y - hqv.y, hs.z - hqv.z, hs.w - hqv.w);
      h4[i] = he;
    } else {
      h4[i] = m4[i];
    }
  }
}

// ---------------------------------------------------------------- preparation
__global__ void cast_kernel(const float* __restrict__ in, bf16* __restrict__ out, int64_t n) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    out[i] = __float2bfloat16(in[i]);
}

template <typename TO>
__global__ void transpose_kernel(const float* __restrict__ in, TO* __restrict__ out, int K, int N) {
  __shared__ float tile[32][33];
  const int n0 = blockIdx.x * 32, k0 = blockIdx.y * 32;
  for (int i = threadIdx.y; i < 32; i += blockDim.y) {
    const int k = k0 + i, n = n0 + threadIdx.x;
    tile[i][threadIdx.x] = (k < K && n < N) ? in[static_cast<int64_t>(k) * N + n] : 0.0f;
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += blockDim.y) {
    const int n = n0 + i, k = k0 + threadIdx.x;
    if (n < N && k < K) {
      if constexpr (sizeof(TO) == 2)
        out[static_cast<int64_t>(n) * K + k] = __float2bfloat16(tile[threadIdx.x][i]);
      else
        out[static_cast<int64_t>(n) * K + k] = tile[threadIdx.x][i];
    }
  }
}

template <typename TO>
__global__ void copy2d_kernel(const float* __restrict__ in, int64_t spitch, TO* __restrict__ out,
                              int64_t dpitch, int rows, int cols) {
  const int64_t total = static_cast<int64_t>(rows) * cols;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i / cols, c = i % cols;
    const float v = in[r * spitch + c];
    if constexpr (sizeof(TO) == 2)
      out[r * dpitch + c] = __float2bfloat16(v);
    else
      out[r * dpitch + c] = v;
  }
}

template <typename TW, int PRE, int POST>
cudaError_t gemv_launch(const float* x, const StepItem* items, const TW* W, const float* bias,
                        float* out, int Bw, int K, int Nout, cudaStream_t s) {
  const size_t smem = static_cast<size_t>(8) * K * sizeof(float);
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(cond_gemv_kernel<TW, PRE, POST>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, 8 * 4096 * 4);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  cond_gemv_kernel<TW, PRE, POST><<<(Nout + 63) / 64, 256, smem, s>>>(x, items, W, bias, out, Bw, K, Nout);
  return cudaGetLastError();
}

template <typename TW>
cudaError_t gemv_pre_post(const float* x, const StepItem* items, const TW* W, const float* bias,
                          float* out, int Bw, int K, int Nout, int pre, int post, cudaStream_t s) {
  if (pre == kPreFeatures && post == 1) return gemv_launch<TW, kPreFeatures, 1>(x, items, W, bias, out, Bw, K, Nout, s);
  if (pre == kPreNone && post == 0) return gemv_launch<TW, kPreNone, 0>(x, items, W, bias, out, Bw, K, Nout, s);
  if (pre == kPreSilu && post == 0) return gemv_launch<TW, kPreSilu, 0>(x, items, W, bias, out, Bw, K, Nout, s);
  return cudaErrorInvalidValue;
}

unsigned row_blocks(int64_t rows) { return static_cast<unsigned>((rows + kRowWarps - 1) / kRowWarps); }

}  // namespace

cudaError_t cond_gemv(const float* x, const StepItem* items, const void* W, bool w_bf16,
                      const float* bias, float* out, int Bw, int K, int Nout, int pre, int post,
                      cudaStream_t s) {
  if (Bw <= 0) return cudaSuccess;
  if (K > 4096 || (Nout & 1)) return cudaErrorInvalidValue;
  return w_bf16 ? gemv_pre_post<bf16>(x, items, static_cast<const bf16*>(W), bias, out, Bw, K, Nout, pre, post, s)
                : gemv_pre_post<float>(x, items, static_cast<const float*>(W), bias, out, Bw, K, Nout, pre, post, s);
}

cudaError_t embed_tokens(float* h, float* xhist, int64_t stage_stride, const StepItem* items,
                         const float* x, int T, const float* obs_emb, const float* vid_w,
                         const float* vid_b, const float* act_w, const float* act_b,
                         const float* pos, int Bw, int No, int Nv, int vd, int Na, int ad, int d,
                         cudaStream_t s) {
  if (Bw <= 0) return cudaSuccess;
  const int64_t rows = static_cast<int64_t>(Bw) * (No + Nv + Na);
  embed_kernel<<<row_blocks(rows), 32 * kRowWarps, 0, s>>>(h, xhist, stage_stride, items, x, T,
                                                           obs_emb, vid_w, vid_b, act_w, act_b,
                                                           pos, Bw, No, Nv, vd, Na, ad, d);
  return cudaGetLastError();
}

#define WAM_NV4_CASES(X) X(1) X(2) X(3) X(4) X(5) X(6) X(7) X(8) X(9) X(10) X(11) X(12)

cudaError_t ln_modulate(const float* h, float* hcopy, const float* mods, int64_t mod_stride,
                        int shift_off, int scale_off, const int* item_map, void* out,
                        bool out_bf16, int M, int d, int rows_per_item, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  if (d % 128 != 0) return cudaErrorInvalidValue;
  const unsigned grid = row_blocks(M);
  const int nv4 = d / 128;
#define WAM_LN_CASE(NV)                                                                            \
  case NV:                                                                                         \
    if (out_bf16)                                                                                  \
      ln_mod_kernel<NV, bf16><<<grid, 256, 0, s>>>(h, hcopy, mods, mod_stride, shift_off,          \
                                                   scale_off, item_map, static_cast<bf16*>(out), M, \
                                                   d, rows_per_item);                              \
    else                                                                                           \
      ln_mod_kernel<NV, float><<<grid, 256, 0, s>>>(h, hcopy, mods, mod_stride, shift_off,         \
                                                    scale_off, item_map, static_cast<float*>(out), \
                                                    M, d, rows_per_item);                          \
    break;
  switch (nv4) {
    WAM_NV4_CASES(WAM_LN_CASE)
    default: return cudaErrorInvalidValue;
  }
#undef WAM_LN_CASE
  return cudaGetLastError();
}

cudaError_t final_euler(const float* h, const StepItem* items, const float* mods,
                        int64_t mod_stride, int fin_off, const float* vout_w,
                        const float* vout_b, const float* aout_w, const float* aout_b, float* x,
                        float* xhist, float* vhist, int64_t stage_stride, int T, int Bw, int No,
                        int Nv, int vd, int Na, int ad, int d, cudaStream_t s) {
  if (Bw <= 0) return cudaSuccess;
  if (d % 128 != 0 || vd > 16 || ad > 16) return cudaErrorInvalidValue;
  const unsigned grid = row_blocks(static_cast<int64_t>(Bw) * (Nv + Na));
#define WAM_FE_CASE(NV)                                                                       \
  case NV:                                                                                    \
    final_euler_kernel<NV><<<grid, 256, 0, s>>>(h, items, mods, mod_stride, fin_off, vout_w,  \
                                                vout_b, aout_w, aout_b, x, xhist, vhist,      \
                                                stage_stride, T, Bw, No, Nv, vd, Na, ad, d); \
    break;
  switch (d / 128) {
    WAM_NV4_CASES(WAM_FE_CASE)
    default: return cudaErrorInvalidValue;
  }
#undef WAM_FE_CASE
  return cudaGetLastError();
}

int tr_num_chunks(int T, int V) {
  const int a = (V + kTrChunk - 1) / kTrChunk;
  const int b = (T - V + kTrChunk - 1) / kTrChunk;
  return (a > b ? a : b) > 0 ? (a > b ? a : b) : 1;
}

cudaError_t tr_rms_partial(const AdaptItem* items, const float* xhist, int64_t stage_stride,
                           int K, int B, int T, int V, int nch, double* partial, cudaStream_t s) {
  dim3 grid(nch, 2, B);
  tr_rms_partial_kernel<<<grid, 256, 0, s>>>(items, xhist, stage_stride, K, T, V, nch, partial);
  return cudaGetLastError();
}

cudaError_t adapt_apply(const AdaptItem* items, const double* partial, int nch, float* x,
                        float* xb0, const float* xhist, int64_t stage_stride, int K,
                        const float* eps, const float* obs_new, float* obs, int B, int T, int V,
                        int Na, int ad, int64_t obs_elems, int normalize, int video_mode,
                        cudaStream_t s) {
  const int traj_blocks = (T + 255) / 256 < 64 ? (T + 255) / 256 : 64;
  const int obs_blocks = static_cast<int>((obs_elems + 255) / 256 < 64 ? (obs_elems + 255) / 256 : 64);
  dim3 grid(traj_blocks + obs_blocks, B);
  adapt_apply_kernel<<<grid, 256, 0, s>>>(items, partial, nch, x, xb0, xhist, stage_stride, K,
                                          eps, obs_new, obs, T, V, Na, ad, obs_elems, normalize,
                                          video_mode, traj_blocks);
  return cudaGetLastError();
}

int or_num_chunks(int64_t comp_elems) {
  return static_cast<int>((comp_elems + kOrChunk - 1) / kOrChunk);
}

cudaError_t or_score_partial(const float* pred, const float* real, int B, int64_t obs_elems,
                             int M, const float* inv_delta4, int nch, double* partial,
                             cudaStream_t s) {
  dim3 grid(nch, M, B);
  const float4 idl = make_float4(inv_delta4[0], inv_delta4[1], inv_delta4[2], inv_delta4[3]);
  or_partial_kernel<<<grid, 256, 0, s>>>(pred, real, obs_elems, M, idl, nch, partial);
  return cudaGetLastError();
}

int rr_num_chunks(int64_t branch_elems_max) {
  return static_cast<int>((branch_elems_max + kProbeChunk - 1) / kProbeChunk);
}

cudaError_t rr_probe_partial(const float* h, const float* hq, const float* pa,
                             const StepItem* items, int Bw, int N, int d, int split_row, int nch,
                             double* partial, cudaStream_t s) {
  if (Bw <= 0) return cudaSuccess;
  dim3 grid(nch, 2, Bw);
  rr_probe_kernel<<<grid, 256, 0, s>>>(h, hq, pa, items, N, d, split_row, nch, partial);
  return cudaGetLastError();
}

cudaError_t rr_gate(const double* partial, int Bw, int nch, int64_t n0, int64_t n1, double amin,
                    double amax, double eps, double gcos, double gfit, RRGate* out,
                    cudaStream_t s) {
  if (Bw <= 0) return cudaSuccess;
  rr_gate_kernel<<<(Bw * 2 + 63) / 64, 64, 0, s>>>(partial, Bw, nch, n0, n1, amin, amax, eps,
                                                   gcos, gfit, out);
  return cudaGetLastError();
}

cudaError_t rr_apply(float* h, const float* hm, const float* hq, float* pa, float* ra,
                     const StepItem* items, const RRApply* ap, int Bw, int N, int d,
                     int split_row, cudaStream_t s) {
  if (Bw <= 0) return cudaSuccess;
  const int64_t n4 = static_cast<int64_t>(N) * d / 4;
  const int bx = static_cast<int>((n4 + 255) / 256 < 1024 ? (n4 + 255) / 256 : 1024);
  dim3 grid(bx, Bw);
  rr_apply_kernel<<<grid, 256, 0, s>>>(h, hm, hq, pa, ra, items, ap, N, d, split_row);
  return cudaGetLastError();
}

cudaError_t cast_f32_bf16(const float* in, bf16* out, int64_t n, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int64_t blocks = (n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096;
  cast_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(in, out, n);
  return cudaGetLastError();
}

cudaError_t transpose_cast(const float* in, void* out, bool out_bf16, int K, int N,
                           cudaStream_t s) {
  dim3 grid((N + 31) / 32, (K + 31) / 32), block(32, 8);
  if (out_bf16)
    transpose_kernel<bf16><<<grid, block, 0, s>>>(in, static_cast<bf16*>(out), K, N);
  else
    transpose_kernel<float><<<grid, block, 0, s>>>(in, static_cast<float*>(out), K, N);
  return cudaGetLastError();
}

cudaError_t copy_cast_2d(const float* in, int64_t spitch, void* out, bool out_bf16,
                         int64_t dpitch, int rows, int cols, cudaStream_t s) {
  const int64_t total = static_cast<int64_t>(rows) * cols;
  const int64_t blocks = (total + 255) / 256 < 4096 ? (total + 255) / 256 : 4096;
  if (out_bf16)
    copy2d_kernel<bf16><<<static_cast<unsigned>(blocks), 256, 0, s>>>(in, spitch, static_cast<bf16*>(out), dpitch, rows, cols);
  else
    copy2d_kernel<float><<<static_cast<unsigned>(blocks), 256, 0, s>>>(in, spitch, static_cast<float*>(out), dpitch, rows, cols);
  return cudaGetLastError();
}

}  // namespace wam
