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
// out = x . W for a few items (the episodes of a step) and a [K, Nout] weight.  The input row of
// each item is formed while staging: the timestep features of the item's sigma, or
// act(sum over `in_splits` partial rows + in_bias).  A block owns CPB output columns (CPT per
// lane, 16-byte weight loads) and one K slice; its 8 warps split the slice and combine in
// shared memory.  With `splits` > 1 every block writes a partial row per K slice (no bias),
// which the next stage reduces in a fixed order; with one split the bias is added here.
template <typename TW> struct WVec;
template <> struct WVec<bf16> {
  static constexpr int kCPT = 8;
  static WAM_DEV void load(const bf16* W, int64_t idx, float (&w)[8]) {
    const uint4 u = __ldg(reinterpret_cast<const uint4*>(W + idx));
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(h[i]);
      w[2 * i] = f.x;
      w[2 * i + 1] = f.y;
    }
  }
};
template <> struct WVec<float> {
  static constexpr int kCPT = 4;
  static WAM_DEV void load(const float* W, int64_t idx, float (&w)[4]) {
    const float4 f = __ldg(reinterpret_cast<const float4*>(W + idx));
    w[0] = f.x;
    w[1] = f.y;
    w[2] = f.z;
    w[3] = f.w;
  }
};

// LPR lanes share one weight row piece of CPB = LPR * CPT columns; with LPR = 16 a warp works on
// two rows at a time (its half-warps take alternate rows of its K range) and a block covers half as
// many columns, so the bf16 modulation weight spreads over twice as many blocks (at one episode 222
// blocks of 256 columns filled 1.5 waves of the SMs and left the read latency-bound).
template <typename TW, int KB, int LPR>
__global__ void __launch_bounds__(256) cond_gemv_kernel(const float* __restrict__ in_part, int in_splits,
                                                        const float* __restrict__ in_bias, int in_act,
                                                        int features, const StepItem* __restrict__ items,
                                                        const TW* __restrict__ W, int K, int Nout, int Bw,
                                                        int kslice, float* __restrict__ out,
                                                        const float* __restrict__ out_bias) {
  pdl_wait();
  pdl_launch_dependents();
  constexpr int CPT = WVec<TW>::kCPT;
  constexpr int CPB = LPR * CPT;
  constexpr int HW = 32 / LPR;            // rows a warp works on at a time
  extern __shared__ float smem[];
  float* sx = smem;                       // [KB][kslice]
  float* red = smem + KB * kslice;        // [8][KB][CPB]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int sub = lane / LPR, lc = lane % LPR;
  const int k_beg = blockIdx.y * kslice;
  const int k_len = max(0, min(K, k_beg + kslice) - k_beg);
  const int col0 = blockIdx.x * CPB + lc * CPT;
  const int kw = (k_len + 7) / 8;
  const int kw0 = warp * kw, kw1 = min(k_len, kw0 + kw);
  const int64_t part_stride = static_cast<int64_t>(Bw) * K;
  for (int b0 = 0; b0 < Bw; b0 += KB) {
    const int nb = min(KB, Bw - b0);
    for (int i = threadIdx.x; i < KB * k_len; i += 256) {
      const int bi = i / k_len, kk = i - bi * k_len, k = k_beg + kk;
      float v = 0.0f;
      if (bi < nb) {
        if (features) {
          // cos / sin of 1000 sigma 10000^(-j/half), argument formed in float64
          const int half = K / 2;
          const int j = k < half ? k : k - half;
          const double f = exp(-log(10000.0) * static_cast<double>(j) / half);
          const double a = 1000.0 * items[b0 + bi].sigma * f;
          v = static_cast<float>(k < half ? cos(a) : sin(a));
        } else {
          float acc = in_bias != nullptr ? in_bias[k] : 0.0f;
          for (int sp = 0; sp < in_splits; ++sp) acc += in_part[sp * part_stride + static_cast<int64_t>(b0 + bi) * K + k];
          v = in_act ? silu_f(acc) : acc;
        }
      }
      sx[bi * kslice + kk] = v;
    }
    __syncthreads();
    float acc[KB][CPT];
#pragma unroll
    for (int bi = 0; bi < KB; ++bi)
#pragma unroll
      for (int c = 0; c < CPT; ++c) acc[bi][c] = 0.0f;
    if (col0 < Nout) {
      // eight weight rows in flight per thread before their first use (the weights stream from
      // HBM once per step; fewer loads in flight left the read latency-bound at one item)
      constexpr int kBatch = 8;
      int kk = kw0 + sub;
      for (; kk + HW * (kBatch - 1) < kw1; kk += HW * kBatch) {
        float w[kBatch][CPT];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) WVec<TW>::load(W, static_cast<int64_t>(k_beg + kk + HW * u) * Nout + col0, w[u]);
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
#pragma unroll
          for (int bi = 0; bi < KB; ++bi) {
            const float xv = sx[bi * kslice + kk + HW * u];
#pragma unroll
            for (int c = 0; c < CPT; ++c) acc[bi][c] = fmaf(xv, w[u][c], acc[bi][c]);
          }
        }
      }
      for (; kk < kw1; kk += HW) {
        float w[CPT];
        WVec<TW>::load(W, static_cast<int64_t>(k_beg + kk) * Nout + col0, w);
#pragma unroll
        for (int bi = 0; bi < KB; ++bi) {
          const float xv = sx[bi * kslice + kk];
#pragma unroll
          for (int c = 0; c < CPT; ++c) acc[bi][c] = fmaf(xv, w[c], acc[bi][c]);
        }
      }
    }
    if constexpr (HW == 2) {   // the half-warps' alternate rows, combined in a fixed order
#pragma unroll
      for (int bi = 0; bi < KB; ++bi)
#pragma unroll
        for (int c = 0; c < CPT; ++c) acc[bi][c] += __shfl_xor_sync(0xffffffffu, acc[bi][c], 16);
    }
    if (sub == 0) {
#pragma unroll
      for (int bi = 0; bi < KB; ++bi)
#pragma unroll
        for (int c = 0; c < CPT; ++c) red[(warp * KB + bi) * CPB + lc * CPT + c] = acc[bi][c];
    }
    __syncthreads();
    for (int i = threadIdx.x; i < nb * CPB; i += 256) {
      const int bi = i / CPB, cc = i - bi * CPB;
      const int col = blockIdx.x * CPB + cc;
      if (col < Nout) {
        float sum = 0.0f;
#pragma unroll
        for (int w = 0; w < 8; ++w) sum += red[(w * KB + bi) * CPB + cc];
        if (out_bias != nullptr) sum += out_bias[col];
        out[static_cast<int64_t>(blockIdx.y) * Bw * Nout + static_cast<int64_t>(b0 + bi) * Nout + col] = sum;
      }
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------- token embedding
// One warp per group of kEmbRows consecutive token rows and one 128-column slice (blockIdx.y): each
// lane loads the embedding weights of its float4 column once and applies them to every video (or
// action) row of the group, so the weight reads from L1 shrink by the group size (one warp per row
// read 16 weight values per output value and was bound by L1, not HBM).  The trajectory values of
// the group's rows sit in shared memory; the slice-0 warps record them in the stage history.  Per
// output: acc = b, then acc = fma(x_i, W_i, acc) for i in order, then + pos.  The position values
// of four rows are requested before their products, and the register budget keeps two blocks per
// SM (46 vs 51 us per launch at 8 serving episodes, 11.7 vs 13.5 us at one episode).
constexpr int kEmbRows = 8;

__global__ void __launch_bounds__(256, 2) embed_kernel(
    float* __restrict__ h, float* __restrict__ xhist, int64_t stage_stride,
    const StepItem* __restrict__ items, const float* __restrict__ x, int T,
    const float* __restrict__ obs_emb, const float* __restrict__ vid_w,
    const float* __restrict__ vid_b, const float* __restrict__ act_w,
    const float* __restrict__ act_b, const float* __restrict__ pos, int Bw, int No, int Nv,
    int vd, int Na, int ad, int d) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ float xs[kRowWarps][kEmbRows][16];
  __shared__ int rinfo[kRowWarps][kEmbRows][3];   // kind (-1 none, 0 obs, 1 video, 2 action), n, episode
  const int N = No + Nv + Na;
  const int wib = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t row0 = (static_cast<int64_t>(blockIdx.x) * kRowWarps + wib) * kEmbRows;
  const int64_t rows = static_cast<int64_t>(Bw) * N;
  if (row0 >= rows) return;
  if (lane < kEmbRows) {
    const int64_t gw = row0 + lane;
    int kind = -1, n = 0, ep = 0;
    if (gw < rows) {
      const int w = static_cast<int>(gw / N);
      n = static_cast<int>(gw % N);
      ep = items[w].ep;
      kind = n < No ? 0 : (n < No + Nv ? 1 : 2);
    }
    rinfo[wib][lane][0] = kind;
    rinfo[wib][lane][1] = n;
    rinfo[wib][lane][2] = ep;
  }
  __syncwarp();
  // the group's trajectory values, and the record of the latent entering this stage
  bool any_v = false, any_a = false;
  for (int j = lane; j < kEmbRows * 16; j += 32) {
    const int r = j >> 4, i = j & 15;
    const int kind = rinfo[wib][r][0], n = rinfo[wib][r][1], ep = rinfo[wib][r][2];
    float v = 0.0f;
    if (kind >= 1) {
      const int in_dim = kind == 1 ? vd : ad;
      const int64_t xoff = static_cast<int64_t>(ep) * T +
                           (kind == 1 ? static_cast<int64_t>(n - No) * vd
                                      : static_cast<int64_t>(Nv) * vd + static_cast<int64_t>(n - No - Nv) * ad);
      if (i < in_dim) {
        v = x[xoff + i];
        if (blockIdx.y == 0) {
          const int stage = items[(row0 + r) / N].stage;
          xhist[static_cast<int64_t>(stage) * stage_stride + xoff + i] = v;
        }
      }
    }
    xs[wib][r][i] = v;
  }
#pragma unroll
  for (int r = 0; r < kEmbRows; ++r) {
    any_v |= rinfo[wib][r][0] == 1;
    any_a |= rinfo[wib][r][0] == 2;
  }
  __syncwarp();
  const int d4 = d / 4;
  const int c = blockIdx.y * 32 + lane;
  if (c < d4) {
#pragma unroll
    for (int r = 0; r < kEmbRows; ++r) {
      if (rinfo[wib][r][0] != 0) continue;
      const int n = rinfo[wib][r][1], ep = rinfo[wib][r][2];
      const float4 a = reinterpret_cast<const float4*>(obs_emb + (static_cast<int64_t>(ep) * No + n) * d)[c];
      const float4 p = reinterpret_cast<const float4*>(pos + static_cast<int64_t>(n) * d)[c];
      reinterpret_cast<float4*>(h + (row0 + r) * d)[c] = make_float4(a.x + p.x, a.y + p.y, a.z + p.z, a.w + p.w);
    }
    for (int kind = 1; kind <= 2; ++kind) {
      if (kind == 1 ? !any_v : !any_a) continue;
      const int in_dim = kind == 1 ? vd : ad;
      const float4* W4 = reinterpret_cast<const float4*>(kind == 1 ? vid_w : act_w);
      float4 wv[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) wv[i] = i < in_dim ? W4[static_cast<int64_t>(i) * d4 + c] : make_float4(0.f, 0.f, 0.f, 0.f);
      const float4 bias = reinterpret_cast<const float4*>(kind == 1 ? vid_b : act_b)[c];
      // the position values of four rows requested before their products (a round trip per four
      // rows instead of one per row)
#pragma unroll
      for (int r0 = 0; r0 < kEmbRows; r0 += 4) {
      float4 pv[4];
#pragma unroll
      for (int q = 0; q < 4; ++q)
        pv[q] = rinfo[wib][r0 + q][0] == kind
                    ? reinterpret_cast<const float4*>(pos + static_cast<int64_t>(rinfo[wib][r0 + q][1]) * d)[c]
                    : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int r = r0 + q;
        if (rinfo[wib][r][0] != kind) continue;
        float4 acc = bias;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          if (i < in_dim) {
            const float xi = xs[wib][r][i];
            acc.x = fmaf(xi, wv[i].x, acc.x);
            acc.y = fmaf(xi, wv[i].y, acc.y);
            acc.z = fmaf(xi, wv[i].z, acc.z);
            acc.w = fmaf(xi, wv[i].w, acc.w);
          }
        }
        const float4 p = pv[q];
        reinterpret_cast<float4*>(h + (row0 + r) * d)[c] = make_float4(acc.x + p.x, acc.y + p.y, acc.z + p.z, acc.w + p.w);
      }
      }
    }
  }
}

// ---------------------------------------------------------------- LN modulate
template <int NV4, typename TO>
__global__ void __launch_bounds__(256) ln_mod_kernel(const float* __restrict__ h,
                                                     float* __restrict__ hcopy,
                                                     const float* __restrict__ mods,
                                                     int64_t mod_stride, int shift_off,
                                                     int scale_off,
                                                     const int* __restrict__ item_map,
                                                     TO* __restrict__ out, int M, int d,
                                                     int rows_per_item) {
  pdl_wait();
  pdl_launch_dependents();
  const int64_t row = static_cast<int64_t>(blockIdx.x) * kRowWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= M) return;
  const float4* hr = reinterpret_cast<const float4*>(h + row * d);
  int item = static_cast<int>(row / rows_per_item);
  if (item_map != nullptr) item = item_map[item];
  const float* shift = mods + item * mod_stride + shift_off;
  const float* scale = mods + item * mod_stride + scale_off;
  // the row and its modulation are requested together: one memory round trip, not two
  float4 v[NV4], sh[NV4], sc[NV4];
#pragma unroll
  for (int i = 0; i < NV4; ++i) {
    v[i] = hr[lane + 32 * i];
    sh[i] = *reinterpret_cast<const float4*>(shift + (lane + 32 * i) * 4);
    sc[i] = *reinterpret_cast<const float4*>(scale + (lane + 32 * i) * 4);
  }
  if (hcopy != nullptr) {
    float4* cr = reinterpret_cast<float4*>(hcopy + row * d);
#pragma unroll
    for (int i = 0; i < NV4; ++i) cr[lane + 32 * i] = v[i];
  }
  float mean, rstd;
  row_stats<NV4>(v, d, mean, rstd);
#pragma unroll
  for (int i = 0; i < NV4; ++i) {
    const int c = (lane + 32 * i) * 4;
    Act<TO>::store4(out + row * d + c, fmaf((v[i].x - mean) * rstd, 1.0f + sc[i].x, sh[i].x),
                    fmaf((v[i].y - mean) * rstd, 1.0f + sc[i].y, sh[i].y),
                    fmaf((v[i].z - mean) * rstd, 1.0f + sc[i].z, sh[i].z),
                    fmaf((v[i].w - mean) * rstd, 1.0f + sc[i].w, sh[i].w));
  }
}

// ---------------------------------------------------------------- final layer + Euler
// Modulated LN of a token row, the output head (16 columns; the [d, 16] heads are zero-padded),
// the Euler update of that token's trajectory values and their retention.  The modulation is
// folded into the head once per work item (final_head_prep_kernel): LN(h)(1+scale)+shift
// times W equals xhat . W' + c with W'[k][j] = (1+scale[k]) W[k][j] and
// c[j] = b[j] + sum_k shift[k] W[k][j], where xhat = (h - mean) rstd.  A block serves a
// contiguous range of one item's video (or action) rows and copies only that head's W'.
//
// Float32 precision mode: SIMT dot products, a warp per row pair (each weight read from shared
// memory serves both rows).  Bf16 precision mode: the head is a [rows, d] x [d, 16] product on
// the tensor cores (mma.sync m16n8k16, bf16 operands, float32 accumulation), a warp per 16-row
// tile, with the row statistics gathered from the same loads; 16 products per loaded element
// would otherwise bound the kernel on the FMA pipe instead of HBM.

// Reduce-scatter 16 partial outputs over the warp: lane l ends with output (l & 15).
WAM_DEV float reduce_scatter16(float (&acc)[16], int lane) {
#pragma unroll
  for (int sft = 8; sft >= 1; sft >>= 1) {
    const bool upper = (lane & sft) != 0;
#pragma unroll
    for (int j = 0; j < sft; ++j) {
      const float send = upper ? acc[j] : acc[j + sft];
      const float keep = upper ? acc[j + sft] : acc[j];
      acc[j] = keep + __shfl_xor_sync(0xffffffffu, send, sft);
    }
  }
  return acc[0] + __shfl_xor_sync(0xffffffffu, acc[0], 16);
}

// Normalised row: xhat = (h - mean) rstd, lane-strided float4s (element c = 4 (lane + 32 i)).
template <int NV4>
WAM_DEV void ln_row(const float* __restrict__ hrow, int d, int lane, float4 (&y)[NV4]) {
  const float4* hr = reinterpret_cast<const float4*>(hrow);
#pragma unroll
  for (int i = 0; i < NV4; ++i) y[i] = hr[lane + 32 * i];
  float mean, rstd;
  row_stats<NV4>(y, d, mean, rstd);
#pragma unroll
  for (int i = 0; i < NV4; ++i)
    y[i] = make_float4((y[i].x - mean) * rstd, (y[i].y - mean) * rstd, (y[i].z - mean) * rstd, (y[i].w - mean) * rstd);
}

// Which rows a block of the final kernel serves: blocks [0, vblocks) split an item's video rows,
// the rest its action rows, in contiguous ranges of `gran`-row units.
struct HeadRange {
  bool video;
  int beg, end;  // token rows within the head
};
WAM_DEV HeadRange head_range(int bx, int vblocks, int ablocks, int Nv, int Na, int gran) {
  HeadRange r;
  r.video = bx < vblocks;
  const int part = r.video ? bx : bx - vblocks;
  const int nparts = r.video ? vblocks : ablocks;
  const int nrows = r.video ? Nv : Na;
  const int units = (nrows + gran - 1) / gran;
  const int per = (units + nparts - 1) / nparts;
  r.beg = min(nrows, part * per * gran);
  r.end = min(nrows, (part + 1) * per * gran);
  return r;
}

// Euler update x <- x + dsigma v of one trajectory value (its current value xv read earlier, so
// that callers can issue those loads before any store), retained as x^{k+1} and v^k.
WAM_DEV void euler_store(const StepItem& it, int64_t idx, float xv, float vel, float* __restrict__ x,
                         float* __restrict__ xhist, float* __restrict__ vhist, int64_t stage_stride) {
  const float xn = static_cast<float>(static_cast<double>(xv) + it.dsigma * static_cast<double>(vel));
  x[idx] = xn;
  xhist[static_cast<int64_t>(it.stage + 1) * stage_stride + idx] = xn;
  vhist[static_cast<int64_t>(it.stage) * stage_stride + idx] = vel;
}

// Head preparation, one block per (head, work item): W' = (1 + scale) W in the layout its
// final kernel reads (float32 [16][d], or bf16 [16][d + 8]), c[j] = b[j] + sum_k shift[k] W[k][j]
// and, for the bf16 layout, colsum[j] = sum_k W'_bf16[k][j].  Thread t covers k = t, t + 256, ..:
// one pass over the [d, 16] head with every load of the pass issued together, then a block
// reduction of the 32 sums.  Writes hw + (item * 2 + head) * head_stride bytes and
// hc[(item * 2 + head) * 32 + (0..15: c, 16..31: colsum)].
template <bool HB>
__global__ void __launch_bounds__(256) final_head_prep_kernel(
    const float* __restrict__ mods, int64_t mod_stride, int fin_off, const float* __restrict__ vout_w,
    const float* __restrict__ vout_b, const float* __restrict__ aout_w, const float* __restrict__ aout_b,
    int d, int vd, int ad, int Nv, int Na, uint8_t* __restrict__ hw, int64_t head_stride, float* __restrict__ hc) {
  __shared__ float red[8][32];
  pdl_wait();
  pdl_launch_dependents();
  const int head = blockIdx.x, w = blockIdx.y;
  if ((head == 0 ? Nv : Na) == 0) return;
  const float* Wg = head == 0 ? vout_w : aout_w;
  const float* shift = mods + w * mod_stride + fin_off;
  const float* scale = shift + d;
  uint8_t* dst = hw + (static_cast<int64_t>(w) * 2 + head) * head_stride;
  const int ld = d + 8;
  float cacc[16], sacc[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) cacc[j] = sacc[j] = 0.0f;
  for (int k = threadIdx.x; k < d; k += blockDim.x) {
    const float4* wr = reinterpret_cast<const float4*>(Wg + static_cast<int64_t>(k) * 16);
    const float4 q0 = wr[0], q1 = wr[1], q2 = wr[2], q3 = wr[3];
    const float wv[16] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w,
                          q2.x, q2.y, q2.z, q2.w, q3.x, q3.y, q3.z, q3.w};
    const float sc = 1.0f + scale[k], sh = shift[k];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const float wp = wv[j] * sc;
      cacc[j] = fmaf(sh, wv[j], cacc[j]);
      if constexpr (HB) {
        const bf16 b = __float2bfloat16(wp);
        reinterpret_cast<bf16*>(dst)[j * ld + k] = b;
        sacc[j] += __bfloat162float(b);
      } else {
        reinterpret_cast<float*>(dst)[j * d + k] = wp;
      }
    }
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const float a = warp_sum(cacc[j]);
    const float b = warp_sum(sacc[j]);
    if (lane == 0) {
      red[warp][j] = a;
      red[warp][16 + j] = b;
    }
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = 0.0f;
    for (int q = 0; q < static_cast<int>(blockDim.x >> 5); ++q) v += red[q][threadIdx.x];
    const int j = threadIdx.x & 15;
    const int od = head == 0 ? vd : ad;
    if (threadIdx.x < 16) v += j < od ? (head == 0 ? vout_b : aout_b)[j] : 0.0f;
    hc[(static_cast<int64_t>(w) * 2 + head) * 32 + threadIdx.x] = v;
  }
}

// Copy `bytes` (a multiple of 16) from global to shared memory, eight 16-byte loads in flight
// per thread.
WAM_DEV void copy_to_smem(void* sdst, const void* gsrc, int bytes) {
  const uint4* src = static_cast<const uint4*>(gsrc);
  uint4* dst = static_cast<uint4*>(sdst);
  const int n = bytes / 16;
  for (int i0 = threadIdx.x; i0 < n; i0 += 8 * blockDim.x) {
    uint4 v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int i = i0 + u * blockDim.x;
      if (i < n) v[u] = src[i];
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int i = i0 + u * blockDim.x;
      if (i < n) dst[i] = v[u];
    }
  }
}

// grid (video blocks + action blocks per item, items); block = 8 warps.
template <int NV4>
__global__ void __launch_bounds__(256, NV4 <= 8 ? 2 : 1) final_euler_kernel(
    const float* __restrict__ h, const StepItem* __restrict__ items, float* __restrict__ x,
    float* __restrict__ xhist, float* __restrict__ vhist, int64_t stage_stride, int T, int No,
    int Nv, int vd, int Na, int ad, int d, int vblocks, int ablocks, const uint8_t* __restrict__ hw,
    int64_t head_stride, const float* __restrict__ hc) {
  extern __shared__ __align__(16) uint8_t fe_smem[];
  __shared__ float cvec[16];
  pdl_wait();
  pdl_launch_dependents();
  const int w = blockIdx.y;
  const HeadRange hr = head_range(blockIdx.x, vblocks, ablocks, Nv, Na, 2);
  if (hr.beg >= hr.end) return;  // whole block: no barrier below is skipped by only some threads
  const bool video = hr.video;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int hidx = w * 2 + (video ? 0 : 1);
  float* Ws = reinterpret_cast<float*>(fe_smem);  // [16][d], prepared by final_head_prep_kernel
  copy_to_smem(Ws, hw + hidx * head_stride, 16 * d * 4);
  if (threadIdx.x < 16) cvec[threadIdx.x] = hc[hidx * 32 + threadIdx.x];
  const int od = video ? vd : ad;
  __syncthreads();
  const StepItem it = items[w];
  const int N = No + Nv + Na;
  const int row0 = No + (video ? 0 : Nv);  // first token row of this head
  const int64_t tbase = static_cast<int64_t>(it.ep) * T + (video ? 0 : static_cast<int64_t>(Nv) * vd);
  for (int r = hr.beg + 2 * warp; r < hr.end; r += 2 * kRowWarps) {
    const bool two = r + 1 < hr.end;
    const int64_t i0 = tbase + static_cast<int64_t>(r) * od + lane, i1 = i0 + od;
    const float x0 = lane < od ? x[i0] : 0.0f;
    const float x1 = (lane < od && two) ? x[i1] : 0.0f;
    float4 y0[NV4], y1[NV4];
    ln_row<NV4>(h + (static_cast<int64_t>(w) * N + row0 + r) * d, d, lane, y0);
    if (two) ln_row<NV4>(h + (static_cast<int64_t>(w) * N + row0 + r + 1) * d, d, lane, y1);
    float acc0[16], acc1[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) acc0[j] = acc1[j] = 0.0f;
#pragma unroll
    for (int i = 0; i < NV4; ++i) {
      const int c = (lane + 32 * i) * 4;
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const float4 wv = *reinterpret_cast<const float4*>(Ws + j * d + c);
        acc0[j] = fmaf(y0[i].x, wv.x, fmaf(y0[i].y, wv.y, fmaf(y0[i].z, wv.z, fmaf(y0[i].w, wv.w, acc0[j]))));
        if (two)
          acc1[j] = fmaf(y1[i].x, wv.x, fmaf(y1[i].y, wv.y, fmaf(y1[i].z, wv.z, fmaf(y1[i].w, wv.w, acc1[j]))));
      }
    }
    const float out0 = reduce_scatter16(acc0, lane);
    const float out1 = reduce_scatter16(acc1, lane);
    if (lane < od) {
      const float cj = cvec[lane];
      euler_store(it, i0, x0, out0 + cj, x, xhist, vhist, stage_stride);
      if (two) euler_store(it, i1, x1, out1 + cj, x, xhist, vhist, stage_stride);
    }
  }
}

WAM_DEV uint32_t bf16x2_bits(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

WAM_DEV void mma_bf16_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                            uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

constexpr int kFtWarps = 4;   // warps per block of the tensor-core final kernel (one K quarter each)
constexpr int kFtUnroll = 8;  // k-steps of 16 whose loads are issued together

// Bf16 precision mode.  A block takes 16-row tiles one at a time; warp q covers the K quarter
// [q d / 4, (q + 1) d / 4) of the tile, so a row tile costs few dependent load batches even at
// one episode.  Lane (g = lane / 4, c = lane % 4) loads rows g and g + 8 at columns
// k0 + 4c .. k0 + 4c + 3 of every 16-column step; the fragment's logical k order
// {2c, 2c+1, 2c+8, 2c+9} is mapped to these physical columns for both operands (a sum over k
// does not depend on the order), so each row slice is one 16-byte load.  Row statistics are
// accumulated from the same values around a per-row reference K (the row's first element) and
// the tensor cores see bf16(h - K):  sum_k (h_k - mean) W'_kj = acc_j - (mean - K) colsum_j.
// The four quarters' partial accumulators and sums meet in shared memory and are added in
// warp order by warp 0, which applies the Euler update.  W' is the prepared bf16 [16][d + 8]
// copy (the pad makes the 8-byte reads of a warp conflict-free).
__global__ void __launch_bounds__(32 * kFtWarps) final_euler_tc_kernel(
    const float* __restrict__ h, const StepItem* __restrict__ items, float* __restrict__ x,
    float* __restrict__ xhist, float* __restrict__ vhist, int64_t stage_stride, int T, int No,
    int Nv, int vd, int Na, int ad, int d, int vblocks, int ablocks, const uint8_t* __restrict__ hw,
    int64_t head_stride, const float* __restrict__ hc) {
  extern __shared__ __align__(16) uint8_t fe_smem[];
  __shared__ float cvec[16], colsum[16];
  __shared__ float part[kFtWarps][12][32];  // per quarter: 8 accumulators + 4 row sums, per lane
  pdl_wait();
  pdl_launch_dependents();
  const int w = blockIdx.y;
  const HeadRange hr = head_range(blockIdx.x, vblocks, ablocks, Nv, Na, 16);
  if (hr.beg >= hr.end) return;  // whole block: no barrier below is skipped by only some threads
  const bool video = hr.video;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int ld = d + 8;
  const int hidx = w * 2 + (video ? 0 : 1);
  bf16* Ws = reinterpret_cast<bf16*>(fe_smem);  // [16][d + 8], prepared by final_head_prep_kernel
  copy_to_smem(Ws, hw + hidx * head_stride, 16 * ld * 2);
  if (threadIdx.x < 32) (threadIdx.x < 16 ? cvec : colsum)[threadIdx.x & 15] = hc[hidx * 32 + threadIdx.x];
  const int od = video ? vd : ad;
  __syncthreads();
  const StepItem it = items[w];
  const int N = No + Nv + Na;
  const int row0 = No + (video ? 0 : Nv);
  const int64_t tbase = static_cast<int64_t>(it.ep) * T + (video ? 0 : static_cast<int64_t>(Nv) * vd);
  const int g = lane >> 2, c = lane & 3;
  const int ks = d / kFtWarps;  // K quarter (a multiple of 32: d is a multiple of 128)
  const uint32_t wsa = static_cast<uint32_t>(__cvta_generic_to_shared(Ws)) + static_cast<uint32_t>(warp * ks * 2);
  for (int r0 = hr.beg; r0 < hr.end; r0 += 16) {
    const int ra = r0 + g, rb = r0 + g + 8;
    const bool va = ra < hr.end, vb = rb < hr.end;
    const float* rowa = h + (static_cast<int64_t>(w) * N + row0 + (va ? ra : r0)) * d;
    const float* rowb = h + (static_cast<int64_t>(w) * N + row0 + (vb ? rb : r0)) * d;
    const float Ka = va ? rowa[0] : 0.0f, Kb = vb ? rowb[0] : 0.0f;
    const float* pa = rowa + warp * ks + 4 * c;
    const float* pb = rowb + warp * ks + 4 * c;
    // This warp finishes accumulator entries 2 warp and 2 warp + 1 (n-tile warp / 2; row g for
    // even warps, g + 8 for odd; columns 2c, 2c + 1): their trajectory values are read now.
    const bool top = (warp & 1) == 0;
    const int jbase = 8 * (warp >> 1) + 2 * c;
    const bool vrow = top ? va : vb;
    const int64_t ibase = tbase + static_cast<int64_t>(top ? ra : rb) * od;
    float xv[2];
#pragma unroll
    for (int e = 0; e < 2; ++e) xv[e] = (vrow && jbase + e < od) ? x[ibase + jbase + e] : 0.0f;
    float acc0[4] = {0.f, 0.f, 0.f, 0.f}, acc1[4] = {0.f, 0.f, 0.f, 0.f};
    float s1a = 0.f, s2a = 0.f, s1b = 0.f, s2b = 0.f;
    for (int k0 = 0; k0 < ks; k0 += 16 * kFtUnroll) {
      float4 xa[kFtUnroll], xb[kFtUnroll];
#pragma unroll
      for (int u = 0; u < kFtUnroll; ++u) {
        const bool in = k0 + 16 * u < ks;
        xa[u] = (va && in) ? *reinterpret_cast<const float4*>(pa + k0 + 16 * u) : make_float4(Ka, Ka, Ka, Ka);
        xb[u] = (vb && in) ? *reinterpret_cast<const float4*>(pb + k0 + 16 * u) : make_float4(Kb, Kb, Kb, Kb);
      }
#pragma unroll
      for (int u = 0; u < kFtUnroll; ++u) {
        const int kk = k0 + 16 * u;
        if (kk >= ks) break;
        const float a0 = xa[u].x - Ka, a1 = xa[u].y - Ka, a2 = xa[u].z - Ka, a3 = xa[u].w - Ka;
        const float b0 = xb[u].x - Kb, b1 = xb[u].y - Kb, b2 = xb[u].z - Kb, b3 = xb[u].w - Kb;
        s1a += (a0 + a1) + (a2 + a3);
        s2a = fmaf(a0, a0, fmaf(a1, a1, fmaf(a2, a2, fmaf(a3, a3, s2a))));
        s1b += (b0 + b1) + (b2 + b3);
        s2b = fmaf(b0, b0, fmaf(b1, b1, fmaf(b2, b2, fmaf(b3, b3, s2b))));
        const uint32_t A0 = bf16x2_bits(a0, a1), A2 = bf16x2_bits(a2, a3);
        const uint32_t A1 = bf16x2_bits(b0, b1), A3 = bf16x2_bits(b2, b3);
        uint32_t B0, B1, C0, C1;  // outputs g (n-tile 0) and g + 8 (n-tile 1), columns kk + 4c ..
        asm volatile("ld.shared.v2.b32 {%0, %1}, [%2];"
                     : "=r"(B0), "=r"(B1)
                     : "r"(wsa + static_cast<uint32_t>((g * ld + kk + 4 * c) * 2)));
        asm volatile("ld.shared.v2.b32 {%0, %1}, [%2];"
                     : "=r"(C0), "=r"(C1)
                     : "r"(wsa + static_cast<uint32_t>(((g + 8) * ld + kk + 4 * c) * 2)));
        mma_bf16_16816(acc0, A0, A1, A2, A3, B0, B1);
        mma_bf16_16816(acc1, A0, A1, A2, A3, C0, C1);
      }
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      part[warp][e][lane] = acc0[e];
      part[warp][4 + e][lane] = acc1[e];
    }
    part[warp][8][lane] = s1a;
    part[warp][9][lane] = s2a;
    part[warp][10][lane] = s1b;
    part[warp][11][lane] = s2b;
    __syncthreads();
    {
      // the row's sums (entries 8, 9 for row g; 10, 11 for row g + 8), added over the quarters in
      // warp order, then over the 4 lanes that share the row
      const int se = top ? 8 : 10;
      float s1 = part[0][se][lane], s2 = part[0][se + 1][lane];
#pragma unroll
      for (int q = 1; q < kFtWarps; ++q) {
        s1 += part[q][se][lane];
        s2 += part[q][se + 1][lane];
      }
      s1 += __shfl_xor_sync(0xffffffffu, s1, 1);
      s1 += __shfl_xor_sync(0xffffffffu, s1, 2);
      s2 += __shfl_xor_sync(0xffffffffu, s2, 1);
      s2 += __shfl_xor_sync(0xffffffffu, s2, 2);
      const float inv_d = 1.0f / static_cast<float>(d);
      const float m = s1 * inv_d;  // mean - K
      const float rs = rsqrtf(fmaxf(s2 * inv_d - m * m, 0.0f) + 1e-6f);
      // accumulator layout: entries 4 n + {0, 1} row g, 4 n + {2, 3} row g + 8 of n-tile n
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int pe = 2 * warp + e;
        const int j = jbase + e;
        if (!vrow || j >= od) continue;
        float tot = part[0][pe][lane];
#pragma unroll
        for (int q = 1; q < kFtWarps; ++q) tot += part[q][pe][lane];
        const float vel = rs * (tot - m * colsum[j]) + cvec[j];
        euler_store(it, ibase + j, xv[e], vel, x, xhist, vhist, stage_stride);
      }
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------- Trajectory Remapping
__global__ void __launch_bounds__(256) tr_rms_partial_kernel(const AdaptItem* __restrict__ items,
                                                             const float* __restrict__ xhist,
                                                             int64_t stage_stride, int K, int T,
                                                             int V, int nch,
                                                             double* __restrict__ partial) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ float red[2][8];
  const int b = blockIdx.z, br = blockIdx.y, ch = blockIdx.x;
  const AdaptItem it = items[b];
  float hi = 0.0f, lo = 0.0f;
  if (it.op == kAdaptTR) {
    const int beg = br == 0 ? 0 : V;
    const int len = br == 0 ? V : T - V;
    const float* xr = xhist + it.r * stage_stride + static_cast<int64_t>(b) * T + beg;
    const float* xb = xhist + K * stage_stride + static_cast<int64_t>(b) * T + beg;
    const int end = min(len, (ch + 1) * kTrChunk);
    // every load of the chunk issued before the first use (the chunk is 8 rows of the block)
    constexpr int kPer = kTrChunk / 256;
    static_assert(kTrChunk % 256 == 0, "TR chunk is whole rows of the block");
    float a[kPer], c[kPer];
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int i = ch * kTrChunk + u * 256 + threadIdx.x;
      a[u] = i < end ? xr[i] : 0.0f;
      c[u] = i < end ? xb[i] : 0.0f;
    }
    // sum of (x^r - x_bar)^2 in double-float (float64 runs at a small fraction of the float32
    // rate on this part); the block total is scaled by 1 / sigma_r^2 once, in float64
#pragma unroll
    for (int u = 0; u < kPer; ++u) df_add_sq_diff(a[u], c[u], hi, lo);
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
    partial[(static_cast<int64_t>(b) * 2 + br) * nch + ch] =
        it.op == kAdaptTR ? s * (1.0 / (it.sigma_r * it.sigma_r)) : 0.0;
  }
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
  pdl_wait();
  pdl_launch_dependents();
  __shared__ double rms[2], gain[2];
  __shared__ float gain_hi[2], gain_lo[2];
  __shared__ int zero[2];
  const int b = blockIdx.y;
  const AdaptItem it = items[b];
  if (it.op == kAdaptNone && !it.bind_obs) return;
  if (static_cast<int>(blockIdx.x) >= traj_blocks) {
    if (!it.bind_obs) return;
    // obs_elems = No * d with d a multiple of 128: whole float4s, four in flight per thread
    const int64_t n4 = obs_elems / 4;
    const float4* src = reinterpret_cast<const float4*>(obs_new + static_cast<int64_t>(b) * obs_elems);
    float4* dst = reinterpret_cast<float4*>(obs + static_cast<int64_t>(b) * obs_elems);
    const int64_t stride = static_cast<int64_t>(gridDim.x - traj_blocks) * blockDim.x;
    int64_t i = static_cast<int64_t>(blockIdx.x - traj_blocks) * blockDim.x + threadIdx.x;
    for (; i + 3 * stride < n4; i += 4 * stride) {
      const float4 v0 = src[i], v1 = src[i + stride], v2 = src[i + 2 * stride], v3 = src[i + 3 * stride];
      dst[i] = v0;
      dst[i + stride] = v1;
      dst[i + 2 * stride] = v2;
      dst[i + 3 * stride] = v3;
    }
    for (; i < n4; i += stride) dst[i] = src[i];
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
    // direction scale of Eq. 2 for this branch: sigma_b0 / (sigma_r rms); one float64 division
    // here instead of two per element
    gain[threadIdx.x] = zero[threadIdx.x] ? 0.0 : it.sigma_b0 / (it.sigma_r * rms[threadIdx.x]);
    // the gain as a float pair for the per-element remap (float64 arithmetic per element bound
    // this kernel on GB300's float64 rate)
    gain_hi[threadIdx.x] = static_cast<float>(gain[threadIdx.x]);
    gain_lo[threadIdx.x] = static_cast<float>(gain[threadIdx.x] - static_cast<double>(gain_hi[threadIdx.x]));
  }
  __syncthreads();
  const int64_t bo = static_cast<int64_t>(b) * T;
  const float* xr = xhist + it.r * stage_stride + bo;
  const float* xb = xhist + K * stage_stride + bo;
  const int stride = traj_blocks * blockDim.x;
  // Four elements per thread and pass, every load issued before the first store.
  for (int j0 = blockIdx.x * blockDim.x + threadIdx.x; j0 < T; j0 += 4 * stride) {
    float val[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int j = j0 + u * stride;
      val[u] = 0.0f;
      if (j >= T) continue;
      if (it.op == kAdaptCold) {
        val[u] = eps[bo + j];
      } else if (it.op == kAdaptRestart) {
        val[u] = xb0[bo + j];
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
          val[u] = df_remap(xr[src], xb[src], gain_hi[br], gain_lo[br]);
        } else {
          val[u] = static_cast<float>(it.sigma_b0 * static_cast<double>(eps[bo + j]));
        }
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int j = j0 + u * stride;
      if (j >= T) continue;
      x[bo + j] = val[u];
      if (it.op != kAdaptRestart) xb0[bo + j] = val[u];
    }
  }
}

// ---------------------------------------------------------------- Observation Rebinding
__global__ void __launch_bounds__(256) or_partial_kernel(const float* __restrict__ pred,
                                                         const float* __restrict__ real,
                                                         int64_t obs_elems, int M,
                                                         float4 inv_delta, int nch,
                                                         double* __restrict__ partial) {
  pdl_wait();
  pdl_launch_dependents();
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
  pdl_wait();
  pdl_launch_dependents();
  __shared__ float red3[8][3];
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
  // the chunk is 8 float4 rows of the block: two batches of four rows, loads issued first
  for (int64_t i0 = beg4 + threadIdx.x; i0 < end4; i0 += 4 * blockDim.x) {
    float4 hv[4], qv[4], av[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t i = i0 + u * blockDim.x;
      const bool in = i < end4;
      hv[u] = in ? h4[i] : make_float4(0.f, 0.f, 0.f, 0.f);
      qv[u] = in ? q4[i] : make_float4(0.f, 0.f, 0.f, 0.f);
      av[u] = in ? a4[i] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float p0 = hv[u].x - qv[u].x, p1 = hv[u].y - qv[u].y, p2 = hv[u].z - qv[u].z, p3 = hv[u].w - qv[u].w;
      sia += (p0 * av[u].x + p1 * av[u].y) + (p2 * av[u].z + p3 * av[u].w);
      saa += (av[u].x * av[u].x + av[u].y * av[u].y) + (av[u].z * av[u].z + av[u].w * av[u].w);
      sii += (p0 * p0 + p1 * p1) + (p2 * p2 + p3 * p3);
    }
  }
  // The three block sums share one barrier: float32 warp trees, then thread 0 adds the warps in
  // order; the chunk partials are combined in float64 by the gate.  (Float64 arithmetic runs at
  // a small fraction of the float32 rate here: a float64 tree per chunk bounded this kernel.)
  const float w0 = warp_sum(sia), w1 = warp_sum(saa), w2 = warp_sum(sii);
  const int wi = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) {
    red3[wi][0] = w0;
    red3[wi][1] = w1;
    red3[wi][2] = w2;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float t0 = 0.0f, t1 = 0.0f, t2 = 0.0f;
    for (int v = 0; v < (blockDim.x >> 5); ++v) {
      t0 += red3[v][0];
      t1 += red3[v][1];
      t2 += red3[v][2];
    }
    double* out = partial + ((static_cast<int64_t>(w) * 2 + br) * nch + ch) * 3;
    out[0] = t0;
    out[1] = t1;
    out[2] = t2;
  }
}

// alpha (Eq. 7), cosine and relative fit (Eq. 8) per (item, branch): one warp per pair, the
// partial sums combined lane-strided then by a fixed shuffle tree (deterministic order).
__global__ void rr_gate_kernel(const double* __restrict__ partial, int Bw, int nch, int64_t n0,
                               int64_t n1, double amin, double amax, double eps, double gcos,
                               double gfit, RRGate* __restrict__ out) {
  pdl_wait();
  pdl_launch_dependents();
  const int i = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (i >= Bw * 2) return;
  const double* p = partial + static_cast<int64_t>(i) * nch * 3;
  double sia = 0.0, saa = 0.0, sii = 0.0;
  for (int c = lane; c < nch; c += 32) {
    sia += p[3 * c];
    saa += p[3 * c + 1];
    sii += p[3 * c + 2];
  }
  sia = warp_sum_d(sia);
  saa = warp_sum_d(saa);
  sii = warp_sum_d(sii);
  if (lane != 0) return;
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

// Device-side RR decision of a single work item (§3.3 branch rule: every non-empty branch must
// pass Eq. 8): writes the item's apply mode and factors, appends the decision to a ring of records
// for the host's bookkeeping, and, inside a CUDA graph, sets the conditional that runs the middle
// layers (1 = rejected: run them and refresh; 0 = accepted: inject).
__global__ void rr_decide_kernel(const RRGate* __restrict__ g, int has0, int has1, RRApply* __restrict__ ap,
                                 RRDecision* __restrict__ ring, unsigned long long* __restrict__ ring_n,
                                 int ring_cap, cudaGraphConditionalHandle handle, int set_handle) {
  pdl_wait();
  pdl_launch_dependents();
  if (threadIdx.x != 0) return;
  const bool pass = (!has0 || g[0].pass) && (!has1 || g[1].pass);
  RRApply a;
  a.mode = pass ? kRRInject : kRRRefresh;
  a.cidx = 0;
  a.alpha0 = pass ? static_cast<float>(g[0].alpha) : 0.0f;
  a.alpha1 = pass ? static_cast<float>(g[1].alpha) : 0.0f;
  ap[0] = a;
  const unsigned long long n = *ring_n;
  RRDecision r;
  r.accept = pass ? 1 : 0;
  r.pad = 0;
  for (int b = 0; b < 2; ++b) {
    const bool has = b == 0 ? has0 : has1;
    r.alpha[b] = has ? static_cast<float>(g[b].alpha) : 0.0f;
    r.cos[b] = has ? static_cast<float>(g[b].cos) : 0.0f;
    r.fit[b] = has ? static_cast<float>(g[b].fit) : 0.0f;
  }
  ring[n % static_cast<unsigned long long>(ring_cap)] = r;
  *ring_n = n + 1;
  if (set_handle) cudaGraphSetConditional(handle, pass ? 0u : 1u);
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
  pdl_wait();
  pdl_launch_dependents();
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

// Copy the items that must run the middle layers into the compact middle-layer buffer.
__global__ void __launch_bounds__(256) rr_gather_kernel(float* __restrict__ hm, const float* __restrict__ h,
                                                        const int* __restrict__ map, int64_t item4) {
  pdl_wait();
  pdl_launch_dependents();
  const int c = blockIdx.y;
  const float4* src = reinterpret_cast<const float4*>(h) + static_cast<int64_t>(map[c]) * item4;
  float4* dst = reinterpret_cast<float4*>(hm) + static_cast<int64_t>(c) * item4;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < item4;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    dst[i] = src[i];
}

// ---------------------------------------------------------------- diagnostics (App. E)
// Per-block float64 partial sums of a.b, a.a, b.b and (a-b).(a-b) over the elements i < n whose
// column i mod row_len is below cols (row_len = cols = n for a whole vector).
__global__ void __launch_bounds__(256) diag_partial_kernel(const float* __restrict__ a, const float* __restrict__ b,
                                                           int64_t n, int64_t row_len, int64_t cols,
                                                           double* __restrict__ partial) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ double red[8];
  double s0 = 0.0, s1 = 0.0, s2 = 0.0, s3 = 0.0;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    if (i % row_len >= cols) continue;
    const double x = a[i], y = b[i], e = x - y;
    s0 += x * y;
    s1 += x * x;
    s2 += y * y;
    s3 += e * e;
  }
  s0 = block_sum_d(s0, red);
  s1 = block_sum_d(s1, red);
  s2 = block_sum_d(s2, red);
  s3 = block_sum_d(s3, red);
  if (threadIdx.x == 0) {
    double* p = partial + static_cast<int64_t>(blockIdx.x) * 4;
    p[0] = s0;
    p[1] = s1;
    p[2] = s2;
    p[3] = s3;
  }
}

// ---------------------------------------------------------------- preparation
__global__ void cast_kernel(const float* __restrict__ in, bf16* __restrict__ out, int64_t n) {
  pdl_wait();
  pdl_launch_dependents();
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

template <typename TW, int KB>
cudaError_t gemv_launch(const CondGemv& g, cudaStream_t s) {
  constexpr int LPR = sizeof(TW) == 2 ? 16 : 32;   // the bf16 modulation weight: half-warp rows
  constexpr int CPB = LPR * WVec<TW>::kCPT;
  const int kslice = (g.K + g.splits - 1) / g.splits;
  const size_t smem = sizeof(float) * (static_cast<size_t>(KB) * kslice + 8 * KB * CPB);
  if (smem > 200 * 1024) return cudaErrorInvalidValue;
  // The limit only ever grows (per device): contexts on other host threads launch the same kernel
  // with other sizes, and lowering it between their set and their launch would fail that launch.
  static PerDeviceSmem smem_rec;
  cudaError_t e = ensure_max_smem(smem_rec, cond_gemv_kernel<TW, KB, LPR>, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid((g.Nout + CPB - 1) / CPB, g.splits);
  launch_pdl(cond_gemv_kernel<TW, KB, LPR>, dim3(grid), dim3(256), smem, s, g.in_part, g.in_splits, g.in_bias, g.in_act, g.features,
                                                   g.items, static_cast<const TW*>(g.W), g.K, g.Nout, g.Bw,
                                                   kslice, g.out, g.out_bias);
  return cudaGetLastError();
}

template <typename TW>
cudaError_t gemv_items(const CondGemv& g, cudaStream_t s) {
  if (g.Bw == 1) return gemv_launch<TW, 1>(g, s);
  if (g.Bw == 2) return gemv_launch<TW, 2>(g, s);
  if (g.Bw <= 4) return gemv_launch<TW, 4>(g, s);
  return gemv_launch<TW, 8>(g, s);
}

unsigned row_blocks(int64_t rows) { return static_cast<unsigned>((rows + kRowWarps - 1) / kRowWarps); }

}  // namespace

cudaError_t cond_gemv(const CondGemv& g, cudaStream_t s) {
  if (g.Bw <= 0) return cudaSuccess;
  if (g.Nout % (g.w_bf16 ? 8 : 4) != 0 || g.splits < 1) return cudaErrorInvalidValue;
  return g.w_bf16 ? gemv_items<bf16>(g, s) : gemv_items<float>(g, s);
}

cudaError_t embed_tokens(float* h, float* xhist, int64_t stage_stride, const StepItem* items,
                         const float* x, int T, const float* obs_emb, const float* vid_w,
                         const float* vid_b, const float* act_w, const float* act_b,
                         const float* pos, int Bw, int No, int Nv, int vd, int Na, int ad, int d,
                         cudaStream_t s) {
  if (Bw <= 0) return cudaSuccess;
  const int64_t rows = static_cast<int64_t>(Bw) * (No + Nv + Na);
  const int64_t groups = (rows + kEmbRows - 1) / kEmbRows;
  launch_pdl(embed_kernel, dim3(row_blocks(groups), (d / 4 + 31) / 32), dim3(32 * kRowWarps), 0, s, h, xhist, stage_stride, items, x, T,
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
      launch_pdl(ln_mod_kernel<NV, bf16>, dim3(grid), dim3(256), 0, s, h, hcopy, mods, mod_stride, shift_off,          \
                                                   scale_off, item_map, static_cast<bf16*>(out), M, \
                                                   d, rows_per_item);                              \
    else                                                                                           \
      launch_pdl(ln_mod_kernel<NV, float>, dim3(grid), dim3(256), 0, s, h, hcopy, mods, mod_stride, shift_off,         \
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

int64_t final_head_bytes(int d) {
  const int64_t a = static_cast<int64_t>(16) * (d + 8) * 2, b = static_cast<int64_t>(16) * d * 4;
  const int64_t m = a > b ? a : b;
  return (m + 15) / 16 * 16;
}

cudaError_t final_euler(const float* h, const StepItem* items, const float* mods,
                        int64_t mod_stride, int fin_off, const float* vout_w,
                        const float* vout_b, const float* aout_w, const float* aout_b, float* x,
                        float* xhist, float* vhist, int64_t stage_stride, int T, int Bw, int No,
                        int Nv, int vd, int Na, int ad, int d, bool head_bf16, uint8_t* head_ws,
                        float* head_const, cudaStream_t s) {
  if (Bw <= 0) return cudaSuccess;
  if (d % 128 != 0 || vd > 16 || ad > 16) return cudaErrorInvalidValue;  // heads padded to 16
  const int num_sms = device_sm_count();
  const int64_t hstride = final_head_bytes(d);
  if (head_bf16)
    launch_pdl(final_head_prep_kernel<true>, dim3(2, Bw), dim3(256), 0, s, mods, mod_stride, fin_off, vout_w, vout_b,
               aout_w, aout_b, d, vd, ad, Nv, Na, head_ws, hstride, head_const);
  else
    launch_pdl(final_head_prep_kernel<false>, dim3(2, Bw), dim3(256), 0, s, mods, mod_stride, fin_off, vout_w, vout_b,
               aout_w, aout_b, d, vd, ad, Nv, Na, head_ws, hstride, head_const);
  // An item's video rows are split over blocks so that all blocks are resident at once (the
  // register limit: four 4-warp blocks of the tensor-core kernel or two 8-warp blocks of the SIMT
  // kernel per SM), with at least a 16-row tile per tensor-core block or a row pair per SIMT
  // warp; its action rows take one block (one per 16-row tile).
  const int rows_per_block = head_bf16 ? 16 : 2 * kRowWarps;
  const int want = ((head_bf16 ? 4 : 2) * num_sms + Bw - 1) / Bw;
  const int vmax = (Nv + rows_per_block - 1) / rows_per_block;
  const int vblocks = Nv == 0 ? 0 : (want < vmax ? (want > 1 ? want : 1) : vmax);
  const int ablocks = Na == 0 ? 0 : (head_bf16 ? (Na + 15) / 16 : 1);
  const size_t smem = head_bf16 ? static_cast<size_t>(16) * (d + 8) * sizeof(bf16) : static_cast<size_t>(16) * d * 4;
  dim3 grid(vblocks + ablocks, Bw);
#define WAM_SET_SMEM(KERNEL)                                                                       \
  {                                                                                                \
    static PerDeviceSmem smem_rec; /* per device: contexts may run on several GPUs */             \
    const cudaError_t e = ensure_max_smem(smem_rec, KERNEL, static_cast<int>(smem));               \
    if (e != cudaSuccess) return e;                                                                \
  }
  if (head_bf16) {
    WAM_SET_SMEM(final_euler_tc_kernel)
    launch_pdl(final_euler_tc_kernel, grid, dim3(32 * kFtWarps), smem, s, h, items, x, xhist, vhist, stage_stride, T,
               No, Nv, vd, Na, ad, d, vblocks, ablocks, static_cast<const uint8_t*>(head_ws), hstride,
               static_cast<const float*>(head_const));
    return cudaGetLastError();
  }
#define WAM_FE_CASE(NV)                                                                             \
  case NV:                                                                                          \
    WAM_SET_SMEM(final_euler_kernel<NV>)                                                            \
    launch_pdl(final_euler_kernel<NV>, grid, dim3(256), smem, s, h, items, x, xhist, vhist, stage_stride, T, No, \
               Nv, vd, Na, ad, d, vblocks, ablocks, static_cast<const uint8_t*>(head_ws), hstride,  \
               static_cast<const float*>(head_const));                                              \
    break;
  switch (d / 128) {
    WAM_NV4_CASES(WAM_FE_CASE)
    default: return cudaErrorInvalidValue;
  }
#undef WAM_FE_CASE
#undef WAM_SET_SMEM
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
  launch_pdl(tr_rms_partial_kernel, dim3(grid), dim3(256), 0, s, items, xhist, stage_stride, K, T, V, nch, partial);
  return cudaGetLastError();
}

cudaError_t adapt_apply(const AdaptItem* items, const double* partial, int nch, float* x,
                        float* xb0, const float* xhist, int64_t stage_stride, int K,
                        const float* eps, const float* obs_new, float* obs, int B, int T, int V,
                        int Na, int ad, int64_t obs_elems, int normalize, int video_mode,
                        cudaStream_t s) {
  const int traj_blocks = (T + 1023) / 1024 < 64 ? (T + 1023) / 1024 : 64;  // ~4 elements per thread
  const int obs_blocks = static_cast<int>((obs_elems + 255) / 256 < 64 ? (obs_elems + 255) / 256 : 64);
  dim3 grid(traj_blocks + obs_blocks, B);
  launch_pdl(adapt_apply_kernel, dim3(grid), dim3(256), 0, s, items, partial, nch, x, xb0, xhist, stage_stride, K,
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
  launch_pdl(or_partial_kernel, dim3(grid), dim3(256), 0, s, pred, real, obs_elems, M, idl, nch, partial);
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
  launch_pdl(rr_probe_kernel, dim3(grid), dim3(256), 0, s, h, hq, pa, items, N, d, split_row, nch, partial);
  return cudaGetLastError();
}

cudaError_t rr_gate(const double* partial, int Bw, int nch, int64_t n0, int64_t n1, double amin,
                    double amax, double eps, double gcos, double gfit, RRGate* out,
                    cudaStream_t s) {
  if (Bw <= 0) return cudaSuccess;
  launch_pdl(rr_gate_kernel, dim3((Bw * 2 * 32 + 127) / 128), dim3(128), 0, s, partial, Bw, nch, n0, n1, amin, amax, eps,
                                                           gcos, gfit, out);
  return cudaGetLastError();
}

cudaError_t rr_decide(const RRGate* g, int has0, int has1, RRApply* ap, RRDecision* ring, unsigned long long* ring_n,
                      int ring_cap, cudaGraphConditionalHandle handle, int set_handle, cudaStream_t s) {
  launch_pdl(rr_decide_kernel, dim3(1), dim3(32), 0, s, g, has0, has1, ap, ring, ring_n, ring_cap, handle, set_handle);
  return cudaGetLastError();
}

cudaError_t rr_apply(float* h, const float* hm, const float* hq, float* pa, float* ra,
                     const StepItem* items, const RRApply* ap, int Bw, int N, int d,
                     int split_row, cudaStream_t s) {
  if (Bw <= 0) return cudaSuccess;
  const int64_t n4 = static_cast<int64_t>(N) * d / 4;
  const int bx = static_cast<int>((n4 + 255) / 256 < 1024 ? (n4 + 255) / 256 : 1024);
  dim3 grid(bx, Bw);
  launch_pdl(rr_apply_kernel, dim3(grid), dim3(256), 0, s, h, hm, hq, pa, ra, items, ap, N, d, split_row);
  return cudaGetLastError();
}

cudaError_t rr_gather(float* hm, const float* h, const int* map, int nmid, int64_t item_elems, cudaStream_t s) {
  if (nmid <= 0) return cudaSuccess;
  const int64_t item4 = item_elems / 4;
  const int bx = static_cast<int>((item4 + 255) / 256 < 512 ? (item4 + 255) / 256 : 512);
  launch_pdl(rr_gather_kernel, dim3(bx, nmid), dim3(256), 0, s, hm, h, map, item4);
  return cudaGetLastError();
}

cudaError_t diag_partial(const float* a, const float* b, int64_t n, int64_t row_len, int64_t cols, int nblocks,
                         double* partial, cudaStream_t s) {
  if (n <= 0 || nblocks <= 0 || row_len <= 0) return cudaErrorInvalidValue;
  launch_pdl(diag_partial_kernel, dim3(nblocks), dim3(256), 0, s, a, b, n, row_len, cols, partial);
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
