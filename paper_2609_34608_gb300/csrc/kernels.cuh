// Internal interfaces of the non-GEMM, non-attention kernels (elementwise.cu).
#pragma once

#include "common.cuh"

namespace wam {

// One work item (episode) of a denoising step.
struct StepItem {
  int32_t ep;      // episode index in the state
  int32_t stage;   // stage k the step starts from
  double sigma;    // sigma_k
  double dsigma;   // sigma_{k+1} - sigma_k
};

// Per-episode adaptation op (wam_adapt_state).
enum AdaptOp : int32_t { kAdaptNone = 0, kAdaptTR = 1, kAdaptCold = 2, kAdaptRestart = 3 };
struct AdaptItem {
  int32_t op;
  int32_t shift;
  int32_t r;        // retained stage
  int32_t bind_obs; // copy the new condition into the state
  double sigma_r;
  double sigma_b0;
};

// RR gate result of one (item, branch).
struct RRGate {
  double alpha, cos, fit;
  int32_t pass;
  int32_t pad;
};

// One device-side RR decision (single work item), as the host records it in the step log.
struct RRDecision {
  int32_t accept, pad;
  float alpha[2], cos[2], fit[2];
};

// RR apply mode of one item after the gate.
enum RRMode : int32_t { kRRNone = 0, kRRInject = 1, kRRRefresh = 2, kRRCopyBack = 3 };
struct RRApply {
  int32_t mode;
  int32_t cidx;     // row block of the item in the middle-layer buffer
  float alpha0, alpha1;
};

constexpr int kTrChunk = 2048;     // elements per TR reduction block
constexpr int kProbeChunk = 8192;  // elements per RR probe block
constexpr int kOrChunk = 8192;     // elements per OR score block

// One conditioning GEMV: out[split][b][n] = sum over the split's K slice of x[b][k] W[k][n]
// (+ out_bias[n] when splits == 1), x[b][k] = timestep features of items[b].sigma when
// `features`, else act(in_bias[k] + sum over in_splits partial rows of in_part).
struct CondGemv {
  const float* in_part;
  int in_splits;
  const float* in_bias;
  int in_act;     // 1: SiLU
  int features;   // 1: sinusoidal timestep features (K of them)
  const StepItem* items;
  const void* W;  // [K, Nout]
  bool w_bf16;
  int K, Nout, Bw, splits;
  float* out;
  const float* out_bias;
};
cudaError_t cond_gemv(const CondGemv& g, cudaStream_t s);

cudaError_t embed_tokens(float* h, float* xhist, int64_t stage_stride, const StepItem* items,
                         const float* x, int T, const float* obs_emb, const float* vid_w,
                         const float* vid_b, const float* act_w, const float* act_b,
                         const float* pos, int Bw, int No, int Nv, int vd, int Na, int ad, int d,
                         cudaStream_t s);

cudaError_t ln_modulate(const float* h, float* hcopy, const float* mods, int64_t mod_stride,
                        int shift_off, int scale_off, const int* item_map, void* out,
                        bool out_bf16, int M, int d, int rows_per_item, cudaStream_t s);

cudaError_t final_euler(const float* h, const StepItem* items, const float* mods,
                        int64_t mod_stride, int fin_off, const float* vout_w,
                        const float* vout_b, const float* aout_w, const float* aout_b, float* x,
                        float* xhist, float* vhist, int64_t stage_stride, int T, int Bw, int No,
                        int Nv, int vd, int Na, int ad, int d, bool head_bf16, uint8_t* head_ws,
                        float* head_const, cudaStream_t s);
// Bytes per (work item, head) of the prepared-head scratch of final_euler (head_ws holds
// 2 * items of them; head_const 64 floats per item).
int64_t final_head_bytes(int d);

int tr_num_chunks(int T, int V);
cudaError_t tr_rms_partial(const AdaptItem* items, const float* xhist, int64_t stage_stride,
                           int K, int B, int T, int V, int nch, double* partial, cudaStream_t s);
cudaError_t adapt_apply(const AdaptItem* items, const double* partial, int nch, float* x,
                        float* xb0, const float* xhist, int64_t stage_stride, int K,
                        const float* eps, const float* obs_new, float* obs, int B, int T, int V,
                        int Na, int ad, int64_t obs_elems, int normalize, int video_mode,
                        cudaStream_t s);

int or_num_chunks(int64_t comp_elems);
cudaError_t or_score_partial(const float* pred, const float* real, int B, int64_t obs_elems,
                             int M, const float* inv_delta4, int nch, double* partial,
                             cudaStream_t s);

int rr_num_chunks(int64_t branch_elems_max);
cudaError_t rr_probe_partial(const float* h, const float* hq, const float* pa,
                             const StepItem* items, int Bw, int N, int d, int split_row, int nch,
                             double* partial, cudaStream_t s);
cudaError_t rr_gate(const double* partial, int Bw, int nch, int64_t n0, int64_t n1, double amin,
                    double amax, double eps, double gcos, double gfit, RRGate* out,
                    cudaStream_t s);
// hm[c] = h[map[c]] for the nmid items that run the middle layers (rows of N*d floats)
cudaError_t rr_gather(float* hm, const float* h, const int* map, int nmid, int64_t item_elems, cudaStream_t s);
// App. E diagnostics: nblocks x {a.b, a.a, b.b, (a-b).(a-b)} float64 partials over the elements
// whose column (index mod row_len) is below cols.
cudaError_t diag_partial(const float* a, const float* b, int64_t n, int64_t row_len, int64_t cols, int nblocks,
                         double* partial, cudaStream_t s);
// The RR decision of work item 0 taken on the device (see rr_decide_kernel).
cudaError_t rr_decide(const RRGate* g, int has0, int has1, RRApply* ap, RRDecision* ring, unsigned long long* ring_n,
                      int ring_cap, cudaGraphConditionalHandle handle, int set_handle, cudaStream_t s);
cudaError_t rr_apply(float* h, const float* hm, const float* hq, float* pa, float* ra,
                     const StepItem* items, const RRApply* ap, int Bw, int N, int d,
                     int split_row, cudaStream_t s);

cudaError_t cast_f32_bf16(const float* in, bf16* out, int64_t n, cudaStream_t s);
// out[n, k] = in[k, n] for a [K, N] float32 matrix, as bf16 or float32
cudaError_t transpose_cast(const float* in, void* out, bool out_bf16, int K, int N,
                           cudaStream_t s);
// copy a [rows, cols] float32 block (source pitch spitch floats) into dst (pitch dpitch elems)
cudaError_t copy_cast_2d(const float* in, int64_t spitch, void* out, bool out_bf16,
                         int64_t dpitch, int rows, int cols, cudaStream_t s);

}  // namespace wam
