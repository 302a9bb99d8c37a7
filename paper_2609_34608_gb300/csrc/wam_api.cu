// C ABI of the WAMachine hot path: context / state management and the host-side orchestration
// of one denoising step (conditioning, embedding, DiT layers with the Residual Rescaling
// branch, final layer + Euler), of Trajectory Remapping and of Observation Rebinding.
// Every step of the path runs in this library's kernels; the host only sequences launches,
// keeps the per-episode bookkeeping of §3.4 and takes the two data-dependent decisions
// (RR gate, OR acceptance) after reading their device-computed statistics.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <deque>
#include <map>
#include <new>
#include <string>
#include <thread>
#include <tuple>
#include <vector>

#include "kernels.cuh"
#include "wam.h"
#include "wam_ops.h"

using namespace wam;

namespace {

constexpr int kRingSlots = 64;
constexpr size_t kSlotBytes = 16384;
constexpr int kMaxBatch = 256;
constexpr int kT1Splits = 8;  // K splits of the two conditioning-MLP GEMVs
constexpr int kT2Splits = 8;
// Largest row count (episodes x tokens) of a layer range run by the fused row-chain kernel.  Above
// it the per-projection GEMMs pick wider tiles and fill the GPU on their own.
constexpr int kChainMaxRows = 16384;
constexpr int kDecCap = 1024;   // device RR decisions in flight between the GPU and the host

struct LayerW {
  void* qkv_wt = nullptr;
  void* out_wt = nullptr;
  void* up_wt = nullptr;
  void* down_wt = nullptr;
  float* qkv_b = nullptr;
  float* out_b = nullptr;
  float* up_b = nullptr;
  float* down_b = nullptr;
  GemmOperand tm_qkv, tm_out, tm_up, tm_down;   // also with 64-row boxes
};

struct ProfSpan {
  int kclass;
  cudaEvent_t a, b;
  double flops, bytes;
};

enum Path : int32_t { kPathCold = 0, kPathPrefix = 1, kPathRefresh = 2 };

struct EpisodeMeta {
  int32_t stage = -1;
  int32_t hist_from = 0;
  int32_t b0 = 0;
  int32_t kappa = 0;
  int32_t finished = 0;
  int32_t since_bind = 0;
  int32_t path = kPathCold;
  int32_t rr_valid = 0;
  int32_t path_steps = 0;
};

}  // namespace

struct wam_ctx {
  wam_config cfg;
  int L, d, H, R, No, Nv, vd, Na, ad, N, T, V, K, dff, Bmax;
  // first row of the RR action branch: No + Nv for a joint model; N for a video-only model
  // (one branch, all rows) and 0 for an action-only model (one branch, all rows)
  int split;
  int64_t mod_n;
  bool bf16;
  cudaStream_t stream = nullptr;
  int device = 0, num_sms = 0;
  std::string err;
  std::vector<double> sigma;
  std::vector<void*> allocs;
  // weights
  void* obs_wt = nullptr;
  float* obs_b = nullptr;
  float *vid_w, *vid_b, *act_w, *act_b, *pos;
  float *t_w1, *t_b1, *t_w2, *t_b2;
  void* mod_w = nullptr;
  float* mod_b = nullptr;
  std::vector<LayerW> layers;
  float *vout_w, *vout_b, *aout_w, *aout_b;
  GemmOperand tm_obs_w;
  // activations (batch_max episodes)
  float *h = nullptr, *hq = nullptr, *hm = nullptr;
  void *xln = nullptr, *qkv = nullptr, *att = nullptr, *u = nullptr, *obs_lp = nullptr;
  GemmOperand tm_xln, tm_att, tm_u, tm_obs_lp;
  // tensor-core attention (head dim 64): V^T per (episode, head) and the TMA maps it reads
  bool tc_attn = false;
  void* vt = nullptr;
  int vt_ld = 0;
  AttnMaps attn_maps;
  float *t1 = nullptr, *cvec = nullptr, *mods = nullptr;
  StepItem* d_items = nullptr;
  int* d_map = nullptr;
  // fused row-chain kernel (dit_chain.cu), off unless enabled: for bf16 models with the
  // tensor-core attention when a layer range covers at most kChainMaxRows rows; its completion
  // counters
  bool chain_ok = false;
  bool layer_fusion = false;
  bool chain_phases = true;   // grid-wide phase boundaries instead of per-row-block dependencies
  int* d_chain_ctr = nullptr;
  // profiling: per-task records of the fused launches (allocated on first use)
  wam_chain_task* d_trace = nullptr;
  int trace_cap = 0, trace_used = 0, trace_launches = 0;
  // Device-side RR branching for a single work item (§3.3 at one episode): the whole step around
  // the gate is one CUDA graph whose conditional node runs the middle layers only when the gate
  // rejects, so the host never waits for the decision.  Decisions come back through a ring of
  // records copied to pinned memory after each call and folded into the step log and the reuse
  // statistics when the host next looks (or when the ring would overflow).
  bool dev_branch = true;
  bool dev_branch_ok = true;
  cudaStream_t aux_stream = nullptr;    // captures the conditional body
  int* d_map0 = nullptr;                // {0}: item map of the single gathered item
  RRDecision* d_dec = nullptr;          // [kDecCap] ring of decisions
  unsigned long long* d_dec_n = nullptr;
  RRDecision* h_dec = nullptr;          // pinned mirror of the ring
  unsigned long long dec_queued = 0, dec_copied = 0, dec_resolved = 0;
  struct PendingDec {
    wam_state* st;
    int log_idx;   // -1 once the state's log moved on
  };
  std::deque<PendingDec> dec_pending;
  std::deque<std::pair<cudaEvent_t, unsigned long long>> dec_batches;   // (copy done, records up to)
  std::map<std::tuple<const void*, const void*>, cudaGraphExec_t> rr_graphs;
  std::map<std::tuple<const void*, const void*>, int> rr_graph_uses;
  std::map<cudaGraphExec_t, long long> graph_kernels;   // kernels per graph (launch counting)
  // CUDA graphs of layer ranges: key (first layer, end layer, episodes, stream buffer, item map,
  // layer that also saves h_q or -1) -> executable graph, captured on a range's second use
  bool graph_replay = true;
  bool graphs_ok = true;
  std::map<std::tuple<int, int, int, const void*, const void*, int>, cudaGraphExec_t> layer_graphs;
  std::map<std::tuple<int, int, int, const void*, const void*, int>, int> layer_graph_uses;
  // conditioning once per distinct sigma of a call: those sigmas (capacity Ucap = max(batch,
  // steps)), their modulation rows, and the work item -> row index a step gathers with
  int Ucap = 0;
  StepItem* d_uitems = nullptr;
  int* d_uidx = nullptr;
  float* mods_u = nullptr;
  RRApply* d_rrapply = nullptr;
  RRGate* d_gate = nullptr;
  AdaptItem* d_adapt = nullptr;
  double* d_part = nullptr;
  size_t part_doubles = 0;
  float* d_eps = nullptr;
  float* d_obs_new = nullptr;
  // final layer: each work item's modulated output heads, prepared once per step
  uint8_t* d_fhead = nullptr;
  float* d_fconst = nullptr;
  int* d_err = nullptr;
  // pinned host staging
  uint8_t* ring = nullptr;
  cudaEvent_t ring_ev[kRingSlots];
  bool ring_used[kRingSlots];
  int ring_next = 0;
  uint8_t* readback = nullptr;
  size_t readback_bytes = 0;
  wam_stats stats;
  bool prof_on = false;
  std::vector<ProfSpan> spans;
  std::vector<cudaEvent_t> evpool;
  size_t evnext = 0;
};

struct wam_state {
  wam_ctx* ctx = nullptr;
  int B = 0;
  float* x = nullptr;      // [B,T]
  float* xhist = nullptr;  // [K+1,B,T]
  float* vhist = nullptr;  // [K,B,T]
  float* xb0 = nullptr;    // [B,T]
  float* obs = nullptr;    // [B,No,d]
  float* obs_emb = nullptr;
  float* pa = nullptr;     // [B,N,d]
  float* ra = nullptr;
  std::vector<void*> allocs;
  std::vector<EpisodeMeta> meta;
  std::vector<wam_step_record> log;
};

namespace {

int fail(wam_ctx* c, int code, const std::string& msg) {
  if (c) c->err = msg;
  return code;
}

int fail_cuda(wam_ctx* c, const char* what, cudaError_t e) {
  return fail(c, e == cudaErrorMemoryAllocation ? WAM_ERR_OOM : WAM_ERR_CUDA,
              std::string(what) + ": " + cudaGetErrorString(e));
}

#define CK(x)                                           \
  do {                                                  \
    cudaError_t e_ = (x);                               \
    if (e_ != cudaSuccess) return fail_cuda(c, #x, e_); \
  } while (0)

#define TRY(x)              \
  do {                      \
    int r_ = (x);           \
    if (r_ != WAM_OK) return r_; \
  } while (0)

template <typename T>
int dalloc(wam_ctx* c, std::vector<void*>& reg, T** p, size_t count) {
  void* q = nullptr;
  cudaError_t e = cudaMalloc(&q, count * sizeof(T) > 0 ? count * sizeof(T) : 16);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(c, WAM_ERR_OOM, "device allocation of " + std::to_string(count * sizeof(T)) + " bytes failed");
  }
  reg.push_back(q);
  *p = static_cast<T*>(q);
  return WAM_OK;
}

bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

cudaEvent_t next_event(wam_ctx* c) {
  if (c->evnext == c->evpool.size()) {
    cudaEvent_t e;
    cudaEventCreate(&e);
    c->evpool.push_back(e);
  }
  return c->evpool[c->evnext++];
}

// Launch bookkeeping: counts every kernel and, while profiling, brackets it with events.
struct Span {
  wam_ctx* c;
  int kc;
  double fl, by;
  cudaEvent_t a = nullptr;
  Span(wam_ctx* c_, int kc_, double fl_ = 0.0, double by_ = 0.0) : c(c_), kc(kc_), fl(fl_), by(by_) {
    c->stats.n_kernel_launches++;
    if (c->prof_on) {
      a = next_event(c);
      cudaEventRecord(a, c->stream);
    }
  }
  ~Span() {
    if (a != nullptr) {
      cudaEvent_t b = next_event(c);
      cudaEventRecord(b, c->stream);
      c->spans.push_back({kc, a, b, fl, by});
    }
  }
};

// Host -> device upload of a small control array through a pinned ring slot.
int upload(wam_ctx* c, void* dst, const void* src, size_t n) {
  if (n == 0) return WAM_OK;
  if (n > kSlotBytes) return fail(c, WAM_ERR_INVALID_ARG, "control upload too large");
  const int s = c->ring_next;
  c->ring_next = (c->ring_next + 1) % kRingSlots;
  if (c->ring_used[s]) CK(cudaEventSynchronize(c->ring_ev[s]));
  std::memcpy(c->ring + s * kSlotBytes, src, n);
  CK(cudaMemcpyAsync(dst, c->ring + s * kSlotBytes, n, cudaMemcpyHostToDevice, c->stream));
  CK(cudaEventRecord(c->ring_ev[s], c->stream));
  c->ring_used[s] = true;
  return WAM_OK;
}

// Device -> host read of small statistics, followed by a stream synchronisation and a check of
// the device error word.
int readback(wam_ctx* c, void* dst, const void* src, size_t n) {
  if (n + sizeof(int) > c->readback_bytes) return fail(c, WAM_ERR_INVALID_ARG, "readback too large");
  CK(cudaMemcpyAsync(c->readback, src, n, cudaMemcpyDeviceToHost, c->stream));
  CK(cudaMemcpyAsync(c->readback + n, c->d_err, sizeof(int), cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  int derr = 0;
  std::memcpy(&derr, c->readback + n, sizeof(int));
  if (derr != 0) {
    cudaMemsetAsync(c->d_err, 0, sizeof(int), c->stream);
    return fail(c, WAM_ERR_TIMEOUT, "a bounded device-side wait gave up");
  }
  std::memcpy(dst, c->readback, n);
  return WAM_OK;
}

int sync_check(wam_ctx* c) {
  int dummy = 0;
  return readback(c, &dummy, c->d_err, sizeof(int));
}

// ---------------------------------------------------------------------------------- GEMM
EpiArgs epi_args(const float* bias, void* C, const float* gate, int64_t gstride, int rpi, const int* map) {
  EpiArgs e;
  e.bias = bias;
  e.C = C;
  e.gate = gate;
  e.gate_stride = gstride;
  e.rows_per_item = rpi;
  e.item_map = map;
  e.vt = nullptr;
  e.vt_ld = 0;
  return e;
}

int gemm(wam_ctx* c, const GemmOperand* ta, const void* A, const GemmOperand* tb, const void* Wt,
         int M, int N, int K, int epi, const EpiArgs& e) {
  const double out_b = (epi == kEpiResidF32) ? 8.0 : (epi == kEpiF32 ? 4.0 : (c->bf16 ? 2.0 : 4.0));
  const double in_b = c->bf16 ? 2.0 : 4.0;
  Span sp(c, WAM_KCLASS_GEMM, 2.0 * M * N * K, in_b * (double(M) * K + double(N) * K) + out_b * double(M) * N);
  if (c->bf16) {
    CK(tc_gemm(*ta, *tb, M, N, K, epi, e, c->num_sms, c->d_err, c->stream, nullptr,
               tc_gemm_plan(M, N, K, epi == kEpiResidF32, tb->r64, c->num_sms)));
  } else {
    CK(simt_gemm(static_cast<const float*>(A), static_cast<const float*>(Wt), M, N, K, epi, e, c->stream));
  }
  return WAM_OK;
}


int ln_mod(wam_ctx* c, const float* hb, float* hcopy, int shift_off, int scale_off, const int* map, int M) {
  const double by = double(M) * c->d * (4.0 + (c->bf16 ? 2.0 : 4.0) + (hcopy ? 4.0 : 0.0));
  Span sp(c, WAM_KCLASS_NORM, 0.0, by);
  CK(ln_modulate(hb, hcopy, c->mods, c->mod_n, shift_off, scale_off, map, c->xln, c->bf16, M, c->d, c->N, c->stream));
  return WAM_OK;
}

// One adaLN DiT block on `Bw` items stored contiguously in hb.
int run_layer(wam_ctx* c, int l, float* hb, int Bw, const int* map, float* hcopy) {
  const int M = Bw * c->N, d = c->d;
  const int base = l * 6 * d;
  LayerW& w = c->layers[l];
  TRY(ln_mod(c, hb, hcopy, base, base + d, map, M));
  {
    EpiArgs eq = epi_args(w.qkv_b, c->qkv, nullptr, 0, c->N, nullptr);
    if (c->tc_attn) {
      eq.vt = static_cast<bf16*>(c->vt);
      eq.vt_ld = c->vt_ld;
    }
    TRY(gemm(c, &c->tm_xln, c->xln, &w.tm_qkv, w.qkv_wt, M, 3 * d, d, c->tc_attn ? kEpiQkvVt : kEpiBf16, eq));
  }
  {
    const double el = c->bf16 ? 2.0 : 4.0;
    Span sp(c, WAM_KCLASS_ATTN, 4.0 * Bw * double(c->N) * c->N * d, el * 4.0 * M * d);
    if (c->tc_attn)
      CK(attention_tc(c->attn_maps, static_cast<bf16*>(c->att), Bw, c->N, d, c->H, c->d_err, c->stream));
    else if (c->bf16)
      CK(attention_bf16(static_cast<const bf16*>(c->qkv), static_cast<bf16*>(c->att), Bw, c->N, d, c->H, c->stream));
    else
      CK(attention_f32(static_cast<const float*>(c->qkv), static_cast<float*>(c->att), Bw, c->N, d, c->H, c->stream));
  }
  TRY(gemm(c, &c->tm_att, c->att, &w.tm_out, w.out_wt, M, d, d, kEpiResidF32,
           epi_args(w.out_b, hb, c->mods + base + 2 * d, c->mod_n, c->N, map)));
  TRY(ln_mod(c, hb, nullptr, base + 3 * d, base + 4 * d, map, M));
  TRY(gemm(c, &c->tm_xln, c->xln, &w.tm_up, w.up_wt, M, c->dff, d, kEpiGeluBf16,
           epi_args(w.up_b, c->u, nullptr, 0, c->N, nullptr)));
  TRY(gemm(c, &c->tm_u, c->u, &w.tm_down, w.down_wt, M, d, c->dff, kEpiResidF32,
           epi_args(w.down_b, hb, c->mods + base + 5 * d, c->mod_n, c->N, map)));
  return WAM_OK;
}

// The row-local work between two attentions as one fused launch: the tail of layer `lt`
// (out-projection .. MLP down) and / or the head of layer `lh` (LN + QKV), -1 for none.
int run_chain(wam_ctx* c, int lt, int lh, float* hb, int Bw, const int* map, float* hcopy) {
  const int M = Bw * c->N, d = c->d;
  ChainParams p;
  std::memset(&p, 0, sizeof(p));
  p.M = M;
  p.Mt = (M + 127) / 128;
  p.d = d;
  p.dff = c->dff;
  p.has_tail = lt >= 0;
  p.has_head = lh >= 0;
  p.mods = c->mods;
  p.mod_stride = c->mod_n;
  p.item_map = map;
  p.rows_per_item = c->N;
  p.h = hb;
  p.hq = hcopy;
  p.xln = static_cast<bf16*>(c->xln);
  p.ctr = c->d_chain_ctr;
  p.dev_err = c->d_err;
  p.phase_barrier = c->chain_phases ? 1 : 0;
  ChainMaps maps{&c->tm_att.r128_k2, &c->tm_xln.r128_k2, &c->tm_u.r128_k2, &c->tm_xln.r128_k2,
                 &c->tm_xln.r128_k2, &c->tm_xln.r128_k2, &c->tm_xln.r128_k2};
  double flops = 0.0, bytes = 0.0;
  if (lt >= 0) {
    LayerW& w = c->layers[lt];
    const int base = lt * 6 * d;
    p.e_out = epi_args(w.out_b, hb, c->mods + base + 2 * d, c->mod_n, c->N, map);
    p.e_up = epi_args(w.up_b, c->u, nullptr, 0, c->N, nullptr);
    p.e_down = epi_args(w.down_b, hb, c->mods + base + 5 * d, c->mod_n, c->N, map);
    p.shift2_off = base + 3 * d;
    p.scale2_off = base + 4 * d;
    maps.out_w = &w.tm_out.r64_k2;     // 64-column tiles of the d-wide projections
    maps.up_w = &w.tm_up.r128_k2;
    maps.down_w = &w.tm_down.r64_k2;
    flops += 2.0 * M * (double(d) * d + 2.0 * double(d) * c->dff);
    bytes += 2.0 * (double(d) * d + 2.0 * double(d) * c->dff) + double(M) * (2.0 * d + 16.0 * d + 4.0 * c->dff);
  }
  if (lh >= 0) {
    LayerW& w = c->layers[lh];
    const int base = lh * 6 * d;
    p.e_qkv = epi_args(w.qkv_b, c->qkv, nullptr, 0, c->N, nullptr);
    p.e_qkv.vt = static_cast<bf16*>(c->vt);
    p.e_qkv.vt_ld = c->vt_ld;
    p.shift1_off = base;
    p.scale1_off = base + d;
    maps.qkv_w = &w.tm_qkv.r128_k2;
    flops += 2.0 * M * 3.0 * double(d) * d;
    bytes += 6.0 * double(d) * d + double(M) * (4.0 * d + 4.0 * d + 6.0 * d + (hcopy ? 4.0 * d : 0.0));
  }
  if (c->prof_on && c->d_trace != nullptr) {
    const int n = dit_chain_tasks(p);
    p.trace = c->d_trace + c->trace_used;
    p.trace_cap = std::max(0, std::min(n, c->trace_cap - c->trace_used));
    p.trace_launch = c->trace_launches++;
    c->trace_used += p.trace_cap;
  }
  Span sp(c, WAM_KCLASS_GEMM, flops, bytes);
  CK(dit_chain(maps, p, c->num_sms, c->stream));
  return WAM_OK;
}

int run_attention(wam_ctx* c, int Bw) {
  const int M = Bw * c->N, d = c->d;
  const double el = c->bf16 ? 2.0 : 4.0;
  Span sp(c, WAM_KCLASS_ATTN, 4.0 * Bw * double(c->N) * c->N * d, el * 4.0 * M * d);
  if (c->tc_attn)
    CK(attention_tc(c->attn_maps, static_cast<bf16*>(c->att), Bw, c->N, d, c->H, c->d_err, c->stream));
  else if (c->bf16)
    CK(attention_bf16(static_cast<const bf16*>(c->qkv), static_cast<bf16*>(c->att), Bw, c->N, d, c->H, c->stream));
  else
    CK(attention_f32(static_cast<const float*>(c->qkv), static_cast<float*>(c->att), Bw, c->N, d, c->H, c->stream));
  return WAM_OK;
}

// Layers [l0, l1) of the episodes in hb (item map `map`, or none), saving h_q at layer `hq_layer`
// (or -1).  The ~7 launches per layer have fixed arguments for a given key, so a range is
// captured into a CUDA graph on its second use (the first runs eagerly, which also sets every
// kernel attribute outside capture) and replayed afterwards: one graph launch instead of the
// per-kernel launch gaps.  Profiling (per-kernel events) and a failed capture run eagerly.
int run_layers(wam_ctx* c, int l0, int l1, float* hb, int Bw, const int* map, int hq_layer) {
  if (l0 >= l1) return WAM_OK;
  const bool fused = c->chain_ok && c->layer_fusion && Bw * c->N <= kChainMaxRows;
  auto eager = [&]() -> int {
    if (!fused) {
      for (int l = l0; l < l1; ++l) TRY(run_layer(c, l, hb, Bw, map, l == hq_layer ? c->hq : nullptr));
      return WAM_OK;
    }
    // head of l0, then per layer: attention, and the tail of l fused with the head of l + 1
    TRY(run_chain(c, -1, l0, hb, Bw, map, l0 == hq_layer ? c->hq : nullptr));
    for (int l = l0; l < l1; ++l) {
      TRY(run_attention(c, Bw));
      const int nx = l + 1 < l1 ? l + 1 : -1;
      TRY(run_chain(c, l, nx, hb, Bw, map, nx >= 0 && nx == hq_layer ? c->hq : nullptr));
    }
    return WAM_OK;
  };
  if (!c->graph_replay || !c->graphs_ok || c->prof_on) return eager();
  // the fused and unfused launch sequences of one range are different graphs
  const auto key = std::make_tuple(l0, l1, fused ? -Bw : Bw, static_cast<const void*>(hb), static_cast<const void*>(map),
                                   hq_layer);
  const auto hit = c->layer_graphs.find(key);
  if (hit != c->layer_graphs.end()) {
    CK(cudaGraphLaunch(hit->second, c->stream));
    c->stats.n_kernel_launches += c->graph_kernels[hit->second];
    return WAM_OK;
  }
  if (++c->layer_graph_uses[key] < 2) return eager();
  cudaGraph_t g = nullptr;
  if (cudaStreamBeginCapture(c->stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
    cudaGetLastError();
    c->graphs_ok = false;
    return eager();
  }
  const long long k0 = c->stats.n_kernel_launches;
  const int rc = eager();
  const cudaError_t ec = cudaStreamEndCapture(c->stream, &g);
  cudaGraphExec_t ex = nullptr;
  if (rc == WAM_OK && ec == cudaSuccess && g != nullptr && cudaGraphInstantiate(&ex, g, 0) == cudaSuccess) {
    cudaGraphDestroy(g);
    c->layer_graphs[key] = ex;
    c->graph_kernels[ex] = c->stats.n_kernel_launches - k0;   // counted once while capturing
    CK(cudaGraphLaunch(ex, c->stream));
    return WAM_OK;
  }
  // Capture not possible here: nothing of it ran; run the range eagerly from now on.
  if (g != nullptr) cudaGraphDestroy(g);
  cudaGetLastError();
  c->err.clear();
  c->graphs_ok = false;
  return eager();
}

// Folds device RR decisions whose copies have landed (all of them when `block`) into the step log
// and the reuse statistics (App. D.2): until then a device-decided step counts as evaluated in
// full.
int resolve_decisions(wam_ctx* c, bool block) {
  const int e = c->cfg.rr_e, sq = c->cfg.rr_s;
  while (!c->dec_batches.empty()) {
    auto& b = c->dec_batches.front();
    if (block) {
      CK(cudaEventSynchronize(b.first));
    } else {
      const cudaError_t q = cudaEventQuery(b.first);
      if (q == cudaErrorNotReady) {
        cudaGetLastError();
        break;
      }
      if (q != cudaSuccess) return fail_cuda(c, "RR decision copy", q);
    }
    for (; c->dec_resolved < b.second; ++c->dec_resolved) {
      const RRDecision& r = c->h_dec[c->dec_resolved % kDecCap];
      const wam_ctx::PendingDec pd = c->dec_pending.front();
      c->dec_pending.pop_front();
      if (r.accept) {
        c->stats.n_reuse++;
        c->stats.b_skip += e - sq;
        c->stats.n_layer_evals -= e - sq;
      }
      if (pd.st != nullptr && pd.log_idx >= 0 && pd.log_idx < static_cast<int>(pd.st->log.size())) {
        wam_step_record& rec = pd.st->log[pd.log_idx];
        rec.rr_accept = r.accept;
        for (int br = 0; br < 2; ++br) {
          rec.alpha[br] = r.alpha[br];
          rec.cos[br] = r.cos[br];
          rec.fit[br] = r.fit[br];
        }
      }
    }
    cudaEventDestroy(b.first);
    c->dec_batches.pop_front();
  }
  return WAM_OK;
}

// Copies the decision records of this call's device-branched steps to the host ring.
int queue_decision_copy(wam_ctx* c) {
  if (c->dec_queued == c->dec_copied) return WAM_OK;
  const unsigned long long a = c->dec_copied, b = c->dec_queued;
  const size_t sz = sizeof(RRDecision);
  const size_t i0 = a % kDecCap, i1 = b % kDecCap;
  if (i0 < i1 || b - a == 0) {
    CK(cudaMemcpyAsync(c->h_dec + i0, c->d_dec + i0, sz * (i1 - i0), cudaMemcpyDeviceToHost, c->stream));
  } else {   // wraps around the ring
    CK(cudaMemcpyAsync(c->h_dec + i0, c->d_dec + i0, sz * (kDecCap - i0), cudaMemcpyDeviceToHost, c->stream));
    if (i1 > 0) CK(cudaMemcpyAsync(c->h_dec, c->d_dec, sz * i1, cudaMemcpyDeviceToHost, c->stream));
  }
  cudaEvent_t ev;
  CK(cudaEventCreateWithFlags(&ev, cudaEventDisableTiming));
  CK(cudaEventRecord(ev, c->stream));
  c->dec_batches.emplace_back(ev, b);
  c->dec_copied = b;
  return WAM_OK;
}

// One RR step of a single work item with the decision on the device: layers [0, s) (saving
// h_q), the probe and gate, the decision, the middle layers under a graph conditional (rejected
// only), the injection or refresh, layers [e, L).  Captured on the second use per state and
// replayed.  Returns WAM_OK with *done = false when the caller should run the host-branching
// path instead (first use, or capture not possible).
int rr_step_device(wam_ctx* c, wam_state* st, int nch, bool* done) {
  *done = false;
  const int N = c->N, d = c->d, L = c->L;
  const int q = c->cfg.rr_q, s = c->cfg.rr_s, e = c->cfg.rr_e, split = c->split;
  const auto key = std::make_tuple(static_cast<const void*>(st->pa), static_cast<const void*>(st->ra));
  auto hit = c->rr_graphs.find(key);
  if (hit == c->rr_graphs.end()) {
    if (++c->rr_graph_uses[key] < 2) return WAM_OK;
    if (c->aux_stream == nullptr) {
      if (cudaStreamCreateWithFlags(&c->aux_stream, cudaStreamNonBlocking) != cudaSuccess) {
        cudaGetLastError();
        c->dev_branch_ok = false;
        return WAM_OK;
      }
    }
    const long long k0 = c->stats.n_kernel_launches;
    cudaGraph_t g = nullptr;
    if (cudaStreamBeginCapture(c->stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
      cudaGetLastError();
      c->dev_branch_ok = false;
      return WAM_OK;
    }
    int rc = WAM_OK;
    bool capture_ok = true;
    for (int l = 0; l < s && rc == WAM_OK; ++l) rc = run_layer(c, l, c->h, 1, nullptr, l == q ? c->hq : nullptr);
    if (rc == WAM_OK) {
      Span sp(c, WAM_KCLASS_RR_PROBE, 0.0, 12.0 * double(N) * d);
      capture_ok = rr_probe_partial(c->h, c->hq, st->pa, c->d_items, 1, N, d, split, nch, c->d_part, c->stream) ==
                   cudaSuccess;
    }
    if (rc == WAM_OK && capture_ok) {
      Span sp(c, WAM_KCLASS_RR_PROBE);
      capture_ok = rr_gate(c->d_part, 1, nch, int64_t(split) * d, int64_t(N - split) * d, c->cfg.rr_alpha_min,
                           c->cfg.rr_alpha_max, c->cfg.rr_eps, c->cfg.rr_gamma_cos, c->cfg.rr_gamma_fit, c->d_gate,
                           c->stream) == cudaSuccess;
    }
    cudaGraph_t cg = nullptr;
    const cudaGraphNode_t* deps = nullptr;
    size_t nd = 0;
    cudaStreamCaptureStatus cs;
    cudaGraphConditionalHandle hdl = 0;
    if (rc == WAM_OK && capture_ok)
      capture_ok = cudaStreamGetCaptureInfo(c->stream, &cs, nullptr, &cg, &deps, nullptr, &nd) == cudaSuccess &&
                   cudaGraphConditionalHandleCreate(&hdl, cg, 0, 0) == cudaSuccess;
    if (rc == WAM_OK && capture_ok) {
      Span sp(c, WAM_KCLASS_RR_PROBE);
      capture_ok = rr_decide(c->d_gate, split > 0, split < N, c->d_rrapply, c->d_dec, c->d_dec_n, kDecCap, hdl, 1,
                             c->stream) == cudaSuccess;
    }
    cudaGraphNode_t cn = nullptr;
    cudaGraph_t body = nullptr;
    if (rc == WAM_OK && capture_ok) {
      cudaGraphNodeParams cp = {};
      cp.type = cudaGraphNodeTypeConditional;
      cp.conditional.handle = hdl;
      cp.conditional.type = cudaGraphCondTypeIf;
      cp.conditional.size = 1;
      capture_ok = cudaStreamGetCaptureInfo(c->stream, &cs, nullptr, &cg, &deps, nullptr, &nd) == cudaSuccess &&
                   cudaGraphAddNode(&cn, cg, deps, nullptr, nd, &cp) == cudaSuccess &&
                   cudaStreamUpdateCaptureDependencies(c->stream, &cn, nullptr, 1, cudaStreamSetCaptureDependencies) ==
                       cudaSuccess;
      body = capture_ok ? cp.conditional.phGraph_out[0] : nullptr;
    }
    if (rc == WAM_OK && capture_ok) {
      // the rejected branch: gather the item, run the middle layers on it
      capture_ok = cudaStreamBeginCaptureToGraph(c->aux_stream, body, nullptr, nullptr, 0,
                                                 cudaStreamCaptureModeThreadLocal) == cudaSuccess;
      if (capture_ok) {
        cudaStream_t main = c->stream;
        c->stream = c->aux_stream;
        {
          Span sp(c, WAM_KCLASS_RR_APPLY, 0.0, 8.0 * double(N) * d);
          if (rr_gather(c->hm, c->h, c->d_map0, 1, int64_t(N) * d, c->stream) != cudaSuccess) capture_ok = false;
        }
        for (int l = s; l < e && rc == WAM_OK && capture_ok; ++l) rc = run_layer(c, l, c->hm, 1, c->d_map0, nullptr);
        c->stream = main;
        cudaGraph_t bo = nullptr;
        if (cudaStreamEndCapture(c->aux_stream, &bo) != cudaSuccess) capture_ok = false;
      }
    }
    if (rc == WAM_OK && capture_ok) {
      Span sp(c, WAM_KCLASS_RR_APPLY, 0.0, 24.0 * double(N) * d);
      capture_ok = rr_apply(c->h, c->hm, c->hq, st->pa, st->ra, c->d_items, c->d_rrapply, 1, N, d, split, c->stream) ==
                   cudaSuccess;
    }
    for (int l = e; l < L && rc == WAM_OK && capture_ok; ++l) rc = run_layer(c, l, c->h, 1, nullptr, nullptr);
    const cudaError_t ec = cudaStreamEndCapture(c->stream, &g);
    cudaGraphExec_t ex = nullptr;
    if (rc == WAM_OK && capture_ok && ec == cudaSuccess && g != nullptr &&
        cudaGraphInstantiate(&ex, g, 0) == cudaSuccess) {
      cudaGraphDestroy(g);
      hit = c->rr_graphs.emplace(key, ex).first;
      c->graph_kernels[ex] = c->stats.n_kernel_launches - k0;
      c->stats.n_kernel_launches = k0;   // counted again when launched below
    } else {
      // nothing of the capture ran: use the host-branching path from now on
      if (g != nullptr) cudaGraphDestroy(g);
      cudaGetLastError();
      c->err.clear();
      c->stats.n_kernel_launches = k0;
      c->dev_branch_ok = false;
      return WAM_OK;
    }
  }
  if (c->dec_queued - c->dec_resolved >= kDecCap) {
    TRY(queue_decision_copy(c));
    TRY(resolve_decisions(c, true));
  }
  CK(cudaGraphLaunch(hit->second, c->stream));
  c->stats.n_kernel_launches += c->graph_kernels[hit->second];
  c->dec_queued++;
  *done = true;
  return WAM_OK;
}

int obs_embed(wam_ctx* c, wam_state* st) {
  const int M = st->B * c->No;
  if (c->bf16) {
    {
      Span sp(c, WAM_KCLASS_EMBED, 0.0, 6.0 * M * c->d);
      CK(cast_f32_bf16(st->obs, static_cast<bf16*>(c->obs_lp), int64_t(M) * c->d, c->stream));
    }
    TRY(gemm(c, &c->tm_obs_lp, c->obs_lp, &c->tm_obs_w, c->obs_wt, M, c->d, c->d, kEpiF32,
             epi_args(c->obs_b, st->obs_emb, nullptr, 0, c->No, nullptr)));
  } else {
    TRY(gemm(c, nullptr, st->obs, nullptr, c->obs_wt, M, c->d, c->d, kEpiF32,
             epi_args(c->obs_b, st->obs_emb, nullptr, 0, c->No, nullptr)));
  }
  return WAM_OK;
}

bool rr_enabled(const wam_ctx* c) {
  const wam_config& g = c->cfg;
  return g.rr_policy != WAM_RR_OFF && 0 < g.rr_q && g.rr_q < g.rr_s && g.rr_s < g.rr_e && g.rr_e < g.n_layers;
}

// Run every episode `n[b]` steps from its current stage (§3.2 native solver, §3.3 RR).
int run_steps(wam_ctx* c, wam_state* st, const std::vector<int>& n) {
  const int B = st->B;
  const int d = c->d, N = c->N, L = c->L;
  const int64_t stage_stride = int64_t(B) * c->T;
  const bool rr_on = rr_enabled(c);
  const int q = c->cfg.rr_q, s = c->cfg.rr_s, e = c->cfg.rr_e;
  const int split_row = c->split;
  TRY(obs_embed(c, st));
  int max_n = 0;
  for (int b = 0; b < B; ++b) max_n = std::max(max_n, n[b]);
  // decisions of earlier calls whose copies have landed; the rest lose their log entry
  TRY(resolve_decisions(c, false));
  for (auto& pd : c->dec_pending)
    if (pd.st == st) pd.log_idx = -1;
  st->log.clear();
  std::vector<StepItem> items, uitems;
  std::vector<int> uidx;
  // The conditioning depends on sigma alone (exact equality: equal sigmas give bit-identical
  // modulations), and every stage each episode runs in this call is known now, so one pass over
  // the conditioning weights computes the modulation rows of all distinct sigmas of the call;
  // each step then gathers its work items' rows (none to gather with one item and one sigma).
  for (int b = 0; b < B; ++b)
    for (int j = 0; j < n[b]; ++j) {
      const int k = st->meta[b].stage + j;
      if (k < 0 || k >= c->K) continue;
      bool seen = false;
      for (const StepItem& u : uitems) seen = seen || u.sigma == c->sigma[k];
      if (seen) continue;
      StepItem it;
      it.ep = b;
      it.stage = k;
      it.sigma = c->sigma[k];
      it.dsigma = c->sigma[k + 1] - c->sigma[k];
      uitems.push_back(it);
    }
  const int U = static_cast<int>(uitems.size());
  if (U > c->Ucap) return fail(c, WAM_ERR_INVALID_ARG, "more distinct noise levels than denoising steps");
  const bool cond_in_place = B == 1 && U == 1;
  if (U > 0) {
    TRY(upload(c, c->d_uitems, uitems.data(), sizeof(StepItem) * U));
    float* cond_out = cond_in_place ? c->mods : c->mods_u;
    // features -> W1 (split K) -> SiLU -> W2 (split K) -> SiLU -> every layer's modulation; each
    // stage reduces the previous stage's K-split partial rows in a fixed order
    {
      Span sp(c, WAM_KCLASS_COND, 2.0 * U * 256 * d, 4.0 * 256 * d);
      const CondGemv g{nullptr, 0, nullptr, 0, 1, c->d_uitems, c->t_w1, false, 256, d, U, kT1Splits, c->t1, nullptr};
      CK(cond_gemv(g, c->stream));
    }
    {
      Span sp(c, WAM_KCLASS_COND, 2.0 * U * d * d, 4.0 * d * d);
      const CondGemv g{c->t1, kT1Splits, c->t_b1, 1, 0, c->d_uitems, c->t_w2, false, d, d, U, kT2Splits, c->cvec, nullptr};
      CK(cond_gemv(g, c->stream));
    }
    {
      Span sp(c, WAM_KCLASS_COND, 2.0 * U * d * c->mod_n, (c->bf16 ? 2.0 : 4.0) * d * c->mod_n);
      const CondGemv g{c->cvec, kT2Splits, c->t_b2, 1, 0, c->d_uitems, c->mod_w, c->bf16, d, static_cast<int>(c->mod_n),
                       U, 1, cond_out, c->mod_b};
      CK(cond_gemv(g, c->stream));
    }
  }
  std::vector<int> rr_path, gate_ok;
  std::vector<RRGate> gates(2 * B);
  std::vector<RRApply> ap(B);
  std::vector<int> midmap;
  for (int i = 0; i < max_n; ++i) {
    items.clear();
    for (int b = 0; b < B; ++b) {
      if (n[b] <= i) continue;
      const int k = st->meta[b].stage;
      StepItem it;
      it.ep = b;
      it.stage = k;
      it.sigma = c->sigma[k];
      it.dsigma = c->sigma[k + 1] - c->sigma[k];
      items.push_back(it);
    }
    const int Bw = static_cast<int>(items.size());
    TRY(upload(c, c->d_items, items.data(), sizeof(StepItem) * Bw));
    // this step's modulation rows: work item w takes the call's row of its sigma
    if (!cond_in_place) {
      uidx.assign(Bw, 0);
      for (int w = 0; w < Bw; ++w)
        for (int j = 0; j < U; ++j)
          if (uitems[j].sigma == items[w].sigma) {
            uidx[w] = j;
            break;
          }
      TRY(upload(c, c->d_uidx, uidx.data(), sizeof(int) * Bw));
      Span sp(c, WAM_KCLASS_COND, 0.0, 8.0 * Bw * c->mod_n);
      CK(rr_gather(c->mods, c->mods_u, c->d_uidx, Bw, c->mod_n, c->stream));
    }
    {
      Span sp(c, WAM_KCLASS_EMBED, 0.0, 4.0 * Bw * double(N) * d * 2.0);
      CK(embed_tokens(c->h, st->xhist, stage_stride, c->d_items, st->x, c->T, st->obs_emb, c->vid_w, c->vid_b,
                      c->act_w, c->act_b, c->pos, Bw, c->No, c->Nv, c->vd, c->Na, c->ad, d, c->stream));
    }
    // RR eligibility per item (App. B.1 policies)
    rr_path.assign(Bw, 0);
    gate_ok.assign(Bw, 0);
    bool any_rr = false, any_gate = false;
    for (int w = 0; w < Bw; ++w) {
      const EpisodeMeta& m = st->meta[items[w].ep];
      if (!rr_on) continue;
      const bool path_ok = c->cfg.rr_policy == WAM_RR_ALL_PATHS ||
                           (c->cfg.rr_policy == WAM_RR_PREFIX_PATH && m.path == kPathPrefix);
      if (!path_ok) continue;
      rr_path[w] = 1;
      any_rr = true;
      const bool allowed = c->cfg.rr_policy == WAM_RR_ALL_PATHS || m.path_steps >= 1;
      if (allowed && m.rr_valid) {
        gate_ok[w] = 1;
        any_gate = true;
      }
    }
    std::vector<int> accepted(Bw, 0);
    bool dev_step = false;   // this step's RR decision is taken on the device (work item 0)
    if (any_rr && Bw == 1 && gate_ok[0] && c->dev_branch && c->dev_branch_ok && c->graph_replay && c->graphs_ok &&
        !c->prof_on) {
      const int nch = rr_num_chunks(int64_t(std::max(split_row, N - split_row)) * d);
      TRY(rr_step_device(c, st, nch, &dev_step));
    }
    if (dev_step) {
      // layers, gate, middle layers or injection and the tail all ran in the step's graph
    } else if (!any_rr) {
      TRY(run_layers(c, 0, L, c->h, Bw, nullptr, -1));
    } else {
      TRY(run_layers(c, 0, s, c->h, Bw, nullptr, q));
      if (any_gate) {
        const int nch = rr_num_chunks(int64_t(std::max(split_row, N - split_row)) * d);
        {
          Span sp(c, WAM_KCLASS_RR_PROBE, 0.0, 12.0 * Bw * double(N) * d);
          CK(rr_probe_partial(c->h, c->hq, st->pa, c->d_items, Bw, N, d, split_row, nch, c->d_part, c->stream));
        }
        {
          Span sp(c, WAM_KCLASS_RR_PROBE);
          CK(rr_gate(c->d_part, Bw, nch, int64_t(split_row) * d, int64_t(N - split_row) * d, c->cfg.rr_alpha_min,
                     c->cfg.rr_alpha_max, c->cfg.rr_eps, c->cfg.rr_gamma_cos, c->cfg.rr_gamma_fit, c->d_gate, c->stream));
        }
        TRY(readback(c, gates.data(), c->d_gate, sizeof(RRGate) * 2 * Bw));
        // every non-empty branch must pass (§3.3); a single-branch model has one
        for (int w = 0; w < Bw; ++w)
          if (gate_ok[w] && (split_row == 0 || gates[2 * w].pass) && (split_row == N || gates[2 * w + 1].pass))
            accepted[w] = 1;
      }
      midmap.clear();
      for (int w = 0; w < Bw; ++w) {
        ap[w].cidx = 0;
        ap[w].alpha0 = ap[w].alpha1 = 0.0f;
        if (accepted[w]) {
          ap[w].mode = kRRInject;
          ap[w].alpha0 = static_cast<float>(gates[2 * w].alpha);
          ap[w].alpha1 = static_cast<float>(gates[2 * w + 1].alpha);
        } else {
          ap[w].mode = rr_path[w] ? kRRRefresh : kRRCopyBack;
          ap[w].cidx = static_cast<int>(midmap.size());
          midmap.push_back(w);
        }
      }
      const int nmid = static_cast<int>(midmap.size());
      if (nmid > 0) {
        TRY(upload(c, c->d_map, midmap.data(), sizeof(int) * nmid));
        {
          Span sp(c, WAM_KCLASS_RR_APPLY, 0.0, 8.0 * nmid * double(N) * d);
          CK(rr_gather(c->hm, c->h, c->d_map, nmid, int64_t(N) * d, c->stream));
        }
        TRY(run_layers(c, s, e, c->hm, nmid, c->d_map, -1));
      }
      TRY(upload(c, c->d_rrapply, ap.data(), sizeof(RRApply) * Bw));
      {
        // algorithmic bytes per element: inject 12 (h, R_a in; h out), refresh 24 (h_s, h_e, h_q
        // in; R_a, p_a, h out), copy-back 8
        double per = 0.0;
        for (int w = 0; w < Bw; ++w) per += ap[w].mode == kRRInject ? 12.0 : (ap[w].mode == kRRRefresh ? 24.0 : 8.0);
        Span sp(c, WAM_KCLASS_RR_APPLY, 0.0, per * double(N) * d);
        CK(rr_apply(c->h, c->hm, c->hq, st->pa, st->ra, c->d_items, c->d_rrapply, Bw, N, d, split_row, c->stream));
      }
      TRY(run_layers(c, e, L, c->h, Bw, nullptr, -1));
    }
    {
      Span sp(c, WAM_KCLASS_FINAL, 2.0 * Bw * double(c->Nv * c->vd + c->Na * c->ad) * d,
              4.0 * Bw * double(c->Nv + c->Na) * d + 16.0 * Bw * c->T);
      CK(final_euler(c->h, c->d_items, c->mods, c->mod_n, 6 * L * d, c->vout_w, c->vout_b, c->aout_w, c->aout_b,
                     st->x, st->xhist, st->vhist, stage_stride, c->T, Bw, c->No, c->Nv, c->vd, c->Na, c->ad, d,
                     c->bf16, c->d_fhead, c->d_fconst, c->stream));
    }
    // bookkeeping (§3.4) and reuse statistics (App. D.2)
    for (int w = 0; w < Bw; ++w) {
      EpisodeMeta& m = st->meta[items[w].ep];
      wam_step_record rec;
      std::memset(&rec, 0, sizeof(rec));
      rec.episode = items[w].ep;
      rec.stage = m.stage;
      rec.rr_active = rr_path[w];
      rec.rr_attempt = gate_ok[w];
      rec.rr_accept = accepted[w];
      if (gate_ok[w]) {
        for (int br = 0; br < 2; ++br) {
          if (br == 0 ? split_row == 0 : split_row == N) continue;  // empty branch
          rec.alpha[br] = static_cast<float>(gates[2 * w + br].alpha);
          rec.cos[br] = static_cast<float>(gates[2 * w + br].cos);
          rec.fit[br] = static_cast<float>(gates[2 * w + br].fit);
        }
      }
      if (dev_step) c->dec_pending.push_back(wam_ctx::PendingDec{st, static_cast<int>(st->log.size())});
      st->log.push_back(rec);
      c->stats.n_episode_steps++;
      c->stats.n_layer_evals += accepted[w] ? (L - (e - s)) : L;
      if (rr_path[w]) {
        c->stats.b_dense += L;
        m.rr_valid = 1;
      }
      if (gate_ok[w]) c->stats.n_attempt++;
      if (accepted[w]) {
        c->stats.n_reuse++;
        c->stats.b_skip += e - s;
      }
      m.stage++;
      m.since_bind++;
      m.path_steps++;
      if (m.stage == c->K) m.finished = 1;
    }
  }
  return queue_decision_copy(c);
}

int copy_out(wam_ctx* c, wam_state* st, float* actions_out, float* video_out, bool& host_out) {
  if (actions_out != nullptr && c->Na > 0) {
    const size_t w = sizeof(float) * c->Na * c->ad;
    CK(cudaMemcpy2DAsync(actions_out, w, st->x + c->V, sizeof(float) * c->T, w, st->B, cudaMemcpyDefault, c->stream));
    host_out = host_out || !is_device_ptr(actions_out);
  }
  if (video_out != nullptr && c->V > 0) {
    const size_t w = sizeof(float) * c->V;
    CK(cudaMemcpy2DAsync(video_out, w, st->x, sizeof(float) * c->T, w, st->B, cudaMemcpyDefault, c->stream));
    host_out = host_out || !is_device_ptr(video_out);
  }
  return WAM_OK;
}

int validate_cfg(const wam_config* g, std::string& why) {
  if (g == nullptr) return why = "null config", WAM_ERR_INVALID_ARG;
  if (g->n_layers < 1 || g->d_model < 1 || g->n_heads < 1 || g->mlp_ratio < 1 || g->n_obs < 1 ||
      g->video_dim < 1 || g->action_dim < 1 || g->n_steps < 1 || g->batch_max < 1)
    return why = "every size must be >= 1", WAM_ERR_INVALID_ARG;
  if (g->n_video < 0 || g->n_action < 0 || g->n_video + g->n_action < 1)
    return why = "n_video and n_action must be >= 0, not both 0", WAM_ERR_INVALID_ARG;
  if (g->d_model % g->n_heads != 0) return why = "d_model must be a multiple of n_heads", WAM_ERR_INVALID_ARG;
  if (g->precision != WAM_PREC_FP32 && g->precision != WAM_PREC_BF16) return why = "unknown precision", WAM_ERR_INVALID_ARG;
  if (g->batch_max > kMaxBatch) return why = "batch_max above 256", WAM_ERR_UNSUPPORTED;
  if (g->d_model % 128 != 0 || g->d_model > 1536) return why = "d_model must be a multiple of 128, at most 1536", WAM_ERR_UNSUPPORTED;
  if (g->video_dim > 16 || g->action_dim > 16) return why = "video_dim and action_dim must be <= 16", WAM_ERR_UNSUPPORTED;
  const int dh = g->d_model / g->n_heads;
  if (g->precision == WAM_PREC_BF16 && !attention_bf16_supported(dh)) return why = "bf16 attention supports head dim 64 or 72", WAM_ERR_UNSUPPORTED;
  if (g->precision == WAM_PREC_FP32 && dh > 128) return why = "fp32 attention supports head dim <= 128", WAM_ERR_UNSUPPORTED;
  if (!(g->sched_shift > 0.0f)) return why = "sched_shift must be > 0", WAM_ERR_INVALID_ARG;
  if (g->tr_entry_stage < 0 || g->tr_entry_stage >= g->n_steps) return why = "tr_entry_stage outside [0, K)", WAM_ERR_INVALID_ARG;
  if (g->tr_retain_stage >= g->n_steps || g->tr_retain_stage < -1) return why = "tr_retain_stage outside [-1, K)", WAM_ERR_INVALID_ARG;
  if (g->rr_policy < 0 || g->rr_policy > 2) return why = "unknown rr_policy", WAM_ERR_INVALID_ARG;
  if (g->rr_policy != WAM_RR_OFF &&
      !(0 < g->rr_q && g->rr_q < g->rr_s && g->rr_s < g->rr_e && g->rr_e < g->n_layers))
    return why = "RR needs 0 < q < s < e < n_layers", WAM_ERR_INVALID_ARG;
  if (g->or_n_components < 1 || g->or_n_components > 4 || g->n_obs % g->or_n_components != 0)
    return why = "or_n_components must be 1..4 and divide n_obs", WAM_ERR_INVALID_ARG;
  for (int m = 0; m < g->or_n_components; ++m)
    if (!(g->or_deltas[m] > 0.0f) || !(g->or_weights[m] >= 0.0f)) return why = "OR deltas must be > 0, weights >= 0", WAM_ERR_INVALID_ARG;
  if (g->or_kappa_max < 0) return why = "or_kappa_max must be >= 0", WAM_ERR_INVALID_ARG;
  const int64_t mod_n = int64_t(6 * g->n_layers + 2) * g->d_model;
  if (mod_n % 2 != 0) return why = "modulation width must be even", WAM_ERR_UNSUPPORTED;
  return WAM_OK;
}

size_t weight_count(const wam_config* g) {
  const size_t d = g->d_model, L = g->n_layers, R = g->mlp_ratio, N = size_t(g->n_obs) + g->n_video + g->n_action;
  const size_t vd = g->video_dim, ad = g->action_dim;
  size_t n = d * d + d + vd * d + d + ad * d + d + N * d + 256 * d + d + d * d + d;
  n += L * (d * 6 * d + 6 * d + d * 3 * d + 3 * d + d * d + d + d * R * d + R * d + R * d * d + d);
  n += d * 2 * d + 2 * d + d * vd + vd + d * ad + ad;
  return n;
}

int build_weights(wam_ctx* c, const float* src) {
  const int d = c->d, L = c->L, dff = c->dff;
  const bool b16 = c->bf16;
  const size_t wel = b16 ? 2 : 4;
  size_t off = 0;
  auto take = [&](size_t n) {
    const float* p = src + off;
    off += n;
    return p;
  };
  auto dmat = [&](void** out, size_t n) -> int {
    void* p = nullptr;
    if (cudaMalloc(&p, n * wel) != cudaSuccess) {
      cudaGetLastError();
      return fail(c, WAM_ERR_OOM, "weight allocation failed");
    }
    c->allocs.push_back(p);
    *out = p;
    return WAM_OK;
  };
  auto dvec = [&](float** out, const float* from, size_t n) -> int {
    TRY(dalloc(c, c->allocs, out, n));
    CK(cudaMemcpyAsync(*out, from, n * sizeof(float), cudaMemcpyDeviceToDevice, c->stream));
    return WAM_OK;
  };
  auto tmat = [&](void** out, const float* from, int K, int Nn) -> int {  // [K,N] -> [N,K]
    TRY(dmat(out, size_t(K) * Nn));
    CK(transpose_cast(from, *out, b16, K, Nn, c->stream));
    return WAM_OK;
  };
  TRY(tmat(&c->obs_wt, take(size_t(d) * d), d, d));
  TRY(dvec(&c->obs_b, take(d), d));
  TRY(dvec(&c->vid_w, take(size_t(c->vd) * d), size_t(c->vd) * d));
  TRY(dvec(&c->vid_b, take(d), d));
  TRY(dvec(&c->act_w, take(size_t(c->ad) * d), size_t(c->ad) * d));
  TRY(dvec(&c->act_b, take(d), d));
  TRY(dvec(&c->pos, take(size_t(c->N) * d), size_t(c->N) * d));
  TRY(dvec(&c->t_w1, take(size_t(256) * d), size_t(256) * d));
  TRY(dvec(&c->t_b1, take(d), d));
  TRY(dvec(&c->t_w2, take(size_t(d) * d), size_t(d) * d));
  TRY(dvec(&c->t_b2, take(d), d));
  TRY(dmat(&c->mod_w, size_t(d) * c->mod_n));
  TRY(dalloc(c, c->allocs, &c->mod_b, c->mod_n));
  c->layers.resize(L);
  for (int l = 0; l < L; ++l) {
    LayerW& w = c->layers[l];
    const float* ada_w = take(size_t(d) * 6 * d);
    CK(copy_cast_2d(ada_w, 6 * d, static_cast<uint8_t*>(c->mod_w) + size_t(l) * 6 * d * wel, b16, c->mod_n, d, 6 * d, c->stream));
    CK(cudaMemcpyAsync(c->mod_b + size_t(l) * 6 * d, take(6 * d), sizeof(float) * 6 * d, cudaMemcpyDeviceToDevice, c->stream));
    TRY(tmat(&w.qkv_wt, take(size_t(d) * 3 * d), d, 3 * d));
    TRY(dvec(&w.qkv_b, take(3 * d), 3 * d));
    TRY(tmat(&w.out_wt, take(size_t(d) * d), d, d));
    TRY(dvec(&w.out_b, take(d), d));
    TRY(tmat(&w.up_wt, take(size_t(d) * dff), d, dff));
    TRY(dvec(&w.up_b, take(dff), dff));
    TRY(tmat(&w.down_wt, take(size_t(dff) * d), dff, d));
    TRY(dvec(&w.down_b, take(d), d));
  }
  CK(copy_cast_2d(take(size_t(d) * 2 * d), 2 * d, static_cast<uint8_t*>(c->mod_w) + size_t(L) * 6 * d * wel, b16, c->mod_n, d, 2 * d, c->stream));
  CK(cudaMemcpyAsync(c->mod_b + size_t(L) * 6 * d, take(2 * d), sizeof(float) * 2 * d, cudaMemcpyDeviceToDevice, c->stream));
  // output heads padded to 16 columns (zeros beyond video_dim / action_dim): 64-byte rows
  auto head = [&](float** w, float** bvec, int od) -> int {
    TRY(dalloc(c, c->allocs, w, size_t(d) * 16));
    TRY(dalloc(c, c->allocs, bvec, 16));
    CK(cudaMemsetAsync(*w, 0, sizeof(float) * d * 16, c->stream));
    CK(cudaMemsetAsync(*bvec, 0, sizeof(float) * 16, c->stream));
    CK(copy_cast_2d(take(size_t(d) * od), od, *w, false, 16, d, od, c->stream));
    CK(cudaMemcpyAsync(*bvec, take(od), sizeof(float) * od, cudaMemcpyDeviceToDevice, c->stream));
    return WAM_OK;
  };
  TRY(head(&c->vout_w, &c->vout_b, c->vd));
  TRY(head(&c->aout_w, &c->aout_b, c->ad));
  if (off != weight_count(&c->cfg)) return fail(c, WAM_ERR_INVALID_ARG, "internal weight layout mismatch");
  return WAM_OK;
}

int encode(wam_ctx* c, GemmOperand* m, const void* base, uint64_t rows, uint64_t K, bool rows64 = false) {
  const int r = tc_encode_gemm_operand(m, base, rows, K, rows64);
  if (r != 0) return fail(c, WAM_ERR_CUDA, "cuTensorMapEncodeTiled failed (" + std::to_string(r) + ")");
  return WAM_OK;
}

int create_impl(wam_ctx* c, const wam_config* cfg, const float* weights, size_t n_weights, void* stream) {
  std::string why;
  const int v = validate_cfg(cfg, why);
  if (v != WAM_OK) return fail(c, v, why);
  if (weights == nullptr || n_weights != weight_count(cfg)) return fail(c, WAM_ERR_INVALID_ARG, "weights null or n_weights != wam_weight_count(cfg)");
  c->cfg = *cfg;
  c->L = cfg->n_layers;
  c->d = cfg->d_model;
  c->H = cfg->n_heads;
  c->R = cfg->mlp_ratio;
  c->No = cfg->n_obs;
  c->Nv = cfg->n_video;
  c->vd = cfg->video_dim;
  c->Na = cfg->n_action;
  c->ad = cfg->action_dim;
  c->N = c->No + c->Nv + c->Na;
  c->split = c->Na == 0 ? c->N : (c->Nv == 0 ? 0 : c->No + c->Nv);
  c->V = c->Nv * c->vd;
  c->T = c->V + c->Na * c->ad;
  c->K = cfg->n_steps;
  c->dff = c->R * c->d;
  c->Bmax = cfg->batch_max;
  c->mod_n = int64_t(6 * c->L + 2) * c->d;
  c->bf16 = cfg->precision == WAM_PREC_BF16;
  c->stream = static_cast<cudaStream_t>(stream);
  std::memset(&c->stats, 0, sizeof(c->stats));
  for (int k = 0; k <= c->K; ++k) {
    const double t = 1.0 - double(k) / c->K;
    const double sft = cfg->sched_shift;
    c->sigma.push_back(sft * t / (1.0 + (sft - 1.0) * t));
  }
  CK(cudaGetDevice(&c->device));
  CK(cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device));
  if (c->bf16) {
    int major = 0, minor = 0;
    CK(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, c->device));
    CK(cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, c->device));
    if (major != 10) return fail(c, WAM_ERR_UNSUPPORTED, "bf16 tensor-core kernels need a Blackwell (sm_10x) device");
  }
  if (c->bf16 && (c->dff % 128 != 0 || (3 * c->d) % 128 != 0))
    return fail(c, WAM_ERR_UNSUPPORTED, "GEMM widths must be multiples of 128");
  // weights: bring the flat buffer to the device once, then convert
  const float* wdev = weights;
  float* tmp = nullptr;
  if (!is_device_ptr(weights)) {
    if (cudaMalloc(&tmp, n_weights * sizeof(float)) != cudaSuccess) {
      cudaGetLastError();
      return fail(c, WAM_ERR_OOM, "weight staging allocation failed");
    }
    cudaError_t e = cudaMemcpyAsync(tmp, weights, n_weights * sizeof(float), cudaMemcpyHostToDevice, c->stream);
    if (e != cudaSuccess) {
      cudaFree(tmp);
      return fail_cuda(c, "weight upload", e);
    }
    wdev = tmp;
  }
  const int rw = build_weights(c, wdev);
  cudaError_t se = cudaStreamSynchronize(c->stream);
  if (tmp) cudaFree(tmp);
  if (rw != WAM_OK) return rw;
  if (se != cudaSuccess) return fail_cuda(c, "weight conversion", se);
  // activations
  const size_t rows = size_t(c->Bmax) * c->N;
  const size_t el = c->bf16 ? 2 : 4;
  uint8_t *xln, *qkv, *att, *u, *olp;
  TRY(dalloc(c, c->allocs, &c->h, rows * c->d));
  TRY(dalloc(c, c->allocs, &c->hq, rows * c->d));
  TRY(dalloc(c, c->allocs, &c->hm, rows * c->d));
  TRY(dalloc(c, c->allocs, &xln, rows * c->d * el));
  TRY(dalloc(c, c->allocs, &qkv, rows * 3 * c->d * el));
  TRY(dalloc(c, c->allocs, &att, rows * c->d * el));
  TRY(dalloc(c, c->allocs, &u, rows * c->dff * el));
  TRY(dalloc(c, c->allocs, &olp, size_t(c->Bmax) * c->No * c->d * el));
  c->xln = xln;
  c->qkv = qkv;
  c->att = att;
  c->u = u;
  c->obs_lp = olp;
  c->Ucap = std::max(c->Bmax, c->K);
  TRY(dalloc(c, c->allocs, &c->t1, size_t(kT1Splits) * c->Ucap * c->d));
  TRY(dalloc(c, c->allocs, &c->cvec, size_t(kT2Splits) * c->Ucap * c->d));
  TRY(dalloc(c, c->allocs, &c->mods, size_t(c->Bmax) * c->mod_n));
  TRY(dalloc(c, c->allocs, &c->d_items, c->Bmax));
  TRY(dalloc(c, c->allocs, &c->d_map, c->Bmax));
  TRY(dalloc(c, c->allocs, &c->d_uitems, c->Ucap));
  TRY(dalloc(c, c->allocs, &c->d_uidx, c->Bmax));
  TRY(dalloc(c, c->allocs, &c->mods_u, size_t(c->Ucap) * c->mod_n));
  TRY(dalloc(c, c->allocs, &c->d_rrapply, c->Bmax));
  TRY(dalloc(c, c->allocs, &c->d_gate, 2 * c->Bmax));
  TRY(dalloc(c, c->allocs, &c->d_adapt, c->Bmax));
  TRY(dalloc(c, c->allocs, &c->d_eps, size_t(c->Bmax) * c->T));
  TRY(dalloc(c, c->allocs, &c->d_obs_new, size_t(c->Bmax) * c->No * c->d));
  TRY(dalloc(c, c->allocs, &c->d_fhead, size_t(c->Bmax) * 2 * size_t(final_head_bytes(c->d))));
  TRY(dalloc(c, c->allocs, &c->d_fconst, size_t(c->Bmax) * 64));
  TRY(dalloc(c, c->allocs, &c->d_err, 1));
  CK(cudaMemset(c->d_err, 0, sizeof(int)));
  TRY(dalloc(c, c->allocs, &c->d_map0, 1));
  CK(cudaMemset(c->d_map0, 0, sizeof(int)));
  TRY(dalloc(c, c->allocs, &c->d_dec, kDecCap));
  TRY(dalloc(c, c->allocs, &c->d_dec_n, 1));
  CK(cudaMemset(c->d_dec_n, 0, sizeof(unsigned long long)));
  CK(cudaHostAlloc(reinterpret_cast<void**>(&c->h_dec), sizeof(RRDecision) * kDecCap, cudaHostAllocDefault));
  // scratch for the float64 partial sums of TR / OR / RR reductions
  const int split = c->split;
  const size_t p_tr = size_t(c->Bmax) * 2 * tr_num_chunks(c->T, c->V);
  const size_t p_or = size_t(c->Bmax) * cfg->or_n_components * or_num_chunks(int64_t(c->No / cfg->or_n_components) * c->d);
  const size_t p_rr = size_t(c->Bmax) * 2 * 3 * rr_num_chunks(int64_t(std::max(split, c->N - split)) * c->d);
  c->part_doubles = std::max(p_tr, std::max(p_or, p_rr));
  TRY(dalloc(c, c->allocs, &c->d_part, c->part_doubles));
  if (c->bf16) {
    // A operands also with 64-row boxes: the clustered GEMM multicasts 64-row halves of A
    TRY(encode(c, &c->tm_xln, c->xln, rows, c->d, true));
    TRY(encode(c, &c->tm_att, c->att, rows, c->d, true));
    TRY(encode(c, &c->tm_u, c->u, rows, c->dff, true));
    TRY(encode(c, &c->tm_obs_lp, c->obs_lp, size_t(c->Bmax) * c->No, c->d, true));
    TRY(encode(c, &c->tm_obs_w, c->obs_wt, c->d, c->d));
    c->tc_attn = c->d / c->H == 64 || c->d / c->H == 72;
    if (c->tc_attn) {
      c->vt_ld = attention_tc_vt_ld(c->N);
      uint8_t* vt = nullptr;
      TRY(dalloc(c, c->allocs, &vt, size_t(c->Bmax) * c->d * c->vt_ld * 2));
      CK(cudaMemsetAsync(vt, 0, size_t(c->Bmax) * c->d * c->vt_ld * 2, c->stream));
      c->vt = vt;
      if (attention_tc_encode(&c->attn_maps, c->qkv, c->vt, c->Bmax, c->N, c->d, c->H, c->vt_ld) != 0)
        return fail(c, WAM_ERR_CUDA, "cuTensorMapEncodeTiled failed for the attention operands");
    }
    c->chain_ok = c->tc_attn && dit_chain_supported(c->d, c->dff) && c->d % 128 == 0;
    if (c->chain_ok) {
      const int nctr = dit_chain_counters(static_cast<int>(rows));
      TRY(dalloc(c, c->allocs, &c->d_chain_ctr, nctr));
      CK(cudaMemsetAsync(c->d_chain_ctr, 0, sizeof(int) * nctr, c->stream));
    }
    for (LayerW& w : c->layers) {
      // every weight also with 64-row boxes: 64-wide tiles and the B halves of 128-wide CTA pairs
      TRY(encode(c, &w.tm_qkv, w.qkv_wt, 3 * c->d, c->d, true));
      TRY(encode(c, &w.tm_out, w.out_wt, c->d, c->d, true));
      TRY(encode(c, &w.tm_up, w.up_wt, c->dff, c->d, true));
      TRY(encode(c, &w.tm_down, w.down_wt, c->d, c->dff, true));
    }
  }
  CK(cudaHostAlloc(reinterpret_cast<void**>(&c->ring), kRingSlots * kSlotBytes, cudaHostAllocDefault));
  for (int i = 0; i < kRingSlots; ++i) {
    CK(cudaEventCreateWithFlags(&c->ring_ev[i], cudaEventDisableTiming));
    c->ring_used[i] = false;
  }
  c->readback_bytes = std::max<size_t>(c->part_doubles * sizeof(double), sizeof(RRGate) * 2 * c->Bmax) + 64;
  CK(cudaHostAlloc(reinterpret_cast<void**>(&c->readback), c->readback_bytes, cudaHostAllocDefault));
  return WAM_OK;
}

void destroy_impl(wam_ctx* c) {
  if (!c->allocs.empty()) cudaStreamSynchronize(c->stream);
  for (auto& kv : c->layer_graphs) cudaGraphExecDestroy(kv.second);
  c->layer_graphs.clear();
  for (auto& kv : c->rr_graphs) cudaGraphExecDestroy(kv.second);
  c->rr_graphs.clear();
  for (auto& b : c->dec_batches) cudaEventDestroy(b.first);
  c->dec_batches.clear();
  if (c->aux_stream) cudaStreamDestroy(c->aux_stream);
  if (c->h_dec) cudaFreeHost(c->h_dec);
  for (void* p : c->allocs) cudaFree(p);
  c->allocs.clear();
  if (c->ring) {
    cudaFreeHost(c->ring);
    for (int i = 0; i < kRingSlots; ++i)
      if (c->ring_ev[i]) cudaEventDestroy(c->ring_ev[i]);
  }
  if (c->readback) cudaFreeHost(c->readback);
  for (cudaEvent_t e : c->evpool) cudaEventDestroy(e);
}

int field_ptr(wam_ctx* c, const wam_state* st, int field, int index, void** p, size_t* bytes) {
  const size_t BT = size_t(st->B) * c->T;
  switch (field) {
    case WAM_FIELD_X: *p = st->x; *bytes = BT * 4; return WAM_OK;
    case WAM_FIELD_X_STAGE:
      if (index < 0 || index > c->K) return fail(c, WAM_ERR_INVALID_ARG, "stage index out of range");
      *p = st->xhist + size_t(index) * BT; *bytes = BT * 4; return WAM_OK;
    case WAM_FIELD_V_STEP:
      if (index < 0 || index >= c->K) return fail(c, WAM_ERR_INVALID_ARG, "step index out of range");
      *p = st->vhist + size_t(index) * BT; *bytes = BT * 4; return WAM_OK;
    case WAM_FIELD_X_INIT: *p = st->xb0; *bytes = BT * 4; return WAM_OK;
    case WAM_FIELD_OBS: *p = st->obs; *bytes = size_t(st->B) * c->No * c->d * 4; return WAM_OK;
    case WAM_FIELD_RR_P:
    case WAM_FIELD_RR_R:
      if (st->pa == nullptr) return fail(c, WAM_ERR_BAD_STATE, "RR is off for this context");
      *p = field == WAM_FIELD_RR_P ? st->pa : st->ra;
      *bytes = size_t(st->B) * c->N * c->d * 4;
      return WAM_OK;
    default: return fail(c, WAM_ERR_INVALID_ARG, "unknown field");
  }
}

}  // namespace

// =========================================================================================
// Public C ABI
// =========================================================================================
extern "C" {

size_t wam_weight_count(const wam_config* cfg) {
  std::string why;
  if (validate_cfg(cfg, why) == WAM_ERR_INVALID_ARG) return 0;
  return weight_count(cfg);
}

int wam_create(const wam_config* cfg, const float* weights, size_t n_weights, void* stream, wam_ctx** out) {
  if (out == nullptr) return WAM_ERR_INVALID_ARG;
  *out = nullptr;
  wam_ctx* c = new (std::nothrow) wam_ctx();
  if (c == nullptr) return WAM_ERR_OOM;
  std::memset(c->ring_ev, 0, sizeof(c->ring_ev));
  int r;
  try {  // no exception crosses the C ABI
    r = create_impl(c, cfg, weights, n_weights, stream);
  } catch (const std::bad_alloc&) {
    r = fail(c, WAM_ERR_OOM, "host allocation failed");
  } catch (...) {
    r = fail(c, WAM_ERR_CUDA, "unexpected host exception");
  }
  if (r != WAM_OK) {
    std::fprintf(stderr, "wam_create: %s\n", c->err.c_str());
    destroy_impl(c);
    delete c;
    return r;
  }
  *out = c;
  return WAM_OK;
}

void wam_destroy(wam_ctx* c) {
  if (c == nullptr) return;
  destroy_impl(c);
  delete c;
}

const char* wam_last_error(const wam_ctx* c) { return c ? c->err.c_str() : "null context"; }

int wam_set_stream(wam_ctx* c, void* stream) {
  if (c == nullptr) return WAM_ERR_INVALID_ARG;
  c->stream = static_cast<cudaStream_t>(stream);
  return WAM_OK;
}

int wam_state_create(wam_ctx* c, int32_t batch, wam_state** out) try {
  if (c == nullptr || out == nullptr) return WAM_ERR_INVALID_ARG;
  *out = nullptr;
  if (batch < 1 || batch > c->Bmax) return fail(c, WAM_ERR_INVALID_ARG, "batch outside [1, batch_max]");
  wam_state* st = new (std::nothrow) wam_state();
  if (st == nullptr) return fail(c, WAM_ERR_OOM, "host allocation failed");
  st->ctx = c;
  st->B = batch;
  const size_t BT = size_t(batch) * c->T;
  auto cleanup = [&](int r) {
    for (void* p : st->allocs) cudaFree(p);
    delete st;
    return r;
  };
  int r;
  if ((r = dalloc(c, st->allocs, &st->x, BT)) != WAM_OK) return cleanup(r);
  if ((r = dalloc(c, st->allocs, &st->xhist, BT * (c->K + 1))) != WAM_OK) return cleanup(r);
  if ((r = dalloc(c, st->allocs, &st->vhist, BT * c->K)) != WAM_OK) return cleanup(r);
  if ((r = dalloc(c, st->allocs, &st->xb0, BT)) != WAM_OK) return cleanup(r);
  if ((r = dalloc(c, st->allocs, &st->obs, size_t(batch) * c->No * c->d)) != WAM_OK) return cleanup(r);
  if ((r = dalloc(c, st->allocs, &st->obs_emb, size_t(batch) * c->No * c->d)) != WAM_OK) return cleanup(r);
  if (rr_enabled(c)) {
    if ((r = dalloc(c, st->allocs, &st->pa, size_t(batch) * c->N * c->d)) != WAM_OK) return cleanup(r);
    if ((r = dalloc(c, st->allocs, &st->ra, size_t(batch) * c->N * c->d)) != WAM_OK) return cleanup(r);
  }
  cudaError_t e = cudaSuccess;
  e = e == cudaSuccess ? cudaMemsetAsync(st->xhist, 0, BT * (c->K + 1) * 4, c->stream) : e;
  e = e == cudaSuccess ? cudaMemsetAsync(st->vhist, 0, BT * c->K * 4, c->stream) : e;
  if (st->pa) {
    e = e == cudaSuccess ? cudaMemsetAsync(st->pa, 0, size_t(batch) * c->N * c->d * 4, c->stream) : e;
    e = e == cudaSuccess ? cudaMemsetAsync(st->ra, 0, size_t(batch) * c->N * c->d * 4, c->stream) : e;
  }
  if (e != cudaSuccess) return cleanup(fail_cuda(c, "state init", e));
  st->meta.assign(batch, EpisodeMeta());
  *out = st;
  return WAM_OK;
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

void wam_state_destroy(wam_state* st) {
  if (st == nullptr) return;
  if (st->ctx) {
    cudaStreamSynchronize(st->ctx->stream);
    resolve_decisions(st->ctx, true);
    for (auto& pd : st->ctx->dec_pending)
      if (pd.st == st) pd.st = nullptr;
    // graphs that embed this state's buffers
    for (auto it = st->ctx->rr_graphs.begin(); it != st->ctx->rr_graphs.end();) {
      if (std::get<0>(it->first) == st->pa) {
        cudaGraphExecDestroy(it->second);
        st->ctx->rr_graph_uses.erase(it->first);
        it = st->ctx->rr_graphs.erase(it);
      } else {
        ++it;
      }
    }
  }
  for (void* p : st->allocs) cudaFree(p);
  delete st;
}

int wam_adapt_state(wam_ctx* c, wam_state* st, const float* new_obs, const int32_t* executed_shift,
                    const int32_t* entry_stage, const float* fresh_noise, int32_t* status_out) try {
  if (c == nullptr || st == nullptr || st->ctx != c) return WAM_ERR_INVALID_ARG;
  if (new_obs == nullptr) return fail(c, WAM_ERR_INVALID_ARG, "new_obs is required");
  const int B = st->B;
  const wam_config& g = c->cfg;
  std::vector<AdaptItem> ad(B);
  std::vector<int32_t> status(B, 0);
  std::vector<EpisodeMeta> meta = st->meta;  // committed only on success
  std::vector<int> rebind;                   // episodes needing the consistency score
  bool need_eps = false, any_tr = false;
  wam_stats dstats;
  std::memset(&dstats, 0, sizeof(dstats));
  for (int b = 0; b < B; ++b) {
    AdaptItem& a = ad[b];
    std::memset(&a, 0, sizeof(a));
    EpisodeMeta& m = meta[b];
    const int shift = executed_shift ? executed_shift[b] : 0;
    const int entry = entry_stage ? entry_stage[b] : g.tr_entry_stage;
    if (shift < 0) return fail(c, WAM_ERR_INVALID_ARG, "executed_shift must be >= 0");
    if (entry == WAM_ENTRY_COLD) {
      a.op = kAdaptCold;
      a.bind_obs = 1;
      need_eps = true;
      m = EpisodeMeta();
      m.stage = 0;
      status[b] = WAM_ADAPT_COLD_INIT;
    } else if (m.finished) {
      const int b0 = entry;
      const int r = g.tr_retain_stage < 0 ? b0 : g.tr_retain_stage;
      if (b0 < 0 || b0 >= c->K) return fail(c, WAM_ERR_INVALID_ARG, "entry stage outside [0, K)");
      if (r < m.hist_from || r >= c->K) return fail(c, WAM_ERR_BAD_STATE, "retained stage not produced by the last replan");
      a.op = kAdaptTR;
      a.shift = shift;
      a.r = r;
      a.sigma_r = c->sigma[r];
      a.sigma_b0 = c->sigma[b0];
      a.bind_obs = 1;
      need_eps = true;
      any_tr = true;
      m.stage = b0;
      m.b0 = b0;
      m.hist_from = b0;
      m.finished = 0;
      m.since_bind = 0;
      m.path = kPathPrefix;
      m.path_steps = 0;
      dstats.n_noninitial++;
      status[b] = m.kappa >= g.or_kappa_max ? WAM_ADAPT_TR_INIT_NO_PREFIX : WAM_ADAPT_TR_INIT;
    } else if (m.stage < 0) {
      return fail(c, WAM_ERR_BAD_STATE, "episode has no state yet (start it cold)");
    } else {
      if (shift != 0) return fail(c, WAM_ERR_BAD_STATE, "rebinding an in-flight replan takes no shift");
      a.bind_obs = 1;
      if (m.since_bind == 0) {
        m.kappa = 0;
        m.path = kPathRefresh;
        m.path_steps = 0;
        status[b] = WAM_ADAPT_REFRESH;
      } else {
        rebind.push_back(b);
      }
    }
  }
  if (need_eps && fresh_noise == nullptr) return fail(c, WAM_ERR_INVALID_ARG, "fresh_noise is required for remapping / cold starts");
  const size_t obs_elems = size_t(c->No) * c->d;
  CK(cudaMemcpyAsync(c->d_obs_new, new_obs, sizeof(float) * obs_elems * B, cudaMemcpyDefault, c->stream));
  if (need_eps) CK(cudaMemcpyAsync(c->d_eps, fresh_noise, sizeof(float) * size_t(B) * c->T, cudaMemcpyDefault, c->stream));
  if (!rebind.empty()) {
    // Eq. 4: weighted RMS of the per-component normalised RMSE between the bound (predicted)
    // condition and the new (real) one; partial sums on the device, combined here in float64.
    const int M = g.or_n_components;
    const int nch = or_num_chunks(int64_t(c->No / M) * c->d);
    float inv_delta[4] = {1.f, 1.f, 1.f, 1.f};
    for (int m = 0; m < M; ++m) inv_delta[m] = 1.0f / g.or_deltas[m];
    {
      Span sp(c, WAM_KCLASS_ADAPT, 0.0, 8.0 * B * obs_elems);
      CK(or_score_partial(st->obs, c->d_obs_new, B, int64_t(obs_elems), M, inv_delta, nch, c->d_part, c->stream));
    }
    std::vector<double> part(size_t(B) * M * nch);
    TRY(readback(c, part.data(), c->d_part, sizeof(double) * part.size()));
    const double comp = double(c->No / M) * c->d;
    for (int b : rebind) {
      double num = 0.0, den = 0.0;
      for (int m = 0; m < M; ++m) {
        double s = 0.0;
        for (int k = 0; k < nch; ++k) s += part[(size_t(b) * M + m) * nch + k];
        const double e2 = s / comp;  // e_m^2
        num += g.or_weights[m] * e2;
        den += g.or_weights[m];
      }
      const double S = std::sqrt(num / den);
      EpisodeMeta& m = meta[b];
      dstats.n_start++;
      if (S < g.or_tau && m.kappa < g.or_kappa_max) {
        m.kappa++;
        m.since_bind = 0;
        dstats.n_bind++;
        status[b] = WAM_ADAPT_REBIND_ACCEPT;
      } else {
        ad[b].op = kAdaptRestart;
        m.stage = m.b0;
        m.kappa = 0;
        m.since_bind = 0;
        m.path = kPathRefresh;
        m.path_steps = 0;
        status[b] = WAM_ADAPT_REBIND_RESTART;
      }
    }
  }
  TRY(upload(c, c->d_adapt, ad.data(), sizeof(AdaptItem) * B));
  const int64_t stage_stride = int64_t(B) * c->T;
  const int nch = tr_num_chunks(c->T, c->V);
  if (any_tr) {
    Span sp(c, WAM_KCLASS_ADAPT, 0.0, 8.0 * B * c->T);
    CK(tr_rms_partial(c->d_adapt, st->xhist, stage_stride, c->K, B, c->T, c->V, nch, c->d_part, c->stream));
  }
  {
    Span sp(c, WAM_KCLASS_ADAPT, 0.0, 16.0 * B * c->T + 8.0 * B * obs_elems);
    CK(adapt_apply(c->d_adapt, c->d_part, nch, st->x, st->xb0, st->xhist, stage_stride, c->K, c->d_eps, c->d_obs_new,
                   st->obs, B, c->T, c->V, c->Na, c->ad, int64_t(obs_elems), g.tr_normalize, g.tr_video_mode, c->stream));
  }
  st->meta = meta;
  c->stats.n_noninitial += dstats.n_noninitial;
  c->stats.n_start += dstats.n_start;
  c->stats.n_bind += dstats.n_bind;
  if (status_out) std::memcpy(status_out, status.data(), sizeof(int32_t) * B);
  return WAM_OK;
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

int wam_continue(wam_ctx* c, wam_state* st, const int32_t* n_steps, float* actions_out, float* video_out) try {
  if (c == nullptr || st == nullptr || st->ctx != c || n_steps == nullptr) return WAM_ERR_INVALID_ARG;
  std::vector<int> n(st->B);
  for (int b = 0; b < st->B; ++b) {
    n[b] = n_steps[b];
    const EpisodeMeta& m = st->meta[b];
    if (n[b] < 0) return fail(c, WAM_ERR_INVALID_ARG, "n_steps must be >= 0");
    if (n[b] == 0) continue;
    if (m.stage < 0 || m.finished) return fail(c, WAM_ERR_BAD_STATE, "episode is not adapted (finished or never started)");
    if (m.stage + n[b] > c->K) return fail(c, WAM_ERR_INVALID_ARG, "stage + n_steps exceeds K");
  }
  TRY(run_steps(c, st, n));
  bool host_out = false;
  TRY(copy_out(c, st, actions_out, video_out, host_out));
  if (host_out) TRY(sync_check(c));
  return WAM_OK;
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

int wam_continue_many(int32_t n, wam_ctx* const* ctxs, wam_state* const* states, const int32_t* const* n_steps,
                      float* const* actions_out, float* const* video_out, int32_t* status_out) try {
  if (n < 1 || ctxs == nullptr || states == nullptr || n_steps == nullptr) return WAM_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i) {
    if (ctxs[i] == nullptr || states[i] == nullptr || states[i]->ctx != ctxs[i] || n_steps[i] == nullptr)
      return WAM_ERR_INVALID_ARG;
    for (int j = 0; j < i; ++j)
      if (ctxs[j] == ctxs[i]) return fail(ctxs[i], WAM_ERR_INVALID_ARG, "a context appears twice");
  }
  std::vector<int> rc(n, WAM_OK);
  auto run = [&](int i) {
    wam_ctx* c = ctxs[i];
    if (cudaSetDevice(c->device) != cudaSuccess) {
      cudaGetLastError();
      rc[i] = fail(c, WAM_ERR_CUDA, "cudaSetDevice failed on a worker thread");
      return;
    }
    rc[i] = wam_continue(c, states[i], n_steps[i], actions_out ? actions_out[i] : nullptr,
                         video_out ? video_out[i] : nullptr);
  };
  // One host thread per context, so the host-side gate decisions of one branch never hold back
  // the launches of another; the GPU overlaps the contexts' streams.
  std::vector<std::thread> workers;
  int spawned = 1;
  try {
    workers.reserve(n - 1);
    for (; spawned < n; ++spawned) workers.emplace_back(run, spawned);
  } catch (...) {
    // no thread available: the rest run on this thread after the spawned ones
  }
  run(0);
  for (auto& t : workers) t.join();
  for (int i = spawned; i < n; ++i) run(i);
  int first = WAM_OK;
  for (int i = 0; i < n; ++i) {
    if (status_out) status_out[i] = rc[i];
    if (first == WAM_OK) first = rc[i];
  }
  return first;
} catch (const std::bad_alloc&) {
  return fail((n > 0 && ctxs != nullptr ? ctxs[0] : nullptr), WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail((n > 0 && ctxs != nullptr ? ctxs[0] : nullptr), WAM_ERR_CUDA, "unexpected host exception");
}

int wam_sample_cold(wam_ctx* c, wam_state* st, const float* obs, const float* noise, int32_t n_steps, float* actions_out) try {
  if (c == nullptr || st == nullptr || st->ctx != c || obs == nullptr || noise == nullptr) return WAM_ERR_INVALID_ARG;
  if (n_steps < 1 || n_steps > c->K) return fail(c, WAM_ERR_INVALID_ARG, "n_steps outside [1, K]");
  std::vector<int32_t> entry(st->B, WAM_ENTRY_COLD);
  TRY(wam_adapt_state(c, st, obs, nullptr, entry.data(), noise, nullptr));
  std::vector<int32_t> n(st->B, n_steps);
  return wam_continue(c, st, n.data(), actions_out, nullptr);
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

int wam_get_stats(wam_ctx* c, wam_stats* out) {
  if (c == nullptr || out == nullptr) return WAM_ERR_INVALID_ARG;
  TRY(resolve_decisions(c, true));
  *out = c->stats;
  return WAM_OK;
}

int wam_reset_stats(wam_ctx* c) {
  if (c == nullptr) return WAM_ERR_INVALID_ARG;
  // decisions of steps already run belong to the counts being cleared
  TRY(queue_decision_copy(c));
  TRY(resolve_decisions(c, true));
  std::memset(&c->stats, 0, sizeof(c->stats));
  return WAM_OK;
}

int wam_state_log(const wam_state* st, wam_step_record* out, int32_t capacity, int32_t* n_out) {
  if (st == nullptr || n_out == nullptr || (capacity > 0 && out == nullptr)) return WAM_ERR_INVALID_ARG;
  if (st->ctx != nullptr) TRY(resolve_decisions(st->ctx, true));
  const int n = std::min<int>(capacity, static_cast<int>(st->log.size()));
  if (n > 0) std::memcpy(out, st->log.data(), sizeof(wam_step_record) * n);
  *n_out = static_cast<int32_t>(st->log.size());
  return WAM_OK;
}

int wam_state_read(wam_ctx* c, const wam_state* st, int32_t field, int32_t index, void* out, size_t n_bytes) try {
  if (c == nullptr || st == nullptr || out == nullptr || st->ctx != c) return WAM_ERR_INVALID_ARG;
  if (field == WAM_FIELD_META) {
    const size_t need = size_t(st->B) * 8 * sizeof(int32_t);
    if (n_bytes != need) return fail(c, WAM_ERR_INVALID_ARG, "META needs B*8 int32");
    int32_t* o = static_cast<int32_t*>(out);
    for (int b = 0; b < st->B; ++b) {
      const EpisodeMeta& m = st->meta[b];
      const int32_t v[8] = {m.stage, m.hist_from, m.b0, m.kappa, m.finished, m.since_bind, m.path, m.rr_valid};
      std::memcpy(o + 8 * b, v, sizeof(v));
    }
    return WAM_OK;
  }
  void* p = nullptr;
  size_t bytes = 0;
  TRY(field_ptr(c, st, field, index, &p, &bytes));
  if (n_bytes != bytes) return fail(c, WAM_ERR_INVALID_ARG, "n_bytes does not match the field size");
  CK(cudaMemcpyAsync(out, p, bytes, cudaMemcpyDefault, c->stream));
  if (!is_device_ptr(out)) TRY(sync_check(c));
  return WAM_OK;
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

int wam_state_write(wam_ctx* c, wam_state* st, int32_t field, int32_t index, const void* in, size_t n_bytes) try {
  if (c == nullptr || st == nullptr || in == nullptr || st->ctx != c) return WAM_ERR_INVALID_ARG;
  if (field == WAM_FIELD_META) {
    const size_t need = size_t(st->B) * 8 * sizeof(int32_t);
    if (n_bytes != need) return fail(c, WAM_ERR_INVALID_ARG, "META needs B*8 int32");
    const int32_t* v = static_cast<const int32_t*>(in);
    for (int b = 0; b < st->B; ++b) {
      const int32_t* e = v + 8 * b;
      if (e[0] < -1 || e[0] > c->K || e[1] < 0 || e[1] > c->K || e[2] < 0 || e[2] >= c->K || e[3] < 0 || e[6] < 0 || e[6] > 2)
        return fail(c, WAM_ERR_INVALID_ARG, "META values out of range");
    }
    for (int b = 0; b < st->B; ++b) {
      const int32_t* e = v + 8 * b;
      EpisodeMeta& m = st->meta[b];
      m.stage = e[0];
      m.hist_from = e[1];
      m.b0 = e[2];
      m.kappa = e[3];
      m.finished = e[4];
      m.since_bind = e[5];
      m.path = e[6];
      m.rr_valid = e[7];
      m.path_steps = 0;
    }
    return WAM_OK;
  }
  void* p = nullptr;
  size_t bytes = 0;
  TRY(field_ptr(c, st, field, index, &p, &bytes));
  if (n_bytes != bytes) return fail(c, WAM_ERR_INVALID_ARG, "n_bytes does not match the field size");
  CK(cudaMemcpyAsync(p, in, bytes, cudaMemcpyDefault, c->stream));
  if (!is_device_ptr(in)) CK(cudaStreamSynchronize(c->stream));
  return WAM_OK;
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

int wam_sync(wam_ctx* c) try {
  if (c == nullptr) return WAM_ERR_INVALID_ARG;
  return sync_check(c);
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

// ------------------------------------------------------------------- diagnostics (App. E)
namespace {

// {a.b, a.a, b.b, (a-b).(a-b)} in float64 over the elements whose column (index mod row_len) is
// below cols; host inputs are staged into the context's scratch first.  Blocks' partials are
// summed on the host in block order.
int diag_sums(wam_ctx* c, const float* a, const float* b, int64_t n, int64_t row_len, int64_t cols, double out[4]) {
  const size_t cap = size_t(c->Bmax) * c->N * c->d;
  if (n <= 0 || size_t(n) > cap) return fail(c, WAM_ERR_INVALID_ARG, "diagnostic length outside [1, batch_max*tokens*d_model]");
  const float* da = a;
  const float* db = b;
  if (!is_device_ptr(a)) {
    CK(cudaMemcpyAsync(c->hq, a, size_t(n) * sizeof(float), cudaMemcpyHostToDevice, c->stream));
    da = c->hq;
  }
  if (!is_device_ptr(b)) {
    CK(cudaMemcpyAsync(c->hm, b, size_t(n) * sizeof(float), cudaMemcpyHostToDevice, c->stream));
    db = c->hm;
  }
  int nb = static_cast<int>(std::min<int64_t>(256, (n + 1023) / 1024));
  nb = std::max(1, std::min<int>(nb, static_cast<int>(c->part_doubles / 4)));
  CK(diag_partial(da, db, n, row_len, cols, nb, c->d_part, c->stream));
  std::vector<double> p(size_t(nb) * 4);
  TRY(readback(c, p.data(), c->d_part, sizeof(double) * p.size()));
  for (int q = 0; q < 4; ++q) out[q] = 0.0;
  for (int i = 0; i < nb; ++i)
    for (int q = 0; q < 4; ++q) out[q] += p[size_t(i) * 4 + q];
  return WAM_OK;
}

}  // namespace

int wam_diag_similarity(wam_ctx* c, const float* a, const float* b, int64_t n, double* cos_out, double* rel_l2_out) try {
  if (c == nullptr || a == nullptr || b == nullptr || cos_out == nullptr || rel_l2_out == nullptr) return WAM_ERR_INVALID_ARG;
  double v[4];
  TRY(diag_sums(c, a, b, n, n, n, v));
  const double na = std::sqrt(v[1]), nb = std::sqrt(v[2]), dist = std::sqrt(v[3]);
  *cos_out = (na > 0.0 && nb > 0.0) ? v[0] / (na * nb) : 0.0;
  *rel_l2_out = nb > 0.0 ? dist / nb : (dist == 0.0 ? 0.0 : HUGE_VAL);
  return WAM_OK;
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

int wam_diag_action_rmse(wam_ctx* c, const float* a, const float* b, int32_t n_rows, int32_t row_len, int32_t dims,
                         double* out) try {
  if (c == nullptr || a == nullptr || b == nullptr || out == nullptr || n_rows <= 0 || row_len <= 0 || dims <= 0 ||
      dims > row_len)
    return WAM_ERR_INVALID_ARG;
  double v[4];
  TRY(diag_sums(c, a, b, int64_t(n_rows) * row_len, row_len, dims, v));
  *out = std::sqrt(v[3] / (double(n_rows) * dims));
  return WAM_OK;
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

}  // extern "C"

namespace {

// Conditioning and token embedding of one episode at its pending stage k into context scratch
// (work item 0: modulations row 0, residual stream c->h); the state itself is not modified (the
// observation embedding is recomputed from the bound observation, which it derives from).
int diag_embed_item(wam_ctx* c, wam_state* st, int episode) {
  const int k = st->meta[episode].stage;
  const int d = c->d;
  StepItem it;
  it.ep = episode;
  it.stage = k;
  it.sigma = c->sigma[k];
  it.dsigma = c->sigma[k + 1] - c->sigma[k];
  TRY(upload(c, c->d_items, &it, sizeof(StepItem)));
  TRY(obs_embed(c, st));
  {
    const CondGemv g{nullptr, 0, nullptr, 0, 1, c->d_items, c->t_w1, false, 256, d, 1, kT1Splits, c->t1, nullptr};
    CK(cond_gemv(g, c->stream));
  }
  {
    const CondGemv g{c->t1, kT1Splits, c->t_b1, 1, 0, c->d_items, c->t_w2, false, d, d, 1, kT2Splits, c->cvec, nullptr};
    CK(cond_gemv(g, c->stream));
  }
  {
    const CondGemv g{c->cvec, kT2Splits, c->t_b2, 1, 0, c->d_items, c->mod_w, c->bf16, d, static_cast<int>(c->mod_n),
                     1, 1, c->mods, c->mod_b};
    CK(cond_gemv(g, c->stream));
  }
  // the embedding records the latent it reads: point that record at scratch (stage stride 0)
  CK(embed_tokens(c->h, c->hq, 0, c->d_items, st->x, c->T, st->obs_emb, c->vid_w, c->vid_b, c->act_w, c->act_b,
                  c->pos, 1, c->No, c->Nv, c->vd, c->Na, c->ad, d, c->stream));
  return WAM_OK;
}

// Output head + Euler kernel of work item 0 written to scratch only: x, x^{k+1} and v^k of a
// stand-in item (episode 0, stage 0, stage stride 0) in three separate T-float buffers, the
// velocity ending in `v_out`.
int diag_final(wam_ctx* c, const float* hb, float* x_scratch, float* xn_scratch, float* v_out) {
  StepItem s;
  s.ep = 0;
  s.stage = 0;
  s.sigma = 0.0;
  s.dsigma = 0.0;
  TRY(upload(c, c->d_uitems, &s, sizeof(StepItem)));
  CK(final_euler(hb, c->d_uitems, c->mods, c->mod_n, 6 * c->L * c->d, c->vout_w, c->vout_b, c->aout_w, c->aout_b,
                 x_scratch, xn_scratch, v_out, 0, c->T, 1, c->No, c->Nv, c->vd, c->Na, c->ad, c->d, c->bf16, c->d_fhead,
                 c->d_fconst, c->stream));
  return WAM_OK;
}

}  // namespace

extern "C" {

int wam_diag_layer_deltas(wam_ctx* c, wam_state* st, int32_t episode, double* out) try {
  if (c == nullptr || st == nullptr || st->ctx != c || out == nullptr || episode < 0 || episode >= st->B)
    return WAM_ERR_INVALID_ARG;
  const int k = st->meta[episode].stage;
  if (k < 0 || k >= c->K) return fail(c, WAM_ERR_BAD_STATE, "the episode has no pending denoising stage");
  const int d = c->d, N = c->N;
  TRY(diag_embed_item(c, st, episode));
  for (int l = 0; l < c->L; ++l) {
    CK(cudaMemcpyAsync(c->hm, c->h, size_t(N) * d * sizeof(float), cudaMemcpyDeviceToDevice, c->stream));
    TRY(run_layer(c, l, c->h, 1, nullptr, nullptr));
    double v[4];
    TRY(diag_sums(c, c->h, c->hm, int64_t(N) * d, int64_t(N) * d, int64_t(N) * d, v));
    out[l] = std::sqrt(v[3]) / std::sqrt(v[2]);
  }
  return WAM_OK;
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

int wam_diag_reuse_error(wam_ctx* c, wam_state* st, int32_t episode, double* e_out, double* alpha_out) try {
  if (c == nullptr || st == nullptr || st->ctx != c || e_out == nullptr || episode < 0 || episode >= st->B)
    return WAM_ERR_INVALID_ARG;
  const int k = st->meta[episode].stage;
  if (k < 0 || k >= c->K) return fail(c, WAM_ERR_BAD_STATE, "the episode has no pending denoising stage");
  const wam_config& g = c->cfg;
  if (!(0 < g.rr_q && g.rr_q < g.rr_s && g.rr_s < g.rr_e && g.rr_e < g.n_layers))
    return fail(c, WAM_ERR_INVALID_ARG, "the profile has no RR layer boundaries 0 < q < s < e < n_layers");
  if (!st->meta[episode].rr_valid) return fail(c, WAM_ERR_BAD_STATE, "the episode has no retained layer state");
  const int d = c->d, N = c->N, L = c->L, T = c->T;
  const int q = g.rr_q, s = g.rr_s, e = g.rr_e;
  const int split_row = c->split;
  TRY(diag_embed_item(c, st, episode));
  // head and probe layers: h = h_s, hq = h_q
  for (int l = 0; l < s; ++l) TRY(run_layer(c, l, c->h, 1, nullptr, l == q ? c->hq : nullptr));
  // Eq. 7 factors against the retained probe residual (the Eq. 8 checks are not applied)
  const int nch = rr_num_chunks(int64_t(std::max(split_row, N - split_row)) * d);
  CK(rr_probe_partial(c->h, c->hq, st->pa, c->d_items, 1, N, d, split_row, nch, c->d_part, c->stream));
  CK(rr_gate(c->d_part, 1, nch, int64_t(split_row) * d, int64_t(N - split_row) * d, g.rr_alpha_min, g.rr_alpha_max,
             g.rr_eps, g.rr_gamma_cos, g.rr_gamma_fit, c->d_gate, c->stream));
  RRGate gates[2];
  TRY(readback(c, gates, c->d_gate, sizeof(gates)));
  // velocity scratch: three T-float buffers for each pass, past the h_q rows no longer needed
  float* xs = c->d_eps;
  float* full_v = c->hq;
  float* full_xn = c->hq + T;
  float* reuse_v = c->hq + 2 * T;
  // full computation: middle and tail layers on a copy of h_s
  CK(cudaMemcpyAsync(c->hm, c->h, size_t(N) * d * sizeof(float), cudaMemcpyDeviceToDevice, c->stream));
  for (int l = s; l < L; ++l) TRY(run_layer(c, l, c->hm, 1, nullptr, nullptr));
  TRY(diag_final(c, c->hm, xs, full_xn, full_v));
  // reuse: h_e = h_s + alpha R_a per branch (Eq. 9), then the tail layers
  RRApply ap;
  ap.mode = kRRInject;
  ap.cidx = 0;
  ap.alpha0 = static_cast<float>(gates[0].alpha);
  ap.alpha1 = static_cast<float>(gates[1].alpha);
  TRY(upload(c, c->d_rrapply, &ap, sizeof(RRApply)));
  CK(rr_apply(c->h, c->hm, c->hq, st->pa, st->ra, c->d_items, c->d_rrapply, 1, N, d, split_row, c->stream));
  for (int l = e; l < L; ++l) TRY(run_layer(c, l, c->h, 1, nullptr, nullptr));
  TRY(diag_final(c, c->h, xs, full_xn, reuse_v));
  double v[4];
  TRY(diag_sums(c, reuse_v, full_v, T, T, T, v));
  *e_out = std::sqrt(v[3]) / std::sqrt(v[2]);
  if (alpha_out != nullptr) {
    alpha_out[0] = split_row == 0 ? 0.0 : gates[0].alpha;
    alpha_out[1] = split_row == N ? 0.0 : gates[1].alpha;
  }
  return WAM_OK;
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

int wam_set_graph_replay(wam_ctx* c, int32_t enable) {
  if (c == nullptr) return WAM_ERR_INVALID_ARG;
  c->graph_replay = enable != 0;
  return WAM_OK;
}

int wam_set_device_branching(wam_ctx* c, int32_t enable) {
  if (c == nullptr) return WAM_ERR_INVALID_ARG;
  c->dev_branch = enable != 0;
  return WAM_OK;
}

int wam_set_layer_fusion(wam_ctx* c, int32_t enable) {
  if (c == nullptr) return WAM_ERR_INVALID_ARG;
  c->layer_fusion = enable != 0;
  return WAM_OK;
}

int wam_gemm_tile_width(const wam_ctx* c, int32_t M, int32_t N, int32_t K, int32_t epilogue) {
  if (c == nullptr || M < 0 || N <= 0 || K <= 0) return WAM_ERR_INVALID_ARG;
  if (!c->bf16) return WAM_ERR_UNSUPPORTED;
  // 64-wide tiles for the residual projections (measured faster there at small M), 64-row weight
  // boxes for every projection (128-wide CTA pairs)
  return tc_gemm_plan(M, N, K, epilogue == kEpiResidF32, true, c->num_sms).bn;
}

int wam_profile_enable(wam_ctx* c, int32_t enable) try {
  if (c == nullptr) return WAM_ERR_INVALID_ARG;
  CK(cudaStreamSynchronize(c->stream));
  c->spans.clear();
  c->evnext = 0;
  c->prof_on = enable != 0;
  if (c->prof_on && c->chain_ok && c->d_trace == nullptr) {
    constexpr int kTraceRecords = 1 << 18;   // 16 MB of task records
    TRY(dalloc(c, c->allocs, &c->d_trace, kTraceRecords));
    c->trace_cap = kTraceRecords;
  }
  if (c->d_trace != nullptr) CK(cudaMemsetAsync(c->d_trace, 0, sizeof(wam_chain_task) * c->trace_cap, c->stream));
  c->trace_used = 0;
  c->trace_launches = 0;
  return WAM_OK;
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

int wam_profile_chain_trace(wam_ctx* c, wam_chain_task* out, int32_t capacity, int32_t* n_out) try {
  if (c == nullptr || n_out == nullptr || (out == nullptr && capacity > 0) || capacity < 0) return WAM_ERR_INVALID_ARG;
  CK(cudaStreamSynchronize(c->stream));
  const int n = std::min(capacity, c->trace_used);
  if (n > 0) CK(cudaMemcpy(out, c->d_trace, sizeof(wam_chain_task) * n, cudaMemcpyDeviceToHost));
  *n_out = capacity == 0 ? c->trace_used : n;
  return WAM_OK;
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

int wam_profile_read(wam_ctx* c, wam_kclass_timing* out) try {
  if (c == nullptr || out == nullptr) return WAM_ERR_INVALID_ARG;
  CK(cudaStreamSynchronize(c->stream));
  for (int k = 0; k < WAM_KCLASS_COUNT; ++k) out[k] = wam_kclass_timing{0, 0.0, 0.0, 0.0};
  for (const ProfSpan& s : c->spans) {
    float ms = 0.0f;
    CK(cudaEventElapsedTime(&ms, s.a, s.b));
    wam_kclass_timing& t = out[s.kclass];
    t.launches++;
    t.ms += ms;
    t.flops += s.flops;
    t.bytes += s.bytes;
  }
  return WAM_OK;
} catch (const std::bad_alloc&) {
  return fail(c, WAM_ERR_OOM, "host allocation failed");
} catch (...) {
  return fail(c, WAM_ERR_CUDA, "unexpected host exception");
}

}  // extern "C"
